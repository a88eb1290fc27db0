// Single-token decode GQA attention over the retained cache.
//
// For each session of the last append (one token each), each KV head h and
// its G = 4 query heads: out = softmax(RoPE(q, p) . k / sqrt(D)) v over every
// resident key (the compacted region, then the live region, the token's own
// key included).
//
// Inside a CTA each of the 4 warps streams its own pages through a TMA
// bulk-copy ring in shared memory, computes scores on CUDA cores (packed fp32
// FMA), keeps a running max/sum with warp shuffles, and the CTA merges its
// warps.  Two ways to spread the pages over CTAs (split-K):
//   - stream-K (many sessions): the call's (session, head, page) units are cut
//     into equal contiguous ranges, one per CTA; partial results go to global
//     slots and the last CTA to arrive for a pair merges them (log-sum-exp);
//   - clusters (few sessions): each (session, head) pair gets a cluster of
//     CTAs that split its pages; the partial states are merged through
//     distributed shared memory, with no global partials or atomics.
#include <cooperative_groups.h>

#include "kvc_internal.cuh"

namespace cg = cooperative_groups;

namespace kvc {

namespace {

constexpr unsigned FULL = 0xFFFFFFFFu;
constexpr int DEC_WARPS = 4;
constexpr int DEC_THREADS = DEC_WARPS * 32;
constexpr int G = 4;  // query heads per KV head
static_assert(DEC_WARPS == G, "the split-K merge maps one warp to one query row");
constexpr float LOG2E = 1.4426950408889634f;
constexpr int STAGES = 2;         // per-warp K/V ring depth
constexpr int MAX_PARTS = 64;     // stream-K parts per (session, head), merge buffer size

template <typename T, int D>
struct DecCfg {
  static constexpr int ESZ = sizeof(T);
  static constexpr int ROW_BYTES = D * ESZ;
  static_assert(ROW_BYTES == 256, "decode kernel assumes 256-byte K/V rows");
  static constexpr int VEC = 16 / ESZ;     // elements per 16-byte lane chunk (QK)
  static constexpr int PVD = D / 32;       // dims per lane (PV)
  static constexpr int TILE = PS * ROW_BYTES;  // one page of one head: 4 KiB
  // shared memory per warp: STAGES x (K tile + V tile) + scores + probability
  // pairs (p, p) + alpha
  static constexpr int WARP_BYTES = STAGES * 2 * TILE + (G * PS + 2 * PS * G + G) * 4 + 16;
  // The cross-warp merge (and the CTA result) reuse the stage buffers once every
  // warp is done with its pages.
  static constexpr int MERGE_FLOATS = DEC_WARPS * G * D + DEC_WARPS * G * 2;
  static constexpr int RESULT_FLOATS = G * D + G * 2;
  static_assert((MERGE_FLOATS + RESULT_FLOATS) * 4 <= DEC_WARPS * WARP_BYTES,
                "merge area must fit in the stages");
  static constexpr int SMEM = DEC_WARPS * WARP_BYTES + DEC_WARPS * STAGES * 8 +
                              MAX_PARTS * G * 4 + 64;
};

template <typename T>
__device__ inline void load_vec(const uint8_t* p, float* f);
template <>
__device__ inline void load_vec<__nv_bfloat16>(const uint8_t* p, float* f) {
  const uint4 w = *reinterpret_cast<const uint4*>(p);
  f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
  f[4] = bf16lo(w.z); f[5] = bf16hi(w.z); f[6] = bf16lo(w.w); f[7] = bf16hi(w.w);
}
template <>
__device__ inline void load_vec<float>(const uint8_t* p, float* f) {
  const float4 w = *reinterpret_cast<const float4*>(p);
  f[0] = w.x; f[1] = w.y; f[2] = w.z; f[3] = w.w;
}

template <typename T>
__device__ inline void load_pv(const uint8_t* p, float* f);
template <>
__device__ inline void load_pv<__nv_bfloat16>(const uint8_t* p, float* f) {
  const uint2 w = *reinterpret_cast<const uint2*>(p);
  f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
}
template <>
__device__ inline void load_pv<float>(const uint8_t* p, float* f) {
  const float2 w = *reinterpret_cast<const float2*>(p);
  f[0] = w.x; f[1] = w.y;
}

// Shared-memory map of one CTA, as seen by one warp.
template <typename T, int D>
struct Smem {
  using C = DecCfg<T, D>;
  uint8_t* tiles;     // this warp's [STAGES][2][TILE]
  float* s_sc;        // [G][PS] scores
  float2* s_p2;       // [PS][G] probability pairs (p, p)
  float* s_alpha;     // [G]
  float* m_o;         // [W][G][D] warp partial outputs (aliases the stages)
  float* m_ml;        // [W][G][2]
  float* r_o;         // [G][D] CTA result (aliases the stages)
  float* r_ml;        // [G][2]
  uint64_t* wbars;    // this warp's [STAGES]
  float* s_scale;     // [MAX_PARTS][G]
  __device__ Smem(uint8_t* smem, int warp) {
    uint8_t* wbase = smem + warp * C::WARP_BYTES;
    tiles = wbase;
    s_sc = reinterpret_cast<float*>(wbase + STAGES * 2 * C::TILE);
    s_p2 = reinterpret_cast<float2*>(s_sc + G * PS);
    s_alpha = reinterpret_cast<float*>(s_p2 + PS * G);
    m_o = reinterpret_cast<float*>(smem);
    m_ml = m_o + DEC_WARPS * G * D;
    r_o = m_ml + DEC_WARPS * G * 2;
    r_ml = r_o + G * D;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + DEC_WARPS * C::WARP_BYTES);
    wbars = bars + warp * STAGES;
    s_scale = reinterpret_cast<float*>(bars + DEC_WARPS * STAGES);
  }
};

// Blocks [blk_begin, blk_begin + nblk) of one (session, head) pair; warp w takes
// blocks blk_begin + w, + w + 4, ...  Page ids are fetched 32 at a time (lane j
// holds the id of the warp's block win + j), so one round trip serves 32 loads.
template <typename T, int D>
struct Segment {
  using C = DecCfg<T, D>;
  SeqInfo si;
  int head, blk_begin, nblk, n_my;
  const int32_t* hrow;
  const int32_t* lrow;
  int pwin, pid;

  __device__ void init(const Dev& d, const SeqInfo& s, int h, int b0, int nb, int warp) {
    si = s;
    head = h;
    blk_begin = b0;
    nblk = nb;
    n_my = (nblk > warp) ? (nblk - warp + DEC_WARPS - 1) / DEC_WARPS : 0;
    hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    pwin = -32;
    pid = 0;
  }

  // Load the K and V tiles of this warp's k-th block (called by the whole warp).
  __device__ void issue(const Dev& d, int layer, const Smem<T, D>& sm, uint32_t loads, int k,
                        int warp, int lane) {
    if (k >= pwin + 32) {
      pwin = k & ~31;
      const int j = pwin + lane;
      pid = j < n_my ? block_page(si, hrow, lrow, blk_begin + warp + j * DEC_WARPS) : 0;
    }
    const int page = __shfl_sync(FULL, pid, k - pwin);
    if (lane == 0) {
      const uint32_t n = loads + k;
      const int st = n % STAGES;
      uint8_t* dst = sm.tiles + st * 2 * C::TILE;
      const T* kp = reinterpret_cast<const T*>(d.pool) +
                    pool_offset_elems(d, page, layer, 0, head, 0);
      mbar_arrive_expect_tx(&sm.wbars[st], 2 * C::TILE);
      bulk_g2s(dst, kp, C::TILE, &sm.wbars[st]);
      bulk_g2s(dst + C::TILE, kp + (size_t)d.kv_heads * PS * D, C::TILE, &sm.wbars[st]);
    }
  }

  __device__ void prefetch(const Dev& d, int layer, const Smem<T, D>& sm, uint32_t loads,
                           int warp, int lane) {
    // The stage buffers may have been written by the previous merge.
    if (lane == 0) fence_proxy_async_smem();
    for (int k = 0; k < min(STAGES, n_my); ++k) issue(d, layer, sm, loads, k, warp, lane);
  }
};

// Query rows of the G heads of `head`, rotated at the token's position and scaled
// by log2(e)/sqrt(D).  Lane c holds 16-byte chunk c of each row; its rotate-half
// partner is chunk c ^ 8.
template <typename T, int D>
__device__ void load_q(const Dev& d, const SeqInfo& si, int head, const T* q, float qk_scale,
                       int lane, float (&qr)[G][DecCfg<T, D>::VEC]) {
  using C = DecCfg<T, D>;
  const int c = lane & 15;
  const uint8_t* qrow =
      reinterpret_cast<const uint8_t*>(q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G) * D);
  const float2* cs = d.rope + (size_t)si.pos_first * (D / 2) + (c & 7) * C::VEC;
  const bool lo = c < 8;
  float2 t[C::VEC];
#pragma unroll
  for (int e = 0; e < C::VEC; ++e) t[e] = cs[e];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float x[C::VEC], y[C::VEC];
    load_vec<T>(qrow + g * C::ROW_BYTES + c * 16, x);
    load_vec<T>(qrow + g * C::ROW_BYTES + (c ^ 8) * 16, y);
#pragma unroll
    for (int e = 0; e < C::VEC; ++e)
      qr[g][e] = (lo ? fmaf(x[e], t[e].x, -y[e] * t[e].y) : fmaf(x[e], t[e].x, y[e] * t[e].y)) *
                 qk_scale;
  }
}

// Stream this warp's blocks of the segment: scores, online softmax, P V.  The first
// STAGES blocks must have been issued (Segment::prefetch).  Returns the first block
// whose wait gave up, or -1.
template <typename T, int D>
__device__ int stream_pages(const Dev& d, int layer, Segment<T, D>& sg, const Smem<T, D>& sm,
                            uint32_t loads, const float (&qr)[G][DecCfg<T, D>::VEC],
                            float& m_run, float& l_run, float2 (&acc)[G][DecCfg<T, D>::PVD / 2],
                            int warp, int lane) {
  using C = DecCfg<T, D>;
  const int half = lane >> 4, c = lane & 15;
  for (int k = 0; k < sg.n_my; ++k) {
    const uint32_t n = loads + k;
    const int st = n % STAGES;
    if (!__all_sync(FULL, mbar_wait(d, &sm.wbars[st], (n / STAGES) & 1))) return k;
    const uint8_t* kt = sm.tiles + st * 2 * C::TILE;
    const uint8_t* vt = kt + C::TILE;
    const BlockRange br = block_range(sg.si, sg.blk_begin + warp + k * DEC_WARPS);

    // Scores: lanes 0-15 take even keys, 16-31 odd keys; each lane a 16-byte chunk.
#pragma unroll
    for (int i = 0; i < PS / 2; ++i) {
      const int key = 2 * i + half;
      float kf[C::VEC];
      load_vec<T>(kt + key * C::ROW_BYTES + c * 16, kf);
      float a[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        // Even and odd dims accumulate in the two halves of a packed pair.
        float2 acc2 = make_float2(0.f, 0.f);
#pragma unroll
        for (int e = 0; e < C::VEC; e += 2)
          acc2 = __ffma2_rn(make_float2(qr[g][e], qr[g][e + 1]), make_float2(kf[e], kf[e + 1]),
                            acc2);
        a[g] = acc2.x + acc2.y;
      }
      // Reduce-scatter of 4 sums over 16 lanes, then all-reduce over 4.
      const bool up8 = lane & 8;
      const float r0 = __shfl_xor_sync(FULL, up8 ? a[0] : a[2], 8);
      const float r1 = __shfl_xor_sync(FULL, up8 ? a[1] : a[3], 8);
      const float b0 = (up8 ? a[2] : a[0]) + r0;
      const float b1 = (up8 ? a[3] : a[1]) + r1;
      const bool up4 = lane & 4;
      float v = (up4 ? b1 : b0) + __shfl_xor_sync(FULL, up4 ? b0 : b1, 4);
      v += __shfl_xor_sync(FULL, v, 2);
      v += __shfl_xor_sync(FULL, v, 1);
      if ((lane & 3) == 0) {
        const int g = (up8 ? 2 : 0) + (up4 ? 1 : 0);
        sm.s_sc[g * PS + key] = (key >= br.lo && key < br.hi) ? v : -INFINITY;
      }
    }
    __syncwarp();
    // Online softmax: lane handles row lane>>3, keys 2*(lane&7) and +1.
    {
      const int g = lane >> 3, kk = (lane & 7) * 2;
      const float s0 = sm.s_sc[g * PS + kk], s1 = sm.s_sc[g * PS + kk + 1];
      float mx = fmaxf(s0, s1);
      mx = fmaxf(mx, __shfl_xor_sync(FULL, mx, 4));
      mx = fmaxf(mx, __shfl_xor_sync(FULL, mx, 2));
      mx = fmaxf(mx, __shfl_xor_sync(FULL, mx, 1));
      const float m_new = fmaxf(m_run, mx);
      const float p0 = exp2_safe(s0, m_new), p1 = exp2_safe(s1, m_new);
      const float alpha = exp2_safe(m_run, m_new);
      float rs = p0 + p1;
      rs += __shfl_xor_sync(FULL, rs, 4);
      rs += __shfl_xor_sync(FULL, rs, 2);
      rs += __shfl_xor_sync(FULL, rs, 1);
      l_run = l_run * alpha + rs;
      m_run = m_new;
      sm.s_p2[kk * G + g] = make_float2(p0, p0);
      sm.s_p2[(kk + 1) * G + g] = make_float2(p1, p1);
      if ((lane & 7) == 0) sm.s_alpha[g] = alpha;
    }
    __syncwarp();
    // PV: lane owns dims [PVD*lane, PVD*lane + PVD) of all G rows, as packed pairs.
    {
      const float4 al = *reinterpret_cast<const float4*>(sm.s_alpha);
      const float alv[G] = {al.x, al.y, al.z, al.w};
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int j = 0; j < C::PVD / 2; ++j)
          acc[g][j] = __fmul2_rn(acc[g][j], make_float2(alv[g], alv[g]));
#pragma unroll
      for (int key = 0; key < PS; ++key) {
        const float4 p01 = *reinterpret_cast<const float4*>(sm.s_p2 + key * G);
        const float4 p23 = *reinterpret_cast<const float4*>(sm.s_p2 + key * G + 2);
        const float2 pp[G] = {make_float2(p01.x, p01.y), make_float2(p01.z, p01.w),
                              make_float2(p23.x, p23.y), make_float2(p23.z, p23.w)};
        float vf[C::PVD];
        load_pv<T>(vt + key * C::ROW_BYTES + lane * C::PVD * C::ESZ, vf);
#pragma unroll
        for (int j = 0; j < C::PVD / 2; ++j) {
          const float2 v2 = make_float2(vf[2 * j], vf[2 * j + 1]);
#pragma unroll
          for (int g = 0; g < G; ++g) acc[g][j] = __ffma2_rn(pp[g], v2, acc[g][j]);
        }
      }
    }
    __syncwarp();
    if (k + STAGES < sg.n_my) {
      if (lane == 0) fence_proxy_async_smem();
      sg.issue(d, layer, sm, loads, k + STAGES, warp, lane);
    }
  }
  return -1;
}

// After every warp of the CTA has finished (caller syncs): publish the warps'
// partial states; after a second sync, merge_elem gives the CTA's (M, L, O) of
// element e = g * D + dd.
template <typename T, int D>
__device__ void publish_warp(const Smem<T, D>& sm, float m_run, float l_run,
                             const float2 (&acc)[G][DecCfg<T, D>::PVD / 2], int warp, int lane) {
  using C = DecCfg<T, D>;
  if ((lane & 7) == 0) {
    sm.m_ml[(warp * G + (lane >> 3)) * 2 + 0] = m_run;
    sm.m_ml[(warp * G + (lane >> 3)) * 2 + 1] = l_run;
  }
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int j = 0; j < C::PVD / 2; ++j)
      *reinterpret_cast<float2*>(&sm.m_o[(warp * G + g) * D + lane * C::PVD + 2 * j]) = acc[g][j];
}

template <typename T, int D>
__device__ void merge_elem(const Smem<T, D>& sm, int e, float& M, float& L, float& O) {
  const int g = e / D, dd = e % D;
  float mw[DEC_WARPS];
  M = -INFINITY;
#pragma unroll
  for (int w = 0; w < DEC_WARPS; ++w) {
    mw[w] = sm.m_ml[(w * G + g) * 2];
    M = fmaxf(M, mw[w]);
  }
  L = 0.f;
  O = 0.f;
#pragma unroll
  for (int w = 0; w < DEC_WARPS; ++w) {
    const float sc = exp2_safe(mw[w], M);
    L += sm.m_ml[(w * G + g) * 2 + 1] * sc;
    O += sm.m_o[(w * G + g) * D + dd] * sc;
  }
}

__device__ inline void init_warp_barriers(uint64_t* wbars, int lane) {
  if (lane == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(&wbars[s], 1);
    fence_mbar_init();
  }
}

// ---------------------------------------------------------------------------
// Stream-K kernel.
// ---------------------------------------------------------------------------
template <typename T, int D>
__global__ void __launch_bounds__(DEC_THREADS) attn_decode_kernel(Dev d, int layer,
                                                                  const T* __restrict__ q,
                                                                  T* __restrict__ out,
                                                                  float qk_scale, int min_units) {
  using C = DecCfg<T, D>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const Smem<T, D> sm(smem, warp);
  __shared__ int s_last, s_abort;
  init_warp_barriers(sm.wbars, lane);
  if (tid == 0) s_abort = 0;
  __syncthreads();
  // The next attention call may start its CTAs as soon as slots free up.  Before
  // pdl_wait() this kernel reads only what the append wrote (work list, page
  // tables, K/V pages); q, outputs, partials and counters come after it.
  pdl_launch_dependents();
  bool waited = false;

  // The call's (session, KV head, page) units, session-major, are cut into n_cta
  // equal contiguous ranges, one per CTA.  A range covers "segments" (the part of
  // one (session, head) pair inside it); only its first and last segments can be
  // partial, and they go to partial slots 2c and 2c+1.
  const int H = d.kv_heads;
  const int U = d.g->n_dec_items;  // units of this call
  const int n_seq = d.g->n_seq;
  // n_cta: at most the grid, at least min_units units per CTA, and small enough that
  // no (session, head) pair spans more than MAX_PARTS CTAs (the merge's buffer).
  const int nb_max = max(1, d.g->dec_nb_max);
  const int c_parts = (int)((int64_t)U * (MAX_PARTS - 2) / (nb_max + MAX_PARTS - 2));
  const int n_cta = max(1, min((int)gridDim.x, min((U + min_units - 1) / min_units, c_parts)));
  if ((int)blockIdx.x >= n_cta) return;
  const int cta = blockIdx.x;
  auto start_of = [&](int cc) { return (int)((int64_t)cc * U / n_cta); };
  auto owner = [&](int64_t u) { return (int)(((u + 1) * n_cta - 1) / U); };
  const int u_begin = start_of(cta), u_end = start_of(cta + 1);
  uint32_t loads = 0;  // loads issued (== consumed) by this warp so far

  for (int u = u_begin; u < u_end;) {
    // Session of unit u: the last one whose first unit is <= u.
    int lo = 0, hi = n_seq - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (d.seq[mid].dec_base <= u) lo = mid; else hi = mid - 1;
    }
    const int seq = lo;
    const SeqInfo si = d.seq[seq];
    const int nb = si.n_blocks;
    const int head = (u - si.dec_base) / nb;
    const int pair_start = si.dec_base + head * nb, pair_end = pair_start + nb;
    const int seg_end = min(u_end, pair_end);

    Segment<T, D> sg;
    sg.init(d, si, head, u - pair_start, seg_end - u, warp);
    sg.prefetch(d, layer, sm, loads, warp, lane);
    if (!waited) {
      pdl_wait();
      waited = true;
    }
    float qr[G][C::VEC];
    load_q<T, D>(d, si, head, q, qk_scale, lane, qr);
    float m_run = -INFINITY, l_run = 0.f;  // for row lane >> 3
    float2 acc[G][C::PVD / 2];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < C::PVD / 2; ++j) acc[g][j] = make_float2(0.f, 0.f);
    const int failed_at = stream_pages<T, D>(d, layer, sg, sm, loads, qr, m_run, l_run, acc,
                                             warp, lane);
    if (failed_at >= 0 && lane == 0) s_abort = 1;
    __syncthreads();
    if (s_abort) {
      // Some wait gave up: each warp drains the copies it still has in flight
      // (bounded waits), then the whole CTA stops together.
      if (failed_at >= 0) {
        for (int k = failed_at; k < min(sg.n_my, failed_at + STAGES); ++k) {
          const uint32_t n = loads + k;
          mbar_wait(d, &sm.wbars[n % STAGES], (n / STAGES) & 1);
        }
      }
      return;
    }
    loads += sg.n_my;

    // Merge the four warps' partial softmax states (stage buffers are free now).
    publish_warp<T, D>(sm, m_run, l_run, acc, warp, lane);
    __syncthreads();
    const bool whole = u == pair_start && seg_end == pair_end;
    const int slot = 2 * cta + (u == u_begin ? 0 : 1);
    for (int e = tid; e < G * D; e += DEC_THREADS) {
      float M, L, O;
      merge_elem<T, D>(sm, e, M, L, O);
      const int g = e / D, dd = e % D;
      if (whole) {
        out[((size_t)si.q_row0 * d.q_heads + head * G + g) * D + dd] = from_float<T>(O / L);
      } else {
        d.dec_part_o[((size_t)slot * G + g) * D + dd] = O;
        if (dd == 0) d.dec_part_ml[(size_t)slot * G + g] = make_float2(M, L);
      }
    }
    if (!whole) {
      // The CTAs cf..cl own the pair's units; the last of them to arrive merges.
      const int cf = owner(pair_start), cl = owner(pair_end - 1);
      const int nch = cl - cf + 1;
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int old = atomicAdd(&d.dec_count[seq * H + head], 1);
        s_last = (old == nch - 1);
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        // Slot of CTA cc's part of this pair: its first segment (2cc) unless the
        // pair began inside cf's range after its first unit (then 2cf+1).
        const int first_slot = start_of(cf) != pair_start ? 2 * cf + 1 : 2 * cf;
        auto slot_of = [&](int cc) { return cc == cf ? first_slot : 2 * cc; };
        // Log-sum-exp merge: warp g reduces row g's maxima and sums over the parts,
        // leaving each part's weight divided by the total in shared memory; then all
        // threads sum the weighted partial outputs with independent loads in flight.
        {
          const int g = warp;  // DEC_WARPS == G
          float M = -INFINITY;
          for (int ch = lane; ch < nch; ch += 32)
            M = fmaxf(M, __ldcg(&d.dec_part_ml[(size_t)slot_of(cf + ch) * G + g]).x);
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(FULL, M, o));
          float L = 0.f;
          for (int ch = lane; ch < nch; ch += 32) {
            const float2 ml = __ldcg(&d.dec_part_ml[(size_t)slot_of(cf + ch) * G + g]);
            const float sc = exp2_safe(ml.x, M);
            sm.s_scale[ch * G + g] = sc;
            L += ml.y * sc;
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(FULL, L, o);
          const float inv = 1.f / L;
          __syncwarp();
          for (int ch = lane; ch < nch; ch += 32) sm.s_scale[ch * G + g] *= inv;
        }
        __syncthreads();
        constexpr int EPT = G * D / DEC_THREADS;
        float O[EPT];
#pragma unroll
        for (int i = 0; i < EPT; ++i) O[i] = 0.f;
        // Eight parts per iteration: 8 x EPT independent loads in flight per thread.
        int ch = 0;
        for (; ch + 8 <= nch; ch += 8) {
          float a[8][EPT];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float* b = d.dec_part_o + (size_t)slot_of(cf + ch + k) * G * D;
#pragma unroll
            for (int i = 0; i < EPT; ++i) a[k][i] = __ldcg(b + tid + i * DEC_THREADS);
          }
#pragma unroll
          for (int k = 0; k < 8; ++k)
#pragma unroll
            for (int i = 0; i < EPT; ++i)
              O[i] += a[k][i] * sm.s_scale[(ch + k) * G + (tid + i * DEC_THREADS) / D];
        }
        for (; ch < nch; ++ch) {
          const float* b0 = d.dec_part_o + (size_t)slot_of(cf + ch) * G * D;
#pragma unroll
          for (int i = 0; i < EPT; ++i) {
            const int g = (tid + i * DEC_THREADS) / D;
            O[i] += __ldcg(b0 + tid + i * DEC_THREADS) * sm.s_scale[ch * G + g];
          }
        }
#pragma unroll
        for (int i = 0; i < EPT; ++i) {
          const int e = tid + i * DEC_THREADS;
          out[((size_t)si.q_row0 * d.q_heads + head * G) * D + e] = from_float<T>(O[i]);
        }
        if (tid == 0) d.dec_count[seq * H + head] = 0;
      }
    }
    __syncthreads();
    u = seg_end;
  }
}

// ---------------------------------------------------------------------------
// Cluster kernel: one cluster of CTAs per (session, head) pair; rank r takes
// the r-th of `csize` equal slices of the pair's pages.  The CTA results are
// merged by rank 0 through distributed shared memory.
// ---------------------------------------------------------------------------
template <typename T, int D>
__global__ void __launch_bounds__(DEC_THREADS) attn_decode_cluster_kernel(
    Dev d, int layer, const T* __restrict__ q, T* __restrict__ out, float qk_scale) {
  using C = DecCfg<T, D>;
  extern __shared__ __align__(128) uint8_t smem[];
  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const Smem<T, D> sm(smem, warp);
  const int rank = (int)cluster.block_rank(), csize = (int)cluster.num_blocks();
  const int pair = blockIdx.x / csize;
  const int H = d.kv_heads;
  const int seq = pair / H, head = pair % H;
  init_warp_barriers(sm.wbars, lane);
  __syncthreads();
  pdl_launch_dependents();

  const SeqInfo si = d.seq[seq];
  const int nb = si.n_blocks;
  const int b0 = (int)((int64_t)rank * nb / csize), b1 = (int)((int64_t)(rank + 1) * nb / csize);
  Segment<T, D> sg;
  sg.init(d, si, head, b0, b1 - b0, warp);
  sg.prefetch(d, layer, sm, 0, warp, lane);
  pdl_wait();
  float qr[G][C::VEC];
  load_q<T, D>(d, si, head, q, qk_scale, lane, qr);
  float m_run = -INFINITY, l_run = 0.f;
  float2 acc[G][C::PVD / 2];
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int j = 0; j < C::PVD / 2; ++j) acc[g][j] = make_float2(0.f, 0.f);
  const int failed_at = stream_pages<T, D>(d, layer, sg, sm, 0, qr, m_run, l_run, acc, warp,
                                           lane);
  if (failed_at >= 0) {
    // A wait gave up (error recorded): drain this warp's copies, contribute nothing.
    for (int k = failed_at; k < min(sg.n_my, failed_at + STAGES); ++k)
      mbar_wait(d, &sm.wbars[k % STAGES], (k / STAGES) & 1);
    m_run = -INFINITY;
    l_run = 0.f;
  }
  __syncthreads();
  publish_warp<T, D>(sm, m_run, l_run, acc, warp, lane);
  __syncthreads();
  for (int e = tid; e < G * D; e += DEC_THREADS) {
    float M, L, O;
    merge_elem<T, D>(sm, e, M, L, O);
    sm.r_o[e] = O;
    if ((e % D) == 0) {
      sm.r_ml[(e / D) * 2 + 0] = M;
      sm.r_ml[(e / D) * 2 + 1] = L;
    }
  }
  // Every rank's result is in its shared memory; rank 0 reads them all.  Every
  // CTA reaches both cluster barriers (all earlier waits are bounded).
  cluster.sync();
  if (rank == 0) {
    for (int e = tid; e < G * D; e += DEC_THREADS) {
      const int g = e / D;
      float M = -INFINITY;
      for (int r = 0; r < csize; ++r) M = fmaxf(M, cluster.map_shared_rank(sm.r_ml, r)[g * 2]);
      float L = 0.f, O = 0.f;
      for (int r = 0; r < csize; ++r) {
        const float* rml = cluster.map_shared_rank(sm.r_ml, r);
        const float sc = exp2_safe(rml[g * 2], M);
        L += rml[g * 2 + 1] * sc;
        O += cluster.map_shared_rank(sm.r_o, r)[e] * sc;
      }
      out[((size_t)si.q_row0 * d.q_heads + head * G) * D + e] = from_float<T>(O / L);
    }
  }
  // Keep this CTA's shared memory alive until rank 0 has read it.
  cluster.sync();
}

template <typename T, int D>
const void* dec_kernel_ptr() {
  return reinterpret_cast<const void*>(&attn_decode_kernel<T, D>);
}

template <typename T, int D>
int dec_smem() {
  return DecCfg<T, D>::SMEM;
}

// Largest cluster size (16, else 8, else 0) with which the cluster kernel can run.
template <typename T, int D>
int cluster_size_for() {
  const void* fn = reinterpret_cast<const void*>(&attn_decode_cluster_kernel<T, D>);
  const int smem = dec_smem<T, D>();
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return 0;
  cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaGetLastError();
  for (int cs : {16, 8}) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cs);
    cfg.blockDim = dim3(DEC_THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) == cudaSuccess && n > 0) return cs;
    cudaGetLastError();
  }
  return 0;
}

template <typename T, int D>
cudaError_t launch_cluster(const Dev& d, int layer, const T* q, T* out, float scale, int n_pairs,
                           int cs, bool pdl, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_pairs * cs);
  cfg.blockDim = dim3(DEC_THREADS);
  cfg.dynamicSmemBytes = dec_smem<T, D>();
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, &attn_decode_cluster_kernel<T, D>, d, layer, q, out, scale);
}

}  // namespace

int decode_grid_ctas(const Dev& d) {
  const void* fn = d.esz == 2 ? dec_kernel_ptr<__nv_bfloat16, 128>() : dec_kernel_ptr<float, 64>();
  const int smem = d.esz == 2 ? dec_smem<__nv_bfloat16, 128>() : dec_smem<float, 64>();
  cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, DEC_THREADS, smem);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return max(1, per_sm) * sms;
}

// Minimum (session, kv head, page) units per CTA of the stream-K split.
constexpr int DEC_MIN_UNITS = 12;

cudaError_t launch_attn_decode(const Dev& d, int layer, const void* q, void* out, int n_seq,
                               bool pdl, cudaStream_t s) {
  static thread_local int grid_bf16 = 0, grid_f32 = 0, cs_bf16 = -1, cs_f32 = -1;
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  // Every CTA of the stream-K split may write two partial slots.
  const int max_grid = d.max_dec_items / 2;
  const int n_pairs = n_seq * d.kv_heads;
  if (d.esz == 2) {
    if (!grid_bf16) grid_bf16 = min(max_grid, decode_grid_ctas(d));
    if (cs_bf16 < 0) cs_bf16 = cluster_size_for<__nv_bfloat16, 128>();
    // Few pairs: one cluster per pair, if the clusters fit in one wave.
    if (cs_bf16 > 0 && n_pairs * cs_bf16 <= grid_bf16)
      return launch_cluster<__nv_bfloat16, 128>(d, layer, static_cast<const __nv_bfloat16*>(q),
                                                static_cast<__nv_bfloat16*>(out), scale, n_pairs,
                                                cs_bf16, pdl, s);
    return launch_ex(&attn_decode_kernel<__nv_bfloat16, 128>, dim3(grid_bf16), dim3(DEC_THREADS),
                     dec_smem<__nv_bfloat16, 128>(), s, pdl, d, layer,
                     static_cast<const __nv_bfloat16*>(q), static_cast<__nv_bfloat16*>(out), scale,
                     DEC_MIN_UNITS);
  }
  if (!grid_f32) grid_f32 = min(max_grid, decode_grid_ctas(d));
  if (cs_f32 < 0) cs_f32 = cluster_size_for<float, 64>();
  if (cs_f32 > 0 && n_pairs * cs_f32 <= grid_f32)
    return launch_cluster<float, 64>(d, layer, static_cast<const float*>(q),
                                     static_cast<float*>(out), scale, n_pairs, cs_f32, pdl, s);
  return launch_ex(&attn_decode_kernel<float, 64>, dim3(grid_f32), dim3(DEC_THREADS),
                   dec_smem<float, 64>(), s, pdl, d, layer, static_cast<const float*>(q),
                   static_cast<float*>(out), scale, DEC_MIN_UNITS);
}

}  // namespace kvc
