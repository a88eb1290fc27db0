// Single-token decode GQA attention over the retained cache.
//
// For each session of the last append (one token each), each KV head h and
// its G = 4 query heads: out = softmax(RoPE(q, p) . k / sqrt(D)) v over every
// resident key (the compacted region, then the live region, the token's own
// key included).  Work is split over pages (split-K): a persistent grid walks
// (session-chunk, kv-head) items; inside a CTA each warp streams its own
// pages through a TMA bulk-copy ring in shared memory, computes scores on
// CUDA cores (fp32 FMA), keeps a running max/sum with warp shuffles, and the
// CTA writes either the output or a (max, sum, acc) partial; the last CTA of
// a (session, head) merges the partials (log-sum-exp).
#include "kvc_internal.cuh"

namespace kvc {

namespace {

constexpr unsigned FULL = 0xFFFFFFFFu;
constexpr int DEC_WARPS = 4;
constexpr int DEC_THREADS = DEC_WARPS * 32;
constexpr int G = 4;  // query heads per KV head
static_assert(DEC_WARPS == G, "the split-K merge maps one warp to one query row");
constexpr float LOG2E = 1.4426950408889634f;

template <typename T, int D, int STAGES>
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
  // The cross-warp merge reuses the stage buffers once every warp is done.
  static constexpr int MERGE_BYTES = DEC_WARPS * G * (D + 2) * 4;
  static_assert(MERGE_BYTES <= DEC_WARPS * WARP_BYTES, "merge area must fit in the stages");
  static constexpr int MAX_CHUNKS = 64;  // split-K chunks per session (work-list cap)
  static constexpr int SMEM = DEC_WARPS * WARP_BYTES + DEC_WARPS * STAGES * 8 +
                              MAX_CHUNKS * G * 4 + 64;
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

template <typename T, int D, int STAGES>
__global__ void __launch_bounds__(DEC_THREADS) attn_decode_kernel(Dev d, int layer,
                                                                  const T* __restrict__ q,
                                                                  T* __restrict__ out,
                                                                  float qk_scale, int min_units) {
  using C = DecCfg<T, D, STAGES>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint8_t* wbase = smem + warp * C::WARP_BYTES;
  uint8_t* tiles = wbase;                                            // [STAGES][2][TILE]
  float* s_sc = reinterpret_cast<float*>(wbase + STAGES * 2 * C::TILE);  // [G][PS]
  float2* s_p2 = reinterpret_cast<float2*>(s_sc + G * PS);         // [PS][G] pairs (p, p)
  float* s_alpha = reinterpret_cast<float*>(s_p2 + PS * G);          // [G]
  float* m_o = reinterpret_cast<float*>(smem);   // [W][G][D], aliases the stages
  float* m_ml = m_o + DEC_WARPS * G * D;          // [W][G][2]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + DEC_WARPS * C::WARP_BYTES);
  uint64_t* wbars = bars + warp * STAGES;
  float* s_scale = reinterpret_cast<float*>(bars + DEC_WARPS * STAGES);  // [MAX_CHUNKS][G]
  __shared__ int s_last, s_abort;

  if (lane == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(&wbars[s], 1);
    fence_mbar_init();
  }
  if (tid == 0) s_abort = 0;
  __syncthreads();
  // The next attention call may start its CTAs as soon as slots free up.  Before
  // pdl_wait() this kernel reads only what the append wrote (work list, page
  // tables, K/V pages); q, outputs, partials and counters come after it.
  pdl_launch_dependents();
  bool waited = false;

  // Stream-K split: the call's (session, KV head, page) units, session-major,
  // are cut into n_cta equal contiguous ranges, one per CTA.  A range covers
  // "segments" (the part of one (session, head) pair inside it); only its first
  // and last segments can be partial, and they go to partial slots 2c and 2c+1.
  const int H = d.kv_heads;
  const int U = d.g->n_dec_items;   // units of this call
  const int n_seq = d.g->n_seq;
  // n_cta: at most the grid, at least min_units units per CTA, and small enough that
  // no (session, head) pair spans more than MAX_CHUNKS CTAs (the merge's buffer).
  const int nb_max = max(1, d.g->dec_nb_max);
  const int c_parts = (int)((int64_t)U * (C::MAX_CHUNKS - 2) / (nb_max + C::MAX_CHUNKS - 2));
  const int n_cta = max(1, min((int)gridDim.x, min((U + min_units - 1) / min_units, c_parts)));
  if ((int)blockIdx.x >= n_cta) return;
  const int cta = blockIdx.x;
  auto start_of = [&](int cc) { return (int)((int64_t)cc * U / n_cta); };
  auto owner = [&](int64_t u) { return (int)(((u + 1) * n_cta - 1) / U); };
  const int u_begin = start_of(cta), u_end = start_of(cta + 1);
  const size_t head_stride = (size_t)PS * D;  // elements between heads in a page
  uint32_t loads = 0;  // loads issued (== consumed) by this warp so far
  const int half = lane >> 4, c = lane & 15;

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
    const int blk_begin = u - pair_start;
    const int32_t* hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    const int32_t* lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    const int pos = si.pos_first;  // the single token of this session

    const int nblk = seg_end - u;
    const int n_my = (nblk > warp) ? (nblk - warp + DEC_WARPS - 1) / DEC_WARPS : 0;
    // Page ids of this warp's blocks, 32 at a time: lane j holds block (win + j),
    // so one round trip to the page table serves 32 loads.  Called warp-wide.
    int pwin = -32, pid = 0;
    auto issue = [&](int k) {
      if (k >= pwin + 32) {
        pwin = k & ~31;
        const int j = pwin + lane;
        pid = j < n_my ? block_page(si, hrow, lrow, blk_begin + warp + j * DEC_WARPS) : 0;
      }
      const int page = __shfl_sync(FULL, pid, k - pwin);
      if (lane == 0) {
        const uint32_t n = loads + k;
        const int st = n % STAGES;
        uint8_t* dst = tiles + st * 2 * C::TILE;
        const T* kp = reinterpret_cast<const T*>(d.pool) +
                      pool_offset_elems(d, page, layer, 0, head, 0);
        mbar_arrive_expect_tx(&wbars[st], 2 * C::TILE);
        bulk_g2s(dst, kp, C::TILE, &wbars[st]);
        bulk_g2s(dst + C::TILE, kp + H * head_stride, C::TILE, &wbars[st]);
      }
    };
    // The stage buffers were written by the previous merge: fence before TMA reuse.
    if (lane == 0) fence_proxy_async_smem();
    for (int k = 0; k < min(STAGES, n_my); ++k) issue(k);

    if (!waited) {
      pdl_wait();
      waited = true;
    }
    // Query rows of the G heads, rotated at `pos`, scaled by log2(e)/sqrt(D).  Lane c
    // holds 16-byte chunk c of each row; its rotate-half partner is chunk c ^ 8.
    float qr[G][C::VEC];
    {
      const uint8_t* qrow = reinterpret_cast<const uint8_t*>(
          q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G) * D);
      const float2* cs = d.rope + (size_t)pos * (D / 2) + (c & 7) * C::VEC;
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

    float m_run = -INFINITY, l_run = 0.f;  // for row g_sm = lane >> 3
    float2 acc[G][C::PVD / 2];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < C::PVD / 2; ++j) acc[g][j] = make_float2(0.f, 0.f);

    int failed_at = -1;  // first block whose wait gave up
    for (int k = 0; k < n_my; ++k) {
      const uint32_t n = loads + k;
      const int st = n % STAGES;
      const uint32_t parity = (n / STAGES) & 1;
      if (!__all_sync(FULL, mbar_wait(d, &wbars[st], parity))) {
        failed_at = k;
        break;
      }
      const uint8_t* kt = tiles + st * 2 * C::TILE;
      const uint8_t* vt = kt + C::TILE;
      const BlockRange br = block_range(si, blk_begin + warp + k * DEC_WARPS);

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
          s_sc[g * PS + key] = (key >= br.lo && key < br.hi) ? v : -INFINITY;
        }
      }
      __syncwarp();
      // Online softmax: lane handles row lane>>3, keys 2*(lane&7) and +1.
      {
        const int g = lane >> 3, kk = (lane & 7) * 2;
        const float s0 = s_sc[g * PS + kk], s1 = s_sc[g * PS + kk + 1];
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
        s_p2[kk * G + g] = make_float2(p0, p0);
        s_p2[(kk + 1) * G + g] = make_float2(p1, p1);
        if ((lane & 7) == 0) s_alpha[g] = alpha;
      }
      __syncwarp();
      // PV: lane owns dims [PVD*lane, PVD*lane + PVD) of all G rows, as packed pairs.
      {
        const float4 al = *reinterpret_cast<const float4*>(s_alpha);
        const float alv[G] = {al.x, al.y, al.z, al.w};
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int j = 0; j < C::PVD / 2; ++j)
            acc[g][j] = __fmul2_rn(acc[g][j], make_float2(alv[g], alv[g]));
#pragma unroll
        for (int key = 0; key < PS; ++key) {
          const float4 p01 = *reinterpret_cast<const float4*>(s_p2 + key * G);
          const float4 p23 = *reinterpret_cast<const float4*>(s_p2 + key * G + 2);
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
      if (k + STAGES < n_my) {
        if (lane == 0) fence_proxy_async_smem();
        issue(k + STAGES);
      }
    }
    if (failed_at >= 0 && lane == 0) s_abort = 1;
    __syncthreads();
    if (s_abort) {
      // Some wait gave up: each warp drains the copies it still has in flight
      // (bounded waits), then the whole CTA stops together.
      if (failed_at >= 0) {
        for (int k = failed_at; k < min(n_my, failed_at + STAGES); ++k) {
          const uint32_t n = loads + k;
          mbar_wait(d, &wbars[n % STAGES], (n / STAGES) & 1);
        }
      }
      return;
    }
    loads += n_my;

    // Merge the four warps' partial softmax states (stage buffers are free now).
    __syncthreads();
    if ((lane & 7) == 0) {
      m_ml[(warp * G + (lane >> 3)) * 2 + 0] = m_run;
      m_ml[(warp * G + (lane >> 3)) * 2 + 1] = l_run;
    }
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < C::PVD / 2; ++j)
        *reinterpret_cast<float2*>(&m_o[(warp * G + g) * D + lane * C::PVD + 2 * j]) = acc[g][j];
    __syncthreads();
    const bool whole = u == pair_start && seg_end == pair_end;
    const int slot = 2 * cta + (u == u_begin ? 0 : 1);
    for (int e = tid; e < G * D; e += DEC_THREADS) {
      const int g = e / D, dd = e % D;
      float mw[DEC_WARPS], M = -INFINITY;
#pragma unroll
      for (int w = 0; w < DEC_WARPS; ++w) {
        mw[w] = m_ml[(w * G + g) * 2];
        M = fmaxf(M, mw[w]);
      }
      float L = 0.f, O = 0.f;
#pragma unroll
      for (int w = 0; w < DEC_WARPS; ++w) {
        const float sc = exp2_safe(mw[w], M);
        L += m_ml[(w * G + g) * 2 + 1] * sc;
        O += m_o[(w * G + g) * D + dd] * sc;
      }
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
            s_scale[ch * G + g] = sc;
            L += ml.y * sc;
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(FULL, L, o);
          const float inv = 1.f / L;
          __syncwarp();
          for (int ch = lane; ch < nch; ch += 32) s_scale[ch * G + g] *= inv;
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
              O[i] += a[k][i] * s_scale[(ch + k) * G + (tid + i * DEC_THREADS) / D];
        }
        for (; ch < nch; ++ch) {
          const float* b0 = d.dec_part_o + (size_t)slot_of(cf + ch) * G * D;
#pragma unroll
          for (int i = 0; i < EPT; ++i) {
            const int g = (tid + i * DEC_THREADS) / D;
            O[i] += __ldcg(b0 + tid + i * DEC_THREADS) * s_scale[ch * G + g];
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

constexpr int DEC_STAGES = 2;

template <typename T, int D>
const void* dec_kernel_ptr() {
  return reinterpret_cast<const void*>(&attn_decode_kernel<T, D, DEC_STAGES>);
}

template <typename T, int D>
int dec_smem() {
  return DecCfg<T, D, DEC_STAGES>::SMEM;
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

// Minimum (session, kv head, page) units per CTA: below this, launch fewer CTAs.
constexpr int DEC_MIN_UNITS = 12;

cudaError_t launch_attn_decode(const Dev& d, int layer, const void* q, void* out, int n_seq,
                               bool pdl, cudaStream_t s) {
  (void)n_seq;
  static thread_local int grid_bf16 = 0, grid_f32 = 0;
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  // Every CTA may write two partial slots.
  const int max_grid = d.max_dec_items / 2;
  if (d.esz == 2) {
    if (!grid_bf16) grid_bf16 = min(max_grid, decode_grid_ctas(d));
    return launch_ex(&attn_decode_kernel<__nv_bfloat16, 128, DEC_STAGES>, dim3(grid_bf16),
                     dim3(DEC_THREADS), dec_smem<__nv_bfloat16, 128>(), s, pdl, d, layer,
                     static_cast<const __nv_bfloat16*>(q), static_cast<__nv_bfloat16*>(out), scale,
                     DEC_MIN_UNITS);
  }
  if (!grid_f32) grid_f32 = min(max_grid, decode_grid_ctas(d));
  return launch_ex(&attn_decode_kernel<float, 64, DEC_STAGES>, dim3(grid_f32), dim3(DEC_THREADS),
                   dec_smem<float, 64>(), s, pdl, d, layer, static_cast<const float*>(q),
                   static_cast<float*>(out), scale, DEC_MIN_UNITS);
}

}  // namespace kvc
