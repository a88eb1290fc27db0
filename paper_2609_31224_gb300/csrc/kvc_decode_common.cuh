// Device code shared by the two decode translation units (stream-K in
// kvc_attn_decode.cu, pair split in kvc_attn_decode_split.cu): CTA shapes, the
// per-warp page pipeline, the page loops (tensor cores for bfloat16, CUDA cores for
// binary32), the cross-warp merge and the log-sum-exp merge of split-K partial
// states.
#pragma once

#include "kvc_launch.cuh"

namespace kvc {

namespace {

constexpr unsigned FULL = 0xFFFFFFFFu;
constexpr int G = 4;  // query heads per KV head
constexpr float LOG2E = 1.4426950408889634f;
constexpr int MAX_PARTS = 64;     // partial states per (session, head) pair, at most

// One CTA shape: WARPS warps, each streaming its own pages through a STAGES-deep
// ring of K/V tiles.  MMA (bfloat16 only): the page loop runs on the tensor cores
// (mma.sync), with tiles staged by 2-D TMA in the 128-byte-swizzled layout;
// otherwise on CUDA cores with tiles staged by 1-D bulk copies.
template <typename T_, int D_, int WARPS_, int STAGES_, bool MMA_ = false>
struct DecCfg {
  using T = T_;
  static constexpr int D = D_, WARPS = WARPS_, STAGES = STAGES_, THREADS = WARPS * 32;
  static constexpr int ESZ = sizeof(T);
  static constexpr bool MMA = MMA_ && ESZ == 2;
  static constexpr int ROW_BYTES = D * ESZ;
  static_assert(ROW_BYTES == 256, "decode kernel assumes 256-byte K/V rows");
  static constexpr int VEC = 16 / ESZ;     // elements per 16-byte lane chunk (QK)
  static constexpr int PVD = D / 32;       // dims per lane (PV)
  static constexpr int TILE = PS * ROW_BYTES;  // one page of one head: 4 KiB
  // Shared memory (from a 1024-aligned base): every warp's STAGES x (K tile + V
  // tile), then per warp: scores + probability pairs (p, p) + alpha.
  static constexpr int TILES = WARPS * STAGES * 2 * TILE;
  static constexpr int SCRATCH = (G * PS + 2 * PS * G + G) * 4 + 16;
  static_assert(SCRATCH % 16 == 0, "scratch stays 16-byte aligned");
  // The cross-warp merge reuses the stage buffers once every warp is done with
  // its pages.
  static constexpr int MERGE_FLOATS = WARPS * G * D + WARPS * G * 2;
  static constexpr int RESULT_FLOATS = G * 2 + WARPS * G;
  static_assert((MERGE_FLOATS + RESULT_FLOATS) * 4 <= TILES, "merge area must fit in the stages");
  static constexpr int SMEM =
      1024 + TILES + WARPS * SCRATCH + WARPS * STAGES * 8 + MAX_PARTS * G * 4 + 64;
};

// Stream-K kernel: 4 warps (one per query row in the split-K merge), 2-deep rings,
// three CTAs per SM; tensor-core pages for bfloat16.
template <typename T, int D>
using SkCfg = DecCfg<T, D, 4, 2, true>;
// Pair-split kernel: 16 warps, one tile pair each, one CTA per SM; with few
// sessions every page of the call is in flight at once.  Its pages are latency-
// bound, so for bfloat16 they run on the tensor cores (fewer instructions per page).
constexpr int SP_WARPS = 16, SP_STAGES = 1;
template <typename T, int D>
using SpCfg = DecCfg<T, D, SP_WARPS, SP_STAGES, true>;
// Pair-split kernel for calls with too many pairs for SpCfg: stream-K's CTA shape
// (three CTAs per SM), with the tensor-core page loop for bfloat16 too (measured
// 28.6 against 31.4 us per launch at 10 sessions, 49.7 against 51.8 at 19).
constexpr bool SP4_MMA = true;
template <typename T, int D>
using Sp4Cfg = DecCfg<T, D, 4, 2, SP4_MMA>;

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
template <class C>
struct Smem {
  uint8_t* tiles;     // this warp's [STAGES][2][TILE]
  float* s_sc;        // [G][PS] scores
  float2* s_p2;       // [PS][G] probability pairs (p, p)
  float* s_alpha;     // [G]
  float* m_o;         // [W][G][D] warp partial outputs (aliases the stages)
  float* m_ml;        // [W][G][2]
  float* r_ml;        // [G][2] CTA (max, sum) per row
  float* s_wsc;       // [W][G] weight of each warp's part (aliases the stages)
  uint64_t* wbars;    // this warp's [STAGES]
  float* s_scale;     // [MAX_PARTS][G]
  // The tensor-core page loop keeps the bfloat16 probabilities P^T [G rows][PS
  // keys] in s_sc.
  __device__ Smem(uint8_t* raw, int warp) {
    // Offset into the shared array itself (keeps the accesses shared-memory ones).
    uint8_t* smem = raw + ((1024u - (smem_u32(raw) & 1023u)) & 1023u);
    tiles = smem + warp * C::STAGES * 2 * C::TILE;
    uint8_t* scratch = smem + C::TILES + warp * C::SCRATCH;
    s_sc = reinterpret_cast<float*>(scratch);
    s_p2 = reinterpret_cast<float2*>(s_sc + G * PS);
    s_alpha = reinterpret_cast<float*>(s_p2 + PS * G);
    m_o = reinterpret_cast<float*>(smem);
    m_ml = m_o + C::WARPS * G * C::D;
    r_ml = m_ml + C::WARPS * G * 2;
    s_wsc = r_ml + G * 2;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::TILES + C::WARPS * C::SCRATCH);
    wbars = bars + warp * C::STAGES;
    s_scale = reinterpret_cast<float*>(bars + C::WARPS * C::STAGES);
  }
};

// Blocks [blk_begin, blk_begin + nblk) of one (session, head) pair; warp w takes
// blocks blk_begin + w, + w + WARPS, ...  Page ids are fetched 32 at a time (lane j
// holds the id of the warp's block win + j), so one round trip serves 32 loads.
template <class C>
struct Segment {
  using T = typename C::T;
  static constexpr int D = C::D;
  SeqInfo si;
  int head, blk_begin, nblk, n_my;
  const int32_t* hrow;
  const int32_t* lrow;
  int pwin, pid;
  const CUtensorMap* map_lo;  // tensor maps of the pool (tensor-core page loop only)
  const CUtensorMap* map_hi;

  __device__ void init(const Dev& d, const SeqInfo& s, int h, int b0, int nb, int warp,
                       const CUtensorMap* mlo = nullptr, const CUtensorMap* mhi = nullptr) {
    map_lo = mlo;
    map_hi = mhi;
    si = s;
    head = h;
    blk_begin = b0;
    nblk = nb;
    n_my = (nblk > warp) ? (nblk - warp + C::WARPS - 1) / C::WARPS : 0;
    hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    pwin = -32;
    pid = 0;
  }

  // Load the K and V tiles of this warp's k-th block (called by the whole warp).
  __device__ void issue(const Dev& d, int layer, const Smem<C>& sm, uint32_t loads, int k,
                        int warp, int lane) {
    if (k >= pwin + 32) {
      pwin = k & ~31;
      const int j = pwin + lane;
      pid = j < n_my ? block_page(si, hrow, lrow, blk_begin + warp + j * C::WARPS) : 0;
    }
    const int page = __shfl_sync(FULL, pid, k - pwin);
    if (lane == 0) {
      const uint32_t n = loads + k;
      const int st = n % C::STAGES;
      uint8_t* dst = sm.tiles + st * 2 * C::TILE;
      mbar_arrive_expect_tx(&sm.wbars[st], 2 * C::TILE);
      if constexpr (C::MMA) {
        // Pool rows of the K and V tiles, each as two swizzled 64-column boxes.
        const int krow = (((page * d.layers + layer) * 2) * d.kv_heads + head) * PS;
        const int vrow = krow + d.kv_heads * PS;
        tma_load_2d(dst, map_lo, 0, krow, &sm.wbars[st]);
        tma_load_2d(dst + C::TILE / 2, map_hi, 0, krow, &sm.wbars[st]);
        tma_load_2d(dst + C::TILE, map_lo, 0, vrow, &sm.wbars[st]);
        tma_load_2d(dst + C::TILE + C::TILE / 2, map_hi, 0, vrow, &sm.wbars[st]);
      } else {
        const T* kp = reinterpret_cast<const T*>(d.pool) +
                      pool_offset_elems(d, page, layer, 0, head, 0);
        bulk_g2s(dst, kp, C::TILE, &sm.wbars[st]);
        bulk_g2s(dst + C::TILE, kp + (size_t)d.kv_heads * PS * D, C::TILE, &sm.wbars[st]);
      }
    }
  }

  __device__ void prefetch(const Dev& d, int layer, const Smem<C>& sm, uint32_t loads,
                           int warp, int lane) {
    // The stage buffers may have been written by the previous merge.
    if (lane == 0) fence_proxy_async_smem();
    for (int k = 0; k < min(C::STAGES, n_my); ++k) issue(d, layer, sm, loads, k, warp, lane);
  }
};

// Query rows of the G heads of `head`, rotated at the token's position and scaled
// by log2(e)/sqrt(D).  Lane c = lane & 7 holds 16-byte chunk c of each row
// (qr[g][0, VEC)) and its rotate-half partner, chunk c + 8 (qr[g][VEC, 2 VEC)).
template <class C>
__device__ void load_q(const Dev& d, const SeqInfo& si, int head, const typename C::T* q,
                       float qk_scale, int lane, float (&qr)[G][2 * C::VEC]) {
  using T = typename C::T;
  constexpr int D = C::D;
  static_assert(D / 2 * C::ESZ == 128, "rotate-half partner is chunk c + 8");
  const int c = lane & 7;
  const uint8_t* qrow =
      reinterpret_cast<const uint8_t*>(q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G) * D);
  const float2* cs = d.rope + (size_t)si.pos_first * (D / 2) + c * C::VEC;
  float2 t[C::VEC];
#pragma unroll
  for (int e = 0; e < C::VEC; ++e) t[e] = cs[e];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float x[C::VEC], y[C::VEC];
    load_vec<T>(qrow + g * C::ROW_BYTES + c * 16, x);
    load_vec<T>(qrow + g * C::ROW_BYTES + 128 + c * 16, y);
#pragma unroll
    for (int e = 0; e < C::VEC; ++e) {
      qr[g][e] = fmaf(x[e], t[e].x, -y[e] * t[e].y) * qk_scale;
      qr[g][C::VEC + e] = fmaf(y[e], t[e].x, x[e] * t[e].y) * qk_scale;
    }
  }
}

// Fused layer write (per-layer order): the session's new token K (rotated at its
// position, the append kernel's binary32 arithmetic) and V of this layer and head,
// read from the caller's [total][Hkv][D] rows, go into the pool slot and into the
// K/V tile just loaded from it (whose copy of that row may be stale).  Called by
// the warp that streams the pair's last block, which holds the token.
template <class C>
__device__ void patch_new_row(const Dev& d, int layer, const SeqInfo& si, int head,
                              const typename C::T* nk, const typename C::T* nv, uint8_t* kt,
                              int lane) {
  using T = typename C::T;
  constexpr int D = C::D, HALF = D / 2;
  const int gs = d.tok_slot[si.q_row0];
  const int page = gs / PS, slot = gs % PS;
  const T* kin = nk + ((size_t)si.q_row0 * d.kv_heads + head) * D;
  const T* vin = nv + ((size_t)si.q_row0 * d.kv_heads + head) * D;
  const float2* cs = d.rope + (size_t)si.pos_first * HALF;
  T* kp = reinterpret_cast<T*>(d.pool) + pool_offset_elems(d, page, layer, 0, head, slot);
  T* vp = reinterpret_cast<T*>(d.pool) + pool_offset_elems(d, page, layer, 1, head, slot);
  // Byte offset of element j of the row within a tile (linear, or two swizzled
  // 64-column boxes for the tensor-core loop).
  auto at = [&](int j) -> int {
    if constexpr (C::MMA)
      return (j >> 6) * (C::TILE / 2) + slot * 128 + ((((j & 63) >> 3) ^ (slot & 7)) << 4) +
             (j & 7) * C::ESZ;
    else
      return slot * C::ROW_BYTES + j * C::ESZ;
  };
  // Every load of the row is issued before any store (one round trip): lane owns the
  // rotate-half pairs (j, j + D/2) for j = lane + 32 i and the V elements lane + 32 i.
  constexpr int KP = HALF / 32, VP = D / 32;
  static_assert(HALF % 32 == 0, "whole pairs per lane");
  float x1[KP], x2[KP];
  float2 c[KP];
  T vv[VP];
#pragma unroll
  for (int i = 0; i < KP; ++i) {
    const int j = lane + 32 * i;
    x1[i] = to_float<T>(kin[j]);
    x2[i] = to_float<T>(kin[j + HALF]);
    c[i] = cs[j];
  }
#pragma unroll
  for (int i = 0; i < VP; ++i) vv[i] = vin[lane + 32 * i];
#pragma unroll
  for (int i = 0; i < KP; ++i) {
    const int j = lane + 32 * i;
    const T y1 = from_float<T>(fmaf(x1[i], c[i].x, -x2[i] * c[i].y));
    const T y2 = from_float<T>(fmaf(x2[i], c[i].x, x1[i] * c[i].y));
    *reinterpret_cast<T*>(kt + at(j)) = y1;
    *reinterpret_cast<T*>(kt + at(j + HALF)) = y2;
    kp[j] = y1;
    kp[j + HALF] = y2;
  }
#pragma unroll
  for (int i = 0; i < VP; ++i) {
    const int j = lane + 32 * i;
    *reinterpret_cast<T*>(kt + C::TILE + at(j)) = vv[i];
    vp[j] = vv[i];
  }
  __syncwarp();
}

// Stream this warp's blocks of the segment: scores, online softmax, P V.  The first
// STAGES blocks must have been issued (Segment::prefetch).  Returns the first block
// whose wait gave up, or -1.
template <class C, bool FUSED>
__device__ int stream_pages(const Dev& d, int layer, Segment<C>& sg, const Smem<C>& sm,
                            uint32_t loads, const float (&qr)[G][2 * C::VEC], float& m_run,
                            float& l_run, float2 (&acc)[G][C::PVD / 2], int warp, int lane,
                            const typename C::T* new_k, const typename C::T* new_v) {
  using T = typename C::T;
  const int kq = lane >> 3, c = lane & 7;
  const bool up4 = lane & 4, up2 = lane & 2;
  const int my_g = (up4 ? 2 : 0) + (up2 ? 1 : 0);  // row whose score this lane ends with
  for (int k = 0; k < sg.n_my; ++k) {
    const uint32_t n = loads + k;
    const int st = n % C::STAGES;
    if (!__all_sync(FULL, mbar_wait(d, &sm.wbars[st], (n / C::STAGES) & 1))) return k;
    const uint8_t* kt = sm.tiles + st * 2 * C::TILE;
    const uint8_t* vt = kt + C::TILE;
    const int blk = sg.blk_begin + warp + k * C::WARPS;
    if constexpr (FUSED) {
      if (blk == sg.si.n_blocks - 1)
        patch_new_row<C>(d, layer, sg.si, sg.head, new_k, new_v, sm.tiles + st * 2 * C::TILE,
                         lane);
    }
    const BlockRange br = block_range(sg.si, blk);
    const bool interior = br.lo == 0 && br.hi == PS;

    // Scores: the 8 lanes 8j..8j+7 take key 4i + j, lane c its chunks c and c + 8.
#pragma unroll
    for (int i = 0; i < PS / 4; ++i) {
      const int key = 4 * i + kq;
      float k0[C::VEC], k1[C::VEC];
      load_vec<T>(kt + key * C::ROW_BYTES + c * 16, k0);
      load_vec<T>(kt + key * C::ROW_BYTES + 128 + c * 16, k1);
      float a[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        // Even and odd dims accumulate in the two halves of a packed pair.
        float2 acc2 = make_float2(0.f, 0.f);
#pragma unroll
        for (int e = 0; e < C::VEC; e += 2) {
          acc2 = __ffma2_rn(make_float2(qr[g][e], qr[g][e + 1]), make_float2(k0[e], k0[e + 1]),
                            acc2);
          acc2 = __ffma2_rn(make_float2(qr[g][C::VEC + e], qr[g][C::VEC + e + 1]),
                            make_float2(k1[e], k1[e + 1]), acc2);
        }
        a[g] = acc2.x + acc2.y;
      }
      // Reduce-scatter of the 4 sums over the key's 8 lanes (xor 4, then xor 2),
      // then a pair sum (xor 1): lane ends with row my_g's score.
      const float r0 = __shfl_xor_sync(FULL, up4 ? a[0] : a[2], 4);
      const float r1 = __shfl_xor_sync(FULL, up4 ? a[1] : a[3], 4);
      const float b0 = (up4 ? a[2] : a[0]) + r0;
      const float b1 = (up4 ? a[3] : a[1]) + r1;
      float v = (up2 ? b1 : b0) + __shfl_xor_sync(FULL, up2 ? b0 : b1, 2);
      v += __shfl_xor_sync(FULL, v, 1);
      if ((lane & 1) == 0)
        sm.s_sc[my_g * PS + key] = (interior || (key >= br.lo && key < br.hi)) ? v : -INFINITY;
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
      // Rescale only when some row's running max moved (warp-uniform).
      if (al.x != 1.f || al.y != 1.f || al.z != 1.f || al.w != 1.f) {
        const float alv[G] = {al.x, al.y, al.z, al.w};
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int j = 0; j < C::PVD / 2; ++j)
            acc[g][j] = __fmul2_rn(acc[g][j], make_float2(alv[g], alv[g]));
      }
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
    if (k + C::STAGES < sg.n_my) {
      if (lane == 0) fence_proxy_async_smem();
      sg.issue(d, layer, sm, loads, k + C::STAGES, warp, lane);
    }
  }
  return -1;
}

// After every warp of the CTA has finished (caller syncs): publish the warps'
// partial states.
template <class C>
__device__ void publish_warp(const Smem<C>& sm, float m_run, float l_run,
                             const float2 (&acc)[G][C::PVD / 2], int warp, int lane) {
  constexpr int D = C::D;
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

// After publish_warp and a sync: warp g < G reduces row g over the warps (max M,
// sum L, each warp's weight exp2(m_w - M)); ends with a sync, after which
// sm.r_ml holds (M, L) per row and merge_warps_elem(e) the row's unnormalised
// output element e = g * D + dd.
template <class C>
__device__ void merge_warps(const Smem<C>& sm, int warp, int lane) {
  static_assert(C::WARPS <= 32, "one lane per warp");
  if (warp < G) {
    const int g = warp;
    float m = -INFINITY, l = 0.f;
    if (lane < C::WARPS) {
      const float2 ml = *reinterpret_cast<const float2*>(&sm.m_ml[(lane * G + g) * 2]);
      m = ml.x;
      l = ml.y;
    }
    float M = m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(FULL, M, o));
    const float w = exp2_safe(m, M);
    float L = l * w;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(FULL, L, o);
    if (lane < C::WARPS) sm.s_wsc[lane * G + g] = w;
    if (lane == 0) {
      sm.r_ml[g * 2 + 0] = M;
      sm.r_ml[g * 2 + 1] = L;
    }
  }
  __syncthreads();
}

template <class C>
__device__ inline float merge_warps_elem(const Smem<C>& sm, int e) {
  constexpr int D = C::D;
  const int g = e / D, dd = e % D;
  float O = 0.f;
#pragma unroll
  for (int w = 0; w < C::WARPS; ++w) O += sm.m_o[(w * G + g) * D + dd] * sm.s_wsc[w * G + g];
  return O;
}

// Arrive at a pair's counter after this CTA's partial state is written; true in
// the last of `parts` CTAs to arrive.  One thread's acquire-release atomic after
// the CTA barrier publishes every thread's partial writes and, in the last CTA,
// orders the loads of the other parts after it.  Called by every thread.
__device__ inline bool arrive_last(int* counter, int parts, int tid, int* s_flag) {
  __syncthreads();
  if (tid == 0) *s_flag = arrive_acq_rel(counter, parts);
  __syncthreads();
  return *s_flag;
}

template <class C>
__device__ inline void init_warp_barriers(uint64_t* wbars, int lane) {
  if (lane == 0) {
    for (int s = 0; s < C::STAGES; ++s) mbar_init(&wbars[s], 1);
    fence_mbar_init();
  }
}

// Warp-wide L2 prefetch of the query rows of `head` and the token's RoPE row, so
// that load_q after pdl_wait() hits L2.
template <class C>
__device__ inline void prefetch_q(const Dev& d, const SeqInfo& si, int head,
                                  const typename C::T* q, int lane) {
  const uintptr_t qa =
      reinterpret_cast<uintptr_t>(q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G) * C::D);
  const uintptr_t ra = reinterpret_cast<uintptr_t>(d.rope + (size_t)si.pos_first * (C::D / 2));
  const uintptr_t q0 = qa & ~uintptr_t(127), r0 = ra & ~uintptr_t(127);
  const int nq = (int)((qa + G * C::ROW_BYTES - q0 + 127) / 128);  // <= 9 lines
  const int nr = (int)((ra + C::D * 4 - r0 + 127) / 128);          // <= 5 lines
  if (lane < nq) prefetch_l2(reinterpret_cast<const void*>(q0 + 128 * lane));
  else if (lane >= 16 && lane - 16 < nr)
    prefetch_l2(reinterpret_cast<const void*>(r0 + 128 * (lane - 16)));
}

// Log-sum-exp merge of the nch <= MAX_PARTS partial states of one (session, head)
// pair into its G output rows (orow: row of query head head * G).  part(i) is the
// slot holding part i.  Warp g < G reduces row g's maxima and sums from one pass
// over the parts' (m, l) and leaves each part's weight, divided by the total, in
// shared memory; then every thread sums its elements' weighted partial outputs
// with up to 32 independent loads in flight.  Called by every thread of the CTA.
template <class C, typename PartFn>
__device__ void merge_parts(const Dev& d, const Smem<C>& sm, int nch, PartFn part,
                            typename C::T* orow, int tid, int warp, int lane) {
  using T = typename C::T;
  constexpr int D = C::D;
  static_assert(C::WARPS >= G, "one warp per query row");
  constexpr int EPT = (G * D + C::THREADS - 1) / C::THREADS;  // elements per thread
  constexpr int CH = 32 / EPT > 0 ? 32 / EPT : 1;              // parts per batch of loads
  auto load_batch = [&](int c0, float (&a)[CH][EPT]) {
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const bool ok = c0 + i < nch;
      const float* b = d.dec_part_o + (size_t)(ok ? part(c0 + i) : 0) * G * D;
#pragma unroll
      for (int t = 0; t < EPT; ++t) {
        const int e = tid + t * C::THREADS;
        a[i][t] = (ok && e < G * D) ? __ldcg(b + e) : 0.f;
      }
    }
  };
  // The first batch of partial outputs is in flight while the weights are formed.
  float a[CH][EPT];
  load_batch(0, a);
  if (warp < G) {
    const int g = warp;
    constexpr int PL = MAX_PARTS / 32;  // parts per lane
    float2 ml[PL];
    float M = -INFINITY;
#pragma unroll
    for (int i = 0; i < PL; ++i) {
      const int ch = lane + 32 * i;
      ml[i] = ch < nch ? __ldcg(&d.dec_part_ml[(size_t)part(ch) * G + g])
                       : make_float2(-INFINITY, 0.f);
      M = fmaxf(M, ml[i].x);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(FULL, M, o));
    float sc[PL], L = 0.f;
#pragma unroll
    for (int i = 0; i < PL; ++i) {
      sc[i] = exp2_safe(ml[i].x, M);
      L += ml[i].y * sc[i];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(FULL, L, o);
    const float inv = 1.f / L;
#pragma unroll
    for (int i = 0; i < PL; ++i)
      if (lane + 32 * i < nch) sm.s_scale[(lane + 32 * i) * G + g] = sc[i] * inv;
  }
  __syncthreads();
  float O[EPT];
#pragma unroll
  for (int t = 0; t < EPT; ++t) O[t] = 0.f;
  for (int c0 = 0;;) {
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      if (c0 + i >= nch) break;
#pragma unroll
      for (int t = 0; t < EPT; ++t) {
        const int e = tid + t * C::THREADS;
        if (e < G * D) O[t] += a[i][t] * sm.s_scale[(c0 + i) * G + e / D];
      }
    }
    c0 += CH;
    if (c0 >= nch) break;
    load_batch(c0, a);
  }
#pragma unroll
  for (int t = 0; t < EPT; ++t) {
    const int e = tid + t * C::THREADS;
    if (e < G * D) orow[e] = from_float<T>(O[t]);
  }
}

// ---------------------------------------------------------------------------
// Tensor-core page loop (bfloat16, D = 128).  Per page of 16 keys and the G = 4
// query rows of one KV head, with the keys as the MMA's M dimension:
//   S^T [16 keys x 8 rows]  = K [16 x 128] . Q^T [128 x 8]        (8 k-steps)
//   O^T [128 dims x 8 rows] += V^T [128 x 16 keys] . P^T [16 x 8]  (8 m-tiles)
// with mma.sync m16n8k16 (bf16 in, fp32 accumulate); rows 4..7 are zero padding.
// Lane (g, t) = (lane >> 2, lane & 3) holds S^T for keys g, g + 8 and rows 2t,
// 2t + 1, so it owns the softmax state of rows 2t, 2t + 1 (valid for t < 2), and
// O^T for dims 16 mt + g (+ 8) of the same rows.  Tiles are two 64-column boxes
// (2 KiB, 16 rows of 128 B) with the 128-byte swizzle: 16-byte chunk c of row r
// sits at chunk c ^ (r & 7), so ldmatrix reads of 8 rows hit 8 distinct banks.
// ---------------------------------------------------------------------------
__device__ inline uint32_t swz(int row, int col) {  // col: a multiple of 8 in [0, 128)
  return (col >> 6) * 2048 + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4);
}

__device__ inline void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr)
               : "memory");
}

__device__ inline void ldsm_x4_trans(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr)
               : "memory");
}

__device__ inline void mma_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                 uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ inline uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Query rows of `head`, rotated at the token's position, scaled by log2(e)/sqrt(D)
// and rounded to bfloat16, as the B operand Q^T of the score products: lane (g, t)
// with g < G holds dims 16 ks + 2t, +1 (qb[ks][0]) and 16 ks + 2t + 8, +9
// (qb[ks][1]) of row g; lanes g >= G hold the zero rows.  Dims d and d + 64 (k-steps
// ks and ks + 4 of the same lane) are rotated together.
template <class C>
__device__ void load_q_mma(const Dev& d, const SeqInfo& si, int head, const typename C::T* q,
                           float qk_scale, int lane, uint32_t (&qb)[8][2]) {
  static_assert(C::D == 128, "tensor-core page loop assumes D = 128");
  const int g = lane >> 2, t = lane & 3;
  if (g >= G) {
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) qb[ks][0] = qb[ks][1] = 0u;
    return;
  }
  const uint32_t* qrow = reinterpret_cast<const uint32_t*>(
      q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G + g) * C::D);
  const float2* cs = d.rope + (size_t)si.pos_first * (C::D / 2);
  uint32_t w[8][2];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    w[ks][0] = qrow[8 * ks + t];
    w[ks][1] = qrow[8 * ks + t + 4];
  }
  float2 c[4][4];
#pragma unroll
  for (int ks = 0; ks < 4; ++ks)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      c[ks][2 * j] = cs[16 * ks + 2 * t + 8 * j];
      c[ks][2 * j + 1] = cs[16 * ks + 2 * t + 8 * j + 1];
    }
#pragma unroll
  for (int ks = 0; ks < 4; ++ks)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const float x0 = bf16lo(w[ks][j]), x1 = bf16hi(w[ks][j]);          // dims < 64
      const float y0 = bf16lo(w[ks + 4][j]), y1 = bf16hi(w[ks + 4][j]);  // dims + 64
      const float2 c0 = c[ks][2 * j], c1 = c[ks][2 * j + 1];
      qb[ks][j] = pack_bf16x2(fmaf(x0, c0.x, -y0 * c0.y) * qk_scale,
                              fmaf(x1, c1.x, -y1 * c1.y) * qk_scale);
      qb[ks + 4][j] = pack_bf16x2(fmaf(y0, c0.x, x0 * c0.y) * qk_scale,
                                  fmaf(y1, c1.x, x1 * c1.y) * qk_scale);
    }
}

// stream_pages on the tensor cores.  m_run / l_run: running max and this lane's
// partial sum of rows 2t, 2t + 1 (the sum is completed over g by publish_warp_mma).
template <class C, bool FUSED>
__device__ int stream_pages_mma(const Dev& d, int layer, Segment<C>& sg, const Smem<C>& sm,
                                uint32_t loads, const uint32_t (&qb)[8][2], float (&m_run)[2],
                                float (&l_run)[2], float (&o)[8][4], int warp, int lane,
                                const typename C::T* new_k, const typename C::T* new_v) {
  const int g = lane >> 2, t = lane & 3;
  // ldmatrix row of this lane: K (A = K, keys x dims) and V (A = V^T via .trans).
  const int k_key = (lane & 7) + 8 * ((lane >> 3) & 1), k_col = 8 * (lane >> 4);
  const int v_key = (lane & 7) + 8 * (lane >> 4), v_col = 8 * ((lane >> 3) & 1);
  __nv_bfloat16* pt = reinterpret_cast<__nv_bfloat16*>(sm.s_sc);  // P^T as [G][PS]
  for (int k = 0; k < sg.n_my; ++k) {
    const uint32_t n = loads + k;
    const int st = n % C::STAGES;
    if (!__all_sync(FULL, mbar_wait(d, &sm.wbars[st], (n / C::STAGES) & 1))) return k;
    uint8_t* kt = sm.tiles + st * 2 * C::TILE;
    const int blk = sg.blk_begin + warp + k * C::WARPS;
    if constexpr (FUSED) {
      if (blk == sg.si.n_blocks - 1)
        patch_new_row<C>(d, layer, sg.si, sg.head, new_k, new_v, kt, lane);
    }
    const uint32_t kb = smem_u32(kt), vb = kb + C::TILE;

    float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      uint32_t a[4];
      ldsm_x4(a, kb + swz(k_key, 16 * ks + k_col));
      mma_16816(s, a, qb[ks][0], qb[ks][1]);
    }
    const BlockRange br = block_range(sg.si, blk);
    if (!(br.lo == 0 && br.hi == PS)) {
      if (g < br.lo || g >= br.hi) s[0] = s[1] = -INFINITY;
      if (g + 8 < br.lo || g + 8 >= br.hi) s[2] = s[3] = -INFINITY;
    }
    // Online softmax of rows 2t (s0, s2) and 2t + 1 (s1, s3) over the page's keys.
    float mx0 = fmaxf(s[0], s[2]), mx1 = fmaxf(s[1], s[3]);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      mx0 = fmaxf(mx0, __shfl_xor_sync(FULL, mx0, off));
      mx1 = fmaxf(mx1, __shfl_xor_sync(FULL, mx1, off));
    }
    const float mn0 = fmaxf(m_run[0], mx0), mn1 = fmaxf(m_run[1], mx1);
    const float p0 = exp2_safe(s[0], mn0), p2 = exp2_safe(s[2], mn0);
    const float p1 = exp2_safe(s[1], mn1), p3 = exp2_safe(s[3], mn1);
    const float al0 = exp2_safe(m_run[0], mn0), al1 = exp2_safe(m_run[1], mn1);
    l_run[0] = l_run[0] * al0 + (p0 + p2);
    l_run[1] = l_run[1] * al1 + (p1 + p3);
    m_run[0] = mn0;
    m_run[1] = mn1;
    // P^T to the B-operand layout through shared memory: lane (g, t < 2) writes
    // P[row][key] for its two rows and keys g, g + 8; lane (g < G, t) reads keys
    // 2t, 2t + 1 and 2t + 8, 2t + 9 of row g.
    __syncwarp();
    if (t < 2) {
      pt[(2 * t) * PS + g] = __float2bfloat16_rn(p0);
      pt[(2 * t + 1) * PS + g] = __float2bfloat16_rn(p1);
      pt[(2 * t) * PS + g + 8] = __float2bfloat16_rn(p2);
      pt[(2 * t + 1) * PS + g + 8] = __float2bfloat16_rn(p3);
    }
    __syncwarp();
    uint32_t pb0 = 0u, pb1 = 0u;
    if (g < G) {
      pb0 = *reinterpret_cast<const uint32_t*>(pt + g * PS + 2 * t);
      pb1 = *reinterpret_cast<const uint32_t*>(pt + g * PS + 2 * t + 8);
    }
    if (__any_sync(FULL, al0 != 1.f || al1 != 1.f)) {
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        o[mt][0] *= al0;
        o[mt][1] *= al1;
        o[mt][2] *= al0;
        o[mt][3] *= al1;
      }
    }
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      uint32_t a[4];
      ldsm_x4_trans(a, vb + swz(v_key, 16 * mt + v_col));
      mma_16816(o[mt], a, pb0, pb1);
    }
    __syncwarp();
    if (k + C::STAGES < sg.n_my) {
      if (lane == 0) fence_proxy_async_smem();
      sg.issue(d, layer, sm, loads, k + C::STAGES, warp, lane);
    }
  }
  return -1;
}

// publish_warp for the tensor-core state: completes each row's sum over the lanes
// holding its keys and writes (m, l) and the row's unnormalised output.
template <class C>
__device__ void publish_warp_mma(const Smem<C>& sm, const float (&m_run)[2],
                                 const float (&l_run)[2], const float (&o)[8][4], int warp,
                                 int lane) {
  constexpr int D = C::D;
  const int g = lane >> 2, t = lane & 3;
  float l0 = l_run[0], l1 = l_run[1];
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    l0 += __shfl_xor_sync(FULL, l0, off);
    l1 += __shfl_xor_sync(FULL, l1, off);
  }
  if (t < 2) {
    const int r0 = warp * G + 2 * t, r1 = r0 + 1;
    if (g == 0) {
      sm.m_ml[r0 * 2 + 0] = m_run[0];
      sm.m_ml[r0 * 2 + 1] = l0;
      sm.m_ml[r1 * 2 + 0] = m_run[1];
      sm.m_ml[r1 * 2 + 1] = l1;
    }
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      sm.m_o[r0 * D + 16 * mt + g] = o[mt][0];
      sm.m_o[r1 * D + 16 * mt + g] = o[mt][1];
      sm.m_o[r0 * D + 16 * mt + g + 8] = o[mt][2];
      sm.m_o[r1 * D + 16 * mt + g + 8] = o[mt][3];
    }
  }
}

}  // namespace

}  // namespace kvc
