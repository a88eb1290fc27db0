// Single-token decode attention, pair-split kernel (calls of few sessions): CTA
// c takes slice c % k of (session, KV head) pair c / k, the pair's pages cut into
// k equal slices, so that every page of a small call is in flight at once.  The
// bfloat16 pages run on the tensor cores (mma.sync) in both CTA shapes.  With 16
// warps (one CTA per SM) the partial states are tagged 64-bit words merged after a
// relaxed arrival; with 4 warps (three CTAs per SM) the acquire-release arrival of
// stream-K is used.
#include "kvc_decode_common.cuh"

// Shape constants of the CUDA-core loop are unused by the tensor-core shapes.
#pragma nv_diag_suppress 177

namespace kvc {

namespace {

// Tagged partial state of slot `slot`: G * D output words, then (m, l) per row.
template <class C>
__device__ inline unsigned long long* tagged_slot(const Dev& d, int slot) {
  return d.dec_tagged + (size_t)slot * (G * C::D + 2 * G);
}

// Write this CTA's merged warps (merge_warps done) as the tagged partial state of
// `slot`.  Called by every thread.
template <class C>
__device__ void publish_tagged(const Dev& d, const Smem<C>& sm, int slot, uint32_t tag,
                               int tid) {
  unsigned long long* ts = tagged_slot<C>(d, slot);
  for (int e = tid; e < G * C::D; e += C::THREADS) st_tagged(ts + e, tag, merge_warps_elem<C>(sm, e));
  if (tid < 2 * G) st_tagged(ts + G * C::D + tid, tag, sm.r_ml[tid]);
}

// Re-read, all in one pass, the words of w[] (loaded from p(i)) whose tag is not
// yet `tag`, until every word carries it: the stores of the other CTAs were issued
// before their arrivals and land within a round trip or two, so reloading every
// stale word at once costs about one round trip instead of one per stale word.
// Gives up (KVC_DERR_WAIT) after WAIT_LIMIT_CYCLES, keeping the stale values.
template <int N, typename PtrFn>
__device__ inline void settle_tagged(const Dev& d, unsigned long long (&w)[N], uint32_t tag,
                                     PtrFn p) {
  long long t0 = 0;
  for (bool first = true;; first = false) {
    bool stale = false;
#pragma unroll
    for (int i = 0; i < N; ++i) {
      if ((uint32_t)(w[i] >> 32) != tag) {
        w[i] = ld_tagged(p(i));
        stale = true;
      }
    }
    if (!stale) return;
    if (first) {
      t0 = clock64();
    } else if (clock64() - t0 > WAIT_LIMIT_CYCLES) {
      set_error(d, KVC_DERR_WAIT);
      return;
    }
  }
}

// merge_parts over the tagged states of slots slot0 .. slot0 + nch - 1 of this
// launch (tag): every load is a single 64-bit word whose tag says whether its
// store has landed.
template <class C>
__device__ void merge_tagged(const Dev& d, const Smem<C>& sm, int nch, int slot0, uint32_t tag,
                             typename C::T* orow, int tid, int warp, int lane) {
  using T = typename C::T;
  constexpr int D = C::D, TW = G * D + 2 * G;
  static_assert(C::WARPS >= G, "one warp per query row");
  constexpr int EPT = (G * D + C::THREADS - 1) / C::THREADS;
  constexpr int CH = 24 / EPT > 0 ? 24 / EPT : 1;
  const unsigned long long* base = tagged_slot<C>(d, slot0);
  const unsigned long long filler = (unsigned long long)tag << 32;  // 0.0f, current tag
  unsigned long long a[CH * EPT];
  auto word = [&](int c0, int j) -> const unsigned long long* {
    return base + (size_t)(c0 + j / EPT) * TW + tid + (j % EPT) * C::THREADS;
  };
  auto load_batch = [&](int c0) {
#pragma unroll
    for (int j = 0; j < CH * EPT; ++j) {
      const int e = tid + (j % EPT) * C::THREADS;
      a[j] = (c0 + j / EPT < nch && e < G * D) ? ld_tagged(word(c0, j)) : filler;
    }
  };
  load_batch(0);
  if (warp < G) {
    const int g = warp;
    constexpr int PL = MAX_PARTS / 32;
    unsigned long long wml[2 * PL];
    auto ml_word = [&](int j) -> const unsigned long long* {
      return base + (size_t)(lane + 32 * (j / 2)) * TW + G * D + 2 * g + (j % 2);
    };
#pragma unroll
    for (int j = 0; j < 2 * PL; ++j)
      wml[j] = lane + 32 * (j / 2) < nch ? ld_tagged(ml_word(j)) : filler;
    settle_tagged(d, wml, tag, ml_word);
    float m[PL], l[PL], M = -INFINITY;
#pragma unroll
    for (int i = 0; i < PL; ++i) {
      const int ch = lane + 32 * i;
      m[i] = ch < nch ? __uint_as_float((uint32_t)wml[2 * i]) : -INFINITY;
      l[i] = ch < nch ? __uint_as_float((uint32_t)wml[2 * i + 1]) : 0.f;
      M = fmaxf(M, m[i]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(FULL, M, o));
    float sc[PL], L = 0.f;
#pragma unroll
    for (int i = 0; i < PL; ++i) {
      sc[i] = exp2_safe(m[i], M);
      L += l[i] * sc[i];
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
    settle_tagged(d, a, tag, [&](int j) { return word(c0, j); });
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      if (c0 + i >= nch) break;
#pragma unroll
      for (int t = 0; t < EPT; ++t) {
        const int e = tid + t * C::THREADS;
        if (e < G * D)
          O[t] += __uint_as_float((uint32_t)a[i * EPT + t]) * sm.s_scale[(c0 + i) * G + e / D];
      }
    }
    c0 += CH;
    if (c0 >= nch) break;
    load_batch(c0);
  }
#pragma unroll
  for (int t = 0; t < EPT; ++t) {
    const int e = tid + t * C::THREADS;
    if (e < G * D) orow[e] = from_float<T>(O[t]);
  }
}

// A wait of this warp's page loop gave up at page failed_at (error recorded):
// drain the copies it still has in flight (bounded waits).  Pair-split layout
// (loads start at 0).
template <class C>
__device__ inline void drain_after_failure(const Dev& d, const Smem<C>& sm, const Segment<C>& sg,
                                           int failed_at) {
  if (failed_at < 0) return;
  for (int j = failed_at; j < min(sg.n_my, failed_at + C::STAGES); ++j)
    mbar_wait(d, &sm.wbars[j % C::STAGES], (j / C::STAGES) & 1);
}

// ---------------------------------------------------------------------------
// Pair-split kernel (few sessions): CTA c takes slice c % k of pair c / k, the
// pair's pages cut into k equal slices.  Each CTA's pages are issued before it
// waits on the previous kernel; the k partial states of a pair are merged by
// the last of its CTAs to finish.
// ---------------------------------------------------------------------------
template <typename T, int D, bool FUSED, class C>
__global__ void __launch_bounds__(C::THREADS) attn_decode_split_kernel(
    Dev d, int layer, const __grid_constant__ CUtensorMap map_lo,
    const __grid_constant__ CUtensorMap map_hi, const T* __restrict__ q, T* __restrict__ out,
    float qk_scale, int k, uint32_t epoch, const T* new_k, const T* new_v) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const Smem<C> sm(smem, warp);
  __shared__ int s_last;
  const int pair = blockIdx.x / k, slice = blockIdx.x % k;
  const int seq = pair / d.kv_heads, head = pair % d.kv_heads;
  init_warp_barriers<C>(sm.wbars, lane);
  __syncthreads();
  pdl_launch_dependents();

  const SeqInfo si = d.seq[seq];
  const int nb = si.n_blocks;
  const int b0 = (int)((int64_t)slice * nb / k), b1 = (int)((int64_t)(slice + 1) * nb / k);
  Segment<C> sg;
  sg.init(d, si, head, b0, b1 - b0, warp, &map_lo, &map_hi);
  sg.prefetch(d, layer, sm, 0, warp, lane);
  if (warp == 0) prefetch_q<C>(d, si, head, q, lane);
  pdl_wait();
  int failed_at;
  if constexpr (C::MMA) {
    uint32_t qb[8][2];
    load_q_mma<C>(d, si, head, q, qk_scale, lane, qb);
    float m2[2] = {-INFINITY, -INFINITY}, l2[2] = {0.f, 0.f};
    float o[8][4];
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    failed_at = stream_pages_mma<C, FUSED>(d, layer, sg, sm, 0, qb, m2, l2, o, warp, lane,
                                           new_k, new_v);
    if (failed_at >= 0) {
      m2[0] = m2[1] = -INFINITY;
      l2[0] = l2[1] = 0.f;
    }
    drain_after_failure<C>(d, sm, sg, failed_at);
    __syncthreads();
    publish_warp_mma<C>(sm, m2, l2, o, warp, lane);
  } else {
    float qr[G][2 * C::VEC];
    load_q<C>(d, si, head, q, qk_scale, lane, qr);
    float m_run = -INFINITY, l_run = 0.f;
    float2 acc[G][C::PVD / 2];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < C::PVD / 2; ++j) acc[g][j] = make_float2(0.f, 0.f);
    failed_at = stream_pages<C, FUSED>(d, layer, sg, sm, 0, qr, m_run, l_run, acc, warp, lane,
                                       new_k, new_v);
    if (failed_at >= 0) {
      m_run = -INFINITY;
      l_run = 0.f;
    }
    drain_after_failure<C>(d, sm, sg, failed_at);
    __syncthreads();
    publish_warp<C>(sm, m_run, l_run, acc, warp, lane);
  }
  __syncthreads();
  merge_warps<C>(sm, warp, lane);
  T* orow = out + ((size_t)si.q_row0 * d.q_heads + head * G) * D;
  const int slot = blockIdx.x;
  if (k > 1 && epoch != 0) {
    publish_tagged<C>(d, sm, slot, epoch, tid);
    __syncthreads();
    if (tid == 0) s_last = arrive_relaxed(&d.dec_count[pair], k);
    __syncthreads();
    if (!s_last) return;
    merge_tagged<C>(d, sm, k, pair * k, epoch, orow, tid, warp, lane);
    if (tid == 0) d.dec_count[pair] = 0;
    return;
  }
  for (int e = tid; e < G * D; e += C::THREADS) {
    const float O = merge_warps_elem<C>(sm, e);
    const int g = e / D;
    if (k == 1) {
      orow[e] = from_float<T>(O / sm.r_ml[g * 2 + 1]);
    } else {
      d.dec_part_o[(size_t)slot * G * D + e] = O;
      if ((e % D) == 0)
        d.dec_part_ml[(size_t)slot * G + g] = make_float2(sm.r_ml[g * 2], sm.r_ml[g * 2 + 1]);
    }
  }
  if (k == 1) return;
  if (!arrive_last(&d.dec_count[pair], k, tid, &s_last)) return;
  merge_parts<C>(d, sm, k, [&](int ch) { return pair * k + ch; }, orow, tid, warp, lane);
  if (tid == 0) d.dec_count[pair] = 0;
}

// Resident CTAs of the pair-split kernel with CTA shape C (one wave).
template <typename T, int D, class C>
int split_slots() {
  const void* fn = reinterpret_cast<const void*>(&attn_decode_split_kernel<T, D, false, C>);
  const int smem = C::SMEM;
  cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaFuncSetAttribute(reinterpret_cast<const void*>(&attn_decode_split_kernel<T, D, true, C>),
                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, C::THREADS, smem);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return max(0, per_sm) * sms;
}

template <typename T, int D, class C>
cudaError_t launch_split(const Dev& d, int layer, const CUtensorMap& map_lo,
                         const CUtensorMap& map_hi, const void* q, void* out, float scale, int k,
                         uint32_t epoch, const void* new_k, const void* new_v, int n_pairs,
                         bool pdl, cudaStream_t s) {
  const bool fused = new_k != nullptr;
  return launch_ex(fused ? &attn_decode_split_kernel<T, D, true, C>
                         : &attn_decode_split_kernel<T, D, false, C>,
                   dim3(n_pairs * k), dim3(C::THREADS), C::SMEM, s, pdl, d, layer, map_lo, map_hi,
                   static_cast<const T*>(q), static_cast<T*>(out), scale, k, epoch,
                   static_cast<const T*>(new_k), static_cast<const T*>(new_v));
}

}  // namespace

int decode_split_slots(int esz, bool wide) {
  if (esz == 2)
    return wide ? split_slots<__nv_bfloat16, 128, SpCfg<__nv_bfloat16, 128>>()
                : split_slots<__nv_bfloat16, 128, Sp4Cfg<__nv_bfloat16, 128>>();
  return wide ? split_slots<float, 64, SpCfg<float, 64>>() : split_slots<float, 64, Sp4Cfg<float, 64>>();
}

bool decode_split_uses_tma(int esz, bool wide) {
  if (esz == 2) return wide ? SpCfg<__nv_bfloat16, 128>::MMA : Sp4Cfg<__nv_bfloat16, 128>::MMA;
  return false;
}

cudaError_t launch_attn_decode_split(const Dev& d, bool wide, int layer, const CUtensorMap& map_lo,
                                     const CUtensorMap& map_hi, const void* q, void* out,
                                     float scale, int k, uint32_t epoch, const void* new_k,
                                     const void* new_v, int n_pairs, bool pdl, cudaStream_t s) {
  if (d.esz == 2) {
    if (wide)
      return launch_split<__nv_bfloat16, 128, SpCfg<__nv_bfloat16, 128>>(
          d, layer, map_lo, map_hi, q, out, scale, k, epoch, new_k, new_v, n_pairs, pdl, s);
    return launch_split<__nv_bfloat16, 128, Sp4Cfg<__nv_bfloat16, 128>>(
        d, layer, map_lo, map_hi, q, out, scale, k, epoch, new_k, new_v, n_pairs, pdl, s);
  }
  if (wide)
    return launch_split<float, 64, SpCfg<float, 64>>(d, layer, map_lo, map_hi, q, out, scale, k,
                                                     epoch, new_k, new_v, n_pairs, pdl, s);
  return launch_split<float, 64, Sp4Cfg<float, 64>>(d, layer, map_lo, map_hi, q, out, scale, k,
                                                    epoch, new_k, new_v, n_pairs, pdl, s);
}

}  // namespace kvc
