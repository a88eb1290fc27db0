// Single-token decode GQA attention over the retained cache.
//
// For each session of the last append (one token each), each KV head h and
// its G = 4 query heads: out = softmax(RoPE(q, p) . k / sqrt(D)) v over every
// resident key (the compacted region, then the live region, the token's own
// key included).
//
// Inside a CTA each warp streams its own pages through a TMA copy ring in shared
// memory and computes its scores and P V products, on the tensor cores (mma.sync)
// for bfloat16 and on CUDA cores (packed fp32 FMA) for binary32, keeping a running
// max/sum; the CTA then merges its warps.  Two ways to spread the pages over CTAs
// (split-K):
//   - stream-K (many sessions): the call's (session, head, page) units are cut
//     into equal contiguous ranges, one per CTA of 4 warps (three CTAs per SM);
//   - pair split (fewer sessions): each (session, head) pair's pages are cut into
//     k slices, one per CTA, so that a call's CTAs fill the GPU in one wave.
// Either way partial states go to global slots and the last CTA to arrive for a
// pair merges them (log-sum-exp).  Stream-K publishes them with an acquire-release
// arrival.  The 16-warp pair split, whose launches are latency-bound, writes each
// partial value as a word tagged with the launch and arrives with a relaxed atomic,
// so no release fence sits on its critical path; the merging CTA re-reads the words
// whose tag is not yet current.  Launches captured into a graph (where a replay
// would repeat the tag) use the acquire-release arrival.
//
// This file holds the stream-K kernel; the pair-split kernel is in
// kvc_attn_decode_split.cu and the dispatch between the tiers in
// kvc_decode_dispatch.cu.
#include "kvc_decode_common.cuh"

namespace kvc {

namespace {

// ---------------------------------------------------------------------------
// Stream-K kernel.
// ---------------------------------------------------------------------------
template <typename T, int D, bool FUSED>
__global__ void __launch_bounds__(SkCfg<T, D>::THREADS) attn_decode_kernel(
    Dev d, int layer, const __grid_constant__ CUtensorMap map_lo,
    const __grid_constant__ CUtensorMap map_hi, const T* __restrict__ q, T* __restrict__ out,
    float qk_scale, int min_units, const T* new_k, const T* new_v) {
  using C = SkCfg<T, D>;
  static_assert(C::WARPS == G, "the split-K merge maps one warp to one query row");
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const Smem<C> sm(smem, warp);
  __shared__ int s_last, s_abort;
  init_warp_barriers<C>(sm.wbars, lane);
  if (tid == 0) s_abort = 0;
  __syncthreads();
  // The next attention call may start its CTAs as soon as slots free up.  Before
  // pdl_wait() this kernel reads only what the append wrote (work list, page
  // tables, K/V pages); q, outputs, partials and counters come after it.
  pdl_launch_dependents();
  bool waited = false;

  // Stream-K: this CTA's contiguous range of the call's units (UnitSplit).
  const int H = d.kv_heads;
  const UnitSplit us = unit_split(d, gridDim.x, min_units, MAX_PARTS);
  if ((int)blockIdx.x >= us.n_cta) return;
  const int cta = blockIdx.x;
  const int u_begin = us.start_of(cta), u_end = us.start_of(cta + 1);
  uint32_t loads = 0;  // loads issued (== consumed) by this warp so far

  for (int u = u_begin; u < u_end;) {
    const UnitSeg seg = unit_segment(d, u, u_end);
    const SeqInfo& si = seg.si;
    const int seq = seg.seq, head = seg.head;
    const int pair_start = seg.pair_start, pair_end = seg.pair_end, seg_end = seg.end;

    Segment<C> sg;
    sg.init(d, si, head, u - pair_start, seg_end - u, warp, &map_lo, &map_hi);
    sg.prefetch(d, layer, sm, loads, warp, lane);
    if (!waited) {
      if (warp == 0) prefetch_q<C>(d, si, head, q, lane);
      pdl_wait();
      waited = true;
    }
    int failed_at;
    // The page loop's state: tensor-core fragments (bfloat16) or CUDA-core rows.
    float m2[2] = {-INFINITY, -INFINITY}, l2[2] = {0.f, 0.f};
    float o[8][4];
    float m_run = -INFINITY, l_run = 0.f;  // for row lane >> 3
    float2 acc[G][C::PVD / 2];
    if constexpr (C::MMA) {
      uint32_t qb[8][2];
      load_q_mma<C>(d, si, head, q, qk_scale, lane, qb);
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
      failed_at = stream_pages_mma<C, FUSED>(d, layer, sg, sm, loads, qb, m2, l2, o, warp, lane,
                                             new_k, new_v);
    } else {
      float qr[G][2 * C::VEC];
      load_q<C>(d, si, head, q, qk_scale, lane, qr);
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int j = 0; j < C::PVD / 2; ++j) acc[g][j] = make_float2(0.f, 0.f);
      failed_at = stream_pages<C, FUSED>(d, layer, sg, sm, loads, qr, m_run, l_run, acc, warp,
                                         lane, new_k, new_v);
    }
    if (failed_at >= 0 && lane == 0) s_abort = 1;
    __syncthreads();
    if (s_abort) {
      // Some wait gave up: each warp drains the copies it still has in flight
      // (bounded waits), then the whole CTA stops together.
      if (failed_at >= 0) {
        for (int k = failed_at; k < min(sg.n_my, failed_at + C::STAGES); ++k) {
          const uint32_t n = loads + k;
          mbar_wait(d, &sm.wbars[n % C::STAGES], (n / C::STAGES) & 1);
        }
      }
      return;
    }
    loads += sg.n_my;

    // Merge the four warps' partial softmax states (stage buffers are free now).
    if constexpr (C::MMA)
      publish_warp_mma<C>(sm, m2, l2, o, warp, lane);
    else
      publish_warp<C>(sm, m_run, l_run, acc, warp, lane);
    __syncthreads();
    merge_warps<C>(sm, warp, lane);
    const bool whole = u == pair_start && seg_end == pair_end;
    const int slot = 2 * cta + (u == u_begin ? 0 : 1);
    for (int e = tid; e < G * D; e += C::THREADS) {
      const float O = merge_warps_elem<C>(sm, e);
      const int g = e / D, dd = e % D;
      if (whole) {
        out[((size_t)si.q_row0 * d.q_heads + head * G + g) * D + dd] =
            from_float<T>(O / sm.r_ml[g * 2 + 1]);
      } else {
        d.dec_part_o[((size_t)slot * G + g) * D + dd] = O;
        if (dd == 0)
          d.dec_part_ml[(size_t)slot * G + g] = make_float2(sm.r_ml[g * 2], sm.r_ml[g * 2 + 1]);
      }
    }
    if (!whole) {
      // The CTAs cf..cl own the pair's units; the last of them to arrive merges.
      const int cf = us.owner(pair_start), cl = us.owner(pair_end - 1);
      const int nch = cl - cf + 1;
      if (arrive_last(&d.dec_count[seq * H + head], nch, tid, &s_last)) {
        const int first_slot = us.slot_of(cf, cf, pair_start);
        merge_parts<C>(d, sm, nch, [&](int ch) { return ch ? 2 * (cf + ch) : first_slot; },
                       out + ((size_t)si.q_row0 * d.q_heads + head * G) * D, tid, warp, lane);
        if (tid == 0) d.dec_count[seq * H + head] = 0;
      }
    }
    __syncthreads();
    u = seg_end;
  }
}

// Resident CTAs of the stream-K kernel (its grid), capped by the partial slots.
template <typename T, int D>
int stream_k_grid(const Dev& d) {
  const void* fn = reinterpret_cast<const void*>(&attn_decode_kernel<T, D, false>);
  const int smem = SkCfg<T, D>::SMEM;
  cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaFuncSetAttribute(reinterpret_cast<const void*>(&attn_decode_kernel<T, D, true>),
                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, SkCfg<T, D>::THREADS, smem);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // Every CTA of the stream-K split may write two partial slots.
  return min(d.dec_slots / 2, max(1, per_sm) * sms);
}

}  // namespace

int decode_stream_k_grid(const Dev& d) {
  return d.esz == 2 ? stream_k_grid<__nv_bfloat16, 128>(d) : stream_k_grid<float, 64>(d);
}

cudaError_t launch_attn_decode_streamk(const Dev& d, int layer, const CUtensorMap& map_lo,
                                       const CUtensorMap& map_hi, const void* q, void* out,
                                       float scale, int grid, int min_units, const void* new_k,
                                       const void* new_v, bool pdl, cudaStream_t s) {
  if (d.esz == 2) {
    using T = __nv_bfloat16;
    const T* nk = static_cast<const T*>(new_k);
    const T* nv = static_cast<const T*>(new_v);
    return launch_ex(nk ? &attn_decode_kernel<T, 128, true> : &attn_decode_kernel<T, 128, false>,
                     dim3(grid), dim3(SkCfg<T, 128>::THREADS), SkCfg<T, 128>::SMEM, s, pdl, d,
                     layer, map_lo, map_hi, static_cast<const T*>(q), static_cast<T*>(out), scale,
                     min_units, nk, nv);
  }
  const float* nk = static_cast<const float*>(new_k);
  const float* nv = static_cast<const float*>(new_v);
  return launch_ex(nk ? &attn_decode_kernel<float, 64, true> : &attn_decode_kernel<float, 64, false>,
                   dim3(grid), dim3(SkCfg<float, 64>::THREADS), SkCfg<float, 64>::SMEM, s, pdl, d,
                   layer, map_lo, map_hi, static_cast<const float*>(q), static_cast<float*>(out),
                   scale, min_units, nk, nv);
}

}  // namespace kvc
