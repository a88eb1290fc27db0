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
  // shared memory per warp: STAGES x (K tile + V tile) + scores + probs + alpha
  static constexpr int WARP_BYTES = STAGES * 2 * TILE + (G * PS + PS * G + G) * 4 + 16;
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
                                                                  float qk_scale) {
  using C = DecCfg<T, D, STAGES>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint8_t* wbase = smem + warp * C::WARP_BYTES;
  uint8_t* tiles = wbase;                                            // [STAGES][2][TILE]
  float* s_sc = reinterpret_cast<float*>(wbase + STAGES * 2 * C::TILE);  // [G][PS]
  float* s_p = s_sc + G * PS;                                        // [PS][G]
  float* s_alpha = s_p + PS * G;                                     // [G]
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

  const int n_items = d.g->n_dec_items * d.kv_heads;
  const size_t head_stride = (size_t)PS * D;  // elements between heads in a page
  uint32_t loads = 0;  // loads issued (== consumed) by this warp so far
  const int half = lane >> 4, c = lane & 15;

  for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
    const int item = it / d.kv_heads, head = it % d.kv_heads;
    const Item itm = d.dec_items[item];
    const SeqInfo si = d.seq[itm.seq];
    const int32_t* hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    const int32_t* lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    const int pos = si.pos_first;  // the single token of this session

    const int nblk = itm.blk_end - itm.blk_begin;
    const int n_my = (nblk > warp) ? (nblk - warp + DEC_WARPS - 1) / DEC_WARPS : 0;
    // Page ids of this warp's blocks, 32 at a time: lane j holds block (win + j),
    // so one round trip to the page table serves 32 loads.  Called warp-wide.
    int pwin = -32, pid = 0;
    auto issue = [&](int k) {
      if (k >= pwin + 32) {
        pwin = k & ~31;
        const int j = pwin + lane;
        pid = j < n_my ? block_page(si, hrow, lrow, itm.blk_begin + warp + j * DEC_WARPS) : 0;
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
        bulk_g2s(dst + C::TILE, kp + d.kv_heads * head_stride, C::TILE, &wbars[st]);
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
    float acc[G][C::PVD];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < C::PVD; ++j) acc[g][j] = 0.f;

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
      const BlockRange br = block_range(si, itm.blk_begin + warp + k * DEC_WARPS);

      // Scores: lanes 0-15 take even keys, 16-31 odd keys; each lane a 16-byte chunk.
#pragma unroll
      for (int i = 0; i < PS / 2; ++i) {
        const int key = 2 * i + half;
        float kf[C::VEC];
        load_vec<T>(kt + key * C::ROW_BYTES + c * 16, kf);
        float a[G];
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float s = 0.f;
#pragma unroll
          for (int e = 0; e < C::VEC; ++e) s = fmaf(qr[g][e], kf[e], s);
          a[g] = s;
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
        s_p[kk * G + g] = p0;
        s_p[(kk + 1) * G + g] = p1;
        if ((lane & 7) == 0) s_alpha[g] = alpha;
      }
      __syncwarp();
      // PV: lane owns dims [PVD*lane, PVD*lane + PVD) of all G rows.
      {
        const float4 al = *reinterpret_cast<const float4*>(s_alpha);
        const float alv[G] = {al.x, al.y, al.z, al.w};
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int j = 0; j < C::PVD; ++j) acc[g][j] *= alv[g];
#pragma unroll
        for (int key = 0; key < PS; ++key) {
          const float4 pk = *reinterpret_cast<const float4*>(s_p + key * G);
          float vf[C::PVD];
          load_pv<T>(vt + key * C::ROW_BYTES + lane * C::PVD * C::ESZ, vf);
#pragma unroll
          for (int j = 0; j < C::PVD; ++j) {
            acc[0][j] = fmaf(pk.x, vf[j], acc[0][j]);
            acc[1][j] = fmaf(pk.y, vf[j], acc[1][j]);
            acc[2][j] = fmaf(pk.z, vf[j], acc[2][j]);
            acc[3][j] = fmaf(pk.w, vf[j], acc[3][j]);
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
      for (int j = 0; j < C::PVD; ++j) m_o[(warp * G + g) * D + lane * C::PVD + j] = acc[g][j];
    __syncthreads();
    const int slot = (si.dec_base + itm.chunk) * d.kv_heads + head;
    const bool single = si.dec_chunks == 1;
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
      if (single) {
        out[((size_t)si.q_row0 * d.q_heads + head * G + g) * D + dd] = from_float<T>(O / L);
      } else {
        d.dec_part_o[((size_t)slot * G + g) * D + dd] = O;
        if (dd == 0) d.dec_part_ml[(size_t)slot * G + g] = make_float2(M, L);
      }
    }
    if (!single) {
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int old = atomicAdd(&d.dec_count[itm.seq * d.kv_heads + head], 1);
        s_last = (old == si.dec_chunks - 1);
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        // Log-sum-exp merge of the session's chunks: warp g reduces row g's maxima and
        // sums over the chunks (lanes stride the chunks), leaving each chunk's weight
        // divided by the total in shared memory; then all threads sum the weighted
        // partial outputs over (row, dim) with independent loads in flight.
        const int s0 = si.dec_base * d.kv_heads + head;
        const int nch = si.dec_chunks;
        {
          const int g = warp;  // DEC_WARPS == G
          float M = -INFINITY;
          for (int ch = lane; ch < nch; ch += 32)
            M = fmaxf(M, __ldcg(&d.dec_part_ml[(size_t)(s0 + ch * d.kv_heads) * G + g]).x);
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(FULL, M, o));
          float L = 0.f;
          for (int ch = lane; ch < nch; ch += 32) {
            const float2 ml = __ldcg(&d.dec_part_ml[(size_t)(s0 + ch * d.kv_heads) * G + g]);
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
        // Each thread owns EPT output elements; per chunk it issues their loads
        // together (two chunks per iteration), so many loads are in flight.
        constexpr int EPT = G * D / DEC_THREADS;
        const size_t cstride = (size_t)d.kv_heads * G * D;
        const float* base = d.dec_part_o + (size_t)s0 * G * D;
        float O[EPT];
#pragma unroll
        for (int i = 0; i < EPT; ++i) O[i] = 0.f;
        int ch = 0;
        for (; ch + 2 <= nch; ch += 2) {
          float a0[EPT], a1[EPT];
#pragma unroll
          for (int i = 0; i < EPT; ++i) {
            a0[i] = __ldcg(base + ch * cstride + tid + i * DEC_THREADS);
            a1[i] = __ldcg(base + (ch + 1) * cstride + tid + i * DEC_THREADS);
          }
#pragma unroll
          for (int i = 0; i < EPT; ++i) {
            const int g = (tid + i * DEC_THREADS) / D;
            O[i] += a0[i] * s_scale[ch * G + g] + a1[i] * s_scale[(ch + 1) * G + g];
          }
        }
        for (; ch < nch; ++ch) {
#pragma unroll
          for (int i = 0; i < EPT; ++i) {
            const int g = (tid + i * DEC_THREADS) / D;
            O[i] += __ldcg(base + ch * cstride + tid + i * DEC_THREADS) * s_scale[ch * G + g];
          }
        }
#pragma unroll
        for (int i = 0; i < EPT; ++i) {
          const int e = tid + i * DEC_THREADS;
          out[((size_t)si.q_row0 * d.q_heads + head * G) * D + e] = from_float<T>(O[i]);
        }
        if (tid == 0) d.dec_count[itm.seq * d.kv_heads + head] = 0;
      }
    }
    __syncthreads();
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

cudaError_t launch_attn_decode(const Dev& d, int layer, const void* q, void* out, int n_seq,
                               bool pdl, cudaStream_t s) {
  (void)n_seq;
  static thread_local int grid_bf16 = 0, grid_f32 = 0;
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  if (d.esz == 2) {
    if (!grid_bf16) grid_bf16 = decode_grid_ctas(d);
    return launch_ex(&attn_decode_kernel<__nv_bfloat16, 128, DEC_STAGES>, dim3(grid_bf16),
                     dim3(DEC_THREADS), dec_smem<__nv_bfloat16, 128>(), s, pdl, d, layer,
                     static_cast<const __nv_bfloat16*>(q), static_cast<__nv_bfloat16*>(out), scale);
  }
  if (!grid_f32) grid_f32 = decode_grid_ctas(d);
  return launch_ex(&attn_decode_kernel<float, 64, DEC_STAGES>, dim3(grid_f32), dim3(DEC_THREADS),
                   dec_smem<float, 64>(), s, pdl, d, layer, static_cast<const float*>(q),
                   static_cast<float*>(out), scale);
}

}  // namespace kvc
