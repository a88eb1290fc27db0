// Chunked-prefill GQA attention over the retained cache.
//
// For each session of the last append (T <= 32 tokens, e.g. the 17 acoustic
// positions of a one-second unit), each KV head and its G = 4 query heads, the
// T*G query rows attend to every resident key at or before their own position
// (causal inside the chunk).  Split-K work items as in decode.
//
// bfloat16 runs on the tcgen05 tensor cores (kvc_attn_prefill_tc.cu); this
// file holds the launcher, the TMA tensor maps over the pool and the binary32
// CUDA-core kernel (one thread per query row).
#include <cuda.h>

#include <algorithm>

#include "kvc_launch.cuh"

namespace kvc {

namespace {

constexpr int PF_D = 128;  // head dim of the bfloat16 pool views
constexpr int G = 4;
constexpr float LOG2E = 1.4426950408889634f;

// ---------------------------------------------------------------------------
// binary32 prefill on CUDA cores: one thread per query row (T*G <= 128).
// ---------------------------------------------------------------------------
constexpr int F32_D = 64;
constexpr int F32_THREADS = 128;
constexpr int F32_TILE = PS * F32_D * 4;  // 4 KiB

__global__ void __launch_bounds__(F32_THREADS) attn_prefill_f32_kernel(
    Dev d, int layer, const float* __restrict__ q, float* __restrict__ out, float qk_scale) {
  __shared__ __align__(128) uint8_t tiles[2][2 * F32_TILE];
  __shared__ uint64_t bars[2];
  __shared__ int s_last;
  const int tid = threadIdx.x;
  if (tid == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
  }
  __syncthreads();
  const int H = d.kv_heads;
  const int n_items = d.g->n_pf_items * H;
  uint32_t loads = 0;
  for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
    const int item = it / H, head = it % H;
    const Item itm = d.pf_items[item];
    const SeqInfo si = d.seq[itm.seq];
    const int32_t* hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    const int32_t* lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    const int R = si.t * G;
    const int n_res = si.n_hist + si.n_live;
    const int r = tid;
    const bool live = r < R;
    const int t = r / G, g = r % G;
    const int qlog = n_res - si.t + t;
    float qr[F32_D], acc[F32_D];
    if (live) {
      const float* qrow = q + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * F32_D;
      const float2* cs = d.rope + (size_t)(si.pos_first + t) * (F32_D / 2);
#pragma unroll
      for (int j = 0; j < F32_D / 2; ++j) {
        const float a = qrow[j], b = qrow[j + F32_D / 2];
        const float2 c = cs[j];
        qr[j] = fmaf(a, c.x, -b * c.y) * qk_scale;
        qr[j + F32_D / 2] = fmaf(b, c.x, a * c.y) * qk_scale;
      }
    }
#pragma unroll
    for (int j = 0; j < F32_D; ++j) acc[j] = 0.f;
    float m = -INFINITY, l = 0.f;
    const int nblk = itm.blk_end - itm.blk_begin;
    auto issue = [&](int k) {
      const BlockRef br = block_ref(si, hrow, lrow, itm.blk_begin + k);
      const int st = (loads + k) & 1;
      const float* kp = reinterpret_cast<const float*>(d.pool) +
                        pool_offset_elems(d, br.page, layer, 0, head, 0);
      mbar_arrive_expect_tx(&bars[st], 2 * F32_TILE);
      bulk_g2s(tiles[st], kp, F32_TILE, &bars[st]);
      bulk_g2s(tiles[st] + F32_TILE, kp + (size_t)H * PS * F32_D, F32_TILE, &bars[st]);
    };
    if (tid == 0) {
      for (int k = 0; k < min(2, nblk); ++k) issue(k);
    }
    bool failed = false;
    for (int k = 0; k < nblk; ++k) {
      const uint32_t n = loads + k;
      if (!__syncthreads_and(mbar_wait(d, &bars[n & 1], (n >> 1) & 1))) {
        failed = true;
        break;
      }
      const float* kt = reinterpret_cast<const float*>(tiles[n & 1]);
      const float* vt = kt + PS * F32_D;
      const BlockRef br = block_ref(si, hrow, lrow, itm.blk_begin + k);
      if (live) {
        float s[PS];
        float mx = -INFINITY;
#pragma unroll
        for (int key = 0; key < PS; ++key) {
          float a = 0.f;
#pragma unroll
          for (int j = 0; j < F32_D; ++j) a = fmaf(qr[j], kt[key * F32_D + j], a);
          const bool v = key >= br.lo && key < br.hi && br.base + key <= qlog;
          s[key] = v ? a : -INFINITY;
          mx = fmaxf(mx, s[key]);
        }
        const float mn = fmaxf(m, mx);
        const float al = exp2_safe(m, mn);
        float rs = 0.f;
#pragma unroll
        for (int key = 0; key < PS; ++key) {
          s[key] = exp2_safe(s[key], mn);
          rs += s[key];
        }
        l = l * al + rs;
        m = mn;
#pragma unroll
        for (int j = 0; j < F32_D; ++j) {
          float a = acc[j] * al;
#pragma unroll
          for (int key = 0; key < PS; ++key) a = fmaf(s[key], vt[key * F32_D + j], a);
          acc[j] = a;
        }
      }
      __syncthreads();
      if (tid == 0 && k + 2 < nblk) {
        fence_proxy_async_smem();
        issue(k + 2);
      }
    }
    if (failed) return;  // CTA-uniform (__syncthreads_and)
    loads += nblk;
    const bool single = si.pf_chunks == 1;
    const int slot = (si.pf_base + itm.chunk) * H + head;
    if (live) {
      if (single) {
        float* orow = out + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * F32_D;
        for (int j = 0; j < F32_D; ++j) orow[j] = acc[j] / l;
      } else {
        float* prow = d.pf_part_o + ((size_t)slot * (PF_MAX_TOKENS * G) + r) * PF_D;
        for (int j = 0; j < F32_D; ++j) prow[j] = acc[j];
        d.pf_part_ml[(size_t)slot * (PF_MAX_TOKENS * G) + r] = make_float2(m, l);
      }
    }
    if (!single) {
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int old = atomicAdd(&d.pf_count[itm.seq * H + head], 1);
        s_last = (old == si.pf_chunks - 1);
      }
      __syncthreads();
      if (s_last && live) {
        __threadfence();
        const int s0 = si.pf_base * H + head;
        float M = -INFINITY;
        for (int ch = 0; ch < si.pf_chunks; ++ch)
          M = fmaxf(M, __ldcg(&d.pf_part_ml[(size_t)(s0 + ch * H) * (PF_MAX_TOKENS * G) + r]).x);
        float Lsum = 0.f;
        float* orow = out + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * F32_D;
        for (int j = 0; j < F32_D; ++j) acc[j] = 0.f;
        for (int ch = 0; ch < si.pf_chunks; ++ch) {
          const size_t sl = (size_t)(s0 + ch * H) * (PF_MAX_TOKENS * G) + r;
          const float2 ml = __ldcg(&d.pf_part_ml[sl]);
          const float sc = exp2_safe(ml.x, M);
          Lsum += ml.y * sc;
          for (int j = 0; j < F32_D; ++j) acc[j] += __ldcg(&d.pf_part_o[sl * PF_D + j]) * sc;
        }
        for (int j = 0; j < F32_D; ++j) orow[j] = acc[j] / Lsum;
      }
      __syncthreads();
      if (s_last && tid == 0) d.pf_count[itm.seq * H + head] = 0;
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Host side: tensor maps over the pool (two 2-D views, dims 0-63 and 64-127).
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &p, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

struct PoolMaps {
  const uint8_t* pool = nullptr;
  uint64_t rows = 0;
  CUtensorMap lo, hi;
  bool ok = false;
};

uint64_t pool_rows(const Dev& d) {
  return (uint64_t)d.n_pages * d.layers * 2 * d.kv_heads * PS;
}

bool make_pool_maps(const Dev& d, PoolMaps& m) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  const uint64_t rows = pool_rows(d);
  cuuint64_t dims[2] = {64, rows};
  cuuint64_t strides[1] = {(cuuint64_t)PF_D * 2};
  cuuint32_t box[2] = {64, PS};
  cuuint32_t estr[2] = {1, 1};
  CUresult r1 = enc(&m.lo, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)d.pool, dims, strides, box,
                    estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  CUresult r2 = enc(&m.hi, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, (void*)(d.pool + 128), dims,
                    strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  m.ok = (r1 == CUDA_SUCCESS && r2 == CUDA_SUCCESS);
  m.pool = d.pool;
  m.rows = rows;
  return m.ok;
}

}  // namespace

bool pool_tensor_maps(const Dev& d, CUtensorMap* lo, CUtensorMap* hi) {
  // Keyed on the pool's address and extent: a later context may get the same address
  // for a pool of another shape.
  static thread_local PoolMaps maps;
  if (!maps.ok || maps.pool != d.pool || maps.rows != pool_rows(d)) {
    if (!make_pool_maps(d, maps)) return false;
  }
  *lo = maps.lo;
  *hi = maps.hi;
  return true;
}

namespace {

template <int MT>
int pf_grid(const void* fn, int threads, int smem) {
  cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, smem);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return max(1, per_sm) * sms;
}

}  // namespace

int prefill_grid_ctas(const Dev& d) {
  if (d.esz == 2)
    return pf_grid<0>(prefill_tc_kernel_ptr(), prefill_tc_threads(), prefill_tc_smem());
  return pf_grid<0>(reinterpret_cast<const void*>(&attn_prefill_f32_kernel), F32_THREADS, 0);
}

cudaError_t launch_attn_prefill(const Dev& d, int layer, const void* q, void* out, int n_seq,
                                int max_t, bool pdl, cudaStream_t s, const void* new_k,
                                const void* new_v) {
  (void)n_seq;
  (void)max_t;
  if (d.esz == 2) {
    static thread_local int gtc = 0;
    CUtensorMap lo, hi;
    if (!pool_tensor_maps(d, &lo, &hi)) return cudaErrorInvalidValue;
    if (!gtc) gtc = pf_grid<0>(prefill_tc_kernel_ptr(), prefill_tc_threads(), prefill_tc_smem());
    // Each CTA of the stream-K split may write two partial slots.
    return launch_attn_prefill_tc(d, layer, lo, hi, q, out, std::min(gtc, d.max_pf_items / 2),
                                  pdl, s, new_k, new_v);
  }
  if (new_k != nullptr) return cudaErrorInvalidValue;  // binary32: the API writes the rows first
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  static thread_local int gf = 0;
  if (!gf) gf = pf_grid<0>(reinterpret_cast<const void*>(&attn_prefill_f32_kernel), F32_THREADS, 0);
  attn_prefill_f32_kernel<<<gf, F32_THREADS, 0, s>>>(d, layer, static_cast<const float*>(q),
                                                     static_cast<float*>(out), scale);
  return cudaGetLastError();
}

}  // namespace kvc
