// kvc_attn_decode_noalloc: the single-token decode attention of
// kvc_attn_decode, with its split-K scratch (per-chunk partial results and the
// per-(session, kv-head) arrival counters) held in a fixed array in device
// global memory owned by this library, instead of in the caller's metadata
// workspace.  The entry point allocates nothing.
//
// The array is a file-scope static __device__ object: every CUDA context that
// loads the library (one per device for runtime-API callers, who share the
// device's primary context) holds its own copy (NOALLOC_SCRATCH_BYTES) until the
// context is destroyed or the process exits.  All calls in one context share that
// copy, so calls whose kernels overlap on the GPU (different streams, or
// different library contexts over the same CUDA context) race on it and must be
// serialised by the caller.
#include <algorithm>
#include <mutex>

#include "kvc_launch.cuh"

namespace kvc {

namespace {

constexpr unsigned FULL = 0xFFFFFFFFu;
constexpr int NA_WARPS = 4;
constexpr int NA_THREADS = NA_WARPS * 32;
constexpr int G = 4;
constexpr int NA_STAGES = 2;
constexpr float LOG2E = 1.4426950408889634f;

// Capacity of the static scratch: partial slots of (session, chunk, kv-head),
// each G x D floats (D <= 128) plus G (max, sum) pairs, and one counter per
// (session, kv-head).
constexpr int NA_MAX_SLOTS = 4096;
constexpr int NA_MAX_PAIRS = 4096;   // (session, kv-head) pairs per call
constexpr int NA_MAX_CHUNKS = 16;    // chunks per session
constexpr size_t NA_PART_O_BYTES = (size_t)NA_MAX_SLOTS * G * 128 * sizeof(float);
constexpr size_t NA_PART_ML_BYTES = (size_t)NA_MAX_SLOTS * G * sizeof(float2);
constexpr size_t NA_COUNT_BYTES = (size_t)NA_MAX_PAIRS * sizeof(int32_t);
constexpr size_t NOALLOC_SCRATCH_BYTES = NA_PART_O_BYTES + NA_PART_ML_BYTES + NA_COUNT_BYTES;

static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

template <typename T, int D>
struct NaCfg {
  static constexpr int ESZ = sizeof(T);
  static constexpr int ROW_BYTES = D * ESZ;
  static_assert(ROW_BYTES == 256, "decode variant assumes 256-byte K/V rows");
  static constexpr int VEC = 16 / ESZ;
  static constexpr int PVD = D / 32;
  static constexpr int TILE = PS * ROW_BYTES;
  static constexpr int WARP_BYTES = NA_STAGES * 2 * TILE + (G * PS + PS * G + G) * 4 + 16;
  static constexpr int MERGE_BYTES = NA_WARPS * G * (D + 2) * 4;
  static_assert(MERGE_BYTES <= NA_WARPS * WARP_BYTES, "merge area must fit in the stages");
  static constexpr int SMEM = NA_WARPS * WARP_BYTES + NA_WARPS * NA_STAGES * 8 +
                              NA_MAX_CHUNKS * G * 4 + 64;
};

template <typename T>
__device__ inline void na_load_vec(const uint8_t* p, float* f);
template <>
__device__ inline void na_load_vec<__nv_bfloat16>(const uint8_t* p, float* f) {
  const uint4 w = *reinterpret_cast<const uint4*>(p);
  f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
  f[4] = bf16lo(w.z); f[5] = bf16hi(w.z); f[6] = bf16lo(w.w); f[7] = bf16hi(w.w);
}
template <>
__device__ inline void na_load_vec<float>(const uint8_t* p, float* f) {
  const float4 w = *reinterpret_cast<const float4*>(p);
  f[0] = w.x; f[1] = w.y; f[2] = w.z; f[3] = w.w;
}

template <typename T>
__device__ inline void na_load_pv(const uint8_t* p, float* f);
template <>
__device__ inline void na_load_pv<__nv_bfloat16>(const uint8_t* p, float* f) {
  const uint2 w = *reinterpret_cast<const uint2*>(p);
  f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
}
template <>
__device__ inline void na_load_pv<float>(const uint8_t* p, float* f) {
  const float2 w = *reinterpret_cast<const float2*>(p);
  f[0] = w.x; f[1] = w.y;
}

// Work item it -> (session i of the last append, chunk c of `cs`, kv head):
// every session is cut into `cs` chunks of its resident pages, so the number of
// partial slots is n_seq * cs * Hkv, which the host checks against NA_MAX_SLOTS.
template <typename T, int D>
__global__ void __launch_bounds__(NA_THREADS) attn_decode_noalloc_kernel(
    Dev d, int layer, const T* __restrict__ q, T* __restrict__ out, float qk_scale, int n_seq,
    int cs, float* __restrict__ part_o, float2* __restrict__ part_ml, int32_t* count) {
  using C = NaCfg<T, D>;
  extern __shared__ __align__(128) uint8_t smem[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint8_t* tiles = smem + warp * C::WARP_BYTES;
  float* s_sc = reinterpret_cast<float*>(tiles + NA_STAGES * 2 * C::TILE);
  float* s_p = s_sc + G * PS;
  float* s_alpha = s_p + PS * G;
  float* m_o = reinterpret_cast<float*>(smem);
  float* m_ml = m_o + NA_WARPS * G * D;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NA_WARPS * C::WARP_BYTES);
  uint64_t* wbars = bars + warp * NA_STAGES;
  float* s_scale = reinterpret_cast<float*>(bars + NA_WARPS * NA_STAGES);
  __shared__ int s_last, s_abort;
  if (lane == 0) {
    for (int s = 0; s < NA_STAGES; ++s) mbar_init(&wbars[s], 1);
    fence_mbar_init();
  }
  if (tid == 0) s_abort = 0;
  __syncthreads();

  const int H = d.kv_heads;
  const int n_items = n_seq * cs * H;
  const size_t head_stride = (size_t)PS * D;
  uint32_t loads = 0;
  const int half = lane >> 4, c = lane & 15;

  for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
    const int head = it % H;
    const int rest = it / H;
    const int seq = rest / cs, chunk = rest % cs;
    const SeqInfo si = d.seq[seq];
    const int32_t* hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    const int32_t* lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    const int blk_begin = (int)((int64_t)chunk * si.n_blocks / cs);
    const int blk_end = (int)((int64_t)(chunk + 1) * si.n_blocks / cs);

    float qr[G][C::VEC];
    {
      const T* qrow = q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G) * D;
      const float2* cs2 = d.rope + (size_t)si.pos_first * (D / 2);
#pragma unroll
      for (int g = 0; g < G; ++g) {
#pragma unroll
        for (int e = 0; e < C::VEC; ++e) {
          const int dd = c * C::VEC + e;
          const bool lo = dd < D / 2;
          const int j = lo ? dd : dd - D / 2;
          const float x = to_float<T>(qrow[g * D + dd]);
          const float y = to_float<T>(qrow[g * D + (lo ? dd + D / 2 : dd - D / 2)]);
          const float2 t = cs2[j];
          qr[g][e] = (lo ? fmaf(x, t.x, -y * t.y) : fmaf(x, t.x, y * t.y)) * qk_scale;
        }
      }
    }

    const int nblk = blk_end - blk_begin;
    const int n_my = (nblk > warp) ? (nblk - warp + NA_WARPS - 1) / NA_WARPS : 0;
    auto issue = [&](int k) {
      const BlockRef br = block_ref(si, hrow, lrow, blk_begin + warp + k * NA_WARPS);
      const uint32_t n = loads + k;
      const int st = n % NA_STAGES;
      uint8_t* dst = tiles + st * 2 * C::TILE;
      const T* kp = reinterpret_cast<const T*>(d.pool) +
                    pool_offset_elems(d, br.page, layer, 0, head, 0);
      mbar_arrive_expect_tx(&wbars[st], 2 * C::TILE);
      bulk_g2s(dst, kp, C::TILE, &wbars[st]);
      bulk_g2s(dst + C::TILE, kp + H * head_stride, C::TILE, &wbars[st]);
    };
    if (lane == 0) {
      fence_proxy_async_smem();
      for (int k = 0; k < min(NA_STAGES, n_my); ++k) issue(k);
    }

    float m_run = -INFINITY, l_run = 0.f;
    float acc[G][C::PVD];
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int j = 0; j < C::PVD; ++j) acc[g][j] = 0.f;

    int failed_at = -1;
    for (int k = 0; k < n_my; ++k) {
      const uint32_t n = loads + k;
      const int st = n % NA_STAGES;
      if (!__all_sync(FULL, mbar_wait(d, &wbars[st], (n / NA_STAGES) & 1))) {
        failed_at = k;
        break;
      }
      const uint8_t* kt = tiles + st * 2 * C::TILE;
      const uint8_t* vt = kt + C::TILE;
      const BlockRef br = block_ref(si, hrow, lrow, blk_begin + warp + k * NA_WARPS);
#pragma unroll
      for (int i = 0; i < PS / 2; ++i) {
        const int key = 2 * i + half;
        float kf[C::VEC];
        na_load_vec<T>(kt + key * C::ROW_BYTES + c * 16, kf);
        float a[G];
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float s = 0.f;
#pragma unroll
          for (int e = 0; e < C::VEC; ++e) s = fmaf(qr[g][e], kf[e], s);
          a[g] = s;
        }
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
          na_load_pv<T>(vt + key * C::ROW_BYTES + lane * C::PVD * C::ESZ, vf);
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
      if (lane == 0 && k + NA_STAGES < n_my) {
        fence_proxy_async_smem();
        issue(k + NA_STAGES);
      }
    }
    if (failed_at >= 0 && lane == 0) s_abort = 1;
    __syncthreads();
    if (s_abort) {
      if (failed_at >= 0) {
        for (int k = failed_at; k < min(n_my, failed_at + NA_STAGES); ++k) {
          const uint32_t n = loads + k;
          mbar_wait(d, &wbars[n % NA_STAGES], (n / NA_STAGES) & 1);
        }
      }
      return;
    }
    loads += n_my;

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
    const int slot = (seq * cs + chunk) * H + head;
    const bool single = cs == 1;
    for (int e = tid; e < G * D; e += NA_THREADS) {
      const int g = e / D, dd = e % D;
      float mw[NA_WARPS], M = -INFINITY;
#pragma unroll
      for (int w = 0; w < NA_WARPS; ++w) {
        mw[w] = m_ml[(w * G + g) * 2];
        M = fmaxf(M, mw[w]);
      }
      float L = 0.f, O = 0.f;
#pragma unroll
      for (int w = 0; w < NA_WARPS; ++w) {
        const float sc = exp2_safe(mw[w], M);
        L += m_ml[(w * G + g) * 2 + 1] * sc;
        O += m_o[(w * G + g) * D + dd] * sc;
      }
      if (single) {
        out[((size_t)si.q_row0 * d.q_heads + head * G + g) * D + dd] = from_float<T>(O / L);
      } else {
        part_o[((size_t)slot * G + g) * D + dd] = O;
        if (dd == 0) part_ml[(size_t)slot * G + g] = make_float2(M, L);
      }
    }
    if (!single) {
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int old = atomicAdd(&count[seq * H + head], 1);
        s_last = (old == cs - 1);
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        const int s0 = seq * cs * H + head;
        {
          const int g = warp;
          float M = -INFINITY;
          for (int ch = lane; ch < cs; ch += 32)
            M = fmaxf(M, __ldcg(&part_ml[(size_t)(s0 + ch * H) * G + g]).x);
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(FULL, M, o));
          float L = 0.f;
          for (int ch = lane; ch < cs; ch += 32) {
            const float2 ml = __ldcg(&part_ml[(size_t)(s0 + ch * H) * G + g]);
            const float sc = exp2_safe(ml.x, M);
            s_scale[ch * G + g] = sc;
            L += ml.y * sc;
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) L += __shfl_xor_sync(FULL, L, o);
          const float inv = 1.f / L;
          __syncwarp();
          for (int ch = lane; ch < cs; ch += 32) s_scale[ch * G + g] *= inv;
        }
        __syncthreads();
        for (int e = tid; e < G * D; e += NA_THREADS) {
          const int g = e / D, dd = e % D;
          float O = 0.f;
          for (int ch = 0; ch < cs; ++ch)
            O += __ldcg(&part_o[((size_t)(s0 + ch * H) * G + g) * D + dd]) * s_scale[ch * G + g];
          out[((size_t)si.q_row0 * d.q_heads + head * G + g) * D + dd] = from_float<T>(O);
        }
        if (tid == 0) count[seq * H + head] = 0;
      }
    }
    __syncthreads();
  }
}

// Per-CUDA-context set-up, done by the first call made in a context (with that
// context current): the array's device address in this context (each context
// loads its own copy of the module), the SM count, and, for each kernel instance,
// the shared-memory attribute and its resident CTAs per SM.  Contexts are told
// apart by their unique id (cuCtxGetId), which is never reused, so a context that
// replaces a destroyed one at the same address gets its own set-up.
struct NaSetup {
  unsigned long long ctx_id;
  uint8_t* scratch;
  int sms;
  int per_sm[2];  // [0] binary32 / D = 64, [1] bfloat16 / D = 128
};
constexpr int NA_MAX_CONTEXTS = 64;
NaSetup g_setup[NA_MAX_CONTEXTS];
int g_n_setup = 0;
std::mutex g_setup_mu;

typedef CUresult (*PfnCtxGetCurrent)(CUcontext*);
typedef CUresult (*PfnCtxGetId)(CUcontext, unsigned long long*);

cudaError_t driver_fn(const char* name, void** fn) {
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPoint(name, fn, cudaEnableDefault, &q);
  if (e != cudaSuccess) return e;
  return (q == cudaDriverEntryPointSuccess && *fn) ? cudaSuccess : cudaErrorNotSupported;
}

template <typename T, int D>
cudaError_t kernel_per_sm(int* per_sm) {
  const void* fn = reinterpret_cast<const void*>(&attn_decode_noalloc_kernel<T, D>);
  const int smem = NaCfg<T, D>::SMEM;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, fn, NA_THREADS, smem);
  if (e != cudaSuccess) return e;
  return *per_sm > 0 ? cudaSuccess : cudaErrorInvalidConfiguration;
}

cudaError_t setup_for_current_context(NaSetup* out) {
  static PfnCtxGetCurrent get_current = nullptr;
  static PfnCtxGetId get_id = nullptr;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  cudaError_t e;
  if (!get_current || !get_id) {
    void* f1 = nullptr;
    void* f2 = nullptr;
    if ((e = driver_fn("cuCtxGetCurrent", &f1)) != cudaSuccess) return e;
    if ((e = driver_fn("cuCtxGetId", &f2)) != cudaSuccess) return e;
    get_current = reinterpret_cast<PfnCtxGetCurrent>(f1);
    get_id = reinterpret_cast<PfnCtxGetId>(f2);
  }
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  void* p = nullptr;
  if (!ctx) {
    // No context current on this thread yet: the runtime makes the device's
    // primary context current on this lookup.
    if ((e = cudaGetSymbolAddress(&p, g_noalloc_scratch)) != cudaSuccess) return e;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return cudaErrorDeviceUninitialized;
  }
  unsigned long long id = 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  for (int i = 0; i < g_n_setup; ++i)
    if (g_setup[i].ctx_id == id) {
      *out = g_setup[i];
      return cudaSuccess;
    }
  NaSetup s = {};
  s.ctx_id = id;
  if ((e = cudaGetSymbolAddress(&p, g_noalloc_scratch)) != cudaSuccess) return e;
  s.scratch = static_cast<uint8_t*>(p);
  int dev = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&s.sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return e;
  if ((e = kernel_per_sm<float, 64>(&s.per_sm[0])) != cudaSuccess) return e;
  if ((e = kernel_per_sm<__nv_bfloat16, 128>(&s.per_sm[1])) != cudaSuccess) return e;
  // A full table only means later contexts repeat the set-up on every call.
  if (g_n_setup < NA_MAX_CONTEXTS) g_setup[g_n_setup++] = s;
  *out = s;
  return cudaSuccess;
}

// Chunks per session: about four work items per resident CTA over the call,
// limited by the static scratch and by NA_MAX_CHUNKS.
int noalloc_chunks(int pairs, int resident_ctas) {
  int cs = std::max(1, 4 * resident_ctas / std::max(1, pairs));
  cs = std::min(cs, NA_MAX_CHUNKS);
  cs = std::min(cs, NA_MAX_SLOTS / std::max(1, pairs));
  return std::max(1, cs);
}

template <typename T, int D>
cudaError_t launch_typed(const Dev& d, int layer, const void* q, void* out, int n_seq,
                         const NaSetup& su, cudaStream_t s) {
  const int per_sm = su.per_sm[sizeof(T) == 2 ? 1 : 0];
  const int grid = per_sm * su.sms;
  const int cs = noalloc_chunks(n_seq * d.kv_heads, grid);
  float* part_o = reinterpret_cast<float*>(su.scratch);
  float2* part_ml = reinterpret_cast<float2*>(su.scratch + NA_PART_O_BYTES);
  int32_t* count = reinterpret_cast<int32_t*>(su.scratch + NA_PART_O_BYTES + NA_PART_ML_BYTES);
  // The counters must start at zero; the array keeps whatever the last call left.
  cudaError_t e = cudaMemsetAsync(count, 0, (size_t)n_seq * d.kv_heads * sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  attn_decode_noalloc_kernel<T, D><<<grid, NA_THREADS, NaCfg<T, D>::SMEM, s>>>(
      d, layer, static_cast<const T*>(q), static_cast<T*>(out), scale, n_seq, cs, part_o,
      part_ml, count);
  return cudaGetLastError();
}

}  // namespace

int noalloc_max_pairs() { return NA_MAX_PAIRS; }

cudaError_t launch_attn_decode_noalloc(const Dev& d, int layer, const void* q, void* out,
                                       int n_seq, cudaStream_t s) {
  NaSetup su;
  cudaError_t e = setup_for_current_context(&su);
  if (e != cudaSuccess) return e;
  if (d.esz == 2) return launch_typed<__nv_bfloat16, 128>(d, layer, q, out, n_seq, su, s);
  return launch_typed<float, 64>(d, layer, q, out, n_seq, su, s);
}

}  // namespace kvc
