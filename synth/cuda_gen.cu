// Device-side generator for the synthetic Q/K/V inputs (the same definition as
// synth/values.py, bit for bit): SplitMix64 (Steele, Lea & Flood, OOPSLA 2014)
// counter hash per element, Irwin-Hall(4) over its four 16-bit fields, scaled
// in binary32, optionally rounded to bfloat16.  Input generation only.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cstring>

namespace {

constexpr uint64_t GAMMA = 0x9E3779B97F4A7C15ull;

__host__ __device__ inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// dst[l][t][h][d] = value(seed, tag, session[t], l, pos[t], h, d)
template <typename T>
__global__ void fill_kernel(T* dst, uint64_t base, float ih_scale, float scale, int apply_scale,
                            int layers, int n_tok, int heads, int head_dim,
                            const int32_t* __restrict__ tok_session,
                            const int32_t* __restrict__ tok_pos) {
  const int64_t n = (int64_t)layers * n_tok * heads * head_dim;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int d = (int)(i % head_dim);
    int64_t r = i / head_dim;
    const int h = (int)(r % heads);
    r /= heads;
    const int t = (int)(r % n_tok);
    const int l = (int)(r / n_tok);
    const uint64_t idx = ((uint64_t)tok_session[t] << 42) | ((uint64_t)l << 36) |
                         ((uint64_t)tok_pos[t] << 14) | ((uint64_t)h << 8) | (uint64_t)d;
    const uint64_t hsh = mix64(base + (idx + 1) * GAMMA);
    const int s = (int)(hsh & 0xFFFF) + (int)((hsh >> 16) & 0xFFFF) + (int)((hsh >> 32) & 0xFFFF) +
                  (int)((hsh >> 48) & 0xFFFF);
    float x = __fmul_rn((float)(s - 131070), ih_scale);
    if (apply_scale) x = __fmul_rn(x, scale);
    if constexpr (sizeof(T) == 2)
      dst[i] = __float2bfloat16_rn(x);
    else
      dst[i] = x;
  }
}

}  // namespace

extern "C" {

// Fill a [layers][n_tok][heads][head_dim] tensor (bfloat16 if dtype == 1,
// binary32 if dtype == 0).  tok_session / tok_pos are device arrays [n_tok].
// ih_scale_bits: binary32 bits of sqrt(3)/65536.  Returns a cudaError_t value.
int synth_fill(void* dst, int dtype, uint64_t seed, int tag, uint32_t ih_scale_bits, float scale,
               int layers, int n_tok, int heads, int head_dim, const int32_t* tok_session,
               const int32_t* tok_pos, void* stream) {
  const uint64_t base = mix64((((seed << 2) | (uint64_t)tag)) + GAMMA);
  float ih;
  memcpy(&ih, &ih_scale_bits, 4);
  const int apply = scale != 1.0f;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t n = (int64_t)layers * n_tok * heads * head_dim;
  if (n == 0) return 0;
  int blocks = (int)((n + 255) / 256);
  if (blocks > 152 * 64) blocks = 152 * 64;
  if (dtype == 1)
    fill_kernel<__nv_bfloat16><<<blocks, 256, 0, s>>>(static_cast<__nv_bfloat16*>(dst), base, ih,
                                                      scale, apply, layers, n_tok, heads,
                                                      head_dim, tok_session, tok_pos);
  else
    fill_kernel<float><<<blocks, 256, 0, s>>>(static_cast<float*>(dst), base, ih, scale, apply,
                                              layers, n_tok, heads, head_dim, tok_session,
                                              tok_pos);
  return (int)cudaGetLastError();
}

}  // extern "C"
