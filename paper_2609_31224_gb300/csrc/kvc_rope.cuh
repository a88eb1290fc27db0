// Rotate-half RoPE of one pair of a key row, shared by every kernel that writes
// keys into the pool, so that the stored bytes do not depend on the path.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace kvc {

// (x1, x2) = (k[j], k[j + D/2]); c = (cos, sin) of the position's angle for dim j
// (the binary32 table); binary32 arithmetic.
__device__ inline void rope_pair(float x1, float x2, float2 c, float& y1, float& y2) {
  y1 = fmaf(x1, c.x, -x2 * c.y);
  y2 = fmaf(x2, c.x, x1 * c.y);
}

// The elements of a 16-byte chunk as binary32, and back (round to nearest even for
// bfloat16), without taking the chunk's address (which would put it in local memory).
template <typename T>
struct Chunk16;
template <>
struct Chunk16<__nv_bfloat16> {
  static constexpr int N = 8;
  __device__ static void unpack(const uint4& w, float (&f)[8]) {
    const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(u[i] << 16);
      f[2 * i + 1] = __uint_as_float(u[i] & 0xFFFF0000u);
    }
  }
  __device__ static uint4 pack(const float (&f)[8]) {
    uint32_t u[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 v = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
      u[i] = *reinterpret_cast<const uint32_t*>(&v);
    }
    return make_uint4(u[0], u[1], u[2], u[3]);
  }
};
template <>
struct Chunk16<float> {
  static constexpr int N = 4;
  __device__ static void unpack(const uint4& w, float (&f)[4]) {
    f[0] = __uint_as_float(w.x);
    f[1] = __uint_as_float(w.y);
    f[2] = __uint_as_float(w.z);
    f[3] = __uint_as_float(w.w);
  }
  __device__ static uint4 pack(const float (&f)[4]) {
    return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                      __float_as_uint(f[3]));
  }
};

}  // namespace kvc
