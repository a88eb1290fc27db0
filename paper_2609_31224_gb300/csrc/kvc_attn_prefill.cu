// Chunked-prefill GQA attention over the retained cache.
//
// For each session of the last append (T <= 32 tokens, e.g. the 17 acoustic
// positions of a one-second unit), each KV head and its G = 4 query heads, the
// T*G query rows attend to every resident key at or before their own position
// (causal inside the chunk).  Split-K work items as in decode.
//
// bfloat16: one CTA = one producer warp + MT consumer warps (16 query rows
// each).  The producer streams K/V pages through a ring of shared-memory
// stages with 2-D TMA (128-byte swizzle, one 2 KiB panel per half head-dim);
// consumers compute S = Q K^T and O += P V with bf16 tensor-core MMAs
// (fp32 accumulate) and keep the online softmax per row in registers.
// binary32: CUDA-core kernel, one thread per query row.
#include <cuda.h>

#include "kvc_internal.cuh"

namespace kvc {

namespace {

constexpr unsigned FULL = 0xFFFFFFFFu;
constexpr int G = 4;
constexpr float LOG2E = 1.4426950408889634f;

// ---------------------------------------------------------------------------
// bfloat16 tensor-core prefill.
// ---------------------------------------------------------------------------
constexpr int PF_D = 128;
constexpr int PF_STAGES = 4;
constexpr int PANEL = PS * 128;           // 16 rows x 128 bytes
constexpr int PAGE_TILE = 4 * PANEL;      // K lo, K hi, V lo, V hi
constexpr int STAGE_BYTES = 2 * PAGE_TILE;  // two pages = 32 keys

__device__ inline void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                   uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ inline void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                               uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ inline void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                 uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ inline void mma_bf16(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, "
      "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ inline uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Address of the 16-byte chunk `chunk` (0..15 over the 128 dims) of row `key`
// (0..15) of a K or V page tile (SW128: chunk index XOR row % 8 inside a panel).
__device__ inline uint32_t tile_addr(uint32_t tile, int key, int chunk) {
  const int panel = chunk >> 3, c = chunk & 7;
  return tile + panel * PANEL + key * 128 + ((c ^ (key & 7)) << 4);
}

template <int MT>
__global__ void __launch_bounds__((MT + 1) * 32) attn_prefill_bf16_kernel(
    Dev d, int layer, const __grid_constant__ CUtensorMap map_lo,
    const __grid_constant__ CUtensorMap map_hi, const __nv_bfloat16* __restrict__ q,
    __nv_bfloat16* __restrict__ out, float qk_scale) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + PF_STAGES * STAGE_BYTES);
  uint64_t* empty = full + PF_STAGES;
  __shared__ int s_last, s_abort;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool producer = warp == MT;
  if (tid == 0) {
    for (int s = 0; s < PF_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], MT);
    }
    fence_mbar_init();
    s_abort = 0;
  }
  __syncthreads();

  const int n_items = d.g->n_pf_items * d.kv_heads;
  const int H = d.kv_heads, L = d.layers;
  uint32_t used = 0;  // stages used so far (same count on both sides)

  for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
    const int item = it / H, head = it % H;
    const Item itm = d.pf_items[item];
    const SeqInfo si = d.seq[itm.seq];
    const int32_t* hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
    const int32_t* lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
    const int nblk = itm.blk_end - itm.blk_begin;
    const int n_st = (nblk + 1) / 2;

    if (producer) {
      if (lane == 0) {
        for (int k = 0; k < n_st; ++k) {
          const uint32_t n = used + k;
          const int st = n % PF_STAGES;
          if (!mbar_wait(d, &empty[st], ((n / PF_STAGES) & 1) ^ 1)) {
            s_abort = 1;
            break;
          }
          const int npg = min(2, nblk - 2 * k);
          mbar_arrive_expect_tx(&full[st], npg * PAGE_TILE);
          for (int pg = 0; pg < npg; ++pg) {
            const BlockRef br = block_ref(si, hrow, lrow, itm.blk_begin + 2 * k + pg);
            uint8_t* dst = smem + st * STAGE_BYTES + pg * PAGE_TILE;
            const int rk = (((br.page * L + layer) * 2 + 0) * H + head) * PS;
            const int rv = rk + H * PS;
            tma_load_2d(dst, &map_lo, 0, rk, &full[st]);
            tma_load_2d(dst + PANEL, &map_hi, 0, rk, &full[st]);
            tma_load_2d(dst + 2 * PANEL, &map_lo, 0, rv, &full[st]);
            tma_load_2d(dst + 3 * PANEL, &map_hi, 0, rv, &full[st]);
          }
        }
      }
      __syncwarp();
    } else {
      // Consumer warp `warp` owns query rows [16*warp, 16*warp + 16).
      const int R = si.t * G;
      const int n_res = si.n_hist + si.n_live;
      const int r_a = warp * 16 + (lane >> 2), r_b = r_a + 8;
      const int qlog_a = n_res - si.t + r_a / G, qlog_b = n_res - si.t + r_b / G;
      const bool rows_live = warp * 16 < R;
      // Q fragments (A operand, 16 x 128), rotated at each row's position.
      uint32_t qa[8][4];
      {
        const float2* cs = d.rope;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
          for (int h2 = 0; h2 < 2; ++h2) {      // row a / row b
#pragma unroll
            for (int k8 = 0; k8 < 2; ++k8) {    // dims +0 / +8
              const int r = h2 ? r_b : r_a;
              const int dd = ks * 16 + k8 * 8 + 2 * (lane & 3);
              float v0 = 0.f, v1 = 0.f;
              if (r < R) {
                const int t = r / G, g = r % G;
                const __nv_bfloat16* qrow =
                    q + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * PF_D;
                const float2* c = cs + (size_t)(si.pos_first + t) * (PF_D / 2);
                float vv[2];
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                  const int x = dd + e;
                  const bool lo = x < PF_D / 2;
                  const int j = lo ? x : x - PF_D / 2;
                  const float a = __bfloat162float(qrow[x]);
                  const float b = __bfloat162float(qrow[lo ? x + PF_D / 2 : x - PF_D / 2]);
                  const float2 t2 = c[j];
                  vv[e] = (lo ? fmaf(a, t2.x, -b * t2.y) : fmaf(a, t2.x, b * t2.y)) * qk_scale;
                }
                v0 = vv[0];
                v1 = vv[1];
              }
              qa[ks][h2 + 2 * k8] = pack_bf16(v0, v1);
            }
          }
        }
      }
      float o[16][4];
#pragma unroll
      for (int j = 0; j < 16; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
      float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;

      for (int k = 0; k < n_st; ++k) {
        const uint32_t n = used + k;
        const int st = n % PF_STAGES;
        if (!__all_sync(FULL, mbar_wait(d, &full[st], (n / PF_STAGES) & 1))) {
          if (lane == 0) s_abort = 1;
          break;
        }
        const int npg = min(2, nblk - 2 * k);
        if (rows_live) {
          const uint32_t stage = smem_u32(smem + st * STAGE_BYTES);
          float s[4][4];
#pragma unroll
          for (int j = 0; j < 4; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
          // S = Q K^T over the stage's 32 keys (n-tiles j: keys 8j..8j+7).
#pragma unroll
          for (int pg = 0; pg < 2; ++pg) {
            if (pg < npg) {
              const uint32_t kt = stage + pg * PAGE_TILE;
#pragma unroll
              for (int ks = 0; ks < 8; ++ks) {
                // x4: (keys 0-7, chunk 2ks), (keys 0-7, 2ks+1), (keys 8-15, 2ks), (keys 8-15, 2ks+1)
                const int mi = lane >> 3, rr = lane & 7;
                const int key = (mi >> 1) * 8 + rr, chunk = 2 * ks + (mi & 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4(tile_addr(kt, key, chunk), b0, b1, b2, b3);
                mma_bf16(s[2 * pg], qa[ks], b0, b1);
                mma_bf16(s[2 * pg + 1], qa[ks], b2, b3);
              }
            }
          }
          // Mask, online softmax (rows a and b of this thread).
          float mx_a = -INFINITY, mx_b = -INFINITY;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int pg = j >> 1;
            const BlockRef br =
                block_ref(si, hrow, lrow, itm.blk_begin + 2 * k + min(pg, npg - 1));
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int slot = (j & 1) * 8 + 2 * (lane & 3) + e;
              const bool v = pg < npg && slot >= br.lo && slot < br.hi;
              const int lg = br.base + slot;
              if (!(v && lg <= qlog_a && r_a < R)) s[j][e] = -INFINITY;
              if (!(v && lg <= qlog_b && r_b < R)) s[j][2 + e] = -INFINITY;
              mx_a = fmaxf(mx_a, s[j][e]);
              mx_b = fmaxf(mx_b, s[j][2 + e]);
            }
          }
          mx_a = fmaxf(mx_a, __shfl_xor_sync(FULL, mx_a, 1));
          mx_a = fmaxf(mx_a, __shfl_xor_sync(FULL, mx_a, 2));
          mx_b = fmaxf(mx_b, __shfl_xor_sync(FULL, mx_b, 1));
          mx_b = fmaxf(mx_b, __shfl_xor_sync(FULL, mx_b, 2));
          const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
          const float al_a = exp2_safe(m_a, mn_a), al_b = exp2_safe(m_b, mn_b);
          float rs_a = 0.f, rs_b = 0.f;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            s[j][0] = exp2_safe(s[j][0], mn_a);
            s[j][1] = exp2_safe(s[j][1], mn_a);
            s[j][2] = exp2_safe(s[j][2], mn_b);
            s[j][3] = exp2_safe(s[j][3], mn_b);
            rs_a += s[j][0] + s[j][1];
            rs_b += s[j][2] + s[j][3];
          }
          rs_a += __shfl_xor_sync(FULL, rs_a, 1);
          rs_a += __shfl_xor_sync(FULL, rs_a, 2);
          rs_b += __shfl_xor_sync(FULL, rs_b, 1);
          rs_b += __shfl_xor_sync(FULL, rs_b, 2);
          l_a = l_a * al_a + rs_a;
          l_b = l_b * al_b + rs_b;
          m_a = mn_a;
          m_b = mn_b;
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            o[j][0] *= al_a;
            o[j][1] *= al_a;
            o[j][2] *= al_b;
            o[j][3] *= al_b;
          }
          // O += P V (k-steps: keys 0-15 of page 0, keys 0-15 of page 1).
#pragma unroll
          for (int pg = 0; pg < 2; ++pg) {
            if (pg < npg) {
              uint32_t pa[4];
              pa[0] = pack_bf16(s[2 * pg][0], s[2 * pg][1]);
              pa[1] = pack_bf16(s[2 * pg][2], s[2 * pg][3]);
              pa[2] = pack_bf16(s[2 * pg + 1][0], s[2 * pg + 1][1]);
              pa[3] = pack_bf16(s[2 * pg + 1][2], s[2 * pg + 1][3]);
              const uint32_t vt = stage + pg * PAGE_TILE + 2 * PANEL;
#pragma unroll
              for (int nj = 0; nj < 8; ++nj) {
                // x4.trans: (keys 0-7, chunk nj*2), (keys 8-15, nj*2), (keys 0-7, nj*2+1), (keys 8-15, nj*2+1)
                const int mi = lane >> 3, rr = lane & 7;
                const int key = (mi & 1) * 8 + rr, chunk = 2 * nj + (mi >> 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(tile_addr(vt, key, chunk), b0, b1, b2, b3);
                mma_bf16(o[2 * nj], pa, b0, b1);
                mma_bf16(o[2 * nj + 1], pa, b2, b3);
              }
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[st]);
      }
      // Per-row results: rows a (o[..][0..1]) and b (o[..][2..3]).
      if (rows_live) {
        const bool single = si.pf_chunks == 1;
        const int slot = (si.pf_base + itm.chunk) * H + head;
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int r = h2 ? r_b : r_a;
          if (r >= R) continue;
          const float m = h2 ? m_b : m_a, l = h2 ? l_b : l_a;
          const int t = r / G, g = r % G;
          if (single) {
            __nv_bfloat16* orow = out + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * PF_D;
            const float inv = 1.f / l;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int dd = j * 8 + 2 * (lane & 3);
              *reinterpret_cast<uint32_t*>(orow + dd) =
                  pack_bf16(o[j][2 * h2] * inv, o[j][2 * h2 + 1] * inv);
            }
          } else {
            float* prow = d.pf_part_o + ((size_t)slot * (PF_MAX_TOKENS * G) + r) * PF_D;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int dd = j * 8 + 2 * (lane & 3);
              *reinterpret_cast<float2*>(prow + dd) = make_float2(o[j][2 * h2], o[j][2 * h2 + 1]);
            }
            if ((lane & 3) == 0)
              d.pf_part_ml[(size_t)slot * (PF_MAX_TOKENS * G) + r] = make_float2(m, l);
          }
        }
      }
    }
    used += n_st;
    __syncthreads();
    if (s_abort) return;
    if (si.pf_chunks > 1) {
      __threadfence();
      __syncthreads();
      if (tid == 0) {
        const int old = atomicAdd(&d.pf_count[itm.seq * H + head], 1);
        s_last = (old == si.pf_chunks - 1);
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        const int R = si.t * G;
        const int s0 = si.pf_base * H + head;
        for (int e = tid; e < R * PF_D; e += blockDim.x) {
          const int r = e / PF_D, dd = e % PF_D;
          float M = -INFINITY;
          for (int ch = 0; ch < si.pf_chunks; ++ch)
            M = fmaxf(M, __ldcg(&d.pf_part_ml[(size_t)(s0 + ch * H) * (PF_MAX_TOKENS * G) + r]).x);
          float Lsum = 0.f, O = 0.f;
          for (int ch = 0; ch < si.pf_chunks; ++ch) {
            const size_t sl = (size_t)(s0 + ch * H) * (PF_MAX_TOKENS * G) + r;
            const float2 ml = __ldcg(&d.pf_part_ml[sl]);
            const float sc = exp2_safe(ml.x, M);
            Lsum += ml.y * sc;
            O += __ldcg(&d.pf_part_o[sl * PF_D + dd]) * sc;
          }
          const int t = r / G, g = r % G;
          out[((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * PF_D + dd] =
              __float2bfloat16_rn(O / Lsum);
        }
        if (tid == 0) d.pf_count[itm.seq * H + head] = 0;
      }
      __syncthreads();
    }
  }
}

constexpr int PF_SMEM = PF_STAGES * STAGE_BYTES + 2 * PF_STAGES * 8 + 1024;

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
  CUtensorMap lo, hi;
  bool ok = false;
};

bool make_pool_maps(const Dev& d, PoolMaps& m) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  const uint64_t rows = (uint64_t)d.n_pages * d.layers * 2 * d.kv_heads * PS;
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
  return m.ok;
}

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
    return pf_grid<5>(reinterpret_cast<const void*>(&attn_prefill_bf16_kernel<5>), 6 * 32,
                      PF_SMEM);
  return pf_grid<0>(reinterpret_cast<const void*>(&attn_prefill_f32_kernel), F32_THREADS, 0);
}

cudaError_t launch_attn_prefill(const Dev& d, int layer, const void* q, void* out, int n_seq,
                                int max_t, cudaStream_t s) {
  (void)n_seq;
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  if (d.esz == 2) {
    static thread_local PoolMaps maps;
    static thread_local int g5 = 0, g8 = 0;
    if (!maps.ok || maps.pool != d.pool) {
      if (!make_pool_maps(d, maps)) return cudaErrorInvalidValue;
    }
    if (max_t * G <= 5 * 16) {
      if (!g5)
        g5 = pf_grid<5>(reinterpret_cast<const void*>(&attn_prefill_bf16_kernel<5>), 6 * 32,
                        PF_SMEM);
      attn_prefill_bf16_kernel<5><<<g5, 6 * 32, PF_SMEM, s>>>(
          d, layer, maps.lo, maps.hi, static_cast<const __nv_bfloat16*>(q),
          static_cast<__nv_bfloat16*>(out), scale);
    } else {
      if (!g8)
        g8 = pf_grid<8>(reinterpret_cast<const void*>(&attn_prefill_bf16_kernel<8>), 9 * 32,
                        PF_SMEM);
      attn_prefill_bf16_kernel<8><<<g8, 9 * 32, PF_SMEM, s>>>(
          d, layer, maps.lo, maps.hi, static_cast<const __nv_bfloat16*>(q),
          static_cast<__nv_bfloat16*>(out), scale);
    }
  } else {
    static thread_local int gf = 0;
    if (!gf)
      gf = pf_grid<0>(reinterpret_cast<const void*>(&attn_prefill_f32_kernel), F32_THREADS, 0);
    attn_prefill_f32_kernel<<<gf, F32_THREADS, 0, s>>>(d, layer, static_cast<const float*>(q),
                                                       static_cast<float*>(out), scale);
  }
  return cudaGetLastError();
}

}  // namespace kvc
