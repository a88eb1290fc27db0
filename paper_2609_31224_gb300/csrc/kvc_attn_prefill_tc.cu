// Chunked-prefill GQA attention on the 5th-generation tensor cores (tcgen05 +
// TMEM), bfloat16 K/V/q, fp32 softmax and accumulation.
//
// The call's (session, KV head, page) units are cut into equal contiguous
// ranges, one per CTA (stream-K); per segment (the part of one (session, KV
// head) pair in a range) the T*G query rows (T <= 32 tokens, G = 4 heads) form
// the M = 128 rows of an MMA tile, the rows past T*G being zero padding.  A
// pair split over several CTAs is merged by the last of them (log-sum-exp).
// Warp roles in one CTA:
//   warps 0, 6 producers: 2-D TMA loads (128-byte swizzle) of the K (warp 0)
//             and V (warp 6) tiles of 4 pages (64 keys) per stage into a
//             shared-memory ring whose K and V halves are released separately;
//   warps 1, 7 MMA issuers: one elected thread each issues tcgen05.mma, warp
//             1 S = Q K^T (N = 64, Q from TMEM, K from shared memory) into a
//             double-buffered TMEM tile, warp 7 O += P V (N = 128, P from
//             TMEM, V from shared memory) into TMEM; completion is signalled
//             with tcgen05.commit on mbarriers;
//   warps 2-5 softmax: each thread owns one TMEM lane (= one query row):
//             it builds its rotated, scaled query row in shared memory,
//             reads its row of S from TMEM, masks (resident slots, causal
//             inside the chunk), keeps the running max/sum, writes P as
//             bfloat16 to a swizzled shared buffer, rescales O in TMEM when
//             the row maximum grows by more than 2^8, and finally reads O.
// All waits are bounded; a timeout records KVC_DERR_WAIT and the CTA stops.
#include <cuda.h>

#include "kvc_launch.cuh"
#include "kvc_rope.cuh"

namespace kvc {

namespace {

constexpr int G = 4;
constexpr int D = 128;
constexpr int M = 128;                       // MMA rows (query rows, padded)
constexpr int NK = 64;                       // keys per stage (4 pages)
constexpr int TC_STAGES = 6;                 // K/V stages of the ring (a 7-stage ring measured slower)
constexpr int KV_PANEL = NK * 128;           // 64 rows x 128 B = 8 KiB
constexpr int STAGE = 4 * KV_PANEL;          // K lo, K hi, V lo, V hi = 32 KiB
// Tensor memory (512 columns x 128 lanes of 32 bits; lane = query row):
//   S0 [0,64) S1 [64,128)  fp32 scores of two stages
//   O  [128,256)           fp32 output accumulator
//   P0 [256,288) P1 [288,320)  bfloat16 probabilities (2 per column), MMA A operand
//   Q  [320,384)           bfloat16 rotated, scaled query rows, MMA A operand
constexpr int TMEM_COLS = 512;
constexpr int S_COL = 0, O_COL = 128, P_COL = 256, Q_COL = 320;
constexpr float LOG2E = 1.4426950408889634f;
constexpr float RESCALE_LOG2 = 8.f;          // rescale O only when the max grows by > 2^8
constexpr int THREADS = 8 * 32;
constexpr int PF_MIN_UNITS = 16;              // pages per CTA of the stream-K split, at least
constexpr int PF_MAX_PARTS = 1 << 16;        // no limit on CTAs per pair (merged row by row)
constexpr unsigned FULL = 0xFFFFFFFFu;

// Shared memory map (offsets from a 1024-aligned base): the K/V ring, barriers.
constexpr int OFF_KV = 0;
constexpr int OFF_BAR = OFF_KV + TC_STAGES * STAGE;
enum {
  B_K_FULL = 0,                          // [TC_STAGES] K half of a stage loaded
  B_K_EMPTY = B_K_FULL + TC_STAGES,      // [TC_STAGES] ... and read by S = Q K^T
  B_V_FULL = B_K_EMPTY + TC_STAGES,      // [TC_STAGES] V half loaded
  B_V_EMPTY = B_V_FULL + TC_STAGES,      // [TC_STAGES] ... and read by O += P V
  B_S_FULL = B_V_EMPTY + TC_STAGES,      // [2]
  B_S_EMPTY = B_S_FULL + 2,              // [2]
  B_P_FULL = B_S_EMPTY + 2,              // [2]
  B_P_EMPTY = B_P_FULL + 2,              // [2]
  // [2] P V product j complete: barrier j % 2, phase j / 2.  One barrier per P
  // buffer keeps every waiter at most one phase behind (P V products j - 3 and
  // earlier are known complete when j is waited for), so parity waits are exact.
  B_O = B_P_EMPTY + 2,
  B_Q = B_O + 2,                         // one phase per segment (query tile ready)
  B_FINAL = B_Q + 1,                     // every MMA of the CTA complete (both issuers)
  // Fused layer write: one phase per segment holding chunk slots, completed when the
  // softmax warps have written those rows into the pool.
  B_ROWS = B_FINAL + 1,
  N_BARS = B_ROWS + 1
};
constexpr int OFF_TMEM_ADDR = OFF_BAR + N_BARS * 8;
constexpr int TC_SMEM = OFF_TMEM_ADDR + 16 + 1024;  // + alignment slack
static_assert(TC_SMEM <= 227 * 1024, "shared memory per CTA");

// -- tcgen05 helpers ------------------------------------------------------------------
__device__ inline void tmem_alloc(uint32_t* smem_dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(smem_dst)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ inline void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ inline void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ inline void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ inline void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
// D (TMEM) (+)= A B with A read from tensor memory (M lanes, K/2 columns of
// bfloat16 pairs) and B from shared memory.
__device__ inline void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                 uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Each thread of the warp reads 32 consecutive fp32 columns of its TMEM lane.
__device__ inline void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ inline void tmem_st32(uint32_t taddr, const uint32_t* w) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
          taddr),
      "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7]),
      "r"(w[8]), "r"(w[9]), "r"(w[10]), "r"(w[11]), "r"(w[12]), "r"(w[13]), "r"(w[14]),
      "r"(w[15]), "r"(w[16]), "r"(w[17]), "r"(w[18]), "r"(w[19]), "r"(w[20]), "r"(w[21]),
      "r"(w[22]), "r"(w[23]), "r"(w[24]), "r"(w[25]), "r"(w[26]), "r"(w[27]), "r"(w[28]),
      "r"(w[29]), "r"(w[30]), "r"(w[31])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ inline void tmem_st32(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
          taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor, 128-byte swizzle: `sbo` bytes between 8-row
// groups; `lbo` bytes between 64-element groups of the contiguous dimension
// (MN-major operands only).
__device__ inline uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFF);
  d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version of this architecture
  d |= (uint64_t)2 << 61;  // 128-byte swizzle
  return d;
}

// The per-layer write of the chunk rows of tokens [t0, t1) of a session (its call
// row q_row0, positions from pos_first) for KV head `head`, by the 128 softmax
// threads (thread index ts): V rows copied, K rows rotated at their positions, in
// 16-byte chunks, every load of an item issued before its stores.  Each thread then
// orders its writes before later tensor copies (async proxy).
__device__ inline void write_chunk_rows(const Dev& d, int layer, const SeqInfo& si, int head,
                                        const __nv_bfloat16* new_k, const __nv_bfloat16* new_v,
                                        int t0, int t1, int ts) {
  // Item (token, c): 16-byte chunk c of the first half of the K row with its
  // rotate-half partner, and chunks c and c + 8 of the V row.
  constexpr int VEC = 8, HALF = D / 2, KC = HALF / VEC;
  __nv_bfloat16* pool = reinterpret_cast<__nv_bfloat16*>(d.pool);
  const int H = d.kv_heads;
  const int n = (t1 - t0) * KC;
  for (int idx = ts; idx < n; idx += 128) {
    const int t = t0 + idx / KC, c = idx % KC;
    const size_t in_row = ((size_t)(si.q_row0 + t) * H + head) * D + c * VEC;
    const uint4 ka = *reinterpret_cast<const uint4*>(new_k + in_row);
    const uint4 kb = *reinterpret_cast<const uint4*>(new_k + in_row + HALF);
    const uint4 va = *reinterpret_cast<const uint4*>(new_v + in_row);
    const uint4 vb = *reinterpret_cast<const uint4*>(new_v + in_row + HALF);
    const float2* t2 = d.rope + (size_t)(si.pos_first + t) * HALF + c * VEC;
    float2 cs[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e) cs[e] = t2[e];
    const int gs = d.tok_slot[si.q_row0 + t];
    float xa[VEC], xb[VEC], ya[VEC], yb[VEC];
    Chunk16<__nv_bfloat16>::unpack(ka, xa);
    Chunk16<__nv_bfloat16>::unpack(kb, xb);
#pragma unroll
    for (int e = 0; e < VEC; ++e) rope_pair(xa[e], xb[e], cs[e], ya[e], yb[e]);
    __nv_bfloat16* kd = pool + pool_offset_elems(d, gs / PS, layer, 0, head, gs % PS) + c * VEC;
    __nv_bfloat16* vd = pool + pool_offset_elems(d, gs / PS, layer, 1, head, gs % PS) + c * VEC;
    *reinterpret_cast<uint4*>(kd) = Chunk16<__nv_bfloat16>::pack(ya);
    *reinterpret_cast<uint4*>(kd + HALF) = Chunk16<__nv_bfloat16>::pack(yb);
    *reinterpret_cast<uint4*>(vd) = va;
    *reinterpret_cast<uint4*>(vd + HALF) = vb;
  }
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Chunk tokens [t0, t1) of a session whose slots lie in its blocks [b_lo, b_hi).
__device__ inline void chunk_tokens_in(const SeqInfo& si, int b_lo, int b_hi, int& t0, int& t1) {
  const int sl_first = si.live_head + si.n_live - si.t;  // live slot of the first token
  const int lo = (b_lo - si.n_hist_pages) * PS, hi = (b_hi - si.n_hist_pages) * PS;
  t0 = max(0, lo - sl_first);
  t1 = min(si.t, hi - sl_first);
}

// Instruction descriptor, kind::f16: D fp32, A and B bf16, A K-major, B K- or MN-major.
__host__ __device__ constexpr uint32_t instr_desc(int n, int m, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
         ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ inline uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ inline float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The segment after `s` in a range ending at u_end, given s.end < u_end: s then ends
// at its pair's end, and the next segment is the next pair from its first unit, the
// session's next KV head or the next session's first one.  Unlike unit_segment, no
// search over the sessions (a chain of dependent loads) is needed.
__device__ inline UnitSeg next_segment(const Dev& d, const UnitSeg& s, int u_end) {
  UnitSeg n;
  if (s.head + 1 < d.kv_heads) {
    n.seq = s.seq;
    n.si = s.si;
    n.head = s.head + 1;
  } else {
    n.seq = s.seq + 1;
    n.si = d.seq[n.seq];
    n.head = 0;
  }
  const int nb = n.si.n_blocks;
  n.pair_start = n.si.unit_base + n.head * nb;
  n.pair_end = n.pair_start + nb;
  n.u = s.end;
  n.end = min(u_end, n.pair_end);
  return n;
}

// FUSED (the per-layer order): the chunk's K (rotated at each token's position) and
// V of this layer are not in the pool yet; new_k / new_v hold them ([total][Hkv][D],
// the append's token order).  The producer warp that loads a stage holding chunk
// slots of its (session, head) first writes those rows into the pool (the CTA
// owning a (session, head, page) unit is the only reader of that unit in the
// launch), then orders the writes before its tensor copy of the stage.
template <bool FUSED>
__global__ void __launch_bounds__(THREADS, 1) attn_prefill_tc_kernel(
    Dev d, int layer, const __grid_constant__ CUtensorMap map_lo,
    const __grid_constant__ CUtensorMap map_hi, const __nv_bfloat16* __restrict__ q,
    __nv_bfloat16* __restrict__ out, float qk_scale, const __nv_bfloat16* __restrict__ new_k,
    const __nv_bfloat16* __restrict__ new_v) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_TMEM_ADDR);
  __shared__ int s_abort_flag, s_last;
  volatile int& s_abort = s_abort_flag;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  if (tid == 0) {
    for (int s = 0; s < TC_STAGES; ++s) {
      mbar_init(&bars[B_K_FULL + s], 1);
      mbar_init(&bars[B_K_EMPTY + s], 1);
      mbar_init(&bars[B_V_FULL + s], 1);
      mbar_init(&bars[B_V_EMPTY + s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars[B_S_FULL + s], 1);
      mbar_init(&bars[B_S_EMPTY + s], 4);
      mbar_init(&bars[B_P_FULL + s], 4);
      mbar_init(&bars[B_P_EMPTY + s], 1);
    }
    mbar_init(&bars[B_O + 0], 1);
    mbar_init(&bars[B_O + 1], 1);
    mbar_init(&bars[B_Q], 4);
    mbar_init(&bars[B_FINAL], 2);
    mbar_init(&bars[B_ROWS], 4);
    fence_mbar_init();
    s_abort = 0;
  }
  // Zero the K/V ring once: the keys of partly filled stages only ever hold finite
  // values (their weights are 0, and 0 times a stale NaN would not be 0).
  for (int i = tid; i < OFF_BAR / 16; i += THREADS)
    reinterpret_cast<uint4*>(smem)[i] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Before pdl_wait() only the append's data is read (work list, page tables, K/V
  // pages); the softmax warps wait before reading q or writing any result.
  pdl_launch_dependents();

  const int H = d.kv_heads, L = d.layers;
  // Stream-K: this CTA's contiguous range of the call's units (UnitSplit); the three
  // roles walk the same segments of it.
  const UnitSplit us = unit_split(d, gridDim.x, PF_MIN_UNITS, PF_MAX_PARTS);
  const int cta = blockIdx.x;
  const bool active = cta < us.n_cta;
  const int u_begin = active ? us.start_of(cta) : 0, u_end = active ? us.start_of(cta + 1) : 0;
  const uint32_t sKV = smem_u32(smem + OFF_KV);

  if (warp == 0 || warp == 6) {
    // ---------------- producers ----------------
    // Warp 0 loads the K halves of the stages, warp 6 the V halves, each with its
    // own full/empty barriers: a K half is free again once S = Q K^T of its stage
    // is complete, a V half once O += P V is, so the K loads run ahead of the V
    // loads by up to the ring depth.  The whole warp walks the segments; lane j
    // fetches the page id of block (window + j) so that one round trip serves 32
    // blocks, and lane 0 issues the TMA loads with the ids shuffled to it.
    const bool is_v = warp == 6;
    const int b_full = is_v ? B_V_FULL : B_K_FULL, b_empty = is_v ? B_V_EMPTY : B_K_EMPTY;
    uint32_t n = 0;  // stages produced
    bool stop = false;
    uint32_t rows_seen = 0;  // segments holding chunk slots, before this one
    (void)rows_seen;
    UnitSeg seg;
    for (int u = u_begin; u < u_end && !stop;) {
      seg = u == u_begin ? unit_segment(d, u, u_end) : next_segment(d, seg, u_end);
      u = seg.end;
      const int head = seg.head;
      const SeqInfo& si = seg.si;
      const int32_t* hrow = d.hist_pt + (size_t)si.sid * d.max_pages_per_session;
      const int32_t* lrow = d.live_pt + (size_t)si.sid * d.max_pages_per_session;
      const int blk0 = seg.blk_begin(), nblk = seg.end - seg.u;
      const int n_st = (nblk + 3) / 4;
      int pid = 0;
      if (is_v) {
        // The segment's query rows (T tokens x G heads, 1 KiB per token) and rotary
        // rows (512 B per token) into L2 ahead of the softmax warps, which read them
        // when the segment starts.  A prefetch changes nothing that a later load
        // observes, so it may run before the previous kernel has finished.
        const char* qb = reinterpret_cast<const char*>(
            q + ((size_t)si.q_row0 * d.q_heads + (size_t)head * G) * D);
        const char* rb = reinterpret_cast<const char*>(d.rope + (size_t)si.pos_first * (D / 2));
        const size_t qstride = (size_t)d.q_heads * D * sizeof(__nv_bfloat16);
        for (int x = lane; x < si.t * 12; x += 32) {
          const int tt = x / 12, line = x % 12;
          prefetch_l2(line < 8 ? qb + tt * qstride + line * 128 : rb + (size_t)tt * 512 + (line - 8) * 128);
        }
      }
      for (int k = 0; k < n_st; ++k, ++n) {
        const int b0 = 4 * k;
        if ((b0 & 31) == 0) {
          const int bj = b0 + lane;
          pid = bj < nblk ? block_page(si, hrow, lrow, blk0 + bj) : 0;
        }
        const int st = n % TC_STAGES;
        int ok = 1;
        if (lane == 0) ok = mbar_wait(d, &bars[b_empty + st], ((n / TC_STAGES) & 1) ^ 1);
        ok = __shfl_sync(FULL, ok, 0);
        if (!ok) {
          if (lane == 0) s_abort = 1;
          stop = true;
          break;
        }
        const int npg = min(4, nblk - b0);
        int pages[4];
#pragma unroll
        for (int pg = 0; pg < 4; ++pg) pages[pg] = __shfl_sync(FULL, pid, (b0 & 31) + pg);
        if constexpr (FUSED) {
          // A stage holding chunk slots is copied only once the softmax warps have
          // written the segment's rows (they do so when the segment starts).
          int t0, t1;
          chunk_tokens_in(si, blk0 + b0, blk0 + b0 + npg, t0, t1);
          if (t0 < t1) {
            int ok = 1;
            if (lane == 0) ok = mbar_wait(d, &bars[B_ROWS], rows_seen & 1);
            if (!__shfl_sync(FULL, ok, 0)) {
              if (lane == 0) s_abort = 1;
              stop = true;
              break;
            }
          }
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&bars[b_full + st], npg * 2 * 2048);
          uint8_t* base = smem + OFF_KV + st * STAGE + (is_v ? 2 * KV_PANEL : 0);
          for (int pg = 0; pg < npg; ++pg) {
            // Pool rows of this page's K (kv = 0) or V (kv = 1) tile of `head`.
            const int row = (((pages[pg] * L + layer) * 2 + (is_v ? 1 : 0)) * H + head) * PS;
            tma_load_2d(base + pg * 2048, &map_lo, 0, row, &bars[b_full + st]);
            tma_load_2d(base + KV_PANEL + pg * 2048, &map_hi, 0, row, &bars[b_full + st]);
          }
        }
      }
      if constexpr (FUSED) {
        int t0, t1;
        chunk_tokens_in(si, blk0, blk0 + nblk, t0, t1);
        if (t0 < t1) ++rows_seen;
      }
      stop = stop || __any_sync(FULL, s_abort != 0);
    }
  } else if (warp == 1 || warp == 7) {
    // ---------------- MMA issuers ----------------
    // One elected thread each: warp 1 issues S = Q K^T of every stage, warp 7
    // O += P V.  Their products use different accumulators, and each thread's
    // tcgen05.commit tracks only its own MMAs, so the two streams interleave in
    // the tensor pipe and neither waits behind the other's issue cost.
    if (lane == 0) {
      uint32_t n = 0;  // K/V stages of the earlier segments
      if (warp == 1) {
        constexpr uint32_t ID_S = instr_desc(NK, M, false);
        uint32_t sc = 0;     // S tiles issued
        uint32_t segs = 0;   // segments started
        UnitSeg seg;
        for (int u = u_begin; u < u_end && !s_abort; ++segs) {
          seg = u == u_begin ? unit_segment(d, u, u_end) : next_segment(d, seg, u_end);
          u = seg.end;
          const int n_st = (seg.end - seg.u + 3) / 4;
          if (!mbar_wait(d, &bars[B_Q], segs & 1)) {
            s_abort = 1;
            break;
          }
          tc_fence_after();
          for (int k = 0; k < n_st && !s_abort; ++k) {
            const int st = (n + k) % TC_STAGES;
            const int sb = sc % 2;
            if (!mbar_wait(d, &bars[B_K_FULL + st], ((n + k) / TC_STAGES) & 1) ||
                !mbar_wait(d, &bars[B_S_EMPTY + sb], ((sc / 2) & 1) ^ 1)) {
              s_abort = 1;
              break;
            }
            tc_fence_after();
            const uint32_t kbase = sKV + st * STAGE;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              // 16 dims per step: 8 TMEM columns of Q; 32 bytes of a swizzled K row.
              const uint32_t kb = kbase + (kk >> 2) * KV_PANEL + (kk & 3) * 32;
              tc_mma_ts(tmem + S_COL + sb * NK, tmem + Q_COL + kk * 8, smem_desc(kb, 0, 1024),
                        ID_S, kk > 0 ? 1u : 0u);
            }
            tc_commit(&bars[B_S_FULL + sb]);
            tc_commit(&bars[B_K_EMPTY + st]);
            ++sc;
          }
          n += n_st;
        }
      } else {
        constexpr uint32_t ID_PV = instr_desc(D, M, true);
        uint32_t pv = 0;  // P V products issued
        UnitSeg seg;
        for (int u = u_begin; u < u_end && !s_abort;) {
          seg = u == u_begin ? unit_segment(d, u, u_end) : next_segment(d, seg, u_end);
          u = seg.end;
          const int n_st = (seg.end - seg.u + 3) / 4;
          for (int k = 0; k < n_st && !s_abort; ++k) {
            const int st = (n + k) % TC_STAGES;
            const int pb = pv % 2;
            if (!mbar_wait(d, &bars[B_V_FULL + st], ((n + k) / TC_STAGES) & 1) ||
                !mbar_wait(d, &bars[B_P_FULL + pb], (pv / 2) & 1)) {
              s_abort = 1;
              break;
            }
            tc_fence_after();
            const uint32_t vbase = sKV + st * STAGE + 2 * KV_PANEL;
#pragma unroll
            for (int kk = 0; kk < NK / 16; ++kk) {
              // 16 keys per step: 8 TMEM columns of P; 16 rows of the V panels.  The
              // first product of a segment overwrites O (its previous contents were
              // read by the epilogue before this segment's first P was written).
              const uint32_t vb = vbase + kk * 16 * 128;
              tc_mma_ts(tmem + O_COL, tmem + P_COL + pb * (NK / 2) + kk * 8,
                        smem_desc(vb, KV_PANEL, 1024), ID_PV, (k > 0 || kk > 0) ? 1u : 0u);
            }
            tc_commit(&bars[B_V_EMPTY + st]);
            tc_commit(&bars[B_P_EMPTY + pb]);
            tc_commit(&bars[B_O + pb]);
            ++pv;
          }
          n += n_st;
        }
      }
      // No MMA may still be running when the tensor memory is released.
      tc_commit(&bars[B_FINAL]);
      mbar_wait(d, &bars[B_FINAL], 0);
    }
  } else {
    // ---------------- softmax / epilogue ----------------
    // A failed (timed-out) wait makes the warp "dead": it then skips waits and
    // work but still walks the same items, arrivals and named barriers, so the
    // other softmax warps never wait for it.
    const int quarter = warp & 3;              // TMEM lanes 32*quarter .. +31
    const int r = quarter * 32 + lane;         // this thread's query row
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    uint32_t sc = 0, pv = 0;
    bool dead = false;
    pdl_wait();
    auto wait = [&](uint64_t* bar, uint32_t parity) {
      if (dead) return;
      dead = !__all_sync(FULL, mbar_wait(d, bar, parity));
      if (dead && lane == 0) s_abort = 1;
    };
    UnitSeg seg;
    for (int u = u_begin; u < u_end;) {
      seg = u == u_begin ? unit_segment(d, u, u_end) : next_segment(d, seg, u_end);
      const int first = seg.u == u_begin;
      u = seg.end;
      const int head = seg.head;
      const SeqInfo& si = seg.si;
      const int blk0 = seg.blk_begin(), nblk = seg.end - seg.u;
      const int n_st = (nblk + 3) / 4;
      const int R = si.t * G;
      const bool live = r < R;
      const int t = r / G, g = r % G;
      const int qlog = si.n_hist + si.n_live - si.t + t;
      // The previous segment's products are complete (its epilogue waited for the
      // last one), so the query tile in tensor memory can be overwritten.  Every
      // lane writes its row: the query (bfloat16 pairs, dims 0..127 in columns
      // 0..63), or zeros for padding rows.
      if (!dead) {
        uint32_t qw[D / 2];
        if (live) {
          // Chunk c (dims 8c..8c+7) of the first half pairs with chunk c of the second.
          const uint4* qrow = reinterpret_cast<const uint4*>(
              q + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * D);
          const float4* cs =
              reinterpret_cast<const float4*>(d.rope + (size_t)(si.pos_first + t) * (D / 2));
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 wa = qrow[c], wb = qrow[c + 8];
            const uint32_t ua[4] = {wa.x, wa.y, wa.z, wa.w}, ub[4] = {wb.x, wb.y, wb.z, wb.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const float4 t4 = cs[c * 4 + h];  // (cos, sin) of dims 8c + 2h, 8c + 2h + 1
              const float a0 = bf16lo(ua[h]), a1 = bf16hi(ua[h]);
              const float b0 = bf16lo(ub[h]), b1 = bf16hi(ub[h]);
              qw[4 * c + h] = pack_bf16(fmaf(a0, t4.x, -b0 * t4.y) * qk_scale,
                                        fmaf(a1, t4.z, -b1 * t4.w) * qk_scale);
              qw[D / 4 + 4 * c + h] = pack_bf16(fmaf(b0, t4.x, a0 * t4.y) * qk_scale,
                                                fmaf(b1, t4.z, a1 * t4.w) * qk_scale);
            }
          }
        } else {
#pragma unroll
          for (int j = 0; j < D / 2; ++j) qw[j] = 0u;
        }
        tmem_st32(trow + Q_COL, qw);
        tmem_st32(trow + Q_COL + 32, qw + 32);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars[B_Q]);
      if constexpr (FUSED) {
        int t0, t1;
        chunk_tokens_in(si, blk0, blk0 + nblk, t0, t1);
        if (t0 < t1) {
          if (!dead) write_chunk_rows(d, layer, si, head, new_k, new_v, t0, t1, r);
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars[B_ROWS]);
        }
      }

      // Blocks that may need a mask: the partly filled last history page, the
      // first live page when it starts mid-page, and every block from the one
      // holding the chunk's first query on (causal).  A stage of four pages that
      // avoids them all is interior.
      const int nhp = si.n_hist_pages;
      const int b_hist_part = (si.n_hist % PS) ? nhp - 1 : -PS;
      const int b_live_part = si.live_head ? nhp : -PS;
      const int sl_first = si.live_head + si.n_live - si.t;  // live slot of the first query
      const int b_causal = nhp + sl_first / PS + ((sl_first % PS) == PS - 1 ? 1 : 0);
      float m_used = -INFINITY, l = 0.f;
      for (int k = 0; k < n_st; ++k) {
        const int sb = sc % 2, pb = pv % 2;
        wait(&bars[B_S_FULL + sb], (sc / 2) & 1);
        tc_fence_after();
        float s[NK];
        tmem_ld32(trow + S_COL + sb * NK, s);
        tmem_ld32(trow + S_COL + sb * NK + 32, s + 32);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[B_S_EMPTY + sb]);
        ++sc;
        // Mask the keys that are not resident slots or lie after the row's query.
        // Interior stages (four full pages, every key before the chunk's first
        // query) need no mask.  Padding rows (r >= T*G) are left unmasked: their
        // products stay finite and their outputs are never written.
        const int npg = min(4, nblk - 4 * k);
        const int b0 = blk0 + 4 * k;
        const bool interior = npg == 4 && b0 + 3 < b_causal &&
                              (unsigned)(b_hist_part - b0) > 3u && (unsigned)(b_live_part - b0) > 3u;
        if (!interior) {
          BlockRange brs[4];
#pragma unroll
          for (int pg = 0; pg < 4; ++pg) brs[pg] = block_range(si, b0 + min(pg, npg - 1));
#pragma unroll
          for (int pg = 0; pg < 4; ++pg) {
#pragma unroll
            for (int j = 0; j < PS; ++j) {
              const bool v = pg < npg && j >= brs[pg].lo && j < brs[pg].hi &&
                             brs[pg].base + j <= qlog;
              float& x = s[pg * PS + j];
              x = (v || !live) ? x : -INFINITY;
            }
          }
        }
        // Row maximum over 8 independent chains.
        float m8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) m8[i] = s[i];
#pragma unroll
        for (int j = 8; j < NK; ++j) m8[j % 8] = fmaxf(m8[j % 8], s[j]);
        float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                         fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
        if (dead || !live) mx = -INFINITY;
        // Rescale O (in TMEM) and l only when the row maximum grows by > 2^8; this
        // waits for the previous P V product.  Every lane of the warp takes part
        // in the TMEM accesses; lanes that need no rescale use factor 1.
        const bool need = mx > m_used + RESCALE_LOG2;
        const bool have_o = pv > 0 && m_used != -INFINITY;
        if (__any_sync(FULL, need && have_o)) {
          wait(&bars[B_O + (pv - 1) % 2], ((pv - 1) / 2) & 1);
          tc_fence_after();
          const float f = (need && have_o) ? exp2f(m_used - mx) : 1.f;
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(trow + O_COL + c * 32, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= f;
            tmem_st32(trow + O_COL + c * 32, o);
          }
          tc_fence_before();
        }
        if (need) {
          if (have_o) l *= exp2f(m_used - mx);
          m_used = mx;
        }
        // P = exp2(s - m_used) as bfloat16 pairs into TMEM buffer pb (row r, 32 columns).
        wait(&bars[B_P_EMPTY + pb], ((pv / 2) & 1) ^ 1);
        // Masked keys are -inf and give 0; a row with no finite key yet uses 0 as
        // its reference so that no -inf - -inf appears; padding rows get weight 0.
        const float mref = !live ? INFINITY : (m_used == -INFINITY ? 0.f : m_used);
        float rs[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        uint32_t pw[NK / 2];
#pragma unroll
        for (int j = 0; j < NK; j += 2) {
          const float p0 = ex2(s[j] - mref), p1 = ex2(s[j + 1] - mref);
          rs[j % 8] += p0;
          rs[j % 8 + 1] += p1;
          pw[j / 2] = pack_bf16(p0, p1);
        }
        l += ((rs[0] + rs[1]) + (rs[2] + rs[3])) + ((rs[4] + rs[5]) + (rs[6] + rs[7]));
        if (!dead) tmem_st32(trow + P_COL + pb * (NK / 2), pw);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars[B_P_FULL + pb]);
        ++pv;
      }
      // Epilogue: wait for the last P V, read O.
      wait(&bars[B_O + (pv - 1) % 2], ((pv - 1) / 2) & 1);
      tc_fence_after();
      const bool single = seg.whole();
      const int slot = 2 * cta + (first ? 0 : 1);
      const size_t prow0 = (size_t)slot * (PF_MAX_TOKENS * G) + r;
      const bool write = live && !dead;
      const float inv = 1.f / l;
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        float o[32];
        tmem_ld32(trow + O_COL + c * 32, o);
        if (write && single) {
          __nv_bfloat16* orow =
              out + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * D + c * 32;
#pragma unroll
          for (int i = 0; i < 32; i += 8)
            *reinterpret_cast<uint4*>(orow + i) =
                make_uint4(pack_bf16(o[i] * inv, o[i + 1] * inv),
                           pack_bf16(o[i + 2] * inv, o[i + 3] * inv),
                           pack_bf16(o[i + 4] * inv, o[i + 5] * inv),
                           pack_bf16(o[i + 6] * inv, o[i + 7] * inv));
        } else if (write) {
          float* prow = d.pf_part_o + prow0 * D + c * 32;
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(prow + i) = make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
        }
      }
      tc_fence_before();
      if (!single) {
        // Split-K: publish this part's (O, max, sum); the last CTA to arrive for the
        // (session, head) merges every part, one thread per query row.  All four
        // softmax warps reach both named barriers on every such segment.
        if (write) d.pf_part_ml[prow0] = make_float2(m_used, l);
        const int cf = us.owner(seg.pair_start), nch = us.owner(seg.pair_end - 1) - cf + 1;
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (warp == 2 && lane == 0)
          s_last = arrive_acq_rel(&d.pf_count[seg.seq * H + head], nch);
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (s_last) {
          // The merge runs in tensor memory: this CTA's own part is still in the O
          // columns (the next segment's first P V overwrites them only after this),
          // and each other part's row is loaded whole, all its words at once, and
          // added there.  The first other part's row is loaded together with every
          // part's (max, sum), so a pair of two parts costs one round trip.  Every
          // lane takes part in the tensor-memory accesses; rows that are padding (or
          // of a warp whose wait gave up) weigh 0 and write nothing.
          const int first_slot = us.slot_of(cf, cf, seg.pair_start);
          const int own = cta - cf;
          auto prow = [&](int ch) {
            return (size_t)(ch ? 2 * (cf + ch) : first_slot) * (PF_MAX_TOKENS * G) + r;
          };
          auto load_row = [&](int ch, float4 (&v)[D / 4]) {
            const float4* src = reinterpret_cast<const float4*>(d.pf_part_o + prow(ch) * D);
#pragma unroll
            for (int i = 0; i < D / 4; ++i)
              v[i] = write ? __ldcg(src + i) : make_float4(0.f, 0.f, 0.f, 0.f);
          };
          const int f0 = own == 0 ? 1 : 0;  // first other part
          float4 v[D / 4];
          load_row(f0, v);
          constexpr int MB = 8;
          float2 ml[MB];
          auto load_ml = [&](int c0) {
#pragma unroll
            for (int i = 0; i < MB; ++i)
              ml[i] = (write && c0 + i < nch && c0 + i != own) ? __ldcg(&d.pf_part_ml[prow(c0 + i)])
                                                               : make_float2(-INFINITY, 0.f);
          };
          float Mx = write ? m_used : -INFINITY;
          load_ml(0);
#pragma unroll
          for (int i = 0; i < MB; ++i) Mx = fmaxf(Mx, ml[i].x);
          const float ml_f0_x = f0 < MB ? (f0 == 0 ? ml[0].x : ml[1].x) : -INFINITY;
          float Ls = 0.f;
#pragma unroll
          for (int i = 0; i < MB; ++i) Ls += ml[i].y * exp2_safe(ml[i].x, Mx);
          for (int c0 = MB; c0 < nch; c0 += MB) {
            load_ml(c0);
#pragma unroll
            for (int i = 0; i < MB; ++i) Mx = fmaxf(Mx, ml[i].x);
          }
          if (nch > MB) {  // the sum again, against the final maximum
            Ls = 0.f;
            for (int c0 = 0; c0 < nch; c0 += MB) {
              load_ml(c0);
#pragma unroll
              for (int i = 0; i < MB; ++i) Ls += ml[i].y * exp2_safe(ml[i].x, Mx);
            }
          }
          if (write) Ls += l * exp2_safe(m_used, Mx);
          const float invL = write ? 1.f / Ls : 0.f;
          const float s_own = write ? exp2_safe(m_used, Mx) : 0.f;
          // Own part scaled, plus the first other part.
          float s_f = write ? exp2_safe(ml_f0_x, Mx) : 0.f;
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(trow + O_COL + c * 32, o);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float4 w4 = v[c * 8 + i];
              o[4 * i] = o[4 * i] * s_own + w4.x * s_f;
              o[4 * i + 1] = o[4 * i + 1] * s_own + w4.y * s_f;
              o[4 * i + 2] = o[4 * i + 2] * s_own + w4.z * s_f;
              o[4 * i + 3] = o[4 * i + 3] * s_own + w4.w * s_f;
            }
            tmem_st32(trow + O_COL + c * 32, o);
          }
          // The remaining parts (pairs over three or more CTAs), one row at a time.
          for (int ch = f0 + 1; ch < nch; ++ch) {
            if (ch == own) continue;
            load_row(ch, v);
            s_f = write ? exp2_safe(__ldcg(&d.pf_part_ml[prow(ch)]).x, Mx) : 0.f;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
              float o[32];
              tmem_ld32(trow + O_COL + c * 32, o);
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const float4 w4 = v[c * 8 + i];
                o[4 * i] += w4.x * s_f;
                o[4 * i + 1] += w4.y * s_f;
                o[4 * i + 2] += w4.z * s_f;
                o[4 * i + 3] += w4.w * s_f;
              }
              tmem_st32(trow + O_COL + c * 32, o);
            }
          }
          __nv_bfloat16* orow = out + ((size_t)(si.q_row0 + t) * d.q_heads + head * G + g) * D;
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(trow + O_COL + c * 32, o);
            if (write) {
#pragma unroll
              for (int i = 0; i < 32; i += 8)
                *reinterpret_cast<uint4*>(orow + c * 32 + i) = make_uint4(
                    pack_bf16(o[i] * invL, o[i + 1] * invL), pack_bf16(o[i + 2] * invL, o[i + 3] * invL),
                    pack_bf16(o[i + 4] * invL, o[i + 5] * invL),
                    pack_bf16(o[i + 6] * invL, o[i + 7] * invL));
            }
          }
          tc_fence_before();
          if (warp == 2 && lane == 0) d.pf_count[seg.seq * H + head] = 0;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, TMEM_COLS);
}

}  // namespace

const void* prefill_tc_kernel_ptr() {
  return reinterpret_cast<const void*>(&attn_prefill_tc_kernel<false>);
}
int prefill_tc_smem() { return TC_SMEM; }
int prefill_tc_threads() { return THREADS; }

cudaError_t launch_attn_prefill_tc(const Dev& d, int layer, const CUtensorMap& lo,
                                   const CUtensorMap& hi, const void* q, void* out, int grid,
                                   bool pdl, cudaStream_t s, const void* new_k, const void* new_v) {
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  if (new_k != nullptr) {
    static thread_local const cudaError_t attr = cudaFuncSetAttribute(
        reinterpret_cast<const void*>(&attn_prefill_tc_kernel<true>),
        cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM);
    if (attr != cudaSuccess) return attr;
  }
  return launch_ex(new_k != nullptr ? &attn_prefill_tc_kernel<true> : &attn_prefill_tc_kernel<false>,
                   dim3(grid), dim3(THREADS), TC_SMEM, s, pdl, d, layer, lo, hi,
                   static_cast<const __nv_bfloat16*>(q), static_cast<__nv_bfloat16*>(out), scale,
                   static_cast<const __nv_bfloat16*>(new_k), static_cast<const __nv_bfloat16*>(new_v));
}

}  // namespace kvc
