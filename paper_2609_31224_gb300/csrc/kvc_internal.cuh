// Internal definitions of the kvc library: device state, metadata layout and
// the PTX helpers (mbarrier, bulk copy) the kernels share.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kvc.h"

namespace kvc {

constexpr int PS = 16;          // positions per page
constexpr int MAX_SEQ = 512;    // sessions per call
constexpr int TYPE_MASK = 0x7F;
constexpr long long WAIT_LIMIT_CYCLES = 4000000000LL;  // ~2 s at 2 GHz

// Per-session device state.  The retained sequence is the hist region
// (n_hist positions, densely packed from slot 0 of hist page 0) followed by
// the live region (n_live positions from slot live_head of live page 0).
struct SessState {
  int32_t pos_next;
  int32_t unit_cur;
  int32_t n_hist;
  int32_t n_hist_pages;
  int32_t live_head;
  int32_t n_live;
  int32_t n_live_pages;
  int32_t last_chunk;
  int32_t n_evicted;
  int32_t peak_resident;
  int32_t pad[6];
};
static_assert(sizeof(SessState) == 64, "SessState size");

// Snapshot of one session of the last append, read by the attention kernels.
struct SeqInfo {
  int32_t sid;
  int32_t t;            // tokens in the chunk
  int32_t q_row0;       // first query row of this session in q/out
  int32_t pos_first;    // position of the chunk's first token
  int32_t n_hist;
  int32_t n_hist_pages;
  int32_t live_head;
  int32_t n_live;
  int32_t n_blocks;     // n_hist_pages + n_live_pages
  int32_t pad0;
  int32_t unit_base;    // first (session, kv head, page) unit of this session
  int32_t pf_chunks;
  int32_t pf_base;
  int32_t pad[3];
};
static_assert(sizeof(SeqInfo) == 64, "SeqInfo size");

// One split-K work item: blocks [blk_begin, blk_end) of one session.
struct Item {
  int32_t seq;
  int32_t chunk;
  int32_t blk_begin;
  int32_t blk_end;
};

struct DevGlobals {
  int32_t err;
  int32_t n_seq;
  int64_t pages_used;
  int32_t n_units;
  int32_t n_pf_items;
  int32_t n_moves;
  int32_t total_tokens;
  int32_t nb_max;   // largest n_blocks among the last append's sessions
  int32_t pad[7];
};

// Device pointers into the caller's workspace plus the shape, passed by value.
struct Dev {
  // shape
  int32_t n_sessions, layers, q_heads, kv_heads, head_dim, group;
  int32_t esz;                 // bytes per element
  int32_t max_pages_per_session, max_positions, max_seq, max_tokens;
  int64_t budget;
  int32_t window;
  int32_t policy, sink, recent;  // KVC_POLICY_*
  int64_t n_pages;
  int32_t bitmap_words;
  int32_t max_moves;
  int32_t dec_slots;           // decode partial slots (two per CTA of a split)
  int32_t max_pf_items;        // prefill chunk items (binary32) / partial slots (bfloat16)
  // memory
  uint8_t* pool;
  SessState* sess;
  int32_t* hist_pt;            // [n_sessions][max_pages_per_session]
  int32_t* live_pt;            // [n_sessions][max_pages_per_session]
  int32_t* meta_pos;           // [n_pages * PS]
  int32_t* meta_unit;          // [n_pages * PS]
  uint8_t* meta_type;          // [n_pages * PS]
  uint32_t* bitmap;            // 1 = page in use
  DevGlobals* g;
  float2* rope;                // [max_positions][D/2] (cos, sin)
  SeqInfo* seq;                // [max_seq]
  Item* pf_items;              // [max_pf_items]
  int32_t* tok_slot;           // [max_tokens] page * PS + slot
  int32_t* tok_pos;            // [max_tokens]
  int2* moves;                 // [max_moves] (src page*PS+slot, dst page*PS+slot)
  int32_t* alloc_list;         // [max_alloc] pages handed out by the last allocation
  int32_t max_alloc;
  float* dec_part_o;           // [dec_slots][G][D]
  float2* dec_part_ml;         // [dec_slots][G] (m, l) in log2 units
  unsigned long long* dec_tagged;  // [dec_tag_slots][G * D + 2 G] tagged partial states
  int32_t dec_tag_slots;
  float* pf_part_o;            // [max_pf_items][PF_ROWS][D]
  float2* pf_part_ml;          // [max_pf_items][PF_ROWS]
  int32_t* dec_count;          // [max_seq * kv_heads] arrival counters
  int32_t* pf_count;           // [max_seq * kv_heads]
};

constexpr int PF_MAX_TOKENS = 32;  // tokens per session per prefill call
constexpr int MAX_CHUNKS_PER_SEQ = 64;  // split-K chunks per session and call

__host__ __device__ inline size_t pool_offset_elems(const Dev& d, int page, int layer, int kv,
                                                    int head, int slot) {
  return ((((size_t)page * d.layers + layer) * 2 + kv) * d.kv_heads + head) * (size_t)PS *
             d.head_dim + (size_t)slot * d.head_dim;
}

// Page and valid slot range [lo, hi) of virtual block b of a session; the
// logical (retained-order) index of slot s is base + s.
struct BlockRef {
  int page, lo, hi, base;
};

__device__ inline BlockRef block_ref(const SeqInfo& si, const int32_t* hist_row,
                                     const int32_t* live_row, int b) {
  BlockRef r;
  if (b < si.n_hist_pages) {
    r.page = hist_row[b];
    r.lo = 0;
    r.hi = min(PS, si.n_hist - b * PS);
    r.base = b * PS;
  } else {
    int lb = b - si.n_hist_pages;
    int s0 = lb * PS;
    r.page = live_row[lb];
    r.lo = max(0, si.live_head - s0);
    r.hi = min(PS, si.live_head + si.n_live - s0);
    r.base = si.n_hist + s0 - si.live_head;
  }
  return r;
}

// ---------------------------------------------------------------------------
// Stream-K split of an attention call's (session, KV head, page) units.  Units
// are ordered session-major, then head, then page; seq[i].unit_base is session
// i's first.  The U units are cut into n_cta equal contiguous ranges, one per
// CTA.  A range covers "segments", the parts of (session, head) pairs inside it;
// only its first and last segments can be partial, and their partial states go
// to slots 2c and 2c + 1.  The CTAs owner(pair_start) .. owner(pair_end - 1)
// share a pair, and the last of them to finish merges it.
// ---------------------------------------------------------------------------
struct UnitSplit {
  int U, n_cta;
  __device__ int start_of(int c) const { return (int)((int64_t)c * U / n_cta); }
  __device__ int owner(int64_t u) const { return (int)(((u + 1) * n_cta - 1) / U); }
  // Slot of CTA cc's part of a pair whose first CTA is cf: cc's first segment,
  // except in cf when the pair begins after the start of cf's range.
  __device__ int slot_of(int cc, int cf, int pair_start) const {
    return cc != cf ? 2 * cc : (start_of(cf) != pair_start ? 2 * cf + 1 : 2 * cf);
  }
};

// At most `grid` CTAs, at least `min_units` units each, and few enough that no
// pair spans more than `max_parts` CTAs.
__device__ inline UnitSplit unit_split(const Dev& d, int grid, int min_units, int max_parts) {
  UnitSplit s;
  s.U = d.g->n_units;
  const int nb_max = max(1, d.g->nb_max);
  const int c_parts = (int)((int64_t)s.U * (max_parts - 2) / (nb_max + max_parts - 2));
  s.n_cta = max(1, min(grid, min((s.U + min_units - 1) / min_units, c_parts)));
  return s;
}

struct UnitSeg {
  int seq, head;             // session of the call, KV head
  int pair_start, pair_end;  // the pair's units
  int u, end;                // this segment's units [u, end)
  SeqInfo si;
  __device__ int blk_begin() const { return u - pair_start; }
  __device__ int blk_end() const { return end - pair_start; }
  __device__ bool whole() const { return u == pair_start && end == pair_end; }
};

// The segment that starts at unit u of a range ending at u_end.
__device__ inline UnitSeg unit_segment(const Dev& d, int u, int u_end) {
  int lo = 0, hi = d.g->n_seq - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (d.seq[mid].unit_base <= u) lo = mid;
    else hi = mid - 1;
  }
  UnitSeg s;
  s.seq = lo;
  s.si = d.seq[lo];
  const int nb = s.si.n_blocks;
  s.head = (u - s.si.unit_base) / nb;
  s.pair_start = s.si.unit_base + s.head * nb;
  s.pair_end = s.pair_start + nb;
  s.u = u;
  s.end = min(u_end, s.pair_end);
  return s;
}

// Arrive at a pair's counter once this CTA's partial state is written; true in
// the last of `parts` arrivals.  The caller synchronises the participating
// threads before (so that their partial writes precede the arrival) and after
// (so that, in the last CTA, the loads of the other parts follow it); one
// thread's acquire-release atomic then publishes and acquires at GPU scope.
__device__ inline bool arrive_acq_rel(int* counter, int parts) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(counter) : "memory");
  return old == parts - 1;
}

// Valid slot range [lo, hi) and logical base of virtual block b, without
// touching memory (the page id is looked up separately, see block_page).
struct BlockRange {
  int lo, hi, base;
};

__device__ inline BlockRange block_range(const SeqInfo& si, int b) {
  BlockRange r;
  if (b < si.n_hist_pages) {
    r.lo = 0;
    r.hi = min(PS, si.n_hist - b * PS);
    r.base = b * PS;
  } else {
    const int s0 = (b - si.n_hist_pages) * PS;
    r.lo = max(0, si.live_head - s0);
    r.hi = min(PS, si.live_head + si.n_live - s0);
    r.base = si.n_hist + s0 - si.live_head;
  }
  return r;
}

__device__ inline int block_page(const SeqInfo& si, const int32_t* hist_row,
                                 const int32_t* live_row, int b) {
  return b < si.n_hist_pages ? hist_row[b] : live_row[b - si.n_hist_pages];
}

__device__ inline void set_error(const Dev& d, int bits) { atomicOr(&d.g->err, bits); }

// Tagged partial states.  A CTA writes each value of its partial state as one
// 64-bit word, (tag << 32) | binary32 bits, and arrives with a relaxed atomic: no
// release fence waits for its stores.  The last CTA to arrive reads each word
// with a single-copy-atomic 64-bit load and re-reads (bounded) any word whose tag
// is not yet the launch's: the stores it waits for were issued before their CTAs'
// arrivals, so the wait needs no other CTA to make progress.
__device__ inline void st_tagged(unsigned long long* p, uint32_t tag, float v) {
  const unsigned long long w = ((unsigned long long)tag << 32) | __float_as_uint(v);
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}
__device__ inline unsigned long long ld_tagged(const unsigned long long* p) {
  unsigned long long w;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(w) : "l"(p) : "memory");
  return w;
}
__device__ inline bool arrive_relaxed(int* counter, int parts) {
  int old;
  asm volatile("atom.relaxed.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(counter) : "memory");
  return old == parts - 1;
}

// ---------------------------------------------------------------------------
// PTX helpers: mbarrier and bulk (TMA) copies global -> shared.
// ---------------------------------------------------------------------------
__device__ inline uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ inline void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

__device__ inline void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ inline void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ inline void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ inline void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ inline bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: returns false (and records KVC_DERR_WAIT) if the phase does
// not complete within WAIT_LIMIT_CYCLES.
__device__ inline bool mbar_wait(const Dev& d, uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > WAIT_LIMIT_CYCLES) {
      set_error(d, KVC_DERR_WAIT);
      return false;
    }
  }
  return true;
}

// 1-D bulk copy (TMA engine): `bytes` (multiple of 16) from 16-byte aligned
// global memory into 16-byte aligned shared memory, completing on `bar`.
__device__ inline void bulk_g2s(void* dst_smem, const void* src_gmem, uint32_t bytes,
                                uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// 2-D tensor copy (TMA engine) of the box at column x, row y of `map` into
// shared memory, completing on `bar`.
__device__ inline void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                   uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// Programmatic dependent launch: let the next kernel in the stream start its
// CTAs early, and wait until the previous kernel's writes are visible.
__device__ inline void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ inline void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Hint to bring the 128-byte line holding p into L2.  It has no effect on what
// later loads observe (L2 is the coherence point), so it may run before
// pdl_wait() on data the previous kernel is still writing.
__device__ inline void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// Launch with an optional programmatic-stream-serialization attribute.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_ex(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t s, bool pdl, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ---------------------------------------------------------------------------
// Small numeric helpers.
// ---------------------------------------------------------------------------
__device__ inline float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ inline float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <typename T>
__device__ inline T from_float(float x);
template <>
__device__ inline float from_float<float>(float x) {
  return x;
}
template <>
__device__ inline __nv_bfloat16 from_float<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

template <typename T>
__device__ inline float to_float(T x);
template <>
__device__ inline float to_float<float>(float x) {
  return x;
}
template <>
__device__ inline float to_float<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

// exp2 with -inf - -inf treated as 0 weight.
__device__ inline float exp2_safe(float x, float m) {
  return (m == -INFINITY) ? 0.f : exp2f(x - m);
}

}  // namespace kvc
