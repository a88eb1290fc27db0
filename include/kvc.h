/*
 * kvc.h - C interface of the GB300 library for acoustic-to-text KV eviction
 * and retained-cache GQA attention ("Acoustic-to-Text KV Compression for
 * Full-Duplex Speech Models", Sec. 3.1 and Sec. 3.3).
 *
 * The library keeps, per streaming session, a paged K/V cache for every
 * layer.  Each fed position carries a type tag (acoustic, ASR delimiter,
 * transcript, text).  kvc_evict applies the online eviction rule of
 * Sec. 3.3: while the resident count exceeds the budget B, the acoustic and
 * structural positions of the oldest unit outside the W most recent units
 * are dropped; transcript, response text and the system prefix stay, and
 * kept keys keep their original rotary positions.  The attention calls run
 * over whatever is resident.
 *
 * Conventions for every call:
 *  - Device memory (pool, metadata workspace, q/k/v/out, types) is owned by
 *    the caller and must outlive the context.  The library never calls a
 *    device allocator; kvc_attn_decode_noalloc uses one fixed array that the
 *    library itself defines.
 *  - Calls taking a stream are asynchronous on it (cudaStream_t passed as
 *    void*; NULL is the legacy default stream), except where a comment says
 *    "synchronises".
 *  - Arguments are validated on the host before any launch; on error the
 *    call returns a negative status, launches nothing and changes no state.
 *    kvc_last_error() then describes the failure (thread-local string).
 *  - Kernels never trap.  A capacity check that can only fail on the device
 *    records a code in a device error word and leaves the state as it was;
 *    the next synchronising call returns KVC_EDEVICE (kvc_device_status
 *    reports the recorded code).
 *  - Layouts are row-major and contiguous.  The element type (binary32 or
 *    bfloat16) is fixed at creation for K, V, q and out alike.
 *  - One context serves one host thread and one stream at a time: its
 *    launches share the context's scratch (split-K slots, arrival counters)
 *    and its host mirrors, so calls on it must be ordered on one stream (or
 *    on streams ordered by events) and not made concurrently.  Independent
 *    contexts share nothing.
 */
#ifndef KVC_H
#define KVC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct kvc_ctx kvc_ctx;

/* Element types. */
enum { KVC_F32 = 0, KVC_BF16 = 1 };

/* Token type tags (low 7 bits of a type byte).  Sec. 3.3: ACOUSTIC (unit
 * marker, audio tokens, native decision, terminators) and ASR_DELIM are
 * evictable; TRANSCRIPT and TEXT (response text, system prefix) are kept. */
enum { KVC_ACOUSTIC = 0, KVC_ASR_DELIM = 1, KVC_TRANSCRIPT = 2, KVC_TEXT = 3 };
/* Flag on the first position of a duplex unit (Sec. 3.1); it opens a new
 * unit.  Positions fed before the first flag belong to unit -1 (the system
 * prefix) and are never evicted. */
#define KVC_UNIT_BEGIN 0x80

/* Eviction policies.  KVC_POLICY_UNIT is the rule of Sec. 3.3 (the default).
 * The two others run on the same state for comparison:
 *  - KVC_POLICY_POSITION: the position-granular reading of the same rule:
 *    single evictable positions, oldest first, of the units outside the W most
 *    recent ones, until the resident count fits in B or none is left;
 *  - KVC_POLICY_SINK_RECENT: the StreamingLLM baseline of Table 1 (footnote:
 *    attention-sink tokens plus 2,000 recent positions), type-blind: each
 *    kvc_evict drops every position p with sink <= p < pos_next - recent; B and
 *    W play no part. */
enum { KVC_POLICY_UNIT = 0, KVC_POLICY_POSITION = 1, KVC_POLICY_SINK_RECENT = 2 };

/* Status codes. */
enum {
  KVC_OK = 0,
  KVC_EINVAL = -1,   /* bad argument */
  KVC_ENOMEM = -2,   /* page pool or a capacity would overflow */
  KVC_ECUDA = -3,    /* a CUDA runtime call failed */
  KVC_ESTATE = -4,   /* call out of order (e.g. attention without append) */
  KVC_EDEVICE = -5   /* a kernel recorded a failed check (kvc_device_status) */
};

/* Device error codes (bits of the device error word). */
enum {
  KVC_DERR_POOL = 1,         /* no free page where the host expected one */
  KVC_DERR_PAGE_TABLE = 2,   /* a session's page list is full */
  KVC_DERR_POSITION = 4,     /* position beyond max_positions */
  KVC_DERR_MOVES = 8,        /* eviction move list full */
  KVC_DERR_WAIT = 16         /* a pipeline wait gave up (bounded spin) */
};

typedef struct kvc_config {
  int32_t n_sessions;            /* session ids are 0 .. n_sessions-1 */
  int32_t layers;                /* L */
  int32_t q_heads;               /* Hq */
  int32_t kv_heads;              /* Hkv; Hq % Hkv == 0, G = Hq / Hkv */
  int32_t head_dim;              /* D */
  int32_t page_size;             /* positions per page; 16 */
  int64_t budget;                /* B (Sec. 3.3); < 0 means unbounded */
  int32_t window;                /* W >= 0 most recent units are never evicted */
  int32_t dtype;                 /* KVC_F32 or KVC_BF16 */
  double rope_base;              /* rotary base, e.g. 10000 */
  int64_t n_pages;               /* pool capacity in pages */
  int32_t max_pages_per_session; /* capacity of each of a session's two page lists */
  int32_t max_positions;         /* positions fed to one session stay below this */
  int32_t max_seq_per_call;      /* sessions per call, <= 512 */
  int32_t max_tokens_per_call;   /* tokens per kvc_append_chunk call */
  int32_t policy;                /* KVC_POLICY_*; 0 = the rule of Sec. 3.3 */
  int32_t sink;                  /* KVC_POLICY_SINK_RECENT: first positions always kept */
  int32_t recent;                /* KVC_POLICY_SINK_RECENT: most recent positions kept */
} kvc_config;

/* Supported shapes: (KVC_BF16, head_dim 128) and (KVC_F32, head_dim 64), with
 * G = Hq / Hkv = 4 and page_size 16. */

typedef struct kvc_session_info {
  int32_t pos_next;       /* next position id (= positions fed so far) */
  int32_t unit_cur;       /* current unit, -1 before the first unit marker */
  int32_t n_hist;         /* retained positions in the compacted (hist) region */
  int32_t n_hist_pages;
  int32_t live_head;      /* consumed slots at the front of the first live page */
  int32_t n_live;         /* positions in the live region */
  int32_t n_live_pages;
  int32_t resident;       /* n_hist + n_live */
  int32_t n_evicted;      /* positions evicted so far */
  int32_t peak_resident;  /* largest resident count seen after an append */
} kvc_session_info;

/* Bytes of pool and metadata workspace a configuration needs.
 * Pool layout: page-major, [n_pages][L][2 (K,V)][Hkv][page_size][D] elements.
 * Returns KVC_EINVAL for unsupported or inconsistent configurations. */
int kvc_query_sizes(const kvc_config* cfg, size_t* pool_bytes, size_t* meta_bytes);

/* Create a context over caller-owned device memory (d_pool, d_meta, sizes
 * from kvc_query_sizes or larger; 256-byte aligned).  Zeroes the pool,
 * initialises the metadata and the rotary table (cos/sin of p * base^(-2i/D)
 * evaluated in binary64, stored in binary32), then synchronises `stream`. */
int kvc_create(kvc_ctx** out, const kvc_config* cfg, void* d_pool, size_t pool_bytes,
               void* d_meta, size_t meta_bytes, void* stream);

/* Free the host-side context.  Device memory stays the caller's. */
void kvc_destroy(kvc_ctx* ctx);

/* Feed tokens to sessions (one chunk per session): assign original position
 * ids (Sec. 3.3: they advance with every fed token), open a unit at each
 * KVC_UNIT_BEGIN, rotate K at its position (rotate-half RoPE) and write K, V
 * and the {position, type, unit} tags at the live tail, allocating the lowest
 * free pages in (call order, token order).
 *   n_seq        number of sessions in the call, 1 .. max_seq_per_call
 *   h_sessions   host [n_seq] distinct session ids
 *   h_cu_tokens  host [n_seq+1] token offsets, h_cu_tokens[0] = 0, every
 *                session gets >= 1 token; total <= max_tokens_per_call
 *   d_types      device [total] type bytes
 *   d_k, d_v     device [L][total][Hkv][D] un-rotated keys / values, or both NULL
 *                to write the layers one by one with kvc_append_kv_layer
 * Returns KVC_ENOMEM (nothing launched) if the pool cannot hold the chunk.
 * The chunk's queries are what the following attention calls answer. */
int kvc_append_chunk(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions,
                     const int32_t* h_cu_tokens, const uint8_t* d_types, const void* d_k,
                     const void* d_v, void* stream);

/* Per-layer K/V of the last append, for the model's real order (layer l's K/V
 * exist only after layer l's projections): call kvc_append_chunk with d_k =
 * d_v = NULL (positions, units, pages and tags only), then this for each layer
 * before that layer's attention.  Writes K rotated at its position and V into
 * the chunk's slots.  Attention on a layer whose K/V are not written returns
 * KVC_ESTATE.
 *   layer      0 .. L-1
 *   d_k, d_v   device [total][Hkv][D], total and order as in the last append */
int kvc_append_kv_layer(kvc_ctx* ctx, int layer, const void* d_k, const void* d_v, void* stream);

/* Decode attention of one layer fused with that layer's K/V write (the
 * per-layer order, after kvc_append_chunk without K/V): the new tokens' K
 * (rotated at their positions) and V of the layer are written into their slots
 * and attended in the same launch.  Same results and stored bytes as
 * kvc_append_kv_layer followed by kvc_attn_decode.
 *   d_k, d_v   device [n_seq][Hkv][D], the layer's rows of the appended tokens
 *   other arguments as for kvc_attn_decode */
int kvc_attn_decode_kv(kvc_ctx* ctx, int layer, const void* d_k, const void* d_v,
                       const void* d_q, void* d_out, void* stream);

/* Online eviction (Sec. 3.3) for each listed session, run by the caller after
 * a unit: while resident > B, evict the ACOUSTIC and ASR_DELIM positions of
 * the oldest unit u with 0 <= u <= unit_cur - W that still has some; stop
 * when resident <= B or no such unit remains (the variants of KVC_POLICY_*
 * decide positions instead, see there).  The live slots whose positions the
 * call decided form a prefix of the live region: its survivors move (all
 * layers, 16-byte copies) to the compacted region in position order, and
 * consumed live pages are freed.
 *   d_resident_out  optional device [n_seq] int64: resident count afterwards
 * Invalidates the last append's queries for attention. */
int kvc_evict(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions, int64_t* d_resident_out,
              void* stream);

/* Chunked-prefill GQA attention of one layer for the queries of the last
 * appended chunk.  Sec. 3.1: the model consumes speech in one-second duplex units
 * (a unit marker, about ten audio tokens and the native decision, 17 positions in
 * the workloads here), so each unit's positions enter the language model together
 * as one chunk.  Sec. 3.3: attention runs over whatever the online eviction left
 * resident, and the kept keys are used at their original rotary positions, never
 * re-encoded.  Query t of a session sits at its own position and sees every
 * resident key at or before it (causal inside the chunk):
 * softmax(RoPE(q, p_t) . k / sqrt(D)) v, with the keys stored already rotated at
 * their positions.  Softmax in binary32; for bfloat16 the q.k and P.v products run
 * on tensor cores (tcgen05) with q and P rounded to bfloat16 and binary32
 * accumulation; binary32 calls stay on CUDA cores.
 *   layer   0 .. L-1
 *   d_q     device [total][Hq][D] un-rotated queries, total and order as in
 *           the last kvc_append_chunk; chunks of at most 32 tokens
 *   d_out   device [total][Hq][D]
 * KVC_ESTATE if no append precedes it (or an evict/release came after). */
int kvc_attn_prefill_chunk(kvc_ctx* ctx, int layer, const void* d_q, void* d_out,
                           void* stream);

/* Chunked-prefill attention of one layer fused with that layer's K/V write (the
 * per-layer order, after kvc_append_chunk without K/V; Sec. 3.1: a layer's keys
 * and values of the unit's positions exist only once that layer has run): the
 * chunk's K (rotated at its positions) and V of the layer are written into their
 * slots and attended in the same call.  Same results and stored bytes as
 * kvc_append_kv_layer followed by kvc_attn_prefill_chunk.  For bfloat16 the write
 * happens inside the attention launch; for binary32 it is a separate launch first.
 *   d_k, d_v   device [total][Hkv][D], the layer's rows of the appended chunk,
 *              total and order as in the last append; 16-byte aligned
 *   other arguments as for kvc_attn_prefill_chunk */
int kvc_attn_prefill_chunk_kv(kvc_ctx* ctx, int layer, const void* d_k, const void* d_v,
                              const void* d_q, void* d_out, void* stream);

/* Single-token decode GQA attention of one layer.  Sec. 3.1: after the unit's
 * first decision the model decodes, one token at a time, the transcription
 * segment (<|asr_start|>, up to 64 transcript tokens, <|asr_end|>) and, in SPEAK
 * units, the response text.  Sec. 3.3: each such token attends to the retained
 * cache (the system prefix, transcripts and text of every unit, and the acoustic
 * states of the units the eviction has not reached) with the kept keys at their
 * original rotary positions.  The last append gave each of its n_seq sessions
 * exactly one token; that token attends to every resident key, itself included.
 * Split-K over pages with a log-sum-exp merge.
 * Precision: for bfloat16 the page products run on tensor cores with q and P
 * rounded to bfloat16 and binary32 accumulation and softmax, in every call size;
 * binary32 calls run on CUDA cores in binary32.  The split of a session's pages
 * over CTAs (and so the order of the partial sums) depends on how many sessions
 * share its call, so its output can differ in the last bits with that number;
 * both stay within the attention tolerance.
 *   d_q     device [n_seq][Hq][D] un-rotated queries (call order of the append)
 *   d_out   device [n_seq][Hq][D]
 * May be captured into a CUDA graph: a launch made while `stream` is capturing
 * merges its split-K parts with an acquire-release arrival, so replays are
 * correct; eager launches tag their parts with a per-context launch counter. */
int kvc_attn_decode(kvc_ctx* ctx, int layer, const void* d_q, void* d_out, void* stream);

/* kvc_attn_decode without caller-provided scratch.  The paper has no
 * counterpart.  It is for callers that cannot allocate device memory for
 * scratch when they decode: for example a real-time duplex loop that must not
 * stall on the implicit device synchronisation cudaMalloc and cudaFree can
 * cause inside a one-second unit, or a host application whose device memory is
 * owned by another framework that forbids allocations from outside it.
 *
 * Same arguments, layouts and result as kvc_attn_decode (within the attention
 * tolerance: the split-K chunking differs).  The split-K partial results and
 * arrival counters live in one fixed array in device global memory that the
 * library defines (8.1 MiB in each CUDA context that loads the library, held until
 * the context is destroyed or the process exits), so this call allocates nothing.
 *   - Limit: at most 4096 (session, kv-head) pairs per call, i.e. the last
 *     append's n_seq * kv_heads <= 4096; larger calls return KVC_EINVAL with a
 *     message and launch nothing.
 *   - Each CUDA context holds its own copy of the array (runtime-API callers share
 *     one primary context per device).  The first call made in a context, with
 *     that context current, looks up the array's device address there (and the
 *     SM count and the kernel's occupancy); make that first call before any
 *     stream capture.
 *   - Every call shares its context's array and clears the counters it needs;
 *     calls whose kernels can overlap on the GPU (other streams, other library
 *     contexts over the same CUDA context) race on it, so serialise them. */
int kvc_attn_decode_noalloc(kvc_ctx* ctx, int layer, const void* d_q, void* d_out, void* stream);

/* Resident count of one session (n_hist + n_live), including the system
 * prefix and text (Sec. 3.3).  Synchronises the device. */
int kvc_resident_size(kvc_ctx* ctx, int session, int64_t* h_out);

/* End sessions: free all their pages and reset them to position 0. */
int kvc_release(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions, void* stream);

/* Copy one session's state to host buffers (synchronises).  Page lists go to
 * h_hist_pages / h_live_pages (capacity max_pages_per_session each); the
 * resident positions' {position, type, unit} go, in retained order, to
 * h_pos / h_type / h_unit (capacity `cap` entries each).  Any pointer but
 * h_info may be NULL. */
int kvc_export_state(kvc_ctx* ctx, int session, kvc_session_info* h_info,
                     int32_t* h_hist_pages, int32_t* h_live_pages, int32_t* h_pos,
                     uint8_t* h_type, int32_t* h_unit, int64_t cap);

/* Copy the stored (rotated) K and V of one layer of one session, in retained
 * order, to host buffers [cap][Hkv][D] each (synchronises). */
int kvc_export_kv(kvc_ctx* ctx, int session, int layer, void* h_k, void* h_v, int64_t cap);

/* Transcript export for query-time re-encoding (Sec. 4.2: task queries use
 * only the incoming-speech transcript, re-encoded after the streaming cache is
 * discarded).  Gathers one session's retained TRANSCRIPT positions, in position
 * order, with their stored K (rotated at the original position) and V of every
 * layer.  Asynchronous on stream; uses the eviction move list as scratch (stream
 * order keeps it apart from kvc_evict).  Leaves the cache unchanged.
 *   session    0 .. n_sessions-1
 *   cap        capacity in positions of the outputs; 0 <= cap <= the move list's
 *              capacity (max_seq_per_call * max_pages_per_session * page_size)
 *   d_pos_out  device [cap] int32: original positions
 *   d_k_out, d_v_out  device [L][cap][Hkv][D] each, the cache's element type,
 *              16-byte aligned
 *   d_count    device int32: number of TRANSCRIPT positions retained; the first
 *              min(count, cap) of them are written */
int kvc_export_transcript(kvc_ctx* ctx, int session, int64_t cap, int32_t* d_pos_out,
                          void* d_k_out, void* d_v_out, int32_t* d_count, void* stream);

/* Free pages in the pool and the device error word (synchronises). */
int kvc_device_status(kvc_ctx* ctx, int64_t* h_free_pages, int32_t* h_error_bits);

/* Description of the last failure on this thread ("" if none). */
const char* kvc_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* KVC_H */
