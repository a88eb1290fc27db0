// Host side of the C interface declared in include/kvc.h: argument checks,
// workspace layout, host mirrors for exact pool-exhaustion detection, launches.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "kvc_launch.cuh"

using namespace kvc;

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

#define KVC_CUDA(call)                                                             \
  do {                                                                             \
    cudaError_t e_ = (call);                                                       \
    if (e_ != cudaSuccess)                                                         \
      return fail(KVC_ECUDA, "%s failed: %s", #call, cudaGetErrorString(e_));     \
  } while (0)

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct Sizes {
  int max_moves, max_alloc, dec_slots, dec_tag_slots, max_pf_items;
};

Sizes derive_sizes(const kvc_config& c) {
  Sizes s;
  const int64_t mv = (int64_t)c.max_seq_per_call * c.max_pages_per_session * PS;
  s.max_moves = (int)std::min<int64_t>(mv, 1 << 26);
  s.max_alloc = s.max_moves / PS + c.max_tokens_per_call / PS + 2 * c.max_seq_per_call + 1;
  // Decode partial slots: two per CTA of the stream-K split (grid <= 2048 CTAs).
  s.dec_slots = 4096;
  // Tagged partial slots of the pair-split decode (one per CTA of its one-wave grid).
  s.dec_tag_slots = 2048;
  // Prefill partial slots: the binary32 kernel's chunk list, and two per CTA of the
  // bfloat16 kernel's stream-K split.
  s.max_pf_items = (int)std::min<int64_t>(2048, std::max<int64_t>(512, (int64_t)c.max_seq_per_call * c.kv_heads * 4));
  return s;
}

// Lay out the metadata workspace; with base == nullptr only the size is computed.
size_t layout_meta(const kvc_config& c, uint8_t* base, Dev* d) {
  const Sizes z = derive_sizes(c);
  const int G = c.q_heads / c.kv_heads;
  size_t off = 0;
  auto take = [&](size_t bytes) -> uint8_t* {
    off = align_up(off, 256);
    uint8_t* p = base ? base + off : nullptr;
    off += bytes;
    return p;
  };
  const int64_t slots = c.n_pages * PS;
  const int words = (int)((c.n_pages + 31) / 32);
  const size_t pt = (size_t)c.n_sessions * c.max_pages_per_session * sizeof(int32_t);
  uint8_t* sess = take((size_t)c.n_sessions * sizeof(SessState));
  uint8_t* hist = take(pt);
  uint8_t* live = take(pt);
  uint8_t* mpos = take(slots * 4);
  uint8_t* munit = take(slots * 4);
  uint8_t* mtype = take(slots);
  uint8_t* bitmap = take((size_t)words * 4);
  uint8_t* glob = take(sizeof(DevGlobals));
  uint8_t* rope = take((size_t)c.max_positions * (c.head_dim / 2) * sizeof(float2));
  uint8_t* seq = take((size_t)c.max_seq_per_call * sizeof(SeqInfo));
  uint8_t* pi = take((size_t)z.max_pf_items * sizeof(Item));
  uint8_t* ts = take((size_t)c.max_tokens_per_call * 4);
  uint8_t* tp = take((size_t)c.max_tokens_per_call * 4);
  uint8_t* mv = take((size_t)z.max_moves * sizeof(int2));
  uint8_t* al = take((size_t)z.max_alloc * 4);
  uint8_t* dpo = take((size_t)z.dec_slots * G * c.head_dim * 4);
  uint8_t* dpm = take((size_t)z.dec_slots * G * sizeof(float2));
  uint8_t* dtg = take((size_t)z.dec_tag_slots * (G * c.head_dim + 2 * G) * 8);
  uint8_t* ppo = take((size_t)z.max_pf_items * PF_MAX_TOKENS * G * 128 * 4);
  uint8_t* ppm = take((size_t)z.max_pf_items * PF_MAX_TOKENS * G * sizeof(float2));
  uint8_t* dc = take((size_t)c.max_seq_per_call * c.kv_heads * 4);
  uint8_t* pc = take((size_t)c.max_seq_per_call * c.kv_heads * 4);
  off = align_up(off, 256);
  if (d) {
    d->sess = reinterpret_cast<SessState*>(sess);
    d->hist_pt = reinterpret_cast<int32_t*>(hist);
    d->live_pt = reinterpret_cast<int32_t*>(live);
    d->meta_pos = reinterpret_cast<int32_t*>(mpos);
    d->meta_unit = reinterpret_cast<int32_t*>(munit);
    d->meta_type = mtype;
    d->bitmap = reinterpret_cast<uint32_t*>(bitmap);
    d->g = reinterpret_cast<DevGlobals*>(glob);
    d->rope = reinterpret_cast<float2*>(rope);
    d->seq = reinterpret_cast<SeqInfo*>(seq);
    d->pf_items = reinterpret_cast<Item*>(pi);
    d->tok_slot = reinterpret_cast<int32_t*>(ts);
    d->tok_pos = reinterpret_cast<int32_t*>(tp);
    d->moves = reinterpret_cast<int2*>(mv);
    d->alloc_list = reinterpret_cast<int32_t*>(al);
    d->dec_part_o = reinterpret_cast<float*>(dpo);
    d->dec_part_ml = reinterpret_cast<float2*>(dpm);
    d->dec_tagged = reinterpret_cast<unsigned long long*>(dtg);
    d->dec_tag_slots = z.dec_tag_slots;
    d->pf_part_o = reinterpret_cast<float*>(ppo);
    d->pf_part_ml = reinterpret_cast<float2*>(ppm);
    d->dec_count = reinterpret_cast<int32_t*>(dc);
    d->pf_count = reinterpret_cast<int32_t*>(pc);
    d->max_moves = z.max_moves;
    d->max_alloc = z.max_alloc;
    d->dec_slots = z.dec_slots;
    d->max_pf_items = z.max_pf_items;
    d->bitmap_words = words;
  }
  return off;
}

int check_config(const kvc_config* c) {
  if (!c) return fail(KVC_EINVAL, "config is NULL");
  if (c->n_sessions < 1) return fail(KVC_EINVAL, "n_sessions must be >= 1");
  if (c->layers < 1 || c->layers > 64) return fail(KVC_EINVAL, "layers must be in 1..64");
  if (c->kv_heads < 1 || c->kv_heads > 64) return fail(KVC_EINVAL, "kv_heads must be in 1..64");
  if (c->q_heads != 4 * c->kv_heads)
    return fail(KVC_EINVAL, "q_heads must be 4 * kv_heads (GQA group of 4)");
  if (c->page_size != PS) return fail(KVC_EINVAL, "page_size must be 16");
  if (!((c->dtype == KVC_BF16 && c->head_dim == 128) || (c->dtype == KVC_F32 && c->head_dim == 64)))
    return fail(KVC_EINVAL, "supported (dtype, head_dim): (KVC_BF16, 128), (KVC_F32, 64)");
  if (c->window < 0) return fail(KVC_EINVAL, "window must be >= 0");
  if (c->policy < KVC_POLICY_UNIT || c->policy > KVC_POLICY_SINK_RECENT)
    return fail(KVC_EINVAL, "policy must be one of KVC_POLICY_UNIT, _POSITION, _SINK_RECENT");
  if (c->policy == KVC_POLICY_SINK_RECENT && (c->sink < 0 || c->recent < 0))
    return fail(KVC_EINVAL, "sink and recent must be >= 0");
  if (!(c->rope_base > 0.0)) return fail(KVC_EINVAL, "rope_base must be > 0");
  if (c->n_pages < 1) return fail(KVC_EINVAL, "n_pages must be >= 1");
  const int64_t rows = c->n_pages * c->layers * 2 * c->kv_heads * PS;
  if (rows >= (1LL << 31)) return fail(KVC_EINVAL, "pool too large for 32-bit row coordinates");
  if (c->max_pages_per_session < 1) return fail(KVC_EINVAL, "max_pages_per_session must be >= 1");
  if (c->max_positions < 1 || c->max_positions > (1 << 24))
    return fail(KVC_EINVAL, "max_positions must be in 1..2^24");
  if (c->max_seq_per_call < 1 || c->max_seq_per_call > MAX_SEQ)
    return fail(KVC_EINVAL, "max_seq_per_call must be in 1..%d", MAX_SEQ);
  if (c->max_seq_per_call > c->n_sessions)
    return fail(KVC_EINVAL, "max_seq_per_call must be <= n_sessions");
  if (c->max_tokens_per_call < 1 || c->max_tokens_per_call > (1 << 20))
    return fail(KVC_EINVAL, "max_tokens_per_call must be in 1..2^20");
  return KVC_OK;
}

}  // namespace

struct kvc_ctx {
  kvc_config cfg;
  Dev d;
  // Host mirrors.
  std::vector<int32_t> tail_mod;  // (live_head + n_live) % PS, exact
  std::vector<int32_t> pos_next;  // exact
  int64_t used_ub = 0;            // upper bound of pages in use after enqueued work
  int64_t delta_since_readback = 0;
  bool readback_pending = false;
  cudaEvent_t ev = nullptr;
  int64_t* h_readback = nullptr;  // pinned
  // Last append (queries of the following attention calls).
  bool attn_valid = false;
  int last_n_seq = 0, last_total = 0, last_max_t = 0;
  int attn_since_append = 0;  // attention launches since the last append (or layer write)
  uint64_t layers_written = 0;  // layers whose K/V of the last append are in the pool
  bool last_single = false;
  int pf_target = 0;
  uint32_t dec_epoch = 0;  // tag of the last decode launch's partial states
};

namespace {

int check_sessions(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions) {
  if (n_seq < 1 || n_seq > ctx->cfg.max_seq_per_call)
    return fail(KVC_EINVAL, "n_seq=%d outside 1..%d", n_seq, ctx->cfg.max_seq_per_call);
  if (!h_sessions) return fail(KVC_EINVAL, "h_sessions is NULL");
  std::vector<uint8_t> seen(ctx->cfg.n_sessions, 0);
  for (int i = 0; i < n_seq; ++i) {
    const int s = h_sessions[i];
    if (s < 0 || s >= ctx->cfg.n_sessions) return fail(KVC_EINVAL, "session id %d out of range", s);
    if (seen[s]) return fail(KVC_EINVAL, "session id %d repeated in one call", s);
    seen[s] = 1;
  }
  return KVC_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// Tag for the next decode launch's partial states, or 0 (fenced arrival) while
// the stream is being captured: a graph replays a launch with the tag it was
// captured with, which older words in the slots may carry.  When the counter
// wraps the slots are cleared first, so no word keeps a tag that comes round again.
cudaError_t next_decode_epoch(kvc_ctx* ctx, cudaStream_t s, uint32_t* epoch) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(s, &st);
  if (e != cudaSuccess) return e;
  if (st != cudaStreamCaptureStatusNone) {
    *epoch = 0;
    return cudaSuccess;
  }
  if (++ctx->dec_epoch == 0) {
    const int G = ctx->cfg.q_heads / ctx->cfg.kv_heads;
    e = cudaMemsetAsync(ctx->d.dec_tagged, 0,
                        (size_t)ctx->d.dec_tag_slots * (G * ctx->cfg.head_dim + 2 * G) * 8, s);
    if (e != cudaSuccess) return e;
    ctx->dec_epoch = 1;
  }
  *epoch = ctx->dec_epoch;
  return cudaSuccess;
}

void enqueue_readback(kvc_ctx* ctx, cudaStream_t s) {
  cudaMemcpyAsync(ctx->h_readback, &ctx->d.g->pages_used, sizeof(int64_t), cudaMemcpyDeviceToHost,
                  s);
  cudaEventRecord(ctx->ev, s);
  ctx->readback_pending = true;
  ctx->delta_since_readback = 0;
}

int sync_and_check(kvc_ctx* ctx) {
  KVC_CUDA(cudaDeviceSynchronize());
  int32_t err = 0;
  KVC_CUDA(cudaMemcpy(&err, &ctx->d.g->err, sizeof(err), cudaMemcpyDeviceToHost));
  if (err) return fail(KVC_EDEVICE, "device error bits 0x%x recorded by a kernel", err);
  return KVC_OK;
}

}  // namespace

extern "C" {

const char* kvc_last_error(void) { return g_err.c_str(); }

int kvc_query_sizes(const kvc_config* cfg, size_t* pool_bytes, size_t* meta_bytes) {
  int rc = check_config(cfg);
  if (rc) return rc;
  const size_t esz = cfg->dtype == KVC_BF16 ? 2 : 4;
  if (pool_bytes)
    *pool_bytes = (size_t)cfg->n_pages * cfg->layers * 2 * cfg->kv_heads * PS * cfg->head_dim * esz;
  if (meta_bytes) *meta_bytes = layout_meta(*cfg, nullptr, nullptr);
  return KVC_OK;
}

int kvc_create(kvc_ctx** out, const kvc_config* cfg, void* d_pool, size_t pool_bytes, void* d_meta,
               size_t meta_bytes, void* stream) {
  g_err.clear();
  if (!out) return fail(KVC_EINVAL, "out is NULL");
  *out = nullptr;
  int rc = check_config(cfg);
  if (rc) return rc;
  size_t need_pool = 0, need_meta = 0;
  kvc_query_sizes(cfg, &need_pool, &need_meta);
  if (!d_pool || !d_meta) return fail(KVC_EINVAL, "d_pool / d_meta must be device pointers");
  if ((reinterpret_cast<uintptr_t>(d_pool) & 255) || (reinterpret_cast<uintptr_t>(d_meta) & 255))
    return fail(KVC_EINVAL, "d_pool and d_meta must be 256-byte aligned");
  if (pool_bytes < need_pool)
    return fail(KVC_EINVAL, "pool_bytes %zu < required %zu", pool_bytes, need_pool);
  if (meta_bytes < need_meta)
    return fail(KVC_EINVAL, "meta_bytes %zu < required %zu", meta_bytes, need_meta);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  kvc_ctx* ctx = new kvc_ctx();
  ctx->cfg = *cfg;
  Dev& d = ctx->d;
  memset(&d, 0, sizeof(d));
  d.n_sessions = cfg->n_sessions;
  d.layers = cfg->layers;
  d.q_heads = cfg->q_heads;
  d.kv_heads = cfg->kv_heads;
  d.head_dim = cfg->head_dim;
  d.group = cfg->q_heads / cfg->kv_heads;
  d.esz = cfg->dtype == KVC_BF16 ? 2 : 4;
  d.max_pages_per_session = cfg->max_pages_per_session;
  d.max_positions = cfg->max_positions;
  d.max_seq = cfg->max_seq_per_call;
  d.max_tokens = cfg->max_tokens_per_call;
  d.budget = cfg->budget;
  d.window = cfg->window;
  d.policy = cfg->policy;
  d.sink = cfg->sink;
  d.recent = cfg->recent;
  d.n_pages = cfg->n_pages;
  d.pool = static_cast<uint8_t*>(d_pool);
  layout_meta(*cfg, static_cast<uint8_t*>(d_meta), &d);
  ctx->tail_mod.assign(cfg->n_sessions, 0);
  ctx->pos_next.assign(cfg->n_sessions, 0);
  auto cleanup = [&](int code) {
    if (ctx->ev) cudaEventDestroy(ctx->ev);
    if (ctx->h_readback) cudaFreeHost(ctx->h_readback);
    delete ctx;
    return code;
  };
  if (cudaEventCreateWithFlags(&ctx->ev, cudaEventDisableTiming) != cudaSuccess ||
      cudaMallocHost(&ctx->h_readback, sizeof(int64_t)) != cudaSuccess)
    return cleanup(fail(KVC_ECUDA, "event / pinned readback allocation failed"));
  if (cudaMemsetAsync(d_pool, 0, need_pool, s) != cudaSuccess ||
      cudaMemsetAsync(d_meta, 0, need_meta, s) != cudaSuccess ||
      launch_init(d, cfg->rope_base, s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
    return cleanup(fail(KVC_ECUDA, "initialisation failed: %s",
                        cudaGetErrorString(cudaGetLastError())));
  ctx->pf_target = 3 * prefill_grid_ctas(d);
  *out = ctx;
  return KVC_OK;
}

void kvc_destroy(kvc_ctx* ctx) {
  if (!ctx) return;
  if (ctx->ev) cudaEventDestroy(ctx->ev);
  if (ctx->h_readback) cudaFreeHost(ctx->h_readback);
  delete ctx;
}

int kvc_append_chunk(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions, const int32_t* h_cu_tokens,
                     const uint8_t* d_types, const void* d_k, const void* d_v, void* stream) {
  g_err.clear();
  if (!ctx) return fail(KVC_EINVAL, "ctx is NULL");
  int rc = check_sessions(ctx, n_seq, h_sessions);
  if (rc) return rc;
  if (!h_cu_tokens) return fail(KVC_EINVAL, "h_cu_tokens is NULL");
  if (!d_types) return fail(KVC_EINVAL, "d_types must be non-NULL");
  if ((d_k == nullptr) != (d_v == nullptr))
    return fail(KVC_EINVAL, "d_k and d_v must both be given or both be NULL");
  if (d_k && (!aligned16(d_k) || !aligned16(d_v)))
    return fail(KVC_EINVAL, "d_k / d_v must be 16-byte aligned");
  if (h_cu_tokens[0] != 0) return fail(KVC_EINVAL, "h_cu_tokens[0] must be 0");
  int64_t need = 0;
  int max_t = 0;
  bool single = true;
  for (int i = 0; i < n_seq; ++i) {
    const int t = h_cu_tokens[i + 1] - h_cu_tokens[i];
    if (t < 1) return fail(KVC_EINVAL, "session %d gets %d tokens (must be >= 1)", h_sessions[i], t);
    max_t = std::max(max_t, t);
    single = single && t == 1;
    const int sid = h_sessions[i];
    if ((int64_t)ctx->pos_next[sid] + t > ctx->cfg.max_positions)
      return fail(KVC_ENOMEM, "session %d would exceed max_positions=%d", sid, ctx->cfg.max_positions);
    const int r = ctx->tail_mod[sid];
    need += (r + t + PS - 1) / PS - (r > 0 ? 1 : 0);
  }
  const int total = h_cu_tokens[n_seq];
  if (total > ctx->cfg.max_tokens_per_call)
    return fail(KVC_EINVAL, "%d tokens > max_tokens_per_call=%d", total, ctx->cfg.max_tokens_per_call);
  if (ctx->used_ub + need > ctx->cfg.n_pages && ctx->readback_pending) {
    KVC_CUDA(cudaEventSynchronize(ctx->ev));
    ctx->used_ub = *ctx->h_readback + ctx->delta_since_readback;
    ctx->readback_pending = false;
  }
  if (ctx->used_ub + need > ctx->cfg.n_pages)
    return fail(KVC_ENOMEM, "page pool exhausted: %lld in use (upper bound), %lld needed, %lld total",
                (long long)ctx->used_ub, (long long)need, (long long)ctx->cfg.n_pages);
  AppendArgs a;
  a.n_seq = n_seq;
  a.total = total;
  // Only the binary32 prefill kernel reads the per-session chunk list.
  a.pf_target = ctx->d.esz == 4 ? ctx->pf_target : 0;
  a.pf_min_blocks = 4;
  for (int i = 0; i < n_seq; ++i) a.sessions[i] = h_sessions[i];
  for (int i = 0; i <= n_seq; ++i) a.cu[i] = h_cu_tokens[i];
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  KVC_CUDA(launch_append(ctx->d, a, d_types, d_k, d_v, single, s));
  for (int i = 0; i < n_seq; ++i) {
    const int sid = h_sessions[i];
    const int t = h_cu_tokens[i + 1] - h_cu_tokens[i];
    ctx->tail_mod[sid] = (ctx->tail_mod[sid] + t) % PS;
    ctx->pos_next[sid] += t;
  }
  ctx->used_ub += need;
  ctx->delta_since_readback += need;
  ctx->attn_valid = true;
  ctx->attn_since_append = 0;
  ctx->layers_written = d_k ? (ctx->cfg.layers == 64 ? ~0ull : (1ull << ctx->cfg.layers) - 1) : 0;
  ctx->last_n_seq = n_seq;
  ctx->last_total = total;
  ctx->last_max_t = max_t;
  ctx->last_single = single;
  return KVC_OK;
}

int kvc_append_kv_layer(kvc_ctx* ctx, int layer, const void* d_k, const void* d_v, void* stream) {
  g_err.clear();
  if (!ctx) return fail(KVC_EINVAL, "ctx is NULL");
  if (layer < 0 || layer >= ctx->cfg.layers)
    return fail(KVC_EINVAL, "layer %d outside 0..%d", layer, ctx->cfg.layers - 1);
  if (!d_k || !d_v) return fail(KVC_EINVAL, "d_k / d_v must be non-NULL");
  if (!aligned16(d_k) || !aligned16(d_v)) return fail(KVC_EINVAL, "d_k / d_v must be 16-byte aligned");
  if (!ctx->attn_valid)
    return fail(KVC_ESTATE, "kvc_append_kv_layer needs a preceding kvc_append_chunk (no evict/release after it)");
  KVC_CUDA(launch_append_layers(ctx->d, ctx->last_total, layer, 1, d_k, d_v,
                                static_cast<cudaStream_t>(stream)));
  ctx->layers_written |= 1ull << layer;
  // The next attention launch must not start early: its prologue loads pages
  // this write may still be filling.
  ctx->attn_since_append = 0;
  return KVC_OK;
}

int kvc_evict(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions, int64_t* d_resident_out,
              void* stream) {
  g_err.clear();
  if (!ctx) return fail(KVC_EINVAL, "ctx is NULL");
  int rc = check_sessions(ctx, n_seq, h_sessions);
  if (rc) return rc;
  SeqArgs a;
  a.n_seq = n_seq;
  for (int i = 0; i < n_seq; ++i) a.sessions[i] = h_sessions[i];
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  KVC_CUDA(launch_evict(ctx->d, a, d_resident_out, s));
  ctx->used_ub += n_seq;  // an evict adds at most one page per session, net
  enqueue_readback(ctx, s);
  ctx->attn_valid = false;
  return KVC_OK;
}

int kvc_release(kvc_ctx* ctx, int n_seq, const int32_t* h_sessions, void* stream) {
  g_err.clear();
  if (!ctx) return fail(KVC_EINVAL, "ctx is NULL");
  int rc = check_sessions(ctx, n_seq, h_sessions);
  if (rc) return rc;
  SeqArgs a;
  a.n_seq = n_seq;
  for (int i = 0; i < n_seq; ++i) a.sessions[i] = h_sessions[i];
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  KVC_CUDA(launch_release(ctx->d, a, s));
  for (int i = 0; i < n_seq; ++i) {
    ctx->tail_mod[h_sessions[i]] = 0;
    ctx->pos_next[h_sessions[i]] = 0;
  }
  enqueue_readback(ctx, s);
  ctx->attn_valid = false;
  return KVC_OK;
}

static int check_attn(kvc_ctx* ctx, int layer, const void* d_q, void* d_out,
                      bool writes_layer = false) {
  if (!ctx) return fail(KVC_EINVAL, "ctx is NULL");
  if (layer < 0 || layer >= ctx->cfg.layers)
    return fail(KVC_EINVAL, "layer %d outside 0..%d", layer, ctx->cfg.layers - 1);
  if (!d_q || !d_out) return fail(KVC_EINVAL, "d_q / d_out must be non-NULL");
  if (!aligned16(d_q) || !aligned16(d_out)) return fail(KVC_EINVAL, "d_q / d_out must be 16-byte aligned");
  if (!ctx->attn_valid)
    return fail(KVC_ESTATE, "attention needs a preceding kvc_append_chunk (no evict/release after it)");
  if (!writes_layer && !((ctx->layers_written >> layer) & 1))
    return fail(KVC_ESTATE, "layer %d's K/V of the last append are not written (kvc_append_kv_layer)",
                layer);
  return KVC_OK;
}

int kvc_attn_decode(kvc_ctx* ctx, int layer, const void* d_q, void* d_out, void* stream) {
  g_err.clear();
  int rc = check_attn(ctx, layer, d_q, d_out);
  if (rc) return rc;
  if (!ctx->last_single)
    return fail(KVC_ESTATE, "decode needs exactly one appended token per session");
  // The first attention launch after an append follows the kernel that wrote the
  // new token's K/V, so it does not start early; later ones may.
  uint32_t epoch = 0;
  KVC_CUDA(next_decode_epoch(ctx, static_cast<cudaStream_t>(stream), &epoch));
  KVC_CUDA(launch_attn_decode(ctx->d, layer, d_q, d_out, ctx->last_n_seq,
                              ctx->attn_since_append > 0, static_cast<cudaStream_t>(stream),
                              epoch));
  ++ctx->attn_since_append;
  return KVC_OK;
}

int kvc_attn_decode_kv(kvc_ctx* ctx, int layer, const void* d_k, const void* d_v,
                      const void* d_q, void* d_out, void* stream) {
  g_err.clear();
  int rc = check_attn(ctx, layer, d_q, d_out, true);
  if (rc) return rc;
  if (!d_k || !d_v) return fail(KVC_EINVAL, "d_k / d_v must be non-NULL");
  if (!aligned16(d_k) || !aligned16(d_v)) return fail(KVC_EINVAL, "d_k / d_v must be 16-byte aligned");
  if (!ctx->last_single)
    return fail(KVC_ESTATE, "decode needs exactly one appended token per session");
  // Launches after the append may start early: the new rows go into the tiles
  // after their loads, and the previous launch writes another layer's rows only.
  uint32_t epoch = 0;
  KVC_CUDA(next_decode_epoch(ctx, static_cast<cudaStream_t>(stream), &epoch));
  KVC_CUDA(launch_attn_decode(ctx->d, layer, d_q, d_out, ctx->last_n_seq,
                              ctx->attn_since_append > 0, static_cast<cudaStream_t>(stream),
                              epoch, d_k, d_v));
  ctx->layers_written |= 1ull << layer;
  ++ctx->attn_since_append;
  return KVC_OK;
}

int kvc_attn_decode_noalloc(kvc_ctx* ctx, int layer, const void* d_q, void* d_out,
                            void* stream) {
  g_err.clear();
  int rc = check_attn(ctx, layer, d_q, d_out);
  if (rc) return rc;
  if (!ctx->last_single)
    return fail(KVC_ESTATE, "decode needs exactly one appended token per session");
  const int pairs = ctx->last_n_seq * ctx->cfg.kv_heads;
  if (pairs > noalloc_max_pairs())
    return fail(KVC_EINVAL,
                "kvc_attn_decode_noalloc handles at most %d (session, kv-head) pairs per call; "
                "this call has %d sessions x %d kv heads = %d",
                noalloc_max_pairs(), ctx->last_n_seq, ctx->cfg.kv_heads, pairs);
  KVC_CUDA(launch_attn_decode_noalloc(ctx->d, layer, d_q, d_out, ctx->last_n_seq,
                                      static_cast<cudaStream_t>(stream)));
  return KVC_OK;
}

int kvc_attn_prefill_chunk(kvc_ctx* ctx, int layer, const void* d_q, void* d_out, void* stream) {
  g_err.clear();
  int rc = check_attn(ctx, layer, d_q, d_out);
  if (rc) return rc;
  if (ctx->last_max_t > PF_MAX_TOKENS)
    return fail(KVC_EINVAL, "prefill chunks are limited to %d tokens per session", PF_MAX_TOKENS);
  KVC_CUDA(launch_attn_prefill(ctx->d, layer, d_q, d_out, ctx->last_n_seq, ctx->last_max_t,
                               ctx->attn_since_append > 0, static_cast<cudaStream_t>(stream)));
  ++ctx->attn_since_append;
  return KVC_OK;
}


int kvc_attn_prefill_chunk_kv(kvc_ctx* ctx, int layer, const void* d_k, const void* d_v,
                              const void* d_q, void* d_out, void* stream) {
  g_err.clear();
  int rc = check_attn(ctx, layer, d_q, d_out, true);
  if (rc) return rc;
  if (!d_k || !d_v) return fail(KVC_EINVAL, "d_k / d_v must be non-NULL");
  if (!aligned16(d_k) || !aligned16(d_v)) return fail(KVC_EINVAL, "d_k / d_v must be 16-byte aligned");
  if (ctx->last_max_t > PF_MAX_TOKENS)
    return fail(KVC_EINVAL, "prefill chunks are limited to %d tokens per session", PF_MAX_TOKENS);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (ctx->d.esz == 2) {
    // Launches after the append may start early: a stage holding chunk slots is
    // copied only after its rows are written, and the previous launch writes
    // another layer's rows only.
    KVC_CUDA(launch_attn_prefill(ctx->d, layer, d_q, d_out, ctx->last_n_seq, ctx->last_max_t,
                                 ctx->attn_since_append > 0, s, d_k, d_v));
  } else {
    // Binary32 (CUDA-core prefill): the rows first, then the attention, unoverlapped.
    KVC_CUDA(launch_append_layers(ctx->d, ctx->last_total, layer, 1, d_k, d_v, s));
    KVC_CUDA(launch_attn_prefill(ctx->d, layer, d_q, d_out, ctx->last_n_seq, ctx->last_max_t,
                                 false, s));
  }
  ctx->layers_written |= 1ull << layer;
  ++ctx->attn_since_append;
  return KVC_OK;
}

int kvc_resident_size(kvc_ctx* ctx, int session, int64_t* h_out) {
  g_err.clear();
  if (!ctx || !h_out) return fail(KVC_EINVAL, "ctx / h_out is NULL");
  if (session < 0 || session >= ctx->cfg.n_sessions)
    return fail(KVC_EINVAL, "session id %d out of range", session);
  int rc = sync_and_check(ctx);
  if (rc) return rc;
  SessState st;
  KVC_CUDA(cudaMemcpy(&st, ctx->d.sess + session, sizeof(st), cudaMemcpyDeviceToHost));
  *h_out = (int64_t)st.n_hist + st.n_live;
  return KVC_OK;
}

int kvc_export_state(kvc_ctx* ctx, int session, kvc_session_info* h_info, int32_t* h_hist_pages,
                     int32_t* h_live_pages, int32_t* h_pos, uint8_t* h_type, int32_t* h_unit,
                     int64_t cap) {
  g_err.clear();
  if (!ctx || !h_info) return fail(KVC_EINVAL, "ctx / h_info is NULL");
  if (session < 0 || session >= ctx->cfg.n_sessions)
    return fail(KVC_EINVAL, "session id %d out of range", session);
  int rc = sync_and_check(ctx);
  if (rc) return rc;
  SessState st;
  KVC_CUDA(cudaMemcpy(&st, ctx->d.sess + session, sizeof(st), cudaMemcpyDeviceToHost));
  h_info->pos_next = st.pos_next;
  h_info->unit_cur = st.unit_cur;
  h_info->n_hist = st.n_hist;
  h_info->n_hist_pages = st.n_hist_pages;
  h_info->live_head = st.live_head;
  h_info->n_live = st.n_live;
  h_info->n_live_pages = st.n_live_pages;
  h_info->resident = st.n_hist + st.n_live;
  h_info->n_evicted = st.n_evicted;
  h_info->peak_resident = st.peak_resident;
  const size_t row = (size_t)session * ctx->cfg.max_pages_per_session;
  std::vector<int32_t> hp(st.n_hist_pages), lp(st.n_live_pages);
  if (st.n_hist_pages)
    KVC_CUDA(cudaMemcpy(hp.data(), ctx->d.hist_pt + row, hp.size() * 4, cudaMemcpyDeviceToHost));
  if (st.n_live_pages)
    KVC_CUDA(cudaMemcpy(lp.data(), ctx->d.live_pt + row, lp.size() * 4, cudaMemcpyDeviceToHost));
  if (h_hist_pages) std::copy(hp.begin(), hp.end(), h_hist_pages);
  if (h_live_pages) std::copy(lp.begin(), lp.end(), h_live_pages);
  const int n = st.n_hist + st.n_live;
  if (h_pos || h_type || h_unit) {
    if (n > cap) return fail(KVC_EINVAL, "cap %lld < resident %d", (long long)cap, n);
    std::vector<int32_t> pos(PS), unit(PS);
    std::vector<uint8_t> type(PS);
    auto fetch_page = [&](int page) -> int {
      KVC_CUDA(cudaMemcpy(pos.data(), ctx->d.meta_pos + (size_t)page * PS, PS * 4, cudaMemcpyDeviceToHost));
      KVC_CUDA(cudaMemcpy(unit.data(), ctx->d.meta_unit + (size_t)page * PS, PS * 4, cudaMemcpyDeviceToHost));
      KVC_CUDA(cudaMemcpy(type.data(), ctx->d.meta_type + (size_t)page * PS, PS, cudaMemcpyDeviceToHost));
      return KVC_OK;
    };
    int i = 0;
    for (int b = 0; b < st.n_hist_pages; ++b) {
      if ((rc = fetch_page(hp[b]))) return rc;
      for (int s = 0; s < PS && b * PS + s < st.n_hist; ++s, ++i) {
        if (h_pos) h_pos[i] = pos[s];
        if (h_type) h_type[i] = type[s];
        if (h_unit) h_unit[i] = unit[s];
      }
    }
    for (int b = 0; b < st.n_live_pages; ++b) {
      if ((rc = fetch_page(lp[b]))) return rc;
      for (int s = 0; s < PS; ++s) {
        const int j = b * PS + s;
        if (j < st.live_head || j >= st.live_head + st.n_live) continue;
        if (h_pos) h_pos[i] = pos[s];
        if (h_type) h_type[i] = type[s];
        if (h_unit) h_unit[i] = unit[s];
        ++i;
      }
    }
  }
  return KVC_OK;
}

int kvc_export_transcript(kvc_ctx* ctx, int session, int64_t cap, int32_t* d_pos_out,
                          void* d_k_out, void* d_v_out, int32_t* d_count, void* stream) {
  g_err.clear();
  if (!ctx || !d_count) return fail(KVC_EINVAL, "ctx / d_count is NULL");
  if (session < 0 || session >= ctx->cfg.n_sessions)
    return fail(KVC_EINVAL, "session id %d out of range", session);
  if (cap < 0 || cap > ctx->d.max_moves)
    return fail(KVC_EINVAL, "cap must be in 0..%d", ctx->d.max_moves);
  if (cap > 0 && (!d_pos_out || !d_k_out || !d_v_out))
    return fail(KVC_EINVAL, "output buffers are NULL");
  if (cap > 0 && (!aligned16(d_k_out) || !aligned16(d_v_out)))
    return fail(KVC_EINVAL, "d_k_out / d_v_out must be 16-byte aligned");
  KVC_CUDA(launch_transcript(ctx->d, session, (int)cap, d_pos_out, d_k_out, d_v_out, d_count,
                             static_cast<cudaStream_t>(stream)));
  return KVC_OK;
}

int kvc_export_kv(kvc_ctx* ctx, int session, int layer, void* h_k, void* h_v, int64_t cap) {
  g_err.clear();
  if (!ctx || !h_k || !h_v) return fail(KVC_EINVAL, "ctx / h_k / h_v is NULL");
  if (session < 0 || session >= ctx->cfg.n_sessions)
    return fail(KVC_EINVAL, "session id %d out of range", session);
  if (layer < 0 || layer >= ctx->cfg.layers) return fail(KVC_EINVAL, "layer out of range");
  int rc = sync_and_check(ctx);
  if (rc) return rc;
  SessState st;
  KVC_CUDA(cudaMemcpy(&st, ctx->d.sess + session, sizeof(st), cudaMemcpyDeviceToHost));
  const int n = st.n_hist + st.n_live;
  if (n > cap) return fail(KVC_EINVAL, "cap %lld < resident %d", (long long)cap, n);
  const Dev& d = ctx->d;
  const size_t row = (size_t)session * ctx->cfg.max_pages_per_session;
  std::vector<int32_t> hp(st.n_hist_pages), lp(st.n_live_pages);
  if (st.n_hist_pages)
    KVC_CUDA(cudaMemcpy(hp.data(), d.hist_pt + row, hp.size() * 4, cudaMemcpyDeviceToHost));
  if (st.n_live_pages)
    KVC_CUDA(cudaMemcpy(lp.data(), d.live_pt + row, lp.size() * 4, cudaMemcpyDeviceToHost));
  const size_t vec = (size_t)d.head_dim * d.esz;              // one head row
  const size_t blk = (size_t)d.kv_heads * PS * vec;           // K (or V) of one page-layer
  std::vector<uint8_t> kb(blk), vb(blk);
  uint8_t* ko = static_cast<uint8_t*>(h_k);
  uint8_t* vo = static_cast<uint8_t*>(h_v);
  int i = 0;
  auto emit = [&](int page, int s_lo, int s_hi) -> int {
    const size_t base = pool_offset_elems(d, page, layer, 0, 0, 0) * d.esz;
    KVC_CUDA(cudaMemcpy(kb.data(), d.pool + base, blk, cudaMemcpyDeviceToHost));
    KVC_CUDA(cudaMemcpy(vb.data(), d.pool + base + blk, blk, cudaMemcpyDeviceToHost));
    for (int s = s_lo; s < s_hi; ++s, ++i)
      for (int h = 0; h < d.kv_heads; ++h) {
        memcpy(ko + ((size_t)i * d.kv_heads + h) * vec, kb.data() + ((size_t)h * PS + s) * vec, vec);
        memcpy(vo + ((size_t)i * d.kv_heads + h) * vec, vb.data() + ((size_t)h * PS + s) * vec, vec);
      }
    return KVC_OK;
  };
  for (int b = 0; b < st.n_hist_pages; ++b)
    if ((rc = emit(hp[b], 0, std::min(PS, st.n_hist - b * PS)))) return rc;
  for (int b = 0; b < st.n_live_pages; ++b) {
    const int lo = std::max(0, st.live_head - b * PS);
    const int hi = std::min(PS, st.live_head + st.n_live - b * PS);
    if (hi > lo && (rc = emit(lp[b], lo, hi))) return rc;
  }
  return KVC_OK;
}

int kvc_device_status(kvc_ctx* ctx, int64_t* h_free_pages, int32_t* h_error_bits) {
  g_err.clear();
  if (!ctx) return fail(KVC_EINVAL, "ctx is NULL");
  KVC_CUDA(cudaDeviceSynchronize());
  DevGlobals g;
  KVC_CUDA(cudaMemcpy(&g, ctx->d.g, sizeof(g), cudaMemcpyDeviceToHost));
  if (h_free_pages) *h_free_pages = ctx->cfg.n_pages - g.pages_used;
  if (h_error_bits) *h_error_bits = g.err;
  ctx->used_ub = g.pages_used;
  ctx->delta_since_readback = 0;
  ctx->readback_pending = false;
  return KVC_OK;
}

}  // extern "C"
