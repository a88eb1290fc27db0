// Cache bookkeeping kernels: initialisation, append (positions, units, page
// allocation, RoPE'd K and V writes), online eviction (Sec. 3.3) with
// compaction, and session release.
//
// Allocation rule: pages are taken lowest free id first, in the call's
// session order then token order (append) or session order (evict: all
// sessions' compacted-region pages are allocated before any live page is
// freed).  This makes page tables a deterministic function of the calls.
#include "kvc_launch.cuh"
#include "kvc_rope.cuh"

namespace kvc {

namespace {

constexpr int META_THREADS = 1024;
constexpr unsigned FULL = 0xFFFFFFFFu;

__device__ inline unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}
__device__ inline unsigned lanemask_le() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_le;" : "=r"(m));
  return m;
}

// Block-wide exclusive scan of one int per thread (blockDim.x == 1024).
__device__ int block_exclusive_scan(int v, int* total, int* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(FULL, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = s_warp[lane];
    int xs = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(FULL, xs, o);
      if (lane >= o) xs += y;
    }
    s_warp[lane] = xs - w;  // exclusive warp offsets
    if (lane == 31) s_warp[32] = xs;
  }
  __syncthreads();
  int r = s_warp[warp] + x - v;
  *total = s_warp[32];
  __syncthreads();
  return r;
}

__device__ int block_max(int v, int* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(FULL, v, o));
  if (lane == 0) s_warp[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int w = s_warp[lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w = max(w, __shfl_xor_sync(FULL, w, o));
    if (lane == 0) s_warp[32] = w;
  }
  __syncthreads();
  int r = s_warp[32];
  __syncthreads();
  return r;
}

// Take the k lowest free page ids, mark them used and write them, ascending,
// to d.alloc_list[0..k).  Returns false (and marks nothing) if fewer than k
// pages are free.  Block-uniform result.
__device__ bool block_alloc_lowest(const Dev& d, int k, int* s_warp) {
  __shared__ int s_found;
  if (k == 0) return true;
  if (threadIdx.x == 0) s_found = 0;
  __syncthreads();
  for (int w0 = 0; w0 < d.bitmap_words; w0 += META_THREADS) {
    const int w = w0 + threadIdx.x;
    uint32_t freebits = 0;
    if (w < d.bitmap_words) {
      freebits = ~d.bitmap[w];
      const int64_t first = (int64_t)w * 32;
      if (first + 32 > d.n_pages) {
        const int valid = (int)(d.n_pages - first);
        freebits &= (valid >= 32) ? 0xFFFFFFFFu : ((1u << valid) - 1u);
      }
    }
    int total;
    const int found = s_found;
    const int base = found + block_exclusive_scan(__popc(freebits), &total, s_warp);
    if (w < d.bitmap_words && base < k && freebits) {
      uint32_t take = 0;
      int idx = base;
      uint32_t fb = freebits;
      while (fb && idx < k) {
        const int bit = __ffs(fb) - 1;
        fb &= fb - 1;
        d.alloc_list[idx++] = w * 32 + bit;
        take |= 1u << bit;
      }
      d.bitmap[w] |= take;
    }
    __syncthreads();
    if (threadIdx.x == 0) s_found = min(k, found + total);
    __syncthreads();
    if (s_found >= k) return true;
  }
  // Not enough pages: roll back what was marked.
  const int got = s_found;
  for (int i = threadIdx.x; i < got; i += META_THREADS) {
    const int p = d.alloc_list[i];
    atomicAnd(&d.bitmap[p >> 5], ~(1u << (p & 31)));
  }
  __syncthreads();
  return false;
}

__device__ inline bool evictable_type(int t) { return t == KVC_ACOUSTIC || t == KVC_ASR_DELIM; }

// ---------------------------------------------------------------------------
// Initialisation.
// ---------------------------------------------------------------------------
__global__ void init_state_kernel(Dev d) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < d.n_sessions) {
    SessState s = {};
    s.unit_cur = -1;
    d.sess[i] = s;
  }
  if (i < d.bitmap_words) {
    const int64_t first = (int64_t)i * 32;
    uint32_t w = 0;
    if (first + 32 > d.n_pages) {
      const int valid = (int)(d.n_pages - first);
      w = (valid >= 32) ? 0u : ~((1u << valid) - 1u);
    }
    d.bitmap[i] = w;
  }
}

// cos/sin of p * base^(-2i/D), evaluated in binary64 and stored in binary32.
__global__ void init_rope_kernel(Dev d, double base) {
  const int half = d.head_dim / 2;
  const int64_t n = (int64_t)d.max_positions * half;
  for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < n;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int p = (int)(idx / half), i = (int)(idx % half);
    const double theta = pow(base, -2.0 * (double)i / (double)d.head_dim);
    double sn, cs;
    sincos((double)p * theta, &sn, &cs);
    d.rope[idx] = make_float2((float)cs, (float)sn);
  }
}

// ---------------------------------------------------------------------------
// Append, part 1 (one CTA): page demand, allocation, positions and units
// (warp ballot over UNIT_BEGIN flags), slot tags, state update and the
// split-K work lists of the attention calls that follow.
// ---------------------------------------------------------------------------
__device__ void build_worklist(const Dev& d, int n_seq, int nb, int target, int min_blocks,
                               int max_items, Item* items, int* s_warp, int* s_total_items) {
  const int i = threadIdx.x;
  int total_blocks;
  (void)block_exclusive_scan(i < n_seq ? nb : 0, &total_blocks, s_warp);
  int per = max(min_blocks, (int)(((int64_t)total_blocks * d.kv_heads + target - 1) / target));
  int chunks = 0, base = 0, total_items = 0;
  for (int iter = 0; iter < 32; ++iter) {
    chunks = (i < n_seq) ? min(MAX_CHUNKS_PER_SEQ, (nb + per - 1) / per) : 0;
    base = block_exclusive_scan(chunks, &total_items, s_warp);
    if ((int64_t)total_items * d.kv_heads <= max_items) break;
    per *= 2;
  }
  if (i < n_seq) {
    SeqInfo& si = d.seq[i];
    si.pf_chunks = chunks;
    si.pf_base = base;
    for (int c = 0; c < chunks; ++c) {
      Item it;
      it.seq = i;
      it.chunk = c;
      it.blk_begin = (int)((int64_t)c * nb / chunks);
      it.blk_end = (int)((int64_t)(c + 1) * nb / chunks);
      items[base + c] = it;
    }
  }
  if (threadIdx.x == 0) *s_total_items = total_items;
  __syncthreads();
}

// A failed append leaves the state as it was and gives the K/V writer and the
// attention kernels nothing to do.
__device__ void abandon_append(const Dev& d) {
  d.g->total_tokens = 0;
  d.g->n_units = 0;
  d.g->n_pf_items = 0;
}

__global__ void __launch_bounds__(META_THREADS) append_plan_kernel(Dev d, AppendArgs a,
                                                                   const uint8_t* types) {
  __shared__ int s_warp[33];
  __shared__ int s_bad;
  __shared__ int s_total_dec, s_total_pf;
  const int i = threadIdx.x;
  const int n_seq = a.n_seq;
  if (i == 0) s_bad = 0;
  __syncthreads();

  // 1. Page demand per session (thread i <-> session i of the call).
  int sid = 0, t_len = 0, need = 0;
  SessState st = {};
  if (i < n_seq) {
    sid = a.sessions[i];
    st = d.sess[sid];
    t_len = a.cu[i + 1] - a.cu[i];
    const int tail = st.live_head + st.n_live;
    need = (tail + t_len + PS - 1) / PS - st.n_live_pages;
    if (st.n_live_pages + need > d.max_pages_per_session) atomicOr(&s_bad, KVC_DERR_PAGE_TABLE);
    if (st.pos_next + t_len > d.max_positions) atomicOr(&s_bad, KVC_DERR_POSITION);
  }
  __syncthreads();
  if (s_bad) {
    if (i == 0) {
      set_error(d, s_bad);
      abandon_append(d);
    }
    return;
  }
  int total_need;
  const int off = block_exclusive_scan(need, &total_need, s_warp);
  if (total_need > d.max_alloc || !block_alloc_lowest(d, total_need, s_warp)) {
    if (i == 0) {
      set_error(d, KVC_DERR_POOL);
      abandon_append(d);
    }
    return;
  }
  // 2. New live pages, in call order then token order.
  if (i < n_seq) {
    int32_t* row = d.live_pt + (size_t)sid * d.max_pages_per_session;
    for (int j = 0; j < need; ++j) row[st.n_live_pages + j] = d.alloc_list[off + j];
  }
  __syncthreads();

  // 3. Positions, units and slot tags: one warp per session.
  const int lane = i & 31, warp = i >> 5;
  for (int q = warp; q < n_seq; q += META_THREADS / 32) {
    const int qs = a.sessions[q];
    const SessState s0 = d.sess[qs];
    const int tq = a.cu[q + 1] - a.cu[q];
    const int g0 = a.cu[q];
    const int tail = s0.live_head + s0.n_live;
    const int32_t* row = d.live_pt + (size_t)qs * d.max_pages_per_session;
    int unit_run = s0.unit_cur;
    for (int t0 = 0; t0 < tq; t0 += 32) {
      const int t = t0 + lane;
      const bool valid = t < tq;
      const int ty = valid ? (int)types[g0 + t] : 0;
      const unsigned flags = __ballot_sync(FULL, valid && (ty & KVC_UNIT_BEGIN));
      const int unit = unit_run + __popc(flags & lanemask_le());
      if (valid) {
        const int slot = tail + t;
        const int gs = row[slot / PS] * PS + (slot % PS);
        d.meta_pos[gs] = s0.pos_next + t;
        d.meta_unit[gs] = unit;
        d.meta_type[gs] = (uint8_t)(ty & TYPE_MASK);
        d.tok_slot[g0 + t] = gs;
        d.tok_pos[g0 + t] = s0.pos_next + t;
      }
      unit_run += __popc(flags);
    }
    __syncwarp();
    if (lane == 0) {
      SessState s1 = s0;
      s1.pos_next = s0.pos_next + tq;
      s1.unit_cur = unit_run;
      s1.n_live = s0.n_live + tq;
      s1.last_chunk = tq;
      d.sess[qs] = s1;  // n_live_pages updated below by the owning thread
    }
  }
  __syncthreads();
  int nb = 0;
  if (i < n_seq) {
    SessState s1 = d.sess[sid];
    s1.n_live_pages = st.n_live_pages + need;
    s1.peak_resident = max(s1.peak_resident, s1.n_hist + s1.n_live);
    d.sess[sid] = s1;
    nb = s1.n_hist_pages + s1.n_live_pages;
    SeqInfo si = {};
    si.sid = sid;
    si.t = t_len;
    si.q_row0 = a.cu[i];
    si.pos_first = st.pos_next;
    si.n_hist = s1.n_hist;
    si.n_hist_pages = s1.n_hist_pages;
    si.live_head = s1.live_head;
    si.n_live = s1.n_live;
    si.n_blocks = nb;
    d.seq[i] = si;
  }
  __syncthreads();
  // 4. Split-K work for the attention calls.  The decode and bfloat16 prefill
  // kernels split the call's (session, kv head, page) units evenly over their CTAs
  // (stream-K): they need each session's first unit, the total and the largest
  // session.  The binary32 prefill kernel takes the per-session chunk list.
  {
    int total_units;
    const int ubase = block_exclusive_scan(i < n_seq ? nb * d.kv_heads : 0, &total_units, s_warp);
    const int nb_max = block_max(i < n_seq ? nb : 0, s_warp);
    if (i < n_seq) d.seq[i].unit_base = ubase;
    if (i == 0) {
      s_total_dec = total_units;
      d.g->nb_max = nb_max;
    }
    __syncthreads();
  }
  if (a.pf_target > 0) {
    build_worklist(d, n_seq, nb, a.pf_target, a.pf_min_blocks, d.max_pf_items, d.pf_items,
                   s_warp, &s_total_pf);
  } else if (i == 0) {
    s_total_pf = 0;
  }
  if (i == 0) {
    d.g->n_seq = n_seq;
    d.g->total_tokens = a.total;
    d.g->n_units = s_total_dec;
    d.g->n_pf_items = s_total_pf;
    d.g->pages_used += total_need;
  }
}

// Append, part 2: K rotated at its position (rotate-half, binary32 math on
// the binary32 table), V copied, both into the page slots of part 1.
// grid = (tokens, layers); K/V input layout [L][total][Hkv][D].
template <typename T>
__global__ void __launch_bounds__(256) append_kv_kernel(Dev d, int total, int layer0, const T* k,
                                                        const T* v) {
  // Input layer blockIdx.y of k/v is cache layer layer0 + blockIdx.y.
  const int g = blockIdx.x, l = layer0 + blockIdx.y;
  if (g >= d.g->total_tokens) return;  // the plan kernel failed (device error recorded)
  const int D = d.head_dim, half = D / 2, H = d.kv_heads;
  const int gs = d.tok_slot[g];
  const int pos = d.tok_pos[g];
  const int page = gs / PS, slot = gs % PS;
  const T* kin = k + ((size_t)blockIdx.y * total + g) * H * D;
  const T* vin = v + ((size_t)blockIdx.y * total + g) * H * D;
  T* pool = reinterpret_cast<T*>(d.pool);
  const float2* cs = d.rope + (size_t)pos * half;
  for (int idx = threadIdx.x; idx < H * half; idx += blockDim.x) {
    const int h = idx / half, j = idx % half;
    const float x1 = to_float<T>(kin[h * D + j]);
    const float x2 = to_float<T>(kin[h * D + j + half]);
    float y1, y2;
    rope_pair(x1, x2, cs[j], y1, y2);
    T* dst = pool + pool_offset_elems(d, page, l, 0, h, slot);
    dst[j] = from_float<T>(y1);
    dst[j + half] = from_float<T>(y2);
  }
  const int vec = 16 / (int)sizeof(T);
  for (int idx = threadIdx.x; idx < H * D / vec; idx += blockDim.x) {
    const int h = (idx * vec) / D, j = (idx * vec) % D;
    const uint4 x = *reinterpret_cast<const uint4*>(vin + h * D + j);
    *reinterpret_cast<uint4*>(pool + pool_offset_elems(d, page, l, 1, h, slot) + j) = x;
  }
}

// ---------------------------------------------------------------------------
// Append of exactly one token per session (the decode rounds): thread i plans
// session i of the call (page demand, lowest-free allocation in call order,
// position, unit, slot tags, state, the attention calls' work split); when k and
// v are given the CTA then writes the tokens' rotated K and V of every layer.
// Same state, tags and stored bytes as the general plan kernel followed by
// append_kv_kernel.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(META_THREADS) append_single_kernel(Dev d, AppendArgs a,
                                                                     const uint8_t* types,
                                                                     const T* k, const T* v) {
  __shared__ int s_warp[33];
  __shared__ int s_bad, s_total_pf;
  __shared__ int s_gs[MAX_SEQ], s_pos[MAX_SEQ];
  const int i = threadIdx.x;
  const int n_seq = a.n_seq;
  const int mpps = d.max_pages_per_session;
  if (i == 0) s_bad = 0;
  __syncthreads();

  int sid = 0, need = 0, ty = 0, page = 0;
  SessState st = {};
  if (i < n_seq) {
    sid = a.sessions[i];
    st = d.sess[sid];
    ty = (int)types[i];
    const int tail = st.live_head + st.n_live;
    need = (tail + PS) / PS - st.n_live_pages;
    if (need < 0 || need > 1 || st.n_live_pages + need > mpps)
      atomicOr(&s_bad, KVC_DERR_PAGE_TABLE);
    if (st.pos_next + 1 > d.max_positions) atomicOr(&s_bad, KVC_DERR_POSITION);
    if (need == 0) page = d.live_pt[(size_t)sid * mpps + tail / PS];
  }
  __syncthreads();
  if (s_bad) {
    if (i == 0) {
      set_error(d, s_bad);
      abandon_append(d);
    }
    return;
  }
  int total_need;
  const int off = block_exclusive_scan(need, &total_need, s_warp);
  if (total_need > 0 && (total_need > d.max_alloc || !block_alloc_lowest(d, total_need, s_warp))) {
    if (i == 0) {
      set_error(d, KVC_DERR_POOL);
      abandon_append(d);
    }
    return;
  }
  int nb = 0;
  SeqInfo si = {};
  if (i < n_seq) {
    const int tail = st.live_head + st.n_live;
    if (need) {
      page = d.alloc_list[off];
      d.live_pt[(size_t)sid * mpps + st.n_live_pages] = page;
    }
    const int gs = page * PS + tail % PS;
    const int unit = st.unit_cur + ((ty & KVC_UNIT_BEGIN) ? 1 : 0);
    d.meta_pos[gs] = st.pos_next;
    d.meta_unit[gs] = unit;
    d.meta_type[gs] = (uint8_t)(ty & TYPE_MASK);
    d.tok_slot[i] = gs;
    d.tok_pos[i] = st.pos_next;
    s_gs[i] = gs;
    s_pos[i] = st.pos_next;
    SessState s1 = st;
    s1.pos_next = st.pos_next + 1;
    s1.unit_cur = unit;
    s1.n_live = st.n_live + 1;
    s1.last_chunk = 1;
    s1.n_live_pages = st.n_live_pages + need;
    s1.peak_resident = max(st.peak_resident, s1.n_hist + s1.n_live);
    d.sess[sid] = s1;
    nb = s1.n_hist_pages + s1.n_live_pages;
    si.sid = sid;
    si.t = 1;
    si.q_row0 = i;
    si.pos_first = st.pos_next;
    si.n_hist = s1.n_hist;
    si.n_hist_pages = s1.n_hist_pages;
    si.live_head = s1.live_head;
    si.n_live = s1.n_live;
    si.n_blocks = nb;
  }
  // Split-K work of the attention calls (as in append_plan_kernel).
  int total_units;
  const int ubase = block_exclusive_scan(i < n_seq ? nb * d.kv_heads : 0, &total_units, s_warp);
  const int nb_max = block_max(i < n_seq ? nb : 0, s_warp);
  if (i < n_seq) {
    si.unit_base = ubase;
    d.seq[i] = si;
  }
  __syncthreads();
  s_total_pf = 0;
  if (a.pf_target > 0)
    build_worklist(d, n_seq, nb, a.pf_target, a.pf_min_blocks, d.max_pf_items, d.pf_items,
                   s_warp, &s_total_pf);
  if (i == 0) {
    d.g->n_seq = n_seq;
    d.g->total_tokens = n_seq;
    d.g->n_units = total_units;
    d.g->nb_max = nb_max;
    d.g->n_pf_items = s_total_pf;
    d.g->pages_used += total_need;
  }
  if (k == nullptr) return;
  __syncthreads();
  // K rotated at the token's position and V, every layer and head: one 16-byte chunk
  // of the first half of a K row with its rotate-half partner per K item, one 16-byte
  // chunk of V per V item; K/V input layout [L][n_seq][Hkv][D].  Each thread loads
  // its items of a pass before it stores any, so their loads are in flight together.
  using CK = Chunk16<T>;
  constexpr int VEC = CK::N, UK = sizeof(T) == 2 ? 1 : 2, UV = 4;
  const int D = d.head_dim, half = D / 2, H = d.kv_heads, L = d.layers;
  T* pool = reinterpret_cast<T*>(d.pool);
  const int kc = half / VEC, vc = D / VEC;
  const int n_k = n_seq * L * H * kc, n_v = n_seq * L * H * vc;
  for (int base = i; base < n_k; base += UK * META_THREADS) {
    uint4 wa[UK], wb[UK];
    float2 cs[UK][VEC];
    int64_t dst_off[UK];
#pragma unroll
    for (int u = 0; u < UK; ++u) {
      const int idx = base + u * META_THREADS;
      dst_off[u] = -1;
      if (idx < n_k) {
        const int c = idx % kc, r = idx / kc, h = r % H, q = (r / H) % n_seq, l = r / H / n_seq;
        const T* kin = k + (((size_t)l * n_seq + q) * H + h) * D + c * VEC;
        wa[u] = *reinterpret_cast<const uint4*>(kin);
        wb[u] = *reinterpret_cast<const uint4*>(kin + half);
        const float2* t2 = d.rope + (size_t)s_pos[q] * half + c * VEC;
#pragma unroll
        for (int e = 0; e < VEC; ++e) cs[u][e] = t2[e];
        const int gs = s_gs[q];
        dst_off[u] = (int64_t)(pool_offset_elems(d, gs / PS, l, 0, h, gs % PS) + c * VEC);
      }
    }
#pragma unroll
    for (int u = 0; u < UK; ++u) {
      if (dst_off[u] < 0) break;
      float xa[VEC], xb[VEC], ya[VEC], yb[VEC];
      CK::unpack(wa[u], xa);
      CK::unpack(wb[u], xb);
#pragma unroll
      for (int e = 0; e < VEC; ++e) {
        float y1, y2;
        rope_pair(xa[e], xb[e], cs[u][e], y1, y2);
        ya[e] = y1;
        yb[e] = y2;
      }
      *reinterpret_cast<uint4*>(pool + dst_off[u]) = CK::pack(ya);
      *reinterpret_cast<uint4*>(pool + dst_off[u] + half) = CK::pack(yb);
    }
  }
  for (int base = i; base < n_v; base += UV * META_THREADS) {
    uint4 x[UV];
    int64_t dst_off[UV];
#pragma unroll
    for (int u = 0; u < UV; ++u) {
      const int idx = base + u * META_THREADS;
      dst_off[u] = -1;
      if (idx < n_v) {
        const int c = idx % vc, r = idx / vc, h = r % H, q = (r / H) % n_seq, l = r / H / n_seq;
        x[u] = *reinterpret_cast<const uint4*>(v + (((size_t)l * n_seq + q) * H + h) * D + c * VEC);
        const int gs = s_gs[q];
        dst_off[u] = (int64_t)(pool_offset_elems(d, gs / PS, l, 1, h, gs % PS) + c * VEC);
      }
    }
#pragma unroll
    for (int u = 0; u < UV; ++u) {
      if (dst_off[u] < 0) break;
      *reinterpret_cast<uint4*>(pool + dst_off[u]) = x[u];
    }
  }
}

// ---------------------------------------------------------------------------
// Evict, part 1 (one CTA): the rule of Sec. 3.3 for each session (one warp
// each), compacted-region page allocation, survivor move list, slot tags,
// freeing of consumed live pages, state update.
// ---------------------------------------------------------------------------
struct LiveSlot {
  int unit, type, gs, pos;
};

__device__ inline LiveSlot live_slot(const Dev& d, const SessState& st, const int32_t* row,
                                     int j) {
  const int slot = st.live_head + j;
  const int gs = row[slot / PS] * PS + (slot % PS);
  LiveSlot r;
  r.gs = gs;
  r.unit = d.meta_unit[gs];
  r.type = d.meta_type[gs];
  r.pos = d.meta_pos[gs];
  return r;
}

// Whether a slot inside the consumed live prefix is dropped: its type under the
// rule of Sec. 3.3 and its position-granular variant; its position under the
// sink + recent variant.
__device__ inline bool slot_evicted(const Dev& d, const LiveSlot& ls) {
  if (d.policy == KVC_POLICY_SINK_RECENT) return ls.pos >= d.sink;
  return ls.unit >= 0 && evictable_type(ls.type);
}

// Length of the live prefix a position-granular evict consumes: up to and
// including the need-th evictable slot of a unit <= lim (fewer if fewer exist;
// those units are a prefix of the live region).  One warp.
__device__ int position_variant_end(const Dev& d, const SessState& st, const int32_t* row,
                                    int lim, int need, int lane) {
  int cnt = 0, end = 0;
  for (int w0 = 0; w0 < st.n_live; w0 += 32) {
    const int j = w0 + lane;
    const bool valid = j < st.n_live;
    LiveSlot ls = {INT_MAX, 0, 0, 0};
    if (valid) ls = live_slot(d, st, row, j);
    const unsigned stop = __ballot_sync(FULL, !valid || ls.unit > lim);
    const int first_stop = stop ? __ffs(stop) - 1 : 32;
    const unsigned ev = __ballot_sync(FULL, lane < first_stop && ls.unit >= 0 &&
                                                evictable_type(ls.type));
    const int n_ev = __popc(ev);
    if (cnt + n_ev >= need) {
      unsigned m = ev;  // drop the (need - cnt - 1) lowest set bits: the next is the need-th
      for (int k = need - cnt - 1; k > 0; --k) m &= m - 1;
      return w0 + (__ffs(m) - 1) + 1;
    }
    if (ev) end = w0 + (31 - __clz(ev)) + 1;
    cnt += n_ev;
    if (stop) break;
  }
  return end;
}

// Length of the live prefix a sink + recent evict consumes: every live slot
// whose position is below pos_next - recent (positions ascend along the region).
__device__ int sink_recent_end(const Dev& d, const SessState& st, const int32_t* row,
                               int lane) {
  const int hi = st.pos_next - d.recent;
  int end = 0;
  for (int w0 = 0; w0 < st.n_live; w0 += 32) {
    const int j = w0 + lane;
    const bool in = j < st.n_live && live_slot(d, st, row, j).pos < hi;
    const unsigned b = __ballot_sync(FULL, in);
    end += __popc(b);
    if (b != FULL) break;
  }
  return end;
}

__global__ void __launch_bounds__(META_THREADS) evict_plan_kernel(Dev d, SeqArgs a,
                                                                  int64_t* resident_out) {
  __shared__ int s_warp[33];
  __shared__ int s_end[MAX_SEQ], s_surv[MAX_SEQ], s_nev[MAX_SEQ];
  __shared__ int s_hneed[MAX_SEQ], s_hoff[MAX_SEQ], s_moff[MAX_SEQ];
  __shared__ int s_bad;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_seq = a.n_seq;
  if (tid == 0) s_bad = 0;

  // Phase 1: plan.  For live slot j with unit u >= 0 the unit-level test is
  //   u <= unit_cur - W  and  R0 - (evictable positions before u's first slot) > B,
  // which holds for a prefix of the units; u* is the newest unit with an
  // evictable position that passes it, and `end` is the live prefix of units <= u*.
  for (int q = warp; q < n_seq; q += META_THREADS / 32) {
    const int sid = a.sessions[q];
    const SessState st = d.sess[sid];
    const int32_t* row = d.live_pt + (size_t)sid * d.max_pages_per_session;
    const int r0 = st.n_hist + st.n_live;
    const int lim = st.unit_cur - d.window;
    int ustar = -2;
    if (d.policy == KVC_POLICY_UNIT && d.budget >= 0 && (int64_t)r0 > d.budget &&
        st.n_live > 0) {
      int e_before = 0;        // evictable slots before this window
      int prev_unit = INT_MIN; // unit of the slot just before this window
      int e_at_prev_start = 0; // evictable count before prev_unit's first slot
      for (int w0 = 0; w0 < st.n_live; w0 += 32) {
        const int j = w0 + lane;
        const bool valid = j < st.n_live;
        LiveSlot ls = {INT_MAX, 0, 0, 0};
        if (valid) ls = live_slot(d, st, row, j);
        const bool ev = valid && ls.unit >= 0 && evictable_type(ls.type);
        const unsigned bal_ev = __ballot_sync(FULL, ev);
        const int e_excl = e_before + __popc(bal_ev & lanemask_lt());
        int up = __shfl_up_sync(FULL, ls.unit, 1);
        if (lane == 0) up = prev_unit;
        const unsigned starts = __ballot_sync(FULL, valid && ls.unit != up);
        const unsigned mine = starts & lanemask_le();
        const int src = mine ? 31 - __clz(mine) : 0;
        const int e_src = __shfl_sync(FULL, e_excl, src);
        const int e_ustart = mine ? e_src : e_at_prev_start;
        const bool cond = (ls.unit < 0) ||
                          (ls.unit <= lim && (int64_t)(r0 - e_ustart) > d.budget);
        const unsigned stops = __ballot_sync(FULL, valid && !cond);
        const int first_stop = stops ? __ffs(stops) - 1 : 32;
        int cand = (lane < first_stop && ev) ? ls.unit : -2;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) cand = max(cand, __shfl_xor_sync(FULL, cand, o));
        ustar = max(ustar, cand);
        if (stops) break;
        const int last = min(31, st.n_live - 1 - w0);
        prev_unit = __shfl_sync(FULL, ls.unit, last);
        e_at_prev_start = __shfl_sync(FULL, e_ustart, last);
        e_before += __popc(bal_ev);
      }
    }
    // The consumed live prefix: units <= u* under the rule; for the variants its
    // length is decided first.
    int end = 0, surv = 0, nev = 0;
    int vend = -1;
    if (d.policy == KVC_POLICY_POSITION) {
      vend = (d.budget >= 0 && (int64_t)r0 > d.budget)
                 ? position_variant_end(d, st, row, lim, (int)(r0 - d.budget), lane)
                 : 0;
    } else if (d.policy == KVC_POLICY_SINK_RECENT) {
      vend = sink_recent_end(d, st, row, lane);
    }
    if (ustar >= 0 || vend > 0) {
      for (int w0 = 0; w0 < st.n_live; w0 += 32) {
        const int j = w0 + lane;
        const bool valid = j < st.n_live;
        LiveSlot ls = {INT_MAX, 0, 0, 0};
        if (valid) ls = live_slot(d, st, row, j);
        const bool in = valid && (vend >= 0 ? j < vend : ls.unit <= ustar);
        const bool ev = in && slot_evicted(d, ls);
        const unsigned bin = __ballot_sync(FULL, in);
        end += __popc(bin);
        nev += __popc(__ballot_sync(FULL, ev));
        surv += __popc(__ballot_sync(FULL, in && !ev));
        if (bin != FULL) break;
      }
    }
    if (lane == 0) {
      s_end[q] = end;
      s_surv[q] = surv;
      s_nev[q] = nev;
    }
  }
  __syncthreads();

  // Phase 2: compacted-region page demand, move offsets, allocation.
  int hneed = 0, surv = 0;
  if (tid < n_seq) {
    const SessState st = d.sess[a.sessions[tid]];
    surv = s_surv[tid];
    hneed = (st.n_hist + surv + PS - 1) / PS - st.n_hist_pages;
    if (st.n_hist_pages + hneed > d.max_pages_per_session) atomicOr(&s_bad, KVC_DERR_PAGE_TABLE);
  }
  int total_h, total_moves;
  const int hoff = block_exclusive_scan(hneed, &total_h, s_warp);
  const int moff = block_exclusive_scan(surv, &total_moves, s_warp);
  if (tid < n_seq) {
    s_hneed[tid] = hneed;
    s_hoff[tid] = hoff;
    s_moff[tid] = moff;
  }
  if (tid == 0 && total_moves > d.max_moves) s_bad |= KVC_DERR_MOVES;
  if (tid == 0 && total_h > d.max_alloc) s_bad |= KVC_DERR_POOL;
  __syncthreads();
  if (s_bad) {
    if (tid == 0) {
      set_error(d, s_bad);
      d.g->n_moves = 0;
    }
    return;
  }
  if (!block_alloc_lowest(d, total_h, s_warp)) {
    if (tid == 0) {
      set_error(d, KVC_DERR_POOL);
      d.g->n_moves = 0;
    }
    return;
  }

  // Phase 3: one warp per session.
  __shared__ int s_freed;
  if (tid == 0) s_freed = 0;
  __syncthreads();
  for (int q = warp; q < n_seq; q += META_THREADS / 32) {
    const int sid = a.sessions[q];
    const SessState st = d.sess[sid];
    int32_t* hrow = d.hist_pt + (size_t)sid * d.max_pages_per_session;
    int32_t* lrow = d.live_pt + (size_t)sid * d.max_pages_per_session;
    const int end = s_end[q];
    for (int j = lane; j < s_hneed[q]; j += 32)
      hrow[st.n_hist_pages + j] = d.alloc_list[s_hoff[q] + j];
    __syncwarp();
    int done = 0;  // survivors placed so far
    for (int w0 = 0; w0 < end; w0 += 32) {
      const int j = w0 + lane;
      const bool in = j < end;
      LiveSlot ls = {0, 0, 0, 0};
      if (in) ls = live_slot(d, st, lrow, j);
      const bool sv = in && !slot_evicted(d, ls);
      const unsigned bal = __ballot_sync(FULL, sv);
      if (sv) {
        const int k = done + __popc(bal & lanemask_lt());
        const int di = st.n_hist + k;
        const int dgs = hrow[di / PS] * PS + (di % PS);
        d.moves[s_moff[q] + k] = make_int2(ls.gs, dgs);
        d.meta_pos[dgs] = d.meta_pos[ls.gs];
        d.meta_unit[dgs] = ls.unit;
        d.meta_type[dgs] = (uint8_t)ls.type;
      }
      done += __popc(bal);
    }
    __syncwarp();
    const int consumed = st.live_head + end;
    const int nfree = consumed / PS;
    for (int j = lane; j < nfree; j += 32) {
      const int p = lrow[j];
      atomicAnd(&d.bitmap[p >> 5], ~(1u << (p & 31)));
    }
    __syncwarp();
    const int remain = st.n_live_pages - nfree;
    if (nfree > 0) {
      for (int j0 = 0; j0 < remain; j0 += 32) {
        const int j = j0 + lane;
        const int v = (j < remain) ? lrow[j + nfree] : 0;
        __syncwarp();
        if (j < remain) lrow[j] = v;
        __syncwarp();
      }
    }
    if (lane == 0) {
      SessState s1 = st;
      s1.n_hist = st.n_hist + s_surv[q];
      s1.n_hist_pages = st.n_hist_pages + s_hneed[q];
      s1.live_head = consumed - nfree * PS;
      s1.n_live = st.n_live - end;
      s1.n_live_pages = remain;
      s1.n_evicted = st.n_evicted + s_nev[q];
      d.sess[sid] = s1;
      if (resident_out) resident_out[q] = (int64_t)(s1.n_hist + s1.n_live);
      atomicAdd(&s_freed, nfree);
    }
  }
  __syncthreads();
  if (tid == 0) {
    d.g->n_moves = total_moves;
    d.g->pages_used += total_h - s_freed;
  }
}

// Evict, part 2: move survivors' K/V for every layer, kv slot and head.
// Work unit: 16 bytes; grid-stride over moves x L x 2 x Hkv x (D*esz/16).
__global__ void __launch_bounds__(256) evict_copy_kernel(Dev d) {
  const int n_moves = d.g->n_moves;
  const int vec_per_row = d.head_dim * d.esz / 16;
  const int rows_per_move = d.layers * 2 * d.kv_heads;
  const int64_t total = (int64_t)n_moves * rows_per_move * vec_per_row;
  const size_t row_bytes = (size_t)d.head_dim * d.esz;
  for (int64_t u = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; u < total;
       u += (int64_t)gridDim.x * blockDim.x) {
    const int v = (int)(u % vec_per_row);
    const int64_t r = u / vec_per_row;
    const int rr = (int)(r % rows_per_move);
    const int m = (int)(r / rows_per_move);
    const int h = rr % d.kv_heads;
    const int kv = (rr / d.kv_heads) % 2;
    const int l = rr / (2 * d.kv_heads);
    const int2 mv = d.moves[m];
    const size_t so = pool_offset_elems(d, mv.x / PS, l, kv, h, mv.x % PS) * d.esz;
    const size_t dof = pool_offset_elems(d, mv.y / PS, l, kv, h, mv.y % PS) * d.esz;
    const uint4 x = *reinterpret_cast<const uint4*>(d.pool + so + (size_t)v * 16);
    *reinterpret_cast<uint4*>(d.pool + dof + (size_t)v * 16) = x;
    (void)row_bytes;
  }
}

// ---------------------------------------------------------------------------
// Transcript export (Sec. 4.2): one session's retained TRANSCRIPT positions in
// retained (= position) order.  Part 1 (one CTA): compaction of the retained
// slots by type (block scan); the global slots go to the move list, used as
// scratch, and the positions to pos_out.  Part 2: K and V rows of every layer.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(META_THREADS) transcript_gather_kernel(Dev d, int sid, int cap,
                                                                         int32_t* pos_out,
                                                                         int32_t* count) {
  __shared__ int s_warp[33];
  const SessState st = d.sess[sid];
  const int n = st.n_hist + st.n_live;
  const int32_t* hrow = d.hist_pt + (size_t)sid * d.max_pages_per_session;
  const int32_t* lrow = d.live_pt + (size_t)sid * d.max_pages_per_session;
  int done = 0;
  for (int b0 = 0; b0 < n; b0 += META_THREADS) {
    const int i = b0 + threadIdx.x;
    int gs = 0;
    bool tr = false;
    if (i < n) {
      if (i < st.n_hist) {
        gs = hrow[i / PS] * PS + i % PS;
      } else {
        const int j = st.live_head + i - st.n_hist;
        gs = lrow[j / PS] * PS + j % PS;
      }
      tr = d.meta_type[gs] == KVC_TRANSCRIPT;
    }
    int total;
    const int idx = done + block_exclusive_scan(tr ? 1 : 0, &total, s_warp);
    if (tr && idx < cap) {
      pos_out[idx] = d.meta_pos[gs];
      d.moves[idx] = make_int2(gs, 0);
    }
    done += total;
    __syncthreads();  // s_warp is reused by the next scan
  }
  if (threadIdx.x == 0) {
    *count = done;
    d.g->n_moves = min(done, cap);
  }
}

// Rows [L][cap][Hkv][D] of K and V; 16-byte units, grid-stride.
__global__ void __launch_bounds__(256) transcript_copy_kernel(Dev d, int cap, uint8_t* k_out,
                                                              uint8_t* v_out) {
  const int n = d.g->n_moves;
  const int vec_per_row = d.head_dim * d.esz / 16;
  const int64_t total = (int64_t)n * d.layers * 2 * d.kv_heads * vec_per_row;
  for (int64_t u = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; u < total;
       u += (int64_t)gridDim.x * blockDim.x) {
    const int v = (int)(u % vec_per_row);
    int64_t r = u / vec_per_row;
    const int h = (int)(r % d.kv_heads);
    r /= d.kv_heads;
    const int kv = (int)(r % 2);
    r /= 2;
    const int i = (int)(r % n);
    const int l = (int)(r / n);
    const int gs = d.moves[i].x;
    const size_t src = pool_offset_elems(d, gs / PS, l, kv, h, gs % PS) * d.esz + (size_t)v * 16;
    const size_t dst =
        (((size_t)l * cap + i) * d.kv_heads + h) * d.head_dim * d.esz + (size_t)v * 16;
    *reinterpret_cast<uint4*>((kv ? v_out : k_out) + dst) =
        *reinterpret_cast<const uint4*>(d.pool + src);
  }
}

// Release (one CTA): free every page of the listed sessions and reset them.
__global__ void __launch_bounds__(META_THREADS) release_kernel(Dev d, SeqArgs a) {
  __shared__ int s_freed;
  if (threadIdx.x == 0) s_freed = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int q = warp; q < a.n_seq; q += META_THREADS / 32) {
    const int sid = a.sessions[q];
    const SessState st = d.sess[sid];
    const int32_t* hrow = d.hist_pt + (size_t)sid * d.max_pages_per_session;
    const int32_t* lrow = d.live_pt + (size_t)sid * d.max_pages_per_session;
    for (int j = lane; j < st.n_hist_pages; j += 32) {
      const int p = hrow[j];
      atomicAnd(&d.bitmap[p >> 5], ~(1u << (p & 31)));
    }
    for (int j = lane; j < st.n_live_pages; j += 32) {
      const int p = lrow[j];
      atomicAnd(&d.bitmap[p >> 5], ~(1u << (p & 31)));
    }
    __syncwarp();
    if (lane == 0) {
      SessState s = {};
      s.unit_cur = -1;
      d.sess[sid] = s;
      atomicAdd(&s_freed, st.n_hist_pages + st.n_live_pages);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) d.g->pages_used -= s_freed;
}

}  // namespace

cudaError_t launch_init(const Dev& d, double rope_base, cudaStream_t s) {
  const int n = max(d.n_sessions, d.bitmap_words);
  init_state_kernel<<<(n + 255) / 256, 256, 0, s>>>(d);
  init_rope_kernel<<<1024, 256, 0, s>>>(d, rope_base);
  return cudaGetLastError();
}

cudaError_t launch_append(const Dev& d, const AppendArgs& a, const uint8_t* types, const void* k,
                          const void* v, bool single, cudaStream_t s) {
  if (single) {
    // One CTA writes the K/V rows only for a one-session call (a few hundred KiB at
    // most); larger calls keep the plan in one CTA and spread the rows over
    // append_kv_kernel's grid.
    const bool fuse_kv = a.n_seq == 1;
    if (d.esz == 2)
      append_single_kernel<__nv_bfloat16><<<1, META_THREADS, 0, s>>>(
          d, a, types, static_cast<const __nv_bfloat16*>(fuse_kv ? k : nullptr),
          static_cast<const __nv_bfloat16*>(fuse_kv ? v : nullptr));
    else
      append_single_kernel<float><<<1, META_THREADS, 0, s>>>(
          d, a, types, static_cast<const float*>(fuse_kv ? k : nullptr),
          static_cast<const float*>(fuse_kv ? v : nullptr));
    if (fuse_kv || k == nullptr) return cudaGetLastError();
    return launch_append_layers(d, a.total, 0, d.layers, k, v, s);
  }
  append_plan_kernel<<<1, META_THREADS, 0, s>>>(d, a, types);
  if (k == nullptr) return cudaGetLastError();  // plan only: layers follow one by one
  return launch_append_layers(d, a.total, 0, d.layers, k, v, s);
}

cudaError_t launch_append_layers(const Dev& d, int total, int layer0, int n_layers, const void* k,
                                 const void* v, cudaStream_t s) {
  dim3 grid(total, n_layers);
  if (d.esz == 2)
    append_kv_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(
        d, total, layer0, static_cast<const __nv_bfloat16*>(k),
        static_cast<const __nv_bfloat16*>(v));
  else
    append_kv_kernel<float><<<grid, 256, 0, s>>>(d, total, layer0, static_cast<const float*>(k),
                                                 static_cast<const float*>(v));
  return cudaGetLastError();
}

cudaError_t launch_evict(const Dev& d, const SeqArgs& a, int64_t* resident_out, cudaStream_t s) {
  evict_plan_kernel<<<1, META_THREADS, 0, s>>>(d, a, resident_out);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  evict_copy_kernel<<<sms * 4, 256, 0, s>>>(d);
  return cudaGetLastError();
}

cudaError_t launch_transcript(const Dev& d, int session, int cap, int32_t* pos_out, void* k_out,
                              void* v_out, int32_t* count, cudaStream_t s) {
  transcript_gather_kernel<<<1, META_THREADS, 0, s>>>(d, session, cap, pos_out, count);
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  transcript_copy_kernel<<<sms * 4, 256, 0, s>>>(d, cap, static_cast<uint8_t*>(k_out),
                                                 static_cast<uint8_t*>(v_out));
  return cudaGetLastError();
}

cudaError_t launch_release(const Dev& d, const SeqArgs& a, cudaStream_t s) {
  release_kernel<<<1, META_THREADS, 0, s>>>(d, a);
  return cudaGetLastError();
}

}  // namespace kvc
