"""Drive the CUDA library with a synthetic workload, one duplex step at a time.

A step advances every active session by one unit (Sec. 3.1): one append of
the 17 acoustic positions and the chunked-prefill attention of every layer,
then the segment/response tokens one at a time (append + decode attention of
every layer), then one eviction call (Sec. 3.3).  Inputs come from the
seeded generators of this package (on the device, bit-identical to
``synth.values``); nothing here computes any part of the method.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

from . import gpu as G
from . import values as V
from .script import (ACOUSTIC, ACOUSTIC_PER_UNIT, UNIT_BEGIN, SessionScript, Workload,
                     schedule)


def resident_bound(w: Workload, sc: SessionScript) -> tuple[int, int]:
    """(upper bound of resident positions, total positions) of one session.

    After an eviction the resident count is at most max(B, protected + window
    positions); one unit's growth comes on top before the next eviction.
    """
    unit_len = [ACOUSTIC_PER_UNIT + (0 if t < 0 else t + 2) + x
                for t, x in zip(sc.n_transcript.tolist(), sc.n_text.tolist())]
    total = sc.prefix_len + sum(unit_len)
    if w.budget < 0:
        return total, total
    protected = sc.prefix_len + int(np.maximum(sc.n_transcript, 0).sum()) + int(sc.n_text.sum())
    top = sorted(unit_len, reverse=True)
    window_pos = sum(top[:w.window + 1])
    bound = max(w.budget, protected + window_pos) + top[0]
    return min(bound, total), total


def cache_sizing(w: Workload, scripts: list[SessionScript], concurrent: int | None = None) -> dict:
    ps = w.page_size
    bounds = [resident_bound(w, s) for s in scripts]
    per_sess_pages = [b // ps + 4 + (b // ps + 2) for b, _ in bounds]  # + evict transient
    k = len(scripts) if concurrent is None else concurrent
    n_pages = sum(sorted(per_sess_pages, reverse=True)[:k]) + 16
    max_t = max(ACOUSTIC_PER_UNIT, max(s.prefix_len for s in scripts))
    return dict(
        n_pages=n_pages,
        max_pages_per_session=max(per_sess_pages),
        max_positions=max(t for _, t in bounds) + 1,
        max_seq_per_call=min(len(scripts), 512),
        max_tokens_per_call=min(len(scripts), 512) * max_t,
    )


@dataclass
class Call:
    """One append and the attention calls that answer its queries."""
    kind: str                      # "prefill" or "decode"
    sessions: np.ndarray           # int32, call order
    cu: np.ndarray                 # int32 token offsets
    positions: list                # per session, positions of its tokens
    types: object = None           # device uint8 [total]
    types_host: np.ndarray = None  # the same, on the host
    k: object = None               # device [L][total][Hkv][D]
    v: object = None
    q: object = None               # device [L][total][Hq][D]
    out: object = None             # device [total][Hq][D]
    raw: tuple = None              # host pointers / device addresses for the raw calls


@dataclass
class Step:
    index: int
    pairs: list
    calls: list = field(default_factory=list)
    evict_sessions: np.ndarray = None


class Driver:
    def __init__(self, w: Workload, scripts: list[SessionScript], cache=None, device="cuda",
                 sizing: dict | None = None):
        import torch
        from paper_2609_31224_gb300 import KVCache
        self.torch = torch
        self.w = w
        self.scripts = {s.session: s for s in scripts}
        self.sched = schedule(scripts)
        self.device = device
        self.sizing = sizing or cache_sizing(w, scripts)
        self.cache = cache or KVCache(n_sessions=w.n_sessions, layers=w.layers,
                                      q_heads=w.q_heads, kv_heads=w.kv_heads,
                                      head_dim=w.head_dim, budget=w.budget, window=w.window,
                                      dtype=w.dtype, rope_base=w.rope_base,
                                      page_size=w.page_size, policy=w.policy, sink=w.sink,
                                      recent=w.recent, device=device, **self.sizing)
        self.pos = np.zeros(w.n_sessions, dtype=np.int64)  # host copy of positions fed
        self.tdtype = torch.bfloat16 if w.dtype == "bf16" else torch.float32
        self.step_index = 0
        self.stream = torch.cuda.current_stream().cuda_stream
        self.resident_out = torch.zeros(self.sizing["max_seq_per_call"], dtype=torch.int64,
                                        device=device)

    # -- inputs ----------------------------------------------------------------------------
    def _fill(self, tag, heads, tok_sess, tok_pos, scale):
        t = self.torch.empty((self.w.layers, len(tok_sess), heads, self.w.head_dim),
                             dtype=self.tdtype, device=self.device)
        G.fill(t, self.w.dtype, self.w.seed, tag,
               self.torch.as_tensor(tok_sess, dtype=self.torch.int32, device=self.device),
               self.torch.as_tensor(tok_pos, dtype=self.torch.int32, device=self.device),
               scale)
        return t

    def _make_call(self, kind, sessions, types_per_session, with_q: bool) -> Call:
        torch = self.torch
        w = self.w
        sess = np.asarray(sessions, dtype=np.int32)
        counts = [len(t) for t in types_per_session]
        cu = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
        positions, tok_sess, tok_pos = [], [], []
        for s, n in zip(sess.tolist(), counts):
            p = list(range(int(self.pos[s]), int(self.pos[s]) + n))
            self.pos[s] += n
            positions.append(p)
            tok_sess += [s] * n
            tok_pos += p
        c = Call(kind=kind, sessions=sess, cu=cu, positions=positions)
        c.types_host = np.concatenate(types_per_session).astype(np.uint8)
        c.types = torch.as_tensor(c.types_host, device=self.device)
        c.k = self._fill(V.TAG_K, w.kv_heads, tok_sess, tok_pos, w.kv_scale)
        c.v = self._fill(V.TAG_V, w.kv_heads, tok_sess, tok_pos, w.kv_scale)
        if with_q:
            c.q = self._fill(V.TAG_Q, w.q_heads, tok_sess, tok_pos, w.q_scale)
            c.out = torch.empty((int(cu[-1]), w.q_heads, w.head_dim), dtype=self.tdtype,
                                device=self.device)
        self._bind(c)
        return c

    def _bind(self, c: Call) -> None:
        """Precompute the raw call arguments (done outside any timed region)."""
        from paper_2609_31224_gb300._lib import host_i32
        s_arr, s_p = host_i32(c.sessions)
        c_arr, c_p = host_i32(c.cu)
        q_ptrs = None
        if c.q is not None:
            base, stride = c.q.data_ptr(), c.q.stride(0) * c.q.element_size()
            q_ptrs = [base + l * stride for l in range(self.w.layers)]
        c.raw = (s_arr, s_p, c_arr, c_p, c.types.data_ptr(), c.k.data_ptr(), c.v.data_ptr(),
                 q_ptrs, None if c.out is None else c.out.data_ptr())

    def prepare_step(self, with_q: bool = True) -> Step:
        """Generate (on the device) every input of the next step; advances host positions."""
        pairs = self.sched[self.step_index]
        st = Step(index=self.step_index, pairs=pairs)
        self.step_index += 1
        if not pairs:
            return st
        # System prefix of sessions starting now (appended without attention).
        pre = [(s, self.scripts[s]) for s, u in pairs if u == 0 and self.scripts[s].prefix_len]
        if pre:
            st.calls.append(self._make_call("prefix", [s for s, _ in pre],
                                            [sc.prefix_types() for _, sc in pre], False))
        sessions = [s for s, _ in pairs]
        st.calls.append(self._make_call(
            "prefill", sessions, [self.scripts[s].prefill_types() for s in sessions], with_q))
        dec = {s: self.scripts[s].decode_types(u) for s, u in pairs}
        rounds = max((len(t) for t in dec.values()), default=0)
        for r in range(rounds):
            act = [s for s in sessions if len(dec[s]) > r]
            st.calls.append(self._make_call("decode", act, [dec[s][r:r + 1] for s in act],
                                            with_q))
        st.evict_sessions = np.asarray(sessions, dtype=np.int32)
        return st

    # -- API calls ---------------------------------------------------------------------------
    def run_call(self, c: Call, attention: bool = True, on_attention=None,
                 on_append=None, per_layer: bool = False) -> int:
        """Append + (optionally) every layer's attention. Returns kernels launched.

        per_layer: the model's order; the append carries no K/V and each layer's K/V
        are written by that layer's attention call (kvc_attn_decode_kv,
        kvc_attn_prefill_chunk_kv), or, for calls without attention, just before it
        would run (kvc_append_kv_layer)."""
        cache = self.cache
        _, s_p, _, c_p, t_ptr, k_ptr, v_ptr, q_ptrs, o_ptr = c.raw
        stream = self.stream
        cache.append_chunk_raw(len(c.sessions), s_p, c_p, t_ptr, None if per_layer else k_ptr,
                               None if per_layer else v_ptr, stream)
        if on_append is not None:
            on_append(c)
        launches = 1 if per_layer else 2
        do_attn = attention and c.q is not None and c.kind != "prefix"
        fn = cache.attn_prefill_raw if c.kind == "prefill" else cache.attn_decode_raw
        kv_stride = c.k.stride(0) * c.k.element_size()
        for layer in range(self.w.layers):
            kl, vl = k_ptr + layer * kv_stride, v_ptr + layer * kv_stride
            if per_layer and do_attn:
                # The layer's K/V write fused into its attention call.
                fused = (cache.attn_decode_kv_raw if c.kind == "decode"
                         else cache.attn_prefill_kv_raw)
                fused(layer, kl, vl, q_ptrs[layer], o_ptr, stream)
                launches += 1 if (c.kind == "decode" or self.w.dtype == "bf16") else 2
                if on_attention is not None:
                    on_attention(c, layer)
                continue
            if per_layer:
                cache.append_kv_layer_raw(layer, kl, vl, stream)
                launches += 1
            if do_attn:
                fn(layer, q_ptrs[layer], o_ptr, stream)
                launches += 1
                if on_attention is not None:
                    on_attention(c, layer)
        return launches

    def run_step(self, st: Step, attention: bool = True, on_attention=None,
                 on_evict=None, on_append=None, per_layer: bool = False) -> int:
        launches = 0
        for c in st.calls:
            launches += self.run_call(c, attention, on_attention, on_append, per_layer)
        if st.evict_sessions is not None and len(st.evict_sessions):
            self.cache.evict(st.evict_sessions, self.resident_out)
            launches += 2
            if on_evict is not None:
                on_evict(st)
        return launches

    def release(self, sessions) -> None:
        """End sessions (kvc_release): their positions start over at 0; later steps feed
        them the rest of their scripts."""
        self.cache.release(np.asarray(sessions, dtype=np.int32))
        for s in sessions:
            self.pos[s] = 0

    def fast_forward(self, n_steps: int) -> None:
        """Advance the cache state without attention (attention does not change state)."""
        for _ in range(n_steps):
            st = self.prepare_step(with_q=False)
            self.run_step(st, attention=False)
            del st
