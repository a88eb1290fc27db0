"""Lockstep runner: the CUDA library (through synth.driver) and the oracle fed the
same calls with the same seeded inputs, compared call by call."""
from __future__ import annotations

import numpy as np

from oracle.cache import OracleCache, OracleConfig
from synth import values as V

TOL = {"bf16": (2e-2, 1e-2, 1e-2), "f32": (1e-4, 1e-4, 1e-5)}  # atol, rtol, normwise


def assert_close(gpu: np.ndarray, ref: np.ndarray, dtype: str, what: str = "",
                 tol=None) -> dict:
    atol, rtol, normwise = TOL[dtype] if tol is None else tol
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    err = np.abs(gpu - ref)
    bad = err > atol + rtol * np.abs(ref)
    nw = float(np.linalg.norm(gpu - ref) / max(np.linalg.norm(ref), 1e-30))
    stats = {"max_abs": float(err.max()), "normwise": nw,
             "max_rel": float((err / np.maximum(np.abs(ref), 1e-6)).max())}
    assert not bad.any(), f"{what}: {int(bad.sum())} elements out of tolerance, {stats}"
    assert nw <= normwise, f"{what}: normwise error {nw} > {normwise}"
    return stats


def compare_state(gpu_state: dict, ref_state: dict, what: str = "") -> None:
    for key in ("pos_next", "unit_cur", "n_hist", "live_head", "n_live", "hist_pages",
                "live_pages", "resident", "n_evicted", "peak_resident", "pos", "type", "unit"):
        assert gpu_state[key] == ref_state[key], f"{what}: {key} differs"


class Lockstep:
    MEMO_ENTRIES = 40

    def __init__(self, driver, w, tol=None):
        self.drv = driver
        self.w = w
        self.tol = tol
        self.orc = OracleCache(OracleConfig(
            n_sessions=w.n_sessions, layers=w.layers, q_heads=w.q_heads, kv_heads=w.kv_heads,
            head_dim=w.head_dim, page_size=w.page_size, budget=w.budget, window=w.window,
            dtype=w.dtype, rope_base=w.rope_base, n_pages=driver.sizing["n_pages"],
            policy=w.policy, sink=w.sink, recent=w.recent))
        self.stats = []
        self.n_compared = 0
        self.compared_calls = set()
        self._memo = {}

    def _generate_kv(self, s, layer, positions):
        w = self.w
        k = V.layer_tensor(w.seed, V.TAG_K, s, layer, positions, w.kv_heads, w.head_dim,
                           w.dtype, w.kv_scale)
        v = V.layer_tensor(w.seed, V.TAG_V, s, layer, positions, w.kv_heads, w.head_dim,
                           w.dtype, w.kv_scale)
        return k, v

    def kv_source(self, s, layer, positions):
        """Raw K and V rows of `positions`, from the seeded generator.  Rows already
        generated for (s, layer) are reused (the generator is a pure function of
        (seed, tensor, session, layer, position, head, dim)); at most MEMO_ENTRIES
        (session, layer) entries are kept, least recently used dropped first."""
        positions = np.asarray(positions, dtype=np.int64)
        key = (int(s), int(layer))
        memo = self._memo.pop(key, None)
        if memo is None:
            memo = (np.empty(0, np.int64), None, None)
        mpos, mk, mv = memo
        missing = np.setdiff1d(positions, mpos)
        if missing.size:
            nk, nv = self._generate_kv(s, layer, missing)
            nk, nv = nk.astype(np.float32), nv.astype(np.float32)
            if mk is None:
                mpos, mk, mv = missing, nk, nv
            else:
                mpos = np.concatenate([mpos, missing])
                mk, mv = np.concatenate([mk, nk]), np.concatenate([mv, nv])
                order = np.argsort(mpos, kind="stable")
                mpos, mk, mv = mpos[order], mk[order], mv[order]
        self._memo[key] = (mpos, mk, mv)
        while len(self._memo) > self.MEMO_ENTRIES:
            self._memo.pop(next(iter(self._memo)))
        idx = np.searchsorted(mpos, positions)
        return mk[idx].astype(np.float64), mv[idx].astype(np.float64)

    def q_raw(self, s, layer, positions):
        w = self.w
        return V.layer_tensor(w.seed, V.TAG_Q, s, layer, positions, w.q_heads, w.head_dim,
                              w.dtype, w.q_scale)

    def on_append(self, c) -> None:
        """Feed the oracle the call just appended on the device."""
        self.orc.append_chunk(c.sessions.tolist(),
                              [c.types_host[c.cu[i]:c.cu[i + 1]] for i in range(len(c.sessions))])

    def compare_call(self, c, layer, sessions=None, what="") -> None:
        """Compare the device output of `c` at `layer` (just computed) with the oracle, for
        the listed sessions of the call (all of them when None)."""
        out = c.out.float().cpu().numpy()
        chosen = [i for i, s in enumerate(c.sessions.tolist())
                  if sessions is None or s in sessions]
        if not chosen:
            return
        sess = [int(c.sessions[i]) for i in chosen]
        qs = [self.q_raw(s, layer, c.positions[i]) for i, s in zip(chosen, sess)]
        refs = self.orc.attend(layer, qs, self.kv_source, sessions=sess)
        for i, ref in zip(chosen, refs):
            got = out[c.cu[i]:c.cu[i + 1]]
            self.stats.append(assert_close(
                got, ref, self.w.dtype,
                f"{what} {c.kind} ({len(c.sessions)} sessions) layer {layer} "
                f"session {int(c.sessions[i])}", self.tol))
            self.n_compared += 1
        self.compared_calls.add((id(c), len(c.sessions)))

    def run_step(self, attn_pred=None, session_pred=None, check_state=True,
                 state_sessions=None, per_layer=False, select=None):
        """One duplex step on both sides.

        attn_pred(step, call_kind, call_index, layer) -> bool selects attention calls to
        compare; session_pred(session) -> bool selects the sessions compared in them.
        select(step, call, call_index, layer) -> None (skip), "all" or a set of sessions
        replaces both when given.
        """
        st = self.drv.prepare_step()
        call_idx = {}

        def on_append(c):
            self.on_append(c)
            call_idx[id(c)] = len(call_idx)

        def on_attention(c, layer):
            if select is not None:
                chosen = select(st.index, c, call_idx[id(c)], layer)
                if chosen is None:
                    return
                self.compare_call(c, layer, None if chosen == "all" else set(chosen),
                                  f"step {st.index}")
                return
            if attn_pred is None or not attn_pred(st.index, c.kind, call_idx[id(c)], layer):
                return
            chosen = None if session_pred is None else {
                int(s) for s in c.sessions.tolist() if session_pred(int(s))}
            self.compare_call(c, layer, chosen, f"step {st.index}")

        def on_evict(step):
            res = self.orc.evict(step.evict_sessions.tolist())
            if not check_state:
                return
            got_res = self.drv.resident_out[:len(res)].cpu().numpy().tolist()
            assert got_res == res, f"step {step.index}: resident counts differ"
            for s in (step.evict_sessions.tolist() if state_sessions is None else
                      [x for x in step.evict_sessions.tolist() if x in state_sessions]):
                compare_state(self.drv.cache.export_state(s), self.orc.state(s),
                              f"step {step.index} session {s}")

        self.drv.run_step(st, attention=True, on_attention=on_attention, on_evict=on_evict,
                          on_append=on_append, per_layer=per_layer)
        return st

    def decode_call(self, sessions, layers, token_type=2) -> None:
        """An extra decode call outside the script: one token of `token_type` (default
        TRANSCRIPT) for each listed session, appended on both sides; every output of the
        listed layers compared."""
        c = self.drv._make_call("decode", list(sessions),
                                [np.array([token_type], np.uint8)] * len(sessions), True)
        layers = set(layers)
        self.drv.run_call(c, on_append=self.on_append,
                          on_attention=lambda cc, layer: layer in layers and self.compare_call(
                              cc, layer, None, f"extra call of {len(sessions)}"))

    def release(self, sessions) -> None:
        """kvc_release on both sides, then every released session's state compared."""
        self.drv.release(sessions)
        self.orc.release(list(sessions))
        for s in sessions:
            compare_state(self.drv.cache.export_state(s), self.orc.state(s), f"released {s}")
