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
                "live_pages", "resident", "n_evicted", "pos", "type", "unit"):
        assert gpu_state[key] == ref_state[key], f"{what}: {key} differs"


class Lockstep:
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

    def kv_source(self, s, layer, positions):
        w = self.w
        k = V.layer_tensor(w.seed, V.TAG_K, s, layer, positions, w.kv_heads, w.head_dim,
                           w.dtype, w.kv_scale)
        v = V.layer_tensor(w.seed, V.TAG_V, s, layer, positions, w.kv_heads, w.head_dim,
                           w.dtype, w.kv_scale)
        return k, v

    def q_raw(self, s, layer, positions):
        w = self.w
        return V.layer_tensor(w.seed, V.TAG_Q, s, layer, positions, w.q_heads, w.head_dim,
                              w.dtype, w.q_scale)

    def run_step(self, attn_pred=None, session_pred=None, check_state=True,
                 state_sessions=None, per_layer=False):
        """One duplex step on both sides.

        attn_pred(step, call_kind, call_index, layer) -> bool selects attention calls to
        compare; session_pred(session) -> bool selects the sessions compared in them.
        """
        st = self.drv.prepare_step()
        call_idx = {}

        def on_append(c):
            self.orc.append_chunk(c.sessions.tolist(),
                                  [c.types_host[c.cu[i]:c.cu[i + 1]]
                                   for i in range(len(c.sessions))])
            call_idx[id(c)] = len(call_idx)

        def on_attention(c, layer):
            if attn_pred is None or not attn_pred(st.index, c.kind, call_idx[id(c)], layer):
                return
            out = c.out.float().cpu().numpy()
            chosen = [i for i, s in enumerate(c.sessions.tolist())
                      if session_pred is None or session_pred(s)]
            if not chosen:
                return
            sess = [int(c.sessions[i]) for i in chosen]
            qs = [self.q_raw(s, layer, c.positions[i]) for i, s in zip(chosen, sess)]
            refs = self.orc.attend(layer, qs, self.kv_source, sessions=sess)
            for i, ref in zip(chosen, refs):
                got = out[c.cu[i]:c.cu[i + 1]]
                self.stats.append(assert_close(
                    got, ref, self.w.dtype,
                    f"step {st.index} {c.kind} layer {layer} session {int(c.sessions[i])}",
                    self.tol))
                self.n_compared += 1

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
