"""The oracle behind calls that mirror the library's: append, evict, attend.

State per session: the policy record (``policy.SessionPolicy``) and the page
layout (``layout.SessionLayout``).  K/V values are not stored: a ``kv_source``
callable returns the raw (already dtype-rounded) input K and V of any
positions, and the oracle applies RoPE (``rope``) and the storage rounding
(``numerics``) itself before the float64 attention (``attention``).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from .attention import gqa_attention
from .layout import PagePool, SessionLayout
from .numerics import round_storage
from .policy import SessionPolicy
from .rope import rope
from synth.script import TRANSCRIPT


@dataclass
class OracleConfig:
    n_sessions: int
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    page_size: int
    budget: int
    window: int
    dtype: str
    rope_base: float
    n_pages: int
    policy: str = "unit"
    sink: int = 0
    recent: int = 0


class OracleCache:
    def __init__(self, cfg: OracleConfig):
        self.cfg = cfg
        self.policy = [SessionPolicy(cfg.budget, cfg.window, cfg.policy, cfg.sink, cfg.recent)
                       for _ in range(cfg.n_sessions)]
        self.layout = [SessionLayout(cfg.page_size) for _ in range(cfg.n_sessions)]
        self.pool = PagePool(cfg.n_pages)
        self.last_append: list[tuple[int, list[int]]] | None = None

    # -- library mirror ---------------------------------------------------------
    def append_chunk(self, sessions, types_per_session) -> None:
        done = []
        for s, types in zip(sessions, types_per_session):
            positions = self.policy[s].append(types)
            self.layout[s].append(positions, self.pool)
            done.append((s, positions))
        self.last_append = done

    def evict(self, sessions) -> list[int]:
        plans = []
        for s in sessions:
            pol, lay = self.policy[s], self.layout[s]
            pol.evict()
            # The live slots whose positions this evict decided form a prefix of the
            # live region: the survivors among them move to the compacted region.
            if pol.frontier is not None:
                end = sum(1 for p in lay.live_pos if p < pol.frontier)
                survivors = [p for p in lay.live_pos[:end] if not pol.evicted[p]]
            else:
                end, survivors = 0, []
            plans.append((s, end, survivors))
        for s, end, survivors in plans:
            self.layout[s].move_survivors(end, survivors, self.pool)
        for s, end, _ in plans:
            self.layout[s].consume_live(end, self.pool)
        self.last_append = None
        for s in sessions:
            assert self.layout[s].retained_positions() == self.policy[s].retained_positions()
        return [self.policy[s].resident() for s in sessions]

    def release(self, sessions) -> None:
        """End sessions: free every page, start over at position 0."""
        for s in sessions:
            for pid in self.layout[s].hist_pages + self.layout[s].live_pages:
                self.pool.release(pid)
            self.policy[s] = SessionPolicy(self.cfg.budget, self.cfg.window, self.cfg.policy,
                                           self.cfg.sink, self.cfg.recent)
            self.layout[s] = SessionLayout(self.cfg.page_size)
        self.last_append = None

    def transcript_positions(self, s: int) -> list[int]:
        """Retained TRANSCRIPT positions in retained order (what query-time re-encoding
        reads after the streaming cache is discarded, Sec. 4.2)."""
        pol = self.policy[s]
        return [p for p in pol.retained_positions() if pol.type[p] == TRANSCRIPT]

    def resident_size(self, s: int) -> int:
        return self.policy[s].resident()

    def state(self, s: int) -> dict:
        """The bit-exact comparison set of one session."""
        pol, lay = self.policy[s], self.layout[s]
        pos = lay.retained_positions()
        return {
            "pos_next": pol.pos_next,
            "unit_cur": pol.unit_cur,
            "n_hist": lay.n_hist,
            "live_head": lay.live_head,
            "n_live": lay.n_live,
            "hist_pages": list(lay.hist_pages),
            "live_pages": list(lay.live_pages),
            "resident": pol.resident(),
            "n_evicted": pol.pos_next - pol.resident(),
            "peak_resident": pol.peak_resident,
            "pos": pos,
            "type": [pol.type[p] for p in pos],
            "unit": [pol.unit[p] for p in pos],
        }

    # -- attention ----------------------------------------------------------------
    def stored_keys(self, s: int, layer: int, positions, kv_source):
        k_raw, v = kv_source(s, layer, positions)
        k = round_storage(rope(k_raw, np.asarray(positions)[:, None], self.cfg.rope_base),
                          self.cfg.dtype)
        return k, np.asarray(v, dtype=np.float64)

    def attend(self, layer: int, q_per_session, kv_source, sessions=None):
        """Attention for the queries of the last appended chunk.

        ``q_per_session[i]`` is ``[T_i][Hq][D]`` raw query input of the i-th session of
        the last append (or of ``sessions``, a subset of it).  Returns float64 outputs.
        """
        assert self.last_append is not None, "attention needs a preceding append"
        chosen = self.last_append if sessions is None else [
            a for a in self.last_append if a[0] in set(sessions)]
        outs = []
        for (s, q_pos), q in zip(chosen, q_per_session):
            keys = self.layout[s].retained_positions()
            k, v = self.stored_keys(s, layer, keys, kv_source)
            q_rot = rope(q, np.asarray(q_pos)[:, None], self.cfg.rope_base)
            outs.append(gqa_attention(q_rot, k, v, q_pos, keys))
        return outs
