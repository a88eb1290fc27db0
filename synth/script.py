"""Seeded synthetic session scripts shaped like the paper's duplex streams.

A duplex unit is one second of speech (Sec. 3.1): a unit marker, about ten
audio tokens and the native decision, which the workloads bundle as 17
ACOUSTIC positions (the paper's "17 for the acoustic history", Sec. 1).  After
the first decision comes the transcription segment: an ASR delimiter, the
transcript tokens, a closing delimiter (Sec. 3.1).  In speaking units the
response text follows the segment.  The 17 acoustic positions are one
chunked-prefill call; every later token is one single-token decode.

Scripts are plain data (token counts per unit) drawn from numpy's PCG64 with a
recorded seed, so the oracle and the GPU driver consume the identical script.
Nothing here evaluates the eviction policy or attention.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

# Token type tags (low 7 bits) and the unit-start flag.  The numbering is the
# one the C interface fixes; it is restated here so that this module stays
# independent of the library.
ACOUSTIC, ASR_DELIM, TRANSCRIPT, TEXT = 0, 1, 2, 3
UNIT_BEGIN = 0x80

ACOUSTIC_PER_UNIT = 17
SEGMENT_CAP = 64  # at most 64 transcript tokens per segment (Sec. 3.1)


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: model shape, policy parameters and session mix."""
    name: str
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    dtype: str                   # "f32" or "bf16"
    page_size: int
    budget: int                  # < 0: unbounded
    window: int
    n_sessions: int
    units: int                   # units per session when lengths are fixed
    unit_range: tuple | None = None   # (lo, hi) units per session, uniform, when set
    offset_max: int = 0          # session i starts at step U{0..offset_max}
    turns: bool = False          # speaking turns about every 60 units
    turn_len: tuple = (20, 80)
    turn_period: int = 60
    turn_jitter: int = 5
    transcript_mean: float = 3.0
    p_no_segment: float = 0.0
    p_long_segment: float = 0.0
    long_segment: tuple = (10, 30)
    prefix_len: int = 0          # system-prefix tokens before the first unit
    seed: int = 0
    q_scale: float = 1.0
    kv_scale: float = 1.0
    rope_base: float = 10000.0
    policy: str = "unit"         # eviction policy: "unit" (Sec. 3.3), "position", "sink_recent"
    sink: int = 0                # sink_recent: first positions kept
    recent: int = 0              # sink_recent: most recent positions kept

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    @property
    def kv_bytes_per_position(self) -> int:
        """K+V bytes of one position over all layers."""
        esz = 2 if self.dtype == "bf16" else 4
        return self.layers * self.kv_heads * self.head_dim * 2 * esz

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workloads of the benchmark description.
TINY_F32 = Workload(name="tiny-f32-1x4x1x64-60u-B512-W5", layers=1, q_heads=4, kv_heads=1,
                    head_dim=64, dtype="f32", page_size=16, budget=512, window=5,
                    n_sessions=1, units=60)
SINGLE_BF16 = Workload(name="single-bf16-32L-32q8kv-d128-600u-B4096-W10", layers=32, q_heads=32,
                       kv_heads=8, head_dim=128, dtype="bf16", page_size=16, budget=4096,
                       window=10, n_sessions=1, units=600, turns=True)
SINGLE_BF16_UNBOUNDED = SINGLE_BF16.with_(name="single-bf16-32L-32q8kv-d128-600u-Binf-W10",
                                          budget=-1)
BATCH64_BF16 = SINGLE_BF16.with_(name="batch64-bf16-32L-32q8kv-d128-600u-off300-B4096-W10",
                                 n_sessions=64, offset_max=300)


def stress256(budget: int, window: int) -> Workload:
    return SINGLE_BF16.with_(name=f"stress256-bf16-32L-32q8kv-d128-10to60min-B{budget}-W{window}",
                             n_sessions=256, unit_range=(600, 3600), budget=budget,
                             window=window, p_no_segment=0.05, p_long_segment=0.02)


WORKLOADS = {
    "tiny": TINY_F32,
    "single": SINGLE_BF16,
    "single-unbounded": SINGLE_BF16_UNBOUNDED,
    "batch64": BATCH64_BF16,
}


@dataclass
class SessionScript:
    """Per-unit token counts of one session."""
    session: int
    offset: int                       # first step at which the session is active
    n_transcript: np.ndarray          # per unit; -1 = no segment in this unit
    n_text: np.ndarray                # per unit; response tokens after the segment
    prefix_len: int = 0

    @property
    def n_units(self) -> int:
        return len(self.n_transcript)

    def prefill_types(self) -> np.ndarray:
        t = np.full(ACOUSTIC_PER_UNIT, ACOUSTIC, dtype=np.uint8)
        t[0] |= UNIT_BEGIN
        return t

    def decode_types(self, unit: int) -> np.ndarray:
        """Token types decoded one at a time after the unit's acoustic chunk."""
        n_tr = int(self.n_transcript[unit])
        seg = [] if n_tr < 0 else [ASR_DELIM] + [TRANSCRIPT] * n_tr + [ASR_DELIM]
        return np.array(seg + [TEXT] * int(self.n_text[unit]), dtype=np.uint8)

    def prefix_types(self) -> np.ndarray:
        return np.full(self.prefix_len, TEXT, dtype=np.uint8)

    def unit_types(self, unit: int) -> np.ndarray:
        return np.concatenate([self.prefill_types(), self.decode_types(unit)])

    def all_types(self, n_units: int | None = None) -> np.ndarray:
        n = self.n_units if n_units is None else n_units
        parts = [self.prefix_types()] + [self.unit_types(u) for u in range(n)]
        return np.concatenate(parts).astype(np.uint8)


def session_script(w: Workload, session: int) -> SessionScript:
    rng = np.random.default_rng(np.random.SeedSequence([w.seed, session]))
    n_units = w.units if w.unit_range is None else int(rng.integers(w.unit_range[0],
                                                                    w.unit_range[1] + 1))
    offset = int(rng.integers(0, w.offset_max + 1)) if w.offset_max > 0 else 0
    n_tr = np.minimum(rng.poisson(w.transcript_mean, size=n_units), SEGMENT_CAP).astype(np.int32)
    if w.p_long_segment > 0:
        long = rng.random(n_units) < w.p_long_segment
        lo, hi = w.long_segment
        n_tr = np.where(long, rng.integers(lo, hi + 1, size=n_units), n_tr).astype(np.int32)
    if w.p_no_segment > 0:
        none = rng.random(n_units) < w.p_no_segment
        n_tr = np.where(none, -1, n_tr).astype(np.int32)
    n_text = np.zeros(n_units, dtype=np.int32)
    if w.turns:
        j = 0
        while True:
            u = w.turn_period * j + (w.turn_period - 1) + int(
                rng.integers(-w.turn_jitter, w.turn_jitter + 1))
            if u >= n_units:
                break
            n_text[max(u, 0)] = int(rng.integers(w.turn_len[0], w.turn_len[1] + 1))
            j += 1
    return SessionScript(session=session, offset=offset, n_transcript=n_tr, n_text=n_text,
                         prefix_len=w.prefix_len)


def workload_scripts(w: Workload) -> list[SessionScript]:
    return [session_script(w, s) for s in range(w.n_sessions)]


def schedule(scripts: list[SessionScript]) -> list[list[tuple[int, int]]]:
    """Per step, the (session, unit) pairs that advance: every active session moves one unit."""
    n_steps = max(s.offset + s.n_units for s in scripts)
    out = []
    for step in range(n_steps):
        out.append([(s.session, step - s.offset) for s in scripts
                    if s.offset <= step < s.offset + s.n_units])
    return out


def steady_state_step(w: Workload, scripts: list[SessionScript]) -> int:
    """First step at which every session is active and its unit count would exceed
    the budget's worth of positions (approximate; used only to place a timing window)."""
    per_unit = ACOUSTIC_PER_UNIT + 2 + w.transcript_mean
    ramp = int(np.ceil((w.budget if w.budget >= 0 else 0) / per_unit)) + w.window + 2
    return max(s.offset for s in scripts) + ramp
