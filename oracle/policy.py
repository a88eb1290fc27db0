"""Online KV eviction policy of Sec. 3.3 ("Online KV Eviction"), executed literally.

The paper's rule, restated:

* After each duplex unit, count the resident KV positions, system prefix and
  text included, and compare that count with the budget B.
* While the count exceeds B, evict the acoustic and structural states of the
  oldest unit outside the W most recent units (the retention window).
* Stop when the count fits in B or when no eligible unit remains.
* Evicted: unit marker, audio tokens, native decision, ASR delimiters and
  terminators.  Kept: transcript tokens, response text, the system prefix.
* Position ids advance with every fed token whatever is evicted, so kept keys
  keep their original rotary positions.

Readings where the text leaves a choice:

1. Granularity: a unit's evictable positions go together, in one step.
2. Window: the W most recent units include the unit just finished, so unit u
   is eligible when ``0 <= u <= unit_cur - W``; W = 0 makes every unit eligible.
3. ASR delimiters are evictable with their unit.
4. Unit marker, audio tokens and decision are tagged ACOUSTIC.
5. Positions fed before the first unit marker (system prefix) have unit -1 and
   are never eligible, whatever their type.
6. Eviction runs only when the caller asks, after a whole unit.
7. When no eligible unit remains the resident count may stay above B.

Two variants run on the same state, for comparison with the rule above:

* ``position``: the position-granular reading of the rule (reading 1 taken the
  other way): evict single evictable positions, oldest first, among the units
  outside the window, until the count fits in B or none is left.
* ``sink_recent``: the StreamingLLM baseline of Table 1 (attention-sink tokens
  plus a window of recent positions, type-blind): after each unit, every
  position p with ``sink <= p < pos_next - recent`` is evicted.  B plays no part.

Each evict call also sets ``frontier``: every position below it has been
decided (kept or evicted) by this call or an earlier one, which is what the
page layout consumes.
"""
from __future__ import annotations

from synth.script import ACOUSTIC, ASR_DELIM, UNIT_BEGIN

EVICTABLE_TYPES = frozenset({ACOUSTIC, ASR_DELIM})
TYPE_MASK = 0x7F
POLICIES = ("unit", "position", "sink_recent")


class SessionPolicy:
    """Per-session state of the policy: one record per fed position."""

    def __init__(self, budget: int, window: int, policy: str = "unit", sink: int = 0,
                 recent: int = 0):
        assert policy in POLICIES
        self.budget = budget          # < 0: unbounded
        self.window = window
        self.policy = policy
        self.sink = sink              # sink_recent only
        self.recent = recent          # sink_recent only
        self.frontier = None          # set by evict(); None: nothing decided by that call
        self._pos_scan = 0            # position variant: no evictable position below this
        self.type: list[int] = []     # low 7 bits of the fed tag
        self.unit: list[int] = []     # -1 before the first unit marker
        self.evicted: list[bool] = []
        self.unit_cur = -1
        self.unit_positions: dict[int, list[int]] = {}
        self._oldest_candidate = 0    # every unit below this has nothing left to evict
        self.peak_resident = 0

    # -- feeding -----------------------------------------------------------
    @property
    def pos_next(self) -> int:
        return len(self.type)

    def append(self, tags) -> list[int]:
        """Feed tokens; returns their position ids (pos_next, pos_next+1, ...)."""
        out = []
        for tag in tags:
            tag = int(tag)
            if tag & UNIT_BEGIN:
                self.unit_cur += 1
            p = len(self.type)
            self.type.append(tag & TYPE_MASK)
            self.unit.append(self.unit_cur)
            self.evicted.append(False)
            self.unit_positions.setdefault(self.unit_cur, []).append(p)
            out.append(p)
        self.peak_resident = max(self.peak_resident, self.resident())
        return out

    # -- the rule ------------------------------------------------------------
    def resident(self) -> int:
        return self.evicted.count(False)

    def is_evictable(self, p: int) -> bool:
        return self.unit[p] >= 0 and self.type[p] in EVICTABLE_TYPES

    def unit_has_evictable(self, u: int) -> bool:
        return any(self.is_evictable(p) and not self.evicted[p]
                   for p in self.unit_positions.get(u, ()))

    def oldest_eligible_unit(self):
        """Smallest u with 0 <= u <= unit_cur - W holding an evictable, resident position."""
        last = self.unit_cur - self.window
        u = self._oldest_candidate
        while u <= last:
            if self.unit_has_evictable(u):
                return u
            u += 1
        return None

    def evict(self) -> list[int]:
        """Run the eviction loop once (after a unit).  Returns the evicted units in order
        (unit rule) or the evicted positions in order (the two variants)."""
        if self.policy == "position":
            return self._evict_positions()
        if self.policy == "sink_recent":
            return self._evict_sink_recent()
        self.frontier = None
        evicted_units = []
        r = self.resident()
        while True:
            if self.budget < 0 or r <= self.budget:
                break
            u = self.oldest_eligible_unit()
            if u is None:
                break
            for p in self.unit_positions[u]:
                if self.is_evictable(p) and not self.evicted[p]:
                    self.evicted[p] = True
                    r -= 1
            evicted_units.append(u)
            # Units below u now hold nothing evictable (u was the oldest such
            # unit), and no position can join them later; the current unit can
            # still grow, so the scan never starts past it.
            self._oldest_candidate = min(u + 1, self.unit_cur)
        if evicted_units:
            u_star = evicted_units[-1]
            self.frontier = next((p for p in range(self.pos_next) if self.unit[p] > u_star),
                                 self.pos_next)
        return evicted_units

    def _evict_positions(self) -> list[int]:
        """Position-granular variant: the R - B oldest evictable resident positions of
        units 0 .. unit_cur - W (fewer if fewer exist)."""
        self.frontier = None
        need = self.resident() - self.budget
        if self.budget < 0 or need <= 0:
            return []
        last = self.unit_cur - self.window
        victims = []
        for p in range(self._pos_scan, self.pos_next):
            if len(victims) == need or self.unit[p] > last:
                break
            if self.is_evictable(p) and not self.evicted[p]:
                victims.append(p)
        for p in victims:
            self.evicted[p] = True
        if victims:
            # Every evictable position below the last victim is evicted now (victims
            # are the oldest, and eligible units form a prefix), so later scans start
            # past it.
            self.frontier = victims[-1] + 1
            self._pos_scan = self.frontier
        return victims

    def _evict_sink_recent(self) -> list[int]:
        """Sink + recent variant: evict every position in [sink, pos_next - recent)."""
        hi = self.pos_next - self.recent
        victims = [p for p in range(self.sink, hi) if not self.evicted[p]]
        for p in victims:
            self.evicted[p] = True
        self.frontier = max(hi, 0)
        return victims

    # -- views -----------------------------------------------------------------
    def retained_positions(self) -> list[int]:
        return [p for p, e in enumerate(self.evicted) if not e]

    def evicted_mask(self) -> list[bool]:
        return list(self.evicted)
