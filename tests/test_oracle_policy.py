"""Pins for the oracle's eviction policy and page layout (Sec. 3.3, "Online KV Eviction").

Each pin comes from outside the oracle: hand-worked examples, an exhaustive
enumeration of eviction sets that satisfy the wording of the rule, and the
invariants the rule implies.
"""
import itertools
import json
import os

import numpy as np
import pytest

from oracle.cache import OracleCache, OracleConfig
from oracle.policy import SessionPolicy
from synth.script import ACOUSTIC, ASR_DELIM, TEXT, TRANSCRIPT, UNIT_BEGIN

EVICTABLE = {ACOUSTIC, ASR_DELIM}


def _cache(budget, window, ps=4, n_pages=64, n_sessions=1):
    return OracleCache(OracleConfig(n_sessions=n_sessions, layers=1, q_heads=1, kv_heads=1,
                                    head_dim=4, page_size=ps, budget=budget, window=window,
                                    dtype="f32", rope_base=10000.0, n_pages=n_pages))


# -- hand-worked examples ----------------------------------------------------------------

def _golden(golden_dir):
    with open(os.path.join(golden_dir, "eviction_examples.json")) as f:
        return json.load(f)["examples"]


def test_hand_worked_examples(golden_dir):
    for ex in _golden(golden_dir):
        c = _cache(ex["budget"], ex["window"], ex["page_size"], ex["n_pages"])
        if ex.get("prefix"):
            c.append_chunk([0], [ex["prefix"]])
        got = []
        at_end = ex.get("evict_only_at_end", False)
        for i, unit in enumerate(ex["units"]):
            c.append_chunk([0], [unit])
            if not at_end or i == len(ex["units"]) - 1:
                before = set(c.policy[0].retained_positions())
                res = c.evict([0])[0]
                after = set(c.policy[0].retained_positions())
                units = sorted({c.policy[0].unit[p] for p in before - after})
                got.append({"resident": res, "evicted_units": units})
        assert got == ex["after_each_evict"], ex["name"]
        st = c.state(0)
        fin = ex["final"]
        assert st["pos"] == fin["retained"], ex["name"]
        for key in ("hist_pages", "n_hist", "live_pages", "live_head", "n_live"):
            assert st[key] == fin[key], (ex["name"], key)
        assert sorted(c.pool._free) == fin["free_pages"], ex["name"]


# -- brute force over every eviction set --------------------------------------------------

def _brute_force_evicted_units(types, units, evicted, unit_cur, budget, window):
    """Enumerate all sets of units; keep those that satisfy the rule's wording.

    A set S of units is the rule's outcome when
      (a) each member is eligible: 0 <= u <= unit_cur - W and holds a resident
          evictable position;
      (b) it is oldest-first: an eligible unit older than a member is a member;
      (c) it stops correctly: after removing S, the count fits in B or no
          eligible unit is left;
      (d) it does not overshoot: before its newest member is removed, the count
          still exceeded B.
    """
    n = len(types)

    def resident_after(s):
        return sum(1 for p in range(n) if not evicted[p]
                   and not (units[p] in s and types[p] in EVICTABLE and units[p] >= 0))

    eligible = sorted({units[p] for p in range(n) if not evicted[p] and units[p] >= 0
                       and units[p] <= unit_cur - window and types[p] in EVICTABLE})
    answers = []
    for r in range(len(eligible) + 1):
        for combo in itertools.combinations(eligible, r):
            s = set(combo)
            if any(u not in s and u < max(s, default=-10) for u in eligible):
                continue
            after = resident_after(s)
            left = [u for u in eligible if u not in s]
            if budget >= 0 and not (after <= budget or not left):
                continue
            if budget < 0 and s:
                continue
            if s:
                prev = s - {max(s)}
                if not resident_after(prev) > budget:
                    continue
            answers.append(s)
    return answers


def _random_script(rng, n_units, max_len):
    tags = []
    for _ in range(n_units):
        k = int(rng.integers(1, max_len + 1))
        body = [int(rng.choice([ACOUSTIC, ASR_DELIM, TRANSCRIPT, TEXT])) for _ in range(k)]
        body[0] |= UNIT_BEGIN
        tags.append(body)
    return tags


@pytest.mark.parametrize("seed", range(300))
def test_brute_force_unique_choice(seed):
    rng = np.random.default_rng(seed)
    n_units = int(rng.integers(1, 5))
    prefix = [int(rng.choice([ACOUSTIC, TEXT])) for _ in range(int(rng.integers(0, 3)))]
    script = _random_script(rng, n_units, 6)
    budget = int(rng.integers(-1, 12))
    window = int(rng.integers(0, 4))
    pol = SessionPolicy(budget, window)
    pol.append(prefix)
    evict_points = set(rng.choice(n_units, size=int(rng.integers(1, n_units + 1)),
                                  replace=False).tolist()) | {n_units - 1}
    for i, unit in enumerate(script):
        pol.append(unit)
        if i not in evict_points:
            continue
        before = list(pol.evicted)
        answers = _brute_force_evicted_units(pol.type, pol.unit, before, pol.unit_cur,
                                             budget, window)
        assert len(answers) == 1, answers
        got = pol.evict()
        assert set(got) == answers[0]
        assert got == sorted(got)


# -- invariants of the rule ------------------------------------------------------------------

def _run_random_session(seed, budget, window, n_units=40, evict_every=1):
    rng = np.random.default_rng(seed)
    pol = SessionPolicy(budget, window)
    pol.append([TEXT] * int(rng.integers(0, 5)))
    history = []
    for u in range(n_units):
        unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 20))
        if rng.random() < 0.8:
            unit += [ASR_DELIM] + [TRANSCRIPT] * int(rng.poisson(3)) + [ASR_DELIM]
        if rng.random() < 0.1:
            unit += [TEXT] * int(rng.integers(1, 40))
        pol.append(unit)
        if u % evict_every == 0:
            r_before = pol.resident()
            was = list(pol.evicted)
            evicted_units = pol.evict()
            history.append((u, r_before, evicted_units, was))
    return pol, history


@pytest.mark.parametrize("budget,window", [(-1, 5), (0, 0), (0, 3), (50, 2), (100, 5),
                                           (200, 10), (30, 0), (400, 1)])
def test_policy_invariants(budget, window):
    for seed in range(8):
        pol, history = _run_random_session(seed, budget, window)
        n = pol.pos_next
        for p in range(n):
            if pol.evicted[p]:
                # (ii) only evictable positions of units >= 0 ever go
                assert pol.unit[p] >= 0 and pol.type[p] in EVICTABLE
        # (ii) transcripts, text and the prefix stay
        for p in range(n):
            if pol.type[p] in (TRANSCRIPT, TEXT) or pol.unit[p] < 0:
                assert not pol.evicted[p]
        # (ii) every position of the W most recent units stays
        for p in range(n):
            if pol.unit[p] > pol.unit_cur - window:
                assert not pol.evicted[p]
        # (i) after the last evict: fits, or nothing eligible remains
        r = pol.resident()
        if budget >= 0 and r > budget:
            assert pol.oldest_eligible_unit() is None
        # (iii) evicted units form a prefix of the units in age order
        gone = sorted({pol.unit[p] for p in range(n) if pol.evicted[p]})
        assert gone == list(range(len(gone)))
        # (v) unbounded evicts nothing
        if budget < 0:
            assert not any(pol.evicted)
        for _, r_before, evicted_units, _ in history:
            assert evicted_units == sorted(evicted_units)


def test_floor_budget_evicts_every_eligible_unit():
    """B = 0 (Table 3's floor) leaves only protected positions and the window."""
    for window in (0, 1, 5):
        pol, _ = _run_random_session(3, 0, window)
        for p in range(pol.pos_next):
            eligible = 0 <= pol.unit[p] <= pol.unit_cur - window
            assert pol.evicted[p] == (eligible and pol.type[p] in EVICTABLE)


def test_budget_shape_like_table3():
    """End <= B and Peak <= B + one unit's growth, on 17+segment units (Table 3 shape)."""
    rng = np.random.default_rng(0)
    # Unit counts chosen so that transcripts plus the window stay below B, as in
    # the paper's sessions (End < B there); beyond that the stop rule applies.
    for budget, n_units in ((512, 100), (1024, 250), (2048, 400)):
        pol = SessionPolicy(budget, 5)
        peak, max_growth = 0, 0
        for u in range(n_units):
            unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * 16 + [ASR_DELIM] + \
                [TRANSCRIPT] * int(rng.poisson(3)) + [ASR_DELIM]
            max_growth = max(max_growth, len(unit))
            pol.append(unit)
            peak = max(peak, pol.resident())
            pol.evict()
            assert pol.resident() <= budget
        assert budget < peak <= budget + max_growth


def test_mid_unit_evict_with_zero_window_keeps_scanning_current_unit():
    """W = 0 lets the current unit go; tokens fed later to the same unit stay eligible."""
    pol = SessionPolicy(0, 0)
    pol.append([ACOUSTIC | UNIT_BEGIN, ACOUSTIC])
    assert pol.evict() == [0]
    pol.append([ACOUSTIC, TRANSCRIPT])
    assert pol.evict() == [0]
    assert pol.retained_positions() == [3]


# -- layout contract -----------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_layout_invariants_many_sessions(seed):
    rng = np.random.default_rng(seed)
    n_sessions, ps = 5, 4
    c = _cache(int(rng.integers(5, 60)), int(rng.integers(0, 4)), ps=ps, n_pages=4000,
               n_sessions=n_sessions)
    total = c.pool.n_pages
    for step in range(60):
        active = sorted(rng.choice(n_sessions, size=int(rng.integers(1, n_sessions + 1)),
                                   replace=False).tolist())
        chunks = []
        for s in active:
            unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 9))
            unit += [ASR_DELIM] + [TRANSCRIPT] * int(rng.poisson(2)) + [ASR_DELIM]
            chunks.append(unit)
        c.append_chunk(active, chunks)
        c.evict(active)
        seen = set()
        used = 0
        for s in range(n_sessions):
            st = c.state(s)
            lay = c.layout[s]
            # retained logical order is ascending position
            assert st["pos"] == sorted(st["pos"])
            # pages are exactly as many as the regions need
            assert len(lay.hist_pages) == -(-lay.n_hist // ps)
            assert len(lay.live_pages) == -(-(lay.live_head + lay.n_live) // ps)
            assert 0 <= lay.live_head < ps
            # no page appears twice, within or across sessions
            for pid in lay.hist_pages + lay.live_pages:
                assert pid not in seen
                seen.add(pid)
            used += len(lay.hist_pages) + len(lay.live_pages)
            # every retained position has a distinct (page, slot)
            slots = {lay.slot_of_logical(i) for i in range(len(st["pos"]))}
            assert len(slots) == len(st["pos"])
        assert used + c.pool.free_count() == total


# -- policy variants -------------------------------------------------------------------------

def _brute_force_position_victims(pol, budget, window):
    """Every set S of resident evictable positions of units 0..unit_cur-W that is
    oldest-first, brings the count within B (or takes them all) and removes no more
    than needed; the variant's choice must be the unique such set."""
    n = pol.pos_next
    last = pol.unit_cur - window
    elig = [p for p in range(n) if not pol.evicted[p] and pol.unit[p] >= 0
            and pol.unit[p] <= last and pol.type[p] in EVICTABLE]
    r = sum(1 for p in range(n) if not pol.evicted[p])
    answers = []
    for k in range(len(elig) + 1):
        for combo in itertools.combinations(elig, k):
            s = set(combo)
            if any(q not in s and q < max(s, default=-1) for q in elig):
                continue  # not oldest-first
            fits = budget < 0 or r - len(s) <= budget
            if budget >= 0 and not (fits or len(s) == len(elig)):
                continue
            if budget < 0 and s:
                continue
            if s and budget >= 0 and r - (len(s) - 1) <= budget:
                continue  # one fewer would have been enough
            answers.append(s)
    return answers


@pytest.mark.parametrize("seed", range(200))
def test_position_variant_brute_force(seed):
    rng = np.random.default_rng(1000 + seed)
    n_units = int(rng.integers(1, 5))
    budget = int(rng.integers(-1, 12))
    window = int(rng.integers(0, 4))
    pol = SessionPolicy(budget, window, policy="position")
    pol.append([int(rng.choice([ACOUSTIC, TEXT])) for _ in range(int(rng.integers(0, 3)))])
    for unit in _random_script(rng, n_units, 6):
        pol.append(unit)
        answers = _brute_force_position_victims(pol, budget, window)
        assert len(answers) == 1, answers
        got = pol.evict()
        assert set(got) == answers[0] and got == sorted(got)
        if got:
            assert pol.frontier == got[-1] + 1


@pytest.mark.parametrize("budget,window", [(0, 0), (0, 3), (50, 2), (200, 10), (30, 0)])
def test_position_variant_invariants(budget, window):
    for seed in range(6):
        rng = np.random.default_rng(seed)
        pol = SessionPolicy(budget, window, policy="position")
        pol.append([TEXT] * int(rng.integers(0, 5)))
        for u in range(40):
            unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 20))
            if rng.random() < 0.8:
                unit += [ASR_DELIM] + [TRANSCRIPT] * int(rng.poisson(3)) + [ASR_DELIM]
            pol.append(unit)
            got = pol.evict()
            last = pol.unit_cur - window
            left = [p for p in range(pol.pos_next) if not pol.evicted[p] and pol.unit[p] >= 0
                    and pol.unit[p] <= last and pol.type[p] in EVICTABLE]
            # (i) fits in B, or nothing eligible is left
            if pol.resident() > budget:
                assert not left
            # (ii) an evict that removes anything lands exactly on B unless it ran out
            if got:
                assert pol.resident() == budget or not left
            # (iii) only evictable positions of units >= 0 ever go
            for p in range(pol.pos_next):
                if pol.evicted[p]:
                    assert pol.unit[p] >= 0 and pol.type[p] in EVICTABLE
            # (iv) oldest first: no resident eligible evictable position is older than
            # an evicted one
            gone = [p for p in range(pol.pos_next) if pol.evicted[p]]
            if gone:
                assert not any(p < gone[-1] for p in left)


def test_position_variant_is_finer_than_unit_rule():
    """Same script, same B and W: the variant keeps at least as many positions after
    every evict and lands exactly on B whenever it evicts."""
    rng = np.random.default_rng(5)
    a = SessionPolicy(300, 3)
    b = SessionPolicy(300, 3, policy="position")
    for u in range(60):
        unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * 16 + [ASR_DELIM] + \
            [TRANSCRIPT] * int(rng.poisson(3)) + [ASR_DELIM]
        a.append(unit)
        b.append(unit)
        a.evict()
        got = b.evict()
        assert b.resident() >= a.resident()
        if got:
            assert b.resident() == 300


@pytest.mark.parametrize("sink,recent", [(0, 0), (4, 0), (0, 16), (4, 16), (4, 2000), (40, 7)])
def test_sink_recent_variant_closed_form(sink, recent):
    rng = np.random.default_rng(sink * 31 + recent)
    pol = SessionPolicy(-1, 0, policy="sink_recent", sink=sink, recent=recent)
    pol.append([TEXT] * 3)
    for u in range(50):
        unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 20)) + \
            [ASR_DELIM] + [TRANSCRIPT] * int(rng.poisson(3)) + [ASR_DELIM]
        pol.append(unit)
        pol.evict()
        n = pol.pos_next
        want = [p for p in range(n) if p < sink or p >= n - recent]
        assert pol.retained_positions() == want
        assert pol.frontier == max(n - recent, 0)


@pytest.mark.parametrize("policy", ["position", "sink_recent"])
@pytest.mark.parametrize("seed", range(4))
def test_layout_invariants_policy_variants(policy, seed):
    rng = np.random.default_rng(seed)
    n_sessions, ps = 4, 4
    c = OracleCache(OracleConfig(n_sessions=n_sessions, layers=1, q_heads=1, kv_heads=1,
                                 head_dim=4, page_size=ps, budget=int(rng.integers(5, 60)),
                                 window=int(rng.integers(0, 4)), dtype="f32",
                                 rope_base=10000.0, n_pages=4000, policy=policy, sink=3,
                                 recent=int(rng.integers(0, 30))))
    total = c.pool.n_pages
    for step in range(50):
        active = sorted(rng.choice(n_sessions, size=int(rng.integers(1, n_sessions + 1)),
                                   replace=False).tolist())
        chunks = []
        for s in active:
            unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 9))
            unit += [ASR_DELIM] + [TRANSCRIPT] * int(rng.poisson(2)) + [ASR_DELIM]
            chunks.append(unit)
        c.append_chunk(active, chunks)
        c.evict(active)
        used, seen = 0, set()
        for s in range(n_sessions):
            st, lay = c.state(s), c.layout[s]
            assert st["pos"] == sorted(st["pos"])
            assert len(lay.hist_pages) == -(-lay.n_hist // ps)
            assert len(lay.live_pages) == -(-(lay.live_head + lay.n_live) // ps)
            for pid in lay.hist_pages + lay.live_pages:
                assert pid not in seen
                seen.add(pid)
            used += len(lay.hist_pages) + len(lay.live_pages)
        assert used + c.pool.free_count() == total


@pytest.mark.parametrize("policy", ["unit", "position"])
def test_transcript_export_keeps_every_transcript(policy):
    """Transcripts are never evicted by the rule (or its position-granular reading), so the
    transcript record after any number of evicts is every TRANSCRIPT position fed."""
    rng = np.random.default_rng(11)
    c = _cache(40, 1, n_sessions=2)
    c.policy = [SessionPolicy(40, 1, policy=policy) for _ in range(2)]
    fed = {0: [], 1: []}
    for _ in range(30):
        chunks = []
        for s in (0, 1):
            unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 9)) + [ASR_DELIM] + \
                [TRANSCRIPT] * int(rng.poisson(2)) + [ASR_DELIM] + [TEXT] * int(rng.integers(0, 3))
            base = c.policy[s].pos_next
            fed[s] += [base + i for i, t in enumerate(unit) if t == TRANSCRIPT]
            chunks.append(unit)
        c.append_chunk([0, 1], chunks)
        c.evict([0, 1])
    for s in (0, 1):
        assert c.transcript_positions(s) == fed[s]
        assert any(c.policy[s].evicted)


# -- release -------------------------------------------------------------------------------

def _unit_chunk(rng, text=False):
    unit = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * int(rng.integers(0, 9)) + [ASR_DELIM] + \
        [TRANSCRIPT] * int(rng.poisson(2)) + [ASR_DELIM]
    return unit + ([TEXT] * int(rng.integers(1, 6)) if text else [])


@pytest.mark.parametrize("policy,sink,recent", [("unit", 0, 0), ("position", 0, 0),
                                                ("sink_recent", 3, 25)])
def test_release_then_refeed_equals_a_fresh_session(policy, sink, recent):
    """A released session starts over under the cache's own policy: fed the same units
    afterwards it evicts exactly what a fresh session fed those units evicts (policy
    record, peak, frontier), its page lists have the same shape, and every page it held
    went back to the pool.  A release that rebuilt the session under the default rule
    would diverge from the fresh position-granular or sink + recent session at its first
    evict past the budget."""
    budget, window, ps = 20, 1, 4

    def cache(n_sessions):
        return OracleCache(OracleConfig(n_sessions=n_sessions, layers=1, q_heads=1, kv_heads=1,
                                        head_dim=4, page_size=ps, budget=budget, window=window,
                                        dtype="f32", rope_base=10000.0, n_pages=400,
                                        policy=policy, sink=sink, recent=recent))

    rng = np.random.default_rng(5)
    before = [_unit_chunk(rng, text=(i % 7 == 3)) for i in range(25)]
    after = [_unit_chunk(rng, text=(i % 5 == 2)) for i in range(30)]
    other = [_unit_chunk(rng) for _ in range(25)]
    used = cache(2)
    for a, b in zip(before, other):
        used.append_chunk([0, 1], [a, b])
        used.evict([0, 1])
    assert any(used.policy[0].evicted)
    free_before = used.pool.free_count()
    held = len(used.layout[0].hist_pages) + len(used.layout[0].live_pages)
    used.release([0])
    assert used.pool.free_count() == free_before + held
    assert used.state(0)["pos_next"] == 0 and used.state(0)["peak_resident"] == 0
    fresh = cache(1)
    for a in after:
        used.append_chunk([0], [a])
        fresh.append_chunk([0], [a])
        assert used.evict([0]) == fresh.evict([0])
        pu, pf = used.policy[0], fresh.policy[0]
        assert (pu.policy, pu.sink, pu.recent) == (policy, sink, recent)
        assert pu.evicted == pf.evicted and pu.frontier == pf.frontier
        su, sf = used.state(0), fresh.state(0)
        for key in ("pos_next", "unit_cur", "n_hist", "live_head", "n_live", "resident",
                    "n_evicted", "peak_resident", "pos", "type", "unit"):
            assert su[key] == sf[key], key
        assert len(su["hist_pages"]) == len(sf["hist_pages"])
        assert len(su["live_pages"]) == len(sf["live_pages"])
    assert any(fresh.policy[0].evicted)


def test_release_of_the_only_session_restores_the_page_ids():
    """With one session, a release frees the whole pool, so the lowest-free-id allocator
    hands out the same page ids as in a fresh cache."""
    rng = np.random.default_rng(9)
    units = [_unit_chunk(rng, text=(i % 6 == 0)) for i in range(20)]
    a, b = _cache(15, 2), _cache(15, 2)
    for u in units[:12]:
        a.append_chunk([0], [u])
        a.evict([0])
    a.release([0])
    assert a.pool.free_count() == a.pool.n_pages
    for u in units:
        a.append_chunk([0], [u])
        b.append_chunk([0], [u])
        a.evict([0])
        b.evict([0])
        assert a.state(0) == b.state(0)
