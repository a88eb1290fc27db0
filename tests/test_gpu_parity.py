"""GPU parity: the CUDA path against the oracle on the same seeded inputs.

Bit-exact: eviction masks (retained position lists), resident counts, page
tables, live head/size and per-slot {position, type, unit}.  Floating point:
|gpu - ref| <= atol + rtol |ref| elementwise (bf16: 2e-2 + 1e-2 |ref|; fp32:
1e-4 + 1e-4 |ref|) and a normwise bound (bf16 1e-2, fp32 1e-5); the reference is
the float64 oracle on the same rounded inputs.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from harness import Lockstep, assert_close, compare_state  # noqa: E402
from synth import script as S  # noqa: E402
from synth import values as V  # noqa: E402
from synth.driver import Driver, cache_sizing  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_31224_gb300 import build
    from synth import gpu
    build.build()
    gpu.build()


def test_device_generator_matches_numpy():
    from synth import gpu
    for dtype in ("bf16", "f32"):
        sess = torch.tensor([0, 3, 3, 7], dtype=torch.int32, device="cuda")
        pos = torch.tensor([0, 5, 4095, 123456], dtype=torch.int32, device="cuda")
        t = torch.empty((3, 4, 8, 128), dtype=torch.bfloat16 if dtype == "bf16" else torch.float32,
                        device="cuda")
        for tag, scale in ((V.TAG_K, 1.0), (V.TAG_Q, 0.25)):
            gpu.fill(t, dtype, 11, tag, sess, pos, scale)
            got = t.float().cpu().numpy()
            want = V.values(11, tag, sess.cpu().numpy()[None, :, None, None],
                            np.arange(3)[:, None, None, None],
                            pos.cpu().numpy()[None, :, None, None],
                            np.arange(8)[None, None, :, None], np.arange(128)[None, None, None, :],
                            dtype, scale)
            assert np.array_equal(got, want)


def _lockstep(w, n_units=None, sizing=None, tol=None):
    scripts = S.workload_scripts(w)
    if n_units is not None:
        for sc in scripts:
            sc.n_transcript = sc.n_transcript[:n_units]
            sc.n_text = sc.n_text[:n_units]
    drv = Driver(w, scripts, sizing=sizing)
    return Lockstep(drv, w, tol=tol), scripts


def test_tiny_f32_every_call_every_evict():
    """60 units, fp32: every attention output and every post-evict state."""
    ls, scripts = _lockstep(S.TINY_F32)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda *a: True)
    assert ls.n_compared > 60 * 6
    st = ls.drv.cache.export_state(0)
    assert st["resident"] <= 512 and st["n_evicted"] > 0


def test_tiny_f32_prefix_window0_floor_budget():
    w = S.TINY_F32.with_(prefix_len=37, window=0, budget=0, seed=3)
    ls, _ = _lockstep(w, n_units=25)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda *a: True)
    st = ls.drv.cache.export_state(0)
    # floor budget: only prefix + transcripts remain
    assert all(t in (2, 3) or u < 0 for t, u in zip(st["type"], st["unit"]))


@pytest.mark.parametrize("budget,window,seed", [(64, 1, 1), (200, 3, 2), (-1, 5, 4),
                                                (17, 0, 5), (1000, 50, 6)])
def test_small_bf16_mixed_segments(budget, window, seed):
    """bf16, 2 layers, 3 sessions with offsets, empty/long segments and speaking turns."""
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=3, offset_max=4, budget=budget,
                            window=window, seed=seed, p_no_segment=0.1, p_long_segment=0.1,
                            turn_period=12, turn_jitter=2, prefix_len=5)
    ls, _ = _lockstep(w, n_units=40)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda step, kind, i, layer: layer == 1 or step % 5 == 0)
    assert ls.n_compared > 100


@pytest.mark.parametrize("policy,budget,window,sink,recent", [
    ("position", 64, 2, 0, 0), ("position", 0, 0, 0, 0), ("position", 100, 5, 0, 0),
    ("sink_recent", 64, 0, 4, 40), ("sink_recent", 64, 0, 0, 7), ("sink_recent", 64, 0, 37, 0)])
def test_policy_variants_small_bf16(policy, budget, window, sink, recent):
    """The position-granular and sink + recent variants of the eviction step on the
    same kernels: every state bit-exact after every evict, every output compared."""
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=3, budget=budget, window=window, seed=21,
                            turn_period=10, turn_jitter=1, policy=policy, sink=sink,
                            recent=recent)
    ls, _ = _lockstep(w, n_units=40)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda *a: True)
    assert ls.n_compared > 0
    assert any(ls.drv.cache.export_state(s)["n_evicted"] > 0 for s in range(3))


@pytest.mark.parametrize("policy", ["position", "sink_recent"])
def test_policy_variants_tiny_f32(policy):
    w = S.TINY_F32.with_(policy=policy, sink=4, recent=300)
    ls, _ = _lockstep(w)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda *a: True)
    assert ls.drv.cache.export_state(0)["n_evicted"] > 0


def test_position_variant_single_session_full_size():
    """The position-granular variant on the full-size single-session workload: every evict
    bit-exact (the resident count lands on B exactly), attention sampled."""
    ls, _ = _lockstep(S.SINGLE_BF16.with_(policy="position"))
    samples = {190, 420, 599}
    for step in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda st, kind, i, layer: st in samples and layer in (0, 31)
                    and i in (0, 1))
    st = ls.drv.cache.export_state(0)
    assert st["resident"] == 4096


def test_transcript_export():
    """Transcript export (Sec. 4.2): positions bit-exact against the oracle, K and V
    bit-exact against the stored rows of those positions, count exact, and a short
    capacity keeps the first positions."""
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=3, budget=64, window=2, seed=5,
                            p_no_segment=0.1, p_long_segment=0.1, turn_period=12, turn_jitter=2)
    ls, _ = _lockstep(w, n_units=40)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=None)
    cache = ls.drv.cache
    for s in range(3):
        want = ls.orc.transcript_positions(s)
        st = cache.export_state(s)
        pos, k, v, count = cache.export_transcript(s, st["resident"])
        torch.cuda.synchronize()
        n = int(count.item())
        assert n == len(want) > 0
        assert pos[:n].cpu().numpy().tolist() == want
        idx = [st["pos"].index(p) for p in want]
        for layer in range(w.layers):
            ks, vs = cache.export_kv(s, layer)
            assert np.array_equal(k[layer, :n].float().cpu().numpy(), ks[idx])
            assert np.array_equal(v[layer, :n].float().cpu().numpy(), vs[idx])
        pos2, k2, _, count2 = cache.export_transcript(s, 3)
        torch.cuda.synchronize()
        assert int(count2.item()) == n
        assert pos2.cpu().numpy().tolist() == want[:3]
        assert torch.equal(k2[:, :3], k[:, :3])


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_per_layer_append(dtype):
    """The model's order: appends without K/V, each layer's K/V written just before that
    layer's attention; state and every output as with whole-chunk appends."""
    w = (S.SINGLE_BF16.with_(layers=3, n_sessions=3, budget=80, window=2, seed=13,
                             turn_period=10, turn_jitter=1) if dtype == "bf16"
         else S.TINY_F32.with_(units=30))
    ls, _ = _lockstep(w, n_units=30)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda *a: True, per_layer=True)
    assert ls.n_compared > 0


def test_per_layer_append_batch64_prefill():
    """The model's order at the 64-session prefill size: every prefill call (64 sessions x
    17 positions) writes its layer's rows inside the tensor-core attention launch
    (kvc_attn_prefill_chunk_kv) and every decode call inside the decode launch; all
    outputs of sampled layers compared with the oracle, every evict bit-exact."""
    w = S.SINGLE_BF16.with_(layers=4, n_sessions=64, budget=300, window=2, seed=41,
                            offset_max=2, turn_period=9, turn_jitter=1)
    ls, _ = _lockstep(w, n_units=18)
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda st, kind, i, layer: layer in (0, 3) and
                    (kind == "prefill" or st % 4 == 0), per_layer=True)
    assert ls.n_compared > 64 * 2 * 10


def test_fused_layer_write_stores_the_same_bytes():
    """Whole-chunk appends and the per-layer order (separate writes for prefill chunks,
    writes fused into the decode launches) leave bit-identical K/V in every layer."""
    w = S.SINGLE_BF16.with_(layers=3, n_sessions=2, budget=60, window=1, seed=3,
                            turn_period=8, turn_jitter=1)
    scripts = S.workload_scripts(w)
    for sc in scripts:
        sc.n_transcript = sc.n_transcript[:25]
        sc.n_text = sc.n_text[:25]
    a, b = Driver(w, scripts), Driver(w, scripts)
    for _ in range(len(a.sched)):
        a.run_step(a.prepare_step())
        b.run_step(b.prepare_step(), per_layer=True)
    torch.cuda.synchronize()
    for s in range(2):
        assert a.cache.export_state(s)["pos"] == b.cache.export_state(s)["pos"]
        for layer in range(w.layers):
            ka, va = a.cache.export_kv(s, layer)
            kb, vb = b.cache.export_kv(s, layer)
            assert np.array_equal(ka, kb) and np.array_equal(va, vb)


def test_attention_needs_the_layer_written():
    from paper_2609_31224_gb300._lib import KvcError
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=1, units=3)
    drv = Driver(w, S.workload_scripts(w))
    st = drv.prepare_step()
    c = [c for c in st.calls if c.kind == "prefill"][0]
    drv.cache.append_chunk(c.sessions, c.cu, c.types, None, None)
    with pytest.raises(KvcError, match="ESTATE"):
        drv.cache.attn_prefill_chunk(0, c.q[0], c.out)
    drv.cache.append_kv_layer(0, c.k[0], c.v[0])
    drv.cache.attn_prefill_chunk(0, c.q[0], c.out)
    with pytest.raises(KvcError, match="ESTATE"):
        drv.cache.attn_prefill_chunk(1, c.q[1], c.out)
    torch.cuda.synchronize()


def test_sharp_attention_bf16():
    """Larger query scale makes the softmax peaked, so a wrong key order shows.

    Logits have standard deviation 6 here, and the tensor-core path rounds the rotated
    query and the probabilities to bfloat16 (relative 2^-9): a logit moves by about
    6 * 2^-9 / sqrt(3) = 0.007, a weight by 0.7 %, an output by up to a few 1e-2.  The
    elementwise bound is therefore 6e-2 + 1e-2 |ref|; the normwise bound stays 1e-2,
    which a wrong key, mask or order exceeds by far."""
    w = S.SINGLE_BF16.with_(layers=1, n_sessions=2, budget=96, window=2, seed=9, q_scale=6.0,
                            turn_period=10, turn_jitter=1)
    ls, _ = _lockstep(w, n_units=30, tol=(6e-2, 1e-2, 1e-2))
    for _ in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda *a: True)
    assert max(s["max_abs"] for s in ls.stats) > 0  # outputs were compared


def test_single_session_full_size_metadata_and_sampled_attention():
    """600 units, 32 layers, B=4096, W=10: every evict bit-exact; attention sampled."""
    ls, _ = _lockstep(S.SINGLE_BF16)
    samples = {0, 1, 50, 186, 187, 300, 420, 599}
    for step in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda st, kind, i, layer: st in samples and
                    (layer in (0, 31) or (kind == "decode" and i == 1 and layer == 17)))
    st = ls.drv.cache.export_state(0)
    assert st["resident"] <= 4096
    assert st["peak_resident"] > 4096


@pytest.mark.parametrize("budget", [8192, 0])
def test_single_session_full_size_table3_budgets(budget):
    """Table 3's other budgets on the full-size single-session workload (32 layers, 600
    units): B = 8K and the B = 0 floor.  Every evict bit-exact, peak resident count
    included (End and Peak of Table 3 are the device's resident and peak_resident at the
    end); attention sampled."""
    ls, _ = _lockstep(S.SINGLE_BF16.with_(budget=budget))
    last = len(ls.drv.sched) - 1
    samples = {300, last}
    for step in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda st, kind, i, layer: st in samples and layer == 0
                    and i in (0, 1))
    st = ls.drv.cache.export_state(0)
    ref = ls.orc.state(0)
    assert (st["resident"], st["peak_resident"]) == (ref["resident"], ref["peak_resident"])
    if budget > 0:
        assert st["resident"] <= budget < st["peak_resident"]
    else:
        assert all(t in (2, 3) or u > ref["unit_cur"] - S.SINGLE_BF16.window
                   for t, u in zip(st["type"], st["unit"]))
    assert ls.n_compared >= 4


@pytest.mark.parametrize("policy", ["unit", "position", "sink_recent"])
def test_release_and_reuse(policy):
    """kvc_release ends sessions mid-run; fed the rest of their scripts from position 0 they
    evict as fresh sessions under the same policy.  Every state bit-exact after the release
    and after every evict, every attention output compared."""
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=3, budget=60, window=1, seed=31,
                            turn_period=9, turn_jitter=1, policy=policy, sink=3, recent=30)
    ls, _ = _lockstep(w, n_units=36)
    for _ in range(15):
        ls.run_step(attn_pred=lambda *a: True)
    free0, _ = ls.drv.cache.device_status()
    held = sum(len(ls.orc.layout[s].hist_pages) + len(ls.orc.layout[s].live_pages)
               for s in (0, 2))
    ls.release([0, 2])
    free1, err = ls.drv.cache.device_status()
    assert err == 0 and free1 == free0 + held
    for _ in range(len(ls.drv.sched) - 15):
        ls.run_step(attn_pred=lambda *a: True)
    for s in (0, 2):
        assert ls.drv.cache.export_state(s)["n_evicted"] > 0
    assert ls.n_compared > 100


def test_single_session_unbounded_full_size():
    """No-eviction run of the single-session workload (B = infinity): every evict is a
    no-op checked bit-exact, the cache grows to every fed position (about 13.7K), and
    attention over the longest contexts is sampled late in the session."""
    ls, scripts = _lockstep(S.SINGLE_BF16_UNBOUNDED)
    samples = {0, 300, 598, 599}
    for step in range(len(ls.drv.sched)):
        ls.run_step(attn_pred=lambda st, kind, i, layer: st in samples and
                    (layer in (0, 31) or (kind == "decode" and i == 1 and layer == 17)))
    st = ls.drv.cache.export_state(0)
    total = len(scripts[0].all_types())
    assert st["resident"] == total and st["n_evicted"] == 0
    assert st["peak_resident"] == total > 13000
    assert ls.n_compared >= 8


@pytest.mark.parametrize("budget,window", [(2048, 5), (2048, 20), (8192, 5), (8192, 20)])
def test_stress_shard(budget, window):
    """The 256-session stress workload (10-60 minute sessions, 5% units without a segment,
    2% long segments of 10-30 tokens) at each (B, W) grid point, on a shard of four
    sessions (one per stride of 64) run until well past the budget: every evict
    bit-exact, attention sampled at the edges of the run."""
    w = S.stress256(budget, window)
    n_units = budget // 20 + 60
    scripts = []
    for sid in (3, 67, 131, 195):
        sc = S.session_script(w, sid)
        sc.n_transcript = sc.n_transcript[:n_units]
        sc.n_text = sc.n_text[:n_units]
        scripts.append(sc)
    # The shard must exercise both segment edge cases.
    assert sum(int((sc.n_transcript < 0).sum()) for sc in scripts) > 0
    assert sum(int((sc.n_transcript >= 10).sum()) for sc in scripts) > 0
    drv = Driver(w, scripts)
    ls = Lockstep(drv, w)
    last = len(drv.sched) - 1
    samples = {0, last // 2, last - 1, last}
    for step in range(len(drv.sched)):
        ls.run_step(attn_pred=lambda st, kind, i, layer: st in samples and layer in (0, 31)
                    and i in (0, 1, 2))
    for sc in scripts:
        st = drv.cache.export_state(sc.session)
        assert st["n_evicted"] > 0
        assert st["peak_resident"] > budget
    assert ls.n_compared >= 16


def _sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def _decode_tier(n_seq, kv_heads):
    """Decode kernel the library dispatches for a call of n_seq sessions: the 16-warp pair
    split (one CTA per SM) while every (session, KV head) pair gets five slices, the 4-warp
    pair split while it gets one of the three CTAs per SM, else stream-K."""
    pairs = n_seq * kv_heads
    if 5 * pairs <= _sms():
        return "split16"
    if pairs <= 3 * _sms():
        return "split4"
    return "streamk"


def test_decode_4warp_tier_at_full_budget():
    """Decode calls of 10-19 sessions (the 4-warp pair split with three slices or more per
    pair on 152 SMs) at full budget,
    every output of every session compared with the oracle: the first two natural decode
    rounds of that size in a step of a 19-session shard of the 64-session workload at its
    steady state, then calls of exactly 10, 12, 16 and 19 sessions (one transcript token
    each)."""
    w = S.BATCH64_BF16
    scripts = S.workload_scripts(w)
    shard = sorted(scripts, key=lambda sc: sc.offset)[:19]
    drv = Driver(w, shard)
    ls = Lockstep(drv, w)
    steady = S.steady_state_step(w, shard)
    for _ in range(steady):
        ls.run_step(check_state=False)
    tiers = {}
    picked = []

    def select(step, c, i, layer):
        if c.kind != "decode" or layer != 0:
            return None
        tier = _decode_tier(len(c.sessions), w.kv_heads)
        if tier != "split4" or len(picked) >= 2:
            return None
        picked.append(len(c.sessions))
        tiers.setdefault(tier, set()).add(len(c.sessions))
        return "all"

    ls.run_step(select=select)
    for n in (10, 12, 16, 19):
        ls.decode_call([sc.session for sc in shard[:n]], layers=(0, 31) if n == 10 else (0,))
        tiers.setdefault(_decode_tier(n, w.kv_heads), set()).add(n)
    for sc in shard:
        st = drv.cache.export_state(sc.session)
        assert st["resident"] >= 4000 and st["n_evicted"] > 0
    if _sms() == 152:
        assert {10, 12, 16, 19} <= tiers["split4"]
        assert len(picked) == 2
    assert ls.n_compared >= 10 * 2 + 12 + 16 + 19


def test_f32_decode_every_tier():
    """Binary32 decode in every dispatch tier: 480 sessions of the tiny binary32 shape (one
    KV head each) starting together, so that a step's decode rounds shrink from 480
    sessions (stream-K) through the 4-warp pair split with one, two and more slices per
    pair down to the 16-warp pair split; every output of every decode call of every
    third step compared with the oracle, every evict bit-exact."""
    w = S.TINY_F32.with_(n_sessions=480, offset_max=2, budget=64, window=1, seed=7)
    ls, _ = _lockstep(w, n_units=12)
    seen = set()

    def select(step, c, i, layer):
        if c.kind != "decode" or step % 3:
            return None
        seen.add(_decode_tier(len(c.sessions), w.kv_heads))
        return "all"

    for _ in range(len(ls.drv.sched)):
        ls.run_step(select=select)
    if _sms() == 152:
        assert {"streamk", "split4", "split16"} <= seen
    assert ls.n_compared > 1000


def test_decode_4warp_tier_one_and_two_slices():
    """Decode calls of 20-57 sessions, where the 4-warp pair split gives every (session, KV
    head) pair two slices (20-28 sessions, merged by the last to arrive) or one (29-57, no
    merge), at full budget: a 57-session shard of the 64-session workload brought to its
    steady state, then calls of exactly 20, 28, 29, 40 and 57 sessions (one transcript
    token each), every output of layer 0 compared with the oracle."""
    w = S.BATCH64_BF16
    scripts = S.workload_scripts(w)
    shard = sorted(scripts, key=lambda sc: sc.offset)[:57]
    drv = Driver(w, shard)
    ls = Lockstep(drv, w)
    steady = S.steady_state_step(w, shard)
    for _ in range(steady):
        ls.run_step(check_state=False)
    for n in (20, 28, 29, 40, 57):
        ls.decode_call([sc.session for sc in shard[:n]], layers=(0,))
        if _sms() == 152:
            assert _decode_tier(n, w.kv_heads) == "split4"
    for sc in shard[:20]:
        st = drv.cache.export_state(sc.session)
        assert st["resident"] >= 4000 and st["n_evicted"] > 0
    assert ls.n_compared >= 20 + 28 + 29 + 40 + 57


def test_batch64_sampled_at_full_size():
    """64 sessions, offsets U{0..300}, run through the benchmark's timed window (its 20
    steps from the steady state): the state of every session bit-exact at sampled steps and
    after every evict of the window; attention in the benchmark's launch configuration at
    three steps of the window: the prefill call and the first decode round of each kernel
    tier present (stream-K for >= 58 sessions, the 4-warp pair split for 4-57, the
    16-warp tensor-core pair split for <= 3, and a one-session round)."""
    w = S.BATCH64_BF16
    scripts = S.workload_scripts(w)
    drv = Driver(w, scripts)
    ls = Lockstep(drv, w)
    start = S.steady_state_step(w, scripts)
    stop = start + 20
    check = set(range(0, start, 97))
    sampled = {start: 0, start + 9: 13, stop - 1: 31}   # step -> layer compared
    seen = set()

    def select(step, c, i, layer):
        if sampled.get(step) != layer:
            return None
        if c.kind == "prefill":
            return {0, 21, 42, 63}
        n = len(c.sessions)
        tier = "one" if n == 1 else _decode_tier(n, w.kv_heads)
        if (tier, step) in seen:
            return None
        seen.add((tier, step))
        stride = {"streamk": 16, "split4": 5, "split16": 3, "one": 1}[tier]
        return {int(x) for x in c.sessions[::stride]}

    for step in range(stop):
        if step >= start or step in check:
            ls.run_step(select=select)
        else:
            # The oracle replays the policy without comparing every state.
            ls.run_step(check_state=False)
    tiers = {t for t, _ in seen}
    assert {"streamk", "split16"} <= tiers
    if _sms() == 152:
        assert "split4" in tiers
    assert ls.n_compared >= 30


def test_compaction_is_a_pure_move():
    """Stored K/V of retained positions are byte-identical before and after evict."""
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=2, budget=100, window=2, seed=12)
    scripts = S.workload_scripts(w)
    for sc in scripts:
        sc.n_transcript = sc.n_transcript[:20]
        sc.n_text = sc.n_text[:20]
    drv = Driver(w, scripts)
    moved = 0
    for _ in range(len(drv.sched)):
        st = drv.prepare_step()
        for c in st.calls:
            drv.run_call(c)
        before = {}
        for s in st.evict_sessions.tolist():
            meta = drv.cache.export_state(s)
            for layer in (0, 1):
                k, v = drv.cache.export_kv(s, layer)
                before[(s, layer)] = dict(zip(meta["pos"], zip(k, v)))
        drv.cache.evict(st.evict_sessions)
        for s in st.evict_sessions.tolist():
            meta = drv.cache.export_state(s)
            for layer in (0, 1):
                k, v = drv.cache.export_kv(s, layer)
                for p, kk, vv in zip(meta["pos"], k, v):
                    kb, vb = before[(s, layer)][p]
                    assert np.array_equal(kk, kb) and np.array_equal(vv, vb)
                    moved += 1
    assert moved > 0


def test_stored_keys_match_oracle_rotation():
    """K is stored rotated at its original position (within one storage ulp)."""
    from oracle.numerics import round_bf16
    from oracle.rope import rope
    w = S.SINGLE_BF16.with_(layers=1, n_sessions=1, budget=-1, seed=2)
    scripts = S.workload_scripts(w)
    for sc in scripts:
        sc.n_transcript = sc.n_transcript[:8]
        sc.n_text = sc.n_text[:8]
    drv = Driver(w, scripts)
    for _ in range(len(drv.sched)):
        drv.run_step(drv.prepare_step(), attention=False)
    meta = drv.cache.export_state(0)
    k, v = drv.cache.export_kv(0, 0)
    pos = np.asarray(meta["pos"])
    raw = V.layer_tensor(w.seed, V.TAG_K, 0, 0, pos, w.kv_heads, w.head_dim, "bf16")
    exact = rope(raw, pos[:, None], w.rope_base)
    want = round_bf16(exact)
    # The kernel rotates in binary32 with a binary32 cos/sin table: error at most a few
    # 2^-24 of the terms |x_i| + |x_{i+D/2}|, then one bfloat16 rounding of the result.
    half = w.head_dim // 2
    terms = np.abs(raw) + np.abs(np.concatenate([raw[..., half:], raw[..., :half]], axis=-1))
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(exact), 1e-30))) - 7)
    assert (np.abs(k - want) <= ulp + 2.0 ** -21 * terms).all()
    assert np.mean(k == want) > 0.99
    assert np.array_equal(v, V.layer_tensor(w.seed, V.TAG_V, 0, 0, pos, w.kv_heads,
                                            w.head_dim, "bf16"))


def test_error_codes():
    from paper_2609_31224_gb300 import KVCache, KvcError
    c = KVCache(n_sessions=2, layers=1, q_heads=4, kv_heads=1, head_dim=64, budget=8, window=0,
                dtype="f32", n_pages=3, max_pages_per_session=4, max_positions=100,
                max_seq_per_call=2, max_tokens_per_call=64)
    q = torch.zeros((64, 4, 64), device="cuda")
    out = torch.zeros_like(q)
    with pytest.raises(KvcError) as e:
        c.attn_decode(0, q, out)
    assert e.value.code == -4  # no append yet
    types = torch.zeros(64, dtype=torch.uint8, device="cuda")
    kv = torch.zeros((1, 64, 1, 64), device="cuda")
    with pytest.raises(KvcError) as e:
        c.append_chunk([0], [0, 60], types, kv, kv)
    assert e.value.code == -2  # 60 tokens need 4 pages, the pool has 3
    c.append_chunk([0], [0, 20], types, kv, kv)
    with pytest.raises(KvcError) as e:
        c.attn_decode(0, q, out)
    assert e.value.code == -4  # decode needs one token per session
    with pytest.raises(KvcError) as e:
        c.append_chunk([1], [0, 20], types, kv, kv)
    assert e.value.code == -2  # pool has 3 pages, 2 in use
    with pytest.raises(KvcError) as e:
        c.append_chunk([0, 0], [0, 1, 2], types, kv, kv)
    assert e.value.code == -1  # repeated session
    with pytest.raises(KvcError) as e:
        c.attn_prefill_chunk(5, q, out)
    assert e.value.code == -1  # bad layer
    c.evict([0])
    with pytest.raises(KvcError) as e:
        c.attn_prefill_chunk(0, q, out)
    assert e.value.code == -4  # evict invalidates the queries
    free, err = c.device_status()
    assert err == 0 and free >= 1
    c.release([0])
    free, err = c.device_status()
    assert free == 3


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_decode_graph_replay_matches_eager(dtype):
    """Decode launches captured in a CUDA graph merge their split-K partial states after
    a fenced arrival (a replay repeats the captured arguments); eager launches tag each
    partial word with the launch.  Both merge in the same order, so the outputs are
    bit-identical, across replays and for eager launches after them."""
    w = S.SINGLE_BF16.with_(layers=2, n_sessions=12, units=80, seed=5)
    if dtype == "f32":
        w = w.with_(dtype="f32", head_dim=64)
    drv = Driver(w, S.workload_scripts(w))
    drv.fast_forward(60)
    torch.cuda.synchronize()
    for n in (1, 4, 12):
        c = drv._make_call("decode", list(range(n)), [np.array([3], np.uint8)] * n, True)
        drv.cache.append_chunk(c.sessions, c.cu, c.types, c.k, c.v)
        eager = []
        for layer in range(w.layers):
            drv.cache.attn_decode(layer, c.q[layer], c.out)
            eager.append(c.out.clone())
        outs = [torch.empty_like(c.out) for _ in range(w.layers)]
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.graph(g, stream=s):
            for layer in range(w.layers):
                drv.cache.attn_decode(layer, c.q[layer], outs[layer], stream=s)
        for _ in range(3):
            for o in outs:
                o.zero_()
            g.replay()
            torch.cuda.synchronize()
            for layer in range(w.layers):
                assert torch.equal(outs[layer], eager[layer]), (n, layer)
        for layer in range(w.layers):
            drv.cache.attn_decode(layer, c.q[layer], c.out)
            assert torch.equal(c.out, eager[layer]), (n, layer)
        del g
        torch.cuda.synchronize()
