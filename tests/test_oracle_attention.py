"""Pins for the oracle's RoPE, storage rounding and attention.

Pinned against closed forms (single key, identical keys), a scalar brute force
written with ``math`` only, the complex-number form of rotary embeddings, the
relative-position property RoPE exists for, torch's bfloat16 conversion, and
the retained-set / masked-full-cache equivalence of the eviction method.
"""
import math

import numpy as np
import pytest
import torch

from oracle.attention import gqa_attention, softmax_attention
from oracle.cache import OracleCache, OracleConfig
from oracle.numerics import round_bf16
from oracle.rope import rope
from synth.script import ACOUSTIC, ASR_DELIM, TEXT, TRANSCRIPT, UNIT_BEGIN


# -- attention -----------------------------------------------------------------------------

def _scalar_attention(q, k, v, visible, scale):
    """Brute force: one query row at a time with math.exp and math.fsum."""
    out = []
    for r in range(len(q)):
        scores = [scale * math.fsum(q[r][i] * k[j][i] for i in range(len(q[r])))
                  if visible[r][j] else None for j in range(len(k))]
        m = max(s for s in scores if s is not None)
        w = [math.exp(s - m) if s is not None else 0.0 for s in scores]
        z = math.fsum(w)
        out.append([math.fsum(w[j] * v[j][d] for j in range(len(k))) / z
                    for d in range(len(v[0]))])
    return np.array(out)


@pytest.mark.parametrize("seed", range(20))
def test_attention_matches_scalar_brute_force(seed):
    rng = np.random.default_rng(seed)
    r, n, d = int(rng.integers(1, 6)), int(rng.integers(1, 40)), int(rng.integers(1, 9))
    q, k, v = rng.normal(size=(r, d)), rng.normal(size=(n, d)), rng.normal(size=(n, d))
    visible = rng.random((r, n)) < 0.7
    visible[:, 0] = True
    scale = 1.0 / math.sqrt(d)
    got = softmax_attention(q, k, v, visible, scale)
    want = _scalar_attention(q.tolist(), k.tolist(), v.tolist(), visible.tolist(), scale)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_single_key_returns_its_value():
    rng = np.random.default_rng(1)
    q, k, v = rng.normal(size=(3, 8)), rng.normal(size=(1, 8)), rng.normal(size=(1, 8))
    out = softmax_attention(q, k, v, np.ones((3, 1), bool), 0.3)
    assert np.array_equal(out, np.repeat(v, 3, axis=0))


def test_identical_keys_average_values():
    rng = np.random.default_rng(2)
    k = np.repeat(rng.normal(size=(1, 16)), 50, axis=0)
    v = rng.normal(size=(50, 16))
    out = softmax_attention(rng.normal(size=(4, 16)), k, v, np.ones((4, 50), bool), 0.25)
    np.testing.assert_allclose(out, np.repeat(v.mean(0, keepdims=True), 4, axis=0),
                               rtol=1e-13, atol=1e-13)


def test_gqa_heads_share_kv_heads_and_mask_is_causal():
    rng = np.random.default_rng(3)
    t, hq, hkv, d, n = 3, 8, 2, 4, 10
    q = rng.normal(size=(t, hq, d))
    k, v = rng.normal(size=(n, hkv, d)), rng.normal(size=(n, hkv, d))
    k_pos = np.arange(n) * 2
    q_pos = np.array([13, 14, 18])
    out = gqa_attention(q, k, v, q_pos, k_pos)
    for h in range(hq):
        for i in range(t):
            vis = [[bool(kp <= q_pos[i]) for kp in k_pos]]
            want = _scalar_attention([q[i, h].tolist()], k[:, h // 4].tolist(),
                                     v[:, h // 4].tolist(), vis, 1 / math.sqrt(d))
            np.testing.assert_allclose(out[i, h], want[0], rtol=1e-12, atol=1e-12)


# -- RoPE ----------------------------------------------------------------------------------

def test_rope_matches_complex_form():
    """Rotate-half RoPE is multiplication of (x_i + i x_{i+D/2}) by exp(i p theta_i)."""
    rng = np.random.default_rng(4)
    d, base = 64, 10000.0
    x = rng.normal(size=(7, d))
    pos = np.array([0, 1, 5, 100, 4095, 60000, 123456])
    got = rope(x, pos, base)
    z = x[:, : d // 2] + 1j * x[:, d // 2:]
    theta = np.array([base ** (-2.0 * i / d) for i in range(d // 2)])
    rot = z * np.exp(1j * pos[:, None] * theta[None, :])
    want = np.concatenate([rot.real, rot.imag], axis=1)
    np.testing.assert_allclose(got, want, rtol=1e-9, atol=1e-9)


def test_rope_identity_at_zero_and_norm_preserving():
    rng = np.random.default_rng(5)
    x = rng.normal(size=(5, 128))
    assert np.array_equal(rope(x, np.zeros(5), 10000.0), x)
    y = rope(x, np.arange(5) * 977, 10000.0)
    np.testing.assert_allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1),
                               rtol=1e-13)


def test_rope_scores_depend_only_on_relative_position():
    rng = np.random.default_rng(6)
    q, k = rng.normal(size=128), rng.normal(size=128)
    for p, pk in [(10, 3), (500, 17), (4000, 3999)]:
        s0 = rope(q, p, 10000.0) @ rope(k, pk, 10000.0)
        for shift in (1, 77, 10_000):
            s1 = rope(q, p + shift, 10000.0) @ rope(k, pk + shift, 10000.0)
            assert abs(s1 - s0) < 1e-8 * max(1.0, abs(s0))


# -- storage rounding ------------------------------------------------------------------------

def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(7)
    x = np.concatenate([rng.normal(size=20000) * 10.0 ** rng.integers(-6, 6, size=20000),
                        # exact ties between two bf16 neighbours, both parities
                        1.0 + np.array([1, 3, 5, 7]) * 2.0 ** -8,
                        -(2.0 + np.array([1, 3]) * 2.0 ** -7),
                        [0.0, -0.0, 1e-40]])
    want = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(round_bf16(x), want)


# -- the method's invariant: retained set == masked full cache --------------------------------

def _tiny_values(n_pos, layers, heads, d, seed):
    rng = np.random.default_rng(seed)
    k = rng.normal(size=(layers, n_pos, heads, d))
    v = rng.normal(size=(layers, n_pos, heads, d))
    return k, v


@pytest.mark.parametrize("budget,window", [(20, 1), (0, 0), (40, 3)])
def test_retained_attention_equals_masked_full_attention(budget, window):
    hq, hkv, d = 4, 2, 8
    rng = np.random.default_rng(8)
    k_all, v_all = _tiny_values(400, 1, hkv, d, 9)

    def source(s, layer, positions):
        return k_all[layer, positions], v_all[layer, positions]

    cfg = dict(n_sessions=1, layers=1, q_heads=hq, kv_heads=hkv, head_dim=d, page_size=4,
               window=window, dtype="f32", rope_base=10000.0, n_pages=200)
    evicting = OracleCache(OracleConfig(budget=budget, **cfg))
    full = OracleCache(OracleConfig(budget=-1, **cfg))
    checked = 0
    for u in range(12):
        chunk = [ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * 5
        tail = [ASR_DELIM] + [TRANSCRIPT] * int(rng.integers(0, 4)) + [ASR_DELIM]
        for cache in (evicting, full):
            cache.append_chunk([0], [chunk])
        q = rng.normal(size=(len(chunk), hq, d))
        got = evicting.attend(0, [q], source)[0]
        # Full cache, with every evicted position masked out of the keys.
        keys = full.layout[0].retained_positions()
        kept = set(evicting.policy[0].retained_positions())
        k, v = full.stored_keys(0, 0, keys, source)
        mask_keys = [i for i, p in enumerate(keys) if p in kept]
        q_pos = evicting.last_append[0][1]
        want = gqa_attention(rope(q, np.asarray(q_pos)[:, None], 10000.0), k[mask_keys],
                             v[mask_keys], q_pos, np.asarray(keys)[mask_keys])
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)
        checked += len(keys) - len(mask_keys)
        for tok in tail:
            for cache in (evicting, full):
                cache.append_chunk([0], [[tok]])
        for cache in (evicting, full):
            cache.evict([0])
    assert checked > 0  # the comparison did exercise evicted keys


def test_unbounded_cache_is_plain_causal_attention():
    hq, hkv, d = 2, 1, 4
    k_all, v_all = _tiny_values(100, 1, hkv, d, 10)

    def source(s, layer, positions):
        return k_all[layer, positions], v_all[layer, positions]

    c = OracleCache(OracleConfig(n_sessions=1, layers=1, q_heads=hq, kv_heads=hkv, head_dim=d,
                                 page_size=4, budget=-1, window=0, dtype="f32",
                                 rope_base=10000.0, n_pages=50))
    rng = np.random.default_rng(11)
    for u in range(5):
        c.append_chunk([0], [[ACOUSTIC | UNIT_BEGIN] + [ACOUSTIC] * 6 + [TEXT]])
        c.evict([0])
    c.append_chunk([0], [[ACOUSTIC | UNIT_BEGIN, ACOUSTIC, ACOUSTIC]])
    q = rng.normal(size=(3, hq, d))
    got = c.attend(0, [q], source)[0]
    n = c.policy[0].pos_next
    pos = np.arange(n)
    from oracle.numerics import round_f32
    k = round_f32(rope(k_all[0, :n], pos[:, None], 10000.0))
    qr = rope(q, np.arange(n - 3, n)[:, None], 10000.0)
    for t in range(3):
        for h in range(hq):
            vis = [[j <= n - 3 + t for j in range(n)]]
            want = _scalar_attention([qr[t, h].tolist()], k[:, 0].tolist(),
                                     v_all[0, :n, 0].tolist(), vis, 1 / math.sqrt(d))
            np.testing.assert_allclose(got[t, h], want[0], rtol=1e-11, atol=1e-12)
