"""The seeded input generators: published SplitMix64 outputs, value statistics and
script shape.  These generators feed both the oracle and the CUDA path."""
import numpy as np
import pytest

from synth import script as S
from synth import values as V


def test_splitmix64_published_outputs():
    """First outputs of SplitMix64 from state 0 (the reference C implementation by
    Vigna, used to seed the xoshiro family)."""
    assert V.splitmix64_stream(0, 3) == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4,
                                         0x06C45D188009454F]


def test_vectorised_hash_equals_scalar_stream():
    base = V.stream_base(7, V.TAG_K)
    assert V.hash64(7, V.TAG_K, np.arange(10)).tolist() == V.splitmix64_stream(base, 10)


def test_values_are_deterministic_and_roughly_standard_normal():
    x = V.values(0, V.TAG_V, 0, np.arange(4)[:, None], np.arange(4000)[None, :], 0, 0, "f32")
    y = V.values(0, V.TAG_V, 0, np.arange(4)[:, None], np.arange(4000)[None, :], 0, 0, "f32")
    assert np.array_equal(x, y)
    assert abs(float(x.mean())) < 0.03
    assert abs(float(x.var()) - 1.0) < 0.03
    # Irwin-Hall(4) of 16-bit fields is bounded by 2 sqrt(3)
    assert float(np.abs(x).max()) <= 2 * np.sqrt(3) + 1e-6
    z = V.values(1, V.TAG_V, 0, np.arange(4)[:, None], np.arange(4000)[None, :], 0, 0, "f32")
    assert not np.array_equal(x, z)


def test_irwin_hall_value_from_hash_by_hand():
    h = V.mix64_int(V.stream_base(0, V.TAG_Q) + V.GAMMA)  # element index 0
    s = sum((h >> (16 * i)) & 0xFFFF for i in range(4))
    want = np.float32(s - 131070) * np.float32(np.sqrt(3.0) / 65536.0)
    got = V.values_f32(0, V.TAG_Q, 0, 0, 0, 0, 0)
    assert got.item() == want


def test_bf16_storage_is_round_to_nearest_even():
    import torch
    x = V.values_f32(3, V.TAG_K, 1, 0, np.arange(2000), np.arange(8)[:, None], 3)
    got = V.values(3, V.TAG_K, 1, 0, np.arange(2000), np.arange(8)[:, None], 3, "bf16")
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(got, want)


def test_script_shape_single_session():
    sc = S.session_script(S.SINGLE_BF16, 0)
    assert sc.n_units == 600
    n_tr = sc.n_transcript
    assert (n_tr >= 0).all()
    assert 2.7 < n_tr.mean() < 3.3
    turns = np.nonzero(sc.n_text)[0]
    assert 8 <= len(turns) <= 11
    assert ((sc.n_text[turns] >= 20) & (sc.n_text[turns] <= 80)).all()
    gaps = np.diff(turns)
    assert (gaps >= 50).all() and (gaps <= 70).all()
    types = sc.unit_types(0)
    assert types[0] == S.ACOUSTIC | S.UNIT_BEGIN
    assert (types[1:17] == S.ACOUSTIC).all()
    assert types[17] == S.ASR_DELIM


def test_script_stress_mix():
    w = S.stress256(2048, 5)
    scripts = [S.session_script(w, s) for s in range(32)]
    n_tr = np.concatenate([s.n_transcript for s in scripts])
    assert 0.035 < float((n_tr < 0).mean()) < 0.065
    assert 0.01 < float((n_tr >= 10).mean()) < 0.035
    lens = [s.n_units for s in scripts]
    assert min(lens) >= 600 and max(lens) <= 3600


def test_schedule_offsets():
    w = S.BATCH64_BF16
    scripts = S.workload_scripts(w)
    sched = S.schedule(scripts)
    offs = [s.offset for s in scripts]
    assert 0 <= min(offs) and max(offs) <= 300
    assert len(sched) == max(offs) + 600
    assert sum(len(x) for x in sched) == 64 * 600
    step = S.steady_state_step(w, scripts)
    assert len(sched[step]) == 64
