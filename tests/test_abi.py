"""The C-ABI library builds for sm_103a, loads, exports every symbol declared in
include/kvc.h, and validates arguments on the host (no GPU needed)."""
import ctypes
import os
import re

import pytest

from paper_2609_31224_gb300 import _lib as L
from paper_2609_31224_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return L.load_library()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "kvc.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kvc_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 13
    for n in names:
        assert hasattr(lib, n), n
    assert set(L.EXPORTED) == set(names)


def _cfg(**kw):
    base = dict(n_sessions=4, layers=2, q_heads=32, kv_heads=8, head_dim=128, page_size=16,
                budget=4096, window=10, dtype=L.KVC_BF16, rope_base=10000.0, n_pages=1024,
                max_pages_per_session=512, max_positions=20000, max_seq_per_call=4,
                max_tokens_per_call=68)
    base.update(kw)
    return L.Config(**base)


def test_query_sizes_pool_formula(lib):
    pool, meta = L.query_sizes(_cfg())
    assert pool == 1024 * 2 * 2 * 8 * 16 * 128 * 2
    assert meta > 0 and meta % 256 == 0
    pool32, _ = L.query_sizes(_cfg(dtype=L.KVC_F32, head_dim=64, q_heads=4, kv_heads=1))
    assert pool32 == 1024 * 2 * 2 * 1 * 16 * 64 * 4


@pytest.mark.parametrize("bad", [
    dict(q_heads=16),                      # G != 4
    dict(page_size=32),
    dict(head_dim=64),                     # bf16 needs 128
    dict(dtype=L.KVC_F32),                 # f32 needs 64
    dict(window=-1),
    dict(n_pages=0),
    dict(max_seq_per_call=5),              # > n_sessions
    dict(layers=0),
    dict(rope_base=0.0),
    dict(max_positions=0),
])
def test_invalid_configs_are_rejected_on_the_host(lib, bad):
    pool, meta = ctypes.c_size_t(), ctypes.c_size_t()
    rc = lib.kvc_query_sizes(ctypes.byref(_cfg(**bad)), ctypes.byref(pool), ctypes.byref(meta))
    assert rc == -1
    assert lib.kvc_last_error()
    ctx = ctypes.c_void_p()
    rc = lib.kvc_create(ctypes.byref(ctx), ctypes.byref(_cfg(**bad)), None, 0, None, 0, None)
    assert rc == -1 and not ctx.value


def test_create_rejects_small_or_unaligned_buffers(lib):
    pool, meta = L.query_sizes(_cfg())
    ctx = ctypes.c_void_p()
    assert lib.kvc_create(ctypes.byref(ctx), ctypes.byref(_cfg()), 256, pool - 1, 512, meta,
                          None) == -1
    assert lib.kvc_create(ctypes.byref(ctx), ctypes.byref(_cfg()), 258, pool, 512, meta,
                          None) == -1
    assert b"aligned" in lib.kvc_last_error()
    assert lib.kvc_create(None, ctypes.byref(_cfg()), 256, pool, 512, meta, None) == -1


def test_null_context_is_rejected(lib):
    s = (ctypes.c_int32 * 1)(0)
    assert lib.kvc_evict(None, 1, s, None, None) == -1
    assert lib.kvc_attn_decode(None, 0, None, None, None) == -1
    out = ctypes.c_int64()
    assert lib.kvc_resident_size(None, 0, ctypes.byref(out)) == -1
    assert lib.kvc_append_kv_layer(None, 0, None, None, None) == -1
    assert lib.kvc_export_transcript(None, 0, 0, None, None, None, None, None) == -1
    assert lib.kvc_last_error()
    lib.kvc_destroy(None)


def test_policy_fields_are_validated(lib):
    pool, meta = ctypes.c_size_t(), ctypes.c_size_t()
    for bad in ({"policy": 3}, {"policy": -1}, {"policy": 2, "sink": -1},
                {"policy": 2, "recent": -5}):
        assert lib.kvc_query_sizes(ctypes.byref(_cfg(**bad)), ctypes.byref(pool),
                                   ctypes.byref(meta)) == -1
        assert b"policy" in lib.kvc_last_error() or b"sink" in lib.kvc_last_error()
    for good in ({"policy": 1}, {"policy": 2, "sink": 4, "recent": 2000}):
        assert lib.kvc_query_sizes(ctypes.byref(_cfg(**good)), ctypes.byref(pool),
                                   ctypes.byref(meta)) == 0


def test_synth_generator_builds():
    from synth import gpu
    assert os.path.exists(gpu.build())
