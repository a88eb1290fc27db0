"""kvc_attn_decode_noalloc: decode attention whose split-K scratch lives in a
fixed array inside the library, for callers that cannot allocate device memory
while they decode (a real-time loop that must not stall on the device
synchronisation an allocation can cause, or an application whose device memory
belongs to another framework).  It must give the same result as
kvc_attn_decode, within the tolerance of the attention parity tests, on calls
made one after another (the array keeps the previous call's contents).

This file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from harness import assert_close  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_31224_gb300 import build
    from synth import gpu
    build.build()
    gpu.build()


def _driver(w, units):
    from synth import script as S
    from synth.driver import Driver
    scripts = S.workload_scripts(w)
    for sc in scripts:
        sc.n_transcript = sc.n_transcript[:units]
        sc.n_text = sc.n_text[:units]
    return Driver(w, scripts)


def _decode_both(drv, c, layer):
    """Existing entry point, then the no-allocation one, on the same queries."""
    lib, ctx = drv.cache.lib, drv.cache.ctx
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    ref = torch.empty_like(c.out)
    got = torch.full_like(c.out, float("nan"))
    assert lib.kvc_attn_decode(ctx, layer, c.q[layer].data_ptr(), ref.data_ptr(), stream) == 0
    rc = lib.kvc_attn_decode_noalloc(ctx, layer, c.q[layer].data_ptr(), got.data_ptr(), stream)
    assert rc == 0, lib.kvc_last_error()
    torch.cuda.synchronize()
    return got.float().cpu().numpy(), ref.float().cpu().numpy()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_noalloc_decode_matches_decode_on_consecutive_calls(dtype):
    from synth import script as S
    if dtype == "bf16":
        w = S.SINGLE_BF16.with_(layers=2, n_sessions=5, offset_max=3, budget=150, window=2,
                                seed=21, turn_period=7, turn_jitter=1)
    else:
        w = S.TINY_F32.with_(n_sessions=3, offset_max=2, budget=120, window=2, seed=22)
    drv = _driver(w, 18)
    compared = 0
    for _ in range(len(drv.sched)):
        st = drv.prepare_step()
        for c in st.calls:
            drv.cache.append_chunk(c.sessions, c.cu, c.types, c.k, c.v)
            if c.kind != "decode":
                continue
            # Two calls in a row (two layers, or the same layer twice), each compared.
            for layer in ([0, w.layers - 1] if w.layers > 1 else [0, 0]):
                got, ref = _decode_both(drv, c, layer)
                assert np.isfinite(got).all()
                assert_close(got, ref, dtype, f"step {st.index} layer {layer}")
                compared += 1
        if st.evict_sessions is not None:
            drv.cache.evict(st.evict_sessions)
    assert compared >= 20


def test_noalloc_decode_rejects_calls_beyond_its_scratch():
    from paper_2609_31224_gb300 import KVCache, KvcError
    # 65 sessions x 64 kv heads = 4160 (session, kv-head) pairs > 4096.
    c = KVCache(n_sessions=65, layers=1, q_heads=256, kv_heads=64, head_dim=128, budget=-1,
                window=0, dtype="bf16", n_pages=80, max_pages_per_session=2, max_positions=8,
                max_seq_per_call=65, max_tokens_per_call=65)
    types = torch.zeros(65, dtype=torch.uint8, device="cuda")
    kv = torch.zeros((1, 65, 64, 128), dtype=torch.bfloat16, device="cuda")
    c.append_chunk(list(range(65)), list(range(66)), types, kv, kv)
    q = torch.zeros((65, 256, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros_like(q)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = c.lib.kvc_attn_decode_noalloc(c.ctx, 0, q.data_ptr(), out.data_ptr(), stream)
    assert rc == -1
    assert b"4096" in c.lib.kvc_last_error()
    c.attn_decode(0, q, out)   # the workspace entry point still serves this call
    torch.cuda.synchronize()
