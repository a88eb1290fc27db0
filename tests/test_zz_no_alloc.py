"""kvc_attn_decode_noalloc: decode attention whose split-K scratch lives in a
fixed array inside the library, for callers that cannot allocate device memory
while they decode (a real-time loop that must not stall on the device
synchronisation an allocation can cause, or an application whose device memory
belongs to another framework).  It must give the same result as
kvc_attn_decode, within the tolerance of the attention parity tests, on calls
made one after another (the array keeps the previous call's contents), and
match the CPU oracle as the other decode paths do.

This file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from harness import Lockstep, assert_close  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_31224_gb300 import build
    from synth import gpu
    build.build()
    gpu.build()


def _lockstep(w, units):
    from synth import script as S
    from synth.driver import Driver
    scripts = S.workload_scripts(w)
    for sc in scripts:
        sc.n_transcript = sc.n_transcript[:units]
        sc.n_text = sc.n_text[:units]
    return Lockstep(Driver(w, scripts), w)


def _decode_both(drv, c, layer):
    """Existing entry point into a scratch buffer, then the no-allocation one into the
    call's output buffer, on the same queries."""
    lib, ctx = drv.cache.lib, drv.cache.ctx
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    ref = torch.empty_like(c.out)
    c.out.fill_(float("nan"))
    assert lib.kvc_attn_decode(ctx, layer, c.q[layer].data_ptr(), ref.data_ptr(), stream) == 0
    rc = lib.kvc_attn_decode_noalloc(ctx, layer, c.q[layer].data_ptr(), c.out.data_ptr(), stream)
    assert rc == 0, lib.kvc_last_error()
    torch.cuda.synchronize()
    return c.out.float().cpu().numpy(), ref.float().cpu().numpy()


def _run(ls, dtype, layers, oracle_pred):
    """Every step of the lockstep run; each decode call answered by both entry points at
    `layers` (two calls in a row), compared with each other, and the decode calls that
    oracle_pred(index of the decode call, call) selects also compared with the oracle."""
    drv = ls.drv
    compared, n_dec = 0, 0
    for _ in range(len(drv.sched)):
        st = drv.prepare_step()
        for c in st.calls:
            drv.cache.append_chunk(c.sessions, c.cu, c.types, c.k, c.v)
            ls.on_append(c)
            if c.kind != "decode":
                continue
            for layer in layers:
                got, ref = _decode_both(drv, c, layer)
                assert np.isfinite(got).all()
                assert_close(got, ref, dtype, f"step {st.index} layer {layer}")
                if oracle_pred(n_dec, c):
                    ls.compare_call(c, layer, None, f"no-allocation step {st.index}")
                compared += 1
            n_dec += 1
        if st.evict_sessions is not None:
            drv.cache.evict(st.evict_sessions)
            ls.orc.evict(st.evict_sessions.tolist())
    return compared


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_noalloc_decode_matches_decode_and_oracle_on_consecutive_calls(dtype):
    from synth import script as S
    if dtype == "bf16":
        w = S.SINGLE_BF16.with_(layers=2, n_sessions=5, offset_max=3, budget=150, window=2,
                                seed=21, turn_period=7, turn_jitter=1)
        layers = [0, 1]
    else:
        w = S.TINY_F32.with_(n_sessions=3, offset_max=2, budget=120, window=2, seed=22)
        layers = [0, 0]
    ls = _lockstep(w, 18)
    assert _run(ls, dtype, layers, lambda i, c: i % 3 == 0) >= 20
    assert ls.n_compared >= 20


def test_noalloc_decode_single_chunk_calls():
    """Decode rounds of all 120 sessions: 120 x 8 KV heads = 960 (session, KV head) pairs,
    more than four work items per resident CTA (3 x 152), so every pair is one chunk and
    its CTA writes the output directly (no partial state, no merge).  Those calls are
    compared with the oracle; the smaller rounds with the workspace entry point."""
    from synth import script as S
    w = S.SINGLE_BF16.with_(layers=1, n_sessions=120, budget=-1, seed=23, turns=False)
    ls = _lockstep(w, 3)
    assert _run(ls, "bf16", [0, 0], lambda i, c: len(c.sessions) == 120) >= 4
    assert ls.n_compared >= 4 * 120


def test_noalloc_decode_rejects_calls_beyond_its_scratch():
    from paper_2609_31224_gb300 import KVCache
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
