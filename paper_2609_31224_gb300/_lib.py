"""Thin ctypes binding of ``libkvc.so`` (include/kvc.h).

Argument marshalling only: every step of eviction, compaction and attention
runs in the library's CUDA kernels.  PyTorch provides the device memory
(pool and metadata workspace) and the stream.  There is no fallback: if the
library is missing or the device is not a CUDA GPU, the calls raise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libkvc.so")

KVC_F32, KVC_BF16 = 0, 1
KVC_ACOUSTIC, KVC_ASR_DELIM, KVC_TRANSCRIPT, KVC_TEXT = 0, 1, 2, 3
KVC_UNIT_BEGIN = 0x80
KVC_POLICY_UNIT, KVC_POLICY_POSITION, KVC_POLICY_SINK_RECENT = 0, 1, 2
POLICIES = {"unit": KVC_POLICY_UNIT, "position": KVC_POLICY_POSITION,
            "sink_recent": KVC_POLICY_SINK_RECENT}
STATUS = {0: "KVC_OK", -1: "KVC_EINVAL", -2: "KVC_ENOMEM", -3: "KVC_ECUDA", -4: "KVC_ESTATE",
          -5: "KVC_EDEVICE"}

EXPORTED = ["kvc_query_sizes", "kvc_create", "kvc_destroy", "kvc_append_chunk",
            "kvc_append_kv_layer", "kvc_evict",
            "kvc_attn_prefill_chunk", "kvc_attn_prefill_chunk_kv", "kvc_attn_decode",
            "kvc_attn_decode_kv",
            "kvc_attn_decode_noalloc",
            "kvc_resident_size", "kvc_release",
            "kvc_export_state", "kvc_export_kv", "kvc_export_transcript", "kvc_device_status",
            "kvc_last_error"]


class KvcError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS.get(code, code)}: {msg}")
        self.code = code


class Config(ctypes.Structure):
    _fields_ = [("n_sessions", ctypes.c_int32), ("layers", ctypes.c_int32),
                ("q_heads", ctypes.c_int32), ("kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("budget", ctypes.c_int64), ("window", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("rope_base", ctypes.c_double),
                ("n_pages", ctypes.c_int64), ("max_pages_per_session", ctypes.c_int32),
                ("max_positions", ctypes.c_int32), ("max_seq_per_call", ctypes.c_int32),
                ("max_tokens_per_call", ctypes.c_int32), ("policy", ctypes.c_int32),
                ("sink", ctypes.c_int32), ("recent", ctypes.c_int32)]


class SessionInfo(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "pos_next", "unit_cur", "n_hist", "n_hist_pages", "live_head", "n_live",
        "n_live_pages", "resident", "n_evicted", "peak_resident")]


_lib = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libkvc.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2609_31224_gb300.build.build()")
    lib = ctypes.CDLL(path)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    p_i32 = ctypes.POINTER(ctypes.c_int32)
    lib.kvc_query_sizes.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(ctypes.c_size_t),
                                    ctypes.POINTER(ctypes.c_size_t)]
    lib.kvc_create.argtypes = [ctypes.POINTER(vp), ctypes.POINTER(Config), vp, ctypes.c_size_t,
                               vp, ctypes.c_size_t, vp]
    lib.kvc_destroy.argtypes = [vp]
    lib.kvc_destroy.restype = None
    lib.kvc_append_chunk.argtypes = [vp, ctypes.c_int, p_i32, p_i32, vp, vp, vp, vp]
    lib.kvc_append_kv_layer.argtypes = [vp, ctypes.c_int, vp, vp, vp]
    lib.kvc_evict.argtypes = [vp, ctypes.c_int, p_i32, vp, vp]
    lib.kvc_attn_prefill_chunk.argtypes = [vp, ctypes.c_int, vp, vp, vp]
    lib.kvc_attn_decode.argtypes = [vp, ctypes.c_int, vp, vp, vp]
    lib.kvc_attn_decode_kv.argtypes = [vp, ctypes.c_int, vp, vp, vp, vp, vp]
    lib.kvc_attn_prefill_chunk_kv.argtypes = [vp, ctypes.c_int, vp, vp, vp, vp, vp]
    lib.kvc_attn_decode_noalloc.argtypes = [vp, ctypes.c_int, vp, vp, vp]
    lib.kvc_resident_size.argtypes = [vp, ctypes.c_int, ctypes.POINTER(i64)]
    lib.kvc_release.argtypes = [vp, ctypes.c_int, p_i32, vp]
    lib.kvc_export_state.argtypes = [vp, ctypes.c_int, ctypes.POINTER(SessionInfo), p_i32, p_i32,
                                     p_i32, ctypes.POINTER(ctypes.c_uint8), p_i32, i64]
    lib.kvc_export_kv.argtypes = [vp, ctypes.c_int, ctypes.c_int, vp, vp, i64]
    lib.kvc_export_transcript.argtypes = [vp, ctypes.c_int, i64, vp, vp, vp, vp, vp]
    lib.kvc_device_status.argtypes = [vp, ctypes.POINTER(i64), ctypes.POINTER(i32)]
    lib.kvc_last_error.restype = ctypes.c_char_p
    for name in EXPORTED:
        if name not in ("kvc_destroy", "kvc_last_error"):
            getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def _check(rc: int) -> None:
    if rc != 0:
        raise KvcError(rc, load_library().kvc_last_error().decode())


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _ptr_i32(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def host_i32(a):
    """(array, ctypes pointer) for a host int32 argument; keep the array alive."""
    arr = _i32(a)
    return arr, _ptr_i32(arr)


def _stream(stream):
    import torch
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def query_sizes(cfg: Config) -> tuple[int, int]:
    lib = load_library()
    pool, meta = ctypes.c_size_t(), ctypes.c_size_t()
    _check(lib.kvc_query_sizes(ctypes.byref(cfg), ctypes.byref(pool), ctypes.byref(meta)))
    return pool.value, meta.value


class KVCache:
    """A kvc context over torch-allocated device memory (pool + metadata workspace)."""

    def __init__(self, *, n_sessions: int, layers: int, q_heads: int, kv_heads: int,
                 head_dim: int, budget: int, window: int, dtype: str, n_pages: int,
                 max_pages_per_session: int, max_positions: int, max_seq_per_call: int,
                 max_tokens_per_call: int, page_size: int = 16, rope_base: float = 10000.0,
                 policy: str = "unit", sink: int = 0, recent: int = 0,
                 device: str = "cuda", stream=None):
        import torch
        self.lib = load_library()
        self.cfg = Config(n_sessions, layers, q_heads, kv_heads, head_dim, page_size, budget,
                          window, KVC_BF16 if dtype == "bf16" else KVC_F32, rope_base, n_pages,
                          max_pages_per_session, max_positions, max_seq_per_call,
                          max_tokens_per_call, POLICIES[policy], sink, recent)
        self.dtype = dtype
        self.torch_dtype = torch.bfloat16 if dtype == "bf16" else torch.float32
        pool_bytes, meta_bytes = query_sizes(self.cfg)
        self.pool = torch.empty(pool_bytes, dtype=torch.uint8, device=device)
        self.meta = torch.empty(meta_bytes, dtype=torch.uint8, device=device)
        self.ctx = ctypes.c_void_p()
        _check(self.lib.kvc_create(ctypes.byref(self.ctx), ctypes.byref(self.cfg),
                                   self.pool.data_ptr(), pool_bytes, self.meta.data_ptr(),
                                   meta_bytes, _stream(stream)))

    def close(self) -> None:
        if getattr(self, "ctx", None) and self.ctx.value:
            self.lib.kvc_destroy(self.ctx)
            self.ctx = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- hot path, raw form: pointers and stream handle as Python ints ------------------
    # For per-token loops where tensor indexing and stream lookup would dominate:
    # ``sess_p`` / ``cu_p`` are ctypes int32 pointers (see ``host_i32``), the rest
    # are device addresses and a cudaStream_t value.
    def append_chunk_raw(self, n_seq, sess_p, cu_p, types_ptr, k_ptr, v_ptr, stream) -> None:
        rc = self.lib.kvc_append_chunk(self.ctx, n_seq, sess_p, cu_p, types_ptr, k_ptr, v_ptr,
                                       stream)
        if rc:
            _check(rc)

    def attn_decode_raw(self, layer, q_ptr, out_ptr, stream) -> None:
        rc = self.lib.kvc_attn_decode(self.ctx, layer, q_ptr, out_ptr, stream)
        if rc:
            _check(rc)

    def attn_prefill_kv_raw(self, layer, k_ptr, v_ptr, q_ptr, out_ptr, stream) -> None:
        rc = self.lib.kvc_attn_prefill_chunk_kv(self.ctx, layer, k_ptr, v_ptr, q_ptr, out_ptr,
                                                stream)
        if rc:
            _check(rc)

    def attn_decode_kv_raw(self, layer, k_ptr, v_ptr, q_ptr, out_ptr, stream) -> None:
        rc = self.lib.kvc_attn_decode_kv(self.ctx, layer, k_ptr, v_ptr, q_ptr, out_ptr, stream)
        if rc:
            _check(rc)

    def attn_prefill_raw(self, layer, q_ptr, out_ptr, stream) -> None:
        rc = self.lib.kvc_attn_prefill_chunk(self.ctx, layer, q_ptr, out_ptr, stream)
        if rc:
            _check(rc)

    # -- hot path -------------------------------------------------------------------
    def append_chunk(self, sessions, cu_tokens, types, k, v, stream=None) -> None:
        s, cu = _i32(sessions), _i32(cu_tokens)
        _check(self.lib.kvc_append_chunk(self.ctx, len(s), _ptr_i32(s), _ptr_i32(cu),
                                         types.data_ptr(), None if k is None else k.data_ptr(),
                                         None if v is None else v.data_ptr(), _stream(stream)))

    def append_kv_layer(self, layer: int, k, v, stream=None) -> None:
        """One layer's K/V [total][Hkv][D] of the last append (after an append without K/V)."""
        _check(self.lib.kvc_append_kv_layer(self.ctx, layer, k.data_ptr(), v.data_ptr(),
                                            _stream(stream)))

    def append_kv_layer_raw(self, layer, k_ptr, v_ptr, stream) -> None:
        rc = self.lib.kvc_append_kv_layer(self.ctx, layer, k_ptr, v_ptr, stream)
        if rc:
            _check(rc)

    def evict(self, sessions, resident_out=None, stream=None) -> None:
        s = _i32(sessions)
        _check(self.lib.kvc_evict(self.ctx, len(s), _ptr_i32(s),
                                  None if resident_out is None else resident_out.data_ptr(),
                                  _stream(stream)))

    def attn_prefill_chunk(self, layer: int, q, out, stream=None) -> None:
        _check(self.lib.kvc_attn_prefill_chunk(self.ctx, layer, q.data_ptr(), out.data_ptr(),
                                               _stream(stream)))

    def attn_decode(self, layer: int, q, out, stream=None) -> None:
        _check(self.lib.kvc_attn_decode(self.ctx, layer, q.data_ptr(), out.data_ptr(),
                                        _stream(stream)))

    def release(self, sessions, stream=None) -> None:
        s = _i32(sessions)
        _check(self.lib.kvc_release(self.ctx, len(s), _ptr_i32(s), _stream(stream)))

    # -- synchronising queries -------------------------------------------------------
    def resident_size(self, session: int) -> int:
        out = ctypes.c_int64()
        _check(self.lib.kvc_resident_size(self.ctx, session, ctypes.byref(out)))
        return out.value

    def export_state(self, session: int) -> dict:
        info = SessionInfo()
        cap_p = self.cfg.max_pages_per_session
        _check(self.lib.kvc_export_state(self.ctx, session, ctypes.byref(info), None, None, None,
                                         None, None, 0))
        hist = np.zeros(max(1, cap_p), dtype=np.int32)
        live = np.zeros(max(1, cap_p), dtype=np.int32)
        n = info.resident
        pos = np.zeros(max(1, n), dtype=np.int32)
        typ = np.zeros(max(1, n), dtype=np.uint8)
        unit = np.zeros(max(1, n), dtype=np.int32)
        _check(self.lib.kvc_export_state(self.ctx, session, ctypes.byref(info), _ptr_i32(hist),
                                         _ptr_i32(live), _ptr_i32(pos),
                                         typ.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)),
                                         _ptr_i32(unit), n))
        return {
            "pos_next": info.pos_next, "unit_cur": info.unit_cur, "n_hist": info.n_hist,
            "live_head": info.live_head, "n_live": info.n_live,
            "hist_pages": hist[:info.n_hist_pages].tolist(),
            "live_pages": live[:info.n_live_pages].tolist(), "resident": info.resident,
            "n_evicted": info.n_evicted, "peak_resident": info.peak_resident,
            "pos": pos[:n].tolist(), "type": typ[:n].tolist(), "unit": unit[:n].tolist(),
        }

    def export_kv(self, session: int, layer: int):
        """Stored (rotated) K and V of one layer in retained order, as float32 numpy arrays."""
        n = self.resident_size(session)
        h, d = self.cfg.kv_heads, self.cfg.head_dim
        np_dt = np.uint16 if self.dtype == "bf16" else np.float32
        k = np.zeros((max(1, n), h, d), dtype=np_dt)
        v = np.zeros((max(1, n), h, d), dtype=np_dt)
        _check(self.lib.kvc_export_kv(self.ctx, session, layer, k.ctypes.data, v.ctypes.data, n))
        if self.dtype == "bf16":
            k = (k.astype(np.uint32) << 16).view(np.float32)
            v = (v.astype(np.uint32) << 16).view(np.float32)
        return k[:n], v[:n]

    def export_transcript(self, session: int, cap: int, stream=None):
        """Retained TRANSCRIPT positions of a session (Sec. 4.2), with their stored K and V
        of every layer: device tensors (positions [cap] int32, K and V [L][cap][Hkv][D],
        count [1] int32), filled asynchronously on the stream."""
        import torch
        dev = self.pool.device
        shape = (self.cfg.layers, max(1, cap), self.cfg.kv_heads, self.cfg.head_dim)
        pos = torch.zeros(max(1, cap), dtype=torch.int32, device=dev)
        k = torch.zeros(shape, dtype=self.torch_dtype, device=dev)
        v = torch.zeros(shape, dtype=self.torch_dtype, device=dev)
        count = torch.zeros(1, dtype=torch.int32, device=dev)
        _check(self.lib.kvc_export_transcript(self.ctx, session, cap, pos.data_ptr(), k.data_ptr(),
                                              v.data_ptr(), count.data_ptr(), _stream(stream)))
        return pos, k, v, count

    def device_status(self) -> tuple[int, int]:
        free, err = ctypes.c_int64(), ctypes.c_int32()
        _check(self.lib.kvc_device_status(self.ctx, ctypes.byref(free), ctypes.byref(err)))
        return free.value, err.value
