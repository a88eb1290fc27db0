"""Counter-based synthetic Q/K/V values (host side, numpy).

Every value is a pure function of its coordinates, so any consumer can
regenerate exactly the element it needs without storing the stream:

    value(seed, tensor, session, layer, pos, head, dim)

Definition (shared bit-for-bit with ``synth/cuda_gen.cu``):

* SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014): ``next()`` adds ``GAMMA`` to the state and
  returns ``mix64(state)``, where ``mix64`` is the variant-13 finaliser.
* Stream base for a tensor: the first SplitMix64 output from the state
  ``(seed << 2) | tag`` (tag 1 = Q, 2 = K, 3 = V).
* Element hash: output number ``idx + 1`` of the stream that starts at that
  base, i.e. ``mix64(base + (idx + 1) * GAMMA)``, with the packed index
  ``idx = session<<42 | layer<<36 | pos<<14 | head<<8 | dim``.
* Irwin-Hall(4) on the four 16-bit fields of the hash: ``S = u0+u1+u2+u3``;
  ``x = fl32(S - 131070) * fl32(sqrt(3)/65536)`` rounded once in binary32.
  ``S - 131070`` is exact in binary32, so the only rounding is the product.
  The result has mean 0 and variance ``1 - 2**-32``.
* Optional per-tensor scale: one more binary32 product (skipped when 1.0).
* Storage: binary32 as is, or bfloat16 by round-to-nearest-even of that
  binary32.

This module holds input generation only: nothing here computes any part of
the eviction policy, the cache layout or attention.
"""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB

TAG_Q, TAG_K, TAG_V = 1, 2, 3

# binary32 bits of sqrt(3)/65536, the scale that gives Irwin-Hall(4) of
# 16-bit uniforms unit variance.
IH_SCALE_F32 = np.float32(np.sqrt(3.0) / 65536.0)
IH_SCALE_BITS = int(IH_SCALE_F32.view(np.uint32))
IH_CENTER = 131070  # 2 * 65535

SESSION_SHIFT, LAYER_SHIFT, POS_SHIFT, HEAD_SHIFT = 42, 36, 14, 8
MAX_SESSION = 1 << 22
MAX_LAYER = 64
MAX_POS = 1 << 22
MAX_HEAD = 64
MAX_DIM = 256


def mix64_int(z: int) -> int:
    """SplitMix64 finaliser on a Python int (mod 2**64)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def splitmix64_stream(state: int, n: int) -> list[int]:
    """The first ``n`` outputs of SplitMix64 started at ``state``."""
    out = []
    for _ in range(n):
        state = (state + GAMMA) & MASK64
        out.append(mix64_int(state))
    return out


def stream_base(seed: int, tag: int) -> int:
    return splitmix64_stream(((seed << 2) | tag) & MASK64, 1)[0]


def _mix64_np(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(MIX1)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(MIX2)
        return z ^ (z >> np.uint64(31))


def packed_index(session, layer, pos, head, dim) -> np.ndarray:
    """Broadcast the five coordinates into the packed 64-bit element index."""
    s = np.asarray(session, dtype=np.uint64)
    l = np.asarray(layer, dtype=np.uint64)
    p = np.asarray(pos, dtype=np.uint64)
    h = np.asarray(head, dtype=np.uint64)
    d = np.asarray(dim, dtype=np.uint64)
    return ((s << np.uint64(SESSION_SHIFT)) | (l << np.uint64(LAYER_SHIFT))
            | (p << np.uint64(POS_SHIFT)) | (h << np.uint64(HEAD_SHIFT)) | d)


def hash64(seed: int, tag: int, idx) -> np.ndarray:
    """Element hashes: output ``idx + 1`` of the tensor's SplitMix64 stream."""
    base = np.uint64(stream_base(seed, tag))
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix64_np(base + (idx + np.uint64(1)) * np.uint64(GAMMA))


def values_f32(seed: int, tag: int, session, layer, pos, head, dim,
               scale: float = 1.0) -> np.ndarray:
    """binary32 values at the broadcast coordinates (before storage rounding)."""
    h = hash64(seed, tag, packed_index(session, layer, pos, head, dim))
    m16 = np.uint64(0xFFFF)
    s = ((h & m16) + ((h >> np.uint64(16)) & m16) + ((h >> np.uint64(32)) & m16)
         + ((h >> np.uint64(48)) & m16)).astype(np.int64)
    x = (s - IH_CENTER).astype(np.float32) * IH_SCALE_F32
    if np.float32(scale) != np.float32(1.0):
        x = x * np.float32(scale)
    return x.astype(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round binary32 to bfloat16 (nearest, ties to even); returns uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (b >> np.uint64(16)) & np.uint64(1)
    r = (b + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def values(seed: int, tag: int, session, layer, pos, head, dim, dtype: str,
           scale: float = 1.0) -> np.ndarray:
    """Stored input values as binary32 numbers (bf16 values are exact in binary32)."""
    x = values_f32(seed, tag, session, layer, pos, head, dim, scale)
    if dtype == "bf16":
        return bf16_bits_to_f32(f32_to_bf16_bits(x))
    if dtype == "f32":
        return x
    raise ValueError(f"unknown dtype {dtype!r}")


def chunk_tensor(seed: int, tag: int, session: int, positions, layers: int, heads: int,
                 head_dim: int, dtype: str, scale: float = 1.0) -> np.ndarray:
    """Values of one session's tokens as ``[layers][len(positions)][heads][head_dim]``."""
    pos = np.asarray(positions, dtype=np.int64)
    l = np.arange(layers)[:, None, None, None]
    p = pos[None, :, None, None]
    h = np.arange(heads)[None, None, :, None]
    d = np.arange(head_dim)[None, None, None, :]
    return values(seed, tag, session, l, p, h, d, dtype, scale)


def layer_tensor(seed: int, tag: int, session: int, layer: int, positions, heads: int,
                 head_dim: int, dtype: str, scale: float = 1.0) -> np.ndarray:
    """Values of one layer for the given positions as ``[len(positions)][heads][head_dim]``."""
    pos = np.asarray(positions, dtype=np.int64)
    p = pos[:, None, None]
    h = np.arange(heads)[None, :, None]
    d = np.arange(head_dim)[None, None, :]
    return values(seed, tag, session, layer, p, h, d, dtype, scale)
