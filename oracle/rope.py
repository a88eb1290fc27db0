"""Rotary position embedding at original positions, in float64.

Sec. 3.3: position ids advance with every fed token and the kept keys keep
their original rotary positions.  The paper does not name the RoPE variant;
the reading used here is rotate-half (pairs ``(i, i + D/2)``) with
``theta_i = base ** (-2 i / D)`` and angle ``p * theta_i``:

    x'[i]       = x[i] cos(p theta_i) - x[i + D/2] sin(p theta_i)
    x'[i + D/2] = x[i + D/2] cos(p theta_i) + x[i] sin(p theta_i)
"""
from __future__ import annotations

import numpy as np


def inv_freq(head_dim: int, base: float) -> np.ndarray:
    i = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(base), -2.0 * i / head_dim)


def rope(x: np.ndarray, positions, base: float) -> np.ndarray:
    """Rotate ``x[..., D]`` where ``positions`` broadcasts against ``x[..., 0]``."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    ang = np.asarray(positions, dtype=np.float64)[..., None] * inv_freq(d, base)
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)
