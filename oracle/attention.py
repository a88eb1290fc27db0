"""Exact softmax attention over the retained keys, in float64.

For a query row ``q`` (already rotated at its position) and the visible keys
``j``: ``out = sum_j softmax_j(q . k_j / sqrt(D)) v_j``.  The visible keys of
a query at position ``p_q`` are the retained keys with position ``<= p_q``:
everything the eviction policy of Sec. 3.3 kept, plus the causal part of the
chunk that was just fed.  GQA: query head ``h`` reads KV head ``h // G``.
"""
from __future__ import annotations

import numpy as np


def softmax_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, visible: np.ndarray,
                      scale: float) -> np.ndarray:
    """q ``[R][D]``, k ``[N][D]``, v ``[N][Dv]``, visible ``[R][N]`` bool -> ``[R][Dv]``."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    s = (q @ k.T) * scale
    s = np.where(visible, s, -np.inf)
    m = np.max(s, axis=1, keepdims=True)
    p = np.exp(s - m)
    p = np.where(visible, p, 0.0)
    return (p @ v) / np.sum(p, axis=1, keepdims=True)


def gqa_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, q_pos, k_pos) -> np.ndarray:
    """q ``[T][Hq][D]`` at positions ``q_pos``; k, v ``[N][Hkv][D]`` at ``k_pos``.

    Returns ``[T][Hq][D]``.  Key j is visible to query t when ``k_pos[j] <= q_pos[t]``.
    """
    t_len, hq, d = q.shape
    hkv = k.shape[1]
    g = hq // hkv
    visible = np.asarray(k_pos)[None, :] <= np.asarray(q_pos)[:, None]
    out = np.empty((t_len, hq, v.shape[2]), dtype=np.float64)
    for h in range(hq):
        kh = h // g
        out[:, h, :] = softmax_attention(q[:, h, :], k[:, kh, :], v[:, kh, :], visible,
                                         1.0 / np.sqrt(d))
    return out
