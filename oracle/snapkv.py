"""O5: SnapKV prefill compression, RocketKV stage 1 (Section 2.1, RocketKV paragraph).

The paper: the first stage uses aggregated attention scores between the input
context and an observation window at the end of the prompt to find and keep
the most relevant tokens.

Readings where the paper is silent:
* the window is the last W prompt positions; window query i (position T-W+i)
  attends causally to keys 0..T-W+i;
* s[j] = sum over the group's G heads and the W window queries of the softmax
  probability of key j, for prefix keys j < T-W;
* pooled[j] = max of s over |j'-j| <= k//2 within the prefix (max-pool,
  stride 1, padding with -inf);
* keep = the top (keep-W) prefix positions under (pooled desc, position asc)
  plus all W window positions, gathered in ascending position order;
  keep >= T keeps everything.
"""
from __future__ import annotations

import numpy as np

from . import order


def window_scores_all(qw, K, scale=None):
    """Column sums [T] over all keys for one kv-head (prefix and window keys).

    qw [G, W, D] window queries at positions T-W..T-1, K [T, D] keys.
    """
    qw = np.asarray(qw, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    G, W, D = qw.shape
    T = K.shape[0]
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    s_all = np.zeros(T)
    for h in range(G):
        s = scale * (qw[h] @ K.T)                          # [W, T]
        rows = (T - W + np.arange(W))[:, None]
        s = np.where(np.arange(T)[None, :] <= rows, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        e = np.exp(s - m)
        s_all += (e / e.sum(axis=1, keepdims=True)).sum(axis=0)
    return s_all


def window_scores(qw, K, scale=None):
    """s [T-W]: the window's aggregated scores of the prefix keys."""
    W = np.asarray(qw).shape[1]
    T = np.asarray(K).shape[0]
    return window_scores_all(qw, K, scale)[: T - W]


def max_pool(s, kernel: int) -> np.ndarray:
    """pooled[j] = max(s[j-r .. j+r]) clipped to the array, r = kernel // 2."""
    s = np.asarray(s, dtype=np.float64)
    n = s.shape[0]
    r = kernel // 2
    return np.array([s[max(0, j - r): min(n, j + r + 1)].max() for j in range(n)])


def keep_positions(pooled, T: int, W: int, keep: int) -> np.ndarray:
    """Kept positions (ascending) given pooled prefix scores [T-W]."""
    if keep >= T:
        return np.arange(T)
    prefix = np.arange(T - W)
    top = order.topk_desc(pooled, prefix, keep - W)
    return np.concatenate([top, np.arange(T - W, T)])


def compress(qw, K, V, W: int, kernel: int, keep: int, scale=None):
    """(kept positions, K[kept], V[kept], s, pooled) for one kv-head."""
    T = K.shape[0]
    if keep >= T:
        pos = np.arange(T)
        return pos, np.asarray(K), np.asarray(V), None, None
    s = window_scores(qw, K, scale)
    pooled = max_pool(s, kernel)
    pos = keep_positions(pooled, T, W, keep)
    return pos, np.asarray(K)[pos], np.asarray(V)[pos], s, pooled
