"""Total orders for ranking decisions (ties broken by lowest index).

Every selection in the three methods of Section 2.1 (H2O keeps the tokens
with the highest accumulated score; SnapKV keeps the tokens with the highest
pooled window score; the sparse-attention stage keeps the best pages) is a
top-k under the order "value descending, index ascending".  Eviction of the
single lowest-scored token is the last element under that same order.
"""
from __future__ import annotations

import numpy as np


def rank_desc(values, index) -> np.ndarray:
    """Permutation sorting by (value desc, index asc)."""
    values = np.asarray(values, dtype=np.float64)
    index = np.asarray(index)
    return np.lexsort((index, -values))


def topk_desc(values, index, k: int) -> np.ndarray:
    """The k best entries of ``index`` under (value desc, index asc), ascending."""
    if k <= 0:
        return np.zeros(0, dtype=np.asarray(index).dtype)
    perm = rank_desc(values, index)
    return np.sort(np.asarray(index)[perm[:k]])


def last_desc(values, index):
    """The entry of ``index`` that ranks last under (value desc, index asc):
    the lowest value; among equal lowest values, the highest index."""
    perm = rank_desc(values, index)
    return np.asarray(index)[perm[-1]]
