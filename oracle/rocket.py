"""O6: RocketKV stage 2, hybrid sparse attention at decode (Section 2.1, RocketKV paragraph).

The paper: at each decoding step attention reads only a subset of the earlier
tokens.  Readings where the paper is silent, in the spirit of a page-level upper
bound on q.k:

* the compressed cache is cut into pages of P consecutive slots; page p's
  metadata is the per-dimension min and max of its (post-rotation) keys;
* dims = the r_d dimensions with the largest a_i = sum_h |q_{h,i}| over the
  group's G heads (ties: lower dimension);
* score_p = sum_h sum_{i in dims} max(q_{h,i} kmin[p,i], q_{h,i} kmax[p,i]);
* candidates: the full pages strictly before the page that holds the current
  (newest) token; the top k_p under (score desc, page asc) are attended, plus
  the tail (the current token's page, 1..P tokens), always.
"""
from __future__ import annotations

import numpy as np

from . import attention, order


def page_minmax(K, page: int, n_pages: int):
    """kmin, kmax [n_pages, D] over slots [p*page, (p+1)*page) of K [n, D]."""
    K = np.asarray(K, dtype=np.float64)
    kmin = np.stack([K[p * page:(p + 1) * page].min(axis=0) for p in range(n_pages)]) if n_pages else np.zeros((0, K.shape[1]))
    kmax = np.stack([K[p * page:(p + 1) * page].max(axis=0) for p in range(n_pages)]) if n_pages else np.zeros((0, K.shape[1]))
    return kmin, kmax


def select_dims(q, r_d: int) -> np.ndarray:
    """The r_d dims with the largest sum_h |q_h,i| (ties: lower dim), ascending."""
    q = np.asarray(q, dtype=np.float64)
    a = np.abs(q).sum(axis=0)
    return order.topk_desc(a, np.arange(q.shape[1]), r_d)


def page_scores(q, kmin, kmax, dims) -> np.ndarray:
    q = np.asarray(q, dtype=np.float64)[:, dims]              # [G, r]
    lo = kmin[:, dims][None, :, :] * q[:, None, :]            # [G, P, r]
    hi = kmax[:, dims][None, :, :] * q[:, None, :]
    return np.maximum(lo, hi).sum(axis=2).sum(axis=0)


def n_scored_pages(n: int, page: int) -> int:
    """Full pages before the page of the newest token (n tokens cached)."""
    return (n - 1) // page


def select_pages(q, K, n: int, page: int, k_p: int, r_d: int):
    """(selected page ids ascending, scores) for a cache of n tokens."""
    ns = n_scored_pages(n, page)
    kmin, kmax = page_minmax(K[:n], page, ns)
    dims = select_dims(q, r_d)
    sc = page_scores(q, kmin, kmax, dims)
    sel = order.topk_desc(sc, np.arange(ns), min(k_p, ns))
    return sel, sc


def attended_slots(sel, n: int, page: int) -> np.ndarray:
    ns = n_scored_pages(n, page)
    toks = [np.arange(p * page, (p + 1) * page) for p in sel]
    toks.append(np.arange(ns * page, n))
    return np.concatenate(toks)


def decode(q, K, V, n: int, page: int, k_p: int, r_d: int, scale=None, forced_pages=None):
    """Sparse decode over compact cache slots 0..n-1 (newest token at n-1).

    Returns (out [G, D], selected pages, scores).  ``forced_pages`` replaces
    the oracle's own selection (parity protocol, after a tie check).
    """
    sel, sc = select_pages(q, K, n, page, k_p, r_d)
    if forced_pages is not None:
        sel = np.sort(np.asarray(forced_pages))
    slots = attended_slots(sel, n, page)
    out = attention.attend(q, np.asarray(K)[slots], np.asarray(V)[slots], scale)[0]
    return out, sel, sc
