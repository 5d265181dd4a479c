"""O4: H2O heavy-hitter eviction (Section 2.1, H2O paragraph; Table 1).

The paper: H2O tracks, for every cached token, an accumulated attention score
(how much attention the token receives from later tokens) and, once the cache
exceeds its budget, evicts older tokens with the lowest accumulated score; a
setting p% keeps p percent of the prompt's tokens.

Readings where the paper is silent:
* budget = H heavy + R recent tokens, H = R = floor(p/200 * T_prompt)
  (or as given); it stays fixed during decode;
* grouped-query attention: one kept set per kv-head, scored by the sum over
  the G query heads of the group;
* prefill: acc0[j] = sum over the group's heads and all prompt queries i >= j
  of the causal softmax probability p_{h,i}(j) (a column sum);
* initial keep: the R most recent positions plus the top-H of the rest under
  (acc desc, position asc);
* decode step: append the new token (acc 0), attend over the whole cache,
  add sum_h p_h(j) to every cached token's acc, then, while the cache holds
  more than H + R tokens, evict among all but the R most recent positions the
  token that ranks last under (acc desc, position asc): the lowest acc, and on
  an exact tie the higher position.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from . import attention, order


def budget(T_prompt: int, pct: float):
    """(H, R) for an H2O setting keeping pct percent of the prompt."""
    h = int(np.floor(pct / 200.0 * T_prompt))
    return h, h


def prefill_scores(qp, K, scale=None, block: int = 1024):
    """acc0 [T] for one kv-head: causal column sums over the group's heads.

    qp [G, T, D] prompt queries, K [T, D] prompt keys.  Query i attends keys
    0..i.  Rows are visited in blocks only to bound memory.
    """
    qp = np.asarray(qp, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    G, T, D = qp.shape
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    acc = np.zeros(T)
    for h in range(G):
        for i0 in range(0, T, block):
            i1 = min(T, i0 + block)
            s = scale * (qp[h, i0:i1] @ K.T)                       # [rows, T]
            cols = np.arange(T)[None, :]
            rows = np.arange(i0, i1)[:, None]
            s = np.where(cols <= rows, s, -np.inf)
            m = s.max(axis=1, keepdims=True)
            e = np.exp(s - m)
            acc += (e / e.sum(axis=1, keepdims=True)).sum(axis=0)
    return acc


def initial_keep(acc0, H: int, R: int) -> np.ndarray:
    """Kept prompt positions (ascending): R most recent + top-H of the rest."""
    T = acc0.shape[0]
    if H + R >= T:
        return np.arange(T)
    recent = np.arange(T - R, T)
    rest = np.arange(0, T - R)
    heavy = order.topk_desc(acc0[rest], rest, H)
    return np.sort(np.concatenate([heavy, recent]))


@dataclasses.dataclass
class H2OHead:
    """State of one (batch entry, kv-head): kept tokens and their scores."""
    pos: np.ndarray     # [n] int positions
    k: np.ndarray       # [n, D]
    v: np.ndarray       # [n, D]
    acc: np.ndarray     # [n] float64


def from_prefill(qp, K, V, H: int, R: int, scale=None) -> H2OHead:
    acc0 = prefill_scores(qp, K, scale)
    keep = initial_keep(acc0, H, R)
    return H2OHead(keep.copy(), np.asarray(K)[keep], np.asarray(V)[keep], acc0[keep].copy())


def recent_candidates(pos, R: int) -> np.ndarray:
    """Indices (into pos) of tokens that may be evicted: all but the R most recent."""
    if R <= 0:
        return np.arange(pos.shape[0])
    rank = np.argsort(-pos, kind="stable")
    return np.sort(rank[R:])


def decode_step(st: H2OHead, q, k_new, v_new, pos_new: int, H: int, R: int, scale=None,
                forced_victim=None):
    """One decode step.  Returns (out [G,D], new state, evicted position or None,
    the candidate scores used for the eviction decision).

    ``forced_victim`` (a position) replaces the oracle's own eviction choice;
    the parity protocol uses it only after checking that choice is within
    tolerance of a tie.
    """
    pos = np.concatenate([st.pos, [pos_new]])
    k = np.concatenate([st.k, np.asarray(k_new)[None]])
    v = np.concatenate([st.v, np.asarray(v_new)[None]])
    acc = np.concatenate([st.acc, [0.0]])
    out, s, m, l = attention.attend(q, k, v, scale)
    acc = acc + attention.probabilities(s, m, l).sum(axis=0)
    evicted = None
    cand_info = None
    if pos.shape[0] > H + R:
        cand = recent_candidates(pos, R)
        cand_info = (pos[cand].copy(), acc[cand].copy())
        victim = order.last_desc(acc[cand], pos[cand]) if forced_victim is None else forced_victim
        idx = int(np.nonzero(pos == victim)[0][0])
        keep = np.ones(pos.shape[0], bool)
        keep[idx] = False
        evicted = int(victim)
        pos, k, v, acc = pos[keep], k[keep], v[keep], acc[keep]
    return out, H2OHead(pos, k, v, acc), evicted, cand_info
