"""O1: softmax attention of one decode query over an attended set (fp64).

Every configuration in Table 1 ends in the same operation: the decode query of
each head attends to the cached keys/values the configuration keeps (all of
them for FP16 and KVQuant, the kept set for H2O, the selected pages for the
sparse-attention stage of RocketKV; Section 2.1).  With grouped-query
attention the G query heads of a group share one key/value head.

    s_h(t)  = scale * q_h . k_t                 scale = 1/sqrt(D) by default
    m_h     = max_t s_h(t)
    l_h     = sum_t exp(s_h(t) - m_h)
    out_h   = sum_t exp(s_h(t) - m_h) v_t / l_h
"""
from __future__ import annotations

import numpy as np


def attend(q, K, V, scale=None):
    """Attention of query rows ``q`` [G, D] over keys ``K`` [n, D], values ``V`` [n, D].

    All inputs are widened exactly to float64.  Returns ``(out [G,D], s [G,n],
    m [G], l [G])``.
    """
    q = np.asarray(q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    if scale is None:
        scale = 1.0 / np.sqrt(q.shape[-1])
    s = scale * (q @ K.T)
    m = s.max(axis=1)
    e = np.exp(s - m[:, None])
    l = e.sum(axis=1)
    out = (e @ V) / l[:, None]
    return out, s, m, l


def probabilities(s, m, l):
    """Softmax probabilities p_h(t) = exp(s_h(t) - m_h) / l_h."""
    return np.exp(s - m[:, None]) / l[:, None]


def decode_gqa(q, K, V, scale=None):
    """Full decode attention for all heads of one batch entry.

    q [Hq, D]; K, V [Hkv, n, D]; query head h reads key/value head h // G.
    Returns out [Hq, D] float64.
    """
    q = np.asarray(q)
    Hq, D = q.shape
    Hkv = K.shape[0]
    G = Hq // Hkv
    out = np.zeros((Hq, D))
    for j in range(Hkv):
        out[j * G:(j + 1) * G] = attend(q[j * G:(j + 1) * G], K[j], V[j], scale)[0]
    return out
