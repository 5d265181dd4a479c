"""Pins for oracle.h2o, oracle.snapkv and oracle.rocket (CPU only).

Brute force on tiny inputs, the limits where each method reduces to full
attention, conservation laws of the accumulated scores, the cross-pin
SnapKV(W=T, pool 1) == H2O prefill scores, torch's max_pool1d, and the
page-score upper bound.
"""
import math

import numpy as np
import torch

from oracle import attention, h2o, rocket, snapkv


def _rand(shape, seed):
    return np.random.default_rng(seed).normal(size=shape).astype(np.float16)


# --------------------------------------------------------------------- H2O

def test_prefill_scores_brute_force():
    G, T, D = 2, 9, 4
    qp, K = _rand((G, T, D), 0), _rand((T, D), 1)
    acc = h2o.prefill_scores(qp, K, block=4)
    ref = [0.0] * T
    for h in range(G):
        for i in range(T):
            w = [math.exp(sum(float(qp[h, i, d]) * float(K[j, d]) for d in range(D)) / 2.0) for j in range(i + 1)]
            z = sum(w)
            for j in range(i + 1):
                ref[j] += w[j] / z
    assert np.allclose(acc, ref, atol=1e-13)
    assert abs(acc.sum() - G * T) < 1e-11          # each causal row sums to one


def test_initial_keep_brute_force():
    rng = np.random.default_rng(2)
    acc = rng.integers(0, 4, size=30).astype(np.float64)      # ties
    keep = h2o.initial_keep(acc, 5, 7)
    rest = sorted(range(23), key=lambda j: (-acc[j], j))[:5]
    assert list(keep) == sorted(rest + list(range(23, 30)))
    assert list(h2o.initial_keep(acc, 20, 20)) == list(range(30))


def _run_h2o(G, T, D, steps, H, R, seed):
    qp, K, V = _rand((G, T, D), seed), _rand((T + steps, D), seed + 1), _rand((T + steps, D), seed + 2)
    q = _rand((steps, G, D), seed + 3)
    st = h2o.from_prefill(qp, K[:T], V[:T], H, R)
    outs, evs, sts = [], [], []
    for s in range(steps):
        out, st, ev, _ = h2o.decode_step(st, q[s], K[T + s], V[T + s], T + s, H, R)
        outs.append(out)
        evs.append(ev)
        sts.append(st)
    return qp, K, V, q, outs, evs, sts


def test_h2o_large_budget_is_full_attention():
    G, T, D, steps = 2, 20, 8, 6
    qp, K, V, q, outs, evs, _ = _run_h2o(G, T, D, steps, 100, 100, 10)
    assert all(e is None for e in evs)
    for s in range(steps):
        ref = attention.attend(q[s], K[:T + s + 1], V[:T + s + 1])[0]
        assert np.array_equal(outs[s], ref)


def test_h2o_invariants_and_brute_force():
    G, T, D, steps, H, R = 2, 24, 6, 10, 4, 5
    qp, K, V, q, outs, evs, sts = _run_h2o(G, T, D, steps, H, R, 20)
    # brute force: recompute every kept token's score from explicit softmax rows
    acc0 = h2o.prefill_scores(qp, K[:T])
    alive = {int(j): acc0[j] for j in h2o.initial_keep(acc0, H, R)}
    for s in range(steps):
        alive[T + s] = 0.0
        toks = sorted(alive)
        for h in range(G):
            logits = [float(np.dot(q[s, h].astype(np.float64), K[t].astype(np.float64))) / math.sqrt(D) for t in toks]
            mx = max(logits)
            w = [math.exp(x - mx) for x in logits]
            z = sum(w)
            for t, wt in zip(toks, w):
                alive[t] += wt / z
        if len(alive) > H + R:
            recent = set(sorted(alive)[-R:])
            cand = [t for t in alive if t not in recent]
            victim = sorted(cand, key=lambda t: (-alive[t], t))[-1]
            assert victim == evs[s]
            del alive[victim]
        st = sts[s]
        assert st.pos.shape[0] == H + R
        assert set(range(T + s + 1 - R, T + s + 1)) <= set(st.pos.tolist())
        for p_, a in zip(st.pos, st.acc):
            assert abs(alive[int(p_)] - a) < 1e-12
    # per step the scores added over the cache sum to G
    st_prev = h2o.from_prefill(qp, K[:T], V[:T], H, R)
    _, st1, ev, _ = h2o.decode_step(st_prev, q[0], K[T], V[T], T, 10**6, 0)
    assert ev is None
    assert abs(st1.acc.sum() - st_prev.acc.sum() - G) < 1e-12


def test_h2o_eviction_tie_evicts_higher_position():
    st = h2o.H2OHead(np.array([0, 1, 2]), np.zeros((3, 2)), np.zeros((3, 2)), np.array([1.0, 1.0, 1.0]))
    # a query orthogonal to every key adds the same probability to all
    _, st2, ev, _ = h2o.decode_step(st, np.array([[0.0, 0.0]]), np.zeros(2), np.zeros(2), 3, 2, 1)
    assert ev == 2


# ------------------------------------------------------------------ SnapKV

def test_snap_window_equal_to_prompt_is_h2o_prefill():
    G, T, D = 2, 40, 8
    qp, K = _rand((G, T, D), 30), _rand((T, D), 31)
    s_all = snapkv.window_scores_all(qp, K)
    assert np.allclose(s_all, h2o.prefill_scores(qp, K), atol=1e-13)
    assert np.array_equal(snapkv.max_pool(s_all, 1), s_all)


def test_snap_scores_sum_and_brute_force():
    G, T, W, D = 2, 30, 5, 4
    qw, K = _rand((G, W, D), 32), _rand((T, D), 33)
    s_all = snapkv.window_scores_all(qw, K)
    assert abs(s_all.sum() - G * W) < 1e-12
    ref = np.zeros(T)
    for h in range(G):
        for i in range(W):
            pos = T - W + i
            w = np.array([math.exp(float(np.dot(qw[h, i].astype(np.float64), K[j].astype(np.float64))) / 2.0) for j in range(pos + 1)])
            ref[:pos + 1] += w / w.sum()
    assert np.allclose(s_all, ref, atol=1e-13)


def test_max_pool_matches_torch():
    s = np.random.default_rng(34).normal(size=101)
    ref = torch.nn.functional.max_pool1d(torch.from_numpy(s)[None, None], 7, 1, 3)[0, 0].numpy()
    assert np.array_equal(snapkv.max_pool(s, 7), ref)


def test_snap_keep_brute_force_and_identity():
    rng = np.random.default_rng(35)
    T, W, keep = 50, 6, 20
    pooled = rng.integers(0, 6, size=T - W).astype(np.float64)
    got = snapkv.keep_positions(pooled, T, W, keep)
    ref = sorted(sorted(range(T - W), key=lambda j: (-pooled[j], j))[:keep - W]) + list(range(T - W, T))
    assert list(got) == ref
    K, V = _rand((T, 4), 36), _rand((T, 4), 37)
    pos, Kc, Vc, _, _ = snapkv.compress(_rand((2, W, 4), 38), K, V, W, 7, T)
    assert list(pos) == list(range(T)) and np.array_equal(Kc, K)


# ------------------------------------------------------------------ Rocket

def test_page_score_upper_bound_full_dims():
    G, n, D, P = 4, 96, 16, 16
    q, K = _rand((G, D), 40).astype(np.float64), _rand((n, D), 41)
    kmin, kmax = rocket.page_minmax(K, P, n // P)
    sc = rocket.page_scores(q, kmin, kmax, np.arange(D))
    for p in range(n // P):
        for t in range(p * P, (p + 1) * P):
            assert sc[p] >= (q @ K[t].astype(np.float64)).sum() - 1e-12


def test_rocket_all_pages_is_full_attention():
    G, n, D, P = 2, 83, 8, 16
    q, K, V = _rand((G, D), 42), _rand((n, D), 43), _rand((n, D), 44)
    out, sel, _ = rocket.decode(q, K, V, n, P, 100, 4)
    assert list(sel) == list(range((n - 1) // P))
    ref = attention.attend(q, K, V)[0]
    assert np.allclose(out, ref, atol=1e-14)   # same set, different summation order


def test_rocket_selection_brute_force():
    G, n, D, P, kp, rd = 3, 16 * 12 + 5, 10, 16, 4, 3
    q, K = _rand((G, D), 45), _rand((n, D), 46)
    sel, sc = rocket.select_pages(q, K, n, P, kp, rd)
    qd = q.astype(np.float64)
    a = [sum(abs(qd[h, i]) for h in range(G)) for i in range(D)]
    dims = sorted(sorted(range(D), key=lambda i: (-a[i], i))[:rd])
    ns = (n - 1) // P
    scores = []
    for p in range(ns):
        pk = K[p * P:(p + 1) * P].astype(np.float64)
        scores.append(sum(max(qd[h, i] * pk[:, i].min(), qd[h, i] * pk[:, i].max()) for h in range(G) for i in dims))
    assert np.allclose(sc, scores, atol=1e-13)
    assert list(sel) == sorted(sorted(range(ns), key=lambda p: (-scores[p], p))[:kp])
    slots = rocket.attended_slots(sel, n, P)
    assert set(range(ns * P, n)) <= set(slots.tolist()) and len(slots) == kp * P + (n - ns * P)


def test_rocket_tail_page_when_newest_completes_a_page():
    assert rocket.n_scored_pages(4097, 16) == 256
    assert rocket.n_scored_pages(4096, 16) == 255      # newest token fills page 255: it is the tail
    assert rocket.n_scored_pages(1, 16) == 0
