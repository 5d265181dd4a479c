"""Pins for oracle.attention, oracle.rope and oracle.order (CPU only).

Each pin checks the oracle against something other than itself: a value worked
out by hand, a closed form, brute-force Python loops, or an independent library
routine (torch's fp64 scaled-dot-product attention, complex multiplication).
"""
import math

import numpy as np
import pytest
import torch

from oracle import attention, order, rope


def test_hand_worked_two_token_example():
    # q=[1,0], k0=[1,0], k1=[0,1], scale 1: weights e/(e+1), 1/(e+1).
    out, s, m, l = attention.attend(np.array([[1.0, 0.0]]), np.array([[1.0, 0.0], [0.0, 1.0]]),
                                    np.array([[1.0, 2.0], [3.0, 4.0]]), scale=1.0)
    e = math.e
    assert np.allclose(out[0], [(e * 1 + 3) / (e + 1), (e * 2 + 4) / (e + 1)], rtol=0, atol=1e-15)
    assert m[0] == 1.0 and abs(l[0] - (1 + math.exp(-1))) < 1e-15


def test_brute_force_loops():
    rng = np.random.default_rng(0)
    G, n, D = 3, 7, 5
    q, K, V = rng.normal(size=(G, D)), rng.normal(size=(n, D)), rng.normal(size=(n, D))
    out = attention.attend(q, K, V)[0]
    for h in range(G):
        logits = [sum(q[h, d] * K[t, d] for d in range(D)) / math.sqrt(D) for t in range(n)]
        w = [math.exp(x) for x in logits]
        z = sum(w)
        for d in range(D):
            ref = sum(w[t] * V[t, d] for t in range(n)) / z
            assert abs(out[h, d] - ref) < 1e-13


def test_torch_sdpa_fp64():
    rng = np.random.default_rng(1)
    Hq, Hkv, n, D = 8, 2, 300, 64
    q = rng.normal(size=(Hq, D)).astype(np.float16)
    K = rng.normal(size=(Hkv, n, D)).astype(np.float16)
    V = rng.normal(size=(Hkv, n, D)).astype(np.float16)
    out = attention.decode_gqa(q, K, V)
    G = Hq // Hkv
    Kt = torch.from_numpy(K.astype(np.float64)).repeat_interleave(G, 0)
    Vt = torch.from_numpy(V.astype(np.float64)).repeat_interleave(G, 0)
    qt = torch.from_numpy(q.astype(np.float64))[:, None, :]
    ref = torch.nn.functional.scaled_dot_product_attention(qt, Kt, Vt)[:, 0, :].numpy()
    assert np.abs(out - ref).max() < 1e-12


def test_closed_forms():
    rng = np.random.default_rng(2)
    V = rng.normal(size=(9, 4))
    K = np.tile(rng.normal(size=(1, 4)), (9, 1))          # identical keys -> mean of V
    out = attention.attend(rng.normal(size=(2, 4)), K, V)[0]
    assert np.allclose(out, V.mean(axis=0)[None, :], atol=1e-14)
    K = np.zeros((9, 4))
    K[5, 0] = 1e3                                           # one dominant key -> its value
    out = attention.attend(np.array([[1.0, 0, 0, 0]]), K, V)[0]
    assert np.allclose(out[0], V[5], atol=1e-12)


def test_probabilities_sum_to_one():
    rng = np.random.default_rng(3)
    _, s, m, l = attention.attend(rng.normal(size=(4, 8)), rng.normal(size=(50, 8)), rng.normal(size=(50, 8)))
    assert np.allclose(attention.probabilities(s, m, l).sum(axis=1), 1.0, atol=1e-14)


def test_rope_complex_form():
    # rotate-half == multiplication of (x_i + i x_{i+D/2}) by exp(i p w_i)
    rng = np.random.default_rng(4)
    D, theta = 16, 10000.0
    x = rng.normal(size=(5, D))
    pos = np.array([0, 1, 7, 100, 4095])
    y = rope.apply(x, pos, theta)
    w = np.array([theta ** (-2.0 * i / D) for i in range(D // 2)])
    for r in range(5):
        z = (x[r, :D // 2] + 1j * x[r, D // 2:]) * np.exp(1j * pos[r] * w)
        assert np.allclose(y[r, :D // 2], z.real, atol=1e-12)
        assert np.allclose(y[r, D // 2:], z.imag, atol=1e-12)


def test_rope_invariants():
    rng = np.random.default_rng(5)
    D = 64
    x = rng.normal(size=(3, D))
    assert np.allclose(rope.apply(x, np.zeros(3, int), 10000.0), x, atol=0)
    y = rope.apply(x, np.array([5, 9, 1000]), 10000.0)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), atol=1e-12)
    # relative-position property: <R_m q, R_n k> depends on m - n only
    q, k = rng.normal(size=(1, D)), rng.normal(size=(1, D))
    a = rope.apply(q, np.array([17]), 10000.0) @ rope.apply(k, np.array([5]), 10000.0).T
    b = rope.apply(q, np.array([112]), 10000.0) @ rope.apply(k, np.array([100]), 10000.0).T
    assert abs(a - b).max() < 1e-11
    # D=2, p=1: plain 2x2 rotation by 1 radian
    y = rope.apply(np.array([[1.0, 0.0]]), np.array([1]), 10000.0)
    assert np.allclose(y[0], [math.cos(1.0), math.sin(1.0)], atol=1e-15)


def test_order_against_sorted():
    rng = np.random.default_rng(6)
    vals = rng.integers(0, 5, size=40).astype(np.float64)     # many exact ties
    idx = rng.permutation(100)[:40]
    brute = sorted(zip(vals, idx), key=lambda t: (-t[0], t[1]))
    assert list(order.topk_desc(vals, idx, 11)) == sorted(i for _, i in brute[:11])
    assert order.last_desc(vals, idx) == brute[-1][1]
    assert order.topk_desc(vals, idx, 0).size == 0
