"""Pins for oracle.kvquant (CPU only).

Closed-form properties of the quantizer: half-step error bound, nearest
centroid, exact outlier restore, exact outlier counts on distinct data,
k-means on planted clusters, brute-force level search, and two limits of the
fused decode (16-bit codes approach FP16 attention; all-outlier storage equals
it exactly).
"""
import math

import numpy as np

from oracle import attention, kvquant, rope

F32 = np.float32


def _data(n, D, seed, scale_ch=None):
    rng = np.random.default_rng(seed)
    x = rng.normal(size=(n, D))
    if scale_ch is not None:
        x *= scale_ch[None, :]
    return x.astype(np.float16)


def test_uniform_half_step_and_exact_outliers():
    D = 16
    k = _data(600, D, 0, scale_ch=np.geomspace(0.1, 10, D))
    v = _data(600, D, 1)
    for bits in (2, 3, 4):
        p = kvquant.calibrate(k[:512], v[:512], bits, "uniform", 0.01)
        qh = kvquant.quantize_head(k, v, p)
        kd = kvquant.dequantize_keys(qh.k_codes, qh.k_mask, k, p)
        err = np.abs(kd - k.astype(np.float64))
        bound = p.k_scale.astype(np.float64)[None, :] * (0.5 + 1e-6)
        assert np.all(err[~qh.k_mask] <= np.broadcast_to(bound, err.shape)[~qh.k_mask])
        assert np.all(err[qh.k_mask] == 0)
        vd = kvquant.dequantize_values(qh.v_codes, qh.v_mask, qh.v_lo, qh.v_scale, v, p)
        err = np.abs(vd - v.astype(np.float64))
        bound = qh.v_scale.astype(np.float64)[:, None] * (0.5 + 1e-6)
        assert np.all(err[~qh.v_mask] <= np.broadcast_to(bound, err.shape)[~qh.v_mask])
        assert np.all(err[qh.v_mask] == 0)
        assert qh.k_codes.max() <= (1 << bits) - 1 and qh.k_codes.min() >= 0


def test_uniform_codes_brute_force_levels():
    rng = np.random.default_rng(7)
    x = rng.normal(size=2000).astype(np.float16).astype(F32)
    lo, hi = F32(-1.5), F32(2.0)
    for bits in (2, 3, 4):
        L = (1 << bits) - 1
        scale = F32((hi - lo) / F32(L))
        codes = kvquant._uniform_codes(x, lo, scale, L + 1)
        levels = lo + np.arange(L + 1) * np.float64(scale)
        xc = np.clip(x.astype(np.float64), lo, hi)
        d = np.abs(xc[:, None] - levels[None, :])
        best = d.argmin(axis=1)
        near_tie = np.sort(d, axis=1)[:, 1] - np.sort(d, axis=1)[:, 0] < 1e-5 * float(scale)
        assert np.all((codes == best) | near_tie)


def test_outlier_counts_on_distinct_data():
    # distinct values per channel/token -> counts are exact
    N, D, frac = 1000, 8, 0.01
    rng = np.random.default_rng(8)
    k = np.stack([rng.permutation(np.arange(N)) for _ in range(D)], 1).astype(np.float16) / np.float16(8)
    nt = kvquant.n_tail(N, frac)
    t_lo, t_hi = kvquant.key_thresholds(k, frac)
    mask = (k.astype(F32) < t_lo) | (k.astype(F32) > t_hi)
    assert np.all(mask.sum(axis=0) == 2 * nt)          # 2*ceil(0.005*1000) = 10 per channel
    v = np.stack([rng.permutation(np.arange(64)) for _ in range(50)]).astype(np.float16)
    vm = kvquant.value_outlier_mask(v, kvquant.n_value_outliers(64, frac))
    assert np.all(vm.sum(axis=1) == 1)                  # ceil(0.01*64) = 1
    assert kvquant.n_value_outliers(128, 0.01) == 2
    # the value outliers are the entries of largest magnitude
    big = np.argmax(np.abs(v.astype(np.float64)), axis=1)
    assert np.all(vm[np.arange(50), big])


def test_value_outlier_tie_goes_to_lower_channel():
    v = np.array([[3.0, -3.0, 1.0, 3.0]], np.float16)
    vm = kvquant.value_outlier_mask(v, 2)
    assert list(np.nonzero(vm[0])[0]) == [0, 1]


def test_kmeans_recovers_planted_clusters():
    rng = np.random.default_rng(9)
    centers = np.array([-3.0, -1.0, 0.5, 2.5])
    x = np.sort(np.concatenate([c + 0.01 * rng.normal(size=200) for c in centers]))
    c = kvquant.lloyd_1d(x, 4)
    assert np.allclose(np.sort(c), centers, atol=0.01)
    # fixed point: each centroid is the mean of the points nearest to it
    a = np.argmin(np.abs(x[:, None] - c[None, :]), axis=1)
    for j in range(4):
        assert abs(c[j] - x[a == j].mean()) < 1e-12


def test_kmeans_brute_force_two_clusters():
    # for 2 clusters of 1-D data the optimum is the best split of the sorted data;
    # Lloyd from quantile init reaches it on well separated data
    x = np.array([0.0, 0.1, 0.2, 5.0, 5.3, 5.9])
    best = min(range(1, 6), key=lambda s: ((x[:s] - x[:s].mean()) ** 2).sum() + ((x[s:] - x[s:].mean()) ** 2).sum())
    c = kvquant.lloyd_1d(x, 2)
    assert np.allclose(np.sort(c), [x[:best].mean(), x[best:].mean()], atol=1e-15)


def test_finalize_codebook_strictly_increasing():
    cb = kvquant.finalize_codebook([1.0, 1.0, 1.0, 0.5])
    assert cb.dtype == np.float16
    assert np.all(np.diff(cb.astype(np.float64)) > 0)
    assert cb[0] == 0.5 and cb[1] == 1.0
    assert cb[2] == np.nextafter(np.float16(1.0), np.float16(2.0))


def test_nuq_nearest_centroid():
    D = 8
    k = _data(700, D, 10, scale_ch=np.geomspace(0.2, 5, D))
    v = _data(700, D, 11)
    for bits in (2, 3, 4):
        p = kvquant.calibrate(k[:600], v[:600], bits, "nuq", 0.01)
        qh = kvquant.quantize_head(k, v, p)
        kd = kvquant.dequantize_keys(qh.k_codes, qh.k_mask, k, p)
        x = k.astype(np.float64)
        best = np.min(np.abs(x[:, :, None] - p.k_cb.astype(np.float64)[None, :, :]), axis=2)
        got = np.abs(x - kd)
        # nearest up to the fp32 rounding of the decision midpoint
        assert np.all(got[~qh.k_mask] <= best[~qh.k_mask] + 1e-6 * (1 + np.abs(x[~qh.k_mask])))
        assert np.all(got[qh.k_mask] == 0)
        u = kvquant.normalized(v, qh.v_lo, qh.v_scale).astype(np.float64)
        cbv = p.v_cb.astype(np.float64)
        bestu = np.min(np.abs(u[:, :, None] - cbv[None, :, :]), axis=2)
        gotu = np.abs(u - np.take_along_axis(np.broadcast_to(cbv, (u.shape[0], D, 1 << bits)),
                                             qh.v_codes[:, :, None], 2)[:, :, 0])
        assert np.all(gotu[~qh.v_mask] <= bestu[~qh.v_mask] + 1e-6)


def test_nuq_codebook_in_range_and_sorted():
    k = _data(512, 4, 12)
    p = kvquant.calibrate(k, k, 3, "nuq", 0.01)
    for c in range(4):
        cb = p.k_cb[c].astype(np.float64)
        assert np.all(np.diff(cb) > 0)
        assert cb[0] >= p.t_lo[c] - 1e-3 and cb[-1] <= p.t_hi[c] + 1e-3
        assert np.all(p.v_cb[c].astype(np.float64) >= 0) and np.all(p.v_cb[c].astype(np.float64) <= 1.0 + 1e-3)


def _fp16_reference(q, k, v, theta):
    kr = rope.apply(k.astype(np.float64), np.arange(k.shape[0]), theta)
    return attention.attend(q, kr, v.astype(np.float64))[0]


def test_sixteen_bit_approaches_fp16():
    rng = np.random.default_rng(13)
    D, n = 64, 256
    k = _data(n, D, 14)
    v = _data(n, D, 15)
    q = rng.normal(size=(4, D)).astype(np.float16)
    p = kvquant.calibrate(k, v, 16, "uniform", 0.01)
    qh = kvquant.quantize_head(k, v, p)
    out = kvquant.decode_head(q, qh, p, 10000.0)
    ref = _fp16_reference(q, k, v, 10000.0)
    assert np.abs(out - ref).max() < 1e-4
    p4 = kvquant.calibrate(k, v, 4, "uniform", 0.01)
    out4 = kvquant.decode_head(q, kvquant.quantize_head(k, v, p4), p4, 10000.0)
    assert np.abs(out4 - ref).max() > 10 * np.abs(out - ref).max()   # 4-bit is visibly coarser


def test_all_outliers_equals_fp16_exactly():
    rng = np.random.default_rng(16)
    D, n = 32, 100
    k = _data(n, D, 17)
    v = _data(n, D, 18)
    q = rng.normal(size=(2, D)).astype(np.float16)
    for mode in ("uniform", "nuq"):
        p = kvquant.calibrate(k, v, 4, mode, 1.0)
        qh = kvquant.quantize_head(k, v, p)
        assert qh.k_mask.all() and qh.v_mask.all()
        out = kvquant.decode_head(q, qh, p, 10000.0)
        assert np.array_equal(out, _fp16_reference(q, k, v, 10000.0))


def test_calibration_limits():
    assert kvquant.n_cal(512) == 512 and kvquant.n_cal(8192) == 4096
    assert kvquant.n_tail(4096, 0.01) == math.ceil(20.48) == 21


def _values_with_planted_outliers(n, D, seed):
    """N(0,1) values with, per token, two entries pushed far outside the rest (+-40, +-25)."""
    rng = np.random.default_rng(seed)
    v = rng.normal(size=(n, D))
    for t in range(n):
        a, b = rng.choice(D, size=2, replace=False)
        v[t, a] = 40.0 * (1 if rng.random() < 0.5 else -1)
        v[t, b] = 25.0 * (1 if rng.random() < 0.5 else -1)
    return v.astype(np.float16)


def test_value_range_is_the_inlier_range():
    """(lo, hi) of a token = min / max over its entries that are not value outliers, checked
    against a plain loop; with the two planted outliers per token a range over all entries
    would reach +-25..40 and fails here."""
    D, n = 32, 60
    v = _values_with_planted_outliers(n, D, 21)
    mask = kvquant.value_outlier_mask(v, 2)
    lo, hi = kvquant.value_range(v, mask)
    for t in range(n):
        inl = [float(v[t, c]) for c in range(D) if not mask[t, c]]
        assert lo[t] == np.float32(min(inl)) and hi[t] == np.float32(max(inl)), t
        assert hi[t] < 5.0 and lo[t] > -5.0            # the planted outliers are excluded
    # a row whose entries are all outliers has the empty range (0, 0)
    lo1, hi1 = kvquant.value_range(v[:1], np.ones((1, D), bool))
    assert lo1[0] == 0 and hi1[0] == 0


def test_nuq_values_nearest_level_in_value_space():
    """Value-side twin of the key pin: every inlier dequantizes to the nearest of the token's
    levels lo + scale * c_j (up to the fp32 rounding of u and of the decision midpoints), and
    every outlier to its exact fp16 value.  Dropping lo, skipping the de-normalisation or
    taking the range over all entries each breaks this."""
    D, n = 16, 400
    v = _values_with_planted_outliers(n, D, 22)
    k = _data(n, D, 23)
    for bits in (2, 3, 4):
        p = kvquant.calibrate(k[:300], v[:300], bits, "nuq", 0.02)
        qh = kvquant.quantize_head(k, v, p)
        vd = kvquant.dequantize_values(qh.v_codes, qh.v_mask, qh.v_lo, qh.v_scale, v, p)
        x = v.astype(np.float64)
        levels = (qh.v_lo.astype(np.float64)[:, None, None]
                  + qh.v_scale.astype(np.float64)[:, None, None] * p.v_cb.astype(np.float64)[None, :, :])
        best = np.min(np.abs(x[:, :, None] - levels), axis=2)
        got = np.abs(x - vd)
        slack = 1e-6 * (1.0 + qh.v_scale.astype(np.float64))[:, None]
        inl = ~qh.v_mask
        assert np.all(got[inl] <= (best + slack)[inl])
        # the level grid spans the inlier range: no inlier is farther than the widest gap
        assert np.all(got[inl] <= np.broadcast_to(qh.v_scale.astype(np.float64)[:, None], got.shape)[inl])
        assert np.all(got[qh.v_mask] == 0)
        assert qh.v_mask.sum() == kvquant.n_value_outliers(D, 0.02) * n


def test_many_centroid_nuq_approaches_fp16():
    """Many-centroid limit of the NUQ path (oracle only): as the centroids per channel grow from
    2^4 to 2^6 and 2^8 (keys and values), the fused decode approaches FP16 attention, ending
    within 5e-3 of it; a value path that skipped the de-normalisation or dropped lo would stay
    O(1) away at any bit width."""
    rng = np.random.default_rng(24)
    D, n = 32, 1024
    k = _data(n, D, 25, scale_ch=np.geomspace(0.3, 3, D))
    v = _data(n, D, 26)
    q = rng.normal(size=(4, D)).astype(np.float16)
    ref = _fp16_reference(q, k, v, 10000.0)
    errs = []
    for bits in (4, 6, 8):
        p = kvquant.calibrate(k, v, bits, "nuq", 0.01)
        out = kvquant.decode_head(q, kvquant.quantize_head(k, v, p), p, 10000.0)
        errs.append(np.abs(out - ref).max())
    assert errs[0] > errs[1] > errs[2]
    assert errs[2] < 5e-3 and errs[2] * 5 < errs[0]
