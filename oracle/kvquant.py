"""O3: KVQuant-style b-bit KV cache (Section 2.1, KVQuant paragraph; Table 1).

The paper states the method's intent: keys are quantized per channel, because
outliers concentrate in consistent channels, and outlier values are kept in
uncompressed FP16; a setting is named by its bit width b in {2, 3, 4}.  The
remaining choices are readings of what the paper leaves open:

* keys are quantized before the rotary embedding, per (layer, kv-head,
  channel); values per (token, kv-head);
* key outliers: per channel, with N_cal calibration tokens and
  n_t = ceil(frac/2 * N_cal) per tail (frac taken as an fp32 parameter), t_lo = sorted[n_t] and
  t_hi = sorted[N_cal-1-n_t]; an entry is an outlier iff x < t_lo or x > t_hi;
* value outliers: the n_v = ceil(frac * D) entries of largest |x| per token
  (ties: lower channel first);
* uniform mode: lo/hi = the inlier range, scale = fl32(fl32(hi-lo)/(2^b-1)),
  code = clamp(rint(fl32(fl32(x-lo)/scale)), 0, 2^b-1), every operation a
  correctly rounded fp32 operation; dequant = lo + code*scale;
* non-uniform (NUQ) mode: 2^b centroids per channel from 1-D Lloyd k-means
  (quantile initialisation, 25 iterations, means summed in ascending order in
  fp64, empty clusters keep their centroid), rounded to fp16, sorted, and
  made strictly increasing by one-ulp nudges; code = #{j : x > mu_j} with the
  fp32 midpoints mu_j = fl32(fl32(c_j + c_{j+1}) * 0.5); value centroids act
  on u = fl32(fl32(x - lo_t) / fl32(hi_t - lo_t));
* an outlier keeps a dense code (that of its clamped value), and dequant
  replaces it by the stored fp16 value exactly.

Codes are decided with numpy float32 arithmetic, which is IEEE correctly
rounded and never fused, so they are defined bit for bit.  Dequantized values
and attention are float64.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

from . import attention, rope

F32 = np.float32


def n_cal(T_prompt: int) -> int:
    """Calibration tokens: the first min(T_prompt, 4096) prompt tokens."""
    return min(int(T_prompt), 4096)


def frac32(frac: float) -> float:
    """The outlier fraction is an fp32 parameter; counts use its fp32 value."""
    return float(np.float32(frac))


def n_tail(N: int, frac: float) -> int:
    return int(math.ceil(frac32(frac) / 2.0 * N))


def n_value_outliers(D: int, frac: float) -> int:
    return min(D, int(math.ceil(frac32(frac) * D)))


# ----------------------------------------------------------------------------
# calibration
# ----------------------------------------------------------------------------

def key_thresholds(kcal, frac: float):
    """Per-channel (t_lo, t_hi) fp32 from calibration keys ``kcal`` [N, D] (fp16).

    If 2*n_t >= N every entry is an outlier (t_lo=+inf, t_hi=-inf).
    """
    x = np.asarray(kcal, dtype=np.float16).astype(F32)
    N, D = x.shape
    nt = n_tail(N, frac)
    if 2 * nt >= N:
        return np.full(D, np.inf, F32), np.full(D, -np.inf, F32)
    srt = np.sort(x, axis=0)
    return srt[nt].copy(), srt[N - 1 - nt].copy()


def lloyd_1d(xs_sorted, K: int, iters: int = 25) -> np.ndarray:
    """1-D Lloyd k-means on ascending data; returns K float64 centroids.

    Initial centroid j is the data point at quantile (j + 0.5)/K.  Each
    iteration assigns every point to its nearest centroid (ties: lower index)
    and moves each centroid to the mean of its points (sum taken in ascending
    data order in float64); a centroid with no points keeps its value.
    """
    x = np.asarray(xs_sorted, dtype=np.float64)
    n = x.shape[0]
    if n == 0:
        return np.zeros(K)
    c = np.array([x[min(n - 1, int(math.floor((j + 0.5) * n / K)))] for j in range(K)])
    for _ in range(iters):
        a = np.argmin(np.abs(x[:, None] - c[None, :]), axis=1)
        for j in range(K):
            mem = x[a == j]
            if mem.size:
                c[j] = np.cumsum(mem)[-1] / mem.size
    return c


def finalize_codebook(c) -> np.ndarray:
    """Round centroids to fp16, sort, and make them strictly increasing."""
    c16 = np.sort(np.asarray(c, dtype=np.float64).astype(np.float16))
    for j in range(1, c16.shape[0]):
        if c16[j] <= c16[j - 1]:
            c16[j] = np.nextafter(c16[j - 1], np.float16(np.inf))
    return c16


def midpoints(cb16) -> np.ndarray:
    """fp32 decision midpoints mu_j = fl32(fl32(c_j + c_{j+1}) * 0.5)."""
    c = np.asarray(cb16, dtype=np.float16).astype(F32)
    return ((c[:-1] + c[1:]).astype(F32) * F32(0.5)).astype(F32)


def value_outlier_mask(x16, n_v: int):
    """[n, D] bool: the n_v entries of largest |x| per row (ties: lower channel).

    A stable sort on -|x| keeps equal magnitudes in channel order.
    """
    x = np.asarray(x16, dtype=np.float16).astype(np.float64)
    n, D = x.shape
    mask = np.zeros((n, D), dtype=bool)
    if n_v <= 0:
        return mask
    order = np.argsort(-np.abs(x), axis=1, kind="stable")
    np.put_along_axis(mask, order[:, :n_v], True, axis=1)
    return mask


def value_range(x16, mask):
    """Per-row fp32 (lo, hi) over inliers (0, 0 when a row has no inlier)."""
    x = np.asarray(x16, dtype=np.float16).astype(F32)
    has = (~mask).any(axis=1)
    lo = np.where(mask, F32(np.inf), x).min(axis=1).astype(F32)
    hi = np.where(mask, F32(-np.inf), x).max(axis=1).astype(F32)
    return np.where(has, lo, F32(0)).astype(F32), np.where(has, hi, F32(0)).astype(F32)


def normalized(x16, lo, s):
    """u = fl32(fl32(x - lo) / s) per row (0 where s == 0)."""
    x = np.asarray(x16, dtype=np.float16).astype(F32)
    d = (x - lo[:, None]).astype(F32)
    safe = np.where(s == 0, F32(1), s).astype(F32)
    u = (d / safe[:, None]).astype(F32)
    return np.where((s == 0)[:, None], F32(0), u).astype(F32)


@dataclasses.dataclass
class QuantParams:
    """Calibration of one (layer, kv-head): everything quantize/dequantize read."""
    bits: int
    mode: str                  # "uniform" | "nuq"
    frac: float
    t_lo: np.ndarray           # [D] fp32 key inlier range
    t_hi: np.ndarray           # [D] fp32
    k_lo: np.ndarray           # [D] fp32 (uniform) key offset
    k_scale: np.ndarray        # [D] fp32 (uniform) key step
    k_cb: np.ndarray | None    # [D, 2^b] fp16 (nuq) key centroids
    v_cb: np.ndarray | None    # [D, 2^b] fp16 (nuq) value centroids on u in [0,1]


def calibrate(kcal, vcal, bits: int, mode: str, frac: float) -> QuantParams:
    """Learn one (layer, kv-head)'s parameters from calibration keys/values [N, D]."""
    kcal = np.asarray(kcal, dtype=np.float16)
    vcal = np.asarray(vcal, dtype=np.float16)
    N, D = kcal.shape
    K = 1 << bits
    t_lo, t_hi = key_thresholds(kcal, frac)
    levels = F32(K - 1)
    finite = np.isfinite(t_lo) & np.isfinite(t_hi)
    k_lo = np.where(finite, t_lo, F32(0)).astype(F32)
    k_hi = np.where(finite, t_hi, F32(0)).astype(F32)
    k_scale = ((k_hi - k_lo).astype(F32) / levels).astype(F32)
    k_cb = v_cb = None
    if mode == "nuq":
        x = kcal.astype(F32)
        k_cb = np.zeros((D, K), np.float16)
        for c in range(D):
            col = np.sort(x[:, c])
            inl = col[(col >= t_lo[c]) & (col <= t_hi[c])]
            k_cb[c] = finalize_codebook(lloyd_1d(inl, K))
        mask = value_outlier_mask(vcal, n_value_outliers(D, frac))
        lo, hi = value_range(vcal, mask)
        s = (hi - lo).astype(F32)
        u = normalized(vcal, lo, s)
        v_cb = np.zeros((D, K), np.float16)
        for c in range(D):
            v_cb[c] = finalize_codebook(lloyd_1d(np.sort(u[:, c][~mask[:, c]]), K))
    return QuantParams(bits, mode, frac, t_lo, t_hi, k_lo, k_scale, k_cb, v_cb)


# ----------------------------------------------------------------------------
# quantize / dequantize
# ----------------------------------------------------------------------------

def _uniform_codes(x32, lo, scale, K):
    safe = np.where(scale == 0, F32(1), scale).astype(F32)
    r = ((x32 - lo).astype(F32) / safe).astype(F32)
    code = np.clip(np.rint(r), 0, K - 1)
    return np.where(scale == 0, 0, code).astype(np.int64)


def _nuq_codes(x32, cb16):
    mu = midpoints(cb16)
    return (x32[:, None] > mu[None, :]).sum(axis=1).astype(np.int64)


def quantize_keys(k16, p: QuantParams):
    """Keys [n, D] fp16 -> (codes [n, D] int, outlier mask [n, D] bool)."""
    x = np.asarray(k16, dtype=np.float16).astype(F32)
    n, D = x.shape
    K = 1 << p.bits
    mask = (x < p.t_lo[None, :]) | (x > p.t_hi[None, :])
    if p.mode == "uniform":
        codes = _uniform_codes(x, p.k_lo[None, :], p.k_scale[None, :], K)
    else:
        codes = np.zeros((n, D), np.int64)
        for c in range(D):
            codes[:, c] = _nuq_codes(x[:, c], p.k_cb[c])
    return codes, mask


def dequantize_keys(codes, mask, k16, p: QuantParams):
    """fp64 pre-rotation keys; outliers restored from the fp16 values ``k16``."""
    if p.mode == "uniform":
        deq = p.k_lo.astype(np.float64)[None, :] + codes * p.k_scale.astype(np.float64)[None, :]
    else:
        cb = p.k_cb.astype(np.float64)
        deq = np.take_along_axis(cb[None, :, :].repeat(codes.shape[0], 0), codes[:, :, None], 2)[:, :, 0]
    return np.where(mask, np.asarray(k16, dtype=np.float16).astype(np.float64), deq)


def quantize_values(v16, p: QuantParams):
    """Values [n, D] fp16 -> (codes, outlier mask, lo [n] fp32, scale [n] fp32).

    uniform: scale = fl32(fl32(hi - lo)/(2^b - 1)); nuq: scale = fl32(hi - lo).
    """
    v16 = np.asarray(v16, dtype=np.float16)
    n, D = v16.shape
    K = 1 << p.bits
    mask = value_outlier_mask(v16, n_value_outliers(D, p.frac))
    lo, hi = value_range(v16, mask)
    x = v16.astype(F32)
    if p.mode == "uniform":
        scale = ((hi - lo).astype(F32) / F32(K - 1)).astype(F32)
        codes = _uniform_codes(x, lo[:, None], scale[:, None], K)
    else:
        scale = (hi - lo).astype(F32)
        u = normalized(v16, lo, scale)
        codes = np.zeros((n, D), np.int64)
        for c in range(D):
            codes[:, c] = _nuq_codes(u[:, c], p.v_cb[c])
    return codes, mask, lo, scale


def dequantize_values(codes, mask, lo, scale, v16, p: QuantParams):
    lo64 = lo.astype(np.float64)[:, None]
    sc64 = scale.astype(np.float64)[:, None]
    if p.mode == "uniform":
        deq = lo64 + codes * sc64
    else:
        cb = p.v_cb.astype(np.float64)
        u = np.take_along_axis(cb[None, :, :].repeat(codes.shape[0], 0), codes[:, :, None], 2)[:, :, 0]
        deq = lo64 + sc64 * u
    return np.where(mask, np.asarray(v16, dtype=np.float16).astype(np.float64), deq)


@dataclasses.dataclass
class QuantizedHead:
    """Quantized cache of one (batch entry, kv-head): n tokens at positions 0..n-1."""
    k_codes: np.ndarray
    k_mask: np.ndarray
    k_raw: np.ndarray      # fp16 keys (only read at outlier positions)
    v_codes: np.ndarray
    v_mask: np.ndarray
    v_lo: np.ndarray
    v_scale: np.ndarray
    v_raw: np.ndarray


def quantize_head(k16, v16, p: QuantParams) -> QuantizedHead:
    kc, km = quantize_keys(k16, p)
    vc, vm, lo, sc = quantize_values(v16, p)
    return QuantizedHead(kc, km, np.asarray(k16, np.float16), vc, vm, lo, sc,
                         np.asarray(v16, np.float16))


def decode_head(q, qh: QuantizedHead, p: QuantParams, theta: float, n=None, scale=None):
    """Fused-dequant decode attention of query rows q [G, D] over tokens 0..n-1.

    k_t = rope(dequant_K(t), t), v_t = dequant_V(t).  Returns out [G, D] fp64.
    """
    n = qh.k_codes.shape[0] if n is None else n
    kd = dequantize_keys(qh.k_codes[:n], qh.k_mask[:n], qh.k_raw[:n], p)
    kr = rope.apply(kd, np.arange(n), theta)
    vd = dequantize_values(qh.v_codes[:n], qh.v_mask[:n], qh.v_lo[:n], qh.v_scale[:n], qh.v_raw[:n], p)
    return attention.attend(q, kr, vd, scale)[0]
