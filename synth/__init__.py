"""Seeded synthetic inputs shared by the CUDA path, the oracle and the bench.

This module draws random tensors and holds none of the method's arithmetic:
no attention, rotation, quantization or selection happens here.  Every tensor
is a pure function of ``(seed, tensor id)``.

Small cases use numpy's counter-based Philox generator (host arrays, fp16).
Full-size workloads use ``torch.Generator`` on the device (same recipe, drawn
where the data lives); the oracle then reads back the slices it checks.

Recipes (the workloads of the evaluation, Section 3.1, made long-context):

* plain: K, V, q ~ N(0, 1) rounded to fp16.
* key outlier channels: selected key channels multiplied by a factor
  (``x10`` on the four lowest channels for the tiny all-configs case).
* per-channel key scale: each (layer, kv-head, channel) key channel is
  multiplied by a scale drawn log-uniform in [0.1, 10].
* heavy hitters: a fraction of positions gets ``k += beta * u_g`` and every
  query gets ``q += alpha * u_g`` with ``u_g`` a fixed unit vector per kv-head;
  with ``alpha * beta / sqrt(D) = ln 20`` such a key draws about 20x the
  attention mass of a plain one.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

# Tensor ids: one stream per tensor kind, so adding a tensor never shifts others.
TID_K, TID_V, TID_Q, TID_QP, TID_KSCALE, TID_HEAVY_POS, TID_HEAVY_DIR, TID_KNEW, TID_VNEW = range(1, 10)


def philox(seed: int, tid: int) -> np.random.Generator:
    """Counter-based Philox4x64 stream keyed by (seed, tensor id)."""
    return np.random.Generator(np.random.Philox(key=(int(seed) << 20) | int(tid)))


def normal_f16(shape, seed: int, tid: int) -> np.ndarray:
    """N(0,1) draws rounded to fp16 (round-to-nearest-even by numpy)."""
    return philox(seed, tid).standard_normal(size=shape).astype(np.float16)


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shapes and method parameters of one synthetic decode workload."""
    name: str
    B: int
    L: int
    Hq: int
    Hkv: int
    D: int
    T: int                      # prompt (prefilled context) length
    steps: int                  # decode steps
    theta: float = 10000.0
    # KVQuant
    bits: int = 4
    quant_mode: str = "uniform"  # "uniform" | "nuq"
    outlier_frac: float = 0.01
    key_outlier_channels: tuple = ()
    key_outlier_factor: float = 1.0
    key_scale_loguniform: tuple | None = None   # (lo, hi) per-channel key scale
    # H2O
    h2o_heavy: int = 0
    h2o_recent: int = 0
    # RocketKV
    snap_window: int = 0
    snap_pool: int = 7
    snap_keep: int = 0
    page: int = 16
    topk_pages: int = 0
    topq_dims: int = 0
    # heavy-hitter structure
    heavy_frac: float = 0.0
    heavy_boost: float = 20.0

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def heavy_alpha(self) -> float:
        """alpha = beta with alpha*beta/sqrt(D) = ln(boost)."""
        return math.sqrt(math.log(self.heavy_boost) * math.sqrt(self.D))


def tiny() -> Workload:
    """The tiny all-configs case: 1 layer, GQA 8/2, D=64, T=512, 16 steps."""
    return Workload(name="tiny", B=1, L=1, Hq=8, Hkv=2, D=64, T=512, steps=16,
                    bits=4, quant_mode="uniform", outlier_frac=0.01,
                    key_outlier_channels=(0, 1, 2, 3), key_outlier_factor=10.0,
                    h2o_heavy=64, h2o_recent=64,
                    snap_window=16, snap_pool=7, snap_keep=256, page=16,
                    topk_pages=8, topq_dims=16)


def kvquant_8k(bits: int = 4) -> Workload:
    """KVQuant decode at 32/8/128 GQA, 32 layers, B=8, T=8192, NUQ codebooks."""
    return Workload(name=f"kvquant_nuq{bits}_b8_t8192", B=8, L=32, Hq=32, Hkv=8, D=128,
                    T=8192, steps=128, bits=bits, quant_mode="nuq", outlier_frac=0.01,
                    key_scale_loguniform=(0.1, 10.0))


def h2o_16k(budget_pct: int = 20) -> Workload:
    """H2O decode at 32/8/128, 32 layers, B=16, T=16384, budget split heavy/recent."""
    T = 16384
    half = int(math.floor(budget_pct / 200.0 * T))
    return Workload(name=f"h2o{budget_pct}_b16_t16384", B=16, L=32, Hq=32, Hkv=8, D=128,
                    T=T, steps=256, h2o_heavy=half, h2o_recent=half,
                    heavy_frac=0.05, heavy_boost=20.0)


def rocket_32k(budget: int = 1024) -> Workload:
    """RocketKV-style decode at 32/8/128, 32 layers, B=4, T=32768, keep 4096."""
    return Workload(name=f"rocket{budget}_b4_t32768", B=4, L=32, Hq=32, Hkv=8, D=128,
                    T=32768, steps=256, snap_window=32, snap_pool=7,
                    snap_keep=min(32768, 4 * budget), page=16, topk_pages=budget // 16,
                    topq_dims=32, heavy_frac=0.05, heavy_boost=20.0)


# ----------------------------------------------------------------------------
# host (numpy) generation, for cases the oracle runs whole
# ----------------------------------------------------------------------------

def host_inputs(w: Workload, seed: int) -> dict:
    """All tensors of a workload as fp16 numpy arrays (small cases only).

    Keys: k [L,B,Hkv,T+steps,D] (prompt tokens then the appended ones; for
    KVQuant these are pre-rotation keys, for the other methods post-rotation
    keys), v likewise, q [steps,L,B,Hq,D] decode queries (post-rotation),
    q_prompt [L,B,Hq,T,D] prompt queries (post-rotation).
    """
    n = w.T + w.steps
    k = normal_f16((w.L, w.B, w.Hkv, n, w.D), seed, TID_K).astype(np.float32)
    v = normal_f16((w.L, w.B, w.Hkv, n, w.D), seed, TID_V)
    q = normal_f16((w.steps, w.L, w.B, w.Hq, w.D), seed, TID_Q).astype(np.float32)
    qp = normal_f16((w.L, w.B, w.Hq, w.T, w.D), seed, TID_QP).astype(np.float32)
    if w.key_outlier_channels:
        k[..., list(w.key_outlier_channels)] *= w.key_outlier_factor
    if w.key_scale_loguniform is not None:
        lo, hi = w.key_scale_loguniform
        u = philox(seed, TID_KSCALE).random(size=(w.L, 1, w.Hkv, 1, w.D))
        k *= np.exp(np.log(lo) + u * (np.log(hi) - np.log(lo)))
    if w.heavy_frac > 0:
        g = philox(seed, TID_HEAVY_DIR).standard_normal(size=(w.L, 1, w.Hkv, 1, w.D))
        g /= np.linalg.norm(g, axis=-1, keepdims=True)
        heavy = philox(seed, TID_HEAVY_POS).random(size=(w.L, w.B, w.Hkv, n, 1)) < w.heavy_frac
        a = w.heavy_alpha
        k += a * g * heavy
        gq = np.repeat(g, w.G, axis=2)          # [L,1,Hq,1,D]
        q += a * gq[None, :, :, :, 0, :]
        qp += a * gq
    return dict(k=k.astype(np.float16), v=v, q=q.astype(np.float16),
                q_prompt=qp.astype(np.float16))


# ----------------------------------------------------------------------------
# device (torch) generation, for full-size workloads
# ----------------------------------------------------------------------------

def _tgen(seed: int, tid: int, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) << 20) | int(tid))
    return g


def device_layer_inputs(w: Workload, seed: int, layer: int, device="cuda", n_tokens=None,
                        with_prompt_queries: bool = False) -> dict:
    """Tensors of one layer drawn on ``device`` (fp16), same recipe as host_inputs.

    Returns k, v [B,Hkv,n,D] with n = n_tokens or T+steps, and q [steps,B,Hq,D];
    q_prompt [B,Hq,T,D] when asked.  Distinct layers use distinct streams.
    """
    import torch
    n = w.T + w.steps if n_tokens is None else n_tokens
    base = layer * 64
    k = torch.randn((w.B, w.Hkv, n, w.D), generator=_tgen(seed, base + TID_K, device),
                    device=device, dtype=torch.float32)
    v = torch.randn((w.B, w.Hkv, n, w.D), generator=_tgen(seed, base + TID_V, device),
                    device=device, dtype=torch.float32).half()
    q = torch.randn((w.steps, w.B, w.Hq, w.D), generator=_tgen(seed, base + TID_Q, device),
                    device=device, dtype=torch.float32)
    qp = None
    if with_prompt_queries:
        qp = torch.randn((w.B, w.Hq, w.T, w.D), generator=_tgen(seed, base + TID_QP, device),
                         device=device, dtype=torch.float32)
    if w.key_outlier_channels:
        k[..., list(w.key_outlier_channels)] *= w.key_outlier_factor
    if w.key_scale_loguniform is not None:
        lo, hi = w.key_scale_loguniform
        u = torch.rand((1, w.Hkv, 1, w.D), generator=_tgen(seed, base + TID_KSCALE, device),
                       device=device)
        k *= torch.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))
    if w.heavy_frac > 0:
        g = torch.randn((1, w.Hkv, 1, w.D), generator=_tgen(seed, base + TID_HEAVY_DIR, device),
                        device=device)
        g = g / g.norm(dim=-1, keepdim=True)
        heavy = torch.rand((w.B, w.Hkv, n, 1), generator=_tgen(seed, base + TID_HEAVY_POS, device),
                           device=device) < w.heavy_frac
        a = w.heavy_alpha
        k += a * g * heavy
        gq = g.repeat_interleave(w.G, dim=1)    # [1,Hq,1,D]
        q += a * gq[:, :, 0, :].unsqueeze(0)
        if qp is not None:
            qp += a * gq
    out = dict(k=k.half(), v=v, q=q.half())
    if qp is not None:
        out["q_prompt"] = qp.half()
    return out


# ----------------------------------------------------------------------------
# the configuration sweep: every method at four (context, batch) points
# ----------------------------------------------------------------------------

SWEEP_POINTS = ((4096, 32), (16384, 16), (65536, 4), (131072, 1))


def sweep(method: str, level: int, T: int, B: int) -> Workload:
    """One configuration of the sweep at context T and batch B (32/8/128 GQA, 32 layers).

    method "fp16" (level ignored), "kvquant" (level = bits, NUQ, per-channel key scales),
    "h2o" (level = budget percent, split heavy/recent), "rocket" (level = token budget; keep
    min(T, 4 * budget) after prefill, budget / 16 pages attended over 32 of 128 dims)."""
    common = dict(B=B, L=32, Hq=32, Hkv=8, D=128, T=T, steps=64)
    if method == "fp16":
        return Workload(name=f"fp16_b{B}_t{T}", **common)
    if method == "kvquant":
        return Workload(name=f"kvquant_nuq{level}_b{B}_t{T}", bits=level, quant_mode="nuq", outlier_frac=0.01,
                        key_scale_loguniform=(0.1, 10.0), **common)
    if method == "h2o":
        half = int(math.floor(level / 200.0 * T))
        return Workload(name=f"h2o{level}_b{B}_t{T}", h2o_heavy=half, h2o_recent=half, heavy_frac=0.05,
                        heavy_boost=20.0, **common)
    if method == "rocket":
        return Workload(name=f"rocket{level}_b{B}_t{T}", snap_window=32, snap_pool=7, snap_keep=min(T, 4 * level),
                        page=16, topk_pages=level // 16, topq_dims=32, heavy_frac=0.05, heavy_boost=20.0, **common)
    raise ValueError(method)


SWEEP_CONFIGS = (("fp16", 0), ("kvquant", 4), ("kvquant", 3), ("kvquant", 2), ("h2o", 10), ("h2o", 20),
                 ("h2o", 40), ("rocket", 1024), ("rocket", 2048), ("rocket", 4096))
