"""Device-memory plumbing for libmkv: caches, calibration tables, workspace.

PyTorch only allocates here (torch tensors own the memory); the returned
objects carry the ctypes structs of include/mkv.h pointing into them.
"""
from __future__ import annotations

import dataclasses

from . import (MKV_FP16, MKV_H2O, MKV_KVQUANT, MKV_ROCKET, mkv_cache, mkv_quant_params, mkv_workspace_size,
               n_value_outliers)


@dataclasses.dataclass
class Cache:
    """One layer's cache: torch tensors plus the mkv_cache struct over them."""
    cfg: object
    T_cap: int
    t: dict
    c: mkv_cache


def _ptr(x):
    return 0 if x is None else x.data_ptr()


def alloc_cache(cfg, T_cap: int, device="cuda", k_out_cap: int | None = None) -> Cache:
    """Zeroed cache of T_cap slots for cfg.method (T_len = 0, H2O slots empty)."""
    import torch
    B, Hkv, D = cfg.B, cfg.Hkv, cfg.D
    t = {"T_len": torch.zeros(B, dtype=torch.int32, device=device)}
    if cfg.method in (MKV_FP16, MKV_H2O, MKV_ROCKET):
        t["k"] = torch.zeros((B, Hkv, T_cap, D), dtype=torch.float16, device=device)
        t["v"] = torch.zeros((B, Hkv, T_cap, D), dtype=torch.float16, device=device)
    if cfg.method == MKV_H2O:
        t["pos"] = torch.full((B, Hkv, T_cap), -1, dtype=torch.int32, device=device)
        t["acc"] = torch.zeros((B, Hkv, T_cap), dtype=torch.float32, device=device)
        t["slot"] = torch.zeros((B, Hkv), dtype=torch.int32, device=device)
    if cfg.method == MKV_ROCKET:
        npg = T_cap // 16
        t["kmin"] = torch.zeros((B, Hkv, D, npg), dtype=torch.float16, device=device)
        t["kmax"] = torch.zeros((B, Hkv, D, npg), dtype=torch.float16, device=device)
    if cfg.method == MKV_KVQUANT:
        row = D * cfg.bits // 8
        nv = n_value_outliers(D, cfg.outlier_frac)
        if k_out_cap is None:   # 4x the nominal outlier rate (data beyond the calibration range)
            k_out_cap = int(T_cap * D * min(1.0, max(cfg.outlier_frac, 1e-6) * 4)) + 1024
        t["k_codes"] = torch.zeros((B, Hkv, T_cap, row), dtype=torch.uint8, device=device)
        t["v_codes"] = torch.zeros((B, Hkv, T_cap, row), dtype=torch.uint8, device=device)
        t["v_params"] = torch.zeros((B, Hkv, T_cap, 2), dtype=torch.float32, device=device)
        t["v_out"] = torch.zeros((B, Hkv, T_cap, max(nv, 1)), dtype=torch.int32, device=device)
        t["k_out_off"] = torch.zeros((B, Hkv, T_cap + 1), dtype=torch.int32, device=device)
        t["k_out"] = torch.zeros((B, Hkv, k_out_cap), dtype=torch.int32, device=device)
    c = mkv_cache()
    c.T_cap = T_cap
    for name, _ in mkv_cache._fields_:
        if name in t:
            setattr(c, name, _ptr(t[name]))
    c.k_out_cap = t["k_out"].shape[-1] if "k_out" in t else 0
    return Cache(cfg, T_cap, t, c)


@dataclasses.dataclass
class QuantParams:
    t: dict
    c: mkv_quant_params


def alloc_quant_params(cfg, rope_len: int, device="cuda") -> QuantParams:
    """Calibration tables of one layer (zeros) and a rope table of rope_len rows."""
    import torch
    Hkv, D, K = cfg.Hkv, cfg.D, 1 << cfg.bits
    t = {
        "t_lo": torch.zeros((Hkv, D), dtype=torch.float32, device=device),
        "t_hi": torch.zeros((Hkv, D), dtype=torch.float32, device=device),
        "k_lo": torch.zeros((Hkv, D), dtype=torch.float32, device=device),
        "k_scale": torch.zeros((Hkv, D), dtype=torch.float32, device=device),
        "k_cb": torch.zeros((Hkv, D, K), dtype=torch.float16, device=device),
        "v_cb": torch.zeros((Hkv, D, K), dtype=torch.float16, device=device),
        "k_dq": torch.zeros((Hkv, D, K), dtype=torch.float32, device=device),
        "v_tbl": torch.zeros((Hkv, D, K), dtype=torch.float16, device=device),
        "rope": torch.zeros((rope_len, D // 2, 2), dtype=torch.float32, device=device),
    }
    c = mkv_quant_params()
    for name, _ in mkv_quant_params._fields_:
        if name in t:
            setattr(c, name, _ptr(t[name]))
    c.rope_len = rope_len
    return QuantParams(t, c)


def workspace(cfg, T_cap: int, device="cuda"):
    """(tensor, nbytes) of the workspace mkv_workspace_size asks for, zero-filled
    (its leading counters must start at zero; the library keeps them zero)."""
    import torch
    n = mkv_workspace_size(cfg, T_cap)
    return torch.zeros(n, dtype=torch.uint8, device=device), n
