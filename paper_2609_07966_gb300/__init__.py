"""Python binding of libmkv (include/mkv.h): argument marshalling only.

Every function here has the name of the C entry point it calls and forwards
plain integers (device pointers, sizes, a stream handle).  All computation runs
in the CUDA kernels of libmkv.so; if the library is missing this module raises
on first use -- there is no CPU or PyTorch fallback.
"""
from __future__ import annotations

import ctypes
import math
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmkv.so")

MKV_ABI_VERSION = 1
MKV_OK, MKV_ERR_INVALID_ARG, MKV_ERR_UNSUPPORTED, MKV_ERR_CUDA, MKV_ERR_CAPACITY, MKV_ERR_WORKSPACE, \
    MKV_ERR_TIMEOUT = range(7)
MKV_FP16, MKV_KVQUANT, MKV_H2O, MKV_ROCKET = range(4)
MKV_QUANT_UNIFORM, MKV_QUANT_NUQ = range(2)
MKV_FLAG_K_OUTLIER_OVERFLOW = 0x1
MKV_FLAG_CACHE_FULL = 0x2
MKV_FLAG_WAIT_TIMEOUT = 0x4

_STATUS_NAMES = {0: "MKV_OK", 1: "MKV_ERR_INVALID_ARG", 2: "MKV_ERR_UNSUPPORTED", 3: "MKV_ERR_CUDA",
                 4: "MKV_ERR_CAPACITY", 5: "MKV_ERR_WORKSPACE", 6: "MKV_ERR_TIMEOUT"}


class mkv_config(ctypes.Structure):
    _fields_ = [("abi_version", ctypes.c_uint32), ("method", ctypes.c_int32),
                ("B", ctypes.c_int32), ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32), ("D", ctypes.c_int32),
                ("softmax_scale", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("bits", ctypes.c_int32), ("quant_mode", ctypes.c_int32), ("outlier_frac", ctypes.c_float),
                ("h2o_heavy", ctypes.c_int32), ("h2o_recent", ctypes.c_int32),
                ("snap_window", ctypes.c_int32), ("snap_pool", ctypes.c_int32), ("snap_keep", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("topk_pages", ctypes.c_int32), ("topq_dims", ctypes.c_int32)]


class mkv_candidate(ctypes.Structure):
    _fields_ = [("method", ctypes.c_int32), ("level", ctypes.c_int32), ("latency", ctypes.c_double),
                ("memory", ctypes.c_double), ("accuracy", ctypes.c_double)]


class mkv_cache(ctypes.Structure):
    _fields_ = [("T_cap", ctypes.c_int64), ("T_len", ctypes.c_void_p), ("k", ctypes.c_void_p),
                ("v", ctypes.c_void_p), ("pos", ctypes.c_void_p), ("acc", ctypes.c_void_p),
                ("slot", ctypes.c_void_p), ("kmin", ctypes.c_void_p), ("kmax", ctypes.c_void_p),
                ("k_codes", ctypes.c_void_p), ("v_codes", ctypes.c_void_p), ("v_params", ctypes.c_void_p),
                ("v_out", ctypes.c_void_p), ("k_out_off", ctypes.c_void_p), ("k_out", ctypes.c_void_p),
                ("k_out_cap", ctypes.c_int64)]


class mkv_quant_params(ctypes.Structure):
    _fields_ = [("t_lo", ctypes.c_void_p), ("t_hi", ctypes.c_void_p), ("k_lo", ctypes.c_void_p),
                ("k_scale", ctypes.c_void_p), ("k_cb", ctypes.c_void_p), ("v_cb", ctypes.c_void_p),
                ("k_dq", ctypes.c_void_p), ("v_tbl", ctypes.c_void_p), ("rope", ctypes.c_void_p),
                ("rope_len", ctypes.c_int64)]


class MkvError(RuntimeError):
    """A libmkv call returned a status other than MKV_OK."""

    def __init__(self, status: int, call: str, detail: str):
        super().__init__(f"{call} -> {_STATUS_NAMES.get(status, status)}: {detail}")
        self.status = status


_lib = None
_P = ctypes.c_void_p
_CFG = ctypes.POINTER(mkv_config)
_CACHE = ctypes.POINTER(mkv_cache)
_QP = ctypes.POINTER(mkv_quant_params)
_SIGS = {
    "mkv_workspace_size": [_CFG, ctypes.c_int64, ctypes.POINTER(ctypes.c_size_t)],
    "mkv_cache_bytes": [_CFG, ctypes.c_int64, ctypes.POINTER(ctypes.c_size_t), ctypes.POINTER(ctypes.c_size_t)],
    "mkv_rope_table": [ctypes.c_int32, ctypes.c_float, ctypes.c_int64, _P, _P],
    "mkv_get_status": [_P, ctypes.POINTER(ctypes.c_uint32)],
    "mkv_wait_timeout_selftest": [ctypes.c_int32, _P],
    "mkv_append_kv": [_CFG, _P, _P, _CACHE, _P],
    "mkv_decode_attention": [_CFG, _P, _CACHE, _QP, _P, _P, _P, ctypes.c_size_t, _P],
    "mkv_kvquant_calibrate": [_CFG, _P, _P, ctypes.c_int64, ctypes.c_int64, _QP, _P, ctypes.c_size_t, _P],
    "mkv_quant_prepare": [_CFG, _QP, _P],
    "mkv_quantize_kv": [_CFG, _QP, _P, _P, ctypes.c_int64, _CACHE, _P],
    "mkv_h2o_prefill": [_CFG, _P, _P, _P, ctypes.c_int64, _CACHE, _P, ctypes.c_size_t, _P],
    "mkv_h2o_update": [_CFG, _CACHE, _P, ctypes.c_size_t, _P],
    "mkv_snap_compress": [_CFG, _P, _P, _P, ctypes.c_int64, _CACHE, _P, _P, ctypes.c_size_t, _P],
    "mkv_rocket_select": [_CFG, _P, _CACHE, _P, _P],
    "mkv_rocket_decode": [_CFG, _P, _CACHE, _P, _P, _P],
    "mkv_rocket_step": [_CFG, _P, _P, _P, _CACHE, _P, _P, _P],
    "mkv_decode_step": [_CFG, _P, _P, _P, _CACHE, _P, _P, ctypes.c_size_t, _P],
    "mkv_kvquant_step": [_CFG, _QP, _P, _P, _P, _CACHE, _P, _P, ctypes.c_size_t, _P],
    "mkv_select_config": [ctypes.POINTER(mkv_candidate), ctypes.c_int32, ctypes.c_double, ctypes.c_double,
                          ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32)],
    "mkv_decode_attention_noalloc": [_CFG, _P, _CACHE, _P, _P],
}


def lib():
    """Load libmkv.so (built by ``__graft_entry__.build()``); raise if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"libmkv.so is not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, args in _SIGS.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        L.mkv_last_error.restype = ctypes.c_char_p
        L.mkv_last_error.argtypes = []
        _lib = L
    return _lib


def exported_symbols():
    """Names of the ABI entry points declared in include/mkv.h."""
    return sorted(list(_SIGS) + ["mkv_last_error"])


def mkv_last_error() -> str:
    return lib().mkv_last_error().decode()


def _call(name, *args):
    st = getattr(lib(), name)(*args)
    if st != MKV_OK:
        raise MkvError(st, name, mkv_last_error())


def config(method: int, B: int, Hq: int, Hkv: int, D: int, **kw) -> mkv_config:
    """An mkv_config with ABI version set; keyword fields as in mkv.h."""
    c = mkv_config()
    c.abi_version = MKV_ABI_VERSION
    c.method, c.B, c.Hq, c.Hkv, c.D = method, B, Hq, Hkv, D
    c.rope_theta = kw.pop("rope_theta", 10000.0)
    c.page_size = kw.pop("page_size", 16)
    c.snap_pool = kw.pop("snap_pool", 7)
    for k, v in kw.items():
        if not hasattr(c, k):
            raise TypeError(f"mkv_config has no field {k}")
        setattr(c, k, v)
    return c


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(stream)


def mkv_workspace_size(cfg: mkv_config, T_cap: int) -> int:
    n = ctypes.c_size_t(0)
    _call("mkv_workspace_size", ctypes.byref(cfg), T_cap, ctypes.byref(n))
    return n.value


def mkv_cache_bytes(cfg: mkv_config, T: int):
    r, p = ctypes.c_size_t(0), ctypes.c_size_t(0)
    _call("mkv_cache_bytes", ctypes.byref(cfg), T, ctypes.byref(r), ctypes.byref(p))
    return r.value, p.value


def mkv_rope_table(D: int, theta: float, T_max: int, table: int, stream=None):
    _call("mkv_rope_table", D, theta, T_max, table, _stream(stream))


def mkv_get_status(stream=None) -> int:
    """Status-word bits (0 when clean).  Synchronizes the stream."""
    f = ctypes.c_uint32(0)
    st = lib().mkv_get_status(_stream(stream), ctypes.byref(f))
    if st not in (MKV_OK, MKV_ERR_CAPACITY, MKV_ERR_TIMEOUT):
        raise MkvError(st, "mkv_get_status", mkv_last_error())
    return f.value


def mkv_wait_timeout_selftest(ms: int, stream=None):
    """Launch the device wait-timeout diagnostic (include/mkv.h); read the flag with mkv_get_status."""
    _call("mkv_wait_timeout_selftest", ms, _stream(stream))


def mkv_append_kv(cfg, k_new: int, v_new: int, cache: mkv_cache, stream=None):
    _call("mkv_append_kv", ctypes.byref(cfg), k_new, v_new, ctypes.byref(cache), _stream(stream))


def mkv_decode_attention(cfg, q: int, cache: mkv_cache, qparams, page_idx: int, out: int, ws: int,
                         ws_bytes: int, stream=None):
    _call("mkv_decode_attention", ctypes.byref(cfg), q, ctypes.byref(cache),
          ctypes.byref(qparams) if qparams is not None else None, page_idx, out, ws, ws_bytes,
          _stream(stream))


def mkv_decode_attention_noalloc(cfg, q: int, cache: mkv_cache, out: int, stream=None):
    _call("mkv_decode_attention_noalloc", ctypes.byref(cfg), q, ctypes.byref(cache), out, _stream(stream))


def mkv_kvquant_calibrate(cfg, k_cal: int, v_cal: int, N_cal: int, row_stride: int, qparams, ws: int,
                          ws_bytes: int, stream=None):
    _call("mkv_kvquant_calibrate", ctypes.byref(cfg), k_cal, v_cal, N_cal, row_stride, ctypes.byref(qparams),
          ws, ws_bytes, _stream(stream))


def mkv_quant_prepare(cfg, qparams, stream=None):
    _call("mkv_quant_prepare", ctypes.byref(cfg), ctypes.byref(qparams), _stream(stream))


def mkv_quantize_kv(cfg, qparams, k_pre: int, v: int, n_tokens: int, cache: mkv_cache, stream=None):
    _call("mkv_quantize_kv", ctypes.byref(cfg), ctypes.byref(qparams), k_pre, v, n_tokens, ctypes.byref(cache),
          _stream(stream))


def mkv_h2o_prefill(cfg, q_prompt: int, full_k: int, full_v: int, T: int, cache: mkv_cache, ws: int,
                    ws_bytes: int, stream=None):
    _call("mkv_h2o_prefill", ctypes.byref(cfg), q_prompt, full_k, full_v, T, ctypes.byref(cache), ws, ws_bytes,
          _stream(stream))


def mkv_h2o_update(cfg, cache: mkv_cache, ws: int, ws_bytes: int, stream=None):
    _call("mkv_h2o_update", ctypes.byref(cfg), ctypes.byref(cache), ws, ws_bytes, _stream(stream))


def mkv_snap_compress(cfg, q_window: int, full_k: int, full_v: int, T: int, cache: mkv_cache, kept_pos: int,
                      ws: int, ws_bytes: int, stream=None):
    _call("mkv_snap_compress", ctypes.byref(cfg), q_window, full_k, full_v, T, ctypes.byref(cache), kept_pos,
          ws, ws_bytes, _stream(stream))


def mkv_rocket_select(cfg, q: int, cache: mkv_cache, page_idx_out: int, stream=None):
    _call("mkv_rocket_select", ctypes.byref(cfg), q, ctypes.byref(cache), page_idx_out, _stream(stream))


def mkv_rocket_decode(cfg, q: int, cache: mkv_cache, page_idx_out, out: int, stream=None):
    _call("mkv_rocket_decode", ctypes.byref(cfg), q, ctypes.byref(cache), page_idx_out or None, out,
          _stream(stream))


def mkv_decode_step(cfg, q: int, k_new: int, v_new: int, cache: mkv_cache, out: int, ws: int, ws_bytes: int,
                    stream=None):
    _call("mkv_decode_step", ctypes.byref(cfg), q, k_new, v_new, ctypes.byref(cache), out, ws, ws_bytes,
          _stream(stream))


def mkv_kvquant_step(cfg, qparams, q: int, k_new: int, v_new: int, cache: mkv_cache, out: int, ws: int,
                     ws_bytes: int, stream=None):
    _call("mkv_kvquant_step", ctypes.byref(cfg), ctypes.byref(qparams), q, k_new, v_new, ctypes.byref(cache), out,
          ws, ws_bytes, _stream(stream))


def mkv_rocket_step(cfg, q: int, k_new: int, v_new: int, cache: mkv_cache, page_idx_out, out: int, stream=None):
    _call("mkv_rocket_step", ctypes.byref(cfg), q, k_new, v_new, ctypes.byref(cache), page_idx_out or None, out,
          _stream(stream))


def n_value_outliers(D: int, frac: float) -> int:
    import ctypes as _ct
    f32 = _ct.c_float(frac).value
    return min(D, int(math.ceil(f32 * D)))


def mkv_select_config(cands, L_max: float, M_max: float):
    """cands: sequence of (method, level, latency, memory, accuracy).  Returns (index, within_budget)."""
    arr = (mkv_candidate * len(cands))(*[mkv_candidate(int(m), int(lv), float(l), float(mm), float(a))
                                          for (m, lv, l, mm, a) in cands])
    chosen, within = ctypes.c_int32(-1), ctypes.c_int32(-1)
    _call("mkv_select_config", arr, len(cands), float(L_max), float(M_max), ctypes.byref(chosen),
          ctypes.byref(within))
    return chosen.value, bool(within.value)
