"""Host-side checks of the C ABI (no GPU needed).

The library must load, export every entry point include/mkv.h declares, and
reject bad arguments on the host with the documented status codes before
launching anything.
"""
import ctypes
import os
import re

import pytest

import paper_2609_07966_gb300 as mkv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(mkv.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    return mkv.lib()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "mkv.h")).read()
    return sorted(set(re.findall(r"^(?:mkv_status|const char\*)\s+(mkv_\w+)\(", text, re.M)))


def test_exports_every_declared_symbol(L):
    decl = declared_symbols()
    assert len(decl) >= 14
    for name in decl:
        assert hasattr(L, name), name
    assert decl == mkv.exported_symbols()


def _cfg(**kw):
    base = dict(method=mkv.MKV_FP16, B=2, Hq=8, Hkv=2, D=64)
    base.update(kw)
    m = base.pop("method")
    return mkv.config(m, base.pop("B"), base.pop("Hq"), base.pop("Hkv"), base.pop("D"), **base)


def _status(L, cfg, T=128):
    n = ctypes.c_size_t(0)
    return L.mkv_workspace_size(ctypes.byref(cfg) if cfg is not None else None, T, ctypes.byref(n)), n.value


def test_config_validation(L):
    assert _status(L, _cfg())[0] == mkv.MKV_OK
    assert _status(L, None)[0] == mkv.MKV_ERR_INVALID_ARG
    c = _cfg()
    c.abi_version = 99
    assert _status(L, c)[0] == mkv.MKV_ERR_INVALID_ARG
    assert _status(L, _cfg(D=96))[0] == mkv.MKV_ERR_UNSUPPORTED
    assert _status(L, _cfg(Hq=12, Hkv=4))[0] == mkv.MKV_ERR_UNSUPPORTED      # G = 3
    assert _status(L, _cfg(Hq=9, Hkv=2))[0] == mkv.MKV_ERR_INVALID_ARG       # Hq % Hkv
    assert _status(L, _cfg(method=mkv.MKV_KVQUANT, bits=5, outlier_frac=0.01))[0] == mkv.MKV_ERR_UNSUPPORTED
    assert _status(L, _cfg(method=mkv.MKV_KVQUANT, bits=4, outlier_frac=1.5))[0] == mkv.MKV_ERR_INVALID_ARG
    assert _status(L, _cfg(method=mkv.MKV_H2O))[0] == mkv.MKV_ERR_INVALID_ARG  # zero budget
    assert _status(L, _cfg(method=mkv.MKV_ROCKET, topk_pages=8, topq_dims=16, snap_window=16,
                           snap_keep=256, page_size=32))[0] == mkv.MKV_ERR_UNSUPPORTED
    assert "page_size" in mkv.mkv_last_error()


def test_workspace_grows_with_context(L):
    small = _status(L, _cfg(), 256)[1]
    big = _status(L, _cfg(), 65536)[1]
    assert 0 < small <= big


def test_cache_bytes_model():
    cfg = mkv.config(mkv.MKV_FP16, 1, 32, 8, 128)
    res, peak = mkv.mkv_cache_bytes(cfg, 1000)
    assert res == peak == 8 * 1000 * 128 * 2 * 2          # 128 KiB per token over 32 layers
    q4 = mkv.config(mkv.MKV_KVQUANT, 1, 32, 8, 128, bits=4, outlier_frac=0.01)
    r4, p4 = mkv.mkv_cache_bytes(q4, 1000)
    assert 0.25 < r4 / res < 0.35 and p4 == r4 + res
    h = mkv.config(mkv.MKV_H2O, 1, 32, 8, 128, h2o_heavy=100, h2o_recent=100)
    rh, ph = mkv.mkv_cache_bytes(h, 1000)
    assert rh == 8 * 200 * (512 + 8) and ph == rh + res


def test_pointer_checks_reject_before_launch(L):
    cfg = _cfg()
    cache = mkv.mkv_cache()
    cache.T_cap = 128
    st = L.mkv_append_kv(ctypes.byref(cfg), None, None, ctypes.byref(cache), None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    st = L.mkv_decode_attention(ctypes.byref(cfg), None, ctypes.byref(cache), None, None, None, None, 0, None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    cache.T_len = 8
    cache.k = 16
    cache.v = 32
    st = L.mkv_decode_attention(ctypes.byref(cfg), 64, ctypes.byref(cache), None, None, 128, None, 0, None)
    assert st == mkv.MKV_ERR_WORKSPACE
    qcfg = _cfg(method=mkv.MKV_KVQUANT, bits=4, outlier_frac=0.01)
    st = L.mkv_append_kv(ctypes.byref(qcfg), 8, 8, ctypes.byref(cache), None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    st = L.mkv_rope_table(96, 10000.0, 10, 8, None)
    assert st == mkv.MKV_ERR_UNSUPPORTED


def test_rocket_fused_step_checks(L):
    """The fused RocketKV step is ROCKET-only, needs q/out, aligned page bounds, and a cache short
    enough for its shared memory; every rejection happens on the host."""
    rc = mkv.config(mkv.MKV_ROCKET, 1, 32, 8, 128, snap_window=32, snap_pool=7, snap_keep=4096, page_size=16,
                    topk_pages=64, topq_dims=32)
    cache = mkv.mkv_cache()
    cache.T_cap, cache.T_len, cache.k, cache.v, cache.kmin, cache.kmax = 4208, 8, 256, 512, 768, 1024
    st = L.mkv_rocket_decode(ctypes.byref(_cfg()), 64, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    st = L.mkv_rocket_decode(ctypes.byref(rc), None, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    cache.kmin = 770                                   # not 16-byte aligned
    st = L.mkv_rocket_decode(ctypes.byref(rc), 64, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_INVALID_ARG and "aligned" in mkv.mkv_last_error()
    cache.kmin = 768
    cache.T_cap = 1 << 20                              # 65536 pages: beyond the fused step
    st = L.mkv_rocket_decode(ctypes.byref(rc), 64, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_UNSUPPORTED and "mkv_rocket_select" in mkv.mkv_last_error()


def test_rocket_step_checks(L):
    """The one-launch RocketKV step also needs the token's rows, and counts its CTAs in the top
    8 bits of T_len: 8 * Hkv <= 256; every rejection happens on the host."""
    rc = mkv.config(mkv.MKV_ROCKET, 1, 32, 8, 128, snap_window=32, snap_pool=7, snap_keep=4096, page_size=16,
                    topk_pages=64, topq_dims=32)
    cache = mkv.mkv_cache()
    cache.T_cap, cache.T_len, cache.k, cache.v, cache.kmin, cache.kmax = 4208, 8, 256, 512, 768, 1024
    st = L.mkv_rocket_step(ctypes.byref(rc), 64, None, 96, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    st = L.mkv_rocket_step(ctypes.byref(rc), 64, 88, 96, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_INVALID_ARG and "aligned" in mkv.mkv_last_error()
    wide = mkv.config(mkv.MKV_ROCKET, 1, 40, 40, 64, snap_window=32, snap_pool=7, snap_keep=256, page_size=16,
                      topk_pages=4, topq_dims=16)
    cache.T_cap = 256
    st = L.mkv_rocket_step(ctypes.byref(wide), 64, 80, 96, ctypes.byref(cache), None, 128, None)
    assert st == mkv.MKV_ERR_UNSUPPORTED and "8 * Hkv" in mkv.mkv_last_error()


def test_decode_step_checks(L):
    """mkv_decode_step is for FP16 and H2O, needs the token's rows 16-byte aligned and counts its
    CTAs in the top 8 bits of T_len: Hkv x splits <= 255; every rejection happens on the host."""
    fc = mkv.config(mkv.MKV_FP16, 1, 32, 8, 128)
    cache = mkv.mkv_cache()
    cache.T_cap, cache.T_len, cache.k, cache.v = 8192, 8, 256, 512
    big = ctypes.c_size_t(1 << 40)
    st = L.mkv_decode_step(ctypes.byref(fc), 64, None, 96, ctypes.byref(cache), 128, 4096, big, None)
    assert st == mkv.MKV_ERR_INVALID_ARG
    st = L.mkv_decode_step(ctypes.byref(fc), 64, 88, 96, ctypes.byref(cache), 128, 4096, big, None)
    assert st == mkv.MKV_ERR_INVALID_ARG and "aligned" in mkv.mkv_last_error()
    st = L.mkv_decode_step(ctypes.byref(fc), 64, 80, 96, ctypes.byref(cache), 128, 4096, ctypes.c_size_t(16),
                           None)
    assert st == mkv.MKV_ERR_WORKSPACE
    kq = mkv.config(mkv.MKV_KVQUANT, 1, 32, 8, 128, bits=4)
    st = L.mkv_decode_step(ctypes.byref(kq), 64, 80, 96, ctypes.byref(cache), 128, 4096, big, None)
    assert st == mkv.MKV_ERR_INVALID_ARG and "FP16 and H2O" in mkv.mkv_last_error()
    cache.T_cap = 1 << 20                      # 38 splits per unit x 8 kv-heads > 255 CTAs per entry
    st = L.mkv_decode_step(ctypes.byref(fc), 64, 80, 96, ctypes.byref(cache), 128, 4096, big, None)
    assert st == mkv.MKV_ERR_UNSUPPORTED and "splits" in mkv.mkv_last_error()
    cache.T_cap = 1 << 24
    st = L.mkv_decode_step(ctypes.byref(fc), 64, 80, 96, ctypes.byref(cache), 128, 4096, big, None)
    assert st == mkv.MKV_ERR_UNSUPPORTED


def test_kvquant_step_checks(L):
    """mkv_kvquant_step is for KVQUANT, needs its inputs and a workspace, and counts the CTAs that read
    T_len[b] in its top 8 bits (T_cap < 2^24); every rejection happens on the host."""
    kq = mkv.config(mkv.MKV_KVQUANT, 1, 32, 8, 128, bits=4)
    qp = mkv.mkv_quant_params()
    for name in ("t_lo", "t_hi", "k_lo", "k_scale", "k_dq", "v_tbl", "rope"):
        setattr(qp, name, 1 << 20)
    qp.k_cb, qp.v_cb, qp.rope_len = 1 << 20, 1 << 20, 1 << 16
    cache = mkv.mkv_cache()
    cache.T_cap, cache.T_len = 8192, 8
    cache.k_codes, cache.v_codes, cache.v_params, cache.v_out = 1 << 12, 1 << 13, 1 << 14, 1 << 15
    cache.k_out_off, cache.k_out, cache.k_out_cap = 1 << 16, 1 << 17, 4096
    big = ctypes.c_size_t(1 << 40)
    args = lambda cfg, kn: (ctypes.byref(cfg), ctypes.byref(qp), 64, kn, 96, ctypes.byref(cache), 128, 4096, big, None)
    fc = mkv.config(mkv.MKV_FP16, 1, 32, 8, 128)
    assert L.mkv_kvquant_step(*args(fc, 80)) == mkv.MKV_ERR_INVALID_ARG
    assert "KVQUANT" in mkv.mkv_last_error()
    assert L.mkv_kvquant_step(*args(kq, None)) == mkv.MKV_ERR_INVALID_ARG
    st = L.mkv_kvquant_step(ctypes.byref(kq), ctypes.byref(qp), 64, 80, 96, ctypes.byref(cache), 128, 4096,
                            ctypes.c_size_t(16), None)
    assert st == mkv.MKV_ERR_WORKSPACE
    cache.T_cap, qp.rope_len = 1 << 24, 1 << 25
    st = L.mkv_kvquant_step(*args(kq, 80))
    assert st == mkv.MKV_ERR_UNSUPPORTED and "2^24" in mkv.mkv_last_error()



def test_kvquant_step_accepts_the_tested_shapes(L):
    """The host checks of mkv_kvquant_step let the shapes the GPU tests and the bench use through to
    the launch (on a machine without a GPU the launch itself then fails with MKV_ERR_CUDA): many
    one-chunk units per CTA, the 8 x 8K bench shape, a short cache and 128K at B = 1."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("would launch on the GPU")
    for B, Hkv, T_cap in [(40, 4, 64), (8, 8, 8320), (3, 2, 256), (1, 8, 131072 + 200)]:
        kq = mkv.config(mkv.MKV_KVQUANT, B, 4 * Hkv, Hkv, 128, bits=4)
        qp = mkv.mkv_quant_params()
        for name in ("t_lo", "t_hi", "k_lo", "k_scale", "k_dq", "v_tbl", "rope"):
            setattr(qp, name, 1 << 20)
        qp.k_cb, qp.v_cb, qp.rope_len = 1 << 20, 1 << 20, T_cap + 64
        cache = mkv.mkv_cache()
        cache.T_cap, cache.T_len = T_cap, 8
        cache.k_codes, cache.v_codes, cache.v_params, cache.v_out = 1 << 12, 1 << 13, 1 << 14, 1 << 15
        cache.k_out_off, cache.k_out, cache.k_out_cap = 1 << 16, 1 << 17, 4096
        st = L.mkv_kvquant_step(ctypes.byref(kq), ctypes.byref(qp), 64, 80, 96, ctypes.byref(cache), 128, 4096,
                                ctypes.c_size_t(1 << 40), None)
        assert st == mkv.MKV_ERR_CUDA, (B, Hkv, T_cap, st, mkv.mkv_last_error())
