"""GPU parity: KVQuant calibration, quantization (codes bit-exact) and fused decode.

The oracle's calibration is the reference; the GPU's own calibration must
reproduce it bit for bit (same fp32 thresholds, same fp16 centroids), the
GPU quantizer must produce the oracle's codes, outlier sets and per-token
value parameters exactly, and the fused decode must match the oracle's fp64
dequant + rotation + attention within the attention tolerance.
"""
import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
import synth
from oracle import kvquant, rope as orope
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, to_dev, torch_cuda

pytestmark = pytest.mark.gpu


def unpack(rows, D, bits):
    """GPU packed rows [..., D*bits/8] -> codes [..., D] (pair i = channels i, i+D/2)."""
    rows = np.asarray(rows, dtype=np.uint8)
    lead = rows.shape[:-1]
    flat = rows.reshape(-1, rows.shape[-1])
    bitsarr = np.unpackbits(flat, axis=1, bitorder="little")
    out = np.zeros((flat.shape[0], D), np.int64)
    NP = D // 2
    for i in range(NP):
        base = 2 * bits * i
        for k in range(bits):
            out[:, i] |= bitsarr[:, base + k].astype(np.int64) << k
            out[:, i + NP] |= bitsarr[:, base + bits + k].astype(np.int64) << k
    return out.reshape(*lead, D)


def make_cfg(B, Hq, Hkv, D, bits, mode, frac=0.01, theta=10000.0):
    return mkv.config(mkv.MKV_KVQUANT, B, Hq, Hkv, D, bits=bits,
                      quant_mode=mkv.MKV_QUANT_NUQ if mode == "nuq" else mkv.MKV_QUANT_UNIFORM,
                      outlier_frac=frac, rope_theta=theta)


def upload_params(qp, plist, dev):
    import torch
    f = lambda key: torch.from_numpy(np.stack([getattr(p, key) for p in plist]).astype(np.float32)).to(dev)
    qp.t["t_lo"].copy_(f("t_lo"))
    qp.t["t_hi"].copy_(f("t_hi"))
    qp.t["k_lo"].copy_(f("k_lo"))
    qp.t["k_scale"].copy_(f("k_scale"))
    if plist[0].k_cb is not None:
        qp.t["k_cb"].copy_(torch.from_numpy(np.stack([p.k_cb for p in plist])).to(dev))
        qp.t["v_cb"].copy_(torch.from_numpy(np.stack([p.v_cb for p in plist])).to(dev))


def _data(B, Hkv, n, D, seed, key_scale=True, outlier_channels=()):
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((B, Hkv, n, D))
    if key_scale:
        k *= np.exp(rng.uniform(np.log(0.1), np.log(10.0), (1, Hkv, 1, D)))
    for c in outlier_channels:
        k[..., c] *= 10.0
    v = rng.standard_normal((B, Hkv, n, D))
    return k.astype(np.float16), v.astype(np.float16)


def _oracle_params(k, v, Ncal, bits, mode, frac):
    return [kvquant.calibrate(k[0, h, :Ncal], v[0, h, :Ncal], bits, mode, frac) for h in range(k.shape[1])]


@pytest.mark.parametrize("bits,mode,D,N", [(4, "uniform", 64, 512), (2, "nuq", 128, 700),
                                           (3, "nuq", 128, 1024), (4, "nuq", 64, 333)])
def test_calibration_bit_exact(bits, mode, D, N):
    torch = torch_cuda()
    dev = torch.device("cuda")
    Hkv = 2
    k, v = _data(1, Hkv, N + 5, D, seed=bits * 100 + D)
    plist = _oracle_params(k, v, N, bits, mode, 0.01)
    cfg = make_cfg(1, 4 * Hkv, Hkv, D, bits, mode)
    qp = caches.alloc_quant_params(cfg, 64, device=dev)
    ws, nws = caches.workspace(cfg, N + 5, device=dev)
    kd, vd = to_dev(k[0], dev), to_dev(v[0], dev)
    mkv.mkv_kvquant_calibrate(cfg, kd.data_ptr(), vd.data_ptr(), N, N + 5, qp.c, ws.data_ptr(), nws)
    torch.cuda.synchronize()
    for key in ("t_lo", "t_hi") + (("k_lo", "k_scale") if mode == "uniform" else ()):
        ref = np.stack([getattr(p, key) for p in plist]).astype(np.float32)
        got = qp.t[key].cpu().numpy()
        assert np.array_equal(got.view(np.uint32), ref.view(np.uint32)), key
    if mode == "nuq":
        for key in ("k_cb", "v_cb"):
            ref = np.stack([getattr(p, key) for p in plist])
            got = qp.t[key].cpu().numpy()
            bad = (got.view(np.uint16) != ref.view(np.uint16)).sum()
            assert bad == 0, f"{key}: {bad} centroids differ"


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_calibration_bit_exact_bench_size(bits):
    """The bench's calibration: N_cal = 4096 tokens, D = 128, 2^b NUQ centroids per channel, keys with
    per-channel scales log-uniform in [0.1, 10]: thresholds and fp16 centroids bit-exact."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    N, D, Hkv = 4096, 128, 1
    k, v = _data(1, Hkv, N, D, seed=400 + bits)
    plist = _oracle_params(k, v, N, bits, "nuq", 0.01)
    cfg = make_cfg(1, 4 * Hkv, Hkv, D, bits, "nuq")
    qp = caches.alloc_quant_params(cfg, 64, device=dev)
    ws, nws = caches.workspace(cfg, N, device=dev)
    kd, vd = to_dev(k[0], dev), to_dev(v[0], dev)
    mkv.mkv_kvquant_calibrate(cfg, kd.data_ptr(), vd.data_ptr(), N, N, qp.c, ws.data_ptr(), nws)
    torch.cuda.synchronize()
    for key in ("t_lo", "t_hi"):
        ref = np.stack([getattr(p, key) for p in plist]).astype(np.float32)
        assert np.array_equal(qp.t[key].cpu().numpy().view(np.uint32), ref.view(np.uint32)), key
    for key in ("k_cb", "v_cb"):
        ref = np.stack([getattr(p, key) for p in plist])
        bad = (qp.t[key].cpu().numpy().view(np.uint16) != ref.view(np.uint16)).sum()
        assert bad == 0, f"{key}: {bad} centroids differ"


def _quantized_cache(cfg, k, v, plist, T, steps, dev, T_cap=None):
    """Bulk-quantize T tokens, then append `steps` single tokens; returns cache, qparams."""
    torch = torch_cuda()
    T_cap = T_cap or (T + steps + 8)
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    qp = caches.alloc_quant_params(cfg, max(T_cap, 64), device=dev)
    upload_params(qp, plist, dev)
    mkv.mkv_quant_prepare(cfg, qp.c)
    mkv.mkv_rope_table(cfg.D, cfg.rope_theta, qp.c.rope_len, qp.t["rope"].data_ptr())
    kp, vp = to_dev(k[:, :, :T], dev), to_dev(v[:, :, :T], dev)
    mkv.mkv_quantize_kv(cfg, qp.c, kp.data_ptr(), vp.data_ptr(), T, cache.c)
    for s in range(steps):
        kn, vn = to_dev(k[:, :, T + s:T + s + 1], dev), to_dev(v[:, :, T + s:T + s + 1], dev)
        mkv.mkv_quantize_kv(cfg, qp.c, kn.data_ptr(), vn.data_ptr(), 1, cache.c)
    torch.cuda.synchronize()
    assert mkv.mkv_get_status() == 0
    return cache, qp


@pytest.mark.parametrize("bits,mode,D", [(4, "uniform", 64), (2, "nuq", 128), (3, "nuq", 128), (4, "nuq", 128),
                                         (3, "uniform", 64)])
def test_quantize_bit_exact(bits, mode, D):
    torch = torch_cuda()
    dev = torch.device("cuda")
    B, Hkv, T, steps = 2, 2, 300, 5
    k, v = _data(B, Hkv, T + steps, D, seed=bits + D, outlier_channels=(0, 1))
    plist = _oracle_params(k, v, T, bits, mode, 0.01)
    cfg = make_cfg(B, 4 * Hkv, Hkv, D, bits, mode)
    cache, _ = _quantized_cache(cfg, k, v, plist, T, steps, dev)
    n = T + steps
    kc = unpack(cache.t["k_codes"][:, :, :n].cpu().numpy(), D, bits)
    vc = unpack(cache.t["v_codes"][:, :, :n].cpu().numpy(), D, bits)
    vpar = cache.t["v_params"][:, :, :n].cpu().numpy()
    off = cache.t["k_out_off"].cpu().numpy()
    kout = cache.t["k_out"].cpu().numpy().view(np.uint32)
    vout = cache.t["v_out"][:, :, :n].cpu().numpy().view(np.uint32)
    nv = kvquant.n_value_outliers(D, 0.01)
    assert int(cache.t["T_len"][0]) == n
    for b in range(B):
        for h in range(Hkv):
            qh = kvquant.quantize_head(k[b, h, :n], v[b, h, :n], plist[h])
            assert np.array_equal(kc[b, h], qh.k_codes), f"key codes b{b} h{h}"
            assert np.array_equal(vc[b, h], qh.v_codes), f"value codes b{b} h{h}"
            assert np.array_equal(vpar[b, h, :, 0].view(np.uint32), qh.v_lo.view(np.uint32))
            assert np.array_equal(vpar[b, h, :, 1].view(np.uint32), qh.v_scale.view(np.uint32))
            for t in range(n):
                ents = kout[b, h, off[b, h, t]:off[b, h, t + 1]]
                assert all(int(e >> 24) == t % 64 for e in ents), f"key outlier token field b{b} h{h} t{t}"
                got = {(int((e >> 16) & 0xff), int(e & 0xffff)) for e in ents}
                chans = np.nonzero(qh.k_mask[t])[0]
                ref = {(int(c), int(k[b, h, t, c].view(np.uint16))) for c in chans}
                assert got == ref, f"key outliers b{b} h{h} t{t}"
                got = {(int(e >> 16), int(e & 0xffff)) for e in vout[b, h, t, :nv]}
                chans = np.nonzero(qh.v_mask[t])[0]
                ref = {(int(c), int(v[b, h, t, c].view(np.uint16))) for c in chans}
                assert got == ref, f"value outliers b{b} h{h} t{t}"


def _decode_vs_oracle(B, Hq, Hkv, D, bits, mode, T, steps, seed, frac=0.01, outlier_channels=(), key_scale=True,
                      T_cap=None, check=None):
    torch = torch_cuda()
    dev = torch.device("cuda")
    k, v = _data(B, Hkv, T + steps, D, seed=seed, key_scale=key_scale, outlier_channels=outlier_channels)
    q = np.random.default_rng(seed + 1).standard_normal((steps, B, Hq, D)).astype(np.float16)
    plist = _oracle_params(k, v, min(T, 4096), bits, mode, frac)
    cfg = make_cfg(B, Hq, Hkv, D, bits, mode, frac)
    cache, qp = _quantized_cache(cfg, k, v, plist, T, 0, dev, T_cap=T_cap or (T + steps + 8))
    ws, nws = caches.workspace(cfg, cache.T_cap, device=dev)
    G = Hq // Hkv
    for s in range(steps):
        kn, vn = to_dev(k[:, :, T + s:T + s + 1], dev), to_dev(v[:, :, T + s:T + s + 1], dev)
        mkv.mkv_quantize_kv(cfg, qp.c, kn.data_ptr(), vn.data_ptr(), 1, cache.c)
        qt = to_dev(q[s], dev)
        out = torch.empty_like(qt)
        mkv.mkv_decode_attention(cfg, qt.data_ptr(), cache.c, qp.c, 0, out.data_ptr(), ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        n = T + s + 1
        for b in (check if check is not None else range(B)):
            for h in range(Hkv):
                qh = kvquant.quantize_head(k[b, h, :n], v[b, h, :n], plist[h])
                ref = kvquant.decode_head(q[s, b, h * G:(h + 1) * G], qh, plist[h], cfg.rope_theta)
                assert_close(got[b, h * G:(h + 1) * G], ref, f"step {s} b{b} h{h}")


def test_decode_tiny_workload():
    """The tiny all-configs case: 4-bit uniform, 1% outliers, 4 key channels x10, 16 steps."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = synth.tiny()
    x = synth.host_inputs(w, seed=1)
    k, v = x["k"][0], x["v"][0]
    plist = _oracle_params(k, v, w.T, w.bits, w.quant_mode, w.outlier_frac)
    cfg = make_cfg(w.B, w.Hq, w.Hkv, w.D, w.bits, w.quant_mode, w.outlier_frac, w.theta)
    cache, qp = _quantized_cache(cfg, k, v, plist, w.T, 0, dev, T_cap=w.T + w.steps)
    ws, nws = caches.workspace(cfg, cache.T_cap, device=dev)
    for s in range(w.steps):
        kn, vn = to_dev(k[:, :, w.T + s:w.T + s + 1], dev), to_dev(v[:, :, w.T + s:w.T + s + 1], dev)
        mkv.mkv_quantize_kv(cfg, qp.c, kn.data_ptr(), vn.data_ptr(), 1, cache.c)
        qt = to_dev(x["q"][s, 0], dev)
        out = torch.empty_like(qt)
        mkv.mkv_decode_attention(cfg, qt.data_ptr(), cache.c, qp.c, 0, out.data_ptr(), ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        n = w.T + s + 1
        for h in range(w.Hkv):
            qh = kvquant.quantize_head(k[0, h, :n], v[0, h, :n], plist[h])
            ref = kvquant.decode_head(x["q"][s, 0, 0, h * w.G:(h + 1) * w.G], qh, plist[h], w.theta)
            assert_close(got[0, h * w.G:(h + 1) * w.G], ref, f"step {s} h{h}")


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_decode_nuq_llama_shape(bits):
    _decode_vs_oracle(B=2, Hq=32, Hkv=8, D=128, bits=bits, mode="nuq", T=1000, steps=2, seed=40 + bits)


@pytest.mark.parametrize("D,G", [(64, 1), (64, 8), (128, 2)])
def test_decode_shapes_ragged(D, G):
    _decode_vs_oracle(B=3, Hq=2 * G, Hkv=2, D=D, bits=4, mode="uniform", T=97, steps=2, seed=D + G)


def test_decode_all_outliers_equals_fp16_path():
    """outlier_frac = 1: every entry is stored exactly, so the fused path is plain attention."""
    _decode_vs_oracle(B=1, Hq=8, Hkv=2, D=64, bits=2, mode="uniform", T=130, steps=1, seed=77, frac=1.0)


def test_decode_dense_outliers():
    """outlier_frac = 0.1 at the Llama shape: ~13 key outliers per token, so each attention warp
    restores several rounds of entries, many beyond the staged ones, and pairs with outliers in
    both channels (i and i + D/2) of a token are common."""
    _decode_vs_oracle(B=2, Hq=32, Hkv=8, D=128, bits=4, mode="nuq", T=700, steps=1, seed=12, frac=0.1)


def test_quantize_capacity_flag():
    """An append past T_cap writes nothing, keeps T_len and raises MKV_FLAG_CACHE_FULL."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    k, v = _data(1, 2, 40, 64, seed=3)
    plist = _oracle_params(k, v, 32, 4, "uniform", 0.01)
    cfg = make_cfg(1, 4, 2, 64, 4, "uniform")
    cache, qp = _quantized_cache(cfg, k, v, plist, 32, 0, dev, T_cap=32)
    before = cache.t["k_codes"].clone()
    kn, vn = to_dev(k[:, :, 32:33], dev), to_dev(v[:, :, 32:33], dev)
    mkv.mkv_quantize_kv(cfg, qp.c, kn.data_ptr(), vn.data_ptr(), 1, cache.c)
    assert mkv.mkv_get_status() == mkv.MKV_FLAG_CACHE_FULL
    assert int(cache.t["T_len"][0]) == 32
    assert torch.equal(before, cache.t["k_codes"])


def test_decode_full_size_sampled():
    """B=8, T=8192, 32/8/128, NUQ 4-bit: one layer, every kv-head of batch entries 0 and 7."""
    _decode_vs_oracle(B=8, Hq=32, Hkv=8, D=128, bits=4, mode="nuq", T=8192, steps=1, seed=99, check=(0, 7))


def test_decode_many_units_ragged_lengths():
    """More (batch, kv-head) units than SMs and a different length per batch entry (0 .. T): the
    CTAs' equal runs of chunks cross unit boundaries, units are merged from several CTAs, and a
    batch entry with no tokens gets a zero output."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    B, Hq, Hkv, D, bits, T = 40, 8, 4, 64, 3, 150
    k, v = _data(B, Hkv, T, D, seed=5)
    plist = _oracle_params(k, v, T, bits, "uniform", 0.01)
    cfg = make_cfg(B, Hq, Hkv, D, bits, "uniform", 0.01)
    cache, qp = _quantized_cache(cfg, k, v, plist, T, 0, dev, T_cap=T + 8)
    lens = [(37 * b) % (T + 1) for b in range(B)]
    assert 0 in lens and max(lens) > 128
    cache.t["T_len"].copy_(torch.tensor(lens, dtype=cache.t["T_len"].dtype, device=dev))
    ws, nws = caches.workspace(cfg, cache.T_cap, device=dev)
    q = np.random.default_rng(6).standard_normal((B, Hq, D)).astype(np.float16)
    qt = to_dev(q, dev)
    out = torch.empty_like(qt)
    G = Hq // Hkv
    for rep in range(2):                      # the ticket counters return to zero after a call
        mkv.mkv_decode_attention(cfg, qt.data_ptr(), cache.c, qp.c, 0, out.data_ptr(), ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        for b in range(B):
            n = lens[b]
            for h in range(Hkv):
                rows = got[b, h * G:(h + 1) * G]
                if n == 0:
                    assert np.all(rows == 0.0), f"empty b{b} h{h}"
                    continue
                qh = kvquant.quantize_head(k[b, h, :n], v[b, h, :n], plist[h])
                ref = kvquant.decode_head(q[b, h * G:(h + 1) * G], qh, plist[h], cfg.rope_theta)
                assert_close(rows, ref, f"call {rep} b{b} h{h} n{n}")
