"""GPU parity of the fused KVQuant step (mkv_kvquant_step, Section 2.1 KVQuant paragraph): one
launch that quantizes the step's token into the cache and attends over it must leave exactly the
cache that mkv_quantize_kv (one token) leaves and produce exactly the output of
mkv_decode_attention after it, on twin caches; at the bench's shape it is also compared with the
fp64 oracle."""
import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
from oracle import kvquant
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, to_dev, torch_cuda
from test_gpu_kvquant import _data, _oracle_params, _quantized_cache, make_cfg

pytestmark = pytest.mark.gpu

CACHE_KEYS = ("k_codes", "v_codes", "v_params", "v_out", "k_out_off", "k_out", "T_len")


def _twin(cache, cfg, dev):
    torch = torch_cuda()
    other = caches.alloc_cache(cfg, cache.T_cap, device=dev, k_out_cap=cache.c.k_out_cap)
    for key in CACHE_KEYS:
        other.t[key].copy_(cache.t[key])
    torch.cuda.synchronize()
    return other


def _same(a, b, what):
    torch = torch_cuda()
    for key in CACHE_KEYS:
        x, y = a.t[key], b.t[key]
        if x.dtype.is_floating_point:
            x, y = x.view(torch.int32), y.view(torch.int32)
        assert torch.equal(x, y), f"{what}: {key} differs"


def _run_twins(B, Hq, Hkv, D, bits, mode, T, T_cap, steps, seed, lens=None, frac=0.01):
    """Steps on twin caches: (quantize + decode) against the fused step; returns the last outputs."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    k, v = _data(B, Hkv, T_cap + steps + 1, D, seed=seed)      # one spare token for a further step
    plist = _oracle_params(k, v, min(T, 4096), bits, mode, frac)
    cfg = make_cfg(B, Hq, Hkv, D, bits, mode, frac)
    a, qp = _quantized_cache(cfg, k, v, plist, T, 0, dev, T_cap=T_cap)
    if lens is not None:
        a.t["T_len"].copy_(torch.tensor(lens, dtype=a.t["T_len"].dtype, device=dev))
    c = _twin(a, cfg, dev)
    wa, na = caches.workspace(cfg, T_cap, device=dev)
    wc, nc = caches.workspace(cfg, T_cap, device=dev)
    rng = np.random.default_rng(seed + 7)
    flags_seen = 0
    for s in range(steps):
        # the step's token: rows the caches do not hold (per batch entry at its own length)
        kn = to_dev(np.ascontiguousarray(k[:, :, T_cap + s]), dev)
        vn = to_dev(np.ascontiguousarray(v[:, :, T_cap + s]), dev)
        q = to_dev(rng.standard_normal((B, Hq, D)).astype(np.float16), dev)
        oa, oc = torch.empty_like(q), torch.empty_like(q)
        mkv.mkv_quantize_kv(cfg, qp.c, kn.data_ptr(), vn.data_ptr(), 1, a.c)
        mkv.mkv_decode_attention(cfg, q.data_ptr(), a.c, qp.c, 0, oa.data_ptr(), wa.data_ptr(), na)
        fa = mkv.mkv_get_status()
        mkv.mkv_kvquant_step(cfg, qp.c, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), c.c, oc.data_ptr(),
                             wc.data_ptr(), nc)
        fc = mkv.mkv_get_status()
        assert fa == fc, f"step {s}: flags {fa} {fc}"
        flags_seen |= fc
        assert torch.equal(oa.view(torch.int16), oc.view(torch.int16)), f"step {s}: outputs differ"
        _same(a, c, f"step {s}")
    return flags_seen, cfg, c, qp, k, v, plist


def test_step_equals_quantize_then_decode():
    """Three batch entries at lengths 0, 126 and 250 of 256 (the first token of a cache, tokens
    crossing chunk and CTA boundaries, and an entry that fills at step 6 and is then not appended:
    MKV_FLAG_CACHE_FULL, length kept, attends to its tokens); NUQ 4-bit, 32/8/128-like groups."""
    flags, _, c, _, _, _, _ = _run_twins(B=3, Hq=8, Hkv=2, D=128, bits=4, mode="nuq", T=250, T_cap=256, steps=12,
                                         seed=61, lens=[0, 126, 250])
    assert flags == mkv.MKV_FLAG_CACHE_FULL
    assert [int(x) for x in c.t["T_len"]] == [12, 138, 256]


@pytest.mark.parametrize("bits,mode,D,G", [(3, "uniform", 64, 2), (2, "nuq", 128, 4), (4, "uniform", 64, 8)])
def test_step_many_units_per_cta(bits, mode, D, G):
    """A short cache (T_cap = 64: one chunk per unit) with 40 batch entries x 4 kv-heads: every CTA
    holds the new tokens of several units and touches several batch entries; ragged lengths
    including empty caches; 2-, 3- and 4-bit, uniform and NUQ, D = 64 (idle quantizer threads)."""
    B, Hkv = 40, 4
    lens = [(11 * b) % 60 for b in range(B)]
    flags, _, c, _, _, _, _ = _run_twins(B=B, Hq=G * Hkv, Hkv=Hkv, D=D, bits=bits, mode=mode, T=60, T_cap=64,
                                         steps=3, seed=70 + bits, lens=lens)
    assert flags == 0
    assert [int(x) for x in c.t["T_len"]] == [n + 3 for n in lens]


def test_step_dense_outliers():
    """outlier_frac = 0.1: ~13 key outliers per token, entries beyond the decode's staged ones, and
    n_v = 13 value outliers (ranked by counting rather than by rounds of maxima)."""
    flags, *_ = _run_twins(B=2, Hq=32, Hkv=8, D=128, bits=4, mode="nuq", T=700, T_cap=776, steps=2, seed=81,
                           frac=0.1)
    assert flags == 0


def test_step_bench_shape_vs_oracle():
    """The bench's shape (B=8, T=8192, 32/8/128, NUQ 4-bit): two fused steps bit-identical to
    quantize + decode, the last one's outputs against the oracle's fp64 decode over T+2 tokens for
    every kv-head of batch entries 0 and 7."""
    T, steps = 8192, 2
    _, cfg, c, qp, k, v, plist = _run_twins(B=8, Hq=32, Hkv=8, D=128, bits=4, mode="nuq", T=T, T_cap=T + 128,
                                            steps=steps, seed=99)
    torch = torch_cuda()
    dev = torch.device("cuda")
    T_cap = T + 128
    # one more fused step, its output checked against the oracle over the appended tokens
    kn = to_dev(np.ascontiguousarray(k[:, :, T_cap + steps]), dev)
    vn = to_dev(np.ascontiguousarray(v[:, :, T_cap + steps]), dev)
    q = np.random.default_rng(5).standard_normal((8, 32, 128)).astype(np.float16)
    qt = to_dev(q, dev)
    out = torch.empty_like(qt)
    ws, nws = caches.workspace(cfg, T_cap, device=dev)
    mkv.mkv_kvquant_step(cfg, qp.c, qt.data_ptr(), kn.data_ptr(), vn.data_ptr(), c.c, out.data_ptr(),
                         ws.data_ptr(), nws)
    assert mkv.mkv_get_status() == 0
    got = out.float().cpu().numpy()
    G = 4
    for b in (0, 7):
        for h in range(8):
            kk = np.concatenate([k[b, h, :T], k[b, h, T_cap:T_cap + steps + 1]])
            vv = np.concatenate([v[b, h, :T], v[b, h, T_cap:T_cap + steps + 1]])
            qh = kvquant.quantize_head(kk, vv, plist[h])
            ref = kvquant.decode_head(q[b, h * G:(h + 1) * G], qh, plist[h], cfg.rope_theta)
            assert_close(got[b, h * G:(h + 1) * G], ref, f"b{b} h{h}")
    assert [int(x) for x in c.t["T_len"]] == [T + steps + 1] * 8
