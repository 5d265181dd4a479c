"""GPU parity at the size sweep's extreme shapes: FP16 at (T, B) = (128K, 1) and (4K, 32), NUQ 4-bit
KVQuant at 64K, H2O with 10 % and 40 % budgets, and RocketKV token budgets 2048 and 4096 (keep 8192
and 16384, 128 and 256 chosen pages) -- sampled (batch, kv-head) units against the oracle."""
import dataclasses

import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
import synth
from oracle import attention
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, torch_cuda
from test_gpu_h2o import run_h2o
from test_gpu_kvquant import _decode_vs_oracle
from test_gpu_rocket import run_rocket

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("T,B", [(131072, 1), (4096, 32)])
def test_fp16_sweep_extremes(T, B):
    """The longest and the widest FP16 sweep shapes: device-generated caches, two append +
    decode steps, the first and the last (batch, kv-head) unit against the oracle."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    Hq, Hkv, D, steps = 32, 8, 128, 2
    G = Hq // Hkv
    cfg = mkv.config(mkv.MKV_FP16, B, Hq, Hkv, D)
    T_cap = T + steps
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    gen = torch.Generator(device=dev).manual_seed(T + B)
    cache.t["k"].copy_(torch.randn(cache.t["k"].shape, generator=gen, device=dev).half())
    cache.t["v"].copy_(torch.randn(cache.t["v"].shape, generator=gen, device=dev).half())
    cache.t["T_len"].fill_(T)
    ws, nws = caches.workspace(cfg, T_cap, device=dev)
    units = [(0, 0), (B - 1, Hkv - 1)]
    for s in range(steps):
        kn = torch.randn((B, Hkv, D), generator=gen, device=dev).half()
        vn = torch.randn((B, Hkv, D), generator=gen, device=dev).half()
        q = torch.randn((B, Hq, D), generator=gen, device=dev).half()
        out = torch.empty_like(q)
        mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), cache.c)
        mkv.mkv_decode_attention(cfg, q.data_ptr(), cache.c, None, 0, out.data_ptr(), ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        n = T + s + 1
        for (b, h) in units:
            k = cache.t["k"][b, h, :n].cpu().numpy()
            v = cache.t["v"][b, h, :n].cpu().numpy()
            assert np.array_equal(k[-1].view(np.uint16), kn[b, h].cpu().numpy().view(np.uint16))
            ref = attention.attend(q[b, h * G:(h + 1) * G].cpu().numpy(), k, v)[0]
            assert_close(got[b, h * G:(h + 1) * G], ref, f"fp16 T{T} B{B} step {s} b{b} h{h}")
    assert mkv.mkv_get_status() == 0


def test_kvquant_sweep_long_context():
    """NUQ 4-bit at T = 65536 (the sweep's 64K point), one appended token, every kv-head of the
    last batch entry against the oracle."""
    _decode_vs_oracle(B=2, Hq=32, Hkv=8, D=128, bits=4, mode="nuq", T=65536, steps=1, seed=64, check=(1,))


@pytest.mark.parametrize("budget", [10, 40])
def test_h2o_sweep_budgets(budget):
    """The sweep's other H2O budgets at T = 16384 (heavy-hitter inputs): prefill keep and four
    decode steps with eviction, two units in lockstep with the oracle."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = dataclasses.replace(synth.h2o_16k(budget), B=2)
    x = synth.device_layer_inputs(w, seed=20 + budget, layer=0, device=dev, n_tokens=w.T + 4,
                                  with_prompt_queries=True)
    run_h2o(w.B, w.Hq, w.Hkv, w.D, w.T, 4, w.h2o_heavy, w.h2o_recent, x["k"], x["v"], x["q_prompt"], x["q"][:4], dev,
            False, [(0, 0), (1, 7)], f"h2o{budget}")


@pytest.mark.parametrize("budget,fused", [(2048, True), (4096, "step")])
def test_rocket_sweep_budgets(budget, fused):
    """The sweep's larger RocketKV budgets at T = 32768 (keep 4 x budget, 128 / 256 chosen pages
    of 512 / 1024): SnapKV compression and four decode steps, two units in lockstep."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = dataclasses.replace(synth.rocket_32k(budget), B=1)
    x = synth.device_layer_inputs(w, seed=30 + budget // 1024, layer=0, device=dev, n_tokens=w.T + 4,
                                  with_prompt_queries=True)
    QW = x["q_prompt"][:, :, w.T - w.snap_window:].contiguous()
    run_rocket(w.B, w.Hq, w.Hkv, w.D, w.T, 4, w.snap_window, w.snap_pool, w.snap_keep, w.topk_pages, w.topq_dims,
               x["k"], x["v"], QW, x["q"][:4], dev, False, [(0, 0), (0, 7)], f"rocket{budget}", fused)
