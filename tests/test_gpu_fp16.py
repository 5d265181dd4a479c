"""GPU parity: FP16 decode attention (append + split-KV decode + combine) vs the oracle."""
import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
import synth
from oracle import attention
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, to_dev, torch_cuda

pytestmark = pytest.mark.gpu


def _run_fp16(B, Hq, Hkv, D, T_lens, T_cap, steps, seed, dev):
    """Prefill T_lens[b] tokens, then `steps` append+decode steps; returns outs and the inputs."""
    torch = torch_cuda()
    rng = np.random.default_rng(seed)
    n = max(T_lens) + steps
    K = rng.standard_normal((B, Hkv, n, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, n, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    cfg = mkv.config(mkv.MKV_FP16, B, Hq, Hkv, D)
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    for b in range(B):
        cache.t["k"][b, :, :T_lens[b]] = to_dev(K[b, :, :T_lens[b]], dev)
        cache.t["v"][b, :, :T_lens[b]] = to_dev(V[b, :, :T_lens[b]], dev)
    cache.t["T_len"].copy_(torch.tensor(T_lens, dtype=torch.int32))
    ws, nws = caches.workspace(cfg, T_cap, device=dev)
    outs = []
    for s in range(steps):
        kn = np.stack([K[b, :, T_lens[b] + s] for b in range(B)])
        vn = np.stack([V[b, :, T_lens[b] + s] for b in range(B)])
        kt, vt, qt = to_dev(kn, dev), to_dev(vn, dev), to_dev(Q[s], dev)
        out = torch.empty_like(qt)
        mkv.mkv_append_kv(cfg, kt.data_ptr(), vt.data_ptr(), cache.c)
        mkv.mkv_decode_attention(cfg, qt.data_ptr(), cache.c, None, 0, out.data_ptr(), ws.data_ptr(), nws)
        outs.append(out.float().cpu().numpy())
    assert mkv.mkv_get_status() == 0
    return outs, K, V, Q


def _ref(K, V, q, b, n):
    return attention.decode_gqa(q[b], K[b, :, :n], V[b, :, :n])


def test_tiny_all_steps():
    torch = torch_cuda()
    w = synth.tiny()
    x = synth.host_inputs(w, seed=1)
    dev = torch.device("cuda")
    cfg = mkv.config(mkv.MKV_FP16, w.B, w.Hq, w.Hkv, w.D)
    T_cap = w.T + w.steps
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    cache.t["k"][:, :, :w.T] = to_dev(x["k"][0, :, :, :w.T], dev)
    cache.t["v"][:, :, :w.T] = to_dev(x["v"][0, :, :, :w.T], dev)
    cache.t["T_len"].fill_(w.T)
    ws, nws = caches.workspace(cfg, T_cap, device=dev)
    for s in range(w.steps):
        kt = to_dev(x["k"][0, :, :, w.T + s], dev)
        vt = to_dev(x["v"][0, :, :, w.T + s], dev)
        qt = to_dev(x["q"][s, 0], dev)
        out = torch.empty_like(qt)
        mkv.mkv_append_kv(cfg, kt.data_ptr(), vt.data_ptr(), cache.c)
        mkv.mkv_decode_attention(cfg, qt.data_ptr(), cache.c, None, 0, out.data_ptr(), ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        for b in range(w.B):
            ref = attention.decode_gqa(x["q"][s, 0, b], x["k"][0, b, :, :w.T + s + 1], x["v"][0, b, :, :w.T + s + 1])
            assert_close(got[b], ref, f"step {s} b {b}")
    assert int(cache.t["T_len"][0]) == w.T + w.steps


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("G", [1, 2, 4, 8])
def test_shapes_ragged(D, G):
    torch = torch_cuda()
    dev = torch.device("cuda")
    Hkv = 2
    T_lens = [0, 1, 63, 65, 777]
    outs, K, V, Q = _run_fp16(len(T_lens), G * Hkv, Hkv, D, T_lens, 1024, 2, seed=D * 10 + G, dev=dev)
    for s in range(2):
        for b, T in enumerate(T_lens):
            assert_close(outs[s][b], _ref(K, V, Q[s], b, T + s + 1), f"G{G} D{D} T{T} s{s}")


def test_long_context_single_entry():
    torch = torch_cuda()
    dev = torch.device("cuda")
    outs, K, V, Q = _run_fp16(1, 32, 8, 128, [40000], 40064, 1, seed=5, dev=dev)
    assert_close(outs[0][0], _ref(K, V, Q[0], 0, 40001), "T=40001")


def test_kvquant_shape_sampled():
    """Llama-shaped 32/8/128 at B=8, T=8192 (the KVQuant workload's shape), every head checked."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    outs, K, V, Q = _run_fp16(8, 32, 8, 128, [8192] * 8, 8320, 1, seed=6, dev=dev)
    for b in (0, 3, 7):
        assert_close(outs[0][b], _ref(K, V, Q[0], b, 8193), f"b{b}")


def test_capacity_flag():
    torch = torch_cuda()
    dev = torch.device("cuda")
    cfg = mkv.config(mkv.MKV_FP16, 1, 4, 1, 64)
    cache = caches.alloc_cache(cfg, 4, device=dev)
    cache.t["T_len"].fill_(4)
    kn = torch.zeros((1, 1, 64), dtype=torch.float16, device=dev)
    mkv.mkv_append_kv(cfg, kn.data_ptr(), kn.data_ptr(), cache.c)
    assert mkv.mkv_get_status() == mkv.MKV_FLAG_CACHE_FULL
    assert int(cache.t["T_len"][0]) == 4
    assert mkv.mkv_get_status() == 0      # reading clears the word


def test_step_equals_append_then_decode():
    """mkv_decode_step against mkv_append_kv + mkv_decode_attention on twin caches, over steps whose
    tokens cross chunk and split boundaries and fill one batch entry: identical outputs, K/V rows and
    lengths; a full cache is not appended, keeps its length, raises MKV_FLAG_CACHE_FULL and attends
    to its tokens."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(45)
    B, Hq, Hkv, D = 3, 8, 2, 128
    T0, T_cap, steps = [1, 126, 250], 256, 12          # entry 2 is full from step 6 on
    cfg = mkv.config(mkv.MKV_FP16, B, Hq, Hkv, D)
    K = rng.standard_normal((B, Hkv, T_cap + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T_cap + steps, D)).astype(np.float16)
    twins = []
    for _ in range(2):
        cache = caches.alloc_cache(cfg, T_cap, device=dev)
        cache.t["k"].copy_(to_dev(K[:, :, :T_cap], dev))
        cache.t["v"].copy_(to_dev(V[:, :, :T_cap], dev))
        cache.t["T_len"].copy_(torch.tensor(T0, dtype=torch.int32))
        ws, nws = caches.workspace(cfg, T_cap, device=dev)
        twins.append((cache, ws, nws))
    (a, wa, na), (c, wc, nc) = twins
    full_seen = False
    for s in range(steps):
        kn = to_dev(K[:, :, T_cap + s], dev)           # rows the caches do not hold yet
        vn = to_dev(V[:, :, T_cap + s], dev)
        q = to_dev(rng.standard_normal((B, Hq, D)).astype(np.float16), dev)
        oa, oc = torch.empty_like(q), torch.empty_like(q)
        will_fill = [int(a.t["T_len"][b]) >= T_cap for b in range(B)]
        mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), a.c)
        fa = mkv.mkv_get_status()
        mkv.mkv_decode_attention(cfg, q.data_ptr(), a.c, None, 0, oa.data_ptr(), wa.data_ptr(), na)
        mkv.mkv_decode_step(cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), c.c, oc.data_ptr(), wc.data_ptr(), nc)
        fc = mkv.mkv_get_status()
        assert fa == fc == (mkv.MKV_FLAG_CACHE_FULL if any(will_fill) else 0), f"step {s}: flags {fa} {fc}"
        full_seen |= any(will_fill)
        assert torch.equal(oa.view(torch.int16), oc.view(torch.int16)), f"step {s}: outputs differ"
        assert torch.equal(a.t["T_len"], c.t["T_len"]), f"step {s}: T_len"
        for key in ("k", "v"):
            assert torch.equal(a.t[key].view(torch.int16), c.t[key].view(torch.int16)), f"step {s}: {key}"
    assert full_seen
    assert [int(x) for x in c.t["T_len"]] == [1 + steps, 126 + steps, T_cap]


def test_step_vs_oracle_bench_shape():
    """mkv_decode_step at the FP16 bench shape (B=8, T=8192, 32/8/128, the bench's T_cap): two steps
    against fp64 attention over the T+1 and T+2 tokens, every head of batch entries 0, 4 and 7."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(47)
    B, Hq, Hkv, D, T, steps = 8, 32, 8, 128, 8192, 2
    T_cap = T + 4 * 25 + 8 + 64
    cfg = mkv.config(mkv.MKV_FP16, B, Hq, Hkv, D)
    K = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    cache.t["k"][:, :, :T] = to_dev(K[:, :, :T], dev)
    cache.t["v"][:, :, :T] = to_dev(V[:, :, :T], dev)
    cache.t["T_len"].fill_(T)
    ws, nws = caches.workspace(cfg, T_cap, device=dev)
    for s in range(steps):
        kn, vn = to_dev(K[:, :, T + s], dev), to_dev(V[:, :, T + s], dev)
        qt = to_dev(Q[s], dev)
        out = torch.empty_like(qt)
        mkv.mkv_decode_step(cfg, qt.data_ptr(), kn.data_ptr(), vn.data_ptr(), cache.c, out.data_ptr(),
                            ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        for b in (0, 4, 7):
            assert_close(got[b], _ref(K, V, Q[s], b, T + s + 1), f"step {s} b{b}")
    assert mkv.mkv_get_status() == 0
    assert [int(x) for x in cache.t["T_len"]] == [T + steps] * B
