"""GPU parity: H2O prefill scores + initial keep, and decode steps with eviction."""
import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
import synth
from oracle import attention, h2o
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, to_dev, torch_cuda
from lockstep import check_evict, check_topk, record, tiny_seed

pytestmark = pytest.mark.gpu


def _state(cache, b, h):
    pos = cache.t["pos"][b, h].cpu().numpy()
    acc = cache.t["acc"][b, h].cpu().numpy()
    held = pos >= 0
    return pos, acc, held


def run_h2o(B, Hq, Hkv, D, T, steps, H, R, K, V, QP, Q, dev, exact, units, tag, step_api=False):
    """K, V [B,Hkv,T+steps,D]; QP [B,Hq,T,D]; Q [steps,B,Hq,D] (device tensors).
    units: (b, kv-head) pairs checked against the oracle in lockstep.
    step_api: each step through mkv_decode_step (the token's append and the attention in one
    launch, as the bench runs it) instead of mkv_append_kv + mkv_decode_attention."""
    torch = torch_cuda()
    G = Hq // Hkv
    cfg = mkv.config(mkv.MKV_H2O, B, Hq, Hkv, D, h2o_heavy=H, h2o_recent=R)
    T_cap = H + R + 1
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    ws, nws = caches.workspace(cfg, max(T, T_cap), device=dev)
    Kp, Vp = K[:, :, :T].contiguous(), V[:, :, :T].contiguous()
    mkv.mkv_h2o_prefill(cfg, QP.data_ptr(), Kp.data_ptr(), Vp.data_ptr(), T, cache.c, ws.data_ptr(), nws)
    torch.cuda.synchronize()
    host = {}
    near = decisions = 0
    for (b, h) in units:
        k = K[b, h].cpu().numpy()
        v = V[b, h].cpu().numpy()
        qp = QP[b, h * G:(h + 1) * G].cpu().numpy()
        acc0 = h2o.prefill_scores(qp, k[:T])
        pos, acc, held = _state(cache, b, h)
        got_keep = np.sort(pos[held])
        rest = np.arange(max(T - R, 0))
        heavy_got = got_keep[got_keep < T - R]
        near += check_topk(acc0[rest], rest, min(H, rest.shape[0]), heavy_got, exact, f"{tag} keep b{b} h{h}")
        decisions += 1
        assert set(range(max(T - R, 0), T)) <= set(got_keep.tolist())
        # scores of the kept tokens: fp32 GPU column sums vs fp64
        np.testing.assert_allclose(acc[held], acc0[pos[held]], rtol=2e-4, atol=1e-5)
        st = h2o.H2OHead(got_keep.copy(), k[got_keep], v[got_keep], acc0[got_keep].copy())
        host[(b, h)] = (k, v, st)
    for s in range(steps):
        kn = K[:, :, T + s].contiguous()
        vn = V[:, :, T + s].contiguous()
        q = Q[s].contiguous()
        out = torch.empty_like(q)
        if step_api:
            # the cache as the append would leave it: the new position in each (b, kv-head)'s next slot
            pos_before = cache.t["pos"].clone()
            sl = cache.t["slot"].long()
            pos_before.scatter_(2, sl.unsqueeze(2), torch.full_like(sl.unsqueeze(2), T + s, dtype=pos_before.dtype))
            mkv.mkv_decode_step(cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), cache.c, out.data_ptr(),
                                ws.data_ptr(), nws)
        else:
            mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), cache.c)
            pos_before = cache.t["pos"].clone()
            mkv.mkv_decode_attention(cfg, q.data_ptr(), cache.c, None, 0, out.data_ptr(), ws.data_ptr(), nws)
        mkv.mkv_h2o_update(cfg, cache.c, ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        for (b, h) in units:
            k, v, st = host[(b, h)]
            qh = Q[s, b, h * G:(h + 1) * G].cpu().numpy()
            ref, st2, ev, cand = h2o.decode_step(st, qh, k[T + s], v[T + s], T + s, H, R)
            assert_close(got[b, h * G:(h + 1) * G], ref, f"{tag} step {s} b{b} h{h}")
            before = set(pos_before[b, h][pos_before[b, h] >= 0].tolist())
            pos, acc, held = _state(cache, b, h)
            after = set(pos[held].tolist())
            gone = sorted(before - after)
            if cand is None:
                assert gone == [] and ev is None
            else:
                assert len(gone) == 1, f"{tag} step {s}: evicted {gone}"
                n = check_evict(cand[0], cand[1], gone[0], exact, f"{tag} step {s} b{b} h{h}")
                near += n
                decisions += 1
                if n:
                    _, st2, _, _ = h2o.decode_step(st, qh, k[T + s], v[T + s], T + s, H, R, forced_victim=gone[0])
            ordr = np.argsort(st2.pos)
            np.testing.assert_array_equal(np.sort(pos[held]), st2.pos[ordr])
            gacc = dict(zip(pos[held].tolist(), acc[held].tolist()))
            np.testing.assert_allclose([gacc[p] for p in st2.pos[ordr]], st2.acc[ordr], rtol=2e-4, atol=1e-5)
            host[(b, h)] = (k, v, st2)
    assert mkv.mkv_get_status() == 0
    record(f"h2o {tag}{' (one-launch step)' if step_api else ''}", near, decisions)
    return near


def test_tiny_exact():
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = synth.tiny()
    x = synth.host_inputs(w, seed=tiny_seed())
    K, V = to_dev(x["k"][0], dev), to_dev(x["v"][0], dev)
    QP, Q = to_dev(x["q_prompt"][0], dev), to_dev(x["q"][:, 0], dev)
    for step_api in (False, True):
        near = run_h2o(w.B, w.Hq, w.Hkv, w.D, w.T, w.steps, w.h2o_heavy, w.h2o_recent, K, V, QP, Q, dev, True,
                       [(0, 0), (0, 1)], f"tiny{'-step' if step_api else ''}", step_api)
        assert near == 0


def test_budget_covers_context_is_full_attention():
    """Budget >= prompt + steps: nothing is evicted and every step is full attention."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(5)
    B, Hq, Hkv, D, T, steps = 2, 8, 2, 128, 100, 4
    K = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    QP = rng.standard_normal((B, Hq, T, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    near = run_h2o(B, Hq, Hkv, D, T, steps, 80, 80, to_dev(K, dev), to_dev(V, dev), to_dev(QP, dev), to_dev(Q, dev),
                   dev, False, [(0, 0), (1, 1)], "full")
    assert near == 0


@pytest.mark.parametrize("G,D", [(1, 64), (8, 128)])
def test_shapes_lockstep(G, D):
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(G * 7 + D)
    B, Hkv, T, steps = 2, 2, 333, 6
    Hq = G * Hkv
    K = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    QP = rng.standard_normal((B, Hq, T, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    run_h2o(B, Hq, Hkv, D, T, steps, 30, 20, to_dev(K, dev), to_dev(V, dev), to_dev(QP, dev), to_dev(Q, dev), dev,
            False, [(0, 0), (1, 1)], f"G{G}D{D}")


def test_full_size_lockstep():
    """B=16, T=16384, 32/8/128, 20% budget (1638 heavy + 1638 recent), heavy-hitter inputs, the
    bench's one-launch step (mkv_decode_step + mkv_h2o_update): one layer, 64 steps, four
    (batch, kv-head) units in lockstep with the oracle."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = synth.h2o_16k(20)
    n = 64
    x = synth.device_layer_inputs(w, seed=11, layer=0, device=dev, n_tokens=w.T + n, with_prompt_queries=True)
    run_h2o(w.B, w.Hq, w.Hkv, w.D, w.T, n, w.h2o_heavy, w.h2o_recent, x["k"], x["v"], x["q_prompt"],
            x["q"][:n], dev, False, [(0, 0), (5, 3), (10, 6), (15, 7)], "h2o20-b16-t16384", step_api=True)


def test_step_equals_append_then_decode():
    """mkv_decode_step against mkv_append_kv + mkv_decode_attention on twin H2O caches, each step
    followed by mkv_h2o_update, over steps that evict and reuse slots: identical outputs, rows,
    positions, scores, chosen slots and lengths."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(46)
    B, Hq, Hkv, D, T, H, R, steps = 2, 8, 2, 64, 300, 64, 64, 10
    cfg = mkv.config(mkv.MKV_H2O, B, Hq, Hkv, D, h2o_heavy=H, h2o_recent=R)
    T_cap = H + R + 1
    K = to_dev(rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16), dev)
    V = to_dev(rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16), dev)
    QP = to_dev(rng.standard_normal((B, Hq, T, D)).astype(np.float16), dev)
    Kp, Vp = K[:, :, :T].contiguous(), V[:, :, :T].contiguous()
    twins = []
    for _ in range(2):
        cache = caches.alloc_cache(cfg, T_cap, device=dev)
        ws, nws = caches.workspace(cfg, max(T, T_cap), device=dev)
        mkv.mkv_h2o_prefill(cfg, QP.data_ptr(), Kp.data_ptr(), Vp.data_ptr(), T, cache.c, ws.data_ptr(), nws)
        twins.append((cache, ws, nws))
    (a, wa, na), (c, wc, nc) = twins
    keys = ("k", "v", "pos", "acc", "slot", "T_len")

    def same(x, y):
        if x.dtype == torch.float16:
            return torch.equal(x.view(torch.int16), y.view(torch.int16))
        return torch.equal(x, y)

    for key in keys:
        assert same(a.t[key], c.t[key]), f"prefill: {key}"
    for s in range(steps):
        kn = K[:, :, T + s].contiguous()
        vn = V[:, :, T + s].contiguous()
        q = to_dev(rng.standard_normal((B, Hq, D)).astype(np.float16), dev)
        oa, oc = torch.empty_like(q), torch.empty_like(q)
        full = s == 4                       # batch entry 1, kv-head 0 has no free slot at this step
        if full:
            len_before = [int(x) for x in a.t["T_len"]]
            saved = int(a.t["slot"][1, 0])
            for cc in (a, c):
                cc.t["slot"][1, 0] = T_cap
        mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), a.c)
        fa = mkv.mkv_get_status()
        mkv.mkv_decode_attention(cfg, q.data_ptr(), a.c, None, 0, oa.data_ptr(), wa.data_ptr(), na)
        mkv.mkv_h2o_update(cfg, a.c, wa.data_ptr(), na)
        mkv.mkv_decode_step(cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), c.c, oc.data_ptr(), wc.data_ptr(), nc)
        fc = mkv.mkv_get_status()
        mkv.mkv_h2o_update(cfg, c.c, wc.data_ptr(), nc)
        assert mkv.mkv_get_status() == 0
        want = mkv.MKV_FLAG_CACHE_FULL if full else 0
        assert fa == fc == want, f"step {s}: flags {fa} {fc}"
        if full:                            # no kv-head of that batch entry was appended; length kept
            assert int(c.t["T_len"][1]) == len_before[1] and int(c.t["T_len"][0]) == len_before[0] + 1
            for cc in (a, c):               # nothing was evicted there: give the slot back
                cc.t["slot"][1, 0] = saved
        assert torch.equal(oa.view(torch.int16), oc.view(torch.int16)), f"step {s}: outputs differ"
        for key in keys:
            assert same(a.t[key], c.t[key]), f"step {s}: {key}"
    assert int(c.t["T_len"][0]) == T + steps and int(c.t["T_len"][1]) == T + steps - 1
