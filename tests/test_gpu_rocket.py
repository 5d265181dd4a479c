"""GPU parity: SnapKV prefill compression, page metadata, page selection and sparse decode,
both as two calls (mkv_rocket_select + mkv_decode_attention), as the fused step
(mkv_rocket_decode) and as the whole step with the token's append (mkv_rocket_step)."""
import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
import synth
from oracle import attention, rocket, snapkv
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, to_dev, torch_cuda
from lockstep import check_topk, record, tiny_seed

pytestmark = pytest.mark.gpu


def run_rocket(B, Hq, Hkv, D, T, steps, W, pool, keep, kp, rd, K, V, QW, Q, dev, exact, units, tag, fused=False):
    """K, V [B,Hkv,T+steps,D]; QW [B,Hq,W,D] window queries; Q [steps,B,Hq,D] (device tensors).
    fused: False (two calls), True (append + mkv_rocket_decode), "step" (mkv_rocket_step)."""
    torch = torch_cuda()
    G = Hq // Hkv
    cfg = mkv.config(mkv.MKV_ROCKET, B, Hq, Hkv, D, snap_window=W, snap_pool=pool, snap_keep=keep,
                     page_size=16, topk_pages=kp, topq_dims=rd)
    kept_n = min(T, keep)
    T_cap = (kept_n + steps + 15) // 16 * 16
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    ws, nws = caches.workspace(cfg, max(T, T_cap), device=dev)
    kept_pos = torch.zeros((B, Hkv, kept_n), dtype=torch.int32, device=dev)
    Kp, Vp = K[:, :, :T].contiguous(), V[:, :, :T].contiguous()
    mkv.mkv_snap_compress(cfg, QW.data_ptr(), Kp.data_ptr(), Vp.data_ptr(), T, cache.c, kept_pos.data_ptr(),
                          ws.data_ptr(), nws)
    torch.cuda.synchronize()
    assert int(cache.t["T_len"][0]) == kept_n
    near = decisions = 0
    host = {}
    for (b, h) in units:
        k = K[b, h].cpu().numpy()
        v = V[b, h].cpu().numpy()
        qw = QW[b, h * G:(h + 1) * G].cpu().numpy()
        got = kept_pos[b, h].cpu().numpy()
        assert np.all(np.diff(got) > 0), "kept positions must ascend"
        if keep >= T:
            assert np.array_equal(got, np.arange(T))
        else:
            s = snapkv.window_scores(qw, k[:T])
            pooled = snapkv.max_pool(s, pool)
            pre = np.arange(T - W)
            near += check_topk(pooled, pre, keep - W, got[got < T - W], exact, f"{tag} snap b{b} h{h}")
            decisions += 1
            assert np.array_equal(got[got >= T - W], np.arange(T - W, T))
        # the compact cache holds exactly the kept rows, and page min/max match
        gk = cache.t["k"][b, h, :kept_n].cpu().numpy()
        assert np.array_equal(gk.view(np.uint16), k[got].view(np.uint16))
        npg = kept_n // 16
        kmin, kmax = rocket.page_minmax(k[got], 16, npg)
        assert np.array_equal(cache.t["kmin"][b, h, :, :npg].cpu().numpy().T.astype(np.float64), kmin)
        assert np.array_equal(cache.t["kmax"][b, h, :, :npg].cpu().numpy().T.astype(np.float64), kmax)
        host[(b, h)] = (list(k[got]), list(v[got]), k, v)
    page_idx = torch.zeros((B, Hkv, kp), dtype=torch.int32, device=dev)
    for s in range(steps):
        kn = K[:, :, T + s].contiguous()
        vn = V[:, :, T + s].contiguous()
        q = Q[s].contiguous()
        out = torch.empty_like(q)
        if fused == "step":
            page_idx.fill_(-7)
            mkv.mkv_rocket_step(cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), cache.c, page_idx.data_ptr(),
                                out.data_ptr())
        elif fused:
            mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), cache.c)
            page_idx.fill_(-7)
            mkv.mkv_rocket_decode(cfg, q.data_ptr(), cache.c, page_idx.data_ptr(), out.data_ptr())
        else:
            mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), cache.c)
            mkv.mkv_rocket_select(cfg, q.data_ptr(), cache.c, page_idx.data_ptr())
            mkv.mkv_decode_attention(cfg, q.data_ptr(), cache.c, None, page_idx.data_ptr(), out.data_ptr(),
                                     ws.data_ptr(), nws)
        got = out.float().cpu().numpy()
        pidx = page_idx.cpu().numpy()
        for (b, h) in units:
            Kc, Vc, k, v = host[(b, h)]
            Kc.append(k[T + s])
            Vc.append(v[T + s])
            n = len(Kc)
            qh = q[b, h * G:(h + 1) * G].cpu().numpy()
            sel_ref, scores = rocket.select_pages(qh, np.array(Kc), n, 16, kp, rd)
            sel_got = pidx[b, h][pidx[b, h] >= 0]
            assert np.all(np.diff(sel_got) > 0), "pages must ascend"
            ns = rocket.n_scored_pages(n, 16)
            nn = check_topk(scores, np.arange(ns), min(kp, ns), sel_got, exact, f"{tag} pages step {s} b{b} h{h}")
            near += nn
            decisions += 1
            ref, _, _ = rocket.decode(qh, np.array(Kc), np.array(Vc), n, 16, kp, rd, forced_pages=sel_got)
            assert_close(got[b, h * G:(h + 1) * G], ref, f"{tag} step {s} b{b} h{h}")
    assert mkv.mkv_get_status() == 0
    record(f"rocket {tag} ({ {False: 'two calls', True: 'fused decode', 'step': 'one-launch step'}[fused] })", near, decisions)
    return near


@pytest.mark.parametrize("fused", [False, True, "step"])
def test_tiny_exact(fused):
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = synth.tiny()
    x = synth.host_inputs(w, seed=tiny_seed())
    K, V = to_dev(x["k"][0], dev), to_dev(x["v"][0], dev)
    QW = to_dev(x["q_prompt"][0, :, :, w.T - w.snap_window:], dev)
    Q = to_dev(x["q"][:, 0], dev)
    near = run_rocket(w.B, w.Hq, w.Hkv, w.D, w.T, w.steps, w.snap_window, w.snap_pool, w.snap_keep, w.topk_pages,
                      w.topq_dims, K, V, QW, Q, dev, True, [(0, 0), (0, 1)], "tiny", fused)
    assert near == 0


@pytest.mark.parametrize("fused", [False, True, "step"])
def test_keep_everything_is_full_attention(fused):
    """keep >= T and k_p >= pages: every step attends the whole cache."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(8)
    B, Hq, Hkv, D, T, steps = 2, 8, 2, 64, 150, 3
    K = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    QW = rng.standard_normal((B, Hq, 8, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    run_rocket(B, Hq, Hkv, D, T, steps, 8, 7, 160, 64, 16, to_dev(K, dev), to_dev(V, dev), to_dev(QW, dev),
               to_dev(Q, dev), dev, False, [(0, 0), (1, 1)], "all", fused)


@pytest.mark.parametrize("G,D,fused", [(1, 128, False), (8, 64, False), (1, 128, True), (8, 64, True),
                                       (4, 128, True), (2, 64, True), (4, 128, "step"), (8, 64, "step")])
def test_shapes_lockstep(G, D, fused):
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(G + D)
    B, Hkv, T, steps, W = 2, 2, 700, 5, 16
    Hq = G * Hkv
    K = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    QW = rng.standard_normal((B, Hq, W, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    run_rocket(B, Hq, Hkv, D, T, steps, W, 7, 300, 6, D // 4, to_dev(K, dev), to_dev(V, dev), to_dev(QW, dev),
               to_dev(Q, dev), dev, False, [(0, 1), (1, 0)], f"G{G}D{D}", fused)


@pytest.mark.parametrize("G,D,W", [(8, 64, 40), (4, 128, 100), (2, 128, 130)])
def test_window_spanning_query_blocks(G, D, W):
    """Observation windows longer than one 128-row query block (W > 128/G): the prefill scoring's
    column sums over several query blocks with the window's position offset (the one-block window
    kernel does not apply), its row statistics over split key ranges; kept sets in lockstep."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(100 * G + W)
    B, Hkv, T, steps = 2, 2, 1500, 3
    Hq = G * Hkv
    K = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T + steps, D)).astype(np.float16)
    QW = rng.standard_normal((B, Hq, W, D)).astype(np.float16)
    Q = rng.standard_normal((steps, B, Hq, D)).astype(np.float16)
    run_rocket(B, Hq, Hkv, D, T, steps, W, 7, 400, 6, D // 4, to_dev(K, dev), to_dev(V, dev), to_dev(QW, dev),
               to_dev(Q, dev), dev, False, [(0, 1), (1, 0)], f"W{W}G{G}D{D}")


@pytest.mark.parametrize("fused", [False, True, "step"])
def test_full_size_lockstep(fused):
    """B=4, T=32768 -> keep 4096, W=32, pool 7, top-64 pages over top-32 dims: one layer in
    lockstep with the oracle -- 16 steps on two (batch, kv-head) units for the two-call and fused
    paths, 48 steps on four units for the one-launch step the bench runs."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    w = synth.rocket_32k(1024)
    n, units = (48, [(0, 0), (1, 2), (2, 5), (3, 7)]) if fused == "step" else (16, [(0, 0), (3, 7)])
    x = synth.device_layer_inputs(w, seed=12, layer=0, device=dev, n_tokens=w.T + n, with_prompt_queries=True)
    QW = x["q_prompt"][:, :, w.T - w.snap_window:].contiguous()
    tag = "rocket1024-b4-t32768" + {False: "-two-calls", True: "-fused", "step": "-step"}[fused]
    run_rocket(w.B, w.Hq, w.Hkv, w.D, w.T, n, w.snap_window, w.snap_pool, w.snap_keep, w.topk_pages,
               w.topq_dims, x["k"], x["v"], QW, x["q"][:n], dev, False, units, tag, fused)


def test_fused_short_contexts():
    """T_len of 0, 1, 16, 17 and 40 in one batch (no candidate page, one partial page, a full page
    plus the newest token's page...): the fused step against the oracle, page list -1 padded."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(31)
    lens = [0, 1, 16, 17, 40]
    B, Hq, Hkv, D, kp, rd = len(lens), 8, 2, 64, 2, 16
    G = Hq // Hkv
    T_cap = 48
    cfg = mkv.config(mkv.MKV_ROCKET, B, Hq, Hkv, D, snap_window=8, snap_pool=7, snap_keep=64, page_size=16,
                     topk_pages=kp, topq_dims=rd)
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    K = rng.standard_normal((B, Hkv, T_cap, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T_cap, D)).astype(np.float16)
    cache.t["k"].copy_(to_dev(K, dev))
    cache.t["v"].copy_(to_dev(V, dev))
    for b in range(B):
        for h in range(Hkv):
            npg = T_cap // 16
            kmin, kmax = rocket.page_minmax(K[b, h], 16, npg)
            cache.t["kmin"][b, h] = to_dev(kmin.T.astype(np.float16), dev)
            cache.t["kmax"][b, h] = to_dev(kmax.T.astype(np.float16), dev)
    cache.t["T_len"].copy_(torch.tensor(lens, dtype=torch.int32))
    q = to_dev(rng.standard_normal((B, Hq, D)).astype(np.float16), dev)
    out = torch.full_like(q, float("nan"))
    page_idx = torch.full((B, Hkv, kp), -7, dtype=torch.int32, device=dev)
    mkv.mkv_rocket_decode(cfg, q.data_ptr(), cache.c, page_idx.data_ptr(), out.data_ptr())
    got = out.float().cpu().numpy()
    pidx = page_idx.cpu().numpy()
    for b, n in enumerate(lens):
        for h in range(Hkv):
            qh = q[b, h * G:(h + 1) * G].cpu().numpy()
            if n == 0:
                assert np.all(got[b, h * G:(h + 1) * G] == 0) and np.all(pidx[b, h] == -1)
                continue
            sel, _ = rocket.select_pages(qh, K[b, h, :n], n, 16, kp, rd)
            assert pidx[b, h][pidx[b, h] >= 0].tolist() == sel.tolist()
            assert np.all(pidx[b, h][len(sel):] == -1)
            ref, _, _ = rocket.decode(qh, K[b, h, :n], V[b, h, :n], n, 16, kp, rd)
            assert_close(got[b, h * G:(h + 1) * G], ref, f"n={n} h{h}")


def test_step_equals_append_then_decode():
    """mkv_rocket_step against mkv_append_kv + mkv_rocket_decode on twin caches, over 40 steps that
    complete pages and then fill the cache: identical outputs, page lists, K/V rows, page bounds and
    lengths; a full cache is not appended, keeps its length, raises MKV_FLAG_CACHE_FULL and
    attends to its tokens."""
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(44)
    B, Hq, Hkv, D, kp, rd = 3, 8, 2, 128, 4, 32
    T0, T_cap, steps = [20, 47, 64], 96, 40           # entry 2 is full from step 32 on
    cfg = mkv.config(mkv.MKV_ROCKET, B, Hq, Hkv, D, snap_window=8, snap_pool=7, snap_keep=64, page_size=16,
                     topk_pages=kp, topq_dims=rd)
    K = rng.standard_normal((B, Hkv, T_cap + steps, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T_cap + steps, D)).astype(np.float16)
    twins = []
    for _ in range(2):
        cache = caches.alloc_cache(cfg, T_cap, device=dev)
        cache.t["k"].copy_(to_dev(K[:, :, :T_cap], dev))
        cache.t["v"].copy_(to_dev(V[:, :, :T_cap], dev))
        for b in range(B):
            for h in range(Hkv):
                npg = T0[b] // 16
                kmin, kmax = rocket.page_minmax(K[b, h, :T0[b]], 16, npg)
                cache.t["kmin"][b, h, :, :npg] = to_dev(kmin.T.astype(np.float16), dev)
                cache.t["kmax"][b, h, :, :npg] = to_dev(kmax.T.astype(np.float16), dev)
        cache.t["T_len"].copy_(torch.tensor(T0, dtype=torch.int32))
        twins.append(cache)
    a, c = twins
    full_seen = False
    for s in range(steps):
        kn = to_dev(K[:, :, T_cap + s], dev)          # rows the caches do not hold yet
        vn = to_dev(V[:, :, T_cap + s], dev)
        q = to_dev(rng.standard_normal((B, Hq, D)).astype(np.float16), dev)
        oa, oc = torch.empty_like(q), torch.empty_like(q)
        pa = torch.full((B, Hkv, kp), -7, dtype=torch.int32, device=dev)
        pc = torch.full_like(pa, -7)
        will_fill = [int(a.t["T_len"][b]) >= T_cap for b in range(B)]
        mkv.mkv_append_kv(cfg, kn.data_ptr(), vn.data_ptr(), a.c)
        fa = mkv.mkv_get_status()
        mkv.mkv_rocket_decode(cfg, q.data_ptr(), a.c, pa.data_ptr(), oa.data_ptr())
        mkv.mkv_rocket_step(cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), c.c, pc.data_ptr(), oc.data_ptr())
        fc = mkv.mkv_get_status()
        assert fa == fc == (mkv.MKV_FLAG_CACHE_FULL if any(will_fill) else 0), f"step {s}: flags {fa} {fc}"
        full_seen |= any(will_fill)
        assert torch.equal(oa.view(torch.int16), oc.view(torch.int16)), f"step {s}: outputs differ"
        assert torch.equal(pa, pc), f"step {s}: page lists differ"
        for key in ("T_len", "k", "v", "kmin", "kmax"):
            assert torch.equal(a.t[key].view(torch.int16) if key != "T_len" else a.t[key],
                               c.t[key].view(torch.int16) if key != "T_len" else c.t[key]), f"step {s}: {key}"
    assert full_seen
