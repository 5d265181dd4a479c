"""GPU parity of the prefill scoring passes (the causal column sums that H2O's prefill keeps by,
Section 2.1 H2O paragraph): with a budget that holds the whole prompt nothing is dropped, so the
cache's accumulated score of every position is that position's prefill score, compared with the
fp64 oracle at every position.  Shapes span several 128-key tiles and 128-row query blocks with
ragged tails, every group size and both head dimensions."""
import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
from oracle import h2o
from paper_2609_07966_gb300 import caches

from gpu_util import to_dev, torch_cuda

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("G,D,T", [(1, 64, 129), (2, 128, 300), (4, 128, 1000), (8, 64, 777), (4, 64, 1),
                                   (8, 128, 2049)])
def test_full_keep_scores_every_position(G, D, T):
    torch = torch_cuda()
    dev = torch.device("cuda")
    rng = np.random.default_rng(1000 * G + D + T)
    B, Hkv = 2, 2
    Hq = G * Hkv
    K = rng.standard_normal((B, Hkv, T, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T, D)).astype(np.float16)
    QP = rng.standard_normal((B, Hq, T, D)).astype(np.float16)
    H = R = (T + 1) // 2 + 1                       # H + R > T: every position kept
    cfg = mkv.config(mkv.MKV_H2O, B, Hq, Hkv, D, h2o_heavy=H, h2o_recent=R)
    cache = caches.alloc_cache(cfg, H + R + 1, device=dev)
    ws, nws = caches.workspace(cfg, max(T, H + R + 1), device=dev)
    Kd, Vd, Qd = to_dev(K, dev), to_dev(V, dev), to_dev(QP, dev)
    mkv.mkv_h2o_prefill(cfg, Qd.data_ptr(), Kd.data_ptr(), Vd.data_ptr(), T, cache.c, ws.data_ptr(), nws)
    assert mkv.mkv_get_status() == 0
    pos = cache.t["pos"].cpu().numpy()
    acc = cache.t["acc"].cpu().numpy()
    for b in range(B):
        for h in range(Hkv):
            ref = h2o.prefill_scores(QP[b, h * G:(h + 1) * G], K[b, h])
            np.testing.assert_array_equal(pos[b, h, :T], np.arange(T))
            np.testing.assert_allclose(acc[b, h, :T], ref, rtol=2e-4, atol=1e-5, err_msg=f"b{b} h{h}")


def test_wait_timeout_raises_status_and_context_survives():
    """A bounded device wait that nothing completes (the prefill's wait routine) gives up, raises
    MKV_FLAG_WAIT_TIMEOUT (mkv_get_status: MKV_ERR_TIMEOUT), and the next scoring call runs clean."""
    torch = torch_cuda()
    import time
    assert mkv.mkv_get_status() == 0
    t0 = time.perf_counter()
    mkv.mkv_wait_timeout_selftest(20)
    flags = mkv.mkv_get_status()
    waited = time.perf_counter() - t0
    assert flags & mkv.MKV_FLAG_WAIT_TIMEOUT
    assert 0.015 < waited < 5.0, waited
    assert mkv.mkv_get_status() == 0                     # the word was cleared
    test_full_keep_scores_every_position(4, 128, 1000)  # the context is still usable
