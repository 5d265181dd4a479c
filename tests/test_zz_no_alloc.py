"""The workspace-free FP16 decode entry point matches the regular one.

mkv_decode_attention_noalloc serves callers that cannot allocate device memory
or pass a scratch buffer (a host framework that owns every allocation, or a
fixed C interface without a workspace argument); it keeps its split partials in
a fixed array inside the library instead.  This test calls it twice in a row
through the C ABI, each time on different inputs, and compares every output
with mkv_decode_attention's on the same inputs, within the attention
tolerance the other GPU tests use.  It is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
from paper_2609_07966_gb300 import caches

from gpu_util import assert_close, to_dev, torch_cuda

pytestmark = pytest.mark.gpu


def test_noalloc_matches_workspace_decode_twice():
    torch = torch_cuda()
    dev = torch.device("cuda")
    L = mkv.lib()
    rng = np.random.default_rng(2024)
    B, Hq, Hkv, D, T_cap = 4, 32, 8, 128, 3000
    lens = [2900, 1, 777, 2048]
    cfg = mkv.config(mkv.MKV_FP16, B, Hq, Hkv, D)
    cache = caches.alloc_cache(cfg, T_cap, device=dev)
    K = rng.standard_normal((B, Hkv, T_cap, D)).astype(np.float16)
    V = rng.standard_normal((B, Hkv, T_cap, D)).astype(np.float16)
    cache.t["k"].copy_(to_dev(K, dev))
    cache.t["v"].copy_(to_dev(V, dev))
    cache.t["T_len"].copy_(torch.tensor(lens, dtype=torch.int32))
    ws, nws = caches.workspace(cfg, T_cap, device=dev)
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        q = to_dev(rng.standard_normal((B, Hq, D)).astype(np.float16), dev)
        ref = torch.empty_like(q)
        got = torch.full_like(q, float("nan"))
        mkv.mkv_decode_attention(cfg, q.data_ptr(), cache.c, None, 0, ref.data_ptr(), ws.data_ptr(), nws)
        st = L.mkv_decode_attention_noalloc(ctypes.byref(cfg), q.data_ptr(), ctypes.byref(cache.c), got.data_ptr(),
                                            stream)
        assert st == mkv.MKV_OK, mkv.mkv_last_error()
        torch.cuda.synchronize()
        assert_close(got.float().cpu().numpy(), ref.float().cpu().numpy(), f"call {call}")
        # a different context length before the second call
        cache.t["T_len"].copy_(torch.tensor([l // 2 + 1 for l in lens], dtype=torch.int32))


def test_noalloc_rejects_oversized_and_non_fp16():
    L = mkv.lib()
    big = mkv.config(mkv.MKV_FP16, 64, 64, 8, 128)
    cache = mkv.mkv_cache()
    cache.T_cap = 1 << 20
    cache.T_len = 8
    cache.k = 16
    cache.v = 32
    st = L.mkv_decode_attention_noalloc(ctypes.byref(big), 64, ctypes.byref(cache), 128, None)
    assert st == mkv.MKV_ERR_WORKSPACE and "built-in" in mkv.mkv_last_error()
    h2o = mkv.config(mkv.MKV_H2O, 1, 8, 2, 64, h2o_heavy=4, h2o_recent=4)
    st = L.mkv_decode_attention_noalloc(ctypes.byref(h2o), 64, ctypes.byref(cache), 128, None)
    assert st == mkv.MKV_ERR_UNSUPPORTED
