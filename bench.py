"""Decode-attention throughput over a compressed KV cache on one GB300.

One step = one decode step of the whole hot path over all 32 layers of a
Llama-3-8B-shaped attention (32 query / 8 KV heads, D = 128) for the batch:
per layer, append the new token to the compressed cache (KVQuant: quantize it)
and run decode attention over the cache.  tokens/s = batch / step time.

Default workload: KVQuant NUQ 4-bit, B = 8, context 8192 (the KVQuant decode
configuration); other workloads via --workload.  Inputs are synthetic and
seeded (synth), every layer has its own cache buffers, and one step reads
more than the 129 MB L2 holds, so no flush is needed between steps.

Besides the headline workload the line carries ``per_config`` (the other configurations at their own
sizes: FP16 8K, KVQuant 3/2-bit, H2O 20 % at 16K, RocketKV 1024 at 32K) and ``sweep``: the ten
configurations (FP16; KVQuant NUQ 4/3/2-bit; H2O 10/20/40 %; RocketKV budgets 1024/2048/4096) at
contexts 4K/16K/64K/128K with batch 32/16/4/1, each a 32-layer step.  There the H2O decode cache is
filled directly with the budget's heavy and recent slots (scoring a 128K prompt is not part of a
decode step).  Every row gives the step time, tokens/s, the decode launch's algorithmic bytes,
GB/s and fraction of the measured and of the 8 TB/s peak, and the resident and peak KV bytes.

Under torchrun each rank runs an independent replica on its own GPU (the
units -- batch entries, heads, layers -- are independent; no collective).
--impl reference times the fp64 CPU oracle on a bounded sample instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

for _v in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "OMP_NUM_THREADS"):
    os.environ.setdefault(_v, "1")          # the CPU oracle runs on one core

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

WORKLOADS = {
    "kvquant4": lambda: synth.kvquant_8k(4),
    "kvquant3": lambda: synth.kvquant_8k(3),
    "kvquant2": lambda: synth.kvquant_8k(2),
    "fp16": lambda: synth.Workload(name="fp16_b8_t8192", B=8, L=32, Hq=32, Hkv=8, D=128, T=8192, steps=128),
    "h2o20": lambda: synth.h2o_16k(20),
    "rocket1024": lambda: synth.rocket_32k(1024),
}
METHOD_OF = {"kvquant4": "kvquant", "kvquant3": "kvquant", "kvquant2": "kvquant", "fp16": "fp16",
             "h2o20": "h2o", "rocket1024": "rocket"}
METRIC = "compressed-KV decode attn tokens/s and HBM GB/s (fraction of ~8 TB/s) per config"


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples (50 ms) around the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.rows = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == 7:
                self.rows.append(parts)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait()
        self.thread.join(timeout=2)
        sm = [float(r[0]) for r in self.rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4) if r[3 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.rows)}


# --------------------------------------------------------------------------- GPU arm

# Algorithmic bytes of one decode launch of one layer (the compressed-KV bytes the method must read),
# per (batch, kv-head) unit: the roofline's numerator.

def alg_bytes_fp16(units: int, T: int, D: int) -> int:
    """K and V rows of the T tokens, fp16."""
    return units * T * D * 2 * 2


def alg_bytes_kvquant(units: int, T: int, D: int, bits: int, n_v: int, n_key_outliers: int) -> int:
    """Per token: key and value codes (D*bits/8 bytes each), the value range (lo, scale: 8 B), n_v
    value outliers of 4 B and the key-outlier CSR offset (4 B); plus 4 B per key-outlier entry."""
    return units * T * (2 * (D * bits // 8) + 8 + 4 * n_v + 4) + 4 * n_key_outliers


def alg_bytes_h2o(units: int, held: int, D: int) -> int:
    """K and V rows of the held slots, fp16."""
    return units * held * D * 2 * 2


def overhead_bytes_h2o(units: int, slots: int, G: int) -> int:
    """What the H2O decode moves besides the model: each slot's position (4 B, the mask) and the G
    fp32 logits it writes for the score update."""
    return units * slots * (4 + 4 * G)


def alg_bytes_rocket(units: int, n: int, D: int, k_p: int, r_d: int, page: int = 16) -> int:
    """The full pages before the newest token's page are candidates; per candidate page the chosen
    r_d dims' min and max (fp16); K and V rows of the k_p chosen pages and of the tail page (the
    newest token's, 1..page tokens)."""
    ns = (n - 1) // page if n > 0 else 0
    tail = n - page * ns
    return units * ((min(k_p, ns) * page + tail) * D * 2 * 2 + ns * r_d * 2 * 2)


class Runner:
    """All layers of one workload resident on the device, plus the step."""

    def __init__(self, name: str, w, dev, seed: int, extra_steps: int, method: str | None = None,
                 synthetic_h2o_cache: bool = False):
        """synthetic_h2o_cache: fill the H2O decode cache (heavy + recent slots, their positions and
        scores) directly from the seeded inputs instead of scoring the whole prompt (the sweep's long
        contexts); the decode step then does exactly the same work."""
        import torch
        import paper_2609_07966_gb300 as mkv
        from paper_2609_07966_gb300 import caches
        self.torch, self.mkv, self.name, self.w, self.dev = torch, mkv, name, w, dev
        self.method = method or METHOD_OF[name]
        B, Hq, Hkv, D = w.B, w.Hq, w.Hkv, w.D
        mk = {"fp16": mkv.MKV_FP16, "kvquant": mkv.MKV_KVQUANT, "h2o": mkv.MKV_H2O, "rocket": mkv.MKV_ROCKET}
        kw = {}
        if self.method == "kvquant":
            kw = dict(bits=w.bits, quant_mode=mkv.MKV_QUANT_NUQ if w.quant_mode == "nuq" else mkv.MKV_QUANT_UNIFORM,
                      outlier_frac=w.outlier_frac, rope_theta=w.theta)
        elif self.method == "h2o":
            kw = dict(h2o_heavy=w.h2o_heavy, h2o_recent=w.h2o_recent)
        elif self.method == "rocket":
            kw = dict(snap_window=w.snap_window, snap_pool=w.snap_pool, snap_keep=w.snap_keep, page_size=w.page,
                      topk_pages=w.topk_pages, topq_dims=w.topq_dims)
        self.cfg = mkv.config(mk[self.method], B, Hq, Hkv, D, **kw)
        if self.method == "h2o":
            self.T_cap = w.h2o_heavy + w.h2o_recent + 1
        elif self.method == "rocket":
            self.T_cap = (min(w.T, w.snap_keep) + extra_steps + 15) // 16 * 16
        else:
            self.T_cap = w.T + extra_steps + 64
        self.layers = []
        self.q, self.kn, self.vn, self.out, self.pidx = [], [], [], [], []
        # prefill-side calls need workspace for the whole prompt
        self.ws, self.nws = caches.workspace(self.cfg, max(self.T_cap, w.T), device=dev)
        if self.method == "h2o":
            # layer l's score update reads the logits its decode left in the workspace, and nothing of
            # layer l + 1 depends on it: it runs on a side stream while the next layer decodes, the
            # layers alternating between two workspaces (a decode first waits for the last update
            # that read its workspace)
            self.ws_alt, _ = caches.workspace(self.cfg, max(self.T_cap, w.T), device=dev)
            self.side = torch.cuda.Stream(device=dev)
            self.overlap = True                 # False: the updates in line on the main stream
            self.dec_ev = [torch.cuda.Event() for _ in range(2)]
            self.upd_ev = [torch.cuda.Event() for _ in range(2)]
        if self.method == "kvquant":
            self.rope = torch.empty((self.T_cap, D // 2, 2), dtype=torch.float32, device=dev)
            mkv.mkv_rope_table(D, w.theta, self.T_cap, self.rope.data_ptr())
        t_setup = time.perf_counter()
        for l in range(w.L):
            syn = self.method == "h2o" and synthetic_h2o_cache
            n_tok = w.h2o_heavy + w.h2o_recent + 1 if syn else w.T + 1
            x = synth.device_layer_inputs(w, seed, l, device=dev, n_tokens=n_tok,
                                          with_prompt_queries=self.method in ("h2o", "rocket") and not syn)
            cache = caches.alloc_cache(self.cfg, self.T_cap, device=dev)
            qp = None
            if self.method == "fp16":
                cache.t["k"][:, :, :w.T] = x["k"][:, :, :w.T]
                cache.t["v"][:, :, :w.T] = x["v"][:, :, :w.T]
                cache.t["T_len"].fill_(w.T)
            elif self.method == "kvquant":
                qp = caches.alloc_quant_params(self.cfg, 1, device=dev)
                qp.t["rope"] = self.rope
                qp.c.rope = self.rope.data_ptr()
                qp.c.rope_len = self.T_cap
                ncal = min(w.T, 4096)
                k0, v0 = x["k"][0].contiguous(), x["v"][0].contiguous()     # batch entry 0 calibrates
                mkv.mkv_kvquant_calibrate(self.cfg, k0.data_ptr(), v0.data_ptr(), ncal, w.T + 1, qp.c,
                                          self.ws.data_ptr(), self.nws)
                kp = x["k"][:, :, :w.T].contiguous()
                vp = x["v"][:, :, :w.T].contiguous()
                mkv.mkv_quantize_kv(self.cfg, qp.c, kp.data_ptr(), vp.data_ptr(), w.T, cache.c)
                del kp, vp
            elif self.method == "h2o" and syn:
                n = w.h2o_heavy + w.h2o_recent
                cache.t["k"][:, :, :n] = x["k"][:, :, :n]
                cache.t["v"][:, :, :n] = x["v"][:, :, :n]
                pos = torch.empty(n, dtype=torch.int32, device=dev)
                hv = torch.arange(w.h2o_heavy, device=dev, dtype=torch.int64)
                pos[:w.h2o_heavy] = (hv * (w.T - w.h2o_recent) // max(w.h2o_heavy, 1)).to(torch.int32)
                pos[w.h2o_heavy:] = torch.arange(w.T - w.h2o_recent, w.T, device=dev, dtype=torch.int32)
                cache.t["pos"][:, :, :n] = pos
                g = torch.Generator(device=dev)
                g.manual_seed(seed * 1000 + l)
                cache.t["acc"][:, :, :n] = torch.rand((B, Hkv, n), generator=g, device=dev)
                cache.t["slot"].fill_(n)
                cache.t["T_len"].fill_(w.T)
            elif self.method == "h2o":
                kp = x["k"][:, :, :w.T].contiguous()
                vp = x["v"][:, :, :w.T].contiguous()
                mkv.mkv_h2o_prefill(self.cfg, x["q_prompt"].data_ptr(), kp.data_ptr(), vp.data_ptr(), w.T, cache.c,
                                    self.ws.data_ptr(), self.nws)
                del kp, vp
            else:
                kp = x["k"][:, :, :w.T].contiguous()
                vp = x["v"][:, :, :w.T].contiguous()
                qw = x["q_prompt"][:, :, w.T - w.snap_window:].contiguous()
                mkv.mkv_snap_compress(self.cfg, qw.data_ptr(), kp.data_ptr(), vp.data_ptr(), w.T, cache.c, 0,
                                      self.ws.data_ptr(), self.nws)
                del kp, vp, qw
                self.pidx.append(torch.zeros((B, Hkv, w.topk_pages), dtype=torch.int32, device=dev))
            self.layers.append((cache, qp))
            self.q.append(x["q"][0].contiguous())
            self.kn.append(x["k"][:, :, n_tok - 1].contiguous())
            self.vn.append(x["v"][:, :, n_tok - 1].contiguous())
            self.out.append(torch.empty((B, Hq, D), dtype=torch.float16, device=dev))
            del x
        torch.cuda.synchronize()
        self.setup_s = time.perf_counter() - t_setup
        flags = mkv.mkv_get_status()
        assert flags == 0, f"device status flags {flags:#x} after setup"
        self.graph = None
        self.step_fused = True
        # RocketKV: the fused one-launch step unless this shape is too large for it (then append,
        # page choice and sparse attention as three calls)
        # The fused step ranks and attends within one cluster per unit, which suits the 64 pages of
        # the 1024-token budget; with more pages and many units the split-KV decode over the page
        # list (three launches) can be faster.  Above 64 pages both are timed and the faster kept.
        self.rocket_fused = self.method == "rocket"
        if self.rocket_fused:
            try:
                mkv.mkv_rocket_decode(self.cfg, self.q[0].data_ptr(), self.layers[0][0].c, 0, self.out[0].data_ptr())
                torch.cuda.synchronize()
            except mkv.MkvError as e:
                if e.status != mkv.MKV_ERR_UNSUPPORTED:
                    raise
                self.rocket_fused = False
            if self.rocket_fused and w.topk_pages > 64:
                t_fused = time_decode_launches(self, 3)
                self.rocket_fused = False
                t_split = time_decode_launches(self, 3)
                self.rocket_fused = t_fused <= t_split

    def choose_kvquant_step(self, reps=3):
        """KVQuant: the one-launch step (mkv_kvquant_step) or quantize + decode, whichever is faster on
        this shape (both leave the same cache and output bits); a few eager steps of each, timed with
        CUDA events.  Returns both times (ms per step)."""
        torch = self.torch
        t = {}
        for fused in (True, False):
            self.step_fused = fused
            self.step()
            torch.cuda.synchronize()
            st = torch.cuda.current_stream()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            for _ in range(reps):
                self.step()
            e1.record(st)
            torch.cuda.synchronize()
            t[fused] = e0.elapsed_time(e1) / reps
        self.step_fused = t[True] <= t[False]
        return {"one_launch_step": t[True], "quantize_then_decode": t[False],
                "chosen": "one_launch_step" if self.step_fused else "quantize_then_decode"}

    def append(self, l, kn=None, vn=None):
        mkv = self.mkv
        cache, qp = self.layers[l]
        kn = self.kn[l] if kn is None else kn
        vn = self.vn[l] if vn is None else vn
        if self.method == "kvquant":
            mkv.mkv_quantize_kv(self.cfg, qp.c, kn.data_ptr(), vn.data_ptr(), 1, cache.c)
        else:
            mkv.mkv_append_kv(self.cfg, kn.data_ptr(), vn.data_ptr(), cache.c)

    def decode(self, l, q=None, out=None):
        mkv = self.mkv
        cache, qp = self.layers[l]
        q = self.q[l] if q is None else q
        out = self.out[l] if out is None else out
        if self.method == "rocket":           # page choice + sparse attention in one launch
            if self.rocket_fused:
                mkv.mkv_rocket_decode(self.cfg, q.data_ptr(), cache.c, 0, out.data_ptr())
            else:
                pidx = self.pidx[l]
                mkv.mkv_rocket_select(self.cfg, q.data_ptr(), cache.c, pidx.data_ptr())
                mkv.mkv_decode_attention(self.cfg, q.data_ptr(), cache.c, None, pidx.data_ptr(), out.data_ptr(),
                                         self.ws.data_ptr(), self.nws)
            return
        mkv.mkv_decode_attention(self.cfg, q.data_ptr(), cache.c, qp.c if qp else None, 0, out.data_ptr(),
                                 self.ws.data_ptr(), self.nws)

    def layer_step(self, l, q=None, kn=None, vn=None, out=None):
        """One layer of one decode step: append the token, attend (RocketKV: choose pages and attend),
        (update scores)."""
        mkv = self.mkv
        cache, _ = self.layers[l]
        if self.method == "rocket" and not self.rocket_fused:
            self.append(l, kn, vn)
            self.decode(l, q, out)
            return
        if self.method == "rocket":           # append, page choice and attention in one launch
            kn = self.kn[l] if kn is None else kn
            vn = self.vn[l] if vn is None else vn
            q = self.q[l] if q is None else q
            out = self.out[l] if out is None else out
            mkv.mkv_rocket_step(self.cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), cache.c, 0, out.data_ptr())
            return
        torch = self.torch
        ws = self.ws if self.method != "h2o" or l % 2 == 0 else self.ws_alt
        if self.method == "h2o" and self.overlap and l >= 2:
            # (layers 0 and 1 follow the previous step's updates, joined at its end)
            torch.cuda.current_stream().wait_event(self.upd_ev[l % 2])
        if self.method in ("fp16", "h2o", "kvquant") and self.step_fused:
            # append (KVQuant: quantize) and attention in one launch, then (H2O) the update
            kn = self.kn[l] if kn is None else kn
            vn = self.vn[l] if vn is None else vn
            q = self.q[l] if q is None else q
            out = self.out[l] if out is None else out
            try:
                if self.method == "kvquant":
                    mkv.mkv_kvquant_step(self.cfg, self.layers[l][1].c, q.data_ptr(), kn.data_ptr(), vn.data_ptr(),
                                         cache.c, out.data_ptr(), ws.data_ptr(), self.nws)
                else:
                    mkv.mkv_decode_step(self.cfg, q.data_ptr(), kn.data_ptr(), vn.data_ptr(), cache.c,
                                        out.data_ptr(), ws.data_ptr(), self.nws)
            except mkv.MkvError as e:
                # too many splits for the step's ticket counter: nothing was launched; two calls instead
                if e.status != mkv.MKV_ERR_UNSUPPORTED:
                    raise
                self.step_fused = False
                return self.layer_step(l, q, kn, vn, out)
        else:
            self.append(l, kn, vn)
            if self.method == "h2o":
                q = self.q[l] if q is None else q
                out = self.out[l] if out is None else out
                mkv.mkv_decode_attention(self.cfg, q.data_ptr(), cache.c, None, 0, out.data_ptr(), ws.data_ptr(),
                                         self.nws)
            else:
                self.decode(l, q, out)
        if self.method == "h2o" and self.overlap:   # the update on the side stream, after this decode
            main = torch.cuda.current_stream()
            self.dec_ev[l % 2].record(main)
            self.side.wait_event(self.dec_ev[l % 2])
            mkv.mkv_h2o_update(self.cfg, cache.c, ws.data_ptr(), self.nws, stream=self.side.cuda_stream)
            self.upd_ev[l % 2].record(self.side)
        elif self.method == "h2o":
            mkv.mkv_h2o_update(self.cfg, cache.c, ws.data_ptr(), self.nws)

    def join_side(self):
        """The main stream waits for the side stream's score updates (end of a step)."""
        if self.method == "h2o" and self.overlap:
            self.torch.cuda.current_stream().wait_stream(self.side)

    def step(self):
        for l in range(self.w.L):
            self.layer_step(l)
        self.join_side()

    def capture(self):
        torch = self.torch
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.step()                          # warm the launch paths outside capture
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self.step()
        torch.cuda.synchronize()

    def run_step(self):
        if self.graph is not None:
            self.graph.replay()
        else:
            self.step()

    def launches_per_step(self):
        # per layer: FP16 / H2O / KVQuant append (KVQuant: quantize) and attention in one launch (H2O:
        # + score update); RocketKV append, page choice and attention in one launch
        per = {"fp16": 1 if self.step_fused else 2, "kvquant": 1 if self.step_fused else 2,
               "h2o": 2 if self.step_fused else 3,
               "rocket": 1 if self.rocket_fused else 3}[self.method]
        return per * self.w.L

    def decode_bytes(self):
        """Algorithmic bytes one decode launch reads for one layer now (the per-unit byte models of
        the compressed KV cache), the attended tokens, and bytes of implementation overhead the
        launch also moves (reported apart, not in the roofline)."""
        w = self.w
        cache, _ = self.layers[0]
        units = w.B * w.Hkv
        T = int(cache.t["T_len"][0])
        if self.method == "fp16":
            return alg_bytes_fp16(units, T, w.D), T, 0
        if self.method == "kvquant":
            nv = self.mkv.n_value_outliers(w.D, w.outlier_frac)
            n_kout = int(cache.t["k_out_off"][:, :, T].sum())
            return alg_bytes_kvquant(units, T, w.D, w.bits, nv, n_kout), T, 0
        if self.method == "h2o":
            held = int(cache.t["pos"][0, 0].ge(0).sum())
            slots = min(self.T_cap, w.h2o_heavy + w.h2o_recent + 1)
            return alg_bytes_h2o(units, held, w.D), held, overhead_bytes_h2o(units, slots, w.G)
        # the fused step reads only the chosen dims' page bounds: no overhead beyond the model
        return alg_bytes_rocket(units, T, w.D, w.topk_pages, w.topq_dims), T, 0


def time_steps(runner, steps, warmup):
    torch = runner.torch
    for _ in range(warmup):
        runner.run_step()
    torch.cuda.synchronize()
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(steps):
        runner.run_step()
    e1.record(st)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def time_decode_launches(runner, reps):
    """Average duration of one mkv_decode_attention call (one fused decode kernel per layer):
    a CUDA graph of every layer's decode call, replayed `reps` times between CUDA events on the
    launching stream (graph replay removes host launch overhead; the cache is not modified)."""
    torch = runner.torch
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for l in range(runner.w.L):
            runner.decode(l)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for l in range(runner.w.L):
            runner.decode(l)
    for _ in range(2):
        g.replay()
    st = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(st)
    for _ in range(reps):
        g.replay()
    b.record(st)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / (reps * runner.w.L)


def time_e2e(runner, steps, warmup, graph=True):
    """Through the public API with host buffers: per step, one H2D copy of every layer's q and
    new k/v from pinned memory (packed in one buffer), the step's API calls, and one D2H copy of
    every layer's output.  graph: the step (copies included) captured once in a CUDA graph and
    replayed, as a serving loop runs it; otherwise eager launches."""
    torch = runner.torch
    w = runner.w
    ins = [t for l in range(w.L) for t in (runner.q[l], runner.kn[l], runner.vn[l])]
    sizes = [t.numel() for t in ins]
    h_in = torch.cat([t.reshape(-1).cpu() for t in ins]).pin_memory()
    d_in = torch.empty_like(h_in, device=runner.q[0].device)
    views, off = [], 0
    for t, n in zip(ins, sizes):
        views.append(d_in[off:off + n].view(t.shape))
        off += n
    o_shape, o_n = runner.out[0].shape, runner.out[0].numel()
    d_out = torch.empty(w.L * o_n, dtype=runner.out[0].dtype, device=runner.out[0].device)
    h_out = torch.empty(d_out.shape, dtype=d_out.dtype).pin_memory()
    outs = [d_out[l * o_n:(l + 1) * o_n].view(o_shape) for l in range(w.L)]

    def one():
        d_in.copy_(h_in, non_blocking=True)
        for l in range(w.L):
            runner.layer_step(l, views[3 * l], views[3 * l + 1], views[3 * l + 2], outs[l])
        runner.join_side()
        h_out.copy_(d_out, non_blocking=True)

    run = one
    if graph:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            one()                             # the launch paths warmed outside capture
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            one()
        run = g.replay
    for _ in range(warmup):
        run()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        run()
    torch.cuda.synchronize()
    dt = (time.perf_counter() - t0) / steps
    h2d = h_in.numel() * h_in.element_size()
    d2h = h_out.numel() * h_out.element_size()
    return dt, h2d, d2h


def slowest_rank_ms(ms: float, dev) -> float:
    """Step time of the slowest rank: every rank gets the max over ranks (one rank: unchanged).
    Ranks are independent replicas (each decodes its own batch, no collective on the data path),
    so the whole-job value is the units of all ranks over this time."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms
    t = torch.tensor([ms], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_tokens_per_s(batch: int, world: int, ms: float) -> float:
    """Tokens per second of the whole job: every rank decodes `batch` tokens per step."""
    return batch * world / (ms * 1e-3)


def source_digest(path: str) -> str:
    """SHA-256 over a kernel source and every header it includes from its own directory, followed
    recursively (each file once, in the order first reached), so the digest changes whenever any
    code compiled into the kernel's translation unit from this repository changes."""
    import hashlib
    import re
    h = hashlib.sha256()
    seen, todo = set(), [os.path.abspath(path)]
    while todo:
        f = todo.pop(0)
        if f in seen or not os.path.exists(f):
            continue
        seen.add(f)
        text = open(f, "rb").read()
        h.update(os.path.basename(f).encode() + b"\0" + text)
        for inc in re.findall(rb'#include\s+"([^"]+)"', text):
            todo.append(os.path.join(os.path.dirname(f), inc.decode()))
    return h.hexdigest()


def captured_traffic(workload: str):
    """DRAM bytes (read + write) of one decode launch from the committed ncu capture of this workload,
    or None when there is none or the kernel source (with its included headers) changed since."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    ent = json.load(open(path)).get(workload)
    if ent is None:
        return None
    src = os.path.join(ROOT, ent["source"])
    if not os.path.exists(src) or source_digest(src) != ent["source_sha256"]:
        return None
    return ent["dram_bytes_read"] + ent["dram_bytes_write"]


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d.get("hbm_gbs", 6800.0), "measured"
    return 6800.0, "fallback"


def measure_config(name, w, dev, seed, method, steps, warmup, peak, no_graph=False, synthetic_h2o_cache=False):
    """One configuration: device-timed 32-layer step (graph replays), the decode launch's duration and
    algorithmic bytes, and the KV bytes; a row of the per-configuration table."""
    import torch
    rx = Runner(name, w, dev, seed, extra_steps=4 * (steps + warmup) + 8, method=method,
                synthetic_h2o_cache=synthetic_h2o_cache)
    paths = rx.choose_kvquant_step() if rx.method == "kvquant" else None
    if not no_graph:
        rx.capture()
    msx = time_steps(rx, steps, warmup)
    bx, tx, ox = rx.decode_bytes()
    dx = time_decode_launches(rx, 10)
    rres, rpk = rx.mkv.mkv_cache_bytes(rx.cfg, w.T)
    gbs = bx / (dx * 1e-3) / 1e9
    row = {"tokens_per_s": w.B / (msx * 1e-3), "ms_per_step": msx, "batch": w.B, "context": w.T,
           "decode_launch_ms": dx, "decode_alg_bytes": bx, "decode_overhead_bytes": ox, "attended_tokens": tx,
           "decode_gbs": gbs, "frac_of_measured_peak": gbs / peak, "frac_of_8000": gbs / 8000.0,
           "kv_bytes_resident": rres * w.L, "kv_bytes_peak": rpk * w.L, "setup_s": rx.setup_s,
           "gpu_launches_per_step": rx.launches_per_step()}
    if rx.method == "h2o" and synthetic_h2o_cache:
        row["note"] = "decode cache filled directly with the budget's heavy + recent slots (no prefill scoring)"
    if paths is not None:
        row["step_paths_ms"] = paths
    if rx.method in ("fp16", "h2o") and not rx.step_fused:
        row["note"] = "append and attention as two launches (too many splits for the one-launch step)"
    if rx.method == "rocket" and not rx.rocket_fused:
        row["note"] = "append, page choice and split-KV attention over the page list as three launches"
    del rx
    torch.cuda.empty_cache()
    return row


def tensor_peak():
    """(dense fp16/bf16 TFLOP/s burst peak, how it was obtained): fp16 runs at the bf16 rate."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        if "bf16_tflops" in d:
            return d["bf16_tflops"], "measured (cuBLAS bf16 burst; fp16 has the same tensor rate)"
    return 1900.0, "fallback"


def prefill_scoring_flops(B: int, Hq: int, D: int, T: int, rows: int) -> float:
    """FLOPs of the prefill scoring for `rows` query rows at positions T - rows .. T - 1 over T keys:
    2 products (row statistics, then column sums) x 2 D per causal (row, key) pair per query head."""
    W = rows
    pairs = W * (T - W) + W * (W + 1) / 2          # row i (position T - W + i) sees T - W + i + 1 keys
    return 2 * 2 * D * pairs * B * Hq


def measure_setup(dev, seed, reps=5, warmup=3, batch=None):
    """The prefill-side calls timed apart from decode, one layer each: mkv_h2o_prefill on the H2O
    workload (causal scores over the whole prompt, then the heavy + recent keep and gather) and
    mkv_snap_compress on the RocketKV workload (the observation window's scores, pooling, keep and
    gather).  Their scoring is two tcgen05 products of the causal Q K^T (row statistics, then column
    sums): FLOPs = 2 passes x 2 D per causal (query row, key) pair per query head -- the least an
    exact column sum does without storing the T x T scores."""
    import torch
    import paper_2609_07966_gb300 as mkv
    from paper_2609_07966_gb300 import caches
    peak, kind = tensor_peak()
    out = {}
    for name in ("h2o20", "rocket1024"):
        w = WORKLOADS[name]()
        if batch is not None:
            import dataclasses
            w = dataclasses.replace(w, B=batch)
        x = synth.device_layer_inputs(w, seed, 0, device=dev, n_tokens=w.T, with_prompt_queries=True)
        kp = x["k"][:, :, :w.T].contiguous()
        vp = x["v"][:, :, :w.T].contiguous()
        if name == "h2o20":
            cfg = mkv.config(mkv.MKV_H2O, w.B, w.Hq, w.Hkv, w.D, h2o_heavy=w.h2o_heavy, h2o_recent=w.h2o_recent)
            T_cap = w.h2o_heavy + w.h2o_recent + 1
            qp = x["q_prompt"].contiguous()
            rows = w.T
            call = "mkv_h2o_prefill"
        else:
            cfg = mkv.config(mkv.MKV_ROCKET, w.B, w.Hq, w.Hkv, w.D, snap_window=w.snap_window,
                             snap_pool=w.snap_pool, snap_keep=w.snap_keep, page_size=w.page,
                             topk_pages=w.topk_pages, topq_dims=w.topq_dims)
            T_cap = (min(w.T, w.snap_keep) + 15) // 16 * 16
            qp = x["q_prompt"][:, :, w.T - w.snap_window:].contiguous()
            rows = w.snap_window
            call = "mkv_snap_compress"
        del x
        cache = caches.alloc_cache(cfg, T_cap, device=dev)
        ws, nws = caches.workspace(cfg, max(w.T, T_cap), device=dev)
        if name == "h2o20":
            fn = lambda: mkv.mkv_h2o_prefill(cfg, qp.data_ptr(), kp.data_ptr(), vp.data_ptr(), w.T, cache.c,
                                             ws.data_ptr(), nws)
        else:
            fn = lambda: mkv.mkv_snap_compress(cfg, qp.data_ptr(), kp.data_ptr(), vp.data_ptr(), w.T, cache.c, 0,
                                               ws.data_ptr(), nws)
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        st = torch.cuda.current_stream()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for a, b in ev:
            a.record(st)
            fn()
            b.record(st)
        torch.cuda.synchronize()
        ms = statistics.median(a.elapsed_time(b) for a, b in ev)
        flops = prefill_scoring_flops(w.B, w.Hq, w.D, w.T, rows)
        tf = flops / (ms * 1e-3) / 1e12
        out[name] = {"call": call, "workload": f"{w.name}, one layer", "batch": w.B, "context": w.T,
                     "query_rows": rows, "ms": ms, "status": mkv.mkv_get_status(),
                     "roofline": {"bound": "tensor", "achieved": tf, "peak": peak, "unit": "TFLOP/s",
                                  "frac": tf / peak, "peak_kind": kind, "flops_per_call": flops,
                                  "note": "the whole call (scoring, keep, gather) timed; FLOPs of the scoring"}}
        del qp, kp, vp, cache, ws
        torch.cuda.empty_cache()
    return out


# --------------------------------------------------------------------------- CPU oracle arm

def oracle_tokens_per_s(name: str, w, budget_s: float, seed: int = 0):
    """The fp64 oracle's decode step, timed on one (layer, batch, kv-head) unit of the
    workload repeated until ``budget_s`` seconds of oracle work; scaled to the step.

    Returns (tokens/s for the whole workload, sample description)."""
    from oracle import attention, kvquant
    method = METHOD_OF[name]
    rng = np.random.default_rng(seed)
    T = w.T
    scale = np.exp(rng.uniform(np.log(0.1), np.log(10), w.D)) if method == "kvquant" else 1.0
    k = (rng.standard_normal((T + 1, w.D)) * scale).astype(np.float16)
    v = rng.standard_normal((T + 1, w.D)).astype(np.float16)
    q = rng.standard_normal((w.G, w.D)).astype(np.float16)
    if method == "kvquant":
        p = kvquant.calibrate(k[:min(T, 4096)], v[:min(T, 4096)], w.bits, w.quant_mode, w.outlier_frac)
        qh = kvquant.quantize_head(k[:T], v[:T], p)

        def unit():
            new = kvquant.quantize_head(k[T:T + 1], v[T:T + 1], p)     # the step's append
            full = kvquant.QuantizedHead(*[np.concatenate([a, b]) for a, b in zip(
                (qh.k_codes, qh.k_mask, qh.k_raw, qh.v_codes, qh.v_mask, qh.v_lo, qh.v_scale, qh.v_raw),
                (new.k_codes, new.k_mask, new.k_raw, new.v_codes, new.v_mask, new.v_lo, new.v_scale, new.v_raw))])
            kvquant.decode_head(q, full, p, w.theta)
    elif method == "h2o":
        from oracle import h2o
        n = w.h2o_heavy + w.h2o_recent
        st = h2o.H2OHead(np.arange(n), k[:n], v[:n], np.abs(rng.standard_normal(n)))

        def unit():
            h2o.decode_step(st, q, k[n], v[n], T, w.h2o_heavy, w.h2o_recent)
    elif method == "rocket":
        from oracle import rocket
        n = min(T, w.snap_keep) + 1

        def unit():
            rocket.decode(q, k[:n], v[:n], n, w.page, w.topk_pages, w.topq_dims)
    else:
        def unit():
            attention.attend(q, k, v)
    t_units, n_units = 0.0, 0
    while t_units < budget_s and n_units < 1000:
        t0 = time.perf_counter()
        unit()
        t_units += time.perf_counter() - t0
        n_units += 1
    per_unit = t_units / n_units
    step_s = per_unit * w.B * w.Hkv * w.L
    sample = (f"{n_units} decodes of one (layer, batch, kv-head) unit of {name} at T={T} "
              f"({per_unit * 1e3:.1f} ms each), scaled to the step's B*Hkv*L={w.B * w.Hkv * w.L} units")
    return w.B / step_s, sample


def _oracle_worker(args):
    name, wd, budget, seed = args
    return oracle_tokens_per_s(name, synth.Workload(**wd), budget, seed)[0]


def oracle_tokens_per_s_all_cores(name: str, w, budget_s: float, seed: int = 0):
    """The same oracle timing on every host core at once: one single-threaded worker process per core
    (spawned, so no CUDA state is inherited), each decoding its own units; tokens/s add up."""
    import dataclasses
    import multiprocessing as mp
    n = os.cpu_count() or 1
    with mp.get_context("spawn").Pool(n) as pool:
        vals = pool.map(_oracle_worker, [(name, dataclasses.asdict(w), budget_s, seed + i) for i in range(n)])
    return float(sum(vals)), n


# --------------------------------------------------------------------------- main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="mkv", choices=["mkv", "reference"])
    ap.add_argument("--workload", default="kvquant4", choices=sorted(WORKLOADS))
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle work for cpu_baseline")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--layers", type=int, default=None,
                    help="profiling only: fewer layers than the workload (the line is then not a bench number)")
    ap.add_argument("--per-config", default="fp16,kvquant3,kvquant2,h2o20,rocket1024",
                    help="other workloads measured after the headline one (comma list, '' for none)")
    ap.add_argument("--sweep", type=int, default=1,
                    help="1: also measure the ten configurations at contexts 4K/16K/64K/128K (batch 32/16/4/1)")
    ap.add_argument("--sweep-steps", type=int, default=5, help="timed steps per sweep configuration")
    ap.add_argument("--cpu-all-cores", type=int, default=1, help="1: also time the oracle on every host core")
    ap.add_argument("--setup", type=int, default=1,
                    help="1: also time the prefill-side calls (H2O prefill, SnapKV compression) on their workloads")
    ap.add_argument("--only-setup", type=int, default=0,
                    help="profiling: time only the prefill-side calls and print their JSON (not a bench line)")
    ap.add_argument("--setup-batch", type=int, default=None,
                    help="profiling: batch of the prefill-side workloads (a smaller case for ncu)")
    ap.add_argument("--profile", action="store_true",
                    help="profiling only: run warmup + steps and exit (for ncu), no JSON line")
    args = ap.parse_args()

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    w = WORKLOADS[args.workload]()
    if args.layers is not None:
        import dataclasses
        w = dataclasses.replace(w, L=args.layers)
    config = {"workload": w.name, "method": METHOD_OF[args.workload], "batch": w.B, "context": w.T, "layers": w.L,
              "heads_q": w.Hq, "heads_kv": w.Hkv, "head_dim": w.D, "l2": "inputs larger than L2 (no flush)"}

    if args.impl == "reference":
        if rank != 0:
            return
        steps = max(1, args.steps)
        vals, sample = [], ""
        budget = min(args.cpu_budget, 120.0 / (steps + args.warmup))
        for i in range(args.warmup + steps):
            v, sample = oracle_tokens_per_s(args.workload, w, budget, seed=args.seed + i)
            if i >= args.warmup:
                vals.append(v)
        value = statistics.mean(vals)
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
                "steps": steps, "warmup": args.warmup, "ms_per_step": 1e3 * w.B / value,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic", "config": config,
                "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle", "sample": sample,
                                 "extrapolated": True},
                "extrapolated": True,
                "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import torch
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if args.only_setup:
        print(json.dumps({"setup": measure_setup(dev, args.seed, batch=args.setup_batch)}))
        return

    total = args.warmup + args.steps
    runner = Runner(args.workload, w, dev, args.seed + rank, extra_steps=4 * total + 8)
    step_paths = runner.choose_kvquant_step() if runner.method == "kvquant" else None
    if not args.no_graph:
        runner.capture()
    if args.profile:
        for _ in range(total):
            runner.run_step()
        torch.cuda.synchronize()
        return

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    time.sleep(0.3)                              # first samples before the warm-up begins
    ms = time_steps(runner, args.steps, args.warmup)
    clk = clocks.stop()
    clk["window"] = "sampled every 50 ms from just before the warm-up to the end of the timed steps"
    ms = slowest_rank_ms(ms, dev)
    if world > 1:
        torch.distributed.barrier()

    alg_bytes, T_now, ovh_bytes = runner.decode_bytes()
    dec_ms = time_decode_launches(runner, 10)
    e2e_s, h2d, d2h = time_e2e(runner, max(1, min(args.steps, 5)), 1, graph=not args.no_graph)
    peak, peak_kind = peaks()
    achieved = alg_bytes / (dec_ms * 1e-3) / 1e9
    value = whole_job_tokens_per_s(w.B, world, ms)
    res, pk = runner.mkv.mkv_cache_bytes(runner.cfg, w.T)
    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f16" if runner.method != "kvquant" else f"u{w.bits}+f16",
            "data": "synthetic (seeded, device-generated)", "config": config,
            "gpu_launches": runner.launches_per_step() * args.steps,
            "e2e": {"value": w.B * world / e2e_s, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "cuda_graph": not args.no_graph},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": captured_traffic(args.workload),
                         "kernel": "mkv_decode_attention (one fused split-KV decode kernel), one layer",
                         "peak_kind": peak_kind, "frac_of_8000": achieved / 8000.0,
                         "alg_bytes_per_launch": alg_bytes, "overhead_bytes_per_launch": ovh_bytes,
                         "context_at_measure": T_now,
                         "avg_launch_ms": dec_ms},
            "kv_bytes": {"resident": res * w.L, "peak": pk * w.L, "unit": "bytes, all layers"},
            "clocks": clk}
    if step_paths is not None:
        line["step_paths_ms"] = step_paths     # the faster path is the timed one
    del runner
    torch.cuda.empty_cache()
    if world == 1 and args.per_config:
        line["per_config"] = {}
        for name in [n for n in args.per_config.split(",") if n and n != args.workload]:
            wx = WORKLOADS[name]()
            if args.layers is not None:
                import dataclasses
                wx = dataclasses.replace(wx, L=args.layers)
            line["per_config"][wx.name] = measure_config(name, wx, dev, args.seed, METHOD_OF[name], args.steps,
                                                         args.warmup, peak, args.no_graph)
    if world == 1 and args.sweep:
        # the ten configurations at contexts 4K/16K/64K/128K with batch 32/16/4/1
        line["sweep"] = {}
        t_sw = time.perf_counter()
        for (T, B) in synth.SWEEP_POINTS:
            for (meth, level) in synth.SWEEP_CONFIGS:
                wx = synth.sweep(meth, level, T, B)
                if args.layers is not None:
                    import dataclasses
                    wx = dataclasses.replace(wx, L=args.layers)
                line["sweep"][wx.name] = measure_config(wx.name, wx, dev, args.seed, meth, args.sweep_steps, 3,
                                                        peak, args.no_graph, synthetic_h2o_cache=True)
        line["sweep_wall_s"] = time.perf_counter() - t_sw
    if world == 1 and args.setup:
        line["setup"] = measure_setup(dev, args.seed, batch=args.setup_batch)
    if rank == 0:
        if world == 1:
            v, sample = oracle_tokens_per_s(args.workload, w, args.cpu_budget, seed=args.seed)
            line["cpu_baseline"] = {"value": v, "unit": "tokens/s", "cores": 1, "kind": "oracle", "sample": sample,
                                    "extrapolated": True}
            if args.cpu_all_cores:
                va, n = oracle_tokens_per_s_all_cores(args.workload, w, args.cpu_budget, seed=args.seed)
                line["cpu_baseline_all_cores"] = {
                    "value": va, "unit": "tokens/s", "cores": n, "kind": "oracle", "extrapolated": True,
                    "sample": f"{n} single-threaded worker processes (nproc = {n}), each as the one-core sample"}
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
