"""fp64 CPU oracle for compressed-KV decode attention.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports this package:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg (``cpu_baseline`` and ``--impl reference``) may import or run it.

It is a plain, slow, obviously-correct restatement of what each candidate
KV-cache configuration of the paper computes at a decode step (Section 2.1:
the KVQuant, H2O and RocketKV paragraphs; Table 1 lists the configurations),
written with numpy in float64.  Where a decision is defined by an fp32 formula
(quantization codes) it is evaluated with numpy float32 scalars/arrays, which
are IEEE correctly rounded and never contracted into FMAs.

It shares no code with the CUDA path.  Inputs come from ``synth`` (random
numbers only) or from other oracle functions.

Modules
  attention  -- softmax attention over an attended set, GQA decode      (O1)
  rope       -- rotate-half rotary embedding                             (O2)
  kvquant    -- calibration, quantize / dequantize, fused decode         (O3)
  h2o        -- prefill scores, initial keep, decode step with eviction  (O4)
  snapkv     -- observation-window scores, pooling, keep selection       (O5)
  rocket     -- page min/max, dims, page scores, sparse decode           (O6)
  order      -- the total orders used for every ranking decision        (O7)
  selector   -- the configuration choice over predicted costs (Section 2.3) (O8)

Parity status: every function is pinned by tests in ``tests/test_oracle_*``
against closed forms, invariants, brute force or an independent library
routine.  No function is "parity unpinned".
"""
