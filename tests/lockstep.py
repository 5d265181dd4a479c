"""Decision-parity protocol for selections the GPU makes in fp32 and the oracle in fp64.

On the tiny case (inputs drawn with a recorded minimum decision margin) the
GPU's kept sets, evictions and pages must equal the oracle's exactly.  On the
large cases a differing decision is accepted only if every differing item's
oracle score lies within EPS of the boundary score (a near-tie); the oracle
then adopts the GPU's choice so the comparison continues on the same state.
Near-ties are counted and reported.
"""
import json
import os

import numpy as np

from oracle import order

EPS_REL, EPS_ABS = 1e-5, 1e-7
HERE = os.path.dirname(os.path.abspath(__file__))


def record(tag, near, decisions):
    """Report a lockstep run's near-tie count: printed, and appended as a JSON line to the file named
    by MKV_NEAR_TIES_OUT when that is set (the committed summary is made from those lines)."""
    print(f"NEAR-TIES {tag}: {near} of {decisions} decisions")
    path = os.environ.get("MKV_NEAR_TIES_OUT")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps({"run": tag, "near_ties": int(near), "decisions": int(decisions)}) + "\n")


def tiny_seed():
    with open(os.path.join(HERE, "golden", "tiny_seed.json")) as f:
        return json.load(f)["seed"]


def check_topk(values, index, k, got, exact, what=""):
    """Compare a GPU top-k set with the oracle's; returns the number of near-ties (0 or 1).

    values/index: the oracle's candidate scores; got: the GPU's chosen subset."""
    values = np.asarray(values, dtype=np.float64)
    index = np.asarray(index)
    ref = set(order.topk_desc(values, index, k).tolist())
    got = set(np.asarray(got).tolist())
    if ref == got:
        return 0
    assert not exact, f"{what}: selection differs on a margin-seeded case: {sorted(ref ^ got)[:8]}"
    assert len(got) == len(ref), f"{what}: GPU chose {len(got)} items, oracle {len(ref)}"
    perm = order.rank_desc(values, index)
    boundary = values[perm[k - 1]]
    pos_of = {int(i): j for j, i in enumerate(index.tolist())}
    for item in ref ^ got:
        v = values[pos_of[int(item)]]
        assert abs(v - boundary) <= EPS_REL * abs(boundary) + EPS_ABS, \
            f"{what}: item {item} score {v!r} is not a near-tie of the boundary {boundary!r}"
    return 1


def check_evict(cand_pos, cand_acc, got_victim, exact, what=""):
    """Compare the GPU's evicted position with the oracle's (last under acc desc, pos asc)."""
    ref = int(order.last_desc(cand_acc, cand_pos))
    if ref == int(got_victim):
        return 0
    assert not exact, f"{what}: evicted {got_victim}, oracle {ref}"
    acc_of = dict(zip(np.asarray(cand_pos).tolist(), np.asarray(cand_acc, dtype=np.float64).tolist()))
    assert int(got_victim) in acc_of, f"{what}: GPU evicted {got_victim}, not a candidate"
    a, b = acc_of[ref], acc_of[int(got_victim)]
    assert abs(a - b) <= EPS_REL * abs(a) + EPS_ABS, f"{what}: eviction {got_victim} vs {ref} is not a near-tie"
    return 1
