"""The host selector (Section 2.3): the oracle's restatement pinned by hand-worked choices over
Table 1's costs, and the C ABI's mkv_select_config identical to the oracle on random candidate
sets.  CPU only."""
import json
import os

import numpy as np
import pytest

import paper_2609_07966_gb300 as mkv
from oracle import selector

HERE = os.path.dirname(os.path.abspath(__file__))


def _table1():
    t = json.load(open(os.path.join(HERE, "golden", "table1_costs.json")))
    names = [r[0] for r in t["rows"]]
    cands = [(r[1], r[2], r[4], r[5], r[3]) for r in t["rows"]]   # (method, level, latency, memory, accuracy)
    return names, cands


# (L_max s, M_max MB) -> expected configuration, each worked by hand from the rule and Table 1
HAND = [
    (5, 50, "FP16", True),            # FP16 fits (2.01 s, 34.47 MB): chosen at once
    (4, 40, "FP16", True),
    (3, 10, "H2O 20%", True),         # only H2O 20% fits (2.70 s, 6.29 MB)
    (25, 10, "KVQuant 3-bit", True),  # fit: KVQuant 3/2-bit, H2O 20%; least compressed: KVQuant 3 (0.609)
                                      # vs H2O 20% (0.507)
    (25, 20, "KVQuant 4-bit", True),  # FP16 over memory; least compressed KVQuant 4 (0.630) vs H2O 60% (0.627)
    (3, 20, "H2O 60%", True),         # only H2O fits: its least compressed setting
    (4, 31, "H2O 60%", True),         # H2O 60% (0.627) vs RocketKV 8x (0.464); KVQuant over latency
    (1, 5, "H2O 20%", False),         # nothing fits: v = L/1 + M/5 is smallest for H2O 20% (3.958)
]


@pytest.mark.parametrize("L,M,want,within", HAND)
def test_oracle_hand_worked(L, M, want, within):
    names, cands = _table1()
    i, ok = selector.select(cands, L, M)
    assert (names[i], ok) == (want, within)


@pytest.mark.parametrize("L,M,want,within", HAND)
def test_library_hand_worked(L, M, want, within):
    names, cands = _table1()
    i, ok = mkv.mkv_select_config(cands, L, M)
    assert (names[i], ok) == (want, within)


def test_violation_tie_goes_to_accuracy_then_index():
    # both over budget with the same violation 2 + 1 = 1 + 2; the more accurate wins, then the first
    c = [(1, 4, 2.0, 1.0, 0.5), (2, 60, 1.0, 2.0, 0.7), (3, -8, 1.0, 2.0, 0.7)]
    assert selector.select(c, 1.0, 1.0) == (1, False)
    assert mkv.mkv_select_config(c, 1.0, 1.0) == (1, False)


def test_level_and_accuracy_ties_go_to_the_lower_index():
    c = [(2, 40, 1, 1, 0.5), (2, 40, 1, 1, 0.9), (1, 4, 1, 1, 0.5)]
    # H2O's least compressed survivor is index 0 (tie on level), then 0.5 vs KVQuant's 0.5: index 0
    assert selector.select(c, 2, 2) == (0, True)
    assert mkv.mkv_select_config(c, 2, 2) == (0, True)


def test_library_matches_oracle_on_random_sets():
    rng = np.random.default_rng(77)
    for trial in range(3000):
        n = int(rng.integers(1, 12))
        cands = []
        for _ in range(n):
            m = int(rng.integers(0, 4))
            lv = int(rng.integers(-3, 4))
            # coarse values so that ties in cost, violation and accuracy occur
            cands.append((m, lv, float(rng.integers(0, 8)) / 2, float(rng.integers(0, 8)) / 2,
                          float(rng.integers(0, 4)) / 4))
        L, M = float(rng.integers(1, 8)) / 2, float(rng.integers(1, 8)) / 2
        assert mkv.mkv_select_config(cands, L, M) == selector.select(cands, L, M), (trial, cands, L, M)


def test_rejects_bad_arguments():
    ok = [(0, 0, 1.0, 1.0, 0.5)]
    for bad in ([(4, 0, 1.0, 1.0, 0.5)], [(1, 0, -1.0, 1.0, 0.5)], [(1, 0, float("nan"), 1.0, 0.5)]):
        with pytest.raises(mkv.MkvError):
            mkv.mkv_select_config(bad, 1.0, 1.0)
    with pytest.raises(mkv.MkvError):
        mkv.mkv_select_config(ok, 0.0, 1.0)
    with pytest.raises(mkv.MkvError):
        mkv.mkv_select_config([], 1.0, 1.0)
