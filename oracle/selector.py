"""MetaKV's configuration choice (Section 2.3), restated step by step.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Given each candidate configuration's predicted end-to-end latency, peak
memory and probability of a correct answer, and the user's budgets L_max and
M_max (Section 2.3, the selection pipeline):
  step 3  budget filter: keep the candidates within both budgets;
  step 4  if the uncompressed FP16 configuration survives, choose it;
  step 5  otherwise keep, per method, only its least compressed survivor;
  step 6  a single remaining candidate is chosen;
  step 7  otherwise the highest predicted accuracy wins.
If nothing survives the filter, the candidate with the smallest relative
violation v_c = L_c / L_max + M_c / M_max is chosen, the accuracy breaking
ties.  Remaining ties (the paper does not order them) go to the lower index.

A candidate is a tuple (method, level, latency, memory, accuracy); method
0 = FP16, 1 = KVQuant, 2 = H2O, 3 = RocketKV, and a larger level means less
compression within the method (KVQuant bits, H2O budget percent, RocketKV
minus its compression ratio).
"""
from __future__ import annotations

FP16 = 0


def select(cands, L_max: float, M_max: float):
    """(index of the chosen candidate, whether it is within both budgets)."""
    ok = [i for i, c in enumerate(cands) if c[2] <= L_max and c[3] <= M_max]            # step 3
    if not ok:
        v = [c[2] / L_max + c[3] / M_max for c in cands]
        return min(range(len(cands)), key=lambda i: (v[i], -cands[i][4], i)), False
    for i in ok:                                                                        # step 4
        if cands[i][0] == FP16:
            return i, True
    least = {}                                                                          # step 5
    for i in ok:
        m = cands[i][0]
        if m not in least or cands[i][1] > cands[least[m]][1]:
            least[m] = i
    rest = sorted(least.values())
    if len(rest) == 1:                                                                  # step 6
        return rest[0], True
    return min(rest, key=lambda i: (-cands[i][4], i)), True                             # step 7
