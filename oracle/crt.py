"""Brute-force evaluation of the linear layer over Z_Q (pin P2; test only).

Every residue vector (one value per RNS limb) is lifted to its unique
representative in Z_Q, Q = prod q_l, with the Chinese remainder theorem.  The
layer of Sec. 4.2 (signed sums scaled by gamma, plus raw PMults; Eq.
"routed-example") is then evaluated with exact Python integers, with no
modular reduction until the very end, and the result is reduced modulo each
q_l.  Because Z_Q is isomorphic to the product of the Z_{q_l} (CRT), the
per-limb oracle must reproduce these residues exactly.  This pins the oracle's
modular reduction and its limb indexing with arithmetic that shares nothing
with it.  Intended for tiny inputs (a few dozen coefficients).
"""
from __future__ import annotations

from typing import List, Sequence

import numpy as np


def crt_lift(residues: Sequence[int], moduli: Sequence[int]) -> int:
    Q = 1
    for q in moduli:
        Q *= q
    x = 0
    for r, q in zip(residues, moduli):
        Mi = Q // q
        x += int(r) * Mi * pow(Mi, -1, q)
    return x % Q


def eval_over_ZQ(plan, moduli: Sequence[int], inputs: np.ndarray,
                 plaintexts: np.ndarray) -> np.ndarray:
    moduli = [int(q) for q in moduli]
    L = len(moduli)
    n_in, _, _, n = inputs.shape
    Q = 1
    for q in moduli:
        Q *= q
    X = [[[crt_lift([inputs[i, c, l, k] for l in range(L)], moduli) for k in range(n)]
          for c in range(2)] for i in range(n_in)]
    P = [[crt_lift([plaintexts[p, l, k] for l in range(L)], moduli) for k in range(n)]
         for p in range(plaintexts.shape[0])]
    out = np.zeros((plan.n_out, 2, L, n), dtype=np.uint64)
    t = plan.terms
    for j in range(plan.n_out):
        lo, hi = int(plan.term_offsets[j]), int(plan.term_offsets[j + 1])
        for c in range(2):
            for k in range(n):
                signed = {}
                total = 0
                for e in range(lo, hi):
                    i = int(t["input"][e])
                    if t["kind"][e] == 1:
                        g = int(t["group"][e])
                        signed[g] = signed.get(g, 0) + int(t["sign"][e]) * X[i][c][k]
                    else:
                        total += P[int(t["pt"][e])][k] * X[i][c][k]
                for g, s in signed.items():
                    total += P[int(plan.group_scale_pt[g])][k] * s
                total %= Q
                for l in range(L):
                    out[j, c, l, k] = total % moduli[l]
    return out
