"""Tiny-N CKKS round trip through the oracle (pin P3; test only).

CKKS (Sec. 2.2, "Ciphertexts and Slots") packs a vector of real numbers into
the slots of one ciphertext; a PMult multiplies slot by slot and Add/Sub add
slot by slot.  This module builds a textbook CKKS instance with exact Python
integers, small enough to run in seconds:

  * encoding: the canonical embedding, evaluated directly (O(N^2)) at the
    primitive 2N-th roots of unity zeta^(5^j) (slot j) and their conjugates,
    coefficients rounded after scaling by Delta;
  * RNS/NTT form: each coefficient vector reduced mod q_l and evaluated at the
    odd powers psi^(2t+1) of a primitive 2N-th root psi mod q_l (direct O(N^2)
    evaluation; slot order t is the natural one);
  * secret-key encryption: s uniform ternary, a uniform, e rounded Gaussian
    with sigma 3.2; ct = (-a*s + m + e, a);
  * decryption c0 + c1*s, inverse NTT, CRT lift, centring, decoding with
    1/(Delta^2) after the plaintext products.

A linear layer evaluated by the oracle on such ciphertexts must decrypt to
the float64 slot-wise mat-vec  y_j = sum_g gamma_g * sum_i t_i x_i +
sum_raw w_e * x_i  within the CKKS error (the paper compares its compiled
layers with an FP64 computation the same way, Sec. 6 RQ1 "Exact
Compilation").  The check is independent of the oracle's formula: a wrong
sign, operand or dropped term changes the decrypted real numbers.
"""
from __future__ import annotations

import cmath
import math
from typing import List, Sequence

import numpy as np


def _primitive_2n_root(q: int, N: int) -> int:
    for g in range(2, 10000):
        psi = pow(g, (q - 1) // (2 * N), q)
        if pow(psi, N, q) == q - 1:
            return psi
    raise ValueError("no primitive 2N-th root found")


class TinyCKKS:
    def __init__(self, N: int, moduli: Sequence[int], delta_bits: int, seed: int = 1):
        assert N & (N - 1) == 0 and N >= 8
        self.N = N
        self.moduli = [int(q) for q in moduli]
        for q in self.moduli:
            assert (q - 1) % (2 * N) == 0
        self.Q = 1
        for q in self.moduli:
            self.Q *= q
        self.delta = 1 << delta_bits
        self.rng = np.random.default_rng(seed)
        M = 2 * N
        # slot j sits at zeta^(5^j); its conjugate at zeta^(-5^j)
        self.rot = [pow(5, j, M) for j in range(N // 2)]
        self.zeta = [cmath.exp(1j * math.pi * r / N) for r in range(M)]
        # per-limb evaluation matrices  W[t][k] = psi^((2t+1) k)
        self.fwd = []
        self.inv = []
        for q in self.moduli:
            psi = _primitive_2n_root(q, N)
            W = [[pow(psi, (2 * t + 1) * k % M, q) for k in range(N)] for t in range(N)]
            psi_inv = pow(psi, -1, q)
            n_inv = pow(N, -1, q)
            Wi = [[pow(psi_inv, (2 * t + 1) * k % M, q) * n_inv % q for t in range(N)]
                  for k in range(N)]
            self.fwd.append(W)
            self.inv.append(Wi)

    # -- encoding ------------------------------------------------------------
    def encode(self, z: Sequence[float], scale: int) -> List[int]:
        """Integer coefficients m with m(zeta^(5^j)) ~= scale * z_j."""
        N, M = self.N, 2 * self.N
        out = []
        for k in range(N):
            acc = 0j
            for j, zj in enumerate(z):
                acc += zj * self.zeta[(-self.rot[j] * k) % M]
            out.append(int(round(2.0 * scale * acc.real / N)))
        return out

    def decode(self, m: Sequence[int], scale: float) -> np.ndarray:
        N, M = self.N, 2 * self.N
        z = []
        for j in range(N // 2):
            acc = 0j
            for k, mk in enumerate(m):
                acc += mk * self.zeta[(self.rot[j] * k) % M]
            z.append(acc.real / scale)
        return np.array(z)

    # -- RNS / NTT ----------------------------------------------------------
    def to_ntt(self, coeffs: Sequence[int]) -> np.ndarray:
        """[L][N] residues of the evaluation form of an integer polynomial."""
        out = np.zeros((len(self.moduli), self.N), dtype=np.uint64)
        for l, q in enumerate(self.moduli):
            c = [int(x) % q for x in coeffs]
            W = self.fwd[l]
            for t in range(self.N):
                out[l, t] = sum(W[t][k] * c[k] for k in range(self.N)) % q
        return out

    def from_ntt(self, ev: np.ndarray) -> List[int]:
        """Centred integer coefficients from [L][N] evaluation-form residues."""
        per_limb = []
        for l, q in enumerate(self.moduli):
            Wi = self.inv[l]
            v = [int(x) for x in ev[l]]
            per_limb.append([sum(Wi[k][t] * v[t] for t in range(self.N)) % q
                             for k in range(self.N)])
        out = []
        for k in range(self.N):
            x = 0
            for l, q in enumerate(self.moduli):
                Mi = self.Q // q
                x += per_limb[l][k] * Mi * pow(Mi, -1, q)
            x %= self.Q
            if x > self.Q // 2:
                x -= self.Q
            out.append(x)
        return out

    # -- keys and encryption ---------------------------------------------
    def keygen(self) -> List[int]:
        self.s = [int(v) for v in self.rng.integers(-1, 2, self.N)]
        self.s_ntt = self.to_ntt(self.s)
        return self.s

    def encrypt(self, z: Sequence[float]) -> np.ndarray:
        """[2][L][N] evaluation-form ciphertext of slot vector z at scale Delta."""
        m = self.encode(z, self.delta)
        e = [int(round(v)) for v in self.rng.normal(0.0, 3.2, self.N)]
        me = self.to_ntt([a + b for a, b in zip(m, e)])
        ct = np.zeros((2, len(self.moduli), self.N), dtype=np.uint64)
        for l, q in enumerate(self.moduli):
            a = [int(v) for v in self.rng.integers(0, q, self.N, dtype=np.uint64)]
            for t in range(self.N):
                ct[1, l, t] = a[t]
                ct[0, l, t] = (int(me[l, t]) - a[t] * int(self.s_ntt[l, t])) % q
        return ct

    def decrypt_decode(self, ct: np.ndarray, scale: float) -> np.ndarray:
        ev = np.zeros((len(self.moduli), self.N), dtype=np.uint64)
        for l, q in enumerate(self.moduli):
            for t in range(self.N):
                ev[l, t] = (int(ct[0, l, t]) + int(ct[1, l, t]) * int(self.s_ntt[l, t])) % q
        return self.decode(self.from_ntt(ev), scale)

    def encode_plaintext(self, w: Sequence[float]) -> np.ndarray:
        """[L][N] evaluation-form plaintext of slot vector w at scale Delta."""
        return self.to_ntt(self.encode(w, self.delta))


def float_layer(plan, x: np.ndarray, pt_slots: np.ndarray) -> np.ndarray:
    """Slot-wise float64 reference of the layer: x [n_in][slots], pt_slots
    [n_pt][slots] (real weights / reconstruction factors)."""
    t = plan.terms
    y = np.zeros((plan.n_out, x.shape[1]))
    for j in range(plan.n_out):
        for e in range(int(plan.term_offsets[j]), int(plan.term_offsets[j + 1])):
            i = int(t["input"][e])
            if t["kind"][e] == 1:
                gamma = pt_slots[int(plan.group_scale_pt[int(t["group"][e])])]
                y[j] += int(t["sign"][e]) * gamma * x[i]
            else:
                y[j] += pt_slots[int(t["pt"][e])] * x[i]
    return y
