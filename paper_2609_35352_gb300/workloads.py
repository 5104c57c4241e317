"""Seeded synthetic workloads for the hybrid packed-CKKS linear layer.

This module is the single source of inputs for both the CUDA path and the
CPU oracle.  It holds no arithmetic of the method itself (no modular
accumulation, no products): it only chooses parameters (RNS moduli), plan
structure (which (output, input) pair takes the raw or the signed route, the
scale groups, the DAG of shared signed sums) and residues.

Randomness
----------
Every random number comes from one counter-based generator, SplitMix64
(Steele, Lea, Flood, "Fast splittable pseudorandom number generators",
OOPSLA 2014; the constants are the published ones).  Value number ``n`` of a
stream with key ``K`` is ``mix64(K + (n + 1) * GOLDEN)``.  A residue modulo
``q`` is the high word of the 128-bit product ``x * q`` (Lemire's
multiply-shift map without the rejection step; its bias is below q / 2^64,
about 6e-5 for the 50-bit primes used here), so each residue is a pure
function of (seed, stream, flat index) and can be regenerated one by one on
the host for any sampled coordinate.  The CUDA fill kernel in
``csrc/workload_fill.cu`` implements the same definition on the device; a GPU
test checks the two agree.

Layouts (all little-endian uint64 residues, row-major):
  inputs      [n_in ][2][L][N]   (c0, c1 of each ciphertext, NTT form)
  plaintexts  [n_pt ][L][N]
  outputs     [n_out][2][L][N]

The layer shapes follow the paper's evaluated layers (Sec. 6, Table
"eval-linear-compilation" and Table "implementation-layouts"): a VGG11-style
convolution (144 rotated inputs -> 16 outputs), a ViT-B-style BSGS projection
(32 -> 24), a BERT-base-style FFN under column packing (96 -> 96), and the
64-ciphertext weighted sum of the motivation table (Sec. 3.1).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15
MIX1 = 0xBF58476D1CE4E5B9
MIX2 = 0x94D049BB133111EB

# stream ids inside one workload seed
STREAM_INPUTS = 1
STREAM_PLAINTEXTS = 2
STREAM_PLAN = 3

TERM_RAW = 0
TERM_TERNARY = 1
TERM_RAW_CONST = 2   # raw term whose plaintext is one value in every slot

# numpy mirrors of the C structs declared in include/fiona.h
TERM_DTYPE = np.dtype([("input", "<u4"), ("pt", "<u4"), ("group", "<u4"),
                       ("kind", "i1"), ("sign", "i1"), ("reserved", "<u2")])
CHILD_DTYPE = np.dtype([("ref", "<u4"), ("is_node", "i1"), ("sign", "i1"),
                        ("reserved", "<u2")])
USE_DTYPE = np.dtype([("output", "<u4"), ("group", "<u4"), ("node", "<u4"),
                      ("sign", "i1"), ("reserved", "u1", (3,))])
assert TERM_DTYPE.itemsize == 16 and CHILD_DTYPE.itemsize == 8 and USE_DTYPE.itemsize == 16


# ----------------------------------------------------------------------------
# SplitMix64, scalar (python int) and vectorised (numpy uint64) forms
# ----------------------------------------------------------------------------
def mix64(z: int) -> int:
    z &= MASK64
    z = ((z ^ (z >> 30)) * MIX1) & MASK64
    z = ((z ^ (z >> 27)) * MIX2) & MASK64
    return z ^ (z >> 31)


def stream_key(seed: int, stream: int) -> int:
    """Key of stream ``stream`` under ``seed``: one SplitMix64 output."""
    return mix64((seed + (stream + 1) * GOLDEN) & MASK64)


def raw64(key: int, index: int) -> int:
    return mix64((key + (index + 1) * GOLDEN) & MASK64)


def _mix64_np(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * np.uint64(MIX1)
    z = z ^ (z >> np.uint64(27))
    z = z * np.uint64(MIX2)
    return z ^ (z >> np.uint64(31))


def raw64_np(key: int, index: np.ndarray) -> np.ndarray:
    idx = np.asarray(index, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + (idx + np.uint64(1)) * np.uint64(GOLDEN)
        return _mix64_np(z)


def mulhi64_np(x: np.ndarray, q: np.ndarray) -> np.ndarray:
    """High 64 bits of the 128-bit product x*q for uint64 arrays (32-bit split)."""
    x = np.asarray(x, dtype=np.uint64)
    q = np.asarray(q, dtype=np.uint64)
    m32 = np.uint64(0xFFFFFFFF)
    s32 = np.uint64(32)
    xl, xh = x & m32, x >> s32
    ql, qh = q & m32, q >> s32
    ll = xl * ql
    lh = xl * qh
    hl = xh * ql
    hh = xh * qh
    mid = (ll >> s32) + (lh & m32) + (hl & m32)
    return hh + (lh >> s32) + (hl >> s32) + (mid >> s32)


def residues_np(key: int, flat_index: np.ndarray, q: np.ndarray) -> np.ndarray:
    """Uniform residues in [0, q): high word of raw64 * q."""
    return mulhi64_np(raw64_np(key, flat_index), q)


class PlanRng:
    """Sequential SplitMix64 stream for plan structure (route choice, DAG)."""

    def __init__(self, seed: int, stream: int = STREAM_PLAN):
        self.key = stream_key(seed, stream)
        self.ctr = 0

    def next64(self) -> int:
        v = raw64(self.key, self.ctr)
        self.ctr += 1
        return v

    def below(self, n: int) -> int:
        return (self.next64() * n) >> 64

    def shuffle(self, items: list) -> None:
        for i in range(len(items) - 1, 0, -1):
            j = self.below(i + 1)
            items[i], items[j] = items[j], items[i]

    def sample(self, population: Sequence, k: int) -> list:
        pool = list(population)
        out = []
        for _ in range(k):
            j = self.below(len(pool))
            out.append(pool[j])
            pool[j] = pool[-1]
            pool.pop()
        return out


# ----------------------------------------------------------------------------
# RNS moduli: the L largest primes below 2^bits with q = 1 (mod 2N)
# ----------------------------------------------------------------------------
_MR_BASES = (2, 3, 5, 7, 11, 13, 17, 19, 23, 29, 31, 37)


def is_prime(n: int) -> bool:
    """Deterministic Miller-Rabin for n < 3.3e24 (bases 2..37)."""
    if n < 2:
        return False
    for p in _MR_BASES:
        if n % p == 0:
            return n == p
    d, s = n - 1, 0
    while d % 2 == 0:
        d //= 2
        s += 1
    for a in _MR_BASES:
        x = pow(a, d, n)
        if x in (1, n - 1):
            continue
        for _ in range(s - 1):
            x = x * x % n
            if x == n - 1:
                break
        else:
            return False
    return True


def ntt_primes(N: int, bits: int, L: int) -> List[int]:
    """The L largest primes q < 2^bits with q = 1 (mod 2N), descending."""
    step = 2 * N
    q = ((1 << bits) - 1) // step * step + 1
    if q >= (1 << bits):
        q -= step
    out = []
    while len(out) < L:
        if q <= step:
            raise ValueError("ran out of NTT-friendly primes")
        if is_prime(q):
            out.append(q)
        q -= step
    return out


# ----------------------------------------------------------------------------
# Plan description (mirrors the arguments of fiona_plan_create)
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class Plan:
    n_in: int
    n_out: int
    n_pt: int
    term_offsets: np.ndarray          # uint32 [n_out + 1]
    terms: np.ndarray                 # TERM_DTYPE [n_terms]
    group_scale_pt: np.ndarray        # uint32 [n_groups]
    group_output: np.ndarray          # uint32 [n_groups]
    node_offsets: np.ndarray          # uint32 [n_nodes + 1]
    children: np.ndarray              # CHILD_DTYPE
    uses: np.ndarray                  # USE_DTYPE

    @property
    def n_groups(self) -> int:
        return int(self.group_scale_pt.shape[0])

    @property
    def n_nodes(self) -> int:
        return int(self.node_offsets.shape[0]) - 1

    @property
    def n_uses(self) -> int:
        return int(self.uses.shape[0])

    def output_terms(self, j: int) -> np.ndarray:
        return self.terms[self.term_offsets[j]:self.term_offsets[j + 1]]

    def counts(self) -> Dict[str, int]:
        t = self.terms
        raw = int(np.sum((t["kind"] == TERM_RAW) | (t["kind"] == TERM_RAW_CONST)))
        tern = t["kind"] == TERM_TERNARY
        return {
            "raw": raw,
            "plus": int(np.sum(tern & (t["sign"] == 1))),
            "minus": int(np.sum(tern & (t["sign"] == -1))),
            "zero": int(np.sum(tern & (t["sign"] == 0))),
            "nonzero": raw + int(np.sum(tern & (t["sign"] != 0))),
        }


def scale_classes(plan: Plan, n_class: int = 2, kind: str = "routes", seed: int = 0) -> np.ndarray:
    """A scale class per plaintext (uint8, < n_class), for a layer whose
    plaintexts are encoded at several scales.  "routes": the scale groups'
    gamma plaintexts in class 0, the raw weights in class 1 (the two routes
    at different scales); "random": seeded uniform classes."""
    cls = np.zeros(plan.n_pt, dtype=np.uint8)
    if n_class < 2:
        return cls
    if kind == "routes":
        t = plan.terms
        raw = t["pt"][(t["kind"] == TERM_RAW) | (t["kind"] == TERM_RAW_CONST)]
        cls[np.unique(raw).astype(np.int64)] = 1
        cls[np.unique(plan.group_scale_pt).astype(np.int64)] = 0
    else:
        rng = PlanRng(seed ^ 0x5CA1E, STREAM_PLAN)
        for p in range(plan.n_pt):
            cls[p] = rng.below(n_class)
    return cls


def class_subplan(plan: Plan, pt_class: np.ndarray, s: int) -> Plan:
    """The layer restricted to the terms whose plaintext (a scale group's
    gamma for signed terms) has class s; every output kept, the DAG dropped."""
    t = plan.terms
    per_output = []
    for j in range(plan.n_out):
        rows = []
        for e in range(int(plan.term_offsets[j]), int(plan.term_offsets[j + 1])):
            pt = int(plan.group_scale_pt[t["group"][e]]) if t["kind"][e] == TERM_TERNARY else int(t["pt"][e])
            if int(pt_class[pt]) == s:
                rows.append((int(t["input"][e]), int(t["kind"][e]), int(t["sign"][e]), int(t["pt"][e]),
                             int(t["group"][e])))
        per_output.append(rows)
    return build_plan(plan.n_in, plan.n_out, per_output, plan.n_pt, list(plan.group_scale_pt),
                      list(plan.group_output), [], [])


def min_bytes(plan: Plan, L: int, N: int) -> int:
    """Minimal HBM bytes of one evaluation: each input read by a nonzero term
    (both polys), each plaintext a raw term or a used scale group reads, and
    each output, one limb-poly of N * 8 bytes per limb, moved once; a
    plaintext read only as a constant (TERM_RAW_CONST) counts one residue per
    limb.  A count, the same as fiona_plan_stats.bytes_min."""
    t = plan.terms
    raw = (t["kind"] == TERM_RAW) | (t["kind"] == TERM_RAW_CONST)
    signed = (t["kind"] == TERM_TERNARY) & (t["sign"] != 0)
    inputs = set(int(i) for i in t["input"][raw | signed])
    whole = set(int(p) for p in t["pt"][t["kind"] == TERM_RAW])
    whole |= set(int(plan.group_scale_pt[g]) for g in set(int(g) for g in t["group"][signed]))
    const = set(int(p) for p in t["pt"][t["kind"] == TERM_RAW_CONST]) - whole
    return L * N * 8 * (2 * len(inputs) + len(whole) + 2 * plan.n_out) + len(const) * L * 8


def build_plan(n_in: int, n_out: int, per_output: List[List[Tuple[int, int, int, int, int]]],
                n_pt: int, group_scale_pt: List[int], group_output: List[int],
                nodes: List[List[Tuple[int, int, int]]],
                uses: List[Tuple[int, int, int, int]]) -> Plan:
    """per_output[j] = [(input, kind, sign, pt, group), ...]; nodes[k] = [(ref, is_node, sign)]."""
    offs = [0]
    rows = []
    for j in range(n_out):
        for (i, kind, sign, pt, grp) in per_output[j]:
            rows.append((i, pt, grp, kind, sign, 0))
        offs.append(len(rows))
    terms = np.array(rows, dtype=TERM_DTYPE) if rows else np.zeros(0, TERM_DTYPE)
    noffs = [0]
    crows = []
    for ch in nodes:
        for (ref, is_node, sign) in ch:
            crows.append((ref, is_node, sign, 0))
        noffs.append(len(crows))
    children = np.array(crows, dtype=CHILD_DTYPE) if crows else np.zeros(0, CHILD_DTYPE)
    urows = [(o, g, k, s, (0, 0, 0)) for (o, g, k, s) in uses]
    uses_arr = np.array(urows, dtype=USE_DTYPE) if urows else np.zeros(0, USE_DTYPE)
    return Plan(n_in=n_in, n_out=n_out, n_pt=n_pt,
                term_offsets=np.array(offs, dtype=np.uint32), terms=terms,
                group_scale_pt=np.array(group_scale_pt, dtype=np.uint32),
                group_output=np.array(group_output, dtype=np.uint32),
                node_offsets=np.array(noffs, dtype=np.uint32), children=children,
                uses=uses_arr)


def dense_hybrid_plan(rng: PlanRng, n_in: int, n_out: int, n_plus: int, n_minus: int,
                      n_zero: int, group_per_term: bool = False,
                      dag_share: float = 0.0, dag_m: int = 4) -> Plan:
    """Dense bipartite layer: every (output, input) pair is one execution group.

    Exact route counts: the pairs are shuffled (Fisher-Yates) and the first
    n_plus take t=+1, the next n_minus t=-1, the next n_zero t=0, the rest the
    raw route.  With ``dag_share`` > 0, shared signed sums are generated first
    (m inputs, k in {2,3} outputs, so the paper's saving estimate km-m-k is
    positive) until the covered nonzero ternary terms reach that share.
    Scale groups: one per output (the output's packed reconstruction factors),
    or one per ternary term when ``group_per_term``.
    """
    assigned: Dict[Tuple[int, int], int] = {}
    nodes: List[List[Tuple[int, int, int]]] = []
    dag_uses: List[Tuple[int, int, int]] = []     # (output, node, sigma)
    target = dag_share * (n_plus + n_minus)
    covered = 0
    attempts = 0
    while covered < target:
        attempts += 1
        if attempts > 100000:
            raise RuntimeError("DAG generation did not converge")
        ins = sorted(rng.sample(range(n_in), dag_m))
        signs = [1 if rng.below(2) else -1 for _ in ins]
        k = 2 + rng.below(2)
        cands = [j for j in range(n_out) if all((j, i) not in assigned for i in ins)]
        if len(cands) < k:
            continue
        outs = sorted(rng.sample(cands, k))
        node_id = len(nodes)
        nodes.append([(i, 0, s) for i, s in zip(ins, signs)])
        for o in outs:
            sigma = 1 if rng.below(2) else -1
            for i, s in zip(ins, signs):
                assigned[(o, i)] = sigma * s
            dag_uses.append((o, node_id, sigma))
        covered += len(outs) * len(ins)
    pre_plus = sum(1 for v in assigned.values() if v == 1)
    pre_minus = sum(1 for v in assigned.values() if v == -1)
    if pre_plus > n_plus or pre_minus > n_minus:
        raise RuntimeError("DAG covers more signed terms than the route counts allow")
    free = [(j, i) for j in range(n_out) for i in range(n_in) if (j, i) not in assigned]
    rng.shuffle(free)
    rp, rm, rz = n_plus - pre_plus, n_minus - pre_minus, n_zero
    route: Dict[Tuple[int, int], Tuple[int, int]] = {}
    for idx, pair in enumerate(free):
        if idx < rp:
            route[pair] = (TERM_TERNARY, 1)
        elif idx < rp + rm:
            route[pair] = (TERM_TERNARY, -1)
        elif idx < rp + rm + rz:
            route[pair] = (TERM_TERNARY, 0)
        else:
            route[pair] = (TERM_RAW, 0)
    for pair, v in assigned.items():
        route[pair] = (TERM_TERNARY, v)

    # plaintext ids: raw plaintexts first (term order), then scale plaintexts
    per_output: List[List[Tuple[int, int, int, int, int]]] = []
    n_raw = sum(1 for v in route.values() if v[0] == TERM_RAW)
    next_raw = 0
    group_scale_pt: List[int] = []
    group_output: List[int] = []
    out_group: Dict[int, int] = {}
    for j in range(n_out):
        row = []
        for i in range(n_in):
            kind, sign = route[(j, i)]
            if kind == TERM_RAW:
                row.append((i, TERM_RAW, 0, next_raw, 0))
                next_raw += 1
            else:
                if group_per_term:
                    g = len(group_output)
                    group_output.append(j)
                    group_scale_pt.append(n_raw + g)
                else:
                    if j not in out_group:
                        out_group[j] = len(group_output)
                        group_output.append(j)
                        group_scale_pt.append(n_raw + out_group[j])
                    g = out_group[j]
                row.append((i, TERM_TERNARY, sign, 0, g))
        per_output.append(row)
    n_pt = n_raw + len(group_output)
    uses = [(o, out_group[o], k, s) for (o, k, s) in dag_uses]
    return build_plan(n_in, n_out, per_output, n_pt, group_scale_pt, group_output,
                       nodes, uses)


# ----------------------------------------------------------------------------
# Workloads
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class Workload:
    name: str
    N: int
    moduli: List[int]
    plan: Plan
    seed: int
    fill: str = "uniform"        # "uniform" residues, or "max" (every residue q-1)
    const_pts: int = 0           # plaintexts [0, const_pts) are constant per limb

    @property
    def L(self) -> int:
        return len(self.moduli)

    @property
    def moduli_np(self) -> np.ndarray:
        return np.array(self.moduli, dtype=np.uint64)

    def key(self, stream: int) -> int:
        return stream_key(self.seed, stream)

    # -- residues on the host ------------------------------------------------
    def _fill(self, stream: int, outer: int) -> np.ndarray:
        L, N = self.L, self.N
        shape = (outer, L, N)
        q = self.moduli_np.reshape(1, L, 1)
        if self.fill == "max":
            return np.broadcast_to(q - np.uint64(1), shape).copy()
        flat = np.arange(outer * L * N, dtype=np.uint64).reshape(shape)
        if stream == STREAM_PLAINTEXTS and self.const_pts:
            # a constant plaintext repeats its limb's first residue
            flat[: self.const_pts] = flat[: self.const_pts, :, :1]
        return residues_np(self.key(stream), flat, q)

    def host_inputs(self) -> np.ndarray:
        n = self.plan.n_in
        return self._fill(STREAM_INPUTS, 2 * n).reshape(n, 2, self.L, self.N)

    def host_plaintexts(self) -> np.ndarray:
        return self._fill(STREAM_PLAINTEXTS, self.plan.n_pt)

    def input_values(self, i, c, l, k) -> np.ndarray:
        """Residues of input i, poly c, limb l, coefficient k (broadcasting)."""
        i, c, l, k = np.broadcast_arrays(*(np.asarray(v, dtype=np.uint64) for v in (i, c, l, k)))
        q = self.moduli_np[l.astype(np.int64)]
        if self.fill == "max":
            return q - np.uint64(1)
        flat = ((i * np.uint64(2) + c) * np.uint64(self.L) + l) * np.uint64(self.N) + k
        return residues_np(self.key(STREAM_INPUTS), flat, q)

    def plaintext_values(self, p, l, k) -> np.ndarray:
        p, l, k = np.broadcast_arrays(*(np.asarray(v, dtype=np.uint64) for v in (p, l, k)))
        q = self.moduli_np[l.astype(np.int64)]
        if self.fill == "max":
            return q - np.uint64(1)
        k = np.where(p < np.uint64(self.const_pts), np.uint64(0), k)
        flat = (p * np.uint64(self.L) + l) * np.uint64(self.N) + k
        return residues_np(self.key(STREAM_PLAINTEXTS), flat, q)

    # -- sizes ------------------------------------------------------------------
    def input_bytes(self) -> int:
        return self.plan.n_in * 2 * self.L * self.N * 8

    def plaintext_bytes(self) -> int:
        return self.plan.n_pt * self.L * self.N * 8

    def output_bytes(self) -> int:
        return self.plan.n_out * 2 * self.L * self.N * 8


SEED_BASE = 0xF10A0000

# Shapes of the configurations (Sec. 6 layers; Sec. 3.1 weighted sum)
WORKLOADS = ("tiny", "tiny-dag", "worked-example", "wsum-pmult", "wsum-ternary",
             "wsum-hybrid", "vgg", "vit", "bert", "bert-const", "overflow60", "overflow50")


def make_workload(name: str, N: Optional[int] = None, L: Optional[int] = None,
                  bits: Optional[int] = None) -> Workload:
    """Build a named workload; N, L and bits override the defaults (for
    reduced-size parity cases with the same plan structure)."""
    def primes(n_default, L_default, b_default):
        n_ = N or n_default
        return n_, ntt_primes(n_, bits or b_default, L or L_default)

    if name == "tiny":
        seed = SEED_BASE + 0
        n, qs = primes(1 << 12, 3, 40)
        # 8 x 4 = 32 pairs, 60% ternary (19): +1 40%, -1 40%, 0 20%; 40% raw
        plan = dense_hybrid_plan(PlanRng(seed), 8, 4, n_plus=8, n_minus=8, n_zero=3,
                                 group_per_term=True)
        return Workload(name, n, qs, plan, seed)
    if name == "tiny-dag":
        seed = SEED_BASE + 0 + 256
        n, qs = primes(1 << 12, 3, 40)
        return Workload(name, n, qs, _tiny_dag_plan(PlanRng(seed)), seed)
    if name == "worked-example":
        seed = SEED_BASE + 0 + 512
        n, qs = primes(1 << 10, 3, 40)
        return Workload(name, n, qs, worked_example_plan(), seed)
    if name.startswith("wsum-"):
        v = {"wsum-pmult": 0, "wsum-ternary": 1, "wsum-hybrid": 2}[name]
        seed = SEED_BASE + 1 + 16 * v
        n, qs = primes(1 << 16, 24, 50)
        rng = PlanRng(seed)
        if v == 0:
            plan = dense_hybrid_plan(rng, 64, 1, 0, 0, 0)
        elif v == 1:
            plan = dense_hybrid_plan(rng, 64, 1, 32, 32, 0)
        else:
            plan = dense_hybrid_plan(rng, 64, 1, 16, 16, 0)
        return Workload(name, n, qs, plan, seed)
    if name == "vgg":
        seed = SEED_BASE + 2
        n, qs = primes(1 << 16, 20, 50)
        plan = dense_hybrid_plan(PlanRng(seed), 144, 16, 819, 819, 182)
        return Workload(name, n, qs, plan, seed)
    if name == "vit":
        seed = SEED_BASE + 3
        n, qs = primes(1 << 16, 16, 50)
        plan = dense_hybrid_plan(PlanRng(seed), 32, 24, 225, 225, 49, dag_share=0.25)
        return Workload(name, n, qs, plan, seed)
    if name == "bert":
        seed = SEED_BASE + 4
        n, qs = primes(1 << 16, 12, 50)
        plan = dense_hybrid_plan(PlanRng(seed), 96, 96, 2198, 2198, 488, dag_share=0.30)
        return Workload(name, n, qs, plan, seed)
    if name == "bert-const":
        # the BERT layer with its raw weights broadcast to every slot (single-
        # weight column packing): every raw plaintext is constant per limb
        seed = SEED_BASE + 4
        n, qs = primes(1 << 16, 12, 50)
        plan = dense_hybrid_plan(PlanRng(seed), 96, 96, 2198, 2198, 488, dag_share=0.30)
        return Workload(name, n, qs, constant_raw_plan(plan), seed, const_pts=plan.counts()["raw"])
    if name in ("overflow60", "overflow50"):
        # worst case for lazy reduction: every residue q-1 and more terms per
        # output than the accumulators hold without a fold (60-bit primes:
        # 256 products of 128 bits, 16 signed residues of 64 bits; 50-bit
        # primes on the radix-2^26 path: 2047 products, 64 packed residues)
        seed = SEED_BASE + 5
        bits_ = 60 if name == "overflow60" else 50
        n, qs = primes(1 << 10, 3, bits_)
        plan = _overflow_plan(PlanRng(seed), 400 if bits_ == 60 else 2100)
        return Workload(name, n, qs, plan, seed, fill="max")
    raise KeyError(name)


def constant_raw_plan(plan: Plan) -> Plan:
    """The same plan with every raw term marked constant (raw plaintexts
    come first, so they are plaintexts [0, raw count))."""
    terms = plan.terms.copy()
    raw = terms["kind"] == TERM_RAW
    assert not raw.any() or int(terms["pt"][raw].max()) < int(raw.sum())
    terms["kind"][raw] = TERM_RAW_CONST
    return dataclasses.replace(plan, terms=terms)


def worked_example_plan() -> Plan:
    """The routed example of Sec. 4.2 (Eq. "routed-example"), 0-based:
    y_1 = g1*A_1 - g1*A_3 + g_{1,2}*A_2 + g_{1,4}*A_4
    y_2 = g2*A_1 - g2*A_3 + g_{2,2}*A_2          (g_{2,4} has t = 0)
    with the shared signed sum U = A_1 - A_3 of Eq. "shared-example".
    Plaintexts: 0 = g_{1,2}, 1 = g_{1,4}, 2 = g_{2,2}, 3 = gamma_1, 4 = gamma_2.
    """
    R, T = TERM_RAW, TERM_TERNARY
    per_output = [
        [(0, T, 1, 0, 0), (1, R, 0, 0, 0), (2, T, -1, 0, 0), (3, R, 0, 1, 0)],
        [(0, T, 1, 0, 1), (1, R, 0, 2, 0), (2, T, -1, 0, 1), (3, T, 0, 0, 1)],
    ]
    nodes = [[(0, 0, 1), (2, 0, -1)]]
    uses = [(0, 0, 0, 1), (1, 1, 0, 1)]
    return build_plan(4, 2, per_output, 5, [3, 4], [0, 1], nodes, uses)


def _tiny_dag_plan(rng: PlanRng) -> Plan:
    """8 -> 4 layer with a two-level DAG: U0 = A0 - A1, U1 = U0 + A2.
    y0 uses +U1, y1 uses -U1, y2 uses +U0, y3 uses -U0 (plus direct terms)."""
    R, T = TERM_RAW, TERM_TERNARY
    fixed = {
        0: {0: 1, 1: -1, 2: 1},
        1: {0: -1, 1: 1, 2: -1},
        2: {0: 1, 1: -1},
        3: {0: -1, 1: 1},
    }
    per_output = []
    n_raw = 0
    layout = []
    for j in range(4):
        row = []
        for i in range(8):
            if i in fixed[j]:
                row.append(("t", fixed[j][i]))
            else:
                r = rng.below(5)
                if r < 2:
                    row.append(("r", 0))
                    n_raw += 1
                elif r == 2:
                    row.append(("t", 1))
                elif r == 3:
                    row.append(("t", -1))
                else:
                    row.append(("t", 0))
        layout.append(row)
    raw_id = 0
    for j in range(4):
        row = []
        for i, (kind, s) in enumerate(layout[j]):
            if kind == "r":
                row.append((i, R, 0, raw_id, 0))
                raw_id += 1
            else:
                row.append((i, T, s, 0, j))
        per_output.append(row)
    nodes = [[(0, 0, 1), (1, 0, -1)], [(0, 1, 1), (2, 0, 1)]]
    uses = [(0, 0, 1, 1), (1, 1, 1, -1), (2, 2, 0, 1), (3, 3, 0, -1)]
    return build_plan(8, 4, per_output, n_raw + 4, [n_raw + j for j in range(4)],
                       [0, 1, 2, 3], nodes, uses)


def _overflow_plan(rng: PlanRng, n_raw_long: int) -> Plan:
    """Worst case for lazy reduction on 60-bit primes: more products per output
    than a 128-bit accumulator holds (256 for q near 2^60), and long signed
    sums.  Inputs repeat (duplicate pairs sum), so 100 inputs suffice."""
    R, T = TERM_RAW, TERM_TERNARY
    n_in = 100
    per_output = []
    pt = 0
    # output 0: 300 raw products interleaved with 300 signed terms (1 scale)
    row = []
    for e in range(600):
        i = (e // 2) % n_in
        if e % 2 == 0:
            row.append((i, R, 0, pt, 0))
            pt += 1
        else:
            row.append((i, T, 1 if (e // 2) % 3 else -1, 0, 0))
    per_output.append(row)
    # output 1: 600 signed terms, all +1 (the signed accumulator's worst case)
    per_output.append([(e % n_in, T, 1, 0, 1) for e in range(600)])
    # output 2: n_raw_long raw products
    row = []
    for e in range(n_raw_long):
        row.append((e % n_in, R, 0, pt, 0))
        pt += 1
    per_output.append(row)
    n_raw = pt
    return build_plan(n_in, 3, per_output, n_raw + 2, [n_raw, n_raw + 1], [0, 1], [], [])
