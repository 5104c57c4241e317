"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself:
  * the worked example of Sec. 4.2 (Eq. "routed-example", Eq. "shared-example");
  * P1 exact distributivity: the hybrid result equals the all-PMult result in
    which every signed term becomes a raw term with plaintext t*gamma;
  * P2 brute force over Z_Q with CRT (Python integers);
  * P3 a tiny CKKS encode/encrypt/decrypt round trip against a float64
    slot-wise mat-vec, max-abs error <= 1e-3 at scale 2^40;
  * closed forms: t = 0, gamma = 1, +A - A, all residues q-1 (lazy bounds);
  * a planted-mistake check: mutated copies of oracle.c fail these pins.
"""
import os
import shutil

import numpy as np
import pytest

import oracle
from oracle import ckks_tiny, crt
from paper_2609_35352_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small_inputs(wl, n):
    """Host residues of a workload truncated to the first n coefficients."""
    i = np.arange(wl.plan.n_in).reshape(-1, 1, 1, 1)
    c = np.arange(2).reshape(1, -1, 1, 1)
    l = np.arange(wl.L).reshape(1, 1, -1, 1)
    k = np.arange(n).reshape(1, 1, 1, -1)
    X = wl.input_values(i, c, l, k)
    p = np.arange(wl.plan.n_pt).reshape(-1, 1, 1)
    P = wl.plaintext_values(p, l.reshape(1, -1, 1), k.reshape(1, 1, -1))
    return X, P


# -- worked example of Sec. 4.2 ---------------------------------------------
def test_worked_example_equations():
    wl = W.make_workload("worked-example")
    n = 16
    X, P = small_inputs(wl, n)
    y = oracle.linear_eval(wl.plan, wl.moduli, X, P)
    y_dag = oracle.linear_eval_dag(wl.plan, wl.moduli, X, P)
    # plaintext ids: 0 = g_{1,2}, 1 = g_{1,4}, 2 = g_{2,2}, 3 = gamma_1, 4 = gamma_2
    for l, q in enumerate(wl.moduli):
        for c in range(2):
            for k in range(n):
                A = [int(X[i, c, l, k]) for i in range(4)]
                g12, g14, g22, ga1, ga2 = (int(P[p, l, k]) for p in range(5))
                # Eq. routed-example, term by term
                y1 = (ga1 * A[0] - ga1 * A[2] + g12 * A[1] + g14 * A[3]) % q
                y2 = (ga2 * A[0] - ga2 * A[2] + g22 * A[1]) % q
                # Eq. shared-example, with U = A_1 - A_3
                U = A[0] - A[2]
                assert (ga1 * U + g12 * A[1] + g14 * A[3]) % q == y1
                assert (ga2 * U + g22 * A[1]) % q == y2
                assert int(y[0, c, l, k]) == y1 and int(y[1, c, l, k]) == y2
                assert int(y_dag[0, c, l, k]) == y1 and int(y_dag[1, c, l, k]) == y2


def test_worked_example_golden_counts_are_the_papers():
    vals = {}
    with open(os.path.join(GOLDEN, "worked_example_counts.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split()
                vals[k] = int(v)
    # numbers printed in Sec. 4.2: seven PMults, five after grouping, one
    # subtraction saved by sharing; one rescale per output after combining
    assert vals["pmult_per_term"] == 7 and vals["pmult_grouped"] == 5
    assert vals["addsub_flat"] - vals["addsub_shared"] == 1
    assert vals["rescale_combined"] * 2 == vals["rescale_separate"]


# -- P1: exact distributivity -------------------------------------------------
def all_pmult_equivalent(wl, X, P):
    """Rewrite every signed term as a raw term with plaintext t*gamma (mod q)."""
    plan = wl.plan
    q = wl.moduli_np.reshape(1, -1, 1)
    new_pts = [P]
    per_output = []
    next_pt = plan.n_pt
    t = plan.terms
    for j in range(plan.n_out):
        row = []
        for e in range(int(plan.term_offsets[j]), int(plan.term_offsets[j + 1])):
            i = int(t["input"][e])
            if t["kind"][e] == W.TERM_RAW:
                row.append((i, W.TERM_RAW, 0, int(t["pt"][e]), 0))
                continue
            s = int(t["sign"][e])
            gamma = P[int(plan.group_scale_pt[int(t["group"][e])])][None]
            if s == 1:
                pt = gamma
            elif s == -1:
                pt = (q - gamma) % q
            else:
                pt = np.zeros_like(gamma)
            new_pts.append(pt.astype(np.uint64))
            row.append((i, W.TERM_RAW, 0, next_pt, 0))
            next_pt += 1
        per_output.append(row)
    P2 = np.concatenate(new_pts, axis=0)
    plan2 = W.build_plan(plan.n_in, plan.n_out, per_output, next_pt, [], [], [], [])
    return plan2, P2


@pytest.mark.parametrize("name", ["tiny", "tiny-dag", "worked-example", "vit"])
def test_P1_distributivity(name):
    wl = W.make_workload(name, N=1024 if name == "vit" else None, L=2 if name == "vit" else None)
    X, P = small_inputs(wl, 32)
    y = oracle.linear_eval(wl.plan, wl.moduli, X, P)
    plan2, P2 = all_pmult_equivalent(wl, X, P)
    y2 = oracle.linear_eval(plan2, wl.moduli, X, P2)
    np.testing.assert_array_equal(y, y2)


# -- P2: CRT over the full modulus Q --------------------------------------------
@pytest.mark.parametrize("name", ["tiny", "tiny-dag", "worked-example"])
def test_P2_crt_bruteforce(name):
    wl = W.make_workload(name)
    X, P = small_inputs(wl, 8)
    y = oracle.linear_eval(wl.plan, wl.moduli, X, P)
    ref = crt.eval_over_ZQ(wl.plan, wl.moduli, X, P)
    np.testing.assert_array_equal(y, ref)
    if wl.plan.n_nodes:
        np.testing.assert_array_equal(oracle.linear_eval_dag(wl.plan, wl.moduli, X, P), ref)


def test_P2_crt_sixty_bit_primes():
    # the widest primes the library accepts: products near 2^120
    qs = W.ntt_primes(1024, 60, 3)
    wl = W.make_workload("tiny")
    wl = W.Workload("tiny60", 1024, qs, wl.plan, wl.seed)
    X, P = small_inputs(wl, 8)
    np.testing.assert_array_equal(oracle.linear_eval(wl.plan, qs, X, P),
                                  crt.eval_over_ZQ(wl.plan, qs, X, P))


# -- P3: tiny CKKS round trip ---------------------------------------------------
def ckks_case(lib=None, seed=7):
    N = 64
    qs = W.ntt_primes(N, 40, 3)
    ck = ckks_tiny.TinyCKKS(N, qs, delta_bits=40, seed=seed)
    ck.keygen()
    plan = W.make_workload("tiny").plan
    rng = np.random.default_rng(seed)
    slots = N // 2
    x = rng.uniform(-1, 1, (plan.n_in, slots))
    w = rng.uniform(-1, 1, (plan.n_pt, slots))
    # scale plaintexts hold reconstruction factors gamma > 0 (mean |W|, Sec. 4.1)
    for g in plan.group_scale_pt:
        w[int(g)] = rng.uniform(0.05, 1.0, slots)
    cts = np.stack([ck.encrypt(x[i]) for i in range(plan.n_in)])
    pts = np.stack([ck.encode_plaintext(w[p]) for p in range(plan.n_pt)])
    y_ct = oracle.linear_eval(plan, qs, cts, pts, lib=lib)
    dec = np.stack([ck.decrypt_decode(y_ct[j], float(ck.delta) ** 2) for j in range(plan.n_out)])
    ref = ckks_tiny.float_layer(plan, x, w)
    return float(np.max(np.abs(dec - ref)))


def test_P3_ckks_round_trip():
    err = ckks_case()
    assert err <= 1e-3, err


# -- closed forms -----------------------------------------------------------------
def test_closed_form_zero_and_identity():
    qs = W.ntt_primes(1024, 40, 3)
    R, T = W.TERM_RAW, W.TERM_TERNARY
    per_output = [
        [(0, T, 0, 0, 0), (1, T, 0, 0, 0)],          # all t = 0  -> 0
        [(1, T, 1, 0, 1)],                            # +A_1 scaled by gamma = 1 -> A_1
        [(0, T, 1, 0, 2), (0, T, -1, 0, 2)],          # +A_0 - A_0 -> 0
        [],                                           # no terms -> 0
        [(1, T, -1, 0, 3)],                           # -A_1 * 1 -> q - A_1
    ]
    plan = W.build_plan(2, 5, per_output, 2, [0, 1, 1, 1], [0, 1, 2, 4], [], [])
    wl = W.Workload("closed", 1024, qs, plan, 99)
    X, P = small_inputs(wl, 64)
    P[1] = 1  # gamma == 1 in every limb and slot
    y = oracle.linear_eval(plan, qs, X, P)
    q = wl.moduli_np.reshape(1, -1, 1)
    assert not y[0].any() and not y[2].any() and not y[3].any()
    np.testing.assert_array_equal(y[1], X[1])
    np.testing.assert_array_equal(y[4], (q - X[1]) % q)


@pytest.mark.parametrize("name", ["overflow60", "overflow50"])
def test_closed_form_all_max_residues(name):
    """Every residue q-1 = -1: a raw product is (+1), a signed term t*(-1)
    scaled by gamma = -1 is (+t); so y = #raw + sum(t) (mod q)."""
    wl = W.make_workload(name)
    X, P = small_inputs(wl, 4)
    y = oracle.linear_eval(wl.plan, wl.moduli, X, P)
    t = wl.plan.terms
    for j in range(wl.plan.n_out):
        sl = slice(int(wl.plan.term_offsets[j]), int(wl.plan.term_offsets[j + 1]))
        raw = int(np.sum(t["kind"][sl] == W.TERM_RAW))
        sgn = int(np.sum(t["sign"][sl][t["kind"][sl] == W.TERM_TERNARY]))
        for l, q in enumerate(wl.moduli):
            assert np.all(y[j, :, l] == np.uint64((raw + sgn) % q))


def test_constant_raw_terms_read_residue_zero():
    """Kind 2 (constant plaintext) is the raw route on the plaintext whose
    every coefficient is the limb's first residue: the same outputs as kind 0
    on that broadcast plaintext, and different ones on the original."""
    wl = W.make_workload("bert-const", N=1024, L=2)
    X, P = small_inputs(wl, 16)
    P = P.copy()
    P[: wl.const_pts] = W.residues_np(123, np.arange(P[: wl.const_pts].size, dtype=np.uint64).reshape(
        P[: wl.const_pts].shape), wl.moduli_np.reshape(1, -1, 1))  # not constant
    got = oracle.linear_eval(wl.plan, wl.moduli, X, P)
    flat = W.constant_raw_plan(wl.plan)
    flat.terms["kind"][flat.terms["kind"] == W.TERM_RAW_CONST] = W.TERM_RAW
    Pb = P.copy()
    Pb[: wl.const_pts] = P[: wl.const_pts, :, :1]
    assert np.array_equal(got, oracle.linear_eval(flat, wl.moduli, X, Pb))
    assert not np.array_equal(got, oracle.linear_eval(flat, wl.moduli, X, P))


def test_duplicate_pairs_sum():
    """Two groups on the same (output, input) pair add (plain summation)."""
    qs = W.ntt_primes(1024, 40, 2)
    R, T = W.TERM_RAW, W.TERM_TERNARY
    dup = W.build_plan(1, 1, [[(0, R, 0, 0, 0), (0, R, 0, 0, 0), (0, T, 1, 0, 0)]], 2, [1], [0],
                       [], [])
    once = W.build_plan(1, 1, [[(0, R, 0, 0, 0), (0, T, 1, 0, 0)]], 2, [1], [0], [], [])
    wl = W.Workload("dup", 1024, qs, dup, 5)
    X, P = small_inputs(wl, 16)
    q = wl.moduli_np.reshape(1, 1, -1, 1)
    a = oracle.linear_eval(dup, qs, X, P).astype(object)
    b = oracle.linear_eval(once, qs, X, P).astype(object)
    raw = (X.astype(object) * P[0][None].astype(object))[0:1] % q.astype(object)
    np.testing.assert_array_equal(a, (b + raw) % q.astype(object))


def test_dag_equals_flat_reduced_bert():
    wl = W.make_workload("bert", N=1024, L=1)
    X, P = small_inputs(wl, 4)
    np.testing.assert_array_equal(oracle.linear_eval(wl.plan, wl.moduli, X, P),
                                  oracle.linear_eval_dag(wl.plan, wl.moduli, X, P))


# -- planted mistakes ----------------------------------------------------------
@pytest.mark.parametrize("name,kind,n_class", [("tiny", "routes", 2), ("tiny-dag", "random", 3),
                                               ("worked-example", "random", 2)])
def test_scale_classes(name, kind, n_class):
    """Plaintexts at several scales (Sec. 4.2 "Combining the Signed and Raw
    Routes": routes combine within one scale): each class's result equals the
    brute-force evaluation over Z_Q of the layer restricted to that class's
    terms (a sub-plan built by filtering the term list), and the class
    results sum to the one-scale evaluation of the whole layer."""
    wl = W.make_workload(name)
    X, P = small_inputs(wl, 6)
    cls = W.scale_classes(wl.plan, n_class, kind, seed=3)
    assert len(set(cls.tolist())) > 1
    y = oracle.linear_eval_classes(wl.plan, wl.moduli, cls, n_class, X, P)
    for s_ in range(n_class):
        sub = W.class_subplan(wl.plan, cls, s_)
        assert np.array_equal(y[:, s_], crt.eval_over_ZQ(sub, wl.moduli, X, P)), s_
    q = np.array(wl.moduli, dtype=object).reshape(1, 1, -1, 1)
    total = (y.astype(object).sum(axis=1) % q).astype(np.uint64)
    assert np.array_equal(total, oracle.linear_eval(wl.plan, wl.moduli, X, P))
    one = oracle.linear_eval_classes(wl.plan, wl.moduli, np.zeros(wl.plan.n_pt, np.uint8), 1, X, P)
    assert np.array_equal(one[:, 0], oracle.linear_eval(wl.plan, wl.moduli, X, P))


def test_planted_class_mistake_is_caught(tmp_path):
    """The raw route's class test taken out of the oracle: the per-class
    brute force catches it."""
    src = open(os.path.join(os.path.dirname(oracle.__file__), "oracle.c")).read()
    old = "if (pt_class && pt_class[term_pt[e]] != want_class)"
    assert old in src
    path = tmp_path / "mutant.c"
    path.write_text(src.replace(old, "if (0)"))
    lib = oracle.load_variant(str(path), str(tmp_path / "libmutant.so"))
    wl = W.make_workload("tiny")
    X, P = small_inputs(wl, 6)
    cls = W.scale_classes(wl.plan, 2, "routes")
    y = oracle.linear_eval_classes(wl.plan, wl.moduli, cls, 2, X, P, lib=lib)
    assert not np.array_equal(y[:, 0], crt.eval_over_ZQ(W.class_subplan(wl.plan, cls, 0), wl.moduli, X, P))


MUTATIONS = {
    "sign_flip": ("s = sub_mod(s, a, q);", "s = add_mod(s, a, q);"),
    "dropped_raw": ("y = add_mod(y, mul_mod(p, a, q), q);", "(void)p; (void)a;"),
    "wrong_poly": ("uint64_t a = inputs[in_idx(term_input[e], c, l, k, L, n_coef)];",
                   "uint64_t a = inputs[in_idx(term_input[e], 1 - c, l, k, L, n_coef)];"),
    "gamma_transposed": ("uint64_t gamma = plaintexts[pt_idx(group_scale_pt[g], l, k, L, n_coef)];",
                         "uint64_t gamma = plaintexts[pt_idx(g, l, k, L, n_coef)];"),
    "no_reduction": ("return (uint64_t)(((u128)a * (u128)b) % q);",
                     "return (uint64_t)((u128)a * (u128)b);"),
}


@pytest.mark.parametrize("mutation", sorted(MUTATIONS))
def test_planted_mistake_is_caught(tmp_path, mutation):
    src = open(os.path.join(os.path.dirname(oracle.__file__), "oracle.c")).read()
    old, new = MUTATIONS[mutation]
    assert old in src
    path = tmp_path / "mutant.c"
    path.write_text(src.replace(old, new))
    lib = oracle.load_variant(str(path), str(tmp_path / "libmutant.so"))
    wl = W.make_workload("tiny")
    X, P = small_inputs(wl, 8)
    bad_p2 = not np.array_equal(oracle.linear_eval(wl.plan, wl.moduli, X, P, lib=lib),
                                crt.eval_over_ZQ(wl.plan, wl.moduli, X, P))
    bad_p3 = ckks_case(lib=lib) > 1e-3
    assert bad_p2 and bad_p3
