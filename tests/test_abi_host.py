"""C-ABI library on the host (no GPU): it loads, exports every function the
headers declare, validates moduli and plans, and reports the paper's
operation counts.  Contexts here use FIONA_DEVICE_NONE (validation only)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_35352_gb300 import build as B
from paper_2609_35352_gb300 import fiona as F
from paper_2609_35352_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()


def declared_functions(header):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fiona_\w+)\s*\(", text)))


@pytest.mark.parametrize("header,path", [("fiona.h", F.LIB_PATH),
                                         ("fiona_workload.h", F.WORKLOAD_LIB_PATH)])
def test_library_exports_every_declared_symbol(header, path):
    lib = ctypes.CDLL(path)
    names = declared_functions(header)
    assert names
    for n in names:
        assert hasattr(lib, n), n
    if header == "fiona.h":
        assert set(F.EXPORTED) <= set(names)
        assert F.lib().fiona_abi_version() == 4


def ctx_none(N=1024, bits=40, L=3):
    return F.Context(N, W.ntt_primes(N, bits, L), device=F.FIONA_DEVICE_NONE)


def test_status_strings():
    assert F.status_str(0) == "ok"
    assert F.status_str(F.FIONA_ERR_PLAN) == "invalid plan"


@pytest.mark.parametrize("moduli,N,code", [
    ([1099511480321 + 2], 1 << 12, F.FIONA_ERR_MODULUS),                  # not 1 mod 2N
    ([(1 << 60) + 1], 1024, F.FIONA_ERR_MODULUS),                         # >= 2^60
    ([1099511480320], 1 << 12, F.FIONA_ERR_MODULUS),                      # even
    ([1099511480321 - 2 * 4096 * 3], 1 << 12, F.FIONA_ERR_MODULUS),        # composite, 1 mod 2N
    ([1099511480321, 1099511480321], 1 << 12, F.FIONA_ERR_MODULUS),       # repeated
    ([1099511480321], 3000, F.FIONA_ERR_ARG),                             # N not a power of 2
    ([1099511480321], 512, F.FIONA_ERR_ARG),                              # N < 2^10
])
def test_bad_moduli_rejected(moduli, N, code):
    if code == F.FIONA_ERR_MODULUS and len(moduli) == 1 and moduli[0] == 1099511480321 - 2 * 4096 * 3:
        assert not W.is_prime(moduli[0])
    with pytest.raises(F.FionaError) as ei:
        F.Context(N, moduli, device=F.FIONA_DEVICE_NONE)
    assert ei.value.status == code


def test_good_moduli_accepted():
    for N, bits, L in [(1 << 12, 40, 3), (1 << 16, 50, 24), (1 << 10, 60, 3), (1 << 17, 59, 2)]:
        ctx = F.Context(N, W.ntt_primes(N, bits, L), device=F.FIONA_DEVICE_NONE)
        ctx.close()


def read_golden_counts():
    vals = {}
    with open(os.path.join(ROOT, "tests", "golden", "worked_example_counts.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split()
                vals[k] = int(v)
    return vals


def test_worked_example_stats_match_paper():
    wl = W.make_workload("worked-example")
    plan = F.Plan(ctx_none(), wl.plan)
    s = plan.stats()
    for k, v in read_golden_counts().items():
        assert s[k] == v, (k, s[k], v)
    assert s["n_nonzero_terms"] == 7 and s["n_skipped_terms"] == 1
    assert s["n_nodes"] == 1 and s["n_uses"] == 2


def test_sharing_saving_matches_km_minus_m_minus_k():
    """A sum of m inputs shared by k outputs: k*m operands accumulated
    separately, versus m-1 Add/Sub to form it plus k operands (Sec. 4.2).
    Counted exactly the saving is (k-1)(m-1) = km - m - k + 1, one more than
    the paper's conservative estimate km - m - k."""
    for name in ("vit", "bert"):
        wl = W.make_workload(name)
        s = F.Plan(ctx_none(1 << 16, 50, 2), wl.plan).stats()
        p = wl.plan
        saving = 0
        for k in range(p.n_nodes):
            m = int(p.node_offsets[k + 1] - p.node_offsets[k])
            users = int(np.sum(p.uses["node"] == k))
            # separately: users*m operands; shared: (m-1) to form + users operands
            saving += users * m - (m - 1) - users
        assert s["addsub_flat"] - s["addsub_shared"] == saving
        assert saving > 0


def test_config_stats_and_bytes():
    wl = W.make_workload("bert")
    s = F.Plan(ctx_none(1 << 16, 50, 12), wl.plan).stats()
    assert s["n_nonzero_terms"] == 8728 and s["n_raw_terms"] == 4332
    assert s["pmult_per_term"] == 4332 + 4396 and s["pmult_grouped"] == 4332 + 96
    limb_poly = 8 * 12 * 65536
    assert s["bytes_min"] == limb_poly * (2 * 96 + 4428 + 2 * 96)
    assert abs(s["bytes_min"] / 1e9 - 30.27) < 0.01   # minimal bytes of the BERT-style layer
    assert s["rescale_separate"] == 192 and s["rescale_combined"] == 96
    w2 = W.make_workload("wsum-hybrid")
    s2 = F.Plan(ctx_none(1 << 16, 50, 24), w2.plan).stats()
    assert abs(s2["bytes_min"] / 1e9 - 2.051) < 0.001


def test_eval_on_validation_only_context_refuses():
    wl = W.make_workload("worked-example")
    plan = F.Plan(ctx_none(), wl.plan)
    assert plan.eval_status(16, 16, 16) == F.FIONA_ERR_NODEVICE


# -- negative plan validation ----------------------------------------------------
def mutate(plan, **kw):
    import copy
    p = copy.deepcopy(plan)
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def expect_plan_error(desc, code=F.FIONA_ERR_PLAN):
    with pytest.raises(F.FionaError) as ei:
        F.Plan(ctx_none(), desc)
    assert ei.value.status == code, F.last_error()


def test_plan_rejects_out_of_range_indices():
    base = W.make_workload("worked-example").plan
    for field, val in (("input", 4), ("pt", 5)):
        p = mutate(base)
        idx = 1  # a raw term
        p.terms[idx][field] = val
        expect_plan_error(p)
    p = mutate(base)
    p.terms[0]["group"] = 7
    expect_plan_error(p)
    p = mutate(base, group_scale_pt=np.array([3, 9], np.uint32))
    expect_plan_error(p)


def test_plan_rejects_bad_sign_and_kind():
    base = W.make_workload("worked-example").plan
    p = mutate(base)
    p.terms[0]["sign"] = 2
    expect_plan_error(p)
    p = mutate(base)
    p.terms[0]["kind"] = 5
    expect_plan_error(p)
    p = mutate(base)
    p.terms[1]["sign"] = 1   # raw term with a sign
    expect_plan_error(p)


def test_plan_rejects_group_of_other_output():
    base = W.make_workload("worked-example").plan
    p = mutate(base)
    p.terms[0]["group"] = 1   # output 0 term in output 1's group
    expect_plan_error(p)


def test_plan_rejects_dag_mismatch_and_overlap():
    base = W.make_workload("worked-example").plan
    # use with the wrong sign: -U does not match +A1 -A3 in output 0
    p = mutate(base)
    p.uses[0]["sign"] = -1
    expect_plan_error(p)
    # two uses of U in the same output overlap (Sec. 4.2: at most one of two
    # overlapping candidates per output)
    p = mutate(base)
    p.uses = np.concatenate([p.uses, p.uses[:1]])
    expect_plan_error(p)
    # node referencing a later node (cycle or wrong order)
    p = mutate(base)
    ch = np.zeros(3, W.CHILD_DTYPE)
    ch[0] = (0, 0, 1, 0)
    ch[1] = (2, 0, -1, 0)
    ch[2] = (0, 1, 1, 0)     # node 1 child = node 0 fine; make node 0 reference node 1
    p.node_offsets = np.array([0, 2, 3], np.uint32)
    p.children = ch.copy()
    p.children[0] = (1, 1, 1, 0)
    expect_plan_error(p)
    # node that expands to the same input twice
    p = mutate(base)
    p.children = np.array([(0, 0, 1, 0), (0, 0, -1, 0)], W.CHILD_DTYPE)
    expect_plan_error(p)


def test_plan_rejects_bad_offsets_and_reserved():
    base = W.make_workload("worked-example").plan
    p = mutate(base, term_offsets=np.array([0, 5, 4], np.uint32))
    expect_plan_error(p)
    p = mutate(base)
    p.terms[0]["reserved"] = 1
    expect_plan_error(p)


def test_edge_plans_accepted():
    # no terms at all, an output with only t = 0 terms, a single raw term
    R, T = W.TERM_RAW, W.TERM_TERNARY
    p = W.build_plan(0, 1, [[]], 0, [], [], [], [])
    s = F.Plan(ctx_none(), p).stats()
    assert s["n_terms"] == 0 and s["bytes_min"] == 2 * 3 * 1024 * 8
    p = W.build_plan(2, 2, [[(0, T, 0, 0, 0), (1, T, 0, 0, 0)], [(1, R, 0, 0, 0)]], 2, [1], [0],
                     [], [])
    s = F.Plan(ctx_none(), p).stats()
    assert s["n_skipped_terms"] == 2 and s["n_scale_groups_used"] == 0
    assert s["n_plaintexts_used"] == 1 and s["n_inputs_used"] == 1


def test_lower_level_arguments():
    """fiona_linear_eval_level checks the level before anything else; a
    validation-only context then refuses to evaluate."""
    wl = W.make_workload("tiny")
    ctx = F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE)
    plan = F.Plan(ctx, wl.plan)
    buf = np.zeros(16, dtype=np.uint64)
    for bad in (0, wl.L + 1):
        assert plan.eval_level_status(bad, buf, buf, buf) == F.FIONA_ERR_ARG
    assert plan.eval_level_status(1, buf, buf, buf) == F.FIONA_ERR_NODEVICE


def test_rescale_arguments_on_the_host():
    """fiona_rescale and fiona_linear_eval_rescale refuse a null ctx or plan
    and a validation-only context before touching any buffer."""
    buf = np.zeros(16, dtype=np.uint64)
    assert F.lib().fiona_rescale(None, None, 2, 1, F.addr(buf), F.addr(buf), 0) == F.FIONA_ERR_ARG
    assert F.lib().fiona_rescale(None, None, 2, 1, F.addr(buf), F.addr(buf), 2) == F.FIONA_ERR_ARG
    ctx = ctx_none()
    assert ctx.rescale_status(2, 1, buf, buf) == F.FIONA_ERR_NODEVICE
    wl = W.make_workload("tiny")
    plan = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan)
    assert plan.eval_rescale_status(2, buf, buf, buf, buf) == F.FIONA_ERR_NODEVICE
    assert F.lib().fiona_linear_eval_rescale(None, None, 2, 0, 0, 0, 0, 0) == F.FIONA_ERR_ARG


def test_constant_raw_terms_count_one_word_per_limb():
    """A plaintext read only by FIONA_TERM_RAW_CONST terms moves L words, not
    L limb-polys; every other count is that of the same layer with plain raw
    terms."""
    a = W.make_workload("bert-const", N=1024, L=3)
    b = W.make_workload("bert", N=1024, L=3)
    sa = F.Plan(F.Context(a.N, a.moduli, device=F.FIONA_DEVICE_NONE), a.plan).stats()
    sb = F.Plan(F.Context(b.N, b.moduli, device=F.FIONA_DEVICE_NONE), b.plan).stats()
    for k in ("n_raw_terms", "n_signed_terms", "n_plaintexts_used", "pmult_grouped", "addsub_shared"):
        assert sa[k] == sb[k], k
    n_raw_pts = a.const_pts
    assert sb["bytes_min"] - sa["bytes_min"] == n_raw_pts * (a.N * a.L * 8 - a.L * 8)
    # a constant term's plaintext index is checked like a raw one's
    bad = a.plan.terms.copy()
    e = int(np.nonzero(bad["kind"] == W.TERM_RAW_CONST)[0][0])
    bad["pt"][e] = a.plan.n_pt
    import dataclasses
    with pytest.raises(F.FionaError):
        F.Plan(F.Context(a.N, a.moduli, device=F.FIONA_DEVICE_NONE), dataclasses.replace(a.plan, terms=bad))


@pytest.mark.parametrize("name", ["tiny", "tiny-dag", "worked-example", "wsum-hybrid", "vgg", "vit", "bert",
                                  "bert-const"])
def test_minimal_bytes_counted_alike(name):
    """The benchmark's configuration counts the minimal bytes from the plan
    description alone (so that both of its arms print the same dict); the
    count equals fiona_plan_stats.bytes_min."""
    wl = W.make_workload(name)
    s = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan).stats()
    assert W.min_bytes(wl.plan, wl.L, wl.N) == s["bytes_min"]


def test_executed_addsub_reaches_the_papers_shared_count(monkeypatch):
    """The worked example (Sec. 4.2) on one warp: the kernel forms U = A_1 - A_3
    once and both outputs read it, so the Add/Sub it executes equal the
    paper's count with sharing (one subtraction saved: 5 -> 4); every other
    plan lies between the shared and the flat count, and the direct kernel
    executes the flat count."""
    monkeypatch.setenv("FIONA_TILED_SHAPE", "2,1,1")
    wl = W.make_workload("worked-example")
    plan = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan)
    s = plan.stats()
    assert s["nodes_materialized"] == 1
    assert s["addsub_executed"] == s["addsub_shared"] == 4 and s["addsub_flat"] == 5
    monkeypatch.delenv("FIONA_TILED_SHAPE")
    for name in ("tiny-dag", "vit", "bert", "vgg"):
        wl = W.make_workload(name)
        plan = F.Plan(F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE), wl.plan)
        s = plan.stats()
        assert s["addsub_shared"] <= s["addsub_executed"] <= s["addsub_flat"], (name, s)
        plan.select_kernel("direct")
        assert plan.stats()["addsub_executed"] == s["addsub_flat"]


def test_scale_class_plans():
    """fiona_plan_create_classes: argument checks, and the plan of a layer
    with two plaintext scales is that of its n_out * 2 results (each output's
    terms split by their plaintext's class, the counts preserved)."""
    wl = W.make_workload("tiny-dag")
    ctx = F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE)
    cls = W.scale_classes(wl.plan, 2, "random", seed=3)
    plan = F.Plan(ctx, wl.plan, pt_class=cls, n_class=2)
    s, s1 = plan.stats(), F.Plan(ctx, wl.plan).stats()
    assert s["n_out"] == 2 * wl.plan.n_out and plan.n_out == 2 * wl.plan.n_out
    for k in ("n_terms", "n_raw_terms", "n_signed_terms", "n_skipped_terms", "n_scale_groups_used"):
        assert s[k] == s1[k], k
    assert s["rescale_combined"] >= s1["rescale_combined"]
    one = F.Plan(ctx, wl.plan, pt_class=np.zeros(wl.plan.n_pt, np.uint8), n_class=1).stats()
    assert one == s1
    with pytest.raises(F.FionaError) as e:
        F.Plan(ctx, wl.plan, pt_class=cls, n_class=0)
    assert e.value.status == F.FIONA_ERR_ARG
    bad = cls.copy()
    bad[0] = 2
    with pytest.raises(F.FionaError) as e:
        F.Plan(ctx, wl.plan, pt_class=bad, n_class=2)
    assert e.value.status == F.FIONA_ERR_PLAN
