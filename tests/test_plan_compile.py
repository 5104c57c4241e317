"""Host plan compiler (fiona_plan_compile, Sec. 4.2): from a dense route
matrix to terms, scale groups and shared signed sums.  CPU only: plans are
checked by fiona_plan_create's validation (every use matches its output's
terms, no term covered twice), by the paper's worked example, and by the
oracle, whose DAG form must equal its flat form."""
import os

import numpy as np
import pytest

import oracle
from paper_2609_35352_gb300 import build as B
from paper_2609_35352_gb300 import fiona as F
from paper_2609_35352_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
R, T = W.TERM_RAW, W.TERM_TERNARY


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()
    oracle.build()


def ctx_none(N=1024, L=2):
    return F.Context(N, W.ntt_primes(N, 40, L), device=F.FIONA_DEVICE_NONE)


def worked_example_routes():
    """Eq. "routed-example" (0-based), plaintexts numbered as in
    workloads.worked_example_plan: 0 = g_{1,2}, 1 = g_{1,4}, 2 = g_{2,2},
    3 = gamma_1, 4 = gamma_2; g_{2,4} is the all-zero group (t = 0)."""
    r = np.zeros((2, 4), F.ROUTE_DTYPE)
    r[0] = [(T, 1, 0, 3), (R, 0, 0, 0), (T, -1, 0, 3), (R, 0, 0, 1)]
    r[1] = [(T, 1, 0, 4), (R, 0, 0, 2), (T, -1, 0, 4), (T, 0, 0, 4)]
    return r


def golden_counts():
    vals = {}
    with open(os.path.join(ROOT, "tests", "golden", "worked_example_counts.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split()
                vals[k] = int(v)
    return vals


def test_worked_example_compiles_to_the_papers_plan():
    """With the exact saving rule the compiler finds U = A_1 - A_3, used by
    both outputs (Eq. "shared-example"), and the plan has the paper's counts:
    7 -> 5 PMults, one Sub saved, 4 -> 2 rescales."""
    d = F.compile_plan(4, 2, 5, worked_example_routes(), share=True, exact=True)
    ref = W.worked_example_plan()
    assert np.array_equal(d.term_offsets, ref.term_offsets)
    assert np.array_equal(d.terms, ref.terms)
    assert d.group_scale_pt.tolist() == [3, 4] and d.group_output.tolist() == [0, 1]
    assert d.node_offsets.tolist() == [0, 2]
    assert [(int(c["ref"]), int(c["sign"])) for c in d.children] == [(0, 1), (2, -1)]
    assert [(int(u["output"]), int(u["group"]), int(u["node"]), int(u["sign"])) for u in d.uses] == \
        [(0, 0, 0, 1), (1, 1, 0, 1)]
    s = F.Plan(ctx_none(), d).stats()
    for k, v in golden_counts().items():
        assert s[k] == v, (k, s[k], v)


def test_conservative_estimate_rejects_the_worked_example():
    """Under the paper's estimate km - m - k the worked example's sum
    (m = 2, k = 2) estimates 0 and is not taken: the paper's acceptance
    rule and its own example disagree, which is why the compiler offers the
    exact rule too.  Grouping still takes 7 PMults to 5."""
    d = F.compile_plan(4, 2, 5, worked_example_routes(), share=True, exact=False)
    assert d.node_offsets.tolist() == [0] and d.uses.shape[0] == 0
    s = F.Plan(ctx_none(), d).stats()
    assert s["pmult_per_term"] == 7 and s["pmult_grouped"] == 5
    assert s["addsub_flat"] == s["addsub_shared"] == 5


def test_sharing_off_gives_grouping_only():
    d = F.compile_plan(4, 2, 5, worked_example_routes(), share=False)
    assert d.node_offsets.tolist() == [0] and d.children.shape[0] == 0


def random_routes(n_in, n_out, n_gamma, seed, p_raw=0.4, p_zero=0.1):
    rng = np.random.default_rng(seed)
    r = np.zeros((n_out, n_in), F.ROUTE_DTYPE)
    n_raw = 0
    for j in range(n_out):
        for i in range(n_in):
            u = rng.random()
            if u < p_raw:
                r[j, i] = (R, 0, 0, n_gamma * n_out + n_raw)
                n_raw += 1
            else:
                t = 0 if u < p_raw + p_zero else int(rng.choice([-1, 1]))
                r[j, i] = (T, t, 0, j * n_gamma + int(rng.integers(n_gamma)))
    return r, n_gamma * n_out + n_raw


@pytest.mark.parametrize("n_in,n_out,n_gamma,exact,seed", [
    (12, 6, 1, False, 1), (12, 6, 1, True, 2), (20, 10, 2, True, 3), (32, 24, 1, False, 4),
])
def test_random_layers_compile_to_valid_plans(n_in, n_out, n_gamma, exact, seed):
    """The compiled plan passes fiona_plan_create's checks; its DAG form
    evaluates (oracle) to the flat form; shared sums save Add/Sub."""
    r, n_pt = random_routes(n_in, n_out, n_gamma, seed)
    d = F.compile_plan(n_in, n_out, n_pt, r, share=True, exact=exact)
    s = F.Plan(ctx_none(), d).stats()
    assert s["n_terms"] == n_in * n_out
    assert s["n_groups"] <= n_out * n_gamma
    if s["n_nodes"]:
        assert s["addsub_shared"] < s["addsub_flat"]
    # every ternary route is a term of its output with the same sign and gamma
    for j in range(n_out):
        for i in range(n_in):
            t = d.terms[d.term_offsets[j] + i]
            assert int(t["input"]) == i and int(t["kind"]) == int(r[j, i]["kind"])
            if t["kind"] == T:
                assert int(t["sign"]) == int(r[j, i]["sign"])
                assert int(d.group_scale_pt[t["group"]]) == int(r[j, i]["pt"])
                assert int(d.group_output[t["group"]]) == j
            else:
                assert int(t["pt"]) == int(r[j, i]["pt"])
    qs = W.ntt_primes(1024, 40, 2)
    wl = W.Workload("compiled", 1024, qs, d, 4242 + seed)
    X, P = wl.host_inputs(), wl.host_plaintexts()
    flat = oracle.linear_eval(d, qs, X[..., :64], P[..., :64])
    dag = oracle.linear_eval_dag(d, qs, X[..., :64], P[..., :64])
    assert np.array_equal(flat, dag)


def test_compiler_rejects_malformed_routes():
    r = worked_example_routes()
    bad = r.copy()
    bad[0, 1]["kind"] = 3
    with pytest.raises(F.FionaError) as e:
        F.compile_plan(4, 2, 5, bad)
    assert e.value.status == F.FIONA_ERR_PLAN
    bad = r.copy()
    bad[1, 0]["pt"] = 5
    with pytest.raises(F.FionaError) as e:
        F.compile_plan(4, 2, 5, bad)
    assert e.value.status == F.FIONA_ERR_PLAN
    bad = r.copy()
    bad[0, 1]["sign"] = 1          # a raw route with a sign
    with pytest.raises(F.FionaError):
        F.compile_plan(4, 2, 5, bad)
