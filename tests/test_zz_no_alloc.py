"""fiona_linear_eval_static, the entry point for callers that cannot allocate
device memory when they evaluate (a runtime that gave all free memory to its
own pool, or a path where cudaMalloc's possible device synchronisation is not
allowed).  Its plan comes from a validation-only context, so nothing was
allocated on the device for it; its results must equal fiona_linear_eval's on
every residue, on consecutive calls.  This file is collected last on purpose."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()


def device_buffers(wl):
    p = wl.plan
    d_in = torch.from_numpy(wl.host_inputs().view(np.int64)).cuda()
    d_pt = torch.from_numpy(wl.host_plaintexts().view(np.int64)).cuda()
    return d_in, d_pt, p.n_out * 2 * wl.L * wl.N


@pytest.mark.parametrize("name,N,L", [("tiny-dag", None, None), ("vit", 2048, 2),
                                      ("overflow60", None, None), ("bert-const", 1024, 2)])
def test_static_entry_matches_linear_eval(name, N, L):
    """bert-const: constant raw plaintexts, which the kernel reads through
    their limb's first residue."""
    wl = W.make_workload(name, N=N, L=L)
    d_in, d_pt, n_out = device_buffers(wl)
    ref_ctx = F.Context(wl.N, wl.moduli, device=0)
    ref_plan = F.Plan(ref_ctx, wl.plan)
    want = torch.empty(n_out, dtype=torch.int64, device="cuda")
    ref_plan.eval(d_in, d_pt, want)

    ctx = F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE)
    plan = F.Plan(ctx, wl.plan)
    got = torch.empty(n_out, dtype=torch.int64, device="cuda")
    stream = torch.cuda.current_stream()
    for call in range(2):
        got.fill_(-1)
        assert plan.eval_static(d_in, d_pt, got, stream=stream) == F.FIONA_OK, F.last_error()
        torch.cuda.synchronize()
        assert torch.equal(got, want), "call %d differs from fiona_linear_eval" % call


def test_static_entry_matches_the_oracle():
    """The static entry point against the CPU oracle directly, on the
    host-generated residues of a small layer with a two-level DAG."""
    import oracle
    oracle.build()
    wl = W.make_workload("tiny-dag")
    X, P = wl.host_inputs(), wl.host_plaintexts()
    want = oracle.linear_eval(wl.plan, wl.moduli, X, P)
    d_in = torch.from_numpy(X.view(np.int64)).cuda()
    d_pt = torch.from_numpy(P.view(np.int64)).cuda()
    ctx = F.Context(wl.N, wl.moduli, device=F.FIONA_DEVICE_NONE)
    plan = F.Plan(ctx, wl.plan)
    got = torch.full((wl.plan.n_out * 2 * wl.L * wl.N,), -1, dtype=torch.int64, device="cuda")
    assert plan.eval_static(d_in, d_pt, got) == F.FIONA_OK, F.last_error()
    torch.cuda.synchronize()
    got = got.cpu().numpy().view(np.uint64).reshape(want.shape)
    assert np.array_equal(got, want)


def test_static_entry_rejects_layers_beyond_the_area():
    # 1000 inputs -> 140 outputs, all raw: 140000 raw terms need 1.1 MB > 1 MiB
    n_in, n_out = 1000, 140
    per_output = [[(i, W.TERM_RAW, 0, j * n_in + i, 0) for i in range(n_in)] for j in range(n_out)]
    desc = W.build_plan(n_in, n_out, per_output, n_in * n_out, [], [], [], [])
    ctx = F.Context(1024, W.ntt_primes(1024, 50, 1), device=F.FIONA_DEVICE_NONE)
    plan = F.Plan(ctx, desc)
    buf = torch.zeros(2, dtype=torch.int64, device="cuda")
    assert plan.eval_static(buf, buf, buf) == F.FIONA_ERR_ARG
    assert "static area" in F.last_error()
