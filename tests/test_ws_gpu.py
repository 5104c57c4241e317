"""GPU parity of the warp-specialised tiled kernel (a producer warp streams
plaintext tiles into shared-memory rings, a stager warp copies the inputs by
TMA), against the CPU oracle, bit-exact; and its bounded waits: a wait made to
run out reports FIONA_ERR_TIMEOUT and leaves the context usable."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402

from gpu_util import DeviceLayer, to_device, to_host  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()


CASES = [
    ("tiny", None, None),
    ("tiny-dag", None, None),
    ("worked-example", None, None),
    ("wsum-hybrid", 2048, 2),
    ("vgg", 1024, 2),
    ("vit", 2048, 2),
    ("bert", 1024, 1),
    ("bert-const", 1024, 1),
    ("overflow60", None, None),
    ("overflow50", None, None),
]
# consumer warps, source regions, ring depth in batches (None: the lowering's choice)
SHAPES = [None, "16,1,3", "15,2,4", "8,2,4", "4,2,3", "12,1,3"]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("name,N,L", CASES)
def test_ws_parity(name, N, L, shape, monkeypatch):
    monkeypatch.setenv("FIONA_TILED_WS", "1")
    if shape:
        monkeypatch.setenv("FIONA_WS_SHAPE", shape)
    wl = W.make_workload(name, N=N, L=L)
    dl = DeviceLayer(wl)
    try:
        dl.plan.select_kernel("tiled")
    except F.FionaError:
        if shape:
            pytest.skip("shape %s does not fit this layer in shared memory" % shape)
        raise
    st = dl.plan.stats()
    assert st["tile_coeffs"] == 64
    if shape:
        assert st["warps_per_cta"] == int(shape.split(",")[0])
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    for _ in range(2):  # the second launch on a dirty output buffer
        dl.run()
        got = dl.outputs()
        mism = np.argwhere(got != want)
        assert mism.shape[0] == 0, "first mismatches (j, c, l, k): %s" % mism[:5].tolist()
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("name,N,L", [("vit", 2048, 3), ("overflow50", None, None)])
def test_ws_lower_level(name, N, L, monkeypatch):
    monkeypatch.setenv("FIONA_TILED_WS", "1")
    wl = W.make_workload(name, N=N, L=L)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan)
    plan.select_kernel("tiled")
    X, P = wl.host_inputs(), wl.host_plaintexts()
    p = wl.plan
    for Le in range(1, wl.L):
        Xl = np.ascontiguousarray(X[:, :, :Le, :])
        Pl = np.ascontiguousarray(P[:, :Le, :])
        d_out = torch.full((p.n_out * 2 * Le * wl.N,), -1, dtype=torch.int64, device="cuda")
        plan.eval_level(Le, to_device(Xl), to_device(Pl), d_out)
        torch.cuda.synchronize()
        got = to_host(d_out).reshape(p.n_out, 2, Le, wl.N)
        assert np.array_equal(got, oracle.linear_eval(p, wl.moduli[:Le], Xl, Pl)), Le
    assert ctx.device_check() == F.FIONA_OK


def test_ws_wait_runs_out(monkeypatch):
    """A test-only plan whose first input copy expects 16 bytes more than it
    issues (and whose waits give up after 2 ms): the consumer warps' wait for
    the tile runs out, the kernel stops, fiona_device_check reports
    FIONA_ERR_TIMEOUT, and the next evaluation on the same context is exact."""
    monkeypatch.setenv("FIONA_TILED_WS", "1")
    monkeypatch.setenv("FIONA_TEST_WS_TIMEOUT", "1")
    wl = W.make_workload("vit", N=2048, L=2)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    dl.run()
    torch.cuda.synchronize()
    assert dl.ctx.device_check() == F.FIONA_ERR_TIMEOUT
    assert dl.ctx.device_check() == F.FIONA_OK  # the flag was cleared
    monkeypatch.delenv("FIONA_TEST_WS_TIMEOUT")
    plan = F.Plan(dl.ctx, wl.plan)
    plan.select_kernel("tiled")
    plan.eval(dl.d_in, dl.d_pt, dl.d_out)
    torch.cuda.synchronize()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    assert np.array_equal(dl.outputs(), want)
    assert dl.ctx.device_check() == F.FIONA_OK
