"""GPU parity of the tiled kernel's tensor-core signed sums (tc_signed.cuh):
every scale group's signed sum formed per tile as one contraction of the
inputs (cut into 10-bit fp16 chunks) with the layer's ternary weights on the
tensor cores, then reduced exactly (Sec. 4.2 "Grouping Reconstruction
Operations": the sum is the same element of Z_q however it is formed).  The
bar is bit-exact equality with the CPU oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402

from gpu_util import DeviceLayer, oracle_at, to_host  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()


# (layer, N, L, shape override "C,W,regions,keep,P" or None): warps per
# tensor-memory quarter 1 to 4, one and two source regions, several tiles per
# CTA (the contraction's barrier and tensor memory reused), residues q - 1
# everywhere (overflow50), shared sums expanded into the groups (vit,
# tiny-dag), a single output (wsum-ternary), inputs not a multiple of 16
# (vit: 32, tiny-dag: 8 -> zero rows of W).
CASES = [
    ("vgg", 1024, 2, None),
    ("vgg", 4096, 3, "1,16,1,-1,16"),
    ("vgg", 4096, 3, "1,12,1,-1,16"),
    ("vgg", 2048, 2, "1,8,0,-1,16"),
    ("vgg", 2048, 2, "1,4,1,-1,16"),
    ("overflow50", None, None, "1,16,1,-1,16"),
    ("vit", 2048, 2, "1,16,1,-1,16"),
    ("tiny-dag", None, None, "1,4,1,-1,16"),
    ("tiny", None, None, "1,8,0,-1,16"),
    ("wsum-ternary", 1024, 3, "1,4,1,-1,16"),
]


@pytest.mark.parametrize("name,N,L,shape", CASES)
def test_tensor_core_sums_parity(name, N, L, shape, monkeypatch):
    monkeypatch.setenv("FIONA_TILED_TC", "1")
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    wl = W.make_workload(name, N=N, L=L)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    st = dl.plan.stats()
    assert st["tensor_core_sums"] > 0, st
    if shape:
        f = [int(v) for v in shape.split(",")]
        assert (st["tile_coeffs"], st["warps_per_cta"]) == (32 * f[0], f[1]), st
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    for _ in range(2):  # the second launch on a dirty output buffer
        dl.run()
        mism = np.argwhere(dl.outputs() != want)
        assert mism.shape[0] == 0, "first mismatches (j, c, l, k): %s" % mism[:5].tolist()
    assert dl.ctx.device_check() == F.FIONA_OK


def test_tensor_core_sums_match_the_alu_sums(monkeypatch):
    """The same layer with the sums on the ALUs (the default) gives the same
    residues, on inputs the device generator fills."""
    wl = W.make_workload("vgg", N=4096, L=2)
    monkeypatch.setenv("FIONA_TILED_TC", "1")
    dl = DeviceLayer(wl, host_inputs=False)
    dl.plan.select_kernel("tiled")
    assert dl.plan.stats()["tensor_core_sums"] == 16
    dl.run()
    got_tc = dl.outputs().copy()
    monkeypatch.delenv("FIONA_TILED_TC")
    alu = F.Plan(dl.ctx, wl.plan)
    alu.select_kernel("tiled")
    assert alu.stats()["tensor_core_sums"] == 0
    dl.d_out.fill_(-1)
    alu.eval(dl.d_in, dl.d_pt, dl.d_out)
    assert np.array_equal(dl.outputs(), got_tc)
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("tc,shape", [("0", "1,16,1,-1,16"), ("1", "1,16,1,-1,16"), ("0", "1,8,0,-1,16")])
def test_tiled_copy_wait_runs_out(tc, shape, monkeypatch):
    """A test-only plan (FIONA_TEST_TILED_TIMEOUT) whose first input copy per
    CTA expects 16 bytes more than its TMA boxes bring, with waits bounded at
    2 ms: every thread's wait for the tile runs out, the CTA stops (thread 0
    waits, bounded, for its copies; the tensor-core variant frees its tensor
    memory), fiona_device_check reports FIONA_ERR_TIMEOUT once, and the next
    evaluation on the same context is exact."""
    monkeypatch.setenv("FIONA_TILED_TC", tc)
    monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    monkeypatch.setenv("FIONA_TEST_TILED_TIMEOUT", "1")
    wl = W.make_workload("vgg", N=2048, L=2)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    assert (dl.plan.stats()["tensor_core_sums"] > 0) == (tc == "1")
    dl.run()
    torch.cuda.synchronize()
    assert dl.ctx.device_check() == F.FIONA_ERR_TIMEOUT
    assert dl.ctx.device_check() == F.FIONA_OK  # the flag was cleared
    monkeypatch.delenv("FIONA_TEST_TILED_TIMEOUT")
    plan = F.Plan(dl.ctx, wl.plan)
    plan.select_kernel("tiled")
    plan.eval(dl.d_in, dl.d_pt, dl.d_out)
    torch.cuda.synchronize()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    assert np.array_equal(dl.outputs(), want)
    assert dl.ctx.device_check() == F.FIONA_OK


def test_tensor_core_sums_full_size(monkeypatch):
    """The full VGG layer (N = 2^16, 20 limbs, inputs filled on the device)
    with the tensor-core sums: outputs at sampled (limb, coefficient)
    coordinates equal the oracle's, every residue is canonical, and every
    residue equals the ALU sums' result."""
    monkeypatch.setenv("FIONA_TILED_TC", "1")
    wl = W.make_workload("vgg")
    dl = DeviceLayer(wl, host_inputs=False)
    dl.plan.select_kernel("tiled")
    assert dl.plan.stats()["tensor_core_sums"] == 16
    dl.run()
    torch.cuda.synchronize()
    rng = np.random.default_rng(43)
    limbs = rng.integers(0, wl.L, 48)
    coefs = rng.integers(0, wl.N, 48)
    coefs[:2] = [0, wl.N - 1]
    want = oracle_at(wl, limbs, coefs)
    out = dl.d_out.view(wl.plan.n_out, 2, wl.L, wl.N)
    got = to_host(out[:, :, torch.from_numpy(limbs).cuda(), torch.from_numpy(coefs).cuda()].contiguous())
    assert np.array_equal(got.reshape(want.shape), want)
    assert dl.ctx.check_residues(dl.d_out, wl.plan.n_out * 2) == F.FIONA_OK
    assert dl.ctx.device_check() == F.FIONA_OK
    first = dl.d_out.clone()
    monkeypatch.delenv("FIONA_TILED_TC")
    alu = F.Plan(dl.ctx, wl.plan)
    alu.select_kernel("tiled")
    assert alu.stats()["tensor_core_sums"] == 0
    dl.d_out.fill_(-1)
    alu.eval(dl.d_in, dl.d_pt, dl.d_out)
    torch.cuda.synchronize()
    assert torch.equal(first, dl.d_out)


def test_tensor_core_sums_with_scale_classes(monkeypatch):
    """Plaintexts at two scales (fiona_plan_create_classes: one result per
    output and class, groups split by their scale plaintext's class) with the
    tensor-core sums: every (output, class) result equals the oracle's."""
    from gpu_util import to_device
    monkeypatch.setenv("FIONA_TILED_TC", "1")
    monkeypatch.setenv("FIONA_TILED_SHAPE", "1,4,1,-1,16")
    wl = W.make_workload("tiny")
    cls = W.scale_classes(wl.plan, 2, "routes", seed=5)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan, pt_class=cls, n_class=2)
    plan.select_kernel("tiled")
    assert plan.stats()["tensor_core_sums"] > 0
    X, P = wl.host_inputs(), wl.host_plaintexts()
    p = wl.plan
    d_out = torch.full((p.n_out * 2 * 2 * wl.L * wl.N,), -1, dtype=torch.int64, device="cuda")
    plan.eval(to_device(X), to_device(P), d_out)
    torch.cuda.synchronize()
    got = to_host(d_out).reshape(p.n_out, 2, 2, wl.L, wl.N)
    want = oracle.linear_eval_classes(p, wl.moduli, cls, 2, X, P)
    mism = np.argwhere(got != want)
    assert mism.shape[0] == 0, "first mismatches (j, s, c, l, k): %s" % mism[:5].tolist()
    assert ctx.device_check() == F.FIONA_OK
