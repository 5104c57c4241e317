"""GPU parity: the CUDA path, called through the C ABI, against the CPU
oracle on the same seeded inputs.  The bar is bit-exact equality of every
residue (integer arithmetic mod q, a unique canonical result)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402

from gpu_util import DeviceLayer, oracle_at, to_device, to_host  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()


# Reduced sizes: the same plan structure, N and L small enough for the oracle
# to finish in seconds, still many coefficient tiles per limb.
SMALL = [
    ("tiny", None, None),
    ("tiny-dag", None, None),
    ("worked-example", None, None),
    ("wsum-pmult", 1024, 3),
    ("wsum-ternary", 1024, 3),
    ("wsum-hybrid", 2048, 2),
    ("vgg", 1024, 2),
    ("vit", 2048, 2),
    ("bert", 1024, 1),
    ("bert-const", 1024, 1),
    ("overflow60", None, None),
    ("overflow50", None, None),
]


@pytest.mark.parametrize("kernel", ["direct", "tiled"])
@pytest.mark.parametrize("name,N,L", SMALL)
def test_elementwise_parity_small(name, N, L, kernel):
    wl = W.make_workload(name, N=N, L=L)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel(kernel)
    assert dl.plan.stats()["kernel"] == F.KERNELS[kernel]
    dl.run()
    got = dl.outputs()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    mism = np.argwhere(got != want)
    assert mism.shape[0] == 0, "first mismatches (j, c, l, k): %s" % mism[:5].tolist()
    # a second launch on a dirty output buffer gives the same result
    dl.run()
    assert np.array_equal(dl.outputs(), want)
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("name,N,L", [("tiny-dag", None, None), ("vgg", 1024, 2), ("vit", 2048, 2),
                                      ("bert-const", 1024, 1), ("overflow50", None, None)])
def test_packed_programs_parity(name, N, L, monkeypatch):
    """The tiled kernel with its signed-sum programs as packed 16-bit indices
    (FIONA_TILED_PACKED=1; the form a schedule takes when the offset form
    does not fit in shared memory) gives the same residues."""
    monkeypatch.setenv("FIONA_TILED_PACKED", "1")
    wl = W.make_workload(name, N=N, L=L)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    assert dl.plan.stats()["source_offsets"] == 0
    dl.run()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    assert np.array_equal(dl.outputs(), want)


@pytest.mark.parametrize("mixed", [False, True])
@pytest.mark.parametrize("N,L", [(1024, 2), (4096, 1)])
def test_all_constant_plaintexts_parity(N, L, mixed, monkeypatch):
    """A layer whose every raw plaintext is constant (bert-const) on the
    12-warp shape: the kernel variant that reads every operation after a
    batch's first as constant, and (FIONA_TILED_KC_MIXED=1) the one that
    tests each operation, give the same residues as the oracle."""
    monkeypatch.setenv("FIONA_TILED_SHAPE", "2,12,1,-1,8")
    if mixed:
        monkeypatch.setenv("FIONA_TILED_KC_MIXED", "1")
    wl = W.make_workload("bert-const", N=N, L=L)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    st = dl.plan.stats()
    assert st["warps_per_cta"] == 12 and st["const_raw_all"] == (0 if mixed else 1)
    dl.run()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    assert np.array_equal(dl.outputs(), want)


# Tiled shapes (coefficients per lane, warps, source regions[, most shared
# sums kept (-1: the lowering's choice)[, operations per batch]]) chosen
# through the lowering's override; every shape must give the same residues.
# A fourth field forces the shared sums in play (0: all expanded), a fifth
# selects batches of 4 (or 8: "2,12,1,-1,8" and "2,8,1,-1,8" take the
# variant built for CTAs of at most 12 warps, two coefficients per lane).
SHAPES = ["2,16,0", "2,8,1", "1,16,1", "1,4,0", "2,12,1,0", "1,8,0,3", "2,8,1,-1,4", "1,16,0,2,4", "2,12,1,-1,8",
          "2,8,1,-1,8"]
SHAPE_CASES = [("tiny-dag", None, None), ("vit", 2048, 2), ("bert", 1024, 1), ("bert-const", 1024, 1),
               ("vgg", 1024, 2),
               ("overflow60", None, None), ("overflow50", None, None)]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("name,N,L", SHAPE_CASES)
def test_tiled_shapes(name, N, L, shape, monkeypatch):
    monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    wl = W.make_workload(name, N=N, L=L)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    st = dl.plan.stats()
    f = [int(v) for v in shape.split(",")]
    if (st["tile_coeffs"], st["warps_per_cta"]) != (32 * f[0], f[1]):
        pytest.skip("shape %s does not fit this layer in shared memory" % shape)
    if len(f) >= 4 and f[3] >= 0:
        assert st["nodes_materialized"] <= f[3]
    dl.run()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    got = dl.outputs()
    mism = np.argwhere(got != want)
    assert mism.shape[0] == 0, "first mismatches (j, c, l, k): %s" % mism[:5].tolist()
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("kernel", ["direct", "tiled"])
@pytest.mark.parametrize("name,N,L,levels", [("tiny", None, None, [1, 2]), ("vit", 2048, 3, [1, 2]),
                                              ("overflow50", None, None, [1])])
def test_lower_level_parity(name, N, L, levels, kernel):
    """fiona_linear_eval_level: buffers holding the first L_eval limbs, the
    same plan; the oracle on the first L_eval moduli."""
    wl = W.make_workload(name, N=N, L=L)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan)
    plan.select_kernel(kernel)
    X, P = wl.host_inputs(), wl.host_plaintexts()
    p = wl.plan
    for Le in levels:
        Xl = np.ascontiguousarray(X[:, :, :Le, :])
        Pl = np.ascontiguousarray(P[:, :Le, :])
        d_out = torch.full((p.n_out * 2 * Le * wl.N,), -1, dtype=torch.int64, device="cuda")
        plan.eval_level(Le, to_device(Xl), to_device(Pl), d_out)
        torch.cuda.synchronize()
        got = to_host(d_out).reshape(p.n_out, 2, Le, wl.N)
        want = oracle.linear_eval(p, wl.moduli[:Le], Xl, Pl)
        mism = np.argwhere(got != want)
        assert mism.shape[0] == 0, (Le, mism[:5].tolist())
    assert plan.eval_level_status(0, to_device(X), to_device(P), d_out) == F.FIONA_ERR_ARG
    assert plan.eval_level_status(wl.L + 1, to_device(X), to_device(P), d_out) == F.FIONA_ERR_ARG


@pytest.mark.parametrize("shape", [None, "2,8,1,64", "1,4,0,64,4"])
def test_compiled_plan_parity(shape, monkeypatch):
    """A dense layer through the host plan compiler (shared sums found by the
    Sec. 4.2 search), evaluated by both kernels (the shapes keep the sums in
    play, so the kernel forms them per tile), against the oracle's flat form."""
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    rng = np.random.default_rng(7)
    n_in, n_out = 24, 12
    r = np.zeros((n_out, n_in), F.ROUTE_DTYPE)
    n_raw = 0
    for j in range(n_out):
        for i in range(n_in):
            u = rng.random()
            if u < 0.3:
                r[j, i] = (W.TERM_RAW, 0, 0, n_out + n_raw)
                n_raw += 1
            else:
                r[j, i] = (W.TERM_TERNARY, 0 if u < 0.35 else int(rng.choice([-1, 1])), 0, j)
    d = F.compile_plan(n_in, n_out, n_out + n_raw, r, share=True, exact=True)
    assert d.node_offsets.shape[0] > 1
    wl = W.Workload("compiled", 2048, W.ntt_primes(2048, 50, 2), d, 99)
    dl = DeviceLayer(wl)
    want = oracle.linear_eval(d, wl.moduli, dl.X, dl.P)
    for kernel in ("direct", "tiled"):
        dl.plan.select_kernel(kernel)
        dl.d_out.fill_(-1)
        dl.run()
        assert np.array_equal(dl.outputs(), want), kernel
    if shape:
        assert dl.plan.stats()["nodes_materialized"] > 0


def test_edge_plans():
    R, T = W.TERM_RAW, W.TERM_TERNARY
    qs = W.ntt_primes(1024, 50, 3)
    plans = [
        W.build_plan(0, 1, [[]], 0, [], [], [], []),                          # no terms
        W.build_plan(2, 2, [[(0, T, 0, 0, 0), (1, T, 0, 0, 0)], [(1, R, 0, 0, 0)]], 2, [1], [0],
                     [], []),                                                  # only t = 0
        W.build_plan(1, 1, [[(0, R, 0, 0, 0), (0, R, 0, 0, 0), (0, T, 1, 0, 0)]], 2, [1], [0],
                     [], []),                                                  # duplicate pair
        W.build_plan(3, 3, [[(2, T, -1, 0, 0)], [(0, T, 1, 0, 1), (1, T, 1, 0, 1)], []], 3,
                     [2, 2], [0, 1], [], []),                                  # ragged outputs
    ]
    for i, p in enumerate(plans):
        wl = W.Workload("edge%d" % i, 1024, qs, p, 1000 + i)
        dl = DeviceLayer(wl)
        want = oracle.linear_eval(p, qs, dl.X, dl.P)
        for kernel in ("direct", "tiled"):
            dl.plan.select_kernel(kernel)
            dl.d_out.fill_(-1)
            dl.run()
            assert np.array_equal(dl.outputs(), want), (i, kernel)



@pytest.mark.parametrize("n_in", [1, 200, 259])
def test_tma_input_boxes(n_in, monkeypatch):
    """One coefficient per lane stages a tile's 2 n_in input polys with TMA
    boxes of at most 256 polys: one box (2 polys), two (400 polys, 200 each)
    and three whose last one overlaps the second (518 polys: boxes of 173 at
    0, 173 and 345)."""
    monkeypatch.setenv("FIONA_TILED_SHAPE", "1,4,0")
    rng = np.random.default_rng(n_in)
    n_out = 3
    r = np.zeros((n_out, n_in), F.ROUTE_DTYPE)
    n_raw = 0
    for j in range(n_out):
        for i in range(n_in):
            if rng.random() < 0.3:
                r[j, i] = (W.TERM_RAW, 0, 0, n_out + n_raw)
                n_raw += 1
            else:
                r[j, i] = (W.TERM_TERNARY, int(rng.choice([-1, 0, 1])), 0, j)
    desc = F.compile_plan(n_in, n_out, n_out + n_raw, r, share=False)
    qs = W.ntt_primes(1024, 50, 2)
    wl = W.Workload("boxes%d" % n_in, 1024, qs, desc, 4200 + n_in)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    assert dl.plan.stats()["tile_coeffs"] == 32
    want = oracle.linear_eval(desc, qs, dl.X, dl.P)
    dl.d_out.fill_(-1)
    dl.run()
    assert np.array_equal(dl.outputs(), want)
    assert dl.ctx.device_check() == F.FIONA_OK

def test_boundary_residues():
    """Residues 0, 1, q-1 and random, on 60-bit primes (widest accepted)."""
    qs = W.ntt_primes(1024, 60, 2)
    wl = W.make_workload("tiny", N=1024)
    wl = W.Workload("tiny60", 1024, qs, wl.plan, wl.seed)
    dl = DeviceLayer(wl)
    X, P = dl.X.copy(), dl.P.copy()
    q = wl.moduli_np.reshape(1, 1, -1, 1)
    X[..., 0:8] = 0
    X[..., 8:16] = 1
    X[..., 16:64] = (q - 1)
    P[..., 32:64] = q.reshape(1, -1, 1) - 1
    P[..., 64:72] = 0
    dl.d_in.copy_(to_device(X))
    dl.d_pt.copy_(to_device(P))
    want = oracle.linear_eval(wl.plan, qs, X, P)
    for kernel in ("direct", "tiled"):
        dl.plan.select_kernel(kernel)
        dl.run()
        assert np.array_equal(dl.outputs(), want), kernel


@pytest.mark.parametrize("kernel,shape", [("direct", None), ("tiled", None), ("tiled", "2,16,0"),
                                          ("tiled", "1,16,1"), ("tiled", "2,12,1,-1,8")])
@pytest.mark.parametrize("bits", [51, 52])
def test_widest_narrow_moduli(bits, kernel, shape, monkeypatch):
    """The radix-2^26 arithmetic at the widest moduli it takes (every q below
    2^52, high digits up to 2^26 - 1): every residue q - 1, and more products
    and signed terms per output than the lazy bounds allow between
    reductions, so that every accumulator comes near its bound; one and two
    coefficients per lane, the 12-warp variant, and the direct kernel."""
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    wl = W.make_workload("overflow50", bits=bits)
    assert all(int(q).bit_length() == bits for q in wl.moduli)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel(kernel)
    st = dl.plan.stats()
    if shape:
        f = [int(v) for v in shape.split(",")]
        if (st["tile_coeffs"], st["warps_per_cta"]) != (32 * f[0], f[1]):
            pytest.skip("shape %s does not fit this layer in shared memory" % shape)
    dl.run()
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    mism = np.argwhere(dl.outputs() != want)
    assert mism.shape[0] == 0, "first mismatches (j, c, l, k): %s" % mism[:5].tolist()
    assert dl.ctx.device_check() == F.FIONA_OK


FULL = ["wsum-pmult", "wsum-ternary", "wsum-hybrid", "vgg", "vit", "bert", "bert-const"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled_parity(name):
    """Full N = 2^16 layer, inputs filled on the device, evaluated with the
    kernel the plan selects by default (the launch the benchmark times);
    outputs compared with the oracle at sampled (limb, coefficient)
    coordinates, every output."""
    wl = W.make_workload(name)
    dl = DeviceLayer(wl, host_inputs=False)
    dl.run()
    torch.cuda.synchronize()
    rng = np.random.default_rng(42)
    n_s = 24 if name.startswith("bert") else 64
    limbs = rng.integers(0, wl.L, n_s)
    coefs = rng.integers(0, wl.N, n_s)
    coefs[:2] = [0, wl.N - 1]
    want = oracle_at(wl, limbs, coefs)
    out = dl.d_out.view(wl.plan.n_out, 2, wl.L, wl.N)
    got = to_host(out[:, :, torch.from_numpy(limbs).cuda(), torch.from_numpy(coefs).cuda()].contiguous())
    assert np.array_equal(got.reshape(want.shape), want)
    # every residue canonical
    assert dl.ctx.check_residues(dl.d_out, wl.plan.n_out * 2) == F.FIONA_OK
    assert dl.ctx.device_check() == F.FIONA_OK
    # the other kernel variant agrees on every residue
    other = "direct" if dl.plan.stats()["kernel"] == F.FIONA_KERNEL_TILED else "tiled"
    first = dl.d_out.clone()
    dl.plan.select_kernel(other)
    dl.d_out.fill_(-1)
    dl.run()
    torch.cuda.synchronize()
    assert torch.equal(first, dl.d_out)


def test_device_fill_matches_host_generator():
    wl = W.make_workload("vit")
    dl = DeviceLayer(wl, host_inputs=False)
    torch.cuda.synchronize()
    rng = np.random.default_rng(3)
    for _ in range(4):
        i, c, l = int(rng.integers(32)), int(rng.integers(2)), int(rng.integers(16))
        k = rng.integers(0, wl.N, 50)
        dev = to_host(dl.d_in.view(32, 2, 16, wl.N)[i, c, l].contiguous())[k]
        assert np.array_equal(dev, wl.input_values(i, c, l, k))
        p = int(rng.integers(wl.plan.n_pt))
        devp = to_host(dl.d_pt.view(wl.plan.n_pt, 16, wl.N)[p, l].contiguous())[k]
        assert np.array_equal(devp, wl.plaintext_values(p, l, k))


def test_constant_plaintexts_are_read_at_residue_zero():
    """FIONA_TERM_RAW_CONST: a constant plaintext's other residues are never
    read -- overwriting them changes no output, on either kernel.  The
    device fill of constant plaintexts matches the host generator."""
    wl = W.make_workload("bert-const", N=2048, L=2)
    dl = DeviceLayer(wl, host_inputs=False)
    torch.cuda.synchronize()
    n_pt, L, N = wl.plan.n_pt, wl.L, wl.N
    pts = dl.d_pt.view(n_pt, L, N)
    k = np.array([0, 1, 17, N - 1])
    for p in (0, wl.const_pts - 1, wl.const_pts):
        assert np.array_equal(to_host(pts[p, 1].contiguous())[k], wl.plaintext_values(p, 1, k))
    want = {}
    for kernel in ("direct", "tiled"):
        dl.plan.select_kernel(kernel)
        dl.run()
        want[kernel] = dl.outputs().copy()
    assert np.array_equal(want["direct"], want["tiled"])
    pts[: wl.const_pts, :, 1:] = -1  # residues that are no residue at all
    for kernel in ("direct", "tiled"):
        dl.plan.select_kernel(kernel)
        dl.d_out.fill_(-1)
        dl.run()
        assert np.array_equal(dl.outputs(), want[kernel]), kernel


def test_host_buffer_path_matches_device_path():
    wl = W.make_workload("vit", N=4096, L=5)
    dl = DeviceLayer(wl)
    dl.run()
    want = dl.outputs()
    h_in = torch.from_numpy(dl.X.view(np.int64)).pin_memory()
    h_out = torch.zeros(want.size, dtype=torch.int64).pin_memory()
    d_in2 = torch.zeros_like(dl.d_in)
    d_out2 = torch.zeros_like(dl.d_out)
    dl.plan.eval_host(h_in, dl.d_pt, h_out, d_in2, d_out2)
    assert np.array_equal(h_out.numpy().view(np.uint64).reshape(want.shape), want)


def test_host_buffer_queries_queued_back_to_back():
    """fiona_linear_eval_host_async: three queries with different inputs,
    queued back to back on the same device buffers (each limb chunk of a
    query ordered after the previous query's kernel and output copy of that
    chunk), into three host outputs: after one synchronisation every output
    equals the device path's result for its own inputs."""
    wl = W.make_workload("vit", N=4096, L=5)
    dl = DeviceLayer(wl)
    p = wl.plan
    rng = np.random.default_rng(11)
    qs = np.asarray(wl.moduli, dtype=np.uint64)
    wants, h_ins, h_outs = [], [], []
    for k in range(3):
        X = (rng.integers(0, 2**62, dl.X.shape, dtype=np.uint64) % qs[None, None, :, None]).astype(np.uint64)
        d_x = torch.from_numpy(X.view(np.int64).reshape(-1)).cuda()
        dl.d_out.fill_(-1)
        dl.plan.eval(d_x, dl.d_pt, dl.d_out)
        wants.append(dl.outputs().copy())
        h_ins.append(torch.from_numpy(X.view(np.int64).reshape(-1)).pin_memory())
        h_outs.append(torch.full((wants[-1].size,), -1, dtype=torch.int64).pin_memory())
    d_in2 = torch.zeros_like(dl.d_in)
    d_out2 = torch.zeros_like(dl.d_out)
    stream = torch.cuda.Stream()
    for k in range(3):
        dl.plan.eval_host_async(h_ins[k], dl.d_pt, h_outs[k], d_in2, d_out2, stream=stream)
    dl.plan.eval_host_join(stream=stream)
    stream.synchronize()
    for k in range(3):
        got = h_outs[k].numpy().view(np.uint64).reshape(wants[k].shape)
        assert np.array_equal(got, wants[k]), k
    assert dl.ctx.device_check() == F.FIONA_OK


def test_stream_and_alignment_errors():
    wl = W.make_workload("tiny")
    dl = DeviceLayer(wl)
    s = torch.cuda.Stream()
    dl.d_out.fill_(0)
    dl.run(stream=s)
    s.synchronize()
    assert np.array_equal(dl.outputs(), oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P))
    # misaligned pointers are refused before any launch
    assert dl.plan.eval_status(dl.d_in.data_ptr() + 8, dl.d_pt, dl.d_out) == F.FIONA_ERR_ARG


def test_check_residues_detects_out_of_range():
    wl = W.make_workload("tiny")
    dl = DeviceLayer(wl)
    assert dl.ctx.check_residues(dl.d_in, 2 * wl.plan.n_in) == F.FIONA_OK
    X = dl.X.copy()
    X[3, 1, 2, 77] = wl.moduli[2]  # residue == q
    dl.d_in.copy_(to_device(X))
    assert dl.ctx.check_residues(dl.d_in, 2 * wl.plan.n_in) == F.FIONA_ERR_RANGE


def test_mul_roof_measures_the_product_rate():
    """fiona_mul_roof returns the whole GPU's product-accumulate rates: both
    positive, within a plausible range for 152 SMs, and the radix-2^26
    Karatsuba form (three 32-bit products) faster than the 64x64 -> 128 one
    (four and a carry chain)."""
    r = F.mul_roof()
    assert 1e11 < r["wide"] < r["narrow"] < 1e14


@pytest.mark.parametrize("bits,L", [(50, 3), (59, 2)])
def test_largest_ring_dimension(bits, L):
    """The tiny layer (8 inputs, 4 outputs, signed, raw and DAG-free) at the
    largest ring dimension the context accepts, N = 2^17, on both kernels,
    narrow (50-bit) and wide (59-bit) arithmetic: element by element."""
    N = 1 << 17
    qs = W.ntt_primes(N, bits, L)
    base = W.make_workload("tiny")
    wl = W.Workload("tiny-2^17", N, qs, base.plan, base.seed + bits)
    dl = DeviceLayer(wl)
    want = oracle.linear_eval(base.plan, qs, dl.X, dl.P)
    for kernel in ("direct", "tiled"):
        dl.plan.select_kernel(kernel)
        dl.d_out.fill_(-1)
        dl.run()
        assert np.array_equal(dl.outputs(), want), kernel


@pytest.mark.parametrize("name,N,L,shape", [("tiny-dag", None, None, "2,1,1"), ("tiny-dag", None, None, "1,2,0"),
                                            ("worked-example", None, None, "2,1,1"),
                                            ("vit", 2048, 2, "2,4,1"), ("vit", 2048, 2, "1,4,1,-1,16"),
                                            ("bert", 1024, 1, "2,8,1"), ("bert", 1024, 1, None),
                                            ("overflow60", None, None, "2,2,1")])
def test_warp_formed_sums(name, N, L, shape, monkeypatch):
    """Shared signed sums formed once per tile by the warp whose outputs use
    them (Sec. 4.2 "Sharing Signed Sums"), read back from the warp's slots:
    the plan reports them formed and every residue equals the oracle's."""
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    wl = W.make_workload(name, N=N, L=L)
    dl = DeviceLayer(wl)
    dl.plan.select_kernel("tiled")
    st = dl.plan.stats()
    if name != "overflow60":
        assert st["nodes_materialized"] > 0, st
    want = oracle.linear_eval(wl.plan, wl.moduli, dl.X, dl.P)
    for _ in range(2):
        dl.run()
        mism = np.argwhere(dl.outputs() != want)
        assert mism.shape[0] == 0, "first mismatches (j, c, l, k): %s" % mism[:5].tolist()
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("kernel", ["direct", "tiled"])
@pytest.mark.parametrize("name,N,L,kind,n_class", [("tiny", None, None, "routes", 2),
                                                   ("tiny-dag", None, None, "random", 3),
                                                   ("vit", 2048, 2, "random", 2),
                                                   ("bert-const", 1024, 1, "routes", 2)])
def test_scale_class_parity(name, N, L, kind, n_class, kernel):
    """Plaintexts at several scales (fiona_plan_create_classes): every
    (output, class) result [n_out][n_class][2][L][N] equals the oracle's."""
    wl = W.make_workload(name, N=N, L=L)
    cls = W.scale_classes(wl.plan, n_class, kind, seed=5)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan, pt_class=cls, n_class=n_class)
    plan.select_kernel(kernel)
    X, P = wl.host_inputs(), wl.host_plaintexts()
    p = wl.plan
    d_out = torch.full((p.n_out * n_class * 2 * wl.L * wl.N,), -1, dtype=torch.int64, device="cuda")
    plan.eval(to_device(X), to_device(P), d_out)
    torch.cuda.synchronize()
    got = to_host(d_out).reshape(p.n_out, n_class, 2, wl.L, wl.N)
    want = oracle.linear_eval_classes(p, wl.moduli, cls, n_class, X, P)
    mism = np.argwhere(got != want)
    assert mism.shape[0] == 0, "first mismatches (j, s, c, l, k): %s" % mism[:5].tolist()
    assert ctx.device_check() == F.FIONA_OK
