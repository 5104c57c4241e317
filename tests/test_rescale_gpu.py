"""GPU parity of the rescale after the layer (fiona_rescale,
fiona_linear_eval_rescale; Sec. 2.2 rescale, Sec. 4.2 one rescale per
combined output) against the oracle's radix-2 NTT path, which
test_rescale_oracle.py pins to the transform's definition, the CRT and exact
division.  The bar is bit-exact equality of every residue."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402

from gpu_util import to_device, to_host  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    oracle.build()


def random_polys(seed, qs, count, N, fill="uniform"):
    """[count][L][N] residues, limb l uniform in [0, q_l) (or all q_l - 1)."""
    L = len(qs)
    q = np.asarray(qs, np.uint64).reshape(1, L, 1)
    if fill == "max":
        return np.broadcast_to(q - np.uint64(1), (count, L, N)).copy()
    flat = np.arange(count * L * N, dtype=np.uint64).reshape(count, L, N)
    return W.residues_np(W.stream_key(seed, W.STREAM_INPUTS), flat, q)


def gpu_rescale(ctx, y, L_cur):
    count, L, N = y.shape
    d_y = to_device(y)
    d_out = torch.full((max(count * (L_cur - 1) * N, 2),), -1, dtype=torch.int64, device="cuda")
    ctx.rescale(L_cur, count, d_y, d_out)
    torch.cuda.synchronize()
    return to_host(d_out)[: count * (L_cur - 1) * N].reshape(count, L_cur - 1, N), \
        to_host(d_y).reshape(count, L, N)


# (N, L, prime bits, polys): one tile per transform (N <= 4096), several
# tiles with R1 = R2 and R1 < R2 (odd log2 N), the largest N the ctx takes,
# 60-bit primes (the ctx's bound) and small ones
CASES = [
    (1024, 3, 50, 3),
    (1024, 2, 20, 5),
    (2048, 4, 60, 2),
    (4096, 3, 40, 2),
    (8192, 3, 50, 2),
    (32768, 4, 59, 1),
    (65536, 5, 50, 2),
    (131072, 3, 50, 1),
]


@pytest.mark.parametrize("N,L,bits,count", CASES)
def test_rescale_parity(N, L, bits, count):
    qs = W.ntt_primes(N, bits, L)
    y = random_polys(N + L + bits, qs, count, N)
    ctx = F.Context(N, qs, device=0)
    got, y_after = gpu_rescale(ctx, y, L)
    want = oracle.rescale(qs, y)
    mism = np.argwhere(got != want)
    assert mism.shape[0] == 0, "first mismatches (poly, limb, k): %s" % mism[:5].tolist()
    # the last limb now holds its coefficients; the other limbs are untouched
    assert np.array_equal(y_after[:, : L - 1], y[:, : L - 1])
    for p in range(count):
        assert np.array_equal(y_after[p, L - 1], oracle.intt(y[p, L - 1], qs[L - 1]))


def test_rescale_matches_the_definition():
    """Against the oracle's O(N^2) transforms, not only its radix-2 ones."""
    N, L = 1024, 3
    qs = W.ntt_primes(N, 45, L)
    y = random_polys(11, qs, 2, N)
    ctx = F.Context(N, qs, device=0)
    got, _ = gpu_rescale(ctx, y, L)
    assert np.array_equal(got, oracle.rescale(qs, y, fast=False))


def test_rescale_extreme_residues():
    """Every residue q_l - 1: the largest operands of each butterfly."""
    N, L = 4096, 4
    qs = W.ntt_primes(N, 60, L)
    y = random_polys(0, qs, 2, N, fill="max")
    ctx = F.Context(N, qs, device=0)
    got, _ = gpu_rescale(ctx, y, L)
    assert np.array_equal(got, oracle.rescale(qs, y))


def test_rescale_lower_levels():
    """L_cur < L: buffers of L_cur limbs, division by q_{L_cur - 1}."""
    N, L = 2048, 6
    qs = W.ntt_primes(N, 50, L)
    ctx = F.Context(N, qs, device=0)
    for Lc in (2, 3, 5, 6):
        y = random_polys(Lc, qs[:Lc], 3, N)
        got, _ = gpu_rescale(ctx, y, Lc)
        assert np.array_equal(got, oracle.rescale(qs[:Lc], y)), Lc


def test_rescale_arguments():
    N, L = 1024, 3
    qs = W.ntt_primes(N, 50, L)
    ctx = F.Context(N, qs, device=0)
    buf = torch.zeros(4 * L * N, dtype=torch.int64, device="cuda")
    out = torch.zeros(4 * L * N, dtype=torch.int64, device="cuda")
    assert ctx.rescale_status(1, 1, buf, out) == F.FIONA_ERR_ARG
    assert ctx.rescale_status(L + 1, 1, buf, out) == F.FIONA_ERR_ARG
    assert ctx.rescale_status(L, 1, buf, buf[(L - 1) * N:]) == F.FIONA_ERR_ARG  # overlap
    assert ctx.rescale_status(L, 1, buf[N:], buf) == F.FIONA_ERR_ARG          # overlap
    assert ctx.rescale_status(L, 1, buf, buf[L * N:]) == F.FIONA_OK           # adjacent
    assert ctx.rescale_status(L, 1, None, out) == F.FIONA_ERR_ARG
    assert ctx.rescale_status(L, 0, None, None) == F.FIONA_OK
    torch.cuda.synchronize()


def test_rescale_full_size_sampled():
    """N = 2^16, L = 24, 192 polys (the BERT layer's 96 outputs, c0 and c1)
    filled on the device by the seeded generator; three polys regenerated on
    the host and rescaled by the oracle."""
    N, L, count = 1 << 16, 24, 192
    qs = W.ntt_primes(N, 50, L)
    ctx = F.Context(N, qs, device=0)
    key = W.stream_key(31, W.STREAM_INPUTS)
    d_y = torch.empty(count * L * N, dtype=torch.int64, device="cuda")
    F.device_fill(d_y, count, L, N, qs, key)
    d_out = torch.full((count * (L - 1) * N,), -1, dtype=torch.int64, device="cuda")
    ctx.rescale(L, count, d_y, d_out)
    torch.cuda.synchronize()
    q = np.asarray(qs, np.uint64).reshape(L, 1)
    for p in (0, 97, count - 1):
        flat = (np.uint64(p * L * N) + np.arange(L * N, dtype=np.uint64)).reshape(L, N)
        y = W.residues_np(key, flat, q).reshape(1, L, N)
        got = to_host(d_out[p * (L - 1) * N:(p + 1) * (L - 1) * N]).reshape(1, L - 1, N)
        assert np.array_equal(got, oracle.rescale(qs, y)), p
    del d_y, d_out


@pytest.mark.parametrize("name,N,L,kernel", [("vit", 2048, 3, "tiled"), ("wsum-hybrid", 2048, 3, "direct"),
                                             ("worked-example", None, None, "tiled")])
def test_eval_rescale_parity(name, N, L, kernel):
    """fiona_linear_eval_rescale at every level >= 2: the layer (oracle
    linear_eval) followed by the rescale (oracle rescale)."""
    wl = W.make_workload(name, N=N, L=L)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan)
    plan.select_kernel(kernel)
    p = wl.plan
    X, P = wl.host_inputs(), wl.host_plaintexts()
    for Le in range(2, wl.L + 1):
        Xl = np.ascontiguousarray(X[:, :, :Le, :])
        Pl = np.ascontiguousarray(P[:, :Le, :])
        work = torch.empty(p.n_out * 2 * Le * wl.N, dtype=torch.int64, device="cuda")
        out = torch.full((p.n_out * 2 * (Le - 1) * wl.N,), -1, dtype=torch.int64, device="cuda")
        plan.eval_rescale(Le, to_device(Xl), to_device(Pl), work, out)
        torch.cuda.synchronize()
        got = to_host(out).reshape(p.n_out * 2, Le - 1, wl.N)
        layer = oracle.linear_eval(p, wl.moduli[:Le], Xl, Pl).reshape(p.n_out * 2, Le, wl.N)
        want = oracle.rescale(wl.moduli[:Le], layer)
        mism = np.argwhere(got != want)
        assert mism.shape[0] == 0, (Le, mism[:5].tolist())
    assert plan.eval_rescale_status(1, to_device(X), to_device(P), work, out) == F.FIONA_ERR_ARG


@pytest.mark.parametrize("N,L,bits,count", [(1024, 3, 50, 3), (2048, 4, 60, 2), (65536, 5, 50, 2),
                                            (131072, 3, 59, 1)])
def test_rounding_rescale_parity(N, L, bits, count):
    """FIONA_RESCALE_ROUND: the nearest quotient (oracle round=True, pinned by
    brute force); the last limb becomes r' = (r + floor(q_last / 2)) mod q_last."""
    qs = W.ntt_primes(N, bits, L)
    y = random_polys(N + 7 * L + bits, qs, count, N)
    ctx = F.Context(N, qs, device=0)
    d_y = to_device(y)
    d_out = torch.full((count * (L - 1) * N,), -1, dtype=torch.int64, device="cuda")
    ctx.rescale(L, count, d_y, d_out, round=True)
    torch.cuda.synchronize()
    got = to_host(d_out).reshape(count, L - 1, N)
    assert np.array_equal(got, oracle.rescale(qs, y, round=True))
    assert not np.array_equal(got, oracle.rescale(qs, y))
    ql = qs[-1]
    last = to_host(d_y).reshape(count, L, N)[:, L - 1]
    for p in range(count):
        r = oracle.intt(y[p, L - 1], ql)
        assert np.array_equal(last[p], (r + np.uint64(ql // 2)) % np.uint64(ql))
    assert ctx.rescale_status(L, count, d_y, d_out, flags=4) == F.FIONA_ERR_ARG


def test_eval_rescale_rounding():
    wl = W.make_workload("vit", N=2048, L=3)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan)
    p = wl.plan
    X, P = wl.host_inputs(), wl.host_plaintexts()
    work = torch.empty(p.n_out * 2 * wl.L * wl.N, dtype=torch.int64, device="cuda")
    out = torch.empty(p.n_out * 2 * (wl.L - 1) * wl.N, dtype=torch.int64, device="cuda")
    plan.eval_rescale(wl.L, to_device(X), to_device(P), work, out, round=True)
    torch.cuda.synchronize()
    layer = oracle.linear_eval(p, wl.moduli, X, P).reshape(p.n_out * 2, wl.L, wl.N)
    assert np.array_equal(to_host(out).reshape(p.n_out * 2, wl.L - 1, wl.N),
                          oracle.rescale(wl.moduli, layer, round=True))


@pytest.mark.parametrize("shape,tile", [(None, 64), ("1,8,1", 32)])
def test_layer_and_rescale_replay_in_a_cuda_graph(shape, tile, monkeypatch):
    """After a first call (which builds the tables), a layer followed by its
    rescale is stream-ordered launches only: it captures into a CUDA graph and
    every replay gives the oracle's residues -- with input tiles staged by
    cp.async (two coefficients per lane) and by TMA tensor copies, whose
    tensor map is a kernel parameter captured with the launch (one)."""
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    wl = W.make_workload("vit", N=2048, L=3)
    ctx = F.Context(wl.N, wl.moduli, device=0)
    plan = F.Plan(ctx, wl.plan)
    assert plan.stats()["tile_coeffs"] == tile
    p = wl.plan
    X, P = wl.host_inputs(), wl.host_plaintexts()
    d_in, d_pt = to_device(X), to_device(P)
    work = torch.empty(p.n_out * 2 * wl.L * wl.N, dtype=torch.int64, device="cuda")
    out = torch.empty(p.n_out * 2 * (wl.L - 1) * wl.N, dtype=torch.int64, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        plan.eval_rescale(wl.L, d_in, d_pt, work, out, stream=s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        plan.eval_rescale(wl.L, d_in, d_pt, work, out, stream=s)
    layer = oracle.linear_eval(p, wl.moduli, X, P).reshape(p.n_out * 2, wl.L, wl.N)
    want = oracle.rescale(wl.moduli, layer)
    for _ in range(3):
        out.fill_(-1)
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(to_host(out).reshape(p.n_out * 2, wl.L - 1, wl.N), want)
