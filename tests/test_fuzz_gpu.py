"""Randomised parity: many small random layers and rescales, each against the
oracle, bit-exact.  Layers: random sizes, route mixes (raw, constant raw,
ternary with zeros), one or several reconstruction factors per output,
shared sums from the plan compiler (both acceptance rules), 40- to 60-bit
primes, N of 2^10 or 2^11, both kernels and a random tiled shape.  Rescales:
random N, level, poly count and quotient rounding."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402

from gpu_util import DeviceLayer, to_device, to_host  # noqa: E402

SHAPES = [None, "2,16,0", "2,8,1", "1,16,1", "1,4,0", "2,8,1,-1,4", "1,8,0,3"]


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    oracle.build()


def random_layer(rng):
    n_in, n_out = int(rng.integers(1, 40)), int(rng.integers(1, 20))
    n_gamma = int(rng.integers(1, 3))
    p_raw, p_const, p_zero = rng.uniform(0, 0.6), rng.uniform(0, 0.3), rng.uniform(0, 0.2)
    r = np.zeros((n_out, n_in), F.ROUTE_DTYPE)
    n_raw = 0
    for j in range(n_out):
        for i in range(n_in):
            u = rng.random()
            if u < p_raw:
                kind = W.TERM_RAW_CONST if rng.random() < p_const else W.TERM_RAW
                r[j, i] = (kind, 0, 0, n_gamma * n_out + n_raw)
                n_raw += 1
            else:
                t = 0 if rng.random() < p_zero else int(rng.choice([-1, 1]))
                r[j, i] = (W.TERM_TERNARY, t, 0, j * n_gamma + int(rng.integers(n_gamma)))
    exact = bool(rng.integers(2))
    return F.compile_plan(n_in, n_out, n_gamma * n_out + n_raw, r, share=bool(rng.integers(4)), exact=exact)


@pytest.mark.parametrize("seed", range(40))
def test_random_layers(seed, monkeypatch):
    rng = np.random.default_rng(1000 + seed)
    shape = SHAPES[seed % len(SHAPES)]
    if shape:
        monkeypatch.setenv("FIONA_TILED_SHAPE", shape)
    desc = random_layer(rng)
    N = int(rng.choice([1024, 2048]))
    bits = int(rng.choice([40, 50, 59]))
    L = int(rng.integers(1, 4))
    wl = W.Workload("fuzz", N, W.ntt_primes(N, bits, L), desc, 5000 + seed)
    dl = DeviceLayer(wl)
    want = oracle.linear_eval(desc, wl.moduli, dl.X, dl.P)
    kernels = ["direct"]
    try:
        dl.plan.select_kernel("tiled")
        kernels.append("tiled")
    except F.FionaError:
        assert shape is not None  # only a forced shape may not fit the layer
    for kernel in kernels:
        dl.plan.select_kernel(kernel)
        dl.d_out.fill_(-1)
        dl.run()
        got = dl.outputs()
        mism = np.argwhere(got != want)
        assert mism.shape[0] == 0, (seed, kernel, shape, mism[:5].tolist())
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("seed", range(24))
def test_random_layers_tensor_core_sums(seed, monkeypatch):
    """Random compiled layers (shared sums expanded into the groups, so the
    weights are small integers, not only +-1), 40- and 50-bit primes, one
    coefficient per lane, 4, 8 or 16 warps: the signed sums on the tensor
    cores against the oracle, bit-exact, where the plan takes them."""
    rng = np.random.default_rng(3000 + seed)
    monkeypatch.setenv("FIONA_TILED_TC", "1")
    monkeypatch.setenv("FIONA_TILED_SHAPE", ["1,4,1,-1,16", "1,8,0,-1,16", "1,16,1,-1,16"][seed % 3])
    desc = random_layer(rng)
    N = int(rng.choice([1024, 2048]))
    bits = int(rng.choice([40, 50]))
    L = int(rng.integers(1, 4))
    wl = W.Workload("fuzz-tc", N, W.ntt_primes(N, bits, L), desc, 7000 + seed)
    dl = DeviceLayer(wl)
    try:
        dl.plan.select_kernel("tiled")
    except F.FionaError:
        pytest.skip("the forced shape does not fit this layer")
    if dl.plan.stats()["tensor_core_sums"] == 0:
        pytest.skip("no signed sums, or more groups than tensor memory holds")
    want = oracle.linear_eval(desc, wl.moduli, dl.X, dl.P)
    dl.run()
    mism = np.argwhere(dl.outputs() != want)
    assert mism.shape[0] == 0, (seed, mism[:5].tolist())
    assert dl.ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("seed", range(16))
def test_random_rescales(seed):
    rng = np.random.default_rng(2000 + seed)
    N = int(rng.choice([1024, 2048, 4096, 16384]))
    L = int(rng.integers(2, 7))
    Lc = int(rng.integers(2, L + 1))
    bits = int(rng.choice([30, 45, 55, 59]))
    count = int(rng.integers(1, 5))
    rnd = bool(rng.integers(2))
    qs = W.ntt_primes(N, bits, L)
    q = np.asarray(qs[:Lc], np.uint64).reshape(1, Lc, 1)
    flat = np.arange(count * Lc * N, dtype=np.uint64).reshape(count, Lc, N)
    y = W.residues_np(W.stream_key(3000 + seed, W.STREAM_INPUTS), flat, q)
    ctx = F.Context(N, qs, device=0)
    d_y = to_device(y)
    d_o = torch.full((count * (Lc - 1) * N,), -1, dtype=torch.int64, device="cuda")
    ctx.rescale(Lc, count, d_y, d_o, round=rnd)
    torch.cuda.synchronize()
    got = to_host(d_o).reshape(count, Lc - 1, N)
    assert np.array_equal(got, oracle.rescale(qs[:Lc], y, round=rnd)), (seed, N, L, Lc, bits, rnd)
