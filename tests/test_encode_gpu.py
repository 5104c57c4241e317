"""GPU plaintext encoding (fiona_ckks_embed, fiona_encode_coeffs,
fiona_encode; Sec. 2.2 "Ciphertexts and Slots") against the encoding
oracle (pinned in test_encode_oracle.py).

fiona_encode_coeffs is integer arithmetic: bit-exact.  fiona_ckks_embed is
fp64: its transform's rounding error is about log2(N) * 2^-53 relative to the
coefficients' scale, below 2e-3 of a unit at Delta = 2^40 and |z| <= 1, so a
coefficient can differ from the oracle's by one only where Delta * m_i lies
that close to a half-integer: every difference must be at most 1, and at most
1% of the coefficients may differ.  Independently of the oracle, decoding
the GPU's coefficients must return the slots within N / (2 Delta)."""
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


def random_slots(seed, count, N, real=False):
    rng = np.random.default_rng(seed)
    re = rng.uniform(-1, 1, (count, N // 2))
    im = np.zeros_like(re) if real else rng.uniform(-1, 1, (count, N // 2))
    return np.ascontiguousarray(np.stack([re, im], axis=-1))  # [count][N/2][2]


def gpu_embed(ctx, slots, scale):
    count, n, _ = slots.shape
    N = 2 * n
    d_s = torch.from_numpy(slots.copy()).cuda()
    d_c = torch.full((count * N,), 7, dtype=torch.int64, device="cuda")
    d_w = torch.empty(count * N * 2, dtype=torch.float64, device="cuda")
    ctx.ckks_embed(count, d_s, scale, d_c, d_w)
    torch.cuda.synchronize()
    return d_c.cpu().numpy().reshape(count, N)


def decode(c, N, scale):
    e = np.array([pow(5, j, 2 * N) for j in range(N // 2)])
    # c(zeta^e) for every e at once: an inverse FFT of length 2N
    vals = np.fft.ifft(np.concatenate([c.astype(np.float64), np.zeros(N)])) * (2 * N)
    return vals[e] / scale


@pytest.mark.parametrize("N,count,real", [(1024, 3, False), (2048, 2, True), (4096, 2, False), (8192, 1, False)])
def test_embed_against_the_oracle(N, count, real):
    qs = W.ntt_primes(N, 50, 2)
    ctx = F.Context(N, qs, device=0)
    slots = random_slots(N, count, N, real)
    scale = 2.0 ** 40
    got = gpu_embed(ctx, slots, scale)
    for p in range(count):
        want = oracle.ckks_embed(slots[p, :, 0] + 1j * slots[p, :, 1], scale)
        d = np.abs(got[p] - want)
        assert d.max() <= 1 and np.count_nonzero(d) <= N // 100, (p, d.max(), np.count_nonzero(d))
        err = np.max(np.abs(decode(got[p], N, scale) - (slots[p, :, 0] + 1j * slots[p, :, 1])))
        assert err <= N / (2 * scale) + 1e-9
    assert ctx.device_check() == F.FIONA_OK


@pytest.mark.parametrize("N", [1 << 16, 1 << 17])
def test_embed_full_size_sampled(N):
    """N = 2^16 and 2^17: the oracle at 512 sampled coefficients, decoding
    everywhere."""
    ctx = F.Context(N, W.ntt_primes(N, 50, 2), device=0)
    slots = random_slots(5, 2, N)
    scale = 2.0 ** 40
    got = gpu_embed(ctx, slots, scale)
    idx = np.random.default_rng(1).choice(N, 512, replace=False).astype(np.uint32)
    for p in range(2):
        z = slots[p, :, 0] + 1j * slots[p, :, 1]
        d = np.abs(got[p, idx] - oracle.ckks_embed(z, scale, idx))
        assert d.max() <= 1 and np.count_nonzero(d) <= 5
        assert np.max(np.abs(decode(got[p], N, scale) - z)) <= N / (2 * scale) + 1e-9


def test_embed_closed_forms():
    """Constant slots -> constant poly; monomial slots -> Delta X^t."""
    N = 4096
    ctx = F.Context(N, W.ntt_primes(N, 50, 2), device=0)
    s = np.zeros((2, N // 2, 2))
    s[0, :, 0] = 0.625
    t = 1234
    e = np.array([pow(5, j, 2 * N) * t % (2 * N) for j in range(N // 2)])
    s[1, :, 0], s[1, :, 1] = np.cos(np.pi * e / N), np.sin(np.pi * e / N)
    got = gpu_embed(ctx, s, 2.0 ** 40)
    want0 = np.zeros(N, np.int64)
    want0[0] = round(0.625 * 2 ** 40)
    want1 = np.zeros(N, np.int64)
    want1[t] = 2 ** 40
    assert np.abs(got[0] - want0).max() <= 1 and np.abs(got[1] - want1).max() <= 1


def random_coeffs(seed, count, N):
    rng = np.random.default_rng(seed)
    c = rng.integers(-2 ** 62, 2 ** 62, size=(count, N), dtype=np.int64)
    c[0, :6] = [np.iinfo(np.int64).min, np.iinfo(np.int64).max, -1, 0, 1, -(2 ** 62)]
    return c


@pytest.mark.parametrize("N,L,bits,count", [(1024, 3, 50, 3), (2048, 2, 60, 2), (8192, 3, 40, 2),
                                            (65536, 12, 50, 2), (131072, 2, 59, 1)])
def test_encode_coeffs_parity(N, L, bits, count):
    qs = W.ntt_primes(N, bits, L)
    ctx = F.Context(N, qs, device=0)
    c = random_coeffs(N + L, count, N)
    d_o = torch.full((count * L * N,), -1, dtype=torch.int64, device="cuda")
    ctx.encode_coeffs(L, count, torch.from_numpy(c).cuda(), d_o)
    torch.cuda.synchronize()
    got = to_host(d_o).reshape(count, L, N)
    assert np.array_equal(got, oracle.encode_coeffs(qs, c))


def test_encode_coeffs_lower_level_and_definition():
    N, L = 1024, 5
    qs = W.ntt_primes(N, 45, L)
    ctx = F.Context(N, qs, device=0)
    c = random_coeffs(3, 2, N)
    for Lc in (1, 3):
        d_o = torch.empty(2 * Lc * N, dtype=torch.int64, device="cuda")
        ctx.encode_coeffs(Lc, 2, torch.from_numpy(c).cuda(), d_o)
        torch.cuda.synchronize()
        assert np.array_equal(to_host(d_o).reshape(2, Lc, N), oracle.encode_coeffs(qs[:Lc], c, fast=False))


def test_encode_is_embed_then_encode_coeffs():
    N, L, count = 4096, 3, 3
    qs = W.ntt_primes(N, 50, L)
    ctx = F.Context(N, qs, device=0)
    slots = random_slots(8, count, N, real=True)
    d_s = torch.from_numpy(slots).cuda()
    c = torch.empty(count * N, dtype=torch.int64, device="cuda")
    w = torch.empty(count * N * 2, dtype=torch.float64, device="cuda")
    out = torch.empty(count * L * N, dtype=torch.int64, device="cuda")
    ctx.encode(L, count, d_s, 2.0 ** 40, c, w, out)
    c2 = torch.empty_like(c)
    out2 = torch.empty_like(out)
    ctx.ckks_embed(count, d_s, 2.0 ** 40, c2, w)
    ctx.encode_coeffs(L, count, c2, out2)
    torch.cuda.synchronize()
    assert torch.equal(c, c2) and torch.equal(out, out2)


def test_encode_errors():
    N = 1024
    qs = W.ntt_primes(N, 50, 2)
    ctx = F.Context(N, qs, device=0)
    s = torch.zeros(N, dtype=torch.float64, device="cuda")
    c = torch.empty(N, dtype=torch.int64, device="cuda")
    w = torch.empty(2 * N, dtype=torch.float64, device="cuda")
    assert ctx.ckks_embed_status(1, s, 0.0, c, w) == F.FIONA_ERR_ARG
    assert ctx.ckks_embed_status(1, s, float("nan"), c, w) == F.FIONA_ERR_ARG
    assert ctx.ckks_embed_status(1, s, 2.0 ** 40, c, s) == F.FIONA_ERR_ARG   # work overlaps the slots
    assert ctx.encode_coeffs_status(0, 1, c, w) == F.FIONA_ERR_ARG
    assert ctx.encode_coeffs_status(3, 1, c, w) == F.FIONA_ERR_ARG
    assert ctx.ckks_embed_status(0, None, 2.0 ** 40, None, None) == F.FIONA_OK
    # a coefficient beyond 2^62: written as 0 and reported once
    big = torch.full((N,), 1e30, dtype=torch.float64, device="cuda")
    ctx.ckks_embed(1, big, 2.0 ** 40, c, w)
    assert ctx.device_check() == F.FIONA_ERR_RANGE
    assert int(c.abs().max()) == 0
    assert ctx.device_check() == F.FIONA_OK
