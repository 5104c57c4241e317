"""Pins of the encoding oracle (oracle/encode.c), CPU only.

- closed forms: a constant slot vector encodes to a constant poly; the slot
  vector of a monomial X^t (z_j = zeta^(5^j t)) encodes to Delta X^t;
- an independent encoder (oracle/ckks_tiny.py: Python complex arithmetic,
  its own tables) gives the same integer coefficients;
- decoding (evaluation at zeta^(5^j), written here with numpy) returns the
  slots within the rounding bound N / (2 Delta);
- NTT form: X^t maps to psi^((2 brv(k) + 1) t) (closed form), a negative
  constant -c to q - c everywhere, and the radix-2 path equals the
  definition path (the transforms themselves are pinned in
  test_rescale_oracle.py).
"""
import cmath
import math

import numpy as np
import pytest

import oracle
from oracle.ckks_tiny import TinyCKKS
from paper_2609_35352_gb300 import workloads as W


@pytest.fixture(scope="module", autouse=True)
def built():
    oracle.build()


def slots_of_monomial(N, t):
    return np.array([cmath.exp(1j * math.pi * (pow(5, j, 2 * N) * t % (2 * N)) / N) for j in range(N // 2)])


def decode(c, N, scale):
    """Slots of the integer poly c: c(zeta^(5^j)) / scale."""
    e = np.array([pow(5, j, 2 * N) for j in range(N // 2)])
    i = np.arange(N)
    zeta = np.exp(1j * np.pi * np.outer(e, i) / N)
    return zeta @ c.astype(np.float64) / scale


@pytest.mark.parametrize("N", [16, 256, 4096])
def test_constant_slots_encode_to_a_constant(N):
    for c in (0.75, -1.25, 3.0):
        got = oracle.ckks_embed(np.full(N // 2, c + 0j), 2 ** 30)
        want = np.zeros(N, np.int64)
        want[0] = round(c * 2 ** 30)
        assert np.array_equal(got, want), c


@pytest.mark.parametrize("N", [16, 512])
def test_monomial_slots_encode_to_the_monomial(N):
    for t in (0, 1, N // 2 - 1, N - 1):
        got = oracle.ckks_embed(slots_of_monomial(N, t), 2 ** 40)
        want = np.zeros(N, np.int64)
        want[t] = 2 ** 40
        assert np.array_equal(got, want), t


def test_independent_encoder_agrees():
    N = 32
    ck = TinyCKKS(N, W.ntt_primes(N, 40, 1), 30, seed=3)
    rng = np.random.default_rng(4)
    for _ in range(3):
        z = rng.uniform(-1, 1, N // 2)
        assert np.array_equal(oracle.ckks_embed(z.astype(np.complex128), 2 ** 30),
                              np.array(ck.encode(list(z), 2 ** 30), np.int64))


@pytest.mark.parametrize("N,bits", [(64, 30), (1024, 40)])
def test_decode_round_trip(N, bits):
    rng = np.random.default_rng(N)
    z = rng.uniform(-1, 1, N // 2) + 1j * rng.uniform(-1, 1, N // 2)
    scale = 2.0 ** bits
    c = oracle.ckks_embed(z, scale)
    err = np.max(np.abs(decode(c, N, scale) - z))
    assert err <= N / (2 * scale) + 1e-9, err


def test_sampled_coefficients_equal_the_full_encoding():
    N = 256
    z = np.random.default_rng(9).uniform(-1, 1, N // 2) + 0j
    full = oracle.ckks_embed(z, 2 ** 40)
    idx = np.array([255, 0, 17, 128], np.uint32)
    assert np.array_equal(oracle.ckks_embed(z, 2 ** 40, idx), full[idx])


def brv(k, bits):
    return int(format(k, "0%db" % bits)[::-1], 2)


@pytest.mark.parametrize("fast", [True, False])
def test_encode_coeffs_closed_forms(fast):
    N, L = 32, 3
    qs = W.ntt_primes(N, 50, L)
    bits = 5
    for t in (0, 1, 7, N - 1):
        c = np.zeros(N, np.int64)
        c[t] = 1
        got = oracle.encode_coeffs(qs, c, fast=fast)[0]
        for l, q in enumerate(qs):
            psi = oracle.min_root(q, N)
            want = [pow(psi, (2 * brv(k, bits) + 1) * t, q) for k in range(N)]
            assert got[l].tolist() == want, (t, l)
    c = np.zeros(N, np.int64)
    c[0] = -5
    got = oracle.encode_coeffs(qs, c, fast=fast)[0]
    for l, q in enumerate(qs):
        assert np.all(got[l] == np.uint64(q - 5))


def test_encode_coeffs_fast_equals_definition_and_handles_extremes():
    N, L = 64, 2
    qs = W.ntt_primes(N, 60, L)
    rng = np.random.default_rng(2)
    c = rng.integers(-2 ** 62, 2 ** 62, size=(2, N), dtype=np.int64)
    c[0, :4] = [np.iinfo(np.int64).min, np.iinfo(np.int64).max, -1, 0]
    a = oracle.encode_coeffs(qs, c, fast=True)
    b = oracle.encode_coeffs(qs, c, fast=False)
    assert np.array_equal(a, b)
    # residues of the extremes, by Python integers, through the inverse transform
    for l, q in enumerate(qs):
        r = oracle.intt(a[0, l], q)
        assert [int(x) for x in r[:4]] == [int(v) % q for v in c[0, :4]]
