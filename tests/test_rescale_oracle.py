"""Pins of the rescale oracle (oracle/rescale.c), CPU only.

- psi is a primitive 2N-th root of unity and the least one (checked against
  the odd powers of a root found independently here);
- the radix-2 transforms equal the definitions, and invert each other;
- the negacyclic convolution theorem: pointwise products in NTT form are
  products in Z_q[X]/(X^N + 1) (schoolbook negacyclic convolution here);
- rescale exactness (brute force over Z_Q with Python integers): the
  rescaled residues are those of (Y - (Y mod q_last)) / q_last, Y the CRT
  value of every coefficient.
"""
import numpy as np
import pytest

import oracle
from paper_2609_35352_gb300 import workloads as W


@pytest.fixture(scope="module", autouse=True)
def built():
    oracle.build()


def rand_res(rng, q, n):
    return np.array([int(x) for x in rng.integers(0, q, size=n, dtype=np.uint64)], dtype=np.uint64)


@pytest.mark.parametrize("N,bits", [(16, 40), (64, 40), (256, 50)])
def test_min_root(N, bits):
    for q in W.ntt_primes(N, bits, 2):
        psi = oracle.min_root(q, N)
        assert pow(psi, N, q) == q - 1 and pow(psi, 2 * N, q) == 1
        # an independent root: g = x^((q-1)/2N) for the first x that gives one
        x = 3
        while pow(pow(x, (q - 1) // (2 * N), q), N, q) != q - 1:
            x += 1
        g = pow(x, (q - 1) // (2 * N), q)
        assert psi == min(pow(g, 2 * j + 1, q) for j in range(N))


@pytest.mark.parametrize("N,bits", [(16, 40), (64, 50), (128, 60)])
def test_fast_transforms_equal_definitions(N, bits):
    rng = np.random.default_rng(N)
    for q in W.ntt_primes(N, bits, 2):
        a = rand_res(rng, q, N)
        A = oracle.ntt(a, q, fast=False)
        assert np.array_equal(oracle.ntt(a, q, fast=True), A)
        assert np.array_equal(oracle.intt(A, q, fast=False), a)
        assert np.array_equal(oracle.intt(A, q, fast=True), a)


def negacyclic(a, b, q):
    N = len(a)
    c = [0] * N
    for i in range(N):
        for j in range(N):
            k = i + j
            if k < N:
                c[k] = (c[k] + int(a[i]) * int(b[j])) % q
            else:
                c[k - N] = (c[k - N] - int(a[i]) * int(b[j])) % q
    return np.array(c, dtype=np.uint64)


@pytest.mark.parametrize("N", [8, 32])
def test_convolution_theorem(N):
    rng = np.random.default_rng(5)
    q = W.ntt_primes(N, 40, 1)[0]
    a, b = rand_res(rng, q, N), rand_res(rng, q, N)
    A, B = oracle.ntt(a, q), oracle.ntt(b, q)
    AB = np.array([(int(x) * int(y)) % q for x, y in zip(A, B)], dtype=np.uint64)
    assert np.array_equal(oracle.intt(AB, q), negacyclic(a, b, q))
    # X * X^(N-1) = X^N = -1
    x = np.zeros(N, np.uint64); x[1] = 1
    y = np.zeros(N, np.uint64); y[N - 1] = 1
    XY = np.array([(int(u) * int(v)) % q for u, v in zip(oracle.ntt(x, q), oracle.ntt(y, q))], dtype=np.uint64)
    want = np.zeros(N, np.uint64); want[0] = q - 1
    assert np.array_equal(oracle.intt(XY, q), want)


@pytest.mark.parametrize("fast", [False, True])
def test_rescale_is_exact_division_by_the_last_prime(fast):
    N, L = 16, 4
    qs = W.ntt_primes(N, 40, L)
    rng = np.random.default_rng(11)
    count = 3
    y = np.zeros((count, L, N), np.uint64)
    for p in range(count):
        for l in range(L):
            y[p, l] = rand_res(rng, qs[l], N)
    out = oracle.rescale(qs, y, fast=fast)
    assert out.shape == (count, L - 1, N)
    Q = 1
    for q in qs:
        Q *= q
    for p in range(count):
        coef = [oracle.intt(y[p, l], qs[l]) for l in range(L)]
        rcoef = [oracle.intt(out[p, l], qs[l]) for l in range(L - 1)]
        for k in range(N):
            Y = 0
            for l, q in enumerate(qs):  # CRT
                Ml = Q // q
                Y = (Y + int(coef[l][k]) * Ml * pow(Ml, -1, q)) % Q
            Yp = (Y - Y % qs[-1]) // qs[-1]
            for l in range(L - 1):
                assert int(rcoef[l][k]) == Yp % qs[l], (p, l, k)


def test_rescale_of_a_multiple_of_the_last_prime():
    """Y = q_last * Z: the rescale returns Z exactly (closed form)."""
    N, L = 8, 3
    qs = W.ntt_primes(N, 40, L)
    import random
    rnd = random.Random(3)
    Z = [rnd.randrange(qs[0] * qs[1]) for _ in range(N)]
    coef = [np.array([(qs[-1] * z) % q for z in Z], np.uint64) for q in qs]
    y = np.stack([oracle.ntt(coef[l], qs[l]) for l in range(L)])[None]
    out = oracle.rescale(qs, y)
    for l in range(L - 1):
        assert np.array_equal(oracle.intt(out[0, l], qs[l]), np.array([z % qs[l] for z in Z], np.uint64))


@pytest.mark.parametrize("fast", [False, True])
def test_rounding_rescale_is_the_nearest_quotient(fast):
    """round=True: the residues of floor((Y + h) / q_last), h = floor(q_last / 2),
    i.e. Y / q_last rounded to the nearest integer (brute force over Z_Q)."""
    N, L = 16, 3
    qs = W.ntt_primes(N, 40, L)
    rng = np.random.default_rng(12)
    y = np.zeros((2, L, N), np.uint64)
    for p in range(2):
        for l in range(L):
            y[p, l] = rand_res(rng, qs[l], N)
    out = oracle.rescale(qs, y, fast=fast, round=True)
    Q = 1
    for q in qs:
        Q *= q
    ql = qs[-1]
    for p in range(2):
        coef = [oracle.intt(y[p, l], qs[l]) for l in range(L)]
        rcoef = [oracle.intt(out[p, l], qs[l]) for l in range(L - 1)]
        for k in range(N):
            Y = 0
            for l, q in enumerate(qs):
                Ml = Q // q
                Y = (Y + int(coef[l][k]) * Ml * pow(Ml, -1, q)) % Q
            Yp = (Y + ql // 2) // ql
            assert abs(Yp * ql - Y) <= ql // 2
            for l in range(L - 1):
                assert int(rcoef[l][k]) == Yp % qs[l], (p, l, k)
