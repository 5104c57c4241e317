"""The narrow reduction of the tiled kernel's accumulators (rns.cuh
reduce_k), restated in Python integers: for a k-bit modulus q and a value
x < 2^(k+63), A = floor(x / 2^(k-1)) and mk = floor(2^(k+63) / q) give a
quotient estimate floor(A mk / 2^64) at most 2 below floor(x / q), so two
conditional subtractions of q leave x mod q.  Checked on random and extreme
values for moduli of 20 to 52 bits, and on the largest value the kernels
reduce: 1024 products of residues q - 1 (the lazy-product budget)."""
import random

from paper_2609_35352_gb300 import workloads as W


def reduce_k(x: int, q: int) -> int:
    k = q.bit_length()
    mk = (1 << (k + 63)) // q
    A = x >> (k - 1)
    assert A < 1 << 64 and mk < 1 << 64
    qe = (A * mk) >> 64
    r = (x - qe * q) % (1 << 64)  # the device computes it modulo 2^64
    assert r < 3 * q
    if r >= q:
        r -= q
    if r >= q:
        r -= q
    return r


def test_reduce_k_random_and_extremes():
    rng = random.Random(20261202)
    for bits in (20, 30, 40, 45, 50, 51, 52):
        for q in W.ntt_primes(1024, bits, 3):
            k = q.bit_length()
            top = (1 << (k + 63)) - 1
            cases = [0, 1, q - 1, q, top, top - 1, 1024 * (q - 1) ** 2, (q - 1) ** 2]
            cases += [rng.randrange(top + 1) for _ in range(2000)]
            cases += [rng.randrange(1 << 64) for _ in range(200)]
            for x in cases:
                assert reduce_k(x, q) == x % q, (q, x)


def test_largest_accumulated_value_is_in_range():
    # at most 1023 products between reductions (a fold adds a residue below q)
    for bits in (40, 50, 52):
        for q in W.ntt_primes(1024, bits, 2):
            x = 1023 * (q - 1) ** 2 + (q - 1)
            assert x < 1 << (q.bit_length() + 63)
            assert reduce_k(x, q) == x % q
