"""The narrow reduction of the tiled kernel's accumulators (rns.cuh
reduce_k), restated in Python integers: for a k-bit modulus q and a value
x < 2^(k+63), A = floor(x / 2^(k-1)) and mk = floor(2^(k+63) / q) give a
quotient estimate floor(A mk / 2^64) at most 2 below floor(x / q), so two
conditional subtractions of q leave x mod q.  Checked on random and extreme
values for moduli of 20 to 52 bits, and on the largest value the kernels
reduce: 1024 products of residues q - 1 (the lazy-product budget).  The
radix-2^26 product path around it (split form, Karatsuba accumulators, the
middle term recovered at the reduction) and the bounds of the lazy signed
sums are restated with explicit 64-bit words at the widest moduli that path
takes (q < 2^52)."""
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


# -- the whole narrow product path (rns.cuh split26, mac26, reduce26) and the
# -- lazy signed sums (tile_math.cuh), restated with explicit 64-bit words

M64 = (1 << 64) - 1


def split26(a: int) -> int:
    return ((a >> 26) << 32) | (a & 0x3FFFFFF)


def mac26(acc, a_s: int, b_s: int):
    """Three 32x32 -> 64-bit products added to (lo, x, hi); every value a
    device register holds is checked to fit it (no wrap)."""
    a0, a1 = a_s & 0xFFFFFFFF, a_s >> 32
    b0, b1 = b_s & 0xFFFFFFFF, b_s >> 32
    ha, hb = a0 + a1, b0 + b1
    assert ha < 1 << 32 and hb < 1 << 32  # the half sums are 32-bit additions
    lo, x, hi = acc[0] + a0 * b0, acc[1] + ha * hb, acc[2] + a1 * b1
    assert max(lo, x, hi) <= M64
    return [lo, x, hi]


def reduce26(acc, q: int) -> int:
    lo, x, hi = acc
    mid = (x - lo - hi) & M64
    # (x1, x0) = lo + mid * 2^26 + hi * 2^52 as the two carry chains form it
    x0 = lo + ((mid << 26) & M64)
    x1 = (mid >> 38) + (x0 >> 64)
    x0 &= M64
    x0 += (hi << 52) & M64
    x1 += (hi >> 12) + (x0 >> 64)
    x0 &= M64
    assert x1 <= M64
    return reduce_k((x1 << 64) | x0, q)


def test_narrow_products_at_the_widest_moduli():
    """1023 products between reductions (kNarrowMacBudget) after a fold, the
    factors residues q - 1 (the largest half sums) or random, for 50- to
    52-bit moduli: no accumulator wraps and the reduction is exact."""
    rng = random.Random(52)
    for bits in (50, 51, 52):
        for q in W.ntt_primes(1024, bits, 2):
            for fill in ("max", "random"):
                def residue():
                    return q - 1 if fill == "max" else rng.randrange(q)
                r = residue()
                acc = [r, r, 0]  # a folded accumulator: lo = x = r, hi = 0
                want = r
                for _ in range(1023):
                    a, b = residue(), residue()
                    acc = mac26(acc, split26(a), split26(b))
                    want += a * b
                assert reduce26(acc, q) == want % q, (q, fill)


def test_narrow_signed_sums_at_the_widest_moduli():
    """The lazy signed sums of the narrow kernels, for 50- to 52-bit moduli.
    Split sources (two coefficients per lane): a packed sum of at most 64
    split words keeps each 32-bit half from carrying into the other, and
    unsplit(P) + 64 q - unsplit(M) is the exact P - M + 64 q below 2^59.
    Canonical sources (one): runs of at most 64 sources with up to six slot
    tiles, P + 128 q - M positive and below 2^60."""
    for bits in (50, 51, 52):
        for q in W.ntt_primes(1024, bits, 2):
            assert 64 * (2 ** 26 - 1) < 1 << 32  # any 64 digits of 26 bits
            w = split26(q - 1)
            packed = 64 * w
            assert packed <= M64
            assert (packed & 0xFFFFFFFF) == 64 * ((q - 1) & 0x3FFFFFF)  # no carry between halves
            value = (packed & 0xFFFFFFFF) + ((packed >> 32) << 26)
            assert value == 64 * (q - 1) and value + 64 * q < 1 << 59
            for p_terms, m_terms in ((64, 0), (0, 64), (64, 64)):
                v = p_terms * (q - 1) + 64 * q - m_terms * (q - 1)
                assert 0 < v < 1 << 59
            for p_terms, m_terms in ((70, 0), (0, 70), (70, 70)):
                v = p_terms * (q - 1) + 128 * q - m_terms * (q - 1)
                assert 0 < v < 1 << 60
