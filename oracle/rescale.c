/*
 * rescale.c -- plain CPU oracle for the rescale that follows the linear
 * layer (Sec. 2.2 "Homomorphic Operations": a PMult raises the scale and a
 * rescale divides by the last prime of the modulus chain; Sec. 4.2
 * "Combining the Signed and Raw Routes": one rescale per output).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this code.  It shares no code,
 * header, table or helper with the CUDA path.
 *
 * Conventions (the evaluator follows the same definitions, written
 * separately):
 *   psi_q    the least primitive 2N-th root of unity modulo q (every
 *            primitive 2N-th root is an odd power of any one of them);
 *   NTT form a polynomial a(X) mod (X^N + 1) is held as
 *              A[k] = a(psi^(2 brv(k) + 1)) mod q,  k = 0..N-1,
 *            brv reversing the log2(N) bits of k (the order the radix-2
 *            Cooley-Tukey transform produces);
 *   rescale  for a poly y with limbs y_0..y_{L-1} in NTT form, and
 *            r = the coefficients of y_{L-1} (inverse NTT mod q_{L-1}),
 *            canonical in [0, q_{L-1}):
 *              y'_l = (y_l - NTT_l(r mod q_l)) * q_{L-1}^{-1}  mod q_l,
 *            l = 0..L-2, i.e. y' = (Y - (Y mod q_{L-1})) / q_{L-1} for the
 *            integer Y in [0, Q) whose residues are y (coefficient-wise);
 *   rounding the same with Y + h in place of Y, h = floor(q_{L-1} / 2), so
 *            that y' = floor((Y + h) / q_{L-1}), Y / q_{L-1} rounded: in
 *            coefficient form r' = (r + h) mod q_{L-1} and the subtracted
 *            poly is r' - h (mod q_l).
 *
 * Two transforms: the definition (an O(N^2) sum, for small N) and the
 * textbook radix-2 transform (Cooley-Tukey forward, Gentleman-Sande
 * inverse), which the tests pin to the definition.  Every operation reduced
 * at once with 128-bit '%'.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef unsigned __int128 u128;

static uint64_t mulm(uint64_t a, uint64_t b, uint64_t q) { return (uint64_t)(((u128)a * b) % q); }
static uint64_t addm(uint64_t a, uint64_t b, uint64_t q) { return (uint64_t)(((u128)a + b) % q); }
static uint64_t subm(uint64_t a, uint64_t b, uint64_t q) { return (uint64_t)(((u128)a + q - b) % q); }

static uint64_t powm(uint64_t b, uint64_t e, uint64_t q)
{
    uint64_t r = 1 % q;
    b %= q;
    while (e) {
        if (e & 1) r = mulm(r, b, q);
        b = mulm(b, b, q);
        e >>= 1;
    }
    return r;
}

/* q prime: a^(q-2) */
static uint64_t invm(uint64_t a, uint64_t q) { return powm(a, q - 2, q); }

static uint32_t log2u(uint32_t n)
{
    uint32_t k = 0;
    while ((1u << k) < n) ++k;
    return k;
}

static uint32_t brv(uint32_t k, uint32_t bits)
{
    uint32_t r = 0;
    for (uint32_t b = 0; b < bits; ++b) r |= ((k >> b) & 1u) << (bits - 1 - b);
    return r;
}

/* The least primitive 2N-th root of unity mod q (q = 1 mod 2N, prime), or 0.
 * x^((q-1)/2N) is a 2N-th root of unity; it is primitive iff its N-th power
 * is q-1.  The primitive ones are its odd powers; the least is kept. */
uint64_t oracle_min_root(uint64_t q, uint32_t N)
{
    const uint64_t M = 2ull * N;
    if ((q - 1) % M) return 0;
    uint64_t g = 0;
    for (uint64_t x = 2; x < q && x < 1000000; ++x) {
        const uint64_t c = powm(x, (q - 1) / M, q);
        if (powm(c, N, q) == q - 1) {
            g = c;
            break;
        }
    }
    if (!g) return 0;
    uint64_t best = g;
    const uint64_t g2 = mulm(g, g, q);
    uint64_t cur = g;
    for (uint32_t j = 1; j < N; ++j) {
        cur = mulm(cur, g2, q);
        if (cur < best) best = cur;
    }
    return best;
}

/* NTT by its definition: A[k] = sum_i a_i psi^((2 brv(k) + 1) i). */
void oracle_ntt_direct(const uint64_t *a, uint64_t *A, uint32_t N, uint64_t q, uint64_t psi)
{
    const uint32_t bits = log2u(N);
    for (uint32_t k = 0; k < N; ++k) {
        const uint64_t x = powm(psi, 2ull * brv(k, bits) + 1, q);
        uint64_t s = 0, xp = 1;
        for (uint32_t i = 0; i < N; ++i) {
            s = addm(s, mulm(a[i], xp, q), q);
            xp = mulm(xp, x, q);
        }
        A[k] = s;
    }
}

/* Inverse by its definition: a_i = N^-1 sum_k A[k] psi^(-(2 brv(k) + 1) i). */
void oracle_intt_direct(const uint64_t *A, uint64_t *a, uint32_t N, uint64_t q, uint64_t psi)
{
    const uint32_t bits = log2u(N);
    const uint64_t ninv = invm(N % q, q), pinv = invm(psi, q);
    for (uint32_t i = 0; i < N; ++i) a[i] = 0;
    for (uint32_t k = 0; k < N; ++k) {
        const uint64_t x = powm(pinv, 2ull * brv(k, bits) + 1, q);
        uint64_t xp = 1;
        for (uint32_t i = 0; i < N; ++i) {
            a[i] = addm(a[i], mulm(A[k], xp, q), q);
            xp = mulm(xp, x, q);
        }
    }
    for (uint32_t i = 0; i < N; ++i) a[i] = mulm(a[i], ninv, q);
}

/* Radix-2 Cooley-Tukey, in place: at the step with m blocks of length 2t,
 * block i pairs (a_j, a_{j+t}) into (a_j + w a_{j+t}, a_j - w a_{j+t}),
 * w = psi^brv_log2N(m + i). */
void oracle_ntt_fast(uint64_t *a, uint32_t N, uint64_t q, uint64_t psi)
{
    const uint32_t bits = log2u(N);
    uint32_t t = N;
    for (uint32_t m = 1; m < N; m *= 2) {
        t /= 2;
        for (uint32_t i = 0; i < m; ++i) {
            const uint64_t w = powm(psi, brv(m + i, bits), q);
            for (uint32_t j = 2 * i * t; j < 2 * i * t + t; ++j) {
                const uint64_t u = a[j], v = mulm(a[j + t], w, q);
                a[j] = addm(u, v, q);
                a[j + t] = subm(u, v, q);
            }
        }
    }
}

/* Radix-2 Gentleman-Sande, in place, the inverse of oracle_ntt_fast:
 * (a_j, a_{j+t}) -> (a_j + a_{j+t}, (a_j - a_{j+t}) w^-1), then N^-1. */
void oracle_intt_fast(uint64_t *a, uint32_t N, uint64_t q, uint64_t psi)
{
    const uint32_t bits = log2u(N);
    const uint64_t pinv = invm(psi, q);
    uint32_t t = 1;
    for (uint32_t m = N / 2; m >= 1; m /= 2) {
        for (uint32_t i = 0; i < m; ++i) {
            const uint64_t w = powm(pinv, brv(m + i, bits), q);
            for (uint32_t j = 2 * i * t; j < 2 * i * t + t; ++j) {
                const uint64_t u = a[j], v = a[j + t];
                a[j] = addm(u, v, q);
                a[j + t] = mulm(subm(u, v, q), w, q);
            }
        }
        t *= 2;
        if (m == 1) break;
    }
    const uint64_t ninv = invm(N % q, q);
    for (uint32_t i = 0; i < N; ++i) a[i] = mulm(a[i], ninv, q);
}

/* Rescale `count` polys: in [count][L][N] (NTT form), out [count][L-1][N].
 * fast != 0 uses the radix-2 transforms, 0 the definitions.  Returns 0, or
 * -1 if an argument cannot be evaluated. */
int oracle_rescale(uint64_t count, uint32_t N, uint32_t L, const uint64_t *moduli, const uint64_t *in,
                   uint64_t *out, int fast, int round)
{
    if (L < 2 || N < 2 || (N & (N - 1))) return -1;
    uint64_t *psi = (uint64_t *)malloc(sizeof(uint64_t) * L);
    uint64_t *r = (uint64_t *)malloc(sizeof(uint64_t) * N);
    uint64_t *t = (uint64_t *)malloc(sizeof(uint64_t) * N);
    uint64_t *u = (uint64_t *)malloc(sizeof(uint64_t) * N);
    int rc = 0;
    if (!psi || !r || !t || !u) rc = -1;
    for (uint32_t l = 0; l < L && !rc; ++l)
        if (!(psi[l] = oracle_min_root(moduli[l], N))) rc = -1;
    const uint64_t ql = moduli[L - 1];
    for (uint64_t p = 0; p < count && !rc; ++p) {
        const uint64_t *y = in + p * L * (uint64_t)N;
        /* coefficients of the last limb */
        if (fast) {
            memcpy(r, y + (uint64_t)(L - 1) * N, sizeof(uint64_t) * N);
            oracle_intt_fast(r, N, ql, psi[L - 1]);
        } else {
            oracle_intt_direct(y + (uint64_t)(L - 1) * N, r, N, ql, psi[L - 1]);
        }
        const uint64_t h = round ? ql / 2 : 0;
        for (uint32_t i = 0; i < N; ++i) r[i] = addm(r[i], h, ql);
        for (uint32_t l = 0; l + 1 < L; ++l) {
            const uint64_t q = moduli[l];
            for (uint32_t i = 0; i < N; ++i) t[i] = subm(r[i] % q, h % q, q);
            if (fast) {
                oracle_ntt_fast(t, N, q, psi[l]);
            } else {
                memcpy(u, t, sizeof(uint64_t) * N);
                oracle_ntt_direct(u, t, N, q, psi[l]);
            }
            const uint64_t qinv = invm(ql % q, q);
            uint64_t *o = out + (p * (L - 1) + l) * (uint64_t)N;
            for (uint32_t k = 0; k < N; ++k) o[k] = mulm(subm(y[(uint64_t)l * N + k], t[k], q), qinv, q);
        }
    }
    free(psi);
    free(r);
    free(t);
    free(u);
    return rc;
}
