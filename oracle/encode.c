/*
 * encode.c -- plain CPU oracle for plaintext encoding (Sec. 2.2 "Ciphertexts
 * and Slots": CKKS packs a vector of numbers into the slots of a plaintext).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this code.  It shares no code,
 * header, table or helper with the CUDA path.
 *
 * Definitions (the evaluator follows the same ones, written separately):
 *   slots    slot j of a plaintext m (a real poly of degree < N) is the value
 *            m(zeta^(5^j)), zeta = exp(i pi / N), j = 0 .. N/2 - 1; its
 *            conjugate is m(zeta^(-5^j));
 *   embed    the coefficients of that m are, by the inversion formula over
 *            the N odd powers of zeta,
 *              m_i = (2/N) sum_j Re(z_j zeta^(-5^j i)),
 *            and encoding at scale Delta rounds them: c_i = round(Delta m_i),
 *            ties away from zero;
 *   NTT form c mod q_l (canonical), then A[k] = c(psi^(2 brv(k) + 1)) mod q_l
 *            (oracle_ntt_fast / oracle_ntt_direct of rescale.c).
 * The sum is taken term by term in long double with powers of zeta from a
 * table of cosl/sinl at exactly reduced exponents.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

void oracle_ntt_fast(uint64_t *a, uint32_t N, uint64_t q, uint64_t psi);
void oracle_ntt_direct(const uint64_t *a, uint64_t *A, uint32_t N, uint64_t q, uint64_t psi);
uint64_t oracle_min_root(uint64_t q, uint32_t N);

/* Coefficients idx[0..n_idx) of the encoding of one slot vector z
 * ([N/2][2] doubles: re, im) at `scale`, into out.  Returns 0, or -1 if a
 * coefficient is not below 2^62 in magnitude (or an argument is invalid). */
int oracle_ckks_embed(uint32_t N, const double *z, double scale, const uint32_t *idx, uint32_t n_idx,
                      int64_t *out)
{
    if (N < 4 || (N & (N - 1))) return -1;
    const uint32_t M = 2 * N, n = N / 2;
    const long double pi = 3.141592653589793238462643383279502884L;
    long double *c = malloc(sizeof(long double) * M), *s = malloc(sizeof(long double) * M);
    uint64_t *p5 = malloc(sizeof(uint64_t) * n);
    int rc = 0;
    if (!c || !s || !p5) rc = -1;
    for (uint32_t e = 0; e < M && !rc; ++e) {
        c[e] = cosl(pi * (long double)e / (long double)N);
        s[e] = sinl(pi * (long double)e / (long double)N);
    }
    if (!rc) {
        p5[0] = 1;
        for (uint32_t j = 1; j < n; ++j) p5[j] = p5[j - 1] * 5 % M;
    }
    for (uint32_t t = 0; t < n_idx && !rc; ++t) {
        const uint64_t i = idx[t];
        if (i >= N) {
            rc = -1;
            break;
        }
        long double acc = 0;
        for (uint32_t j = 0; j < n; ++j) {
            /* Re(z zeta^(-e)) = re cos(pi e / N) + im sin(pi e / N) */
            const uint64_t e = p5[j] * i % M;
            acc += (long double)z[2 * j] * c[e] + (long double)z[2 * j + 1] * s[e];
        }
        const long double v = (long double)scale * 2 * acc / (long double)N;
        if (!(fabsl(v) < 4611686018427387904.0L)) {
            rc = -1;
            break;
        }
        out[t] = (int64_t)llroundl(v);
    }
    free(c);
    free(s);
    free(p5);
    return rc;
}

/* Integer polys coeffs [count][N] to NTT form out [count][L][N] modulo
 * moduli[0..L).  fast != 0 uses the radix-2 transform, 0 the definition.
 * Returns 0, or -1 if a modulus has no primitive 2N-th root. */
int oracle_encode_coeffs(uint32_t N, uint32_t L, const uint64_t *moduli, uint64_t count, const int64_t *coeffs,
                         uint64_t *out, int fast)
{
    uint64_t *t = malloc(sizeof(uint64_t) * N);
    if (!t) return -1;
    int rc = 0;
    for (uint32_t l = 0; l < L && !rc; ++l) {
        const uint64_t q = moduli[l];
        const uint64_t psi = oracle_min_root(q, N);
        if (!psi) {
            rc = -1;
            break;
        }
        for (uint64_t p = 0; p < count; ++p) {
            const int64_t *c = coeffs + p * N;
            uint64_t *o = out + (p * L + l) * (uint64_t)N;
            for (uint32_t i = 0; i < N; ++i) {
                /* c mod q, canonical: |c| as an unsigned word, then negated mod q */
                const uint64_t mag = c[i] >= 0 ? (uint64_t)c[i] : (uint64_t)0 - (uint64_t)c[i];
                const uint64_t r = mag % q;
                t[i] = (c[i] >= 0 || r == 0) ? r : q - r;
            }
            if (fast) {
                for (uint32_t i = 0; i < N; ++i) o[i] = t[i];
                oracle_ntt_fast(o, N, q, psi);
            } else {
                oracle_ntt_direct(t, o, N, q, psi);
            }
        }
    }
    free(t);
    return rc;
}
