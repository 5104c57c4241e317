/*
 * fiona_workload.h -- device-side filler for synthetic benchmark and test
 * inputs (library libfiona_workload.so).  It is not part of the evaluator:
 * it holds none of the layer's arithmetic and exists so that multi-GB
 * synthetic layers can be produced on the GPU without a host round trip.
 *
 * Definition (identical to paper_2609_35352_gb300/workloads.py): value number
 * n of the stream with key K is x = SplitMix64_mix(K + (n + 1) * 0x9E3779B97F4A7C15)
 * (Steele, Lea, Flood 2014), and the residue modulo q is the high word of the
 * 128-bit product x * q.  Element n of a buffer laid out [outer][L][N] uses the
 * modulus of limb (n / N) mod L.
 */
#ifndef FIONA_WORKLOAD_H
#define FIONA_WORKLOAD_H
#include <stdint.h>
#ifdef __cplusplus
extern "C" {
#endif

/* Fill dst[outer][L][N] (device memory, 8-byte aligned) with the residues of
 * stream `key`; moduli is a HOST array of L values.  mode 0 = uniform
 * residues, mode 1 = every residue q-1, mode 2 = uniform residues constant
 * over each limb-poly (element n takes the value of element n - n mod N: a
 * constant plaintext).  Asynchronous on cuda_stream.
 * Returns 0, or -1 on a bad argument, -5 on a CUDA error. */
int fiona_workload_fill(void *cuda_stream, uint64_t *dst, uint64_t outer, uint32_t L, uint32_t N,
                        const uint64_t *moduli, uint64_t key, int mode);

/* Measured integer-multiply roof of the current device: product-accumulates
 * per second over the whole GPU of the layer kernels' own primitives, one
 * 50-bit x 50-bit product each -- narrow: three 32x32 -> 64-bit products of
 * radix-2^26 halves (Karatsuba), the arithmetic of every plan whose moduli
 * are below 2^52; wide: the 64x64 -> 128-bit product-accumulate.  Runs a few
 * milliseconds of kernels on the default stream and synchronizes.
 * Returns 0, or -1 on a null argument, -5 on a CUDA error. */
int fiona_mul_roof(double *narrow_per_s, double *wide_per_s);

/* Measured butterfly roof of the current device: forward NTT butterflies per
 * second over the whole GPU of the rescale's own butterfly (one product by a
 * twiddle with Shoup's precomputed quotient, a sum and a difference); fast:
 * without the conditional subtraction (every modulus below 2^56), general:
 * with it.  Runs a few milliseconds of kernels on the default stream and
 * synchronizes.  Returns 0, or -1 on a null argument, -5 on a CUDA error. */
int fiona_bfly_roof(double *fast_per_s, double *general_per_s);

#ifdef __cplusplus
}
#endif
#endif
