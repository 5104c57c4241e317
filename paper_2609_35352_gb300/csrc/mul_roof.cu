// mul_roof.cu -- measured integer-multiply roof of the GPU (library
// libfiona_workload.so, a measurement aid beside the synthetic filler; not
// part of the evaluator).
//
// Every thread of a full grid runs independent product-accumulate chains of
// the layer kernels' own primitives (rns.cuh) on operands that change every
// step, so that nothing folds away:
//   narrow: rns::mac26, three 32x32 -> 64-bit products of radix-2^26 halves
//           (Karatsuba) into three accumulators -- one 50-bit x 50-bit
//           product per call;
//   wide:   rns::mac, the 64x64 -> 128-bit product-accumulate with carry.
// The rate is products per second of the whole GPU, timed with CUDA events
// after a warm-up launch.  A layer's products per evaluation
// (fiona_plan_stats.wide_products) over its kernel time, divided by this
// rate, is its utilisation of the multiplier roof.
#include <cuda_runtime.h>

#include "fiona_workload.h"
#include "ntt.cuh"
#include "rns.cuh"

namespace {

constexpr int kChains = 4;
constexpr int kSteps = 256;

template <bool NARROW>
__global__ void __launch_bounds__(256) roof_kernel(const uint64_t *seed, uint64_t *sink, uint32_t zero)
{
    uint64_t a[kChains], b[kChains], lo[kChains], mid[kChains], hi[kChains];
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
        // split-form operands: halves below 2^26
        a[c] = (seed[(threadIdx.x + c) & 63] & 0x03FFFFFF03FFFFFFull) | 1;
        b[c] = (seed[(threadIdx.x + 7 * c + 1) & 63] & 0x03FFFFFF03FFFFFFull) | 1;
        lo[c] = mid[c] = hi[c] = 0;
    }
    for (int s = 0; s < kSteps; ++s) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) {
            if (NARROW)
                rns::mac26(lo[c], mid[c], hi[c], a[c], b[c], zero);  // as the layer kernels call it
            else
                rns::mac(lo[c], hi[c], a[c], b[c]);
            // the next step's operands depend on this step (stay in split form)
            a[c] = (a[c] + (lo[c] & 0x0000000F0000000Full)) & 0x03FFFFFF03FFFFFFull;
        }
    }
    uint64_t r = 0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) r += lo[c] ^ mid[c] ^ hi[c];
    sink[blockIdx.x * blockDim.x + threadIdx.x] = r;
}

template <bool NARROW>
double rate(int sms, const uint64_t *seed, uint64_t *sink)
{
    const dim3 grid(sms * 8), block(256);
    roof_kernel<NARROW><<<grid, block>>>(seed, sink, 0);  // warm-up
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    const int reps = 3;
    cudaEventRecord(e0);
    for (int r = 0; r < reps; ++r) roof_kernel<NARROW><<<grid, block>>>(seed, sink, 0);
    cudaEventRecord(e1);
    float ms = 0;
    const bool ok = cudaEventSynchronize(e1) == cudaSuccess && cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess;
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (!ok || ms <= 0) return 0;
    const double products = (double)reps * grid.x * block.x * kSteps * kChains;
    return products / (ms * 1e-3);
}

// Forward NTT butterflies of the rescale (fiona_ntt::ModArith::ct: one
// product by a twiddle with Shoup's precomputed quotient, a sum and a
// difference), FAST = without the conditional subtraction (every modulus
// below 2^56), in kChains independent chains per thread; the twiddle changes
// every step so that nothing folds away.
template <bool FAST>
__global__ void __launch_bounds__(256) bfly_kernel(const uint64_t *seed, uint64_t *sink)
{
    const fiona_ntt::ModArith<FAST> ar{(seed[0] >> 14) | 1};
    uint64_t x[kChains], y[kChains];
    ulonglong2 w[kChains];
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
        x[c] = seed[(threadIdx.x + c) & 63] >> 14;
        y[c] = seed[(threadIdx.x + 7 * c + 1) & 63] >> 14;
        w[c] = make_ulonglong2(seed[(threadIdx.x + 3 * c + 2) & 63] >> 14, seed[(threadIdx.x + 5 * c + 3) & 63]);
    }
    for (int s = 0; s < kSteps; ++s) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) {
            ar.ct(x[c], y[c], w[c]);
            w[c].x ^= y[c] & 0xF;
        }
    }
    uint64_t r = 0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) r += x[c] ^ y[c] ^ w[c].x;
    sink[blockIdx.x * blockDim.x + threadIdx.x] = r;
}

template <bool FAST>
double bfly_rate(int sms, const uint64_t *seed, uint64_t *sink)
{
    const dim3 grid(sms * 8), block(256);
    bfly_kernel<FAST><<<grid, block>>>(seed, sink);  // warm-up
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    const int reps = 3;
    cudaEventRecord(e0);
    for (int r = 0; r < reps; ++r) bfly_kernel<FAST><<<grid, block>>>(seed, sink);
    cudaEventRecord(e1);
    float ms = 0;
    const bool ok = cudaEventSynchronize(e1) == cudaSuccess && cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess;
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    if (!ok || ms <= 0) return 0;
    return (double)reps * grid.x * block.x * kSteps * kChains / (ms * 1e-3);
}

// device buffers of the roof measurements: 64 seed words and one sink word
// per thread of the grid
int roof_buffers(int *sms, uint64_t **seed, uint64_t **sink)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || *sms <= 0)
        return -5;
    if (cudaMalloc(seed, 64 * sizeof(uint64_t)) != cudaSuccess) return -5;
    if (cudaMalloc(sink, (size_t)*sms * 8 * 256 * sizeof(uint64_t)) != cudaSuccess) {
        cudaFree(*seed);
        return -5;
    }
    uint64_t h[64];
    uint64_t x = 0x9E3779B97F4A7C15ull;
    for (auto &v : h) v = (x = x * 6364136223846793005ull + 1442695040888963407ull);
    return cudaMemcpy(*seed, h, sizeof(h), cudaMemcpyHostToDevice) == cudaSuccess ? 0 : -5;
}

}  // namespace

extern "C" int fiona_bfly_roof(double *fast_per_s, double *general_per_s)
{
    if (!fast_per_s || !general_per_s) return -1;
    int sms = 0;
    uint64_t *seed = nullptr, *sink = nullptr;
    int rc = roof_buffers(&sms, &seed, &sink);
    if (rc == 0) {
        *fast_per_s = bfly_rate<true>(sms, seed, sink);
        *general_per_s = bfly_rate<false>(sms, seed, sink);
        if (*fast_per_s <= 0 || *general_per_s <= 0 || cudaGetLastError() != cudaSuccess) rc = -5;
    }
    cudaFree(seed);
    cudaFree(sink);
    return rc;
}

extern "C" int fiona_mul_roof(double *narrow_per_s, double *wide_per_s)
{
    if (!narrow_per_s || !wide_per_s) return -1;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        return -5;
    uint64_t *seed = nullptr, *sink = nullptr;
    if (cudaMalloc(&seed, 64 * sizeof(uint64_t)) != cudaSuccess) return -5;
    if (cudaMalloc(&sink, (size_t)sms * 8 * 256 * sizeof(uint64_t)) != cudaSuccess) {
        cudaFree(seed);
        return -5;
    }
    uint64_t h[64];
    uint64_t x = 0x9E3779B97F4A7C15ull;
    for (auto &v : h) v = (x = x * 6364136223846793005ull + 1442695040888963407ull);
    int rc = cudaMemcpy(seed, h, sizeof(h), cudaMemcpyHostToDevice) == cudaSuccess ? 0 : -5;
    if (rc == 0) {
        *narrow_per_s = rate<true>(sms, seed, sink);
        *wide_per_s = rate<false>(sms, seed, sink);
        if (*narrow_per_s <= 0 || *wide_per_s <= 0 || cudaGetLastError() != cudaSuccess) rc = -5;
    }
    cudaFree(seed);
    cudaFree(sink);
    return rc;
}
