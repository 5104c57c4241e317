// workload_fill.cu -- device filler for synthetic inputs (see
// include/fiona_workload.h).  Shares nothing with the evaluator.
#include <cuda_runtime.h>
#include <stdint.h>

#include "fiona_workload.h"

namespace {

struct Moduli {
    uint64_t q[64];
};

__device__ __forceinline__ uint64_t splitmix_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__global__ void fill_kernel(uint64_t *__restrict__ dst, uint64_t total, uint32_t L, uint32_t N,
                            Moduli mods, uint64_t key, int mode)
{
    for (uint64_t n = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; n < total;
         n += (uint64_t)gridDim.x * blockDim.x) {
        const uint64_t q = mods.q[(n / N) % L];
        if (mode == 1) {
            dst[n] = q - 1;
        } else {
            // mode 2: every element of a limb-poly takes the value of its first
            const uint64_t idx = mode == 2 ? n - n % N : n;
            const uint64_t x = splitmix_mix(key + (idx + 1) * 0x9E3779B97F4A7C15ull);
            dst[n] = __umul64hi(x, q);
        }
    }
}

}  // namespace

extern "C" int fiona_workload_fill(void *stream, uint64_t *dst, uint64_t outer, uint32_t L,
                                   uint32_t N, const uint64_t *moduli, uint64_t key, int mode)
{
    if (!dst || !moduli || L == 0 || L > 64 || N == 0 || mode < 0 || mode > 2) return -1;
    Moduli m{};
    for (uint32_t l = 0; l < L; ++l) m.q[l] = moduli[l];
    const uint64_t total = outer * L * (uint64_t)N;
    if (total == 0) return 0;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int blocks = (sms > 0 ? sms : 128) * 8;
    fill_kernel<<<blocks, 256, 0, (cudaStream_t)stream>>>(dst, total, L, N, m, key, mode);
    return cudaGetLastError() == cudaSuccess ? 0 : -5;
}
