// kernel_direct.cu -- direct evaluation of the hybrid linear layer: one
// thread per (output j, limb l, pair of coefficients).  Each thread walks its
// output's scale groups (signed sum, then one product by gamma, Sec. 4.2
// "Grouping Reconstruction Operations") and raw terms (PMult-MAC), keeps one
// lazy 128-bit accumulator per poly and coefficient, and stores the canonical
// residue (signed and raw routes added before any rescale, Sec. 4.2
// "Combining the Signed and Raw Routes").  Inputs are re-read per output
// (through L2); the tiled kernel reads each input tile once.
#include <cuda_runtime.h>

#include <mutex>

#include "fiona_internal.h"

namespace {

constexpr int kDirectThreads = 128;

// Fixed device area for fiona_linear_eval_static: the limb constants and the
// direct schedule of one layer, copied in by each call.  Every GPU that
// loads this library holds these bytes until the process exits.
constexpr size_t kStaticBytes = FIONA_STATIC_AREA_BYTES;
static __device__ __align__(256) unsigned char g_static_area[kStaticBytes];

__device__ __forceinline__ ulonglong2 ld2(const uint64_t *p)
{
    return __ldg(reinterpret_cast<const ulonglong2 *>(p));
}

__global__ void __launch_bounds__(kDirectThreads)
direct_kernel(const uint64_t *__restrict__ in, const uint64_t *__restrict__ pt,
              uint64_t *__restrict__ out, const LimbConst *__restrict__ limbs,
              const DirOut *__restrict__ outs, const DirSeg *__restrict__ segs,
              const uint32_t *__restrict__ ops, const uint32_t *__restrict__ raw_in,
              const uint32_t *__restrict__ raw_pt, uint32_t N, uint32_t L, uint32_t limb0,
              uint32_t mac_budget)
{
    const uint32_t j = blockIdx.z;
    const uint32_t l = limb0 + blockIdx.y;
    const uint32_t k = (blockIdx.x * kDirectThreads + threadIdx.x) * 2;
    if (k >= N) return;
    const LimbConst m = limbs[l];
    const size_t LN = (size_t)L * N;
    const uint64_t *inl = in + (size_t)l * N + k;
    const uint64_t *ptl = pt + (size_t)l * N + k;

    // acc[c][x]: poly c, coefficient k + x, as (lo, hi)
    uint64_t lo[2][2] = {{0, 0}, {0, 0}}, hi[2][2] = {{0, 0}, {0, 0}};
    uint32_t nprod = 0;
    auto fold_if_full = [&]() {
        if (++nprod >= mac_budget) {
#pragma unroll
            for (int c = 0; c < 2; ++c)
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    lo[c][x] = rns::reduce128(lo[c][x], hi[c][x], m);
                    hi[c][x] = 0;
                }
            nprod = 1;
        }
    };

    const DirOut o = outs[j];
    for (uint32_t s = o.seg_begin; s < o.seg_end; ++s) {
        const DirSeg sg = segs[s];
        uint64_t S[2][2] = {{0, 0}, {0, 0}};
#pragma unroll 4
        for (uint32_t e = sg.op_begin; e < sg.op_end; ++e) {
            const uint32_t w = ops[e];
            const uint32_t i = w & 0x7fffffffu;
            const ulonglong2 a0 = ld2(inl + (size_t)(2 * i) * LN);
            const ulonglong2 a1 = ld2(inl + (size_t)(2 * i + 1) * LN);
            if (w >> 31) {
                S[0][0] = rns::sub_mod(S[0][0], a0.x, m.q);
                S[0][1] = rns::sub_mod(S[0][1], a0.y, m.q);
                S[1][0] = rns::sub_mod(S[1][0], a1.x, m.q);
                S[1][1] = rns::sub_mod(S[1][1], a1.y, m.q);
            } else {
                S[0][0] = rns::add_mod(S[0][0], a0.x, m.q);
                S[0][1] = rns::add_mod(S[0][1], a0.y, m.q);
                S[1][0] = rns::add_mod(S[1][0], a1.x, m.q);
                S[1][1] = rns::add_mod(S[1][1], a1.y, m.q);
            }
        }
        const ulonglong2 g = ld2(ptl + (size_t)sg.scale_pt * LN);
        rns::mac(lo[0][0], hi[0][0], g.x, S[0][0]);
        rns::mac(lo[0][1], hi[0][1], g.y, S[0][1]);
        rns::mac(lo[1][0], hi[1][0], g.x, S[1][0]);
        rns::mac(lo[1][1], hi[1][1], g.y, S[1][1]);
        fold_if_full();
    }
#pragma unroll 2
    for (uint32_t r = o.raw_begin; r < o.raw_end; ++r) {
        const uint32_t i = raw_in[r];
        // bit 31: a constant plaintext, its limb's residue 0 at every coefficient
        const uint32_t wp = raw_pt[r];
        ulonglong2 p = ld2(((wp >> 31) ? ptl - k : ptl) + (size_t)(wp & 0x7fffffffu) * LN);
        if (wp >> 31) p.y = p.x;
        const ulonglong2 a0 = ld2(inl + (size_t)(2 * i) * LN);
        const ulonglong2 a1 = ld2(inl + (size_t)(2 * i + 1) * LN);
        rns::mac(lo[0][0], hi[0][0], p.x, a0.x);
        rns::mac(lo[0][1], hi[0][1], p.y, a0.y);
        rns::mac(lo[1][0], hi[1][0], p.x, a1.x);
        rns::mac(lo[1][1], hi[1][1], p.y, a1.y);
        fold_if_full();
    }
    uint64_t *outl = out + ((size_t)j * 2 * L + l) * N + k;
#pragma unroll
    for (int c = 0; c < 2; ++c) {
        ulonglong2 y;
        y.x = rns::reduce128(lo[c][0], hi[c][0], m);
        y.y = rns::reduce128(lo[c][1], hi[c][1], m);
        *reinterpret_cast<ulonglong2 *>(outl + (size_t)c * LN) = y;
    }
}

__global__ void check_residues_kernel(const uint64_t *__restrict__ data, uint64_t count,
                                      const LimbConst *__restrict__ limbs, uint32_t N, uint32_t L,
                                      int *flag)
{
    const uint64_t total = count * L * (uint64_t)N;
    for (uint64_t idx = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (uint64_t)gridDim.x * blockDim.x) {
        const uint32_t l = (uint32_t)((idx / N) % L);
        if (data[idx] >= limbs[l].q) {
            atomicOr(flag, 1);
            return;
        }
    }
}

}  // namespace

int launch_direct(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                  uint64_t *out, uint32_t l0, uint32_t l1, uint32_t layout_L)
{
    const fiona_ctx *ctx = p->ctx;
    if (l1 <= l0) return FIONA_OK;
    dim3 grid((ctx->N / 2 + kDirectThreads - 1) / kDirectThreads, l1 - l0, p->hp.n_out);
    direct_kernel<<<grid, kDirectThreads, 0, (cudaStream_t)stream>>>(
        in, pt, out, ctx->d_limbs, p->d_dir_out, p->d_dir_seg, p->d_sig_ops, p->d_raw_input,
        p->d_raw_pt, ctx->N, layout_L, l0, p->mac_budget);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "direct kernel launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

const size_t kStaticAreaBytes = kStaticBytes;

// Device address of g_static_area on the current device, looked up once per
// device (host code cannot use the symbol itself as a device pointer).
static int static_area(unsigned char **ptr)
{
    static std::mutex mu;
    static unsigned char *addr[FIONA_MAX_DEVICES] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "static area: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= FIONA_MAX_DEVICES) return set_error(FIONA_ERR_ARG, "static area: device %d", dev);
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_area);
        if (e != cudaSuccess)
            return set_error(FIONA_ERR_CUDA, "static area: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        addr[dev] = (unsigned char *)p;
    }
    *ptr = addr[dev];
    return FIONA_OK;
}

int launch_direct_static(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                         uint64_t *out)
{
    const fiona_ctx *ctx = p->ctx;
    unsigned char *area = nullptr;
    int rc = static_area(&area);
    if (rc) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    // every byte the kernel reads is rewritten here first, in stream order
    cudaError_t e = cudaMemcpyAsync(area, p->static_image.data(), p->static_image.size(),
                                    cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "static area copy: %s", cudaGetErrorString(e));
    const size_t *o = p->static_off;
    dim3 grid((ctx->N / 2 + kDirectThreads - 1) / kDirectThreads, ctx->L, p->hp.n_out);
    direct_kernel<<<grid, kDirectThreads, 0, s>>>(
        in, pt, out, (const LimbConst *)(area + o[0]), (const DirOut *)(area + o[1]),
        (const DirSeg *)(area + o[2]), (const uint32_t *)(area + o[3]), (const uint32_t *)(area + o[4]),
        (const uint32_t *)(area + o[5]), ctx->N, ctx->L, 0, p->mac_budget);
    e = cudaGetLastError();
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "direct kernel launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int launch_check_residues(const fiona_ctx *ctx, void *stream, const uint64_t *data, uint64_t count)
{
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(ctx->d_flag, 0, sizeof(int), s);
    if (e == cudaSuccess) {
        const int blocks = ctx->sm_count > 0 ? ctx->sm_count * 8 : 1024;
        check_residues_kernel<<<blocks, 256, 0, s>>>(data, count, ctx->d_limbs, ctx->N, ctx->L,
                                                     ctx->d_flag);
        e = cudaGetLastError();
    }
    int flag = 0;
    if (e == cudaSuccess) e = cudaMemcpyAsync(&flag, ctx->d_flag, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "check_residues: %s", cudaGetErrorString(e));
    return flag ? set_error(FIONA_ERR_RANGE, "a residue is >= its modulus") : FIONA_OK;
}
