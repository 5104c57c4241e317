// encode.cu -- plaintext encoding on the GPU (Sec. 2.2 "Ciphertexts and
// Slots": CKKS packs a vector of numbers into the slots of a plaintext; the
// evaluated layer's gamma and raw plaintexts are such encodings of the
// model's weights, and the paper's timings include encoding them).
//
// Encoding of a slot vector z (N/2 complex numbers) at scale Delta:
//   1. embedding: m is the real poly of degree < N with m(zeta^(5^j)) = z_j
//      and m(zeta^(-5^j)) = conj(z_j), zeta = exp(i pi / N) (slot j sits at
//      the odd power 5^j mod 2N; the powers +-5^j are every odd residue);
//      the integer coefficients are c_i = round(Delta * m_i), ties away from
//      zero.  By the inversion formula over the odd powers of zeta,
//      m_i = (2/N) Re(u_i) and m_{i+n} = (2/N) Im(u_i), n = N/2, with
//        u_i = sum_j z_j zeta^(-5^j i) = sum_r y_r zeta^(-(4r+1) i),
//      y_r = z_j for 5^j = 4r + 1 mod 2N (the powers of 5 are the residues
//      1 mod 4).  With A[k] = y_brv(k) (n-bit reversal) and psi = zeta^2,
//        u_i = zeta^i sum_k A[k] psi^(-(2 brv(k) + 1) i),
//      which is n times the inverse negacyclic transform of A of size n
//      (ntt.cuh over complex fp64) twisted by zeta^i.  So the inverse low
//      pass gathers A[k] from z, and the inverse high pass multiplies by
//      zeta^i and rounds Delta (2/N) of the real and imaginary parts to the
//      64-bit coefficients i and i + n.
//   2. RNS/NTT form: c_i mod q_l for every limb, then the forward NTT mod
//      q_l (ntt.cuh, the tables the rescale uses), canonical.
// Step 1 is floating point: it reproduces round(Delta m_i) except where
// Delta m_i lies within the transform's rounding error of a half-integer.
// Step 2 is exact.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <vector>

#include "fiona_internal.h"
#include "ntt.cuh"

using namespace fiona_ntt;

namespace {

// in device memory, n = N/2 entries each: the twiddles psi^-brv(k) =
// zeta^(-2 brv(k)) as (cos, sin), the slot index of A[k], and the twists
// zeta^i
struct EncTables {
    const double2 *cinv;
    const uint32_t *gather;
    const double2 *twist;
};

struct EmbArgs {
    const double2 *slots;  // [count][N/2]
    double2 *work;         // [count][N/2]
    int64_t *coeffs;       // [count][N]
    EncTables E;
    double factor;         // Delta (2 / N)
    int *err;              // bit 1: a coefficient reached 2^62 (or was not finite)
};

struct EncArgs {
    const int64_t *coeffs;  // [count][N]
    uint64_t *out;          // [count][Lc][N]
    const NttLimb *T;
    uint32_t Lc;
};

// round(x) as a 64-bit integer; 0 and the range flag when |x| >= 2^62 or x
// is not finite
__device__ __forceinline__ int64_t round_coeff(double x, int *err)
{
    if (fabs(x) < 0x1p62) return llround(x);
    atomicOr(err, 2);
    return 0;
}

// embedding, inverse low stages of the size-n transform (LN = log2 n):
// A[k] gathered from the slots
template <int LN>
__global__ void __launch_bounds__(LowPass<LN>::threads, 2) k_embed_low(EmbArgs A)
{
    using SH = Shape<LN>;
    using PS = LowPass<LN>;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), p = blockIdx.x >> PS::ltiles;
    const uint32_t first = tile << PS::lsubs;
    const size_t base = (size_t)first << PS::s;
    const double2 *z = A.slots + ((size_t)p << LN);
    const uint32_t *gat = A.E.gather + base;
    double2 *w = A.work + ((size_t)p << LN) + base;
    inv_low_pass<LN>(
        smem_raw, A.E.cinv, first, CplxArith{}, [&](uint32_t e) { return z[gat[e]]; },
        [&](uint32_t sub, uint32_t pos, double2 v) { w[(sub << PS::s) + pos] = v; });
}

// embedding, inverse high stages: x zeta^i, rounded Delta (2/N) Re and Im to
// coefficients i and i + n
template <int LN>
__global__ void __launch_bounds__(HighPass<LN>::threads, 2) k_embed_high(EmbArgs A)
{
    using SH = Shape<LN>;
    using PS = HighPass<LN>;
    constexpr uint32_t R2 = 1u << (LN - SH::n1);
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), p = blockIdx.x >> PS::ltiles;
    const uint32_t first = tile << PS::lsubs;
    const double2 *g = A.work + ((size_t)p << LN) + first;
    const double2 *tw = A.E.twist + first;
    int64_t *c = A.coeffs + ((size_t)p << (LN + 1)) + first;
    const double f = A.factor;
    inv_high_pass<LN>(
        smem_raw, A.E.cinv, first, CplxArith{}, [&](uint32_t sub, uint32_t pos) { return g[(size_t)pos * R2 + sub]; },
        [&](uint32_t sub, uint32_t pos, double2 v) {
            const size_t i = (size_t)pos * R2 + sub;
            const double2 u = CplxArith::mul(v, tw[i]);
            c[i] = round_coeff(u.x * f, A.err);
            c[i + (1u << LN)] = round_coeff(u.y * f, A.err);
        });
}

// RNS/NTT form, forward high stages: c mod q_l into out (lazy)
template <int LOGN, bool FAST>
__global__ void __launch_bounds__(HighPass<LOGN>::threads, 3) k_enc_high(EncArgs A)
{
    using SH = Shape<LOGN>;
    using PS = HighPass<LOGN>;
    constexpr uint32_t R2 = 1u << (LOGN - SH::n1);
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), tr = blockIdx.x >> PS::ltiles;
    const uint32_t p = tr / A.Lc, l = tr % A.Lc;
    const uint32_t first = tile << PS::lsubs;
    const int64_t *c = A.coeffs + ((size_t)p << LOGN) + first;
    uint64_t *o = A.out + ((size_t)tr << LOGN) + first;
    const NttLimb &Tl = A.T[l];
    const uint64_t q = Tl.q, mu = Tl.mu64;
    fwd_high_pass<LOGN>(
        smem_raw, Tl.fwd, first, ModArith<FAST>{q},
        [&](uint32_t sub, uint32_t pos) {
            const int64_t v = c[(size_t)pos * R2 + sub];
            // |v| as an unsigned word (exact for every 64-bit v); -|v| is q - r,
            // in (0, q]
            const uint64_t mag = v >= 0 ? (uint64_t)v : 0 - (uint64_t)v;
            const uint64_t r = reduce_any(mag, q, mu);
            return v >= 0 ? r : q - r;
        },
        [&](uint32_t sub, uint32_t pos, uint64_t v) { o[(size_t)pos * R2 + sub] = v; });
}

// RNS/NTT form, forward low stages, canonical store
template <int LOGN, bool FAST>
__global__ void __launch_bounds__(LowPass<LOGN>::threads, 4) k_enc_low(EncArgs A)
{
    using SH = Shape<LOGN>;
    using PS = LowPass<LOGN>;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), tr = blockIdx.x >> PS::ltiles;
    const uint32_t l = tr % A.Lc;
    const uint32_t first = tile << PS::lsubs;
    uint64_t *o = A.out + ((size_t)tr << LOGN) + ((size_t)first << PS::s);
    const NttLimb &Tl = A.T[l];
    const uint64_t q = Tl.q, mu = Tl.mu64;
    fwd_low_pass<LOGN>(
        smem_raw, Tl.fwd, first, ModArith<FAST>{q}, [] {},
        [&](uint32_t sub, uint32_t pos) { return o[(sub << PS::s) + pos]; },
        [&](auto t_of) {
            sweep<PS, uint64_t>([&](uint32_t e) { return t_of(e); },
                                [&](uint32_t e, uint64_t v) { o[e] = reduce_any(v, q, mu); });
        });
}

// ---------------------------------------------------------------------------
// Host
// ---------------------------------------------------------------------------
std::mutex g_enc_mu;

int build_encode_tables(const fiona_ctx *ctx)
{
    std::lock_guard<std::mutex> lock(g_enc_mu);
    if (ctx->d_enc) return FIONA_OK;
    const uint32_t N = ctx->N, n = N / 2, ln = log2u(n), M = 2 * N;
    const size_t tw_bytes = sizeof(double2) * n, gat_bytes = sizeof(uint32_t) * n;
    const size_t bytes = 2 * tw_bytes + gat_bytes;
    std::vector<uint8_t> host(bytes);
    double2 *tw = reinterpret_cast<double2 *>(host.data());
    double2 *twist = reinterpret_cast<double2 *>(host.data() + tw_bytes);
    uint32_t *gat = reinterpret_cast<uint32_t *>(host.data() + 2 * tw_bytes);
    const long double pi = 3.141592653589793238462643383279502884L;
    for (uint32_t k = 0; k < n; ++k) {
        // psi^-brv(k) = zeta^(-2 brv(k)) and zeta^k, zeta = exp(i pi / N)
        const long double a = -2 * pi * (long double)bit_reverse(k, ln) / (long double)N;
        tw[k] = make_double2((double)cosl(a), (double)sinl(a));
        const long double b = pi * (long double)k / (long double)N;
        twist[k] = make_double2((double)cosl(b), (double)sinl(b));
    }
    // slot j sits at the exponent 5^j mod 2N, which is 4r + 1 for one r < n
    std::vector<int64_t> slot_of_r(n, -1);
    uint64_t e5 = 1;
    for (uint32_t j = 0; j < n; ++j) {
        if (e5 % 4 != 1 || slot_of_r[(e5 - 1) / 4] >= 0)
            return set_error(FIONA_ERR_INTERNAL, "encode tables: 5^%u mod 2N = %llu", j, (unsigned long long)e5);
        slot_of_r[(e5 - 1) / 4] = j;
        e5 = e5 * 5 % M;
    }
    for (uint32_t k = 0; k < n; ++k) gat[k] = (uint32_t)slot_of_r[bit_reverse(k, ln)];
    void *dev = nullptr;
    cudaError_t err = cudaMalloc(&dev, bytes);
    if (err != cudaSuccess) return set_error(FIONA_ERR_NOMEM, "encode tables: %s", cudaGetErrorString(err));
    err = cudaMemcpy(dev, host.data(), bytes, cudaMemcpyHostToDevice);
    if (err != cudaSuccess) {
        cudaFree(dev);
        return set_error(FIONA_ERR_CUDA, "encode tables: %s", cudaGetErrorString(err));
    }
    ctx->d_enc = dev;
    return FIONA_OK;
}

typedef void (*EmbKern)(EmbArgs);
typedef void (*EncKern)(EncArgs);

template <int LOGN>
struct Inst {
    static constexpr size_t emb_low = LowPass<LOGN - 1>::template smem_bytes<CplxArith>();
    static constexpr size_t emb_high = HighPass<LOGN - 1>::template smem_bytes<CplxArith>();
    static constexpr size_t enc_low = LowPass<LOGN>::template smem_bytes<ModArith<false>>();
    static constexpr size_t enc_high = HighPass<LOGN>::template smem_bytes<ModArith<false>>();
};

struct Kernels {
    EmbKern emb_low, emb_high;
    EncKern enc_high[2], enc_low[2];
    size_t s_emb_low, s_emb_high, s_enc_high, s_enc_low;
    // log2 tiles per transform and threads per CTA of each pass
    uint32_t lt_emb_low, lt_emb_high, lt_enc_high, lt_enc_low;
    uint32_t t_emb_low, t_emb_high, t_enc_high, t_enc_low;
};

template <int LOGN>
constexpr Kernels kernels_for()
{
    return Kernels{k_embed_low<LOGN - 1>,
                   k_embed_high<LOGN - 1>,
                   {k_enc_high<LOGN, false>, k_enc_high<LOGN, true>},
                   {k_enc_low<LOGN, false>, k_enc_low<LOGN, true>},
                   Inst<LOGN>::emb_low,
                   Inst<LOGN>::emb_high,
                   Inst<LOGN>::enc_high,
                   Inst<LOGN>::enc_low,
                   LowPass<LOGN - 1>::ltiles,
                   HighPass<LOGN - 1>::ltiles,
                   HighPass<LOGN>::ltiles,
                   LowPass<LOGN>::ltiles,
                   LowPass<LOGN - 1>::threads,
                   HighPass<LOGN - 1>::threads,
                   HighPass<LOGN>::threads,
                   LowPass<LOGN>::threads};
}

const Kernels &kernels(uint32_t n)
{
    static const Kernels K[] = {kernels_for<10>(), kernels_for<11>(), kernels_for<12>(), kernels_for<13>(),
                                kernels_for<14>(), kernels_for<15>(), kernels_for<16>(), kernels_for<17>()};
    return K[n - kLogNMin];
}

// the dynamic shared memory limits, once per device and ring dimension
int configure(const fiona_ctx *ctx, uint32_t n)
{
    static bool done[FIONA_MAX_DEVICES][kLogNMax - kLogNMin + 1] = {};
    std::lock_guard<std::mutex> lock(g_enc_mu);
    if (ctx->device < 0 || ctx->device >= FIONA_MAX_DEVICES)
        return set_error(FIONA_ERR_ARG, "encode: device %d", ctx->device);
    if (done[ctx->device][n - kLogNMin]) return FIONA_OK;
    const Kernels &K = kernels(n);
    const std::pair<const void *, size_t> fs[] = {
        {(const void *)K.emb_low, K.s_emb_low},         {(const void *)K.emb_high, K.s_emb_high},
        {(const void *)K.enc_high[0], K.s_enc_high},    {(const void *)K.enc_high[1], K.s_enc_high},
        {(const void *)K.enc_low[0], K.s_enc_low},      {(const void *)K.enc_low[1], K.s_enc_low}};
    for (const auto &f : fs) {
        const cudaError_t e = cudaFuncSetAttribute(f.first, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)f.second);
        if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "encode: kernel attributes: %s", cudaGetErrorString(e));
    }
    done[ctx->device][n - kLogNMin] = true;
    return FIONA_OK;
}

}  // namespace

int launch_embed(const fiona_ctx *ctx, void *stream, uint64_t count, const double *slots, double scale,
                 int64_t *coeffs, double *work)
{
    const uint32_t n = log2u(ctx->N);
    if (n < (uint32_t)kLogNMin || n > (uint32_t)kLogNMax)
        return set_error(FIONA_ERR_ARG, "encode: N = %u outside [2^%d, 2^%d]", ctx->N, kLogNMin, kLogNMax);
    int rc = build_encode_tables(ctx);
    if (rc == FIONA_OK) rc = configure(ctx, n);
    if (rc) return rc;
    if (count == 0) return FIONA_OK;
    const Kernels &K = kernels(n);
    const uint8_t *tab = static_cast<const uint8_t *>(ctx->d_enc);
    EmbArgs a;
    a.E.cinv = reinterpret_cast<const double2 *>(tab);
    a.E.twist = reinterpret_cast<const double2 *>(tab + sizeof(double2) * (ctx->N / 2));
    a.E.gather = reinterpret_cast<const uint32_t *>(tab + 2 * sizeof(double2) * (ctx->N / 2));
    a.factor = 2.0 * scale / (double)ctx->N;
    a.err = ctx->d_kerr;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaSuccess;
    const uint64_t max_polys = ((1ull << 31) - 1) >> std::max(K.lt_emb_low, K.lt_emb_high);
    for (uint64_t p0 = 0; p0 < count && e == cudaSuccess; p0 += max_polys) {
        const uint64_t np = std::min<uint64_t>(count - p0, max_polys);
        a.slots = reinterpret_cast<const double2 *>(slots) + p0 * (ctx->N / 2);
        a.work = reinterpret_cast<double2 *>(work) + p0 * (ctx->N / 2);
        a.coeffs = coeffs + p0 * ctx->N;
        K.emb_low<<<(uint32_t)(np << K.lt_emb_low), K.t_emb_low, K.s_emb_low, s>>>(a);
        K.emb_high<<<(uint32_t)(np << K.lt_emb_high), K.t_emb_high, K.s_emb_high, s>>>(a);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "encode launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int launch_encode_coeffs(const fiona_ctx *ctx, void *stream, uint32_t Lc, uint64_t count, const int64_t *coeffs,
                         uint64_t *out)
{
    const uint32_t n = log2u(ctx->N);
    if (n < (uint32_t)kLogNMin || n > (uint32_t)kLogNMax)
        return set_error(FIONA_ERR_ARG, "encode: N = %u outside [2^%d, 2^%d]", ctx->N, kLogNMin, kLogNMax);
    const NttLimb *T = nullptr;
    int rc = ntt_tables(ctx, &T);
    if (rc == FIONA_OK) rc = configure(ctx, n);
    if (rc) return rc;
    if (count == 0) return FIONA_OK;
    // the reduction-free butterflies need every q_l < 2^56 (inputs are canonical)
    bool fast = true;
    for (uint32_t l = 0; l < Lc; ++l)
        if (ctx->moduli[l] >= (1ull << 56)) fast = false;
    const Kernels &K = kernels(n);
    EncArgs a;
    a.T = T;
    a.Lc = Lc;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaSuccess;
    const uint64_t max_polys = ((1ull << 31) - 1) / ((uint64_t)Lc << std::max(K.lt_enc_high, K.lt_enc_low));
    for (uint64_t p0 = 0; p0 < count && e == cudaSuccess; p0 += max_polys) {
        const uint64_t np = std::min<uint64_t>(count - p0, max_polys);
        a.coeffs = coeffs + p0 * ctx->N;
        a.out = out + p0 * Lc * (uint64_t)ctx->N;
        const uint64_t nt = np * Lc;
        K.enc_high[fast]<<<(uint32_t)(nt << K.lt_enc_high), K.t_enc_high, K.s_enc_high, s>>>(a);
        K.enc_low[fast]<<<(uint32_t)(nt << K.lt_enc_low), K.t_enc_low, K.s_enc_low, s>>>(a);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "encode launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

void free_encode_tables(const fiona_ctx *ctx)
{
    if (ctx->d_enc) cudaFree(ctx->d_enc);
    ctx->d_enc = nullptr;
}
