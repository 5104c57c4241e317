// rescale.cu -- the rescale that follows the layer: every output poly is
// divided by the last prime of its level (Sec. 2.2 "Homomorphic Operations":
// a PMult raises the scale and a rescale restores it; Sec. 4.2 "Combining
// the Signed and Raw Routes": one rescale per output).  For a poly y with
// limbs y_0..y_{Lc-1} in NTT form:
//   r    = coefficients of y_{Lc-1}       (inverse NTT mod q_{Lc-1})
//   y'_l = (y_l - NTT_l(r mod q_l)) * q_{Lc-1}^{-1}  mod q_l,   l < Lc-1,
// the quotient of the CRT value Y by q_{Lc-1} rounded down; rounded to the
// nearest (the variant that adds h = floor(q_{Lc-1} / 2) to Y), r becomes
// r' = (r + h) mod q_{Lc-1} and the subtracted poly r' - h (mod q_l).
// NTT form: A[k] = a(psi^(2 brv(k) + 1)) mod q, psi the least primitive
// 2N-th root of unity mod q (the transform and its passes: ntt.cuh).
//
// The rescale is four launches on the caller's stream: the two inverse passes
// on the last limb of every poly (in place: it becomes the coefficients r,
// canonical), then the two forward passes of every other limb; the first
// reads r and reduces it mod q_l (unless r < 4 q_l already, with every
// q_l < 2^56: then the reduction-free butterflies take it as it is), the
// second applies the subtraction and the product by q_{Lc-1}^{-1}.  The whole
// last limb must be known before any limb can be finished, so the rescale
// cannot share a launch with the layer's kernels, whose CTAs each see one
// tile of coefficients.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "fiona_internal.h"
#include "ntt.cuh"

using namespace fiona_ntt;

namespace {

typedef unsigned __int128 u128;

struct Args {
    uint64_t *polys;   // [count][Lc][N]
    uint64_t *out;     // [count][Lc-1][N]
    const NttLimb *T;
    uint32_t Lc;
    uint32_t round;    // 1: nearest quotient (add h = floor(q_{Lc-1} / 2))
};

// ---------------------------------------------------------------------------
// The four launches.  blockIdx.x = transform * tiles + tile; the transforms
// are the polys (inverse passes) or poly * (Lc - 1) + limb (forward passes).
// ---------------------------------------------------------------------------

// inverse, low stages, on the last limb in place
template <int LOGN>
__global__ void __launch_bounds__(LowPass<LOGN>::threads, 4) k_inv_low(Args A)
{
    using SH = Shape<LOGN>;
    using PS = LowPass<LOGN>;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), p = blockIdx.x >> PS::ltiles;
    const uint32_t first = tile << PS::lsubs;
    uint64_t *g = A.polys + ((size_t)p * A.Lc + (A.Lc - 1)) * (1u << LOGN) + ((size_t)first << PS::s);
    const NttLimb &Tl = A.T[A.Lc - 1];
    inv_low_pass<LOGN>(smem_raw, Tl.inv, first, ModArith<false>{Tl.q}, [&](uint32_t e) { return g[e]; },
                       [&](uint32_t sub, uint32_t pos, uint64_t v) { g[(sub << PS::s) + pos] = v; });
}

// inverse, high stages: stores r = N^-1 x, canonical
template <int LOGN>
__global__ void __launch_bounds__(HighPass<LOGN>::threads, 3) k_inv_high(Args A)
{
    using SH = Shape<LOGN>;
    using PS = HighPass<LOGN>;
    constexpr uint32_t R2 = 1u << (LOGN - SH::n1);
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), p = blockIdx.x >> PS::ltiles;
    const uint32_t first = tile << PS::lsubs;
    uint64_t *g = A.polys + ((size_t)p * A.Lc + (A.Lc - 1)) * (1u << LOGN) + first;
    const NttLimb &Tl = A.T[A.Lc - 1];
    const uint64_t q = Tl.q;
    const ulonglong2 ninv = Tl.ninv;
    const uint64_t h = A.round ? q / 2 : 0;
    inv_high_pass<LOGN>(smem_raw, Tl.inv, first, ModArith<false>{q},
                        [&](uint32_t sub, uint32_t pos) { return g[(size_t)pos * R2 + sub]; },
                        [&](uint32_t sub, uint32_t pos, uint64_t v) {
                            g[(size_t)pos * R2 + sub] = csub(canon4(mul_shoup_lazy(v, ninv, q), q) + h, q);
                        });
}

// forward, high stages: r (the last limb's coefficients), reduced mod q_l
// unless FAST, into out
template <int LOGN, bool FAST>
__global__ void __launch_bounds__(HighPass<LOGN>::threads, 3) k_fwd_high(Args A)
{
    using SH = Shape<LOGN>;
    using PS = HighPass<LOGN>;
    constexpr uint32_t R2 = 1u << (LOGN - SH::n1);
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), tr = blockIdx.x >> PS::ltiles;
    const uint32_t p = tr / (A.Lc - 1), l = tr % (A.Lc - 1);
    const uint32_t first = tile << PS::lsubs;
    const uint64_t *g = A.polys + ((size_t)p * A.Lc + (A.Lc - 1)) * (1u << LOGN) + first;
    uint64_t *o = A.out + (size_t)tr * (1u << LOGN) + first;
    const NttLimb &Tl = A.T[l];
    const uint64_t q = Tl.q, mu = Tl.mu64;
    // rounding: subtract h mod q_l, as + (q_l - h mod q_l); the loaded value
    // then stays below 5 q_l (FAST) or 2 q_l
    const uint64_t hq = A.round ? q - reduce_any(A.T[A.Lc - 1].q / 2, q, mu) : 0;
    fwd_high_pass<LOGN>(
        smem_raw, Tl.fwd, first, ModArith<FAST>{q},
        [&](uint32_t sub, uint32_t pos) {
            const uint64_t v = g[(size_t)pos * R2 + sub];
            return (FAST ? v : reduce_any(v, q, mu)) + hq;
        },
        [&](uint32_t sub, uint32_t pos, uint64_t v) { o[(size_t)pos * R2 + sub] = v; });
}

// forward, low stages, then y' = (y_l - t) * q_{Lc-1}^-1
template <int LOGN, bool FAST>
__global__ void __launch_bounds__(LowPass<LOGN>::threads, 4) k_fwd_low(Args A)
{
    using SH = Shape<LOGN>;
    using PS = LowPass<LOGN>;
    extern __shared__ __align__(16) uint8_t smem_raw[];
    const uint32_t tile = blockIdx.x & ((1u << PS::ltiles) - 1), tr = blockIdx.x >> PS::ltiles;
    const uint32_t p = tr / (A.Lc - 1), l = tr % (A.Lc - 1);
    const uint32_t first = tile << PS::lsubs;
    uint64_t *o = A.out + (size_t)tr * (1u << LOGN) + ((size_t)first << PS::s);
    const uint64_t *y = A.polys + ((size_t)p * A.Lc + l) * (1u << LOGN) + ((size_t)first << PS::s);
    const NttLimb &Tl = A.T[l];
    const uint64_t q = Tl.q;
    const ulonglong2 qi = Tl.qinv[A.Lc - 1];
    // transform values: below 73q (FAST) or 8q; M = 128q or 8q bounds them
    const uint64_t M = (FAST ? 128 : 8) * q;
    fwd_low_pass<LOGN>(
        smem_raw, Tl.fwd, first, ModArith<FAST>{q},
        [&] {
            // y is read only by the epilogue: start bringing it into L2 now
            for (uint32_t e = threadIdx.x * 16; e < PS::tile; e += PS::threads * 16)
                asm volatile("prefetch.global.L2 [%0];\n" ::"l"(y + e));
        },
        [&](uint32_t sub, uint32_t pos) { return o[(sub << PS::s) + pos]; },
        [&](auto t_of) {
            sweep<PS, uint64_t>([&](uint32_t e) { return y[e]; },
                                [&](uint32_t e, uint64_t v) { o[e] = canon4(mul_shoup_lazy(v + M - t_of(e), qi, q), q); });
        });
}

// ---------------------------------------------------------------------------
// Host: tables, built once per context on its first rescale
// ---------------------------------------------------------------------------
uint64_t mulm(uint64_t a, uint64_t b, uint64_t q) { return (uint64_t)((u128)a * b % q); }

uint64_t powm(uint64_t b, uint64_t e, uint64_t q)
{
    uint64_t r = 1 % q;
    b %= q;
    for (; e; e >>= 1) {
        if (e & 1) r = mulm(r, b, q);
        b = mulm(b, b, q);
    }
    return r;
}

ulonglong2 shoup(uint64_t w, uint64_t q) { return make_ulonglong2(w, (uint64_t)(((u128)w << 64) / q)); }

// The least primitive 2N-th root of unity mod q, or 0.  For the first x whose
// c = x^((q-1)/2N) has c^N = -1, c is primitive and the primitive roots are
// its odd powers; the least of them is returned.
uint64_t least_root(uint64_t q, uint32_t N)
{
    const uint64_t M = 2ull * N;
    if ((q - 1) % M) return 0;
    uint64_t g = 0;
    for (uint64_t x = 2; x < 1000000 && x < q; ++x) {
        const uint64_t c = powm(x, (q - 1) / M, q);
        if (powm(c, N, q) == q - 1) {
            g = c;
            break;
        }
    }
    if (!g) return 0;
    const uint64_t g2 = mulm(g, g, q);
    uint64_t best = g, cur = g;
    for (uint32_t j = 1; j < N; ++j) {
        cur = mulm(cur, g2, q);
        best = std::min(best, cur);
    }
    return best;
}

std::mutex g_ntt_mu;

int build_tables(const fiona_ctx *ctx)
{
    std::lock_guard<std::mutex> lock(g_ntt_mu);
    if (ctx->d_ntt) return FIONA_OK;
    const uint32_t N = ctx->N, L = ctx->L;
    const uint32_t n = log2u(N);
    const size_t head = ((sizeof(NttLimb) * L + 255) / 256) * 256;
    const size_t table = sizeof(ulonglong2) * N, qtab = sizeof(ulonglong2) * L;
    const size_t per_limb = 2 * table + ((qtab + 255) / 256) * 256;
    const size_t bytes = head + per_limb * L;
    std::vector<uint8_t> host(bytes, 0);
    std::vector<uint64_t> pw(N);
    void *dev = nullptr;
    cudaError_t e = cudaMalloc(&dev, bytes);
    if (e != cudaSuccess) return set_error(FIONA_ERR_NOMEM, "rescale tables: %s", cudaGetErrorString(e));
    for (uint32_t l = 0; l < L; ++l) {
        const uint64_t q = ctx->moduli[l];
        const uint64_t psi = least_root(q, N);
        if (!psi) {
            cudaFree(dev);
            return set_error(FIONA_ERR_MODULUS, "rescale: modulus %u has no primitive 2N-th root of unity", l);
        }
        const size_t off = head + per_limb * l;
        ulonglong2 *fwd = reinterpret_cast<ulonglong2 *>(host.data() + off);
        ulonglong2 *inv = reinterpret_cast<ulonglong2 *>(host.data() + off + table);
        ulonglong2 *qinv = reinterpret_cast<ulonglong2 *>(host.data() + off + 2 * table);
        // powers of psi, then of psi^-1, placed in bit-reversed order
        for (int dir = 0; dir < 2; ++dir) {
            const uint64_t base = dir == 0 ? psi : powm(psi, q - 2, q);
            pw[0] = 1;
            for (uint32_t i = 1; i < N; ++i) pw[i] = mulm(pw[i - 1], base, q);
            ulonglong2 *dst = dir == 0 ? fwd : inv;
            for (uint32_t k = 0; k < N; ++k) dst[k] = shoup(pw[bit_reverse(k, n)], q);
        }
        for (uint32_t j = l + 1; j < L; ++j) qinv[j] = shoup(powm(ctx->moduli[j] % q, q - 2, q), q);
        NttLimb &T = reinterpret_cast<NttLimb *>(host.data())[l];
        const uint8_t *dbase = static_cast<const uint8_t *>(dev) + off;
        T.fwd = reinterpret_cast<const ulonglong2 *>(dbase);
        T.inv = reinterpret_cast<const ulonglong2 *>(dbase + table);
        T.qinv = reinterpret_cast<const ulonglong2 *>(dbase + 2 * table);
        T.q = q;
        T.mu64 = ~(uint64_t)0 / q;
        T.ninv = shoup(powm(N % q, q - 2, q), q);
    }
    e = cudaMemcpy(dev, host.data(), bytes, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        cudaFree(dev);
        return set_error(FIONA_ERR_CUDA, "rescale tables: %s", cudaGetErrorString(e));
    }
    ctx->d_ntt = dev;
    return FIONA_OK;
}

}  // namespace

int ntt_tables(const fiona_ctx *ctx, const fiona_ntt::NttLimb **limbs)
{
    const int rc = build_tables(ctx);
    if (rc == FIONA_OK) *limbs = reinterpret_cast<const NttLimb *>(ctx->d_ntt);
    return rc;
}

int launch_rescale(const fiona_ctx *ctx, void *stream, uint32_t Lc, uint64_t count, uint64_t *polys, uint64_t *out,
                   bool round)
{
    const NttLimb *T = nullptr;
    const int rc = ntt_tables(ctx, &T);
    if (rc) return rc;
    if (count == 0) return FIONA_OK;
    const uint32_t n = log2u(ctx->N);
    if (n < (uint32_t)kLogNMin || n > (uint32_t)kLogNMax)
        return set_error(FIONA_ERR_ARG, "rescale: N = %u outside [2^%d, 2^%d]", ctx->N, kLogNMin, kLogNMax);
    // the reduction-free forward butterflies need q < 2^56 and r < 4 q_l
    bool fast = true;
    const uint64_t qlast = ctx->moduli[Lc - 1];
    for (uint32_t l = 0; l + 1 < Lc; ++l)
        if (ctx->moduli[l] >= (1ull << 56) || qlast >= 4 * ctx->moduli[l]) fast = false;
    const int ix = (int)n - kLogNMin;
    typedef void (*Kern)(Args);
    static const Kern inv_low[] = {k_inv_low<10>, k_inv_low<11>, k_inv_low<12>, k_inv_low<13>,
                                   k_inv_low<14>, k_inv_low<15>, k_inv_low<16>, k_inv_low<17>};
    static const Kern inv_high[] = {k_inv_high<10>, k_inv_high<11>, k_inv_high<12>, k_inv_high<13>,
                                    k_inv_high<14>, k_inv_high<15>, k_inv_high<16>, k_inv_high<17>};
    static const Kern fwd_high[2][8] = {
        {k_fwd_high<10, false>, k_fwd_high<11, false>, k_fwd_high<12, false>, k_fwd_high<13, false>,
         k_fwd_high<14, false>, k_fwd_high<15, false>, k_fwd_high<16, false>, k_fwd_high<17, false>},
        {k_fwd_high<10, true>, k_fwd_high<11, true>, k_fwd_high<12, true>, k_fwd_high<13, true>,
         k_fwd_high<14, true>, k_fwd_high<15, true>, k_fwd_high<16, true>, k_fwd_high<17, true>}};
    static const Kern fwd_low[2][8] = {
        {k_fwd_low<10, false>, k_fwd_low<11, false>, k_fwd_low<12, false>, k_fwd_low<13, false>,
         k_fwd_low<14, false>, k_fwd_low<15, false>, k_fwd_low<16, false>, k_fwd_low<17, false>},
        {k_fwd_low<10, true>, k_fwd_low<11, true>, k_fwd_low<12, true>, k_fwd_low<13, true>,
         k_fwd_low<14, true>, k_fwd_low<15, true>, k_fwd_low<16, true>, k_fwd_low<17, true>}};
    // per pass: tiles per transform (log2) and threads per CTA
#define FIONA_GEO(P) {P<10>::ltiles, P<11>::ltiles, P<12>::ltiles, P<13>::ltiles, P<14>::ltiles, P<15>::ltiles, P<16>::ltiles, P<17>::ltiles}
#define FIONA_THR(P) {P<10>::threads, P<11>::threads, P<12>::threads, P<13>::threads, P<14>::threads, P<15>::threads, P<16>::threads, P<17>::threads}
    static const int low_lt[] = FIONA_GEO(LowPass), high_lt[] = FIONA_GEO(HighPass);
    static const uint32_t low_thr[] = FIONA_THR(LowPass), high_thr[] = FIONA_THR(HighPass);
#undef FIONA_GEO
#undef FIONA_THR
    const uint32_t lt_low = (uint32_t)low_lt[ix], lt_high = (uint32_t)high_lt[ix];
    const Kern ks[4] = {inv_low[ix], inv_high[ix], fwd_high[fast][ix], fwd_low[fast][ix]};
    typedef ModArith<false> MA;
    static const size_t low_smem[] = {
        LowPass<10>::smem_bytes<MA>(), LowPass<11>::smem_bytes<MA>(), LowPass<12>::smem_bytes<MA>(),
        LowPass<13>::smem_bytes<MA>(), LowPass<14>::smem_bytes<MA>(), LowPass<15>::smem_bytes<MA>(),
        LowPass<16>::smem_bytes<MA>(), LowPass<17>::smem_bytes<MA>()};
    static const size_t high_smem[] = {
        HighPass<10>::smem_bytes<MA>(), HighPass<11>::smem_bytes<MA>(), HighPass<12>::smem_bytes<MA>(),
        HighPass<13>::smem_bytes<MA>(), HighPass<14>::smem_bytes<MA>(), HighPass<15>::smem_bytes<MA>(),
        HighPass<16>::smem_bytes<MA>(), HighPass<17>::smem_bytes<MA>()};
    const size_t smem[4] = {low_smem[ix], high_smem[ix], high_smem[ix], low_smem[ix]};
    cudaError_t e = cudaSuccess;
    {
        // the dynamic shared memory limit, once per device and kernel
        static bool configured[FIONA_MAX_DEVICES][kLogNMax - kLogNMin + 1][2] = {};
        std::lock_guard<std::mutex> lock(g_ntt_mu);
        if (ctx->device < 0 || ctx->device >= FIONA_MAX_DEVICES)
            return set_error(FIONA_ERR_ARG, "rescale: device %d", ctx->device);
        if (!configured[ctx->device][ix][fast]) {
            for (int i = 0; i < 4 && e == cudaSuccess; ++i)
                e = cudaFuncSetAttribute((const void *)ks[i], cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem[i]);
            if (e != cudaSuccess)
                return set_error(FIONA_ERR_CUDA, "rescale: kernel attributes: %s", cudaGetErrorString(e));
            configured[ctx->device][ix][fast] = true;
        }
    }
    // grid.x < 2^31: transforms * tiles, in chunks of whole polys
    const uint64_t max_polys = ((1ull << 31) - 1) / ((uint64_t)(Lc - 1) << std::max(lt_low, lt_high));
    cudaStream_t s = (cudaStream_t)stream;
    for (uint64_t p0 = 0; p0 < count && e == cudaSuccess; p0 += max_polys) {
        const uint64_t np = std::min<uint64_t>(count - p0, max_polys);
        Args a;
        a.polys = polys + p0 * Lc * (uint64_t)ctx->N;
        a.out = out + p0 * (Lc - 1) * (uint64_t)ctx->N;
        a.T = T;
        a.Lc = Lc;
        a.round = round ? 1 : 0;
        const uint64_t nf = np * (Lc - 1);
        ks[0]<<<(uint32_t)(np << lt_low), low_thr[ix], smem[0], s>>>(a);
        ks[1]<<<(uint32_t)(np << lt_high), high_thr[ix], smem[1], s>>>(a);
        ks[2]<<<(uint32_t)(nf << lt_high), high_thr[ix], smem[2], s>>>(a);
        ks[3]<<<(uint32_t)(nf << lt_low), low_thr[ix], smem[3], s>>>(a);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "rescale launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

void free_rescale_tables(const fiona_ctx *ctx)
{
    if (ctx->d_ntt) cudaFree(ctx->d_ntt);
    ctx->d_ntt = nullptr;
}
