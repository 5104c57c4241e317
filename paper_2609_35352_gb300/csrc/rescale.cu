// rescale.cu -- the rescale that follows the layer: every output poly is
// divided by the last prime of its level (Sec. 2.2 "Homomorphic Operations":
// a PMult raises the scale and a rescale restores it; Sec. 4.2 "Combining
// the Signed and Raw Routes": one rescale per output).  For a poly y with
// limbs y_0..y_{Lc-1} in NTT form:
//   r    = coefficients of y_{Lc-1}       (inverse NTT mod q_{Lc-1})
//   y'_l = (y_l - NTT_l(r mod q_l)) * q_{Lc-1}^{-1}  mod q_l,   l < Lc-1.
// NTT form: A[k] = a(psi^(2 brv(k) + 1)) mod q, psi the least primitive
// 2N-th root of unity mod q, brv reversing the log2(N) bits of k.
//
// A transform of N = 2^n points is two passes over memory, each a set of
// independent sub-transforms held in shared memory (N = R1 * R2,
// R1 = 2^floor(n/2)):
//   high pass  the radix-2 stages whose butterfly distance is a multiple of
//              R2: for a fixed low index lo, the R1 elements hi * R2 + lo
//              form one sub-transform (a CTA takes tile / R1 of them, loaded
//              as rows of consecutive elements);
//   low pass   the remaining stages, inside blocks of R2 consecutive
//              elements (a CTA takes tile / R2 blocks).
// Forward stages run high then low (Cooley-Tukey: at the stage with m blocks,
// block i uses psi^brv(m + i)); inverse stages low then high
// (Gentleman-Sande with psi^-brv(m + i), then N^-1).  Products by table
// constants use Shoup's method: with w' = floor(w * 2^64 / q), w < q < 2^63,
// x*w - floor(x*w' / 2^64)*q lies in [0, 2q) for any 64-bit x.
// The rescale is four launches on the caller's stream: the two inverse passes
// on the last limb of every poly (in place: it becomes the coefficients r),
// then the two forward passes of every other limb; the first reads r and
// reduces it mod q_l, the second applies the subtraction and the product by
// q_{Lc-1}^{-1}.  The whole last limb must be known before any limb can be
// finished, so the rescale cannot share a launch with the layer's kernels,
// whose CTAs each see one tile of coefficients.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "fiona_internal.h"

namespace {

typedef unsigned __int128 u128;

constexpr uint32_t kTile = 4096;  // elements of one CTA's sub-transforms (32 KB)
constexpr uint32_t kThreads = 256;

// per limb, in device memory (the tables follow the array of these)
struct NttLimb {
    const ulonglong2 *fwd;   // [N]: (psi^brv(k), Shoup companion)
    const ulonglong2 *inv;   // [N]: (psi^-brv(k), Shoup companion)
    const ulonglong2 *qinv;  // [L]: q_j^-1 mod q (Shoup) for j > this limb, else (0, 0)
    uint64_t q;
    uint64_t mu64;           // floor(2^64 / q)
    ulonglong2 ninv;         // N^-1 mod q (Shoup)
};

struct Geo {
    uint32_t N, n, n1;       // N = 2^n, R1 = 2^n1, R2 = 2^(n - n1)
    uint32_t lt;             // log2(tile), tile = min(kTile, N)
    uint32_t ltiles;         // log2(N / tile): tiles per transform
    uint32_t Lc;             // limbs per poly: the level being rescaled
};

__device__ __forceinline__ uint64_t mul_shoup(uint64_t x, ulonglong2 w, uint64_t q)
{
    const uint64_t qh = __umul64hi(x, w.y);
    const uint64_t r = x * w.x - qh * q;
    return r >= q ? r - q : r;
}

__device__ __forceinline__ uint64_t addq(uint64_t a, uint64_t b, uint64_t q)
{
    const uint64_t s = a + b;
    return s >= q ? s - q : s;
}

__device__ __forceinline__ uint64_t subq(uint64_t a, uint64_t b, uint64_t q) { return a >= b ? a - b : a + (q - b); }

// x mod q for any 64-bit x: floor(x * mu64 / 2^64) is floor(x / q) or one less
__device__ __forceinline__ uint64_t reduce_any(uint64_t x, uint64_t q, uint64_t mu64)
{
    const uint64_t r = x - __umul64hi(x, mu64) * q;
    return r >= q ? r - q : r;
}

// ---------------------------------------------------------------------------
// High pass: columns [col0, col0 + C) with C = tile / R1, rows hi < R1; the
// shared layout is s[hi * C + c].  Global stage st (0 <= st < n1) has
// butterfly distance R1 >> (st + 1) rows.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void high_stages(uint64_t *s, const Geo &G, const NttLimb &T, bool inverse)
{
    const uint32_t lC = G.lt - G.n1, half = 1u << (G.lt - 1);
    for (uint32_t i = 0; i < G.n1; ++i) {
        const uint32_t st = inverse ? G.n1 - 1 - i : i;
        const uint32_t lth = G.n1 - 1 - st;  // log2 of the distance in rows
        const uint32_t m = 1u << st;
        __syncthreads();
        for (uint32_t b = threadIdx.x; b < half; b += kThreads) {
            const uint32_t c = b & ((1u << lC) - 1), k = b >> lC;
            const uint32_t hi = ((k >> lth) << (lth + 1)) | (k & ((1u << lth) - 1));
            uint64_t *u = &s[(hi << lC) + c], *v = &s[((hi + (1u << lth)) << lC) + c];
            const uint64_t x = *u;
            if (!inverse) {
                const uint64_t y = mul_shoup(*v, __ldg(&T.fwd[m + (k >> lth)]), T.q);
                *u = addq(x, y, T.q);
                *v = subq(x, y, T.q);
            } else {
                const uint64_t y = *v;
                *u = addq(x, y, T.q);
                *v = mul_shoup(subq(x, y, T.q), __ldg(&T.inv[m + (k >> lth)]), T.q);
            }
        }
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// Low pass: blocks [row0, row0 + B) with B = tile / R2, lo < R2; the shared
// layout is s[r * R2 + lo].  Global stage st (n1 <= st < n) has butterfly
// distance N >> (st + 1) < R2.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void low_stages(uint64_t *s, const Geo &G, uint32_t row0, const NttLimb &T,
                                           bool inverse)
{
    const uint32_t lR2 = G.n - G.n1, half = 1u << (G.lt - 1);
    for (uint32_t i = 0; i < G.n - G.n1; ++i) {
        const uint32_t st = inverse ? G.n - 1 - i : G.n1 + i;
        const uint32_t ld = G.n - 1 - st;  // log2 of the distance
        const uint32_t m = 1u << st;
        __syncthreads();
        for (uint32_t b = threadIdx.x; b < half; b += kThreads) {
            const uint32_t r = b >> (lR2 - 1), k = b & ((1u << (lR2 - 1)) - 1);
            const uint32_t lo = ((k >> ld) << (ld + 1)) | (k & ((1u << ld) - 1));
            const uint32_t blk = (((row0 + r) << lR2) | lo) >> (ld + 1);
            uint64_t *u = &s[(r << lR2) + lo], *v = u + (1u << ld);
            const uint64_t x = *u;
            if (!inverse) {
                const uint64_t y = mul_shoup(*v, __ldg(&T.fwd[m + blk]), T.q);
                *u = addq(x, y, T.q);
                *v = subq(x, y, T.q);
            } else {
                const uint64_t y = *v;
                *u = addq(x, y, T.q);
                *v = mul_shoup(subq(x, y, T.q), __ldg(&T.inv[m + blk]), T.q);
            }
        }
    }
    __syncthreads();
}

// element e of a high-pass tile -> its index in the poly
__device__ __forceinline__ size_t col_index(uint32_t e, const Geo &G, uint32_t col0)
{
    const uint32_t lC = G.lt - G.n1;
    return ((size_t)(e >> lC) << (G.n - G.n1)) + col0 + (e & ((1u << lC) - 1));
}

// ---------------------------------------------------------------------------
// The four launches.  blockIdx.x = transform * tiles + tile; the transforms
// are the polys (inverse passes) or poly * (Lc - 1) + limb (forward passes).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_inv_low(uint64_t *polys, Geo G, const NttLimb *T)
{
    __shared__ uint64_t s[kTile];
    const uint32_t tile = blockIdx.x & ((1u << G.ltiles) - 1);
    const uint64_t p = blockIdx.x >> G.ltiles;
    const uint32_t row0 = tile << (G.lt - (G.n - G.n1));
    uint64_t *g = polys + (p * G.Lc + (G.Lc - 1)) * G.N + ((size_t)tile << G.lt);
    const NttLimb &Tl = T[G.Lc - 1];
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads) s[e] = g[e];
    low_stages(s, G, row0, Tl, true);
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads) g[e] = s[e];
}

__global__ void __launch_bounds__(kThreads) k_inv_high(uint64_t *polys, Geo G, const NttLimb *T)
{
    __shared__ uint64_t s[kTile];
    const uint32_t tile = blockIdx.x & ((1u << G.ltiles) - 1);
    const uint64_t p = blockIdx.x >> G.ltiles;
    const uint32_t col0 = tile << (G.lt - G.n1);
    uint64_t *g = polys + (p * G.Lc + (G.Lc - 1)) * G.N;
    const NttLimb &Tl = T[G.Lc - 1];
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads) s[e] = g[col_index(e, G, col0)];
    high_stages(s, G, Tl, true);
    const ulonglong2 ninv = Tl.ninv;
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads)
        g[col_index(e, G, col0)] = mul_shoup(s[e], ninv, Tl.q);
}

// r (the last limb's coefficients) mod q_l, then the high forward stages, into out
__global__ void __launch_bounds__(kThreads) k_fwd_high(const uint64_t *polys, uint64_t *out, Geo G,
                                                       const NttLimb *T)
{
    __shared__ uint64_t s[kTile];
    const uint32_t tile = blockIdx.x & ((1u << G.ltiles) - 1);
    const uint64_t t = blockIdx.x >> G.ltiles;
    const uint64_t p = t / (G.Lc - 1);
    const uint32_t l = (uint32_t)(t % (G.Lc - 1));
    const uint32_t col0 = tile << (G.lt - G.n1);
    const uint64_t *g = polys + (p * G.Lc + (G.Lc - 1)) * G.N;
    const NttLimb &Tl = T[l];
    const uint64_t q = Tl.q, mu = Tl.mu64;
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads)
        s[e] = reduce_any(g[col_index(e, G, col0)], q, mu);
    high_stages(s, G, Tl, false);
    uint64_t *o = out + t * G.N;
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads) o[col_index(e, G, col0)] = s[e];
}

// the low forward stages, then y' = (y_l - t) * q_{Lc-1}^-1
__global__ void __launch_bounds__(kThreads) k_fwd_low(const uint64_t *polys, uint64_t *out, Geo G,
                                                      const NttLimb *T)
{
    __shared__ uint64_t s[kTile];
    const uint32_t tile = blockIdx.x & ((1u << G.ltiles) - 1);
    const uint64_t t = blockIdx.x >> G.ltiles;
    const uint64_t p = t / (G.Lc - 1);
    const uint32_t l = (uint32_t)(t % (G.Lc - 1));
    const uint32_t row0 = tile << (G.lt - (G.n - G.n1));
    uint64_t *o = out + t * G.N + ((size_t)tile << G.lt);
    const uint64_t *y = polys + (p * G.Lc + l) * G.N + ((size_t)tile << G.lt);
    const NttLimb &Tl = T[l];
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads) s[e] = o[e];
    low_stages(s, G, row0, Tl, false);
    const ulonglong2 qi = Tl.qinv[G.Lc - 1];
    for (uint32_t e = threadIdx.x; e < (1u << G.lt); e += kThreads)
        o[e] = mul_shoup(subq(y[e], s[e], Tl.q), qi, Tl.q);
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

uint32_t bit_reverse(uint32_t k, uint32_t bits)
{
    uint32_t r = 0;
    for (uint32_t b = 0; b < bits; ++b) r = (r << 1) | ((k >> b) & 1u);
    return r;
}

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

int ensure_tables(const fiona_ctx *ctx)
{
    std::lock_guard<std::mutex> lock(g_ntt_mu);
    if (ctx->d_ntt) return FIONA_OK;
    const uint32_t N = ctx->N, L = ctx->L;
    uint32_t n = 0;
    while ((1u << n) < N) ++n;
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

int launch_rescale(const fiona_ctx *ctx, void *stream, uint32_t Lc, uint64_t count, uint64_t *polys, uint64_t *out)
{
    const int rc = ensure_tables(ctx);
    if (rc) return rc;
    if (count == 0) return FIONA_OK;
    Geo G;
    G.N = ctx->N;
    G.n = 0;
    while ((1u << G.n) < G.N) ++G.n;
    G.n1 = G.n / 2;
    G.lt = std::min<uint32_t>(G.n, 12);
    G.ltiles = G.n - G.lt;
    G.Lc = Lc;
    // grid.x < 2^31: transforms * tiles, in chunks of whole polys
    const uint64_t max_polys = ((1ull << 31) - 1) / ((uint64_t)(Lc - 1) << G.ltiles);
    const NttLimb *T = reinterpret_cast<const NttLimb *>(ctx->d_ntt);
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaSuccess;
    for (uint64_t p0 = 0; p0 < count && e == cudaSuccess; p0 += max_polys) {
        const uint64_t np = std::min<uint64_t>(count - p0, max_polys);
        uint64_t *pp = polys + p0 * Lc * (uint64_t)G.N;
        uint64_t *op = out + p0 * (Lc - 1) * (uint64_t)G.N;
        const uint32_t inv_blocks = (uint32_t)(np << G.ltiles);
        const uint32_t fwd_blocks = (uint32_t)((np * (Lc - 1)) << G.ltiles);
        k_inv_low<<<inv_blocks, kThreads, 0, s>>>(pp, G, T);
        k_inv_high<<<inv_blocks, kThreads, 0, s>>>(pp, G, T);
        k_fwd_high<<<fwd_blocks, kThreads, 0, s>>>(pp, op, G, T);
        k_fwd_low<<<fwd_blocks, kThreads, 0, s>>>(pp, op, G, T);
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
