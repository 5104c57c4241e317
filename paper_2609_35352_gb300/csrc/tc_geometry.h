// tc_geometry.h -- layout of one tile's tensor-core signed sums (the
// contraction of tc_signed.cuh), shared by the lowering and the kernel.
//
// K inputs (a multiple of 16: the contraction's steps; rows of W past the
// layer's inputs are zero), N groups (a multiple of 8, at most 256).  In
// tensor memory chunk j of the inputs (A_j, fp16 pairs: K/2 columns) sits
// at columns a_col(j), the product D_j = A_j W (fp32: N columns) at
// d_col(j); cols() columns in all.  W sits in shared memory as K-major core
// matrices of 8 rows x 16 bytes without swizzle: core matrix (n / 8, k / 8)
// at byte (n / 8) * sbo() + (k / 8) * 128, w_bytes() bytes.
#pragma once
#include <stdint.h>

#if defined(__CUDACC__)
#define TC_HD __host__ __device__
#else
#define TC_HD
#endif

constexpr uint32_t kTcChunks = 5;  // 10-bit chunks of a residue below 2^50

struct TcGeometry {
    uint32_t K, N;
    TC_HD constexpr uint32_t a_col(uint32_t j) const { return j * (K / 2); }
    TC_HD constexpr uint32_t d_base() const { return (kTcChunks * (K / 2) + 15) & ~15u; }
    TC_HD constexpr uint32_t d_col(uint32_t j) const { return d_base() + j * ((N + 15) & ~15u); }
    TC_HD constexpr uint32_t cols() const { return d_col(kTcChunks); }
    TC_HD constexpr uint32_t sbo() const { return (K / 8) * 128; }
    TC_HD constexpr uint32_t w_bytes() const { return N * K * 2; }
};
