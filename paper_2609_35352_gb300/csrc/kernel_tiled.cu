// kernel_tiled.cu -- launch of the tiled evaluation kernel (tiled_kernel.cuh)
// and its variants with packed signed-sum programs; the variants whose
// programs are in the offset form are built in kernel_tiled_off.cu, those
// for CTAs of at most 12 warps in kernel_tiled_w12.cu.
#include "tiled_kernel.cuh"

// kernel_tiled_off.cu: the variant with programs in the offset form, or null
void *tiled_select_offsets(int C, bool narrow, uint32_t P, bool kc);
// kernel_tiled_w12.cu: the 12-warp variants (two coefficients per lane,
// narrow moduli, batches of 8)
void *tiled_select_w12(bool kc, bool off, bool ka);

namespace {

template <uint32_t P, bool KC>
void *select_ptr_p(int C, bool narrow)
{
    if (C == 2)
        return narrow ? reinterpret_cast<void *>(&tiled_kernel<2, true, P, KC>)
                      : reinterpret_cast<void *>(&tiled_kernel<2, false, P, KC>);
    return narrow ? reinterpret_cast<void *>(&tiled_kernel<1, true, P, KC>)
                  : reinterpret_cast<void *>(&tiled_kernel<1, false, P, KC>);
}

// batches of 16: one coefficient per lane only
template <bool KC>
void *select_ptr_16(int C, bool narrow)
{
    if (C != 1) return nullptr;
    return narrow ? reinterpret_cast<void *>(&tiled_kernel<1, true, 16, KC>)
                  : reinterpret_cast<void *>(&tiled_kernel<1, false, 16, KC>);
}

// KC: the variant that reads constant plaintexts (operations marked kOpConst);
// TC: the signed sums on the tensor cores (one coefficient per lane, narrow
// moduli, batches of 16); off: signed-sum programs in the offset form; w12:
// the variant for CTAs of at most 12 warps; ka: every raw plaintext constant
void *select_ptr(int C, bool narrow, uint32_t P, bool kc, bool tc = false, bool off = false, bool w12 = false,
                 bool ka = false)
{
    if (w12) return C == 2 && narrow && P == 8 && !tc ? tiled_select_w12(kc, off, ka) : nullptr;
    if (ka) return nullptr;  // (built for the 12-warp shape only)
    if (off) return tc ? nullptr : tiled_select_offsets(C, narrow, P, kc);
    if (tc) {
        if (C != 1 || !narrow || P != 16) return nullptr;
        return kc ? reinterpret_cast<void *>(&tiled_kernel<1, true, 16, true, true>)
                  : reinterpret_cast<void *>(&tiled_kernel<1, true, 16, false, true>);
    }
    if (P == 16) return kc ? select_ptr_16<true>(C, narrow) : select_ptr_16<false>(C, narrow);
    if (kc) return P == 4 ? select_ptr_p<4, true>(C, narrow) : select_ptr_p<8, true>(C, narrow);
    return P == 4 ? select_ptr_p<4, false>(C, narrow) : select_ptr_p<8, false>(C, narrow);
}

}  // namespace

int tiled_kernel_attributes(int C, bool narrow, uint32_t P, bool kc, bool tc, cudaFuncAttributes *attr, bool off,
                            bool w12, bool ka)
{
    if (!select_ptr(C, narrow, P, kc, tc, off, w12, ka))
        return set_error(FIONA_ERR_ARG, "tiled kernel: no variant with C=%d, P=%u", C, P);
    cudaError_t e = cudaFuncGetAttributes(attr, select_ptr(C, narrow, P, kc, tc, off, w12, ka));
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel attributes: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int tiled_configure_kernel(int C, bool narrow, uint32_t P, bool kc, bool tc, size_t smem, bool off, bool w12,
                           bool ka)
{
    if (!select_ptr(C, narrow, P, kc, tc, off, w12, ka))
        return set_error(FIONA_ERR_ARG, "tiled kernel: no variant with C=%d, P=%u", C, P);
    cudaError_t e = cudaFuncSetAttribute(select_ptr(C, narrow, P, kc, tc, off, w12, ka),
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel attribute: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

namespace {
// cuTensorMapEncodeTiled, from the driver the runtime uses (no link to it)
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    });
    return fn;
}
}  // namespace

// The inputs [n_in][2][L][N] as a 3-D tensor (coefficient, limb, poly) with
// boxes of T coefficients, one limb and `box_rows` polys.
int input_tensor_map(uint32_t N, uint32_t layout_L, uint32_t n_in, uint32_t T, uint32_t box_rows,
                     const uint64_t *in, CUtensorMap *tm)
{
    memset(tm, 0, sizeof(*tm));
    if (!n_in) return FIONA_OK;
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (!enc) return set_error(FIONA_ERR_CUDA, "tiled kernel: cuTensorMapEncodeTiled is not available");
    const cuuint64_t dims[3] = {N, layout_L, 2ull * n_in};
    const cuuint64_t strides[2] = {(cuuint64_t)N * 8, (cuuint64_t)layout_L * N * 8};
    const cuuint32_t box[3] = {T, 1, box_rows};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_UINT64, 3, const_cast<uint64_t *>(in), dims, strides, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return set_error(FIONA_ERR_CUDA, "tiled kernel: input tensor map (error %d)", (int)r);
    return FIONA_OK;
}

// kernel_ws.cu
int launch_ws(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt, uint64_t *out, uint32_t l0,
              uint32_t l1, uint32_t layout_L);

int launch_tiled(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                 uint64_t *out, uint32_t l0, uint32_t l1, uint32_t layout_L)
{
    const TiledSchedule *ts = p->tiled;
    if (!ts) return set_error(FIONA_ERR_ARG, "tiled kernel not available for this plan");
    if (ts->ws) return launch_ws(p, stream, in, pt, out, l0, l1, layout_L);
    if (l1 <= l0) return FIONA_OK;
    TiledArgs a = ts->args;
    a.in = in;
    a.pt = pt;
    a.out = out;
    a.limb0 = l0;
    a.n_limbs = l1 - l0;
    a.L = layout_L;
    a.pt_stride = layout_L * a.N;
    const uint32_t tiles = a.n_limbs * a.tiles_per_limb;
    const uint32_t resident = ts->ctas_per_sm * (uint32_t)std::max(p->ctx->sm_count, 1);
    dim3 grid(std::min(tiles, resident));
    dim3 block(ts->warps * 32);
    cudaStream_t s = (cudaStream_t)stream;
    void *fn = select_ptr(ts->C, ts->narrow, ts->batch, ts->has_const, ts->tc, a.src_offsets != 0, ts->w12,
                          a.kc_all != 0);
    if (!fn) return set_error(FIONA_ERR_INTERNAL, "tiled kernel: no variant for the schedule's shape");
    CUtensorMap tm;  // read by the kernels with one coefficient per lane only
    memset(&tm, 0, sizeof(tm));
    if (ts->C == 1)
        if (const int rc = input_tensor_map(a.N, layout_L, a.n_in, ts->tile, a.box_rows, in, &tm)) return rc;
    void *args[] = {&a, &tm};
    cudaError_t e = cudaLaunchKernel(fn, grid, block, args, ts->smem, s);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}
