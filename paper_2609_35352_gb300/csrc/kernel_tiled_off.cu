// kernel_tiled_off.cu -- the tiled kernel's variants whose signed-sum
// programs are in the offset form (tiled.h), in a translation unit of their
// own so that both sets build in parallel.
#include "tiled_kernel.cuh"

namespace {

template <uint32_t P, bool KC>
void *select_p(int C, bool narrow)
{
    if (C == 2)
        return narrow ? reinterpret_cast<void *>(&tiled_kernel<2, true, P, KC, false, true>)
                      : reinterpret_cast<void *>(&tiled_kernel<2, false, P, KC, false, true>);
    return narrow ? reinterpret_cast<void *>(&tiled_kernel<1, true, P, KC, false, true>)
                  : reinterpret_cast<void *>(&tiled_kernel<1, false, P, KC, false, true>);
}

template <bool KC>
void *select_16(int C, bool narrow)
{
    if (C != 1) return nullptr;
    return narrow ? reinterpret_cast<void *>(&tiled_kernel<1, true, 16, KC, false, true>)
                  : reinterpret_cast<void *>(&tiled_kernel<1, false, 16, KC, false, true>);
}

}  // namespace

void *tiled_select_offsets(int C, bool narrow, uint32_t P, bool kc)
{
    if (P == 16) return kc ? select_16<true>(C, narrow) : select_16<false>(C, narrow);
    if (P != 4 && P != 8) return nullptr;
    if (kc) return P == 4 ? select_p<4, true>(C, narrow) : select_p<8, true>(C, narrow);
    return P == 4 ? select_p<4, false>(C, narrow) : select_p<8, false>(C, narrow);
}
