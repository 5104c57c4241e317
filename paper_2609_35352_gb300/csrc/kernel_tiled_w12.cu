// kernel_tiled_w12.cu -- the tiled kernel's variants with two coefficients
// per lane, narrow moduli and 8-deep plaintext queues for CTAs of at most 12
// warps (up to 168 registers a thread instead of 128: measured on the BERT
// layer, 12 warps with 8 plaintext tiles in flight each beat 16 warps with 4),
// in a translation unit of their own so that the variant sets build in
// parallel; with constant plaintexts also the variant for plans whose every
// raw plaintext is constant.
#include "tiled_kernel.cuh"

void *tiled_select_w12(bool kc, bool off, bool ka)
{
    if (ka)  // every raw plaintext constant (bert-const-like layers)
        return !kc ? nullptr
               : off ? reinterpret_cast<void *>(&tiled_kernel<2, true, 8, true, false, true, 12, true>)
                     : reinterpret_cast<void *>(&tiled_kernel<2, true, 8, true, false, false, 12, true>);
    if (off)
        return kc ? reinterpret_cast<void *>(&tiled_kernel<2, true, 8, true, false, true, 12>)
                  : reinterpret_cast<void *>(&tiled_kernel<2, true, 8, false, false, true, 12>);
    return kc ? reinterpret_cast<void *>(&tiled_kernel<2, true, 8, true, false, false, 12>)
              : reinterpret_cast<void *>(&tiled_kernel<2, true, 8, false, false, false, 12>);
}
