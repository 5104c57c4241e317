// kernel_tiled.cu -- tiled, shared-memory-staged evaluation (not yet built;
// every plan uses the direct kernel).
#include "fiona_internal.h"

int lower_tiled(fiona_plan *) { return FIONA_ERR_ARG; }
void free_tiled(fiona_plan *) {}
int launch_tiled(const fiona_plan *, void *, const uint64_t *, const uint64_t *, uint64_t *,
                 uint32_t, uint32_t)
{
    return set_error(FIONA_ERR_ARG, "tiled kernel not available");
}
