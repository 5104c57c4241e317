// tiled.h -- schedule of the tiled kernel (shared by lower_tiled.cpp and
// kernel_tiled.cu).
//
// One CTA evaluates every output of the layer on one limb and one tile of
// T = 32*C coefficients (C = 1 or 2 coefficients per lane).  Operand space in
// shared memory: sources [0, n_in) are the input tiles, [n_in, n_in+n_nodes)
// the shared signed sums.  Each warp runs a list of jobs; a job is one output
// (or one part of an output split across warps), made of scale-group
// segments (a signed sum over sources, then one product by gamma) and raw
// terms (PMult-MAC).
#pragma once
#include <stdint.h>
#include <vector_types.h>

#include "fiona_internal.h"

constexpr uint32_t kTiledMaxWarps = 16;
constexpr uint32_t kPartBit = 0x80000000u;  // TiledJob::target: partial slot
constexpr uint32_t kNegBit = 0x80000000u;   // op word: subtract the source
constexpr uint32_t kSchedPad = 32;          // zero words after each schedule array

struct TiledJob {
    uint32_t target;  // output index, or kPartBit | partial slot
    uint32_t seg_begin, seg_end;
    uint32_t raw_begin, raw_end;
    uint32_t pad[3];
};

struct TiledSeg {
    uint32_t scale_pt;
    uint32_t op_begin, op_end;
    uint32_t pad;
};

struct TiledArgs {
    const uint64_t *in;
    const uint64_t *pt;
    uint64_t *out;
    const LimbConst *limbs;
    const uint32_t *node_level_off;  // [n_levels + 1] into node_slots
    const uint32_t *node_slots;      // node slot ids, grouped by level
    const uint32_t *node_op_off;     // [2 * n_nodes]: begin, end per node slot
    const uint32_t *node_ops;        // source | kNegBit; each node's list 16-byte aligned
    const uint32_t *warp_job_off;    // [kTiledWarps + 1]
    const TiledJob *jobs;
    const TiledSeg *segs;
    const uint32_t *ops;             // source | kNegBit; each segment 16-byte aligned
    const uint2 *raws;               // (plaintext, input) per raw term; each job 16-byte aligned
    const uint32_t *comb_off;        // [n_comb + 1] into comb_parts
    const uint32_t *comb_out;        // output of each combine
    const uint32_t *comb_parts;      // partial slots to add
    int *err;                        // set to 1 when a bounded wait gives up
    uint32_t N, L, limb0;
    uint32_t n_in, n_nodes, n_levels, n_part, n_comb;
    uint32_t mac_budget;     // products per 128-bit accumulator (generic arithmetic)
    uint32_t signed_budget;  // residues per 64-bit signed sum (generic arithmetic)
};

struct TiledSchedule {
    int C = 2;                 // coefficients per lane
    bool narrow = false;       // every modulus < 2^52: radix-2^26 arithmetic
    uint32_t warps = 8;        // warps per CTA
    uint32_t tile = 64;        // coefficients per CTA
    size_t smem = 0;           // dynamic shared memory per CTA
    uint32_t ctas_per_sm = 0;  // shared-memory occupancy
    DeviceSchedule sched;
    TiledArgs args{};          // device pointers into sched.blob (data pointers unset)
};
