// tiled.h -- schedule of the tiled kernel (shared by lower_tiled.cpp and
// kernel_tiled.cu).
//
// A persistent CTA walks the (limb, coefficient tile) pairs.  For each it
// holds, in shared memory, the tile of every input and of every shared
// signed sum ("sources"), plus one all-zero tile used as padding.  Each warp
// runs a list of jobs; a job is one output (or one part of an output split
// across warps), made of scale-group segments (a signed sum over sources,
// then one product by gamma) and raw terms (PMult-MAC).
//
// Encodings (all offsets precomputed by the lowering, so the kernel does no
// multiplications on addresses):
//   op word   byte offset of a source tile inside the source region
//   segment   gamma's plaintext index times L, then a run of plus words and
//             a run of minus words, each at most `sum_budget` long (longer
//             sums are split into several segments with the same gamma:
//             exact, since gamma*S1 + gamma*S2 = gamma*(S1+S2) mod q)
//   raw term  (plaintext index times L, byte offset of the input tile)
// A warp reads a job's words lane-parallel (word i in lane i) and broadcasts
// them with shuffles, so a job costs a few coalesced loads, not one
// dependent load per term.
#pragma once
#include <stdint.h>
#include <vector_types.h>

#include "fiona_internal.h"

constexpr uint32_t kTiledMaxWarps = 16;
constexpr uint32_t kPartBit = 0x80000000u;  // TiledJob::target: partial slot
constexpr uint32_t kSchedPad = 64;          // zero words after each schedule array

struct TiledJob {
    uint32_t target;  // output index, or kPartBit | partial slot
    uint32_t seg_begin, seg_end;
    uint32_t raw_begin, raw_end;  // in raw terms (8 bytes each)
    uint32_t pad[3];
};

struct TiledSeg {
    uint32_t gamma_ptl;  // plaintext index * L (unused for shared sums)
    uint32_t op_begin;   // index into ops
    uint16_t n_plus;     // plus words
    uint16_t n_minus;    // minus words (they follow the plus words)
    uint32_t pad;
};

struct TiledArgs {
    const uint64_t *in;
    const uint64_t *pt;
    uint64_t *out;
    const LimbConst *limbs;
    const uint32_t *node_level_off;  // [n_levels + 1] into node_slots
    const uint32_t *node_slots;      // node slot ids, grouped by level
    const TiledSeg *node_segs;       // per node slot: its op runs
    const uint32_t *warp_job_off;    // [warps + 1]
    const TiledJob *jobs;
    const TiledSeg *segs;
    const uint32_t *ops;
    const uint2 *raws;               // (plaintext index * L, input tile byte offset)
    const uint32_t *comb_off;        // [n_comb + 1] into comb_parts
    const uint32_t *comb_out;        // output of each combine
    const uint32_t *comb_parts;      // partial slots to add
    int *err;                        // set to 1 when a bounded wait gives up
    uint32_t N, L, log2N;
    uint32_t limb0, n_limbs;         // limb range of this launch
    uint32_t tiles_per_limb;         // N / T
    uint32_t n_in, n_nodes, n_levels, n_part, n_comb;
    uint32_t src_bytes;              // one source region (inputs, then shared sums)
    uint32_t double_buffer;          // 1: two source regions, next tile staged early
    uint32_t mac_budget;             // products per accumulator between folds
};

struct TiledSchedule {
    int C = 2;                 // coefficients per lane
    bool narrow = false;       // every modulus < 2^52: radix-2^26 arithmetic
    uint32_t warps = 8;        // warps per CTA
    uint32_t tile = 64;        // coefficients per CTA tile
    size_t smem = 0;           // dynamic shared memory per CTA
    uint32_t ctas_per_sm = 0;  // occupancy the lowering planned for
    DeviceSchedule sched;
    TiledArgs args{};          // device pointers into sched.blob (data pointers unset)
};
