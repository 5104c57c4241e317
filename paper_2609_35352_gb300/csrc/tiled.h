// tiled.h -- schedule of the tiled kernel (shared by lower_tiled.cpp and
// kernel_tiled.cu).
//
// A persistent CTA walks the (limb, coefficient tile) pairs.  For each it
// holds, in shared memory, the tile of every input and of every shared
// signed sum ("sources").  Each warp runs a fixed program of jobs for every
// tile; a job is one output (or one part of an output split across warps),
// made of scale-group segments (a signed sum over sources, then one product
// by gamma) and raw terms (PMult-MAC).  The whole schedule is one array of
// 32-bit words, copied once per CTA into shared memory:
//
//   node program   per shared sum: n_plus | n_minus << 16, then the words
//   warp program   per job: target, n_seg | n_raw << 16; per segment
//                  n_plus | n_minus << 16 and the words; then one word per
//                  raw term (the input's tile offset)
//   fetch list     per warp, the plaintext tiles its program consumes, in
//                  order (gamma of each segment, then each raw term), as
//                  plaintext index * L
//   combine lists  outputs split across warps: partial slots to add
//
// A "word" naming a source is the byte offset of its tile pair (c0, c1)
// inside the source region.  Sign runs are at most the lazy-sum bound long
// (longer sums are cut into several segments with the same gamma: exact,
// since gamma*S1 + gamma*S2 = gamma*(S1+S2) mod q).
#pragma once
#include <stdint.h>

#include "fiona_internal.h"

constexpr uint32_t kTiledMaxWarps = 16;
constexpr uint32_t kPartBit = 0x80000000u;  // job target: partial slot

struct TiledArgs {
    const uint64_t *in;
    const uint64_t *pt;
    uint64_t *out;
    const LimbConst *limbs;
    const uint32_t *sched;   // schedule words (global), copied to shared memory
    int *err;                // set to 1 when a bounded wait gives up
    // word offsets of the schedule's sections
    uint32_t o_level, o_node_slot, o_node_prog_off, o_prog_off, o_fetch_off, o_comb_off,
        o_comb_out, o_comb_parts;
    uint32_t sched_bytes;    // multiple of 16
    uint32_t N, L, log2N;
    uint32_t limb0, n_limbs;
    uint32_t tiles_per_limb;
    uint32_t n_in, n_nodes, n_levels, n_part, n_comb;
    uint32_t src_bytes;      // one source region (inputs, then shared sums)
    uint32_t double_buffer;  // 1: two source regions, next tile staged early
    uint32_t mac_budget;     // products per accumulator between folds
};

struct TiledSchedule {
    int C = 2;                 // coefficients per lane
    bool narrow = false;       // every modulus < 2^52: radix-2^26 arithmetic
    uint32_t warps = 8;        // warps per CTA
    uint32_t depth = 8;        // plaintext tiles in flight per warp
    uint32_t tile = 64;        // coefficients per CTA tile
    size_t smem = 0;           // dynamic shared memory per CTA
    uint32_t ctas_per_sm = 0;  // occupancy the lowering planned for
    DeviceSchedule sched;
    TiledArgs args{};          // device pointers (data pointers unset)
};
