// tiled.h -- schedule of the tiled kernel (shared by lower_tiled.cpp and
// kernel_tiled.cu).
//
// A persistent CTA walks the (limb, coefficient tile) pairs.  For each it
// holds, in shared memory, the tile of every input and of every materialised
// shared signed sum ("sources"), plus one tile of zeros.  Each warp runs a
// fixed stream of operations for every tile; each operation consumes one
// plaintext tile:
//
//   RAW  acc += pt * source                     (PMult-MAC of a raw term)
//   SEG  acc += gamma * (sum of +sources - sum of -sources)
//        (one scale group, or a piece of it: Sec. 4.2 "Grouping
//        Reconstruction Operations")
//   NOP  padding: acc += pt * 0, with pt a tile another operation of the
//        batch also reads, so the loop body has no branch and no extra HBM
//        traffic
// with flags FOLD (reduce the accumulator before this batch) and LAST (this
// job's result is complete after this batch: reduce, store, clear).  The
// stream is processed in batches of P operations (P = 16, 8 or 4, the number of
// plaintext tiles each warp keeps in flight): every job
// starts a batch and is padded to whole batches; SEG and FOLD only open a
// batch (a SEG's signed sum is formed before its batch) and LAST only closes
// one.  (Measured: a LAST test on every operation, so that jobs could end
// inside a batch and pad less, slows the loop by 15-50%, more than the
// padding it could save.)  A job is one output, or one part of an
// output split across warps whose reduced partial sums are added at the end
// of the tile.
//
// The schedule is one array of 32-bit words (a multiple of 128 bytes, so that
// the source regions after it are aligned for TMA), copied once per CTA into
// shared memory:
//   level offsets   shared sums of level l are nodes [lev[l], lev[l+1])
//   node offsets    word offset of each node's program
//   node programs   n_plus | n_minus << 16, then the plus then the minus
//                   source indices, two 16-bit indices per word (each run
//                   starts on a new word); or, in the offset form
//                   (TiledArgs::src_offsets), a block of four words (the
//                   header, the slot word, a formation's target slot, 0)
//                   and the runs as one 32-bit word per source, its byte
//                   offset s * 2T * 8 in the source region, each run padded
//                   to a multiple of four words: the kernel then forms each
//                   source's address with one addition instead of unpacking
//                   and scaling an index
//   warp table      per warp: op stream offset, op count (a multiple of the
//                   prefetch depth), segment stream offset, target offset,
//                   first warp slot (then padding to eight words)
//   op streams      one word per operation (layout below)
//   segment streams per SEG operation, in order: a program as above
//                   (its formations first: a slot word and a program each,
//                   or in the offset form a program holding its slot)
//   target streams  per job: output index, or kPartBit | partial slot
//   combine lists   per split output: its partial slots
//   (tensor-core sums only) W as fp16 core matrices, then one fp32 constant
//                   per group (tc_signed.cuh)
// Source index s names the tile pair (c0, c1) at s * 2T words of the source
// region: inputs first, then the materialised shared sums in level order,
// then the zero tile.  Programs name warp slots in their slot word (see
// tile_math.cuh signed_sum); a warp's slots are tile pairs of its own, after
// the partial slots, written and read only by that warp (each lane its own
// coefficients).
#pragma once
#include <stdint.h>

#include "fiona_internal.h"
#include "tc_geometry.h"

// most warps per CTA (the kernels are built for it: at most 128 registers a
// thread; a bound of 20 warps measured slower, its register cap spills)
constexpr uint32_t kTiledMaxWarps = 16;
constexpr uint32_t kPartBit = 0x80000000u;  // job target: partial slot

// operation word: [31:14] plaintext index, [13:9] flags, [8:0] source index.
// CONST marks a raw term whose plaintext is constant over the coefficients
// (FIONA_TERM_RAW_CONST): its load reads residue 0 of the limb.  A SEG's
// [8:0] is instead the number of shared signed sums the warp forms into its
// slots before the SEG's own sum: its segment-stream entry is that many
// (slot number, program) pairs, then the SEG's program.
constexpr uint32_t kOpSrcBits = 9;
constexpr uint32_t kOpMaxSources = 1u << kOpSrcBits;
constexpr uint32_t kOpSeg = 1u << 9;
constexpr uint32_t kOpLast = 1u << 10;
constexpr uint32_t kOpFold = 1u << 11;
constexpr uint32_t kOpNop = 1u << 12;
constexpr uint32_t kOpConst = 1u << 13;
constexpr uint32_t kOpPtShift = 14;
constexpr uint32_t kOpMaxPlaintexts = 1u << (32 - kOpPtShift);

// per warp: op offset, op count, seg offset, target offset, first slot
constexpr uint32_t kWarpTableWords = 8;
// test only: the first input copy of each CTA expects 16 bytes that never come
constexpr uint32_t kTiledFlagExtraTx = 1;

struct TiledArgs {
    const uint64_t *in;
    const uint64_t *pt;
    uint64_t *out;
    const LimbConst *limbs;
    const uint32_t *sched;   // schedule words (global), copied to shared memory
    int *err;                // set to 1 when a bounded wait gives up
    // word offsets of the schedule's sections
    uint32_t o_level, o_node_off, o_warp, o_comb_off, o_comb_out, o_comb_parts;
    uint32_t sched_bytes;    // multiple of 16
    uint32_t N, L;
    uint32_t pt_stride;      // L * N: elements between plaintexts
    uint32_t limb0, n_limbs;
    uint32_t tiles_per_limb;
    uint32_t n_in, n_nodes, n_levels, n_part, n_comb;
    uint32_t src_bytes;      // one source region (inputs, shared sums, zero tile)
    uint32_t box_rows;       // input polys per TMA box (<= 256), n_boxes boxes per tile
    uint32_t n_boxes;
    uint32_t double_buffer;  // 1: two source regions, next tile staged early
    uint32_t has_pt;         // 0: the plan has no plaintexts (every load reads the schedule)
    uint32_t n_slots;        // warp slots of the CTA (shared signed sums a warp forms for itself);
                             // a warp's own start at the slot its table entry names
    // tensor-core signed sums (tc_signed.cuh; tc_groups = 0: none): the
    // n_nodes = tc_groups level-0 nodes are formed as one contraction per
    // tile, by the kernel variant built for it, instead of by their programs
    uint32_t tc_groups;
    uint32_t tc_k, tc_n;     // TcGeometry
    uint32_t tc_cols;        // tensor memory columns a CTA allocates
    uint32_t tc_wabs;        // largest sum of |weights| of a group: S + tc_wabs * q > 0
    uint32_t o_tcw, o_tcm;   // word offsets of W (fp16 image) and of the groups' magic constants
    uint64_t wait_ns;        // bound of the waits for input copies and for the contraction
    uint32_t test_flags;     // kTiledFlag* (0 outside tests)
    uint32_t zero;           // always 0, read at run time (rns::mac26)
    uint32_t src_offsets;    // 1: programs in the offset form (source byte offsets), 0: packed indices
    uint32_t kc_all;         // 1: every raw term's plaintext is constant (KA variant): operations after
                             // a batch's first are read as constant, so none of them may be a non-constant RAW
};

// Warp-specialised variant (kernel_ws.cu), two coefficients per lane.  The
// block is W consumer warps (the operation streams, as above) and one stager
// warp that copies each tile's inputs by TMA and, for narrow plans, rewrites
// them in split form.  Each consumer warp copies its own plaintext tiles
// with per-lane asynchronous copies into a ring of D groups of P slots in
// shared memory, D - 1 batches ahead of its use.  The schedule is copied to
// shared memory whole (`smem_sched_bytes`).
constexpr uint32_t kWsMaxWarps = 16;  // consumer warps
constexpr uint32_t kWsFlagExtraTx = 1;  // test only: the first input copy expects 16 bytes that never come

struct WsArgs {
    const uint64_t *in;
    const uint64_t *pt;
    uint64_t *out;
    const LimbConst *limbs;
    const uint32_t *sched;   // schedule words (global), copied to shared memory
    int *err;                // set to 1 when a bounded wait gives up
    uint64_t wait_ns;        // bound of every wait
    uint32_t smem_sched_bytes;
    uint32_t o_warp, o_comb_off, o_comb_out, o_comb_parts;
    uint32_t N, L;
    uint32_t pt_stride;      // L * N
    uint32_t limb0, n_limbs;
    uint32_t tiles_per_limb;
    uint32_t n_in, n_part, n_comb;
    uint32_t src_bytes;      // one source region (inputs, zero tile)
    uint32_t box_rows, n_boxes;
    uint32_t n_buf;          // source regions (1 or 2)
    uint32_t has_pt;
    uint32_t flags;          // kWsFlag*
    uint32_t n_slots;        // warp slots of the CTA (a warp's own start where its table entry says)
};

// Shared-memory layout of the warp-specialised kernel (byte offsets), the
// same on the host and in the kernel.
struct WsLayout {
    uint32_t src0, part0, ring0, slot0, bar0, total;
#if defined(__CUDACC__)
    __host__ __device__
#endif
    WsLayout(uint32_t sched_bytes, uint32_t n_buf, uint32_t src_bytes, uint32_t n_part, uint32_t W, uint32_t D,
             uint32_t P, uint32_t TB, uint32_t S)
    {
        src0 = sched_bytes;
        part0 = src0 + n_buf * src_bytes;
        ring0 = part0 + 2 * n_part * 2 * TB;
        slot0 = ring0 + W * D * P * TB;
        bar0 = slot0 + S * 2 * TB;
        total = bar0 + 8 * 8;
    }
};

struct TiledSchedule {
    int C = 2;                 // coefficients per lane
    bool narrow = false;       // every modulus < 2^52: radix-2^26 arithmetic
    uint32_t warps = 8;        // warps per CTA
    uint32_t tile = 64;        // coefficients per CTA tile
    uint32_t batch = 8;        // P: operations per batch, plaintext tiles in flight per warp
    bool has_const = false;    // some operation reads a constant plaintext (kOpConst)
    size_t smem = 0;           // dynamic shared memory per CTA
    uint32_t ctas_per_sm = 0;  // occupancy the lowering planned for
    uint32_t addsub = 0;       // Add/Sub per evaluation (fiona_plan_stats.addsub_executed)
    uint32_t nodes_kept = 0;   // shared sums materialised per tile
    uint32_t nodes_expanded = 0;  // shared sums expanded into their uses
    DeviceSchedule sched;
    TiledArgs args{};          // device pointers (data pointers unset)
    bool tc = false;           // the scale groups' signed sums run on the tensor cores (args.tc_groups)
    bool w12 = false;          // the variant built for CTAs of at most 12 warps (kernel_tiled_w12.cu)
    bool ws = false;           // the warp-specialised kernel runs this plan
    uint32_t ring = 0;         // its plaintext ring depth D (groups of P slots per warp)
    WsArgs ws_args{};
};
