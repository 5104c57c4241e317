// fiona_internal.h -- structures shared by the host library code and the
// CUDA kernels (not part of the public ABI).
#pragma once
#include <stddef.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "fiona.h"
#include "rns.cuh"

#define FIONA_MAX_LIMBS 64
#define FIONA_MAX_DEVICES 64

// ---------------------------------------------------------------------------
// Direct schedule (one thread per coefficient pair and output): a flat list of
// scale-group segments and raw terms per output.
// ---------------------------------------------------------------------------
struct DirOut {
    uint32_t seg_begin, seg_end;  // into DirSeg[]
    uint32_t raw_begin, raw_end;  // into raw_input[] / raw_pt[]
};
struct DirSeg {
    uint32_t scale_pt;
    uint32_t op_begin, op_end;    // into sig_ops[]: input | (sign < 0) << 31
    uint32_t pad;
};

// ---------------------------------------------------------------------------
// Tiled schedule (one CTA per limb x coefficient tile; inputs staged in shared
// memory by TMA bulk copies; shared signed sums formed once per tile; each
// warp owns a job list).  Defined in lower_tiled.cpp / kernel_tiled.cu.
// ---------------------------------------------------------------------------
struct TiledSchedule;

struct DeviceSchedule {
    void *blob = nullptr;  // one device allocation holding every array below
    size_t bytes = 0;
};

struct fiona_ctx {
    uint32_t N = 0, L = 0;
    int device = FIONA_DEVICE_NONE;
    std::vector<uint64_t> moduli;
    std::vector<LimbConst> limbs;
    uint64_t q_max = 0;
    LimbConst *d_limbs = nullptr;   // device copy of limbs
    int *d_flag = nullptr;          // scratch flag for fiona_check_residues
    int *d_kerr = nullptr;          // set by a kernel whose bounded wait gave up
    int sm_count = 0;
    size_t smem_optin = 0;
    mutable void *d_ntt = nullptr;  // modular NTT tables, built on first use (rescale.cu)
    mutable void *d_enc = nullptr;  // encoder tables, built on first use (encode.cu)
};

struct HostPlan {
    uint32_t n_in = 0, n_out = 0, n_pt = 0, n_groups = 0, n_nodes = 0, n_uses = 0;
    std::vector<uint32_t> term_offsets;
    std::vector<fiona_term> terms;
    std::vector<uint32_t> group_scale_pt, group_output;
    std::vector<uint32_t> node_offsets;
    std::vector<fiona_sum_child> children;
    std::vector<fiona_sum_use> uses;
    // derived by validation
    std::vector<std::vector<std::pair<uint32_t, int>>> node_leaves;  // (input, sign)
    std::vector<int32_t> term_use;  // use index covering term e, or -1
};

struct fiona_plan {
    const fiona_ctx *ctx = nullptr;
    HostPlan hp;
    fiona_plan_stats_t stats{};
    uint32_t mac_budget = 0;     // products a 128-bit accumulator may take before a reduction
    uint32_t signed_budget = 0;  // residues a 64-bit signed accumulator may take
    int kernel = 0;              // 0 = direct, 1 = tiled (what evaluations use)
    // direct schedule (device pointers into sched.blob)
    DeviceSchedule sched;
    const DirOut *d_dir_out = nullptr;
    const DirSeg *d_dir_seg = nullptr;
    const uint32_t *d_sig_ops = nullptr;
    const uint32_t *d_raw_input = nullptr;
    const uint32_t *d_raw_pt = nullptr;
    // tiled schedule
    TiledSchedule *tiled = nullptr;
    // streams for fiona_linear_eval_host(_async), and per limb chunk the
    // events of its last input copy, kernel and output copy: a call orders
    // each chunk after the previous call's use of the same device buffers
    static constexpr uint32_t kHostChunks = 16;
    void *copy_in_stream = nullptr;
    void *copy_out_stream = nullptr;
    void *ev_in[kHostChunks] = {};
    void *ev_kernel[kHostChunks] = {};
    void *ev_out[kHostChunks] = {};
    void *ev_start = nullptr;
    // host image of the direct schedule and the limb constants, copied into
    // the library's fixed device area by fiona_linear_eval_static
    std::vector<uint8_t> static_image;
    size_t static_off[6] = {0, 0, 0, 0, 0, 0};  // limbs, outs, segs, ops, raw_in, raw_pt
};

// kernel_direct.cu.  Launches evaluate limbs [limb_begin, limb_end) of
// buffers laid out with `layout_L` limbs per poly (the ctx's L, or fewer for
// an evaluation at a lower level).
int launch_direct(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                  uint64_t *out, uint32_t limb_begin, uint32_t limb_end, uint32_t layout_L);
int launch_check_residues(const fiona_ctx *ctx, void *stream, const uint64_t *data,
                          uint64_t count);
int launch_direct_static(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                         uint64_t *out);
extern const size_t kStaticAreaBytes;

// lower_tiled.cpp / kernel_tiled.cu
int lower_tiled(fiona_plan *p);
void free_tiled(fiona_plan *p);
int launch_tiled(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                 uint64_t *out, uint32_t limb_begin, uint32_t limb_end, uint32_t layout_L);

// rescale.cu.  Rescales `count` polys [count][Lc][N] (the last limb of each
// is overwritten with its coefficients) into out [count][Lc-1][N].
int launch_rescale(const fiona_ctx *ctx, void *stream, uint32_t Lc, uint64_t count, uint64_t *polys,
                   uint64_t *out, bool round);
void free_rescale_tables(const fiona_ctx *ctx);
namespace fiona_ntt {
struct NttLimb;
}
// the modular NTT tables of every limb (built on the first call)
int ntt_tables(const fiona_ctx *ctx, const fiona_ntt::NttLimb **limbs);

// encode.cu.  Slots [count][N/2] (complex, fp64) -> integer coefficients
// [count][N] (work: [count][N/2] complex); integer coefficients -> RNS NTT
// form [count][Lc][N].
int launch_embed(const fiona_ctx *ctx, void *stream, uint64_t count, const double *slots, double scale,
                 int64_t *coeffs, double *work);
int launch_encode_coeffs(const fiona_ctx *ctx, void *stream, uint32_t Lc, uint64_t count, const int64_t *coeffs,
                         uint64_t *out);
void free_encode_tables(const fiona_ctx *ctx);

// fiona_host.cpp
int set_error(int code, const char *fmt, ...);
