/*
 * fiona.h -- C ABI of the GB300 evaluator for hybrid packed-CKKS linear layers.
 *
 * The operation (Sec. 4.2 of "Fiona: Accelerating FHE Inference with
 * Packing-Aware Ternary Weights", "Exact Compilation of Routed Linear
 * Operators"): every packed output ciphertext y_j of a linear layer is a sum
 * of signed terms and raw terms over input ciphertexts A_i that are already
 * rotated into place (Sec. 2.3, "Packed Evaluation of a Linear Layer"):
 *
 *   y_j = sum_{scale groups g of j} gamma_g * ( sum_{t=+1} A_i - sum_{t=-1} A_i )
 *       + sum_{raw terms e of j}    P_e * A_{i_e}
 *
 * evaluated in RNS, NTT (evaluation) form, where PMult is the element-wise
 * product of residues in each limb and Add/Sub the element-wise modular
 * sum/difference (Sec. 2.2, "Homomorphic Operations").  Terms with t = 0 are
 * skipped (Sec. 4.1, "Packing-Aware Weight Representation").  Each scale
 * group applies its reconstruction-factor plaintext gamma_g once to its signed
 * sum ("Grouping Reconstruction Operations"); signed sums shared by several
 * outputs are formed once and reused with sign +1 or -1 ("Sharing Signed
 * Sums", Eq. "shared-example"); signed and raw products of an output are
 * added before any rescale, so the output is left at scale
 * Delta_ct * Delta_pt and is not rescaled ("Combining the Signed and Raw
 * Routes").  All plaintexts of one layer must be encoded at the same scale
 * and every input must be at the same level and slot arrangement.
 *
 * Memory layouts (row-major uint64 residues in [0, q_l); every buffer must
 * start on a 16-byte boundary, FIONA_ERR_ARG otherwise):
 *   inputs      [n_in ][2][L][N]   c0, c1 of each input ciphertext
 *   plaintexts  [n_pt ][L][N]      raw-group and scale (gamma) plaintexts
 *   outputs     [n_out][2][L][N]   overwritten, canonical residues in [0, q_l)
 *
 * Ownership: fiona_ctx and fiona_plan objects are created and freed by the
 * library (the matching _destroy call).  Every data buffer is owned by the
 * caller; the library neither frees nor retains it after a call returns.
 *
 * Errors: every function that can fail returns a fiona_status (0 = success,
 * negative = failure) and leaves its out-arguments untouched on failure.
 * fiona_last_error() returns a one-line description of the most recent
 * failure in the calling thread.  No entry point synchronises the device,
 * except where stated.  A call that works on a context's device makes it the
 * current device for the call's duration and restores the caller's device
 * on return; if it cannot select it, the call returns FIONA_ERR_CUDA having
 * enqueued nothing.
 */
#ifndef FIONA_H
#define FIONA_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* 4: fiona_plan_stats_t's last two words report the signed-sum program form
 * (source_offsets) and the all-constant-plaintext kernel variant
 * (const_raw_all); the structure's size is unchanged (they were reserved). */
#define FIONA_ABI_VERSION 4

typedef struct fiona_ctx fiona_ctx;   /* N, RNS moduli, per-limb constants on one device */
typedef struct fiona_plan fiona_plan; /* one validated, lowered linear layer */

typedef enum fiona_status {
    FIONA_OK = 0,
    FIONA_ERR_ARG = -1,     /* null pointer, size out of range, misaligned buffer */
    FIONA_ERR_MODULUS = -2, /* a modulus is not an odd prime < 2^60 with q = 1 mod 2N */
    FIONA_ERR_PLAN = -3,    /* the layer description is malformed (see fiona_plan_create) */
    FIONA_ERR_NOMEM = -4,   /* host or device allocation failed */
    FIONA_ERR_CUDA = -5,    /* a CUDA runtime call failed (launch, copy, device) */
    FIONA_ERR_RANGE = -6,   /* fiona_check_residues found a residue >= q_l */
    FIONA_ERR_NODEVICE = -7,/* evaluation requested on a validation-only context */
    FIONA_ERR_TIMEOUT = -8, /* a kernel gave up waiting for its own copies (see fiona_device_check) */
    FIONA_ERR_INTERNAL = -9 /* a lowered schedule failed its own consistency check (a library bug) */
} fiona_status;

/* Kernel variants (fiona_plan_select_kernel).  DIRECT: one thread per output
 * and coefficient pair, inputs read through L2 for every output.  TILED: one
 * CTA per limb and coefficient tile; the tile of every input is copied once
 * into shared memory (bulk asynchronous copies), shared signed sums are
 * formed once per tile, and the warps split the outputs.  AUTO (the default
 * after fiona_plan_create): TILED for layers with more than one output whose
 * tile fits in shared memory, DIRECT otherwise. */
enum { FIONA_KERNEL_AUTO = 0, FIONA_KERNEL_DIRECT = 1, FIONA_KERNEL_TILED = 2 };

/* Pass as `device` to fiona_ctx_create for a validation-only context: plans
 * can be created, validated and inspected with fiona_plan_stats, nothing
 * touches a GPU, and fiona_linear_eval returns FIONA_ERR_NODEVICE. */
#define FIONA_DEVICE_NONE (-1)

/* Route of one term (Sec. 4.1: a pure group takes the signed route, every
 * other group the raw route).  FIONA_TERM_RAW_CONST is a raw term whose
 * plaintext encodes one value in every slot (column packing broadcasts a
 * single weight to all slots, Sec. 6 "BERT"): the encoding of a constant
 * slot vector is a constant poly, so in NTT form every coefficient of limb l
 * holds the same residue.  The kernels read only that residue, the first of
 * each limb (plaintexts[pt][l][0]); the plaintext keeps its [L][N] place in
 * the plaintext buffer, and its other residues are not read. */
enum { FIONA_TERM_RAW = 0, FIONA_TERM_TERNARY = 1, FIONA_TERM_RAW_CONST = 2 };

/* One term = one execution group g_{j,i}: the weights of output j applied to
 * input A_i through one plaintext operand (Sec. 2.3 "Packing Layout and
 * Execution Groups"; Sec. 4.2 notation g_{j,i}).  16 bytes. */
typedef struct fiona_term {
    uint32_t input;   /* i, index of the input ciphertext, < n_in                     */
    uint32_t pt;      /* RAW, RAW_CONST: index of the raw-group plaintext, < n_pt;
                         TERNARY: 0                                                   */
    uint32_t group;   /* TERNARY: scale group, < n_groups, owned by this output; RAW: 0 */
    int8_t kind;      /* FIONA_TERM_RAW, FIONA_TERM_TERNARY or FIONA_TERM_RAW_CONST     */
    int8_t sign;      /* TERNARY: h_g in {-1, 0, +1}; RAW: 0                           */
    uint16_t reserved;/* must be 0                                                      */
} fiona_term;

/* Child of a shared signed sum U_k: an input ciphertext or an earlier shared
 * sum, with sign +1 or -1 (Sec. 4.2 "Sharing Signed Sums").  8 bytes. */
typedef struct fiona_sum_child {
    uint32_t ref;     /* input index (< n_in) or node index (< this node's index) */
    int8_t is_node;   /* 0: ref is an input; 1: ref is a node                      */
    int8_t sign;      /* +1 or -1                                                   */
    uint16_t reserved;/* must be 0                                                  */
} fiona_sum_child;

/* Output `output` takes sign * U_node into the signed sum of its scale group
 * `group`, in place of the signed terms U_node stands for (a sum can be
 * reused with all signs reversed, Sec. 4.2).  16 bytes. */
typedef struct fiona_sum_use {
    uint32_t output;
    uint32_t group;
    uint32_t node;
    int8_t sign;      /* +1 or -1 */
    uint8_t reserved[3];
} fiona_sum_use;

/* Operation counts in the paper's units (Sec. 6 "Measurements" counts weight
 * PMults, Add/Sub and rescales; Table "eval-linear-compilation") and sizes. */
typedef struct fiona_plan_stats_t {
    uint64_t n_terms;             /* all terms, t = 0 included                             */
    uint64_t n_nonzero_terms;     /* raw + signed terms with t != 0 (the unit of terms/s)  */
    uint64_t n_raw_terms;
    uint64_t n_signed_terms;      /* TERNARY terms with t = +1 or -1                        */
    uint64_t n_skipped_terms;     /* TERNARY terms with t = 0                               */
    uint64_t n_scale_groups_used; /* scale groups with at least one signed term            */
    uint64_t n_nodes;
    uint64_t n_uses;
    uint64_t pmult_per_term;      /* term by term: one PMult per raw or signed term        */
    uint64_t pmult_grouped;       /* grouped: one PMult per raw term and per used group    */
    uint64_t addsub_flat;         /* grouped, no sharing: n-1 Add/Sub to combine n operands */
    uint64_t addsub_shared;       /* with each shared sum formed once                       */
    uint64_t rescale_separate;    /* one rescale per route (signed, raw) per output         */
    uint64_t rescale_combined;    /* one rescale per output with any nonzero term           */
    uint64_t n_inputs_used;       /* inputs read by at least one nonzero term               */
    uint64_t n_plaintexts_used;   /* distinct plaintexts read                               */
    uint64_t bytes_min;           /* each used input, plaintext and each output moved once
                                     (a plaintext read only by RAW_CONST terms: L words)     */
    uint64_t wide_products;       /* 64x64->128-bit products per evaluation                 */
    uint32_t N;
    uint32_t L;
    uint32_t n_in, n_out, n_pt, n_groups;
    uint32_t tile_coeffs;         /* coefficients per CTA tile chosen by the lowering       */
    uint32_t warps_per_cta;
    uint32_t smem_bytes;          /* dynamic shared memory per CTA                          */
    uint32_t ctas_per_sm;         /* occupancy the lowering planned for                     */
    uint32_t kernel;              /* variant in use: FIONA_KERNEL_DIRECT or FIONA_KERNEL_TILED */
    uint32_t nodes_materialized;  /* TILED: shared sums formed once per tile, by the block or
                                     by the warp whose outputs use them (a sum several warps
                                     use counts once per warp); the others are expanded into
                                     their uses: same residues, more Add/Sub */
    uint32_t addsub_executed;     /* Add/Sub of the kernel in use, in the units of addsub_flat:
                                     each sum of n operands it forms (shared sums, scale groups,
                                     an output's products, its partial sums) counts n - 1 */
    uint32_t tensor_core_sums;    /* TILED: scale-group signed sums formed per tile as one
                                     contraction on the tensor cores (the groups' terms, shared
                                     sums expanded, exact in fp16 chunks); 0: on the ALUs      */
    uint32_t source_offsets;      /* TILED: 1 if the schedule's signed-sum runs hold source byte
                                     offsets (one addition per source address), 0 if 16-bit
                                     indices packed two per word (used when the larger offset
                                     schedule does not fit in shared memory)                   */
    uint32_t const_raw_all;       /* TILED: 1 if every raw plaintext of the plan is constant and
                                     the kernel variant for that case runs (no per-operation test
                                     of the plaintext's kind after a batch's first operation)   */
} fiona_plan_stats_t;

/* Create a context for ring dimension N (a power of two, 2^10 <= N <= 2^17)
 * and L RNS moduli (1 <= L <= 64) on CUDA device `device` (or
 * FIONA_DEVICE_NONE).  Each modulus must be an odd prime below 2^60 with
 * q = 1 (mod 2N) (an NTT-friendly CKKS prime, Sec. 2.2; the paper's setting
 * is N = 2^16, Sec. 5 "Execution Environment"); the check is a deterministic
 * Miller-Rabin test.  Moduli must be distinct.  The moduli are copied.
 * Errors: FIONA_ERR_ARG, FIONA_ERR_MODULUS, FIONA_ERR_NOMEM, FIONA_ERR_CUDA. */
int fiona_ctx_create(uint32_t N, const uint64_t *moduli, uint32_t L, int device,
                     fiona_ctx **out);
void fiona_ctx_destroy(fiona_ctx *ctx); /* NULL is a no-op; destroy plans first */

/* Validate and lower one linear layer (Sec. 4.2).
 *   terms[term_offsets[j] .. term_offsets[j+1]) are the terms of output j
 *   (CSR, term_offsets has n_out+1 entries, term_offsets[0] = 0).  The term
 *   list is the ground truth of what each output computes.
 *   group_scale_pt[g] is the plaintext holding gamma_g; group_output[g] the
 *   output that owns group g (a scale group belongs to one output).
 *   Nodes k = 0..n_nodes-1 are shared signed sums with children
 *   children[node_offsets[k] .. node_offsets[k+1]); a child node must have a
 *   smaller index (children first), so the DAG is acyclic by construction.
 *   uses[] say which signed terms are evaluated through a shared sum.
 * FIONA_ERR_PLAN if: an index is out of range; a RAW term has sign != 0 or a
 * TERNARY term a sign outside {-1,0,+1}; a reserved field is nonzero; a
 * group's terms belong to another output than group_output[g]; a node has no
 * child, a child sign not +/-1, a child node index >= its own, or expands to
 * the same input twice; a use's node, expanded with its sign, is not matched
 * by the output's TERNARY terms in that group with the same inputs and signs;
 * two uses in one output cover the same term ("at most one of any two
 * overlapping candidates", Sec. 4.2).  Arrays are copied; the caller may free
 * them on return.  The plan keeps a pointer to ctx: destroy it first.
 * The device schedule is uploaded with a synchronous copy. */
int fiona_plan_create(const fiona_ctx *ctx, uint32_t n_in, uint32_t n_out, uint32_t n_pt,
                      const uint32_t *term_offsets, const fiona_term *terms,
                      uint32_t n_groups, const uint32_t *group_scale_pt,
                      const uint32_t *group_output,
                      uint32_t n_nodes, const uint32_t *node_offsets,
                      const fiona_sum_child *children,
                      uint32_t n_uses, const fiona_sum_use *uses, fiona_plan **out);
void fiona_plan_destroy(fiona_plan *plan); /* NULL is a no-op */

/* A layer whose plaintexts are encoded at several scales (Sec. 4.2,
 * "Combining the Signed and Raw Routes": an output's signed and raw routes
 * are added before its one rescale only when their plaintexts share a scale;
 * with different scales each must be rescaled on its own).  pt_class[p] in
 * [0, n_class) is the scale class of plaintext p (a scale group's class is
 * that of its gamma, a raw term's that of its plaintext).  Output j of the
 * description becomes n_class results: result j * n_class + s holds the
 * scale groups and raw terms of output j whose plaintexts have class s,
 * combined (a class with no term of output j gives a result of zeros).  The
 * plan then evaluates like any other with n_out * n_class outputs: the output
 * buffer of fiona_linear_eval (and its variants) is [n_out][n_class][2][L][N],
 * and fiona_plan_stats counts those results as outputs.  Other arguments and
 * errors as fiona_plan_create; FIONA_ERR_ARG if n_class is 0 or above 255,
 * pt_class is null while n_pt > 0, or n_out * n_class exceeds 65535;
 * FIONA_ERR_PLAN if a class is >= n_class.  n_class = 1 is
 * fiona_plan_create. */
int fiona_plan_create_classes(const fiona_ctx *ctx, uint32_t n_in, uint32_t n_out, uint32_t n_pt,
                              const uint32_t *term_offsets, const fiona_term *terms,
                              uint32_t n_groups, const uint32_t *group_scale_pt,
                              const uint32_t *group_output,
                              uint32_t n_nodes, const uint32_t *node_offsets,
                              const fiona_sum_child *children,
                              uint32_t n_uses, const fiona_sum_use *uses,
                              uint32_t n_class, const uint8_t *pt_class, fiona_plan **out);

/* Route of the weights of output j on input i, for the plan compiler.
 * 8 bytes. */
typedef struct fiona_route {
    int8_t kind;      /* FIONA_TERM_RAW, FIONA_TERM_TERNARY or FIONA_TERM_RAW_CONST     */
    int8_t sign;      /* TERNARY: h_g in {-1, 0, +1}; RAW, RAW_CONST: 0                */
    uint16_t reserved;/* must be 0                                                     */
    uint32_t pt;      /* RAW, RAW_CONST: the group's plaintext; TERNARY: the output's reconstruction-
                         factor plaintext gamma (terms with one gamma share one PMult)  */
} fiona_route;

enum {
    FIONA_COMPILE_SHARE = 1,       /* search shared signed sums                        */
    FIONA_COMPILE_SHARE_EXACT = 2  /* with SHARE: accept a sum of m inputs used by k
                                      outputs when (k-1)(m-1) > 0 (the Add/Sub it saves
                                      under the n-1 rule) instead of km-m-k > 0        */
};

/* Host plan compiler (Sec. 4.2): from the dense route matrix
 * routes[j * n_in + i] of a layer to the arrays fiona_plan_create takes.
 *   Terms: one per (output, input) pair, in input order (term_offsets[j] =
 *   j * n_in).  Grouping Reconstruction Operations: the TERNARY terms of one
 *   output with the same gamma form one scale group (groups numbered in
 *   order of first appearance).  Sharing Signed Sums (with
 *   FIONA_COMPILE_SHARE): every pair of scale groups of different outputs
 *   proposes the signed terms they have in common (the same inputs with the
 *   same signs, or with all signs reversed) as a sum; a sum of m inputs that
 *   k groups can take is estimated to save km - m - k Add/Sub (the paper's
 *   conservative count; (k-1)(m-1) with FIONA_COMPILE_SHARE_EXACT), and the
 *   sums are accepted largest estimate first while the estimate over the
 *   groups still free to take them is positive.  A group takes at most one of
 *   any two overlapping sums, so a term is covered at most once.  Nodes are
 *   sums of inputs (one level).
 * Caller-allocated outputs, each with room for n_out * n_in entries
 * (term_offsets and node_offsets: one more): terms, group_scale_pt,
 * group_output, node_offsets, children, uses; counts in *n_groups,
 * *n_nodes, *n_uses.  Pure host code: no context, no device.
 * Errors: FIONA_ERR_ARG (null argument, unknown flag, more than 2^24 pairs),
 * FIONA_ERR_PLAN (a route with an unknown kind, a sign outside its range,
 * a plaintext >= n_pt, or a nonzero reserved field). */
int fiona_plan_compile(uint32_t n_in, uint32_t n_out, uint32_t n_pt, const fiona_route *routes,
                       uint32_t flags, uint32_t *term_offsets, fiona_term *terms, uint32_t *n_groups,
                       uint32_t *group_scale_pt, uint32_t *group_output, uint32_t *n_nodes,
                       uint32_t *node_offsets, fiona_sum_child *children, uint32_t *n_uses,
                       fiona_sum_use *uses);

int fiona_plan_stats(const fiona_plan *plan, fiona_plan_stats_t *out);

/* Choose the kernel variant used by later evaluations of `plan`
 * (FIONA_KERNEL_AUTO, _DIRECT or _TILED).  Both compute the same residues.
 * FIONA_ERR_ARG if the variant cannot run this plan (TILED needs the tile of
 * every input and shared sum to fit in shared memory).  Not thread-safe
 * against concurrent evaluations of the same plan. */
int fiona_plan_select_kernel(fiona_plan *plan, int kernel);

/* Evaluate the layer on the GPU: enqueue the fused kernel on `cuda_stream`
 * (a cudaStream_t; NULL = the legacy default stream) and return at once.
 * `inputs`, `plaintexts`, `outputs` are device pointers of the ctx's device
 * in the layouts above; outputs must not overlap the other two.  Residues
 * must be < q_l (undefined results otherwise; fiona_check_residues checks).
 * Errors: FIONA_ERR_ARG (null or misaligned pointer), FIONA_ERR_NODEVICE,
 * FIONA_ERR_CUDA (launch failure, reported from cudaGetLastError). */
int fiona_linear_eval(const fiona_plan *plan, void *cuda_stream, const uint64_t *inputs,
                      const uint64_t *plaintexts, uint64_t *outputs);

/* Evaluate the layer at a lower level: the ciphertexts and plaintexts hold
 * only the first `L_eval` RNS limbs (moduli q_0 .. q_{L_eval-1}; CKKS drops
 * the last limbs as a ciphertext goes down in level, Sec. 2.2), laid out
 * [n_in][2][L_eval][N], [n_pt][L_eval][N] and [n_out][2][L_eval][N].  One
 * plan serves every level: the layer's routes, groups and shared sums do
 * not depend on the limb count, and every limb is computed independently.
 * Asynchronous like fiona_linear_eval.  Errors: FIONA_ERR_ARG (L_eval
 * outside [1, L], null or misaligned pointer), FIONA_ERR_NODEVICE,
 * FIONA_ERR_CUDA. */
int fiona_linear_eval_level(const fiona_plan *plan, void *cuda_stream, uint32_t L_eval,
                            const uint64_t *inputs, const uint64_t *plaintexts, uint64_t *outputs);

/* Rescale (Sec. 2.2 "Homomorphic Operations": after a PMult the scale is
 * Delta^2 and a rescale divides by the last prime of the current level;
 * Sec. 4.2 "Combining the Signed and Raw Routes": the combined output of a
 * layer is rescaled once).  `polys` holds `count` polys in NTT form at level
 * `L_cur` ([count][L_cur][N], moduli q_0 .. q_{L_cur-1}; a ciphertext is two
 * polys, c0 and c1).  For each poly y, with r the coefficients of its last
 * limb (inverse NTT mod q_{L_cur-1}, canonical in [0, q_{L_cur-1})):
 *   out_l = (y_l - NTT_l(r mod q_l)) * q_{L_cur-1}^{-1}  mod q_l,
 * for l < L_cur - 1, into `out` ([count][L_cur-1][N], canonical): the
 * residues of floor(Y / q_{L_cur-1}) for the CRT value Y of each
 * coefficient.  With FIONA_RESCALE_ROUND in `flags` the quotient is rounded
 * to the nearest integer instead, floor((Y + h) / q_{L_cur-1}) with
 * h = floor(q_{L_cur-1} / 2), as SEAL's rescale does: r is replaced by
 * r' = (r + h) mod q_{L_cur-1} and the subtracted poly by r' - h.  The NTT
 * form is A[k] = a(psi^(2 brv(k) + 1)) mod q_l, psi the least primitive 2N-th
 * root of unity mod q_l and brv the log2(N)-bit reversal; every modulus must
 * be a prime = 1 mod 2N (FIONA_ERR_MODULUS otherwise).
 * The last limb of every input poly is overwritten with r (r' when rounding); the other limbs
 * are only read.  `out` must not overlap `polys`.  Device pointers of the
 * ctx's device, 16-byte aligned.  Asynchronous on `cuda_stream`, except that
 * the first call on a ctx builds its twiddle tables (about 32 N L bytes of
 * device memory, held until fiona_ctx_destroy) synchronously: make it before
 * any stream capture.  Errors: FIONA_ERR_ARG (L_cur outside [2, L], null,
 * misaligned or overlapping buffers, unknown flags), FIONA_ERR_NODEVICE,
 * FIONA_ERR_MODULUS, FIONA_ERR_NOMEM, FIONA_ERR_CUDA. */
enum { FIONA_RESCALE_ROUND = 1 };
int fiona_rescale(const fiona_ctx *ctx, void *cuda_stream, uint32_t L_cur, uint64_t count,
                  uint64_t *polys, uint64_t *out, uint32_t flags);

/* A layer followed by its rescale: evaluates at level L_eval (as
 * fiona_linear_eval_level) into `work` ([n_out][2][L_eval][N]), then
 * rescales the 2 n_out polys of `work` into `outputs`
 * ([n_out][2][L_eval-1][N]), both on `cuda_stream`.  `work` ends with the
 * un-rescaled layer output except in its last limbs, which hold
 * coefficients.  `outputs` must overlap neither `work` nor `inputs`.  `flags`
 * as for fiona_rescale.  Errors as fiona_linear_eval_level and fiona_rescale
 * (L_eval >= 2). */
int fiona_linear_eval_rescale(const fiona_plan *plan, void *cuda_stream, uint32_t L_eval,
                              const uint64_t *inputs, const uint64_t *plaintexts, uint64_t *work,
                              uint64_t *outputs, uint32_t flags);

/* Plaintext encoding on the GPU (Sec. 2.2 "Ciphertexts and Slots": CKKS
 * packs a vector of numbers into the slots of a plaintext; the layer's gamma
 * and raw plaintexts are encodings of the model's weights).
 *
 * fiona_ckks_embed: `slots` holds `count` vectors of N/2 complex numbers
 * ([count][N/2][2] doubles: re, im; real weights have im = 0).  For each,
 * the real poly m of degree < N with m(zeta^(5^j)) = z_j and
 * m(zeta^(-5^j)) = conj(z_j), zeta = exp(i pi / N) (slot j at the odd
 * power 5^j mod 2N), is computed in fp64 and its coefficients
 * round(scale * m_i) (ties away from zero) are written to `coeffs`
 * ([count][N] int64).  `work` is scratch of count * N * 8 bytes.  The
 * rounding is floating point: a coefficient whose exact value lies within
 * the transform's fp64 error of a half-integer may round either way.  A
 * coefficient that is not finite or reaches 2^62 in magnitude is written as
 * 0 and reported by the next fiona_device_check (FIONA_ERR_RANGE).
 *
 * fiona_encode_coeffs: integer polys `coeffs` ([count][N] int64, any value)
 * to RNS NTT form at level L_cur: out[p][l] = NTT_l(coeffs[p] mod q_l)
 * ([count][L_cur][N], canonical; NTT form as for fiona_rescale).  Exact.
 *
 * fiona_encode: fiona_ckks_embed then fiona_encode_coeffs (`coeffs` and
 * `work` as above).
 *
 * Device pointers of the ctx's device, 16-byte aligned, pairwise
 * non-overlapping; asynchronous on `cuda_stream`, except that the first call
 * on a ctx builds its tables (twiddles, slot order; synchronous, before any
 * stream capture).  Errors: FIONA_ERR_ARG (scale not positive, L_cur outside
 * [1, L], null, misaligned or overlapping buffers), FIONA_ERR_NODEVICE,
 * FIONA_ERR_NOMEM, FIONA_ERR_CUDA. */
int fiona_ckks_embed(const fiona_ctx *ctx, void *cuda_stream, uint64_t count, const double *slots,
                     double scale, int64_t *coeffs, double *work);
int fiona_encode_coeffs(const fiona_ctx *ctx, void *cuda_stream, uint32_t L_cur, uint64_t count,
                        const int64_t *coeffs, uint64_t *out);
int fiona_encode(const fiona_ctx *ctx, void *cuda_stream, uint32_t L_cur, uint64_t count,
                 const double *slots, double scale, int64_t *coeffs, double *work, uint64_t *out);

/* End-to-end evaluation from host memory: copies `h_inputs` (host, layout
 * [n_in][2][L][N], pinned for overlap) to the caller's device buffer
 * `d_inputs`, evaluates with the device-resident `d_plaintexts` (the model's
 * weights stay on the GPU), and copies the result through `d_outputs` to
 * `h_outputs` (host, [n_out][2][L][N]).  The work is split into limb chunks
 * (one limb each, at most 16 chunks) so the copies of one chunk overlap the
 * kernel of another (RNS limbs are independent).  Synchronous: returns when
 * h_outputs holds the result.
 * Errors as fiona_linear_eval. */
int fiona_linear_eval_host(const fiona_plan *plan, void *cuda_stream, const uint64_t *h_inputs,
                           const uint64_t *d_plaintexts, uint64_t *h_outputs,
                           uint64_t *d_inputs, uint64_t *d_outputs);

/* The same evaluation, queued only: returns once the copies and kernels are
 * enqueued.  fiona_linear_eval_host_join(plan, cuda_stream) then makes
 * `cuda_stream` wait for the plan's output copies queued so far; h_outputs
 * holds the result once `cuda_stream` has completed after the join
 * (cudaStreamSynchronize, or an event recorded on it).  The input copies of a
 * call wait for the work queued on `cuda_stream` before the call (which
 * includes the kernels of the calls before it, not their output copies).
 * Consecutive calls on one plan may reuse the same device buffers: each limb
 * chunk's input copy waits for the previous call's kernel on that chunk and
 * its kernel for the previous call's output copy of it, so a burst of calls
 * overlaps one query's input copies with the previous query's output copies
 * (the two directions of the host link run at once).  The host buffers
 * belong to a call until its join has completed; the calls on one plan come
 * from one host thread at a time.  Errors as fiona_linear_eval (a CUDA error
 * may also surface at the synchronisation). */
int fiona_linear_eval_host_async(const fiona_plan *plan, void *cuda_stream, const uint64_t *h_inputs,
                                 const uint64_t *d_plaintexts, uint64_t *h_outputs,
                                 uint64_t *d_inputs, uint64_t *d_outputs);
int fiona_linear_eval_host_join(const fiona_plan *plan, void *cuda_stream);

/* Evaluate the layer without allocating any device memory.  The paper has no
 * counterpart: this entry point exists for callers that cannot call
 * cudaMalloc at the time they evaluate -- for example a serving runtime that
 * hands all free device memory to its own pool at start-up (a later
 * cudaMalloc would fail), or a latency-critical path that forbids allocation
 * because cudaMalloc/cudaFree may synchronise the device and take unbounded
 * time.  Such a caller creates its context with FIONA_DEVICE_NONE (so
 * fiona_ctx_create and fiona_plan_create touch no device memory either) and
 * passes device buffers it owns; any plan is accepted.
 * The layer's schedule and the per-limb constants are copied (stream
 * ordered) into one fixed area of FIONA_STATIC_AREA_BYTES that the library
 * reserves in every GPU that loads it, until the process exits; the direct
 * kernel then runs from there on the current device (the ctx's device if it
 * has one).  A layer whose schedule exceeds the area is rejected with
 * FIONA_ERR_ARG (about 16 B per output, 16 B per used scale group, 4 B per
 * signed term and 8 B per raw term, plus 32 B per limb).
 * The first call on a device also looks up the area's device address once
 * (cudaGetSymbolAddress); make that first call before any stream capture.
 * The copy from host memory may wait for work already queued on the stream.
 * All calls share the one area and each call overwrites what it reads, so
 * nothing in it needs clearing; calls whose work can overlap on the GPU (other
 * streams, other threads) race on it and must be ordered by the caller.
 * Errors as fiona_linear_eval. */
#define FIONA_STATIC_AREA_BYTES (1u << 20)
int fiona_linear_eval_static(const fiona_plan *plan, void *cuda_stream, const uint64_t *inputs,
                             const uint64_t *plaintexts, uint64_t *outputs);

/* Debug check of the precondition residue < q_l: scans `count` ciphertext
 * polys or plaintexts ([count][L][N], pass n_in*2 for inputs) on the device
 * and returns FIONA_OK, or FIONA_ERR_RANGE if any residue is >= q_l.
 * Synchronous. */
int fiona_check_residues(const fiona_ctx *ctx, void *cuda_stream, const uint64_t *data,
                         uint64_t count);

/* Report kernel-side failures of earlier calls on this context:
 * synchronises `cuda_stream`, then returns FIONA_ERR_TIMEOUT if a tiled
 * kernel gave up waiting for its bulk copies or its tensor-core contraction
 * (every such wait is bounded; the CTA then stops: the outputs of that
 * evaluation are undefined, the context stays usable), FIONA_ERR_RANGE if an encoding met a
 * coefficient out of range (fiona_ckks_embed), FIONA_ERR_CUDA on a CUDA
 * error, FIONA_OK otherwise; the flags are cleared. */
int fiona_device_check(const fiona_ctx *ctx, void *cuda_stream);

const char *fiona_status_str(int status);
const char *fiona_last_error(void); /* thread-local; "" if none */
int fiona_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* FIONA_H */
