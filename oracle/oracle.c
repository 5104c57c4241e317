/*
 * oracle.c -- plain CPU oracle for the hybrid packed-CKKS linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this code.  It shares no code,
 * header, table or helper with the CUDA path.
 *
 * What it computes (Sec. 4.2, "Exact Compilation of Routed Linear
 * Operators"; PMult and Add/Sub as defined in Sec. 2.2).  The inputs are
 * ciphertexts in RNS, NTT (evaluation) form, so PMult is the element-wise
 * product of residues in every limb (Sec. 2.2, "Homomorphic Operations").
 * Output j of the layer is the sum of its signed terms and its raw terms
 * (Sec. 4.2, first paragraph, Eq. "routed-example"):
 *
 *   y[j][c][l][k] = (  sum over scale groups g of output j:
 *                         gamma_g[l][k] * ( sum_{t=+1} A[i][c][l][k]
 *                                         - sum_{t=-1} A[i][c][l][k] )
 *                    + sum over raw terms e of output j:
 *                         P[pt_e][l][k] * A[i_e][c][l][k] )  mod q_l
 *
 * Terms with t = 0 are skipped (Sec. 4.1, "Packing-Aware Weight
 * Representation").  The grouping, sharing and combining rewrites of Sec. 4.2
 * are exact identities in Z_q, so every correct evaluation order reaches this
 * same canonical residue in [0, q_l).
 *
 * Every operation is reduced at once with 128-bit '%' (schoolbook).  Nothing
 * is blocked, fused, reordered or reduced lazily.
 *
 * oracle_linear_eval_classes evaluates a layer whose plaintexts carry scale
 * classes (encoded at different scales).  The two routes of an output are
 * added only when their plaintexts share a scale (Sec. 4.2, "Combining the
 * Signed and Raw Routes": the routes are combined before the one rescale of
 * the output, which needs one common scale), so each (output j, class s) is
 * its own result: the sum above restricted to the scale groups whose gamma
 * has class s and the raw terms whose plaintext has class s.
 *
 * oracle_linear_eval_dag evaluates the same layer through the DAG of shared
 * signed sums (Sec. 4.2, "Sharing Signed Sums", Eq. "shared-example"): each
 * shared sum U is formed once, and an output that uses sigma*U adds it to its
 * signed sum in place of the terms U covers.  Tests assert both forms agree.
 *
 * Layouts (row-major uint64):
 *   inputs      [n_in ][2][L][n_coef]
 *   plaintexts  [n_pt ][L][n_coef]
 *   outputs     [n_out][2][L][n_coef]   ([n_out][n_class][2][L][n_coef] with classes)
 * Terms of output j are term_*[term_offsets[j] .. term_offsets[j+1]).
 * kind 0 = raw route (uses term_pt), kind 1 = signed route (term_sign in
 * {-1,0,+1}, term_group = scale group whose plaintext is group_scale_pt[g]),
 * kind 2 = raw route whose plaintext encodes one value in every slot: the
 * encoding of a constant slot vector is a constant poly, so every
 * coefficient of limb l is the limb's first residue, plaintexts[pt][l][0].
 *
 * Return 0 on success, -1 on an argument the oracle cannot evaluate.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef unsigned __int128 u128;

static uint64_t add_mod(uint64_t a, uint64_t b, uint64_t q)
{
    return (uint64_t)(((u128)a + (u128)b) % q);
}

static uint64_t sub_mod(uint64_t a, uint64_t b, uint64_t q)
{
    return (uint64_t)(((u128)a + (u128)q - (u128)b) % q);
}

static uint64_t mul_mod(uint64_t a, uint64_t b, uint64_t q)
{
    return (uint64_t)(((u128)a * (u128)b) % q);
}

static size_t in_idx(uint32_t i, uint32_t c, uint32_t l, uint64_t k, uint32_t L, uint64_t n)
{
    return (((size_t)i * 2 + c) * L + l) * n + k;
}

static size_t pt_idx(uint32_t p, uint32_t l, uint64_t k, uint32_t L, uint64_t n)
{
    return ((size_t)p * L + l) * n + k;
}

/* One output coefficient, straight from the definition above.  covered[e]
 * (may be NULL) marks signed terms evaluated through a shared sum instead;
 * extra_signed[g] (may be NULL) is the value those shared sums add to the
 * signed sum of scale group g. */
static uint64_t eval_one(uint32_t j, uint32_t c, uint32_t l, uint64_t k,
                         uint32_t L, uint64_t n_coef, uint64_t q,
                         const uint32_t *term_offsets, const uint32_t *term_input,
                         const int8_t *term_kind, const int8_t *term_sign,
                         const uint32_t *term_pt, const uint32_t *term_group,
                         const uint32_t *group_scale_pt,
                         const uint64_t *inputs, const uint64_t *plaintexts,
                         const uint8_t *covered, const uint64_t *extra_signed,
                         const uint8_t *group_has_use, const uint8_t *pt_class, uint32_t want_class)
{
    uint64_t y = 0;
    uint32_t e0 = term_offsets[j], e1 = term_offsets[j + 1];

    /* signed route: one signed sum per scale group, then one PMult by gamma */
    for (uint32_t e = e0; e < e1; ++e) {
        if (term_kind[e] != 1)
            continue;
        uint32_t g = term_group[e];
        if (pt_class && pt_class[group_scale_pt[g]] != want_class)
            continue;
        /* visit each scale group once: at its first term in this output */
        int first = 1;
        for (uint32_t f = e0; f < e; ++f)
            if (term_kind[f] == 1 && term_group[f] == g) {
                first = 0;
                break;
            }
        if (!first)
            continue;
        uint64_t s = 0;
        for (uint32_t f = e; f < e1; ++f) {
            if (term_kind[f] != 1 || term_group[f] != g)
                continue;
            if (covered && covered[f])
                continue;
            uint64_t a = inputs[in_idx(term_input[f], c, l, k, L, n_coef)];
            if (term_sign[f] == 1)
                s = add_mod(s, a, q);
            else if (term_sign[f] == -1)
                s = sub_mod(s, a, q);
        }
        if (extra_signed && group_has_use[g])
            s = add_mod(s, extra_signed[g], q);
        uint64_t gamma = plaintexts[pt_idx(group_scale_pt[g], l, k, L, n_coef)];
        y = add_mod(y, mul_mod(gamma, s, q), q);
    }

    /* raw route: one PMult per raw group, added at the same scale */
    for (uint32_t e = e0; e < e1; ++e) {
        if (term_kind[e] != 0 && term_kind[e] != 2)
            continue;
        if (pt_class && pt_class[term_pt[e]] != want_class)
            continue;
        uint64_t a = inputs[in_idx(term_input[e], c, l, k, L, n_coef)];
        uint64_t p = plaintexts[pt_idx(term_pt[e], l, term_kind[e] == 2 ? 0 : k, L, n_coef)];
        y = add_mod(y, mul_mod(p, a, q), q);
    }
    return y;
}

static int check_common(uint32_t L, const uint64_t *moduli, uint32_t n_in, uint32_t n_out,
                        uint32_t n_pt, const uint32_t *term_offsets, const uint32_t *term_input,
                        const int8_t *term_kind, const int8_t *term_sign,
                        const uint32_t *term_pt, const uint32_t *term_group,
                        uint32_t n_groups, const uint32_t *group_scale_pt)
{
    for (uint32_t l = 0; l < L; ++l)
        if (moduli[l] < 2)
            return -1;
    for (uint32_t j = 0; j < n_out; ++j)
        if (term_offsets[j + 1] < term_offsets[j])
            return -1;
    for (uint32_t e = 0; e < term_offsets[n_out]; ++e) {
        if (term_input[e] >= n_in)
            return -1;
        if (term_kind[e] == 0 || term_kind[e] == 2) {
            if (term_pt[e] >= n_pt)
                return -1;
        } else if (term_kind[e] == 1) {
            if (term_group[e] >= n_groups || term_sign[e] < -1 || term_sign[e] > 1)
                return -1;
        } else {
            return -1;
        }
    }
    for (uint32_t g = 0; g < n_groups; ++g)
        if (group_scale_pt[g] >= n_pt)
            return -1;
    return 0;
}

int oracle_linear_eval(uint64_t n_coef, uint32_t L, const uint64_t *moduli,
                       uint32_t n_in, uint32_t n_out, uint32_t n_pt,
                       const uint32_t *term_offsets, const uint32_t *term_input,
                       const int8_t *term_kind, const int8_t *term_sign,
                       const uint32_t *term_pt, const uint32_t *term_group,
                       uint32_t n_groups, const uint32_t *group_scale_pt,
                       const uint64_t *inputs, const uint64_t *plaintexts,
                       uint64_t *outputs)
{
    if (check_common(L, moduli, n_in, n_out, n_pt, term_offsets, term_input, term_kind,
                     term_sign, term_pt, term_group, n_groups, group_scale_pt))
        return -1;
    for (uint32_t j = 0; j < n_out; ++j)
        for (uint32_t c = 0; c < 2; ++c)
            for (uint32_t l = 0; l < L; ++l)
                for (uint64_t k = 0; k < n_coef; ++k)
                    outputs[in_idx(j, c, l, k, L, n_coef)] =
                        eval_one(j, c, l, k, L, n_coef, moduli[l], term_offsets, term_input,
                                 term_kind, term_sign, term_pt, term_group, group_scale_pt,
                                 inputs, plaintexts, NULL, NULL, NULL, NULL, 0);
    return 0;
}

int oracle_linear_eval_classes(uint64_t n_coef, uint32_t L, const uint64_t *moduli,
                               uint32_t n_in, uint32_t n_out, uint32_t n_pt,
                               const uint32_t *term_offsets, const uint32_t *term_input,
                               const int8_t *term_kind, const int8_t *term_sign,
                               const uint32_t *term_pt, const uint32_t *term_group,
                               uint32_t n_groups, const uint32_t *group_scale_pt,
                               uint32_t n_class, const uint8_t *pt_class,
                               const uint64_t *inputs, const uint64_t *plaintexts,
                               uint64_t *outputs)
{
    if (check_common(L, moduli, n_in, n_out, n_pt, term_offsets, term_input, term_kind,
                     term_sign, term_pt, term_group, n_groups, group_scale_pt))
        return -1;
    if (n_class == 0)
        return -1;
    for (uint32_t p = 0; p < n_pt; ++p)
        if (pt_class[p] >= n_class)
            return -1;
    for (uint32_t j = 0; j < n_out; ++j)
        for (uint32_t s = 0; s < n_class; ++s)
            for (uint32_t c = 0; c < 2; ++c)
                for (uint32_t l = 0; l < L; ++l)
                    for (uint64_t k = 0; k < n_coef; ++k)
                        outputs[in_idx(j * n_class + s, c, l, k, L, n_coef)] =
                            eval_one(j, c, l, k, L, n_coef, moduli[l], term_offsets, term_input,
                                     term_kind, term_sign, term_pt, term_group, group_scale_pt,
                                     inputs, plaintexts, NULL, NULL, NULL, pt_class, s);
    return 0;
}

/* Expand node `node` into (input, sign) leaves with the accumulated sign
 * `mult`; adds +1/-1 per leaf into leaf_sign[input].  Children that are
 * nodes must have a smaller index (nodes are listed children first). */
static int expand_node(uint32_t node, int mult, const uint32_t *node_offsets,
                       const uint32_t *child_ref, const int8_t *child_is_node,
                       const int8_t *child_sign, uint32_t n_in, int *leaf_sign, int depth)
{
    if (depth > 64)
        return -1;
    for (uint32_t c = node_offsets[node]; c < node_offsets[node + 1]; ++c) {
        int s = mult * child_sign[c];
        if (child_is_node[c]) {
            if (child_ref[c] >= node)
                return -1;
            if (expand_node(child_ref[c], s, node_offsets, child_ref, child_is_node,
                            child_sign, n_in, leaf_sign, depth + 1))
                return -1;
        } else {
            if (child_ref[c] >= n_in)
                return -1;
            leaf_sign[child_ref[c]] += s;
        }
    }
    return 0;
}

int oracle_linear_eval_dag(uint64_t n_coef, uint32_t L, const uint64_t *moduli,
                           uint32_t n_in, uint32_t n_out, uint32_t n_pt,
                           const uint32_t *term_offsets, const uint32_t *term_input,
                           const int8_t *term_kind, const int8_t *term_sign,
                           const uint32_t *term_pt, const uint32_t *term_group,
                           uint32_t n_groups, const uint32_t *group_scale_pt,
                           uint32_t n_nodes, const uint32_t *node_offsets,
                           const uint32_t *child_ref, const int8_t *child_is_node,
                           const int8_t *child_sign,
                           uint32_t n_uses, const uint32_t *use_output,
                           const uint32_t *use_group, const uint32_t *use_node,
                           const int8_t *use_sign,
                           const uint64_t *inputs, const uint64_t *plaintexts,
                           uint64_t *outputs)
{
    if (check_common(L, moduli, n_in, n_out, n_pt, term_offsets, term_input, term_kind,
                     term_sign, term_pt, term_group, n_groups, group_scale_pt))
        return -1;
    uint32_t n_terms = term_offsets[n_out];
    uint8_t *covered = calloc(n_terms ? n_terms : 1, 1);
    int *leaf = calloc(n_in ? n_in : 1, sizeof(int));
    uint64_t *U = calloc((size_t)(n_nodes ? n_nodes : 1) * 2 * L * n_coef, sizeof(uint64_t));
    uint64_t *extra = calloc(n_groups ? n_groups : 1, sizeof(uint64_t));
    uint8_t *has_use = calloc(n_groups ? n_groups : 1, 1);
    int rc = 0;
    if (!covered || !leaf || !U || !extra || !has_use) {
        rc = -1;
        goto done;
    }

    /* mark the terms each use stands for: a use of sigma*U in (output j,
     * group g) replaces exactly the signed terms of U's leaves in that group */
    for (uint32_t u = 0; u < n_uses; ++u) {
        uint32_t j = use_output[u], g = use_group[u], nd = use_node[u];
        if (j >= n_out || g >= n_groups || nd >= n_nodes) {
            rc = -1;
            goto done;
        }
        memset(leaf, 0, sizeof(int) * n_in);
        if (expand_node(nd, use_sign[u], node_offsets, child_ref, child_is_node, child_sign,
                        n_in, leaf, 0)) {
            rc = -1;
            goto done;
        }
        has_use[g] = 1;
        for (uint32_t i = 0; i < n_in; ++i) {
            if (leaf[i] == 0)
                continue;
            int found = 0;
            for (uint32_t e = term_offsets[j]; e < term_offsets[j + 1]; ++e)
                if (term_kind[e] == 1 && term_group[e] == g && term_input[e] == i &&
                    !covered[e] && term_sign[e] == leaf[i]) {
                    covered[e] = 1;
                    found = 1;
                    break;
                }
            if (!found) {
                rc = -1;
                goto done;
            }
        }
    }

    for (uint32_t l = 0; l < L; ++l) {
        uint64_t q = moduli[l];
        for (uint32_t c = 0; c < 2; ++c)
            for (uint64_t k = 0; k < n_coef; ++k) {
                /* each shared signed sum is formed once (children first) */
                for (uint32_t nd = 0; nd < n_nodes; ++nd) {
                    uint64_t s = 0;
                    for (uint32_t ch = node_offsets[nd]; ch < node_offsets[nd + 1]; ++ch) {
                        uint64_t v = child_is_node[ch]
                                         ? U[in_idx(child_ref[ch], c, l, k, L, n_coef)]
                                         : inputs[in_idx(child_ref[ch], c, l, k, L, n_coef)];
                        s = child_sign[ch] > 0 ? add_mod(s, v, q) : sub_mod(s, v, q);
                    }
                    U[in_idx(nd, c, l, k, L, n_coef)] = s;
                }
                for (uint32_t j = 0; j < n_out; ++j) {
                    for (uint32_t u = 0; u < n_uses; ++u)
                        if (use_output[u] == j)
                            extra[use_group[u]] = 0;
                    for (uint32_t u = 0; u < n_uses; ++u) {
                        if (use_output[u] != j)
                            continue;
                        uint64_t v = U[in_idx(use_node[u], c, l, k, L, n_coef)];
                        uint32_t g = use_group[u];
                        extra[g] = use_sign[u] > 0 ? add_mod(extra[g], v, q)
                                                   : sub_mod(extra[g], v, q);
                    }
                    outputs[in_idx(j, c, l, k, L, n_coef)] =
                        eval_one(j, c, l, k, L, n_coef, q, term_offsets, term_input, term_kind,
                                 term_sign, term_pt, term_group, group_scale_pt, inputs,
                                 plaintexts, covered, extra, has_use, NULL, 0);
                }
            }
    }
done:
    free(covered);
    free(leaf);
    free(U);
    free(extra);
    free(has_use);
    return rc;
}
