// fiona_host.cpp -- C ABI entry points: contexts, plan validation, operation
// statistics, schedule upload and evaluation dispatch (host side).
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <new>

#include "fiona_internal.h"
#include "tiled.h"

typedef unsigned __int128 u128;

// ---------------------------------------------------------------------------
// errors
// ---------------------------------------------------------------------------
static thread_local char g_last_error[512];

int set_error(int code, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
    va_end(ap);
    return code;
}

static int cuda_fail(cudaError_t e, const char *what)
{
    return set_error(FIONA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

extern "C" const char *fiona_last_error(void) { return g_last_error; }

extern "C" int fiona_abi_version(void) { return FIONA_ABI_VERSION; }

extern "C" const char *fiona_status_str(int status)
{
    switch (status) {
    case FIONA_OK: return "ok";
    case FIONA_ERR_ARG: return "invalid argument";
    case FIONA_ERR_MODULUS: return "invalid RNS modulus";
    case FIONA_ERR_PLAN: return "invalid plan";
    case FIONA_ERR_NOMEM: return "out of memory";
    case FIONA_ERR_CUDA: return "CUDA error";
    case FIONA_ERR_RANGE: return "residue out of range";
    case FIONA_ERR_NODEVICE: return "context has no device";
    case FIONA_ERR_TIMEOUT: return "kernel wait timed out";
    case FIONA_ERR_INTERNAL: return "internal consistency check failed";
    default: return "unknown status";
    }
}

// Sets the context's device for the duration of a call and restores the
// caller's device afterwards.
struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev)
    {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard()
    {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

// ---------------------------------------------------------------------------
// moduli
// ---------------------------------------------------------------------------
static uint64_t mulmod_u64(uint64_t a, uint64_t b, uint64_t n) { return (uint64_t)((u128)a * b % n); }

static uint64_t powmod_u64(uint64_t a, uint64_t e, uint64_t n)
{
    uint64_t r = 1 % n;
    a %= n;
    while (e) {
        if (e & 1) r = mulmod_u64(r, a, n);
        a = mulmod_u64(a, a, n);
        e >>= 1;
    }
    return r;
}

// Deterministic Miller-Rabin; the first twelve primes as bases are exact for
// every n < 3.3e24 (Sorenson and Webster, 2015), so for every 64-bit n.
static bool is_prime_u64(uint64_t n)
{
    static const uint64_t bases[] = {2, 3, 5, 7, 11, 13, 17, 19, 23, 29, 31, 37};
    if (n < 2) return false;
    for (uint64_t p : bases)
        if (n % p == 0) return n == p;
    uint64_t d = n - 1;
    int s = 0;
    while ((d & 1) == 0) {
        d >>= 1;
        ++s;
    }
    for (uint64_t a : bases) {
        uint64_t x = powmod_u64(a, d, n);
        if (x == 1 || x == n - 1) continue;
        bool composite = true;
        for (int r = 1; r < s; ++r) {
            x = mulmod_u64(x, x, n);
            if (x == n - 1) {
                composite = false;
                break;
            }
        }
        if (composite) return false;
    }
    return true;
}

static LimbConst limb_constants(uint64_t q)
{
    LimbConst c;
    c.q = q;
    const u128 mu = ~(u128)0 / q;  // floor((2^128 - 1) / q) = floor(2^128 / q) for odd q
    c.mu_hi = (uint64_t)(mu >> 64);
    c.mu_lo = (uint64_t)mu;
    c.mu64 = ~(uint64_t)0 / q;     // floor(2^64 / q) for odd q
    uint32_t k = 0;
    while (k < 64 && (q >> k)) ++k;  // bit length of q
    c.km1 = k - 1;
    c.mk = k + 63 < 128 ? (uint64_t)(((u128)1 << (k + 63)) / q) : 0;  // (used for q < 2^52: k + 63 < 116)
    return c;
}

extern "C" int fiona_ctx_create(uint32_t N, const uint64_t *moduli, uint32_t L, int device,
                                fiona_ctx **out)
{
    if (!out || !moduli) return set_error(FIONA_ERR_ARG, "ctx_create: null argument");
    if (N < 1024 || N > 131072 || (N & (N - 1)))
        return set_error(FIONA_ERR_ARG, "ctx_create: N=%u is not a power of two in [2^10, 2^17]", N);
    if (L < 1 || L > FIONA_MAX_LIMBS)
        return set_error(FIONA_ERR_ARG, "ctx_create: L=%u outside [1, %d]", L, FIONA_MAX_LIMBS);
    for (uint32_t l = 0; l < L; ++l) {
        const uint64_t q = moduli[l];
        if (q >= (1ull << 60) || q < 3 || !(q & 1))
            return set_error(FIONA_ERR_MODULUS, "modulus %u (%llu) is not odd and below 2^60", l,
                             (unsigned long long)q);
        if ((q - 1) % (2ull * N) != 0)
            return set_error(FIONA_ERR_MODULUS, "modulus %u (%llu) is not 1 mod 2N", l,
                             (unsigned long long)q);
        if (!is_prime_u64(q))
            return set_error(FIONA_ERR_MODULUS, "modulus %u (%llu) is not prime", l,
                             (unsigned long long)q);
        for (uint32_t m = 0; m < l; ++m)
            if (moduli[m] == q)
                return set_error(FIONA_ERR_MODULUS, "moduli %u and %u are equal", m, l);
    }
    fiona_ctx *ctx = new (std::nothrow) fiona_ctx;
    if (!ctx) return set_error(FIONA_ERR_NOMEM, "ctx_create: host allocation");
    ctx->N = N;
    ctx->L = L;
    ctx->device = device;
    ctx->moduli.assign(moduli, moduli + L);
    for (uint32_t l = 0; l < L; ++l) {
        ctx->limbs.push_back(limb_constants(moduli[l]));
        ctx->q_max = std::max(ctx->q_max, moduli[l]);
    }
    if (device != FIONA_DEVICE_NONE) {
        int count = 0;
        cudaError_t e = cudaGetDeviceCount(&count);
        if (e != cudaSuccess || device < 0 || device >= count) {
            delete ctx;
            return set_error(FIONA_ERR_CUDA, "ctx_create: device %d unavailable (%s)", device,
                             e == cudaSuccess ? "no such device" : cudaGetErrorString(e));
        }
        DeviceGuard g(device);
        int smem = 0;
        cudaDeviceGetAttribute(&ctx->sm_count, cudaDevAttrMultiProcessorCount, device);
        cudaDeviceGetAttribute(&smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, device);
        ctx->smem_optin = (size_t)smem;
        e = cudaMalloc(&ctx->d_limbs, sizeof(LimbConst) * L);
        if (e == cudaSuccess) e = cudaMalloc(&ctx->d_flag, sizeof(int));
        if (e == cudaSuccess) e = cudaMalloc(&ctx->d_kerr, sizeof(int));
        if (e == cudaSuccess) e = cudaMemset(ctx->d_kerr, 0, sizeof(int));
        if (e == cudaSuccess)
            e = cudaMemcpy(ctx->d_limbs, ctx->limbs.data(), sizeof(LimbConst) * L,
                           cudaMemcpyHostToDevice);
        if (e != cudaSuccess) {
            cudaFree(ctx->d_limbs);
            cudaFree(ctx->d_flag);
            cudaFree(ctx->d_kerr);
            delete ctx;
            return e == cudaErrorMemoryAllocation
                       ? set_error(FIONA_ERR_NOMEM, "ctx_create: device allocation")
                       : cuda_fail(e, "ctx_create");
        }
    }
    *out = ctx;
    return FIONA_OK;
}

extern "C" void fiona_ctx_destroy(fiona_ctx *ctx)
{
    if (!ctx) return;
    if (ctx->device != FIONA_DEVICE_NONE) {
        DeviceGuard g(ctx->device);
        cudaFree(ctx->d_limbs);
        cudaFree(ctx->d_flag);
        cudaFree(ctx->d_kerr);
        free_rescale_tables(ctx);
        free_encode_tables(ctx);
    }
    delete ctx;
}

// ---------------------------------------------------------------------------
// plan validation (the rules of Sec. 4.2 as stated in fiona.h)
// ---------------------------------------------------------------------------
static int validate(const fiona_ctx *ctx, HostPlan &hp)
{
    const uint32_t n_out = hp.n_out;
    if (hp.term_offsets.size() != (size_t)n_out + 1 || hp.term_offsets[0] != 0)
        return set_error(FIONA_ERR_PLAN, "term_offsets[0] must be 0");
    for (uint32_t j = 0; j < n_out; ++j)
        if (hp.term_offsets[j + 1] < hp.term_offsets[j])
            return set_error(FIONA_ERR_PLAN, "term_offsets decrease at output %u", j);
    for (uint32_t g = 0; g < hp.n_groups; ++g) {
        if (hp.group_scale_pt[g] >= hp.n_pt)
            return set_error(FIONA_ERR_PLAN, "group %u: scale plaintext %u >= n_pt", g,
                             hp.group_scale_pt[g]);
        if (hp.group_output[g] >= n_out)
            return set_error(FIONA_ERR_PLAN, "group %u: output %u >= n_out", g, hp.group_output[g]);
    }
    for (uint32_t j = 0; j < n_out; ++j)
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &t = hp.terms[e];
            if (t.input >= hp.n_in)
                return set_error(FIONA_ERR_PLAN, "term %u: input %u >= n_in", e, t.input);
            if (t.reserved != 0) return set_error(FIONA_ERR_PLAN, "term %u: reserved != 0", e);
            if (t.kind == FIONA_TERM_RAW || t.kind == FIONA_TERM_RAW_CONST) {
                if (t.pt >= hp.n_pt)
                    return set_error(FIONA_ERR_PLAN, "term %u: plaintext %u >= n_pt", e, t.pt);
                if (t.sign != 0 || t.group != 0)
                    return set_error(FIONA_ERR_PLAN, "term %u: raw term with sign or group", e);
            } else if (t.kind == FIONA_TERM_TERNARY) {
                if (t.sign < -1 || t.sign > 1)
                    return set_error(FIONA_ERR_PLAN, "term %u: sign %d not in {-1,0,1}", e, t.sign);
                if (t.group >= hp.n_groups)
                    return set_error(FIONA_ERR_PLAN, "term %u: group %u >= n_groups", e, t.group);
                if (hp.group_output[t.group] != j)
                    return set_error(FIONA_ERR_PLAN, "term %u: group %u belongs to output %u, not %u",
                                     e, t.group, hp.group_output[t.group], j);
                if (t.pt != 0) return set_error(FIONA_ERR_PLAN, "term %u: ternary term with pt", e);
            } else {
                return set_error(FIONA_ERR_PLAN, "term %u: unknown kind %d", e, t.kind);
            }
        }
    // shared signed sums: expand each node to its leaves (children first)
    if (hp.node_offsets.size() != (size_t)hp.n_nodes + 1 || hp.node_offsets[0] != 0)
        return set_error(FIONA_ERR_PLAN, "node_offsets[0] must be 0");
    hp.node_leaves.assign(hp.n_nodes, {});
    std::vector<int> acc(hp.n_in, 0);
    for (uint32_t k = 0; k < hp.n_nodes; ++k) {
        if (hp.node_offsets[k + 1] <= hp.node_offsets[k])
            return set_error(FIONA_ERR_PLAN, "node %u has no child", k);
        std::vector<uint32_t> touched;
        for (uint32_t c = hp.node_offsets[k]; c < hp.node_offsets[k + 1]; ++c) {
            const fiona_sum_child &ch = hp.children[c];
            if (ch.reserved != 0 || (ch.sign != 1 && ch.sign != -1) ||
                (ch.is_node != 0 && ch.is_node != 1))
                return set_error(FIONA_ERR_PLAN, "node %u child %u: bad sign/flag", k, c);
            if (ch.is_node) {
                if (ch.ref >= k)
                    return set_error(FIONA_ERR_PLAN, "node %u: child node %u not listed before it",
                                     k, ch.ref);
                for (auto &lv : hp.node_leaves[ch.ref]) {
                    if (acc[lv.first] != 0)
                        return set_error(FIONA_ERR_PLAN, "node %u: input %u appears twice", k,
                                         lv.first);
                    acc[lv.first] = lv.second * ch.sign;
                    touched.push_back(lv.first);
                }
            } else {
                if (ch.ref >= hp.n_in)
                    return set_error(FIONA_ERR_PLAN, "node %u: input %u >= n_in", k, ch.ref);
                if (acc[ch.ref] != 0)
                    return set_error(FIONA_ERR_PLAN, "node %u: input %u appears twice", k, ch.ref);
                acc[ch.ref] = ch.sign;
                touched.push_back(ch.ref);
            }
        }
        std::sort(touched.begin(), touched.end());
        for (uint32_t i : touched) {
            hp.node_leaves[k].push_back({i, acc[i]});
            acc[i] = 0;
        }
    }
    // uses: each must match uncovered signed terms of its output's group
    hp.term_use.assign(hp.terms.size(), -1);
    for (uint32_t u = 0; u < hp.n_uses; ++u) {
        const fiona_sum_use &us = hp.uses[u];
        if (us.output >= n_out || us.group >= hp.n_groups || us.node >= hp.n_nodes ||
            (us.sign != 1 && us.sign != -1) || us.reserved[0] || us.reserved[1] || us.reserved[2])
            return set_error(FIONA_ERR_PLAN, "use %u: index out of range or bad sign", u);
        if (hp.group_output[us.group] != us.output)
            return set_error(FIONA_ERR_PLAN, "use %u: group %u does not belong to output %u", u,
                             us.group, us.output);
        for (auto &lv : hp.node_leaves[us.node]) {
            const int want = lv.second * us.sign;
            bool found = false;
            for (uint32_t e = hp.term_offsets[us.output]; e < hp.term_offsets[us.output + 1]; ++e) {
                const fiona_term &t = hp.terms[e];
                if (t.kind == FIONA_TERM_TERNARY && t.group == us.group && t.input == lv.first &&
                    t.sign == want) {
                    if (hp.term_use[e] >= 0) continue;
                    hp.term_use[e] = (int32_t)u;
                    found = true;
                    break;
                }
            }
            if (!found) {
                // distinguish overlap from a plain mismatch for the message
                for (uint32_t e = hp.term_offsets[us.output]; e < hp.term_offsets[us.output + 1];
                     ++e) {
                    const fiona_term &t = hp.terms[e];
                    if (t.kind == FIONA_TERM_TERNARY && t.group == us.group &&
                        t.input == lv.first && t.sign == want && hp.term_use[e] >= 0)
                        return set_error(FIONA_ERR_PLAN,
                                         "use %u overlaps use %d in output %u (input %u)", u,
                                         hp.term_use[e], us.output, lv.first);
                }
                return set_error(FIONA_ERR_PLAN,
                                 "use %u: output %u group %u has no term (input %u, sign %d)", u,
                                 us.output, us.group, lv.first, want);
            }
        }
    }
    (void)ctx;
    return FIONA_OK;
}

// ---------------------------------------------------------------------------
// statistics in the paper's units
// ---------------------------------------------------------------------------
static void compute_stats(const fiona_ctx *ctx, const HostPlan &hp, fiona_plan_stats_t &s)
{
    memset(&s, 0, sizeof s);
    s.N = ctx->N;
    s.L = ctx->L;
    s.n_in = hp.n_in;
    s.n_out = hp.n_out;
    s.n_pt = hp.n_pt;
    s.n_groups = hp.n_groups;
    s.n_nodes = hp.n_nodes;
    s.n_uses = hp.n_uses;
    // pt_used: 1 = read whole (raw or scale plaintext), 2 = only residue 0 of each limb
    std::vector<uint8_t> in_used(hp.n_in, 0), pt_used(hp.n_pt, 0), grp_used(hp.n_groups, 0);
    for (uint32_t j = 0; j < hp.n_out; ++j) {
        uint64_t S = 0, R = 0, ops_direct = 0;
        std::map<uint32_t, uint64_t> uses_in_group;
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &t = hp.terms[e];
            ++s.n_terms;
            if (t.kind == FIONA_TERM_RAW || t.kind == FIONA_TERM_RAW_CONST) {
                ++R;
                in_used[t.input] = 1;
                if (t.kind == FIONA_TERM_RAW)
                    pt_used[t.pt] = 1;
                else if (!pt_used[t.pt])
                    pt_used[t.pt] = 2;
            } else if (t.sign == 0) {
                ++s.n_skipped_terms;
            } else {
                ++S;
                in_used[t.input] = 1;
                if (!grp_used[t.group]) {
                    grp_used[t.group] = 1;
                    pt_used[hp.group_scale_pt[t.group]] = 1;
                }
                if (hp.term_use[e] < 0) ++ops_direct;
            }
        }
        for (uint32_t u = 0; u < hp.n_uses; ++u)
            if (hp.uses[u].output == j) ++ops_direct;  // each use is one operand
        s.n_raw_terms += R;
        s.n_signed_terms += S;
        if (S + R > 0) {
            s.addsub_flat += S + R - 1;
            s.addsub_shared += ops_direct + R - 1;
            s.rescale_combined += 1;
        }
        s.rescale_separate += (S > 0) + (R > 0);
    }
    for (uint32_t k = 0; k < hp.n_nodes; ++k)
        s.addsub_shared += hp.node_offsets[k + 1] - hp.node_offsets[k] - 1;
    for (uint32_t g = 0; g < hp.n_groups; ++g) s.n_scale_groups_used += grp_used[g];
    for (uint8_t v : in_used) s.n_inputs_used += v;
    uint64_t n_pt_whole = 0, n_pt_const = 0;
    for (uint8_t v : pt_used) {
        s.n_plaintexts_used += v != 0;
        n_pt_whole += v == 1;
        n_pt_const += v == 2;
    }
    s.n_nonzero_terms = s.n_raw_terms + s.n_signed_terms;
    s.pmult_per_term = s.n_raw_terms + s.n_signed_terms;
    s.pmult_grouped = s.n_raw_terms + s.n_scale_groups_used;
    const uint64_t limb_poly = (uint64_t)ctx->N * ctx->L * 8;
    s.bytes_min = limb_poly * (2 * s.n_inputs_used + n_pt_whole + 2ull * hp.n_out) + n_pt_const * ctx->L * 8ull;
    s.wide_products = 2ull * ctx->L * ctx->N * s.pmult_grouped;
}

// ---------------------------------------------------------------------------
// direct schedule: per output, its used scale groups (signed operands) and
// its raw terms, evaluated term by term without the DAG
// ---------------------------------------------------------------------------
static int upload(fiona_plan *p, const std::vector<std::pair<const void *, size_t>> &parts,
                  std::vector<size_t> &offsets)
{
    size_t total = 0;
    offsets.clear();
    for (auto &pr : parts) {
        offsets.push_back(total);
        total += (pr.second + 255) & ~(size_t)255;
    }
    if (total == 0) total = 256;
    std::vector<uint8_t> host(total, 0);
    for (size_t i = 0; i < parts.size(); ++i)
        if (parts[i].second) memcpy(host.data() + offsets[i], parts[i].first, parts[i].second);
    cudaError_t e = cudaMalloc(&p->sched.blob, total);
    if (e != cudaSuccess) return set_error(FIONA_ERR_NOMEM, "schedule upload: %s", cudaGetErrorString(e));
    p->sched.bytes = total;
    e = cudaMemcpy(p->sched.blob, host.data(), total, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "schedule upload");
    return FIONA_OK;
}

// The direct kernel's schedule of a plan: per output its scale-group segments
// (each a run of signed operations, bit 31 = subtract) and its raw terms
// (input, plaintext with bit 31 = constant plaintext).
struct DirectSchedule {
    std::vector<DirOut> outs;
    std::vector<DirSeg> segs;
    std::vector<uint32_t> ops, raw_in, raw_pt;
};

static DirectSchedule direct_schedule(const HostPlan &hp)
{
    DirectSchedule d;
    d.outs.resize(hp.n_out);
    for (uint32_t j = 0; j < hp.n_out; ++j) {
        DirOut &o = d.outs[j];
        o.seg_begin = (uint32_t)d.segs.size();
        std::vector<uint32_t> seen;
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &t = hp.terms[e];
            if (t.kind != FIONA_TERM_TERNARY || t.sign == 0) continue;
            if (std::find(seen.begin(), seen.end(), t.group) != seen.end()) continue;
            seen.push_back(t.group);
            DirSeg sg{};
            sg.scale_pt = hp.group_scale_pt[t.group];
            sg.op_begin = (uint32_t)d.ops.size();
            for (uint32_t f = e; f < hp.term_offsets[j + 1]; ++f) {
                const fiona_term &u = hp.terms[f];
                if (u.kind == FIONA_TERM_TERNARY && u.group == t.group && u.sign != 0)
                    d.ops.push_back(u.input | (u.sign < 0 ? 0x80000000u : 0u));
            }
            sg.op_end = (uint32_t)d.ops.size();
            d.segs.push_back(sg);
        }
        o.seg_end = (uint32_t)d.segs.size();
        o.raw_begin = (uint32_t)d.raw_in.size();
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &t = hp.terms[e];
            if (t.kind != FIONA_TERM_RAW && t.kind != FIONA_TERM_RAW_CONST) continue;
            d.raw_in.push_back(t.input);
            d.raw_pt.push_back(t.pt | (t.kind == FIONA_TERM_RAW_CONST ? 0x80000000u : 0u));
        }
        o.raw_end = (uint32_t)d.raw_in.size();
    }
    return d;
}

static int lower_direct(fiona_plan *p)
{
    const DirectSchedule d = direct_schedule(p->hp);
    std::vector<size_t> off;
    int rc = upload(p, {{d.outs.data(), d.outs.size() * sizeof(DirOut)},
                        {d.segs.data(), d.segs.size() * sizeof(DirSeg)},
                        {d.ops.data(), d.ops.size() * 4},
                        {d.raw_in.data(), d.raw_in.size() * 4},
                        {d.raw_pt.data(), d.raw_pt.size() * 4}},
                    off);
    if (rc) return rc;
    uint8_t *b = (uint8_t *)p->sched.blob;
    p->d_dir_out = (const DirOut *)(b + off[0]);
    p->d_dir_seg = (const DirSeg *)(b + off[1]);
    p->d_sig_ops = (const uint32_t *)(b + off[2]);
    p->d_raw_input = (const uint32_t *)(b + off[3]);
    p->d_raw_pt = (const uint32_t *)(b + off[4]);
    return FIONA_OK;
}

// Host image for fiona_linear_eval_static: the limb constants and the direct
// schedule (the same parts as lower_direct's), each part 16-byte aligned.
static void build_static_image(fiona_plan *p)
{
    const DirectSchedule d = direct_schedule(p->hp);
    const std::pair<const void *, size_t> parts[6] = {
        {p->ctx->limbs.data(), p->ctx->limbs.size() * sizeof(LimbConst)},
        {d.outs.data(), d.outs.size() * sizeof(DirOut)},
        {d.segs.data(), d.segs.size() * sizeof(DirSeg)},
        {d.ops.data(), d.ops.size() * 4},
        {d.raw_in.data(), d.raw_in.size() * 4},
        {d.raw_pt.data(), d.raw_pt.size() * 4}};
    size_t total = 0;
    for (int i = 0; i < 6; ++i) {
        p->static_off[i] = total;
        total += (parts[i].second + 15) & ~(size_t)15;
    }
    p->static_image.assign(total, 0);
    for (int i = 0; i < 6; ++i)
        if (parts[i].second) memcpy(p->static_image.data() + p->static_off[i], parts[i].first, parts[i].second);
}

static void release_device(fiona_plan *p)
{
    if (!p->ctx || p->ctx->device == FIONA_DEVICE_NONE) {
        if (p->tiled) free_tiled(p);  // host-only schedule: nothing on a device
        return;
    }
    DeviceGuard g(p->ctx->device);
    if (p->tiled) free_tiled(p);
    cudaFree(p->sched.blob);
    p->sched.blob = nullptr;
    if (p->copy_in_stream) cudaStreamDestroy((cudaStream_t)p->copy_in_stream);
    if (p->copy_out_stream) cudaStreamDestroy((cudaStream_t)p->copy_out_stream);
    p->copy_in_stream = p->copy_out_stream = nullptr;
    for (void **set : {p->ev_in, p->ev_kernel, p->ev_out})
        for (uint32_t c = 0; c < fiona_plan::kHostChunks; ++c)
            if (set[c]) {
                cudaEventDestroy((cudaEvent_t)set[c]);
                set[c] = nullptr;
            }
    if (p->ev_start) cudaEventDestroy((cudaEvent_t)p->ev_start);
    p->ev_start = nullptr;
}

// The tiled schedule is optional: a plan whose tile does not fit in shared
// memory runs on the direct kernel.  A schedule that fails its own check is
// a library bug and is reported.
static int lower_tiled_optional(fiona_plan *p)
{
    const int rc = lower_tiled(p);
    if (rc == FIONA_ERR_INTERNAL) return rc;
    if (rc != FIONA_OK) p->tiled = nullptr;
    set_error(FIONA_OK, "");
    return FIONA_OK;
}

// Kernel choice: TILED for layers with more than one output whose tile fits
// in shared memory (every input is then read from HBM once), DIRECT otherwise
// (a single output has no input reuse to exploit).
static int select_kernel(fiona_plan *p, int which)
{
    int k;
    if (which == FIONA_KERNEL_DIRECT)
        k = 0;
    else if (which == FIONA_KERNEL_TILED)
        k = 1;
    else if (which == FIONA_KERNEL_AUTO)
        k = (p->tiled && p->hp.n_out > 1) ? 1 : 0;
    else
        return set_error(FIONA_ERR_ARG, "select_kernel: unknown variant %d", which);
    if (k == 1 && !p->tiled && p->ctx->device != FIONA_DEVICE_NONE)
        return set_error(FIONA_ERR_ARG, "select_kernel: the tiled kernel cannot run this plan");
    p->kernel = k;
    fiona_plan_stats_t &s = p->stats;
    if (k == 1 && p->tiled) {
        s.kernel = FIONA_KERNEL_TILED;
        s.tile_coeffs = p->tiled->tile;
        s.warps_per_cta = p->tiled->warps;
        s.smem_bytes = (uint32_t)p->tiled->smem;
        s.ctas_per_sm = p->tiled->ctas_per_sm;
        s.nodes_materialized = p->tiled->nodes_kept;
        s.addsub_executed = p->tiled->addsub;
        s.tensor_core_sums = p->tiled->tc ? p->tiled->args.tc_groups : 0;
        s.source_offsets = p->tiled->args.src_offsets;
        s.const_raw_all = p->tiled->args.kc_all;
    } else {
        s.kernel = FIONA_KERNEL_DIRECT;
        s.tile_coeffs = 256;
        s.warps_per_cta = 4;
        s.smem_bytes = 0;
        s.ctas_per_sm = 0;
        s.nodes_materialized = 0;
        s.addsub_executed = (uint32_t)std::min<uint64_t>(s.addsub_flat, 0xffffffffu);
        s.tensor_core_sums = 0;
        s.source_offsets = 0;
        s.const_raw_all = 0;
    }
    return FIONA_OK;
}

extern "C" int fiona_plan_select_kernel(fiona_plan *p, int which)
{
    if (!p) return set_error(FIONA_ERR_ARG, "select_kernel: null plan");
    return select_kernel(p, which);
}

extern "C" int fiona_device_check(const fiona_ctx *ctx, void *stream)
{
    if (!ctx) return set_error(FIONA_ERR_ARG, "device_check: null ctx");
    if (ctx->device == FIONA_DEVICE_NONE)
        return set_error(FIONA_ERR_NODEVICE, "device_check: validation-only context");
    DeviceGuard g(ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "device_check: cannot select device %d", ctx->device);
    cudaStream_t s = (cudaStream_t)stream;
    int flag = 0;
    cudaError_t e = cudaStreamSynchronize(s);
    if (e == cudaSuccess) e = cudaMemcpy(&flag, ctx->d_kerr, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && flag) e = cudaMemset(ctx->d_kerr, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "device_check");
    if (flag & 1) return set_error(FIONA_ERR_TIMEOUT, "a kernel gave up waiting for its bulk copies");
    if (flag & 2) return set_error(FIONA_ERR_RANGE, "an encoded coefficient was not finite or reached 2^62");
    return FIONA_OK;
}

extern "C" int fiona_plan_create(const fiona_ctx *ctx, uint32_t n_in, uint32_t n_out,
                                 uint32_t n_pt, const uint32_t *term_offsets,
                                 const fiona_term *terms, uint32_t n_groups,
                                 const uint32_t *group_scale_pt, const uint32_t *group_output,
                                 uint32_t n_nodes, const uint32_t *node_offsets,
                                 const fiona_sum_child *children, uint32_t n_uses,
                                 const fiona_sum_use *uses, fiona_plan **out)
{
    if (!ctx || !out || !term_offsets) return set_error(FIONA_ERR_ARG, "plan_create: null argument");
    if (n_in > 65535 || n_out > 65535 || n_pt >= (1u << 24) || n_groups >= (1u << 24) ||
        n_nodes > 65535 || n_uses >= (1u << 24))
        return set_error(FIONA_ERR_ARG, "plan_create: size limit exceeded");
    if ((n_groups && (!group_scale_pt || !group_output)) || (n_uses && !uses) ||
        (n_nodes && (!node_offsets || !children)))
        return set_error(FIONA_ERR_ARG, "plan_create: null array with nonzero count");
    const uint64_t n_terms = term_offsets[n_out];
    if (n_terms && !terms) return set_error(FIONA_ERR_ARG, "plan_create: null terms");
    if (n_terms >= (1u << 28)) return set_error(FIONA_ERR_ARG, "plan_create: too many terms");

    fiona_plan *p = new (std::nothrow) fiona_plan;
    if (!p) return set_error(FIONA_ERR_NOMEM, "plan_create: host allocation");
    p->ctx = ctx;
    HostPlan &hp = p->hp;
    hp.n_in = n_in;
    hp.n_out = n_out;
    hp.n_pt = n_pt;
    hp.n_groups = n_groups;
    hp.n_nodes = n_nodes;
    hp.n_uses = n_uses;
    hp.term_offsets.assign(term_offsets, term_offsets + n_out + 1);
    if (hp.term_offsets[0] != 0) {
        delete p;
        return set_error(FIONA_ERR_PLAN, "term_offsets[0] must be 0");
    }
    hp.terms.assign(terms, terms + n_terms);
    if (n_groups) {
        hp.group_scale_pt.assign(group_scale_pt, group_scale_pt + n_groups);
        hp.group_output.assign(group_output, group_output + n_groups);
    }
    if (n_nodes) {
        hp.node_offsets.assign(node_offsets, node_offsets + n_nodes + 1);
        if (hp.node_offsets[0] != 0 || hp.node_offsets[n_nodes] > (1u << 24)) {
            delete p;
            return set_error(FIONA_ERR_PLAN, "node_offsets malformed");
        }
        hp.children.assign(children, children + hp.node_offsets[n_nodes]);
    } else {
        hp.node_offsets.assign(1, 0);
    }
    if (n_uses) hp.uses.assign(uses, uses + n_uses);

    int rc = validate(ctx, hp);
    if (rc) {
        delete p;
        return rc;
    }
    compute_stats(ctx, hp, p->stats);
    // lazy-reduction budgets from the largest modulus
    const u128 qm1 = ctx->q_max - 1;
    const u128 mb = (~(u128)0) / (qm1 * qm1);
    p->mac_budget = (uint32_t)std::min<u128>(mb, 1u << 30);
    const uint64_t sb = ~(uint64_t)0 / (ctx->q_max - 1);
    p->signed_budget = (uint32_t)std::min<uint64_t>(sb, 1u << 30);
    build_static_image(p);

    if (ctx->device != FIONA_DEVICE_NONE) {
        DeviceGuard g(ctx->device);
        if (!g.ok) {
            delete p;
            return set_error(FIONA_ERR_CUDA, "plan_create: cannot select device %d", ctx->device);
        }
        rc = lower_direct(p);
        if (rc == FIONA_OK && hp.n_out > 0) rc = lower_tiled_optional(p);
        if (rc == FIONA_OK) {
            cudaError_t e = cudaStreamCreateWithFlags((cudaStream_t *)&p->copy_in_stream,
                                                      cudaStreamNonBlocking);
            if (e == cudaSuccess)
                e = cudaStreamCreateWithFlags((cudaStream_t *)&p->copy_out_stream,
                                              cudaStreamNonBlocking);
            for (void **set : {p->ev_in, p->ev_kernel, p->ev_out})
                for (uint32_t c = 0; c < fiona_plan::kHostChunks && e == cudaSuccess; ++c)
                    e = cudaEventCreateWithFlags((cudaEvent_t *)&set[c], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags((cudaEvent_t *)&p->ev_start, cudaEventDisableTiming);
            if (e != cudaSuccess) rc = cuda_fail(e, "plan_create: stream");
        }
        if (rc) {
            release_device(p);
            delete p;
            return rc;
        }
    }
    if (ctx->device == FIONA_DEVICE_NONE && hp.n_out > 0) {
        // the tiled lowering (and its schedule check) also runs without a
        // GPU, so a validation-only context reports the shape it would use
        rc = lower_tiled_optional(p);
        if (rc) {
            delete p;
            return rc;
        }
    }
    select_kernel(p, FIONA_KERNEL_AUTO);
    *out = p;
    return FIONA_OK;
}

// Plaintext scale classes: output j of the description becomes results
// j * n_class + s, each holding the terms of j whose plaintext has class s
// (a scale group by its gamma); the validation and lowering are those of the
// expanded layer (Sec. 4.2 "Combining the Signed and Raw Routes": routes are
// combined within one scale only).
extern "C" int fiona_plan_create_classes(const fiona_ctx *ctx, uint32_t n_in, uint32_t n_out, uint32_t n_pt,
                                         const uint32_t *term_offsets, const fiona_term *terms,
                                         uint32_t n_groups, const uint32_t *group_scale_pt,
                                         const uint32_t *group_output, uint32_t n_nodes,
                                         const uint32_t *node_offsets, const fiona_sum_child *children,
                                         uint32_t n_uses, const fiona_sum_use *uses, uint32_t n_class,
                                         const uint8_t *pt_class, fiona_plan **out)
{
    if (n_class == 0 || n_class > 255) return set_error(FIONA_ERR_ARG, "plan_create_classes: n_class %u", n_class);
    if (n_class == 1)
        return fiona_plan_create(ctx, n_in, n_out, n_pt, term_offsets, terms, n_groups, group_scale_pt,
                                 group_output, n_nodes, node_offsets, children, n_uses, uses, out);
    if (!ctx || !out || !term_offsets) return set_error(FIONA_ERR_ARG, "plan_create_classes: null argument");
    if (n_pt && !pt_class) return set_error(FIONA_ERR_ARG, "plan_create_classes: null pt_class");
    if ((uint64_t)n_out * n_class > 65535) return set_error(FIONA_ERR_ARG, "plan_create_classes: too many results");
    if ((n_groups && (!group_scale_pt || !group_output)) || (n_uses && !uses))
        return set_error(FIONA_ERR_ARG, "plan_create_classes: null array with nonzero count");
    const uint64_t n_terms = term_offsets[n_out];
    if (n_terms && !terms) return set_error(FIONA_ERR_ARG, "plan_create_classes: null terms");
    for (uint32_t pi = 0; pi < n_pt; ++pi)
        if (pt_class[pi] >= n_class)
            return set_error(FIONA_ERR_PLAN, "plaintext %u has class %u >= %u", pi, pt_class[pi], n_class);
    // the class of a plaintext index (out-of-range indices are left to the
    // validation of the expanded plan)
    auto cls = [&](uint32_t pt) -> uint32_t { return pt < n_pt ? pt_class[pt] : 0; };
    auto gcls = [&](uint32_t g) -> uint32_t { return g < n_groups ? cls(group_scale_pt[g]) : 0; };
    for (uint32_t j = 0; j < n_out; ++j)
        if (term_offsets[j + 1] < term_offsets[j]) return set_error(FIONA_ERR_PLAN, "term_offsets decrease");
    std::vector<uint32_t> offs(1, 0);
    std::vector<fiona_term> ts;
    ts.reserve(n_terms);
    for (uint32_t j = 0; j < n_out; ++j)
        for (uint32_t s = 0; s < n_class; ++s) {
            for (uint32_t e = term_offsets[j]; e < term_offsets[j + 1]; ++e) {
                const fiona_term &t = terms[e];
                const uint32_t c = t.kind == FIONA_TERM_TERNARY ? gcls(t.group) : cls(t.pt);
                if (c == s) ts.push_back(t);
            }
            offs.push_back((uint32_t)ts.size());
        }
    std::vector<uint32_t> gout(n_groups);
    for (uint32_t g = 0; g < n_groups; ++g)
        gout[g] = group_output[g] < n_out ? group_output[g] * n_class + gcls(g) : n_out * n_class;
    std::vector<fiona_sum_use> us(uses, uses + n_uses);
    for (auto &u : us) u.output = u.output < n_out ? u.output * n_class + gcls(u.group) : n_out * n_class;
    return fiona_plan_create(ctx, n_in, n_out * n_class, n_pt, offs.data(), ts.data(), n_groups, group_scale_pt,
                             gout.data(), n_nodes, node_offsets, children, n_uses, us.data(), out);
}

extern "C" void fiona_plan_destroy(fiona_plan *p)
{
    if (!p) return;
    release_device(p);
    delete p;
}

extern "C" int fiona_plan_stats(const fiona_plan *p, fiona_plan_stats_t *out)
{
    if (!p || !out) return set_error(FIONA_ERR_ARG, "plan_stats: null argument");
    *out = p->stats;
    return FIONA_OK;
}

// ---------------------------------------------------------------------------
// evaluation
// ---------------------------------------------------------------------------
static int check_eval_args(const fiona_plan *p, const void *in, const void *pt, const void *out)
{
    if (!p) return set_error(FIONA_ERR_ARG, "linear_eval: null plan");
    if (p->ctx->device == FIONA_DEVICE_NONE)
        return set_error(FIONA_ERR_NODEVICE, "linear_eval: validation-only context");
    if (!out) return set_error(FIONA_ERR_ARG, "linear_eval: null outputs");
    if ((p->hp.n_in && !in) || (p->hp.n_pt && !pt))
        return set_error(FIONA_ERR_ARG, "linear_eval: null inputs or plaintexts");
    if (((uintptr_t)in | (uintptr_t)pt | (uintptr_t)out) & 15)
        return set_error(FIONA_ERR_ARG, "linear_eval: buffers must be 16-byte aligned");
    return FIONA_OK;
}

static int launch_range(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                        uint64_t *out, uint32_t l0, uint32_t l1, uint32_t layout_L)
{
    if (p->kernel == 1) return launch_tiled(p, stream, in, pt, out, l0, l1, layout_L);
    return launch_direct(p, stream, in, pt, out, l0, l1, layout_L);
}

extern "C" int fiona_linear_eval(const fiona_plan *p, void *stream, const uint64_t *in,
                                 const uint64_t *pt, uint64_t *out)
{
    int rc = check_eval_args(p, in, pt, out);
    if (rc) return rc;
    if (p->hp.n_out == 0) return FIONA_OK;
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval: cannot select device %d", p->ctx->device);
    return launch_range(p, stream, in, pt, out, 0, p->ctx->L, p->ctx->L);
}

extern "C" int fiona_linear_eval_level(const fiona_plan *p, void *stream, uint32_t L_eval,
                                       const uint64_t *in, const uint64_t *pt, uint64_t *out)
{
    if (!p) return set_error(FIONA_ERR_ARG, "linear_eval_level: null plan");
    if (L_eval < 1 || L_eval > p->ctx->L)
        return set_error(FIONA_ERR_ARG, "linear_eval_level: level %u outside [1, %u]", L_eval, p->ctx->L);
    int rc = check_eval_args(p, in, pt, out);
    if (rc) return rc;
    if (p->hp.n_out == 0) return FIONA_OK;
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval_level: cannot select device %d", p->ctx->device);
    return launch_range(p, stream, in, pt, out, 0, L_eval, L_eval);
}

// Queue the host-buffer evaluation: per limb chunk (one limb each, at most
// kHostChunks), its input copy on the plan's input stream, its kernel on
// `stream`, its output copy on the plan's output stream, each ordered after
// the step before it and after the previous call's use of the same chunk of
// d_in (its kernel) and d_out (its output copy); with `join`, `stream` ends
// waiting for the last output copy (a queued call leaves that to
// fiona_linear_eval_host_join, so that the next call's input copies, which
// wait for the work on `stream` before them, need not wait for these output
// copies too).
static int eval_host_enqueue(const fiona_plan *p, cudaStream_t s, const uint64_t *h_in, const uint64_t *d_pt,
                             uint64_t *h_out, uint64_t *d_in, uint64_t *d_out, bool join)
{
    const uint32_t L = p->ctx->L, N = p->ctx->N;
    const size_t pitch = (size_t)L * N * 8;
    cudaStream_t sin = (cudaStream_t)p->copy_in_stream, sout = (cudaStream_t)p->copy_out_stream;
    const uint32_t chunks = std::min<uint32_t>(L, fiona_plan::kHostChunks);
    auto ev = [](void *const *set, uint32_t c) { return (cudaEvent_t)set[c]; };
    // the copies must not run ahead of work already queued on `stream`
    cudaError_t e = cudaEventRecord((cudaEvent_t)p->ev_start, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(sin, (cudaEvent_t)p->ev_start, 0);
    for (uint32_t c = 0; c < chunks && e == cudaSuccess; ++c) {
        const uint32_t l0 = L * c / chunks, l1 = L * (c + 1) / chunks;
        const size_t width = (size_t)(l1 - l0) * N * 8;
        if ((e = cudaStreamWaitEvent(sin, ev(p->ev_kernel, c), 0)) != cudaSuccess) break;
        if (p->hp.n_in) {
            e = cudaMemcpy2DAsync(d_in + (size_t)l0 * N, pitch, h_in + (size_t)l0 * N, pitch, width,
                                  (size_t)p->hp.n_in * 2, cudaMemcpyHostToDevice, sin);
            if (e != cudaSuccess) break;
        }
        if ((e = cudaEventRecord(ev(p->ev_in, c), sin)) != cudaSuccess) break;
        if ((e = cudaStreamWaitEvent(s, ev(p->ev_in, c), 0)) != cudaSuccess) break;
        if ((e = cudaStreamWaitEvent(s, ev(p->ev_out, c), 0)) != cudaSuccess) break;
        if (const int rc = launch_range(p, s, d_in, d_pt, d_out, l0, l1, L)) return rc;
        if ((e = cudaEventRecord(ev(p->ev_kernel, c), s)) != cudaSuccess) break;
        if ((e = cudaStreamWaitEvent(sout, ev(p->ev_kernel, c), 0)) != cudaSuccess) break;
        e = cudaMemcpy2DAsync(h_out + (size_t)l0 * N, pitch, d_out + (size_t)l0 * N, pitch, width,
                              (size_t)p->hp.n_out * 2, cudaMemcpyDeviceToHost, sout);
        if (e == cudaSuccess) e = cudaEventRecord(ev(p->ev_out, c), sout);
    }
    if (e == cudaSuccess && join) e = cudaStreamWaitEvent(s, ev(p->ev_out, chunks - 1), 0);
    if (e != cudaSuccess) return cuda_fail(e, "linear_eval_host");
    return FIONA_OK;
}

static int check_host_args(const fiona_plan *p, const uint64_t *h_in, const uint64_t *d_pt, const uint64_t *h_out,
                           const uint64_t *d_in, const uint64_t *d_out)
{
    int rc = check_eval_args(p, d_in, d_pt, d_out);
    if (rc) return rc;
    if ((p->hp.n_in && !h_in) || !h_out) return set_error(FIONA_ERR_ARG, "linear_eval_host: null host buffer");
    return FIONA_OK;
}

extern "C" int fiona_linear_eval_host(const fiona_plan *p, void *stream, const uint64_t *h_in,
                                      const uint64_t *d_pt, uint64_t *h_out, uint64_t *d_in,
                                      uint64_t *d_out)
{
    if (const int rc = check_host_args(p, h_in, d_pt, h_out, d_in, d_out)) return rc;
    if (p->hp.n_out == 0) return FIONA_OK;
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval_host: cannot select device %d", p->ctx->device);
    cudaStream_t s = (cudaStream_t)stream;
    const int rc = eval_host_enqueue(p, s, h_in, d_pt, h_out, d_in, d_out, true);
    // whatever was queued completes before the call returns
    const cudaError_t e = cudaStreamSynchronize(s);
    const cudaError_t e2 = cudaStreamSynchronize((cudaStream_t)p->copy_out_stream);
    const cudaError_t e3 = cudaStreamSynchronize((cudaStream_t)p->copy_in_stream);
    if (rc) return rc;
    if (e != cudaSuccess) return cuda_fail(e, "linear_eval_host: sync");
    if (e2 != cudaSuccess) return cuda_fail(e2, "linear_eval_host: sync");
    if (e3 != cudaSuccess) return cuda_fail(e3, "linear_eval_host: sync");
    return FIONA_OK;
}

extern "C" int fiona_linear_eval_host_async(const fiona_plan *p, void *stream, const uint64_t *h_in,
                                            const uint64_t *d_pt, uint64_t *h_out, uint64_t *d_in,
                                            uint64_t *d_out)
{
    if (const int rc = check_host_args(p, h_in, d_pt, h_out, d_in, d_out)) return rc;
    if (p->hp.n_out == 0) return FIONA_OK;
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval_host_async: cannot select device %d", p->ctx->device);
    return eval_host_enqueue(p, (cudaStream_t)stream, h_in, d_pt, h_out, d_in, d_out, false);
}

extern "C" int fiona_linear_eval_host_join(const fiona_plan *p, void *stream)
{
    if (!p) return set_error(FIONA_ERR_ARG, "linear_eval_host_join: null plan");
    if (p->ctx->device == FIONA_DEVICE_NONE)
        return set_error(FIONA_ERR_NODEVICE, "linear_eval_host_join: validation-only context");
    if (p->hp.n_out == 0) return FIONA_OK;
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval_host_join: cannot select device %d", p->ctx->device);
    const uint32_t chunks = std::min<uint32_t>(p->ctx->L, fiona_plan::kHostChunks);
    // the output copies run in order on one stream: the last chunk's is the last
    const cudaError_t e = cudaStreamWaitEvent((cudaStream_t)stream, (cudaEvent_t)p->ev_out[chunks - 1], 0);
    if (e != cudaSuccess) return cuda_fail(e, "linear_eval_host_join");
    return FIONA_OK;
}

extern "C" int fiona_linear_eval_static(const fiona_plan *p, void *stream, const uint64_t *in,
                                        const uint64_t *pt, uint64_t *out)
{
    if (!p) return set_error(FIONA_ERR_ARG, "linear_eval_static: null plan");
    if (!out) return set_error(FIONA_ERR_ARG, "linear_eval_static: null outputs");
    if ((p->hp.n_in && !in) || (p->hp.n_pt && !pt))
        return set_error(FIONA_ERR_ARG, "linear_eval_static: null inputs or plaintexts");
    if (((uintptr_t)in | (uintptr_t)pt | (uintptr_t)out) & 15)
        return set_error(FIONA_ERR_ARG, "linear_eval_static: buffers must be 16-byte aligned");
    if (p->static_image.size() > kStaticAreaBytes)
        return set_error(FIONA_ERR_ARG,
                         "linear_eval_static: this layer needs %zu bytes of schedule, more than "
                         "the %zu-byte static area; use fiona_linear_eval",
                         p->static_image.size(), kStaticAreaBytes);
    if (p->hp.n_out == 0) return FIONA_OK;
    // a validation-only context runs on the current device (see the header)
    if (p->ctx->device == FIONA_DEVICE_NONE) return launch_direct_static(p, stream, in, pt, out);
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval_static: cannot select device %d", p->ctx->device);
    return launch_direct_static(p, stream, in, pt, out);
}

static bool overlaps(const void *a, uint64_t a_bytes, const void *b, uint64_t b_bytes)
{
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return a_bytes && b_bytes && x < y + b_bytes && y < x + a_bytes;
}

static int check_rescale_args(const fiona_ctx *ctx, uint32_t L_cur, uint64_t count, const uint64_t *polys,
                              const uint64_t *out, const char *who)
{
    if (!ctx) return set_error(FIONA_ERR_ARG, "%s: null ctx", who);
    if (ctx->device == FIONA_DEVICE_NONE) return set_error(FIONA_ERR_NODEVICE, "%s: validation-only context", who);
    if (L_cur < 2 || L_cur > ctx->L)
        return set_error(FIONA_ERR_ARG, "%s: level %u outside [2, %u]", who, L_cur, ctx->L);
    if (count > (1ull << 40) / ((uint64_t)L_cur * ctx->N))
        return set_error(FIONA_ERR_ARG, "%s: %llu polys", who, (unsigned long long)count);
    if (count == 0) return FIONA_OK;
    if (!polys || !out) return set_error(FIONA_ERR_ARG, "%s: null buffer", who);
    if (((uintptr_t)polys | (uintptr_t)out) & 15)
        return set_error(FIONA_ERR_ARG, "%s: buffers must be 16-byte aligned", who);
    const uint64_t poly_bytes = (uint64_t)ctx->N * 8;
    if (overlaps(polys, count * L_cur * poly_bytes, out, count * (L_cur - 1) * poly_bytes))
        return set_error(FIONA_ERR_ARG, "%s: output overlaps the input", who);
    return FIONA_OK;
}

extern "C" int fiona_rescale(const fiona_ctx *ctx, void *stream, uint32_t L_cur, uint64_t count, uint64_t *polys,
                             uint64_t *out, uint32_t flags)
{
    if (flags & ~(uint32_t)FIONA_RESCALE_ROUND) return set_error(FIONA_ERR_ARG, "rescale: unknown flags 0x%x", flags);
    int rc = check_rescale_args(ctx, L_cur, count, polys, out, "rescale");
    if (rc) return rc;
    DeviceGuard g(ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "rescale: cannot select device %d", ctx->device);
    return launch_rescale(ctx, stream, L_cur, count, polys, out, flags & FIONA_RESCALE_ROUND);
}

extern "C" int fiona_linear_eval_rescale(const fiona_plan *p, void *stream, uint32_t L_eval, const uint64_t *in,
                                         const uint64_t *pt, uint64_t *work, uint64_t *out, uint32_t flags)
{
    if (flags & ~(uint32_t)FIONA_RESCALE_ROUND)
        return set_error(FIONA_ERR_ARG, "linear_eval_rescale: unknown flags 0x%x", flags);
    int rc = check_eval_args(p, in, pt, work);
    if (rc) return rc;
    const uint64_t count = 2ull * p->hp.n_out;
    rc = check_rescale_args(p->ctx, L_eval, count, work, out, "linear_eval_rescale");
    if (rc) return rc;
    const uint64_t poly_bytes = (uint64_t)p->ctx->N * 8;
    if (overlaps(out, count * (L_eval - 1) * poly_bytes, in, 2ull * p->hp.n_in * L_eval * poly_bytes))
        return set_error(FIONA_ERR_ARG, "linear_eval_rescale: output overlaps the inputs");
    if (p->hp.n_out == 0) return FIONA_OK;
    DeviceGuard g(p->ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "linear_eval_rescale: cannot select device %d", p->ctx->device);
    rc = launch_range(p, stream, in, pt, work, 0, L_eval, L_eval);
    if (rc) return rc;
    return launch_rescale(p->ctx, stream, L_eval, count, work, out, flags & FIONA_RESCALE_ROUND);
}

static int check_encode_ctx(const fiona_ctx *ctx, const char *who)
{
    if (!ctx) return set_error(FIONA_ERR_ARG, "%s: null ctx", who);
    if (ctx->device == FIONA_DEVICE_NONE) return set_error(FIONA_ERR_NODEVICE, "%s: validation-only context", who);
    return FIONA_OK;
}

static int check_embed_args(const fiona_ctx *ctx, uint64_t count, const double *slots, double scale,
                            const int64_t *coeffs, const double *work, const char *who)
{
    int rc = check_encode_ctx(ctx, who);
    if (rc) return rc;
    if (!(scale > 0.0) || !std::isfinite(scale)) return set_error(FIONA_ERR_ARG, "%s: scale must be positive", who);
    if (count > (1ull << 40) / ctx->N) return set_error(FIONA_ERR_ARG, "%s: %llu polys", who, (unsigned long long)count);
    if (count == 0) return FIONA_OK;
    if (!slots || !coeffs || !work) return set_error(FIONA_ERR_ARG, "%s: null buffer", who);
    if (((uintptr_t)slots | (uintptr_t)coeffs | (uintptr_t)work) & 15)
        return set_error(FIONA_ERR_ARG, "%s: buffers must be 16-byte aligned", who);
    const uint64_t N = ctx->N;
    if (overlaps(work, count * N * 8, slots, count * N * 8) || overlaps(work, count * N * 8, coeffs, count * N * 8) ||
        overlaps(coeffs, count * N * 8, slots, count * N * 8))
        return set_error(FIONA_ERR_ARG, "%s: overlapping buffers", who);
    return FIONA_OK;
}

static int check_encode_coeff_args(const fiona_ctx *ctx, uint32_t L_cur, uint64_t count, const int64_t *coeffs,
                                   const uint64_t *out, const char *who)
{
    int rc = check_encode_ctx(ctx, who);
    if (rc) return rc;
    if (L_cur < 1 || L_cur > ctx->L) return set_error(FIONA_ERR_ARG, "%s: level %u outside [1, %u]", who, L_cur, ctx->L);
    if (count > (1ull << 40) / ((uint64_t)L_cur * ctx->N))
        return set_error(FIONA_ERR_ARG, "%s: %llu polys", who, (unsigned long long)count);
    if (count == 0) return FIONA_OK;
    if (!coeffs || !out) return set_error(FIONA_ERR_ARG, "%s: null buffer", who);
    if (((uintptr_t)coeffs | (uintptr_t)out) & 15) return set_error(FIONA_ERR_ARG, "%s: buffers must be 16-byte aligned", who);
    const uint64_t N = ctx->N;
    if (overlaps(coeffs, count * N * 8, out, count * L_cur * N * 8))
        return set_error(FIONA_ERR_ARG, "%s: output overlaps the coefficients", who);
    return FIONA_OK;
}

extern "C" int fiona_ckks_embed(const fiona_ctx *ctx, void *stream, uint64_t count, const double *slots,
                                double scale, int64_t *coeffs, double *work)
{
    int rc = check_embed_args(ctx, count, slots, scale, coeffs, work, "ckks_embed");
    if (rc || count == 0) return rc;
    DeviceGuard g(ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "ckks_embed: cannot select device %d", ctx->device);
    return launch_embed(ctx, stream, count, slots, scale, coeffs, work);
}

extern "C" int fiona_encode_coeffs(const fiona_ctx *ctx, void *stream, uint32_t L_cur, uint64_t count,
                                   const int64_t *coeffs, uint64_t *out)
{
    int rc = check_encode_coeff_args(ctx, L_cur, count, coeffs, out, "encode_coeffs");
    if (rc || count == 0) return rc;
    DeviceGuard g(ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "encode_coeffs: cannot select device %d", ctx->device);
    return launch_encode_coeffs(ctx, stream, L_cur, count, coeffs, out);
}

extern "C" int fiona_encode(const fiona_ctx *ctx, void *stream, uint32_t L_cur, uint64_t count, const double *slots,
                            double scale, int64_t *coeffs, double *work, uint64_t *out)
{
    int rc = check_embed_args(ctx, count, slots, scale, coeffs, work, "encode");
    if (rc == FIONA_OK) rc = check_encode_coeff_args(ctx, L_cur, count, coeffs, out, "encode");
    if (rc == FIONA_OK && count) {
        const uint64_t N = ctx->N;
        if (overlaps(out, count * L_cur * N * 8, slots, count * N * 8) ||
            overlaps(out, count * L_cur * N * 8, work, count * N * 8))
            rc = set_error(FIONA_ERR_ARG, "encode: output overlaps the slots or the work area");
    }
    if (rc || count == 0) return rc;
    DeviceGuard g(ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "encode: cannot select device %d", ctx->device);
    rc = launch_embed(ctx, stream, count, slots, scale, coeffs, work);
    if (rc) return rc;
    return launch_encode_coeffs(ctx, stream, L_cur, count, coeffs, out);
}

extern "C" int fiona_check_residues(const fiona_ctx *ctx, void *stream, const uint64_t *data,
                                    uint64_t count)
{
    if (!ctx) return set_error(FIONA_ERR_ARG, "check_residues: null ctx");
    if (ctx->device == FIONA_DEVICE_NONE)
        return set_error(FIONA_ERR_NODEVICE, "check_residues: validation-only context");
    if (count == 0) return FIONA_OK;
    if (!data || ((uintptr_t)data & 15))
        return set_error(FIONA_ERR_ARG, "check_residues: null or misaligned data");
    DeviceGuard g(ctx->device);
    if (!g.ok) return set_error(FIONA_ERR_CUDA, "check_residues: cannot select device %d", ctx->device);
    return launch_check_residues(ctx, stream, data, count);
}
