// lower_tiled.cpp -- lowering of a validated plan to the tiled kernel's
// schedule (host side, once per layer).
//
// * Shared signed sums (Sec. 4.2 "Sharing Signed Sums") become smem sources
//   computed once per tile, in topological levels (children first).  Only
//   sums reachable from a use are kept.
// * Each output's used scale groups become segments: the group's signed terms
//   not covered by a use, plus one source per use (sign sigma), followed by
//   one product by gamma (Sec. 4.2 "Grouping Reconstruction Operations").
// * Outputs are assigned to warps by longest-processing-time first on an
//   estimated cost; with fewer outputs than warps, each output is split into
//   parts whose reduced partial sums are added at the end (an exact identity
//   in Z_q: gamma*(S1+S2) = gamma*S1 + gamma*S2).
// * The tile shape (2 or 1 coefficients per lane, 8 or 16 warps per CTA) is
//   the one that keeps the most 16- or 8-byte loads in flight per SM, given
//   the shared memory the sources need and the kernel's register count.
// * Plans whose moduli are all below 2^52 use the radix-2^26 arithmetic.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>
#include <map>
#include <numeric>

#include "tiled.h"

namespace {

struct OutWork {
    struct Seg {
        uint32_t scale_pt;
        std::vector<uint32_t> ops;
    };
    std::vector<Seg> segs;
    std::vector<std::pair<uint32_t, uint32_t>> raws;  // (input, pt)
    uint64_t cost() const
    {
        uint64_t c = 3 * raws.size();
        for (auto &s : segs) c += s.ops.size() + 3;
        return c;
    }
};

int upload_blob(TiledSchedule *ts, const std::vector<std::pair<const void *, size_t>> &parts,
                std::vector<size_t> &off)
{
    size_t total = 0;
    off.clear();
    for (auto &pr : parts) {
        off.push_back(total);
        total += (pr.second + 255) & ~(size_t)255;
    }
    if (!total) total = 256;
    std::vector<uint8_t> host(total, 0);
    for (size_t i = 0; i < parts.size(); ++i)
        if (parts[i].second) memcpy(host.data() + off[i], parts[i].first, parts[i].second);
    cudaError_t e = cudaMalloc(&ts->sched.blob, total);
    if (e != cudaSuccess) return set_error(FIONA_ERR_NOMEM, "tiled schedule: %s", cudaGetErrorString(e));
    ts->sched.bytes = total;
    e = cudaMemcpy(ts->sched.blob, host.data(), total, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled schedule: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

}  // namespace

struct JobSet {
    std::vector<uint32_t> warp_job_off, ops;
    std::vector<uint32_t> raws;  // (pt, input) pairs; each job's list starts on a 16-byte boundary
    std::vector<TiledJob> jobs;
    std::vector<TiledSeg> segs;
    std::vector<uint32_t> comb_off, comb_out, comb_parts;
    uint32_t n_part = 0;
};

// Jobs for W warps: whole outputs assigned largest first to the least-loaded
// warp; with fewer outputs than warps each output is cut into parts of about
// equal cost whose reduced partial sums are added at the end.
static JobSet build_jobs(const std::vector<OutWork> &work, uint32_t n_out, uint32_t W)
{
    struct Job {
        uint32_t target;
        OutWork w;
    };
    JobSet js;
    std::vector<Job> jobs;
    js.comb_off.assign(1, 0);
    const uint32_t parts = n_out >= W ? 1 : W / std::max<uint32_t>(n_out, 1);
    for (uint32_t j = 0; j < n_out; ++j) {
        const OutWork &w = work[j];
        const uint64_t c = w.cost();
        const uint32_t P = (uint32_t)std::max<uint64_t>(1, std::min<uint64_t>(parts, c / 4));
        if (P == 1) {
            jobs.push_back({j, w});
            continue;
        }
        std::vector<OutWork> chunk(P);
        const uint64_t per = (c + P - 1) / P;
        uint32_t cur = 0;
        uint64_t acc = 0;
        auto advance = [&](uint64_t add) {
            if (acc + add > per && acc > 0 && cur + 1 < P) {
                ++cur;
                acc = 0;
            }
            acc += add;
        };
        for (auto &sg : w.segs) {
            int open = -1;
            advance(3);
            for (uint32_t op : sg.ops) {
                advance(1);
                if (open != (int)cur) {
                    chunk[cur].segs.push_back({sg.scale_pt, {}});
                    open = (int)cur;
                }
                chunk[cur].segs.back().ops.push_back(op);
            }
        }
        for (auto &r : w.raws) {
            advance(3);
            chunk[cur].raws.push_back(r);
        }
        js.comb_out.push_back(j);
        for (uint32_t q = 0; q < P; ++q) {
            if (chunk[q].segs.empty() && chunk[q].raws.empty()) continue;
            jobs.push_back({kPartBit | js.n_part, chunk[q]});
            js.comb_parts.push_back(js.n_part++);
        }
        js.comb_off.push_back((uint32_t)js.comb_parts.size());
    }
    std::vector<uint32_t> order(jobs.size());
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(),
                     [&](uint32_t a, uint32_t b) { return jobs[a].w.cost() > jobs[b].w.cost(); });
    std::vector<uint64_t> load(W, 0);
    std::vector<std::vector<uint32_t>> per_warp(W);
    for (uint32_t o : order) {
        const uint32_t wi = (uint32_t)(std::min_element(load.begin(), load.end()) - load.begin());
        per_warp[wi].push_back(o);
        load[wi] += jobs[o].w.cost() + 1;
    }
    js.warp_job_off.assign(W + 1, 0);
    for (uint32_t wi = 0; wi < W; ++wi) {
        for (uint32_t o : per_warp[wi]) {
            const Job &jb = jobs[o];
            TiledJob t{};
            t.target = jb.target;
            t.seg_begin = (uint32_t)js.segs.size();
            for (auto &sg : jb.w.segs) {
                TiledSeg s{};
                s.scale_pt = sg.scale_pt;
                while (js.ops.size() % 4) js.ops.push_back(0);  // 16-byte aligned start
                s.op_begin = (uint32_t)js.ops.size();
                js.ops.insert(js.ops.end(), sg.ops.begin(), sg.ops.end());
                s.op_end = (uint32_t)js.ops.size();
                js.segs.push_back(s);
            }
            t.seg_end = (uint32_t)js.segs.size();
            if ((js.raws.size() / 2) % 2) js.raws.insert(js.raws.end(), {0u, 0u});
            t.raw_begin = (uint32_t)(js.raws.size() / 2);
            for (auto &r : jb.w.raws) {
                js.raws.push_back(r.second);  // plaintext
                js.raws.push_back(r.first);   // input
            }
            t.raw_end = (uint32_t)(js.raws.size() / 2);
            js.jobs.push_back(t);
        }
        js.warp_job_off[wi + 1] = (uint32_t)js.jobs.size();
    }
    // the kernel prefetches schedule words one chunk ahead of use: pad the
    // ends so those loads stay inside the arrays
    js.ops.insert(js.ops.end(), kSchedPad, 0u);
    js.raws.insert(js.raws.end(), 2 * kSchedPad, 0u);
    return js;
}

size_t tiled_smem_bytes(uint32_t n_src, uint32_t n_part, uint32_t tile)
{
    return ((size_t)n_src + n_part) * 2 * tile * 8 + 16;
}

// kernel_tiled.cu
int tiled_configure_kernel(int C, bool narrow, size_t smem);
int tiled_kernel_attributes(int C, bool narrow, cudaFuncAttributes *attr);

int lower_tiled(fiona_plan *p)
{
    const HostPlan &hp = p->hp;
    const fiona_ctx *ctx = p->ctx;

    // -- shared sums reachable from a use, numbered in index order (children first)
    std::vector<uint8_t> need(hp.n_nodes, 0);
    for (uint32_t u = 0; u < hp.n_uses; ++u) need[hp.uses[u].node] = 1;
    for (int k = (int)hp.n_nodes - 1; k >= 0; --k) {
        if (!need[k]) continue;
        for (uint32_t c = hp.node_offsets[k]; c < hp.node_offsets[k + 1]; ++c)
            if (hp.children[c].is_node) need[hp.children[c].ref] = 1;
    }
    std::vector<int32_t> slot(hp.n_nodes, -1);
    uint32_t n_slots = 0;
    for (uint32_t k = 0; k < hp.n_nodes; ++k)
        if (need[k]) slot[k] = (int32_t)n_slots++;
    const uint32_t n_in = hp.n_in;
    std::vector<uint32_t> level(hp.n_nodes, 0);
    uint32_t n_levels = 0;
    std::vector<uint32_t> node_op_begin, node_op_end, node_ops;
    for (uint32_t k = 0; k < hp.n_nodes; ++k) {
        if (!need[k]) continue;
        uint32_t lev = 0;
        while (node_ops.size() % 4) node_ops.push_back(0);  // 16-byte aligned start
        node_op_begin.push_back((uint32_t)node_ops.size());
        for (uint32_t c = hp.node_offsets[k]; c < hp.node_offsets[k + 1]; ++c) {
            const fiona_sum_child &ch = hp.children[c];
            const uint32_t src = ch.is_node ? n_in + (uint32_t)slot[ch.ref] : ch.ref;
            if (ch.is_node) lev = std::max(lev, level[ch.ref] + 1);
            node_ops.push_back(src | (ch.sign < 0 ? kNegBit : 0u));
        }
        level[k] = lev;
        n_levels = std::max(n_levels, lev + 1);
        node_op_end.push_back((uint32_t)node_ops.size());
    }
    node_ops.insert(node_ops.end(), kSchedPad, 0u);
    // node_op_off: begin/end pairs per node slot
    std::vector<uint32_t> node_op_off;
    for (size_t i = 0; i < node_op_begin.size(); ++i) {
        node_op_off.push_back(node_op_begin[i]);
        node_op_off.push_back(node_op_end[i]);
    }
    std::vector<uint32_t> node_level_off(n_levels + 1, 0), node_slots;
    for (uint32_t lev = 0; lev < n_levels; ++lev) {
        for (uint32_t k = 0; k < hp.n_nodes; ++k)
            if (need[k] && level[k] == lev) node_slots.push_back((uint32_t)slot[k]);
        node_level_off[lev + 1] = (uint32_t)node_slots.size();
    }

    // -- per-output work
    std::vector<OutWork> work(hp.n_out);
    for (uint32_t j = 0; j < hp.n_out; ++j) {
        std::vector<uint32_t> groups;
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &t = hp.terms[e];
            if (t.kind == FIONA_TERM_RAW) {
                work[j].raws.push_back({t.input, t.pt});
            } else if (t.sign != 0 &&
                       std::find(groups.begin(), groups.end(), t.group) == groups.end()) {
                groups.push_back(t.group);
            }
        }
        for (uint32_t g : groups) {
            OutWork::Seg sg;
            sg.scale_pt = hp.group_scale_pt[g];
            for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
                const fiona_term &t = hp.terms[e];
                if (t.kind == FIONA_TERM_TERNARY && t.group == g && t.sign != 0 && hp.term_use[e] < 0)
                    sg.ops.push_back(t.input | (t.sign < 0 ? kNegBit : 0u));
            }
            for (uint32_t u = 0; u < hp.n_uses; ++u)
                if (hp.uses[u].output == j && hp.uses[u].group == g)
                    sg.ops.push_back((n_in + (uint32_t)slot[hp.uses[u].node]) |
                                     (hp.uses[u].sign < 0 ? kNegBit : 0u));
            work[j].segs.push_back(sg);
        }
    }

    // -- candidate shapes: coefficients per lane C and warps per CTA W
    const bool narrow = ctx->q_max < (1ull << 52);
    const uint32_t n_src = n_in + n_slots;
    const size_t budget = (ctx->smem_optin ? ctx->smem_optin : 227 * 1024) - 256;
    const size_t per_sm = 228 * 1024;
    JobSet best_js;
    int best_C = 0;
    uint32_t best_W = 0, best_ctas = 0;
    size_t best_smem = 0;
    uint64_t best_score = 0;
    for (int C : {2, 1}) {
        if (ctx->N % (32u * C)) continue;
        cudaFuncAttributes attr{};
        if (tiled_kernel_attributes(C, narrow, &attr) != FIONA_OK) continue;
        const uint32_t regs = std::max(attr.numRegs, 1);
        for (uint32_t W : {8u, 16u}) {
            JobSet js = build_jobs(work, hp.n_out, W);
            const size_t smem = tiled_smem_bytes(n_src, js.n_part, 32u * C);
            if (smem + attr.sharedSizeBytes > budget) continue;
            const uint32_t by_smem = (uint32_t)(per_sm / (smem + attr.sharedSizeBytes + 1024));
            const uint32_t by_threads = 2048 / (W * 32);
            const uint32_t by_regs = 65536 / (W * 32 * ((regs + 7) & ~7u));
            const uint32_t ctas = std::min({by_smem, by_threads, by_regs});
            if (ctas == 0) continue;
            // bytes a CTA set can have in flight scale with resident warps x C
            const uint64_t score = (uint64_t)ctas * W * C;
            if (score > best_score) {
                best_score = score;
                best_js = std::move(js);
                best_C = C;
                best_W = W;
                best_ctas = ctas;
                best_smem = smem;
            }
        }
    }
    if (!best_score)
        return set_error(FIONA_ERR_ARG, "tiled kernel: %u sources need more shared memory than %zu B",
                         n_src, budget);

    TiledSchedule *ts = new (std::nothrow) TiledSchedule;
    if (!ts) return set_error(FIONA_ERR_NOMEM, "tiled schedule: host allocation");
    ts->C = best_C;
    ts->narrow = narrow;
    ts->warps = best_W;
    ts->tile = 32u * best_C;
    ts->smem = best_smem;
    ts->ctas_per_sm = best_ctas;
    const JobSet &js = best_js;
    int rc = tiled_configure_kernel(best_C, narrow, ts->smem);
    std::vector<size_t> off;
    if (rc == FIONA_OK)
        rc = upload_blob(ts, {{node_level_off.data(), node_level_off.size() * 4},
                              {node_slots.data(), node_slots.size() * 4},
                              {node_op_off.data(), node_op_off.size() * 4},
                              {node_ops.data(), node_ops.size() * 4},
                              {js.warp_job_off.data(), js.warp_job_off.size() * 4},
                              {js.jobs.data(), js.jobs.size() * sizeof(TiledJob)},
                              {js.segs.data(), js.segs.size() * sizeof(TiledSeg)},
                              {js.ops.data(), js.ops.size() * 4},
                              {js.raws.data(), js.raws.size() * 4},
                              {js.comb_off.data(), js.comb_off.size() * 4},
                              {js.comb_out.data(), js.comb_out.size() * 4},
                              {js.comb_parts.data(), js.comb_parts.size() * 4}},
                         off);
    if (rc != FIONA_OK) {
        cudaFree(ts->sched.blob);
        delete ts;
        return rc;
    }
    uint8_t *b = (uint8_t *)ts->sched.blob;
    TiledArgs &a = ts->args;
    a.node_level_off = (const uint32_t *)(b + off[0]);
    a.node_slots = (const uint32_t *)(b + off[1]);
    a.node_op_off = (const uint32_t *)(b + off[2]);
    a.node_ops = (const uint32_t *)(b + off[3]);
    a.warp_job_off = (const uint32_t *)(b + off[4]);
    a.jobs = (const TiledJob *)(b + off[5]);
    a.segs = (const TiledSeg *)(b + off[6]);
    a.ops = (const uint32_t *)(b + off[7]);
    a.raws = (const uint2 *)(b + off[8]);
    a.comb_off = (const uint32_t *)(b + off[9]);
    a.comb_out = (const uint32_t *)(b + off[10]);
    a.comb_parts = (const uint32_t *)(b + off[11]);
    a.limbs = ctx->d_limbs;
    a.err = ctx->d_kerr;
    a.N = ctx->N;
    a.L = ctx->L;
    a.n_in = n_in;
    a.n_nodes = n_slots;
    a.n_levels = n_levels;
    a.n_part = js.n_part;
    a.n_comb = (uint32_t)js.comb_out.size();
    a.mac_budget = p->mac_budget;
    a.signed_budget = p->signed_budget;
    p->tiled = ts;
    return FIONA_OK;
}

void free_tiled(fiona_plan *p)
{
    if (!p->tiled) return;
    cudaFree(p->tiled->sched.blob);
    delete p->tiled;
    p->tiled = nullptr;
}
