// lower_tiled.cpp -- lowering of a validated plan to the tiled kernel's
// schedule (host side, once per layer).
//
// * Shared signed sums (Sec. 4.2 "Sharing Signed Sums") become sources
//   computed once per tile, in topological levels (children first).  Only
//   sums reachable from a use are kept.
// * Each output's used scale groups become segments: the group's signed terms
//   not covered by a use, plus one source per use (sign sigma), summed and
//   then multiplied once by gamma (Sec. 4.2 "Grouping Reconstruction
//   Operations").  Plus and minus operands form two runs, cut so that a run
//   never exceeds the lazy-sum bound (a cut repeats gamma, which is exact).
// * Outputs are assigned to warps by longest-processing-time first on an
//   estimated cost; with fewer outputs than warps, each output is split into
//   parts whose reduced partial sums are added at the end (exact in Z_q).
// * Shape: 2 or 1 coefficients per lane and 8 or 16 warps per CTA, and two
//   source buffers (the next tile staged during this one) when they fit;
//   chosen to keep the most bytes in flight per SM.  Plans whose moduli are
//   all below 2^52 use the radix-2^26 arithmetic.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <numeric>

#include "tiled.h"

namespace {

struct OutWork {
    struct Seg {
        uint32_t scale_pt;
        std::vector<uint32_t> plus, minus;  // source indices
    };
    std::vector<Seg> segs;
    std::vector<std::pair<uint32_t, uint32_t>> raws;  // (input, pt)
    uint64_t cost() const
    {
        uint64_t c = 4 * raws.size();
        for (auto &s : segs) c += s.plus.size() + s.minus.size() + 6;
        return c;
    }
};

struct JobSet {
    std::vector<uint32_t> warp_job_off, ops;
    std::vector<uint2> raws;
    std::vector<TiledJob> jobs;
    std::vector<TiledSeg> segs;
    std::vector<uint32_t> comb_off, comb_out, comb_parts;
    uint32_t n_part = 0;
};

// Segments of one scale group: the group's plus and minus runs as op words,
// each run at most `budget` words long.
void put_segments(JobSet &js, const OutWork::Seg &sg, uint32_t L, uint32_t budget,
                  uint32_t pair_bytes)
{
    size_t pb = 0, mb = 0;
    do {
        const size_t pe = std::min(sg.plus.size(), pb + budget);
        const size_t me = std::min(sg.minus.size(), mb + budget);
        TiledSeg s{};
        s.gamma_ptl = sg.scale_pt * L;
        s.op_begin = (uint32_t)js.ops.size();
        for (size_t i = pb; i < pe; ++i) js.ops.push_back(sg.plus[i] * pair_bytes);
        for (size_t i = mb; i < me; ++i) js.ops.push_back(sg.minus[i] * pair_bytes);
        s.n_plus = (uint16_t)(pe - pb);
        s.n_minus = (uint16_t)(me - mb);
        js.segs.push_back(s);
        pb = pe;
        mb = me;
    } while (pb < sg.plus.size() || mb < sg.minus.size());
}

JobSet build_jobs(const std::vector<OutWork> &work, uint32_t n_out, uint32_t W, uint32_t L,
                  uint32_t pair_bytes, uint32_t budget)
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
        const uint32_t P = (uint32_t)std::max<uint64_t>(1, std::min<uint64_t>(parts, c / 16));
        if (P == 1) {
            jobs.push_back({j, w});
            continue;
        }
        // cut the output's items into P contiguous chunks of about equal cost
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
            advance(6);
            int open = -1;
            auto add = [&](uint32_t src, bool minus) {
                advance(1);
                if (open != (int)cur) {
                    chunk[cur].segs.push_back({sg.scale_pt, {}, {}});
                    open = (int)cur;
                }
                (minus ? chunk[cur].segs.back().minus : chunk[cur].segs.back().plus).push_back(src);
            };
            for (uint32_t s : sg.plus) add(s, false);
            for (uint32_t s : sg.minus) add(s, true);
        }
        for (auto &r : w.raws) {
            advance(4);
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
            for (auto &sg : jb.w.segs) put_segments(js, sg, L, budget, pair_bytes);
            t.seg_end = (uint32_t)js.segs.size();
            t.raw_begin = (uint32_t)js.raws.size();
            for (auto &r : jb.w.raws) js.raws.push_back(make_uint2(r.second * L, r.first * pair_bytes));
            t.raw_end = (uint32_t)js.raws.size();
            js.jobs.push_back(t);
        }
        js.warp_job_off[wi + 1] = (uint32_t)js.jobs.size();
    }
    return js;
}

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

// kernel_tiled.cu
int tiled_configure_kernel(int C, bool narrow, size_t smem);
int tiled_kernel_attributes(int C, bool narrow, cudaFuncAttributes *attr);

int lower_tiled(fiona_plan *p)
{
    const HostPlan &hp = p->hp;
    const fiona_ctx *ctx = p->ctx;
    const bool narrow = ctx->q_max < (1ull << 52);
    // lazy-sum bound in words: 64 split words (rns.cuh), or
    // floor((2^64-1)/(q-1)) canonical residues
    const uint32_t budget = narrow ? 64u : std::min<uint32_t>(p->signed_budget, 1u << 14);

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
    std::vector<OutWork::Seg> node_seg(n_slots);
    for (uint32_t k = 0; k < hp.n_nodes; ++k) {
        if (!need[k]) continue;
        uint32_t lev = 0;
        OutWork::Seg &sg = node_seg[(uint32_t)slot[k]];
        for (uint32_t c = hp.node_offsets[k]; c < hp.node_offsets[k + 1]; ++c) {
            const fiona_sum_child &ch = hp.children[c];
            const uint32_t src = ch.is_node ? n_in + (uint32_t)slot[ch.ref] : ch.ref;
            if (ch.is_node) lev = std::max(lev, level[ch.ref] + 1);
            (ch.sign < 0 ? sg.minus : sg.plus).push_back(src);
        }
        level[k] = lev;
        n_levels = std::max(n_levels, lev + 1);
    }
    for (auto &sg : node_seg)
        if (sg.plus.size() > budget || sg.minus.size() > budget)
            return set_error(FIONA_ERR_ARG, "tiled kernel: a shared sum has more than %u children", budget);
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
            if (t.kind == FIONA_TERM_RAW)
                work[j].raws.push_back({t.input, t.pt});
            else if (t.sign != 0 && std::find(groups.begin(), groups.end(), t.group) == groups.end())
                groups.push_back(t.group);
        }
        for (uint32_t g : groups) {
            OutWork::Seg sg;
            sg.scale_pt = hp.group_scale_pt[g];
            for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
                const fiona_term &t = hp.terms[e];
                if (t.kind == FIONA_TERM_TERNARY && t.group == g && t.sign != 0 && hp.term_use[e] < 0)
                    (t.sign < 0 ? sg.minus : sg.plus).push_back(t.input);
            }
            for (uint32_t u = 0; u < hp.n_uses; ++u)
                if (hp.uses[u].output == j && hp.uses[u].group == g)
                    (hp.uses[u].sign < 0 ? sg.minus : sg.plus)
                        .push_back(n_in + (uint32_t)slot[hp.uses[u].node]);
            work[j].segs.push_back(sg);
        }
    }

    // -- shape
    const size_t budget_smem = (ctx->smem_optin ? ctx->smem_optin : 227 * 1024) - 256;
    const size_t per_sm = 228 * 1024;
    const uint32_t n_src = n_in + n_slots;
    struct Shape {
        int C;
        uint32_t W;
        bool dbl;
        uint32_t ctas;
        uint64_t score;
    };
    std::vector<Shape> shapes;
    for (int C : {2, 1}) {
        if (ctx->N % (32u * C)) continue;
        cudaFuncAttributes attr{};
        if (tiled_kernel_attributes(C, narrow, &attr) != FIONA_OK) continue;
        const uint32_t regs = (std::max(attr.numRegs, 1) + 7) & ~7;
        const uint32_t pair_bytes = 2 * 32u * C * 8;
        for (uint32_t W : {8u, 16u}) {
            const uint32_t n_part_est = hp.n_out >= W ? 0 : W;
            for (bool dbl : {true, false}) {
                if (dbl && n_in == 0) continue;
                const size_t smem = (size_t)n_src * pair_bytes * (dbl ? 2 : 1) +
                                    (size_t)n_part_est * pair_bytes + 16;
                if (smem + attr.sharedSizeBytes > budget_smem) continue;
                const uint32_t by_smem = (uint32_t)(per_sm / (smem + attr.sharedSizeBytes + 1024));
                const uint32_t by_threads = 2048 / (W * 32);
                const uint32_t by_regs = 65536 / (W * 32 * regs);
                const uint32_t ctas = std::min({by_smem, by_threads, by_regs});
                if (!ctas) continue;
                // resident warps x bytes per load (ties: the first listed,
                // double-buffered before single, 8 warps before 16)
                const uint64_t score = (uint64_t)ctas * W * C;
                shapes.push_back({C, W, dbl, ctas, score});
            }
        }
    }
    if (shapes.empty())
        return set_error(FIONA_ERR_ARG, "tiled kernel: %u source tiles do not fit in shared memory", n_src);
    Shape best = *std::max_element(shapes.begin(), shapes.end(),
                                   [](const Shape &a, const Shape &b) { return a.score < b.score; });
    // tuning override "C,W,double": every shape computes the same residues
    if (const char *env = getenv("FIONA_TILED_SHAPE")) {
        int c = 0, w = 0, d = 0;
        if (sscanf(env, "%d,%d,%d", &c, &w, &d) == 3)
            for (auto &s : shapes)
                if (s.C == c && s.W == (uint32_t)w && s.dbl == (d != 0)) best = s;
    }
    const uint32_t T = 32u * best.C, pair_bytes = 2 * T * 8;
    JobSet js = build_jobs(work, hp.n_out, best.W, ctx->L, pair_bytes, budget);
    // shared sums' runs go into the same op array, after the jobs' runs
    std::vector<TiledSeg> node_segs(n_slots);
    for (uint32_t s = 0; s < n_slots; ++s) {
        const size_t before = js.segs.size();
        put_segments(js, node_seg[s], ctx->L, budget, pair_bytes);
        node_segs[s] = js.segs[before];
        js.segs.resize(before);
    }
    // the kernel reads schedule words ahead of use: pad the ends so those
    // reads stay inside the arrays
    js.ops.insert(js.ops.end(), kSchedPad, 0u);
    js.raws.insert(js.raws.end(), kSchedPad, make_uint2(0, 0));
    const size_t smem =
        (size_t)n_src * pair_bytes * (best.dbl ? 2 : 1) + (size_t)js.n_part * pair_bytes + 16;
    if (smem > budget_smem) return set_error(FIONA_ERR_ARG, "tiled kernel: shared memory estimate exceeded");

    TiledSchedule *ts = new (std::nothrow) TiledSchedule;
    if (!ts) return set_error(FIONA_ERR_NOMEM, "tiled schedule: host allocation");
    ts->C = best.C;
    ts->narrow = narrow;
    ts->warps = best.W;
    ts->tile = T;
    ts->smem = smem;
    ts->ctas_per_sm = best.ctas;
    int rc = tiled_configure_kernel(best.C, narrow, smem);
    std::vector<size_t> off;
    if (rc == FIONA_OK)
        rc = upload_blob(ts, {{node_level_off.data(), node_level_off.size() * 4},
                              {node_slots.data(), node_slots.size() * 4},
                              {node_segs.data(), node_segs.size() * sizeof(TiledSeg)},
                              {js.warp_job_off.data(), js.warp_job_off.size() * 4},
                              {js.jobs.data(), js.jobs.size() * sizeof(TiledJob)},
                              {js.segs.data(), js.segs.size() * sizeof(TiledSeg)},
                              {js.ops.data(), js.ops.size() * 4},
                              {js.raws.data(), js.raws.size() * sizeof(uint2)},
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
    a.node_segs = (const TiledSeg *)(b + off[2]);
    a.warp_job_off = (const uint32_t *)(b + off[3]);
    a.jobs = (const TiledJob *)(b + off[4]);
    a.segs = (const TiledSeg *)(b + off[5]);
    a.ops = (const uint32_t *)(b + off[6]);
    a.raws = (const uint2 *)(b + off[7]);
    a.comb_off = (const uint32_t *)(b + off[8]);
    a.comb_out = (const uint32_t *)(b + off[9]);
    a.comb_parts = (const uint32_t *)(b + off[10]);
    a.limbs = ctx->d_limbs;
    a.err = ctx->d_kerr;
    a.N = ctx->N;
    a.L = ctx->L;
    a.log2N = 0;
    while ((1u << a.log2N) < ctx->N) ++a.log2N;
    a.tiles_per_limb = ctx->N / T;
    a.n_in = n_in;
    a.n_nodes = n_slots;
    a.n_levels = n_levels;
    a.n_part = js.n_part;
    a.n_comb = (uint32_t)js.comb_out.size();
    a.src_bytes = n_src * pair_bytes;
    a.double_buffer = best.dbl ? 1 : 0;
    a.mac_budget = narrow ? 64u : p->mac_budget;  // rns.cuh: kNarrowMacBudget
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
