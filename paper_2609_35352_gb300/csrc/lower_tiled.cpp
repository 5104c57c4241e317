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
// * Each warp gets a program (its jobs' words) and a fetch list (the
//   plaintext tiles it consumes, in order); the whole schedule is one word
//   array the kernel copies into shared memory.
// * Shape: 2 or 1 coefficients per lane, 8 or 16 warps per CTA, 16 or 8
//   plaintext tiles in flight per warp, and two source buffers (the next
//   tile staged during this one) when they fit; chosen to keep enough bytes
//   in flight per SM.  Plans whose moduli are all below 2^52 use the
//   radix-2^26 arithmetic.
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

// Jobs for W warps: whole outputs assigned largest first to the least-loaded
// warp; with fewer outputs than warps each output is cut into parts of about
// equal cost whose reduced partial sums are added at the end.
struct JobPlan {
    struct Job {
        uint32_t target;
        OutWork w;
    };
    std::vector<std::vector<Job>> per_warp;
    std::vector<uint32_t> comb_off, comb_out, comb_parts;
    uint32_t n_part = 0;
};

JobPlan build_jobs(const std::vector<OutWork> &work, uint32_t n_out, uint32_t W)
{
    JobPlan jp;
    std::vector<JobPlan::Job> jobs;
    jp.comb_off.assign(1, 0);
    const uint32_t parts = n_out >= W ? 1 : W / std::max<uint32_t>(n_out, 1);
    for (uint32_t j = 0; j < n_out; ++j) {
        const OutWork &w = work[j];
        const uint64_t c = w.cost();
        const uint32_t P = (uint32_t)std::max<uint64_t>(1, std::min<uint64_t>(parts, c / 16));
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
        jp.comb_out.push_back(j);
        for (uint32_t q = 0; q < P; ++q) {
            if (chunk[q].segs.empty() && chunk[q].raws.empty()) continue;
            jobs.push_back({kPartBit | jp.n_part, chunk[q]});
            jp.comb_parts.push_back(jp.n_part++);
        }
        jp.comb_off.push_back((uint32_t)jp.comb_parts.size());
    }
    std::vector<uint32_t> order(jobs.size());
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(),
                     [&](uint32_t a, uint32_t b) { return jobs[a].w.cost() > jobs[b].w.cost(); });
    std::vector<uint64_t> load(W, 0);
    jp.per_warp.assign(W, {});
    for (uint32_t o : order) {
        const uint32_t wi = (uint32_t)(std::min_element(load.begin(), load.end()) - load.begin());
        jp.per_warp[wi].push_back(jobs[o]);
        load[wi] += jobs[o].w.cost() + 1;
    }
    return jp;
}

// Append one scale group's segments (runs of at most `budget` words) to a
// warp program and its gamma fetches to the fetch list.
void put_group(std::vector<uint32_t> &prog, std::vector<uint32_t> &fetch, const OutWork::Seg &sg,
               uint32_t L, uint32_t budget, uint32_t pair_bytes, uint32_t &n_seg)
{
    size_t pb = 0, mb = 0;
    do {
        const size_t pe = std::min(sg.plus.size(), pb + budget);
        const size_t me = std::min(sg.minus.size(), mb + budget);
        prog.push_back((uint32_t)(pe - pb) | ((uint32_t)(me - mb) << 16));
        for (size_t i = pb; i < pe; ++i) prog.push_back(sg.plus[i] * pair_bytes);
        for (size_t i = mb; i < me; ++i) prog.push_back(sg.minus[i] * pair_bytes);
        fetch.push_back(sg.scale_pt * L);
        ++n_seg;
        pb = pe;
        mb = me;
    } while (pb < sg.plus.size() || mb < sg.minus.size());
}

// The whole schedule as one word array (see tiled.h).
struct Sched {
    std::vector<uint32_t> w;
    uint32_t o_level, o_node_slot, o_node_prog_off, o_prog_off, o_fetch_off, o_comb_off, o_comb_out,
        o_comb_parts;
};

Sched encode(const JobPlan &jp, const std::vector<uint32_t> &node_level_off,
             const std::vector<uint32_t> &node_slots, const std::vector<OutWork::Seg> &node_seg,
             uint32_t W, uint32_t L, uint32_t budget, uint32_t pair_bytes)
{
    Sched sc;
    auto &w = sc.w;
    auto put = [&](const std::vector<uint32_t> &v) { w.insert(w.end(), v.begin(), v.end()); };
    sc.o_level = (uint32_t)w.size();
    put(node_level_off);
    sc.o_node_slot = (uint32_t)w.size();
    put(node_slots);
    // node programs: offsets table then programs
    sc.o_node_prog_off = (uint32_t)w.size();
    const size_t n_nodes = node_seg.size();
    w.resize(w.size() + n_nodes + 1);
    for (size_t k = 0; k < n_nodes; ++k) {
        w[sc.o_node_prog_off + k] = (uint32_t)w.size();
        const OutWork::Seg &sg = node_seg[k];
        w.push_back((uint32_t)sg.plus.size() | ((uint32_t)sg.minus.size() << 16));
        for (uint32_t s : sg.plus) w.push_back(s * pair_bytes);
        for (uint32_t s : sg.minus) w.push_back(s * pair_bytes);
    }
    w[sc.o_node_prog_off + n_nodes] = (uint32_t)w.size();
    // warp programs and fetch lists
    std::vector<std::vector<uint32_t>> progs(W), fetches(W);
    for (uint32_t wi = 0; wi < W; ++wi) {
        for (const auto &jb : jp.per_warp[wi]) {
            auto &prog = progs[wi];
            prog.push_back(jb.target);
            const size_t hdr = prog.size();
            prog.push_back(0);
            uint32_t n_seg = 0;
            for (const auto &sg : jb.w.segs) put_group(prog, fetches[wi], sg, L, budget, pair_bytes, n_seg);
            for (const auto &r : jb.w.raws) {
                prog.push_back(r.first * pair_bytes);
                fetches[wi].push_back(r.second * L);
            }
            prog[hdr] = n_seg | ((uint32_t)jb.w.raws.size() << 16);
        }
    }
    sc.o_prog_off = (uint32_t)w.size();
    w.resize(w.size() + W + 1);
    for (uint32_t wi = 0; wi < W; ++wi) {
        w[sc.o_prog_off + wi] = (uint32_t)w.size();
        put(progs[wi]);
    }
    w[sc.o_prog_off + W] = (uint32_t)w.size();
    sc.o_fetch_off = (uint32_t)w.size();
    w.resize(w.size() + W + 1);
    for (uint32_t wi = 0; wi < W; ++wi) {
        w[sc.o_fetch_off + wi] = (uint32_t)w.size();
        put(fetches[wi]);
    }
    w[sc.o_fetch_off + W] = (uint32_t)w.size();
    sc.o_comb_off = (uint32_t)w.size();
    put(jp.comb_off);
    sc.o_comb_out = (uint32_t)w.size();
    put(jp.comb_out);
    sc.o_comb_parts = (uint32_t)w.size();
    put(jp.comb_parts);
    while (w.size() % 4) w.push_back(0);  // a multiple of 16 bytes
    return sc;
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
int tiled_configure_kernel(int C, bool narrow, uint32_t depth, size_t smem);
int tiled_kernel_attributes(int C, bool narrow, uint32_t depth, cudaFuncAttributes *attr);

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

    // -- shape: coefficients per lane C, warps W, ring depth D, source buffers
    const size_t budget_smem = (ctx->smem_optin ? ctx->smem_optin : 227 * 1024) - 256;
    const size_t per_sm = 228 * 1024;
    const uint32_t n_src = n_in + n_slots;
    struct Shape {
        int C;
        uint32_t W, D;
        bool dbl;
        uint32_t ctas;
        size_t smem;
        uint64_t score;
    };
    std::vector<Shape> shapes;
    for (int C : {2, 1}) {
        if (ctx->N % (32u * C)) continue;
        const uint32_t T = 32u * C, pair_bytes = 2 * T * 8;
        for (uint32_t W : {8u, 16u}) {
            const JobPlan jp = build_jobs(work, hp.n_out, W);
            const Sched sc = encode(jp, node_level_off, node_slots, node_seg, W, ctx->L, budget, pair_bytes);
            const size_t sched_bytes = sc.w.size() * 4;
            for (uint32_t D : {16u, 8u}) {
                cudaFuncAttributes attr{};
                if (tiled_kernel_attributes(C, narrow, D, &attr) != FIONA_OK) continue;
                const uint32_t regs = (std::max(attr.numRegs, 1) + 7) & ~7;
                for (bool dbl : {true, false}) {
                    if (dbl && n_in == 0) continue;
                    const size_t smem = sched_bytes + (size_t)n_src * pair_bytes * (dbl ? 2 : 1) +
                                        (size_t)jp.n_part * pair_bytes + (size_t)W * D * T * 8 + 32;
                    if (smem + attr.sharedSizeBytes > budget_smem) continue;
                    const uint32_t by_smem = (uint32_t)(per_sm / (smem + attr.sharedSizeBytes + 1024));
                    const uint32_t by_threads = 2048 / (W * 32);
                    const uint32_t by_regs = 65536 / (W * 32 * regs);
                    const uint32_t ctas = std::min({by_smem, by_threads, by_regs});
                    if (!ctas) continue;
                    // plaintext bytes in flight per SM (enough at about 96 KB),
                    // then resident warps, then wider loads
                    const uint64_t inflight = std::min<uint64_t>((uint64_t)ctas * W * D * T * 8, 96 * 1024);
                    const uint64_t score = (inflight << 16) | ((uint64_t)ctas * W << 4) | (uint64_t)(C * 2 + dbl);
                    shapes.push_back({C, W, D, dbl, ctas, smem, score});
                }
            }
        }
    }
    if (shapes.empty())
        return set_error(FIONA_ERR_ARG, "tiled kernel: %u source tiles do not fit in shared memory", n_src);
    Shape best = *std::max_element(shapes.begin(), shapes.end(),
                                   [](const Shape &a, const Shape &b) { return a.score < b.score; });
    // tuning override "C,W,D,double": every shape computes the same residues
    if (const char *env = getenv("FIONA_TILED_SHAPE")) {
        int c = 0, w = 0, dd = 0, d = 0;
        if (sscanf(env, "%d,%d,%d,%d", &c, &w, &dd, &d) == 4)
            for (auto &s : shapes)
                if (s.C == c && s.W == (uint32_t)w && s.D == (uint32_t)dd && s.dbl == (d != 0)) best = s;
    }
    const uint32_t T = 32u * best.C, pair_bytes = 2 * T * 8;
    const JobPlan jp = build_jobs(work, hp.n_out, best.W);
    const Sched sc = encode(jp, node_level_off, node_slots, node_seg, best.W, ctx->L, budget, pair_bytes);

    TiledSchedule *ts = new (std::nothrow) TiledSchedule;
    if (!ts) return set_error(FIONA_ERR_NOMEM, "tiled schedule: host allocation");
    ts->C = best.C;
    ts->narrow = narrow;
    ts->warps = best.W;
    ts->depth = best.D;
    ts->tile = T;
    ts->smem = best.smem;
    ts->ctas_per_sm = best.ctas;
    int rc = tiled_configure_kernel(best.C, narrow, best.D, ts->smem);
    std::vector<size_t> off;
    if (rc == FIONA_OK) rc = upload_blob(ts, {{sc.w.data(), sc.w.size() * 4}}, off);
    if (rc != FIONA_OK) {
        cudaFree(ts->sched.blob);
        delete ts;
        return rc;
    }
    TiledArgs &a = ts->args;
    a.sched = (const uint32_t *)ts->sched.blob;
    a.o_level = sc.o_level;
    a.o_node_slot = sc.o_node_slot;
    a.o_node_prog_off = sc.o_node_prog_off;
    a.o_prog_off = sc.o_prog_off;
    a.o_fetch_off = sc.o_fetch_off;
    a.o_comb_off = sc.o_comb_off;
    a.o_comb_out = sc.o_comb_out;
    a.o_comb_parts = sc.o_comb_parts;
    a.sched_bytes = (uint32_t)(sc.w.size() * 4);
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
    a.n_part = jp.n_part;
    a.n_comb = (uint32_t)jp.comb_out.size();
    a.src_bytes = n_src * pair_bytes;
    a.double_buffer = best.dbl ? 1 : 0;
    a.mac_budget = narrow ? 1023u : p->mac_budget;  // rns.cuh: kNarrowMacBudget
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
