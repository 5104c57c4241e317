// lower_tiled.cpp -- lowering of a validated plan to the tiled kernel's
// schedule (host side, once per layer).
//
// * Shared signed sums (Sec. 4.2 "Sharing Signed Sums") reachable from a use
//   are materialised once per tile as extra sources, in topological levels
//   (children first), when they save enough additions to pay for that phase
//   and as many as shared memory holds: the sums are ranked by the additions
//   they save, and a sum left out is expanded into its children wherever it
//   is used (the same residues, a few more additions).
// * Each output's used scale groups become SEG operations: the group's
//   signed terms not covered by a use, plus one operand per use (sign
//   sigma), summed and then multiplied once by gamma (Sec. 4.2 "Grouping
//   Reconstruction Operations").  Plus and minus runs longer than the
//   lazy-sum bound are cut into several operations with the same gamma
//   (gamma*S1 + gamma*S2 = gamma*(S1+S2) mod q).  Each raw term is a RAW
//   operation.
// * Outputs are assigned to warps by longest-processing-time first on an
//   estimated cost; an output larger than a warp's fair share is split into
//   parts whose reduced partial sums are added at the end (exact in Z_q).
// * Shape: 2 or 1 coefficients per lane, 4 to 16 warps per CTA, one or two
//   source regions, ranked as described at the choice below.  Plans whose
//   moduli are all below 2^52 use the radix-2^26 arithmetic.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <map>
#include <numeric>
#include <tuple>

#include "tiled.h"

namespace {

constexpr uint32_t kNodeTag = 0x80000000u;  // operand naming a shared sum

// A signed-sum program formed by a warp into one of its slots.
struct Form {
    uint32_t slot;
    std::vector<uint32_t> plus, minus;             // source indices
    std::vector<uint32_t> plus_slots, minus_slots; // warp slots
};

// One SEG operation (after cuts) or the unresolved operand list of a group.
struct Seg {
    uint32_t scale_pt;
    std::vector<uint32_t> plus, minus;              // source indices
    std::vector<uint32_t> plus_slots, minus_slots;  // warp slots (shared sums this warp formed)
    std::vector<Form> forms;                        // sums formed into slots before this one
};

// operands a SEG reads, its formations included
size_t seg_operands(const Seg &s)
{
    size_t n = s.plus.size() + s.minus.size() + s.plus_slots.size() + s.minus_slots.size();
    for (const Form &f : s.forms) n += f.plus.size() + f.minus.size() + f.plus_slots.size() + f.minus_slots.size();
    return n;
}

struct OutWork {
    std::vector<Seg> segs;
    std::vector<std::pair<uint32_t, uint32_t>> raws;  // (source | kOpConst if constant, pt)
};

// Estimated issue cost of operations, in warp instructions, and of the
// resources they draw on (see the shape search).
struct Costs {
    double raw, seg, operand, last, nop;
    double imad_op;          // wide multiplies (quarter rate) per product operation
    double smem_operand;     // shared-memory bytes per source read (both polys)
};

Costs costs_for(int C, bool narrow)
{
    Costs c{};
    if (narrow) {
        c = C == 2 ? Costs{34, 70, 8.5, 90, 6, 12, 1024} : Costs{22, 40, 6, 50, 5, 6, 512};
    } else {
        c = C == 2 ? Costs{60, 80, 8.5, 110, 6, 32, 1024} : Costs{35, 45, 6, 60, 5, 16, 512};
    }
    return c;
}

double work_cost(const OutWork &w, const Costs &k, size_t P)
{  // P: operations per batch
    double c = k.last + k.raw * (double)w.raws.size();
    for (auto &s : w.segs) c += k.seg * (1.0 + 0.5 * (double)s.forms.size()) + k.operand * (double)seg_operands(s);
    // NOP padding: each SEG opens a batch, the job fills its last one
    const size_t ops = w.segs.size() + w.raws.size();
    size_t slots = 0;
    if (w.segs.empty()) {
        slots = (w.raws.size() + P - 1) / P * P;
    } else {
        slots = (w.segs.size() - 1) * P + (1 + w.raws.size() + P - 1) / P * P;
    }
    c += k.nop * (double)(std::max(slots, std::max<size_t>(ops, 1)) - ops);
    return c;
}

struct Job {
    uint32_t target;
    OutWork w;
};

struct JobPlan {
    std::vector<std::vector<Job>> per_warp;
    std::vector<uint32_t> comb_off, comb_out, comb_parts;
    uint32_t n_part = 0;
};

// Cut `w` into P parts of about equal cost (segments are cut between
// operands; each piece keeps its gamma).
std::vector<OutWork> split_work(const OutWork &w, uint32_t P, const Costs &k, size_t batch)
{
    std::vector<OutWork> chunk(P);
    const double per = work_cost(w, k, batch) / P;
    uint32_t cur = 0;
    double acc = 0;
    auto advance = [&](double add) {
        if (acc + add > per && acc > 0 && cur + 1 < P) {
            ++cur;
            acc = 0;
        }
        acc += add;
    };
    for (auto &sg : w.segs) {
        advance(k.seg);
        int open = -1;
        auto add = [&](uint32_t src, bool minus) {
            advance(k.operand);
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
        advance(k.raw);
        chunk[cur].raws.push_back(r);
    }
    return chunk;
}

// Outputs that share signed sums (Sec. 4.2 "Sharing Signed Sums"): per
// shared sum of the plan, the distinct outputs whose groups use it, and what
// keeping it saves.  Used to place such outputs on one warp, which can then
// form the sum once per tile for all of them.
struct Sharing {
    std::vector<std::vector<uint32_t>> users;  // per plan node
    std::vector<double> benefit;               // per plan node
};

// Clusters of outputs for W warps: the users of each shared sum (best saving
// first) are merged while the merged cost stays within one warp's share.
// Returns a cluster id per output (-1: on its own).
std::vector<int> clusters_for(const std::vector<OutWork> &work, uint32_t W, const Costs &k, size_t batch,
                              const Sharing *sh)
{
    std::vector<int> cl(work.size(), -1);
    if (!sh || work.empty()) return cl;
    std::vector<double> cost(work.size());
    double total = 0;
    for (size_t j = 0; j < work.size(); ++j) total += cost[j] = work_cost(work[j], k, batch);
    double cmax = 0;
    for (double c : cost) cmax = std::max(cmax, c);
    const double cap = std::max(total / W, 2 * cmax);  // a pair of outputs always fits
    std::vector<uint32_t> parent(work.size());
    std::iota(parent.begin(), parent.end(), 0);
    std::vector<double> ccost = cost;
    std::function<uint32_t(uint32_t)> find = [&](uint32_t x) { return parent[x] == x ? x : parent[x] = find(parent[x]); };
    std::vector<uint32_t> order(sh->users.size());
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(), [&](uint32_t x, uint32_t y) { return sh->benefit[x] > sh->benefit[y]; });
    for (uint32_t nd : order) {
        const auto &us = sh->users[nd];
        if (us.size() < 2 || sh->benefit[nd] <= 0) continue;
        std::vector<uint32_t> roots;
        for (uint32_t u : us) {
            const uint32_t r = find(u);
            if (std::find(roots.begin(), roots.end(), r) == roots.end()) roots.push_back(r);
        }
        if (roots.size() < 2) continue;
        double c = 0;
        for (uint32_t r : roots) c += ccost[r];
        if (c > cap) continue;
        for (size_t i = 1; i < roots.size(); ++i) parent[roots[i]] = roots[0];
        ccost[roots[0]] = c;
    }
    std::vector<uint32_t> size(work.size(), 0);
    for (size_t j = 0; j < work.size(); ++j) ++size[find((uint32_t)j)];
    for (size_t j = 0; j < work.size(); ++j)
        if (size[find((uint32_t)j)] > 1) cl[j] = (int)find((uint32_t)j);
    return cl;
}

// Jobs for W warps: every output worth splitting is cut into `split` parts
// (more if it costs more than a fair share, total / W), except outputs
// clustered with others (`cl`), which stay whole and together; then the
// units (a cluster's jobs, or one job) are assigned largest first to the
// least-loaded warp.  `makespan` receives the largest warp load.
JobPlan build_jobs_split(const std::vector<OutWork> &work, uint32_t W, const Costs &k, uint32_t split,
                         double &makespan, size_t batch, const std::vector<int> &cl)
{
    JobPlan jp;
    std::vector<Job> jobs;
    std::vector<int> job_cluster;
    jp.comb_off.assign(1, 0);
    double total = 0;
    for (auto &w : work) total += work_cost(w, k, batch);
    const double share = total / W;
    for (uint32_t j = 0; j < work.size(); ++j) {
        const double c = work_cost(work[j], k, batch);
        uint32_t P = (uint32_t)std::max(1.0, std::round(c / std::max(share, 1.0)));
        P = std::min(W, std::max(P, split));
        // a part must be worth its partial slot and final addition
        if (P <= 1 || c < 4 * k.last || cl[j] >= 0) {
            jobs.push_back({j, work[j]});
            job_cluster.push_back(cl[j]);
            continue;
        }
        std::vector<OutWork> chunk = split_work(work[j], P, k, batch);
        jp.comb_out.push_back(j);
        for (auto &ch : chunk) {
            if (ch.segs.empty() && ch.raws.empty()) continue;
            jobs.push_back({kPartBit | jp.n_part, std::move(ch)});
            job_cluster.push_back(-1);
            jp.comb_parts.push_back(jp.n_part++);
        }
        jp.comb_off.push_back((uint32_t)jp.comb_parts.size());
    }
    // units: the jobs of one cluster, or a single job
    std::vector<std::vector<uint32_t>> units;
    std::map<int, uint32_t> unit_of;
    for (uint32_t i = 0; i < jobs.size(); ++i) {
        if (job_cluster[i] < 0) {
            units.push_back({i});
            continue;
        }
        auto it = unit_of.find(job_cluster[i]);
        if (it == unit_of.end()) {
            unit_of[job_cluster[i]] = (uint32_t)units.size();
            units.push_back({i});
        } else {
            units[it->second].push_back(i);
        }
    }
    std::vector<double> jc(jobs.size()), uc(units.size(), 0);
    for (size_t i = 0; i < jobs.size(); ++i) jc[i] = work_cost(jobs[i].w, k, batch);
    for (size_t u = 0; u < units.size(); ++u)
        for (uint32_t i : units[u]) uc[u] += jc[i];
    std::vector<uint32_t> order(units.size());
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(), [&](uint32_t a, uint32_t b) { return uc[a] > uc[b]; });
    std::vector<double> load(W, 0);
    jp.per_warp.assign(W, {});
    for (uint32_t u : order) {
        const uint32_t wi = (uint32_t)(std::min_element(load.begin(), load.end()) - load.begin());
        for (uint32_t i : units[u]) jp.per_warp[wi].push_back(std::move(jobs[i]));
        load[wi] += uc[u];
    }
    makespan = *std::max_element(load.begin(), load.end());
    return jp;
}

// The split (1 to 4 parts per output) with the smallest largest warp load;
// a finer split must gain at least 3% to be taken.  With `sh`, outputs that
// share signed sums are clustered onto warps first.
JobPlan build_jobs_with(const std::vector<OutWork> &work, uint32_t W, const Costs &k, size_t batch,
                        const std::vector<int> &cl, double &best_ms)
{
    JobPlan best = build_jobs_split(work, W, k, 1, best_ms, batch, cl);
    for (uint32_t split = 2; split <= 4; ++split) {
        double ms = 0;
        JobPlan jp = build_jobs_split(work, W, k, split, ms, batch, cl);
        if (ms < 0.97 * best_ms) {
            best_ms = ms;
            best = std::move(jp);
        }
    }
    return best;
}

// Brings the users of shared sums onto one warp by swapping whole outputs of
// similar cost between warps, a sum at a time (best saving first), keeping
// every warp's load within `limit`; outputs already brought together stay.
void colocate(JobPlan &jp, const std::vector<OutWork> &work, const Costs &k, size_t batch, const Sharing &sh,
              double limit)
{
    const uint32_t W = (uint32_t)jp.per_warp.size();
    std::vector<int> warp_of(work.size(), -1), pinned(work.size(), 0);
    std::vector<double> load(W, 0), cost(work.size(), 0);
    for (uint32_t wi = 0; wi < W; ++wi)
        for (const Job &jb : jp.per_warp[wi]) {
            const double c = work_cost(jb.w, k, batch);
            load[wi] += c;
            if (!(jb.target & kPartBit)) {
                warp_of[jb.target] = (int)wi;
                cost[jb.target] = c;
            }
        }
    std::vector<uint32_t> order(sh.users.size());
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(), [&](uint32_t x, uint32_t y) { return sh.benefit[x] > sh.benefit[y]; });
    for (uint32_t nd : order) {
        const auto &us = sh.users[nd];
        if (us.size() < 2 || sh.benefit[nd] <= 0) continue;
        bool whole = true;
        for (uint32_t u : us) whole &= warp_of[u] >= 0;
        if (!whole) continue;
        // the warp already holding most of the users (pinned ones first); of
        // those, the least loaded (it will also form the sum)
        std::vector<int> votes(W, 0);
        for (uint32_t u : us) votes[warp_of[u]] += 1 + 4 * pinned[u];
        uint32_t t = 0;
        for (uint32_t wi = 1; wi < W; ++wi)
            if (votes[wi] > votes[t] || (votes[wi] == votes[t] && load[wi] < load[t])) t = wi;
        std::vector<std::pair<uint32_t, uint32_t>> swaps;  // (user, partner on t)
        std::vector<double> ld = load;
        std::vector<int> taken(work.size(), 0);
        bool ok = true;
        for (uint32_t u : us) {
            if ((uint32_t)warp_of[u] == t) continue;
            if (pinned[u]) {
                ok = false;
                break;
            }
            const uint32_t from = (uint32_t)warp_of[u];
            int best = -1;
            double bd = 0;
            for (size_t v = 0; v < work.size(); ++v) {
                if (warp_of[v] != (int)t || pinned[v] || taken[v] ||
                    std::find(us.begin(), us.end(), (uint32_t)v) != us.end())
                    continue;
                const double lt = ld[t] - cost[v] + cost[u], lf = ld[from] - cost[u] + cost[v];
                if (lt > limit || lf > limit) continue;
                const double d = std::fabs(cost[v] - cost[u]);
                if (best < 0 || d < bd) {
                    best = (int)v;
                    bd = d;
                }
            }
            if (best < 0) {
                ok = false;
                break;
            }
            taken[best] = 1;
            ld[t] += cost[u] - cost[best];
            ld[from] += cost[best] - cost[u];
            swaps.push_back({u, (uint32_t)best});
        }
        if (!ok) continue;
        for (auto &sp : swaps) {
            const uint32_t from = (uint32_t)warp_of[sp.first];
            warp_of[sp.second] = (int)from;
            warp_of[sp.first] = (int)t;
        }
        load = ld;
        for (uint32_t u : us) pinned[u] = 1;
    }
    // rebuild the warps' job lists (parts stay where they were; outputs that
    // share a warp follow one another in index order)
    std::vector<std::vector<Job>> pw(W);
    for (uint32_t wi = 0; wi < W; ++wi)
        for (Job &jb : jp.per_warp[wi])
            if (jb.target & kPartBit) pw[wi].push_back(std::move(jb));
    for (size_t j = 0; j < work.size(); ++j)
        if (warp_of[j] >= 0) pw[warp_of[j]].push_back({(uint32_t)j, work[j]});
    jp.per_warp = std::move(pw);
}

// ... then the users of shared sums are brought together by swaps within 1%
// of the largest warp load (warp balance is worth more than the additions a
// shared sum saves).
JobPlan build_jobs(const std::vector<OutWork> &work, uint32_t W, const Costs &k, size_t batch,
                   const Sharing *sh = nullptr)
{
    double ms = 0;
    JobPlan jp = build_jobs_with(work, W, k, batch, std::vector<int>(work.size(), -1), ms);
    if (sh) colocate(jp, work, k, batch, *sh, 1.01 * ms);
    return jp;
}

// Form of the signed-sum programs in a schedule (tiled.h): 16-bit source
// indices packed two per word, or one 32-bit byte offset (index * PB) per
// source, each program starting on a 16-byte boundary.
struct ProgForm {
    bool offsets = false;
    uint32_t PB = 0;  // bytes of one source tile pair
};

// Program words of a signed sum: n_plus | n_minus << 16, the runs and the
// slot word (counts, then up to six 4-bit slot numbers, plus slots first).
// A formation (`form_slot` >= 0) names the warp slot it fills: the word
// before its program in the packed form, the third word of its program in
// the offset form.
void put_program(std::vector<uint32_t> &w, const std::vector<uint32_t> &plus, const std::vector<uint32_t> &minus,
                 const std::vector<uint32_t> &plus_slots, const std::vector<uint32_t> &minus_slots,
                 const ProgForm &pf, int form_slot = -1)
{
    uint32_t sw = (uint32_t)plus_slots.size() | ((uint32_t)minus_slots.size() << 4);
    uint32_t j = 0;
    for (const auto *ss : {&plus_slots, &minus_slots})
        for (uint32_t sl : *ss) sw |= (sl & 15u) << (8 + 4 * j++);
    const uint32_t h = (uint32_t)plus.size() | ((uint32_t)minus.size() << 16);
    if (pf.offsets) {
        while (w.size() % 4) w.push_back(0);
        w.push_back(h);
        w.push_back(sw);
        w.push_back(form_slot >= 0 ? (uint32_t)form_slot : 0u);
        w.push_back(0);
        for (const auto *run : {&plus, &minus}) {
            for (uint32_t s : *run) w.push_back(s * pf.PB);
            while (w.size() % 4) w.push_back(0);
        }
        return;
    }
    if (form_slot >= 0) w.push_back((uint32_t)form_slot);
    w.push_back(h);
    for (const auto *run : {&plus, &minus})
        for (size_t i = 0; i < run->size(); i += 2)
            w.push_back(run->at(i) | (i + 1 < run->size() ? run->at(i + 1) << 16 : 0u));
    w.push_back(sw);
}

// A program decoded from schedule words (either form).
struct ProgRead {
    uint32_t np = 0, nm = 0;     // plus and minus run lengths
    uint32_t sw = 0;             // slot word
    uint32_t form_slot = 0;      // a formation's target slot
    std::vector<uint32_t> src;   // the plus run's source indices, then the minus run's
    size_t next = 0;             // word just past the program
};

// Decode the program at word p (a formation's, with its target slot, when
// `formation`), reading no word at or past `end`; false if it does not fit,
// is misaligned, or an offset is not a whole source.
bool read_program(const std::vector<uint32_t> &w, size_t p, size_t end, const ProgForm &pf, bool formation,
                  ProgRead &r)
{
    end = std::min(end, w.size());
    r = ProgRead{};
    if (pf.offsets) {
        if (p % 4 || p + 4 > end || pf.PB == 0) return false;
        r.np = w[p] & 0xffffu;
        r.nm = w[p] >> 16;
        r.sw = w[p + 1];
        r.form_slot = w[p + 2];
        if (!formation && w[p + 2]) return false;
        p += 4;
        for (uint32_t n : {r.np, r.nm}) {
            const size_t padded = ((size_t)n + 3) & ~(size_t)3;
            if (p + padded > end) return false;
            for (uint32_t i = 0; i < n; ++i) {
                if (w[p + i] % pf.PB) return false;
                r.src.push_back(w[p + i] / pf.PB);
            }
            p += padded;
        }
        r.next = p;
        return true;
    }
    if (formation) {
        if (p >= end) return false;
        r.form_slot = w[p++];
    }
    if (p >= end) return false;
    r.np = w[p] & 0xffffu;
    r.nm = w[p] >> 16;
    ++p;
    for (uint32_t n : {r.np, r.nm}) {
        if (p + (n + 1) / 2 > end) return false;
        for (uint32_t i = 0; i < n; ++i) r.src.push_back((w[p + i / 2] >> (16 * (i & 1))) & 0xffffu);
        p += (n + 1) / 2;
    }
    if (p >= end) return false;
    r.sw = w[p++];
    r.next = p;
    return true;
}

// The program form of a schedule, from its kernel arguments.
ProgForm prog_form(const TiledArgs &a)
{
    ProgForm pf;
    pf.offsets = a.src_offsets != 0;
    pf.PB = a.src_bytes / (a.n_in + a.n_nodes + 1);
    return pf;
}

// The whole schedule (see tiled.h).
struct Sched {
    std::vector<uint32_t> w;
    uint32_t o_level = 0, o_node_off = 0, o_warp = 0, o_comb_off = 0, o_comb_out = 0, o_comb_parts = 0;
    uint64_t pt_ops = 0;  // plaintext tiles fetched per tile
};

void pad4(std::vector<uint32_t> &w)
{
    while (w.size() % 4) w.push_back(0);
}

Sched encode(const JobPlan &jp, const std::vector<uint32_t> &level_off, const std::vector<Seg> &nodes, uint32_t W,
             uint32_t mac_budget, uint32_t zero_index, uint32_t P, const std::vector<uint32_t> *warp_slots = nullptr,
             const ProgForm &pf = ProgForm{})
{
    Sched sc;
    auto &w = sc.w;
    sc.o_level = 0;
    w.insert(w.end(), level_off.begin(), level_off.end());
    sc.o_node_off = (uint32_t)w.size();
    w.resize(w.size() + nodes.size());
    for (size_t k = 0; k < nodes.size(); ++k) {
        if (pf.offsets) pad4(w);
        w[sc.o_node_off + k] = (uint32_t)w.size();
        put_program(w, nodes[k].plus, nodes[k].minus, {}, {}, pf);
    }
    pad4(w);
    sc.o_warp = (uint32_t)w.size();
    w.resize(w.size() + (size_t)W * kWarpTableWords);
    std::vector<std::vector<uint32_t>> ops(W), segw(W), tgt(W);
    const uint32_t zero_src = zero_index;
    for (uint32_t wi = 0; wi < W; ++wi) {
        auto &o = ops[wi];
        for (const Job &jb : jp.per_warp[wi]) {
            const size_t first = o.size();
            const auto &raws = jb.w.raws;
            const auto &segs = jb.w.segs;
            size_t r = 0;
            auto raw_or_nop = [&]() {
                if (r < raws.size()) {
                    const auto &t = raws[r++];
                    return (t.second << kOpPtShift) | t.first;
                }
                return kOpNop | zero_src;
            };
            // Each SEG opens a batch.  The batches holding them are staggered
            // across warps and jobs, so that the signed sums (shared-memory
            // reads, formed before their batch) of different warps fall at
            // different times of the tile instead of all at its start.  A job
            // starts a batch (`first`) and is padded to whole batches.
            const size_t H = P;
            const size_t len = segs.size() + raws.size();
            const size_t b0 = (first + P - 1) / P * P;  // first batch start in the job
            const size_t nbs = std::max(segs.size(), first + len > b0 ? (first + len - b0 + P - 1) / P : 0);
            std::vector<uint8_t> seg_at(nbs, 0);
            if (!segs.empty()) {
                const size_t step = nbs / segs.size(), phase = (wi * 5 + tgt[wi].size() * 3) % nbs;
                for (size_t k = 0; k < segs.size(); ++k) {
                    size_t b = (phase + k * step) % nbs;
                    while (seg_at[b]) b = (b + 1) % nbs;
                    seg_at[b] = 1;
                }
            }
            size_t k = 0;
            for (size_t p = first; k < segs.size() || r < raws.size(); ++p) {
                if (p % P == 0 && k < segs.size() && seg_at[(p - b0) / P]) {
                    const Seg &sg = segs[k++];
                    for (const Form &f : sg.forms)
                        put_program(segw[wi], f.plus, f.minus, f.plus_slots, f.minus_slots, pf, (int)f.slot);
                    put_program(segw[wi], sg.plus, sg.minus, sg.plus_slots, sg.minus_slots, pf);
                    o.push_back((sg.scale_pt << kOpPtShift) | kOpSeg | (uint32_t)sg.forms.size());
                } else {
                    o.push_back(raw_or_nop());  // a NOP while a SEG waits for its batch
                }
            }
            if (o.size() == first) o.push_back(kOpNop | zero_src);  // an output with no terms
            while (o.size() % H) o.push_back(kOpNop | zero_src);
            o.back() |= kOpLast;
            // at most mac_budget products in an accumulator between reductions
            // (a FOLD opens a batch inside the job)
            auto products = [&](size_t from, size_t to) {
                uint32_t cnt = 0;
                for (size_t i = from; i < to; ++i) cnt += (o[i] & kOpNop) ? 0 : 1;
                return cnt;
            };
            const size_t end = o.size();
            uint32_t nprod = products(first, std::min(b0, end));
            sc.pt_ops += nprod;
            for (size_t b = b0; b < end; b += P) {
                const uint32_t cnt = products(b, std::min(b + P, end));
                if (nprod + cnt > mac_budget) {
                    o[b] |= kOpFold;
                    nprod = 1;
                }
                nprod += cnt;
                sc.pt_ops += cnt;
            }
            tgt[wi].push_back(jb.target);
        }
        while (o.size() % P) o.push_back(kOpNop | zero_src);
        // a NOP loads a plaintext tile that another operation of its batch (or
        // the nearest earlier one) loads too (the same words: same index, same
        // CONST flag)
        uint32_t last_pt = 0, last_const = 0;
        for (size_t b = 0; b < o.size(); b += P) {
            for (size_t i = b; i < b + P; ++i)
                if (!(o[i] & kOpNop)) {
                    last_pt = o[i] >> kOpPtShift;
                    last_const = o[i] & kOpConst;
                    break;
                }
            for (size_t i = b; i < b + P; ++i)
                if (o[i] & kOpNop)
                    o[i] = (o[i] & ((1u << kOpPtShift) - 1) & ~kOpConst) | last_const | (last_pt << kOpPtShift);
        }
    }
    for (uint32_t wi = 0, first = 0; wi < W; ++wi) {
        pad4(w);
        w[sc.o_warp + wi * kWarpTableWords + 0] = (uint32_t)w.size();
        w[sc.o_warp + wi * kWarpTableWords + 1] = (uint32_t)ops[wi].size();
        w[sc.o_warp + wi * kWarpTableWords + 4] = first;
        if (warp_slots) first += (*warp_slots)[wi];
        w.insert(w.end(), ops[wi].begin(), ops[wi].end());
    }
    for (uint32_t wi = 0; wi < W; ++wi) {  // (offset form: every program a multiple of four words)
        w[sc.o_warp + wi * kWarpTableWords + 2] = (uint32_t)w.size();
        w.insert(w.end(), segw[wi].begin(), segw[wi].end());
    }
    for (uint32_t wi = 0; wi < W; ++wi) {
        w[sc.o_warp + wi * kWarpTableWords + 3] = (uint32_t)w.size();
        w.insert(w.end(), tgt[wi].begin(), tgt[wi].end());
    }
    sc.o_comb_off = (uint32_t)w.size();
    w.insert(w.end(), jp.comb_off.begin(), jp.comb_off.end());
    sc.o_comb_out = (uint32_t)w.size();
    w.insert(w.end(), jp.comb_out.begin(), jp.comb_out.end());
    sc.o_comb_parts = (uint32_t)w.size();
    w.insert(w.end(), jp.comb_parts.begin(), jp.comb_parts.end());
    while (w.size() % 32) w.push_back(0);  // a multiple of 128 bytes: the regions after it take TMA copies
    return sc;
}

// Shared sums of the plan (those reachable from a use), their unresolved
// operand lists, and what keeping each one saves.
struct NodeInfo {
    std::vector<uint32_t> ids;                                  // plan node ids in index order
    std::vector<std::vector<std::pair<uint32_t, int>>> kids;    // per plan node: (operand, sign)
    std::vector<double> benefit;                                // per plan node
};

// Resolution of operands against a set of kept shared sums.
struct Resolver {
    const NodeInfo &ni;
    const std::vector<int32_t> &slot;  // per plan node: source index if kept, else -1
    void add(uint32_t opnd, int sign, std::vector<uint32_t> &plus, std::vector<uint32_t> &minus) const
    {
        if (!(opnd & kNodeTag)) {
            (sign < 0 ? minus : plus).push_back(opnd);
            return;
        }
        const uint32_t k = opnd & ~kNodeTag;
        if (slot[k] >= 0) {
            (sign < 0 ? minus : plus).push_back((uint32_t)slot[k]);
            return;
        }
        for (auto &c : ni.kids[k]) add(c.first, sign * c.second, plus, minus);
    }
};

struct Lowered {
    std::vector<OutWork> work;      // resolved, runs cut to the lazy-sum bound
    std::vector<Seg> nodes;         // kept sums in slot order
    std::vector<uint32_t> level_off;
    uint32_t n_levels = 0;
};

// Resolve every operand list against the `keep` set (plan node ids, at most
// `keep_n` of them taken from `rank` order); a kept sum whose own runs would
// exceed `budget` is dropped, since it must be one lazy sum.  Scale groups
// are cut into pieces whose plus and minus runs are at most `budget` long.
Lowered resolve(const HostPlan &hp, const NodeInfo &ni, const std::vector<OutWork> &groups,
                const std::vector<uint32_t> &rank, uint32_t keep_n, uint32_t budget)
{
    const uint32_t n_in = hp.n_in;
    std::vector<uint8_t> kept(hp.n_nodes, 0);
    for (uint32_t i = 0; i < keep_n && i < rank.size(); ++i) kept[rank[i]] = 1;
    std::vector<int32_t> slot(hp.n_nodes, -1);
    std::vector<uint32_t> level(hp.n_nodes, 0);
    Lowered lw;
    for (bool changed = true; changed;) {
        changed = false;
        // slots in index order (children first: a child's index is lower)
        std::fill(slot.begin(), slot.end(), -1);
        uint32_t n = 0;
        for (uint32_t k : ni.ids)
            if (kept[k]) slot[k] = (int32_t)(n_in + n++);
        Resolver rv{ni, slot};
        for (uint32_t k : ni.ids) {
            if (!kept[k]) continue;
            Seg s;
            for (auto &c : ni.kids[k]) rv.add(c.first, c.second, s.plus, s.minus);
            if (s.plus.size() > budget || s.minus.size() > budget) {
                kept[k] = 0;
                changed = true;
                break;
            }
        }
    }
    Resolver rv{ni, slot};
    // kept sums ordered by level, then index
    std::vector<uint32_t> order;
    for (uint32_t k : ni.ids) {
        if (!kept[k]) continue;
        uint32_t lev = 0;
        std::vector<uint32_t> stack;
        for (auto &c : ni.kids[k]) stack.push_back(c.first);
        while (!stack.empty()) {  // kept descendants reached through dropped sums
            const uint32_t o = stack.back();
            stack.pop_back();
            if (!(o & kNodeTag)) continue;
            const uint32_t c = o & ~kNodeTag;
            if (kept[c]) lev = std::max(lev, level[c] + 1);
            else for (auto &g : ni.kids[c]) stack.push_back(g.first);
        }
        level[k] = lev;
        lw.n_levels = std::max(lw.n_levels, lev + 1);
        order.push_back(k);
    }
    std::stable_sort(order.begin(), order.end(), [&](uint32_t a, uint32_t b) { return level[a] < level[b]; });
    // renumber slots in level order
    std::vector<int32_t> slot2(hp.n_nodes, -1);
    for (uint32_t i = 0; i < order.size(); ++i) slot2[order[i]] = (int32_t)(n_in + i);
    Resolver rv2{ni, slot2};
    lw.level_off.assign(lw.n_levels + 1, 0);
    for (uint32_t k : order) {
        Seg s;
        for (auto &c : ni.kids[k]) rv2.add(c.first, c.second, s.plus, s.minus);
        lw.nodes.push_back(std::move(s));
        ++lw.level_off[level[k] + 1];
    }
    for (uint32_t l = 0; l < lw.n_levels; ++l) lw.level_off[l + 1] += lw.level_off[l];
    (void)rv;
    lw.work.resize(groups.size());
    for (size_t j = 0; j < groups.size(); ++j) {
        OutWork &o = lw.work[j];
        o.raws = groups[j].raws;
        for (const Seg &g : groups[j].segs) {
            // g.plus holds tagged operands with their signs folded in: plus and minus lists
            Seg s;
            s.scale_pt = g.scale_pt;
            for (uint32_t op : g.plus) rv2.add(op, +1, s.plus, s.minus);
            for (uint32_t op : g.minus) rv2.add(op, -1, s.plus, s.minus);
            if (s.plus.empty() && s.minus.empty()) continue;
            size_t pb = 0, mb = 0;
            do {  // runs of at most `budget` words
                const size_t pe = std::min(s.plus.size(), pb + budget);
                const size_t me = std::min(s.minus.size(), mb + budget);
                Seg piece;
                piece.scale_pt = s.scale_pt;
                piece.plus.assign(s.plus.begin() + pb, s.plus.begin() + pe);
                piece.minus.assign(s.minus.begin() + mb, s.minus.begin() + me);
                o.segs.push_back(std::move(piece));
                pb = pe;
                mb = me;
            } while (pb < s.plus.size() || mb < s.minus.size());
        }
    }
    return lw;
}

// Shared signed sums formed by the warps that use them (Sec. 4.2 "Sharing
// Signed Sums").  For each warp, every shared sum that the warp's outputs use
// at least twice is formed once per tile, by that warp, into one of its
// slots, right before the first scale group that needs it, and read from
// there by every later use on the warp; a sum's own program may read sums
// formed before it.  Slots are reused once a sum has no use left in the
// tile.  Sums a warp uses once, or that would need more than `max_slots`
// slots, more than six slot operands in one program or runs beyond
// `budget`, are expanded into their terms (the same residues).  Rewrites the
// jobs' scale groups (whole outputs only; parts of split outputs keep their
// expanded terms) and returns the slots per warp and the sums formed per
// tile.
struct LocalResult {
    uint32_t n_slots = 0;              // slots of all warps
    uint32_t formed = 0;               // sums formed per tile, all warps
    std::vector<uint32_t> warp_slots;  // per warp
};

LocalResult localize(JobPlan &jp, const std::vector<OutWork> &groups, const NodeInfo &ni, uint32_t budget,
                     uint32_t max_slots)
{
    LocalResult res;
    res.warp_slots.assign(jp.per_warp.size(), 0);
    const size_t n_nodes = ni.kids.size();
    for (size_t wi = 0; wi < jp.per_warp.size(); ++wi) {
        auto &jobs = jp.per_warp[wi];
        std::vector<uint32_t> uses(n_nodes, 0);
        for (const Job &jb : jobs) {
            if (jb.target & kPartBit) continue;
            for (const Seg &g : groups[jb.target].segs)
                for (const auto *l : {&g.plus, &g.minus})
                    for (uint32_t o : *l)
                        if (o & kNodeTag) ++uses[o & ~kNodeTag];
        }
        std::vector<char> local(n_nodes, 0);
        bool any = false;
        for (size_t k = 0; k < n_nodes; ++k)
            if (uses[k] >= 2) local[k] = any = 1;
        if (!any) continue;
        // operands of an unresolved list against the local set
        struct Res {
            std::vector<uint32_t> plus, minus, np, nm;  // sources; local sums (plan node ids)
        };
        std::function<void(uint32_t, int, Res &)> expand = [&](uint32_t o, int sign, Res &r) {
            if (!(o & kNodeTag)) {
                (sign < 0 ? r.minus : r.plus).push_back(o);
                return;
            }
            const uint32_t k = o & ~kNodeTag;
            if (local[k]) {
                (sign < 0 ? r.nm : r.np).push_back(k);
                return;
            }
            for (auto &c : ni.kids[k]) expand(c.first, sign * c.second, r);
        };
        for (int round = 0; round < 64; ++round) {
            // every scale group of the warp's whole outputs, in stream order
            std::vector<Res> segres;
            std::vector<uint32_t> seg_job, seg_grp;
            for (uint32_t ji = 0; ji < jobs.size(); ++ji) {
                if (jobs[ji].target & kPartBit) continue;
                const auto &gs = groups[jobs[ji].target].segs;
                for (uint32_t gi = 0; gi < gs.size(); ++gi) {
                    Res r;
                    for (uint32_t o : gs[gi].plus) expand(o, +1, r);
                    for (uint32_t o : gs[gi].minus) expand(o, -1, r);
                    segres.push_back(std::move(r));
                    seg_job.push_back(ji);
                    seg_grp.push_back(gi);
                }
            }
            std::vector<Res> nodres(n_nodes);
            for (size_t k = 0; k < n_nodes; ++k)
                if (local[k])
                    for (auto &c : ni.kids[k]) expand(c.first, c.second, nodres[k]);
            // formation points (children first) and last uses
            std::vector<int> formed_at(n_nodes, -1), last(n_nodes, -1);
            std::vector<std::vector<uint32_t>> forms(segres.size());
            std::function<void(uint32_t, int)> need = [&](uint32_t k, int si) {
                last[k] = std::max(last[k], si);
                if (formed_at[k] >= 0) return;
                for (uint32_t c : nodres[k].np) need(c, si);
                for (uint32_t c : nodres[k].nm) need(c, si);
                formed_at[k] = si;
                forms[si].push_back(k);
            };
            for (int si = 0; si < (int)segres.size(); ++si) {
                for (uint32_t k : segres[si].np) need(k, si);
                for (uint32_t k : segres[si].nm) need(k, si);
            }
            // constraints: six slot operands a program, runs within the budget
            int bad = -1;
            auto check = [&](const Res &r, bool is_node) {
                if (r.np.size() + r.nm.size() > 6) return false;
                if (is_node && (r.plus.size() + r.np.size() > budget || r.minus.size() + r.nm.size() > budget))
                    return false;
                return true;
            };
            for (size_t k = 0; k < n_nodes && bad < 0; ++k)
                if (local[k] && formed_at[k] >= 0 && !check(nodres[k], true)) bad = (int)k;
            for (size_t si = 0; si < segres.size() && bad < 0; ++si)
                if (!check(segres[si], false)) {
                    const auto &r = segres[si];
                    bad = (int)(r.np.empty() ? r.nm.back() : r.np.back());
                }
            // slots by lifetime
            std::vector<int> slot(n_nodes, -1);
            uint32_t live_max = 0;
            if (bad < 0) {
                std::vector<char> busy(16, 0);
                for (int si = 0; si < (int)segres.size() && bad < 0; ++si) {
                    for (uint32_t k : forms[si]) {
                        int f = -1;
                        for (uint32_t x = 0; x < max_slots; ++x)
                            if (!busy[x]) {
                                f = (int)x;
                                break;
                            }
                        if (f < 0) {
                            bad = (int)k;
                            break;
                        }
                        busy[f] = 1;
                        slot[k] = f;
                        live_max = std::max(live_max, (uint32_t)f + 1);
                    }
                    for (size_t k = 0; k < n_nodes; ++k)
                        if (slot[k] >= 0 && last[k] == si && busy[slot[k]]) busy[slot[k]] = 0;
                }
            }
            if (bad >= 0) {  // expand the offending sum and try again
                local[bad] = 0;
                continue;
            }
            // rewrite the scale groups of the warp's whole outputs
            std::vector<std::vector<Seg>> newsegs(jobs.size());
            for (size_t si = 0; si < segres.size(); ++si) {
                const Res &r = segres[si];
                const uint32_t ji = seg_job[si];
                const Seg &g = groups[jobs[ji].target].segs[seg_grp[si]];
                std::vector<Form> fs;
                for (uint32_t k : forms[si]) {
                    Form f;
                    f.slot = (uint32_t)slot[k];
                    f.plus = nodres[k].plus;
                    f.minus = nodres[k].minus;
                    for (uint32_t c : nodres[k].np) f.plus_slots.push_back((uint32_t)slot[c]);
                    for (uint32_t c : nodres[k].nm) f.minus_slots.push_back((uint32_t)slot[c]);
                    fs.push_back(std::move(f));
                }
                std::vector<uint32_t> ps, ms;
                for (uint32_t k : r.np) ps.push_back((uint32_t)slot[k]);
                for (uint32_t k : r.nm) ms.push_back((uint32_t)slot[k]);
                if (r.plus.empty() && r.minus.empty() && ps.empty() && ms.empty() && fs.empty()) continue;
                size_t pb = 0, mb = 0;
                bool first = true;
                do {  // runs of at most `budget` operands, slot operands in the first piece
                    Seg piece;
                    piece.scale_pt = g.scale_pt;
                    if (first) {
                        piece.plus_slots = ps;
                        piece.minus_slots = ms;
                        piece.forms = std::move(fs);
                    }
                    const size_t pe = std::min(r.plus.size(), pb + budget - piece.plus_slots.size());
                    const size_t me = std::min(r.minus.size(), mb + budget - piece.minus_slots.size());
                    piece.plus.assign(r.plus.begin() + pb, r.plus.begin() + pe);
                    piece.minus.assign(r.minus.begin() + mb, r.minus.begin() + me);
                    pb = pe;
                    mb = me;
                    first = false;
                    newsegs[ji].push_back(std::move(piece));
                } while (pb < r.plus.size() || mb < r.minus.size());
            }
            for (uint32_t ji = 0; ji < jobs.size(); ++ji)
                if (!(jobs[ji].target & kPartBit)) jobs[ji].w.segs = std::move(newsegs[ji]);
            for (size_t k = 0; k < n_nodes; ++k) res.formed += formed_at[k] >= 0 ? 1 : 0;
            res.warp_slots[wi] = live_max;
            res.n_slots += live_max;
            break;
        }
    }
    return res;
}

// The scale groups' signed sums as one tensor-core contraction per tile
// (tc_signed.cuh): every used group of every output (shared sums expanded
// into their terms) becomes one materialised source, the group's column of
// the weight matrix W, formed per tile before the operation streams run; the
// group's product by gamma is then an ordinary operation on that source.
struct TcPlan {
    bool ok = false;
    std::vector<OutWork> work;  // per output: its raw terms, then one operation per group source
    std::vector<Seg> nodes;     // the group sums, over inputs only
    uint32_t K = 0, N = 0;      // contraction length (inputs, padded to 16) and width (groups, padded to 8)
    uint32_t wabs = 0;          // largest sum of |weights| of a group
    uint32_t cols = 0;          // tensor memory columns a CTA allocates (a power of two)
};

// exact fp16 bits of an integer |v| <= 2048
uint16_t fp16_of_int(int v)
{
    if (v == 0) return 0;
    const uint16_t sgn = v < 0 ? 0x8000 : 0;
    const uint32_t a = (uint32_t)(v < 0 ? -v : v);
    int e = 0;
    while ((a >> (e + 1)) != 0) ++e;
    return (uint16_t)(sgn | ((e + 15) << 10) | ((a << (10 - e)) & 0x3FFu));
}

// net weight of each input in a program's plus and minus lists
std::vector<int> net_weights(const Seg &s, uint32_t n_in)
{
    std::vector<int> w(n_in, 0);
    for (uint32_t i : s.plus) ++w[i];
    for (uint32_t i : s.minus) --w[i];
    return w;
}

TcPlan plan_tc(const HostPlan &hp, const NodeInfo &ni, const std::vector<OutWork> &groups, uint64_t q_max)
{
    TcPlan tc;
    const uint32_t n_in = hp.n_in;
    const std::vector<int32_t> none(hp.n_nodes, -1);
    const Resolver rv{ni, none};
    tc.work.resize(groups.size());
    for (size_t j = 0; j < groups.size(); ++j) {
        tc.work[j].raws = groups[j].raws;
        for (const Seg &g : groups[j].segs) {
            Seg s;
            s.scale_pt = g.scale_pt;
            for (uint32_t op : g.plus) rv.add(op, +1, s.plus, s.minus);
            for (uint32_t op : g.minus) rv.add(op, -1, s.plus, s.minus);
            const std::vector<int> w = net_weights(s, n_in);
            if (std::all_of(w.begin(), w.end(), [](int x) { return x == 0; })) continue;
            tc.work[j].raws.push_back({n_in + (uint32_t)tc.nodes.size(), s.scale_pt});
            tc.nodes.push_back(std::move(s));
        }
    }
    const uint32_t ng = (uint32_t)tc.nodes.size();
    if (!ng || n_in + ng + 1 > kOpMaxSources) return tc;
    tc.K = (n_in + 15) & ~15u;
    tc.N = std::max(8u, (ng + 7) & ~7u);
    if (tc.N > 256) return tc;
    const TcGeometry geo{tc.K, tc.N};
    if (geo.cols() > 512) return tc;
    tc.cols = 32;
    while (tc.cols < geo.cols()) tc.cols *= 2;
    for (const Seg &s : tc.nodes) {
        int cs = 0;
        uint32_t ab = 0;
        for (int x : net_weights(s, n_in)) {
            if (x > 2048 || x < -2048) return tc;
            cs += x;
            ab += (uint32_t)std::abs(x);
        }
        // exact chunk sums in fp32 (2047 * ab < 2^24), the magic constant
        // exact (|1024 cs| < 2^22), S + wabs * q below 2^64
        if (ab > 8191 || std::abs(cs) >= 4096) return tc;
        tc.wabs = std::max(tc.wabs, ab);
    }
    if ((unsigned __int128)2 * tc.wabs * q_max >= ((unsigned __int128)1 << 64)) return tc;
    tc.ok = true;
    return tc;
}

// Append W (fp16, K-major core matrices, tc_signed.cuh) and the groups'
// magic constants to the schedule; returns their word offsets.
void append_tc(std::vector<uint32_t> &w, const TcPlan &tc, uint32_t n_in, uint32_t &o_w, uint32_t &o_magic)
{
    const TcGeometry geo{tc.K, tc.N};
    pad4(w);
    o_w = (uint32_t)w.size();
    w.resize(w.size() + geo.w_bytes() / 4, 0);
    for (uint32_t n = 0; n < tc.nodes.size(); ++n) {
        const std::vector<int> wt = net_weights(tc.nodes[n], n_in);
        for (uint32_t k = 0; k < n_in; ++k) {
            const uint32_t b = (n / 8) * geo.sbo() + (k / 8) * 128 + (n % 8) * 16 + (k % 8) * 2;
            w[o_w + b / 4] |= (uint32_t)fp16_of_int(wt[k]) << (16 * ((b / 2) & 1));
        }
    }
    o_magic = (uint32_t)w.size();
    for (uint32_t n = 0; n < tc.nodes.size(); ++n) {
        const std::vector<int> wt = net_weights(tc.nodes[n], n_in);
        const int cs = std::accumulate(wt.begin(), wt.end(), 0);
        const float magic = 12582912.0f - 1024.0f * (float)cs;
        uint32_t bits;
        memcpy(&bits, &magic, 4);
        w.push_back(bits);
    }
    while (w.size() % 32) w.push_back(0);
}

// Check the contraction's tables against the node programs the schedule
// holds (the sums the linear-map check verified): every weight, the padding
// zero, each magic constant, the bound wabs, and the layout.
const char *check_tc(const std::vector<uint32_t> &w, const TiledArgs &a)
{
    if (!a.tc_groups) return nullptr;
    if (a.tc_groups != a.n_nodes || a.n_levels != 1) return "tensor-core sums: node count";
    const TcGeometry geo{a.tc_k, a.tc_n};
    if (a.tc_k % 16 || a.tc_k < a.n_in || a.tc_n % 8 || a.tc_n < std::max(a.tc_groups, 8u) || a.tc_n > 256 ||
        geo.cols() > a.tc_cols || a.tc_cols > 512 || (a.tc_cols & (a.tc_cols - 1)) || a.tc_cols < 32)
        return "tensor-core sums: geometry";
    if (a.o_tcw % 4 || (size_t)a.o_tcw + geo.w_bytes() / 4 > a.o_tcm || (size_t)a.o_tcm + a.tc_groups > w.size())
        return "tensor-core sums: layout";
    for (uint32_t n = 0; n < a.tc_n; ++n) {
        std::vector<int> want(a.tc_k, 0);
        if (n < a.tc_groups) {  // the node program: plus run, minus run, inputs only
            ProgRead r;
            if (!read_program(w, w[a.o_node_off + n], w.size(), prog_form(a), false, r))
                return "tensor-core sums: node program";
            for (uint32_t i = 0; i < r.np + r.nm; ++i) {
                if (r.src[i] >= a.n_in) return "tensor-core sums: a node reads a non-input";
                want[r.src[i]] += i < r.np ? 1 : -1;
            }
            if (r.sw != 0) return "tensor-core sums: a node reads warp slots";
        }
        int cs = 0;
        uint32_t ab = 0;
        for (uint32_t k = 0; k < a.tc_k; ++k) {
            const uint32_t b = (n / 8) * geo.sbo() + (k / 8) * 128 + (n % 8) * 16 + (k % 8) * 2;
            const uint16_t h = (uint16_t)(w[a.o_tcw + b / 4] >> (16 * ((b / 2) & 1)));
            if (std::abs(want[k]) > 2048 || h != fp16_of_int(want[k])) return "tensor-core sums: weight";
            cs += want[k];
            ab += (uint32_t)std::abs(want[k]);
        }
        if (n < a.tc_groups) {
            const float magic = 12582912.0f - 1024.0f * (float)cs;
            uint32_t bits;
            memcpy(&bits, &magic, 4);
            if (w[a.o_tcm + n] != bits || std::abs(cs) >= 4096 || ab > 8191 || ab > a.tc_wabs)
                return "tensor-core sums: constants";
        }
    }
    return nullptr;
}

// Add/Sub a schedule performs per evaluation, in the units of the paper's
// counts (a sum of n operands costs n - 1): the shared sums formed for the
// block and by warps, every scale group's signed sum, each job's products
// added together, and the partial sums of split outputs.
uint32_t count_addsub(const std::vector<uint32_t> &w, const TiledArgs &a, uint32_t W)
{
    uint64_t n = 0;
    const ProgForm pf = prog_form(a);
    // operands of the program at word p (a formation's when `form`); p is left past it
    auto program = [&](size_t &p, bool form) -> uint64_t {
        ProgRead r;
        if (!read_program(w, p, w.size(), pf, form, r)) return 1;  // (check_schedule rejects the schedule)
        p = r.next;
        return (uint64_t)r.np + r.nm + (r.sw & 15u) + ((r.sw >> 4) & 15u);
    };
    for (uint32_t x = 0; x < a.n_nodes; ++x) {
        size_t p = w[a.o_node_off + x];
        n += program(p, false) - 1;
    }
    for (uint32_t wi = 0; wi < W; ++wi) {
        const size_t t = a.o_warp + (size_t)wi * kWarpTableWords;
        const uint32_t op0 = w[t], n_ops = w[t + 1];
        size_t sp = w[t + 2];
        uint64_t products = 0;
        for (uint32_t f = 0; f < n_ops; ++f) {
            const uint32_t op = w[op0 + f];
            if (op & kOpSeg) {
                for (uint32_t g = 0; g < (op & (kOpMaxSources - 1)); ++g) n += program(sp, true) - 1;
                const uint64_t k = program(sp, false);
                if (k) n += k - 1;
            }
            if (!(op & kOpNop)) ++products;
            if (op & kOpLast) {
                if (products) n += products - 1;
                products = 0;
            }
        }
    }
    for (uint32_t r = 0; r < a.n_comb; ++r) n += w[a.o_comb_off + r + 1] - w[a.o_comb_off + r] - 1;
    return (uint32_t)std::min<uint64_t>(n, 0xffffffffu);
}

int upload_blob(TiledSchedule *ts, const std::vector<uint32_t> &words)
{
    const size_t bytes = std::max<size_t>(words.size() * 4, 256);
    cudaError_t e = cudaMalloc(&ts->sched.blob, bytes);
    if (e != cudaSuccess) return set_error(FIONA_ERR_NOMEM, "tiled schedule: %s", cudaGetErrorString(e));
    ts->sched.bytes = bytes;
    e = cudaMemcpy(ts->sched.blob, words.data(), words.size() * 4, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled schedule: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

// Walk the schedule words exactly as the kernel does and check every index
// and offset it will use: plaintexts, sources, partial slots, outputs, the
// ends of each stream, alignment, and the shared-memory layout.  Returns an
// explanation of the first violation, or null.
const char *check_schedule(const std::vector<uint32_t> &w, const TiledArgs &a, uint32_t W, uint32_t n_out,
                           uint32_t n_pt, size_t smem, uint32_t PB, uint32_t P)
{
    const size_t nw = w.size();
    if (a.sched_bytes != nw * 4 || a.sched_bytes % 128) return "schedule size";
    if (a.n_in && (a.box_rows == 0 || a.box_rows > 256 || a.box_rows > 2 * a.n_in ||
                   (size_t)a.n_boxes * a.box_rows < 2ull * a.n_in || a.n_boxes > 2 * a.n_in))
        return "input boxes";
    const uint32_t n_src = a.n_in + a.n_nodes, zero = n_src;  // the zero tile follows the sources
    if (n_src + 1 > kOpMaxSources) return "too many sources";
    if ((size_t)a.sched_bytes + (size_t)(a.double_buffer ? 2 : 1) * a.src_bytes + (size_t)a.n_part * PB +
            (size_t)a.n_slots * PB + (a.tc_groups ? 32 : 24) >
        smem)
        return "shared-memory layout";
    if (a.src_bytes != (n_src + 1) * PB) return "source region size";
    auto at = [&](size_t i, uint32_t &v) {
        if (i >= nw) return false;
        v = w[i];
        return true;
    };
    // a signed-sum program at word `o` (a formation's, whose target slot is
    // below `slot_lim`, when `form`) whose indices must be below `lim` and
    // whose slot numbers below `slot_lim`; in the offset form every offset a
    // whole source and the program on a 16-byte boundary (read_program)
    const ProgForm pf = prog_form(a);
    if (pf.offsets && pf.PB != PB) return "program form";
    auto program = [&](size_t o, uint32_t lim, size_t end, size_t &next, uint32_t slot_lim, bool form) -> bool {
        ProgRead r;
        if (!read_program(w, o, end, pf, form, r)) return false;
        for (uint32_t x : r.src)
            if (x >= lim) return false;
        if (form && r.form_slot >= slot_lim) return false;
        const uint32_t ns = (r.sw & 15u) + ((r.sw >> 4) & 15u);
        if (ns > 6 || (ns < 6 && (r.sw >> (8 + 4 * ns)) != 0)) return false;
        for (uint32_t j = 0; j < ns; ++j)
            if (((r.sw >> (8 + 4 * j)) & 15u) >= slot_lim) return false;
        next = r.next;
        return true;
    };
    // levels and node programs
    for (uint32_t l = 0; l <= a.n_levels; ++l) {
        uint32_t v;
        if (!at(a.o_level + l, v) || v > a.n_nodes) return "level table";
        if (l > 0 && v < w[a.o_level + l - 1]) return "level order";
    }
    if (a.n_levels && w[a.o_level + a.n_levels] != a.n_nodes) return "level table end";
    for (uint32_t l = 0; l < a.n_levels; ++l)
        for (uint32_t x = w[a.o_level + l]; x < w[a.o_level + l + 1]; ++x) {
            uint32_t off;
            size_t next;
            // a node reads inputs and nodes of lower levels only
            if (!at(a.o_node_off + x, off) || !program(off, a.n_in + w[a.o_level + l], a.o_warp, next, 0, false))
                return "node program";
        }
    // warp streams
    for (uint32_t wi = 0; wi < W; ++wi) {
        const size_t t = a.o_warp + (size_t)wi * kWarpTableWords;
        if (t + kWarpTableWords > nw) return "warp table";
        const uint32_t op0 = w[t], n_ops = w[t + 1], seg0 = w[t + 2], tg0 = w[t + 3];
        if (op0 % 4 || n_ops % P || (size_t)op0 + n_ops > nw) return "op stream";
        // this warp's slots: from its first to the next warp's first (or the end)
        const uint32_t sl0 = w[t + 4], sl1 = wi + 1 < W ? w[t + kWarpTableWords + 4] : a.n_slots;
        if (sl1 < sl0 || sl1 > a.n_slots) return "warp slot table";
        const uint32_t n_wslots = sl1 - sl0;
        size_t sp = seg0, tp = tg0;
        const size_t seg_end = wi + 1 < W ? w[t + kWarpTableWords + 2] : w[a.o_warp + 3];
        const size_t tg_end = wi + 1 < W ? w[t + kWarpTableWords + 3] : a.o_comb_off;
        bool open = false;
        for (uint32_t f = 0; f < n_ops; ++f) {
            const uint32_t op = w[op0 + f];
            const uint32_t pos = f % P;
            if ((op & (kOpSeg | kOpFold)) && pos != 0) return "SEG or FOLD inside a batch";
            if ((op & kOpLast) && pos != P - 1) return "LAST inside a batch";
            // every operation loads a plaintext tile, NOPs included
            if ((op >> kOpPtShift) >= std::max<uint32_t>(n_pt, 1)) return "plaintext index";
            if ((op & kOpConst) && (op & kOpSeg)) return "SEG marked CONST";
            if (a.kc_all && pos != 0 && !(op & (kOpNop | kOpConst))) return "RAW read as constant";
            if (op & kOpNop) {
                if (op & kOpSeg) return "SEG marked NOP";
                if ((op & (kOpMaxSources - 1)) != zero) return "NOP source";
            } else if (op & kOpSeg) {
                size_t next;
                for (uint32_t f = 0; f < (op & (kOpMaxSources - 1)); ++f) {  // formations into warp slots
                    if (!program(sp, n_src, seg_end, next, n_wslots, true)) return "formation program";
                    sp = next;
                }
                if (!program(sp, n_src, seg_end, next, n_wslots, false)) return "segment program";
                sp = next;
                open = true;
            } else {
                if ((op & (kOpMaxSources - 1)) >= n_src) return "source index";
                open = true;
            }
            if (op & kOpLast) {
                uint32_t tg;
                if (tp >= tg_end || !at(tp, tg)) return "target stream";
                ++tp;
                if (tg & kPartBit) {
                    if ((tg & ~kPartBit) >= a.n_part) return "partial slot";
                } else if (tg >= n_out) {
                    return "output index";
                }
                open = false;
            }
        }
        if (open) return "job without LAST";
        if (sp != seg_end) return "segment stream length";
        if (tp != tg_end) return "target stream length";
    }
    // combine lists
    for (uint32_t r = 0; r <= a.n_comb; ++r) {
        uint32_t v;
        if (!at(a.o_comb_off + r, v)) return "combine table";
    }
    for (uint32_t r = 0; r < a.n_comb; ++r) {
        uint32_t o;
        if (!at(a.o_comb_out + r, o) || o >= n_out) return "combine output";
        for (uint32_t q = w[a.o_comb_off + r]; q < w[a.o_comb_off + r + 1]; ++q) {
            uint32_t ps;
            if (!at(a.o_comb_parts + q, ps) || ps >= a.n_part) return "combine part";
        }
    }
    return nullptr;
}

const char *check_linear_map(const std::vector<uint32_t> &w, const TiledArgs &a, uint32_t W, const HostPlan &hp)
{
    using Expr = std::vector<std::pair<uint32_t, int64_t>>;  // (input, coefficient), sorted
    auto add = [](Expr &dst, const Expr &src, int64_t f) {
        Expr out;
        size_t i = 0, j = 0;
        while (i < dst.size() || j < src.size()) {
            if (j == src.size() || (i < dst.size() && dst[i].first < src[j].first)) {
                out.push_back(dst[i++]);
            } else if (i == dst.size() || src[j].first < dst[i].first) {
                out.push_back({src[j].first, src[j].second * f});
                ++j;
            } else {
                const int64_t v = dst[i].second + src[j].second * f;
                if (v) out.push_back({dst[i].first, v});
                ++i;
                ++j;
            }
        }
        dst.swap(out);
    };
    std::vector<Expr> src(a.n_in + a.n_nodes + 1);  // + the zero tile
    for (uint32_t i = 0; i < a.n_in; ++i) src[i] = {{i, 1}};
    std::vector<Expr> slot(std::max<uint32_t>(a.n_slots, 1));  // the current warp's slots
    const ProgForm pf = prog_form(a);
    // a signed-sum program at word p (a formation's when `form`: its target
    // slot goes to *fs); p is left past it (check_schedule has walked every
    // program before)
    auto program = [&](size_t &p, Expr &e, bool form, uint32_t *fs) {
        ProgRead r;
        if (!read_program(w, p, w.size(), pf, form, r)) return;
        for (uint32_t i = 0; i < r.np + r.nm; ++i) add(e, src[r.src[i]], i < r.np ? 1 : -1);
        const uint32_t nps = r.sw & 15u, ns = nps + ((r.sw >> 4) & 15u);
        for (uint32_t j = 0; j < ns; ++j) add(e, slot[(r.sw >> (8 + 4 * j)) & 15u], j < nps ? 1 : -1);
        if (fs) *fs = r.form_slot;
        p = r.next;
    };
    for (uint32_t x = 0; x < a.n_nodes; ++x) {
        size_t p = w[a.o_node_off + x];
        program(p, src[a.n_in + x], false, nullptr);
    }
    // (plaintext, input) -> coefficient, per output and partial slot
    using Map = std::map<std::pair<uint32_t, uint32_t>, int64_t>;
    auto put = [](Map &m, const std::pair<uint32_t, uint32_t> &key, int64_t v) {
        if (!(m[key] += v)) m.erase(key);
    };
    std::vector<Map> out(hp.n_out), part(a.n_part);
    for (uint32_t wi = 0; wi < W; ++wi) {
        const size_t t = a.o_warp + (size_t)wi * kWarpTableWords;
        const uint32_t op0 = w[t], n_ops = w[t + 1];
        size_t sp = w[t + 2], tp = w[t + 3];
        Map job;
        for (auto &x : slot) x.clear();  // a warp's slots are its own
        for (uint32_t f = 0; f < n_ops; ++f) {
            const uint32_t op = w[op0 + f], pt = op >> kOpPtShift;
            if (op & kOpSeg) {
                for (uint32_t g = 0; g < (op & (kOpMaxSources - 1)); ++g) {
                    uint32_t sl = 0;
                    Expr u;
                    program(sp, u, true, &sl);
                    slot[sl] = std::move(u);
                }
                Expr e;
                program(sp, e, false, nullptr);
                for (auto &x : e) put(job, {pt, x.first}, x.second);
            } else if (!(op & kOpNop)) {
                for (auto &x : src[op & (kOpMaxSources - 1)]) put(job, {pt, x.first}, x.second);
            }
            if (op & kOpLast) {
                const uint32_t tg = w[tp++];
                Map &dst = (tg & kPartBit) ? part[tg & ~kPartBit] : out[tg];
                for (auto &x : job) put(dst, x.first, x.second);
                job.clear();
            }
        }
    }
    for (uint32_t r = 0; r < a.n_comb; ++r)
        for (uint32_t q = w[a.o_comb_off + r]; q < w[a.o_comb_off + r + 1]; ++q)
            for (auto &x : part[w[a.o_comb_parts + q]]) put(out[w[a.o_comb_out + r]], x.first, x.second);
    for (uint32_t j = 0; j < hp.n_out; ++j) {
        Map want;
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &tm = hp.terms[e];
            if (tm.kind == FIONA_TERM_RAW || tm.kind == FIONA_TERM_RAW_CONST)
                put(want, {tm.pt, tm.input}, 1);
            else if (tm.sign != 0)
                put(want, {hp.group_scale_pt[tm.group], tm.input}, tm.sign);
        }
        if (want != out[j]) return "an output differs from the plan's terms";
    }
    return nullptr;
}

}  // namespace

// kernel_tiled.cu
// (kernel_tiled.cu; off: the variant whose signed-sum programs are in the offset form)
int tiled_configure_kernel(int C, bool narrow, uint32_t P, bool kc, bool tc, size_t smem, bool off = false,
                           bool w12 = false, bool ka = false);
int tiled_kernel_attributes(int C, bool narrow, uint32_t P, bool kc, bool tc, cudaFuncAttributes *attr,
                            bool off = false, bool w12 = false, bool ka = false);
// kernel_ws.cu
int ws_kernel_attributes(bool narrow, uint32_t P, bool kc, uint32_t W, uint32_t D, cudaFuncAttributes *attr);
int ws_configure_kernel(bool narrow, uint32_t P, bool kc, uint32_t W, uint32_t D, size_t smem);

namespace {

// Lowering for the warp-specialised kernel (kernel_ws.cu): two coefficients
// per lane, W consumer warps plus a stager warp, one or two source regions,
// a ring of D groups of P plaintext slots per consumer warp.  The shape: the
// most consumer warps per SM (up to 16), then the most plaintext bytes in
// flight per SM (up to 64 KB, where HBM reads saturate), then two source
// regions, then deeper rings.  Tuning override FIONA_WS_SHAPE="W,regions,D".
int lower_ws(fiona_plan *p, const NodeInfo &ni, const std::vector<OutWork> &groups, uint32_t budget,
             uint32_t mac_budget, bool narrow, bool has_const, bool device)
{
    const HostPlan &hp = p->hp;
    const fiona_ctx *ctx = p->ctx;
    constexpr uint32_t P = 4, T = 64, TB = T * 8, PB = 2 * TB;
    if (ctx->N % T) return set_error(FIONA_ERR_ARG, "ws kernel: N is not a multiple of %u", T);
    const Costs k = costs_for(2, narrow);
    const std::vector<uint32_t> no_rank;
    const Lowered lw = resolve(hp, ni, groups, no_rank, 0, budget);  // shared sums expanded
    const size_t per_sm = 228 * 1024;
    int fw = 0, fb = 0, fd = 0;
    const char *env = getenv("FIONA_WS_SHAPE");
    const bool forced = env && sscanf(env, "%d,%d,%d", &fw, &fb, &fd) == 3;
    struct Pick {
        uint32_t W = 0, nbuf = 0, D = 0, ctas = 0;
        size_t smem = 0;
        std::tuple<uint32_t, uint32_t, uint32_t, uint32_t> key{};
    } best;
    for (uint32_t W : {16u, 15u, 12u, 8u, 4u})
        for (uint32_t D : {4u, 3u}) {
            cudaFuncAttributes attr{};
            if (!device) {
                attr.numRegs = W > 15 ? 96 : 128;
                attr.sharedSizeBytes = 128;
            } else if (ws_kernel_attributes(narrow, P, has_const, W, D, &attr) != FIONA_OK) {
                continue;
            }
            const size_t smem_cap = (ctx->smem_optin ? ctx->smem_optin : 227 * 1024) - attr.sharedSizeBytes - 64;
            const uint32_t regs = (std::max(attr.numRegs, 1) + 7) & ~7;
            for (uint32_t nbuf : {2u, 1u}) {
                if (forced && (W != (uint32_t)fw || nbuf != (uint32_t)fb || D != (uint32_t)fd)) continue;
                const JobPlan jp = build_jobs(lw.work, W, k, P);
                const Sched sc = encode(jp, lw.level_off, lw.nodes, W, mac_budget, hp.n_in, P);
                const uint32_t src_bytes = (hp.n_in + 1) * PB;
                const WsLayout lay((uint32_t)sc.w.size() * 4, nbuf, src_bytes, jp.n_part, W, D, P, TB, 0);
                if (lay.total > smem_cap) continue;
                const uint32_t threads = (W + 1) * 32;
                const uint32_t warps_alloc = (threads / 32 + 3) & ~3u;  // registers go to warps in fours
                const uint32_t ctas = std::min({(uint32_t)(per_sm / (lay.total + attr.sharedSizeBytes + 1024)),
                                                65536u / (warps_alloc * 32 * regs), 2048u / threads});
                if (!ctas) continue;
                const uint32_t ring = std::min<uint32_t>(ctas * W * (D - 1) * P * TB, 64 * 1024);
                const auto key = std::make_tuple(std::min(ctas * W, 16u), ring, nbuf, D);
                if (best.W == 0 || key > best.key) best = {W, nbuf, D, ctas, lay.total, key};
            }
        }
    if (!best.W) return set_error(FIONA_ERR_ARG, "ws kernel: the input tiles do not fit in shared memory");
    const JobPlan jp = build_jobs(lw.work, best.W, k, P);
    const Sched sc = encode(jp, lw.level_off, lw.nodes, best.W, mac_budget, hp.n_in, P);

    TiledSchedule *ts = new (std::nothrow) TiledSchedule;
    if (!ts) return set_error(FIONA_ERR_NOMEM, "ws schedule: host allocation");
    ts->ws = true;
    ts->C = 2;
    ts->narrow = narrow;
    ts->warps = best.W;
    ts->tile = T;
    ts->batch = P;
    ts->has_const = has_const;
    ts->smem = best.smem;
    ts->ctas_per_sm = best.ctas;
    ts->nodes_kept = 0;
    ts->nodes_expanded = (uint32_t)ni.ids.size();
    ts->ring = best.D;
    WsArgs &a = ts->ws_args;
    a.limbs = ctx->d_limbs;
    a.err = ctx->d_kerr;
    a.wait_ns = 2000000000ull;
    a.smem_sched_bytes = (uint32_t)sc.w.size() * 4;
    a.o_warp = sc.o_warp;
    a.o_comb_off = sc.o_comb_off;
    a.o_comb_out = sc.o_comb_out;
    a.o_comb_parts = sc.o_comb_parts;
    a.N = ctx->N;
    a.L = ctx->L;
    a.pt_stride = ctx->L * ctx->N;
    a.tiles_per_limb = ctx->N / T;
    a.n_in = hp.n_in;
    a.n_part = jp.n_part;
    a.n_comb = (uint32_t)jp.comb_out.size();
    a.src_bytes = (hp.n_in + 1) * PB;
    a.n_boxes = (2 * hp.n_in + 255) / 256;
    a.box_rows = a.n_boxes ? (2 * hp.n_in + a.n_boxes - 1) / a.n_boxes : 0;
    a.n_buf = best.nbuf;
    a.has_pt = hp.n_pt ? 1 : 0;
    a.flags = 0;
    if (const char *t = getenv("FIONA_TEST_WS_TIMEOUT")) {  // test only: a wait that runs out
        if (atoi(t) > 0) {
            a.flags |= kWsFlagExtraTx;
            a.wait_ns = 2000000ull;
        }
    }
    // the schedule checks of the tiled kernel, on a mirror of its arguments
    TiledArgs m{};
    m.sched_bytes = (uint32_t)(sc.w.size() * 4);
    m.o_level = sc.o_level;
    m.o_node_off = sc.o_node_off;
    m.o_warp = sc.o_warp;
    m.o_comb_off = sc.o_comb_off;
    m.o_comb_out = sc.o_comb_out;
    m.o_comb_parts = sc.o_comb_parts;
    m.n_in = hp.n_in;
    m.n_part = jp.n_part;
    m.n_comb = a.n_comb;
    m.src_bytes = a.src_bytes;
    m.box_rows = a.box_rows;
    m.n_boxes = a.n_boxes;
    const char *why = check_schedule(sc.w, m, best.W, hp.n_out, hp.n_pt, (size_t)1 << 30, PB, P);
    ts->addsub = count_addsub(sc.w, m, best.W);
    if (!why) why = check_linear_map(sc.w, m, best.W, hp);
    if (why) {
        delete ts;
        return set_error(FIONA_ERR_INTERNAL, "ws schedule check failed: %s", why);
    }
    if (device) {
        int rc = ws_configure_kernel(narrow, P, has_const, best.W, best.D, ts->smem);
        if (rc == FIONA_OK) rc = upload_blob(ts, sc.w);
        if (rc != FIONA_OK) {
            cudaFree(ts->sched.blob);
            delete ts;
            return rc;
        }
        a.sched = (const uint32_t *)ts->sched.blob;
    }
    p->tiled = ts;
    return FIONA_OK;
}

}  // namespace

int lower_tiled(fiona_plan *p)
{
    const HostPlan &hp = p->hp;
    const fiona_ctx *ctx = p->ctx;
    const bool narrow = ctx->q_max < (1ull << 52);
    const bool device = ctx->device != FIONA_DEVICE_NONE;
    // lazy-sum bound in words: 64 split words (rns.cuh), or
    // floor((2^64-1)/(q-1)) canonical residues
    const uint32_t budget = narrow ? 64u : std::min<uint32_t>(p->signed_budget, 1u << 14);
    const uint32_t mac_budget = narrow ? 1023u : p->mac_budget;  // rns.cuh: kNarrowMacBudget

    if (hp.n_pt >= kOpMaxPlaintexts)
        return set_error(FIONA_ERR_ARG, "tiled kernel: more than %u plaintexts", kOpMaxPlaintexts - 1);
    if (hp.n_in >= kOpMaxSources)
        return set_error(FIONA_ERR_ARG, "tiled kernel: more than %u inputs", kOpMaxSources - 1);

    // -- shared sums reachable from a use
    NodeInfo ni;
    std::vector<uint8_t> need(hp.n_nodes, 0);
    for (uint32_t u = 0; u < hp.n_uses; ++u) need[hp.uses[u].node] = 1;
    for (int k = (int)hp.n_nodes - 1; k >= 0; --k) {
        if (!need[k]) continue;
        for (uint32_t c = hp.node_offsets[k]; c < hp.node_offsets[k + 1]; ++c)
            if (hp.children[c].is_node) need[hp.children[c].ref] = 1;
    }
    ni.kids.resize(hp.n_nodes);
    ni.benefit.assign(hp.n_nodes, 0);
    std::vector<uint32_t> refs(hp.n_nodes, 0);
    for (uint32_t u = 0; u < hp.n_uses; ++u) ++refs[hp.uses[u].node];
    for (uint32_t k = 0; k < hp.n_nodes; ++k) {
        if (!need[k]) continue;
        ni.ids.push_back(k);
        for (uint32_t c = hp.node_offsets[k]; c < hp.node_offsets[k + 1]; ++c) {
            const fiona_sum_child &ch = hp.children[c];
            ni.kids[k].push_back({ch.is_node ? (kNodeTag | ch.ref) : ch.ref, ch.sign < 0 ? -1 : 1});
            if (ch.is_node) ++refs[ch.ref];
        }
    }
    // a kept sum of m operands referenced r times saves about (r - 1) * (m - 1) additions
    for (uint32_t k : ni.ids)
        ni.benefit[k] = ((double)refs[k] - 1.0) * ((double)ni.kids[k].size() - 1.0);
    std::vector<uint32_t> rank = ni.ids;
    std::stable_sort(rank.begin(), rank.end(), [&](uint32_t a, uint32_t b) { return ni.benefit[a] > ni.benefit[b]; });
    while (!rank.empty() && ni.benefit[rank.back()] <= 0) rank.pop_back();

    // -- per-output operand lists (unresolved: tagged shared sums), raw terms
    std::vector<OutWork> groups(hp.n_out);
    for (uint32_t j = 0; j < hp.n_out; ++j) {
        std::vector<uint32_t> gl;
        for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
            const fiona_term &t = hp.terms[e];
            if (t.kind == FIONA_TERM_RAW || t.kind == FIONA_TERM_RAW_CONST)
                groups[j].raws.push_back({t.input | (t.kind == FIONA_TERM_RAW_CONST ? kOpConst : 0u), t.pt});
            else if (t.sign != 0 && std::find(gl.begin(), gl.end(), t.group) == gl.end())
                gl.push_back(t.group);
        }
        for (uint32_t g : gl) {
            Seg sg;
            sg.scale_pt = hp.group_scale_pt[g];
            for (uint32_t e = hp.term_offsets[j]; e < hp.term_offsets[j + 1]; ++e) {
                const fiona_term &t = hp.terms[e];
                if (t.kind == FIONA_TERM_TERNARY && t.group == g && t.sign != 0 && hp.term_use[e] < 0)
                    (t.sign < 0 ? sg.minus : sg.plus).push_back(t.input);
            }
            for (uint32_t u = 0; u < hp.n_uses; ++u)
                if (hp.uses[u].output == j && hp.uses[u].group == g)
                    (hp.uses[u].sign < 0 ? sg.minus : sg.plus).push_back(kNodeTag | hp.uses[u].node);
            groups[j].segs.push_back(std::move(sg));
        }
    }

    // -- the warp-specialised kernel (FIONA_TILED_WS=1)
    if (const char *env = getenv("FIONA_TILED_WS"))
        if (atoi(env) > 0) {
            bool has_const = false;
            for (const fiona_term &t : hp.terms) has_const |= t.kind == FIONA_TERM_RAW_CONST;
            return lower_ws(p, ni, groups, budget, mac_budget, narrow, has_const, device);
        }

    // -- forming shared sums once per tile is a phase of its own (a barrier per
    //    DAG level, no plaintext traffic issued meanwhile): measured on the ViT
    //    and BERT layers it costs more than the additions it saves (9% of the
    //    signed operands with the generated sums, 12-17% with the compiled
    //    ones; VGG's compiled sums, 27%, gain under 1%), so sums are formed
    //    only when they save at least 30%; otherwise every use is expanded
    //    (the same residues).  A tuning override with a fourth field keeps
    //    the sums in play.
    bool force_keep = false;
    if (const char *env = getenv("FIONA_TILED_SHAPE")) {
        int c = 0, w = 0, d = 0, keep = -1;
        force_keep = sscanf(env, "%d,%d,%d,%d", &c, &w, &d, &keep) == 4 && keep >= 0;
    }
    if (!rank.empty() && !force_keep) {
        const Lowered flat = resolve(hp, ni, groups, rank, 0, budget);
        double opnds = 0, save = 0;
        for (auto &w : flat.work)
            for (auto &sg : w.segs) opnds += (double)(sg.plus.size() + sg.minus.size());
        for (uint32_t k : rank) save += ni.benefit[k];
        if (save < 0.30 * opnds) rank.clear();
    }

    // -- outputs sharing signed sums, to be placed on one warp each
    Sharing sharing;
    sharing.users.resize(hp.n_nodes);
    sharing.benefit = ni.benefit;
    for (uint32_t j = 0; j < hp.n_out; ++j)
        for (const Seg &g : groups[j].segs)
            for (const auto *l : {&g.plus, &g.minus})
                for (uint32_t o : *l)
                    if (o & kNodeTag) {
                        auto &us = sharing.users[o & ~kNodeTag];
                        if (us.empty() || us.back() != j) us.push_back(j);
                    }
    const Sharing *sh = ni.ids.empty() ? nullptr : &sharing;

    // -- shape search
    const size_t smem_cap = (ctx->smem_optin ? ctx->smem_optin : 227 * 1024) - 256;
    const size_t per_sm = 228 * 1024;
    const uint32_t sms = ctx->sm_count > 0 ? (uint32_t)ctx->sm_count : 152;
    struct Shape {
        int C = 0;
        uint32_t W = 0, P = 8;
        double pad = 0;               // share of padding operations
        bool dbl = false;
        bool w12 = false;             // the variant for CTAs of at most 12 warps
        double balance = 0;           // mean warp cost / largest warp cost
        uint32_t keep = 0, ctas = 0;  // shared sums requested (top of the ranking)
        size_t smem = 0;
        double est = 0;
    };
    // plans with constant plaintexts run the kernel variant that reads them
    bool has_const = false;
    for (const fiona_term &t : hp.terms) has_const |= t.kind == FIONA_TERM_RAW_CONST;
    std::vector<Shape> shapes;
    for (int C : {2, 1})
    for (uint32_t batch : {16u, 8u, 4u}) {
        if (ctx->N % (32u * C)) continue;
        if (batch == 16 && C != 1) continue;  // the kernels with 16 plaintexts in flight per lane
        const uint32_t T = 32u * C, PB = 2 * T * 8;
        const Costs k = costs_for(C, narrow);
        cudaFuncAttributes attr{};
        if (!device) {  // lowering without a GPU: the build's usual figures
            attr.numRegs = 128;
            attr.sharedSizeBytes = 64;
        } else if (tiled_kernel_attributes(C, narrow, batch, has_const, false, &attr) != FIONA_OK) {
            continue;
        }
        // the variant for CTAs of at most 12 warps (two coefficients per
        // lane, narrow moduli, batches of 8): more registers a thread
        cudaFuncAttributes attr12{};
        bool has12 = C == 2 && batch == 8 && narrow;
        if (has12 && !device) {
            attr12.numRegs = 168;
            attr12.sharedSizeBytes = 64;
        } else if (has12) {
            has12 = tiled_kernel_attributes(C, narrow, batch, has_const, false, &attr12, false, true) == FIONA_OK;
        }
        for (uint32_t W : {16u, 12u, 8u, 4u, 2u, 1u}) {
            const bool w12 = has12 && W <= 12;
            const uint32_t regs = (std::max(w12 ? attr12.numRegs : attr.numRegs, 1) + 7) & ~7;
            // one or two warps only when the tuning override asks for them
            if (W < 4) {
                const char *env = getenv("FIONA_TILED_SHAPE");
                int fc = 0, fw = 0;
                if (!env || sscanf(env, "%d,%d", &fc, &fw) != 2 || fw != (int)W) continue;
            }
            for (bool dbl : {true, false}) {
                if (dbl && hp.n_in == 0) continue;
                const uint32_t nbuf = dbl ? 2 : 1;
                // most shared sums that fit: smem grows with each kept sum
                auto smem_for = [&](uint32_t keep, Lowered &lw, JobPlan &jp, Sched &sc) {
                    lw = resolve(hp, ni, groups, rank, keep, budget);
                    jp = build_jobs(lw.work, W, k, batch, keep ? nullptr : sh);
                    sc = encode(jp, lw.level_off, lw.nodes, W, mac_budget, hp.n_in + (uint32_t)lw.nodes.size(),
                                batch);
                    const uint32_t n_src = hp.n_in + (uint32_t)lw.nodes.size() + 1;  // + the zero tile
                    if (n_src > kOpMaxSources) return (size_t)-1;
                    return sc.w.size() * 4 + (size_t)n_src * PB * nbuf + (size_t)jp.n_part * PB + 32 +
                           attr.sharedSizeBytes;
                };
                Lowered lw;
                JobPlan jp;
                Sched sc;
                uint32_t lo = 0, hi = (uint32_t)rank.size();
                if (smem_for(0, lw, jp, sc) > smem_cap) continue;
                if (smem_for(hi, lw, jp, sc) > smem_cap) {
                    while (lo + 1 < hi) {  // smem_for(lo) fits, smem_for(hi) does not
                        const uint32_t mid = (lo + hi) / 2;
                        if (smem_for(mid, lw, jp, sc) <= smem_cap) lo = mid;
                        else hi = mid;
                    }
                    hi = lo;
                }
                const size_t smem = smem_for(hi, lw, jp, sc);
                const uint32_t by_smem = (uint32_t)(per_sm / (smem + 1024));
                const uint32_t by_threads = 2048 / (W * 32);
                const uint32_t by_regs = 65536 / (W * 32 * regs);
                const uint32_t ctas = std::min({by_smem, by_threads, by_regs, 32u});
                if (!ctas) continue;
                // per-tile demand of one CTA (cycles of the resource it uses)
                double issue = 0, imad = 0, lds = 0, slowest = 0;
                for (uint32_t wi = 0; wi < W; ++wi) {
                    double c = 0;
                    for (const Job &jb : jp.per_warp[wi]) {
                        c += work_cost(jb.w, k, batch);
                        const double prods = (double)(jb.w.raws.size() + jb.w.segs.size());
                        imad += prods * k.imad_op;
                        double opnds = (double)jb.w.raws.size();
                        for (auto &s : jb.w.segs) opnds += (double)(s.plus.size() + s.minus.size());
                        lds += opnds * k.smem_operand / 128.0;
                    }
                    issue += c;
                    slowest = std::max(slowest, c);
                }
                double node_ops = 0;
                for (auto &s : lw.nodes) node_ops += k.seg + k.operand * (double)(s.plus.size() + s.minus.size());
                const double hbm_bytes = (double)(sc.pt_ops + 2ull * hp.n_in + 2ull * hp.n_out) * T * 8;
                const double hbm = hbm_bytes / 22.0;  // about 22 bytes per SM cycle at the measured copy rate
                const double shared = std::max({issue / 4.0, imad, lds, hbm});
                const double serial = slowest * 2.5 + node_ops / W * 2.5 + 150.0 * (lw.n_levels + 2) +
                                      (dbl ? 0.0 : 1500.0 + (double)hp.n_in * PB / 64.0);
                const double tiles = (double)ctx->N / T * ctx->L;
                const double rounds = std::ceil(tiles / ((double)sms * ctas));
                const double per_round = std::max(ctas * shared, serial + (ctas == 1 ? 0.25 * shared : 0.0));
                Shape s;
                s.C = C;
                s.W = W;
                s.P = batch;
                size_t n_ops = 0;
                for (uint32_t wi = 0; wi < W; ++wi) n_ops += sc.w[sc.o_warp + wi * kWarpTableWords + 1];
                s.pad = n_ops ? 1.0 - (double)sc.pt_ops / (double)n_ops : 0.0;
                s.dbl = dbl;
                s.w12 = w12;
                s.balance = slowest > 0 ? issue / W / slowest : 1.0;
                s.keep = hi;
                s.ctas = ctas;
                s.smem = smem - attr.sharedSizeBytes;
                s.est = rounds * per_round;
                shapes.push_back(s);
                if (getenv("FIONA_TILED_DEBUG"))
                    fprintf(stderr,
                            "C=%d P=%u W=%u dbl=%d w12=%d keep=%u sched=%zu parts=%u smem=%zu ctas=%u pad=%.2f est=%.0f\n",
                            C, batch, W, (int)dbl, (int)w12, s.keep, sc.w.size() * 4, jp.n_part, smem, ctas, s.pad,
                            s.est);
            }
        }
    }
    if (shapes.empty()) return set_error(FIONA_ERR_ARG, "tiled kernel: the input tiles do not fit in shared memory");
    // Ranking (from shape sweeps of the layer workloads): a second source
    // region first (the next tile's inputs arrive during this one), then
    // resident warps up to 16 per SM (12 warps of the 12-warp variant count
    // as 16: their deeper plaintext queues keep as many HBM reads in flight
    // as 16 warps with 4), then 2 coefficients per lane (half the
    // per-operation overhead per coefficient), then more CTAs per SM (their
    // per-tile phases overlap), then, with 2 coefficients per lane, the
    // 12-warp variant with batches of 8, batches of 4, and of 8, and with
    // one, batches of 16, then 8 (measured: BERT, one CTA per SM, 5.998 ms
    // with 12 warps x 8 against 6.049 ms with 16 x 4; ViT faster with two
    // CTAs of 8 warps x 4; VGG with 16, its deeper plaintext queue keeping
    // more HBM reads in flight), then the cost estimate.
    auto key = [](const Shape &s) {
        // (the 12-warp variant only where its warps are as evenly loaded as
        // 16 would be: measured on the first 72 inputs of the VGG layer, 16
        // outputs on 12 warps, it ran 1.69 ms against 1.47 ms for 16 x 4)
        const bool deep = s.w12 && s.W == 12 && s.P == 8 && s.balance >= 0.95;
        const int pref = s.C == 2 ? (deep ? 3 : s.P == 4 ? 2 : 1) : (s.P == 16 ? 2 : s.P == 8 ? 1 : 0);
        const uint32_t resident = deep ? 16 : std::min<uint32_t>(s.ctas * s.W, 16);
        return std::make_tuple(s.dbl ? 1 : 0, resident, s.C, s.ctas, pref, -s.est);
    };
    Shape best = *std::max_element(shapes.begin(), shapes.end(),
                                   [&](const Shape &a, const Shape &b) { return key(a) < key(b); });
    // tuning override "C,W,double[,most shared sums kept[,P]]": every shape
    // computes the same residues
    if (const char *env = getenv("FIONA_TILED_SHAPE")) {
        int c = 0, w = 0, d = 0, keep = -1, pb = 8;
        const int n = sscanf(env, "%d,%d,%d,%d,%d", &c, &w, &d, &keep, &pb);
        if (n >= 3)
            for (auto &s : shapes)
                if (s.C == c && s.W == (uint32_t)w && s.dbl == (d != 0) && s.P == (uint32_t)pb) {
                    best = s;
                    if (n >= 4 && keep >= 0) best.keep = std::min(best.keep, (uint32_t)keep);
                }
    }
    const uint32_t T = 32u * best.C, PB = 2 * T * 8;
    const Costs k = costs_for(best.C, narrow);
    const uint32_t nbuf = best.dbl ? 2 : 1;
    Lowered lw;
    JobPlan jp;
    LocalResult loc;
    Sched sc;
    // -- the scale groups' signed sums as one tensor-core contraction per
    //    tile (one coefficient per lane, every q < 2^50, batches of 16, warps
    //    in fours: one per tensor-memory quarter), when its sources, W and
    //    the schedule fit and FIONA_TILED_TC=1 asks for it.  Not the default:
    //    measured on the VGG layer, the contraction's phase (conversion to
    //    fp16 chunks 3.3k cycles a tile, 45 dependent MMAs 4.3k, epilogue
    //    1.8k) costs more than the shared-memory sums it replaces, which
    //    overlap the plaintext loads (3.45 against 2.34 ms a launch)
    bool use_tc = false;
    TcPlan tc;
    uint32_t o_tcw = 0, o_tcm = 0;
    {
        const char *env = getenv("FIONA_TILED_TC");
        const bool allow = env && atoi(env) != 0;
        if (allow && !force_keep && best.C == 1 && narrow && best.P == 16 && best.W % 4 == 0 &&
            ctx->q_max < (1ull << 50))
            tc = plan_tc(hp, ni, groups, ctx->q_max);
        cudaFuncAttributes attr{};
        if (!device) {
            attr.numRegs = 128;
            attr.sharedSizeBytes = 64;
        } else if (tc.ok && tiled_kernel_attributes(1, true, best.P, has_const, true, &attr) != FIONA_OK) {
            tc.ok = false;
        }
        if (tc.ok) {
            const uint32_t ng = (uint32_t)tc.nodes.size();
            Lowered lt;
            lt.work = tc.work;
            lt.nodes = tc.nodes;
            lt.level_off = {0, ng};
            lt.n_levels = 1;
            JobPlan jt = build_jobs(lt.work, best.W, k, best.P, nullptr);
            Sched st = encode(jt, lt.level_off, lt.nodes, best.W, mac_budget, hp.n_in + ng, best.P);
            append_tc(st.w, tc, hp.n_in, o_tcw, o_tcm);
            const size_t smem = st.w.size() * 4 + (size_t)(hp.n_in + ng + 1) * PB * nbuf + (size_t)jt.n_part * PB + 32;
            const uint32_t regs = (std::max(attr.numRegs, 1) + 7) & ~7;
            const uint32_t ctas = std::min({(uint32_t)(per_sm / (smem + attr.sharedSizeBytes + 1024)),
                                            2048 / (best.W * 32), 65536 / (best.W * 32 * regs), 512 / tc.cols});
            if (getenv("FIONA_TILED_DEBUG"))
                fprintf(stderr, "tensor-core sums: groups=%u K=%u N=%u cols=%u smem=%zu ctas=%u\n", ng, tc.K, tc.N,
                        tc.cols, smem, ctas);
            if (smem + attr.sharedSizeBytes <= smem_cap && ctas >= 1) {
                use_tc = true;
                lw = std::move(lt);
                jp = std::move(jt);
                sc = std::move(st);
                best.ctas = ctas;
            }
        }
    }
    if (!use_tc) {
    lw = resolve(hp, ni, groups, rank, best.keep, budget);
    jp = build_jobs(lw.work, best.W, k, best.P, best.keep ? nullptr : sh);
    // shared sums formed by the warps that use them, when no sum is formed
    // for the whole block and the warps' slots fit in shared memory
    // (a tuning override with a fourth field selects the block-level sums instead)
    if (!best.keep && sh && !force_keep && !getenv("FIONA_NO_WARP_SUMS")) {
        for (uint32_t max_slots = 8; max_slots >= 1; max_slots /= 2) {
            JobPlan jt = jp;
            LocalResult r = localize(jt, groups, ni, budget, max_slots);
            Sched st = encode(jt, lw.level_off, lw.nodes, best.W, mac_budget, hp.n_in, best.P, &r.warp_slots);
            // when some warps have more operation slots than others, those
            // set the tile's length: a formation there (its run sums,
            // reduction and store before the batch that needs it) lengthens
            // every tile, so those warps keep their groups expanded (measured
            // on the ViT layer: 0.943 ms with two of its four formations on
            // such warps, 0.906 ms with none formed)
            std::vector<uint32_t> crit;
            if (r.formed && !getenv("FIONA_WARP_SUMS_ANYWHERE")) {
                uint32_t most = 0, least = ~0u;
                for (uint32_t wi = 0; wi < best.W; ++wi) {
                    most = std::max(most, st.w[st.o_warp + wi * kWarpTableWords + 1]);
                    least = std::min(least, st.w[st.o_warp + wi * kWarpTableWords + 1]);
                }
                for (uint32_t wi = 0; wi < best.W && least < most; ++wi)
                    if (r.warp_slots[wi] && st.w[st.o_warp + wi * kWarpTableWords + 1] == most) crit.push_back(wi);
                if (!crit.empty()) {
                    for (uint32_t wi : crit) {  // this warp keeps its expanded groups
                        jt.per_warp[wi] = jp.per_warp[wi];
                        r.n_slots -= r.warp_slots[wi];
                        r.warp_slots[wi] = 0;
                    }
                    r.formed = 0;
                    for (uint32_t wi = 0; wi < best.W; ++wi) r.formed += r.warp_slots[wi] ? 1 : 0;
                    st = encode(jt, lw.level_off, lw.nodes, best.W, mac_budget, hp.n_in, best.P, &r.warp_slots);
                }
            }
            const size_t sm = st.w.size() * 4 + (size_t)(hp.n_in + 1) * PB * (best.dbl ? 2 : 1) +
                              (size_t)jt.n_part * PB + (size_t)r.n_slots * PB + 32;
            if (getenv("FIONA_TILED_DEBUG"))
                fprintf(stderr, "warp sums: max_slots=%u formed=%u slots=%u smem=%zu cap=%zu\n", max_slots, r.formed,
                        r.n_slots, sm, smem_cap);
            if (!r.formed) break;
            // warps whose slots do not fit give up theirs (largest first)
            size_t over = sm > smem_cap - 64 ? sm - (smem_cap - 64) : 0;
            const size_t per_cta = per_sm / std::max(best.ctas, 1u);
            if (sm + 1024 > per_cta) over = std::max(over, sm + 1024 - per_cta);
            if (over && max_slots > 1) continue;
            if (over) {  // one slot a warp: drop warps until the rest fit
                std::vector<uint32_t> keep_w(best.W, 1);
                size_t freed = 0;
                for (uint32_t wi = 0; wi < best.W && freed < over; ++wi)
                    if (r.warp_slots[wi]) {
                        keep_w[wi] = 0;
                        freed += PB;
                    }
                if (freed < over) break;
                JobPlan jk = jp;
                std::vector<std::vector<Job>> saved = jk.per_warp;
                r = localize(jk, groups, ni, budget, 1);
                for (uint32_t wi : crit) keep_w[wi] = 0;
                for (uint32_t wi = 0; wi < best.W; ++wi)
                    if (!keep_w[wi]) {  // this warp keeps its expanded groups
                        jk.per_warp[wi] = saved[wi];
                        r.n_slots -= r.warp_slots[wi];
                        r.warp_slots[wi] = 0;
                    }
                r.formed = 0;  // recount from the schedule below
                jt = std::move(jk);
            }
            jp = std::move(jt);
            loc = r;
            break;
        }
    }
    sc = encode(jp, lw.level_off, lw.nodes, best.W, mac_budget, hp.n_in + (uint32_t)lw.nodes.size(), best.P,
                loc.warp_slots.empty() ? nullptr : &loc.warp_slots);
    if (!loc.warp_slots.empty()) {  // sums formed per tile, from the schedule's formations
        loc.formed = 0;
        for (uint32_t wi = 0; wi < best.W; ++wi) {
            const uint32_t op0 = sc.w[sc.o_warp + wi * kWarpTableWords];
            const uint32_t n = sc.w[sc.o_warp + wi * kWarpTableWords + 1];
            for (uint32_t f = 0; f < n; ++f)
                if (sc.w[op0 + f] & kOpSeg) loc.formed += sc.w[op0 + f] & (kOpMaxSources - 1);
        }
    }
    }  // !use_tc
    auto smem_of = [&](const Sched &x) {
        return x.w.size() * 4 + (size_t)(hp.n_in + lw.nodes.size() + 1) * PB * nbuf + (size_t)jp.n_part * PB +
               (size_t)loc.n_slots * PB + 32;
    };
    // the signed-sum programs in the offset form (the kernel forms each
    // source address with one addition: measured on the VGG layer, whose
    // 1638 signed terms per tile dominate its index decoding), when the
    // larger schedule still fits beside the regions and slots at the
    // occupancy the shape was chosen for; otherwise (BERT, whose two source
    // regions fill the shared memory) the packed indices.  FIONA_TILED_PACKED=1
    // keeps the packed form (the same residues).
    // every raw plaintext constant (the bert-const layers): the 12-warp
    // shape has a kernel variant that reads every operation after a batch's
    // first as constant, without a per-operation test (a SEG only opens a
    // batch).  FIONA_TILED_KC_MIXED=1 keeps the per-operation test.
    bool kc_all = false;
    if (has_const && best.w12 && !use_tc && !(getenv("FIONA_TILED_KC_MIXED") && atoi(getenv("FIONA_TILED_KC_MIXED")) > 0)) {
        kc_all = true;
        for (const fiona_term &t : hp.terms) kc_all &= t.kind != FIONA_TERM_RAW;
    }
    bool offsets = false;
    if (!use_tc && !(getenv("FIONA_TILED_PACKED") && atoi(getenv("FIONA_TILED_PACKED")) > 0)) {
        const Sched so = encode(jp, lw.level_off, lw.nodes, best.W, mac_budget, hp.n_in + (uint32_t)lw.nodes.size(),
                                best.P, loc.warp_slots.empty() ? nullptr : &loc.warp_slots, ProgForm{true, PB});
        const size_t sm_off = smem_of(so);
        // (and only when that kernel variant spills no more than the packed one)
        cudaFuncAttributes attr{}, packed{};
        bool ok = true;
        if (!device) {
            attr.numRegs = 128;
            attr.sharedSizeBytes = 64;
        } else {
            ok = tiled_kernel_attributes(best.C, narrow, best.P, has_const, false, &attr, true, best.w12, kc_all) ==
                     FIONA_OK &&
                 tiled_kernel_attributes(best.C, narrow, best.P, has_const, false, &packed, false, best.w12, kc_all) ==
                     FIONA_OK &&
                 attr.localSizeBytes <= packed.localSizeBytes;
        }
        const uint32_t regs = (std::max(attr.numRegs, 1) + 7) & ~7;
        if (getenv("FIONA_TILED_DEBUG"))
            fprintf(stderr, "offset form: ok=%d smem=%zu+%zu cap=%zu per_sm=%zu ctas=%u regs=%u local=%zu/%zu\n",
                    (int)ok, sm_off, (size_t)attr.sharedSizeBytes, smem_cap, per_sm, best.ctas, regs,
                    (size_t)attr.localSizeBytes, (size_t)packed.localSizeBytes);
        if (ok && sm_off + attr.sharedSizeBytes <= smem_cap &&
            per_sm / (sm_off + attr.sharedSizeBytes + 1024) >= std::max(best.ctas, 1u) &&
            65536 / (best.W * 32 * regs) >= std::max(best.ctas, 1u)) {
            sc = so;
            offsets = true;
        }
    }
    best.smem = smem_of(sc);
    TiledSchedule *ts = new (std::nothrow) TiledSchedule;
    if (!ts) return set_error(FIONA_ERR_NOMEM, "tiled schedule: host allocation");
    ts->C = best.C;
    ts->narrow = narrow;
    ts->warps = best.W;
    ts->tile = T;
    ts->batch = best.P;
    ts->has_const = has_const;
    ts->smem = best.smem;
    ts->ctas_per_sm = best.ctas;
    ts->tc = use_tc;
    ts->w12 = best.w12 && !use_tc;
    // (the group sums of the tensor-core variant are not shared sums: every
    // shared sum is expanded into them)
    ts->nodes_kept = use_tc ? 0 : (uint32_t)lw.nodes.size() + loc.formed;
    ts->nodes_expanded = (uint32_t)ni.ids.size() - std::min<uint32_t>((uint32_t)ni.ids.size(), ts->nodes_kept);
    TiledArgs &a = ts->args;
    a.n_slots = loc.n_slots;
    a.o_level = sc.o_level;
    a.o_node_off = sc.o_node_off;
    a.o_warp = sc.o_warp;
    a.o_comb_off = sc.o_comb_off;
    a.o_comb_out = sc.o_comb_out;
    a.o_comb_parts = sc.o_comb_parts;
    a.sched_bytes = (uint32_t)(sc.w.size() * 4);
    a.limbs = ctx->d_limbs;
    a.err = ctx->d_kerr;
    a.N = ctx->N;
    a.L = ctx->L;
    a.pt_stride = ctx->L * ctx->N;
    a.tiles_per_limb = ctx->N / T;
    a.n_in = hp.n_in;
    a.n_nodes = (uint32_t)lw.nodes.size();
    a.n_levels = lw.n_levels;
    a.n_part = jp.n_part;
    a.n_comb = (uint32_t)jp.comb_out.size();
    a.src_bytes = (hp.n_in + a.n_nodes + 1) * PB;  // + the zero tile
    a.double_buffer = best.dbl ? 1 : 0;
    // TMA boxes of at most 256 polys covering the 2 n_in input polys
    a.n_boxes = (2 * hp.n_in + 255) / 256;
    a.box_rows = a.n_boxes ? (2 * hp.n_in + a.n_boxes - 1) / a.n_boxes : 0;
    a.has_pt = hp.n_pt ? 1 : 0;
    if (use_tc) {
        a.tc_groups = (uint32_t)tc.nodes.size();
        a.tc_k = tc.K;
        a.tc_n = tc.N;
        a.tc_cols = tc.cols;
        a.tc_wabs = tc.wabs;
        a.o_tcw = o_tcw;
        a.o_tcm = o_tcm;
    }
    a.wait_ns = 2000000000ull;
    a.zero = 0;
    a.src_offsets = offsets ? 1 : 0;
    a.kc_all = kc_all ? 1 : 0;
    if (const char *t = getenv("FIONA_TEST_TILED_TIMEOUT")) {  // test only: a copy wait that runs out
        if (atoi(t) > 0 && best.C == 1 && hp.n_in) {
            a.test_flags |= kTiledFlagExtraTx;
            a.wait_ns = 2000000ull;
        }
    }
    ts->addsub = count_addsub(sc.w, a, best.W);
    if (const char *why = check_schedule(sc.w, a, best.W, hp.n_out, hp.n_pt, ts->smem, PB, best.P)) {
        delete ts;
        return set_error(FIONA_ERR_INTERNAL, "tiled schedule check failed: %s", why);
    }
    if (const char *why = check_linear_map(sc.w, a, best.W, hp)) {
        delete ts;
        return set_error(FIONA_ERR_INTERNAL, "tiled schedule check failed: %s", why);
    }
    if (const char *why = check_tc(sc.w, a)) {
        delete ts;
        return set_error(FIONA_ERR_INTERNAL, "tiled schedule check failed: %s", why);
    }
    if (device) {
        int rc = tiled_configure_kernel(best.C, narrow, best.P, has_const, use_tc, ts->smem, offsets, ts->w12, kc_all);
        if (rc == FIONA_OK) rc = upload_blob(ts, sc.w);
        if (rc != FIONA_OK) {
            cudaFree(ts->sched.blob);
            delete ts;
            return rc;
        }
        a.sched = (const uint32_t *)ts->sched.blob;
    }
    p->tiled = ts;
    return FIONA_OK;
}

void free_tiled(fiona_plan *p)
{
    if (!p->tiled) return;
    if (p->tiled->sched.blob) cudaFree(p->tiled->sched.blob);
    delete p->tiled;
    p->tiled = nullptr;
}
