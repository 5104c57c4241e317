// plan_compile.cpp -- the host plan compiler: from a dense route matrix to
// the arrays of fiona_plan_create (Sec. 4.2 "Exact Compilation of Routed
// Linear Operators").
//
// * Terms: one per (output, input) pair, in input order (Sec. 4.2: every
//   pair is one execution group g_{j,i}).
// * Grouping Reconstruction Operations: the signed terms of one output that
//   use the same reconstruction-factor plaintext form one scale group, so
//   their signed sum takes one PMult.
// * Sharing Signed Sums: for every pair of scale groups of different
//   outputs, the signed terms they have in common -- the same inputs with
//   the same signs, or with all signs reversed -- are a candidate sum.  For a
//   candidate of m inputs usable by k groups the saving is estimated as
//   km - m - k (the paper's conservative count), or as the exact
//   (k - 1)(m - 1) when FIONA_COMPILE_SHARE_EXACT is set.  Candidates are
//   taken greedily, largest estimate first, while the estimate over the
//   groups still free to use them stays positive; a group takes at most one
//   of any two overlapping candidates (a term is covered once at most).
#include <algorithm>
#include <map>
#include <vector>

#include "fiona_internal.h"

namespace {

struct Cand {
    std::vector<std::pair<uint32_t, int8_t>> t;  // (input, sign), inputs ascending, first sign +1
    bool operator<(const Cand &o) const { return t < o.t; }
};

Cand canonical(std::vector<std::pair<uint32_t, int8_t>> t)
{
    std::sort(t.begin(), t.end());
    if (!t.empty() && t[0].second < 0)
        for (auto &x : t) x.second = (int8_t)-x.second;
    return Cand{std::move(t)};
}

}  // namespace

extern "C" int fiona_plan_compile(uint32_t n_in, uint32_t n_out, uint32_t n_pt, const fiona_route *routes,
                                  uint32_t flags, uint32_t *term_offsets, fiona_term *terms, uint32_t *n_groups,
                                  uint32_t *group_scale_pt, uint32_t *group_output, uint32_t *n_nodes,
                                  uint32_t *node_offsets, fiona_sum_child *children, uint32_t *n_uses,
                                  fiona_sum_use *uses)
{
    if (flags & ~(uint32_t)(FIONA_COMPILE_SHARE | FIONA_COMPILE_SHARE_EXACT))
        return set_error(FIONA_ERR_ARG, "plan_compile: unknown flags 0x%x", flags);
    if (!term_offsets || !n_groups || !n_nodes || !n_uses)
        return set_error(FIONA_ERR_ARG, "plan_compile: null output argument");
    const uint64_t pairs = (uint64_t)n_in * n_out;
    if (pairs > (1u << 24)) return set_error(FIONA_ERR_ARG, "plan_compile: %llu pairs", (unsigned long long)pairs);
    if (pairs && (!routes || !terms || !group_scale_pt || !group_output || !node_offsets || !children || !uses))
        return set_error(FIONA_ERR_ARG, "plan_compile: null array");
    for (uint64_t e = 0; e < pairs; ++e) {
        const fiona_route &r = routes[e];
        if (r.reserved) return set_error(FIONA_ERR_PLAN, "plan_compile: route %llu reserved field", (unsigned long long)e);
        if (r.kind == FIONA_TERM_RAW || r.kind == FIONA_TERM_RAW_CONST) {
            if (r.sign != 0 || r.pt >= n_pt)
                return set_error(FIONA_ERR_PLAN, "plan_compile: raw route %llu malformed", (unsigned long long)e);
        } else if (r.kind == FIONA_TERM_TERNARY) {
            if (r.sign < -1 || r.sign > 1 || r.pt >= n_pt)
                return set_error(FIONA_ERR_PLAN, "plan_compile: ternary route %llu malformed", (unsigned long long)e);
        } else {
            return set_error(FIONA_ERR_PLAN, "plan_compile: route %llu kind %d", (unsigned long long)e, r.kind);
        }
    }

    // -- terms and scale groups: one group per (output, gamma plaintext)
    std::vector<uint32_t> gsp, gout;
    std::vector<int8_t> sign_of;  // [group][input]: the group's nonzero signs
    term_offsets[0] = 0;
    for (uint32_t j = 0; j < n_out; ++j) {
        std::map<uint32_t, uint32_t> by_gamma;
        for (uint32_t i = 0; i < n_in; ++i) {
            const fiona_route &r = routes[(uint64_t)j * n_in + i];
            fiona_term &t = terms[(uint64_t)j * n_in + i];
            t = fiona_term{};
            t.input = i;
            t.kind = (int8_t)r.kind;
            if (r.kind == FIONA_TERM_RAW || r.kind == FIONA_TERM_RAW_CONST) {
                t.pt = r.pt;
                continue;
            }
            auto it = by_gamma.find(r.pt);
            if (it == by_gamma.end()) {
                it = by_gamma.emplace(r.pt, (uint32_t)gsp.size()).first;
                gsp.push_back(r.pt);
                gout.push_back(j);
                sign_of.resize(sign_of.size() + n_in, 0);
            }
            t.group = it->second;
            t.sign = r.sign;
            sign_of[(size_t)t.group * n_in + i] = r.sign;
        }
        term_offsets[j + 1] = (uint32_t)((uint64_t)(j + 1) * n_in);
    }
    const uint32_t G = (uint32_t)gsp.size();
    for (uint32_t g = 0; g < G; ++g) {
        group_scale_pt[g] = gsp[g];
        group_output[g] = gout[g];
    }
    *n_groups = G;
    *n_nodes = 0;
    *n_uses = 0;
    node_offsets[0] = 0;
    if (!(flags & FIONA_COMPILE_SHARE) || G < 2) return FIONA_OK;

    // -- candidate sums: the common signed terms of two groups of different outputs
    std::vector<Cand> cands;
    {
        std::vector<Cand> all;
        for (uint32_t a = 0; a < G; ++a)
            for (uint32_t b = a + 1; b < G; ++b) {
                if (gout[a] == gout[b]) continue;
                std::vector<std::pair<uint32_t, int8_t>> same, opp;
                const int8_t *sa = &sign_of[(size_t)a * n_in], *sb = &sign_of[(size_t)b * n_in];
                for (uint32_t i = 0; i < n_in; ++i) {
                    if (!sa[i] || !sb[i]) continue;
                    (sa[i] == sb[i] ? same : opp).push_back({i, sa[i]});
                }
                if (same.size() >= 2) all.push_back(canonical(std::move(same)));
                if (opp.size() >= 2) all.push_back(canonical(std::move(opp)));
            }
        std::sort(all.begin(), all.end());
        all.erase(std::unique(all.begin(), all.end(), [](const Cand &x, const Cand &y) { return x.t == y.t; }),
                  all.end());
        cands = std::move(all);
    }
    const bool exact = flags & FIONA_COMPILE_SHARE_EXACT;
    auto estimate = [&](uint64_t m, uint64_t k) -> int64_t {
        return exact ? (int64_t)((k - 1) * (m - 1)) : (int64_t)(k * m) - (int64_t)m - (int64_t)k;
    };
    // groups that can take candidate c with sign sigma, none of its terms covered yet
    std::vector<uint8_t> covered((size_t)G * n_in, 0);
    auto users = [&](const Cand &c, std::vector<std::pair<uint32_t, int8_t>> &out) {
        out.clear();
        for (uint32_t g = 0; g < G; ++g) {
            const int8_t *sg = &sign_of[(size_t)g * n_in];
            const int8_t sigma = sg[c.t[0].first];
            if (!sigma) continue;
            bool ok = true;
            for (auto &x : c.t)
                if (sg[x.first] != sigma * x.second || covered[(size_t)g * n_in + x.first]) {
                    ok = false;
                    break;
                }
            if (ok) out.push_back({g, sigma});
        }
    };
    // initial estimates, then greedy acceptance largest first
    std::vector<std::pair<int64_t, uint32_t>> order;
    std::vector<std::pair<uint32_t, int8_t>> us;
    for (uint32_t c = 0; c < cands.size(); ++c) {
        users(cands[c], us);
        const int64_t est = estimate(cands[c].t.size(), us.size());
        if (est > 0) order.push_back({-est, c});
    }
    std::sort(order.begin(), order.end());
    uint32_t nn = 0, nc = 0, nu = 0;
    for (auto &oc : order) {
        const Cand &c = cands[oc.second];
        users(c, us);
        if (us.size() < 2 || estimate(c.t.size(), us.size()) <= 0) continue;
        for (auto &x : c.t) children[nc++] = fiona_sum_child{x.first, 0, x.second, 0};
        node_offsets[++nn] = nc;
        for (auto &u : us) {
            uses[nu++] = fiona_sum_use{gout[u.first], u.first, nn - 1, u.second, {0, 0, 0}};
            for (auto &x : c.t) covered[(size_t)u.first * n_in + x.first] = 1;
        }
    }
    *n_nodes = nn;
    *n_uses = nu;
    return FIONA_OK;
}
