// Host mask compiler: budgeted greedy selection of dependency-closed units (paper Sec. 3.3).
//
// Units of a layer are the H_kv GQA groups (a KV head with its g query heads; keeping
// the group keeps the Q/K/V rows and the O columns of those heads, which is the GQA
// closure rule of Sec. 3.3) and the df/chan_unit SwiGLU channel units (gate row, up
// row and down column kept together, the SwiGLU closure rule). Unit cost is its
// marginal active FLOPs from Eqs. flop-attn / flop-mlp. Selection is greedy by score
// per active FLOP (Sec. 3.3): exact integer ratio comparison, per-layer targets drawn
// in [r_lo, r_hi] and shifted to meet the global budget, a per-layer greedy fill,
// then a global top-up under the budget and the per-layer cap.
//
// Query-head candidates (Sec. 3.3; Table 1: 64 per 70B layer) are the finer unit: a
// query head keeps its Q rows and O columns, and the closure keeps its KV head, whose
// K and V rows are charged to the first head of the group that is accepted. The greedy
// then ranks every candidate by score over its marginal cost with the closure applied,
// which falls for the other heads of a group once its KV head is on. It runs on lazy
// max-heaps: an entry whose cost went stale is skipped, and the heads of a group are
// pushed again with their lower cost when its KV head comes on.
#include <algorithm>
#include <cmath>
#include <numeric>
#include <queue>
#include <string>

#include "tasp_internal.h"

namespace tasp {

int64_t layer_flops(const Shape& s, int64_t m_q, int64_t m_kv, int64_t c) {
    const int64_t d = s.d, dh = s.dh;
    return 2 * d * dh * (m_q + 2 * m_kv) + 2 * dh * m_q * d + 6 * d * c;
}

bool Shape::same(const Shape& o) const {
    return L == o.L && d == o.d && Hq == o.Hq && Hkv == o.Hkv && dh == o.dh && df == o.df && vocab == o.vocab &&
           cu == o.cu && eps == o.eps && theta == o.theta && seed == o.seed && qg == o.qg;
}

namespace {

constexpr int kFixBits = 24;
constexpr int64_t kFix = int64_t(1) << kFixBits;

int64_t fixed_of(double r) { return (int64_t)std::floor(r * (double)kFix + 0.5); }

struct Unit {
    int layer, idx;  // idx < Hkv: group; else channel unit idx - Hkv
    uint32_t score;
    int64_t cost;
};

// a precedes b in descending score/cost; ties: group before channel unit, lower index, lower layer
bool ratio_first(const Unit& a, const Unit& b, int n_groups, bool layer_major_ties) {
    unsigned __int128 lhs = (unsigned __int128)a.score * (uint64_t)b.cost;
    unsigned __int128 rhs = (unsigned __int128)b.score * (uint64_t)a.cost;
    if (lhs != rhs) return lhs > rhs;
    int ta = a.idx < n_groups ? 0 : 1, tb = b.idx < n_groups ? 0 : 1;
    if (layer_major_ties && a.layer != b.layer) return a.layer < b.layer;
    if (ta != tb) return ta < tb;
    if (a.idx != b.idx) return a.idx < b.idx;
    return a.layer < b.layer;
}

struct Budgets {
    std::vector<int64_t> b, cap;  // per-layer budget and cap
    int64_t B = 0;                // global budget
};

// Per-layer targets t_l = r_lo + (r_hi - r_lo) u24_l / 2^24 in 2^-24 fixed point, shifted by
// the largest common delta with sum_l clamp(t_l + delta) F <= T sum_l F; b_l = floor(clamp(.) F).
int layer_budgets(const Shape& s, const tasp_mask_desc& m, Budgets& out) {
    const int L = s.L;
    const int64_t F = dense_layer_flops(s);
    if (!m.scores || !m.target_u24) return fail(TASP_EINVAL, "greedy mask needs scores and target_u24");
    if (!(m.flop_budget > 0.0 && m.flop_budget <= 1.0) || !(m.r_lo >= 0.0 && m.r_lo <= m.r_hi && m.r_hi <= 1.0))
        return fail(TASP_EINVAL, "greedy mask: budget or retention range out of [0, 1]");
    const int64_t T = fixed_of(m.flop_budget), LO = fixed_of(m.r_lo), HI = fixed_of(m.r_hi);
    if (LO > T) return fail(TASP_EINVAL, "greedy mask: r_lo above the budget");
    std::vector<int64_t> t(L);
    for (int l = 0; l < L; ++l) t[l] = LO + (((HI - LO) * (int64_t)(m.target_u24[l] & 0xFFFFFFu)) >> kFixBits);
    const __int128 b_fix = (__int128)T * (__int128)(F * L);
    auto filled = [&](int64_t delta) {
        __int128 acc = 0;
        for (int l = 0; l < L; ++l) acc += (__int128)std::min(std::max(t[l] + delta, LO), HI) * F;
        return acc;
    };
    int64_t lo = -kFix, hi = kFix, delta;
    if (filled(hi) <= b_fix) {
        delta = hi;
    } else {
        while (hi - lo > 1) {
            int64_t mid = lo + (hi - lo) / 2;
            if (filled(mid) <= b_fix) lo = mid; else hi = mid;
        }
        delta = lo;
    }
    out.b.assign(L, 0);
    out.cap.assign(L, 0);
    for (int l = 0; l < L; ++l) {
        int64_t tt = std::min(std::max(t[l] + delta, LO), HI);
        out.b[l] = (int64_t)(((__int128)tt * F) >> kFixBits);
        out.cap[l] = (int64_t)(((__int128)HI * F) >> kFixBits);
    }
    out.B = (int64_t)(b_fix >> kFixBits);
    return TASP_OK;
}

// Heap entry of the query-head greedy; `cost` is the marginal cost when it was pushed.
struct Cand {
    int layer, idx;  // idx < Hq: query head; else channel unit idx - Hq
    uint32_t score;
    int64_t cost;
};

// Greedy over query heads and channel units with the GQA closure charged on acceptance.
int select_qheads(const Shape& s, const tasp_mask_desc& m, MaskSel& out) {
    const int L = s.L, Hq = s.Hq, g = s.g(), U = s.n_units(), N = Hq + U;
    Budgets bud;
    int rc = layer_budgets(s, m, bud);
    if (rc) return rc;
    out.budget = bud.B;
    const int64_t c_q = layer_flops(s, 1, 0, 0), c_kv = layer_flops(s, 0, 1, 0), c_u = layer_flops(s, 0, 0, s.cu);
    std::vector<std::vector<char>> kept(L, std::vector<char>(N, 0)), kv_on(L, std::vector<char>(s.Hkv, 0));
    std::vector<int64_t> lc(L, 0);
    auto marginal = [&](int l, int i) { return i < Hq ? c_q + (kv_on[l][i / g] ? 0 : c_kv) : c_u; };
    auto score = [&](int l, int i) { return m.scores[(size_t)l * N + i]; };
    // heap order: true when a ranks below b (lower score/cost; on a tie the later in the
    // order query head < channel unit, lower index, and lower layer first (globally) or last)
    auto below = [&](bool layer_major) {
        return [layer_major, Hq](const Cand& a, const Cand& b) {
            unsigned __int128 lhs = (unsigned __int128)a.score * (uint64_t)b.cost;
            unsigned __int128 rhs = (unsigned __int128)b.score * (uint64_t)a.cost;
            if (lhs != rhs) return lhs < rhs;
            int ka = a.idx >= Hq, kb = b.idx >= Hq;
            if (layer_major && a.layer != b.layer) return a.layer > b.layer;
            if (ka != kb) return ka > kb;
            if (a.idx != b.idx) return a.idx > b.idx;
            return a.layer > b.layer;
        };
    };
    auto accept = [&](int l, int i, auto& heap) {
        const int64_t c = marginal(l, i);
        kept[l][i] = 1;
        lc[l] += c;
        if (i < Hq && !kv_on[l][i / g]) {
            kv_on[l][i / g] = 1;
            for (int h = (i / g) * g; h < (i / g + 1) * g; ++h)
                if (!kept[l][h]) heap.push({l, h, score(l, h), marginal(l, h)});
        }
        return c;
    };
    using Heap = std::priority_queue<Cand, std::vector<Cand>, decltype(below(false))>;
    for (int l = 0; l < L; ++l) {
        Heap heap(below(false));
        // forced minimum: the best-scored query head (with its KV head) and channel unit
        int bq = 0, bu = Hq;
        for (int h = 1; h < Hq; ++h) if (score(l, h) > score(l, bq)) bq = h;
        for (int u = Hq + 1; u < N; ++u) if (score(l, u) > score(l, bu)) bu = u;
        for (int i = 0; i < N; ++i) heap.push({l, i, score(l, i), marginal(l, i)});
        accept(l, bq, heap);
        accept(l, bu, heap);
        while (!heap.empty()) {
            Cand c = heap.top();
            heap.pop();
            if (kept[l][c.idx] || c.cost != marginal(l, c.idx)) continue;  // taken or stale
            if (lc[l] + c.cost <= bud.b[l]) accept(l, c.idx, heap);
        }
    }
    int64_t total = 0;
    for (int l = 0; l < L; ++l) total += lc[l];
    Heap heap(below(true));
    for (int l = 0; l < L; ++l)
        for (int i = 0; i < N; ++i)
            if (!kept[l][i]) heap.push({l, i, score(l, i), marginal(l, i)});
    while (!heap.empty()) {
        Cand c = heap.top();
        heap.pop();
        if (kept[c.layer][c.idx] || c.cost != marginal(c.layer, c.idx)) continue;
        if (total + c.cost <= bud.B && lc[c.layer] + c.cost <= bud.cap[c.layer]) total += accept(c.layer, c.idx, heap);
    }
    for (int l = 0; l < L; ++l) {
        for (int h = 0; h < Hq; ++h) if (kept[l][h]) out.qheads[l].push_back(h);
        for (int j = 0; j < s.Hkv; ++j) if (kv_on[l][j]) out.groups[l].push_back(j);
        for (int i = Hq; i < N; ++i) if (kept[l][i]) out.units[l].push_back(i - Hq);
        out.layer_flops[l] = lc[l];
    }
    out.total = total;
    if (total > bud.B) return fail(TASP_EINVAL, "mask exceeds its FLOP budget");
    return TASP_OK;
}

}  // namespace

int select_mask(const Shape& s, const tasp_mask_desc& m, MaskSel& out) {
    const int L = s.L, G = s.Hkv, U = s.n_units();
    out = MaskSel{};
    out.groups.assign(L, {});
    out.qheads.assign(L, {});
    out.units.assign(L, {});
    out.layer_flops.assign(L, 0);
    const int64_t F = dense_layer_flops(s);
    out.dense = F * L;
    const int64_t c_group = layer_flops(s, s.g(), 1, 0);
    const int64_t c_unit = layer_flops(s, 0, 0, s.cu);
    // every query head of the kept groups (the group-granular kinds)
    auto all_heads = [&]() {
        for (int l = 0; l < L; ++l)
            for (int j : out.groups[l])
                for (int h = j * s.g(); h < (j + 1) * s.g(); ++h) out.qheads[l].push_back(h);
    };

    if (m.kind == TASP_MASK_ALL_KEEP) {
        for (int l = 0; l < L; ++l) {
            out.groups[l].resize(G);
            std::iota(out.groups[l].begin(), out.groups[l].end(), 0);
            out.units[l].resize(U);
            std::iota(out.units[l].begin(), out.units[l].end(), 0);
            out.layer_flops[l] = F;
        }
        all_heads();
        out.total = out.budget = out.dense;
        return TASP_OK;
    }
    if (m.kind == TASP_MASK_EXPLICIT || m.kind == TASP_MASK_EXPLICIT_QHEADS) {
        const bool byq = m.kind == TASP_MASK_EXPLICIT_QHEADS;
        const int32_t* keep = byq ? m.keep_qheads : m.keep_groups;
        const int32_t* nkeep = byq ? m.n_qheads : m.n_groups;
        const int nmax = byq ? s.Hq : G;
        if (!keep || !nkeep || !m.keep_units || !m.n_units)
            return fail(TASP_EINVAL, byq ? "explicit query-head mask needs keep_qheads, n_qheads, keep_units, n_units"
                                         : "explicit mask needs keep_groups, n_groups, keep_units, n_units");
        size_t og = 0, ou = 0;
        for (int l = 0; l < L; ++l) {
            int ng = nkeep[l], nu = m.n_units[l];
            if (ng < 0 || ng > nmax || nu < 0 || nu > U) return fail(TASP_EINVAL, "explicit mask: count out of range");
            for (int i = 0; i < ng; ++i) {
                int j = keep[og + i];
                if (j < 0 || j >= nmax || (i && j <= keep[og + i - 1]))
                    return fail(TASP_EINVAL, byq ? "explicit mask: query heads must be ascending and in range"
                                                 : "explicit mask: group indices must be ascending and in range");
                if (!byq) {
                    out.groups[l].push_back(j);
                } else {
                    out.qheads[l].push_back(j);
                    // closure: the KV head of every kept query head (heads ascending, so groups too)
                    if (out.groups[l].empty() || out.groups[l].back() != j / s.g()) out.groups[l].push_back(j / s.g());
                }
            }
            for (int i = 0; i < nu; ++i) {
                int u = m.keep_units[ou + i];
                if (u < 0 || u >= U || (i && u <= m.keep_units[ou + i - 1]))
                    return fail(TASP_EINVAL, "explicit mask: channel units must be ascending and in range");
                out.units[l].push_back(u);
            }
            og += ng;
            ou += nu;
            const int64_t mq = byq ? ng : (int64_t)ng * s.g();
            out.layer_flops[l] = layer_flops(s, mq, (int64_t)out.groups[l].size(), (int64_t)nu * s.cu);
            out.total += out.layer_flops[l];
        }
        if (!byq) all_heads();
        out.budget = out.dense;
        return TASP_OK;
    }
    if (m.kind == TASP_MASK_GREEDY_QHEADS) return select_qheads(s, m, out);
    if (m.kind != TASP_MASK_GREEDY) return fail(TASP_EINVAL, "unknown mask kind");

    Budgets bud;
    int rc = layer_budgets(s, m, bud);
    if (rc) return rc;
    const std::vector<int64_t>& b = bud.b;
    const std::vector<int64_t>& cap = bud.cap;
    const int64_t B = bud.B;
    out.budget = B;

    std::vector<std::vector<char>> kept(L, std::vector<char>(G + U, 0));
    std::vector<int64_t> lc(L, 0);
    auto cost_of = [&](int idx) { return idx < G ? c_group : c_unit; };
    for (int l = 0; l < L; ++l) {
        const uint32_t* sc = m.scores + (size_t)l * (G + U);
        // forced minimum: the best-scored group and channel unit (lowest index on ties)
        int bg = 0, bu = G;
        for (int j = 1; j < G; ++j) if (sc[j] > sc[bg]) bg = j;
        for (int u = G + 1; u < G + U; ++u) if (sc[u] > sc[bu]) bu = u;
        kept[l][bg] = kept[l][bu] = 1;
        lc[l] = c_group + c_unit;
        std::vector<Unit> us;
        us.reserve(G + U);
        for (int i = 0; i < G + U; ++i) us.push_back({l, i, sc[i], cost_of(i)});
        std::sort(us.begin(), us.end(), [&](const Unit& a, const Unit& c) { return ratio_first(a, c, G, false); });
        for (const Unit& u : us)
            if (!kept[l][u.idx] && lc[l] + u.cost <= b[l]) {
                kept[l][u.idx] = 1;
                lc[l] += u.cost;
            }
    }
    int64_t total = 0;
    for (int l = 0; l < L; ++l) total += lc[l];
    std::vector<Unit> rest;
    for (int l = 0; l < L; ++l)
        for (int i = 0; i < G + U; ++i)
            if (!kept[l][i]) rest.push_back({l, i, m.scores[(size_t)l * (G + U) + i], cost_of(i)});
    std::sort(rest.begin(), rest.end(), [&](const Unit& a, const Unit& c) { return ratio_first(a, c, G, true); });
    for (const Unit& u : rest)
        if (total + u.cost <= B && lc[u.layer] + u.cost <= cap[u.layer]) {
            kept[u.layer][u.idx] = 1;
            lc[u.layer] += u.cost;
            total += u.cost;
        }
    for (int l = 0; l < L; ++l) {
        for (int i = 0; i < G; ++i) if (kept[l][i]) out.groups[l].push_back(i);
        for (int i = G; i < G + U; ++i) if (kept[l][i]) out.units[l].push_back(i - G);
        out.layer_flops[l] = lc[l];
    }
    all_heads();
    out.total = total;
    if (total > B) return fail(TASP_EINVAL, "mask exceeds its FLOP budget");
    return TASP_OK;
}

}  // namespace tasp
