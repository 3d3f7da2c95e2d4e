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
#include <algorithm>
#include <cmath>
#include <numeric>
#include <string>

#include "tasp_internal.h"

namespace tasp {

int64_t layer_flops(const Shape& s, int64_t m_q, int64_t m_kv, int64_t c) {
    const int64_t d = s.d, dh = s.dh;
    return 2 * d * dh * (m_q + 2 * m_kv) + 2 * dh * m_q * d + 6 * d * c;
}

bool Shape::same(const Shape& o) const {
    return L == o.L && d == o.d && Hq == o.Hq && Hkv == o.Hkv && dh == o.dh && df == o.df && vocab == o.vocab &&
           cu == o.cu && eps == o.eps && theta == o.theta && seed == o.seed;
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

}  // namespace

int select_mask(const Shape& s, const tasp_mask_desc& m, MaskSel& out) {
    const int L = s.L, G = s.Hkv, U = s.n_units();
    out = MaskSel{};
    out.groups.assign(L, {});
    out.units.assign(L, {});
    out.layer_flops.assign(L, 0);
    const int64_t F = dense_layer_flops(s);
    out.dense = F * L;
    const int64_t c_group = layer_flops(s, s.g(), 1, 0);
    const int64_t c_unit = layer_flops(s, 0, 0, s.cu);

    if (m.kind == TASP_MASK_ALL_KEEP) {
        for (int l = 0; l < L; ++l) {
            out.groups[l].resize(G);
            std::iota(out.groups[l].begin(), out.groups[l].end(), 0);
            out.units[l].resize(U);
            std::iota(out.units[l].begin(), out.units[l].end(), 0);
            out.layer_flops[l] = F;
        }
        out.total = out.budget = out.dense;
        return TASP_OK;
    }
    if (m.kind == TASP_MASK_EXPLICIT) {
        if (!m.keep_groups || !m.n_groups || !m.keep_units || !m.n_units)
            return fail(TASP_EINVAL, "explicit mask needs keep_groups, n_groups, keep_units, n_units");
        size_t og = 0, ou = 0;
        for (int l = 0; l < L; ++l) {
            int ng = m.n_groups[l], nu = m.n_units[l];
            if (ng < 0 || ng > G || nu < 0 || nu > U) return fail(TASP_EINVAL, "explicit mask: count out of range");
            for (int i = 0; i < ng; ++i) {
                int j = m.keep_groups[og + i];
                if (j < 0 || j >= G || (i && j <= m.keep_groups[og + i - 1]))
                    return fail(TASP_EINVAL, "explicit mask: group indices must be ascending and in range");
                out.groups[l].push_back(j);
            }
            for (int i = 0; i < nu; ++i) {
                int u = m.keep_units[ou + i];
                if (u < 0 || u >= U || (i && u <= m.keep_units[ou + i - 1]))
                    return fail(TASP_EINVAL, "explicit mask: channel units must be ascending and in range");
                out.units[l].push_back(u);
            }
            og += ng;
            ou += nu;
            out.layer_flops[l] = layer_flops(s, (int64_t)ng * s.g(), ng, (int64_t)nu * s.cu);
            out.total += out.layer_flops[l];
        }
        out.budget = out.dense;
        return TASP_OK;
    }
    if (m.kind != TASP_MASK_GREEDY) return fail(TASP_EINVAL, "unknown mask kind");
    if (!m.scores || !m.target_u24) return fail(TASP_EINVAL, "greedy mask needs scores and target_u24");
    if (!(m.flop_budget > 0.0 && m.flop_budget <= 1.0) || !(m.r_lo >= 0.0 && m.r_lo <= m.r_hi && m.r_hi <= 1.0))
        return fail(TASP_EINVAL, "greedy mask: budget or retention range out of [0, 1]");

    const int64_t T = fixed_of(m.flop_budget), LO = fixed_of(m.r_lo), HI = fixed_of(m.r_hi);
    if (LO > T) return fail(TASP_EINVAL, "greedy mask: r_lo above the budget");
    // per-layer targets in fixed point, then the common shift delta (largest feasible)
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
    std::vector<int64_t> b(L), cap(L);
    for (int l = 0; l < L; ++l) {
        int64_t tt = std::min(std::max(t[l] + delta, LO), HI);
        b[l] = (int64_t)(((__int128)tt * F) >> kFixBits);
        cap[l] = (int64_t)(((__int128)HI * F) >> kFixBits);
    }
    const int64_t B = (int64_t)(b_fix >> kFixBits);
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
    out.total = total;
    if (total > B) return fail(TASP_EINVAL, "mask exceeds its FLOP budget");
    return TASP_OK;
}

}  // namespace tasp
