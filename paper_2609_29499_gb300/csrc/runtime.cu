// C ABI of the TASP runtime: shared store registry, plan compilation and packing,
// sessions with plan-bound KV caches, CUDA-graph decode steps, introspection.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <atomic>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "tasp_internal.h"

namespace tasp {


// ---------------------------------------------------------------- errors
static thread_local std::string g_err;

void set_error(const std::string& msg) { g_err = msg; }
int fail(int code, const std::string& msg) {
    g_err = msg;
    return code;
}
int cuda_fail(cudaError_t e, const char* what) {
    g_err = std::string(what) + ": " + cudaGetErrorString(e);
    return e == cudaErrorMemoryAllocation ? TASP_ENOMEM : TASP_ECUDA;
}

// ---------------------------------------------------------------- device info
namespace test_hooks {
static std::atomic<long long> g_wait_limit{0};
static std::atomic<int> g_skip{0};
long long wait_limit(long long dflt) {
    const long long v = g_wait_limit.load();
    return v > 0 ? v : dflt;
}
bool take_skip() {
    int v = g_skip.load();
    while (v > 0)
        if (g_skip.compare_exchange_weak(v, v - 1)) return true;
    return false;
}
}  // namespace test_hooks

int device_info(DevInfo& out) {
    static DevInfo cached;
    static std::mutex mu;
    std::lock_guard<std::mutex> lk(mu);
    int dev = 0;
    TASP_CUDA(cudaGetDevice(&dev));
    if (cached.dev != dev) {
        cudaDeviceProp pr;
        TASP_CUDA(cudaGetDeviceProperties(&pr, dev));
        cached.dev = dev;
        cached.sms = pr.multiProcessorCount;
        cached.smem_optin = (int)pr.sharedMemPerBlockOptin;
        cached.smem_per_sm = (int)pr.sharedMemPerMultiprocessor;
        cached.smem_reserved = (int)pr.reservedSharedMemPerBlock;
    }
    out = cached;
    return TASP_OK;
}

// ---------------------------------------------------------------- arena
// Device bytes held by all arenas, and the optional cap on them (0 = none).
static std::atomic<int64_t> g_arena_bytes{0};
static std::atomic<int64_t> g_arena_limit{0};

int Arena::reserve(size_t bytes) {
    cap = (bytes + 255) & ~size_t(255);
    used = 0;
    if (cap == 0) return TASP_OK;
    const int64_t lim = g_arena_limit.load();
    const int64_t now = g_arena_bytes.fetch_add((int64_t)cap) + (int64_t)cap;
    if (lim > 0 && now > lim) {
        g_arena_bytes.fetch_sub((int64_t)cap);
        const size_t want = cap;
        cap = 0;
        return fail(TASP_ENOMEM, "device memory limit reached (" + std::to_string(want) + " more bytes, " +
                                     std::to_string(now - (int64_t)want) + " of " + std::to_string(lim) + " in use)");
    }
    cudaError_t e = cudaMalloc((void**)&base, cap);
    if (e != cudaSuccess) {
        g_arena_bytes.fetch_sub((int64_t)cap);
        base = nullptr;
        cap = 0;
        return cuda_fail(e, "cudaMalloc");
    }
    return TASP_OK;
}
void* Arena::take(size_t bytes) {
    size_t b = (bytes + 255) & ~size_t(255);
    if (used + b > cap) return nullptr;
    void* p = base + used;
    used += b;
    return p;
}
void Arena::release() {
    if (base) {
        cudaFree(base);
        g_arena_bytes.fetch_sub((int64_t)cap);
    }
    base = nullptr;
    cap = used = 0;
}

// Sizing pass helper: records sizes then hands out pointers from a reserved arena.
struct Layout {
    std::vector<size_t> sizes;
    size_t total = 0;
    void add(size_t b) {
        sizes.push_back(b);
        total += (b + 255) & ~size_t(255);
    }
};

static int round16(int v) { return (v + 15) & ~15; }
static int round8(int v) { return (v + 7) & ~7; }

// ---------------------------------------------------------------- store registry
static std::mutex g_mu;
static std::vector<Store*> g_stores;

int validate_shape(const tasp_model_desc* m, Shape& s, bool device) {
    if (!m) return fail(TASP_EINVAL, "model_desc is NULL");
    s.L = m->L; s.d = m->d; s.Hq = m->Hq; s.Hkv = m->Hkv; s.dh = m->dh; s.df = m->df; s.vocab = m->vocab;
    s.cu = m->chan_unit; s.eps = m->rms_eps; s.theta = m->rope_theta; s.seed = m->seed; s.qg = m->quant_group;
    if (s.L < 1 || s.d < 16 || s.d % 16 || s.Hq < 1 || s.Hkv < 1 || s.Hq % s.Hkv || s.dh < 16 || s.dh % 16 ||
        s.dh > 128 || s.df < 1 || s.df % 16 || s.cu < 1 || s.df % s.cu || s.vocab < 0 || !(s.eps > 0.f) ||
        !(s.theta > 0.f))
        return fail(TASP_EINVAL, "invalid model shape (need d, df, dh multiples of 16, dh <= 128, Hq % Hkv == 0, "
                                 "df % chan_unit == 0)");
    if (s.qg < 0 || (s.qg && (s.qg % 16 || ((s.qg / 16) & (s.qg / 16 - 1)) || s.d % s.qg || s.df % s.qg ||
                              s.dh % s.qg || s.cu % s.qg)))
        return fail(TASP_EINVAL, "quant_group must be 0 or 16 times a power of two dividing d, df, dh and chan_unit");
    if (!device) return TASP_OK;
    if (!attn_supported(s.dh, s.g()))
        return fail(TASP_EUNSUP, "attention kernel not built for this (head_dim, query heads per group)");
    if ((int64_t)s.d * 4 > 200 * 1024 || (int64_t)s.df * 4 > 200 * 1024)
        return fail(TASP_EUNSUP, "hidden or SwiGLU width too large for the shared-memory activation stage");
    return TASP_OK;
}

static int store_acquire(const Shape& sh, Store** out) {
    std::lock_guard<std::mutex> lk(g_mu);
    for (Store* st : g_stores)
        if (st->sh.same(sh)) {
            st->refs++;
            *out = st;
            return TASP_OK;
        }
    auto st = std::make_unique<Store>();
    st->sh = sh;
    const size_t d = sh.d, qkv = (size_t)sh.qkv_rows_dense(), hq = (size_t)sh.Hq * sh.dh, df = sh.df;
    Layout lay;
    const size_t G = sh.qg;
    for (int l = 0; l < sh.L; ++l) {
        lay.add(qkv * d); lay.add(d * hq); lay.add(2 * df * d); lay.add(d * df);
        lay.add(qkv * 4); lay.add(d * 4); lay.add(2 * df * 4); lay.add(d * 4); lay.add(d * 4); lay.add(d * 4);
        if (G) { lay.add(qkv * (d / G) * 2); lay.add(d * (hq / G) * 2); lay.add(2 * df * (d / G) * 2); lay.add(d * (df / G) * 2); }
    }
    lay.add(d * 4);
    lay.add((size_t)sh.vocab * d * 2);
    int rc = st->arena.reserve(lay.total);
    if (rc) return rc;
    st->layers.resize(sh.L);
    for (int l = 0; l < sh.L; ++l) {
        LayerStore& ls = st->layers[l];
        ls.qkv = (int8_t*)st->arena.take(qkv * d);
        ls.o = (int8_t*)st->arena.take(d * hq);
        ls.gu = (int8_t*)st->arena.take(2 * df * d);
        ls.down = (int8_t*)st->arena.take(d * df);
        ls.qkv_s = (float*)st->arena.take(qkv * 4);
        ls.o_s = (float*)st->arena.take(d * 4);
        ls.gu_s = (float*)st->arena.take(2 * df * 4);
        ls.down_s = (float*)st->arena.take(d * 4);
        ls.g_attn = (float*)st->arena.take(d * 4);
        ls.g_mlp = (float*)st->arena.take(d * 4);
        if (G) {
            ls.qkv_g = (uint16_t*)st->arena.take(qkv * (d / G) * 2);
            ls.o_g = (uint16_t*)st->arena.take(d * (hq / G) * 2);
            ls.gu_g = (uint16_t*)st->arena.take(2 * df * (d / G) * 2);
            ls.down_g = (uint16_t*)st->arena.take(d * (df / G) * 2);
        }
    }
    st->g_final = (float*)st->arena.take(d * 4);
    st->lm_head = sh.vocab ? (uint16_t*)st->arena.take((size_t)sh.vocab * d * 2) : nullptr;
    st->bytes = lay.total;
    cudaStream_t s;
    cudaError_t ce = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
    if (ce != cudaSuccess) {
        st->arena.release();
        return cuda_fail(ce, "cudaStreamCreateWithFlags");
    }
    rc = store_generate(*st, s);
    cudaError_t e = cudaStreamSynchronize(s);
    cudaStreamDestroy(s);
    if (rc) {
        st->arena.release();
        return rc;
    }
    if (e != cudaSuccess) {
        st->arena.release();
        return cuda_fail(e, "store generation");
    }
    st->refs = 1;
    *out = st.get();
    g_stores.push_back(st.release());
    return TASP_OK;
}

static void store_release(Store* st) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (--st->refs > 0) return;
    st->arena.release();
    g_stores.erase(std::remove(g_stores.begin(), g_stores.end(), st), g_stores.end());
    delete st;
}

// ---------------------------------------------------------------- plan compilation
// Source rows of the qkv panel in the store (per kept group its kept heads' d_h-row blocks,
// then K, then V; store rows are group-major: g head blocks, K, V), source columns of the O
// panel (the kept heads in ascending order), and the role / slot / block tables of partial
// groups (see LayerPlan).
static void layer_tables(const Shape& sh, const LayerPlan& lp, std::vector<int32_t>& hq, std::vector<int32_t>& ho,
                         std::vector<int16_t>& hrole, std::vector<int16_t>& hslot, std::vector<int16_t>& hblk) {
    const int g = sh.g(), dh = sh.dh;
    hq.clear(); ho.clear(); hrole.clear();
    hslot.assign((size_t)lp.m_kv * g, -1);
    hblk.assign((size_t)lp.m_kv * (g + 2), -1);
    std::vector<char> keep_h(sh.Hq, 0);
    for (int h : lp.keep_qheads) keep_h[h] = 1;
    int slot = 0;
    for (int jl = 0; jl < lp.m_kv; ++jl) {
        const int j = lp.keep_groups[jl];
        for (int hh = 0; hh < g + 2; ++hh) {
            if (hh < g && !keep_h[j * g + hh]) continue;
            for (int r = 0; r < dh; ++r) hq.push_back((j * (g + 2) + hh) * dh + r);
            hblk[(size_t)jl * (g + 2) + hh] = (int16_t)hrole.size();
            hrole.push_back((int16_t)(jl * (g + 2) + hh));
            if (hh < g) {
                hslot[(size_t)jl * g + hh] = (int16_t)slot++;
                for (int c = 0; c < dh; ++c) ho.push_back((j * g + hh) * dh + c);
            }
        }
    }
}

static int build_plan(Plan& p, const MaskSel& sel, int panel_mode, bool all_keep) {
    Store& st = *p.store;
    const Shape& sh = st.sh;
    const int g = sh.g(), dh = sh.dh, d = sh.d;
    p.layers.resize(sh.L);
    for (int l = 0; l < sh.L; ++l) {
        LayerPlan& lp = p.layers[l];
        lp.keep_groups = sel.groups[l];
        lp.keep_qheads = sel.qheads[l];
        lp.keep_chans.clear();
        for (int u : sel.units[l])
            for (int i = 0; i < sh.cu; ++i) lp.keep_chans.push_back(u * sh.cu + i);
        lp.m_kv = (int)lp.keep_groups.size();
        lp.m_q = (int)lp.keep_qheads.size();
        lp.c = (int)lp.keep_chans.size();
        lp.qkv_rows = (lp.m_q + 2 * lp.m_kv) * dh;
        lp.gu_rows = 2 * lp.c;
        lp.o_K = lp.m_q * dh;
        lp.dn_K = lp.c;
        lp.g_attn = st.layers[l].g_attn;
        lp.g_mlp = st.layers[l].g_mlp;
    }
    p.all_keep = all_keep;
    p.panel_mode = panel_mode;
    if (all_keep) {
        for (int l = 0; l < sh.L; ++l) {
            LayerPlan& lp = p.layers[l];
            const LayerStore& ls = st.layers[l];
            lp.qkv_w = ls.qkv; lp.qkv_s = ls.qkv_s;
            lp.o_w = ls.o; lp.o_s = ls.o_s; lp.o_ld = sh.Hq * dh;
            lp.gu_w = ls.gu; lp.gu_s = ls.gu_s;
            lp.dn_w = ls.down; lp.dn_s = ls.down_s; lp.dn_ld = sh.df;
            lp.qkv_g = ls.qkv_g; lp.o_g = ls.o_g; lp.gu_g = ls.gu_g; lp.dn_g = ls.down_g;
            if (sh.qg) {
                lp.qkv_gld = lp.gu_gld = d / sh.qg;
                lp.o_gld = sh.Hq * dh / sh.qg;
                lp.dn_gld = sh.df / sh.qg;
            }
        }
        return TASP_OK;
    }
    const int G = sh.qg;  // scale group of a grouped store (0: per-row scales only)
    const bool rowidx = panel_mode == TASP_PANELS_ROW_INDEXED;
    auto ragged = [&](const LayerPlan& lp) { return lp.m_q != lp.m_kv * g; };
    // sizing pass
    Layout lay;
    for (int l = 0; l < sh.L; ++l) {
        const LayerPlan& lp = p.layers[l];
        const size_t ol = round16(lp.o_K), dl = round16(lp.dn_K);
        if (G) {  // group scales in panel order (rows padded to 16 bytes), and the column-group maps of O / down
            lay.add((size_t)lp.qkv_rows * round8(d / G) * 2); lay.add((size_t)lp.gu_rows * round8(d / G) * 2);
            lay.add((size_t)d * round8(lp.o_K / G) * 2); lay.add((size_t)d * round8(lp.dn_K / G) * 2);
            lay.add((size_t)(lp.o_K / G) * 4); lay.add((size_t)(lp.dn_K / G) * 4);
        }
        if (ragged(lp)) {
            lay.add((size_t)(lp.m_q + 2 * lp.m_kv) * 2);
            lay.add((size_t)lp.m_kv * g * 2);
            lay.add((size_t)lp.m_kv * (g + 2) * 2);
        }
        lay.add((size_t)lp.qkv_rows * 4); lay.add((size_t)lp.qkv_rows * 4);  // map, scales
        lay.add((size_t)lp.gu_rows * 4); lay.add((size_t)lp.gu_rows * 4);
        lay.add(ol * 4); lay.add(dl * 4);                                       // column maps
        if (!rowidx) { lay.add((size_t)lp.qkv_rows * d); lay.add((size_t)lp.gu_rows * d); }
        lay.add((size_t)d * ol); lay.add((size_t)d * dl);
    }
    int rc = p.arena.reserve(lay.total);
    if (rc) return rc;
    cudaStream_t s;
    TASP_CUDA(cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking));
    std::vector<int32_t> hq, hg, ho, hd;
    std::vector<int16_t> hrole, hslot, hblk;
    for (int l = 0; l < sh.L && !rc; ++l) {
        LayerPlan& lp = p.layers[l];
        const LayerStore& ls = st.layers[l];
        const int ol = round16(lp.o_K), dl = round16(lp.dn_K);
        layer_tables(sh, lp, hq, ho, hrole, hslot, hblk);
        hg.clear(); hd.clear();
        for (int c : lp.keep_chans) { hg.push_back(2 * c); hg.push_back(2 * c + 1); }
        ho.resize(ol, 0);
        hd = std::vector<int32_t>(lp.keep_chans.begin(), lp.keep_chans.end());
        hd.resize(dl, 0);
        int32_t* dq = (int32_t*)p.arena.take(hq.size() * 4);
        float* sq = (float*)p.arena.take(hq.size() * 4);
        int32_t* dg = (int32_t*)p.arena.take(hg.size() * 4);
        float* sg = (float*)p.arena.take(hg.size() * 4);
        int32_t* dco = (int32_t*)p.arena.take(ho.size() * 4);
        int32_t* dcd = (int32_t*)p.arena.take(hd.size() * 4);
        if (ragged(lp)) {
            int16_t* drole = (int16_t*)p.arena.take(hrole.size() * 2);
            int16_t* dslot = (int16_t*)p.arena.take(hslot.size() * 2);
            int16_t* dblk = (int16_t*)p.arena.take(hblk.size() * 2);
            TASP_CUDA(cudaMemcpyAsync(drole, hrole.data(), hrole.size() * 2, cudaMemcpyHostToDevice, s));
            TASP_CUDA(cudaMemcpyAsync(dslot, hslot.data(), hslot.size() * 2, cudaMemcpyHostToDevice, s));
            TASP_CUDA(cudaMemcpyAsync(dblk, hblk.data(), hblk.size() * 2, cudaMemcpyHostToDevice, s));
            lp.blk_role = drole;
            lp.oslot = dslot;
            lp.blk_of = dblk;
        }
        if (hq.size()) TASP_CUDA(cudaMemcpyAsync(dq, hq.data(), hq.size() * 4, cudaMemcpyHostToDevice, s));
        if (hg.size()) TASP_CUDA(cudaMemcpyAsync(dg, hg.data(), hg.size() * 4, cudaMemcpyHostToDevice, s));
        if (ho.size()) TASP_CUDA(cudaMemcpyAsync(dco, ho.data(), ho.size() * 4, cudaMemcpyHostToDevice, s));
        if (hd.size()) TASP_CUDA(cudaMemcpyAsync(dcd, hd.data(), hd.size() * 4, cudaMemcpyHostToDevice, s));
        if ((rc = gather_f32(sq, ls.qkv_s, dq, (int)hq.size(), s))) break;
        if ((rc = gather_f32(sg, ls.gu_s, dg, (int)hg.size(), s))) break;
        lp.qkv_s = sq;
        lp.gu_s = sg;
        if (G) {
            // qkv / gu: the scale rows follow their weight rows; O / down: the scale columns of
            // the kept column groups (kept heads and channel units are whole groups)
            std::vector<int32_t> cgo, cgd;
            for (size_t k = 0; k < (size_t)lp.o_K; k += G) cgo.push_back(ho[k] / G);
            for (size_t k = 0; k < (size_t)lp.dn_K; k += G) cgd.push_back(lp.keep_chans[k] / G);
            // scale rows padded to 16 bytes (zeros), so that a GEMV stage can take them by bulk copy
            lp.qkv_gld = lp.gu_gld = round8(d / G);
            lp.o_gld = round8(lp.o_K / G);
            lp.dn_gld = round8(lp.dn_K / G);
            uint16_t* gq = (uint16_t*)p.arena.take((size_t)lp.qkv_rows * lp.qkv_gld * 2);
            uint16_t* gg = (uint16_t*)p.arena.take((size_t)lp.gu_rows * lp.gu_gld * 2);
            uint16_t* go = (uint16_t*)p.arena.take((size_t)d * lp.o_gld * 2);
            uint16_t* gd = (uint16_t*)p.arena.take((size_t)d * lp.dn_gld * 2);
            TASP_CUDA(cudaMemsetAsync(gq, 0, (size_t)lp.qkv_rows * lp.qkv_gld * 2, s));
            TASP_CUDA(cudaMemsetAsync(gg, 0, (size_t)lp.gu_rows * lp.gu_gld * 2, s));
            TASP_CUDA(cudaMemsetAsync(go, 0, (size_t)d * lp.o_gld * 2, s));
            TASP_CUDA(cudaMemsetAsync(gd, 0, (size_t)d * lp.dn_gld * 2, s));
            int32_t* dgo = (int32_t*)p.arena.take(cgo.size() * 4);
            int32_t* dgd = (int32_t*)p.arena.take(cgd.size() * 4);
            if (cgo.size()) TASP_CUDA(cudaMemcpyAsync(dgo, cgo.data(), cgo.size() * 4, cudaMemcpyHostToDevice, s));
            if (cgd.size()) TASP_CUDA(cudaMemcpyAsync(dgd, cgd.data(), cgd.size() * 4, cudaMemcpyHostToDevice, s));
            if ((rc = gather_u16_rows(gq, lp.qkv_gld, ls.qkv_g, dq, lp.qkv_rows, d / G, s))) break;
            if ((rc = gather_u16_rows(gg, lp.gu_gld, ls.gu_g, dg, lp.gu_rows, d / G, s))) break;
            if ((rc = gather_u16_cols(go, lp.o_gld, ls.o_g, sh.Hq * dh / G, dgo, d, lp.o_K / G, s))) break;
            if ((rc = gather_u16_cols(gd, lp.dn_gld, ls.down_g, sh.df / G, dgd, d, lp.dn_K / G, s))) break;
            // the host vectors above die at the end of this block: wait for their copies
            cudaError_t ge = cudaStreamSynchronize(s);
            if (ge != cudaSuccess) { rc = cuda_fail(ge, "group scale packing"); break; }
            lp.qkv_g = gq; lp.gu_g = gg; lp.o_g = go; lp.dn_g = gd;
        }
        if (rowidx) {
            lp.qkv_w = ls.qkv; lp.qkv_map = dq;
            lp.gu_w = ls.gu; lp.gu_map = dg;
        } else {
            int8_t* wq = (int8_t*)p.arena.take((size_t)lp.qkv_rows * d);
            int8_t* wg = (int8_t*)p.arena.take((size_t)lp.gu_rows * d);
            if ((rc = gather_rows(wq, ls.qkv, dq, lp.qkv_rows, d, s))) break;
            if ((rc = gather_rows(wg, ls.gu, dg, lp.gu_rows, d, s))) break;
            lp.qkv_w = wq;
            lp.gu_w = wg;
        }
        int8_t* wo = (int8_t*)p.arena.take((size_t)d * ol);
        int8_t* wd = (int8_t*)p.arena.take((size_t)d * dl);
        if ((rc = gather_cols(wo, ol, ls.o, sh.Hq * dh, dco, d, lp.o_K, s))) break;
        if ((rc = gather_cols(wd, dl, ls.down, sh.df, dcd, d, lp.dn_K, s))) break;
        lp.o_w = wo; lp.o_ld = ol; lp.o_s = ls.o_s;
        lp.dn_w = wd; lp.dn_ld = dl; lp.dn_s = ls.down_s;
        // host vectors must outlive the async copies
        cudaError_t e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) { rc = cuda_fail(e, "plan packing"); break; }
    }
    cudaStreamDestroy(s);
    return rc;
}

static void plan_ledger(Plan& p) {
    const Shape& sh = p.store->sh;
    int64_t fl = 0, launched = 0, bytes = 0;
    for (const LayerPlan& lp : p.layers) {
        fl += layer_flops(sh, lp.m_q, lp.m_kv, lp.c);
        launched += 2 * (int64_t)lp.qkv_rows * sh.d + 2 * (int64_t)sh.d * lp.o_K + 2 * (int64_t)lp.gu_rows * sh.d +
                    2 * (int64_t)sh.d * lp.dn_K;
        bytes += (int64_t)lp.qkv_rows * sh.d + (int64_t)sh.d * lp.o_K + (int64_t)lp.gu_rows * sh.d +
                 (int64_t)sh.d * lp.dn_K;
        bytes += 4 * ((int64_t)lp.qkv_rows + (lp.m_kv ? sh.d : 0) + lp.gu_rows + (lp.c ? sh.d : 0));
        if (sh.qg)  // BF16 group scales, 2 bytes per qg weights
            bytes += 2 * (((int64_t)lp.qkv_rows + lp.gu_rows) * (sh.d / sh.qg) +
                          (int64_t)sh.d * ((lp.o_K + lp.dn_K) / sh.qg));
        bytes += 2 * 4 * (int64_t)sh.d;  // norm gains
    }
    bytes += (int64_t)sh.vocab * sh.d * 2 + 4 * (int64_t)sh.d;
    p.flops_retained = fl;
    p.flops_dense = dense_layer_flops(sh) * sh.L;
    p.launched_flops = launched;
    p.weight_bytes_per_token = bytes;
}

static Plan* as_plan(void* h) {
    Plan* p = (Plan*)h;
    return (p && p->magic == PLAN_MAGIC) ? p : nullptr;
}
static Session* as_session(void* h) {
    Session* s = (Session*)h;
    return (s && s->magic == SESSION_MAGIC) ? s : nullptr;
}

// ---------------------------------------------------------------- sessions
static int session_alloc(Plan* p, int max_tokens, Session** out) {
    const Shape& sh = p->store->sh;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    auto se = std::make_unique<Session>();
    se->plan = p;
    se->max_tokens = max_tokens;
    int smax = 1;
    for (const LayerPlan& lp : p->layers)
        smax = std::max(smax, attn_splits(lp.m_kv, max_tokens, di.sms, sh.dh, sh.g(), 8) / 8);  // either cluster size
    se->att_splits_max = smax;
    Layout lay;
    for (const LayerPlan& lp : p->layers) {
        lay.add((size_t)lp.m_kv * max_tokens * sh.dh * 2);
        lay.add((size_t)lp.m_kv * max_tokens * sh.dh * 2);
    }
    const size_t half = sh.dh / 2;
    lay.add((size_t)max_tokens * half * sizeof(float2));
    lay.add(sizeof(int));
    lay.add((size_t)sh.d * 4);
    lay.add((size_t)sh.Hq * sh.dh * 4);
    lay.add((size_t)sh.Hq * sh.dh * 4);
    lay.add((size_t)sh.df * 4);
    const size_t part = (size_t)sh.Hkv * smax * sh.g() * sh.dh * 4;
    const size_t mlb = (size_t)sh.Hkv * smax * sh.g() * 2 * 4;
    lay.add(part);
    lay.add(mlb);
    lay.add((size_t)sh.Hkv * 4);
    lay.add(sizeof(int));
    lay.add((size_t)sh.d * 2);
    lay.add((size_t)sh.vocab * 4);
    lay.add((size_t)sh.d * 4);
    if ((rc = se->arena.reserve(lay.total))) return rc;
    for (const LayerPlan& lp : p->layers) {
        se->K.push_back((uint16_t*)se->arena.take((size_t)lp.m_kv * max_tokens * sh.dh * 2));
        se->V.push_back((uint16_t*)se->arena.take((size_t)lp.m_kv * max_tokens * sh.dh * 2));
        // TMA descriptors of the layer's caches for decode attention
        CUtensorMap mk{}, mv{};
        if (lp.m_kv > 0 && (sh.dh == 64 || sh.dh == 128)) {
            if ((rc = encode_kv_map(&mk, se->K.back(), sh.dh, max_tokens, lp.m_kv))) return rc;
            if ((rc = encode_kv_map(&mv, se->V.back(), sh.dh, max_tokens, lp.m_kv))) return rc;
        }
        se->tmK.push_back(mk);
        se->tmV.push_back(mv);
    }
    se->rope = (float2*)se->arena.take((size_t)max_tokens * half * sizeof(float2));
    se->d_pos = (int*)se->arena.take(sizeof(int));
    se->x = (float*)se->arena.take((size_t)sh.d * 4);
    se->q = (float*)se->arena.take((size_t)sh.Hq * sh.dh * 4);
    se->o = (float*)se->arena.take((size_t)sh.Hq * sh.dh * 4);
    se->h = (float*)se->arena.take((size_t)sh.df * 4);
    se->part = (float*)se->arena.take(part);
    se->ml = (float*)se->arena.take(mlb);
    se->cnt = (int*)se->arena.take((size_t)sh.Hkv * 4);
    se->err = (int*)se->arena.take(sizeof(int));
    se->x_stage = (uint16_t*)se->arena.take((size_t)sh.d * 2);
    se->logits_stage = sh.vocab ? (float*)se->arena.take((size_t)sh.vocab * 4) : nullptr;
    se->hidden_stage = (float*)se->arena.take((size_t)sh.d * 4);
    // zero the whole arena: empty caches, position 0, attention tickets 0
    TASP_CUDA(cudaMemset(se->arena.base, 0, se->arena.cap));
    if ((rc = rope_table(*se, 0))) return rc;
    TASP_CUDA(cudaDeviceSynchronize());
    *out = se.release();
    return TASP_OK;
}

static void session_free(Session* se) {
    if (se->graph.exec) cudaGraphExecDestroy(se->graph.exec);
    se->arena.release();
    se->magic = 0;
    delete se;
}

// Record (or re-record) the step graph of a batch view for a set of caller buffers.
static int record_graph(StepGraph& g, const BatchView& bv, const StepTarget& t) {
    if (g.exec && g.x == t.x_in && g.hidden == t.hidden_out && g.logits == t.logits) return TASP_OK;
    if (g.exec) {
        cudaGraphExecDestroy(g.exec);
        g.exec = nullptr;
    }
    cudaStream_t cs;
    TASP_CUDA(cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking));
    cudaError_t e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeRelaxed);
    if (e != cudaSuccess) {
        cudaStreamDestroy(cs);
        return cuda_fail(e, "cudaStreamBeginCapture");
    }
    int launches = 0;
    int rc = enqueue_batch(bv, t, cs, -1, nullptr, nullptr, &launches);
    cudaGraph_t graph = nullptr;
    e = cudaStreamEndCapture(cs, &graph);
    cudaStreamDestroy(cs);
    if (rc) {
        if (graph) cudaGraphDestroy(graph);
        return rc;
    }
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamEndCapture");
    e = cudaGraphInstantiate(&g.exec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) {
        g.exec = nullptr;
        return cuda_fail(e, "cudaGraphInstantiate");
    }
    g.x = t.x_in;
    g.hidden = t.hidden_out;
    g.logits = t.logits;
    g.launches = launches;
    return TASP_OK;
}

static int session_graph(Session& se, const StepTarget& t) { return record_graph(se.graph, single_view(se), t); }

// ---------------------------------------------------------------- batches
// 2 to 4 sessions of one plan decoded together: every weight byte of a step is read
// once for all of them (the decode step groups sessions per plan). A batch keeps the
// step workspace for its sessions and its own CUDA graph; it is made on first use and
// dropped when one of its sessions is released.
struct Batch {
    std::vector<Session*> ss;
    Arena arena;
    BatchView view;
    uint16_t* x_stage = nullptr;  // BF16 [n][d] step-input staging (device and host-buffer steps)
    float* hidden_stage = nullptr;
    float* logits_stage = nullptr;
    StepGraph graph;
};
static std::map<std::vector<Session*>, Batch*> g_batches;  // guarded by g_mu

static void batch_free(Batch* b) {
    if (b->graph.exec) cudaGraphExecDestroy(b->graph.exec);
    b->arena.release();
    delete b;
}

static int batch_get(Session* const* ss, int n, Batch** out) {
    std::vector<Session*> key(ss, ss + n);
    {
        std::lock_guard<std::mutex> lk(g_mu);
        auto it = g_batches.find(key);
        if (it != g_batches.end()) {
            *out = it->second;
            return TASP_OK;
        }
    }
    const Plan& p = *ss[0]->plan;
    const Shape& sh = p.store->sh;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    const int smax = batch_attn_slots(p, ss, n, di.sms);
    const int64_t xs = sh.d, qs = (int64_t)sh.Hq * sh.dh, hs = (sh.df + 3) & ~3;
    const int64_t ps = (int64_t)sh.Hkv * smax * sh.g() * sh.dh, ms = (int64_t)sh.Hkv * smax * sh.g() * 2;
    Layout lay;
    lay.add((size_t)n * xs * 4);
    lay.add((size_t)n * qs * 4);
    lay.add((size_t)n * qs * 4);
    lay.add((size_t)n * hs * 4);
    lay.add((size_t)n * ps * 4);
    lay.add((size_t)n * ms * 4);
    lay.add((size_t)n * sh.Hkv * 4);
    lay.add(sizeof(int));
    lay.add((size_t)n * sh.d * 2);
    lay.add((size_t)n * sh.d * 4);
    lay.add((size_t)n * sh.vocab * 4);
    auto b = std::make_unique<Batch>();
    b->ss = key;
    if ((rc = b->arena.reserve(lay.total))) return rc;
    BatchView& v = b->view;
    v.n = n;
    for (int i = 0; i < n; ++i) v.ss[i] = ss[i];
    v.x = (float*)b->arena.take((size_t)n * xs * 4);
    v.q = (float*)b->arena.take((size_t)n * qs * 4);
    v.o = (float*)b->arena.take((size_t)n * qs * 4);
    v.h = (float*)b->arena.take((size_t)n * hs * 4);
    v.part = (float*)b->arena.take((size_t)n * ps * 4);
    v.ml = (float*)b->arena.take((size_t)n * ms * 4);
    v.cnt = (int*)b->arena.take((size_t)n * sh.Hkv * 4);
    v.err = (int*)b->arena.take(sizeof(int));
    v.x_stride = xs;
    v.q_stride = qs;
    v.h_stride = hs;
    v.part_stride = ps;
    v.ml_stride = ms;
    v.cnt_stride = sh.Hkv;
    b->x_stage = (uint16_t*)b->arena.take((size_t)n * sh.d * 2);
    b->hidden_stage = (float*)b->arena.take((size_t)n * sh.d * 4);
    b->logits_stage = sh.vocab ? (float*)b->arena.take((size_t)n * sh.vocab * 4) : nullptr;
    cudaError_t e = cudaMemset(b->arena.base, 0, b->arena.cap);  // tickets and the error word start at 0
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        b->arena.release();
        return cuda_fail(e, "batch workspace");
    }
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_batches.find(key);
    if (it != g_batches.end()) {  // made meanwhile by another thread
        b->arena.release();
        *out = it->second;
        return TASP_OK;
    }
    *out = b.get();
    g_batches.emplace(key, b.release());
    return TASP_OK;
}

// Drop every batch that holds session se (the device is idle).
static void batches_drop(Session* se) {
    std::vector<Batch*> gone;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        for (auto it = g_batches.begin(); it != g_batches.end();) {
            if (std::find(it->first.begin(), it->first.end(), se) != it->first.end()) {
                gone.push_back(it->second);
                it = g_batches.erase(it);
            } else {
                ++it;
            }
        }
    }
    for (Batch* b : gone) batch_free(b);
}

// Device error words of the batches that hold session se.
static std::vector<int*> batch_errors(Session* se) {
    std::vector<int*> out;
    std::lock_guard<std::mutex> lk(g_mu);
    for (auto& kv : g_batches)
        if (std::find(kv.first.begin(), kv.first.end(), se) != kv.first.end()) out.push_back(kv.second->view.err);
    return out;
}

static int check_sessions(tasp_session* const* ss, int n, Plan** plan) {
    if (!ss || n < 1) return fail(TASP_EINVAL, "need at least one session");
    Plan* p = nullptr;
    for (int i = 0; i < n; ++i) {
        Session* se = as_session(ss[i]);
        if (!se) return fail(TASP_EINVAL, "invalid session handle");
        if (!p) p = se->plan;
        if (se->plan != p) return fail(TASP_EMASK, "sessions of different plans in one decode step (a KV cache is "
                                                   "never reused across masks)");
        if (se->pos + 1 > se->max_tokens) return fail(TASP_ECAP, "session KV capacity exhausted");
        for (int j = 0; j < i; ++j)
            if (ss[j] == ss[i]) return fail(TASP_EINVAL, "a session appears twice in one decode step");
    }
    *plan = p;
    return TASP_OK;
}

}  // namespace tasp

using namespace tasp;

// ==================================================================== C ABI
extern "C" {

const char* tasp_last_error(void) { return g_err.c_str(); }
const char* tasp_version(void) { return "tasp-gb300 0.1 (sm_103a)"; }

int tasp_dispatch(const float* h_probs, int32_t n, float tau, int32_t* plan) {
    if (!h_probs || !plan || n < 1) return fail(TASP_EINVAL, "dispatch needs n >= 1 probabilities and an output");
    if (!(tau >= 0.f && tau <= 1.f)) return fail(TASP_EINVAL, "tau must lie in [0, 1]");
    int best = 0;
    for (int i = 0; i < n; ++i) {
        if (!std::isfinite(h_probs[i]) || h_probs[i] < 0.f)
            return fail(TASP_EINVAL, "probabilities must be finite and non-negative");
        if (h_probs[i] > h_probs[best]) best = i;
    }
    *plan = h_probs[best] >= tau ? best : n;
    return TASP_OK;
}

int tasp_test_set_wait_limit(int64_t cycles) {
    if (cycles < 0) return fail(TASP_EINVAL, "negative wait limit");
    test_hooks::g_wait_limit.store(cycles);
    return TASP_OK;
}

int tasp_test_skip_gemv_copies(int32_t launches) {
    if (launches < 0) return fail(TASP_EINVAL, "negative launch count");
    test_hooks::g_skip.store(launches);
    return TASP_OK;
}

int tasp_set_memory_limit(int64_t bytes) {
    if (bytes < 0) return fail(TASP_EINVAL, "memory limit must be >= 0");
    g_arena_limit.store(bytes);
    return TASP_OK;
}

int tasp_memory_in_use(int64_t* bytes) {
    if (!bytes) return fail(TASP_EINVAL, "bytes is NULL");
    *bytes = g_arena_bytes.load();
    return TASP_OK;
}

int tasp_mask_select_qheads(const tasp_model_desc* model, const tasp_mask_desc* mask, int32_t* keep_qheads,
                            int32_t* n_qheads, int32_t* keep_groups, int32_t* n_groups, int32_t* keep_units,
                            int32_t* n_units, int64_t* flops) {
    Shape sh;
    int rc = validate_shape(model, sh, false);
    if (rc) return rc;
    if (!mask) return fail(TASP_EINVAL, "mask_desc is NULL");
    MaskSel sel;
    if ((rc = select_mask(sh, *mask, sel))) return rc;
    size_t og = 0, ou = 0, oq = 0;
    for (int l = 0; l < sh.L; ++l) {
        if (n_groups) n_groups[l] = (int32_t)sel.groups[l].size();
        if (n_units) n_units[l] = (int32_t)sel.units[l].size();
        if (n_qheads) n_qheads[l] = (int32_t)sel.qheads[l].size();
        for (int j : sel.groups[l]) if (keep_groups) keep_groups[og++] = j;
        for (int u : sel.units[l]) if (keep_units) keep_units[ou++] = u;
        for (int h : sel.qheads[l]) if (keep_qheads) keep_qheads[oq++] = h;
        if (flops) flops[l] = sel.layer_flops[l];
    }
    if (flops) {
        flops[sh.L] = sel.total;
        flops[sh.L + 1] = sel.budget;
        flops[sh.L + 2] = sel.dense;
    }
    return TASP_OK;
}

int tasp_plan_layout(const tasp_model_desc* model, const tasp_mask_desc* mask, int32_t layer, int32_t* qkv_src,
                     int32_t* o_src, int16_t* role, int16_t* slot, int16_t* blk_of, int32_t* counts) {
    Shape sh;
    int rc = validate_shape(model, sh, false);
    if (rc) return rc;
    if (!mask || !counts) return fail(TASP_EINVAL, "mask_desc or counts is NULL");
    MaskSel sel;
    if ((rc = select_mask(sh, *mask, sel))) return rc;
    if (layer < 0 || layer >= sh.L) return fail(TASP_EINVAL, "layer out of range");
    LayerPlan lp;
    lp.keep_groups = sel.groups[layer];
    lp.keep_qheads = sel.qheads[layer];
    lp.m_kv = (int)lp.keep_groups.size();
    std::vector<int32_t> hq, ho;
    std::vector<int16_t> hrole, hslot, hblk;
    layer_tables(sh, lp, hq, ho, hrole, hslot, hblk);
    counts[0] = (int32_t)hq.size();
    counts[1] = (int32_t)ho.size();
    counts[2] = (int32_t)hrole.size();
    counts[3] = (int32_t)hslot.size();
    counts[4] = (int32_t)hblk.size();
    if (qkv_src) std::copy(hq.begin(), hq.end(), qkv_src);
    if (o_src) std::copy(ho.begin(), ho.end(), o_src);
    if (role) std::copy(hrole.begin(), hrole.end(), role);
    if (slot) std::copy(hslot.begin(), hslot.end(), slot);
    if (blk_of) std::copy(hblk.begin(), hblk.end(), blk_of);
    return TASP_OK;
}

int tasp_mask_select(const tasp_model_desc* model, const tasp_mask_desc* mask, int32_t* keep_groups,
                     int32_t* n_groups, int32_t* keep_units, int32_t* n_units, int64_t* flops) {
    return tasp_mask_select_qheads(model, mask, nullptr, nullptr, keep_groups, n_groups, keep_units, n_units, flops);
}

int tasp_compile_mask(const tasp_model_desc* model, const tasp_mask_desc* mask, tasp_plan** out) {
    if (!out) return fail(TASP_EINVAL, "out is NULL");
    *out = nullptr;
    Shape sh;
    int rc = validate_shape(model, sh);
    if (rc) return rc;
    if (!mask) return fail(TASP_EINVAL, "mask_desc is NULL");
    if (mask->panel_mode != TASP_PANELS_COMPACT && mask->panel_mode != TASP_PANELS_ROW_INDEXED)
        return fail(TASP_EINVAL, "unknown panel mode");
    MaskSel sel;
    if ((rc = select_mask(sh, *mask, sel))) return rc;
    for (int l = 0; l < sh.L; ++l) {
        if (sel.groups[l].empty() && sel.units[l].empty())
            return fail(TASP_EINVAL, "mask leaves a layer empty (layer " + std::to_string(l) + ")");
    }
    Store* st = nullptr;
    if ((rc = store_acquire(sh, &st))) return rc;
    auto p = std::make_unique<Plan>();
    p->store = st;
    if ((rc = build_plan(*p, sel, mask->panel_mode, mask->kind == TASP_MASK_ALL_KEEP))) {
        p->arena.release();
        store_release(st);
        return rc;
    }
    plan_ledger(*p);
    *out = (tasp_plan*)p.release();
    return TASP_OK;
}

int tasp_session_create(tasp_plan* plan, int32_t max_tokens, tasp_session** out) {
    if (!out) return fail(TASP_EINVAL, "out is NULL");
    *out = nullptr;
    Plan* p = as_plan(plan);
    if (!p) return fail(TASP_EINVAL, "invalid plan handle");
    if (max_tokens < 1) return fail(TASP_EINVAL, "max_tokens must be positive");
    Session* se = nullptr;
    int rc = session_alloc(p, max_tokens, &se);
    if (rc) return rc;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        p->live_sessions++;
    }
    *out = (tasp_session*)se;
    return TASP_OK;
}

int tasp_session_fill_synthetic(tasp_session* s, int32_t t_prior, uint64_t kv_seed, void* stream) {
    Session* se = as_session(s);
    if (!se) return fail(TASP_EINVAL, "invalid session handle");
    if (t_prior < 0 || t_prior > se->max_tokens) return fail(TASP_ECAP, "t_prior exceeds the session capacity");
    int rc = kv_fill_synthetic(*se, t_prior, kv_seed, (cudaStream_t)stream);
    if (rc) return rc;
    se->pos = t_prior;
    return TASP_OK;
}

int tasp_session_position(const tasp_session* s, int32_t* pos) {
    Session* se = as_session((void*)s);
    if (!se || !pos) return fail(TASP_EINVAL, "invalid session handle or NULL output");
    *pos = se->pos;
    return TASP_OK;
}

int tasp_session_status(tasp_session* s, int32_t clear, int32_t* device_error) {
    Session* se = as_session(s);
    if (!se || !device_error) return fail(TASP_EINVAL, "invalid session handle or NULL output");
    TASP_CUDA(cudaDeviceSynchronize());
    std::vector<int*> words = batch_errors(se);
    words.push_back(se->err);
    int v = 0;
    for (int* w : words) {
        int x = 0;
        TASP_CUDA(cudaMemcpy(&x, w, sizeof(int), cudaMemcpyDeviceToHost));
        if (clear) TASP_CUDA(cudaMemset(w, 0, sizeof(int)));
        v |= x;
    }
    *device_error = v;
    return TASP_OK;
}

int tasp_decode_step(tasp_session* const* sessions, int32_t n, const void* d_x_bf16, float* d_hidden_out,
                     float* d_logits, void* stream) {
    int rc = check_aligned({{d_x_bf16, 2}, {d_hidden_out, 4}, {d_logits, 4}});
    if (rc) return rc;
    Plan* p = nullptr;
    rc = check_sessions(sessions, n, &p);
    if (rc) return rc;
    if (!d_x_bf16) return fail(TASP_EINVAL, "d_x_bf16 is NULL");
    const Shape& sh = p->store->sh;
    if (d_logits && sh.vocab == 0) return fail(TASP_EINVAL, "logits requested from a model without LM head");
    Session* const* ss = (Session* const*)sessions;
    cudaStream_t st = (cudaStream_t)stream;
    // groups of up to MAX_BATCH sessions share each weight pass
    for (int i0 = 0; i0 < n; i0 += MAX_BATCH) {
        const int m = std::min(MAX_BATCH, n - i0);
        Batch* b = nullptr;
        if (m > 1 && (rc = batch_get(ss + i0, m, &b))) return rc;
        // the inputs go through the group's fixed staging buffer, so the recorded step graph
        // depends only on the output buffers and stays valid while callers vary the inputs
        uint16_t* xs = m == 1 ? ss[i0]->x_stage : b->x_stage;
        TASP_CUDA(cudaMemcpyAsync(xs, (const uint16_t*)d_x_bf16 + (size_t)i0 * sh.d, (size_t)m * sh.d * 2,
                                  cudaMemcpyDeviceToDevice, st));
        StepTarget t;
        t.x_in = xs;
        t.hidden_out = d_hidden_out ? d_hidden_out + (size_t)i0 * sh.d : nullptr;
        t.logits = d_logits ? d_logits + (size_t)i0 * sh.vocab : nullptr;
        StepGraph* g = nullptr;
        if (m == 1) {
            if ((rc = session_graph(*ss[i0], t))) return rc;
            g = &ss[i0]->graph;
        } else {
            if ((rc = record_graph(b->graph, b->view, t))) return rc;
            g = &b->graph;
        }
        TASP_CUDA(cudaGraphLaunch(g->exec, st));
        for (int i = i0; i < i0 + m; ++i) ss[i]->pos += 1;
    }
    return TASP_OK;
}

int tasp_decode_step_host(tasp_session* const* sessions, int32_t n, const void* h_x_bf16, float* h_hidden_out,
                          float* h_logits, void* stream) {
    Plan* p = nullptr;
    int rc = check_sessions(sessions, n, &p);
    if (rc) return rc;
    if (!h_x_bf16) return fail(TASP_EINVAL, "h_x_bf16 is NULL");
    const Shape& sh = p->store->sh;
    if (h_logits && sh.vocab == 0) return fail(TASP_EINVAL, "logits requested from a model without LM head");
    cudaStream_t st = (cudaStream_t)stream;
    Session* const* ss = (Session* const*)sessions;
    for (int i0 = 0; i0 < n; i0 += MAX_BATCH) {
        const int m = std::min(MAX_BATCH, n - i0);
        uint16_t* xs;
        float *hs, *ls;
        StepGraph* g = nullptr;
        Batch* b = nullptr;
        if (m == 1) {
            xs = ss[i0]->x_stage;
            hs = ss[i0]->hidden_stage;
            ls = ss[i0]->logits_stage;
        } else {
            if ((rc = batch_get(ss + i0, m, &b))) return rc;
            xs = b->x_stage;
            hs = b->hidden_stage;
            ls = b->logits_stage;
        }
        TASP_CUDA(cudaMemcpyAsync(xs, (const uint16_t*)h_x_bf16 + (size_t)i0 * sh.d, (size_t)m * sh.d * 2,
                                  cudaMemcpyHostToDevice, st));
        StepTarget t;
        t.x_in = xs;
        t.hidden_out = h_hidden_out ? hs : nullptr;
        t.logits = h_logits ? ls : nullptr;
        if (m == 1) {
            if ((rc = session_graph(*ss[i0], t))) return rc;
            g = &ss[i0]->graph;
        } else {
            if ((rc = record_graph(b->graph, b->view, t))) return rc;
            g = &b->graph;
        }
        TASP_CUDA(cudaGraphLaunch(g->exec, st));
        for (int i = i0; i < i0 + m; ++i) ss[i]->pos += 1;
        if (h_hidden_out)
            TASP_CUDA(cudaMemcpyAsync(h_hidden_out + (size_t)i0 * sh.d, hs, (size_t)m * sh.d * 4,
                                      cudaMemcpyDeviceToHost, st));
        if (h_logits)
            TASP_CUDA(cudaMemcpyAsync(h_logits + (size_t)i0 * sh.vocab, ls, (size_t)m * sh.vocab * 4,
                                      cudaMemcpyDeviceToHost, st));
    }
    TASP_CUDA(cudaStreamSynchronize(st));
    return TASP_OK;
}

int tasp_prefill(tasp_plan* plan, const void* d_embeds_bf16, int32_t T, int32_t max_new_tokens, void* stream,
                 tasp_session** out, float* d_logits_last) {
    if (!out) return fail(TASP_EINVAL, "out is NULL");
    *out = nullptr;
    if (int rc = check_aligned({{d_embeds_bf16, 2}, {d_logits_last, 4}})) return rc;
    Plan* p = as_plan(plan);
    if (!p) return fail(TASP_EINVAL, "invalid plan handle");
    if (!d_embeds_bf16 || T < 1 || max_new_tokens < 0) return fail(TASP_EINVAL, "bad prompt (NULL or T < 1)");
    const Shape& sh = p->store->sh;
    if (d_logits_last && sh.vocab == 0) return fail(TASP_EUNSUP, "logits requested from a model without LM head");
    if (sh.d % 8) return fail(TASP_EUNSUP, "prefill needs d % 8 == 0");
    Session* se = nullptr;
    int rc = session_alloc(p, T + max_new_tokens, &se);
    if (rc) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    rc = prefill_run(*se, (const uint16_t*)d_embeds_bf16, T, st);
    if (!rc) rc = enqueue_set_pos(*se, T, st);
    if (!rc && d_logits_last) rc = enqueue_lm_head(*se, d_logits_last, st);
    if (rc) {
        cudaStreamSynchronize(st);
        session_free(se);
        return rc;
    }
    se->pos = T;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        p->live_sessions++;
    }
    *out = (tasp_session*)se;
    return TASP_OK;
}

int tasp_session_prefill(tasp_session* s, const void* d_embeds_bf16, int32_t T, void* stream, float* d_logits_last) {
    if (int rc = check_aligned({{d_embeds_bf16, 2}, {d_logits_last, 4}})) return rc;
    Session* se = as_session(s);
    if (!se) return fail(TASP_EINVAL, "invalid session handle");
    const Shape& sh = se->plan->store->sh;
    if (!d_embeds_bf16 || T < 1) return fail(TASP_EINVAL, "bad prompt (NULL or T < 1)");
    if (T > se->max_tokens) return fail(TASP_ECAP, "prompt longer than the session capacity");
    if (d_logits_last && sh.vocab == 0) return fail(TASP_EUNSUP, "logits requested from a model without LM head");
    if (sh.d % 8) return fail(TASP_EUNSUP, "prefill needs d % 8 == 0");
    cudaStream_t st = (cudaStream_t)stream;
    int rc = prefill_run(*se, (const uint16_t*)d_embeds_bf16, T, st);
    if (!rc) rc = enqueue_set_pos(*se, T, st);
    if (!rc && d_logits_last) rc = enqueue_lm_head(*se, d_logits_last, st);
    if (rc) return rc;
    se->pos = T;
    return TASP_OK;
}

int tasp_session_kv_export(const tasp_session* s, int32_t layer, int32_t which, void* h_dst, size_t bytes) {
    Session* se = as_session((void*)s);
    if (!se || !h_dst) return fail(TASP_EINVAL, "invalid session or NULL destination");
    const Shape& sh = se->plan->store->sh;
    if (layer < 0 || layer >= sh.L || (which != 0 && which != 1)) return fail(TASP_EINVAL, "bad layer or item");
    const int m = se->plan->layers[layer].m_kv;
    const size_t row = (size_t)sh.dh * 2;
    if (bytes != (size_t)m * se->pos * row)
        return fail(TASP_EINVAL, "kv export size mismatch: expected " + std::to_string((size_t)m * se->pos * row));
    if (bytes == 0) return TASP_OK;
    TASP_CUDA(cudaDeviceSynchronize());
    const uint16_t* src = which == 0 ? se->K[layer] : se->V[layer];
    TASP_CUDA(cudaMemcpy2D(h_dst, (size_t)se->pos * row, src, (size_t)se->max_tokens * row, (size_t)se->pos * row, m,
                           cudaMemcpyDeviceToHost));
    return TASP_OK;
}

int tasp_release(void* handle) {
    if (!handle) return TASP_OK;
    if (Session* se = as_session(handle)) {
        cudaError_t e = cudaDeviceSynchronize();
        batches_drop(se);
        union_drop(se);
        {
            std::lock_guard<std::mutex> lk(g_mu);
            se->plan->live_sessions--;
        }
        session_free(se);
        if (e != cudaSuccess) return cuda_fail(e, "tasp_release");
        return TASP_OK;
    }
    if (Plan* p = as_plan(handle)) {
        {
            std::lock_guard<std::mutex> lk(g_mu);
            if (p->live_sessions > 0) return fail(TASP_EBUSY, "plan still has live sessions");
        }
        cudaError_t e = cudaDeviceSynchronize();
        p->arena.release();
        p->f16_arena.release();
        store_release(p->store);
        p->magic = 0;
        delete p;
        if (e != cudaSuccess) return cuda_fail(e, "tasp_release");
        return TASP_OK;
    }
    return fail(TASP_EINVAL, "unknown handle");
}

int tasp_plan_info_get(const tasp_plan* plan, tasp_plan_info* out) {
    Plan* p = as_plan((void*)plan);
    if (!p || !out) return fail(TASP_EINVAL, "invalid plan handle or NULL output");
    out->L = p->store->sh.L;
    out->panel_bytes = (int64_t)p->arena.cap;
    out->store_bytes = (int64_t)p->store->bytes;
    out->weight_bytes_per_token = p->weight_bytes_per_token;
    out->flops_retained = p->flops_retained;
    out->flops_dense = p->flops_dense;
    out->launched_flops = p->launched_flops;
    return TASP_OK;
}

int tasp_plan_layer_dims(const tasp_plan* plan, int32_t layer, int32_t* out2) {
    Plan* p = as_plan((void*)plan);
    if (!p || !out2 || layer < 0 || layer >= (int)p->layers.size()) return fail(TASP_EINVAL, "bad plan or layer");
    out2[0] = p->layers[layer].m_kv;
    out2[1] = p->layers[layer].c;
    return TASP_OK;
}

int tasp_plan_layer_qheads(const tasp_plan* plan, int32_t layer, int32_t* m_q) {
    Plan* p = as_plan((void*)plan);
    if (!p || !m_q || layer < 0 || layer >= (int)p->layers.size()) return fail(TASP_EINVAL, "bad plan or layer");
    *m_q = p->layers[layer].m_q;
    return TASP_OK;
}

int tasp_plan_export(const tasp_plan* plan, int32_t layer, int32_t item, void* h_dst, size_t bytes) {
    Plan* p = as_plan((void*)plan);
    if (!p || !h_dst || layer < 0 || layer >= (int)p->layers.size()) return fail(TASP_EINVAL, "bad plan, layer or dst");
    const LayerPlan& lp = p->layers[layer];
    const Shape& sh = p->store->sh;
    const size_t d = sh.d;
    auto need = [&](size_t b) { return b == bytes ? TASP_OK : fail(TASP_EINVAL, "export size mismatch: expected " +
                                                                                std::to_string(b)); };
    auto rows_out = [&](const int8_t* w, const int32_t* map, int rows) -> int {
        if (int rc = need((size_t)rows * d)) return rc;
        if (!map) {
            TASP_CUDA(cudaMemcpy(h_dst, w, (size_t)rows * d, cudaMemcpyDeviceToHost));
            return TASP_OK;
        }
        int8_t* tmp = nullptr;
        TASP_CUDA(cudaMalloc((void**)&tmp, std::max<size_t>(16, (size_t)rows * d)));
        int rc = gather_rows(tmp, w, map, rows, (int)d, 0);
        cudaError_t e = cudaMemcpy(h_dst, tmp, (size_t)rows * d, cudaMemcpyDeviceToHost);
        cudaFree(tmp);
        if (rc) return rc;
        if (e != cudaSuccess) return cuda_fail(e, "export");
        return TASP_OK;
    };
    auto cols_out = [&](const int8_t* w, int ld, int K) -> int {
        if (int rc = need(d * (size_t)K)) return rc;
        if (K == 0) return TASP_OK;
        TASP_CUDA(cudaMemcpy2D(h_dst, K, w, ld, K, d, cudaMemcpyDeviceToHost));
        return TASP_OK;
    };
    auto f32_out = [&](const float* v, size_t n) -> int {
        if (int rc = need(n * 4)) return rc;
        if (n) TASP_CUDA(cudaMemcpy(h_dst, v, n * 4, cudaMemcpyDeviceToHost));
        return TASP_OK;
    };
    switch (item) {
        case TASP_EXPORT_KEEP_GROUPS: {
            if (int rc = need(lp.keep_groups.size() * 4)) return rc;
            std::memcpy(h_dst, lp.keep_groups.data(), bytes);
            return TASP_OK;
        }
        case TASP_EXPORT_QKV_G:
        case TASP_EXPORT_O_G:
        case TASP_EXPORT_GU_G:
        case TASP_EXPORT_DOWN_G: {
            if (!sh.qg) return fail(TASP_EINVAL, "the store has no group scales");
            const uint16_t* src = item == TASP_EXPORT_QKV_G ? lp.qkv_g : item == TASP_EXPORT_O_G ? lp.o_g
                                : item == TASP_EXPORT_GU_G ? lp.gu_g : lp.dn_g;
            const int gld = item == TASP_EXPORT_QKV_G ? lp.qkv_gld : item == TASP_EXPORT_O_G ? lp.o_gld
                          : item == TASP_EXPORT_GU_G ? lp.gu_gld : lp.dn_gld;
            const size_t rows = item == TASP_EXPORT_QKV_G ? (size_t)lp.qkv_rows : item == TASP_EXPORT_GU_G ? (size_t)lp.gu_rows
                                                                                                          : (size_t)d;
            const size_t cols = item == TASP_EXPORT_QKV_G || item == TASP_EXPORT_GU_G ? (size_t)(d / sh.qg)
                              : item == TASP_EXPORT_O_G ? (size_t)(lp.o_K / sh.qg) : (size_t)(lp.dn_K / sh.qg);
            if (int rc = need(rows * cols * 2)) return rc;
            if (rows * cols)
                TASP_CUDA(cudaMemcpy2D(h_dst, cols * 2, src, (size_t)gld * 2, cols * 2, rows, cudaMemcpyDeviceToHost));
            return TASP_OK;
        }
        case TASP_EXPORT_KEEP_QHEADS: {
            if (int rc = need(lp.keep_qheads.size() * 4)) return rc;
            std::memcpy(h_dst, lp.keep_qheads.data(), bytes);
            return TASP_OK;
        }
        case TASP_EXPORT_KEEP_CHANS: {
            if (int rc = need(lp.keep_chans.size() * 4)) return rc;
            std::memcpy(h_dst, lp.keep_chans.data(), bytes);
            return TASP_OK;
        }
        case TASP_EXPORT_QKV_W: return rows_out(lp.qkv_w, lp.qkv_map, lp.qkv_rows);
        case TASP_EXPORT_QKV_S: return f32_out(lp.qkv_s, lp.qkv_rows);
        case TASP_EXPORT_O_W: return cols_out(lp.o_w, lp.o_ld, lp.o_K);
        case TASP_EXPORT_O_S: return f32_out(lp.o_s, d);
        case TASP_EXPORT_GU_W: return rows_out(lp.gu_w, lp.gu_map, lp.gu_rows);
        case TASP_EXPORT_GU_S: return f32_out(lp.gu_s, lp.gu_rows);
        case TASP_EXPORT_DOWN_W: return cols_out(lp.dn_w, lp.dn_ld, lp.dn_K);
        case TASP_EXPORT_DOWN_S: return f32_out(lp.dn_s, d);
        default: return fail(TASP_EINVAL, "unknown export item");
    }
}

int tasp_layer_step(tasp_session* s, int32_t layer, const float* d_x_in, float* d_x_out, void* stream) {
    if (int rc = check_aligned({{d_x_in, 4}, {d_x_out, 4}})) return rc;
    Session* se = as_session(s);
    if (!se || !d_x_in || !d_x_out) return fail(TASP_EINVAL, "invalid session or NULL buffers");
    const Shape& sh = se->plan->store->sh;
    if (layer < 0 || layer >= sh.L) return fail(TASP_EINVAL, "layer out of range");
    if (se->pos + 1 > se->max_tokens) return fail(TASP_ECAP, "session KV capacity exhausted");
    cudaStream_t st = (cudaStream_t)stream;
    TASP_CUDA(cudaMemcpyAsync(se->x, d_x_in, (size_t)sh.d * 4, cudaMemcpyDeviceToDevice, st));
    StepTarget t;
    t.advance = false;
    int rc = enqueue_step(*se, t, st, layer, nullptr, nullptr, nullptr);
    if (rc) return rc;
    TASP_CUDA(cudaMemcpyAsync(d_x_out, se->x, (size_t)sh.d * 4, cudaMemcpyDeviceToDevice, st));
    return TASP_OK;
}

struct ProfCtx {
    cudaStream_t s;
    std::vector<cudaEvent_t> ev;
    std::vector<int> kind;
    int err = 0;
};

static void prof_hook(void* c, int kind, bool before) {
    ProfCtx* pc = (ProfCtx*)c;
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) {
        pc->err = 1;
        return;
    }
    cudaEventRecord(e, pc->s);
    pc->ev.push_back(e);
    pc->kind.push_back(before ? -1 : kind);
}

int tasp_profile_step(tasp_session* const* sessions, int32_t n, const void* d_x_bf16, float* d_logits, void* stream,
                      float* h_ms, int32_t* h_count) {
    int rc = check_aligned({{d_x_bf16, 2}, {d_logits, 4}});
    if (rc) return rc;
    Plan* p = nullptr;
    rc = check_sessions(sessions, n, &p);
    if (rc) return rc;
    if (!h_ms || !h_count || !d_x_bf16) return fail(TASP_EINVAL, "NULL buffers");
    const Shape& sh = p->store->sh;
    for (int k = 0; k < TASP_KERNEL_KINDS; ++k) { h_ms[k] = 0.f; h_count[k] = 0; }
    Session* const* ss = (Session* const*)sessions;
    for (int i0 = 0; i0 < n; i0 += MAX_BATCH) {
        const int m = std::min(MAX_BATCH, n - i0);
        BatchView bv;
        if (m == 1) {
            bv = single_view(*ss[i0]);
        } else {
            Batch* b = nullptr;
            if ((rc = batch_get(ss + i0, m, &b))) return rc;
            bv = b->view;
        }
        ProfCtx pc;
        pc.s = (cudaStream_t)stream;
        StepTarget t;
        t.x_in = (const uint16_t*)d_x_bf16 + (size_t)i0 * sh.d;
        t.logits = d_logits ? d_logits + (size_t)i0 * sh.vocab : nullptr;
        rc = enqueue_batch(bv, t, pc.s, -1, prof_hook, &pc, nullptr);
        cudaError_t e = cudaStreamSynchronize(pc.s);
        if (!rc && e == cudaSuccess && !pc.err) {
            for (size_t j = 0; j + 1 < pc.ev.size(); j += 2) {
                float ms = 0.f;
                cudaEventElapsedTime(&ms, pc.ev[j], pc.ev[j + 1]);
                int k = pc.kind[j + 1];
                h_ms[k] += ms;
                h_count[k] += 1;
            }
            for (int i = i0; i < i0 + m; ++i) ss[i]->pos += 1;
        }
        for (cudaEvent_t ev : pc.ev) cudaEventDestroy(ev);
        if (rc) return rc;
        if (e != cudaSuccess) return cuda_fail(e, "profile step");
        if (pc.err) return fail(TASP_ECUDA, "event creation failed");
    }
    return TASP_OK;
}

int tasp_step_launches(tasp_session* const* sessions, int32_t n, int32_t with_logits, int32_t* out) {
    Plan* p = nullptr;
    int rc = check_sessions(sessions, n, &p);
    if (rc) return rc;
    if (!out) return fail(TASP_EINVAL, "NULL output");
    int per = 0;
    for (const LayerPlan& lp : p->layers) per += 1 + (lp.m_kv ? 2 : 0) + (lp.c ? 2 : 0);
    per += (with_logits && p->store->sh.vocab ? 1 : 0) + 1;
    *out = per * ((n + MAX_BATCH - 1) / MAX_BATCH);  // one launch sequence per group of <= 4
    return TASP_OK;
}

}  // extern "C"
