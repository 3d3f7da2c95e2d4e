// Decode step of the compiled sparse path (Sec. 3.3, Fig. 1): the launch sequence of
// one token for n <= 4 sessions of one plan, sm_103a.
//
// Per layer: K1 RMSNorm + QKV GEMV + RoPE + KV append, K2 GQA attention over the kept
// KV groups (attention.cu), K3 O GEMV + residual, K4 RMSNorm + gate/up GEMV +
// SiLU(gate) * up, K5 down GEMV + residual; then the final RMSNorm + dense LM head and the
// position advance. The GEMVs (gemv.cuh) read every weight byte once for all sessions of
// the batch; attention runs one grid over all of them, each on its own KV cache and
// position. Consecutive kernels overlap through programmatic dependent launch, and the
// runtime replays the whole sequence as one CUDA graph.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>
#include <vector>

#include "gemv.cuh"
#include "tasp_internal.h"

namespace tasp {

namespace {

using namespace gemv;

__global__ void set_pos_kernel(int* pos, int v) {
    if (threadIdx.x == 0) *pos = v;
}

struct AdvanceArgs {
    int* pos[MAX_BATCH];
    int n;
};

__global__ void advance_kernel(AdvanceArgs a) {
    pdl_wait();
    pdl_trigger();
    if (threadIdx.x < a.n) *a.pos[threadIdx.x] += 1;
}

// ---------------------------------------------------------------- host side
template <typename Kern, typename Arg>
int launch_pdl(Kern k, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const Arg& a) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    TASP_CUDA(cudaLaunchKernelEx(&cfg, k, a));
    return TASP_OK;
}

Fn pick_any(int nbk, int mode, int R, int XC, bool gs) {
    switch (nbk) {
        case 1: return pick<1>(mode, R, XC, gs);
        case 2: return pick<2>(mode, R, XC, gs);
        default: return pick<4>(mode, R, XC, gs);
    }
}

// Kernel shape for a launch: NB (vectors per weight pass), XC (register chunks per
// thread, NB * XC <= 4), the K pass length and R (rows per stage, <= 32 KB per stage,
// pairs for the rotary / SwiGLU modes).
struct Variant {
    int nbk, XC, R, seg, passes;
};

Variant variant(int mode, int nb, int nchunks, int max_r) {
    Variant v;
    v.nbk = nb <= 1 ? 1 : (nb <= 2 ? 2 : 4);
    const int xc_max = 4 / v.nbk;
    v.XC = 1;
    while (v.XC < xc_max && v.XC * CT < nchunks) v.XC <<= 1;
    v.seg = std::min(nchunks, v.XC * CT);
    v.passes = (nchunks + v.seg - 1) / v.seg;
    int R = 8;
    while (R > 1 && R * v.seg * 16 > 32768) R >>= 1;
    if ((mode == M_QKV || mode == M_GU) && R < 2) R = 2;
    R = std::min(R, max_r);
    if (v.XC == 2) R = std::min(R, 4);
    if (v.XC == 4) R = std::min(R, 2);
    if (v.nbk == 4) R = std::min(R, 4);
    v.R = R;
    return v;
}

std::mutex g_attr_mu;
std::map<const void*, int> g_attr;  // kernel -> dynamic shared memory cap

int launch_gemv(int mode, Params p, cudaStream_t s) {
    if (p.rows == 0 || p.nb == 0) return TASP_OK;
    if (p.nb > MAXNB) return fail(TASP_EINVAL, "more activation vectors than one GEMV pass takes");
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    const Variant v = variant(mode, p.nb, p.nchunks, 8);
    if ((mode == M_QKV || mode == M_GU) && v.passes > 1)
        return fail(TASP_EUNSUP, "hidden size too large for the register-resident activation slices of this batch");
    if (p.gscale && (v.nbk == 1 || mode == M_LM))
        return fail(TASP_EINVAL, "grouped scales on a one-vector or LM-head batched GEMV");
    Fn fn = pick_any(v.nbk, mode, v.R, v.XC, p.gscale != nullptr);
    if (!fn) return fail(TASP_EINVAL, "no GEMV variant for this row length");
    p.seg = v.seg;
    p.passes = v.passes;
    {
        std::lock_guard<std::mutex> lk(g_attr_mu);
        auto it = g_attr.find((const void*)fn);
        if (it == g_attr.end()) {
            cudaFuncAttributes fa;
            TASP_CUDA(cudaFuncGetAttributes(&fa, fn));
            const int cap = di.smem_optin - (int)fa.sharedSizeBytes - 128;
            TASP_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, cap));
            it = g_attr.emplace((const void*)fn, cap).first;
        }
        p.smem_cap = it->second;
    }
    const Smem L = smem_plan(v.R, v.seg * 16, p.smem_cap);
    if (L.nstages < 2) return fail(TASP_EUNSUP, "row too long for the shared-memory ring");
    const int NG = (p.rows + v.R - 1) / v.R;
    const int grid = std::max(1, std::min(NG, di.sms));
    if (mode != M_LM && (int64_t)((NG + grid - 1) / grid) * v.R > EPI_MAXR)
        return fail(TASP_EUNSUP, "more output rows per CTA than the epilogue stages");
    return launch_pdl(fn, dim3(grid), dim3(THREADS), (size_t)L.total, s, p);
}

Params lm_params(const BatchView& bv, float* logits, int64_t logit_stride) {
    const Plan& pl = *bv.ss[0]->plan;
    const Shape& sh = pl.store->sh;
    Params lm{};
    lm.w = reinterpret_cast<const int8_t*>(pl.store->lm_head);
    lm.ld = (int64_t)sh.d * 2;
    lm.rows = sh.vocab;
    lm.K = sh.d;
    lm.nchunks = sh.d / 8;
    lm.nb = bv.n;
    lm.x_resid = bv.x;
    lm.x_stride = bv.x_stride;
    lm.gamma = pl.store->g_final;
    lm.eps = sh.eps;
    lm.logits = logits;
    lm.logit_stride = logit_stride;
    lm.err = bv.err;
    return lm;
}

// One launch of a decode step.
struct Op {
    enum Type { GEMV, ATTN, COPY_HIDDEN, ADVANCE } type;
    int kind;  // KernelKind reported to the profiling hook
    int mode = 0;
    Params p{};
    AttnParams a{};
    int m_kv = 0, S = 0, cs = 16;
};

}  // namespace

BatchView single_view(Session& se) {
    const Shape& sh = se.plan->store->sh;
    BatchView bv;
    bv.n = 1;
    bv.ss[0] = &se;
    bv.x = se.x;
    bv.q = se.q;
    bv.o = se.o;
    bv.h = se.h;
    bv.x_stride = sh.d;
    bv.q_stride = (int64_t)sh.Hq * sh.dh;
    bv.h_stride = sh.df;
    bv.part = se.part;
    bv.ml = se.ml;
    bv.cnt = se.cnt;
    bv.err = se.err;
    return bv;
}

int batch_attn_slots(const Plan& p, const Session* const* ss, int n, int sms) {
    const Shape& sh = p.store->sh;
    int smax = 1;
    for (int b = 0; b < n; ++b)
        for (const LayerPlan& lp : p.layers)
            smax = std::max(smax, attn_splits(lp.m_kv, ss[b]->max_tokens, sms, sh.dh, sh.g(), 8) / 8);  // either size
    return smax;
}

int enqueue_batch(const BatchView& bv, const StepTarget& t, cudaStream_t s, int only_layer, KernelHook hook,
                  void* ctx, int* launches) {
    if (bv.n < 1 || bv.n > MAX_BATCH) return fail(TASP_EINVAL, "a batch holds 1 to 4 sessions");
    const Plan& pl = *bv.ss[0]->plan;
    const Shape& sh = pl.store->sh;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    const int n = bv.n;
    std::vector<Op> ops;
    const int l_begin = only_layer >= 0 ? only_layer : 0;
    const int l_end = only_layer >= 0 ? only_layer + 1 : sh.L;
    auto gemv = [&](int kind, int mode, const Params& p) {
        Op op;
        op.type = Op::GEMV;
        op.kind = kind;
        op.mode = mode;
        op.p = p;
        ops.push_back(op);
    };
    // groupwise store: the row's BF16 scale of each column group of `cols` input columns
    auto set_groups = [&](Params& q, const uint16_t* gs, int cols, int gld) {
        if (!sh.qg) return;
        q.gscale = gs;
        q.gcols = cols / sh.qg;
        q.gld = gld;
        int sft = 0;
        while ((16 << sft) < sh.qg) ++sft;
        q.gshift = sft;
    };
    for (int l = l_begin; l < l_end; ++l) {
        const LayerPlan& lp = pl.layers[l];
        const bool first = (l == 0) && t.x_in != nullptr;
        // K1: RMSNorm + QKV GEMV + RoPE + KV append
        Params p{};
        p.w = lp.qkv_w;
        p.map = lp.qkv_map;
        p.scale = lp.qkv_s;
        p.ld = sh.d;
        p.rows = lp.qkv_rows;
        p.K = sh.d;
        p.nchunks = sh.d / 16;
        p.nb = n;
        p.x_resid = bv.x;
        p.x_stride = bv.x_stride;
        p.x_in = first ? t.x_in : nullptr;
        p.xin_stride = sh.d;
        p.x_resid_init = first ? bv.x : nullptr;
        p.gamma = lp.g_attn;
        p.eps = sh.eps;
        p.q_out = bv.q;
        p.q_stride = bv.q_stride;
        for (int b = 0; b < n; ++b) {
            const Session& se = *bv.ss[b];
            p.k_cache[b] = se.K[l];
            p.v_cache[b] = se.V[l];
            p.max_tokens[b] = se.max_tokens;
            p.rope[b] = se.rope;
            p.pos[b] = se.d_pos;
        }
        p.g = sh.g();
        p.dh = sh.dh;
        p.blk_role = lp.blk_role;
        set_groups(p, lp.qkv_g, sh.d, lp.qkv_gld);
        p.err = bv.err;
        gemv(K_QKV, M_QKV, p);
        // K2: split-KV attention over the retained KV heads of every session
        if (lp.m_kv > 0) {
            AttnParams a{};
            a.q = bv.q;
            a.o = bv.o;
            a.q_stride = bv.q_stride;
            int S = 0, mt = 0;
            for (int b = 0; b < n; ++b) mt = std::max(mt, bv.ss[b]->max_tokens);
            const int cs = attn_cluster_for(lp.m_kv, n, mt, sh.dh, sh.g(), n <= MAX_BATCH);
            for (int b = 0; b < n; ++b) {
                const Session& se = *bv.ss[b];
                a.K[b] = se.K[l];
                a.V[b] = se.V[l];
                a.pos[b] = se.d_pos;
                a.max_tokens[b] = se.max_tokens;
                a.m_kv[b] = lp.m_kv;
                a.oslot[b] = lp.oslot;
                S = std::max(S, attn_splits(lp.m_kv, se.max_tokens, di.sms, sh.dh, sh.g(), cs));
            }
            a.qscale = (float)(1.0 / std::sqrt((double)sh.dh) * 1.4426950408889634);
            a.tma = 1;
            for (int b = 0; b < n; ++b) {
                a.tmK[b] = bv.ss[b]->tmK[l];
                a.tmV[b] = bv.ss[b]->tmV[l];
            }
            a.err = bv.err;
            a.part = t.att_part ? t.att_part : bv.part;
            a.ml = t.att_ml ? t.att_ml : bv.ml;
            a.cnt = t.att_cnt ? t.att_cnt : bv.cnt;
            a.part_stride = bv.part_stride;
            a.ml_stride = bv.ml_stride;
            a.cnt_stride = bv.cnt_stride;
            Op op;
            op.type = Op::ATTN;
            op.kind = K_ATTN;
            op.a = a;
            op.m_kv = lp.m_kv;
            op.S = S;
            op.cs = cs;
            ops.push_back(op);
        }
        // K3: O-projection + residual
        if (lp.m_kv > 0) {
            Params o{};
            o.w = lp.o_w;
            o.scale = lp.o_s;
            o.ld = lp.o_ld;
            o.rows = sh.d;
            o.K = lp.o_K;
            o.nchunks = lp.o_ld / 16;
            o.nb = n;
            o.act = bv.o;
            o.act_stride = bv.q_stride;
            o.resid_out = bv.x;
            o.x_stride = bv.x_stride;
            set_groups(o, lp.o_g, lp.o_K, lp.o_gld);
            o.err = bv.err;
            gemv(K_O, M_O, o);
        }
        // K4: RMSNorm + gate/up GEMV + SiLU(gate) * up
        const bool last = (l == sh.L - 1) && only_layer < 0;
        if (lp.c > 0) {
            Params gu{};
            gu.w = lp.gu_w;
            gu.map = lp.gu_map;
            gu.scale = lp.gu_s;
            gu.ld = sh.d;
            gu.rows = lp.gu_rows;
            gu.K = sh.d;
            gu.nchunks = sh.d / 16;
            gu.nb = n;
            gu.x_resid = bv.x;
            gu.x_stride = bv.x_stride;
            gu.gamma = lp.g_mlp;
            gu.eps = sh.eps;
            gu.h_out = bv.h;
            gu.h_stride = bv.h_stride;
            set_groups(gu, lp.gu_g, sh.d, lp.gu_gld);
            gu.err = bv.err;
            gemv(K_GU, M_GU, gu);
            // K5: down projection + residual
            Params dn{};
            dn.w = lp.dn_w;
            dn.scale = lp.dn_s;
            dn.ld = lp.dn_ld;
            dn.rows = sh.d;
            dn.K = lp.dn_K;
            dn.nchunks = lp.dn_ld / 16;
            dn.nb = n;
            dn.act = bv.h;
            dn.act_stride = bv.h_stride;
            dn.resid_out = bv.x;
            dn.x_stride = bv.x_stride;
            dn.hidden_out = last ? t.hidden_out : nullptr;
            dn.hid_stride = sh.d;
            set_groups(dn, lp.dn_g, lp.dn_K, lp.dn_gld);
            dn.err = bv.err;
            gemv(K_DOWN, M_DOWN, dn);
        } else if (last && t.hidden_out) {
            Op op;
            op.type = Op::COPY_HIDDEN;
            op.kind = K_OTHER;
            ops.push_back(op);
        }
    }
    if (only_layer < 0) {
        if (t.logits) gemv(K_LM, M_LM, lm_params(bv, t.logits, sh.vocab));
        if (t.advance) {
            Op op;
            op.type = Op::ADVANCE;
            op.kind = K_OTHER;
            ops.push_back(op);
        }
    }
    int nl = 0;
    for (const Op& op : ops) {
        if (hook) hook(ctx, op.kind, true);
        switch (op.type) {
            case Op::GEMV:
                rc = op.p.nb == 1 ? launch_gemv_single(op.mode, op.p, s) : launch_gemv(op.mode, op.p, s);
                break;
            case Op::ATTN:
                rc = launch_attention(op.a, sh.dh, sh.g(), op.m_kv, op.S, n, s, op.cs);
                break;
            case Op::COPY_HIDDEN: {
                const cudaError_t e = cudaMemcpy2DAsync(t.hidden_out, (size_t)sh.d * 4, bv.x, (size_t)bv.x_stride * 4,
                                                        (size_t)sh.d * 4, n, cudaMemcpyDeviceToDevice, s);
                rc = e == cudaSuccess ? TASP_OK : cuda_fail(e, "hidden state copy");
                break;
            }
            case Op::ADVANCE: {
                AdvanceArgs aa{};
                aa.n = n;
                for (int b = 0; b < n; ++b) aa.pos[b] = bv.ss[b]->d_pos;
                rc = launch_pdl(advance_kernel, dim3(1), dim3(32), 0, s, aa);
                break;
            }
        }
        if (rc) return rc;
        if (hook) hook(ctx, op.kind, false);
        if (op.type != Op::COPY_HIDDEN) ++nl;
    }
    if (launches) *launches = nl;
    return TASP_OK;
}

int enqueue_step(Session& se, const StepTarget& t, cudaStream_t s, int only_layer, KernelHook hook, void* ctx,
                 int* launches) {
    return enqueue_batch(single_view(se), t, s, only_layer, hook, ctx, launches);
}

int enqueue_lm_heads(const BatchView& bv, float* logits, cudaStream_t s) {
    const Shape& sh = bv.ss[0]->plan->store->sh;
    if (sh.vocab == 0) return fail(TASP_EINVAL, "model has no LM head");
    const Params p = lm_params(bv, logits, sh.vocab);
    return bv.n == 1 ? launch_gemv_single(M_LM, p, s) : launch_gemv(M_LM, p, s);
}

int enqueue_lm_head(Session& se, float* logits, cudaStream_t s) {
    const Shape& sh = se.plan->store->sh;
    if (sh.vocab == 0) return fail(TASP_EINVAL, "model has no LM head");
    return launch_gemv_single(M_LM, lm_params(single_view(se), logits, sh.vocab), s);
}

int enqueue_set_pos(Session& se, int pos, cudaStream_t s) {
    set_pos_kernel<<<1, 32, 0, s>>>(se.d_pos, pos);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

}  // namespace tasp
