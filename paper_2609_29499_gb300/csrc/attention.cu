// GQA decode attention over the retained KV heads of a plan (split-KV), sm_103a.
//
// One CTA handles one (split, kept KV group): a contiguous range of cached positions
// and all g query heads of the group. Its 8 warps take 16-position tiles in turn:
//  * K and V tiles are staged with cp.async (16-byte chunks, zero-filled past the
//    last position) into a padded shared-memory layout read conflict-free by ldmatrix;
//  * S = q K^T and O += P V run on the tensor cores (mma.sync m16n8k16, BF16 in,
//    FP32 accumulate). The 16 rows of the A operand hold the g query heads twice:
//    rows r carry bf16(x) and rows r + 8 carry bf16(x - bf16(x)), so the two halves
//    summed in FP32 reproduce the FP32 queries / probabilities to ~2^-17 relative
//    while K and V are used exactly (the cache is BF16);
//  * online softmax in the log2 domain (scores pre-scaled by log2(e)/sqrt(d_h)).
// Warps merge in shared memory, splits merge through global partials: the last CTA
// of a group (atomic ticket, no waiting) weights each split by 2^(m_s - M) / L.
#include <cuda_bf16.h>

#include <algorithm>

#include "tasp_internal.h"

namespace tasp {

namespace {

constexpr int AT_WARPS = 8;
constexpr int AT_THREADS = AT_WARPS * 32;
constexpr int TILE = 16;
constexpr int SPLITS_MAX = 32;

template <int DH>
struct AttCfg {
    static constexpr int ROWB = DH * 2 + 16;  // padded BF16 row (bytes): 16-byte rotation per row
    static constexpr int TILEB = TILE * ROWB;
    static constexpr int WARPB = 2 * 2 * TILEB;  // two stages of (K, V)
    static constexpr int KS = DH / 16;           // k-steps of q K^T
    static constexpr int NT = DH / 8;            // n-tiles of P V
    static constexpr int CPR = DH * 2 / 16;      // 16-byte chunks per row
    static constexpr int SMEM = AT_WARPS * WARPB;
};

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(a));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// (x0, x1) -> packed BF16 pair (x0 in the low half) of the high parts, and of the residuals
__device__ __forceinline__ void split_pack(float x0, float x1, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(x0, x1);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(x0 - hf.x, x1 - hf.y);
    hi = *reinterpret_cast<const uint32_t*>(&h);
    lo = *reinterpret_cast<const uint32_t*>(&l);
}

template <int DH, int G>
__global__ void __launch_bounds__(AT_THREADS, 1) attn_kernel(const AttnParams p) {
    using C = AttCfg<DH>;
    static_assert(G <= 8, "at most 8 query heads per KV group");
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ float red_m[AT_WARPS][8], red_l[AT_WARPS][8];
    __shared__ float Mh[8], Lh[8];
    __shared__ int is_last;
    const int split = blockIdx.x, jl = blockIdx.y, S = gridDim.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    // Positions before T-1 do not depend on the previous kernel (and L2 is coherent):
    // pull this CTA's K/V range toward L2 before waiting on it.
    const int T = *p.pos + 1;  // written by the previous step, which has completed
    const int chunk = (((T + S - 1) / S) + TILE - 1) / TILE * TILE;
    const int p0 = min(T, split * chunk), p1 = min(T, p0 + chunk);
    const uint16_t* Kg = p.K + (int64_t)jl * p.max_tokens * DH;
    const uint16_t* Vg = p.V + (int64_t)jl * p.max_tokens * DH;
    if (tid == 0 && p1 > p0) prefetch_l2(Kg + (int64_t)p0 * DH, (uint32_t)((p1 - p0) * DH * 2));
    if (tid == 32 && p1 > p0) prefetch_l2(Vg + (int64_t)p0 * DH, (uint32_t)((p1 - p0) * DH * 2));
    pdl_wait();
    pdl_trigger();

    const int h = lane >> 2;        // head row of this lane's fragments
    const int qc = (lane & 3) * 2;  // column pair within an 8-column block
    uint32_t qa[C::KS][4];
#pragma unroll
    for (int ks = 0; ks < C::KS; ++ks)
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int col = ks * 16 + half * 8 + qc;
            float x0 = 0.f, x1 = 0.f;
            if (h < G) {
                const float* qp = p.q + (int64_t)(jl * G + h) * DH + col;
                x0 = qp[0] * p.qscale;
                x1 = qp[1] * p.qscale;
            }
            split_pack(x0, x1, qa[ks][2 * half], qa[ks][2 * half + 1]);
        }

    float acc[C::NT][4];
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;
    uint8_t* wsm = sm + warp * C::WARPB;
    const int ntiles = (p1 - p0 + TILE - 1) / TILE;
    const int my = warp < ntiles ? (ntiles - warp + AT_WARPS - 1) / AT_WARPS : 0;

    auto issue = [&](int ti, int stage) {
        const int base = p0 + ti * TILE;
        uint8_t* kt = wsm + stage * 2 * C::TILEB;
        uint8_t* vt = kt + C::TILEB;
#pragma unroll
        for (int c = lane; c < TILE * C::CPR; c += 32) {
            const int r = c / C::CPR, cc = c - r * C::CPR;
            const int pos = base + r;
            const bool ok = pos < p1;
            const int64_t off = (int64_t)(ok ? pos : p0) * DH + cc * 8;
            cp_async16(smem_u32(kt + r * C::ROWB + cc * 16), Kg + off, ok ? 16 : 0);
            cp_async16(smem_u32(vt + r * C::ROWB + cc * 16), Vg + off, ok ? 16 : 0);
        }
        cp_commit();
    };

    if (my > 0) issue(warp, 0);
    for (int i = 0; i < my; ++i) {
        const int stage = i & 1;
        if (i + 1 < my) {
            issue(warp + AT_WARPS * (i + 1), stage ^ 1);
            cp_wait<1>();
        } else {
            cp_wait<0>();
        }
        __syncwarp();
        const int base = p0 + (warp + AT_WARPS * i) * TILE;
        const uint8_t* kt = wsm + stage * 2 * C::TILEB;
        const uint8_t* vt = kt + C::TILEB;

        float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
        const uint32_t krow = smem_u32(kt + (8 * ((lane >> 4) & 1) + (lane & 7)) * C::ROWB + 16 * ((lane >> 3) & 1));
#pragma unroll
        for (int ks = 0; ks < C::KS; ++ks) {
            uint32_t b00, b01, b10, b11;
            ldsm_x4(krow + ks * 32, b00, b01, b10, b11);
            mma16816(s0, qa[ks], b00, b01);
            mma16816(s1, qa[ks], b10, b11);
        }
        float sc[4] = {s0[0] + s0[2], s0[1] + s0[3], s1[0] + s1[2], s1[1] + s1[3]};
        const int pp[4] = {base + qc, base + qc + 1, base + 8 + qc, base + 9 + qc};
#pragma unroll
        for (int e = 0; e < 4; ++e)
            if (pp[e] >= p1) sc[e] = -INFINITY;
        float mt = fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3]));
        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 1));
        mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 2));
        const float m_new = fmaxf(m_run, mt);  // finite: every tile holds position `base` < p1
        const float corr = exp2f(m_run - m_new);
        float pv[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) pv[e] = exp2f(sc[e] - m_new);
        l_run = l_run * corr + ((pv[0] + pv[1]) + (pv[2] + pv[3]));
        m_run = m_new;
#pragma unroll
        for (int nt = 0; nt < C::NT; ++nt) {
            acc[nt][0] *= corr;
            acc[nt][1] *= corr;
            acc[nt][2] *= corr;
            acc[nt][3] *= corr;
        }
        uint32_t pa[4];
        split_pack(pv[0], pv[1], pa[0], pa[1]);
        split_pack(pv[2], pv[3], pa[2], pa[3]);
        const uint32_t vrow = smem_u32(vt + (8 * ((lane >> 3) & 1) + (lane & 7)) * C::ROWB + 16 * ((lane >> 4) & 1));
#pragma unroll
        for (int nt = 0; nt < C::NT; nt += 2) {
            uint32_t v0, v1, v2, v3;
            ldsm_x4_t(vrow + nt * 16, v0, v1, v2, v3);
            mma16816(acc[nt], pa, v0, v1);
            mma16816(acc[nt + 1], pa, v2, v3);
        }
        __syncwarp();
    }
    l_run += __shfl_xor_sync(0xffffffffu, l_run, 1);
    l_run += __shfl_xor_sync(0xffffffffu, l_run, 2);

    // ---- merge the warps of this CTA (staging memory is reused)
    __syncthreads();
    float* wacc = reinterpret_cast<float*>(sm);  // [AT_WARPS][8][DH]
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) {
        const int dim = nt * 8 + qc;
        float* dst = wacc + (warp * 8 + h) * DH + dim;
        dst[0] = my ? acc[nt][0] + acc[nt][2] : 0.f;
        dst[1] = my ? acc[nt][1] + acc[nt][3] : 0.f;
    }
    if ((lane & 3) == 0) {
        red_m[warp][h] = my ? m_run : -INFINITY;
        red_l[warp][h] = my ? l_run : 0.f;
    }
    __syncthreads();
    float* part = p.part + (int64_t)(jl * S + split) * G * DH;
    for (int it = tid; it < G * DH; it += AT_THREADS) {
        const int hh = it / DH, dim = it - hh * DH;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < AT_WARPS; ++w) M = fmaxf(M, red_m[w][hh]);
        float Ls = 0.f, As = 0.f;
#pragma unroll
        for (int w = 0; w < AT_WARPS; ++w) {
            const float e = (red_m[w][hh] == -INFINITY) ? 0.f : exp2f(red_m[w][hh] - M);
            Ls = fmaf(red_l[w][hh], e, Ls);
            As = fmaf(wacc[(w * 8 + hh) * DH + dim], e, As);
        }
        part[it] = As;
        if (dim == 0) {
            p.ml[((int64_t)(jl * S + split) * G + hh) * 2 + 0] = M;
            p.ml[((int64_t)(jl * S + split) * G + hh) * 2 + 1] = Ls;
        }
    }

    // ---- ticket: the last CTA of this group merges the splits
    __threadfence();
    __syncthreads();
    if (tid == 0) is_last = (atomicAdd(p.cnt + jl, 1) == S - 1);
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    float* wts = reinterpret_cast<float*>(sm);  // [S][G] split weights
    const float* mlg = p.ml + (int64_t)jl * S * G * 2;
    if (tid < S * G) wts[tid] = __ldcg(mlg + 2 * tid);
    __syncthreads();
    if (tid < G) {
        float M = -INFINITY;
        for (int s = 0; s < S; ++s) M = fmaxf(M, wts[s * G + tid]);
        float L = 0.f;
        for (int s = 0; s < S; ++s) {
            const float m = wts[s * G + tid];
            if (m != -INFINITY) L = fmaf(__ldcg(mlg + 2 * (s * G + tid) + 1), exp2f(m - M), L);
        }
        Mh[tid] = M;
        Lh[tid] = L;
    }
    __syncthreads();
    if (tid < S * G) {
        const int hh = tid % G;
        const float m = wts[tid];
        wts[tid] = (m == -INFINITY) ? 0.f : exp2f(m - Mh[hh]) / Lh[hh];
    }
    __syncthreads();
    const float* pg = p.part + (int64_t)jl * S * G * DH;
    for (int it = tid; it < G * DH / 4; it += AT_THREADS) {
        const int hh = it / (DH / 4), d4 = it - hh * (DH / 4);
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
        for (int s = 0; s < S; ++s) {
            const float4 a = __ldcg(reinterpret_cast<const float4*>(pg + ((int64_t)s * G + hh) * DH) + d4);
            const float w = wts[s * G + hh];
            o.x = fmaf(a.x, w, o.x);
            o.y = fmaf(a.y, w, o.y);
            o.z = fmaf(a.z, w, o.z);
            o.w = fmaf(a.w, w, o.w);
        }
        reinterpret_cast<float4*>(p.o + (int64_t)(jl * G + hh) * DH)[d4] = o;
    }
    if (tid == 0) p.cnt[jl] = 0;
}

typedef void (*AttnFn)(const AttnParams);

template <int DH, int G>
AttnFn attn_fn(int* smem) {
    *smem = AttCfg<DH>::SMEM;
    return attn_kernel<DH, G>;
}

AttnFn pick(int dh, int g, int* smem) {
#define TASP_ATT(D, GG) \
    if (dh == D && g == GG) return attn_fn<D, GG>(smem);
    TASP_ATT(64, 1) TASP_ATT(64, 2) TASP_ATT(64, 4) TASP_ATT(64, 8)
    TASP_ATT(128, 1) TASP_ATT(128, 2) TASP_ATT(128, 4) TASP_ATT(128, 8)
#undef TASP_ATT
    return nullptr;
}

}  // namespace

int attn_supported(int dh, int g) {
    int smem = 0;
    return pick(dh, g, &smem) != nullptr;
}

int attn_splits(int m_kv, int max_tokens, int sms) {
    if (m_kv <= 0) return 1;
    int s = std::max(1, sms / m_kv);
    s = std::min(s, SPLITS_MAX);
    s = std::min(s, std::max(1, (max_tokens + TILE - 1) / TILE));
    return s;
}

int attn_splits_max() { return SPLITS_MAX; }

int launch_attention(const AttnParams& a, int dh, int g, int m_kv, int splits, cudaStream_t s) {
    int smem = 0;
    AttnFn fn = pick(dh, g, &smem);
    if (!fn) return fail(TASP_EUNSUP, "attention kernel not built for this (head_dim, query heads per group)");
    static bool attr[2][9] = {};
    bool& done = attr[dh == 128][g];
    if (!done) {
        TASP_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
        done = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(splits, m_kv);
    cfg.blockDim = dim3(AT_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    TASP_CUDA(cudaLaunchKernelEx(&cfg, fn, a));
    return TASP_OK;
}

}  // namespace tasp
