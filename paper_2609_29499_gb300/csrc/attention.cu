// GQA decode attention over the retained KV heads of a plan, sm_103a.
//
// One thread-block cluster of CS CTAs handles one kept KV group (all g query heads of
// the group); its CTAs split the cached positions. Within a CTA:
//  * every 16-position K/V tile of the CTA's range is requested at once, before the
//    programmatic-dependency wait. Decode steps of one plan (TMA = true) load each tile
//    with 3-D TMA boxes (16 positions x 64 dimensions, 128-byte swizzle, read
//    conflict-free by ldmatrix) completing on the tile's own mbarrier, so a warp starts
//    on a tile as soon as it lands; the row of the token this step's QKV kernel writes is
//    copied again after the wait. The union step (up to 16 sessions, no descriptors) uses
//    16-byte cp.async into a padded layout, where only that row waits;
//  * S = q K^T and O += P V run on the tensor cores (mma.sync m16n8k16, BF16 in, FP32
//    accumulate). The 16 rows of the A operand hold the g query heads twice: rows r
//    carry bf16(x) and rows r + 8 carry bf16(x - bf16(x)), so the two halves summed in
//    FP32 reproduce the FP32 queries / probabilities to ~2^-17 relative while K and V
//    are used exactly (the cache is BF16);
//  * online softmax in the log2 domain (scores pre-scaled by log2(e)/sqrt(d_h)); warps
//    merge through shared memory.
// The CTAs of a cluster then merge through distributed shared memory: each CTA stores
// its (max, sum) per head into every CTA and each partial output into the CTA that
// finalizes that (head, dim) slice, one cluster barrier makes the stores visible, and
// each CTA merges its slice from its own shared memory. Contexts longer than one
// cluster holds use several clusters per group;
// their partials go through global scratch and the last cluster (atomic ticket, no
// waiting) merges them.
#include <cuda_bf16.h>

#include <algorithm>
#include <map>
#include <mutex>

#include "tasp_internal.h"
#include "tc_ptx.cuh"

namespace tasp {

namespace {

constexpr int AT_WARPS = 8;
constexpr int AT_THREADS = AT_WARPS * 32;
constexpr int TILE = 16;
constexpr int CLUSTERS_MAX = ATTN_CLUSTERS_MAX;  // clusters per kept group (global merge when > 1)

template <int DH, bool TMA>
struct AttCfg {
    // cp.async layout: rows padded by 16 bytes (a 16-byte rotation per row, read
    // conflict-free by ldmatrix). TMA layout: per 64-dimension half a [16][128 B] box in the
    // 128-byte swizzle (16-byte chunk j of row r stored at chunk j ^ (r & 7)).
    static constexpr int ROWB = DH * 2 + 16;
    static constexpr int HALFB = TILE * 128;    // one 64-dimension half of a tile (TMA layout)
    static constexpr int TILEB = TMA ? TILE * DH * 2 : TILE * ROWB;  // one K or one V tile
    static constexpr int MAXT = DH == 128 ? 24 : 48;  // tiles resident per CTA
    static constexpr int KS = DH / 16;          // k-steps of q K^T
    static constexpr int NT = DH / 8;           // n-tiles of P V
    static constexpr int CPR = DH * 2 / 16;     // 16-byte chunks per row
    static constexpr int SMEM = MAXT * 2 * TILEB + (TMA ? 1024 : 0);  // + alignment of the swizzle atoms
};
// Byte offset of 16-byte chunk c (8 dimensions) of row r in a TMA-layout tile.
__device__ __forceinline__ uint32_t swz_off(int r, int c) {
    return (uint32_t)((c >> 3) * (TILE * 128) + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
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
// cluster primitives (hardware barriers: every CTA of a cluster is co-scheduled)
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_relaxed() {
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.aligned;" ::: "memory"); }
__device__ __forceinline__ void st_cluster(uint32_t addr, float2 v) {
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(addr), "f"(v.x), "f"(v.y) : "memory");
}
__device__ __forceinline__ void st_cluster(uint32_t addr, float4 v) {
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v.x), "f"(v.y), "f"(v.z),
                 "f"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

template <int DH, int G, int CS, bool TMA>
__global__ void __launch_bounds__(AT_THREADS, 1) attn_kernel(const __grid_constant__ AttnParams p) {
    using C = AttCfg<DH, TMA>;
    static_assert(G <= 8, "at most 8 query heads per KV group");
    extern __shared__ __align__(128) uint8_t smraw[];
    uint8_t* const sm =
        TMA ? reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023)) : smraw;
    __shared__ __align__(8) uint64_t tbar[C::MAXT];  // TMA: one mbarrier per tile slot
    __shared__ int abort_flag;
    __shared__ float red_m[AT_WARPS][8], red_l[AT_WARPS][8];
    __shared__ float cm[8], cl[8];              // this CTA's merged (max, sum) per head
    constexpr int ITEMS = G * DH / CS;          // (head, dim) outputs each CTA of the cluster finalizes
    __shared__ __align__(16) float inbox[CS][ITEMS];  // every rank's partial outputs of this CTA's slice
    __shared__ float2 inml[CS][8];                  // every rank's (max, sum) per head
    __shared__ float Mh[8], Lh[8], wts[CLUSTERS_MAX][8];
    __shared__ float we[AT_WARPS][8];  // per-warp weights of each head in the CTA merge
    __shared__ float rw[CS][8];        // per-rank weights of each head in the cluster merge
    __shared__ float Mt[8], Lt[8];     // cluster-wide (max, sum) per head
    __shared__ int is_last;
    const int split = blockIdx.x, jl = blockIdx.y, S = gridDim.x, bz = blockIdx.z;
    if (jl >= p.m_kv[bz]) return;  // the session's plan keeps fewer groups (whole cluster exits)
    const int NC = S / CS, cid = split / CS;
    // session bz of the batch
    const float* const q_in = p.q + bz * p.q_stride;
    float* const o_out = p.o + bz * p.q_stride;
    const int16_t* const oslot = p.oslot[bz];  // NULL: every head of the kept groups, in order
    float* const part = p.part + bz * p.part_stride;
    float* const ml = p.ml + bz * p.ml_stride;
    int* const cnt = p.cnt + bz * p.cnt_stride;
    const int max_tokens = p.max_tokens[bz];
    const uint32_t rank = cluster_rank();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // first half of a cluster barrier: waited on before the first remote store, so every
    // CTA of the cluster is known to be running by then
    cluster_arrive_relaxed();

    const int T = *p.pos[bz] + 1;  // written by the previous step, which has completed
    const int chunk = (((T + S - 1) / S) + TILE - 1) / TILE * TILE;
    const int p0 = min(T, split * chunk), p1 = min(T, p0 + chunk);
    const uint16_t* Kg = p.K[bz] + (int64_t)jl * max_tokens * DH;
    const uint16_t* Vg = p.V[bz] + (int64_t)jl * max_tokens * DH;
    const int ntiles = (p1 - p0 + TILE - 1) / TILE;
    const int dep_tile = (p1 == T && ntiles > 0) ? ntiles - 1 : -1;  // holds this step's new token

    // rows of tile ti into slot `slot`, except position `skip` (zero-filled past p1)
    auto issue = [&](int ti, int slot, int skip) {
        const int base = p0 + ti * TILE;
        uint8_t* kt = sm + slot * 2 * C::TILEB;
        uint8_t* vt = kt + C::TILEB;
#pragma unroll
        for (int c = lane; c < TILE * C::CPR; c += 32) {
            const int r = c / C::CPR, cc = c - r * C::CPR;
            const int pos = base + r;
            if (pos == skip) continue;
            const bool ok = pos < p1;
            const int64_t off = (int64_t)(ok ? pos : p0) * DH + cc * 8;
            cp_async16(smem_u32(kt + r * C::ROWB + cc * 16), Kg + off, ok ? 16 : 0);
            cp_async16(smem_u32(vt + r * C::ROWB + cc * 16), Vg + off, ok ? 16 : 0);
        }
    };

    // TMA: tile ti into slot `slot` (K then V, each DH / 64 boxes of 16 positions), completing
    // on the slot's mbarrier. Positions past p1 hold finite cache contents (the caches start
    // zeroed) or zeros past the capacity; their scores are masked.
    auto issue_tma = [&](int ti, int slot) {
        const uint32_t bar = smem_u32(&tbar[slot]);
        const uint32_t kt = smem_u32(sm + slot * 2 * C::TILEB), vt = kt + C::TILEB;
        tc::mbar_expect_tx(bar, 2 * C::TILEB);
#pragma unroll
        for (int hx = 0; hx < DH / 64; ++hx) {
            tc::tma_load_3d(kt + hx * C::HALFB, &p.tmK[bz], hx * 64, p0 + ti * TILE, jl, bar);
            tc::tma_load_3d(vt + hx * C::HALFB, &p.tmV[bz], hx * 64, p0 + ti * TILE, jl, bar);
        }
    };

    // first batch of tiles; the row of this step's token (written by the QKV kernel) waits
    const int nb0 = min(C::MAXT, ntiles);
    if constexpr (TMA) {
        if (tid == 0) {
            abort_flag = 0;
            for (int t = 0; t < C::MAXT; ++t) tc::mbar_init(smem_u32(&tbar[t]), 1);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncthreads();
        if (lane == 0)
            for (int t = warp; t < nb0; t += AT_WARPS) issue_tma(t, t);
        pdl_wait();
        pdl_trigger();
    } else {
        for (int t = warp; t < nb0; t += AT_WARPS) issue(t, t, t == dep_tile ? T - 1 : -1);
        cp_commit();
        pdl_wait();
        pdl_trigger();
        if (dep_tile >= 0 && dep_tile < nb0 && dep_tile % AT_WARPS == warp && lane < C::CPR) {
            const int r = T - 1 - (p0 + dep_tile * TILE);
            const int64_t off = (int64_t)(T - 1) * DH + lane * 8;
            uint8_t* kt = sm + dep_tile * 2 * C::TILEB;
            cp_async16(smem_u32(kt + r * C::ROWB + lane * 16), Kg + off, 16);
            cp_async16(smem_u32(kt + C::TILEB + r * C::ROWB + lane * 16), Vg + off, 16);
        }
        cp_commit();
    }

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
                const float* qp = q_in + (int64_t)(jl * G + h) * DH + col;
                x0 = qp[0] * p.qscale;
                x1 = qp[1] * p.qscale;
            }
            split_pack(x0, x1, qa[ks][2 * half], qa[ks][2 * half + 1]);
        }

    float acc[C::NT][4];
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;
    bool any = false;

    for (int b0 = 0; b0 < ntiles; b0 += C::MAXT) {
        const int nb = min(C::MAXT, ntiles - b0);
        const uint32_t par = (uint32_t)((b0 / C::MAXT) & 1);
        if (b0 > 0) {  // later batches (very long contexts): reuse this warp's slots
            if constexpr (TMA) {
                // this warp's reads of its slots are done; order them before the async writes
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0)
                    for (int t = warp; t < nb; t += AT_WARPS) issue_tma(b0 + t, t);
            } else {
                for (int t = warp; t < nb; t += AT_WARPS) issue(b0 + t, t, -1);
                cp_commit();
            }
        }
        if constexpr (!TMA) {
            cp_wait_all();
            __syncwarp();
        }
        for (int t = warp; t < nb; t += AT_WARPS) {
            any = true;
            const int base = p0 + (b0 + t) * TILE;
            const uint8_t* kt = sm + t * 2 * C::TILEB;
            const uint8_t* vt = kt + C::TILEB;
            if constexpr (TMA) {
                tc::mbar_wait(smem_u32(&tbar[t]), par, &abort_flag, p.err);
                if (b0 == 0 && b0 + t == dep_tile) {
                    // the box was requested before the QKV kernel wrote this step's token: copy
                    // that row again (K by lanes 0..CPR-1, V by the next CPR lanes)
                    const int r = T - 1 - base;
                    if (lane < 2 * C::CPR) {
                        const int which = lane / C::CPR, c = lane - which * C::CPR;
                        const uint4 v = *reinterpret_cast<const uint4*>((which ? Vg : Kg) + (int64_t)(T - 1) * DH + c * 8);
                        *reinterpret_cast<uint4*>(const_cast<uint8_t*>(which ? vt : kt) + swz_off(r, c)) = v;
                    }
                    __syncwarp();
                }
            }
            float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
            const int kr = 8 * ((lane >> 4) & 1) + (lane & 7), kh = (lane >> 3) & 1;
            const uint32_t krow = TMA ? smem_u32(kt) : smem_u32(kt + kr * C::ROWB + 16 * kh);
#pragma unroll
            for (int ks = 0; ks < C::KS; ++ks) {
                uint32_t b00, b01, b10, b11;
                ldsm_x4(TMA ? krow + swz_off(kr, 2 * ks + kh) : krow + ks * 32, b00, b01, b10, b11);
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
            const int vr = 8 * ((lane >> 3) & 1) + (lane & 7), vh = (lane >> 4) & 1;
            const uint32_t vrow = TMA ? smem_u32(vt) : smem_u32(vt + vr * C::ROWB + 16 * vh);
#pragma unroll
            for (int nt = 0; nt < C::NT; nt += 2) {
                uint32_t v0, v1, v2, v3;
                ldsm_x4_t(TMA ? vrow + swz_off(vr, nt + vh) : vrow + nt * 16, v0, v1, v2, v3);
                mma16816(acc[nt], pa, v0, v1);
                mma16816(acc[nt + 1], pa, v2, v3);
            }
        }
        __syncwarp();
    }
    if constexpr (!TMA) cp_wait_all();  // nothing in flight past this point (also for warps without tiles)
    if constexpr (TMA) {
        // after a wait that gave up, wait once more (bounded on its own) for this warp's last
        // boxes, so no copy lands in shared memory that is reused or released
        if (*(volatile int*)&abort_flag && ntiles > 0) {
            const int lb = (ntiles - 1) / C::MAXT * C::MAXT;
            for (int t = warp; t < min(C::MAXT, ntiles - lb); t += AT_WARPS)
                tc::mbar_wait(smem_u32(&tbar[t]), (uint32_t)((lb / C::MAXT) & 1), &abort_flag, p.err, false);
        }
    }
    l_run += __shfl_xor_sync(0xffffffffu, l_run, 1);
    l_run += __shfl_xor_sync(0xffffffffu, l_run, 2);

    // ---- merge the warps of this CTA (the tile memory is reused)
    constexpr int WS = DH + 4;  // padded row of a warp's partial outputs: conflict-free float2 stores
    __syncthreads();
    float* wacc = reinterpret_cast<float*>(sm);  // [AT_WARPS][8][WS]
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) {
        const int dim = nt * 8 + qc;
        *reinterpret_cast<float2*>(wacc + (warp * 8 + h) * WS + dim) =
            any ? make_float2(acc[nt][0] + acc[nt][2], acc[nt][1] + acc[nt][3]) : make_float2(0.f, 0.f);
    }
    if ((lane & 3) == 0) {
        red_m[warp][h] = any ? m_run : -INFINITY;
        red_l[warp][h] = any ? l_run : 0.f;
    }
    __syncthreads();
    // per head: the maximum over warps, each warp's weight 2^(m_w - M) and the weighted sum
    if (tid < 8) {
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < AT_WARPS; ++w) M = fmaxf(M, red_m[w][tid]);
        float Ls = 0.f;
#pragma unroll
        for (int w = 0; w < AT_WARPS; ++w) {
            const float e = red_m[w][tid] == -INFINITY ? 0.f : exp2f(red_m[w][tid] - M);
            we[w][tid] = e;
            Ls = fmaf(red_l[w][tid], e, Ls);
        }
        cm[tid] = M;
        cl[tid] = Ls;
    }
    __syncthreads();
    // ---- merge the CTAs of the cluster: push each (head, dim) output of this CTA to the
    // rank that finalizes it, and this CTA's (max, sum) of each head to every rank
    cluster_wait();  // every CTA of the cluster is running (first barrier half)
    const uint32_t inbox_a = smem_u32(&inbox[rank][0]), inml_a = smem_u32(&inml[rank][0]);
    if (tid < 8 * CS) {
        const int r = tid >> 3, hh = tid & 7;
        st_cluster(map_to_rank(inml_a + 8 * hh, r), make_float2(cm[hh], cl[hh]));
    }
    for (int it = tid; it < G * DH / 4; it += AT_THREADS) {
        const int hh = it / (DH / 4), d4 = it - hh * (DH / 4);
        float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int w = 0; w < AT_WARPS; ++w) {
            const float e = we[w][hh];
            const float4 v = *reinterpret_cast<const float4*>(wacc + (w * 8 + hh) * WS + d4 * 4);
            a.x = fmaf(v.x, e, a.x);
            a.y = fmaf(v.y, e, a.y);
            a.z = fmaf(v.z, e, a.z);
            a.w = fmaf(v.w, e, a.w);
        }
        const int item = it * 4, k = item / ITEMS;  // ITEMS is a multiple of 4: one owner per float4
        st_cluster(map_to_rank(inbox_a + 4 * (item - k * ITEMS), k), a);
    }
    cluster_sync();  // the pushed values are visible to their owners; nothing is read remotely after this
    // finalize this CTA's slice from its own shared memory
    if (tid < 8) {
        float M = -INFINITY;
#pragma unroll
        for (int r = 0; r < CS; ++r) M = fmaxf(M, inml[r][tid].x);
        float Ls = 0.f;
#pragma unroll
        for (int r = 0; r < CS; ++r) {
            const float e = inml[r][tid].x == -INFINITY ? 0.f : exp2f(inml[r][tid].x - M);
            rw[r][tid] = e;
            Ls = fmaf(inml[r][tid].y, e, Ls);
        }
        Mt[tid] = M;
        Lt[tid] = Ls;
    }
    __syncthreads();
    for (int it = tid; it < ITEMS; it += AT_THREADS) {
        const int item = (int)rank * ITEMS + it;
        const int hh = item / DH, dim = item - hh * DH;
        float As = 0.f;
#pragma unroll
        for (int r = 0; r < CS; ++r) As = fmaf(inbox[r][it], rw[r][hh], As);
        if (NC == 1) {
            const int oh = oslot ? oslot[jl * G + hh] : jl * G + hh;
            if (oh >= 0) o_out[(int64_t)oh * DH + dim] = As / Lt[hh];
        } else {
            part[((int64_t)(jl * NC + cid) * G + hh) * DH + dim] = As;
            if (dim == 0) {
                ml[((int64_t)(jl * NC + cid) * G + hh) * 2 + 0] = Mt[hh];
                ml[((int64_t)(jl * NC + cid) * G + hh) * 2 + 1] = Lt[hh];
            }
        }
    }
    if (NC == 1) return;
    __threadfence();
    cluster_sync();  // every slice of this cluster is written before its ticket is taken

    // ---- several clusters per group: the last one (ticket) merges their partials
    if (rank != 0) return;
    if (tid == 0) is_last = (atomicAdd(cnt + jl, 1) == NC - 1);
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    const float* mlg = ml + (int64_t)jl * NC * G * 2;
    if (tid < G) {
        float M = -INFINITY;
        for (int c = 0; c < NC; ++c) M = fmaxf(M, __ldcg(mlg + 2 * (c * G + tid)));
        float L = 0.f;
        for (int c = 0; c < NC; ++c) {
            const float m = __ldcg(mlg + 2 * (c * G + tid));
            const float w = (m == -INFINITY) ? 0.f : exp2f(m - M);
            wts[c][tid] = w;
            L = fmaf(__ldcg(mlg + 2 * (c * G + tid) + 1), w, L);
        }
        Mh[tid] = M;
        Lh[tid] = L;
    }
    __syncthreads();
    const float* pg = part + (int64_t)jl * NC * G * DH;
    for (int it = tid; it < G * DH / 4; it += AT_THREADS) {
        const int hh = it / (DH / 4), d4 = it - hh * (DH / 4);
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int c = 0; c < NC; ++c) {
            const float4 a = __ldcg(reinterpret_cast<const float4*>(pg + ((int64_t)c * G + hh) * DH) + d4);
            const float w = wts[c][hh] / Lh[hh];
            o.x = fmaf(a.x, w, o.x);
            o.y = fmaf(a.y, w, o.y);
            o.z = fmaf(a.z, w, o.z);
            o.w = fmaf(a.w, w, o.w);
        }
        const int oh = oslot ? oslot[jl * G + hh] : jl * G + hh;
        if (oh >= 0) reinterpret_cast<float4*>(o_out + (int64_t)oh * DH)[d4] = o;
    }
    if (tid == 0) cnt[jl] = 0;
}

typedef void (*AttnFn)(const AttnParams);

template <int DH, int G>
AttnFn attn_fn(int cs, bool tma) {
    if (tma) return cs == 16 ? attn_kernel<DH, G, 16, true> : attn_kernel<DH, G, 8, true>;
    return cs == 16 ? attn_kernel<DH, G, 16, false> : attn_kernel<DH, G, 8, false>;
}

AttnFn pick(int dh, int g, int cs, bool tma = false) {
#define TASP_ATT(D, GG) \
    if (dh == D && g == GG) return attn_fn<D, GG>(cs, tma);
    TASP_ATT(64, 1) TASP_ATT(64, 2) TASP_ATT(64, 4) TASP_ATT(64, 8)
    TASP_ATT(128, 1) TASP_ATT(128, 2) TASP_ATT(128, 4) TASP_ATT(128, 8)
#undef TASP_ATT
    return nullptr;
}

int smem_of(int dh, bool tma = false) {
    if (tma) return dh == 128 ? AttCfg<128, true>::SMEM : AttCfg<64, true>::SMEM;
    return dh == 128 ? AttCfg<128, false>::SMEM : AttCfg<64, false>::SMEM;
}
int maxt_of(int dh) { return dh == 128 ? AttCfg<128, false>::MAXT : AttCfg<64, false>::MAXT; }

// Largest cluster size (16 when the device allows it, else 8) for a kernel.
int cluster_size(AttnFn fn, int dh) {
    static int cached[2] = {0, 0};
    int& c = cached[dh == 128];
    if (c) return c;
    cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_of(dh));
    int cs = 8;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(16, 1);
        cfg.blockDim = dim3(AT_THREADS);
        cfg.dynamicSmemBytes = smem_of(dh);
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 16;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) == cudaSuccess && n >= 1) cs = 16;
    }
    cudaGetLastError();  // a refused non-portable size is not an error of the step
    c = cs;
    return cs;
}

}  // namespace

int attn_supported(int dh, int g) { return pick(dh, g, 8) != nullptr; }

int attn_cluster(int dh, int g) { return cluster_size(pick(dh, g, 16), dh); }

// Splits (CTAs) per kept group: one cluster, or several when the context exceeds what
// one cluster keeps resident.
int attn_splits(int m_kv, int max_tokens, int sms, int dh, int g, int cs_cap) {
    (void)m_kv;
    (void)sms;
    const int cs = std::min(attn_cluster(dh, g), cs_cap);
    const int tiles = (max_tokens + TILE - 1) / TILE;
    int nc = (tiles + cs * maxt_of(dh) - 1) / (cs * maxt_of(dh));
    nc = std::max(1, std::min(nc, CLUSTERS_MAX));
    return nc * cs;
}

int attn_splits_max() { return CLUSTERS_MAX * 16; }

namespace {
// Clusters of `cs` CTAs of the attention kernel that the device holds at once (cached).
int active_clusters(int dh, int g, int cs, bool tma) {
    static std::mutex mu;
    static std::map<int, int> cache;
    const int key = ((dh * 16 + g) * 32 + cs) * 2 + (tma ? 1 : 0);
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
    int n = 0;
    if (AttnFn fn = pick(dh, g, cs, tma)) {
        cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_of(dh, tma));
        if (cs == 16) cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(cs, 1);
        cfg.blockDim = dim3(AT_THREADS);
        cfg.dynamicSmemBytes = smem_of(dh, tma);
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = cs;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) n = 0;
        cudaGetLastError();
    }
    cache.emplace(key, n);
    return n;
}
}  // namespace

int attn_cluster_for(int m_kv, int nb, int max_tokens, int dh, int g, bool tma) {
    const int c16 = attn_cluster(dh, g);
    if (c16 < 16 || m_kv * nb <= 0) return c16;
    auto waves = [&](int cs) {
        const int act = active_clusters(dh, g, cs, tma);
        const int n = m_kv * nb * (attn_splits(m_kv, max_tokens, 0, dh, g, cs) / cs);
        return act > 0 ? (n + act - 1) / act : 1 << 20;
    };
    return waves(8) < waves(16) ? 8 : 16;
}

int launch_attention(const AttnParams& a, int dh, int g, int m_kv, int splits, int nb, cudaStream_t s,
                     int cs_cap) {
    const int cs = std::min(attn_cluster(dh, g), cs_cap);
    const bool tma = a.tma != 0 && nb <= MAX_BATCH;
    AttnFn fn = pick(dh, g, cs, tma);
    if (!fn) return fail(TASP_EUNSUP, "attention kernel not built for this (head_dim, query heads per group)");
    static bool attr[2][9][2][2] = {};
    bool& done = attr[dh == 128][g][cs == 16][tma];
    if (!done) {
        TASP_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_of(dh, tma)));
        if (cs == 16) TASP_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1));
        done = true;
    }
    if (splits % cs) return fail(TASP_EINVAL, "attention splits must be a multiple of the cluster size");
    cudaLaunchConfig_t cfg = {};
    if (nb < 1 || nb > UNION_MAX) return fail(TASP_EINVAL, "attention batch of 1 to 16 sessions");
    cfg.gridDim = dim3(splits, m_kv, nb);
    cfg.blockDim = dim3(AT_THREADS);
    cfg.dynamicSmemBytes = smem_of(dh, tma);
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cs;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    TASP_CUDA(cudaLaunchKernelEx(&cfg, fn, a));
    return TASP_OK;
}

}  // namespace tasp
