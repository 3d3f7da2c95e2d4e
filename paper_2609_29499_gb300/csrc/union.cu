// Union-of-masks batched decode (sm_103a): one step for up to 16 sessions whose plans may
// differ, reading every weight row of the shared store once for all of them.
//
// Each session's plan is the dense layer with its pruned units set to zero (the paper's
// mask-as-zero reading, Sec. 3): so the union step runs the dense projections for all
// sessions at once and applies each session's mask where the units meet it:
//  * Q/K/V: outputs of a group the session's plan drops are not written; the kept ones go
//    to the session's plan-shaped query buffer and KV cache (rotary applied);
//  * attention: per session over its own kept groups (the decode attention kernel, one
//    cluster per (kept group, session)); under a query-head plan the heads a kept group
//    drops are computed but not written (the plan's output-slot table);
//  * O: the session's attention output scattered to dense head order with zeros for the
//    dropped heads (whole groups or single query heads), so their columns contribute nothing;
//  * gate/up: SiLU(gate) * up is zeroed for the channel units the plan drops, so the down
//    projection's columns for them contribute nothing.
//
// The dense projections are skinny GEMMs on the 5th-generation tensor cores: D[rows x 16] =
// W[rows x K] X[16 x K]^T with W the INT8 store panel and X the sessions' activations in
// FP16 (each session scaled by a power of two so its largest entry is below 2^14; exact
// rescaling). Persistent CTAs (three per SM) walk (128-row tile, K slice) units:
//  * warp 0 streams 128 x 128 INT8 weight tiles and the 16 x 128 FP16 activation tile of
//    the same K range with TMA (128-byte swizzle) into a 3-stage ring;
//  * warps 2-5 convert each INT8 tile to FP16 (exact: v + 1152 is built in the FP16 bit
//    pattern 0x6400 | (v ^ 0x80) and 1152 subtracted) in registers, one weight row per
//    thread, and store it into tensor memory (row = TMEM lane, packed FP16 pairs);
//  * warp 1 issues tcgen05.mma (M = 128, N = 16, K = 16) with the weights as the A operand
//    read from tensor memory and the activations from shared memory, into one of two
//    16-column TMEM accumulators;
//  * warps 6-9 read the accumulator (tcgen05.ld) and store the unit's FP32 partial sums.
// The BF16 LM head runs through the same kernel: TMA writes its weight tiles straight into the
// MMA operand layout (no conversion) and the activations are BF16.
// Small finish kernels then sum the K slices in a fixed order, apply the row scales and
// each session's mask, and run the projection's epilogue.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <cmath>
#include <map>
#include <memory>
#include <mutex>

#include "tasp_internal.h"
#include "tc_ptx.cuh"

namespace tasp {

namespace {

using namespace tc;

constexpr int US = UNION_MAX;  // sessions per union step = MMA N
constexpr int SK_BM = 128;     // weight rows per tile (MMA M)
constexpr int SK_BK = 128;     // K (INT8 bytes) per stage
constexpr int SK_NST = 3;       // INT8 + activation stages
constexpr int SK_NST_BF16 = 2;  // BF16 weight + activation stages (the LM head)
constexpr int SK_NA = 1;        // FP16 operand buffers in tensor memory
// CTAs per SM: each small MMA costs its issuing thread ~90 ns, so three CTAs (three issuing
// threads) keep the tensor core busier than one CTA with deep rings (measured with the FP16
// operand in shared memory: 1, 2, 3 CTAs per SM -> 523, 618, 711 tokens/s)
constexpr int SK_CTAS_PER_SM = 3;
// Tensor memory of an INT8 CTA: accumulators at columns 0 and 16, operand buffer b (128 K
// values = 64 columns of FP16 pairs) at 64 + 64 b; a BF16 CTA needs the accumulators only.
constexpr uint32_t SK_TMEM_I8 = 128, SK_TMEM_BF16 = 32;
static_assert(64 + 64 * SK_NA <= SK_TMEM_I8 && SK_CTAS_PER_SM * SK_TMEM_I8 <= 512, "tensor memory of the skinny GEMM");
constexpr int SK_W_BYTES = SK_BM * SK_BK;      // INT8 tile
constexpr int SK_X_BYTES = US * SK_BK * 2;     // FP16 activation tile (two 64-column boxes)
constexpr int SK_A_HALF = SK_BM * 64 * 2;      // BF16 weight box of 64 columns
constexpr int SK_STAGE = SK_W_BYTES + SK_X_BYTES;
constexpr int SK_SMEM = SK_NST * SK_STAGE + 1024;
constexpr int SK_THREADS = 320;
constexpr uint32_t SK_IDESC = idesc_f16(SK_BM, US);
// BF16 weights (the LM head): both operands BF16 (instruction-descriptor A/B format 1)
constexpr uint32_t SK_IDESC_BF16 = SK_IDESC | (1u << 7) | (1u << 10);
constexpr int SK_WB_BF16 = 2 * SK_A_HALF;  // BF16 weight tile 128 x 128 (two 64-column boxes)
constexpr int SK_SMEM_BF16 = SK_NST_BF16 * (SK_WB_BF16 + SK_X_BYTES) + 1024;
constexpr int SK_UNITS_PER_CTA = 3;  // target units per CTA when choosing K slices
constexpr int UN_ATT_CS = 8;         // attention cluster size: 16 sessions fill the GPU with 8-CTA clusters

// Programmatic dependent launch: every union kernel lets the next one launch early and waits
// for the previous one (all of whose writes it may read, and whose reads it may overwrite)
// only where it first touches dependent data.
__device__ __forceinline__ void grid_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

struct SkArgs {
    int rows, K;  // weight panel rows; reduction length (multiple of 128)
    int S, kbs;   // K slices and 128-column blocks per slice
    float* part;  // [S][rows][US] partial sums
    int* err;
    // grouped store: BF16 scales [rows][gld] of qg columns each (NULL: per-row scales, applied
    // by the finish kernels); the converters then make FP16 q s_g 2^SK_GS_EXP, one rounding
    const uint16_t* gs;
    int gld, qg;
};
// power-of-two factor on q s_g in FP16 (undone in FP32 by the finish kernels): keeps the
// products of scales down to ~2^-22 normal in FP16 and weights up to 255 in magnitude in range
constexpr int SK_GS_EXP = 8;

// INT8 x 4 (one word) -> FP16 x 4 (two words), exact.
__device__ __forceinline__ void i8x4_to_h(uint32_t w, uint32_t& lo, uint32_t& hi) {
    const uint32_t u = w ^ 0x80808080u;                  // v + 128 as unsigned bytes
    const uint32_t a = __byte_perm(u, 0x64646464u, 0x5140);  // (0x64, b1, 0x64, b0): 1024 + u per half
    const uint32_t b = __byte_perm(u, 0x64646464u, 0x7362);
    const __half2 k = __halves2half2(__ushort_as_half(0x6480), __ushort_as_half(0x6480));  // 1152
    const __half2 ha = __hsub2(*reinterpret_cast<const __half2*>(&a), k);
    const __half2 hb = __hsub2(*reinterpret_cast<const __half2*>(&b), k);
    lo = *reinterpret_cast<const uint32_t*>(&ha);
    hi = *reinterpret_cast<const uint32_t*>(&hb);
}

// BW: BF16 weights (the LM head), read by the MMAs straight from the stage (no conversion).
// GS: INT8 weights of a grouped store (the converters apply the group scales).
template <bool BW, bool GS = false>
__global__ void __launch_bounds__(SK_THREADS, SK_CTAS_PER_SM)
    skinny_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, const SkArgs a) {
    constexpr int WBYTES = BW ? SK_WB_BF16 : SK_W_BYTES;
    constexpr int STAGE = WBYTES + SK_X_BYTES;
    constexpr int NST = BW ? SK_NST_BF16 : SK_NST;
    constexpr uint32_t TCOLS = BW ? SK_TMEM_BF16 : SK_TMEM_I8;
    extern __shared__ uint8_t smraw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = sm;  // stage s: weight tile, then the activation tile
    __shared__ __align__(8) uint64_t full[NST], empty[NST], afull[SK_NA], aempty[SK_NA], accf[2], acce[2];
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tiles = (a.rows + SK_BM - 1) / SK_BM;
    const int units = tiles * a.S;
    const int nkb = a.K / SK_BK;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < NST; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), BW ? 1 : 4 + 1);  // converter warps (INT8) + the MMAs
        }
        for (int b = 0; b < SK_NA; ++b) {
            mbar_init(smem_u32(&afull[b]), 4);
            mbar_init(smem_u32(&aempty[b]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&accf[b]), 1);
            mbar_init(smem_u32(&acce[b]), 4);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                     "r"(TCOLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = tmem_base;
    grid_trigger();

    if (warp == 0) {
        if (lane == 0) {  // ---- TMA producer
            // the first stages' weight tiles go out before the dependency wait (weights are
            // constant); activations, written by the previous kernel, after it
            int g = 0, xs = 0;  // stages issued, stages whose activation tile is issued
            auto issue_x = [&](int gx, int kb) {
                const uint32_t st = smem_u32(ring + (gx % NST) * STAGE);
                const uint32_t fb = smem_u32(&full[gx % NST]);
                tma_load_2d(st + WBYTES, &tmX, kb * SK_BK, 0, fb);
                tma_load_2d(st + WBYTES + SK_X_BYTES / 2, &tmX, kb * SK_BK + 64, 0, fb);
            };
            int pre_kb[NST];
            for (int u = blockIdx.x; u < units; u += gridDim.x) {
                const int tile = u / a.S, ks = u - tile * a.S;
                const int kb0 = ks * a.kbs, kb1 = min(nkb, kb0 + a.kbs);
                for (int kb = kb0; kb < kb1; ++kb, ++g) {
                    const int s = g % NST;
                    if (g >= NST) mbar_wait(smem_u32(&empty[s]), ((g / NST) - 1) & 1, &abort_flag, a.err);
                    const uint32_t fb = smem_u32(&full[s]);
                    mbar_expect_tx(fb, STAGE);
                    const uint32_t st = smem_u32(ring + s * STAGE);
                    tma_load_2d(st, &tmW, kb * SK_BK, tile * SK_BM, fb);
                    if (BW) tma_load_2d(st + SK_A_HALF, &tmW, kb * SK_BK + 64, tile * SK_BM, fb);
                    if (g < NST) {
                        pre_kb[g] = kb;
                        if (g == NST - 1) {
                            grid_wait();
                            for (; xs <= g; ++xs) issue_x(xs, pre_kb[xs]);
                        }
                    } else {
                        issue_x(g, kb);
                        xs = g + 1;
                    }
                }
            }
            if (xs < g || g == 0) {  // fewer k-blocks than stages: their activations are still due
                grid_wait();
                for (; xs < g; ++xs) issue_x(xs, pre_kb[xs]);
            }
            for (int k = max(0, g - NST); k < g; ++k)  // no copy may outlive the CTA
                mbar_wait(smem_u32(&full[k % NST]), (k / NST) & 1, &abort_flag, a.err, false);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---- MMA issuer
            int g = 0, it = 0;
            for (int u = blockIdx.x; u < units; u += gridDim.x, ++it) {
                const int tile = u / a.S, ks = u - tile * a.S;
                const int kb0 = ks * a.kbs, kb1 = min(nkb, kb0 + a.kbs);
                const int acc = it & 1;
                if (it >= 2) mbar_wait(smem_u32(&acce[acc]), ((it >> 1) - 1) & 1, &abort_flag, a.err);
                fence_after();
                for (int kb = kb0; kb < kb1; ++kb, ++g) {
                    const int s = g % NST, ab = g % SK_NA;
                    if (!BW) mbar_wait(smem_u32(&afull[ab]), (g / SK_NA) & 1, &abort_flag, a.err);
                    mbar_wait(smem_u32(&full[s]), (g / NST) & 1, &abort_flag, a.err);
                    fence_after();
                    const uint32_t sx = smem_u32(ring + s * STAGE + WBYTES);
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint64_t bd = sw128_desc(sx + h * (SK_X_BYTES / 2) + kk * 32);
                            const uint32_t on = (kb > kb0 || h > 0 || kk > 0) ? 1u : 0u;
                            if constexpr (BW)
                                mma_f16(tmem + 16u * acc, sw128_desc(smem_u32(ring + s * STAGE) + h * SK_A_HALF + kk * 32),
                                        bd, SK_IDESC_BF16, on);
                            else  // K 16 = 8 columns of FP16 pairs; K 64 per half
                                mma_f16_tmem_a(tmem + 16u * acc, tmem + 64u + 64u * ab + 32u * h + 8u * kk, bd,
                                               SK_IDESC, on);
                        }
                    if (!BW) commit(smem_u32(&aempty[ab]));
                    commit(smem_u32(&empty[s]));
                }
                commit(smem_u32(&accf[acc]));
            }
        }
    } else if (warp < 6) {  // ---- converters (INT8 weights): thread = weight row = its TMEM lane
      if constexpr (!BW) {
        const int r = 32 * (warp & 3) + lane;  // a warp reaches TMEM lanes 32 (warp % 4) .. + 31
        const uint32_t trow = tmem + ((uint32_t)(32 * (warp & 3)) << 16);
        int g = 0;
        for (int u = blockIdx.x; u < units; u += gridDim.x) {
            const int tile = u / a.S, ks = u - tile * a.S;
            const int kb0 = ks * a.kbs, kb1 = min(nkb, kb0 + a.kbs);
            const int wr = tile * SK_BM + r;  // this thread's weight row (beyond the panel: zero fill)
            const uint16_t* gsr = GS && wr < a.rows ? a.gs + (int64_t)wr * a.gld : nullptr;
            for (int kb = kb0; kb < kb1; ++kb, ++g) {
                const int s = g % NST, ab = g % SK_NA;
                __half2 gsc[8];  // grouped store: the scale of each 16-column chunk, times 2^SK_GS_EXP
                if constexpr (GS) {
                    const int gsh = __ffs(a.qg) - 1;  // the group size is a power of two
                    if (a.qg >= SK_BK) {              // one group covers the whole k-block
                        const float v = gsr ? __uint_as_float((uint32_t)__ldg(gsr + ((kb * SK_BK) >> gsh)) << 16) : 0.f;
                        const __half2 h = __float2half2_rn(ldexpf(v, SK_GS_EXP));
#pragma unroll
                        for (int c = 0; c < 8; ++c) gsc[c] = h;
                    } else {
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            const float v =
                                gsr ? __uint_as_float((uint32_t)__ldg(gsr + ((kb * SK_BK + 16 * c) >> gsh)) << 16) : 0.f;
                            gsc[c] = __float2half2_rn(ldexpf(v, SK_GS_EXP));
                        }
                    }
                }
                mbar_wait(smem_u32(&full[s]), (g / NST) & 1, &abort_flag, a.err);
                if (g >= SK_NA) mbar_wait(smem_u32(&aempty[ab]), ((g / SK_NA) - 1) & 1, &abort_flag, a.err);
                fence_after();  // after the MMAs that last read this operand buffer
                const uint8_t* wrow = ring + s * STAGE + r * 128;
                const int sw = r & 7;  // 128-byte swizzle: 16-byte chunk c of row r sits at c ^ (r % 8)
#pragma unroll
                for (int h = 0; h < 2; ++h) {  // K columns 64 h .. 64 h + 63 -> TMEM columns 32 h ..
                    uint32_t o[32];
#pragma unroll
                    for (int c4 = 0; c4 < 4; ++c4) {
                        const uint4 w = *reinterpret_cast<const uint4*>(wrow + (((4 * h + c4) ^ sw) << 4));
                        i8x4_to_h(w.x, o[8 * c4 + 0], o[8 * c4 + 1]);
                        i8x4_to_h(w.y, o[8 * c4 + 2], o[8 * c4 + 3]);
                        i8x4_to_h(w.z, o[8 * c4 + 4], o[8 * c4 + 5]);
                        i8x4_to_h(w.w, o[8 * c4 + 6], o[8 * c4 + 7]);
                        if constexpr (GS) {  // exact q times an FP16 scale: one rounding of the product
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const __half2 v = __hmul2(*reinterpret_cast<const __half2*>(&o[8 * c4 + i]), gsc[4 * h + c4]);
                                o[8 * c4 + i] = *reinterpret_cast<const uint32_t*>(&v);
                            }
                        }
                    }
                    tmem_st32(trow + 64u + 64u * ab + 32u * h, o);
                }
                asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(smem_u32(&afull[ab]));
                    mbar_arrive(smem_u32(&empty[s]));
                }
            }
        }
      }
    } else {  // ---- epilogue warps 6-9: TMEM lanes 32 (warp % 4) ..
        const int q = warp & 3;
        int it = 0;
        for (int u = blockIdx.x; u < units; u += gridDim.x, ++it) {
            const int tile = u / a.S, ks = u - tile * a.S;
            const int acc = it & 1;
            mbar_wait(smem_u32(&accf[acc]), (it >> 1) & 1, &abort_flag, a.err);
            fence_after();
            uint32_t v[16];
            tmem_ld16(tmem + ((uint32_t)(32 * q) << 16) + 16u * acc, v);
            const int row = tile * SK_BM + 32 * q + lane;
            if (row < a.rows) {
                float4* dst = reinterpret_cast<float4*>(a.part + ((int64_t)ks * a.rows + row) * US);
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    dst[k] = make_float4(__uint_as_float(v[4 * k]), __uint_as_float(v[4 * k + 1]),
                                         __uint_as_float(v[4 * k + 2]), __uint_as_float(v[4 * k + 3]));
            }
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&acce[acc]));
        }
    }
    fence_before();
    __syncthreads();
    fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TCOLS) : "memory");
}

// ------------------------------------------------------------------ activations to FP16
enum PrepMode { PR_NORM = 0, PR_COPY = 1, PR_HEADS = 2 };
struct PrepArgs {
    int mode, K;
    const float* src;          // FP32 [US][src_ld]
    int64_t src_ld;
    const uint16_t* in_bf16;   // PR_NORM on layer 0: the step inputs BF16 [US][K] (also copied to src)
    const float* gamma;        // PR_NORM
    float eps;
    const int* gmap;           // PR_HEADS: [US][Hkv] dense group -> plan group (-1: dropped)
    const int16_t* oslot[US];  // PR_HEADS: the plan's (group slot, head) -> attention output slot, -1 for
                               // a dropped head (NULL: every head of the kept groups, slot jl g + hh)
    int g, dh, Hkv;
    __half* x16;               // [US][ld16] (BF16 bits when bf16)
    int64_t ld16;
    float* xinv;               // [US]: 2^-e of the session's scale
    int bf16;                  // write BF16 (for BF16 weights) instead of FP16
};

constexpr int PREP_CS = 8;  // CTAs (one cluster) per session in prep_kernel

__device__ __forceinline__ float warp_sum(float v) {
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float2 ld_cluster2(const float2* p, uint32_t rank) {
    uint32_t a = smem_u32(p), r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(r) : "memory");
    return v;
}
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Four consecutive entries k..k+3 of the projection input of session b (before the
// RMSNorm factor): x * gamma, a copy, or the plan's heads in dense order.
__device__ __forceinline__ float4 prep_in(const PrepArgs& p, const float* src, int b, int k) {
    if (p.mode == PR_HEADS) {
        const int hd = k / p.dh, j = hd / p.g, hh = hd - j * p.g;
        const int lj = p.gmap[b * p.Hkv + j];
        if (lj < 0) return make_float4(0.f, 0.f, 0.f, 0.f);
        const int slot = p.oslot[b] ? p.oslot[b][lj * p.g + hh] : lj * p.g + hh;
        if (slot < 0) return make_float4(0.f, 0.f, 0.f, 0.f);
        return *reinterpret_cast<const float4*>(src + (int64_t)slot * p.dh + (k - hd * p.dh));
    }
    float4 v = *reinterpret_cast<const float4*>(src + k);
    if (p.mode == PR_NORM) {
        const float4 g = *reinterpret_cast<const float4*>(p.gamma + k);
        v.x *= g.x;
        v.y *= g.y;
        v.z *= g.z;
        v.w *= g.w;
    }
    return v;
}

// One 8-CTA cluster per session: the projection input (RMSNorm(x) * gamma, a copy, or the
// plan's heads scattered to dense order), scaled by 2^e so that its largest magnitude is
// below 2^14, as FP16. Each CTA takes K/8 entries; the cluster combines the sum of squares
// and the largest magnitude through distributed shared memory.
__global__ void __launch_bounds__(256) prep_kernel(const PrepArgs p) {
    grid_wait();
    grid_trigger();
    __shared__ float2 red[8];
    __shared__ float2 tot;  // this CTA's (sum of squares, max |in|)
    const int b = blockIdx.y, rank = blockIdx.x;  // cluster = the session's 8 CTAs along x
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int chunk = (p.K / PREP_CS + 3) & ~3;
    const int k0 = rank * chunk, k1 = min(p.K, k0 + chunk);
    float* x = const_cast<float*>(p.src) + b * p.src_ld;
    if (p.in_bf16) {  // first layer: the residual starts as the step input (this CTA's entries)
        for (int k = k0 + threadIdx.x; k < k1; k += blockDim.x)
            x[k] = __uint_as_float((uint32_t)p.in_bf16[(int64_t)b * p.K + k] << 16);
        __syncthreads();
    }
    float ss = 0.f, mx = 0.f;
    for (int k = k0 + 4 * threadIdx.x; k < k1; k += 4 * blockDim.x) {
        if (p.mode == PR_NORM) {
            const float4 v = *reinterpret_cast<const float4*>(x + k);
            ss = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, ss))));
        }
        const float4 v = prep_in(p, x, b, k);
        mx = fmaxf(mx, fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w))));
    }
    ss = warp_sum(ss);
    mx = warp_max(mx);
    if (lane == 0) red[warp] = make_float2(ss, mx);
    __syncthreads();
    if (threadIdx.x == 0) {
        float2 t = make_float2(0.f, 0.f);
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
            t.x += red[w].x;
            t.y = fmaxf(t.y, red[w].y);
        }
        tot = t;
    }
    cluster_sync_all();
    float2 all = make_float2(0.f, 0.f);
#pragma unroll
    for (int r = 0; r < PREP_CS; ++r) {  // same order in every CTA
        const float2 t = ld_cluster2(&tot, r);
        all.x += t.x;
        all.y = fmaxf(all.y, t.y);
    }
    const float rs = p.mode == PR_NORM ? rsqrtf(all.x / (float)p.K + p.eps) : 1.f;
    const float amax = all.y * rs;
    int e = 0;
    if (amax > 0.f) {
        int ex;
        frexpf(amax, &ex);  // amax < 2^ex
        e = 14 - ex;
    }
    const float sc = ldexpf(rs, e);
    __half* dst = p.x16 + b * p.ld16;
    for (int k = k0 + 4 * threadIdx.x; k < k1; k += 4 * blockDim.x) {
        const float4 v = prep_in(p, x, b, k);
        uint2 o;
        if (p.bf16) {
            const __nv_bfloat162 h0 = __floats2bfloat162_rn(v.x * sc, v.y * sc), h1 = __floats2bfloat162_rn(v.z * sc, v.w * sc);
            o.x = *reinterpret_cast<const uint32_t*>(&h0);
            o.y = *reinterpret_cast<const uint32_t*>(&h1);
        } else {
            const __half2 h0 = __floats2half2_rn(v.x * sc, v.y * sc), h1 = __floats2half2_rn(v.z * sc, v.w * sc);
            o.x = *reinterpret_cast<const uint32_t*>(&h0);
            o.y = *reinterpret_cast<const uint32_t*>(&h1);
        }
        *reinterpret_cast<uint2*>(dst + k) = o;
    }
    if (rank == 0 && threadIdx.x == 0) p.xinv[b] = ldexpf(1.f, -e);
    cluster_sync_all();  // no CTA leaves while others may read its total
}

// ------------------------------------------------------------------ finish kernels
struct FinArgs {
    const float* part;  // [S][rows][US]
    int S, rows, n;
    const float* scale;  // [rows]
    const float* xinv;   // [US]
    float post;          // 2^-SK_GS_EXP for a grouped store, else 1
};
__device__ __forceinline__ float fin_sum(const FinArgs& f, int row, int b) {
    float acc = 0.f;
    for (int s = 0; s < f.S; ++s) acc += f.part[((int64_t)s * f.rows + row) * US + b];
    return acc * f.scale[row] * f.xinv[b] * f.post;
}

// Q/K/V: blockIdx.x = one dense head row block (group j, head hh of g + 2), blockIdx.y = a
// quarter of its rotary pairs; thread = (pair i, session b).
struct QkvFin {
    FinArgs f;
    int g, dh, Hkv;
    const int* gmap;  // [US][Hkv]
    float* q;         // session b: q + b * q_stride, plan-shaped [m_q][dh]
    int64_t q_stride;
    uint16_t* K[US];
    uint16_t* V[US];
    const float2* rope[US];
    const int* pos[US];
    int max_tokens[US];
};
__global__ void finish_qkv_kernel(const QkvFin p) {
    grid_wait();
    grid_trigger();
    const int hb = blockIdx.x, half = p.dh >> 1;
    const int b = threadIdx.x % US, i = blockIdx.y * (blockDim.x / US) + threadIdx.x / US;
    if (b >= p.f.n || i >= half) return;
    const int j = hb / (p.g + 2), hh = hb - j * (p.g + 2);
    const int lj = p.gmap[b * p.Hkv + j];
    if (lj < 0) return;
    const int r0 = hb * p.dh + i;
    float y0 = fin_sum(p.f, r0, b), y1 = fin_sum(p.f, r0 + half, b);
    const int pos = *p.pos[b];
    if (hh <= p.g) {  // rotary on queries and keys
        const float2 cs = p.rope[b][(int64_t)pos * half + i];
        const float ya = y0 * cs.x - y1 * cs.y, yb = y1 * cs.x + y0 * cs.y;
        y0 = ya;
        y1 = yb;
    }
    if (hh < p.g) {
        float* dq = p.q + b * p.q_stride + (int64_t)(lj * p.g + hh) * p.dh;
        dq[i] = y0;
        dq[i + half] = y1;
    } else {
        uint16_t* dst = (hh == p.g ? p.K[b] : p.V[b]) + ((int64_t)lj * p.max_tokens[b] + pos) * p.dh;
        const __nv_bfloat16 a0 = __float2bfloat16_rn(y0), a1 = __float2bfloat16_rn(y1);
        dst[i] = *reinterpret_cast<const uint16_t*>(&a0);
        dst[i + half] = *reinterpret_cast<const uint16_t*>(&a1);
    }
}

// O / down: x_b[row] += s_row * sum; thread = (row, session).
struct ResFin {
    FinArgs f;
    float* x;  // [US][ld]
    int64_t ld;
    float* hidden;  // [n][ld] or nullptr
};
__global__ void finish_resid_kernel(const ResFin p) {
    grid_wait();
    grid_trigger();
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int row = (int)(t / US), b = (int)(t % US);
    if (row >= p.f.rows || b >= p.f.n) return;
    const float v = p.x[b * p.ld + row] + fin_sum(p.f, row, b);
    p.x[b * p.ld + row] = v;
    if (p.hidden) p.hidden[b * p.ld + row] = v;
}

// gate/up (rows interleaved per channel): h_b[c] = SiLU(gate) * up, 0 for dropped units.
struct GuFin {
    FinArgs f;
    float* h;  // [US][ld]
    int64_t ld;
    const uint8_t* keep;  // [US][n_units]
    int n_units, cu;
};
__global__ void finish_gu_kernel(const GuFin p) {
    grid_wait();
    grid_trigger();
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int c = (int)(t / US), b = (int)(t % US);
    if (2 * c >= p.f.rows || b >= p.f.n) return;
    float v = 0.f;
    if (p.keep[b * p.n_units + c / p.cu]) {
        const float a = fin_sum(p.f, 2 * c, b), u = fin_sum(p.f, 2 * c + 1, b);
        v = a / (1.0f + expf(-a)) * u;
    }
    p.h[b * p.ld + c] = v;
}

// LM head: logits_b[row] = sum (no row scale: the head is BF16 as stored).
struct LogitFin {
    FinArgs f;
    float* logits;  // [n][rows]
};
__global__ void finish_logits_kernel(const LogitFin p) {
    grid_wait();
    grid_trigger();
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int row = (int)(t / US), b = (int)(t % US);
    if (row >= p.f.rows || b >= p.f.n) return;
    float acc = 0.f;
    for (int s = 0; s < p.f.S; ++s) acc += p.f.part[((int64_t)s * p.f.rows + row) * US + b];
    p.logits[(int64_t)b * p.f.rows + row] = acc * p.f.xinv[b];
}

struct UnAdvance {
    int* pos[US];
    int n;
};
__global__ void union_advance_kernel(const UnAdvance a) {
    grid_wait();
    if (threadIdx.x < a.n) *a.pos[threadIdx.x] += 1;
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
std::mutex g_enc_mu;

int get_encoder(PFN_cuTensorMapEncodeTiled_v12000* out) {
    std::lock_guard<std::mutex> lk(g_enc_mu);
    if (!g_enc) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
            return fail(TASP_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
        g_enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    *out = g_enc;
    return TASP_OK;
}

// 2-D tensor map of a row-major [rows][cols] buffer (row stride ld_bytes), 128-byte swizzle.
int map2d(CUtensorMap* m, CUtensorMapDataType dt, int esize, const void* base, int rows, int cols, int64_t ld_bytes,
          int box_cols, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc;
    int rc = get_encoder(&enc);
    if (rc) return rc;
    if ((reinterpret_cast<uintptr_t>(base) & 15) || (ld_bytes % 16))
        return fail(TASP_EINVAL, "TMA operand not 16-byte aligned");
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld_bytes};
    cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    (void)esize;
    CUresult r = enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                     CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(TASP_ECUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
    return TASP_OK;
}

// K slices of a projection: about SK_UNITS_PER_CTA units per CTA, no empty slice.
void slices(int rows, int K, int sms, int& S, int& kbs) {
    const int tiles = (rows + SK_BM - 1) / SK_BM, nkb = K / SK_BK;
    S = std::max(1, std::min(nkb, (SK_UNITS_PER_CTA * SK_CTAS_PER_SM * sms + tiles - 1) / tiles));
    kbs = (nkb + S - 1) / S;
    S = (nkb + kbs - 1) / kbs;
}

// Launch with programmatic stream serialization (the kernel waits with griddepcontrol.wait);
// cluster_x > 1 adds a cluster dimension.
template <typename K, typename... A>
int launch_pdl(K kern, dim3 grid, dim3 block, size_t smem, cudaStream_t s, int cluster_x, const A&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = cluster_x;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = cluster_x > 1 ? 2 : 1;
    TASP_CUDA(cudaLaunchKernelEx(&cfg, kern, args...));
    return TASP_OK;
}
template <typename K, typename A>
int launch(K kern, dim3 grid, dim3 block, cudaStream_t s, const A& a) {
    return launch_pdl(kern, grid, block, 0, s, 1, a);
}

// W: INT8 [rows][K], or BF16 [rows][K] when bw (the LM head)
int launch_skinny(const void* W, bool bw, int rows, int K, const __half* x16, int64_t ld16, float* part, int* err,
                  int& S_out, cudaStream_t s, const uint16_t* gs = nullptr, int qg = 0) {
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    if (K % SK_BK) return fail(TASP_EUNSUP, "union decode needs reduction lengths that are multiples of 128");
    CUtensorMap tw, tx;
    if (bw) {
        if ((rc = map2d(&tw, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, W, rows, K, (int64_t)K * 2, 64, SK_BM))) return rc;
        if ((rc = map2d(&tx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, x16, US, K, ld16 * 2, 64, US))) return rc;
    } else {
        if ((rc = map2d(&tw, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, W, rows, K, K, SK_BK, SK_BM))) return rc;
        if ((rc = map2d(&tx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, x16, US, K, ld16 * 2, 64, US))) return rc;
    }
    SkArgs a{};
    a.rows = rows;
    a.K = K;
    slices(rows, K, di.sms, a.S, a.kbs);
    a.part = part;
    a.err = err;
    a.gs = gs;
    a.qg = qg;
    a.gld = qg ? K / qg : 0;
    const int units = ((rows + SK_BM - 1) / SK_BM) * a.S;
    const int grid = std::min(units, SK_CTAS_PER_SM * di.sms);
    if (bw) {
        if ((rc = launch_pdl(skinny_kernel<true>, dim3(grid), dim3(SK_THREADS), SK_SMEM_BF16, s, 1, tw, tx, a))) return rc;
    } else {
        if (gs) {
            if ((rc = launch_pdl(skinny_kernel<false, true>, dim3(grid), dim3(SK_THREADS), SK_SMEM, s, 1, tw, tx, a)))
                return rc;
        } else if ((rc = launch_pdl(skinny_kernel<false>, dim3(grid), dim3(SK_THREADS), SK_SMEM, s, 1, tw, tx, a))) {
            return rc;
        }
    }
    S_out = a.S;
    return TASP_OK;
}

// Workspace and recorded step graph of one set of sessions.
struct UnionWs {
    std::vector<Session*> ss;
    Arena arena;
    float *x = nullptr, *q = nullptr, *o = nullptr, *h = nullptr;
    __half* x16 = nullptr;
    float* xinv = nullptr;
    float* part = nullptr;
    float *apart = nullptr, *aml = nullptr;
    int* acnt = nullptr;
    int* gmap = nullptr;      // [L][US][Hkv]
    uint8_t* keep = nullptr;  // [L][US][n_units]
    int* err = nullptr;
    uint16_t* x_stage = nullptr;
    int64_t ld16 = 0, part_stride = 0, ml_stride = 0;
    int asplits = 0;
    StepGraph graph;
};
std::mutex g_un_mu;
std::map<std::vector<Session*>, std::unique_ptr<UnionWs>> g_un;
bool g_skinny_attr = false;

size_t part_floats(const Shape& sh, int sms) {
    size_t mx = 0;
    auto need = [&](int rows, int K) {
        int S, kbs;
        slices(rows, K, sms, S, kbs);
        mx = std::max(mx, (size_t)S * rows * US);
    };
    need(sh.qkv_rows_dense(), sh.d);
    need(sh.d, sh.Hq * sh.dh);
    need(2 * sh.df, sh.d);
    need(sh.d, sh.df);
    if (sh.vocab) need(sh.vocab, sh.d);
    return mx;
}

int union_get(Session* const* ss, int n, UnionWs** out) {
    std::vector<Session*> key(ss, ss + n);
    std::lock_guard<std::mutex> lk(g_un_mu);
    auto it = g_un.find(key);
    if (it != g_un.end()) {
        *out = it->second.get();
        return TASP_OK;
    }
    const Store& st = *ss[0]->plan->store;
    const Shape& sh = st.sh;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    auto w = std::make_unique<UnionWs>();
    w->ss = key;
    int smax = 1;
    for (int b = 0; b < n; ++b)
        for (const LayerPlan& lp : ss[b]->plan->layers)
            smax = std::max(smax, attn_splits(lp.m_kv, ss[b]->max_tokens, di.sms, sh.dh, sh.g()));
    w->asplits = smax;
    const int kmax = std::max(std::max(sh.d, sh.Hq * sh.dh), sh.df);
    w->ld16 = (kmax + 63) / 64 * 64;
    const size_t pf = part_floats(sh, di.sms);
    const size_t apart = (size_t)sh.Hkv * smax * sh.g() * sh.dh, aml = (size_t)sh.Hkv * smax * sh.g() * 2;
    const size_t nu = (size_t)sh.n_units();
    const size_t sizes[] = {(size_t)US * sh.d * 4,           (size_t)US * sh.Hq * sh.dh * 4, (size_t)US * sh.Hq * sh.dh * 4,
                            (size_t)US * sh.df * 4,          (size_t)US * w->ld16 * 2,       (size_t)US * 4,
                            pf * 4,                          (size_t)US * apart * 4,         (size_t)US * aml * 4,
                            (size_t)US * sh.Hkv * 4,         (size_t)sh.L * US * sh.Hkv * 4, (size_t)sh.L * US * nu,
                            sizeof(int),                     (size_t)US * sh.d * 2};
    size_t total = 0;
    for (size_t z : sizes) total += (z + 255) / 256 * 256;
    if ((rc = w->arena.reserve(total))) return rc;
    w->x = (float*)w->arena.take(sizes[0]);
    w->q = (float*)w->arena.take(sizes[1]);
    w->o = (float*)w->arena.take(sizes[2]);
    w->h = (float*)w->arena.take(sizes[3]);
    w->x16 = (__half*)w->arena.take(sizes[4]);
    w->xinv = (float*)w->arena.take(sizes[5]);
    w->part = (float*)w->arena.take(sizes[6]);
    w->apart = (float*)w->arena.take(sizes[7]);
    w->aml = (float*)w->arena.take(sizes[8]);
    w->acnt = (int*)w->arena.take(sizes[9]);
    w->gmap = (int*)w->arena.take(sizes[10]);
    w->keep = (uint8_t*)w->arena.take(sizes[11]);
    w->err = (int*)w->arena.take(sizes[12]);
    w->x_stage = (uint16_t*)w->arena.take(sizes[13]);
    w->part_stride = (int64_t)apart;
    w->ml_stride = (int64_t)aml;
    TASP_CUDA(cudaMemset(w->arena.base, 0, w->arena.cap));
    // per layer and session: dense group -> plan group, and the kept channel units
    std::vector<int> gm((size_t)sh.L * US * sh.Hkv, -1);
    std::vector<uint8_t> kp((size_t)sh.L * US * nu, 0);
    for (int b = 0; b < n; ++b)
        for (int l = 0; l < sh.L; ++l) {
            const LayerPlan& lp = ss[b]->plan->layers[l];
            for (size_t i = 0; i < lp.keep_groups.size(); ++i)
                gm[((size_t)l * US + b) * sh.Hkv + lp.keep_groups[i]] = (int)i;
            for (int c : lp.keep_chans) kp[((size_t)l * US + b) * nu + c / sh.cu] = 1;
        }
    TASP_CUDA(cudaMemcpy(w->gmap, gm.data(), gm.size() * 4, cudaMemcpyHostToDevice));
    TASP_CUDA(cudaMemcpy(w->keep, kp.data(), kp.size(), cudaMemcpyHostToDevice));
    if (!g_skinny_attr) {  // before any stream capture
        TASP_CUDA(cudaFuncSetAttribute(skinny_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, SK_SMEM));
        TASP_CUDA(cudaFuncSetAttribute(skinny_kernel<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, SK_SMEM));
        TASP_CUDA(cudaFuncSetAttribute(skinny_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       SK_SMEM_BF16));
        g_skinny_attr = true;
    }
    *out = w.get();
    g_un.emplace(key, std::move(w));
    return TASP_OK;
}


// One union step on `s` (inputs in w.x_stage).
int enqueue_union(UnionWs& w, float* hidden, float* logits, cudaStream_t s, int* launches) {
    const int n = (int)w.ss.size();
    const Store& st = *w.ss[0]->plan->store;
    const Shape& sh = st.sh;
    const int g = sh.g(), qd = sh.Hq * sh.dh, nu = sh.n_units();
    int rc = 0, nl = 0;
    auto prep = [&](int mode, const float* src, int64_t src_ld, const uint16_t* in_bf16, const float* gamma, int K,
                    const int* gmap, int bf16 = 0, int layer = -1) -> int {
        PrepArgs p{};
        p.mode = mode;
        p.K = K;
        p.src = src;
        p.src_ld = src_ld;
        p.in_bf16 = in_bf16;
        p.gamma = gamma;
        p.eps = sh.eps;
        p.gmap = gmap;
        if (mode == PR_HEADS)
            for (int b = 0; b < n; ++b) p.oslot[b] = w.ss[b]->plan->layers[layer].oslot;
        p.g = g;
        p.dh = sh.dh;
        p.Hkv = sh.Hkv;
        p.x16 = w.x16;
        p.ld16 = w.ld16;
        p.xinv = w.xinv;
        p.bf16 = bf16;
        ++nl;
        return launch_pdl(prep_kernel, dim3(PREP_CS, n), dim3(256), 0, s, PREP_CS, p);
    };
    auto fin = [&](int S, int rows, const float* scale) {
        FinArgs f{};
        f.part = w.part;
        f.S = S;
        f.rows = rows;
        f.n = n;
        f.scale = scale;
        f.xinv = w.xinv;
        f.post = sh.qg ? std::ldexp(1.0f, -SK_GS_EXP) : 1.0f;
        return f;
    };
    for (int l = 0; l < sh.L; ++l) {
        const LayerStore& ls = st.layers[l];
        const int* gmap = w.gmap + (size_t)l * US * sh.Hkv;
        const bool last = l == sh.L - 1;
        int S = 0;
        // Q/K/V for every session's kept groups
        if ((rc = prep(PR_NORM, w.x, sh.d, l == 0 ? w.x_stage : nullptr, ls.g_attn, sh.d, nullptr))) return rc;
        if ((rc = launch_skinny(ls.qkv, false, sh.qkv_rows_dense(), sh.d, w.x16, w.ld16, w.part, w.err, S, s, ls.qkv_g, sh.qg))) return rc;
        ++nl;
        {
            QkvFin p{};
            p.f = fin(S, sh.qkv_rows_dense(), ls.qkv_s);
            p.g = g;
            p.dh = sh.dh;
            p.Hkv = sh.Hkv;
            p.gmap = gmap;
            p.q = w.q;
            p.q_stride = qd;
            for (int b = 0; b < n; ++b) {
                p.K[b] = w.ss[b]->K[l];
                p.V[b] = w.ss[b]->V[l];
                p.rope[b] = w.ss[b]->rope;
                p.pos[b] = w.ss[b]->d_pos;
                p.max_tokens[b] = w.ss[b]->max_tokens;
            }
            if ((rc = launch(finish_qkv_kernel, dim3(sh.Hkv * (g + 2), 4), dim3(US * (sh.dh / 8)), s, p))) return rc;
            ++nl;
        }
        // attention of each session over its own kept groups
        int mkv = 0;
        for (int b = 0; b < n; ++b) mkv = std::max(mkv, w.ss[b]->plan->layers[l].m_kv);
        if (mkv > 0) {
            AttnParams a{};
            a.q = w.q;
            a.o = w.o;
            a.q_stride = qd;
            for (int b = 0; b < n; ++b) {
                a.K[b] = w.ss[b]->K[l];
                a.V[b] = w.ss[b]->V[l];
                a.pos[b] = w.ss[b]->d_pos;
                a.max_tokens[b] = w.ss[b]->max_tokens;
                a.m_kv[b] = w.ss[b]->plan->layers[l].m_kv;
                a.oslot[b] = w.ss[b]->plan->layers[l].oslot;  // query-head plans: dropped heads are not written
            }
            a.qscale = (float)(1.0 / std::sqrt((double)sh.dh) * 1.4426950408889634);
            a.part = w.apart;
            a.ml = w.aml;
            a.cnt = w.acnt;
            a.part_stride = w.part_stride;
            a.ml_stride = w.ml_stride;
            a.cnt_stride = sh.Hkv;
            DevInfo di;
            if ((rc = device_info(di))) return rc;
            int S_att = 0;
            for (int b = 0; b < n; ++b)
                S_att = std::max(S_att, attn_splits(a.m_kv[b], w.ss[b]->max_tokens, di.sms, sh.dh, g, UN_ATT_CS));
            if ((rc = launch_attention(a, sh.dh, g, mkv, S_att, n, s, UN_ATT_CS))) return rc;
            ++nl;
        }
        // O projection + residual (the dropped heads are zero in the scattered input)
        if ((rc = prep(PR_HEADS, w.o, qd, nullptr, nullptr, qd, gmap, 0, l))) return rc;
        if ((rc = launch_skinny(ls.o, false, sh.d, qd, w.x16, w.ld16, w.part, w.err, S, s, ls.o_g, sh.qg))) return rc;
        ++nl;
        {
            ResFin p{};
            p.f = fin(S, sh.d, ls.o_s);
            p.x = w.x;
            p.ld = sh.d;
            p.hidden = nullptr;
            if ((rc = launch(finish_resid_kernel, dim3((sh.d * US + 255) / 256), dim3(256), s, p))) return rc;
            ++nl;
        }
        // gate/up + SiLU(gate) * up, zero for the dropped channel units
        if ((rc = prep(PR_NORM, w.x, sh.d, nullptr, ls.g_mlp, sh.d, nullptr))) return rc;
        if ((rc = launch_skinny(ls.gu, false, 2 * sh.df, sh.d, w.x16, w.ld16, w.part, w.err, S, s, ls.gu_g, sh.qg))) return rc;
        ++nl;
        {
            GuFin p{};
            p.f = fin(S, 2 * sh.df, ls.gu_s);
            p.h = w.h;
            p.ld = sh.df;
            p.keep = w.keep + (size_t)l * US * nu;
            p.n_units = nu;
            p.cu = sh.cu;
            if ((rc = launch(finish_gu_kernel, dim3((sh.df * US + 255) / 256), dim3(256), s, p))) return rc;
            ++nl;
        }
        // down projection + residual
        if ((rc = prep(PR_COPY, w.h, sh.df, nullptr, nullptr, sh.df, nullptr))) return rc;
        if ((rc = launch_skinny(ls.down, false, sh.d, sh.df, w.x16, w.ld16, w.part, w.err, S, s, ls.down_g, sh.qg))) return rc;
        ++nl;
        {
            ResFin p{};
            p.f = fin(S, sh.d, ls.down_s);
            p.x = w.x;
            p.ld = sh.d;
            p.hidden = last ? hidden : nullptr;
            if ((rc = launch(finish_resid_kernel, dim3((sh.d * US + 255) / 256), dim3(256), s, p))) return rc;
            ++nl;
        }
    }
    // final RMSNorm + LM head (BF16) for all sessions in one weight pass
    if (logits) {
        int S = 0;
        if ((rc = prep(PR_NORM, w.x, sh.d, nullptr, st.g_final, sh.d, nullptr, 1))) return rc;
        if ((rc = launch_skinny(st.lm_head, true, sh.vocab, sh.d, w.x16, w.ld16, w.part, w.err, S, s))) return rc;
        ++nl;
        LogitFin p{};
        p.f = fin(S, sh.vocab, nullptr);
        p.logits = logits;
        if ((rc = launch(finish_logits_kernel, dim3((unsigned)(((int64_t)sh.vocab * US + 255) / 256)), dim3(256), s, p)))
            return rc;
        ++nl;
    }
    UnAdvance ad{};
    ad.n = n;
    for (int b = 0; b < n; ++b) ad.pos[b] = w.ss[b]->d_pos;
    if ((rc = launch(union_advance_kernel, dim3(1), dim3(32), s, ad))) return rc;
    ++nl;
    if (launches) *launches = nl;
    return TASP_OK;
}

int union_check(Session* const* ss, int n, bool step) {
    if (n < 1 || n > US) return fail(TASP_EINVAL, "a union step holds 1 to 16 sessions");
    for (int b = 0; b < n; ++b)
        if (!ss[b] || ss[b]->magic != SESSION_MAGIC) return fail(TASP_EINVAL, "invalid session handle");
    const Store* st = ss[0]->plan->store;
    for (int b = 0; b < n; ++b) {
        if (ss[b]->plan->store != st) return fail(TASP_EMASK, "union step sessions must share one weight store");
        if (step && ss[b]->pos >= ss[b]->max_tokens) return fail(TASP_ECAP, "KV capacity exhausted");
        for (int c = 0; c < b; ++c)
            if (ss[c] == ss[b]) return fail(TASP_EINVAL, "a session appears twice in one step");
    }
    const Shape& sh = st->sh;
    if (sh.d % SK_BK || (sh.Hq * sh.dh) % SK_BK || sh.df % SK_BK)
        return fail(TASP_EUNSUP, "union decode needs d, Hq*dh and d_ff that are multiples of 128");
    return TASP_OK;
}

}  // namespace

void union_drop(Session* se) {
    std::lock_guard<std::mutex> lk(g_un_mu);
    for (auto it = g_un.begin(); it != g_un.end();) {
        if (std::find(it->first.begin(), it->first.end(), se) != it->first.end()) {
            if (it->second->graph.exec) cudaGraphExecDestroy(it->second->graph.exec);
            it->second->arena.release();
            it = g_un.erase(it);
        } else {
            ++it;
        }
    }
}

}  // namespace tasp

using namespace tasp;

extern "C" int tasp_decode_step_union(tasp_session* const* sessions, int32_t n, const void* d_x_bf16,
                                      float* d_hidden_out, float* d_logits, void* stream) {
    if (!sessions || !d_x_bf16) return fail(TASP_EINVAL, "null argument");
    int rc = check_aligned({{d_x_bf16, 2}, {d_hidden_out, 4}, {d_logits, 4}});
    if (rc) return rc;
    Session* const* ss = reinterpret_cast<Session* const*>(sessions);
    rc = union_check(ss, n, true);
    if (rc) return rc;
    const Shape& sh = ss[0]->plan->store->sh;
    if (d_logits && sh.vocab == 0) return fail(TASP_EINVAL, "model has no LM head");
    UnionWs* w = nullptr;
    if ((rc = union_get(ss, n, &w))) return rc;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    TASP_CUDA(cudaMemcpyAsync(w->x_stage, d_x_bf16, (size_t)n * sh.d * 2, cudaMemcpyDeviceToDevice, s));
    StepGraph& gr = w->graph;
    if (!(gr.exec && gr.hidden == d_hidden_out && gr.logits == d_logits)) {
        if (gr.exec) {
            cudaGraphExecDestroy(gr.exec);
            gr.exec = nullptr;
        }
        cudaStream_t cap;
        TASP_CUDA(cudaStreamCreateWithFlags(&cap, cudaStreamNonBlocking));
        cudaGraph_t graph = nullptr;
        TASP_CUDA(cudaStreamBeginCapture(cap, cudaStreamCaptureModeThreadLocal));
        int nl = 0;
        const int erc = enqueue_union(*w, d_hidden_out, d_logits, cap, &nl);
        const cudaError_t ce = cudaStreamEndCapture(cap, &graph);
        cudaStreamDestroy(cap);
        if (erc) {
            if (graph) cudaGraphDestroy(graph);
            return erc;
        }
        if (ce != cudaSuccess) return cuda_fail(ce, "union step capture");
        const cudaError_t ie = cudaGraphInstantiate(&gr.exec, graph, 0);
        cudaGraphDestroy(graph);
        if (ie != cudaSuccess) return cuda_fail(ie, "union step graph instantiation");
        gr.hidden = d_hidden_out;
        gr.logits = d_logits;
        gr.launches = nl;
    }
    TASP_CUDA(cudaGraphLaunch(gr.exec, s));
    for (int b = 0; b < n; ++b) ss[b]->pos += 1;
    return TASP_OK;
}

extern "C" int tasp_union_status(tasp_session* const* sessions, int32_t n, int32_t* device_error, int32_t* launches) {
    if (!sessions) return fail(TASP_EINVAL, "null argument");
    Session* const* ss = reinterpret_cast<Session* const*>(sessions);
    int rc = union_check(ss, n, false);
    if (rc) return rc;
    UnionWs* w = nullptr;
    if ((rc = union_get(ss, n, &w))) return rc;
    int e = 0;
    TASP_CUDA(cudaMemcpy(&e, w->err, sizeof(int), cudaMemcpyDeviceToHost));
    if (device_error) *device_error = e;
    if (launches) *launches = w->graph.launches;
    return TASP_OK;
}
