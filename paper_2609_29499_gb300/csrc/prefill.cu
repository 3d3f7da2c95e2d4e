// Prefill of one prompt with a compiled plan (Fig. 1 "one launch plan for prefill"), sm_103a.
//
// Per layer: row RMSNorm -> QKV GEMM -> rotary + KV-cache write -> causal GQA attention
// over the kept heads -> O GEMM (+ residual) -> row RMSNorm -> gate/up GEMM with fused
// SiLU(gate) * up -> down GEMM (+ residual). The projections are dense GEMMs over the
// plan's compacted panels on the 5th-generation tensor cores:
//  * operands FP16 (INT8 weights are exact in FP16; activations keep 11 significant
//    bits), FP32 accumulators in tensor memory, per-weight-row scales in the epilogue;
//  * one persistent CTA per SM walks 128 x 256 output tiles: warp 0 streams 128 x 64 and
//    256 x 64 operand tiles with TMA (128-byte swizzle) into a 4-stage ring, warp 1
//    allocates 512 TMEM columns (two accumulators) and issues tcgen05.mma (M = 128,
//    N = 256, K = 16 per instruction), warps 2-5 read one accumulator back with tcgen05.ld
//    and apply the epilogue while the MMAs fill the other;
//  * every mbarrier wait is bounded and reports to the session's device error word.
// Attention is a causal flash-attention over the kept heads: for head dim 128 on tcgen05
// (S = Q K^T and O += P V in tensor memory, FP16 operands, softmax warps owning one query
// row each), for head dim 64 on mma.sync with FP16 operands.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cmath>
#include <mutex>

#include "tasp_internal.h"
#include "tc_ptx.cuh"

namespace tasp {

namespace {

// ------------------------------------------------------------------ PTX helpers (tc_ptx.cuh)
using namespace tc;

// Programmatic dependent launch through the prefill chain: each kernel lets the next one launch
// at once, and waits (the previous grid complete, its writes visible) before it reads what the
// previous kernels wrote or writes what they may still read. Only the GEMM's constant weight
// tiles and the kernels' set-up (barriers, tensor memory) come before the wait.
__device__ __forceinline__ void pf_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pf_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ------------------------------------------------------------------ GEMM
// Persistent GEMM on the 5th-generation tensor cores: one CTA per SM walks 128 x BN output
// tiles (M fastest, so the CTAs in flight share weight tiles in L2), with two BN-column TMEM
// accumulators: the MMA warp fills one while the epilogue warps drain the other. BN = 256,
// or 128 when 256-column tiles would not fill one wave of SMs (short prompts).
constexpr int BM = 128, BN = 256, BK = 64;
constexpr int A_BYTES = BM * BK * 2;
constexpr int GEMM_THREADS = 192;

enum EpiMode { EP_STORE = 0, EP_RESID = 1, EP_SWIGLU = 2 };

struct GemmArgs {
    int M, N, K;
    const float* scale;  // [N] scale of each weight row
    float* out;          // STORE: out[m][n] = s_n acc; RESID: out[m][n] += s_n acc
    int ldo;
    __half* hout;        // SWIGLU: hout[m][n/2] = SiLU(s_g gate) * (s_u up), n even = gate
    int ldh;
    int mode;
    int vec;             // rows of out / hout are 16-byte aligned (vector stores)
    int* err;
    int pdl;             // launched as a programmatic dependent: weight tiles of the first stages go
                         // out before the dependency wait
};

// Epilogue of 32 accumulator columns [nb, nb + 32) of one output row.
__device__ __forceinline__ void gemm_epi32(const GemmArgs& g, int row, int nb, const uint32_t (&r)[32]) {
    if (g.vec && nb + 32 <= g.N) {
        float sc[32];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float4 t = __ldg(reinterpret_cast<const float4*>(g.scale + nb) + k);
            sc[4 * k] = t.x;
            sc[4 * k + 1] = t.y;
            sc[4 * k + 2] = t.z;
            sc[4 * k + 3] = t.w;
        }
        if (g.mode == EP_SWIGLU) {
            uint32_t hw[8];
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
                const float a0 = __uint_as_float(r[2 * j]) * sc[2 * j];
                const float b0 = __uint_as_float(r[2 * j + 1]) * sc[2 * j + 1];
                const float a1 = __uint_as_float(r[2 * j + 2]) * sc[2 * j + 2];
                const float b1 = __uint_as_float(r[2 * j + 3]) * sc[2 * j + 3];
                const __half2 h = __floats2half2_rn(a0 / (1.0f + expf(-a0)) * b0, a1 / (1.0f + expf(-a1)) * b1);
                hw[j >> 1] = *reinterpret_cast<const uint32_t*>(&h);
            }
            uint4* dst = reinterpret_cast<uint4*>(g.hout + (int64_t)row * g.ldh + (nb >> 1));
            dst[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            dst[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
        } else {
            float4* o4 = reinterpret_cast<float4*>(g.out + (int64_t)row * g.ldo + nb);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                float4 v = make_float4(__uint_as_float(r[4 * k]) * sc[4 * k], __uint_as_float(r[4 * k + 1]) * sc[4 * k + 1],
                                       __uint_as_float(r[4 * k + 2]) * sc[4 * k + 2],
                                       __uint_as_float(r[4 * k + 3]) * sc[4 * k + 3]);
                if (g.mode == EP_RESID) {
                    const float4 t = o4[k];
                    v.x += t.x;
                    v.y += t.y;
                    v.z += t.z;
                    v.w += t.w;
                }
                o4[k] = v;
            }
        }
        return;
    }
    if (g.mode == EP_SWIGLU) {
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const int n = nb + j;
            if (n + 1 < g.N) {
                const float a = __uint_as_float(r[j]) * g.scale[n];
                const float b = __uint_as_float(r[j + 1]) * g.scale[n + 1];
                g.hout[(int64_t)row * g.ldh + (n >> 1)] = __float2half_rn(a / (1.0f + expf(-a)) * b);
            }
        }
    } else {
        float* o = g.out + (int64_t)row * g.ldo;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int n = nb + j;
            if (n < g.N) {
                const float v = __uint_as_float(r[j]) * g.scale[n];
                if (g.mode == EP_RESID)
                    o[n] += v;
                else
                    o[n] = v;
            }
        }
    }
}

// Warp 0 streams the A (activation) and B (weight) k-blocks of all the CTA's tiles through a
// TMA ring (4 stages at BN = 256, 6 at BN = 128) that runs on across tile boundaries; warp 1
// issues tcgen05.mma; warps 2-5 read an accumulator with tcgen05.ld and run the epilogue.
template <int BNT>
struct PgCfg {
    static constexpr int B_BYTES = BNT * BK * 2;
    static constexpr int STAGES = BNT == 256 ? 4 : 6;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int SMEM = STAGES * STAGE_BYTES + 1024;
    static constexpr uint32_t IDESC = idesc_f16(BM, BNT);
    static constexpr uint32_t TMEM_COLS = 2 * BNT;
};

template <int BNT>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    gemm_persist_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        const GemmArgs g) {
    using C = PgCfg<BNT>;
    constexpr int BN = BNT, PG_STAGES = C::STAGES, PG_STAGE_BYTES = C::STAGE_BYTES;
    constexpr uint32_t IDESC = C::IDESC;
    extern __shared__ uint8_t smraw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_full[PG_STAGES], bar_empty[PG_STAGES], acc_full[2], acc_empty[2];
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mt = (g.M + BM - 1) / BM, ntl = (g.N + BN - 1) / BN;
    const int ntiles = mt * ntl;
    const int nk = (g.K + BK - 1) / BK;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int s = 0; s < PG_STAGES; ++s) {
            mbar_init(smem_u32(&bar_full[s]), 1);
            mbar_init(smem_u32(&bar_empty[s]), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(smem_u32(&acc_full[a]), 1);
            mbar_init(smem_u32(&acc_empty[a]), 4);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                     "r"(C::TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = tmem_base;
    pf_trigger();

    if (warp == 0) {
        if (lane == 0) {  // ---- TMA producer: k-blocks of all this CTA's tiles, back to back
            // the first stages' weight tiles go out before the dependency wait (the panels are
            // constant); the activation tiles, written by the previous kernel, after it
            int kbg = 0;   // k-blocks issued so far
            int pend = 0;  // leading stages whose activation tile is still due (their k-blocks
                           // are the CTA's first ones, walked again here)
            bool waited = !g.pdl;
            auto flush = [&]() {
                pf_wait();
                waited = true;
                int i = 0;
                for (int t2 = blockIdx.x; t2 < ntiles && i < pend; t2 += gridDim.x)
                    for (int kb2 = 0; kb2 < nk && i < pend; ++kb2, ++i)
                        tma_load_2d(smem_u32(sm + i * PG_STAGE_BYTES), &tmA, kb2 * BK, (t2 % mt) * BM,
                                    smem_u32(&bar_full[i]));
            };
            for (int t = blockIdx.x; t < ntiles; t += gridDim.x) {
                const int m0 = (t % mt) * BM, n0 = (t / mt) * BN;
                for (int kb = 0; kb < nk; ++kb, ++kbg) {
                    const int s = kbg % PG_STAGES;
                    if (kbg >= PG_STAGES)
                        mbar_wait(smem_u32(&bar_empty[s]), ((kbg / PG_STAGES) - 1) & 1, &abort_flag, g.err);
                    const uint32_t fb = smem_u32(&bar_full[s]);
                    mbar_expect_tx(fb, PG_STAGE_BYTES);
                    const uint32_t a = smem_u32(sm + s * PG_STAGE_BYTES);
                    if (!waited) {  // kbg < PG_STAGES here
                        tma_load_2d(a + A_BYTES, &tmB, kb * BK, n0, fb);
                        if (++pend == PG_STAGES) flush();
                    } else if (g.pdl) {  // the weight tile first (2,048 tokens: 15.44 against 15.75 ms)
                        tma_load_2d(a + A_BYTES, &tmB, kb * BK, n0, fb);
                        tma_load_2d(a, &tmA, kb * BK, m0, fb);
                    } else {  // the activation tile first (8,192 tokens: 67.9 against 69.2 ms)
                        tma_load_2d(a, &tmA, kb * BK, m0, fb);
                        tma_load_2d(a + A_BYTES, &tmB, kb * BK, n0, fb);
                    }
                }
            }
            if (!waited) flush();  // fewer k-blocks than stages
            for (int k = max(0, kbg - PG_STAGES); k < kbg; ++k)  // no copy may outlive the CTA
                mbar_wait(smem_u32(&bar_full[k % PG_STAGES]), (k / PG_STAGES) & 1, &abort_flag, g.err, false);
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---- MMA issuer
            int kbg = 0, it = 0;
            for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++it) {
                const int a = it & 1;
                if (it >= 2) mbar_wait(smem_u32(&acc_empty[a]), ((it >> 1) - 1) & 1, &abort_flag, g.err);
                fence_after();
                for (int kb = 0; kb < nk; ++kb, ++kbg) {
                    const int s = kbg % PG_STAGES;
                    mbar_wait(smem_u32(&bar_full[s]), (kbg / PG_STAGES) & 1, &abort_flag, g.err);
                    fence_after();
                    const uint32_t sa = smem_u32(sm + s * PG_STAGE_BYTES), sb = sa + A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint32_t accum = (kb > 0 || kk > 0) ? 1u : 0u;
                        asm volatile(
                            "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
                            " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem + (uint32_t)BN * a),
                            "l"(sw128_desc(sa + kk * 32)), "l"(sw128_desc(sb + kk * 32)), "r"(IDESC), "r"(accum)
                            : "memory");
                    }
                    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                                     smem_u32(&bar_empty[s]))
                                 : "memory");
                }
                asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                                 smem_u32(&acc_full[a]))
                             : "memory");
            }
        }
    } else {  // ---- epilogue warps 2..5: TMEM lanes 32 (warp % 4) ..
        pf_wait();  // the outputs (and the residual rows) belong to the chain
        const int q = warp & 3;
        int it = 0;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++it) {
            const int a = it & 1;
            const int m0 = (t % mt) * BM, n0 = (t / mt) * BN;
            mbar_wait(smem_u32(&acc_full[a]), (it >> 1) & 1, &abort_flag, g.err);
            fence_after();
            const int row = m0 + 32 * q + lane;
#pragma unroll 1
            for (int c0 = 0; c0 < BN; c0 += 32) {
                uint32_t r[32];
                asm volatile(
                    "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
                    "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
                    : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
                      "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
                      "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
                      "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
                      "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
                    : "r"(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)BN * a + (uint32_t)c0));
                asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
                if (row < g.M) gemm_epi32(g, row, n0 + c0, r);
            }
            fence_before();
            __syncwarp();
            if (lane == 0)
                asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&acc_empty[a])) : "memory");
        }
    }
    fence_before();
    __syncthreads();
    fence_after();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::TMEM_COLS) : "memory");
}

// ------------------------------------------------------------------ elementwise kernels
// x^ = half(x / sqrt(mean(x^2) + eps) * gamma) per row; row 0 source may be BF16 input embeddings.
__global__ void __launch_bounds__(256) rmsnorm_rows_kernel(const float* __restrict__ X, const uint16_t* x_bf16,
                                                            float* X_init, int d, const float* __restrict__ gamma,
                                                            float eps, __half* out, int ldo) {
    pf_wait();
    pf_trigger();
    __shared__ float red[8];
    const int t = blockIdx.x, tid = threadIdx.x;
    const float* xr = X + (int64_t)t * d;
    float ss = 0.f;
    for (int i = tid; i < d; i += 256) {
        float v;
        if (x_bf16) {
            v = __uint_as_float((uint32_t)x_bf16[(int64_t)t * d + i] << 16);
            X_init[(int64_t)t * d + i] = v;
        } else {
            v = xr[i];
        }
        ss = fmaf(v, v, ss);
    }
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((tid & 31) == 0) red[tid >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    const float inv = 1.0f / sqrtf(__fdiv_rn(tot, (float)d) + eps);
    for (int i = tid; i < d; i += 256) {
        const float v = x_bf16 ? __uint_as_float((uint32_t)x_bf16[(int64_t)t * d + i] << 16) : xr[i];
        out[(int64_t)t * ldo + i] = __float2half_rn((v * inv) * gamma[i]);
    }
}

// The same with 16-byte loads and 8-byte stores (d % 4 == 0, FP32 rows; 16-byte aligned X and
// gamma, 8-byte aligned out rows).
__global__ void __launch_bounds__(256) rmsnorm_rows_vec_kernel(const float* __restrict__ X, int d,
                                                                const float* __restrict__ gamma, float eps,
                                                                __half* out, int ldo) {
    pf_wait();
    pf_trigger();
    __shared__ float red[8];
    const int t = blockIdx.x, tid = threadIdx.x;
    const float4* xr = reinterpret_cast<const float4*>(X + (int64_t)t * d);
    const int n4 = d >> 2;
    float ss = 0.f;
    for (int f = tid; f < n4; f += 256) {
        const float4 v = xr[f];
        ss = fmaf(v.x, v.x, ss);
        ss = fmaf(v.y, v.y, ss);
        ss = fmaf(v.z, v.z, ss);
        ss = fmaf(v.w, v.w, ss);
    }
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((tid & 31) == 0) red[tid >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    const float inv = 1.0f / sqrtf(__fdiv_rn(tot, (float)d) + eps);
    const float4* g4 = reinterpret_cast<const float4*>(gamma);
    uint2* o2 = reinterpret_cast<uint2*>(out + (int64_t)t * ldo);
    for (int f = tid; f < n4; f += 256) {
        const float4 v = xr[f], gm = g4[f];
        const __half2 a = __floats2half2_rn((v.x * inv) * gm.x, (v.y * inv) * gm.y);
        const __half2 b = __floats2half2_rn((v.z * inv) * gm.z, (v.w * inv) * gm.w);
        o2[f] = make_uint2(*reinterpret_cast<const uint32_t*>(&a), *reinterpret_cast<const uint32_t*>(&b));
    }
}

// Projected rows Y [T][qkv rows] (group-major panel order, scaled) -> rotated queries (FP32,
// [m_q][T][dh]) and the plan-bound KV cache (BF16 keys rotated, values as is) at 0..T-1.
// Rotary embedding on q and k, KV-cache write (BF16); optionally also the tensor-core
// attention's operands Qh = FP16(q * qscale) [head][T][dh] and Kh = FP16 of the cached BF16
// keys [group][T][dh] (the transposed values come from v_transpose_kernel).
__global__ void rope_kv_kernel(const float* __restrict__ Y, int ldy, int T, int g, int dh,
                               const float2* __restrict__ rope, float* Qf, uint16_t* Kc, uint16_t* Vc,
                               int max_tokens, __half* Qh, float qscale, __half* Kh,
                               const int16_t* __restrict__ blk_of) {
    pf_wait();
    pf_trigger();
    const int t = blockIdx.x, jl = blockIdx.y;
    const int half = dh >> 1;
    for (int w = threadIdx.x; w < (g + 2) * half; w += blockDim.x) {
        const int hh = w / half, i = w - hh * half;
        // the panel's d_h-column block of (group slot, head); -1: a dropped head, whose query
        // slot is written as zeros (its attention output is never used)
        const int blk = blk_of ? blk_of[jl * (g + 2) + hh] : jl * (g + 2) + hh;
        const int col = blk * dh + i;
        float y0 = blk >= 0 ? Y[(int64_t)t * ldy + col] : 0.f, y1 = blk >= 0 ? Y[(int64_t)t * ldy + col + half] : 0.f;
        if (hh <= g) {
            const float2 cs = rope[(int64_t)t * half + i];
            const float a = y0 * cs.x - y1 * cs.y, b = y1 * cs.x + y0 * cs.y;
            y0 = a;
            y1 = b;
        }
        if (hh < g) {
            const int64_t qrow = (int64_t)(jl * g + hh) * T + t;
            if (Qf) {
                float* q = Qf + qrow * dh;
                q[i] = y0;
                q[i + half] = y1;
            }
            if (Qh) {
                Qh[qrow * dh + i] = __float2half_rn(y0 * qscale);
                Qh[qrow * dh + i + half] = __float2half_rn(y1 * qscale);
            }
        } else {
            uint16_t* dst = (hh == g ? Kc : Vc) + ((int64_t)jl * max_tokens + t) * dh;
            __nv_bfloat16 b0 = __float2bfloat16_rn(y0), b1 = __float2bfloat16_rn(y1);
            dst[i] = *reinterpret_cast<uint16_t*>(&b0);
            dst[i + half] = *reinterpret_cast<uint16_t*>(&b1);
            const __half h0 = __float2half_rn(__bfloat162float(b0)), h1 = __float2half_rn(__bfloat162float(b1));
            if (hh == g && Kh) {
                Kh[((int64_t)jl * T + t) * dh + i] = h0;
                Kh[((int64_t)jl * T + t) * dh + i + half] = h1;
            }
        }
    }
}

// FP16 of the cached BF16 values of one KV group, transposed: VT [group][128][Tp] from
// V [group][max_tokens][128]; 64 tokens per CTA through a shared tile (coalesced both ways).
__global__ void __launch_bounds__(256) v_transpose_kernel(const uint16_t* __restrict__ V, int max_tokens, int T,
                                                           __half* VT, int Tp) {
    pf_wait();
    pf_trigger();
    __shared__ __half tile[128][64 + 8];
    const int t0 = blockIdx.x * 64, jl = blockIdx.y, tid = threadIdx.x;
    const uint16_t* src = V + ((int64_t)jl * max_tokens + t0) * 128;
    for (int c = tid; c < 64 * 16; c += 256) {  // 64 tokens x 16 chunks of 8 dims
        const int tt = c >> 4, dc = (c & 15) * 8;
        uint4 w = make_uint4(0, 0, 0, 0);
        if (t0 + tt < T) w = *reinterpret_cast<const uint4*>(src + (int64_t)tt * 128 + dc);
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            tile[dc + 2 * k][tt] = __float2half_rn(__uint_as_float(u[k] << 16));
            tile[dc + 2 * k + 1][tt] = __float2half_rn(__uint_as_float(u[k] & 0xffff0000u));
        }
    }
    __syncthreads();
    for (int c = tid; c < 128 * 8; c += 256) {  // 128 dims x 8 chunks of 8 tokens
        const int dd = c >> 3, tc = (c & 7) * 8;
        if (t0 + tc + 8 <= Tp)
            *reinterpret_cast<uint4*>(VT + ((int64_t)jl * 128 + dd) * Tp + t0 + tc) =
                *reinterpret_cast<const uint4*>(&tile[dd][tc]);
    }
}

// INT8 panel rows (optionally through a row map) -> FP16 rows with a padded stride. A grouped
// store's rows become q s_g 2^F16_GS_EXP, with s_g the BF16 scale of column group k / qg in
// panel order (gs [rows][gld]): exact in FP32, one rounding to FP16.
constexpr int F16_GS_EXP = 8;  // keeps q s_g normal in FP16 for scales down to ~2^-22
__global__ void i8_to_f16_kernel(const int8_t* __restrict__ src, const int32_t* map, int64_t lds, int K,
                                 __half* dst, int ldd, const uint16_t* __restrict__ gs, int gld, int qg) {
    const int r = blockIdx.x;
    const int8_t* s = src + (int64_t)(map ? map[r] : r) * lds;
    __half* d = dst + (int64_t)r * ldd;
    for (int k = threadIdx.x; k < ldd; k += blockDim.x) {
        if (!gs) {
            d[k] = __int2half_rn(k < K ? (int)s[k] : 0);
        } else {
            const float sg = k < K ? __uint_as_float((uint32_t)gs[(int64_t)r * gld + k / qg] << 16) : 0.f;
            d[k] = __float2half_rn(k < K ? (float)s[k] * ldexpf(sg, F16_GS_EXP) : 0.f);
        }
    }
}

// ------------------------------------------------------------------ causal attention
// Flash attention on mma.sync m16n8k16 with FP16 operands: the BF16 K/V tiles are widened to
// FP16 in shared memory after they land (exact: 8 significant bits fit in 11, for values in
// FP16's normal range), queries and probabilities enter as FP16 (11 significant bits, like
// the GEMM operands of the prefill), accumulation and the online softmax stay FP32.
constexpr int PA_WARPS = 8;
constexpr int PA_QB = PA_WARPS * 16;  // queries per CTA (16 per warp)

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
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
__device__ __forceinline__ void mma16816_f16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_h2(float x0, float x1) {
    const __half2 h = __floats2half2_rn(x0, x1);
    return *reinterpret_cast<const uint32_t*>(&h);
}

// One CTA: one kept query head, 128 consecutive queries (16 per warp: fragment rows r and
// r + 8 of lane l are queries l / 4 and l / 4 + 8 of the warp). Keys stream in tiles of
// PA_KT = 64 through a double-buffered cp.async ring in dynamic shared memory; the online
// softmax is updated once per tile.
constexpr int PA_KT = 64;
template <int DH>
struct PaCfg {
    static constexpr int ROWB = DH * 2 + 16;  // padded row: conflict-free ldmatrix
    static constexpr int TILEB = PA_KT * ROWB;
    static constexpr int SMEM = 2 * 2 * TILEB;  // [stage][K, V]
};

template <int DH>
__global__ void __launch_bounds__(PA_WARPS * 32, 1) attn_prefill_kernel(const float* __restrict__ Qf, const uint16_t* K,
                                                                     const uint16_t* V, int T, int max_tokens, int g,
                                                                     float qscale, __half* O, int ldo,
                                                                     const int16_t* __restrict__ oslot) {
    pf_wait();
    pf_trigger();
    using C = PaCfg<DH>;
    constexpr int ROWB = C::ROWB, TILEB = C::TILEB, KS = DH / 16, NT = DH / 8, CPR = DH * 2 / 16;
    constexpr int SUB = PA_KT / 16;  // 16-key sub-tiles per tile
    extern __shared__ __align__(128) uint8_t pa_sm[];
    auto tile = [&](int st, int kv) { return pa_sm + (2 * st + kv) * TILEB; };
    // grid (heads, query blocks): blocks are scheduled x-fastest, so the longest query blocks
    // of every head run first and the short ones fill the tail
    const int h = blockIdx.x, jl = h / g;
    const int q0 = (gridDim.y - 1 - blockIdx.y) * PA_QB;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int qw = q0 + warp * 16;                // this warp's first query
    const int rq[2] = {qw + (lane >> 2), qw + 8 + (lane >> 2)};  // queries of this lane's fragment rows
    const int qc = (lane & 3) * 2;
    const uint16_t* Kg = K + (int64_t)jl * max_tokens * DH;
    const uint16_t* Vg = V + (int64_t)jl * max_tokens * DH;
    const int kend = min(T, q0 + PA_QB);  // keys needed by this CTA: 0 .. kend-1
    const int ntile = (kend + PA_KT - 1) / PA_KT;

    uint32_t qa[KS][4];
#pragma unroll
    for (int ks = 0; ks < KS; ++ks)
#pragma unroll
        for (int i = 0; i < 4; ++i) {  // a0: row r, k 0-7; a1: row r+8; a2: row r, k 8-15; a3: row r+8
            const int rr = rq[i & 1];
            const int col = ks * 16 + (i >> 1) * 8 + qc;
            float x0 = 0.f, x1 = 0.f;
            if (rr < T) {
                const float* qp = Qf + ((int64_t)h * T + rr) * DH + col;
                x0 = qp[0] * qscale;
                x1 = qp[1] * qscale;
            }
            qa[ks][i] = pack_h2(x0, x1);
        }
    float acc[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};

    auto issue = [&](int kt, int st) {
        uint8_t* kt_s = tile(st, 0);
        uint8_t* vt_s = tile(st, 1);
        for (int c = tid; c < PA_KT * CPR; c += PA_WARPS * 32) {
            const int r = c / CPR, cc = c - r * CPR;
            const int pos = kt * PA_KT + r;
            const bool ok = pos < kend;
            const int64_t off = (int64_t)(ok ? pos : 0) * DH + cc * 8;
            cp_async16(smem_u32(kt_s + r * ROWB + cc * 16), Kg + off, ok ? 16 : 0);
            cp_async16(smem_u32(vt_s + r * ROWB + cc * 16), Vg + off, ok ? 16 : 0);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    // BF16 -> FP16 in place, 8 elements per 16-byte chunk
    auto widen = [&](int st) {
        for (int c = tid; c < 2 * PA_KT * CPR; c += PA_WARPS * 32) {
            const int kv = c / (PA_KT * CPR), rc = c - kv * PA_KT * CPR;
            const int r = rc / CPR, cc = rc - r * CPR;
            uint4* p = reinterpret_cast<uint4*>(tile(st, kv) + r * ROWB + cc * 16);
            uint4 w = *p;
            uint32_t* u = reinterpret_cast<uint32_t*>(&w);
#pragma unroll
            for (int k = 0; k < 4; ++k)
                u[k] = pack_h2(__uint_as_float(u[k] << 16), __uint_as_float(u[k] & 0xffff0000u));
            *p = w;
        }
    };
    if (ntile > 0) issue(0, 0);
    for (int kt = 0; kt < ntile; ++kt) {
        const int st = kt & 1;
        if (kt + 1 < ntile) {
            issue(kt + 1, st ^ 1);
            asm volatile("cp.async.wait_group 1;" ::: "memory");
        } else {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
        }
        __syncthreads();
        widen(st);
        __syncthreads();
        const int base = kt * PA_KT;
        if (base <= qw + 15) {  // some key of the tile is visible to this warp's queries
            const uint8_t* kt_s = tile(st, 0);
            const uint8_t* vt_s = tile(st, 1);
            // scores of the tile: sub-tile u, keys base + 16u + {qc, qc+1} (s[u][0][.]) and
            // + 8 + {qc, qc+1} (s[u][1][.]); element [2i + e]: row r (i = 0) / r + 8, key +e
            float sc[SUB][2][4];
#pragma unroll
            for (int u = 0; u < SUB; ++u)
#pragma unroll
                for (int e = 0; e < 4; ++e) sc[u][0][e] = sc[u][1][e] = 0.f;
            // k-steps outer, sub-tiles inner: 2 SUB independent accumulation chains in flight
            // (sub-tiles past the warp's last query are computed and masked below)
            const uint32_t krow0 =
                smem_u32(kt_s + (8 * ((lane >> 4) & 1) + (lane & 7)) * ROWB + 16 * ((lane >> 3) & 1));
#pragma unroll
            for (int ks = 0; ks < KS; ++ks)
#pragma unroll
                for (int u = 0; u < SUB; ++u) {
                    uint32_t b00, b01, b10, b11;
                    ldsm_x4(krow0 + 16 * u * ROWB + ks * 32, b00, b01, b10, b11);
                    mma16816_f16(sc[u][0], qa[ks], b00, b01);
                    mma16816_f16(sc[u][1], qa[ks], b10, b11);
                }
            float (&pv)[SUB][2][4] = sc;  // probabilities overwrite the scores in place
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                float mt = -INFINITY;
#pragma unroll
                for (int u = 0; u < SUB; ++u)
#pragma unroll
                    for (int hlf = 0; hlf < 2; ++hlf)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int kp = base + 16 * u + 8 * hlf + qc + e;
                            float& v = sc[u][hlf][2 * i + e];
                            if (kp > rq[i] || kp >= kend) v = -INFINITY;  // causal
                            mt = fmaxf(mt, v);
                        }
                mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 1));
                mt = fmaxf(mt, __shfl_xor_sync(0xffffffffu, mt, 2));
                const float m_new = fmaxf(m_run[i], mt);
                // key 0 is visible to every query, so m_new is finite from the first tile on
                // (rows past T are computed like the others and never stored)
                const float corr = m_new == -INFINITY ? 1.f : exp2f(m_run[i] - m_new);
                float ls = 0.f;
#pragma unroll
                for (int u = 0; u < SUB; ++u)
#pragma unroll
                    for (int hlf = 0; hlf < 2; ++hlf)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const float p = m_new == -INFINITY ? 0.f : exp2f(sc[u][hlf][2 * i + e] - m_new);
                            pv[u][hlf][2 * i + e] = p;
                            ls += p;
                        }
                l_run[i] = l_run[i] * corr + ls;
                m_run[i] = m_new;
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    acc[nt][2 * i] *= corr;
                    acc[nt][2 * i + 1] *= corr;
                }
            }
#pragma unroll
            for (int u = 0; u < SUB; ++u) {
                if (base + 16 * u > qw + 15) continue;  // no visible key in this sub-tile
                uint32_t pa[4];
                pa[0] = pack_h2(pv[u][0][0], pv[u][0][1]);  // row r, keys qc, qc+1
                pa[1] = pack_h2(pv[u][0][2], pv[u][0][3]);  // row r+8
                pa[2] = pack_h2(pv[u][1][0], pv[u][1][1]);  // row r, keys 8+qc, 9+qc
                pa[3] = pack_h2(pv[u][1][2], pv[u][1][3]);  // row r+8
                const uint32_t vrow = smem_u32(vt_s + (16 * u + 8 * ((lane >> 3) & 1) + (lane & 7)) * ROWB +
                                               16 * ((lane >> 4) & 1));
#pragma unroll
                for (int nt = 0; nt < NT; nt += 2) {
                    uint32_t v0, v1, v2, v3;
                    ldsm_x4_t(vrow + nt * 16, v0, v1, v2, v3);
                    mma16816_f16(acc[nt], pa, v0, v1);
                    mma16816_f16(acc[nt + 1], pa, v2, v3);
                }
            }
        }
        __syncthreads();  // the stage is refilled two tiles later
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        l_run[i] += __shfl_xor_sync(0xffffffffu, l_run[i], 1);
        l_run[i] += __shfl_xor_sync(0xffffffffu, l_run[i], 2);
        const int oh = oslot ? oslot[h] : h;  // compact O column block; -1: dropped head
        if (rq[i] < T && oh >= 0) {
            const float inv = 1.0f / l_run[i];
            __half* o = O + (int64_t)rq[i] * ldo + oh * DH;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const int dim = nt * 8 + qc;
                *reinterpret_cast<__half2*>(o + dim) = __floats2half2_rn(acc[nt][2 * i] * inv, acc[nt][2 * i + 1] * inv);
            }
        }
    }
}

// ------------------------------------------------------------------ causal attention on tcgen05
// One CTA: 128 queries of one kept head, head dim 128. Keys stream in tiles of 64:
//  * warp 0 loads Q once and, per tile, the FP16 key tile and the transposed FP16 value tile
//    (TMA, 128-byte swizzle) into two 2-slot rings: a key slot is free again once S_j has
//    been computed, a value slot once O += P_j V_j has, so the keys run a tile further ahead
//    (in MMA order the enabling events come as K_j, V_{j-1}, K_{j+1}, V_j, ...);
//  * warp 1 issues S_j = Q K_j^T (M 128, N 64) into one of two TMEM score buffers, and
//    O += P_{j-1} V_{j-1} (M 128, N 128) into the TMEM output, with P read from TMEM;
//  * warps 2-5 own one query row per thread: they read S_j from TMEM, apply the causal mask,
//    keep a running maximum that may lag the true one by up to 8 (log2 units; O in TMEM is
//    rescaled only when it would lag more), write P_j = 2^(S - m) as packed FP16 pairs over
//    the first 32 columns of S_j's buffer (the MMA's A operand), and finally divide O by the
//    running sum.
// The MMAs of a CTA run in issue order, so S_{j+2}, issued after O += P_j V_j, cannot
// overwrite P_j before it is read. Without a shared-memory P tile a CTA takes 97 KB and two
// fit on an SM (8 softmax warps, one CTA's softmax overlapping the other's MMAs).
// Every wait is bounded and reports to the device error word.
constexpr int AT_KT = 64;
constexpr int AT_Q_BYTES = 128 * 128 * 2;
constexpr int AT_K_BYTES = AT_KT * 128 * 2;
constexpr int AT_VT_BYTES = 128 * AT_KT * 2;
constexpr int AT_SMEM = AT_Q_BYTES + 2 * (AT_K_BYTES + AT_VT_BYTES) + 1024;
constexpr uint32_t AT_TMEM_COLS = 256;  // S0 [0, 64), S1 [64, 128), O [128, 256)
constexpr uint32_t IDESC_S = idesc_f16(128, AT_KT), IDESC_O = idesc_f16(128, 128);
constexpr float AT_LAZY = 8.0f;

// 2^x by the ex2.approx.ftz.f32 instruction (relative error ~2^-22; results below 2^-126
// flush to zero, far below what a probability in FP16 can hold).
__device__ __forceinline__ float ex2_ftz(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__global__ void __launch_bounds__(192, 2)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmVT, int T, int g, __half* O, int ldo, int* err,
                   const int16_t* __restrict__ oslot) {
    extern __shared__ uint8_t smraw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
    uint8_t* sq = sm;
    uint8_t* sk = sm + AT_Q_BYTES;                       // key slot s at + s * AT_K_BYTES (two 8 KB halves)
    uint8_t* sv = sm + AT_Q_BYTES + 2 * AT_K_BYTES;      // value slot s at + s * AT_VT_BYTES
    __shared__ __align__(8) uint64_t bar_q, k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], p_full[2],
        p_empty[2], o_done;
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.x, jl = h / g;
    const int oh = oslot ? oslot[h] : h;  // compact O column block of this head; -1: dropped head
    const int q0 = (gridDim.y - 1 - blockIdx.y) * 128;  // the longest query blocks of every head first
    const int kend = min(T, q0 + 128);
    const int ntile = (kend + AT_KT - 1) / AT_KT;
    auto B = [](uint64_t& b) { return smem_u32(&b); };

    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(B(bar_q), 1);
        mbar_init(B(o_done), 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(B(k_full[i]), 1);
            mbar_init(B(k_empty[i]), 1);
            mbar_init(B(v_full[i]), 1);
            mbar_init(B(v_empty[i]), 1);
            mbar_init(B(s_full[i]), 1);
            mbar_init(B(p_full[i]), 4);
            mbar_init(B(p_empty[i]), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base)),
                     "r"(AT_TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = tmem_base;
    pf_wait();  // Q, K and V^T come from the previous kernels; O is rewritten
    pf_trigger();

    if (warp == 0) {
        if (lane == 0) {  // ---- TMA producer
            mbar_expect_tx(B(bar_q), AT_Q_BYTES);
            tma_load_2d(smem_u32(sq), &tmQ, 0, h * T + q0, B(bar_q));
            tma_load_2d(smem_u32(sq + AT_Q_BYTES / 2), &tmQ, 64, h * T + q0, B(bar_q));
            auto load_v = [&](int j) {
                const int s = j & 1;
                if (j >= 2) mbar_wait(B(v_empty[s]), ((j >> 1) - 1) & 1, &abort_flag, err);
                mbar_expect_tx(B(v_full[s]), AT_VT_BYTES);
                tma_load_2d(smem_u32(sv + s * AT_VT_BYTES), &tmVT, j * AT_KT, jl * 128, B(v_full[s]));
            };
            for (int j = 0; j < ntile; ++j) {
                const int s = j & 1;
                if (j >= 2) mbar_wait(B(k_empty[s]), ((j >> 1) - 1) & 1, &abort_flag, err);
                const uint32_t fb = B(k_full[s]);
                mbar_expect_tx(fb, AT_K_BYTES);
                uint8_t* st = sk + s * AT_K_BYTES;
                tma_load_2d(smem_u32(st), &tmK, 0, jl * T + j * AT_KT, fb);
                tma_load_2d(smem_u32(st + AT_K_BYTES / 2), &tmK, 64, jl * T + j * AT_KT, fb);
                if (j >= 1) load_v(j - 1);
            }
            load_v(ntile - 1);
            // no copy may outlive the CTA
            mbar_wait(B(bar_q), 0, &abort_flag, err, false);
            for (int j = max(0, ntile - 2); j < ntile; ++j) {
                mbar_wait(B(k_full[j & 1]), (j >> 1) & 1, &abort_flag, err, false);
                mbar_wait(B(v_full[j & 1]), (j >> 1) & 1, &abort_flag, err, false);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {  // ---- MMA issuer
            mbar_wait(B(bar_q), 0, &abort_flag, err);
            fence_after();
            const uint32_t qa = smem_u32(sq);
            for (int j = 0; j <= ntile; ++j) {
                if (j < ntile) {  // S_j = Q K_j^T into score buffer j % 2
                    const int s = j & 1;
                    // score buffer s is free: S_{j-2} was read and P_{j-2} consumed by O += P_{j-2} V_{j-2},
                    // issued (after the softmax's p_full) before this MMA, and MMAs run in order
                    mbar_wait(B(k_full[s]), (j >> 1) & 1, &abort_flag, err);
                    fence_after();
                    const uint32_t kb = smem_u32(sk + s * AT_K_BYTES);
#pragma unroll
                    for (int blk = 0; blk < 2; ++blk)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_f16(tmem + 64u * s, sw128_desc(qa + blk * (AT_Q_BYTES / 2) + kk * 32),
                                   sw128_desc(kb + blk * (AT_K_BYTES / 2) + kk * 32), IDESC_S, (blk | kk) ? 1u : 0u);
                    commit(B(s_full[s]));
                    commit(B(k_empty[s]));
                }
                if (j >= 1) {  // O += P_{j-1} V_{j-1}
                    const int jp = j - 1, s = jp & 1;
                    mbar_wait(B(p_full[s]), (jp >> 1) & 1, &abort_flag, err);
                    mbar_wait(B(v_full[s]), (jp >> 1) & 1, &abort_flag, err);
                    fence_after();
                    const uint32_t vb = smem_u32(sv + s * AT_VT_BYTES);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)  // K 16 = 8 TMEM columns of packed pairs
                        mma_f16_tmem_a(tmem + 128u, tmem + 64u * s + 8u * kk, sw128_desc(vb + kk * 32), IDESC_O,
                                       (jp > 0 || kk > 0) ? 1u : 0u);
                    commit(B(p_empty[s]));
                    commit(B(v_empty[s]));
                }
            }
            commit(B(o_done));
        }
    } else {  // ---- softmax warps 2..5: TMEM lanes 32 (warp % 4) ..
        const int qw = warp & 3;
        const int row = 32 * qw + lane, qi = q0 + row;
        const uint32_t trow = tmem + ((uint32_t)(32 * qw) << 16);
        float m_run = -INFINITY, l_run = 0.f;
        for (int j = 0; j < ntile; ++j) {
            const int s = j & 1;
            mbar_wait(B(s_full[s]), (j >> 1) & 1, &abort_flag, err);
            fence_after();
            uint32_t v0[32], v1[32];
            tmem_ld32(trow + 64u * s, v0);
            tmem_ld32(trow + 64u * s + 32u, v1);
            asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
            float x[64];
            const int k0 = j * AT_KT;
            const int kv = min(qi + 1, kend) - k0;  // keys k0 + c with c < kv are visible
            if (k0 + AT_KT <= min(q0 + 1, kend)) {  // every row of the CTA sees the whole tile
#pragma unroll
                for (int c = 0; c < 64; ++c) x[c] = __uint_as_float(c < 32 ? v0[c] : v1[c - 32]);
            } else {
#pragma unroll
                for (int c = 0; c < 64; ++c) {
                    const float v = __uint_as_float(c < 32 ? v0[c] : v1[c - 32]);
                    x[c] = c < kv ? v : -INFINITY;  // causal
                }
            }
            float mx[8];  // the row maximum as a tree (independent chains instead of one of 64)
#pragma unroll
            for (int i = 0; i < 8; ++i)
                mx[i] = fmaxf(fmaxf(fmaxf(x[i], x[i + 8]), fmaxf(x[i + 16], x[i + 24])),
                              fmaxf(fmaxf(x[i + 32], x[i + 40]), fmaxf(x[i + 48], x[i + 56])));
            const float mt = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                   fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
            if (j == 0) {
                m_run = mt;  // key 0 is visible to every row
            } else {
                const bool need = mt > m_run + AT_LAZY;
                if (__any_sync(0xffffffffu, need)) {
                    // O must hold P_{j-1} V_{j-1} before it is rescaled
                    mbar_wait(B(p_empty[(j - 1) & 1]), ((j - 1) >> 1) & 1, &abort_flag, err);
                    fence_after();
                    const float corr = need ? exp2f(m_run - mt) : 1.0f;
#pragma unroll 1
                    for (int c0 = 0; c0 < 128; c0 += 32) {
                        uint32_t o[32];
                        tmem_ld32(trow + 128u + c0, o);
                        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
                        for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * corr);
                        tmem_st32(trow + 128u + c0, o);
                    }
                    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                    if (need) {
                        l_run *= corr;
                        m_run = mt;
                    }
                }
            }
            // P_j = 2^(S - m) in FP16 (<= 2^8 by the lag bound), row-sum in FP32 (8 partial sums)
            uint32_t pw[32];
            float lsp[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) lsp[i] = 0.f;
#pragma unroll
            for (int c = 0; c < 64; c += 2) {
                const float p0 = ex2_ftz(x[c] - m_run), p1 = ex2_ftz(x[c + 1] - m_run);
                lsp[(c >> 1) & 7] += p0 + p1;
                pw[c >> 1] = pack_h2(p0, p1);
            }
            l_run += ((lsp[0] + lsp[1]) + (lsp[2] + lsp[3])) + ((lsp[4] + lsp[5]) + (lsp[6] + lsp[7]));
            // S_j's commit covered every earlier MMA, so O += P_{j-2} V_{j-2} has read P_{j-2}
            tmem_st32(trow + 64u * s, pw);  // P_j over the first 32 columns of S_j's buffer
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(p_full[s]));
        }
        mbar_wait(B(o_done), 0, &abort_flag, err);
        fence_after();
        const float inv = 1.0f / l_run;
#pragma unroll 1
        for (int c0 = 0; c0 < 128; c0 += 32) {
            uint32_t o[32];
            tmem_ld32(trow + 128u + c0, o);
            asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
            if (qi < T && oh >= 0) {
                uint32_t hw[16];
#pragma unroll
                for (int c = 0; c < 32; c += 2)
                    hw[c >> 1] = pack_h2(__uint_as_float(o[c]) * inv, __uint_as_float(o[c + 1]) * inv);
                uint4* dst = reinterpret_cast<uint4*>(O + (int64_t)qi * ldo + oh * 128 + c0);
#pragma unroll
                for (int k = 0; k < 4; ++k) dst[k] = make_uint4(hw[4 * k], hw[4 * k + 1], hw[4 * k + 2], hw[4 * k + 3]);
            }
        }
    }
    fence_before();
    __syncthreads();
    fence_after();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(AT_TMEM_COLS) : "memory");
}

// ------------------------------------------------------------------ host side
// Launch with programmatic stream serialization when `pdl` (the kernels above wait with
// griddepcontrol.wait, a no-op in a plain launch). Prompts of up to PDL_MAX_T tokens take it:
// the overlapped launch ramps gave 7.51 -> 6.77 ms at 512 tokens and 16.31 -> 15.43 ms at 2,048,
// while 8,192-token prompts ran ~2% slower with it (68.5 -> 69.8 ms, same box, with the trigger
// at the start or at the end of each GEMM role), where the launch ramps are a small share.
constexpr int PDL_MAX_T = 4096;
template <typename K, typename... A>
int pdl_launch(bool pdl, K kern, dim3 grid, dim3 block, size_t smem, cudaStream_t s, const A&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = pdl ? 1 : 0;
    TASP_CUDA(cudaLaunchKernelEx(&cfg, kern, args...));
    return TASP_OK;
}
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::mutex g_enc_mu;

int encoder(PFN_cuTensorMapEncodeTiled_v12000* out) {
    std::lock_guard<std::mutex> lk(g_enc_mu);
    if (!g_encode) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
            return fail(TASP_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    *out = g_encode;
    return TASP_OK;
}

// 2-D FP16 tensor map of a row-major [rows][ld] buffer (cols used), box = box_rows x 64.
int make_map(CUtensorMap* m, const void* base, int rows, int cols, int ld, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc;
    int rc = encoder(&enc);
    if (rc) return rc;
    if ((reinterpret_cast<uintptr_t>(base) & 15) || (ld * 2) % 16)
        return fail(TASP_EINVAL, "TMA operand not 16-byte aligned");
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(TASP_ECUDA, "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")");
    return TASP_OK;
}

int launch_gemm(const __half* A, int lda, int M, const __half* B, int ldb, int N, int K, GemmArgs ga, cudaStream_t s,
                bool pdl = false) {
    ga.pdl = pdl ? 1 : 0;
    if (M == 0 || N == 0) return TASP_OK;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    // 128-column tiles when 256-column ones would leave SMs of the one wave idle
    const int mt = (M + BM - 1) / BM;
    const bool narrow = mt * ((N + 255) / 256) < di.sms;
    const int bn = narrow ? 128 : 256;
    CUtensorMap ta, tb;
    if ((rc = make_map(&ta, A, M, K, lda, BM))) return rc;
    if ((rc = make_map(&tb, B, N, K, ldb, bn))) return rc;
    ga.vec = ga.mode == EP_SWIGLU ? ((reinterpret_cast<uintptr_t>(ga.hout) & 15) == 0 && ga.ldh % 8 == 0)
                                  : ((reinterpret_cast<uintptr_t>(ga.out) & 15) == 0 && ga.ldo % 4 == 0);
    ga.vec = ga.vec && (reinterpret_cast<uintptr_t>(ga.scale) & 15) == 0;
    static bool attr = false;
    if (!attr) {
        TASP_CUDA(cudaFuncSetAttribute(gemm_persist_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       PgCfg<256>::SMEM));
        TASP_CUDA(cudaFuncSetAttribute(gemm_persist_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       PgCfg<128>::SMEM));
        attr = true;
    }
    const int tiles = mt * ((N + bn - 1) / bn);
    if (narrow) return pdl_launch(pdl, gemm_persist_kernel<128>, dim3(std::min(tiles, di.sms)), dim3(GEMM_THREADS),
                                  (size_t)PgCfg<128>::SMEM, s, ta, tb, ga);
    return pdl_launch(pdl, gemm_persist_kernel<256>, dim3(std::min(tiles, di.sms)), dim3(GEMM_THREADS),
                      (size_t)PgCfg<256>::SMEM, s, ta, tb, ga);
}

int round8(int v) { return (v + 7) & ~7; }

// FP16 copies of a plan's panels for the prefill GEMMs (made on first use, kept by the plan).
int ensure_f16_panels(Plan& p, cudaStream_t s) {
    if (p.f16_ready) return TASP_OK;
    const Shape& sh = p.store->sh;
    size_t total = 0;
    for (const LayerPlan& lp : p.layers) {
        total += ((size_t)lp.qkv_rows * round8(sh.d) + (size_t)sh.d * round8(lp.o_K) + (size_t)lp.gu_rows * round8(sh.d) +
                  (size_t)sh.d * round8(lp.dn_K)) * 2 + 4 * 256;
    }
    int post_n = sh.d;  // rows of the largest panel
    for (const LayerPlan& lp : p.layers) post_n = std::max(post_n, std::max(lp.qkv_rows, lp.gu_rows));
    if (sh.qg) total += (size_t)post_n * 4 + 256;
    int rc = p.f16_arena.reserve(total);
    if (rc) return rc;
    p.f16.resize(sh.L);
    for (int l = 0; l < sh.L; ++l) {
        const LayerPlan& lp = p.layers[l];
        F16Panels& f = p.f16[l];
        f.ld_d = round8(sh.d);
        f.ld_o = round8(lp.o_K);
        f.ld_dn = round8(lp.dn_K);
        f.qkv = (__half*)p.f16_arena.take((size_t)lp.qkv_rows * f.ld_d * 2);
        f.o = (__half*)p.f16_arena.take((size_t)sh.d * f.ld_o * 2);
        f.gu = (__half*)p.f16_arena.take((size_t)lp.gu_rows * f.ld_d * 2);
        f.dn = (__half*)p.f16_arena.take((size_t)sh.d * f.ld_dn * 2);
        const int G = sh.qg;
        if (lp.qkv_rows)
            i8_to_f16_kernel<<<lp.qkv_rows, 256, 0, s>>>(lp.qkv_w, lp.qkv_map, sh.d, sh.d, f.qkv, f.ld_d,
                                                          G ? lp.qkv_g : nullptr, lp.qkv_gld, G);
        if (lp.o_K)
            i8_to_f16_kernel<<<sh.d, 256, 0, s>>>(lp.o_w, nullptr, lp.o_ld, lp.o_K, f.o, f.ld_o, G ? lp.o_g : nullptr,
                                                  lp.o_gld, G);
        if (lp.gu_rows)
            i8_to_f16_kernel<<<lp.gu_rows, 256, 0, s>>>(lp.gu_w, lp.gu_map, sh.d, sh.d, f.gu, f.ld_d,
                                                         G ? lp.gu_g : nullptr, lp.gu_gld, G);
        if (lp.dn_K)
            i8_to_f16_kernel<<<sh.d, 256, 0, s>>>(lp.dn_w, nullptr, lp.dn_ld, lp.dn_K, f.dn, f.ld_dn,
                                                  G ? lp.dn_g : nullptr, lp.dn_gld, G);
        TASP_CUDA(cudaGetLastError());
    }
    std::vector<float> post;
    if (sh.qg) {
        float* d_post = (float*)p.f16_arena.take((size_t)post_n * 4);
        post.assign(post_n, std::ldexp(1.0f, -F16_GS_EXP));
        TASP_CUDA(cudaMemcpyAsync(d_post, post.data(), (size_t)post_n * 4, cudaMemcpyHostToDevice, s));
        p.f16_post = d_post;
    }
    TASP_CUDA(cudaStreamSynchronize(s));
    p.f16_ready = true;
    return TASP_OK;
}

}  // namespace

int gemm_f16_nt(const __half* A, int lda, int M, const __half* B, int ldb, int N, int K, const float* scale, float* C,
                int ldc, int* err, cudaStream_t s) {
    GemmArgs ga{};
    ga.M = M;
    ga.N = N;
    ga.K = K;
    ga.scale = scale;
    ga.out = C;
    ga.ldo = ldc;
    ga.mode = EP_STORE;
    ga.err = err;
    return launch_gemm(A, lda, M, B, ldb, N, K, ga, s);
}

int encode_kv_map(CUtensorMap* m, const uint16_t* base, int dh, int max_tokens, int m_kv) {
    PFN_cuTensorMapEncodeTiled_v12000 enc;
    int rc = encoder(&enc);
    if (rc) return rc;
    if (reinterpret_cast<uintptr_t>(base) & 15) return fail(TASP_EINVAL, "KV cache not 16-byte aligned");
    cuuint64_t dims[3] = {(cuuint64_t)dh, (cuuint64_t)max_tokens, (cuuint64_t)m_kv};
    cuuint64_t strides[2] = {(cuuint64_t)dh * 2, (cuuint64_t)max_tokens * dh * 2};
    cuuint32_t box[3] = {64, 16, 1};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<uint16_t*>(base), dims, strides, box, es,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(TASP_ECUDA, "cuTensorMapEncodeTiled failed for a KV cache (" + std::to_string((int)r) + ")");
    return TASP_OK;
}

int prefill_run(Session& se, const uint16_t* d_embeds, int T, cudaStream_t s) {
    Plan& pl = *se.plan;
    const Shape& sh = pl.store->sh;
    int rc = ensure_f16_panels(pl, s);
    if (rc) return rc;
    int max_rows = 0, max_c = 0, max_oK = 0;
    for (const LayerPlan& lp : pl.layers) {
        max_rows = std::max(max_rows, lp.qkv_rows);
        max_c = std::max(max_c, lp.c);
        max_oK = std::max(max_oK, lp.o_K);
    }
    const int ld_x = round8(sh.d), ld_y = std::max(4, (max_rows + 3) & ~3), ld_o = round8(std::max(8, sh.Hq * sh.dh)),
              ld_h = round8(std::max(8, max_c));
    // workspace (stream-ordered, released at the end of the prefill)
    float *X = nullptr, *Y = nullptr, *Qf = nullptr;
    __half *Xh = nullptr, *O = nullptr, *H = nullptr;
    TASP_CUDA(cudaMallocAsync((void**)&X, (size_t)T * sh.d * 4, s));
    TASP_CUDA(cudaMallocAsync((void**)&Xh, (size_t)T * ld_x * 2, s));
    TASP_CUDA(cudaMallocAsync((void**)&Y, (size_t)T * ld_y * 4, s));
    TASP_CUDA(cudaMallocAsync((void**)&Qf, (size_t)T * sh.Hq * sh.dh * 4, s));
    TASP_CUDA(cudaMallocAsync((void**)&O, (size_t)T * ld_o * 2, s));
    TASP_CUDA(cudaMallocAsync((void**)&H, (size_t)T * ld_h * 2, s));
    TASP_CUDA(cudaMemsetAsync(O, 0, (size_t)T * ld_o * 2, s));
    TASP_CUDA(cudaMemsetAsync(H, 0, (size_t)T * ld_h * 2, s));
    // tensor-core attention operands (head dim 128): scaled FP16 queries, FP16 keys and
    // transposed FP16 values (rows padded to Tp keys, padding zero)
    const bool tc_attn = sh.dh == 128;
    const int Tp = (T + 7) & ~7;
    __half *Qh = nullptr, *Kh = nullptr, *VT = nullptr;
    if (tc_attn) {
        TASP_CUDA(cudaMallocAsync((void**)&Qh, (size_t)sh.Hq * T * 128 * 2, s));
        TASP_CUDA(cudaMallocAsync((void**)&Kh, (size_t)sh.Hkv * T * 128 * 2, s));
        TASP_CUDA(cudaMallocAsync((void**)&VT, (size_t)sh.Hkv * 128 * Tp * 2, s));
        TASP_CUDA(cudaMemsetAsync(VT, 0, (size_t)sh.Hkv * 128 * Tp * 2, s));
        static bool attr = false;
        if (!attr) {
            TASP_CUDA(cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, AT_SMEM));
            attr = true;
        }
    }
    const float qscale = (float)(1.0 / std::sqrt((double)sh.dh) * 1.4426950408889634);
    const bool pdl = T <= PDL_MAX_T;
    bool vec_norm = sh.d % 4 == 0 && ld_x % 4 == 0;
    for (const LayerPlan& lp : pl.layers)
        vec_norm = vec_norm && (reinterpret_cast<uintptr_t>(lp.g_attn) & 15) == 0 &&
                   (reinterpret_cast<uintptr_t>(lp.g_mlp) & 15) == 0;
    {
        static bool attr = false;  // the key/value ring exceeds the default 48 KB of shared memory
        if (!attr) {
            TASP_CUDA(cudaFuncSetAttribute(attn_prefill_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           PaCfg<128>::SMEM));
            TASP_CUDA(cudaFuncSetAttribute(attn_prefill_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           PaCfg<64>::SMEM));
            attr = true;
        }
    }
    for (int l = 0; l < sh.L && !rc; ++l) {
        const LayerPlan& lp = pl.layers[l];
        const F16Panels& f = pl.f16[l];
        if (l == 0 || !vec_norm)  // the first layer also widens the BF16 embeddings into X
            rc = pdl_launch(pdl, rmsnorm_rows_kernel, dim3(T), dim3(256), 0, s, (const float*)X,
                            l == 0 ? d_embeds : nullptr, X, sh.d, lp.g_attn, sh.eps, Xh, ld_x);
        else
            rc = pdl_launch(pdl, rmsnorm_rows_vec_kernel, dim3(T), dim3(256), 0, s, (const float*)X, sh.d, lp.g_attn,
                            sh.eps, Xh, ld_x);
        if (rc) break;
        if (lp.m_kv > 0) {
            GemmArgs ga{};
            ga.M = T; ga.N = lp.qkv_rows; ga.K = sh.d; ga.scale = pl.f16_post ? pl.f16_post : lp.qkv_s; ga.out = Y; ga.ldo = ld_y;
            ga.mode = EP_STORE; ga.err = se.err;
            if ((rc = launch_gemm(Xh, ld_x, T, f.qkv, f.ld_d, lp.qkv_rows, sh.d, ga, s, pdl))) break;
            if ((rc = pdl_launch(pdl, rope_kv_kernel, dim3(T, lp.m_kv), dim3(256), 0, s, (const float*)Y, ld_y, T, sh.g(),
                                 sh.dh, (const float2*)se.rope, tc_attn ? nullptr : Qf, se.K[l], se.V[l],
                                 se.max_tokens, Qh, qscale, Kh, lp.blk_of)))
                break;
            if (tc_attn) {
                if ((rc = pdl_launch(pdl, v_transpose_kernel, dim3((T + 63) / 64, lp.m_kv), dim3(256), 0, s,
                                     (const uint16_t*)se.V[l], se.max_tokens, T, VT, Tp)))
                    break;
                CUtensorMap mq, mk, mv;
                const int mq_rows = lp.m_kv * sh.g() * T;
                if ((rc = make_map(&mq, Qh, mq_rows, 128, 128, 128))) break;
                if ((rc = make_map(&mk, Kh, lp.m_kv * T, 128, 128, AT_KT))) break;
                if ((rc = make_map(&mv, VT, lp.m_kv * 128, Tp, Tp, 128))) break;
                if ((rc = pdl_launch(pdl, attn_tc_kernel, dim3(lp.m_kv * sh.g(), (T + 127) / 128), dim3(192),
                                     (size_t)AT_SMEM, s, mq, mk, mv, T, sh.g(), O, ld_o, se.err, lp.oslot)))
                    break;
            } else {
                const int qb = (T + PA_QB - 1) / PA_QB;
                if ((rc = pdl_launch(pdl, attn_prefill_kernel<64>, dim3(lp.m_kv * sh.g(), qb), dim3(PA_WARPS * 32),
                                     (size_t)PaCfg<64>::SMEM, s, (const float*)Qf, (const uint16_t*)se.K[l],
                                     (const uint16_t*)se.V[l], T, se.max_tokens, sh.g(), qscale, O, ld_o, lp.oslot)))
                    break;
            }
            TASP_CUDA(cudaGetLastError());
            GemmArgs go{};
            go.M = T; go.N = sh.d; go.K = lp.o_K; go.scale = pl.f16_post ? pl.f16_post : lp.o_s; go.out = X; go.ldo = sh.d;
            go.mode = EP_RESID; go.err = se.err;
            if ((rc = launch_gemm(O, ld_o, T, f.o, f.ld_o, sh.d, lp.o_K, go, s, pdl))) break;
        }
        if (lp.c > 0) {
            if (vec_norm)
                rc = pdl_launch(pdl, rmsnorm_rows_vec_kernel, dim3(T), dim3(256), 0, s, (const float*)X, sh.d, lp.g_mlp,
                                sh.eps, Xh, ld_x);
            else
                rc = pdl_launch(pdl, rmsnorm_rows_kernel, dim3(T), dim3(256), 0, s, (const float*)X,
                                (const uint16_t*)nullptr, (float*)nullptr, sh.d, lp.g_mlp, sh.eps, Xh, ld_x);
            if (rc) break;
            GemmArgs gg{};
            gg.M = T; gg.N = lp.gu_rows; gg.K = sh.d; gg.scale = pl.f16_post ? pl.f16_post : lp.gu_s; gg.hout = H; gg.ldh = ld_h;
            gg.mode = EP_SWIGLU; gg.err = se.err;
            if ((rc = launch_gemm(Xh, ld_x, T, f.gu, f.ld_d, lp.gu_rows, sh.d, gg, s, pdl))) break;
            GemmArgs gd{};
            gd.M = T; gd.N = sh.d; gd.K = lp.c; gd.scale = pl.f16_post ? pl.f16_post : lp.dn_s; gd.out = X; gd.ldo = sh.d;
            gd.mode = EP_RESID; gd.err = se.err;
            if ((rc = launch_gemm(H, ld_h, T, f.dn, f.ld_dn, sh.d, lp.c, gd, s, pdl))) break;
        }
    }
    if (!rc) {
        // the last prompt position's residual seeds the session (final norm + LM head read it)
        cudaError_t e = cudaMemcpyAsync(se.x, X + (size_t)(T - 1) * sh.d, (size_t)sh.d * 4, cudaMemcpyDeviceToDevice, s);
        if (e != cudaSuccess) rc = cuda_fail(e, "prefill residual copy");
    }
    cudaFreeAsync(X, s);
    cudaFreeAsync(Xh, s);
    cudaFreeAsync(Y, s);
    cudaFreeAsync(Qf, s);
    cudaFreeAsync(O, s);
    cudaFreeAsync(H, s);
    if (Qh) cudaFreeAsync(Qh, s);
    if (Kh) cudaFreeAsync(Kh, s);
    if (VT) cudaFreeAsync(VT, s);
    return rc;
}

}  // namespace tasp
