// INT8-weight GEMV for decode (and the BF16 LM head), sm_103a, for NB <= 4 activation
// vectors per weight pass (NB sessions decoding on one plan share every weight byte).
//
// Every projection of a decode step is an HBM-bound GEMV over the retained rows of an
// INT8 panel with one FP32 scale per output row (the paper's INT8-weight runtime, Table 1).
// One persistent CTA per SM runs three roles:
//  * a producer warp streams row groups (R rows, one cp.async.bulk per row) into a
//    shared-memory ring of up to 8 stages with full/empty mbarriers; weights never depend
//    on the previous kernel, so it starts before griddepcontrol.wait;
//  * 16 consumer warps: the activation vectors pass once through a 32 KB shared window
//    (coalesced loads, RMSNorm applied on the way), from which each thread takes its
//    slice (16 elements per 16-byte weight chunk) and turns it into block-scaled integers: per
//    chunk one power-of-two scale 2^(e-14) with max|x| < 2^e, each element rounded to
//    X in [-2^14, 2^14] and split X = 256 hi + lo (hi signed byte, lo unsigned byte). The
//    raw INT8 weight words then feed dp4a directly (exact INT32 chunk sums, one FP32 FMA
//    per chunk); R x NB row sums are reduced with a halving butterfly and handed to
//  * an epilogue warp through a ring of partial-sum buffers: it sums across warps and
//    finishes the rows (rotary embedding + KV append, SiLU(gate) * up, residual add, LM
//    head logits) with scales, residual rows and rotary pairs staged in shared memory.
// A thread keeps NB x XC chunks of digits in registers (NB * XC <= 4). Rows longer than
// XC x 512 chunks are streamed in K passes: pass k covers chunks [k S, (k + 1) S) of every
// row of the CTA, the digits are rebuilt for each pass, and the epilogue warp adds the
// pass sums into the residual (or the logits) row by row.
// Every wait is bounded: a timeout sets the device error word and aborts the CTA's later
// waits instead of hanging. A step of one session uses the one-vector kernels of
// gemv_single.cu instead (shorter prologue); these serve groups of 2-4 sessions.
#pragma once

#include <cuda_bf16.h>

#include "tasp_internal.h"

namespace tasp {
namespace gemv {

constexpr int MAXNB = 4;
constexpr int CW = 16;                   // consumer warps
constexpr int CT = CW * 32;              // consumer threads
constexpr int THREADS = CT + 64;         // + producer warp + epilogue warp
constexpr int MAX_STAGES = 8;
constexpr int NRB = 8;                   // partial-sum buffers between consumers and the epilogue warp
constexpr long long WAIT_LIMIT = 4000000000ll;  // clock cycles (~2 s) before a wait gives up
constexpr int ERR_WAIT_TIMEOUT = 1;
constexpr int EPI_MAXR = 512;            // rows per CTA the epilogue warp can stage

enum Mode { M_QKV = 0, M_O = 1, M_GU = 2, M_DOWN = 3, M_LM = 4 };

struct Params {
    const int8_t* w;       // panel (or store) base
    const int32_t* map;    // optional row map: panel row -> source row
    const float* scale;    // per panel row
    int64_t ld;            // row stride in bytes
    int rows, K, nchunks;  // output rows, logical K, 16-byte chunks per row
    int seg;               // chunks per K pass (XC x consumer threads, or nchunks)
    int passes;            // ceil(nchunks / seg); 1 for the rotary / SwiGLU modes
    int nb;                // activation vectors in this launch (<= NB of the kernel)
    // inputs: vector v at base + v * stride
    const float* x_resid;  // QKV / GU / LM: FP32 residual rows to normalize
    const uint16_t* x_in;  // QKV of layer 0: BF16 step inputs (the residual is initialized from them)
    int64_t x_stride, xin_stride;
    float* x_resid_init;   // where CTA 0 stores the initialized residual (stride x_stride)
    const float* gamma;
    float eps;
    const float* act;      // O / DOWN: FP32 activations
    int64_t act_stride;
    // outputs
    float* resid_out;      // O / DOWN: residual rows (+=), stride x_stride
    float* hidden_out;     // DOWN of the last layer: copy of the residual (stride hid_stride)
    int64_t hid_stride;
    float* q_out;          // QKV: rotated queries, stride q_stride
    int64_t q_stride;
    uint16_t* k_cache[MAXNB];
    uint16_t* v_cache[MAXNB];
    int max_tokens[MAXNB];
    const float2* rope[MAXNB];
    const int* pos[MAXNB];
    int g, dh;
    const int16_t* blk_role;  // QKV: role of each d_h-row block (NULL = block index)
    const uint16_t* gscale;   // groupwise store: BF16 scales [panel row][gld] (NULL = per-row only)
    int gcols, gshift;        // scales per row; chunk c uses scale c >> gshift
    int gld;                  // row stride of gscale (elements)
    float* h_out;          // GU: SiLU(gate) * up, stride h_stride
    int64_t h_stride;
    float* logits;         // LM: stride logit_stride
    int64_t logit_stride;
    int* err;              // device error word
    int smem_cap;          // dynamic shared memory available to the launch
};


// Shared-memory plan of one launch (host and device agree on it).
struct Smem {
    int stage_bytes, nstages, total;
};
constexpr int XS_BYTES = CT * 64;  // activation window: one 16-element FP32 chunk per consumer thread

__host__ __device__ inline Smem smem_plan(int R, int seg_bytes, int cap) {
    Smem g;
    g.stage_bytes = ((R * seg_bytes) + 127) & ~127;
    const int bar_bytes = (2 * MAX_STAGES + 2 * NRB) * 8 + 16;
    int ns = (cap - XS_BYTES - bar_bytes) / g.stage_bytes;
    g.nstages = ns > MAX_STAGES ? MAX_STAGES : ns;
    g.total = XS_BYTES + g.nstages * g.stage_bytes + bar_bytes;
    return g;
}

// ------------------------------------------------------------------ PTX helpers
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
typedef unsigned long long u64;
__device__ __forceinline__ u64 pk(float a, float b) {
    u64 r;
    asm("mov.b64 %0, {%1,%2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ float2 upk(u64 v) {
    float2 r;
    asm("mov.b64 {%0,%1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
    return r;
}
__device__ __forceinline__ u64 fma2(u64 a, u64 b, u64 c) {
    u64 d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ uint16_t f32_to_bf16_bits(float v) {
    __nv_bfloat16 b = __float2bfloat16_rn(v);
    return *reinterpret_cast<uint16_t*>(&b);
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(CT) : "memory"); }
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait: after WAIT_LIMIT cycles it records the failure in the device error word
// and makes every later wait of this CTA return at once (abort).
__device__ __forceinline__ void mbar_wait(uint32_t bar, uint32_t parity, int* abort_flag, int* err,
                                          bool honor_abort = true) {
    if (honor_abort && *(volatile int*)abort_flag) return;
    if (mbar_try(bar, parity)) return;
    const long long t0 = clock64();
    while (!mbar_try(bar, parity)) {
        if (clock64() - t0 > WAIT_LIMIT) {
            *(volatile int*)abort_flag = 1;
            if (err) atomicOr(err, ERR_WAIT_TIMEOUT);
            return;
        }
    }
}
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}
__device__ __forceinline__ int dp4a_ss(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.s32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}
__device__ __forceinline__ int dp4a_su(uint32_t a, uint32_t b, int c) {
    int d;
    asm("dp4a.s32.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

// ------------------------------------------------------------------ row addressing
// QKV work rows are ordered so that each even/odd pair holds rows i and i + dh/2 of one
// head (a rotary pair); all other modes use the panel order.
template <int MODE>
__device__ __forceinline__ int panel_row(const Params& p, int w) {
    if (MODE == M_QKV) {
        int hb = w / p.dh, iw = w - hb * p.dh;
        return hb * p.dh + (iw >> 1) + (iw & 1) * (p.dh >> 1);
    }
    return w;
}
template <int MODE>
__device__ __forceinline__ const int8_t* row_ptr(const Params& p, int w) {
    if (w >= p.rows) w = 0;
    int pr = panel_row<MODE>(p, w);
    int src = p.map ? __ldg(p.map + pr) : pr;
    return p.w + (int64_t)src * p.ld;
}

// ------------------------------------------------------------------ activation slices
// 1 / RMS of each vector (RMSNorm modes); every CTA sums in the same fixed order.
template <int NB>
__device__ __forceinline__ void norm_scales(const Params& p, float (*stat)[CW], float (&inv)[NB], int tid) {
    const int n4 = p.K / 4;
#pragma unroll
    for (int v = 0; v < NB; ++v) {
        float ss = 0.f;
        if (v < p.nb) {
            for (int f = tid; f < n4; f += CT) {
                float4 x;
                if (p.x_in) {
                    const uint2 b = __ldcg(reinterpret_cast<const uint2*>(p.x_in + v * p.xin_stride) + f);
                    x = make_float4(__uint_as_float(b.x << 16), __uint_as_float(b.x & 0xffff0000u),
                                    __uint_as_float(b.y << 16), __uint_as_float(b.y & 0xffff0000u));
                    if (p.x_resid_init && blockIdx.x == 0)
                        reinterpret_cast<float4*>(p.x_resid_init + v * p.x_stride)[f] = x;
                } else {
                    x = __ldcg(reinterpret_cast<const float4*>(p.x_resid + v * p.x_stride) + f);
                }
                ss = fmaf(x.x, x.x, ss);
                ss = fmaf(x.y, x.y, ss);
                ss = fmaf(x.z, x.z, ss);
                ss = fmaf(x.w, x.w, ss);
            }
        }
        ss = warp_sum(ss);
        if ((tid & 31) == 0) stat[v][tid >> 5] = ss;
    }
    consumer_sync();
#pragma unroll
    for (int v = 0; v < NB; ++v) {
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < CW; ++w) tot += stat[v][w];
        inv[v] = 1.0f / sqrtf(__fdiv_rn(tot, (float)p.K) + p.eps);
    }
}

// E consecutive activations of vector v starting at element e0 (normalized when inv > 0).
template <int MODE, int E>
__device__ __forceinline__ void slice(const Params& p, int v, int e0, float inv, float (&out)[E]) {
#pragma unroll
    for (int q = 0; q < E / 4; ++q) {
        const int e = e0 + 4 * q;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (MODE == M_O || MODE == M_DOWN) {
            const float* a = p.act + v * p.act_stride;
            if (e + 3 < p.K) {
                x = __ldcg(reinterpret_cast<const float4*>(a + e));
            } else {
                x.x = e + 0 < p.K ? __ldcg(a + e + 0) : 0.f;
                x.y = e + 1 < p.K ? __ldcg(a + e + 1) : 0.f;
                x.z = e + 2 < p.K ? __ldcg(a + e + 2) : 0.f;
                x.w = e + 3 < p.K ? __ldcg(a + e + 3) : 0.f;
            }
        } else if (e < p.K) {  // K is a multiple of 8 for the normalized modes
            if (p.x_in) {
                const uint2 b = __ldcg(reinterpret_cast<const uint2*>(p.x_in + v * p.xin_stride + e));
                x = make_float4(__uint_as_float(b.x << 16), __uint_as_float(b.x & 0xffff0000u),
                                __uint_as_float(b.y << 16), __uint_as_float(b.y & 0xffff0000u));
            } else {
                x = __ldcg(reinterpret_cast<const float4*>(p.x_resid + v * p.x_stride + e));
            }
            const float4 gm = *reinterpret_cast<const float4*>(p.gamma + e);
            x.x = (x.x * inv) * gm.x;
            x.y = (x.y * inv) * gm.y;
            x.z = (x.z * inv) * gm.z;
            x.w = (x.w * inv) * gm.w;
        }
        out[4 * q + 0] = x.x;
        out[4 * q + 1] = x.y;
        out[4 * q + 2] = x.z;
        out[4 * q + 3] = x.w;
    }
}

template <int XC, int NB>
struct XDigits {
    uint32_t hi[NB][XC][4], lo[NB][XC][4];
    float scale[NB][XC];
};

// float4 index swizzle of the activation window: F float4 per chunk (4 for INT8 rows, 2 for
// BF16 rows); thread t reads float4 F t .. F t + F - 1, conflict-free with the swizzle.
template <int F>
__device__ __forceinline__ int swz(int f) {
    return f ^ ((f >> 3) & (F - 1));
}

// Window (v, j) of the activation slices: chunks cb + j * CT + [0, CT) of vector v, read with
// coalesced float4 loads by all consumer threads into shared memory (normalized for the
// RMSNorm modes, zero beyond cb + nvalid); then thread t holds chunk t of the window.
template <int MODE, int F>
__device__ __forceinline__ void stage_window(const Params& p, int v, int cw, int nvalid, float inv, float4* xs,
                                             int tid) {
    consumer_sync();  // every thread has read the previous window
    constexpr int EPC = 4 * F;  // elements per chunk
#pragma unroll
    for (int k = 0; k < F; ++k) {
        const int f = tid + k * CT;  // float4 of the window
        float x[4] = {0.f, 0.f, 0.f, 0.f};
        if (v < p.nb && f / F < nvalid) slice<MODE, 4>(p, v, EPC * cw + 4 * f, inv, x);
        xs[swz<F>(f)] = make_float4(x[0], x[1], x[2], x[3]);
    }
    consumer_sync();
}

// Digits of this thread's chunks cb + tid + j * CT (j < XC) of every vector; chunks at or
// beyond cb + nvalid are zero.
template <int MODE, int XC, int NB>
__device__ __forceinline__ void make_digits(const Params& p, const float (&inv)[NB], XDigits<XC, NB>& xd, int cb,
                                            int nvalid, float4* xs, int tid) {
#pragma unroll
    for (int v = 0; v < NB; ++v)
#pragma unroll
        for (int j = 0; j < XC; ++j) {
            if (v >= p.nb || j * CT >= nvalid) {  // uniform: nothing of this window is used
#pragma unroll
                for (int w = 0; w < 4; ++w) xd.hi[v][j][w] = xd.lo[v][j][w] = 0u;
                xd.scale[v][j] = 0.f;
                continue;
            }
            stage_window<MODE, 4>(p, v, cb + j * CT, nvalid - j * CT, inv[v], xs, tid);
            float x[16];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float4 t = xs[swz<4>(4 * tid + q)];
                x[4 * q + 0] = t.x;
                x[4 * q + 1] = t.y;
                x[4 * q + 2] = t.z;
                x[4 * q + 3] = t.w;
            }
            float m = 0.f;
#pragma unroll
            for (int e = 0; e < 16; ++e) m = fmaxf(m, fabsf(x[e]));
            int ex = 0;
            if (m > 0.f) frexpf(m, &ex);  // m = f * 2^ex, f in [0.5, 1): every |x| < 2^ex
            xd.scale[v][j] = m > 0.f ? ldexpf(1.0f, ex - 14) : 0.f;
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                uint32_t h = 0, l = 0;
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    const int X = m > 0.f ? __float2int_rn(ldexpf(x[4 * w + b], 14 - ex)) : 0;
                    h |= ((uint32_t)(X >> 8) & 0xFFu) << (8 * b);
                    l |= ((uint32_t)X & 0xFFu) << (8 * b);
                }
                xd.hi[v][j][w] = h;
                xd.lo[v][j][w] = l;
            }
        }
}

template <int XC, int NB>
struct XRegs {
    float4 v[NB][XC][2];
};

// LM head: FP32 slices of 8 elements per chunk (BF16 weights), staged the same way.
template <int XC, int NB>
__device__ __forceinline__ void make_xregs(const Params& p, const float (&inv)[NB], XRegs<XC, NB>& xr, int cb,
                                           int nvalid, float4* xs, int tid) {
#pragma unroll
    for (int v = 0; v < NB; ++v)
#pragma unroll
        for (int j = 0; j < XC; ++j) {
            if (v >= p.nb || j * CT >= nvalid) {
                xr.v[v][j][0] = xr.v[v][j][1] = make_float4(0.f, 0.f, 0.f, 0.f);
                continue;
            }
            stage_window<M_LM, 2>(p, v, cb + j * CT, nvalid - j * CT, inv[v], xs, tid);
            xr.v[v][j][0] = xs[swz<2>(2 * tid)];
            xr.v[v][j][1] = xs[swz<2>(2 * tid + 1)];
        }
}

// ------------------------------------------------------------------ dot products
// INT8 rows of one stage . x: per chunk sum(w X) = 256 sum(w hi) + sum(w lo) in exact
// INT32, then acc[r][v] += float(sum) * scale in FP32. GS (grouped store): the chunk's sum
// is also scaled by its row's BF16 group scale, grow[r][(cb + c) >> gshift] (cb = the pass's
// first chunk), read through the cache and shared by the NB vectors.
template <int R, int XC, int NB, bool GS = false>
__device__ __forceinline__ void dot_i8(const uint8_t* __restrict__ stage, int ld, const XDigits<XC, NB>& xd,
                                       int nvalid, int tid, float (&acc)[R][NB],
                                       const uint16_t* const (&grow)[R], int gshift, int cb) {
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const int c = tid + j * CT;
        if (c < nvalid) {
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int4 wv = *reinterpret_cast<const int4*>(stage + (size_t)r * ld + (size_t)c * 16);
                const uint32_t wd[4] = {(uint32_t)wv.x, (uint32_t)wv.y, (uint32_t)wv.z, (uint32_t)wv.w};
                float gsc = 1.0f;
                if constexpr (GS) gsc = __uint_as_float((uint32_t)__ldg(grow[r] + ((cb + c) >> gshift)) << 16);
#pragma unroll
                for (int v = 0; v < NB; ++v) {
                    int sh = 0, sl = 0;
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        sh = dp4a_ss(wd[k], xd.hi[v][j][k], sh);
                        sl = dp4a_su(wd[k], xd.lo[v][j][k], sl);
                    }
                    const float xs = GS ? xd.scale[v][j] * gsc : xd.scale[v][j];
                    acc[r][v] = fmaf(__int2float_rn(sh * 256 + sl), xs, acc[r][v]);
                }
            }
        }
    }
}

// BF16 rows (LM head): 8 weights per 16-byte chunk, packed f32x2 FMAs
template <int R, int XC, int NB>
__device__ __forceinline__ void dot_bf16(const uint8_t* __restrict__ stage, int ld, const XRegs<XC, NB>& xr,
                                         int nvalid, int tid, float (&out)[R][NB]) {
    u64 acc[R][NB];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int v = 0; v < NB; ++v) acc[r][v] = 0ull;
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const int c = tid + j * CT;
        if (c < nvalid) {
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int4 wv = *reinterpret_cast<const int4*>(stage + (size_t)r * ld + (size_t)c * 16);
                const uint32_t w0 = wv.x, w1 = wv.y, w2 = wv.z, w3 = wv.w;
                const u64 p0 = pk(__uint_as_float(w0 << 16), __uint_as_float(w0 & 0xffff0000u));
                const u64 p1 = pk(__uint_as_float(w1 << 16), __uint_as_float(w1 & 0xffff0000u));
                const u64 p2 = pk(__uint_as_float(w2 << 16), __uint_as_float(w2 & 0xffff0000u));
                const u64 p3 = pk(__uint_as_float(w3 << 16), __uint_as_float(w3 & 0xffff0000u));
#pragma unroll
                for (int v = 0; v < NB; ++v) {
                    const float4 x0 = xr.v[v][j][0], x1 = xr.v[v][j][1];
                    acc[r][v] = fma2(p0, pk(x0.x, x0.y), acc[r][v]);
                    acc[r][v] = fma2(p1, pk(x0.z, x0.w), acc[r][v]);
                    acc[r][v] = fma2(p2, pk(x1.x, x1.y), acc[r][v]);
                    acc[r][v] = fma2(p3, pk(x1.z, x1.w), acc[r][v]);
                }
            }
        }
    }
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int v = 0; v < NB; ++v) {
            const float2 a = upk(acc[r][v]);
            out[r][v] = a.x + a.y;
        }
}

// Warp reduction of N sums at once: each butterfly level halves the vector a lane carries,
// so lane l ends with the full sum of entry l / (32 / N).
template <int N>
__device__ __forceinline__ float vec_reduce(float (&v)[N], int lane) {
#pragma unroll
    for (int n = N, o = 16; n > 1; n >>= 1, o >>= 1) {
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < n / 2; ++i) {
            const float send = up ? v[i] : v[i + n / 2];
            const float keep = up ? v[i + n / 2] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    float s = v[0];
#pragma unroll
    for (int o = 16 / N; o >= 1; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    return s;
}

// ------------------------------------------------------------------ epilogue warp
// Copy n floats src(i) -> dst[i] with one warp, eight independent loads in flight per lane
// (a load followed by a shared store per element would wait out each load's latency).
template <typename Src>
__device__ __forceinline__ void warp_stage(float* dst, int n, Src src, int lane) {
    for (int base = 0; base < n; base += 32 * 8) {
        float v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int i = base + lane + 32 * k;
            v[k] = i < n ? src(i) : 0.f;
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int i = base + lane + 32 * k;
            if (i < n) dst[i] = v[k];
        }
    }
}

template <int NB>
struct EpiStage {
    float sc[EPI_MAXR];
    float res[NB][EPI_MAXR];
    float2 rope[NB][64];
    int pos[NB];
    int w_lo;  // first row of the CTA (the host guarantees <= EPI_MAXR rows per CTA)
};

// Lanes split the CW partial sums of each (row, vector) entry k = r * NB + v, then lane k
// (< R * NB) finishes it; rotary / SwiGLU pairs are rows 2t and 2t + 1 (entries k, k + NB).
// A given entry is always finished by the same lane, so the K passes of a row add up in
// program order.
template <int MODE, int R, int NB>
__device__ __forceinline__ void epilogue(const Params& p, const float (*red)[R * NB], int gi, int pass, int lane,
                                         EpiStage<NB>& es) {
    constexpr int N = R * NB;
    constexpr int LPE = 32 / N;  // lanes per entry
    const int k = lane % N;
    float s = 0.f;
#pragma unroll
    for (int w = lane / N; w < CW; w += LPE) s += red[w][k];
#pragma unroll
    for (int o = N; o < 32; o <<= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const int r = k / NB, v = k - r * NB;
    const int w0 = gi * R;
    if (MODE == M_QKV || MODE == M_GU) {
        const float s_other = __shfl_down_sync(0xffffffffu, s, NB);  // row r + 1, same vector
        if (lane < N && (r & 1) == 0 && v < p.nb) {
            const float s0 = s, s1 = s_other;
            const int wa = w0 + r;
            if (wa < p.rows) {
                const float sc0 = es.sc[wa - es.w_lo];
                const float sc1 = es.sc[wa + 1 - es.w_lo];
                if (MODE == M_GU) {
                    const float a = sc0 * s0, b = sc1 * s1;
                    const float silu = a / (1.0f + expf(-a));
                    p.h_out[v * p.h_stride + (wa >> 1)] = silu * b;
                } else {
                    const int half = p.dh >> 1;
                    const int hb = wa / p.dh, i = (wa - hb * p.dh) >> 1;
                    float y0 = sc0 * s0, y1 = sc1 * s1;
                    const int gp2 = p.g + 2;
                    const int code = p.blk_role ? p.blk_role[hb] : hb;
                    const int jl = code / gp2, hh = code - jl * gp2;
                    if (hh <= p.g) {
                        const float2 cs = es.rope[v][i];
                        const float ya = y0 * cs.x - y1 * cs.y, yb = y1 * cs.x + y0 * cs.y;
                        y0 = ya;
                        y1 = yb;
                    }
                    if (hh < p.g) {
                        float* dq = p.q_out + v * p.q_stride + (int64_t)(jl * p.g + hh) * p.dh;
                        dq[i] = y0;
                        dq[i + half] = y1;
                    } else {
                        uint16_t* dst = (hh == p.g ? p.k_cache[v] : p.v_cache[v]) +
                                        ((int64_t)jl * p.max_tokens[v] + es.pos[v]) * p.dh;
                        dst[i] = f32_to_bf16_bits(y0);  // the KV cache is BF16
                        dst[i + half] = f32_to_bf16_bits(y1);
                    }
                }
            }
        }
    } else if (lane < N && v < p.nb) {
        const int row = w0 + r;
        if (row < p.rows) {
            if (MODE == M_LM) {
                float* lg = p.logits + v * p.logit_stride + row;
                if (pass == 0)
                    *lg = s;
                else
                    *lg += s;  // later K passes: the same lane wrote the row before
            } else {
                const float val = es.res[v][row - es.w_lo] + es.sc[row - es.w_lo] * s;
                es.res[v][row - es.w_lo] = val;
                if (pass == p.passes - 1) {
                    p.resid_out[v * p.x_stride + row] = val;
                    if (p.hidden_out) p.hidden_out[v * p.hid_stride + row] = val;
                }
            }
        }
    }
}

// ------------------------------------------------------------------ the kernel
template <int MODE, int R, int XC, int NB, bool GS = false>
__global__ void __launch_bounds__(THREADS, 1) gemv_kernel(const Params p) {
    static_assert(R * NB <= 32, "row x vector entries must fit one warp");
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ float red[NRB][CW][R * NB];
    __shared__ float stat[NB][CW];
    __shared__ int abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int seg_bytes = p.seg * 16;  // row stride inside a stage
    const Smem L = smem_plan(R, seg_bytes, p.smem_cap);
    const int NS = L.nstages;
    float4* xs = reinterpret_cast<float4*>(sm);
    uint8_t* stages = sm + XS_BYTES;
    const uint32_t full0 = smem_u32(stages + NS * L.stage_bytes);
    const uint32_t empty0 = full0 + 8 * MAX_STAGES;
    const uint32_t rfull0 = empty0 + 8 * MAX_STAGES;
    const uint32_t rempty0 = rfull0 + 8 * NRB;
    const int NG = (p.rows + R - 1) / R;
    const int g0 = (int)((int64_t)blockIdx.x * NG / gridDim.x);
    const int g1 = (int)((int64_t)(blockIdx.x + 1) * NG / gridDim.x);
    const int ngrp = g1 - g0;
    const int nitems = ngrp * p.passes;  // stages this CTA consumes: passes x row groups

    if (tid == 0) {
        abort_flag = 0;
        for (int s = 0; s < NS; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, CW);
        }
        for (int b = 0; b < NRB; ++b) {
            mbar_init(rfull0 + 8 * b, CW);
            mbar_init(rempty0 + 8 * b, 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    if (warp == CW) {
        // ---- producer: weights never depend on the previous kernel, so start at once
        pdl_trigger();
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            for (int i = 0; i < nitems; ++i) {
                const int pass = i / ngrp, gi = g0 + (i - pass * ngrp);
                const int cb = pass * p.seg;
                const uint32_t bytes = (uint32_t)(min(p.seg, p.nchunks - cb) * 16);
                if (i >= NS) mbar_wait(empty0 + 8 * s, ph ^ 1, &abort_flag, p.err);
                const int nrow = min(R, p.rows - gi * R);
                mbar_expect_tx(full0 + 8 * s, (uint32_t)nrow * bytes);
                for (int r = 0; r < nrow; ++r)
                    bulk_g2s(smem_u32(stages + (size_t)s * L.stage_bytes + (size_t)r * seg_bytes),
                             row_ptr<MODE>(p, gi * R + r) + (size_t)cb * 16, bytes, full0 + 8 * s);
                if (++s == NS) {
                    s = 0;
                    ph ^= 1;
                }
            }
        }
        if (lane == 0) {
            // never leave while copies into this CTA's shared memory are in flight (even
            // after an abort: this second wait is bounded on its own)
            for (int i = max(0, nitems - NS); i < nitems; ++i)
                mbar_wait(full0 + 8 * (i % NS), (i / NS) & 1, &abort_flag, p.err, false);
        }
        return;
    }
    if (warp == CW + 1) {
        // ---- epilogue warp: stage constants, then finish every row group in order
        __shared__ EpiStage<NB> es;
        const int w_lo = g0 * R, w_hi = min(g1 * R, p.rows);
        if (lane == 0) es.w_lo = w_lo;
        if (MODE != M_LM)  // scales are constant: stage them before the dependency wait
            warp_stage(es.sc, w_hi - w_lo, [&](int i) { return __ldg(p.scale + panel_row<MODE>(p, w_lo + i)); }, lane);
        pdl_wait();
        pdl_trigger();
        if (MODE == M_O || MODE == M_DOWN)
            for (int v = 0; v < p.nb; ++v)
                warp_stage(es.res[v], w_hi - w_lo, [&](int i) { return __ldcg(p.resid_out + v * p.x_stride + w_lo + i); }, lane);
        if (MODE == M_QKV) {
            for (int v = 0; v < p.nb; ++v) {
                const int pos = *p.pos[v];
                if (lane == 0) es.pos[v] = pos;
                for (int i = lane; i < (p.dh >> 1); i += 32)
                    es.rope[v][i] = p.rope[v][(int64_t)pos * (p.dh >> 1) + i];
            }
        }
        __syncwarp();
        int b = 0;
        uint32_t ph = 0;
        for (int i = 0; i < nitems; ++i) {
            const int pass = i / ngrp, gi = g0 + (i - pass * ngrp);
            mbar_wait(rfull0 + 8 * b, ph, &abort_flag, p.err);
            epilogue<MODE, R, NB>(p, red[b], gi, pass, lane, es);
            __syncwarp();
            if (lane == 0) mbar_arrive(rempty0 + 8 * b);
            if (++b == NRB) {
                b = 0;
                ph ^= 1;
            }
        }
        return;
    }

    // ---- consumers
    pdl_wait();
    pdl_trigger();
    float inv[NB];
#pragma unroll
    for (int v = 0; v < NB; ++v) inv[v] = 0.f;
    if (MODE == M_QKV || MODE == M_GU || MODE == M_LM) norm_scales<NB>(p, stat, inv, tid);
    XRegs<XC, NB> xr;     // LM head: FP32 activation slices
    XDigits<XC, NB> xd;   // INT8 modes: block-scaled integer digits of the slices
    int s = 0, b = 0;
    uint32_t sph = 0, bph = 0;
    for (int pass = 0, i = 0; pass < p.passes; ++pass) {
        const int cb = pass * p.seg;
        const int nvalid = min(p.seg, p.nchunks - cb);
        if constexpr (MODE == M_LM)
            make_xregs<XC, NB>(p, inv, xr, cb, nvalid, xs, tid);
        else
            make_digits<MODE, XC, NB>(p, inv, xd, cb, nvalid, xs, tid);
        for (int gi = g0; gi < g1; ++gi, ++i) {
            mbar_wait(full0 + 8 * s, sph, &abort_flag, p.err);
            const uint8_t* st = stages + (size_t)s * L.stage_bytes;
            float acc[R][NB];
            if constexpr (MODE == M_LM) {
                dot_bf16<R, XC, NB>(st, seg_bytes, xr, nvalid, tid, acc);
            } else {
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int v = 0; v < NB; ++v) acc[r][v] = 0.f;
                const uint16_t* grow[R];
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    int w = gi * R + r;
                    if (w >= p.rows) w = 0;  // padding row of a ragged last group: never stored
                    grow[r] = GS ? p.gscale + (size_t)panel_row<MODE>(p, w) * p.gld : nullptr;
                }
                dot_i8<R, XC, NB, GS>(st, seg_bytes, xd, nvalid, tid, acc, grow, p.gshift, cb);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(empty0 + 8 * s);  // this warp is done with the stage
            float vals[R * NB];
#pragma unroll
            for (int r = 0; r < R; ++r)
#pragma unroll
                for (int v = 0; v < NB; ++v) vals[r * NB + v] = acc[r][v];
            const float rs = vec_reduce<R * NB>(vals, lane);
            if (i >= NRB) mbar_wait(rempty0 + 8 * b, bph ^ 1, &abort_flag, p.err);
            if ((lane & (32 / (R * NB) - 1)) == 0) red[b][warp][lane / (32 / (R * NB))] = rs;
            __syncwarp();
            if (lane == 0) mbar_arrive(rfull0 + 8 * b);
            if (++s == NS) {
                s = 0;
                sph ^= 1;
            }
            if (++b == NRB) {
                b = 0;
                bph ^= 1;
            }
        }
    }
}

typedef void (*Fn)(const Params);

// The instantiated variants: NB * XC <= 4 keeps the digit registers of the tuned
// single-vector kernel; R * NB <= 16 bounds the accumulators.
template <int NB, int MODE, bool GS = false>
Fn pick_mode(int R, int XC) {
#define TASP_GEMV_V(r, x) \
    if (R == r && XC == x) return gemv_kernel<MODE, r, x, NB, GS>;
    if constexpr (NB == 1) {
        TASP_GEMV_V(8, 1) TASP_GEMV_V(4, 1) TASP_GEMV_V(2, 1) TASP_GEMV_V(4, 2) TASP_GEMV_V(2, 2) TASP_GEMV_V(2, 4)
        if constexpr (MODE != M_QKV && MODE != M_GU) {
            TASP_GEMV_V(1, 4)  // rotary / SwiGLU pairs need two rows per stage
        }
    } else if constexpr (NB == 2) {
        TASP_GEMV_V(8, 1) TASP_GEMV_V(4, 1) TASP_GEMV_V(2, 1) TASP_GEMV_V(4, 2) TASP_GEMV_V(2, 2)
    } else {
        TASP_GEMV_V(4, 1) TASP_GEMV_V(2, 1)
    }
#undef TASP_GEMV_V
    return nullptr;
}

// gs: the grouped-store variant (INT8 modes with 2 or 4 vectors; one vector of a grouped
// store runs on the single-vector kernels)
template <int NB>
Fn pick_nb(int mode, int R, int XC, bool gs) {
    if (gs) {
        if constexpr (NB == 1) {
            return nullptr;
        } else {
            switch (mode) {
                case M_QKV: return pick_mode<NB, M_QKV, true>(R, XC);
                case M_O: return pick_mode<NB, M_O, true>(R, XC);
                case M_GU: return pick_mode<NB, M_GU, true>(R, XC);
                case M_DOWN: return pick_mode<NB, M_DOWN, true>(R, XC);
                default: return nullptr;
            }
        }
    }
    switch (mode) {
        case M_QKV: return pick_mode<NB, M_QKV>(R, XC);
        case M_O: return pick_mode<NB, M_O>(R, XC);
        case M_GU: return pick_mode<NB, M_GU>(R, XC);
        case M_DOWN: return pick_mode<NB, M_DOWN>(R, XC);
        default: return pick_mode<NB, M_LM>(R, XC);
    }
}

// Kernel variant for (mode, rows per stage R, chunks per thread XC) with NB vectors, per-row
// or grouped scales; nullptr if not built. Each NB is compiled in its own translation unit.
template <int NB>
Fn pick(int mode, int R, int XC, bool gs);
template <>
Fn pick<1>(int mode, int R, int XC, bool gs);
template <>
Fn pick<2>(int mode, int R, int XC, bool gs);
template <>
Fn pick<4>(int mode, int R, int XC, bool gs);

}  // namespace gemv

// One-vector GEMV launch on the single-session kernels (gemv_single.cu).
int launch_gemv_single(int mode, const gemv::Params& p, cudaStream_t s);

}  // namespace tasp
