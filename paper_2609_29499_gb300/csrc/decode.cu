// Decode kernels of the compiled sparse path (batch 1 per plan step), sm_103a.
//
// Every projection is an HBM-bound GEMV over the retained rows of an INT8 panel with
// one FP32 scale per output row (the paper's INT8-weight / BF16-compute runtime,
// Sec. 4 and Table 1). Design:
//  * persistent grid (SMs x resident CTAs), each CTA owns a contiguous range of row
//    groups (R rows) and splits K across its 256 threads in 16-byte chunks, so a row
//    group keeps R x CPT 128-bit streaming loads in flight per thread;
//  * the next group is loaded into a second register buffer and the one after is
//    prefetched into L2 with cp.async.bulk.prefetch while the current one is reduced;
//  * the activation vector (BF16 values) sits in shared memory as FP32 with an XOR
//    swizzle that makes the per-chunk 128-bit reads conflict-free;
//  * INT8 -> FP32 is exact: byte ^ 0x80 is placed in the mantissa of 2^23 with PRMT and
//    2^23 + 128 is subtracted (packed f32x2 add), then packed f32x2 FMAs accumulate;
//    the row scale is applied once after the reduction;
//  * the previous kernel's tail is overlapped with programmatic dependent launch:
//    weights (which never depend on the previous kernel) are fetched before
//    griddepcontrol.wait, activations after it.
// Attention is a split-KV (flash-decoding) kernel over the retained KV heads only; the
// last CTA of each KV group (atomic ticket, no waiting) merges the splits.
#include <cuda_bf16.h>

#include <cmath>
#include <map>
#include <mutex>

#include "tasp_internal.h"

namespace tasp {

namespace {

constexpr int NT = 256;
constexpr int NWARP = NT / 32;
constexpr int ATT_THREADS = 256;
constexpr int ATT_SPLITS_MAX = 64;

enum GemvMode { M_QKV = 0, M_O = 1, M_GU = 2, M_DOWN = 3, M_LM = 4 };

struct GemvParams {
    const int8_t* w;
    const int32_t* map;
    const float* scale;
    int64_t ld;
    int rows, K, nchunks;
    const float* x_resid;
    const uint16_t* x_in;
    float* x_resid_init;
    const float* gamma;
    float eps;
    const uint16_t* act;
    float* resid_out;
    float* hidden_out;
    uint16_t* q_out;
    uint16_t* k_cache;
    uint16_t* v_cache;
    int max_tokens;
    const float2* rope;
    const int* pos;
    int g, dh;
    uint16_t* h_out;
    float* logits;
};

struct AttnParams {
    const uint16_t* q;
    const uint16_t* K;
    const uint16_t* V;
    const int* pos;
    int max_tokens;
    float qscale;  // 1/sqrt(dh) * log2(e)
    float* part;
    int* cnt;
    uint16_t* o;
};

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ int4 ld_stream16(const void* p) {
    int4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.s32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

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
__device__ __forceinline__ u64 add2(u64 a, u64 b) {
    u64 d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ u64 fma2(u64 a, u64 b, u64 c) {
    u64 d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// float4 index swizzle: F = float4s per 16-byte weight chunk (4 for INT8, 2 for BF16)
template <int F>
__device__ __forceinline__ int swz(int f) {
    return f ^ ((f >> 3) & (F - 1));
}

__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ float round_bf16(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }
__device__ __forceinline__ uint16_t f32_to_bf16_bits(float v) {
    __nv_bfloat16 b = __float2bfloat16_rn(v);
    return *reinterpret_cast<uint16_t*>(&b);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// ---------------------------------------------------------------- activation prologues
// x^ = bf16(x * (1/sqrt(mean(x^2) + eps)) * gamma) into swizzled FP32 shared memory.
// Every CTA reduces in the same fixed order, so all CTAs see identical x^.
template <int F>
__device__ void norm_to_smem(const float* __restrict__ x, const uint16_t* __restrict__ x_in, float* x_init,
                             const float* __restrict__ gamma, int d, float eps, int nchunks, float4* xs,
                             float* stat) {
    const int tid = threadIdx.x;
    const int n4 = d / 4;
    float ss = 0.f;
    for (int f = tid; f < n4; f += NT) {
        float4 v;
        if (x_in) {
            uint2 b = *reinterpret_cast<const uint2*>(x_in + 4 * f);
            v = make_float4(__uint_as_float(b.x << 16), __uint_as_float(b.x & 0xffff0000u),
                            __uint_as_float(b.y << 16), __uint_as_float(b.y & 0xffff0000u));
            if (x_init && blockIdx.x == 0) reinterpret_cast<float4*>(x_init)[f] = v;
        } else {
            v = reinterpret_cast<const float4*>(x)[f];
        }
        ss = fmaf(v.x, v.x, ss);
        ss = fmaf(v.y, v.y, ss);
        ss = fmaf(v.z, v.z, ss);
        ss = fmaf(v.w, v.w, ss);
    }
    ss = warp_sum(ss);
    if ((tid & 31) == 0) stat[tid >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < NWARP; ++w) tot += stat[w];
    const float inv = 1.0f / sqrtf(__fdiv_rn(tot, (float)d) + eps);
    const int ntot4 = nchunks * F;  // float4 slots including zero padding
    for (int f = tid; f < ntot4; f += NT) {
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
        if (f < n4) {
            float4 v;
            if (x_in) {
                uint2 b = *reinterpret_cast<const uint2*>(x_in + 4 * f);
                v = make_float4(__uint_as_float(b.x << 16), __uint_as_float(b.x & 0xffff0000u),
                                __uint_as_float(b.y << 16), __uint_as_float(b.y & 0xffff0000u));
            } else {
                v = reinterpret_cast<const float4*>(x)[f];
            }
            float4 gm = reinterpret_cast<const float4*>(gamma)[f];
            o.x = round_bf16((v.x * inv) * gm.x);
            o.y = round_bf16((v.y * inv) * gm.y);
            o.z = round_bf16((v.z * inv) * gm.z);
            o.w = round_bf16((v.w * inv) * gm.w);
        }
        xs[swz<F>(f)] = o;
    }
    __syncthreads();
}

// BF16 activation vector [K] -> swizzled FP32 shared memory (zero padded to nchunks*16)
__device__ void bf16_to_smem(const uint16_t* __restrict__ a, int K, int nchunks, float4* xs) {
    const int tid = threadIdx.x;
    const int ntot4 = nchunks * 4;
    for (int f = tid; f < ntot4; f += NT) {
        float4 o;
        int e = 4 * f;
        o.x = (e + 0 < K) ? bf16_to_f32(a[e + 0]) : 0.f;
        o.y = (e + 1 < K) ? bf16_to_f32(a[e + 1]) : 0.f;
        o.z = (e + 2 < K) ? bf16_to_f32(a[e + 2]) : 0.f;
        o.w = (e + 3 < K) ? bf16_to_f32(a[e + 3]) : 0.f;
        xs[swz<4>(f)] = o;
    }
    __syncthreads();
}

// ---------------------------------------------------------------- row addressing
// QKV work rows are ordered so that each even/odd pair holds rows i and i + dh/2 of
// one head (a rotary pair); all other modes use the panel order.
template <int MODE>
__device__ __forceinline__ int panel_row(const GemvParams& p, int w) {
    if (MODE == M_QKV) {
        int hb = w / p.dh, iw = w - hb * p.dh;
        return hb * p.dh + (iw >> 1) + (iw & 1) * (p.dh >> 1);
    }
    return w;
}

template <int MODE>
__device__ __forceinline__ const int8_t* row_ptr(const GemvParams& p, int w) {
    if (w >= p.rows) w = 0;  // padding row of a ragged last group: loaded, never stored
    int pr = panel_row<MODE>(p, w);
    int src = p.map ? __ldg(p.map + pr) : pr;
    return p.w + (int64_t)src * p.ld;
}

// ---------------------------------------------------------------- the GEMV core
template <int R, int CPT>
struct WRegs {
    int4 v[R][CPT];
};

template <int MODE, int R, int CPT>
__device__ __forceinline__ void load_group(WRegs<R, CPT>& wr, const GemvParams& p, int gi, int tid) {
    const int8_t* rp[R];
#pragma unroll
    for (int r = 0; r < R; ++r) rp[r] = row_ptr<MODE>(p, gi * R + r);
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
        const int c = tid + i * NT;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            if (c < p.nchunks)
                wr.v[r][i] = ld_stream16(rp[r] + (int64_t)c * 16);
            else
                wr.v[r][i] = make_int4(0, 0, 0, 0);
        }
    }
}

template <int MODE, int R>
__device__ __forceinline__ void prefetch_group(const GemvParams& p, int gi, int g1, int tid) {
    if (tid < R && gi < g1) {
        const int w = gi * R + tid;
        if (w < p.rows) prefetch_l2(row_ptr<MODE>(p, w), (uint32_t)(p.nchunks * 16));
    }
}

// INT8 chunk dot products: acc[r] (packed pairs) += w[r] . x
template <int R, int CPT>
__device__ __forceinline__ void dot_i8(const WRegs<R, CPT>& wr, const float4* __restrict__ xs, int nchunks, int tid,
                                       u64 (&acc)[R]) {
    const u64 magic = pk(-8388736.0f, -8388736.0f);  // -(2^23 + 128)
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
        const int c = tid + i * NT;
        if (c < nchunks) {
            float4 xv[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) xv[j] = xs[swz<4>(4 * c + j)];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const uint32_t wd[4] = {(uint32_t)wr.v[r][i].x, (uint32_t)wr.v[r][i].y, (uint32_t)wr.v[r][i].z,
                                        (uint32_t)wr.v[r][i].w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint32_t u = wd[j] ^ 0x80808080u;
                    u64 p01 = pk(__uint_as_float(prmt(u, 0x4B000000u, 0x7540u)),
                                 __uint_as_float(prmt(u, 0x4B000000u, 0x7541u)));
                    u64 p23 = pk(__uint_as_float(prmt(u, 0x4B000000u, 0x7542u)),
                                 __uint_as_float(prmt(u, 0x4B000000u, 0x7543u)));
                    p01 = add2(p01, magic);
                    p23 = add2(p23, magic);
                    acc[r] = fma2(p01, pk(xv[j].x, xv[j].y), acc[r]);
                    acc[r] = fma2(p23, pk(xv[j].z, xv[j].w), acc[r]);
                }
            }
        }
    }
}

// BF16 chunk dot products (LM head): 8 weights per 16-byte chunk
template <int R, int CPT>
__device__ __forceinline__ void dot_bf16(const WRegs<R, CPT>& wr, const float4* __restrict__ xs, int nchunks, int tid,
                                         u64 (&acc)[R]) {
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
        const int c = tid + i * NT;
        if (c < nchunks) {
            const float4 x0 = xs[swz<2>(2 * c)], x1 = xs[swz<2>(2 * c + 1)];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const uint32_t w0 = wr.v[r][i].x, w1 = wr.v[r][i].y, w2 = wr.v[r][i].z, w3 = wr.v[r][i].w;
                acc[r] = fma2(pk(__uint_as_float(w0 << 16), __uint_as_float(w0 & 0xffff0000u)), pk(x0.x, x0.y), acc[r]);
                acc[r] = fma2(pk(__uint_as_float(w1 << 16), __uint_as_float(w1 & 0xffff0000u)), pk(x0.z, x0.w), acc[r]);
                acc[r] = fma2(pk(__uint_as_float(w2 << 16), __uint_as_float(w2 & 0xffff0000u)), pk(x1.x, x1.y), acc[r]);
                acc[r] = fma2(pk(__uint_as_float(w3 << 16), __uint_as_float(w3 & 0xffff0000u)), pk(x1.z, x1.w), acc[r]);
            }
        }
    }
}

// Reduce, then the mode's epilogue for one row group.
template <int MODE, int R, int CPT>
__device__ __forceinline__ void finish_group(const GemvParams& p, const WRegs<R, CPT>& wr, const float4* xs, int gi,
                                             float (*red)[NWARP][R], int parity, int tid) {
    u64 acc[R];
#pragma unroll
    for (int r = 0; r < R; ++r) acc[r] = 0ull;
    if (MODE == M_LM)
        dot_bf16<R, CPT>(wr, xs, p.nchunks, tid, acc);
    else
        dot_i8<R, CPT>(wr, xs, p.nchunks, tid, acc);
    const int lane = tid & 31, warp = tid >> 5;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        float2 a = upk(acc[r]);
        float v = warp_sum(a.x + a.y);
        if (lane == 0) red[parity][warp][r] = v;
    }
    __syncthreads();
    const int w0 = gi * R;
    if (MODE == M_QKV || MODE == M_GU) {
        if (tid < R / 2) {
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int w = 0; w < NWARP; ++w) {
                s0 += red[parity][w][2 * tid];
                s1 += red[parity][w][2 * tid + 1];
            }
            const int wa = w0 + 2 * tid;
            if (wa < p.rows) {
                if (MODE == M_GU) {
                    const float a = p.scale[wa] * s0, b = p.scale[wa + 1] * s1;
                    const float silu = a / (1.0f + expf(-a));
                    p.h_out[wa >> 1] = f32_to_bf16_bits(silu * b);
                } else {
                    const int half = p.dh >> 1;
                    const int hb = wa / p.dh, i = (wa - hb * p.dh) >> 1;
                    const int pr0 = hb * p.dh + i, pr1 = pr0 + half;
                    float y0 = p.scale[pr0] * s0, y1 = p.scale[pr1] * s1;
                    const int gp2 = p.g + 2;
                    const int jl = hb / gp2, hh = hb - jl * gp2;
                    const int pos = *p.pos;
                    if (hh <= p.g) {
                        const float2 cs = p.rope[(int64_t)pos * half + i];
                        const float a = y0 * cs.x - y1 * cs.y, b = y1 * cs.x + y0 * cs.y;
                        y0 = a;
                        y1 = b;
                    }
                    uint16_t* dst;
                    if (hh < p.g)
                        dst = p.q_out + (int64_t)(jl * p.g + hh) * p.dh;
                    else if (hh == p.g)
                        dst = p.k_cache + ((int64_t)jl * p.max_tokens + pos) * p.dh;
                    else
                        dst = p.v_cache + ((int64_t)jl * p.max_tokens + pos) * p.dh;
                    dst[i] = f32_to_bf16_bits(y0);
                    dst[i + half] = f32_to_bf16_bits(y1);
                }
            }
        }
    } else {
        if (tid < R) {
            float s = 0.f;
#pragma unroll
            for (int w = 0; w < NWARP; ++w) s += red[parity][w][tid];
            const int row = w0 + tid;
            if (row < p.rows) {
                if (MODE == M_LM) {
                    p.logits[row] = s;
                } else {
                    const float v = p.resid_out[row] + p.scale[row] * s;
                    p.resid_out[row] = v;
                    if (p.hidden_out) p.hidden_out[row] = v;
                }
            }
        }
    }
}

template <int MODE, int R, int CPT>
__global__ void __launch_bounds__(NT) gemv_kernel(const GemvParams p) {
    extern __shared__ __align__(16) float4 xs[];
    __shared__ float red[2][NWARP][R];
    __shared__ float stat[NWARP];
    const int tid = threadIdx.x;
    const int NG = (p.rows + R - 1) / R;
    const int g0 = (int)((int64_t)blockIdx.x * NG / gridDim.x);
    const int g1 = (int)((int64_t)(blockIdx.x + 1) * NG / gridDim.x);

    // weights never depend on the previous kernel: start streaming them now
    prefetch_group<MODE, R>(p, g0 + 1, g1, tid);
    WRegs<R, CPT> A, B;
    if (g0 < g1) load_group<MODE, R, CPT>(A, p, g0, tid);

    pdl_wait();
    pdl_trigger();
    if (MODE == M_QKV || MODE == M_GU)
        norm_to_smem<4>(p.x_resid, p.x_in, p.x_resid_init, p.gamma, p.K, p.eps, p.nchunks, xs, stat);
    else if (MODE == M_LM)
        norm_to_smem<2>(p.x_resid, nullptr, nullptr, p.gamma, p.K, p.eps, p.nchunks, xs, stat);
    else
        bf16_to_smem(p.act, p.K, p.nchunks, xs);

    for (int gi = g0; gi < g1; gi += 2) {
        if (gi + 1 < g1) load_group<MODE, R, CPT>(B, p, gi + 1, tid);
        prefetch_group<MODE, R>(p, gi + 2, g1, tid);
        finish_group<MODE, R, CPT>(p, A, xs, gi, red, 0, tid);
        if (gi + 1 < g1) {
            if (gi + 2 < g1) load_group<MODE, R, CPT>(A, p, gi + 2, tid);
            prefetch_group<MODE, R>(p, gi + 3, g1, tid);
            finish_group<MODE, R, CPT>(p, B, xs, gi + 1, red, 1, tid);
        }
    }
}

// ---------------------------------------------------------------- attention
template <int DH, int G>
__global__ void __launch_bounds__(ATT_THREADS) attn_kernel(const AttnParams p) {
    constexpr int DPL = DH / 32;
    __shared__ float sm_m[NWARP][G], sm_l[NWARP][G];
    __shared__ float sm_acc[NWARP][G][DH];
    __shared__ int is_last;
    const int split = blockIdx.x, jl = blockIdx.y, S = gridDim.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    // The prior cache does not depend on the previous kernel (only position T-1 does,
    // and L2 is coherent): pull this CTA's K/V range into L2 before waiting.
    const int T = *p.pos + 1;  // written by the previous step, which has completed
    const int chunk = (T + S - 1) / S;
    const int p0 = split * chunk, p1 = min(T, p0 + chunk);
    const uint16_t* Kg = p.K + (int64_t)jl * p.max_tokens * DH;
    const uint16_t* Vg = p.V + (int64_t)jl * p.max_tokens * DH;
    if (tid == 0 && p1 > p0) prefetch_l2(Kg + (int64_t)p0 * DH, (uint32_t)((p1 - p0) * DH * 2));
    if (tid == 32 && p1 > p0) prefetch_l2(Vg + (int64_t)p0 * DH, (uint32_t)((p1 - p0) * DH * 2));
    pdl_wait();
    pdl_trigger();

    float q[G][DPL];
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < DPL; ++e) q[h][e] = bf16_to_f32(p.q[(int64_t)(jl * G + h) * DH + lane * DPL + e]) * p.qscale;
    float m[G], l[G], acc[G][DPL];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int e = 0; e < DPL; ++e) acc[h][e] = 0.f;
    }
    constexpr int UNR = 4;
    for (int t0 = p0 + warp; t0 < p1; t0 += UNR * NWARP) {
        float k[UNR][DPL], v[UNR][DPL];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            const int t = t0 + u * NWARP;
            if (t < p1) {
                const uint16_t* kp = Kg + (int64_t)t * DH + lane * DPL;
                const uint16_t* vp = Vg + (int64_t)t * DH + lane * DPL;
                if constexpr (DPL == 4) {
                    const uint2 kb = *reinterpret_cast<const uint2*>(kp);
                    const uint2 vb = *reinterpret_cast<const uint2*>(vp);
                    k[u][0] = __uint_as_float(kb.x << 16);
                    k[u][1] = __uint_as_float(kb.x & 0xffff0000u);
                    k[u][2] = __uint_as_float(kb.y << 16);
                    k[u][3] = __uint_as_float(kb.y & 0xffff0000u);
                    v[u][0] = __uint_as_float(vb.x << 16);
                    v[u][1] = __uint_as_float(vb.x & 0xffff0000u);
                    v[u][2] = __uint_as_float(vb.y << 16);
                    v[u][3] = __uint_as_float(vb.y & 0xffff0000u);
                } else {
                    const uint32_t kb = *reinterpret_cast<const uint32_t*>(kp);
                    const uint32_t vb = *reinterpret_cast<const uint32_t*>(vp);
                    k[u][0] = __uint_as_float(kb << 16);
                    k[u][1] = __uint_as_float(kb & 0xffff0000u);
                    v[u][0] = __uint_as_float(vb << 16);
                    v[u][1] = __uint_as_float(vb & 0xffff0000u);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            if (t0 + u * NWARP < p1) {
                float sc[G];
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    float a = 0.f;
#pragma unroll
                    for (int e = 0; e < DPL; ++e) a = fmaf(q[h][e], k[u][e], a);
                    sc[h] = warp_sum(a);
                }
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    const float mn = fmaxf(m[h], sc[h]);
                    const float c = exp2f(m[h] - mn);  // m = -inf before the first key gives 0
                    const float pe = exp2f(sc[h] - mn);
                    l[h] = l[h] * c + pe;
#pragma unroll
                    for (int e = 0; e < DPL; ++e) acc[h][e] = fmaf(acc[h][e], c, pe * v[u][e]);
                    m[h] = mn;
                }
            }
        }
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
        if (lane == 0) {
            sm_m[warp][h] = m[h];
            sm_l[warp][h] = l[h];
        }
#pragma unroll
        for (int e = 0; e < DPL; ++e) sm_acc[warp][h][lane * DPL + e] = acc[h][e];
    }
    __syncthreads();
    float* part = p.part + (int64_t)(jl * S + split) * G * (DH + 2);
    for (int it = tid; it < G * DH; it += ATT_THREADS) {
        const int h = it / DH, dim = it - h * DH;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NWARP; ++w) M = fmaxf(M, sm_m[w][h]);
        float Ls = 0.f, As = 0.f;
#pragma unroll
        for (int w = 0; w < NWARP; ++w) {
            const float sc = (sm_m[w][h] == -INFINITY) ? 0.f : exp2f(sm_m[w][h] - M);
            Ls = fmaf(sm_l[w][h], sc, Ls);
            As = fmaf(sm_acc[w][h][dim], sc, As);
        }
        part[h * (DH + 2) + dim] = As;
        if (dim == 0) {
            part[h * (DH + 2) + DH] = M;
            part[h * (DH + 2) + DH + 1] = Ls;
        }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) is_last = (atomicAdd(p.cnt + jl, 1) == S - 1);
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    const float* pg = p.part + (int64_t)jl * S * G * (DH + 2);
    for (int it = tid; it < G * DH; it += ATT_THREADS) {
        const int h = it / DH, dim = it - h * DH;
        float M = -INFINITY;
        for (int sp = 0; sp < S; ++sp) M = fmaxf(M, __ldcg(pg + (sp * G + h) * (DH + 2) + DH));
        float Ls = 0.f, As = 0.f;
        for (int sp = 0; sp < S; ++sp) {
            const float* e = pg + (sp * G + h) * (DH + 2);
            const float ms = __ldcg(e + DH);
            const float sc = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
            Ls = fmaf(__ldcg(e + DH + 1), sc, Ls);
            As = fmaf(__ldcg(e + dim), sc, As);
        }
        p.o[(int64_t)(jl * G + h) * DH + dim] = f32_to_bf16_bits(As / Ls);
    }
    if (tid == 0) p.cnt[jl] = 0;
}

__global__ void advance_kernel(int* pos) {
    pdl_wait();
    pdl_trigger();
    if (threadIdx.x == 0) *pos += 1;
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

typedef void (*GemvFn)(const GemvParams);

struct GemvVariant {
    GemvFn fn;
    int R, CPT;
};

template <int MODE>
GemvVariant pick_variant(int nchunks) {
    const int cpt = (nchunks + NT - 1) / NT;
    if (cpt <= 1) return {gemv_kernel<MODE, 8, 1>, 8, 1};
    if (cpt <= 2) return {gemv_kernel<MODE, 4, 2>, 4, 2};
    if (cpt <= 4) return {gemv_kernel<MODE, 2, 4>, 2, 4};
    return {gemv_kernel<MODE, 2, 8>, 2, 8};
}

GemvVariant pick(int mode, int nchunks) {
    switch (mode) {
        case M_QKV: return pick_variant<M_QKV>(nchunks);
        case M_O: return pick_variant<M_O>(nchunks);
        case M_GU: return pick_variant<M_GU>(nchunks);
        case M_DOWN: return pick_variant<M_DOWN>(nchunks);
        default: return pick_variant<M_LM>(nchunks);
    }
}

std::mutex g_occ_mu;
std::map<std::pair<const void*, size_t>, int> g_occ;

int resident_ctas(const void* fn, int threads, size_t smem, int* out) {
    std::lock_guard<std::mutex> lk(g_occ_mu);
    auto key = std::make_pair(fn, smem);
    auto it = g_occ.find(key);
    if (it != g_occ.end()) {
        *out = it->second;
        return TASP_OK;
    }
    TASP_CUDA(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
    int n = 0;
    TASP_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, threads, smem));
    if (n < 1) return fail(TASP_EINVAL, "GEMV configuration does not fit on an SM");
    g_occ[key] = n;
    *out = n;
    return TASP_OK;
}

int launch_gemv(int mode, const GemvParams& p, cudaStream_t s) {
    if (p.rows == 0) return TASP_OK;
    GemvVariant v = pick(mode, p.nchunks);
    const int F = (mode == M_LM) ? 2 : 4;
    const size_t smem = (size_t)p.nchunks * F * sizeof(float4);
    if (smem > 200 * 1024) return fail(TASP_EINVAL, "activation vector too long for shared memory");
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    int occ = 0;
    if ((rc = resident_ctas((const void*)v.fn, NT, smem, &occ))) return rc;
    const int NG = (p.rows + v.R - 1) / v.R;
    const int grid = std::max(1, std::min(NG, di.sms * occ));
    return launch_pdl(v.fn, dim3(grid), dim3(NT), smem, s, p);
}

typedef void (*AttnFn)(const AttnParams);

AttnFn pick_attn(int dh, int g) {
#define TASP_ATT(D, GG) \
    if (dh == D && g == GG) return attn_kernel<D, GG>;
    TASP_ATT(64, 1) TASP_ATT(64, 2) TASP_ATT(64, 4) TASP_ATT(64, 8)
    TASP_ATT(128, 1) TASP_ATT(128, 2) TASP_ATT(128, 4) TASP_ATT(128, 8)
#undef TASP_ATT
    return nullptr;
}

}  // namespace

int attn_splits(int m_kv, int max_tokens, int sms) {
    if (m_kv <= 0) return 1;
    int s = (2 * sms + m_kv - 1) / m_kv;
    s = std::min(s, ATT_SPLITS_MAX);
    s = std::min(s, std::max(1, (max_tokens + 15) / 16));
    return std::max(1, s);
}

int attn_supported(int dh, int g) { return pick_attn(dh, g) != nullptr; }

int enqueue_step(Session& se, const StepTarget& t, cudaStream_t s, int only_layer, KernelHook hook, void* ctx,
                 int* launches) {
    const Plan& pl = *se.plan;
    const Shape& sh = pl.store->sh;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    int nl = 0;
    const int l_begin = only_layer >= 0 ? only_layer : 0;
    const int l_end = only_layer >= 0 ? only_layer + 1 : sh.L;
    auto pre = [&](int kind) { if (hook) hook(ctx, kind, true); };
    auto post = [&](int kind) { if (hook) hook(ctx, kind, false); ++nl; };
    for (int l = l_begin; l < l_end; ++l) {
        const LayerPlan& lp = pl.layers[l];
        const bool first = (l == 0) && t.x_in != nullptr;
        // K1: RMSNorm + QKV GEMV + RoPE + KV append
        GemvParams p{};
        p.w = lp.qkv_w;
        p.map = lp.qkv_map;
        p.scale = lp.qkv_s;
        p.ld = sh.d;
        p.rows = lp.qkv_rows;
        p.K = sh.d;
        p.nchunks = sh.d / 16;
        p.x_resid = se.x;
        p.x_in = first ? t.x_in : nullptr;
        p.x_resid_init = first ? se.x : nullptr;
        p.gamma = lp.g_attn;
        p.eps = sh.eps;
        p.q_out = se.q;
        p.k_cache = se.K[l];
        p.v_cache = se.V[l];
        p.max_tokens = se.max_tokens;
        p.rope = se.rope;
        p.pos = se.d_pos;
        p.g = sh.g();
        p.dh = sh.dh;
        pre(K_QKV);
        if ((rc = launch_gemv(M_QKV, p, s))) return rc;
        post(K_QKV);
        // K2: split-KV attention over the retained KV heads
        if (lp.m_kv > 0) {
            AttnParams a{};
            a.q = se.q;
            a.K = se.K[l];
            a.V = se.V[l];
            a.pos = se.d_pos;
            a.max_tokens = se.max_tokens;
            a.qscale = (float)(1.0 / std::sqrt((double)sh.dh) * 1.4426950408889634);
            a.part = se.part;
            a.cnt = se.cnt;
            a.o = se.o;
            const int S = attn_splits(lp.m_kv, se.max_tokens, di.sms);
            pre(K_ATTN);
            if ((rc = launch_pdl(pick_attn(sh.dh, sh.g()), dim3(S, lp.m_kv), dim3(ATT_THREADS), 0, s, a))) return rc;
            post(K_ATTN);
        }
        // K3: O-projection + residual
        if (lp.m_kv > 0) {
            GemvParams o{};
            o.w = lp.o_w;
            o.scale = lp.o_s;
            o.ld = lp.o_ld;
            o.rows = sh.d;
            o.K = lp.o_K;
            o.nchunks = lp.o_ld / 16;
            o.act = se.o;
            o.resid_out = se.x;
            pre(K_O);
            if ((rc = launch_gemv(M_O, o, s))) return rc;
            post(K_O);
        }
        // K4: RMSNorm + gate/up GEMV + SiLU(gate) * up
        const bool last = (l == sh.L - 1) && only_layer < 0;
        if (lp.c > 0) {
            GemvParams gu{};
            gu.w = lp.gu_w;
            gu.map = lp.gu_map;
            gu.scale = lp.gu_s;
            gu.ld = sh.d;
            gu.rows = lp.gu_rows;
            gu.K = sh.d;
            gu.nchunks = sh.d / 16;
            gu.x_resid = se.x;
            gu.gamma = lp.g_mlp;
            gu.eps = sh.eps;
            gu.h_out = se.h;
            pre(K_GU);
            if ((rc = launch_gemv(M_GU, gu, s))) return rc;
            post(K_GU);
            // K5: down projection + residual
            GemvParams dn{};
            dn.w = lp.dn_w;
            dn.scale = lp.dn_s;
            dn.ld = lp.dn_ld;
            dn.rows = sh.d;
            dn.K = lp.dn_K;
            dn.nchunks = lp.dn_ld / 16;
            dn.act = se.h;
            dn.resid_out = se.x;
            dn.hidden_out = last ? t.hidden_out : nullptr;
            pre(K_DOWN);
            if ((rc = launch_gemv(M_DOWN, dn, s))) return rc;
            post(K_DOWN);
        } else if (last && t.hidden_out) {
            TASP_CUDA(cudaMemcpyAsync(t.hidden_out, se.x, sizeof(float) * sh.d, cudaMemcpyDeviceToDevice, s));
        }
    }
    if (only_layer < 0) {
        if (t.logits) {
            GemvParams lm{};
            lm.w = reinterpret_cast<const int8_t*>(pl.store->lm_head);
            lm.ld = (int64_t)sh.d * 2;
            lm.rows = sh.vocab;
            lm.K = sh.d;
            lm.nchunks = sh.d / 8;
            lm.x_resid = se.x;
            lm.gamma = pl.store->g_final;
            lm.eps = sh.eps;
            lm.logits = t.logits;
            pre(K_LM);
            if ((rc = launch_gemv(M_LM, lm, s))) return rc;
            post(K_LM);
        }
        if (t.advance) {
            pre(K_OTHER);
            if ((rc = launch_pdl(advance_kernel, dim3(1), dim3(32), 0, s, se.d_pos))) return rc;
            post(K_OTHER);
        }
    }
    if (launches) *launches = nl;
    return TASP_OK;
}

}  // namespace tasp
