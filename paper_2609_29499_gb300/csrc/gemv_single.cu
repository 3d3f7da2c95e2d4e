// Single-session GEMV kernels of the decode step (one activation vector per weight pass).
//
// The same roles as the batched kernels of gemv.cuh (producer warp with a cp.async.bulk +
// mbarrier ring started before griddepcontrol.wait, 16 consumer warps on dp4a over
// block-scaled activation digits, an epilogue warp), specialised for one vector: the
// whole normalized activation vector is staged once in shared memory with coalesced
// loads and read back per chunk, which keeps the kernel prologue short. Measured on
// GB300 this variant is ~2 us per launch faster than the batched template at NB = 1,
// so a single session's step uses it.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>

#include "gemv.cuh"
#include "tasp_internal.h"

namespace tasp {
namespace gemv1 {
namespace {


constexpr int NT = 512;  // consumer threads of a GEMV CTA
constexpr int NWARP = NT / 32;

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
    const float* act;
    float* resid_out;
    float* hidden_out;
    float* q_out;
    uint16_t* k_cache;
    uint16_t* v_cache;
    int max_tokens;
    const float2* rope;
    const int* pos;
    int g, dh;
    const int16_t* blk_role;  // QKV: role of each d_h-row block (NULL = block index)
    const uint16_t* gscale;   // groupwise store: BF16 scales [panel row][gld] (NULL = per-row only)
    int gcols, gshift;        // scales per row; chunk c uses scale c >> gshift
    int gld;                  // row stride of gscale (elements)
    int gstage;               // the producer copies each row's scale row into the stage (gld a multiple of 8)
    float skew;               // start-order split: CTA b takes a share 1 + skew (1 - 2 b / (grid - 1)) of the rows
    float* h_out;
    float* logits;
    int* err;       // device error word (bounded waits that gave up)
    int smem_cap;   // dynamic shared memory available to the launch
    long long wait_limit;  // clock cycles before a bounded wait gives up
    int skip_copies;       // failure-detection test hook: the producer issues no copies
};



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

constexpr int CW = NWARP;                // consumer warps
constexpr int CT = CW * 32;              // consumer threads
constexpr int GEMV_THREADS = CT + 64;    // + producer warp + epilogue warp
constexpr int MAX_STAGES = 8;
constexpr int NRB = 8;                   // partial-sum buffers between consumers and the epilogue warp
constexpr long long WAIT_LIMIT = 4000000000ll;  // clock cycles (~2 s) before a wait gives up
constexpr int ERR_WAIT_TIMEOUT = 1;

__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(CT) : "memory"); }

// ---------------------------------------------------------------- activation slices
// Each consumer thread reads its own chunks of the activation vector straight from global
// memory: chunk c = tid + j * CT holds elements [4F c, 4F c + 4F) (16 for the INT8 modes, 8
// for the BF16 LM head). Nothing is staged in shared memory, so the weight ring gets all of
// it. Elements at or beyond `len` read as zero.
template <int F>
__device__ __forceinline__ void chunk_f32(const float* __restrict__ a, int c, int len, float4 (&v)[F]) {
    const int e0 = 4 * F * c;
    if (e0 + 4 * F <= len) {
#pragma unroll
        for (int e = 0; e < F; ++e) v[e] = reinterpret_cast<const float4*>(a + e0)[e];
    } else {
#pragma unroll
        for (int e = 0; e < F; ++e) {
            const int b = e0 + 4 * e;
            v[e] = make_float4(b < len ? a[b] : 0.f, b + 1 < len ? a[b + 1] : 0.f, b + 2 < len ? a[b + 2] : 0.f,
                               b + 3 < len ? a[b + 3] : 0.f);
        }
    }
}
// BF16 step input (16-byte aligned; len a multiple of 16)
template <int F>
__device__ __forceinline__ void chunk_bf16(const uint16_t* __restrict__ a, int c, int len, float4 (&v)[F]) {
    const int e0 = 4 * F * c;
#pragma unroll
    for (int e = 0; e < F; e += 2) {
        uint4 b = make_uint4(0u, 0u, 0u, 0u);
        if (e0 + 4 * F <= len) b = reinterpret_cast<const uint4*>(a + e0)[e >> 1];
        v[e] = make_float4(__uint_as_float(b.x << 16), __uint_as_float(b.x & 0xffff0000u), __uint_as_float(b.y << 16),
                           __uint_as_float(b.y & 0xffff0000u));
        if (e + 1 < F)
            v[e + 1] = make_float4(__uint_as_float(b.z << 16), __uint_as_float(b.z & 0xffff0000u),
                                   __uint_as_float(b.w << 16), __uint_as_float(b.w & 0xffff0000u));
    }
}

// The residual stream's chunk c (the step input on the first layer).
template <int F>
__device__ __forceinline__ void chunk_resid(const GemvParams& p, int c, float4 (&v)[F]) {
    if (p.x_in)
        chunk_bf16<F>(p.x_in, c, p.K, v);
    else
        chunk_f32<F>(p.x_resid, c, p.K, v);
}

// The consumer's slice held in registers: chunk j of the thread is c = tid + j * CT.
template <int XC, int F>
struct Slice {
    float4 v[XC][F];
};

// Norm gains of this thread's chunks: constant, so they are read before the dependency wait.
template <int XC, int F>
__device__ __forceinline__ void load_gamma(const GemvParams& p, int tid, Slice<XC, F>& g) {
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const int c = tid + j * CT;
        if (c < p.nchunks)
            chunk_f32<F>(p.gamma, c, p.K, g.v[j]);
        else
#pragma unroll
            for (int e = 0; e < F; ++e) g.v[j][e] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
}

// The activation slice: x^ = x * inv * gamma with inv = 1 / sqrt(mean(x^2) + eps) for the norm
// modes, the plain activation otherwise. One read of this thread's chunks after the dependency
// wait; the sum of squares is taken in the same fixed order by every CTA (each thread its
// chunks, then the warps in index order), so all CTAs see identical x^. On the first layer CTA
// 0 also writes the widened step input into the residual buffer.
template <int MODE, int XC, int F>
__device__ __forceinline__ void load_slice(const GemvParams& p, int tid, float* stat, const Slice<XC, F>& g,
                                           Slice<XC, F>& x) {
    constexpr bool NORM = MODE == M_QKV || MODE == M_GU || MODE == M_LM;
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const int c = tid + j * CT;
        if (c < p.nchunks) {
            if (NORM)
                chunk_resid<F>(p, c, x.v[j]);
            else
                chunk_f32<F>(p.act, c, p.K, x.v[j]);
        } else {
#pragma unroll
            for (int e = 0; e < F; ++e) x.v[j][e] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    if (!NORM) return;
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < XC; ++j)
#pragma unroll
        for (int e = 0; e < F; ++e) {
            ss = fmaf(x.v[j][e].x, x.v[j][e].x, ss);
            ss = fmaf(x.v[j][e].y, x.v[j][e].y, ss);
            ss = fmaf(x.v[j][e].z, x.v[j][e].z, ss);
            ss = fmaf(x.v[j][e].w, x.v[j][e].w, ss);
        }
    if (p.x_in && p.x_resid_init && blockIdx.x == 0)
#pragma unroll
        for (int j = 0; j < XC; ++j) {
            const int c = tid + j * CT;
            if (c < p.nchunks && 4 * F * c < p.K)
#pragma unroll
                for (int e = 0; e < F; ++e) reinterpret_cast<float4*>(p.x_resid_init + 4 * F * c)[e] = x.v[j][e];
        }
    ss = warp_sum(ss);
    if ((tid & 31) == 0) stat[tid >> 5] = ss;
    consumer_sync();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < NWARP; ++w) tot += stat[w];
    const float inv = 1.0f / sqrtf(__fdiv_rn(tot, (float)p.K) + p.eps);
#pragma unroll
    for (int j = 0; j < XC; ++j)
#pragma unroll
        for (int e = 0; e < F; ++e) {
            x.v[j][e].x = (x.v[j][e].x * inv) * g.v[j][e].x;
            x.v[j][e].y = (x.v[j][e].y * inv) * g.v[j][e].y;
            x.v[j][e].z = (x.v[j][e].z * inv) * g.v[j][e].z;
            x.v[j][e].w = (x.v[j][e].w * inv) * g.v[j][e].w;
        }
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
// One persistent CTA per SM: warp CW is the producer, warps 0..CW-1 consume.
// The producer streams row groups (R rows, one bulk copy per row) into an NS-stage
// shared-memory ring; stage s has a "full" mbarrier (transaction bytes) and an
// "empty" mbarrier (released by the consumers after their last read of the stage).
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
// Bounded wait: gives up after `limit` cycles, records the failure in the device error
// word and makes every later wait of this CTA return at once (abort), so a lost transfer
// can never hang the GPU; the host reports the error word.
__device__ __forceinline__ void mbar_wait(uint32_t bar, uint32_t parity, int* abort_flag, int* err, long long limit,
                                          bool honor_abort = true) {
    if (honor_abort && *(volatile int*)abort_flag) return;
    if (mbar_try(bar, parity)) return;
    const long long t0 = clock64();
    while (!mbar_try(bar, parity)) {
        if (clock64() - t0 > limit) {
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

// This thread's slice of the activation vector, kept in registers for the whole
// kernel: chunk j of the thread is c = tid + j * CT (16 weight bytes per chunk).
template <int XC, int F>
struct XRegs {
    float4 v[XC][F];
};

// The activation slice of an INT8 GEMV as block-scaled integers: per 16-element chunk
// one power-of-two scale 2^(e-14) with max|x| < 2^e, each element rounded to the integer
// X in [-2^14, 2^14] and split as X = 256 hi + lo (hi signed byte, lo unsigned byte),
// four elements packed per 32-bit word. The INT8 weight words then feed dp4a directly.
template <int XC>
struct XDigits {
    uint32_t hi[XC][4], lo[XC][4];
    float scale[XC];
};

template <int XC>
__device__ __forceinline__ void digits_x(XDigits<XC>& xd, const Slice<XC, 4>& xs) {
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const float4 (&q)[4] = xs.v[j];
        float v[16];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[4 * e + 0] = q[e].x;
            v[4 * e + 1] = q[e].y;
            v[4 * e + 2] = q[e].z;
            v[4 * e + 3] = q[e].w;
        }
        float m = 0.f;
#pragma unroll
        for (int e = 0; e < 16; ++e) m = fmaxf(m, fabsf(v[e]));
        int ex = 0;
        if (m > 0.f) frexpf(m, &ex);  // m = f * 2^ex, f in [0.5, 1): every |x| < 2^ex
        xd.scale[j] = m > 0.f ? ldexpf(1.0f, ex - 14) : 0.f;
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            uint32_t h = 0, l = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const int X = m > 0.f ? __float2int_rn(ldexpf(v[4 * w + b], 14 - ex)) : 0;
                h |= ((uint32_t)(X >> 8) & 0xFFu) << (8 * b);
                l |= ((uint32_t)X & 0xFFu) << (8 * b);
            }
            xd.hi[j][w] = h;
            xd.lo[j][w] = l;
        }
    }
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

// INT8 rows of one stage . x: per chunk sum(w * X) = 256 sum(w * hi) + sum(w * lo) in
// exact INT32, then acc[r] += float(sum) * scale in FP32. GS (groupwise store): the scale
// of the chunk also carries the row's BF16 scale of the chunk's column group.
template <int R, int XC, bool GS>
__device__ __forceinline__ void dot_i8(const uint8_t* __restrict__ stage, int ld, const XDigits<XC>& xd,
                                       int nchunks, int tid, float (&acc)[R], const uint16_t* const (&grow)[R],
                                       int gshift, const uint16_t* __restrict__ gstage, int gld) {
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const int c = tid + j * CT;
        if (c < nchunks) {
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int4 wv = *reinterpret_cast<const int4*>(stage + (size_t)r * ld + (size_t)c * 16);
                const uint32_t wd[4] = {(uint32_t)wv.x, (uint32_t)wv.y, (uint32_t)wv.z, (uint32_t)wv.w};
                int sh = 0, sl = 0;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    sh = dp4a_ss(wd[k], xd.hi[j][k], sh);
                    sl = dp4a_su(wd[k], xd.lo[j][k], sl);
                }
                float xsc = xd.scale[j];
                if constexpr (GS) {
                    // the row's scale of this chunk's column group: staged with the weights, or global
                    const uint16_t sv = gstage ? gstage[r * gld + (c >> gshift)] : __ldg(grow[r] + (c >> gshift));
                    xsc *= __uint_as_float((uint32_t)sv << 16);
                }
                acc[r] = fmaf(__int2float_rn(sh * 256 + sl), xsc, acc[r]);
            }
        }
    }
}

// BF16 rows (LM head): 8 weights per 16-byte chunk
template <int R, int XC>
__device__ __forceinline__ void dot_bf16(const uint8_t* __restrict__ stage, int ld, const XRegs<XC, 2>& xr,
                                         int nchunks, int tid, u64 (&acc)[R]) {
#pragma unroll
    for (int j = 0; j < XC; ++j) {
        const int c = tid + j * CT;
        if (c < nchunks) {
            const float4 x0 = xr.v[j][0], x1 = xr.v[j][1];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int4 wv = *reinterpret_cast<const int4*>(stage + (size_t)r * ld + (size_t)c * 16);
                const uint32_t w0 = wv.x, w1 = wv.y, w2 = wv.z, w3 = wv.w;
                acc[r] = fma2(pk(__uint_as_float(w0 << 16), __uint_as_float(w0 & 0xffff0000u)), pk(x0.x, x0.y), acc[r]);
                acc[r] = fma2(pk(__uint_as_float(w1 << 16), __uint_as_float(w1 & 0xffff0000u)), pk(x0.z, x0.w), acc[r]);
                acc[r] = fma2(pk(__uint_as_float(w2 << 16), __uint_as_float(w2 & 0xffff0000u)), pk(x1.x, x1.y), acc[r]);
                acc[r] = fma2(pk(__uint_as_float(w3 << 16), __uint_as_float(w3 & 0xffff0000u)), pk(x1.z, x1.w), acc[r]);
            }
        }
    }
}

// Warp reduction of R row sums at once: each butterfly level halves the vector a lane
// carries, so lane l ends with the full sum of row l / (32 / R).
template <int R>
__device__ __forceinline__ float row_reduce(float (&v)[R], int lane) {
#pragma unroll
    for (int n = R, o = 16; n > 1; n >>= 1, o >>= 1) {
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
    for (int o = 16 / R; o >= 1; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    return s;
}

// Per-CTA values the epilogue warp stages in shared memory: row scales (constant, read
// before the dependency wait), residual rows (after it) and this position's rotary pairs.
constexpr int EPI_MAXR = 512;
struct EpiStage {
    float sc[EPI_MAXR];
    float res[EPI_MAXR];
    float2 rope[64];
    int w_lo, pos;
    bool ok;  // the CTA's rows fit the staging arrays
};

// Epilogue of one row group, run by the epilogue warp: lanes split the CW partial sums
// of each row, then lanes < R (or < R/2 for rotary / SwiGLU pairs) finish the rows.
template <int MODE, int R>
__device__ __forceinline__ void epilogue(const GemvParams& p, const float (*red)[R], int gi, int lane,
                                         const EpiStage& es) {
    constexpr int LPR = 32 / R;  // lanes per row
    const int r = lane % R;
    float s = 0.f;
#pragma unroll
    for (int w = lane / R; w < CW; w += LPR) s += red[w][r];
#pragma unroll
    for (int o = R; o < 32; o <<= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    // lane r (< R) now holds the full sum of row r of the group
    const int w0 = gi * R;
    if (MODE == M_QKV || MODE == M_GU) {
        const float s_other = __shfl_down_sync(0xffffffffu, s, 1);  // row 2t+1 for lane 2t
        if ((lane & 1) == 0 && lane < R) {
            const float s0 = s, s1 = s_other;
            const int wa = w0 + lane;
            if (wa < p.rows) {
                const float sc0 = es.ok ? es.sc[wa - es.w_lo] : p.scale[panel_row<MODE>(p, wa)];
                const float sc1 = es.ok ? es.sc[wa + 1 - es.w_lo] : p.scale[panel_row<MODE>(p, wa + 1)];
                if (MODE == M_GU) {
                    const float a = sc0 * s0, b = sc1 * s1;
                    const float silu = a / (1.0f + expf(-a));
                    p.h_out[wa >> 1] = silu * b;
                } else {
                    const int half = p.dh >> 1;
                    const int hb = wa / p.dh, i = (wa - hb * p.dh) >> 1;
                    float y0 = sc0 * s0, y1 = sc1 * s1;
                    const int gp2 = p.g + 2;
                    const int code = p.blk_role ? p.blk_role[hb] : hb;
                    const int jl = code / gp2, hh = code - jl * gp2;
                    const int pos = es.pos;
                    if (hh <= p.g) {
                        const float2 cs = es.rope[i];
                        const float ya = y0 * cs.x - y1 * cs.y, yb = y1 * cs.x + y0 * cs.y;
                        y0 = ya;
                        y1 = yb;
                    }
                    if (hh < p.g) {
                        float* dq = p.q_out + (int64_t)(jl * p.g + hh) * p.dh;
                        dq[i] = y0;
                        dq[i + half] = y1;
                    } else {
                        uint16_t* dst = (hh == p.g ? p.k_cache : p.v_cache) + ((int64_t)jl * p.max_tokens + pos) * p.dh;
                        dst[i] = f32_to_bf16_bits(y0);  // the KV cache is BF16
                        dst[i + half] = f32_to_bf16_bits(y1);
                    }
                }
            }
        }
    } else if (lane < R) {
        const int row = w0 + lane;
        if (row < p.rows) {
            if (MODE == M_LM) {
                p.logits[row] = s;
            } else {
                const float base = es.ok ? es.res[row - es.w_lo] : p.resid_out[row];
                const float v = base + (es.ok ? es.sc[row - es.w_lo] : p.scale[row]) * s;
                p.resid_out[row] = v;
                if (p.hidden_out) p.hidden_out[row] = v;
            }
        }
    }
}

// Shared-memory plan of one launch (host and device agree on it).
struct GemvSmem {
    int x_bytes, stage_bytes, nstages, total;
};
__host__ __device__ inline GemvSmem gemv_smem(int nchunks, int F, int R, int ld, int cap, int gscale_bytes = 0) {
    GemvSmem g;
    g.x_bytes = 0;  // the activation slices are read from global memory
    g.stage_bytes = ((R * ld + R * gscale_bytes) + 127) & ~127;  // weight rows, then their scale rows
    const int bar_bytes = (2 * MAX_STAGES + 2 * NRB) * 8 + 16;
    int ns = (cap - g.x_bytes - bar_bytes) / g.stage_bytes;
    g.nstages = ns > MAX_STAGES ? MAX_STAGES : ns;
    g.total = g.x_bytes + g.nstages * g.stage_bytes + bar_bytes;
    return g;
}

template <int MODE, int R, int XC, bool GS>
__global__ void __launch_bounds__(GEMV_THREADS, 1) gemv_kernel(const GemvParams p) {
    extern __shared__ __align__(128) uint8_t sm[];
    __shared__ float red[NRB][CW][R];
    __shared__ float stat[CW];
    __shared__ int abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gsb = GS && p.gstage ? p.gld * 2 : 0;  // bytes of one staged scale row
    const GemvSmem L = gemv_smem(p.nchunks, MODE == M_LM ? 2 : 4, R, (int)p.ld, p.smem_cap, gsb);
    const int NS = L.nstages;
    uint8_t* stages = sm + L.x_bytes;
    const uint32_t full0 = smem_u32(stages + NS * L.stage_bytes);
    const uint32_t empty0 = full0 + 8 * MAX_STAGES;
    const uint32_t rfull0 = empty0 + 8 * MAX_STAGES;
    const uint32_t rempty0 = rfull0 + 8 * NRB;
    const int NG = (p.rows + R - 1) / R;
    // CTAs start in block-index order (each takes the SM the previous kernel frees next), so a
    // launch whose CTAs start spread out gives the later ones a smaller share: with shares
    // 1 + skew (1 - 2 i / (G - 1)), CTA b starts at the prefix NG S(b) / G, S(k) = k (1 + skew)
    // - skew k (k - 1) / (G - 1), S(G) = G. skew = 0: the even split, in integers. FP32 only:
    // FP64 runs at a few operations per clock per SM on this part, microseconds per launch here.
    auto start_of = [&](int b) -> int {
        if (b >= (int)gridDim.x) return NG;
        if (p.skew == 0.f || gridDim.x < 2) return (int)((int64_t)b * NG / gridDim.x);
        const float G = (float)gridDim.x, k = (float)b, sg = p.skew;
        const float S = k * (1.f + sg) - sg * k * (k - 1.f) / (G - 1.f);
        return max(0, min(NG, (int)((float)NG * S / G)));
    };
    const int g0 = start_of(blockIdx.x);
    const int g1 = start_of(blockIdx.x + 1);

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
        if (lane == 0 && !p.skip_copies) {
            int s = 0;
            uint32_t ph = 0;
            for (int gi = g0, i = 0; gi < g1; ++gi, ++i) {
                if (i >= NS) mbar_wait(empty0 + 8 * s, ph ^ 1, &abort_flag, p.err, p.wait_limit);
                const int nrow = min(R, p.rows - gi * R);
                mbar_expect_tx(full0 + 8 * s, (uint32_t)(nrow * (p.ld + gsb)));
                for (int r = 0; r < nrow; ++r) {
                    bulk_g2s(smem_u32(stages + (size_t)s * L.stage_bytes + (size_t)r * p.ld),
                             row_ptr<MODE>(p, gi * R + r), (uint32_t)p.ld, full0 + 8 * s);
                    if (GS && gsb)  // the row's group scales, behind the stage's weight rows
                        bulk_g2s(smem_u32(stages + (size_t)s * L.stage_bytes + (size_t)R * p.ld + (size_t)r * gsb),
                                 p.gscale + (size_t)panel_row<MODE>(p, gi * R + r) * p.gld, (uint32_t)gsb,
                                 full0 + 8 * s);
                }
                if (++s == NS) {
                    s = 0;
                    ph ^= 1;
                }
            }
            // never leave while copies into this CTA's shared memory are in flight (even
            // after an abort: this second wait is bounded on its own)
            for (int gi = max(g0, g1 - NS), i = gi - g0; gi < g1; ++gi, ++i)
                mbar_wait(full0 + 8 * (i % NS), (i / NS) & 1, &abort_flag, p.err, p.wait_limit, false);
        }
        return;
    }
    if (warp == CW + 1) {
        // ---- epilogue warp: cross-warp sums of each row group, then the mode's epilogue
        __shared__ EpiStage es;
        const int w_lo = g0 * R, w_hi = min(g1 * R, p.rows);
        if (lane == 0) {
            es.w_lo = w_lo;
            es.ok = (w_hi - w_lo) <= EPI_MAXR;
        }
        __syncwarp();
        if (MODE != M_LM && es.ok)  // scales are constant: stage them before the dependency wait
            for (int w = w_lo + lane; w < w_hi; w += 32) es.sc[w - w_lo] = p.scale[panel_row<MODE>(p, w)];
        pdl_wait();
        pdl_trigger();
        if ((MODE == M_O || MODE == M_DOWN) && es.ok)
            for (int w = w_lo + lane; w < w_hi; w += 32) es.res[w - w_lo] = p.resid_out[w];
        if (MODE == M_QKV) {
            const int pos = *p.pos;
            if (lane == 0) es.pos = pos;
            for (int i = lane; i < (p.dh >> 1); i += 32) es.rope[i] = p.rope[(int64_t)pos * (p.dh >> 1) + i];
        }
        __syncwarp();
        int b = 0;
        uint32_t ph = 0;
        for (int gi = g0; gi < g1; ++gi) {
            mbar_wait(rfull0 + 8 * b, ph, &abort_flag, p.err, p.wait_limit);
            epilogue<MODE, R>(p, red[b], gi, lane, es);
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
    constexpr int F = MODE == M_LM ? 2 : 4;  // float4s per 16-byte weight chunk
    Slice<XC, F> gam, xsl;
    if (MODE == M_QKV || MODE == M_GU || MODE == M_LM) load_gamma<XC, F>(p, tid, gam);
    pdl_wait();
    pdl_trigger();
    load_slice<MODE, XC, F>(p, tid, stat, gam, xsl);

    XRegs<XC, 2> xr;        // LM head: FP32 activation slice
    XDigits<XC> xd;         // INT8 modes: block-scaled integer digits of the slice
    if constexpr (MODE == M_LM) {
#pragma unroll
        for (int j = 0; j < XC; ++j) {
            xr.v[j][0] = xsl.v[j][0];
            xr.v[j][1] = xsl.v[j][1];
        }
    } else {
        digits_x<XC>(xd, xsl);
    }
    int s = 0, b = 0;
    uint32_t sph = 0, bph = 0;
    for (int gi = g0, i = 0; gi < g1; ++gi, ++i) {
        mbar_wait(full0 + 8 * s, sph, &abort_flag, p.err, p.wait_limit);
        const uint8_t* st = stages + (size_t)s * L.stage_bytes;
        float v[R];
        if constexpr (MODE == M_LM) {
            u64 acc[R];
#pragma unroll
            for (int r = 0; r < R; ++r) acc[r] = 0ull;
            dot_bf16<R, XC>(st, (int)p.ld, xr, p.nchunks, tid, acc);
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const float2 a = upk(acc[r]);
                v[r] = a.x + a.y;
            }
        } else {
#pragma unroll
            for (int r = 0; r < R; ++r) v[r] = 0.f;
            const uint16_t* grow[R];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                int w = gi * R + r;
                if (w >= p.rows) w = 0;  // padding row of a ragged last group: never stored
                grow[r] = GS ? p.gscale + (size_t)panel_row<MODE>(p, w) * p.gld : nullptr;
            }
            dot_i8<R, XC, GS>(st, (int)p.ld, xd, p.nchunks, tid, v, grow, p.gshift,
                              GS && gsb ? reinterpret_cast<const uint16_t*>(st + (size_t)R * p.ld) : nullptr, p.gld);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * s);  // this warp is done with the stage
        const float rs = row_reduce<R>(v, lane);
        if (i >= NRB) mbar_wait(rempty0 + 8 * b, bph ^ 1, &abort_flag, p.err, p.wait_limit);
        if ((lane & (32 / R - 1)) == 0) red[b][warp][lane / (32 / R)] = rs;
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

// ---------------------------------------------------------------- host side
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

template <int MODE, bool GS>
GemvFn gemv_fn(int R, int XC) {
    if (XC <= 1) {
        if (R >= 8) return gemv_kernel<MODE, 8, 1, GS>;
        if (R >= 4) return gemv_kernel<MODE, 4, 1, GS>;
        return gemv_kernel<MODE, 2, 1, GS>;
    }
    if (XC <= 2) {
        if (R >= 4) return gemv_kernel<MODE, 4, 2, GS>;
        return gemv_kernel<MODE, 2, 2, GS>;
    }
    if (XC <= 4) {
        if (R >= 2) return gemv_kernel<MODE, 2, 4, GS>;
        if constexpr (MODE == M_QKV || MODE == M_GU)
            return nullptr;  // rotary / SwiGLU pairs need two rows per stage
        else
            return gemv_kernel<MODE, 1, 4, GS>;
    }
    return nullptr;
}

GemvFn pick(int mode, int R, int XC, bool gs) {
    if (gs) {
        switch (mode) {
            case M_QKV: return gemv_fn<M_QKV, true>(R, XC);
            case M_O: return gemv_fn<M_O, true>(R, XC);
            case M_GU: return gemv_fn<M_GU, true>(R, XC);
            case M_DOWN: return gemv_fn<M_DOWN, true>(R, XC);
            default: return nullptr;  // the LM head is BF16, never grouped
        }
    }
    switch (mode) {
        case M_QKV: return gemv_fn<M_QKV, false>(R, XC);
        case M_O: return gemv_fn<M_O, false>(R, XC);
        case M_GU: return gemv_fn<M_GU, false>(R, XC);
        case M_DOWN: return gemv_fn<M_DOWN, false>(R, XC);
        default: return gemv_fn<M_LM, false>(R, XC);
    }
}

// Rows per stage: the largest power of two with R * row_bytes <= 32 KB (pairs need R >= 2).
int rows_per_stage(int mode, int64_t ld) {
    int R = 8;
    while (R > 1 && (int64_t)R * ld > 32768) R >>= 1;
    if ((mode == M_QKV || mode == M_GU) && R < 2) R = 2;
    return R;
}

std::mutex g_attr_mu;
std::map<const void*, int> g_attr;  // kernel -> dynamic shared memory cap

// Start-order skew of the row split per mode (see the kernel).
constexpr float SKEW_QKV = 0.f, SKEW_O = 0.3f, SKEW_GU = 0.f, SKEW_DOWN = 0.f;

int launch_gemv(int mode, GemvParams p, int* err, cudaStream_t s) {
    if (p.rows == 0) return TASP_OK;
    p.wait_limit = test_hooks::wait_limit(WAIT_LIMIT);
    p.skew = mode == M_O ? SKEW_O : mode == M_GU ? SKEW_GU : mode == M_DOWN ? SKEW_DOWN : mode == M_QKV ? SKEW_QKV : 0.f;
    p.skip_copies = test_hooks::take_skip() ? 1 : 0;
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    int R = rows_per_stage(mode, p.ld);
    int XC = 1;
    while (XC * CT < p.nchunks) XC <<= 1;
    if (XC > 4) return fail(TASP_EUNSUP, "row too long for the register-resident activation slice");
    if (XC == 2 && R > 4) R = 4;
    if (XC == 4 && R > 2) R = 2;
    GemvFn fn = pick(mode, R, XC, p.gscale != nullptr);
    if (!fn) return fail(TASP_EINVAL, "no GEMV variant for this row length");
    p.err = err;
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
    // group scales ride in the stage when their rows are 16-byte multiples (the plans pad them)
    p.gstage = p.gscale && p.gld % 8 == 0 && (reinterpret_cast<uintptr_t>(p.gscale) & 15) == 0 ? 1 : 0;
    const GemvSmem L = gemv_smem(p.nchunks, mode == M_LM ? 2 : 4, R, (int)p.ld, p.smem_cap, p.gstage ? p.gld * 2 : 0);
    if (L.nstages < 2) return fail(TASP_EUNSUP, "row or activation vector too long for the shared-memory ring");
    const int NG = (p.rows + R - 1) / R;
    const int grid = std::max(1, std::min(NG, di.sms));
    return launch_pdl(fn, dim3(grid), dim3(GEMV_THREADS), (size_t)L.total, s, p);
}

}  // namespace
}  // namespace gemv1

// One GEMV launch for one activation vector (the fields of gemv::Params for vector 0).
int launch_gemv_single(int mode, const gemv::Params& q, cudaStream_t s) {
    gemv1::GemvParams p{};
    p.w = q.w;
    p.map = q.map;
    p.scale = q.scale;
    p.ld = q.ld;
    p.rows = q.rows;
    p.K = q.K;
    p.nchunks = q.nchunks;
    p.x_resid = q.x_resid;
    p.x_in = q.x_in;
    p.x_resid_init = q.x_resid_init;
    p.gamma = q.gamma;
    p.eps = q.eps;
    p.act = q.act;
    p.resid_out = q.resid_out;
    p.hidden_out = q.hidden_out;
    p.q_out = q.q_out;
    p.k_cache = q.k_cache[0];
    p.v_cache = q.v_cache[0];
    p.max_tokens = q.max_tokens[0];
    p.rope = q.rope[0];
    p.pos = q.pos[0];
    p.g = q.g;
    p.dh = q.dh;
    p.blk_role = q.blk_role;
    p.gscale = q.gscale;
    p.gcols = q.gcols;
    p.gshift = q.gshift;
    p.gld = q.gld;
    p.h_out = q.h_out;
    p.logits = q.logits;
    return gemv1::launch_gemv(mode, p, q.err, s);
}

}  // namespace tasp
