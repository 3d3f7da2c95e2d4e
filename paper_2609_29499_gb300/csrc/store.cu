// Shared INT8 store generation (synthetic weights + per-row quantization), synthetic KV
// caches, rotary tables and the panel gather kernels used by the packer.
#include <cuda_bf16.h>

#include <cmath>

#include "synth_dev.cuh"
#include "tasp_internal.h"

namespace tasp {

namespace {

constexpr int GQ_THREADS = 256;

// Row source of a store row: which generator stream and which dense row it comes from.
enum RowMode { RM_PLAIN = 0, RM_QKV = 1, RM_GU = 2 };

struct GenQuantArgs {
    int mode;
    uint64_t key0, key1, key2;  // plain: key0; qkv: q, k, v; gu: gate, up
    int rows, cols;
    int g, dh;                 // qkv row decoding
    int8_t* q;                 // [rows][cols]
    float* s;                  // [rows]
    int qg;                    // > 0: group scales of qg columns (s is then set to 1)
    uint16_t* gs;              // [rows][cols / qg] BF16, when qg > 0
};

__device__ __forceinline__ void row_source(const GenQuantArgs& a, int r, uint64_t& key, uint64_t& dense_row) {
    if (a.mode == RM_PLAIN) {
        key = a.key0;
        dense_row = (uint64_t)r;
    } else if (a.mode == RM_GU) {
        key = (r & 1) ? a.key1 : a.key0;
        dense_row = (uint64_t)(r >> 1);
    } else {
        int blk = (a.g + 2) * a.dh;
        int j = r / blk, w = r % blk, hh = w / a.dh, i = w % a.dh;
        if (hh < a.g) {
            key = a.key0;
            dense_row = (uint64_t)((j * a.g + hh) * a.dh + i);
        } else if (hh == a.g) {
            key = a.key1;
            dense_row = (uint64_t)(j * a.dh + i);
        } else {
            key = a.key2;
            dense_row = (uint64_t)(j * a.dh + i);
        }
    }
}

// One CTA per row: regenerate the dense FP32 row into shared memory, reduce max|w|,
// then s = a / 127 and q = clamp(rint(w / s), -127, 127) with IEEE division.
__global__ void __launch_bounds__(GQ_THREADS) gen_quant_kernel(GenQuantArgs a) {
    extern __shared__ float wrow[];
    __shared__ float red[GQ_THREADS / 32];
    int r = blockIdx.x;
    uint64_t key, drow;
    row_source(a, r, key, drow);
    const uint64_t base = drow * (uint64_t)a.cols;
    float m = 0.f;
    for (int j = threadIdx.x; j < a.cols; j += GQ_THREADS) {
        float w = __fmul_rn(sm_normal(key, base + (uint64_t)j), SM_WEIGHT_SIGMA);
        wrow[j] = w;
        m = fmaxf(m, fabsf(w));
    }
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    float amax = 0.f;
#pragma unroll
    for (int w = 0; w < GQ_THREADS / 32; ++w) amax = fmaxf(amax, red[w]);
    if (a.qg) {
        // groupwise (Table 1): per run of qg columns s_g = bf16(fl32(max|w| / 127)), then
        // q = clamp(rint(fl32(w / s_g)), -127, 127); the row scale is 1
        if (threadIdx.x == 0) a.s[r] = 1.0f;
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, ng = a.cols / a.qg;
        int8_t* qrow = a.q + (size_t)r * a.cols;
        for (int gi = warp; gi < ng; gi += GQ_THREADS / 32) {
            float gm = 0.f;
            for (int j = gi * a.qg + lane; j < (gi + 1) * a.qg; j += 32) gm = fmaxf(gm, fabsf(wrow[j]));
            for (int o = 16; o; o >>= 1) gm = fmaxf(gm, __shfl_xor_sync(0xffffffffu, gm, o));
            const __nv_bfloat16 sb = __float2bfloat16_rn(__fdiv_rn(gm, 127.0f));
            const float sg = __bfloat162float(sb);
            if (lane == 0) a.gs[(size_t)r * ng + gi] = *reinterpret_cast<const uint16_t*>(&sb);
            for (int j = gi * a.qg + lane; j < (gi + 1) * a.qg; j += 32) {
                int v = 0;
                if (sg != 0.f) {
                    v = __float2int_rn(__fdiv_rn(wrow[j], sg));
                    v = v > 127 ? 127 : (v < -127 ? -127 : v);
                }
                qrow[j] = (int8_t)v;
            }
        }
        return;
    }
    float s = (amax == 0.f) ? 0.f : __fdiv_rn(amax, 127.0f);
    if (threadIdx.x == 0) a.s[r] = s;
    int8_t* qrow = a.q + (size_t)r * a.cols;
    for (int j = threadIdx.x; j < a.cols; j += GQ_THREADS) {
        int v = 0;
        if (s != 0.f) {
            v = __float2int_rn(__fdiv_rn(wrow[j], s));
            v = v > 127 ? 127 : (v < -127 ? -127 : v);
        }
        qrow[j] = (int8_t)v;
    }
}

// gamma = fl32(1 + fl32(z * 0.02))
__global__ void gamma_kernel(uint64_t key, int n, float* out) {
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) out[i] = __fadd_rn(1.0f, __fmul_rn(sm_normal(key, (uint64_t)i), 0.02f));
}

// BF16 of fl32(z * sigma) for a flat range of n elements
__global__ void bf16_normal_kernel(uint64_t key, uint64_t n, float sigma, uint16_t* out) {
    uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
    uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
    for (; i < n; i += stride) out[i] = sm_bf16_bits(__fmul_rn(sm_normal(key, i), sigma));
}

// KV prior fill: cache[jl][p][i] for p < t_prior, from the stream of the original group.
__global__ void kv_fill_kernel(uint16_t* cache, const int* orig_group, uint64_t seed, int tensor, int layer,
                               int t_prior, int max_tokens, int dh) {
    int jl = blockIdx.y;
    uint64_t key = sm_key(seed, (uint64_t)tensor, (uint64_t)layer, (uint64_t)orig_group[jl]);
    uint64_t n = (uint64_t)t_prior * dh;
    uint16_t* dst = cache + (size_t)jl * max_tokens * dh;
    for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x)
        dst[i] = sm_bf16_bits(sm_normal(key, i));
}

// cos/sin of pos * theta^(-2i/dh), evaluated in double precision.
__global__ void rope_kernel(float2* out, int max_tokens, int half, int dh, double theta) {
    int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= max_tokens * half) return;
    int p = idx / half, i = idx % half;
    double inv = pow(theta, -2.0 * (double)i / (double)dh);
    double s, c;
    sincos((double)p * inv, &s, &c);
    out[idx] = make_float2((float)c, (float)s);
}

__global__ void gather_rows_kernel(int4* dst, const int4* src, const int32_t* map, int K16) {
    int r = blockIdx.x;
    const int4* s = src + (size_t)map[r] * K16;
    int4* d = dst + (size_t)r * K16;
    for (int j = threadIdx.x; j < K16; j += blockDim.x) d[j] = s[j];
}

__global__ void gather_cols_kernel(int8_t* dst, int ld_dst, const int8_t* src, int ld_src, const int32_t* cmap,
                                   int Kc) {
    int r = blockIdx.x;
    const int8_t* s = src + (size_t)r * ld_src;
    int8_t* d = dst + (size_t)r * ld_dst;
    for (int j = threadIdx.x; j < ld_dst; j += blockDim.x) d[j] = (j < Kc) ? s[cmap[j]] : (int8_t)0;
}

__global__ void gather_u16_rows_kernel(uint16_t* dst, int ld_dst, const uint16_t* src, const int32_t* map, int cols) {
    const int r = blockIdx.x;
    const uint16_t* s = src + (size_t)map[r] * cols;
    uint16_t* d = dst + (size_t)r * ld_dst;
    for (int j = threadIdx.x; j < cols; j += blockDim.x) d[j] = s[j];
}

__global__ void gather_u16_cols_kernel(uint16_t* dst, int ld_dst, const uint16_t* src, int ld_src, const int32_t* cmap,
                                       int ncols) {
    const int r = blockIdx.x;
    for (int j = threadIdx.x; j < ncols; j += blockDim.x) dst[(size_t)r * ld_dst + j] = src[(size_t)r * ld_src + cmap[j]];
}

__global__ void gather_f32_kernel(float* dst, const float* src, const int32_t* map, int n) {
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) dst[i] = src[map[i]];
}

int launch_gen_quant(const GenQuantArgs& a, cudaStream_t s) {
    size_t smem = (size_t)a.cols * sizeof(float);
    static bool attr_set = false;
    if (!attr_set) {
        TASP_CUDA(cudaFuncSetAttribute(gen_quant_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
        attr_set = true;
    }
    if (smem > 200 * 1024) return fail(TASP_EINVAL, "row too long for the store generator");
    gen_quant_kernel<<<a.rows, GQ_THREADS, smem, s>>>(a);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

}  // namespace

int store_generate(Store& st, cudaStream_t s) {
    const Shape& sh = st.sh;
    for (int l = 0; l < sh.L; ++l) {
        LayerStore& ls = st.layers[l];
        GenQuantArgs a{};
        a.mode = RM_QKV;
        a.key0 = sm_key(sh.seed, ST_WQ, l, 0);
        a.key1 = sm_key(sh.seed, ST_WK, l, 0);
        a.key2 = sm_key(sh.seed, ST_WV, l, 0);
        a.rows = sh.qkv_rows_dense();
        a.cols = sh.d;
        a.g = sh.g();
        a.dh = sh.dh;
        a.q = ls.qkv;
        a.s = ls.qkv_s;
        a.qg = sh.qg;
        a.gs = ls.qkv_g;
        int rc = launch_gen_quant(a, s);
        if (rc) return rc;
        a = GenQuantArgs{};
        a.mode = RM_PLAIN;
        a.key0 = sm_key(sh.seed, ST_WO, l, 0);
        a.rows = sh.d;
        a.cols = sh.Hq * sh.dh;
        a.q = ls.o;
        a.s = ls.o_s;
        a.qg = sh.qg;
        a.gs = ls.o_g;
        if ((rc = launch_gen_quant(a, s))) return rc;
        a = GenQuantArgs{};
        a.mode = RM_GU;
        a.key0 = sm_key(sh.seed, ST_WGATE, l, 0);
        a.key1 = sm_key(sh.seed, ST_WUP, l, 0);
        a.rows = 2 * sh.df;
        a.cols = sh.d;
        a.q = ls.gu;
        a.s = ls.gu_s;
        a.qg = sh.qg;
        a.gs = ls.gu_g;
        if ((rc = launch_gen_quant(a, s))) return rc;
        a = GenQuantArgs{};
        a.mode = RM_PLAIN;
        a.key0 = sm_key(sh.seed, ST_WDOWN, l, 0);
        a.rows = sh.d;
        a.cols = sh.df;
        a.q = ls.down;
        a.s = ls.down_s;
        a.qg = sh.qg;
        a.gs = ls.down_g;
        if ((rc = launch_gen_quant(a, s))) return rc;
        int nb = (sh.d + 255) / 256;
        gamma_kernel<<<nb, 256, 0, s>>>(sm_key(sh.seed, ST_GAMMA_ATTN, l, 0), sh.d, ls.g_attn);
        gamma_kernel<<<nb, 256, 0, s>>>(sm_key(sh.seed, ST_GAMMA_MLP, l, 0), sh.d, ls.g_mlp);
        TASP_CUDA(cudaGetLastError());
    }
    gamma_kernel<<<(sh.d + 255) / 256, 256, 0, s>>>(sm_key(sh.seed, ST_GAMMA_FINAL, 0, 0), sh.d, st.g_final);
    if (sh.vocab > 0)
        bf16_normal_kernel<<<4096, 256, 0, s>>>(sm_key(sh.seed, ST_LMHEAD, 0, 0), (uint64_t)sh.vocab * sh.d,
                                                SM_WEIGHT_SIGMA, st.lm_head);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

int kv_fill_synthetic(Session& se, int t_prior, uint64_t kv_seed, cudaStream_t s) {
    const Plan& p = *se.plan;
    const Shape& sh = p.store->sh;
    int* d_groups = nullptr;
    // kept-group ids per layer, staged through a small device buffer
    int maxg = sh.Hkv;
    TASP_CUDA(cudaMallocAsync((void**)&d_groups, sizeof(int) * maxg * sh.L, s));
    std::vector<int> hg((size_t)maxg * sh.L, 0);
    for (int l = 0; l < sh.L; ++l)
        for (int j = 0; j < p.layers[l].m_kv; ++j) hg[(size_t)l * maxg + j] = p.layers[l].keep_groups[j];
    TASP_CUDA(cudaMemcpyAsync(d_groups, hg.data(), sizeof(int) * hg.size(), cudaMemcpyHostToDevice, s));
    for (int l = 0; l < sh.L; ++l) {
        int m = p.layers[l].m_kv;
        if (m == 0 || t_prior == 0) continue;
        dim3 grid(64, m);
        kv_fill_kernel<<<grid, 256, 0, s>>>(se.K[l], d_groups + (size_t)l * maxg, kv_seed, ST_KCACHE, l, t_prior,
                                            se.max_tokens, sh.dh);
        kv_fill_kernel<<<grid, 256, 0, s>>>(se.V[l], d_groups + (size_t)l * maxg, kv_seed, ST_VCACHE, l, t_prior,
                                            se.max_tokens, sh.dh);
    }
    TASP_CUDA(cudaGetLastError());
    TASP_CUDA(cudaMemcpyAsync(se.d_pos, &t_prior, sizeof(int), cudaMemcpyHostToDevice, s));
    TASP_CUDA(cudaStreamSynchronize(s));  // host t_prior goes out of scope
    TASP_CUDA(cudaFreeAsync(d_groups, s));
    return TASP_OK;
}

int rope_table(Session& se, cudaStream_t s) {
    const Shape& sh = se.plan->store->sh;
    int half = sh.dh / 2;
    int n = se.max_tokens * half;
    rope_kernel<<<(n + 255) / 256, 256, 0, s>>>(se.rope, se.max_tokens, half, sh.dh, (double)sh.theta);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

int gather_rows(int8_t* dst, const int8_t* src, const int32_t* map, int rows, int K, cudaStream_t s) {
    if (rows == 0) return TASP_OK;
    if (K % 16) return fail(TASP_EINVAL, "gather_rows: K not a multiple of 16");
    gather_rows_kernel<<<rows, 256, 0, s>>>((int4*)dst, (const int4*)src, map, K / 16);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

int gather_cols(int8_t* dst, int ld_dst, const int8_t* src, int ld_src, const int32_t* cmap, int rows, int Kc,
                cudaStream_t s) {
    if (rows == 0) return TASP_OK;
    gather_cols_kernel<<<rows, 256, 0, s>>>(dst, ld_dst, src, ld_src, cmap, Kc);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

int gather_u16_rows(uint16_t* dst, int ld_dst, const uint16_t* src, const int32_t* map, int rows, int cols,
                    cudaStream_t s) {
    if (rows == 0 || cols == 0) return TASP_OK;
    gather_u16_rows_kernel<<<rows, 128, 0, s>>>(dst, ld_dst, src, map, cols);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

int gather_u16_cols(uint16_t* dst, int ld_dst, const uint16_t* src, int ld_src, const int32_t* cmap, int rows,
                    int ncols, cudaStream_t s) {
    if (rows == 0 || ncols == 0) return TASP_OK;
    gather_u16_cols_kernel<<<rows, 128, 0, s>>>(dst, ld_dst, src, ld_src, cmap, ncols);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

int gather_f32(float* dst, const float* src, const int32_t* map, int n, cudaStream_t s) {
    if (n == 0) return TASP_OK;
    gather_f32_kernel<<<(n + 255) / 256, 256, 0, s>>>(dst, src, map, n);
    TASP_CUDA(cudaGetLastError());
    return TASP_OK;
}

}  // namespace tasp
