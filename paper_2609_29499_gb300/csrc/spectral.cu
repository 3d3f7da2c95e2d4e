// Spectral descriptors of the candidate units on the device (Sec. 3.1 "Candidate Units and
// Spectral Features", Eqs. 1-4; Appendix "Exact candidate feature construction").
//
// A candidate's block W (n_r x d, n_r <= d) stacks its pieces of the layer: an attention head h
// its own Q rows, the O columns it feeds (transposed) and its KV group's K and V rows
// ([4 d_h, d]); a channel group its gate rows, up rows and down columns (transposed)
// ([3 chan_unit, d]). The eigenvalues of the normalized Gram matrix, lambda_i = s_i^2 / d, give:
//  * alpha: the maximum-likelihood Pareto exponent of the eigenvalues >= lambda_min,
//    m / sum log(lambda_i / lambda_min), with lambda_min the value among the distinct
//    eigenvalues below the largest that minimizes the Kolmogorov-Smirnov distance between the
//    tail and P(x) = 1 - (x / lambda_min)^-alpha (ties to the smaller lambda_min);
//  * SETOL: the share of the spectrum's mass in that tail;
//  * the effective rank exp(-sum p_i log p_i), p_i = lambda_i / sum_j lambda_j;
//  * the spectral norm s_1 = sqrt(lambda_1 d).
//
// Steps per candidate, all on one stream:
//  1. spec_block_kernel writes the block from the model's counter-based generator, each weight
//     rounded to BF16 (the checkpoint precision the paper reads) and widened to FP16 (exact for
//     every BF16 value in FP16's normal range; the ~0.02% of weights below 2^-14 in magnitude
//     keep 11 bits as FP16 subnormals);
//  2. the Gram matrix B B^T on the tensor cores: the prefill's persistent tcgen05 GEMM (TMA-fed,
//     FP32 accumulation in tensor memory), FP16 products exact;
//  3. the eigenvalues of the symmetric Gram matrix: cuSOLVER's symmetric eigensolver (syevd,
//     no vectors), loaded at run time, as a library step like a matmul;
//  4. spec_stats_kernel: the statistics above in FP64, one CTA per candidate (suffix sums of log
//     lambda give each alpha in O(1); the KS scan is O(n) per candidate lambda_min).
#include <cuda_fp16.h>
#include <cusolverDn.h>
#include <dlfcn.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include "synth_dev.cuh"
#include "tasp_internal.h"

namespace tasp {

namespace {

constexpr int SPEC_FEATURES = 6;  // alpha, r_eff, spectral norm, SETOL, lambda_min, KS distance

struct SpecBlockArgs {
    __half* out;   // [rows][d]
    int rows, d;
    int kind;      // 0: attention head, 1: channel group
    int unit;      // head index or channel-group index
    int dh, g, Hq, df, cu;
    uint64_t k0, k1, k2, k3;  // head: Q, O, K, V keys; channel group: gate, up, down keys
};

__global__ void spec_block_kernel(SpecBlockArgs a) {
    const int r = blockIdx.y;
    for (int col = blockIdx.x * blockDim.x + threadIdx.x; col < a.d; col += gridDim.x * blockDim.x) {
        uint64_t key, idx;
        if (a.kind == 0) {
            const int h = a.unit, j = h / a.g, piece = r / a.dh, i = r - piece * a.dh;
            if (piece == 0) {  // Q row h dh + i
                key = a.k0;
                idx = (uint64_t)(h * a.dh + i) * a.d + col;
            } else if (piece == 1) {  // O column h dh + i of the [d][Hq dh] matrix, as a row
                key = a.k1;
                idx = (uint64_t)col * (uint64_t)(a.Hq * a.dh) + (uint64_t)(h * a.dh + i);
            } else {  // K or V row j dh + i
                key = piece == 2 ? a.k2 : a.k3;
                idx = (uint64_t)(j * a.dh + i) * a.d + col;
            }
        } else {
            const int piece = r / a.cu, i = r - piece * a.cu, c = a.unit * a.cu + i;
            if (piece < 2) {  // gate / up row c
                key = piece == 0 ? a.k0 : a.k1;
                idx = (uint64_t)c * a.d + col;
            } else {  // down column c of the [d][df] matrix, as a row
                key = a.k2;
                idx = (uint64_t)col * (uint64_t)a.df + (uint64_t)c;
            }
        }
        const float w = __fmul_rn(sm_normal(key, idx), SM_WEIGHT_SIGMA);
        const __nv_bfloat16 b = __float2bfloat16_rn(w);
        a.out[(size_t)r * a.d + col] = __float2half_rn(__bfloat162float(b));
    }
}

// Block-wide reduction helpers (256 threads).
constexpr int ST_THREADS = 256;
__device__ double block_sum(double v, double* red) {
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    double t = 0.0;
    for (int w = 0; w < ST_THREADS / 32; ++w) t += red[w];
    return t;
}

// KS distance of the tail lam[k..n-1] against P(x) = 1 - (x / lam[k])^-alpha (T = float: the
// scan; T = double: the final comparison). lg holds log lambda, suf its suffix sums.
template <typename T>
__device__ __forceinline__ T ks_at(const double* lg, const double* suf, int n, int k) {
    const int m = n - k;
    const double lx = lg[k];
    const T alpha = (T)((double)m / (suf[k] - (double)m * lx));
    T D = 0;
    for (int i = 0; i < m; ++i) {
        const T P = (T)1 - exp(-alpha * (T)(lg[k + i] - lx));
        const T hi = (T)(i + 1) / (T)m, lo = (T)i / (T)m;
        D = fmax(D, fmax(hi - P, P - lo));
    }
    return D;
}

// One CTA per candidate (blockIdx.x). w: eigenvalues of each candidate's Gram matrix ascending
// (FP32, row stride w_ld, n_head for the first n_heads candidates, else n_chan); lam_out
// (optional) receives lambda_i = w_i / d descending, candidates back to back; feat the six
// features. The KS scan runs in FP32 over every candidate lambda_min; the ones within
// KS_MARGIN of the FP32 minimum (FP32 rounding moves a distance by ~1e-6) are evaluated again
// in FP64 and the FP64 minimum taken (ties to the smaller lambda_min).
constexpr float KS_MARGIN = 1e-4f;
__global__ void __launch_bounds__(ST_THREADS) spec_stats_kernel(const float* w, int w_ld, int n_heads, int n_head,
                                                               int n_chan, int d, double* lam_out, double* feat) {
    extern __shared__ double sh[];
    const int cand = blockIdx.x;
    const bool head = cand < n_heads;
    const int n = head ? n_head : n_chan;
    const float* wc = w + (size_t)cand * w_ld;
    double* lo_out = lam_out ? lam_out + (head ? (size_t)cand * n_head
                                               : (size_t)n_heads * n_head + (size_t)(cand - n_heads) * n_chan)
                             : nullptr;
    double* fo = feat + (size_t)cand * SPEC_FEATURES;
    double* lam = sh;       // [n] ascending, lambda_i = max(w_i, 0) / d
    double* lg = sh + n;    // [n] log lambda_i (0 for lambda_i = 0)
    double* suf = lg + n;   // [n + 1] suffix sums of log lambda
    float* d32 = reinterpret_cast<float*>(suf + n + 1);  // [n] FP32 KS distance per candidate cut
    __shared__ double red[ST_THREADS / 32];
    __shared__ double bestD[ST_THREADS];
    __shared__ int bestK[ST_THREADS];
    __shared__ float fmin_s;
    const int tid = threadIdx.x;
    for (int i = tid; i < n; i += ST_THREADS) {
        const double v = fmax((double)wc[i], 0.0) / (double)d;
        lam[i] = v;
        lg[i] = v > 0.0 ? log(v) : 0.0;
        if (lo_out) lo_out[n - 1 - i] = v;
    }
    __syncthreads();
    if (tid == 0) {
        double acc = 0.0;
        suf[n] = 0.0;
        for (int i = n - 1; i >= 0; --i) {
            acc += lg[i];
            suf[i] = acc;
        }
    }
    double ls = 0.0;
    for (int i = tid; i < n; i += ST_THREADS) ls += lam[i];
    const double total = block_sum(ls, red);  // (its barriers also publish suf)
    double ent = 0.0;
    for (int i = tid; i < n; i += ST_THREADS)
        if (lam[i] > 0.0) {
            const double p = lam[i] / total;
            ent -= p * log(p);
        }
    ent = block_sum(ent, red);
    // candidate cut k: lambda_min = lam[k], the first index of a distinct positive value below the largest
    const double lmax = lam[n - 1];
    auto is_cut = [&](int k) { return lam[k] > 0.0 && lam[k] < lmax && !(k > 0 && lam[k - 1] == lam[k]); };
    float fmin = INFINITY;
    for (int k = tid; k < n; k += ST_THREADS) {
        const float D = is_cut(k) ? ks_at<float>(lg, suf, n, k) : INFINITY;
        d32[k] = D;
        fmin = fminf(fmin, D);
    }
    for (int o = 16; o; o >>= 1) fmin = fminf(fmin, __shfl_xor_sync(0xffffffffu, fmin, o));
    if ((tid & 31) == 0) red[tid >> 5] = fmin;
    __syncthreads();
    if (tid == 0) {
        float m = INFINITY;
        for (int w2 = 0; w2 < ST_THREADS / 32; ++w2) m = fminf(m, (float)red[w2]);
        fmin_s = m;
    }
    __syncthreads();
    double bD = INFINITY;
    int bK = n;
    for (int k = tid; k < n; k += ST_THREADS) {
        if (!(d32[k] <= fmin_s + KS_MARGIN)) continue;
        const double D = ks_at<double>(lg, suf, n, k);
        if (D < bD) {  // k ascends within a thread: the first (smallest) minimum stays
            bD = D;
            bK = k;
        }
    }
    bestD[tid] = bD;
    bestK[tid] = bK;
    __syncthreads();
    if (tid == 0) {
        double D = INFINITY;
        int k = n;
        for (int t = 0; t < ST_THREADS; ++t)
            if (bestD[t] < D || (bestD[t] == D && bestK[t] < k)) {
                D = bestD[t];
                k = bestK[t];
            }
        double mass = 0.0;
        for (int i = k; i < n; ++i) mass += lam[i];
        const int m = n - k;
        const double x = k < n ? lam[k] : 0.0;
        fo[0] = k < n ? (double)m / (suf[k] - (double)m * log(x)) : 0.0;
        fo[1] = exp(ent);
        fo[2] = sqrt(lmax * (double)d);
        fo[3] = k < n ? mass / total : 0.0;
        fo[4] = x;
        fo[5] = k < n ? D : 0.0;
    }
}

// cuSOLVER's dense symmetric eigensolver, resolved at run time so that the library does not
// depend on it for anything else.
struct Solver {
    decltype(&cusolverDnCreate) create = nullptr;
    decltype(&cusolverDnDestroy) destroy = nullptr;
    decltype(&cusolverDnSetStream) set_stream = nullptr;
    decltype(&cusolverDnSsyevd_bufferSize) buffer_size = nullptr;
    decltype(&cusolverDnSsyevd) syevd = nullptr;
    bool ok = false;
};

std::mutex g_solver_mu;

int solver(Solver** out) {
    static Solver s;
    static bool tried = false;
    std::lock_guard<std::mutex> lk(g_solver_mu);
    if (!tried) {
        tried = true;
        const char* names[] = {"libcusolver.so", "libcusolver.so.12", "libcusolver.so.11",
                               "/usr/local/cuda/lib64/libcusolver.so"};
        void* h = nullptr;
        for (const char* nm : names)
            if ((h = dlopen(nm, RTLD_NOW | RTLD_LOCAL))) break;
        if (h) {
            s.create = (decltype(s.create))dlsym(h, "cusolverDnCreate");
            s.destroy = (decltype(s.destroy))dlsym(h, "cusolverDnDestroy");
            s.set_stream = (decltype(s.set_stream))dlsym(h, "cusolverDnSetStream");
            s.buffer_size = (decltype(s.buffer_size))dlsym(h, "cusolverDnSsyevd_bufferSize");
            s.syevd = (decltype(s.syevd))dlsym(h, "cusolverDnSsyevd");
            s.ok = s.create && s.destroy && s.set_stream && s.buffer_size && s.syevd;
        }
    }
    if (!s.ok) return fail(TASP_EUNSUP, "the symmetric eigensolver (cuSOLVER) could not be loaded");
    *out = &s;
    return TASP_OK;
}

}  // namespace

}  // namespace tasp

using namespace tasp;

extern "C" int tasp_spectral_layer(const tasp_model_desc* model, int32_t layer, double* h_features,
                                   double* h_lambda, double* h_phase_ms, void* stream) {
    Shape sh;
    int rc = validate_shape(model, sh, false);
    if (rc) return rc;
    if (!h_features) return fail(TASP_EINVAL, "h_features is NULL");
    if (layer < 0 || layer >= sh.L) return fail(TASP_EINVAL, "layer out of range");
    const int nh = 4 * sh.dh, nc = 3 * sh.cu;
    if (nh > sh.d || nc > sh.d)
        return fail(TASP_EUNSUP, "candidate blocks taller than the model width (4 dh and 3 chan_unit must be <= d)");
    if (sh.d % 64) return fail(TASP_EUNSUP, "the Gram GEMM needs d to be a multiple of 64");
    Solver* sv = nullptr;
    if ((rc = solver(&sv))) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    const int nunits = sh.df / sh.cu, ncand = sh.Hq + nunits;
    const int nmax = std::max(nh, nc);
    // Candidates go round-robin to NW worker streams, each with its own block, Gram matrix,
    // eigensolver handle and workspace, so that several eigensolves run at once; the statistics
    // of all candidates then run as one launch on the caller's stream. Device temporaries come
    // from the stream-ordered pool and are freed before return.
    constexpr int NW = 8;
    struct Worker {
        cudaStream_t st = nullptr;
        cusolverDnHandle_t hs = nullptr;
        __half* blk = nullptr;
        float *G = nullptr, *work = nullptr;
        cudaEvent_t ev[4] = {};
    } wk[NW];
    float *W = nullptr, *ones = nullptr;
    double *feat = nullptr, *lam = nullptr;
    int* info = nullptr;
    cudaEvent_t e_start = nullptr, e_done = nullptr, e_stats = nullptr;
    int lwork = 0;
    const bool timing = h_phase_ms != nullptr;
    auto cleanup = [&]() {
        cudaStreamSynchronize(s);
        for (Worker& w : wk) {
            if (w.st) cudaStreamSynchronize(w.st);
            if (w.hs) sv->destroy(w.hs);
            for (void* p : {(void*)w.blk, (void*)w.G, (void*)w.work})
                if (p) cudaFree(p);
            for (auto& e : w.ev)
                if (e) cudaEventDestroy(e);
            if (w.st) cudaStreamDestroy(w.st);
            w = Worker{};
        }
        for (void* p : {(void*)W, (void*)ones, (void*)feat, (void*)lam, (void*)info})
            if (p) cudaFree(p);
        W = ones = nullptr;
        feat = lam = nullptr;
        info = nullptr;
        for (cudaEvent_t* e : {&e_start, &e_done, &e_stats})
            if (*e) {
                cudaEventDestroy(*e);
                *e = nullptr;
            }
    };
    auto cu = [&](cudaError_t e, const char* what) -> int {
        if (e == cudaSuccess) return TASP_OK;
        cleanup();
        return cuda_fail(e, what);
    };
    const size_t nlam = (size_t)sh.Hq * nh + (size_t)nunits * nc;
    if ((rc = cu(cudaMalloc((void**)&W, (size_t)ncand * nmax * sizeof(float)), "spectral eigenvalues"))) return rc;
    if ((rc = cu(cudaMalloc((void**)&ones, (size_t)nmax * sizeof(float)), "spectral scales"))) return rc;
    if ((rc = cu(cudaMalloc((void**)&feat, (size_t)ncand * SPEC_FEATURES * sizeof(double)), "spectral features")))
        return rc;
    if ((rc = cu(cudaMalloc((void**)&lam, nlam * sizeof(double)), "spectral lambdas"))) return rc;
    if ((rc = cu(cudaMalloc((void**)&info, (size_t)ncand * sizeof(int)), "spectral info"))) return rc;
    {
        std::vector<float> h1(nmax, 1.0f);
        if ((rc = cu(cudaMemcpy(ones, h1.data(), nmax * sizeof(float), cudaMemcpyHostToDevice), "spectral scales")))
            return rc;
    }
    for (cudaEvent_t* e : {&e_start, &e_done, &e_stats})
        if ((rc = cu(cudaEventCreate(e), "spectral events"))) return rc;
    for (Worker& w : wk) {
        if ((rc = cu(cudaStreamCreateWithFlags(&w.st, cudaStreamNonBlocking), "spectral worker stream"))) return rc;
        if ((rc = cu(cudaMalloc((void**)&w.blk, (size_t)nmax * sh.d * sizeof(__half)), "spectral block"))) return rc;
        if ((rc = cu(cudaMalloc((void**)&w.G, (size_t)nmax * nmax * sizeof(float)), "spectral Gram"))) return rc;
        if (timing)
            for (auto& e : w.ev)
                if ((rc = cu(cudaEventCreate(&e), "spectral timing events"))) return rc;
        if (sv->create(&w.hs) != CUSOLVER_STATUS_SUCCESS) {
            w.hs = nullptr;
            cleanup();
            return fail(TASP_ECUDA, "cusolverDnCreate failed");
        }
        sv->set_stream(w.hs, w.st);
        if (!lwork) {
            int l1 = 0, l2 = 0;
            if (sv->buffer_size(w.hs, CUSOLVER_EIG_MODE_NOVECTOR, CUBLAS_FILL_MODE_LOWER, nh, w.G, nh, W, &l1) !=
                    CUSOLVER_STATUS_SUCCESS ||
                sv->buffer_size(w.hs, CUSOLVER_EIG_MODE_NOVECTOR, CUBLAS_FILL_MODE_LOWER, nc, w.G, nc, W, &l2) !=
                    CUSOLVER_STATUS_SUCCESS) {
                cleanup();
                return fail(TASP_ECUDA, "cusolverDnSsyevd_bufferSize failed");
            }
            lwork = std::max(1, std::max(l1, l2));
        }
        if ((rc = cu(cudaMalloc((void**)&w.work, (size_t)lwork * sizeof(float)), "spectral solver work"))) return rc;
    }
    const size_t st_smem_max = (size_t)(3 * nmax + 1) * sizeof(double) + (size_t)nmax * sizeof(float);
    if ((rc = cu(cudaFuncSetAttribute(spec_stats_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)st_smem_max),
                 "spectral statistics attributes")))
        return rc;
    if ((rc = cu(cudaEventRecord(e_start, s), "spectral start"))) return rc;
    for (Worker& w : wk)
        if ((rc = cu(cudaStreamWaitEvent(w.st, e_start, 0), "spectral start"))) return rc;
    // One host thread per worker: the eigensolver has host-side steps, so one issuing thread
    // would serialize the workers.
    double wphase[NW][3] = {};
    int wrc[NW] = {};
    std::string werr[NW];
    auto run_worker = [&](int wi) {
        Worker& w = wk[wi];
        for (int cidx = wi; cidx < ncand; cidx += NW) {
            const bool head = cidx < sh.Hq;
            const int n = head ? nh : nc;
            SpecBlockArgs a{};
            a.out = w.blk;
            a.rows = n;
            a.d = sh.d;
            a.kind = head ? 0 : 1;
            a.unit = head ? cidx : cidx - sh.Hq;
            a.dh = sh.dh;
            a.g = sh.g();
            a.Hq = sh.Hq;
            a.df = sh.df;
            a.cu = sh.cu;
            if (head) {
                a.k0 = sm_key(sh.seed, ST_WQ, layer, 0);
                a.k1 = sm_key(sh.seed, ST_WO, layer, 0);
                a.k2 = sm_key(sh.seed, ST_WK, layer, 0);
                a.k3 = sm_key(sh.seed, ST_WV, layer, 0);
            } else {
                a.k0 = sm_key(sh.seed, ST_WGATE, layer, 0);
                a.k1 = sm_key(sh.seed, ST_WUP, layer, 0);
                a.k2 = sm_key(sh.seed, ST_WDOWN, layer, 0);
            }
            if (timing) cudaEventRecord(w.ev[0], w.st);
            spec_block_kernel<<<dim3((sh.d + 255) / 256, n), 256, 0, w.st>>>(a);
            cudaError_t e = cudaGetLastError();
            if (e != cudaSuccess) {
                wrc[wi] = cuda_fail(e, "spectral block kernel");
                werr[wi] = tasp_last_error();
                return;
            }
            if (timing) cudaEventRecord(w.ev[1], w.st);
            if (int r = gemm_f16_nt(w.blk, sh.d, n, w.blk, sh.d, n, sh.d, ones, w.G, n, nullptr, w.st)) {
                wrc[wi] = r;
                werr[wi] = tasp_last_error();
                return;
            }
            if (timing) cudaEventRecord(w.ev[2], w.st);
            if (sv->syevd(w.hs, CUSOLVER_EIG_MODE_NOVECTOR, CUBLAS_FILL_MODE_LOWER, n, w.G, n, W + (size_t)cidx * nmax,
                          w.work, lwork, info + cidx) != CUSOLVER_STATUS_SUCCESS) {
                wrc[wi] = fail(TASP_ECUDA, "cusolverDnSsyevd failed");
                werr[wi] = tasp_last_error();
                return;
            }
            if (timing) {
                cudaEventRecord(w.ev[3], w.st);
                cudaEventSynchronize(w.ev[3]);
                for (int i = 0; i < 3; ++i) {
                    float ms = 0.f;
                    cudaEventElapsedTime(&ms, w.ev[i], w.ev[i + 1]);
                    wphase[wi][i] += ms;
                }
            }
        }
    };
    {
        int dev = 0;
        cudaGetDevice(&dev);
        std::vector<std::thread> th;
        for (int wi = 0; wi < NW; ++wi)
            th.emplace_back([&, wi, dev]() {
                cudaSetDevice(dev);
                run_worker(wi);
            });
        for (auto& t : th) t.join();
    }
    for (int wi = 0; wi < NW; ++wi)
        if (wrc[wi]) {
            cleanup();
            return fail(wrc[wi], werr[wi]);
        }
    double phase[4] = {0, 0, 0, 0};
    for (int wi = 0; wi < NW; ++wi)
        for (int i = 0; i < 3; ++i) phase[i] += wphase[wi][i];
    for (Worker& w : wk) {  // the caller's stream waits for every worker
        if ((rc = cu(cudaEventRecord(w.ev[0] ? w.ev[0] : e_done, w.st), "spectral join"))) return rc;
        if ((rc = cu(cudaStreamWaitEvent(s, w.ev[0] ? w.ev[0] : e_done, 0), "spectral join"))) return rc;
    }
    if ((rc = cu(cudaEventRecord(e_done, s), "spectral join"))) return rc;
    spec_stats_kernel<<<ncand, ST_THREADS, st_smem_max, s>>>(W, nmax, sh.Hq, nh, nc, sh.d, lam, feat);
    if ((rc = cu(cudaGetLastError(), "spectral statistics kernel"))) return rc;
    if ((rc = cu(cudaEventRecord(e_stats, s), "spectral statistics"))) return rc;
    std::vector<int> hinfo(ncand, 0);
    if ((rc = cu(cudaMemcpyAsync(hinfo.data(), info, (size_t)ncand * sizeof(int), cudaMemcpyDeviceToHost, s),
                 "spectral info")))
        return rc;
    if ((rc = cu(cudaMemcpyAsync(h_features, feat, (size_t)ncand * SPEC_FEATURES * sizeof(double),
                                 cudaMemcpyDeviceToHost, s),
                 "spectral features copy")))
        return rc;
    if (h_lambda &&
        (rc = cu(cudaMemcpyAsync(h_lambda, lam, nlam * sizeof(double), cudaMemcpyDeviceToHost, s), "spectral lambda copy")))
        return rc;
    if ((rc = cu(cudaStreamSynchronize(s), "spectral copies"))) return rc;
    for (int c = 0; c < ncand; ++c)
        if (hinfo[c] != 0) {
            cleanup();
            return fail(TASP_ECUDA, "the eigensolver did not converge (candidate " + std::to_string(c) + ", info " +
                                        std::to_string(hinfo[c]) + ")");
        }
    if (timing) {
        float ms = 0.f;
        cudaEventElapsedTime(&ms, e_done, e_stats);
        phase[3] = ms;
        for (int i = 0; i < 4; ++i) h_phase_ms[i] = phase[i];
    }
    cleanup();
    return TASP_OK;
}
