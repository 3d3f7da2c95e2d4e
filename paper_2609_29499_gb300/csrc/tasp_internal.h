// Internal structures of the TASP runtime: shared store, plans, sessions, kernel parameters.
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <initializer_list>
#include <string>
#include <vector>

#include "../../include/tasp.h"

namespace tasp {

// ---------------------------------------------------------------- errors
void set_error(const std::string& msg);
int fail(int code, const std::string& msg);

// Caller buffers are accessed element by element: each must be aligned to its element size
// (2 bytes for BF16, 4 for FP32). NULL passes (optional buffers are checked elsewhere).
struct BufAlign {
    const void* p;
    unsigned bytes;
};
inline int check_aligned(std::initializer_list<BufAlign> bufs) {
    for (const BufAlign& b : bufs)
        if (b.p && (reinterpret_cast<uintptr_t>(b.p) % b.bytes))
            return fail(TASP_EINVAL, "a buffer is not aligned to its element size (" + std::to_string(b.bytes) +
                                         " bytes)");
    return TASP_OK;
}
int cuda_fail(cudaError_t e, const char* what);

#define TASP_CUDA(call)                                   \
    do {                                                  \
        cudaError_t e_ = (call);                          \
        if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
    } while (0)

// ---------------------------------------------------------------- shape
struct Shape {
    int L = 0, d = 0, Hq = 0, Hkv = 0, dh = 0, df = 0, vocab = 0, cu = 1;
    int qg = 0;  // scale group (input columns per BF16 scale), 0 = one FP32 scale per row
    float eps = 1e-5f, theta = 500000.f;
    uint64_t seed = 0;
    int g() const { return Hq / Hkv; }
    int n_units() const { return df / cu; }
    int qkv_rows_dense() const { return (Hq + 2 * Hkv) * dh; }
    bool same(const Shape& o) const;
};

// Active-FLOP ledger (Appendix, Eqs. flop-attn and flop-mlp).
int64_t layer_flops(const Shape& s, int64_t m_q, int64_t m_kv, int64_t c);
inline int64_t dense_layer_flops(const Shape& s) { return layer_flops(s, s.Hq, s.Hkv, s.df); }

// Host mask compiler result: per layer kept groups (KV heads), query heads and channel
// units (ascending). For the group-granular kinds `qheads` holds every head of each kept group.
struct MaskSel {
    std::vector<std::vector<int>> groups, qheads, units;
    std::vector<int64_t> layer_flops;
    int64_t total = 0, budget = 0, dense = 0;
};
int select_mask(const Shape& s, const tasp_mask_desc& m, MaskSel& out);

// ---------------------------------------------------------------- device memory arena
struct Arena {
    char* base = nullptr;
    size_t cap = 0, used = 0;
    int reserve(size_t bytes);  // cudaMalloc of the whole arena
    void* take(size_t bytes);   // 256-byte aligned sub-allocation
    void release();
};

// ---------------------------------------------------------------- shared store
// Each projection once, INT8 with one FP32 scale per output row; QKV rows group-major
// (per KV group: its g query heads, then K, then V) and gate/up rows interleaved per
// channel, i.e. the packed layout of the all-keep mask.
struct LayerStore {
    int8_t *qkv, *o, *gu, *down;
    float *qkv_s, *o_s, *gu_s, *down_s, *g_attn, *g_mlp;  // row scales (all 1 in a grouped store)
    // grouped store only: BF16 scales [rows][K / qg] of each projection
    uint16_t *qkv_g = nullptr, *o_g = nullptr, *gu_g = nullptr, *down_g = nullptr;
};

struct Store {
    Shape sh;
    int refs = 0;
    Arena arena;
    std::vector<LayerStore> layers;
    float* g_final = nullptr;
    uint16_t* lm_head = nullptr;  // BF16 [vocab][d]
    size_t bytes = 0;
};

// ---------------------------------------------------------------- plans
struct LayerPlan {
    int m_kv = 0, c = 0;
    int m_q = 0;  // kept query heads (m_kv g unless the mask keeps part of a group)
    std::vector<int> keep_groups, keep_chans, keep_qheads;
    // Partial groups only (NULL when every kept group keeps its g heads):
    // blk_role[b] = role of the qkv panel's d_h-row block b as jl (g + 2) + hh, with jl the
    // kept-group slot and hh the head within the group (< g), g for K or g + 1 for V;
    // oslot[jl g + hh] = the compact position of that head in the O panel's columns, or -1
    // for a dropped head (its query slot stays zero and its attention output is not written).
    const int16_t* blk_role = nullptr;
    const int16_t* oslot = nullptr;
    const int16_t* blk_of = nullptr;  // inverse of blk_role: [m_kv (g + 2)] panel block or -1
    // qkv panel: rows (m_q + 2 m_kv) dh of K = d; row i at qkv_w + (qkv_map ? qkv_map[i] : i) * d
    const int8_t* qkv_w = nullptr;
    const int32_t* qkv_map = nullptr;
    const float* qkv_s = nullptr;
    int qkv_rows = 0;
    // o panel: d rows of K = m_q dh (stride o_ld >= K, multiple of 16, zero padded)
    const int8_t* o_w = nullptr;
    const float* o_s = nullptr;
    int o_K = 0, o_ld = 0;
    // gate/up panel: 2c rows of K = d
    const int8_t* gu_w = nullptr;
    const int32_t* gu_map = nullptr;
    const float* gu_s = nullptr;
    int gu_rows = 0;
    // down panel: d rows of K = c (stride dn_ld)
    const int8_t* dn_w = nullptr;
    const float* dn_s = nullptr;
    int dn_K = 0, dn_ld = 0;
    const float *g_attn = nullptr, *g_mlp = nullptr;
    // grouped store only: BF16 group scales in panel order, [rows][K / qg] (row stride gq_ld
    // for qkv / gu, o_K / qg and dn_K / qg for the column-compacted O / down panels)
    const uint16_t *qkv_g = nullptr, *gu_g = nullptr, *o_g = nullptr, *dn_g = nullptr;
    int qkv_gld = 0, gu_gld = 0, o_gld = 0, dn_gld = 0;  // their row strides (elements)
};

// FP16 copies of a layer's panels (row strides padded to 8 elements) for the prefill GEMMs.
struct F16Panels {
    __half *qkv = nullptr, *o = nullptr, *gu = nullptr, *dn = nullptr;
    int ld_d = 0, ld_o = 0, ld_dn = 0;
};

constexpr uint32_t PLAN_MAGIC = 0x7A5B1A01u;
constexpr uint32_t SESSION_MAGIC = 0x7A5B5E55u;

struct Plan {
    uint32_t magic = PLAN_MAGIC;
    Store* store = nullptr;
    int live_sessions = 0;
    int panel_mode = 0;
    bool all_keep = false;
    std::vector<LayerPlan> layers;
    Arena arena;
    int64_t flops_retained = 0, flops_dense = 0, launched_flops = 0;
    int64_t weight_bytes_per_token = 0;
    bool f16_ready = false;  // FP16 panels made on the first prefill
    Arena f16_arena;
    std::vector<F16Panels> f16;
    // grouped store: the FP16 panels hold q s_g 2^F16_GS_EXP, and the prefill GEMMs scale their
    // rows by this array of 2^-F16_GS_EXP (the store's row scales are all 1); NULL otherwise
    const float* f16_post = nullptr;
};

// ---------------------------------------------------------------- sessions
struct StepGraph {
    cudaGraphExec_t exec = nullptr;
    const void* x = nullptr;
    float* hidden = nullptr;
    float* logits = nullptr;
    int launches = 0;
};

struct Session {
    uint32_t magic = SESSION_MAGIC;
    Plan* plan = nullptr;
    int max_tokens = 0;
    int pos = 0;  // host mirror of the device position
    Arena arena;
    std::vector<uint16_t*> K, V;  // per layer BF16 [m_kv][max_tokens][dh]
    // per layer TMA descriptors of K and V (boxes of 16 positions x 64 dims, 128-byte swizzle)
    std::vector<CUtensorMap> tmK, tmV;
    float2* rope = nullptr;       // [max_tokens][dh/2] (cos, sin)
    int* d_pos = nullptr;
    // workspace of one decode step
    float* x = nullptr;  // FP32 residual [d]
    float* q = nullptr;  // FP32 rotated queries [Hq dh]
    float* o = nullptr;  // FP32 attention output [Hq dh]
    float* h = nullptr;  // FP32 SiLU(gate) * up [df]
    float* part = nullptr;  // attention split partials [Hkv][splits][g][dh]
    float* ml = nullptr;    // attention split (max, sum) [Hkv][splits][g][2]
    int* cnt = nullptr;     // attention split tickets [Hkv]
    int* err = nullptr;     // device error word (0 = no kernel reported a failure)
    int att_splits_max = 0;
    uint16_t* x_stage = nullptr;  // BF16 [d] step-input staging (device and host-buffer steps)
    float* logits_stage = nullptr;
    float* hidden_stage = nullptr;
    StepGraph graph;
};

// ---------------------------------------------------------------- device info
// Failure-detection test hooks (tasp_test_set_wait_limit, tasp_test_skip_gemv_copies): a
// shorter limit for the bounded waits of the one-session GEMVs, and a number of upcoming
// one-session GEMV launches whose producer issues no copies.
namespace test_hooks {
long long wait_limit(long long dflt);  // the limit to launch with
bool take_skip();                      // true (and one fewer pending) if this launch skips its copies
}  // namespace test_hooks

struct DevInfo {
    int dev = -1, sms = 0, smem_optin = 0;
    int smem_per_sm = 0, smem_reserved = 0;  // shared memory of an SM, and reserved per resident CTA
};
int device_info(DevInfo& out);
// Model description -> Shape with every requirement checked (device: also the device limits).
int validate_shape(const tasp_model_desc* m, Shape& s, bool device = true);

// ---------------------------------------------------------------- kernels (launchers)
// store.cu
int store_generate(Store& st, cudaStream_t s);
int kv_fill_synthetic(Session& se, int t_prior, uint64_t kv_seed, cudaStream_t s);
int rope_table(Session& se, cudaStream_t s);
int gather_rows(int8_t* dst, const int8_t* src, const int32_t* map, int rows, int K, cudaStream_t s);
int gather_cols(int8_t* dst, int ld_dst, const int8_t* src, int ld_src, const int32_t* cmap, int rows, int Kc,
                cudaStream_t s);
int gather_f32(float* dst, const float* src, const int32_t* map, int n, cudaStream_t s);
// rows of a [*][cols] uint16 matrix (dst row r, stride ld_dst, = src row map[r])
int gather_u16_rows(uint16_t* dst, int ld_dst, const uint16_t* src, const int32_t* map, int rows, int cols,
                    cudaStream_t s);
// columns of a [rows][ld_src] uint16 matrix (dst [rows][ld_dst] column j = src column cmap[j], j < ncols)
int gather_u16_cols(uint16_t* dst, int ld_dst, const uint16_t* src, int ld_src, const int32_t* cmap, int rows,
                    int ncols, cudaStream_t s);

// attention.cu
constexpr int MAX_BATCH = 4;   // sessions of one plan that share each weight pass
constexpr int UNION_MAX = 16;  // sessions (of any plans) in one union-of-masks step
constexpr int ATTN_CLUSTERS_MAX = 8;  // decode attention clusters per kept group (global merge when > 1)
struct AttnParams {
    // TMA descriptors of session b's K / V cache of this layer (tma != 0, at most MAX_BATCH
    // sessions); otherwise the tiles are loaded with cp.async
    CUtensorMap tmK[MAX_BATCH], tmV[MAX_BATCH];
    int tma;
    int* err;            // device error word (bounded waits that gave up)
    // session b of the launch (blockIdx.z) reads q + b * q_stride, writes o + b * q_stride
    const float* q;      // FP32 rotated queries [m_kv g][dh] (kept groups, all g slots)
    float* o;            // FP32 [m_q][dh], kept heads in O-panel column order
    int64_t q_stride;
    const uint16_t* K[UNION_MAX];  // BF16 [m_kv][max_tokens][dh] of this layer
    const uint16_t* V[UNION_MAX];
    const int* pos[UNION_MAX];     // device position: the step attends to positions 0..pos
    int max_tokens[UNION_MAX];
    int m_kv[UNION_MAX];           // kept groups of the session's plan (grid y covers the largest)
    const int16_t* oslot[UNION_MAX];  // output slot per (group slot, head), NULL = jl g + hh
    float qscale;        // log2(e) / sqrt(dh)
    float* part;         // + b * part_stride
    float* ml;           // + b * ml_stride
    int* cnt;            // + b * cnt_stride; zero between launches
    int64_t part_stride, ml_stride, cnt_stride;
};
int attn_supported(int dh, int g);
int attn_cluster(int dh, int g);  // CTAs per cluster of the attention kernel (16, else 8)
int attn_splits(int m_kv, int max_tokens, int sms, int dh, int g, int cs_cap = 16);
int attn_splits_max();
// Cluster size for one launch of m_kv kept groups x nb sessions: 16, or 8 when 16-CTA clusters
// would take more waves than 8-CTA ones (more clusters than the device holds at once)
int attn_cluster_for(int m_kv, int nb, int max_tokens, int dh, int g, bool tma);
// C[m][n] = scale[n] * sum_k A[m][k] B[n][k] on the tensor cores (prefill.cu's persistent
// tcgen05 GEMM): FP16 A [M][lda], B [N][ldb], FP32 C [M][ldc]; K a multiple of 8.
int gemm_f16_nt(const __half* A, int lda, int M, const __half* B, int ldb, int N, int K, const float* scale, float* C,
                int ldc, int* err, cudaStream_t s);
// TMA descriptor of a BF16 KV cache [m_kv][max_tokens][dh]: 16 positions x 64 dims per box,
// 128-byte swizzle (prefill.cu)
int encode_kv_map(CUtensorMap* m, const uint16_t* base, int dh, int max_tokens, int m_kv);
// cs_cap: largest cluster size to use (16 or 8; many short sessions run better on 8)
int launch_attention(const AttnParams& a, int dh, int g, int m_kv, int splits, int nb, cudaStream_t s,
                     int cs_cap = 16);

// decode.cu
enum KernelKind { K_QKV = 0, K_ATTN = 1, K_O = 2, K_GU = 3, K_DOWN = 4, K_LM = 5, K_OTHER = 6 };

struct StepTarget {
    const uint16_t* x_in = nullptr;  // BF16 [n][d] step inputs (first layer) or nullptr (use residual)
    float* hidden_out = nullptr;     // [n][d]
    float* logits = nullptr;         // [n][vocab]
    bool advance = true;
    // attention split scratch; nullptr = the workspace of the batch view
    float* att_part = nullptr;
    float* att_ml = nullptr;
    int* att_cnt = nullptr;
};

// The n (<= MAX_BATCH) sessions of one plan that a decode step runs together, with the
// step workspace they use: every weight byte is read once for all of them.
struct BatchView {
    int n = 0;
    Session* ss[MAX_BATCH] = {};
    float *x = nullptr, *q = nullptr, *o = nullptr, *h = nullptr;  // FP32 [n][...]
    int64_t x_stride = 0, q_stride = 0, h_stride = 0;
    float* part = nullptr;  // attention partials, session b at + b * part_stride
    float* ml = nullptr;
    int* cnt = nullptr;
    int64_t part_stride = 0, ml_stride = 0, cnt_stride = 0;
    int* err = nullptr;     // device error word of the step
};
// View of one session on its own workspace.
BatchView single_view(Session& se);
// Attention split slots (partials per kept group) a batch view must hold.
int batch_attn_slots(const Plan& p, const Session* const* ss, int n, int sms);

using KernelHook = void (*)(void* ctx, int kind, bool before);

// union.cu: free the union-step workspaces (and graphs) that include this session.
void union_drop(Session* se);
// Final RMSNorm + LM head of a batch view's residuals into logits [n][vocab].
int enqueue_lm_heads(const BatchView& bv, float* logits, cudaStream_t s);
// Enqueue one decode step of a batch (or one isolated layer when only_layer >= 0) on `s`.
int enqueue_batch(const BatchView& bv, const StepTarget& t, cudaStream_t s, int only_layer, KernelHook hook,
                  void* ctx, int* launches);
// The same for one session on its own workspace.
int enqueue_step(Session& se, const StepTarget& t, cudaStream_t s, int only_layer, KernelHook hook, void* ctx,
                 int* launches);
// Final RMSNorm + LM head on the session's residual (se.x) into logits [vocab].
int enqueue_lm_head(Session& se, float* logits, cudaStream_t s);
// Device position of a session := pos.
int enqueue_set_pos(Session& se, int pos, cudaStream_t s);

// prefill.cu: run the prompt [T][d] (BF16) through the plan, filling KV positions 0..T-1
// and leaving the last position's residual in se.x.
int prefill_run(Session& se, const uint16_t* d_embeds, int T, cudaStream_t s);

}  // namespace tasp
