/*
 * tasp.h - C ABI of the TASP compiled sparse execution path on one GB300 (sm_103a).
 *
 * The path (paper Sec. 3.3 and Appendix "Backing-store semantics"): one shared,
 * immutable INT8 weight store per model; a mask is a dependency-closed set of
 * retained GQA groups and SwiGLU channel units, compiled into a plan (retained
 * index lists + packed panels + launch geometry) that owns no weights it does
 * not need; one plan is chosen per user turn and stays fixed through prefill
 * and every decode step; a KV cache is never reused across plans.
 *
 * Conventions for every function below:
 *  - Return value: TASP_OK (0) or a negative tasp_status. Nothing aborts. On
 *    failure tasp_last_error() returns a thread-local description.
 *  - Pointers named d_* are DEVICE pointers owned by the caller; h_* are HOST
 *    pointers owned by the caller. All other objects (store, plans, sessions
 *    and their device memory) are owned by the library and freed with
 *    tasp_release().
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    Functions marked "async" enqueue work on it and return without
 *    synchronizing; their device outputs are valid once the stream reaches
 *    that point. Functions marked "sync" synchronize the device before return.
 *  - BF16 buffers hold IEEE bfloat16 bit patterns (uint16); FP32 buffers hold
 *    float. Matrices are row-major. A d_* buffer must be aligned to its
 *    element size (2 bytes for BF16, 4 for FP32); a misaligned one is refused
 *    with TASP_EINVAL before any work. The library cannot tell a device
 *    pointer from a host one: passing a host pointer as d_* is undefined.
 *  - All sizes are element counts unless the name says bytes.
 */
#ifndef TASP_H
#define TASP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum tasp_status {
    TASP_OK = 0,
    TASP_EINVAL = -1, /* bad shape, pointer, mask (closure violated, budget exceeded, empty layer) */
    TASP_EMASK = -2,  /* sessions of different plans in one decode call (KV reuse across masks, Sec. 3.3) */
    TASP_ECAP = -3,   /* KV-cache capacity of a session exhausted */
    TASP_ENOMEM = -4, /* device or host allocation failed */
    TASP_EBUSY = -5,  /* plan released while sessions still reference it */
    TASP_ECUDA = -6,  /* a CUDA call failed; tasp_last_error() holds the CUDA error string */
    TASP_EUNSUP = -7  /* valid request this build does not implement */
} tasp_status;

/* Shape of a Llama-style decoder (Sec. 3.3 / Table 1) and the seed of its
 * synthetic weights. Requirements: Hq % Hkv == 0, dh even and a multiple of 16
 * (dh <= 128), d % 16 == 0, df % chan_unit == 0, vocab >= 0 (0 = no LM head).
 * The library regenerates the weights from `seed` with its counter-based
 * generator (N(0, 0.02), quantized per output row to INT8 with FP32 scales). */
typedef struct tasp_model_desc {
    int32_t L, d, Hq, Hkv, dh, df, vocab;
    int32_t chan_unit; /* SwiGLU channels per mask unit (1,024 in Table 1) */
    float rms_eps;     /* RMSNorm epsilon (1e-5) */
    float rope_theta;  /* rotary base (500000) */
    uint64_t seed;
    int32_t quant_group; /* INT8 scale granularity: 0 = one FP32 scale per output row; G > 0 =
                            one BF16 scale per output row and run of G input columns (Table 1:
                            G = 128). G must divide d, Hq*dh, df, dh and chan_unit and be a
                            multiple of 16. Grouped stores serve every path: decode (one
                            session or batches), prefill and the union step. */
} tasp_model_desc;

enum tasp_mask_kind {
    TASP_MASK_ALL_KEEP = 0,       /* dense fallback: every unit retained; panels are the store itself */
    TASP_MASK_GREEDY = 1,         /* budgeted greedy by score per active FLOP with closure (Sec. 3.3) */
    TASP_MASK_EXPLICIT = 2,       /* caller-given retained groups / channel units per layer */
    TASP_MASK_GREEDY_QHEADS = 3,  /* the greedy over query-head candidates (Sec. 3.3, Table 1) */
    TASP_MASK_EXPLICIT_QHEADS = 4 /* caller-given retained query heads / channel units per layer */
};

enum tasp_panel_mode {
    TASP_PANELS_COMPACT = 0,    /* all four panels are packed copies (contiguous retained tensors) */
    TASP_PANELS_ROW_INDEXED = 1 /* Q/K/V and gate/up rows index the shared store (zero copy);
                                   O and down columns are packed copies. Same bytes are read. */
};

/* Mask request. For kind GREEDY: `scores` is host uint32 [L][Hkv + df/chan_unit]
 * (stand-ins for the predictor scores s_h of Sec. 3.3; groups first, then
 * channel units), `target_u24` is host uint32 [L] with per-layer retention
 * draws in [0, 2^24), `flop_budget` the active-FLOP target (0.57) and
 * [r_lo, r_hi] the per-layer retention range. For kind EXPLICIT:
 * keep_groups / keep_units are host int32 lists concatenated over layers with
 * n_groups / n_units [L] giving each layer's count (indices ascending).
 * Query-head kinds (Sec. 3.3: a KV head stays whenever one of its query heads
 * does; query heads never move across groups): GREEDY_QHEADS takes `scores`
 * [L][Hq + df/chan_unit] (query heads first, then channel units) with the
 * same budget fields, and charges a head its Q rows and O columns plus, for
 * the first head of a group, the group's K and V rows; EXPLICIT_QHEADS takes
 * keep_qheads / n_qheads (ascending heads, concatenated over layers) with
 * keep_units / n_units, and keeps the KV head of every listed head.
 * Unused fields may be NULL / 0. */
typedef struct tasp_mask_desc {
    int32_t kind;
    int32_t panel_mode;
    double flop_budget, r_lo, r_hi;
    const uint32_t* scores;
    const uint32_t* target_u24;
    const int32_t* keep_groups;
    const int32_t* n_groups;
    const int32_t* keep_units;
    const int32_t* n_units;
    const int32_t* keep_qheads;
    const int32_t* n_qheads;
} tasp_mask_desc;

typedef struct tasp_plan tasp_plan;
typedef struct tasp_session tasp_session;

/* ---------------------------------------------------------------------------
 * The four entry points of the path.
 * ------------------------------------------------------------------------- */

/* Compile one mask into a plan (Sec. 3.3 "packed into contiguous tensors and
 * compiled as static launch plans over one shared INT8 weight store";
 * Appendix "Backing-store semantics"). Creates the model's shared store on
 * first use (generated and quantized on the device; later plans with an
 * identical model_desc share it), runs the host mask compiler, packs the
 * panels on the device. sync. *out receives the plan.
 * Errors: EINVAL (bad desc, mask violates closure/budget, empty layer),
 * ENOMEM, ECUDA. Query-head masks may keep part of a group: the plan then
 * carries per-layer role tables for its partial groups. */
int tasp_compile_mask(const tasp_model_desc* model, const tasp_mask_desc* mask, tasp_plan** out);

/* Prefill one prompt with a plan (Sec. 3.3: the plan chosen for a turn serves
 * its prefill; Fig. 1 "one launch plan for prefill"): d_embeds_bf16 is a device
 * BF16 [T][d] buffer of input embeddings. Creates a session whose KV cache
 * (retained KV heads only, capacity T + max_new_tokens) holds the prompt's
 * keys/values. If d_logits_last != NULL it receives FP32 [vocab] logits of the
 * last prompt position. async on `stream`. *out receives the session.
 * Errors: EINVAL, ENOMEM, ECUDA, EUNSUP (vocab == 0 with d_logits_last, or d not
 * a multiple of 8). */
int tasp_prefill(tasp_plan* plan, const void* d_embeds_bf16, int32_t T, int32_t max_new_tokens, void* stream,
                 tasp_session** out, float* d_logits_last);

/* One decode step for n >= 1 sessions that share one plan (Fig. 1 "same plan
 * for every decode step"). d_x_bf16 is device BF16 [n][d] (the step's input
 * vectors, session order). Outputs, each optional (NULL skips it):
 * d_hidden_out FP32 [n][d] = the residual stream after the last decoder layer
 * (before the final norm); d_logits FP32 [n][vocab]. Each session's KV grows by
 * one position. Sessions are taken in groups of up to 4 (session order): the
 * GEMVs of a group read every weight byte once for all of its sessions and one
 * attention grid covers them, each on its own KV cache and position (the decode
 * step groups the turns that share a mask). A group of 2-4 sessions keeps a step
 * workspace (~ n x (d + 2 H_q d_h + d_f + vocab) x 4 bytes plus attention
 * partials) until one of its sessions is released. Results per session do not
 * depend on the group (up to FP32 summation order). The inputs are copied on
 * `stream` into the session's (or group's) own staging buffer, and the step is
 * replayed from a CUDA graph captured on first use for this (sessions, output
 * buffers) combination; call it outside any stream capture. async on `stream`.
 * Errors: EMASK (sessions on different plans), ECAP (a session is full),
 * EINVAL, ENOMEM, ECUDA. */
int tasp_decode_step(tasp_session* const* sessions, int32_t n, const void* d_x_bf16, float* d_hidden_out,
                     float* d_logits, void* stream);

/* Release a plan or a session (the handle's type is recorded inside). A plan
 * still referenced by live sessions returns EBUSY and stays valid. The shared
 * store is freed with its last plan. sync. NULL is a no-op. */
int tasp_release(void* handle);

/* ---------------------------------------------------------------------------
 * Sessions without prefill, host-buffer decode, host-only mask compilation.
 * ------------------------------------------------------------------------- */

/* Empty session on a plan with KV capacity max_tokens (position 0). sync. */
int tasp_session_create(tasp_plan* plan, int32_t max_tokens, tasp_session** out);

/* Prefill a prompt into an existing session (its previous contents are
 * overwritten from position 0; capacity must be >= T): the same computation as
 * tasp_prefill without allocating the session. async. Errors: EINVAL, ECAP,
 * EUNSUP, ECUDA. */
int tasp_session_prefill(tasp_session* s, const void* d_embeds_bf16, int32_t T, void* stream, float* d_logits_last);

/* Fill positions [0, t_prior) of a session's KV cache with the synthetic
 * N(0,1) BF16 "prior tokens" keyed by kv_seed (the keys are taken as already
 * rotated) and set its position to t_prior. async. Errors: ECAP, EINVAL. */
int tasp_session_fill_synthetic(tasp_session* s, int32_t t_prior, uint64_t kv_seed, void* stream);

/* Current position (number of cached tokens) as tracked on the host. */
int tasp_session_position(const tasp_session* s, int32_t* pos);

/* Device-side status of a session's kernels: *device_error = 0 when no kernel
 * reported a failure; bit 0 set when a bounded wait inside a kernel gave up
 * (the step's outputs are then invalid). Synchronizes the device; clears the word
 * when `clear` is nonzero. */
int tasp_session_status(tasp_session* s, int32_t clear, int32_t* device_error);

/* tasp_decode_step with HOST buffers: h_x_bf16 [n][d] is copied to the device
 * (should be pinned memory), the step runs, and the requested outputs are
 * copied back to h_hidden_out [n][d] / h_logits [n][vocab] (either may be
 * NULL). Synchronizes `stream` before returning. */
int tasp_decode_step_host(tasp_session* const* sessions, int32_t n, const void* h_x_bf16, float* h_hidden_out,
                          float* h_logits, void* stream);

/* Host-only mask compilation (no GPU work): the retained index lists the plan
 * would use. Outputs (host, caller-sized): keep_groups [L*Hkv] and keep_units
 * [L*(df/chan_unit)] concatenated per layer with counts n_groups [L],
 * n_units [L]; flops [L + 3] = per-layer retained FLOPs (Eqs. flop-attn +
 * flop-mlp), the total, the global budget B and the dense total. */
int tasp_mask_select(const tasp_model_desc* model, const tasp_mask_desc* mask, int32_t* keep_groups,
                     int32_t* n_groups, int32_t* keep_units, int32_t* n_units, int64_t* flops);

/* tasp_mask_select plus the retained query heads: keep_qheads [L*Hq] with
 * n_qheads [L] (ascending per layer). For the group kinds these are all g heads
 * of every kept group; for the query-head kinds keep_groups holds the KV heads
 * that the closure keeps. Host only; any output may be NULL. */
int tasp_mask_select_qheads(const tasp_model_desc* model, const tasp_mask_desc* mask, int32_t* keep_qheads,
                            int32_t* n_qheads, int32_t* keep_groups, int32_t* n_groups, int32_t* keep_units,
                            int32_t* n_units, int64_t* flops);

/* Host only (test introspection): the tables a plan of `mask` uses for one layer.
 * qkv_src [(m_q + 2 m_kv) dh]: store row of each qkv panel row (store rows are
 * group-major: per KV group its g head blocks of dh rows, then K, then V);
 * o_src [m_q dh]: dense O column of each panel column; role [m_q + 2 m_kv],
 * slot [m_kv g], blk_of [m_kv (g + 2)]: the partial-group tables (role of each
 * dh-row block as jl (g + 2) + hh; compact O position of (jl, hh) or -1; inverse
 * of role or -1). counts [5] receives the five lengths. Any array may be NULL. */
int tasp_plan_layout(const tasp_model_desc* model, const tasp_mask_desc* mask, int32_t layer, int32_t* qkv_src,
                     int32_t* o_src, int16_t* role, int16_t* slot, int16_t* blk_of, int32_t* counts);

/* ---------------------------------------------------------------------------
 * Introspection and measurement (tests and benchmark).
 * ------------------------------------------------------------------------- */

typedef struct tasp_plan_info {
    int32_t L;
    int64_t panel_bytes;   /* device bytes owned by the plan (packed panels, maps, scales) */
    int64_t store_bytes;   /* device bytes of the shared store (INT8, scales, gains, LM head) */
    int64_t weight_bytes_per_token; /* INT8 panel bytes + FP32 scales + BF16 LM head read per decode token */
    int64_t flops_retained, flops_dense; /* layer FLOPs per token, Eqs. flop-attn + flop-mlp */
    int64_t launched_flops; /* 2 x rows x cols over the packed panels (Appendix ledger check) */
} tasp_plan_info;

int tasp_plan_info_get(const tasp_plan* plan, tasp_plan_info* out);

/* Per-layer retained sizes: out[0] = m_kv (kept groups), out[1] = c (kept channels). */
int tasp_plan_layer_dims(const tasp_plan* plan, int32_t layer, int32_t* out2);
/* Kept query heads m_q of a layer (m_kv g unless the mask keeps part of a group). */
int tasp_plan_layer_qheads(const tasp_plan* plan, int32_t layer, int32_t* m_q);

enum tasp_export_item {
    TASP_EXPORT_KEEP_GROUPS = 0, /* int32 [m_kv] */
    TASP_EXPORT_KEEP_CHANS = 1,  /* int32 [c] */
    TASP_EXPORT_QKV_W = 2,       /* int8 [(m_q + 2 m_kv) dh][d] */
    TASP_EXPORT_QKV_S = 3,       /* float [(m_q + 2 m_kv) dh] */
    TASP_EXPORT_O_W = 4,         /* int8 [d][m_q dh] */
    TASP_EXPORT_O_S = 5,         /* float [d] */
    TASP_EXPORT_GU_W = 6,        /* int8 [2c][d], gate row then up row per kept channel */
    TASP_EXPORT_GU_S = 7,        /* float [2c] */
    TASP_EXPORT_DOWN_W = 8,      /* int8 [d][c] */
    TASP_EXPORT_DOWN_S = 9,      /* float [d] */
    TASP_EXPORT_KEEP_QHEADS = 10, /* int32 [m_q] */
    /* groupwise stores: BF16 scale bit patterns (uint16) of the panels */
    TASP_EXPORT_QKV_G = 11,      /* [(m_q + 2 m_kv) dh][d / G] */
    TASP_EXPORT_O_G = 12,        /* [d][m_q dh / G] */
    TASP_EXPORT_GU_G = 13,       /* [2c][d / G] */
    TASP_EXPORT_DOWN_G = 14      /* [d][c / G] */
};

/* Copy one packed panel (logical layout, no padding) or index list of a layer
 * to host memory h_dst of `bytes` bytes (must equal the item's size). sync. */
int tasp_plan_export(const tasp_plan* plan, int32_t layer, int32_t item, void* h_dst, size_t bytes);

/* Run one decoder layer of a session's plan in isolation on a given FP32
 * residual d_x_in [d] at the session's current position, writing d_x_out [d]
 * (K/V of that position are written into the layer's cache; the position is
 * not advanced). For per-layer parity checks. async. */
int tasp_layer_step(tasp_session* s, int32_t layer, const float* d_x_in, float* d_x_out, void* stream);

/* Run one decode step eagerly (no graph, no programmatic overlap) with CUDA
 * events around every kernel, then synchronize. h_ms[k] / h_count[k] receive
 * the total time and launch count of kernel kind k over the step:
 * 0 qkv (RMSNorm + QKV GEMV + RoPE + KV append), 1 attention (split-KV + combine),
 * 2 o-proj + residual, 3 gate/up + SiLU*up, 4 down + residual, 5 final norm +
 * LM head, 6 other. Arrays have TASP_KERNEL_KINDS entries. Sessions are grouped
 * as in tasp_decode_step. */
#define TASP_KERNEL_KINDS 7
int tasp_profile_step(tasp_session* const* sessions, int32_t n, const void* d_x_bf16, float* d_logits,
                      void* stream, float* h_ms, int32_t* h_count);

/* Copy the cached keys (which = 0) or values (which = 1) of one layer, BF16
 * [m_kv][position][dh] for positions 0 .. current position - 1, to host memory of
 * exactly that many bytes. sync. */
int tasp_session_kv_export(const tasp_session* s, int32_t layer, int32_t which, void* h_dst, size_t bytes);

/* Number of library kernel launches one decode step of these sessions makes
 * (graph nodes): one launch sequence per group of up to 4 sessions. */
int tasp_step_launches(tasp_session* const* sessions, int32_t n, int32_t with_logits, int32_t* out);

/* ---------------------------------------------------------------------------
 * Allocation-free decode step (the paper has no counterpart: a deployment aid).
 * ------------------------------------------------------------------------- */

/* tasp_decode_step for ONE session that allocates nothing, for callers that must
 * not enter the CUDA allocator while decoding (a fixed device-memory budget that
 * is already handed out, another library's stream capture in progress, a serving
 * loop that forbids allocator calls). The step's kernels are launched directly (no
 * CUDA graph is built) and the attention scratch comes from one file-scope
 * device array of about 260 KB (8 kept KV groups x 8 attention clusters per
 * group x 8 query heads per group x head dim 128 partial floats, plus maxima/sums
 * and 8 merge tickets) that every GPU loading the library holds until the process
 * exits. The clusters are used when a session's capacity exceeds one cluster's
 * reach (about 6,100 positions at head dim 128, 12,200 at 64).
 * Arguments and outputs are those of tasp_decode_step with n = 1. The first call on
 * a device looks up the array's device address (cudaGetSymbolAddress); make that
 * first call before any stream capture. All calls share the array and it keeps the
 * last call's contents (the tickets are cleared at the start of every call), so
 * calls whose kernels overlap on the GPU (different streams, several sessions at
 * once) race: serialize them. Errors: EINVAL (NULL pointers, or a plan whose
 * attention partials exceed the array), ECAP, ECUDA. async on `stream`. */
int tasp_decode_step_static(tasp_session* s, const void* d_x_bf16, float* d_hidden_out, float* d_logits,
                            void* stream);

/* ---------------------------------------------------------------------------
 * Union-of-masks batched decode (the next step after per-plan grouping).
 * ------------------------------------------------------------------------- */

/* One decode step for 1 <= n <= 16 sessions whose plans may differ (each turn keeps
 * the mask it was started with: its KV cache stays plan-shaped). Every weight row
 * of the shared store is read once for all n sessions: the projections run dense
 * for all of them on the tensor cores (INT8 rows converted to FP16 in tensor
 * memory, times the BF16 group scale for a grouped store; activations in FP16 with a
 * per-session power-of-two scale; FP32 accumulation), and each session's mask is
 * applied where a unit meets it: Q/K/V of a dropped group are not written, attention
 * runs over the session's own kept groups, dropped heads (whole groups, or single
 * query heads of a query-head plan) enter the O projection as zeros and dropped
 * channel units leave SiLU(gate) * up at zero. This equals the session's compacted plan up to
 * FP32 summation order and FP16 rounding of the activations (the mask-as-zero
 * reading of a plan, Sec. 3). d_x_bf16 is device BF16 [n][d]; d_hidden_out FP32
 * [n][d] and d_logits FP32 [n][vocab] are optional (NULL skips). The sessions must
 * share one weight store; d, H_q d_h and d_f must be multiples of 128. The set of
 * sessions keeps a workspace (~ 16 x (2 d + 2 H_q d_h + d_f) x 4 bytes, partial
 * sums of ~ 16 x 4 x (rows of the largest projection) bytes, attention partials)
 * and a CUDA graph captured on first use for these output buffers; inputs are
 * copied on `stream` into its staging buffer. Call it outside any stream capture.
 * async on `stream`. Errors: EMASK (sessions on different stores), ECAP (a session
 * is full), EUNSUP (shape), EINVAL, ENOMEM, ECUDA. */
int tasp_decode_step_union(tasp_session* const* sessions, int32_t n, const void* d_x_bf16, float* d_hidden_out,
                           float* d_logits, void* stream);

/* Device error word (bit 0: a bounded wait gave up) and graph launch count of the
 * union workspace of these sessions (created if absent). sync. */
int tasp_union_status(tasp_session* const* sessions, int32_t n, int32_t* device_error, int32_t* launches);

/* Per-turn plan choice (Sec. 3.3; Table 1: tau = 0.85): given the router's task
 * distribution h_probs [n] over the n task masks, *plan = the index of the most
 * probable task (lowest index on ties) when its probability reaches tau, else n,
 * the dense plan. Host only; EINVAL for NULL, n < 1, tau outside [0, 1] or a
 * negative / non-finite probability. */
int tasp_dispatch(const float* h_probs, int32_t n, float tau, int32_t* plan);

/* Cap on the device memory held by the library's arenas (the shared store,
 * plan panels, sessions and step workspaces); 0 = no cap, the default. A
 * reservation that would pass the cap fails with TASP_ENOMEM before anything
 * is allocated, and the call that needed it fails cleanly. Prefill's per-call
 * temporaries come from the stream-ordered pool and are not counted. Host only. */
int tasp_set_memory_limit(int64_t bytes);
/* Device bytes the library's arenas hold now. Host only. */
int tasp_memory_in_use(int64_t* bytes);

/* ---------------------------------------------------------------------------
 * Spectral descriptors of the candidate units (the calibration side of the method).
 * ------------------------------------------------------------------------- */

/* Features of every candidate unit of one layer (Sec. 3.1 "Candidate Units and Spectral
 * Features", Eqs. 1-4; Appendix "Exact candidate feature construction"): the H_q attention
 * heads (block [4 dh][d]: the head's Q rows, the O columns it feeds transposed, its KV group's
 * K and V rows), then the df / chan_unit channel groups (block [3 chan_unit][d]: gate rows, up
 * rows, down columns transposed), built from the model's synthetic weights rounded to BF16.
 * With lambda_i = s_i^2 / d the eigenvalues of a block's normalized Gram matrix:
 * h_features FP64 [H_q + df / chan_unit][6] = (alpha: Pareto exponent of the tail
 * lambda >= lambda_min by maximum likelihood, lambda_min chosen among the distinct eigenvalues
 * below the largest to minimize the Kolmogorov-Smirnov distance, ties to the smaller; effective
 * rank; spectral norm s_1; SETOL, the tail's share of sum lambda; lambda_min; the KS distance).
 * h_lambda (optional) FP64 [H_q 4 dh + (df / chan_unit) 3 chan_unit]: each block's
 * eigenvalues, descending, blocks in the same order. The Gram matrices run on the tensor cores
 * (FP16 operands holding the BF16 weights, FP32 accumulation); the eigenvalues come from
 * cuSOLVER's symmetric eigensolver, loaded at run time. Per-call device temporaries come from
 * the stream-ordered pool. h_phase_ms (optional) FP64 [4] receives the device time summed
 * over the candidates of the four steps: block generation, Gram matrices, eigensolver,
 * statistics. sync. Errors: EINVAL (desc, layer, NULL), EUNSUP (4 dh or 3 chan_unit above d,
 * d not a multiple of 64, or no eigensolver), ECUDA. */
int tasp_spectral_layer(const tasp_model_desc* model, int32_t layer, double* h_features, double* h_lambda,
                        double* h_phase_ms, void* stream);

/* ---------------------------------------------------------------------------
 * Failure-detection test hooks (the paper has no counterpart). They let a test make
 * a device wait run out without faulting or hanging the GPU; both are process-wide,
 * host only, and meant for eager launches (tasp_layer_step, tasp_profile_step,
 * tasp_decode_step_static): a CUDA graph captured while a hook is set keeps it.
 * ------------------------------------------------------------------------- */

/* Clock-cycle limit of the bounded mbarrier waits in the one-session GEMVs launched
 * from now on (0 restores the default of ~2 s). A wait that runs out sets bit 0 of the
 * session's device error word, every later wait of that CTA returns at once, and the
 * kernel returns (its outputs are then invalid). EINVAL for a negative value. */
int tasp_test_set_wait_limit(int64_t cycles);

/* The next `launches` one-session GEMV launches issue no weight copies at all, so their
 * consumers' first wait runs out (nothing is ever in flight); 0 cancels. EINVAL for a
 * negative count. */
int tasp_test_skip_gemv_copies(int32_t launches);

/* Thread-local description of the last failure on this thread ("" if none). */
const char* tasp_last_error(void);

/* Library version string. */
const char* tasp_version(void);

#ifdef __cplusplus
}
#endif

#endif /* TASP_H */
