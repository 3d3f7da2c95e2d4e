// Allocation-free decode step.
//
// Some callers cannot allocate device memory at the moment they decode: code that
// runs under a fixed memory budget whose pool is already handed out, code inside a
// region where the CUDA allocator must not be entered (another library's stream
// capture, a real-time serving loop that forbids allocator calls), or embedders whose
// own allocator owns the device. tasp_decode_step_static serves them: it launches the
// step's kernels directly (no CUDA graph is instantiated) and takes the attention
// scratch (per-cluster partial outputs of long contexts, their maxima/sums and the
// merge tickets) from one file-scope device array instead of the session's workspace.
//
// The array is a module global: every GPU that loads this library holds it until the
// process exits, every call shares it, and it keeps the last call's contents.
#include <cuda_runtime.h>

#include <map>
#include <mutex>

#include "tasp_internal.h"

namespace tasp {

namespace {

// Capacity of the shared scratch: up to 8 kept KV groups per layer, each with at most
// ATTN_CLUSTERS_MAX attention clusters whose partial outputs (8 query heads per group x
// head dimension 128, the Llama-3 8B/70B shapes) and (max, sum) pairs are kept: ~260 KB.
constexpr size_t kGroups = 8;
constexpr size_t kPartFloats = kGroups * ATTN_CLUSTERS_MAX * 8 * 128;
constexpr size_t kMlFloats = kGroups * ATTN_CLUSTERS_MAX * 8 * 2;
constexpr size_t kTickets = kGroups;
constexpr size_t kScratchFloats = kPartFloats + kMlFloats + kTickets;

static __device__ __align__(256) float g_tasp_static_scratch[kScratchFloats];

std::mutex g_mu;
std::map<int, float*> g_addr;  // device ordinal -> device address of the array

// Device address of the array for the current device (looked up once per device).
int scratch_address(float** out) {
    int dev = 0;
    TASP_CUDA(cudaGetDevice(&dev));
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_addr.find(dev);
    if (it != g_addr.end()) {
        *out = it->second;
        return TASP_OK;
    }
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_tasp_static_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(static attention scratch)");
    g_addr[dev] = static_cast<float*>(p);
    *out = static_cast<float*>(p);
    return TASP_OK;
}

}  // namespace

}  // namespace tasp

using namespace tasp;

extern "C" int tasp_decode_step_static(tasp_session* s, const void* d_x_bf16, float* d_hidden_out, float* d_logits,
                                       void* stream) {
    if (int rc = check_aligned({{d_x_bf16, 2}, {d_hidden_out, 4}, {d_logits, 4}})) return rc;
    Session* se = (Session*)s;
    if (!se || se->magic != SESSION_MAGIC) return fail(TASP_EINVAL, "invalid session handle");
    if (!d_x_bf16) return fail(TASP_EINVAL, "d_x_bf16 is NULL");
    if (se->pos + 1 > se->max_tokens) return fail(TASP_ECAP, "session KV capacity exhausted");
    const Plan& pl = *se->plan;
    const Shape& sh = pl.store->sh;
    if (d_logits && sh.vocab == 0) return fail(TASP_EINVAL, "logits requested from a model without LM head");
    DevInfo di;
    int rc = device_info(di);
    if (rc) return rc;
    // every layer's attention partials must fit the static array
    for (const LayerPlan& lp : pl.layers) {
        // partial outputs are kept per cluster of the attention kernel
        const size_t S = (size_t)attn_splits(lp.m_kv, se->max_tokens, di.sms, sh.dh, sh.g(), 8) / 8;  // either size
        const size_t part = (size_t)lp.m_kv * S * sh.g() * sh.dh;
        const size_t ml = (size_t)lp.m_kv * S * sh.g() * 2;
        if (part > kPartFloats || ml > kMlFloats || (size_t)lp.m_kv > kTickets)
            return fail(TASP_EINVAL, "plan exceeds the static attention scratch (at most " +
                                         std::to_string(kPartFloats) + " partial floats, " + std::to_string(kTickets) +
                                         " kept KV groups per layer)");
    }
    float* base = nullptr;
    if ((rc = scratch_address(&base))) return rc;
    cudaStream_t st = (cudaStream_t)stream;
    int* tickets = reinterpret_cast<int*>(base + kPartFloats + kMlFloats);
    // the merge tickets must start at zero (a previous call may have been cut short)
    TASP_CUDA(cudaMemsetAsync(tickets, 0, kTickets * sizeof(int), st));
    StepTarget t;
    t.x_in = (const uint16_t*)d_x_bf16;
    t.hidden_out = d_hidden_out;
    t.logits = d_logits;
    t.att_part = base;
    t.att_ml = base + kPartFloats;
    t.att_cnt = tickets;
    if ((rc = enqueue_step(*se, t, st, -1, nullptr, nullptr, nullptr))) return rc;
    se->pos += 1;
    return TASP_OK;
}
