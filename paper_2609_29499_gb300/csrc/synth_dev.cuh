// The library's implementation of the synthetic-data generator (host + device).
//
// Counter-based SplitMix64 (Steele, Lea, Flood, OOPSLA 2014): output n of a
// generator with state `key` is fin(key + (n + 1) * 0x9E3779B97F4A7C15), fin being
// the variant-13 finalizer (xor-shift 30, multiply 0xBF58476D1CE4E5B9, xor-shift
// 27, multiply 0x94D049BB133111EB, xor-shift 31). Streams are keyed by folding
// (seed, tensor id, layer, sub) through k -> fin(k + 0x9E3779B97F4A7C15). A normal
// value is the Irwin-Hall sum of the twelve 16-bit lanes of outputs 3i..3i+2,
// centred by 393210 and scaled by 2^-16 (exact in FP32).
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

namespace tasp {

enum SynthTensor : uint64_t {
    ST_WQ = 1, ST_WK = 2, ST_WV = 3, ST_WO = 4, ST_WGATE = 5, ST_WUP = 6, ST_WDOWN = 7,
    ST_GAMMA_ATTN = 8, ST_GAMMA_MLP = 9, ST_GAMMA_FINAL = 10, ST_LMHEAD = 11,
    ST_KCACHE = 20, ST_VCACHE = 21
};

constexpr uint64_t SM_STEP = 0x9E3779B97F4A7C15ull;
constexpr float SM_WEIGHT_SIGMA = 0.02f;

__host__ __device__ __forceinline__ uint64_t sm_fin(uint64_t v) {
    v ^= v >> 30;
    v *= 0xBF58476D1CE4E5B9ull;
    v ^= v >> 27;
    v *= 0x94D049BB133111EBull;
    v ^= v >> 31;
    return v;
}

__host__ __device__ __forceinline__ uint64_t sm_key(uint64_t seed, uint64_t tensor, uint64_t layer, uint64_t sub) {
    uint64_t k = sm_fin(seed + SM_STEP);
    k = sm_fin((k ^ tensor) + SM_STEP);
    k = sm_fin((k ^ layer) + SM_STEP);
    k = sm_fin((k ^ sub) + SM_STEP);
    return k;
}

__device__ __forceinline__ float sm_normal(uint64_t key, uint64_t i) {
    uint64_t base = key + (3ull * i + 1ull) * SM_STEP;
    uint32_t acc = 0;
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        uint64_t v = sm_fin(base + (uint64_t)k * SM_STEP);
        uint32_t lo = (uint32_t)v, hi = (uint32_t)(v >> 32);
        acc += (lo & 0xFFFFu) + (lo >> 16) + (hi & 0xFFFFu) + (hi >> 16);
    }
    int c = (int)acc - 393210;
    return __fmul_rn(__int2float_rn(c), 1.0f / 65536.0f);
}

__device__ __forceinline__ uint16_t sm_bf16_bits(float v) {
    __nv_bfloat16 b = __float2bfloat16_rn(v);
    return *reinterpret_cast<uint16_t*>(&b);
}

}  // namespace tasp
