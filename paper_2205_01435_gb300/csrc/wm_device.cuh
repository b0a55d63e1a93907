// wm_device.cuh -- device helpers shared by the CUDA kernels of the engine:
// counter-based random numbers, uniform / normal transforms, bf16 operand
// rounding and the LSTM nonlinearities.
//
// Philox-4x32-10 follows Salmon, Moraes, Dror, Shaw, "Parallel random numbers:
// as easy as 1, 2, 3" (SC'11): ten rounds of two 32x32->64 multiplies (words 0
// and 2), the high halves xored into words 1 and 3 with the round key, the key
// advanced by the golden-ratio / sqrt(3) Weyl increments between rounds.
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

namespace wmk {

struct u32x4 { uint32_t x, y, z, w; };

// Stream layout (the header wm.h states the same): key = seed, counter =
// (episode lo, step, purpose << 24 | block, episode hi).
enum : uint32_t { RNG_COMPONENT = 0u, RNG_NORMAL = 1u, RNG_CONTROLLER = 2u };

__device__ __forceinline__ u32x4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                               uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t m0 = 0xD2511F53u, m1 = 0xCD9E8D57u;
        uint32_t hi0 = __umulhi(m0, c0), lo0 = m0 * c0;
        uint32_t hi1 = __umulhi(m1, c2), lo1 = m1 * c2;
        uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return {c0, c1, c2, c3};
}

__device__ __forceinline__ u32x4 rng_draw(unsigned long long seed, unsigned long long episode,
                                          uint32_t step, uint32_t purpose, uint32_t block) {
    return philox4x32_10((uint32_t)episode, step, (purpose << 24) | block,
                         (uint32_t)(episode >> 32), (uint32_t)seed, (uint32_t)(seed >> 32));
}

__device__ __forceinline__ uint32_t u32x4_get(const u32x4 &v, int i) {
    return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

// top 24 bits -> [0, 1), exact in fp32
__device__ __forceinline__ float to_uniform(uint32_t x) { return (float)(x >> 8) * 5.9604644775390625e-8f; }

// One Box-Muller normal: pair (x1, x2), second = false -> r cos, true -> r sin.
__device__ __forceinline__ float box_muller(uint32_t x1, uint32_t x2, bool second) {
    float u1 = to_uniform(x1), u2 = to_uniform(x2);
    float r = sqrtf(-2.0f * logf(1.0f - u1));
    float s, c;
    sincospif(2.0f * u2, &s, &c);
    return r * (second ? s : c);
}

// Both Box-Muller normals of a pair: c = r cos, s = r sin (the values box_muller returns).
__device__ __forceinline__ void box_muller2(uint32_t x1, uint32_t x2, float &c_out, float &s_out) {
    float u1 = to_uniform(x1), u2 = to_uniform(x2);
    float r = sqrtf(-2.0f * logf(1.0f - u1));
    float s, c;
    sincospif(2.0f * u2, &s, &c);
    c_out = r * c;
    s_out = r * s;
}

// The normal of latent dim d at (episode, step).
__device__ __forceinline__ float normal_for_dim(unsigned long long seed, unsigned long long ep,
                                                uint32_t step, int d) {
    u32x4 v = rng_draw(seed, ep, step, RNG_NORMAL, (uint32_t)(d >> 2));
    int pair = (d & 3) >> 1;
    return box_muller(pair ? v.z : v.x, pair ? v.w : v.y, (d & 1) != 0);
}

__device__ __forceinline__ float uniform_for_dim(unsigned long long seed, unsigned long long ep,
                                                 uint32_t step, int d) {
    u32x4 v = rng_draw(seed, ep, step, RNG_COMPONENT, (uint32_t)(d >> 2));
    return to_uniform(u32x4_get(v, d & 3));
}

// Records a device-side error in the status word unless one is already recorded
// (wm_sync returns the first).
__device__ __forceinline__ void report_status(int *status, int code) {
    if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ float round_bf16(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

__device__ __forceinline__ float sigmoidf_(float x) { return 1.0f / (1.0f + expf(-x)); }

}  // namespace wmk
