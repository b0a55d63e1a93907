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

// Bit j of a mask row (null: every action valid).
__device__ __forceinline__ bool action_valid(const uint32_t *mw, int j) {
    return !mw || ((mw[j >> 5] >> (j & 31)) & 1u);
}

// One warp's controller choice over n logits (Sec. 3.4, masks of Sec. 3.1.3).
struct WarpSelect {
    bool sample;                     // tempered draw (else masked argmax)
    float tau;                       // controller temperature
    bool want_lp;                    // compute the log-prob of the choice
    unsigned long long seed, episode;
    uint32_t step;
};

// log pi(a) under softmax(l / tau) over the valid of n actions (every lane returns it)
__device__ inline float warp_logp(const float *l, int n, const uint32_t *mw, int a, float lmax, float tau,
                                  int ld = 1) {
    const int lane = threadIdx.x & 31;
    float S = 0.f;
    for (int j = lane; j < n; j += 32)
        if (action_valid(mw, j)) S += expf((l[j * ld] - lmax) / tau);
#pragma unroll
    for (int off = 16; off; off >>= 1) S += __shfl_xor_sync(0xffffffffu, S, off);
    return (l[a * ld] - lmax) / tau - logf(S);
}

// Masked argmax (lowest index on ties) or a tempered draw by inverse CDF with word `word` of
// the controller's Philox block, over the n logits l[j * ld] with mask words mw (or null).  Returns
// the choice (-1: nothing valid); with want_lp, *logp receives its log-prob under
// softmax(l / tau) over the valid actions (0 if none, or tau = 0).  Called by a full warp.
__device__ inline int warp_select(const WarpSelect &s, const float *l, int n, const uint32_t *mw, int word,
                                  float *logp, int ld = 1) {
    const int lane = threadIdx.x & 31;
    const int A = n;
    float bv = -INFINITY;
    int bi = -1;
    for (int j = lane; j < A; j += 32) {
        if (!action_valid(mw, j)) continue;
        float v = l[j * ld];
        if (bi < 0 || v > bv) { bv = v; bi = j; }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
        float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        bool take = oi >= 0 && (bi < 0 || ov > bv || (ov == bv && oi < bi));
        if (take) { bv = ov; bi = oi; }
    }
    *logp = 0.f;
    if (bi < 0) return bi;
    if (!s.sample) {
        if (s.want_lp && s.tau > 0.f) *logp = warp_logp(l, A, mw, bi, bv, s.tau, ld);
        return bi;
    }
    const float tau = s.tau;
    float S = 0.f;
    for (int j = lane; j < A; j += 32)
        if (action_valid(mw, j)) S += expf((l[j * ld] - bv) / tau);
#pragma unroll
    for (int off = 16; off; off >>= 1) S += __shfl_xor_sync(0xffffffffu, S, off);
    const u32x4 rc = rng_draw(s.seed, s.episode, s.step, RNG_CONTROLLER, 0);
    const float u = to_uniform(word ? rc.y : rc.x);
    const float target = u * S;
    float run = 0.f;
    int last = -1;
    for (int j0 = 0; j0 < A; j0 += 32) {
        int j = j0 + lane;
        bool ok = j < A && action_valid(mw, j);
        float sc = ok ? expf((l[j * ld] - bv) / tau) : 0.f;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            float o = __shfl_up_sync(0xffffffffu, sc, off);
            if (lane >= off) sc += o;
        }
        float cum = run + sc;
        unsigned hit = __ballot_sync(0xffffffffu, ok && target < cum);
        unsigned okm = __ballot_sync(0xffffffffu, ok);
        if (okm) last = j0 + 31 - __clz(okm);
        if (hit) {
            const int a = j0 + __ffs(hit) - 1;
            if (s.want_lp) *logp = (l[a * ld] - bv) / tau - logf(S);
            return a;
        }
        run += __shfl_sync(0xffffffffu, sc, 31);
    }
    if (s.want_lp && last >= 0) *logp = (l[last * ld] - bv) / tau - logf(S);
    return last;
}

// Records a device-side error in the status word unless one is already recorded
// (wm_sync returns the first).
__device__ __forceinline__ void report_status(int *status, int code) {
    if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ float round_bf16(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

__device__ __forceinline__ float sigmoidf_(float x) { return 1.0f / (1.0f + expf(-x)); }

}  // namespace wmk
