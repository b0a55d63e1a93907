// wm_returns.cu -- discounted returns of dream rollouts and each controller
// candidate's fitness (wm_returns).
//
//   G_t = r_t + gamma G_{t+1},  G_T = bootstrap (or 0);  a done step ends the sum
//   fitness[g] = mean of G_0 over the call's episodes of candidate g
//
// The objective the agent maximises is the expected discounted return (Sec. 3.1);
// CMA-ES ranks controller candidates by it (Sec. 3.4).  One thread per episode walks
// its steps backwards, so every access to the time-major [T, B] arrays is coalesced
// across the warp.  The recursion runs in fp64 (a few operations per (episode,
// step), far from any throughput limit), multiply and add rounded separately.
// The fitness of candidate g is summed by one block over the runs of E
// consecutive episodes that belong to g, in a fixed order (deterministic).
#include "wm_internal.h"

namespace {

__global__ void k_returns(int B, int T, double gamma, int stop_at_done, const float *__restrict__ r,
                          const uint8_t *__restrict__ d, const float *__restrict__ boot,
                          float *__restrict__ ret, double *__restrict__ g0) {
    for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < B; b += gridDim.x * blockDim.x) {
        double G = boot ? (double)boot[b] : 0.0;
        for (int t = T - 1; t >= 0; --t) {
            const size_t i = (size_t)t * B + b;
            if (stop_at_done && d[i]) G = 0.0;
            G = __dadd_rn((double)r[i], __dmul_rn(gamma, G));  // no FMA contraction: the
                                                                 // oracle's rounding exactly
            ret[i] = (float)G;
        }
        if (g0) g0[b] = G;
    }
}

// Block g: the mean G_0 of candidate g's episodes of this call.  Global episode e has
// candidate (e / E) mod P, so g owns the runs q = g, g + P, ... of E episodes.
__global__ void k_fitness(int B, unsigned long long ep0, int P, int E, const double *__restrict__ g0,
                          float *__restrict__ fitness) {
    __shared__ double s_sum[256];
    __shared__ long long s_n[256];
    const int g = blockIdx.x;
    const unsigned long long e_lo = ep0, e_hi = ep0 + (unsigned long long)B;  // [e_lo, e_hi)
    const unsigned long long q_lo = e_lo / E, q_hi = (e_hi + E - 1) / E;
    // first run of candidate g at or after q_lo
    unsigned long long q = q_lo + (unsigned long long)(((long long)g - (long long)(q_lo % P) + P) % P);
    double sum = 0.0;
    long long n = 0;
    for (; q < q_hi; q += P) {
        unsigned long long a = q * E, z = a + E;
        if (a < e_lo) a = e_lo;
        if (z > e_hi) z = e_hi;
        for (unsigned long long e = a + threadIdx.x; e < z; e += blockDim.x) {
            sum += g0[e - ep0];
            ++n;
        }
    }
    s_sum[threadIdx.x] = sum;
    s_n[threadIdx.x] = n;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) {
            s_sum[threadIdx.x] += s_sum[threadIdx.x + w];
            s_n[threadIdx.x] += s_n[threadIdx.x + w];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) fitness[g] = s_n[0] ? (float)(s_sum[0] / (double)s_n[0]) : 0.f;
}

}  // namespace

size_t wm_returns_ws(const wm_handle *, int B) { return ((size_t)B * 8 + 255) & ~(size_t)255; }

cudaError_t wm_returns_launch(const wm_handle *h, int B, int T, unsigned long long ep0, float gamma,
                              int stop_at_done, const float *rewards, const uint8_t *done,
                              const float *bootstrap, float *returns, float *fitness, void *ws,
                              cudaStream_t s) {
    double *g0 = (double *)ws;
    int launches = 0;
    if (B > 0) {
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        const int grid = (B + 255) / 256 < 1184 ? (B + 255) / 256 : 1184;
        k_returns<<<grid, 256, 0, s>>>(B, T, (double)gamma, stop_at_done, rewards, done, bootstrap, returns, g0);
        ++launches;
    }
    if (fitness) {
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        if (B > 0) {
            k_fitness<<<h->P, 256, 0, s>>>(B, ep0, h->P, h->E, g0, fitness);
        } else {
            cudaError_t e = cudaMemsetAsync(fitness, 0, (size_t)h->P * 4, s);
            if (e != cudaSuccess) return e;
        }
        ++launches;
    }
    h->last_launches = launches;
    return cudaGetLastError();
}
