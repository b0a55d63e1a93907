// wm_step.cu -- the stepwise kernel family: four launches per dream step.
//
//   1. k_gemm        [z_t; h_t] x [W_z|W_h ; W_c]  -> gate pre-activations and
//                    controller logits (a1, a3 without the action row)
//   2. k_select_cell masked argmax / tempered draw of a_t (a2), the gathered
//                    action row W_a[a_t], the LSTM cell update (a3, a4)
//   3. k_gemm        h' x [W_mdn | w_rew | w_done]  -> head outputs (a5)
//   4. k_sample      per-dim temperature softmax, inverse-CDF component draw,
//                    Gaussian draw, reward / done / freeze (a6, a7, a8) -- or,
//                    in teacher-forced mode, the per-dim mixture NLL (a9)
//
// Every shape is supported (ragged tails are bounds-checked), fp32 SIMT FMA.
// This family is the reference point the fused and tensor-core families are
// compared against, and the fallback for shapes they do not take.
#include <math.h>

#include "wm_device.cuh"
#include "wm_internal.h"

using namespace wmk;

namespace {

constexpr int GBM = 64, GBN = 64, GBK = 16;

// C[m,n] = bias[n] + sum_k A(m,k) W[k,n];  A(m,k) = A1[m,k] for k < K1, else A2[m,k-K1].
template <bool ROUND>
__global__ void __launch_bounds__(256) k_gemm(int M, int N, int K1, int K2,
                                              const float *__restrict__ A1, long lda1,
                                              const float *__restrict__ A2, long lda2,
                                              const float *__restrict__ W, long ldw,
                                              const float *__restrict__ bias,
                                              float *__restrict__ C, long ldc) {
    __shared__ float As[GBK][GBM + 4];
    __shared__ float Ws[GBK][GBN + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const long m0 = (long)blockIdx.y * GBM;
    const int n0 = blockIdx.x * GBN;
    const int K = K1 + K2;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < K; k0 += GBK) {
        for (int i = tid; i < GBM * GBK; i += 256) {
            int r = i / GBK, kk = i % GBK;
            long m = m0 + r;
            int k = k0 + kk;
            float v = 0.f;
            if (m < M && k < K) v = (k < K1) ? A1[m * lda1 + k] : A2[m * lda2 + (k - K1)];
            if (ROUND) v = round_bf16(v);
            As[kk][r] = v;
        }
        for (int i = tid; i < GBK * GBN; i += 256) {
            int kk = i / GBN, c = i % GBN;
            int k = k0 + kk, n = n0 + c;
            Ws[kk][c] = (k < K && n < N) ? W[(long)k * ldw + n] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < GBK; ++kk) {
            float a[4], w[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) w[j] = Ws[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        long m = m0 + ty * 4 + i;
        if (m >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            int n = n0 + tx * 4 + j;
            if (n < N) C[m * ldc + n] = acc[i][j] + bias[n];
        }
    }
}

struct StepParams {
    int B, Z, A, H, K, M, T;
    int teacher;
    int t;
    uint32_t step;
    unsigned long long ep0, seed;
    int ctrl_sample, sigma_sqrt_tau, done_terminates, noop_terminates;
    float ctrl_tau, mdn_tau;
    const float *G;       // [B, ldg]: 4H gate pre-activations (+bias), then A logits
    long ldg;
    const float *Wa;      // [A, 4H]
    const uint32_t *mask; // [T, B, W] or null
    const int32_t *act_in;
    int32_t *act_out;
    float *h, *c;
    uint8_t *frozen;
    float *h_seq, *c_seq;
    const float *heads;   // [B, M+2]
    long ldh;
    const float *z_cur;   // [B, Z] z_t
    float *z_next;        // [B, Z] z_{t+1} (rollout)
    const float *z_target;// [B, Z] z_{t+1} (teacher)
    float *rewards;
    uint8_t *done;
    float *mdn_seq;
    uint8_t *comp_seq;
    const int32_t *lengths;
    double *nll_acc;
    int *status;          // device status word (out-of-range teacher inputs)
    // shaped reward (Sec. 3.1.4, Eq. 2): the heads' columns M+2, M+3 predict runtime and
    // memory accesses; rt / mem carry each episode's last predictions
    int reward_mode;
    float alpha, beta, invalid_reward;
    float *rt, *mem;
    float *rt_seq, *mem_seq;
    // controller population: episode e acts with candidate (e / E) mod P (Wp, bp when P > 1)
    int P, E;
    const float *Wp, *bp;
    float *logp_seq;      // log pi(a_t | z_t, h_t) of the action taken (optional)
    float *value_seq;     // value head, heads column value_col (optional)
    int value_col;
    // hierarchical action: n_xfers xfer logits, then A - n_xfers location logits
    int n_xfers;
    const uint32_t *loc_mask;  // [T, B, NX, WL] or null
    int32_t *loc_out;          // [T, B] the location taken (optional)
    int32_t *loc_cur;          // [B] this step's location (workspace)
};

// a1 for a controller population: the logits of each episode's candidate into the
// controller columns of G.  One block per episode, the input [z_t; h_t] staged in
// shared memory (bf16-rounded on the bf16 path), one column per thread.
template <bool ROUND>
__global__ void __launch_bounds__(128) k_ctrl_pop(StepParams p, const float *__restrict__ z) {
    extern __shared__ float xs[];
    const int b = blockIdx.x, Z = p.Z, H = p.H, A = p.A, KX = Z + H;
    for (int i = threadIdx.x; i < KX; i += blockDim.x) {
        float v = i < Z ? z[(size_t)b * Z + i] : p.h[(size_t)b * H + (i - Z)];
        xs[i] = ROUND ? round_bf16(v) : v;
    }
    __syncthreads();
    const size_t cand = (size_t)(((p.ep0 + b) / (unsigned long long)p.E) % (unsigned long long)p.P);
    const float *W = p.Wp + cand * KX * A, *bias = p.bp + cand * A;
    float *out = const_cast<float *>(p.G) + (size_t)b * p.ldg + 4 * H;
    for (int j = threadIdx.x; j < A; j += blockDim.x) {
        float acc = 0.f;
        for (int i = 0; i < KX; ++i) acc = fmaf(xs[i], W[(size_t)i * A + j], acc);
        out[j] = acc + bias[j];
    }
}

// a2 on one warp over the n logits l: the shared masked argmax / tempered draw.
__device__ int select_warp(const StepParams &p, const float *l, int n, const uint32_t *mw, int b, int word,
                           float *logp) {
    WarpSelect ws;
    ws.sample = p.ctrl_sample && p.ctrl_tau > 0.f;
    ws.tau = p.ctrl_tau;
    ws.want_lp = p.logp_seq != nullptr;
    ws.seed = p.seed;
    ws.episode = p.ep0 + b;
    ws.step = p.step;
    return warp_select(ws, l, n, mw, word, logp);
}

// The step's action: one flat choice of A, or (Sec. 3.1.3) the xfer among the first NX
// logits, then the location among the other L under the chosen xfer's location mask.
// Returns the action (the xfer); *loc receives the location (-1: none), *logp the log-prob
// of the whole action.
__device__ int select_action_warp(const StepParams &p, int b, int *loc, float *logp) {
    const float *l = p.G + (long)b * p.ldg + 4 * p.H;
    const int A = p.A, W = (A + 31) >> 5, NX = p.n_xfers;
    const uint32_t *mw = p.mask ? p.mask + ((size_t)p.t * p.B + b) * W : nullptr;
    *loc = -1;
    if (NX == 0) return select_warp(p, l, A, mw, b, 0, logp);
    const int L = A - NX, WL = (L + 31) >> 5;
    const int x = select_warp(p, l, NX, mw, b, 0, logp);
    if (x >= 0 && x != NX - 1) {
        const uint32_t *lmw = p.loc_mask ? p.loc_mask + (((size_t)p.t * p.B + b) * NX + x) * WL : nullptr;
        float lpl = 0.f;
        *loc = select_warp(p, l + NX, L, lmw, b, 1, &lpl);
        *logp += lpl;
    }
    return x;
}

__global__ void __launch_bounds__(256) k_select_cell(StepParams p) {
    const int b = blockIdx.x;
    __shared__ int s_a, s_a2;
    const bool fz = p.frozen[b] != 0;
    if (threadIdx.x < 32) {
        int a, loc = -1;
        float lp = 0.f;
        if (fz) {
            a = -1;
        } else if (p.teacher) {
            a = p.act_in[(size_t)p.t * p.B + b];
            if (a >= p.A) report_status(p.status, WM_ERR_INVALID_ARG);
            if (a >= p.A || a < 0) a = -1;
        } else {
            a = select_action_warp(p, b, &loc, &lp);
        }
        if (threadIdx.x == 0) {
            s_a = a;
            s_a2 = loc >= 0 ? p.n_xfers + loc : -1;  // the location's action row
            if (!p.teacher) p.act_out[(size_t)p.t * p.B + b] = a;
            if (!p.teacher && p.logp_seq) p.logp_seq[(size_t)p.t * p.B + b] = lp;
            if (p.n_xfers > 0 && !p.teacher) {
                p.loc_cur[b] = loc;
                if (p.loc_out) p.loc_out[(size_t)p.t * p.B + b] = loc;
            }
        }
    }
    __syncthreads();
    const int a = s_a, a2 = s_a2, H = p.H;
    const float *g = p.G + (long)b * p.ldg;
    const float *wa = a >= 0 ? p.Wa + (size_t)a * 4 * H : nullptr;
    const float *wa2 = a2 >= 0 ? p.Wa + (size_t)a2 * 4 * H : nullptr;
    for (int u = threadIdx.x; u < H; u += blockDim.x) {
        const size_t i = (size_t)b * H + u;
        float hv, cv;
        if (fz) {
            hv = p.h[i];
            cv = p.c[i];
        } else {
            float gi = g[u], gf = g[H + u], gg = g[2 * H + u], go = g[3 * H + u];
            if (wa) { gi += wa[u]; gf += wa[H + u]; gg += wa[2 * H + u]; go += wa[3 * H + u]; }
            if (wa2) { gi += wa2[u]; gf += wa2[H + u]; gg += wa2[2 * H + u]; go += wa2[3 * H + u]; }
            cv = sigmoidf_(gf) * p.c[i] + sigmoidf_(gi) * tanhf(gg);
            hv = sigmoidf_(go) * tanhf(cv);
            p.c[i] = cv;
            p.h[i] = hv;
        }
        const size_t o = ((size_t)p.t * p.B + b) * H + u;
        if (p.h_seq) p.h_seq[o] = hv;
        if (p.c_seq) p.c_seq[o] = cv;
    }
}

constexpr float HALF_LOG_2PI = 0.91893853320467274178f;

// a9 for one dim in fp32 (log-sum-exp over the K components).
__device__ float mixture_nll_dim(const float *row, int K, int KZ, int d, float x) {
    const float *lg = row + d * K, *mu = row + KZ + d * K, *ls = row + 2 * KZ + d * K;
    float m = -INFINITY;
    for (int k = 0; k < K; ++k) m = fmaxf(m, lg[k]);
    float s = 0.f;
    for (int k = 0; k < K; ++k) s += expf(lg[k] - m);
    const float lse = m + logf(s);
    float lp[32];
    float tmax = -INFINITY;
    for (int k = 0; k < K; ++k) {
        float zs = (x - mu[k]) * expf(-ls[k]);
        lp[k] = (lg[k] - lse) - 0.5f * zs * zs - ls[k] - HALF_LOG_2PI;
        tmax = fmaxf(tmax, lp[k]);
    }
    float acc = 0.f;
    for (int k = 0; k < K; ++k) acc += expf(lp[k] - tmax);
    return -(tmax + logf(acc));
}

__global__ void __launch_bounds__(128) k_sample(StepParams p) {
    const int b = blockIdx.x;
    const bool fz = p.frozen[b] != 0;
    const int Z = p.Z, K = p.K, M = p.M, KZ = K * Z;
    const float *row = p.heads + (long)b * p.ldh;
    const size_t tb = (size_t)p.t * p.B + b;
    const unsigned long long ep = p.ep0 + b;
    float part = 0.f;
    for (int d = threadIdx.x; d < Z; d += blockDim.x) {
        const size_t zi = (size_t)b * Z + d;
        if (p.teacher) {
            part += mixture_nll_dim(row, K, KZ, d, p.z_target[zi]);
            if (p.mdn_seq) {
                float *ms = p.mdn_seq + tb * M;
                for (int k = 0; k < K; ++k) {
                    ms[d * K + k] = row[d * K + k];
                    ms[KZ + d * K + k] = row[KZ + d * K + k];
                    ms[2 * KZ + d * K + k] = row[2 * KZ + d * K + k];
                }
            }
            continue;
        }
        if (fz) {
            p.z_next[zi] = p.z_cur[zi];
            if (p.mdn_seq) {
                float *ms = p.mdn_seq + tb * M;
                for (int k = 0; k < K; ++k) ms[d * K + k] = ms[KZ + d * K + k] = ms[2 * KZ + d * K + k] = 0.f;
            }
            if (p.comp_seq) p.comp_seq[tb * Z + d] = 255;
            continue;
        }
        const float *lg = row + d * K, *mu = row + KZ + d * K, *ls = row + 2 * KZ + d * K;
        int kc;
        float z;
        if (!(p.mdn_tau > 0.f)) {
            kc = 0;
            for (int k = 1; k < K; ++k) if (lg[k] > lg[kc]) kc = k;
            z = mu[kc];
        } else {
            const float tau = p.mdn_tau;
            float m = -INFINITY;
            for (int k = 0; k < K; ++k) m = fmaxf(m, lg[k] / tau);
            float pk[32], s = 0.f;
            for (int k = 0; k < K; ++k) { pk[k] = expf(lg[k] / tau - m); s += pk[k]; }
            const float u = uniform_for_dim(p.seed, ep, p.step, d);
            kc = K - 1;
            float cum = 0.f;
            for (int k = 0; k < K - 1; ++k) {
                cum += pk[k] / s;
                if (u < cum) { kc = k; break; }
            }
            const float eps = normal_for_dim(p.seed, ep, p.step, d);
            const float scale = p.sigma_sqrt_tau ? sqrtf(tau) : 1.f;
            z = mu[kc] + expf(ls[kc]) * scale * eps;
        }
        p.z_next[zi] = z;
        if (p.comp_seq) p.comp_seq[tb * Z + d] = (uint8_t)kc;
        if (p.mdn_seq) {
            float *ms = p.mdn_seq + tb * M;
            for (int k = 0; k < K; ++k) {
                ms[d * K + k] = lg[k];
                ms[KZ + d * K + k] = mu[k];
                ms[2 * KZ + d * K + k] = ls[k];
            }
        }
    }
    if (p.teacher) {
        __shared__ float red[4];
#pragma unroll
        for (int off = 16; off; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
        __syncthreads();
        if (threadIdx.x == 0) {
            float tot = 0.f;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
            int len = p.lengths ? p.lengths[b] : p.T;
            if (p.t == 0 && (len < 0 || len > p.T)) report_status(p.status, WM_ERR_INVALID_ARG);
            if (p.t < len) p.nll_acc[b] += (double)tot;
        }
        return;
    }
    __syncthreads();  // every thread has read frozen[b] before it may change
    if (threadIdx.x == 0) {
        const bool shaped = p.reward_mode == WM_REWARD_SHAPED;
        if (fz) {
            p.rewards[tb] = 0.f;
            p.done[tb] = 1;
        } else {
            float r = row[M];
            const float dl = row[M + 1];
            const int a = p.act_out[tb];
            const int noop_a = p.n_xfers > 0 ? p.n_xfers - 1 : p.A - 1;
            const bool noop = p.noop_terminates && a == noop_a;
            if (shaped) {  // Eq. 2 on the predictions entering and leaving the step
                const float rt = row[M + 2], mem = row[M + 3];
                // valid: an action was taken (and, for an xfer, a location)
                const bool ok = a >= 0 && (p.n_xfers == 0 || a == noop_a || p.loc_cur[b] >= 0);
                r = ok ? p.alpha * (p.rt[b] - rt) + p.beta * (p.mem[b] - mem) : p.invalid_reward;
                p.rt[b] = rt;
                p.mem[b] = mem;
            }
            p.rewards[tb] = r;
            p.done[tb] = (dl > 0.f || noop) ? 1 : 0;
            if ((p.done_terminates && dl > 0.f) || noop) p.frozen[b] = 1;
        }
        if (shaped && p.rt_seq) p.rt_seq[tb] = p.rt[b];
        if (shaped && p.mem_seq) p.mem_seq[tb] = p.mem[b];
        if (p.value_seq) p.value_seq[tb] = fz ? 0.f : row[p.value_col];
    }
}

__global__ void k_init_state(int B, int H, int Z, const float *h0, const float *c0, const uint8_t *done0,
                             const float *z0, float *h, float *c, uint8_t *frozen, float *z_out,
                             double *nll_acc, const float *rt0, const float *mem0, float *rt, float *mem) {
    const size_t n = (size_t)B * H;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        h[i] = h0 ? h0[i] : 0.f;
        c[i] = c0 ? c0[i] : 0.f;
    }
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < (size_t)B; i += (size_t)gridDim.x * blockDim.x) {
        if (frozen) frozen[i] = done0 ? (done0[i] != 0) : 0;
        if (nll_acc) nll_acc[i] = 0.0;
        if (rt0) {
            rt[i] = rt0[i];
            mem[i] = mem0[i];
        }
    }
    if (z_out)
        for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < (size_t)B * Z; i += (size_t)gridDim.x * blockDim.x)
            z_out[i] = z0[i];
}

__global__ void k_finish(int B, int H, const float *h, const float *c, float *h_final, float *c_final,
                         const double *nll_acc, float *nll) {
    const size_t n = (size_t)B * H;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        if (h_final) h_final[i] = h[i];
        if (c_final) c_final[i] = c[i];
    }
    if (nll)
        for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < (size_t)B; i += (size_t)gridDim.x * blockDim.x)
            nll[i] = (float)nll_acc[i];
}

inline size_t align_up(size_t x) { return (x + 255) & ~(size_t)255; }

struct StepWs {
    float *G, *heads, *h, *c;
    float *rt, *mem;  // shaped reward: each episode's last predictions
    int32_t *loc;     // hierarchical action: the step's location
    uint8_t *frozen;
    double *nll_acc;
};

size_t step_ws_bytes(const wm_handle *hd, int B, bool teacher) {
    const wm_config &c = hd->cfg;
    const size_t H = c.h_dim, A = c.a_dim, M = hd->M, NR = hd->NR;
    size_t s = 0;
    s += align_up((size_t)B * (4 * H + A) * 4);
    s += align_up((size_t)B * (M + NR) * 4);
    s += 2 * align_up((size_t)B * H * 4);
    if (c.reward_mode == WM_REWARD_SHAPED) s += 2 * align_up((size_t)B * 4);
    s += align_up((size_t)B * 4);
    s += align_up((size_t)B);
    if (teacher) s += align_up((size_t)B * 8);
    return s;
}

StepWs carve(const wm_handle *hd, int B, void *ws, bool teacher) {
    const wm_config &c = hd->cfg;
    const size_t H = c.h_dim, A = c.a_dim, M = hd->M, NR = hd->NR;
    char *p = (char *)ws;
    StepWs w{};
    w.G = (float *)p; p += align_up((size_t)B * (4 * H + A) * 4);
    w.heads = (float *)p; p += align_up((size_t)B * (M + NR) * 4);
    w.h = (float *)p; p += align_up((size_t)B * H * 4);
    w.c = (float *)p; p += align_up((size_t)B * H * 4);
    if (c.reward_mode == WM_REWARD_SHAPED) {
        w.rt = (float *)p; p += align_up((size_t)B * 4);
        w.mem = (float *)p; p += align_up((size_t)B * 4);
    }
    w.loc = (int32_t *)p; p += align_up((size_t)B * 4);
    w.frozen = (uint8_t *)p; p += align_up((size_t)B);
    w.nll_acc = teacher ? (double *)p : nullptr;
    return w;
}

void launch_gemm(const wm_handle *hd, bool round, int M, int N, int K1, int K2, const float *A1, long lda1,
                 const float *A2, long lda2, const float *W, long ldw, const float *bias, float *C, long ldc,
                 cudaStream_t s) {
    wm_ktime kt(hd, WM_KERNEL_STEP_GEMM, s);
    dim3 grid((N + GBN - 1) / GBN, (M + GBM - 1) / GBM);
    if (round)
        k_gemm<true><<<grid, 256, 0, s>>>(M, N, K1, K2, A1, lda1, A2, lda2, W, ldw, bias, C, ldc);
    else
        k_gemm<false><<<grid, 256, 0, s>>>(M, N, K1, K2, A1, lda1, A2, lda2, W, ldw, bias, C, ldc);
}

int grid_1d(size_t n) {
    size_t g = (n + 255) / 256;
    if (g > 4096) g = 4096;
    return g < 1 ? 1 : (int)g;
}

StepParams base_params(const wm_handle *hd, int B, int T, const StepWs &w) {
    const wm_config &c = hd->cfg;
    StepParams p{};
    p.B = B; p.Z = c.z_dim; p.A = c.a_dim; p.H = c.h_dim; p.K = c.k_mix; p.M = hd->M; p.T = T;
    p.seed = c.seed;
    p.ctrl_sample = c.ctrl_sample; p.ctrl_tau = c.ctrl_tau; p.mdn_tau = c.mdn_tau;
    p.sigma_sqrt_tau = c.sigma_sqrt_tau; p.done_terminates = c.done_terminates;
    p.noop_terminates = c.noop_terminates;
    p.G = w.G; p.ldg = 4L * c.h_dim + c.a_dim;
    p.Wa = hd->step.Wa;
    p.h = w.h; p.c = w.c; p.frozen = w.frozen;
    p.heads = w.heads; p.ldh = hd->M + hd->NR;
    p.status = hd->status;
    p.reward_mode = c.reward_mode;
    p.alpha = c.reward_alpha; p.beta = c.reward_beta; p.invalid_reward = c.invalid_reward;
    p.rt = w.rt; p.mem = w.mem;
    p.P = hd->P; p.E = hd->E;
    p.Wp = hd->step.Wp; p.bp = hd->step.bp;
    p.value_col = hd->M + hd->NR - 1;
    p.n_xfers = c.n_xfers;
    p.loc_cur = w.loc;
    return p;
}

}  // namespace

size_t wm_step_rollout_ws(const wm_handle *h, int B) { return step_ws_bytes(h, B, false); }
size_t wm_step_nll_ws(const wm_handle *h, int N) { return step_ws_bytes(h, N, true); }

cudaError_t wm_step_rollout(const wm_handle *hd, const wm_rollout_dev &a, void *ws, cudaStream_t s) {
    const wm_config &c = hd->cfg;
    const int B = a.B, T = a.T, Z = c.z_dim, H = c.h_dim, A = c.a_dim;
    if (B == 0) return cudaSuccess;
    StepWs w = carve(hd, B, ws, false);
    const bool round = c.precision == WM_BF16;
    {
        wm_ktime kt(hd, WM_KERNEL_AUX, s);
        const bool shaped = c.reward_mode == WM_REWARD_SHAPED;
        k_init_state<<<grid_1d((size_t)B * H), 256, 0, s>>>(B, H, Z, a.h0, a.c0, a.done0, a.z0, w.h, w.c,
                                                             w.frozen, a.z_out, nullptr,
                                                             shaped ? a.rt0 : nullptr, shaped ? a.mem0 : nullptr,
                                                             w.rt, w.mem);
    }
    StepParams p = base_params(hd, B, T, w);
    p.teacher = 0;
    p.ep0 = a.ep0;
    p.mask = a.mask;
    p.act_out = a.actions;
    p.h_seq = a.h_seq; p.c_seq = a.c_seq;
    p.rewards = a.rewards; p.done = a.done; p.mdn_seq = a.mdn_seq; p.comp_seq = a.comp_seq;
    p.rt_seq = a.rt_seq; p.mem_seq = a.mem_seq;
    p.logp_seq = a.logp_seq;
    p.value_seq = c.value_head ? a.value_seq : nullptr;
    p.loc_mask = a.loc_mask;
    p.loc_out = a.loc_actions;
    const int NH = hd->M + hd->NR;  // head GEMM columns
    const bool pop = hd->P > 1;     // controller logits per candidate, in k_ctrl_pop
    for (int t = 0; t < T; ++t) {
        p.t = t;
        p.step = a.t0 + (uint32_t)t;
        p.z_cur = a.z_out + (size_t)t * B * Z;
        p.z_next = a.z_out + (size_t)(t + 1) * B * Z;
        launch_gemm(hd, round, B, pop ? 4 * H : 4 * H + A, Z, H, p.z_cur, Z, w.h, H, hd->step.Wg, 4L * H + A,
                    hd->step.bg, w.G, 4L * H + A, s);
        if (pop) {
            wm_ktime kt(hd, WM_KERNEL_STEP_GEMM, s);
            const size_t sm = (size_t)(Z + H) * 4;
            if (round) k_ctrl_pop<true><<<B, 128, sm, s>>>(p, p.z_cur);
            else k_ctrl_pop<false><<<B, 128, sm, s>>>(p, p.z_cur);
        }
        {
            wm_ktime kt(hd, WM_KERNEL_STEP_CELL, s);
            k_select_cell<<<B, 256, 0, s>>>(p);
        }
        launch_gemm(hd, round, B, NH, H, 0, w.h, H, nullptr, 0, hd->step.Wh, NH, hd->step.bh, w.heads, NH, s);
        {
            wm_ktime kt(hd, WM_KERNEL_STEP_SAMPLE, s);
            k_sample<<<B, 128, 0, s>>>(p);
        }
    }
    if (a.h_final || a.c_final) {
        wm_ktime kt(hd, WM_KERNEL_AUX, s);
        k_finish<<<grid_1d((size_t)B * H), 256, 0, s>>>(B, H, w.h, w.c, a.h_final, a.c_final, nullptr, nullptr);
    }
    return cudaGetLastError();
}

cudaError_t wm_step_nll(const wm_handle *hd, const wm_nll_dev &a, void *ws, cudaStream_t s) {
    const wm_config &c = hd->cfg;
    const int N = a.N, T = a.T, Z = c.z_dim, H = c.h_dim, A = c.a_dim;
    if (N == 0) return cudaSuccess;
    StepWs w = carve(hd, N, ws, true);
    const bool round = c.precision == WM_BF16;
    {
        wm_ktime kt(hd, WM_KERNEL_AUX, s);
        k_init_state<<<grid_1d((size_t)N * H), 256, 0, s>>>(N, H, Z, nullptr, nullptr, nullptr, nullptr, w.h,
                                                             w.c, w.frozen, nullptr, w.nll_acc, nullptr,
                                                             nullptr, nullptr, nullptr);
    }
    StepParams p = base_params(hd, N, T, w);
    p.teacher = 1;
    p.act_in = a.actions;
    p.h_seq = a.h_seq; p.c_seq = a.c_seq; p.mdn_seq = a.mdn_seq;
    p.lengths = a.lengths;
    p.nll_acc = w.nll_acc;
    for (int t = 0; t < T; ++t) {
        p.t = t;
        p.z_cur = a.z_seq + (size_t)t * N * Z;
        p.z_target = a.z_seq + (size_t)(t + 1) * N * Z;
        launch_gemm(hd, round, N, 4 * H, Z, H, p.z_cur, Z, w.h, H, hd->step.Wg, 4L * H + A, hd->step.bg, w.G,
                    4L * H + A, s);
        {
            wm_ktime kt(hd, WM_KERNEL_STEP_CELL, s);
            k_select_cell<<<N, 256, 0, s>>>(p);
        }
        launch_gemm(hd, round, N, hd->M + hd->NR, H, 0, w.h, H, nullptr, 0, hd->step.Wh, hd->M + hd->NR,
                    hd->step.bh, w.heads, hd->M + hd->NR, s);
        {
            wm_ktime kt(hd, WM_KERNEL_STEP_SAMPLE, s);
            k_sample<<<N, 128, 0, s>>>(p);
        }
    }
    {
        wm_ktime kt(hd, WM_KERNEL_AUX, s);
        k_finish<<<grid_1d((size_t)N * H), 256, 0, s>>>(N, H, w.h, w.c, nullptr, nullptr, w.nll_acc, a.nll);
    }
    return cudaGetLastError();
}
