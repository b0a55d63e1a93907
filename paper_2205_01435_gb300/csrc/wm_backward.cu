// wm_backward.cu -- wm_mdn_nll_backward: the world model's training step, the gradient
// of the teacher-forced mixture NLL (Sec. 4.7) by backpropagation through time
// (Sec. 3.3.2).
//
// Rows are (step, sequence) pairs r = t N + n, time-major like every [T, N, ...] array of
// the library.  Everything that does not depend on the recurrence is batched over all
// N T rows:
//   forward      the teacher-forced pass of the kernel family wm_mdn_nll picks, keeping
//                h_t, c_t and the head outputs of every row
//   X, Y         the GEMM operands of every row, X = [op(z_t); op(h_{t-1})], Y = op(h_t)
//   gates        G = X W_zh (one GEMM) + b + W_a[a_t], then sigma / tanh  (k_bw_gates)
//   dMD          d NLL / d [logit | mu | log sigma] of every counted row     (k_bw_mdn)
//   dY           dMD W_mdn^T (one GEMM): the heads' share of d loss / d h_t
// then the recurrence, t = T-1 .. 0:
//   dG_t         the cell's backward step from dY_t + dH and the carried dc  (k_bw_cell)
//   dH           dG_t W_h^T (one GEMM on N rows): d loss / d h_{t-1}
// and the weight gradients, batched again:
//   dW_z, dW_h   X^T dG (two GEMMs writing the z and h rows of the output)
//   dW_a         per action, the sum of the dG rows that took it          (k_bw_arows)
//   dW_mdn       Y^T dMD (one GEMM);  db_lstm, db_mdn  column sums          (k_bw_colsum)
// The plain GEMMs are cuBLAS calls (bf16 operands and fp32 accumulation on the bf16 path;
// on the fp32 path the library's fp32 emulation, and for the recurrence's dH one bf16 GEMM
// over the operands' hi and lo parts, see k_bw_split3); the rest are the kernels below.
// Every reduction has a fixed order, so results are bit-reproducible.
#include <cublas_v2.h>
#include <cuda_bf16.h>
#include <math.h>

#include "wm_internal.h"

namespace {

constexpr int CHUNKS = 16;  // row chunks of the two-level reductions

template <class T> __device__ __forceinline__ T to_op(float v);
template <> __device__ __forceinline__ float to_op<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 to_op<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// X [NT, Z+H] = [z_t | h_{t-1}] and Y [NT, H] = h_t, in the GEMM operand type (bf16: RNE,
// the forward's operand rounding)
// (a block per row at a time, the row's columns over its threads: no 64-bit divisions)
template <class T>
__global__ void k_bw_build(int N, int TT, int Z, int H, const float *__restrict__ z_seq,
                           const float *__restrict__ hs, T *__restrict__ X, T *__restrict__ Y) {
    const int KX = Z + H;
    const size_t NT = (size_t)N * TT;
    for (size_t r = blockIdx.x; r < NT; r += gridDim.x) {
        const float *hp = r >= (size_t)N ? hs + (r - N) * H : nullptr;  // h_{-1} = 0
        for (int k = threadIdx.x; k < KX; k += blockDim.x) {
            const float v = k < Z ? z_seq[r * Z + k] : (hp ? hp[k - Z] : 0.f);
            X[r * KX + k] = to_op<T>(v);
        }
        for (int k = threadIdx.x; k < H; k += blockDim.x) Y[r * H + k] = to_op<T>(hs[r * H + k]);
    }
}

// gate pre-activations + bias + the action row -> i, f, g, o (in place); a block per row at
// a time, four columns per thread
__global__ void k_bw_gates(size_t NT, int N, int H, int A, float *__restrict__ G, const int32_t *__restrict__ act,
                           const float *__restrict__ Wa, const float *__restrict__ bias) {
    const int H4 = 4 * H;
    for (size_t r = blockIdx.x; r < NT; r += gridDim.x) {
        const int a = act[r];
        const float *wa = (a >= 0 && a < A) ? Wa + (size_t)a * H4 : nullptr;
        float4 *g4 = reinterpret_cast<float4 *>(G + r * H4);
        for (int c4 = threadIdx.x; c4 < H4 / 4; c4 += blockDim.x) {
            const int col = 4 * c4;
            float4 v = g4[c4];
            float x[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                float u = x[j] + bias[col + j];
                if (wa) u += wa[col + j];
                const bool cand = col + j >= 2 * H && col + j < 3 * H;  // the g gate: tanh
                x[j] = cand ? tanhf(u) : 1.f / (1.f + expf(-u));
            }
            g4[c4] = make_float4(x[0], x[1], x[2], x[3]);
        }
    }
}

// d NLL / d [logit | mu | log sigma] of one row's latent dim d (0 past the row's length)
template <class T>
__global__ void k_bw_mdn(int N, int TT, int Z, int K, const float *__restrict__ md, const float *__restrict__ z_seq,
                         const int32_t *__restrict__ lengths, float *__restrict__ dmd, T *__restrict__ dmd_op) {
    const int KZ = K * Z, M = 3 * KZ;
    const size_t NT = (size_t)N * TT;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < NT * Z; i += (size_t)gridDim.x * blockDim.x) {
        const size_t r = i / Z;
        const int d = (int)(i % Z), t = (int)(r / N), n = (int)(r % N);
        int len = lengths ? lengths[n] : TT;
        len = len < 0 ? 0 : (len > TT ? TT : len);
        const float *row = md + r * M;
        float *out = dmd + r * M;
        T *oop = dmd_op + r * M;
        if (t >= len) {
            for (int k = 0; k < K; ++k)
                for (int p = 0; p < 3; ++p) {
                    out[p * KZ + d * K + k] = 0.f;
                    oop[p * KZ + d * K + k] = to_op<T>(0.f);
                }
            continue;
        }
        const float x = z_seq[(r + N) * Z + d];  // the target z_{t+1}
        const float *lg = row + d * K, *mu = row + KZ + d * K, *ls = row + 2 * KZ + d * K;
        float lmax = -INFINITY, s = 0.f, term[32], tmax = -INFINITY, acc = 0.f;
        for (int k = 0; k < K; ++k) lmax = fmaxf(lmax, lg[k]);
        for (int k = 0; k < K; ++k) s += expf(lg[k] - lmax);
        const float logz = lmax + logf(s);
        for (int k = 0; k < K; ++k) {
            const float zs = (x - mu[k]) * expf(-ls[k]);
            term[k] = (lg[k] - logz) - 0.5f * zs * zs - ls[k] - 0.91893853320467274178f;
            tmax = fmaxf(tmax, term[k]);
        }
        for (int k = 0; k < K; ++k) acc += expf(term[k] - tmax);
        const float lse = tmax + logf(acc);
        for (int k = 0; k < K; ++k) {
            const float pi = expf(lg[k] - logz), gam = expf(term[k] - lse);
            const float is = expf(-ls[k]), zs = (x - mu[k]) * is;
            const float v0 = pi - gam, v1 = -gam * zs * is, v2 = gam * (1.f - zs * zs);
            out[d * K + k] = v0;
            out[KZ + d * K + k] = v1;
            out[2 * KZ + d * K + k] = v2;
            oop[d * K + k] = to_op<T>(v0);
            oop[KZ + d * K + k] = to_op<T>(v1);
            oop[2 * KZ + d * K + k] = to_op<T>(v2);
        }
    }
}

// The cell's backward step at t for N rows: dh = dY_t + dH (from step t + 1), and
//   dc = dh o (1 - tanh^2 c_t) + dc_carried;  dG = [dc g i(1-i) | dc c_{t-1} f(1-f) |
//   dc i (1-g^2) | dh tanh(c_t) o(1-o)];  dc_carried <- dc f.
template <class T>
__global__ void k_bw_cell(int N, int H, int t, int first, const float *__restrict__ act, const float *__restrict__ cs,
                          const float *__restrict__ dY, const float *__restrict__ dH, float *__restrict__ dC,
                          float *__restrict__ dG, T *__restrict__ dG_op, __nv_bfloat16 *__restrict__ dG3) {
    const size_t base = (size_t)t * N;
    const int u = blockIdx.x * blockDim.x + threadIdx.x;  // unit; rows n over the grid's y
    if (u >= H) return;
    for (size_t n = blockIdx.y; n < (size_t)N; n += gridDim.y) {
        const size_t i = n * H + u;
        const size_t r = base + n;
        const float *a = act + r * 4 * H;
        const float ig = a[u], fg = a[H + u], gg = a[2 * H + u], og = a[3 * H + u];
        const float c = cs[r * H + u], cp = t > 0 ? cs[(r - N) * H + u] : 0.f;
        const float dh = dY[r * H + u] + (first ? 0.f : dH[i]);
        const float tc = tanhf(c);
        const float dc = dh * og * (1.f - tc * tc) + (first ? 0.f : dC[i]);
        const float g0 = dc * gg * ig * (1.f - ig), g1 = dc * cp * fg * (1.f - fg);
        const float g2 = dc * ig * (1.f - gg * gg), g3 = dh * tc * og * (1.f - og);
        float *o = dG + r * 4 * H;
        T *oo = dG_op + r * 4 * H;
        o[u] = g0; o[H + u] = g1; o[2 * H + u] = g2; o[3 * H + u] = g3;
        oo[u] = to_op<T>(g0); oo[H + u] = to_op<T>(g1); oo[2 * H + u] = to_op<T>(g2); oo[3 * H + u] = to_op<T>(g3);
        if (dG3) {  // this step's row as [hi | hi | lo] for the three-product recurrence GEMM
            __nv_bfloat16 *q = dG3 + n * 12 * H;
            const float gv[4] = {g0, g1, g2, g3};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const __nv_bfloat16 hi = __float2bfloat16_rn(gv[j]);
                q[j * H + u] = hi;
                q[4 * H + j * H + u] = hi;
                q[8 * H + j * H + u] = __float2bfloat16_rn(gv[j] - __bfloat162float(hi));
            }
        }
        dC[i] = dc * fg;
    }
}

// Column sums of a [R, C] matrix, two levels: chunk c of the rows (COLSUM_CHUNKS of them)
// into part[c][C], then the chunks' partials in order.  One thread per column, rows in
// order, a compensated (Kahan) fp32 sum: the error stays near one rounding whatever R,
// and the order, so the result, is fixed.
constexpr int COLSUM_CHUNKS = 64;
__global__ void k_bw_colsum(size_t R, int C, const float *__restrict__ in, float *__restrict__ part) {
    const int col = blockIdx.x * blockDim.x + threadIdx.x, c = blockIdx.y;
    if (col >= C) return;
    const size_t r0 = R * c / COLSUM_CHUNKS, r1 = R * (c + 1) / COLSUM_CHUNKS;
    float s = 0.f, comp = 0.f;
    for (size_t r = r0; r < r1; ++r) {
        const float y = in[r * C + col] - comp;
        const float t = s + y;
        comp = (t - s) - y;
        s = t;
    }
    part[(size_t)c * C + col] = s;
}
__global__ void k_bw_colsum_fin(int C, const float *__restrict__ part, float *__restrict__ out) {
    const int col = blockIdx.x * blockDim.x + threadIdx.x;
    if (col >= C) return;
    double s = 0.0;
    for (int c = 0; c < COLSUM_CHUNKS; ++c) s += part[(size_t)c * C + col];
    out[col] = (float)s;
}

// The action rows of dW_lstm: dW_a[a] = sum of the dG rows whose action is a.  Each row
// chunk is first sorted stably by action (k_bw_rowsort: one block per chunk, rows taken in
// order by one warp 32 at a time, each lane's place among the lanes with the same action
// from a match mask), then block (a, c) sums, in row order, only the rows of chunk c with
// action a, into part[c][a][4H]; then the CHUNKS partials in order.
__global__ void k_bw_rowsort(size_t R, int A, const int32_t *__restrict__ act, int32_t *__restrict__ srows,
                             int32_t *__restrict__ soff) {
    extern __shared__ int s_cnt[];  // [A] counts, then running cursors
    const int c = blockIdx.x;
    const size_t r0 = R * c / CHUNKS, r1 = R * (c + 1) / CHUNKS;
    for (int a = threadIdx.x; a < A; a += blockDim.x) s_cnt[a] = 0;
    __syncthreads();
    for (size_t r = r0 + threadIdx.x; r < r1; r += blockDim.x) {
        const int a = act[r];
        if (a >= 0 && a < A) atomicAdd(&s_cnt[a], 1);
    }
    __syncthreads();
    if (threadIdx.x == 0) {  // exclusive offsets within the chunk
        int run = 0;
        int32_t *off = soff + (size_t)c * (A + 1);
        for (int a = 0; a < A; ++a) {
            const int n = s_cnt[a];
            off[a] = run;
            s_cnt[a] = run;
            run += n;
        }
        off[A] = run;
    }
    __syncthreads();
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        for (size_t b = r0; b < r1; b += 32) {
            const size_t r = b + lane;
            const int a = r < r1 ? act[r] : -1;
            const bool ok = a >= 0 && a < A;
            const uint32_t same = __match_any_sync(0xffffffffu, ok ? a : -1);
            const int rank = __popc(same & ((1u << lane) - 1u));
            int pos = 0;
            if (ok) pos = s_cnt[a] + rank;
            __syncwarp();
            if (ok && rank == 0) s_cnt[a] += __popc(same);  // the lowest lane of each action
            __syncwarp();
            if (ok) srows[r0 + pos] = (int32_t)r;
        }
    }
}
__global__ void k_bw_arows(size_t R, int A, int H4, const int32_t *__restrict__ srows,
                           const int32_t *__restrict__ soff, const float *__restrict__ dG, float *__restrict__ part) {
    const int a = blockIdx.x, c = blockIdx.y;
    const size_t r0 = R * c / CHUNKS;
    const int32_t *off = soff + (size_t)c * (A + 1);
    const int i0 = off[a], i1 = off[a + 1];
    for (int col0 = 0; col0 < H4; col0 += blockDim.x * 4) {
        float s[4] = {0.f, 0.f, 0.f, 0.f};
        const int col = col0 + 4 * threadIdx.x;
        for (int i = i0; i < i1; ++i) {
            const size_t r = (size_t)srows[r0 + i];
            if (col < H4)
                for (int j = 0; j < 4; ++j)
                    if (col + j < H4) s[j] += dG[r * H4 + col + j];
        }
        for (int j = 0; j < 4; ++j)
            if (col + j < H4) part[((size_t)c * A + a) * H4 + col + j] = s[j];
    }
}
__global__ void k_bw_arows_fin(int A, int H4, const float *__restrict__ part, float *__restrict__ out) {
    const size_t n = (size_t)A * H4;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int c = 0; c < CHUNKS; ++c) s += part[(size_t)c * n + i];
        out[i] = s;
    }
}

// bf16 copies of the weights the backward's GEMMs read (bf16 path): W_zh [Z+H, 4H] and
// W_mdn [H, M] from the stepwise family's (already bf16-rounded) fp32 matrices
__global__ void k_bw_cast(size_t rows, int cols, const float *__restrict__ src, long lds, __nv_bfloat16 *__restrict__ dst) {
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < rows * cols; i += (size_t)gridDim.x * blockDim.x)
        dst[i] = __float2bfloat16_rn(src[(i / cols) * lds + i % cols]);
}

// W_h [H, 4H] (the h rows of the gate matrix) as bf16 rows [hi | lo | hi], hi = bf16(w),
// lo = bf16(w - hi): against a [hi | hi | lo] row of dG the K = 12H contraction is
// hi.hi + hi.lo + lo.hi, the fp32 product up to the dropped lo.lo term and the parts'
// residuals (at most about 3 * 2^-16 of each product: bf16's unit roundoff is 2^-8)
__global__ void k_bw_split3(size_t rows, int cols, const float *__restrict__ src, long lds,
                            __nv_bfloat16 *__restrict__ dst) {
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < rows * cols; i += (size_t)gridDim.x * blockDim.x) {
        const size_t r = i / cols;
        const int k = (int)(i % cols);
        const float w = src[r * lds + k];
        const __nv_bfloat16 hi = __float2bfloat16_rn(w), lo = __float2bfloat16_rn(w - __bfloat162float(hi));
        __nv_bfloat16 *d = dst + r * 3 * cols;
        d[k] = hi;
        d[cols + k] = lo;
        d[2 * cols + k] = hi;
    }
}

int grid_of(size_t n) {
    size_t g = (n + 255) / 256;
    if (g > 8192) g = 8192;
    return g < 1 ? 1 : (int)g;
}

inline size_t al(size_t x) { return (x + 255) & ~(size_t)255; }

// Row-major GEMM on cuBLAS: C[m][n] = sum_k A(m,k) B(k,n), A(m,k) = ta ? A[k lda + m] :
// A[m lda + k], B(k,n) = tb ? B[n ldb + k] : B[k ldb + n].  (cuBLAS is column-major: it
// computes C^T = B^T A^T.)  bf16 operands accumulate in fp32; fp32 operands take cuBLAS's
// fp32 emulation on the tensor cores (each operand split into three bf16 parts, fp32-accurate
// products), or plain fp32 where the library does not offer it.
cublasStatus_t gemm(cublasHandle_t hb, bool bf16, bool ta, bool tb, int m, int n, int k, const void *A, long lda,
                    const void *B, long ldb, float *C, long ldc) {
    const float one = 1.f, zero = 0.f;
    const cudaDataType_t dt = bf16 ? CUDA_R_16BF : CUDA_R_32F;
    auto run = [&](cublasComputeType_t ct) {
        return cublasGemmEx(hb, tb ? CUBLAS_OP_T : CUBLAS_OP_N, ta ? CUBLAS_OP_T : CUBLAS_OP_N, n, m, k, &one, B, dt,
                            (int)ldb, A, dt, (int)lda, &zero, C, CUDA_R_32F, (int)ldc, ct, CUBLAS_GEMM_DEFAULT);
    };
    if (bf16) return run(CUBLAS_COMPUTE_32F);
    const cublasStatus_t st = run(CUBLAS_COMPUTE_32F_EMULATED_16BFX9);
    return st == CUBLAS_STATUS_NOT_SUPPORTED ? run(CUBLAS_COMPUTE_32F_PEDANTIC) : st;
}

cudaError_t cublas_err(cublasStatus_t st) {
    return st == CUBLAS_STATUS_SUCCESS ? cudaSuccess
                                       : st == CUBLAS_STATUS_ALLOC_FAILED ? cudaErrorMemoryAllocation
                                                                          : cudaErrorUnknown;
}

}  // namespace

// The forward's outputs at the front of the backward's workspace, then its own buffers.
void wm_bw_carve(const wm_handle *h, int N, int T, void *base, float **hs, float **cs, float **md, float **nll,
                 void **tail) {
    const size_t NT = (size_t)N * T, H = h->cfg.h_dim, M = h->M;
    char *p = (char *)base;
    *hs = (float *)p; p += al(NT * H * 4);
    *cs = (float *)p; p += al(NT * H * 4);
    *md = (float *)p; p += al(NT * M * 4);
    *nll = (float *)p; p += al((size_t)N * 4);
    *tail = p;
}

size_t wm_bw_ws(const wm_handle *h, int N, int T) {
    const wm_config &c = h->cfg;
    const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M, KX = Z + H, H4 = 4 * H;
    const size_t NT = (size_t)N * T, es = c.precision == WM_BF16 ? 2 : 4;
    const size_t part_cols = H4 > M ? H4 : M;
    return al(NT * H * 4) * 2 + al(NT * M * 4) + al((size_t)N * 4)             // h, c, head outputs, nll
           + al(NT * KX * es) + al(NT * H * es)                                // X, Y
           + al(NT * H4 * 4)                                                   // gate activations
           + al(NT * M * 4) + al(NT * M * es)                                  // dMD
           + al(NT * H * 4)                                                    // dY
           + al(NT * H4 * 4) + al(NT * H4 * es)                                // dG
           + 2 * al((size_t)N * H * 4)                                         // dH, dc
           + al((size_t)COLSUM_CHUNKS * part_cols * 4) + al((size_t)CHUNKS * A * H4 * 4)  // partials
           + al(NT * 4) + al((size_t)CHUNKS * (A + 1) * 4)                       // rows sorted by action
           + (es == 4 ? al((size_t)N * 3 * H4 * 2) : 0) + 256;                   // fp32: dG_t as bf16 parts
}

cudaError_t wm_bw_prepare(wm_handle *h) {
    if (!h->cublas) {
        cublasHandle_t hb;
        cublasStatus_t st = cublasCreate(&hb);
        if (st != CUBLAS_STATUS_SUCCESS) return cublas_err(st);
        h->cublas = hb;
        // fp32 GEMMs: the emulation whenever the library has it, and without the scans and
        // patches for infinities and NaNs (every operand here is finite: activations, their
        // gradients and the weights); where the library lacks either setting, its default
        cublasSetEmulationStrategy(hb, CUBLAS_EMULATION_STRATEGY_EAGER);
        cublasSetEmulationSpecialValuesSupport(hb, CUDA_EMULATION_SPECIAL_VALUES_SUPPORT_NONE);
    }
    const wm_config &c = h->cfg;
    if (c.precision == WM_BF16 && !h->bw_wzh) {
        const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M, KX = Z + H;
        cudaError_t e = cudaMalloc(&h->bw_wzh, KX * 4 * H * 2);
        if (e == cudaSuccess) e = cudaMalloc(&h->bw_wm, H * M * 2);
        if (e != cudaSuccess) return e;
        k_bw_cast<<<grid_of(KX * 4 * H), 256>>>(KX, 4 * (int)H, h->step.Wg, (long)(4 * H + A), (__nv_bfloat16 *)h->bw_wzh);
        k_bw_cast<<<grid_of(H * M), 256>>>(H, (int)M, h->step.Wh, (long)(M + h->NR), (__nv_bfloat16 *)h->bw_wm);
        e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return e;
    }
    if (c.precision != WM_BF16 && !h->bw_w3) {
        const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim;
        cudaError_t e = cudaMalloc(&h->bw_w3, H * 12 * H * 2);
        if (e != cudaSuccess) return e;
        k_bw_split3<<<grid_of(H * 4 * H), 256>>>(H, 4 * (int)H, h->step.Wg + Z * (4 * H + A), (long)(4 * H + A),
                                                 (__nv_bfloat16 *)h->bw_w3);
        e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return e;
    }
    if (c.precision != WM_BF16 && !h->bw_wm) {
        // W_mdn without the reward and done columns: the step layout's row stride M + NR is not a
        // multiple of 16 bytes, which keeps cuBLAS off the tensor cores for dY = dMD W_mdn^T
        const size_t H = c.h_dim, M = h->M;
        cudaError_t e = cudaMalloc(&h->bw_wm, H * M * 4);
        if (e == cudaSuccess)
            e = cudaMemcpy2D(h->bw_wm, M * 4, h->step.Wh, (M + h->NR) * 4, M * 4, H, cudaMemcpyDeviceToDevice);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

void wm_bw_free(wm_handle *h) {
    if (h->cublas) cublasDestroy((cublasHandle_t)h->cublas);
    cudaFree(h->bw_wzh);
    cudaFree(h->bw_wm);
    cudaFree(h->bw_w3);
    cudaFree(h->bws);
    h->cublas = h->bw_wzh = h->bw_wm = h->bw_w3 = h->bws = nullptr;
    h->bws_bytes = 0;
}

template <class T>
static cudaError_t bw_run(const wm_handle *h, int N, int TT, const float *z_seq, const int32_t *actions,
                          const int32_t *lengths, const wm_grads &g, const float *hs, const float *cs,
                          const float *md, char *p, cudaStream_t s) {
    const wm_config &c = h->cfg;
    const bool bf = c.precision == WM_BF16;
    const int Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M, KX = Z + H, H4 = 4 * H;
    const size_t NT = (size_t)N * TT;
    cublasHandle_t hb = (cublasHandle_t)h->cublas;
    cublasStatus_t st = cublasSetStream(hb, s);
    if (st != CUBLAS_STATUS_SUCCESS) return cublas_err(st);
    T *X = (T *)p; p += al(NT * KX * sizeof(T));
    T *Y = (T *)p; p += al(NT * H * sizeof(T));
    float *G = (float *)p; p += al(NT * H4 * 4);
    float *dMD = (float *)p; p += al(NT * M * 4);
    T *dMDo = (T *)p; p += al(NT * M * sizeof(T));
    float *dY = (float *)p; p += al(NT * H * 4);
    float *dG = (float *)p; p += al(NT * H4 * 4);
    T *dGo = (T *)p; p += al(NT * H4 * sizeof(T));
    float *dH = (float *)p; p += al((size_t)N * H * 4);
    float *dC = (float *)p; p += al((size_t)N * H * 4);
    float *part = (float *)p; p += al((size_t)COLSUM_CHUNKS * (H4 > M ? H4 : M) * 4);
    float *apart = (float *)p; p += al((size_t)CHUNKS * A * H4 * 4);
    int32_t *srows = (int32_t *)p; p += al(NT * 4);
    int32_t *soff = (int32_t *)p; p += al((size_t)CHUNKS * (A + 1) * 4);
    __nv_bfloat16 *dG3 = bf ? nullptr : (__nv_bfloat16 *)p;  // fp32: dG_t as [hi | hi | lo]
    // weights of the GEMMs: W_zh = the z and h rows of the gate matrix, W_mdn, W_h = W_zh's h rows
    const void *Wzh = bf ? (const void *)h->bw_wzh : (const void *)h->step.Wg;
    const long ldw = bf ? H4 : H4 + A;
    const void *Wm = h->bw_wm;
    const long ldm = M;
    const void *Wh = bf ? (const void *)((const __nv_bfloat16 *)h->bw_wzh + (size_t)Z * H4)
                        : (const void *)(h->step.Wg + (size_t)Z * (H4 + A));
    int launches = 0;
    {
        wm_ktime kt(h, WM_KERNEL_BW, s);
        k_bw_build<T><<<(unsigned)(NT < 8192 ? NT : 8192), 256, 0, s>>>(N, TT, Z, H, z_seq, hs, X, Y);
        ++launches;
    }
    {
        wm_ktime kt(h, WM_KERNEL_BW_GEMM, s);
        st = gemm(hb, bf, false, false, (int)NT, H4, KX, X, KX, Wzh, ldw, G, H4);
        ++launches;
    }
    if (st != CUBLAS_STATUS_SUCCESS) return cublas_err(st);
    {
        wm_ktime kt(h, WM_KERNEL_BW, s);
        k_bw_gates<<<(unsigned)(NT < 8192 ? NT : 8192), 256, 0, s>>>(NT, N, H, A, G, actions, h->step.Wa, h->step.bg);
        k_bw_mdn<T><<<grid_of(NT * Z), 256, 0, s>>>(N, TT, Z, c.k_mix, md, z_seq, lengths, dMD, dMDo);
        launches += 2;
    }
    {
        wm_ktime kt(h, WM_KERNEL_BW_GEMM, s);
        st = gemm(hb, bf, false, true, (int)NT, H, M, dMDo, M, Wm, ldm, dY, H);
        ++launches;
    }
    if (st != CUBLAS_STATUS_SUCCESS) return cublas_err(st);
    for (int t = TT - 1; t >= 0; --t) {
        {
            wm_ktime kt(h, WM_KERNEL_BW, s);
            const dim3 grid((unsigned)((H + 255) / 256), (unsigned)(N < 65535 ? N : 65535));
            k_bw_cell<T><<<grid, 256, 0, s>>>(N, H, t, t == TT - 1, G, cs, dY, dH, dC, dG, dGo, t > 0 ? dG3 : nullptr);
            ++launches;
        }
        if (t > 0) {
            wm_ktime kt(h, WM_KERNEL_BW_GEMM, s);
            // fp32: bf16 operands over K = 12H (three products, fp32 accumulation)
            st = bf ? gemm(hb, true, false, true, N, H, H4, dGo + (size_t)t * N * H4, H4, Wh, ldw, dH, H)
                    : gemm(hb, true, false, true, N, H, 3 * H4, dG3, 3 * H4, h->bw_w3, 3 * H4, dH, H);
            ++launches;
            if (st != CUBLAS_STATUS_SUCCESS) return cublas_err(st);
        }
    }
    {
        wm_ktime kt(h, WM_KERNEL_BW_GEMM, s);
        // z rows and h rows of dW_lstm: X^T dG, straight into the output's row blocks
        st = gemm(hb, bf, true, false, Z, H4, (int)NT, X, KX, dGo, H4, g.W_lstm, H4);
        if (st == CUBLAS_STATUS_SUCCESS)
            st = gemm(hb, bf, true, false, H, H4, (int)NT, X + Z, KX, dGo, H4, g.W_lstm + (size_t)(Z + A) * H4, H4);
        if (st == CUBLAS_STATUS_SUCCESS) st = gemm(hb, bf, true, false, H, M, (int)NT, Y, H, dMDo, M, g.W_mdn, M);
        launches += 3;
    }
    if (st != CUBLAS_STATUS_SUCCESS) return cublas_err(st);
    {
        wm_ktime kt(h, WM_KERNEL_BW, s);
        k_bw_rowsort<<<CHUNKS, 256, (size_t)A * 4, s>>>(NT, A, actions, srows, soff);
        k_bw_arows<<<dim3(A, CHUNKS), 256, 0, s>>>(NT, A, H4, srows, soff, dG, apart);
        k_bw_arows_fin<<<grid_of((size_t)A * H4), 256, 0, s>>>(A, H4, apart, g.W_lstm + (size_t)Z * H4);
        k_bw_colsum<<<dim3((H4 + 255) / 256, COLSUM_CHUNKS), 256, 0, s>>>(NT, H4, dG, part);
        k_bw_colsum_fin<<<(H4 + 255) / 256, 256, 0, s>>>(H4, part, g.b_lstm);
        k_bw_colsum<<<dim3((M + 255) / 256, COLSUM_CHUNKS), 256, 0, s>>>(NT, M, dMD, part);
        k_bw_colsum_fin<<<(M + 255) / 256, 256, 0, s>>>(M, part, g.b_mdn);
        launches += 7;
    }
    h->last_launches += launches;
    return cudaGetLastError();
}

cudaError_t wm_bw_launch(const wm_handle *h, int N, int T, const float *z_seq, const int32_t *actions,
                         const int32_t *lengths, const wm_grads &g, const float *hs, const float *cs,
                         const float *md, void *tail, cudaStream_t s) {
    if (N == 0 || T == 0) {  // no rows: every gradient is 0
        const wm_config &c = h->cfg;
        const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M;
        cudaError_t e = cudaMemsetAsync(g.W_lstm, 0, (Z + A + H) * 4 * H * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(g.b_lstm, 0, 4 * H * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(g.W_mdn, 0, H * M * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(g.b_mdn, 0, M * 4, s);
        return e;
    }
    if (h->cfg.precision == WM_BF16)
        return bw_run<__nv_bfloat16>(h, N, T, z_seq, actions, lengths, g, hs, cs, md, (char *)tail, s);
    return bw_run<float>(h, N, T, z_seq, actions, lengths, g, hs, cs, md, (char *)tail, s);
}
