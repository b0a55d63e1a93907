// wm_small.cu -- the fused family's small-batch member: one launch runs all T dream steps
// in fp32 SIMT arithmetic, one thread-block cluster per tile of EB = 4, 8 or 16 episodes,
// with the model's weights resident in the cluster's shared memory.
//
// It serves the models the tcgen05 member (wm_fused.cu) does not take -- the fp32 path
// (Sec. 3.3.2's MDN-RNN evaluated in fp32) and bf16 models of other shapes, with either
// controller (Sec. 3.4: masked argmax or tempered draw) and either reward (Sec. 3.1.4:
// the linear head or Eq. 2) -- when the batch is small: at most 4 waves of 16-episode
// tiles.  A tile of 16 rows is far below the M = 128 of a tensor-core MMA, and the step is
// bound by its chain of dependent phases, so the products run on the FMA pipes: fp32
// operands (bf16-rounded ones for a bf16 model), fp32 accumulation (paired f32x2 FMAs).
//
// Layout of the work.  CTA r of a cluster of CL owns
//   hidden units [r U, r U + U)                  -> 4U gate columns      (a3, a4)
//   controller columns [r AC, r AC + AC)                                 (a1)
//   latent dims [r DZ, r DZ + DZ)                -> their 3K mixture columns (a5 - a7)
// and computes the NR reward / done (/ runtime, memory) columns itself, so every CTA
// decides reward, done and freezing for every episode of the tile without an exchange
// (its inputs, h', are the same bits in every CTA).  Its weight columns are packed once per
// model into an image in the shared-memory layout and loaded per call by bulk copies.  Every
// CTA holds the operand X = [z_t | h_t] of the tile transposed, X^T [k][episode] (rows of EB
// plus a pad that keeps the k-split lanes on distinct banks), in two frames: step t reads
// frame t & 1 and fills the other.  Step t:
//   1. its gate and controller columns: X W1 + b1, a 4 x 4 register tile per group of S1
//      lanes that split k, reduced over the group by a butterfly
//   2. its logit rows go to every CTA
//   3. one warp per episode: masked argmax / tempered draw over all A logits (every CTA
//      reaches the same action, so it needs no exchange)                   (a2)
//   4. the cell for its units; its h' rows go to every CTA's next frame
//   5. its head columns: h' W2 + b2 (S2 lanes split k)
//   6. one warp per (episode, dim) of its dims: temperature softmax, inverse-CDF component
//      and Gaussian draw (or, when scoring, the dim's mixture NLL); reward, done and
//      freezing per episode; its z' rows go to every CTA's next frame
// Exchanges are st.async DSMEM stores counted on the receivers' mbarriers; each wait is
// bounded, and a CTA that gives up records WM_ERR_TIMEOUT and leaves the step loop.
#include <limits.h>
#include <math.h>
#include <string.h>

#include <mutex>

#include "tc_ptx.cuh"
#include "wm_device.cuh"
#include "wm_internal.h"

using namespace wmk;

namespace {

constexpr int MAX_THREADS = 640;  // launch bound: <= 96 registers, so 5 warps fit one SM
                                  // sub-partition's register file

// Episodes per cluster tile EB (16, 8 or 4: fewer episodes per cluster put more clusters,
// and more lanes per output, on a small batch), and what follows from it: the row stride XS
// of the transposed operands [k][episode] (EB + pad, so that the rows k, ..., k + 7 that the
// 8 lanes of one 16-byte access phase read fall on distinct 4-bank groups), and the lanes
// S1 / S2 that split k in the two products (about 512 lanes for the tiny model's columns).
template <int EB>
struct Tile {
    static constexpr int XS = EB == 16 ? 20 : 12;
    static constexpr int S1 = EB == 16 ? 8 : (EB == 8 ? 16 : 32);
    static constexpr int S2 = EB == 16 ? 16 : 32;
};

// Shared-memory geometry of one CTA (offsets in floats, each a multiple of 4).
struct Geo {
    int EB, XS, CL, KX, U, AC, DZ, G4, NC1, NC1P, NC2, NC2P, AP, W, nthreads;
    int w1, b1, wa, w2, b2, xt, lg, g1, hd, cs, hs, zs, nl, pu, pe, mk, ep;
    int wpart1, wend;  // the weight image: [0, wpart1) W1 and b1, [wpart1, wend) W_a, W2, b2
    size_t smem;
};

// A row stride of n floats rounded up to 4 with n / 4 odd: rows k, k+1, ..., k+7 of a
// 16-byte column then fall on 8 distinct 4-bank groups.
int pad_odd4(int n) {
    int p = (n + 3) & ~3;
    if (((p >> 2) & 1) == 0) p += 4;
    return p;
}

Geo geometry(int Z, int A, int H, int K, int NR, int CL, int EB, int XS, int S1, int S2) {
    Geo g{};
    g.EB = EB;
    g.XS = XS;
    g.CL = CL;
    g.KX = Z + H;
    g.U = (H + CL - 1) / CL;
    g.AC = (A + CL - 1) / CL;
    g.DZ = (Z + CL - 1) / CL;
    g.G4 = 4 * g.U;
    g.NC1 = g.G4 + g.AC;
    g.NC1P = pad_odd4(g.NC1);
    g.NC2 = 3 * K * g.DZ + NR;
    g.NC2P = pad_odd4(g.NC2);
    g.AP = (A + 3) & ~3;
    g.W = (A + 31) / 32;
    int o = 0;
    auto take = [&](long n) {
        const int at = o;
        o += (int)((n + 3) & ~3L);
        return at;
    };
    g.w1 = take((long)g.KX * g.NC1P);
    g.b1 = take(g.NC1P);
    g.wpart1 = o;
    g.wa = take((long)A * g.G4);
    g.w2 = take((long)H * g.NC2P);
    g.b2 = take(g.NC2P);
    g.wend = o;
    g.xt = take(2L * g.KX * XS);
    g.lg = take((long)g.AP * XS);
    g.g1 = take((long)EB * g.G4);
    g.hd = take((long)EB * g.NC2P);
    g.cs = take((long)EB * g.U);
    g.hs = take((long)EB * g.U);
    g.zs = take((long)EB * g.DZ);
    g.nl = take((long)EB * g.DZ);
    g.pu = take(2L * EB * g.DZ);  // the step's Philox uniforms and normals, two steps (double buffer)
    g.pe = take(2L * EB * g.DZ);
    g.mk = take(2L * EB * g.W);  // two steps' mask words (double buffer)
    g.ep = take(8L * EB);  // act, frozen, frozen next, length (int); rt, mem; NLL (double)
    g.smem = (size_t)o * 4;
    const int eg = EB / 4;
    const int l1 = eg * ((g.NC1 + 3) / 4) * S1, l2 = eg * ((g.NC2 + 3) / 4) * S2;
    int n = l1 > l2 ? l1 : l2;
    if (n < 32 * EB) n = 32 * EB;
    n = (n + 31) & ~31;
    g.nthreads = n > 576 ? 576 : n;  // larger products loop over their tiles
    return g;
}

template <int EB>
Geo geometry_for(const wm_handle *h, int CL) {
    const wm_config &c = h->cfg;
    return geometry(c.z_dim, c.a_dim, c.h_dim, c.k_mix, h->NR, CL, EB, Tile<EB>::XS, Tile<EB>::S1, Tile<EB>::S2);
}

struct SmallParams {
    Geo g;
    int B, T, Z, A, H, K, M, NR;
    int round;    // bf16 model: the products take bf16-rounded operands
    int teacher;  // teacher-forced scoring (a9) instead of a rollout
    unsigned long long ep0, seed;
    uint32_t t0;
    int ctrl_sample;
    float ctrl_tau, mdn_tau;
    float inv_tau, sigma_scale;  // 1 / mdn_tau; sqrt(mdn_tau) with sigma_sqrt_tau, else 1
    int sigma_sqrt_tau, done_terminates, noop_terminates;
    int shaped;
    float alpha, beta, invalid_reward;
    // this model's per-rank weight images (the shared-memory layout of [0, wend)), one per
    // cluster rank, img_stride bytes apart
    const unsigned char *img;
    size_t img_stride;
    // rollout
    const float *z0, *h0, *c0;
    const uint8_t *done0;
    const uint32_t *mask;
    float *z_out;
    int32_t *actions;
    float *rewards;
    uint8_t *done;
    float *h_final, *c_final, *h_seq, *c_seq, *mdn_seq;
    uint8_t *comp_seq;
    const float *rt0, *mem0;
    float *rt_seq, *mem_seq;
    // scoring
    const float *z_seq;
    const int32_t *act_in, *lengths;
    float *nll;
    int *status;
    uint32_t test_wait;  // > 0: wait this many polls on a barrier nothing completes, then abort
};

__device__ __forceinline__ double ld_cluster_f64(uint32_t caddr) {
    double v;
    asm volatile("ld.shared::cluster.f64 %0, [%1];" : "=d"(v) : "r"(caddr) : "memory");
    return v;
}

// Asynchronous 4-byte copy global -> shared (cp.async), and the wait for all of this thread's.
__device__ __forceinline__ void cp4(void *dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" :: "r"(tc::smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
// waits until at most N of this thread's committed groups are still in flight
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory"); }

// The gate nonlinearities from the exponential: sigma(x) = 1 / (1 + e^-x), tanh(x) =
// 2 sigma(2x) - 1.  With the exp2-based exponential (relative error ~1e-7 at the gates'
// magnitudes) and a rounded reciprocal, both stay within ~2e-7 of the exact values: far
// inside the fp32 path's 1e-4, and a few instructions each on the step's critical path.
__device__ __forceinline__ float sig_fast(float x) { return __frcp_rn(1.f + __expf(-x)); }
__device__ __forceinline__ float tanh_fast(float x) { return fmaf(2.f, sig_fast(2.f * x), -1.f); }

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
// A signed-integer key with the order of the float (for the warp's integer max reduction).
__device__ __forceinline__ int ord_key(float v) {
    const int i = __float_as_int(v);
    return i >= 0 ? i : i ^ 0x7fffffff;
}

// Index of the largest of the lanes' keys (lowest index on ties) by two warp reductions;
// idx = INT_MAX: the lane has none.  Returns INT_MAX if no lane has one.
__device__ __forceinline__ int redux_argmax(int key, int idx) {
    const int kmax = __reduce_max_sync(0xffffffffu, idx != INT_MAX ? key : INT_MIN);
    return __reduce_min_sync(0xffffffffu, (idx != INT_MAX && key == kmax) ? idx : INT_MAX);
}


// The cluster barrier (release / acquire: the DSMEM stores before it are visible after it),
// or the CTA barrier for a cluster of one.
__device__ __forceinline__ void step_sync(int CL) {
    if (CL > 1) tc::cluster_sync();
    else __syncthreads();
}

constexpr uint32_t WAIT_POLLS = 1u << 26;  // bound of every wait on a peer's data

// Copies n4 16-byte words at src (this CTA's shared memory) to the same offset in every other
// CTA of the cluster with st.async: each store counts its 16 bytes on the receiver's mbarrier
// `mbar` (the same offset in every CTA), so that the receiver waits for the bytes, not on a
// cluster-wide barrier, and the sender issues no fence.
__device__ __forceinline__ void to_peers(const float *src, int n4, int CL, int r, uint32_t mbar) {
    if (CL <= 1 || n4 <= 0) return;
    const uint32_t sa = tc::smem_u32(src);
    const int tot = n4 * (CL - 1);
    for (int i = threadIdx.x; i < tot; i += blockDim.x) {
        int q = i / n4;
        const int j = i - q * n4;
        q += q >= r;
        const uint4 v = reinterpret_cast<const uint4 *>(src)[j];
        const uint32_t dst = tc::map_rank(sa + 16u * (uint32_t)j, (uint32_t)q), mb = tc::map_rank(mbar, (uint32_t)q);
        asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];"
                     :: "r"(dst), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(mb) : "memory");
    }
}

// Waits (bounded) until phase `parity` of this CTA's mbarrier completes (the bulk copies it
// counts have landed); thread 0 polls, the CTA barrier hands data and outcome to every thread.
__device__ __forceinline__ bool wait_local(uint32_t mbar, uint32_t parity, int *flag) {
    if (threadIdx.x == 0) *flag = tc::mbar_wait_bounded(mbar, parity, WAIT_POLLS) ? 1 : 0;
    __syncthreads();
    return *flag != 0;
}

// Waits (bounded) until phase `parity` of this CTA's mbarrier completes, i.e. every peer's
// bytes of this exchange have landed.  Thread 0 polls with cluster-scope acquire; the CTA
// barrier then hands the data, and the outcome, to every thread.  Returns false on expiry
// (the same answer in every thread).
__device__ __forceinline__ bool wait_peers(int CL, uint32_t mbar, uint32_t parity, int *flag) {
    if (CL <= 1) {
        __syncthreads();
        return true;
    }
    if (threadIdx.x == 0) {
        bool ok = false;
        for (uint32_t i = 0; i < WAIT_POLLS && !ok; ++i) {
            uint32_t done;
            asm volatile(
                "{\n\t.reg .pred p;\n\t"
                "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
                "selp.u32 %0, 1, 0, p;\n\t}"
                : "=r"(done) : "r"(mbar), "r"(parity) : "memory");
            ok = done != 0;
        }
        *flag = ok ? 1 : 0;
    }
    __syncthreads();
    return *flag != 0;
}

// One butterfly level over the lanes xor `o` of a group: the lane with bit o set keeps the
// upper half of its N2 * 2 partial sums, the other the lower half, each adding its partner's.
template <int N2>
__device__ __forceinline__ void fold(float *acc, bool up, int o) {
#pragma unroll
    for (int j = 0; j < N2; ++j) {
        const float keep = up ? acc[j + N2] : acc[j];
        const float send = up ? acc[j] : acc[j + N2];
        acc[j] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
}

// Outputs per lane after tile_dot<S>, and the output index of value j of lane s.
template <int S>
struct Fold {
    static constexpr int NV = S >= 16 ? 1 : 16 / S;
    static __device__ __forceinline__ int out(int s, int j) { return S == 32 ? s >> 1 : s * NV + j; }
    static __device__ __forceinline__ bool writer(int s) { return S < 32 || (s & 1) == 0; }
};

// The 4 x 4 tile (episodes e0 .. e0+3, columns c0 .. c0+3) of sum_k X^T[k][e] W[k][c],
// k < K, on a group of S lanes (lane s takes k = s, s + S, ...), reduced over the group by a
// butterfly: lane s returns as value j the sum of output Fold<S>::out(s, j), o = 4 i + jj
// meaning episode e0 + i, column c0 + jj (with S = 32 both lanes of a pair hold it).  Every
// lane of the warp must call it (the reduction shuffles); lanes with on = false contribute
// zeros.  Each output's sum is formed in the same order whatever the tile's position, so an
// episode's results do not depend on the batch it is in.  The products are paired into
// f32x2 FMAs (two fp32 FMAs, each rounded once, as fmaf).  Out of line: both products call
// the one copy, which keeps the step's code within the instruction cache.
template <int S, int XS>
__device__ __noinline__ float2 tile_dot(const float *__restrict__ xt, const float *__restrict__ w, int ldw, int K,
                                        int e0, int c0, int s, bool on) {
    unsigned long long acc2[8];  // (episode pair, column): acc2[2 c + p] = episodes e0 + 2p, e0 + 2p + 1
#pragma unroll
    for (int j = 0; j < 8; ++j) acc2[j] = 0ull;
    if (on) {
        const float *xp = xt + e0, *wp = w + c0;
#pragma unroll 2
        for (int k = s; k < K; k += S) {
            const float4 x = *reinterpret_cast<const float4 *>(xp + k * XS);
            const float4 y = *reinterpret_cast<const float4 *>(wp + k * ldw);
            unsigned long long x01, x23;
            asm("mov.b64 %0, {%1, %2};" : "=l"(x01) : "f"(x.x), "f"(x.y));
            asm("mov.b64 %0, {%1, %2};" : "=l"(x23) : "f"(x.z), "f"(x.w));
            const float yv[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                unsigned long long yy;
                asm("mov.b64 %0, {%1, %1};" : "=l"(yy) : "f"(yv[c]));
                asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(acc2[2 * c]) : "l"(x01), "l"(yy));
                asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(acc2[2 * c + 1]) : "l"(x23), "l"(yy));
            }
        }
    }
    float acc[16];  // acc[4 i + c]: episode e0 + i, column c0 + c
#pragma unroll
    for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int p2 = 0; p2 < 2; ++p2) {
            float lo, hi;
            asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(acc2[2 * c + p2]));
            acc[4 * (2 * p2) + c] = lo;
            acc[4 * (2 * p2 + 1) + c] = hi;
        }
    if (S == 32) {
        fold<8>(acc, (s & 16) != 0, 16);
        fold<4>(acc, (s & 8) != 0, 8);
        fold<2>(acc, (s & 4) != 0, 4);
        fold<1>(acc, (s & 2) != 0, 2);
        acc[0] += __shfl_xor_sync(0xffffffffu, acc[0], 1);
    } else if (S == 16) {
        fold<8>(acc, (s & 8) != 0, 8);
        fold<4>(acc, (s & 4) != 0, 4);
        fold<2>(acc, (s & 2) != 0, 2);
        fold<1>(acc, (s & 1) != 0, 1);
    } else {
        fold<8>(acc, (s & 4) != 0, 4);
        fold<4>(acc, (s & 2) != 0, 2);
        fold<2>(acc, (s & 1) != 0, 1);
    }
    return make_float2(acc[0], Fold<S>::NV > 1 ? acc[1] : 0.f);
}

// Global column of step.Wg [Z+H, 4H+A] behind local column c of W1 (-1: padding).
__device__ __forceinline__ int col1(const Geo &g, int c, int r, int H, int A) {
    if (c < g.G4) {
        const int gi = c / g.U, u = r * g.U + (c - gi * g.U);
        return u < H ? gi * H + u : -1;
    }
    if (c < g.NC1) {
        const int a = r * g.AC + (c - g.G4);
        return a < A ? 4 * H + a : -1;
    }
    return -1;
}

// Global column of step.Wh [H, M+NR] behind local column c of W2 (-1: padding).
__device__ __forceinline__ int col2(const Geo &g, int c, int r, int Z, int K, int M) {
    const int KD = K * g.DZ;
    if (c < 3 * KD) {
        const int part = c / KD, rem = c - part * KD, dd = rem / K, k = rem - dd * K, d = r * g.DZ + dd;
        return d < Z ? part * K * Z + d * K + k : -1;
    }
    if (c < g.NC2) return M + (c - 3 * KD);
    return -1;
}

__device__ __forceinline__ int clampi(int x, int lo, int hi) { return x < lo ? lo : (x > hi ? hi : x); }

// The tempered draw of the controller (Sec. 3.4) for one episode, on a full warp, over the
// logits col[j * ld] (the shared warp selection).
__device__ __noinline__ int select_sampled(const float *col, int ld, int A, const uint32_t *mw, float tau,
                                           unsigned long long seed, unsigned long long episode, uint32_t step) {
    WarpSelect ws;
    ws.sample = true;
    ws.tau = tau;
    ws.want_lp = false;
    ws.seed = seed;
    ws.episode = episode;
    ws.step = step;
    float lp;
    return warp_select(ws, col, A, mw, 0, &lp, ld);
}

// -log sum_k pi_k N(x; mu_k, sigma_k) of one latent dim on a full warp, lane k holding
// component k's logit lgv, mean muv and log sigma lsv (lanes >= K: lgv = -inf): pi the softmax
// of the logits, log sigma used directly, a log-sum-exp over the logits and one over the
// components (a9, the loss of Sec. 4.7).
__device__ __noinline__ float nll_dim(float lgv, float muv, float lsv, float x, bool kv) {
    const float m = warp_max(lgv);
    const float lse = m + logf(warp_sum(kv ? expf(lgv - m) : 0.f));
    const float zk = (x - muv) * expf(-lsv);
    const float lp = kv ? (lgv - lse) - 0.5f * zk * zk - lsv - 0.91893853320467274178f : -INFINITY;
    const float tmax = warp_max(lp);
    return -(tmax + logf(warp_sum(kv ? expf(lp - tmax) : 0.f)));
}

// The step's Philox numbers of one latent dim: the component uniform and the Gaussian draw.
__device__ __noinline__ float2 draw_dim(unsigned long long seed, unsigned long long ep, uint32_t step, int d) {
    return make_float2(uniform_for_dim(seed, ep, step, d), normal_for_dim(seed, ep, step, d));
}

template <int EB>
__global__ void __launch_bounds__(MAX_THREADS, 1) k_small(const __grid_constant__ SmallParams p) {
    using TL = Tile<EB>;
    constexpr int XS = TL::XS, S1 = TL::S1, S2 = TL::S2, EG = EB / 4;
    extern __shared__ __align__(16) float sm[];
    const Geo &g = p.g;
    const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, warp = tid >> 5, nw = nt >> 5;
    const int CL = g.CL, r = CL > 1 ? (int)tc::cluster_rank() : 0;
    const int b0 = (blockIdx.x / CL) * EB, nv = clampi(p.B - b0, 0, EB);
    const int Z = p.Z, A = p.A, H = p.H, K = p.K, KX = g.KX, U = g.U, G4 = g.G4, DZ = g.DZ, W = g.W;
    const int u0 = r * U, a0 = r * g.AC, d0 = r * DZ;
    const int nu = clampi(H - u0, 0, U), na = clampi(A - a0, 0, g.AC), nd = clampi(Z - d0, 0, DZ);
    const int B = p.B, T = p.T, M = p.M, KZ = K * Z;
    const bool teacher = p.teacher != 0, draw = !teacher && p.mdn_tau > 0.f;
    float *w1 = sm + g.w1, *wa = sm + g.wa, *b1 = sm + g.b1, *w2 = sm + g.w2, *b2 = sm + g.b2;
    float *xt = sm + g.xt, *lg = sm + g.lg, *g1 = sm + g.g1, *hd = sm + g.hd;
    float *cs = sm + g.cs, *hs = sm + g.hs, *zs = sm + g.zs, *nl = sm + g.nl;
    float *pu = sm + g.pu, *pe = sm + g.pe;
    uint32_t *mk = reinterpret_cast<uint32_t *>(sm + g.mk);
    // the three exchanges' mbarriers (logits, h', z') and the wait outcome word
    __shared__ __align__(8) unsigned long long xbar[3];
    __shared__ int wflag;
    const uint32_t MB_LG = tc::smem_u32(&xbar[0]), MB_H = tc::smem_u32(&xbar[1]), MB_Z = tc::smem_u32(&xbar[2]);
    int *act = reinterpret_cast<int *>(sm + g.ep), *frz = act + EB, *frzn = act + 2 * EB, *len = act + 3 * EB;
    float *rts = sm + g.ep + 4 * EB, *mems = rts + EB;
    double *nacc = reinterpret_cast<double *>(sm + g.ep + 6 * EB);  // 8-byte aligned: g.ep % 4 == 0
    auto rnd = [&](float v) { return p.round ? round_bf16(v) : v; };
    const int nsd = EB * DZ;  // (episode, dim) items of the rank
    int KP = 1;               // lanes of the mixture reductions: K rounded up to a power of 2
    while (KP < K) KP <<= 1;

    // ---- weights of this CTA's columns (once per call): the rank's packed image, by bulk copies
    // on the TMA engine; part 0 (W1, b1) is waited for before the first product, part 1 (W_a,
    // W2, b2) before the first cell
    __shared__ __align__(8) unsigned long long wbar[2];
    if (tid == 0) {
        tc::mbar_init(tc::smem_u32(&wbar[0]), 1);
        tc::mbar_init(tc::smem_u32(&wbar[1]), 1);
        tc::fence_mbar_init();
        const unsigned char *src = p.img + (size_t)r * p.img_stride;
        const uint32_t base = tc::smem_u32(sm);
        const uint32_t lim[3] = {0u, (uint32_t)g.wpart1 * 4u, (uint32_t)g.wend * 4u};
        for (int part = 0; part < 2; ++part) {
            const uint32_t mb = tc::smem_u32(&wbar[part]);
            tc::mbar_arrive_expect_tx(mb, lim[part + 1] - lim[part]);
            for (uint32_t off = lim[part]; off < lim[part + 1]; off += 32768u) {
                const uint32_t n = lim[part + 1] - off < 32768u ? lim[part + 1] - off : 32768u;
                tc::bulk_load_global(base + off, src + off, n, mb);
            }
        }
    }
    // step 0's Philox numbers (step t + 1's are drawn during step t's sampling)
    if (draw && T > 0)
        for (int i = tid; i < nsd; i += nt) {
            const int e = i / DZ, d = d0 + (i - e * DZ);
            if (e >= nv || d >= Z) continue;
            const float2 ue = draw_dim(p.seed, p.ep0 + b0 + e, p.t0, d);
            pu[i] = ue.x;
            pe[i] = ue.y;
        }
    // step 0's mask words; step t + 1's are fetched during step t
    if (!teacher && p.mask && T > 0)
        for (int i = tid; i < EB * W; i += nt) {
            const int e = i / W;
            if (e < nv) cp4(mk + i, p.mask + ((size_t)b0 + e) * W + (i - e * W));
        }
    cp_commit();
    // ---- state: frame 0 of X (every row: z_0 and h_0 of the whole tile), the rank's c, h, z
    for (int k = warp; k < KX; k += nw)
        if (lane < XS) {
            const int e = lane;
            float v = 0.f;
            if (e < nv) {
                const size_t b = (size_t)b0 + e;
                if (k < Z) v = teacher ? p.z_seq[b * Z + k] : p.z0[b * Z + k];
                else if (!teacher && p.h0) v = p.h0[b * H + (k - Z)];
            }
            xt[k * XS + e] = rnd(v);
            xt[(KX + k) * XS + e] = 0.f;
        }
    for (int i = tid; i < EB * U; i += nt) {
        const int e = i / U, u = u0 + (i - e * U);
        const bool ok = !teacher && e < nv && u < H;
        cs[i] = ok && p.c0 ? p.c0[((size_t)b0 + e) * H + u] : 0.f;
        hs[i] = ok && p.h0 ? p.h0[((size_t)b0 + e) * H + u] : 0.f;
    }
    for (int i = tid; i < nsd; i += nt) {
        const int e = i / DZ, d = d0 + (i - e * DZ);
        const bool ok = !teacher && e < nv && d < Z;
        zs[i] = ok ? p.z0[((size_t)b0 + e) * Z + d] : 0.f;
        if (ok) p.z_out[((size_t)b0 + e) * Z + d] = zs[i];  // frame 0 of the trajectory
    }
    if (tid < EB) {
        const int e = tid;
        const size_t b = (size_t)b0 + e;
        frz[e] = e >= nv ? 1 : (!teacher && p.done0 && p.done0[b] != 0 ? 1 : 0);
        frzn[e] = frz[e];
        act[e] = -1;
        int L = T;
        if (teacher && e < nv && p.lengths) {
            L = p.lengths[b];
            if (r == 0 && (L < 0 || L > T)) report_status(p.status, WM_ERR_INVALID_ARG);
        }
        len[e] = L;
        const bool sh = p.shaped && !teacher && e < nv;  // scoring takes no runtime / memory state
        rts[e] = sh ? p.rt0[b] : 0.f;
        mems[e] = sh ? p.mem0[b] : 0.f;
        nacc[e] = 0.0;
    }
    cp_wait<0>();  // step 0's mask words have landed (the barriers below publish them)
    // bytes each exchange brings from the peers (their slices differ at ragged edges)
    uint32_t in_lg = 0, in_h = 0, in_z = 0;
    for (int q = 0; q < CL; ++q)
        if (q != r) {
            in_lg += (uint32_t)clampi(A - q * g.AC, 0, g.AC) * XS * 4;
            in_h += (uint32_t)clampi(H - q * U, 0, U) * XS * 4;
            in_z += (uint32_t)clampi(Z - q * DZ, 0, DZ) * XS * 4;
        }
    if (tid == 0) {
        for (int i = 0; i < 3; ++i) tc::mbar_init(tc::smem_u32(&xbar[i]), 1);
        tc::fence_mbar_init();
        if (CL > 1 && T > 0) {  // phase 0 of the logits and h' exchanges (z': in step 0)
            tc::mbar_arrive_expect_tx(MB_LG, in_lg);
            tc::mbar_arrive_expect_tx(MB_H, in_h);
        }
    }
    // the injected wait: a barrier nothing completes, polled at most test_wait times; every
    // CTA gives up the same way, so the abort is uniform across the cluster
    bool abort = false;
    if (p.test_wait) {
        __shared__ __align__(8) unsigned long long never;
        const uint32_t bar = tc::smem_u32(&never);
        if (tid == 0) {
            tc::mbar_init(bar, 1);
            tc::fence_mbar_init();
        }
        __syncthreads();
        if (tid == 0) {
            tc::mbar_wait_bounded(bar, 0, p.test_wait);
            report_status(p.status, WM_ERR_TIMEOUT);
        }
        abort = true;
    }
    bool w_rest = false;  // whether the second weight part has been waited for
    if (!wait_local(tc::smem_u32(&wbar[0]), 0, &wflag)) {  // W1, b1
        if (tid == 0) report_status(p.status, WM_ERR_TIMEOUT);
        abort = true;
    }
    step_sync(CL);  // every CTA of the cluster is running, its mbarriers initialised

    const int CG1 = (g.NC1 + 3) / 4, CG2 = (g.NC2 + 3) / 4;
    for (int t = 0; t < T && !abort; ++t) {
        float *xc = xt + (t & 1) * KX * XS, *xn = xt + ((t + 1) & 1) * KX * XS;
        const uint32_t step = p.t0 + (uint32_t)t;
        // Each exchange's mbarrier completes one phase per step.  The arrive that sets a phase's
        // expected bytes is made by the CTA's last thread (in a phase where its warp is idle),
        // after the mbarrier's previous phase has completed: the logits' for step t + 1 during
        // the cell of step t, the h' one during the head product, the z' one during the
        // selection.  Peers' bytes may land before the arrive (the transaction count goes
        // negative meanwhile); they cannot land before the previous phase completed, since a
        // peer sends step t + 1's data only after it has this CTA's data of step t, which this
        // CTA sends after reading its own of step t.
        const bool zx = t + 1 < T;  // the last step sends no z'
        const bool last_thread = tid == nt - 1 && CL > 1;
        uint32_t *mkc = mk + (t & 1) * EB * W;  // this step's mask words (double buffer)
        // 1. gate pre-activations and logits of the rank's columns
        {
            const int ng = nt / S1, tiles = EG * CG1, gid = tid / S1, s = tid % S1;
            for (int base = 0; base < tiles; base += ng) {
                const int ti = base + gid;
                const bool on = ti < tiles;
                const int eg = on ? ti % EG : 0, cg = on ? ti / EG : 0;
                const float2 v2 = tile_dot<S1, XS>(xc, w1, g.NC1P, KX, 4 * eg, 4 * cg, s, on);
                const float v[2] = {v2.x, v2.y};
                if (on && Fold<S1>::writer(s)) {
#pragma unroll
                    for (int j = 0; j < Fold<S1>::NV; ++j) {
                        const int o = Fold<S1>::out(s, j), e = 4 * eg + (o >> 2), c = 4 * cg + (o & 3);
                        const float y = v[j] + b1[c];
                        if (c < G4) g1[e * G4 + c] = y;
                        else if (c < g.NC1 && a0 + (c - G4) < A) lg[(a0 + (c - G4)) * XS + e] = y;
                    }
                }
            }
        }
        cp_wait<0>();  // this step's mask words (fetched during the previous step)
        __syncthreads();
        // 2. the rank's logit rows to every CTA
        to_peers(lg + a0 * XS, na * XS / 4, CL, r, MB_LG);
        if (!wait_peers(CL, MB_LG, t & 1, &wflag)) {
            if (tid == 0) report_status(p.status, WM_ERR_TIMEOUT);
            abort = true;
            break;
        }
        // 3. the action of each episode (a2), the same in every CTA
        if (last_thread && zx) tc::mbar_arrive_expect_tx(MB_Z, in_z);  // phase t of the z' exchange
        if (warp < EB) {
            const int e = warp;
            const size_t b = (size_t)b0 + e;
            int a = -1;
            if (!frz[e]) {
                if (teacher) {
                    a = p.act_in[(size_t)t * B + b];
                    if (a >= A && r == 0 && lane == 0) report_status(p.status, WM_ERR_INVALID_ARG);
                    if (a >= A || a < 0) a = -1;
                } else if (!(p.ctrl_sample && p.ctrl_tau > 0.f)) {
                    // masked argmax, lowest index on ties
                    const uint32_t *mw = p.mask ? mkc + e * W : nullptr;
                    int key = INT_MIN, bj = INT_MAX;
                    for (int j = lane; j < A; j += 32) {
                        if (mw && !((mw[j >> 5] >> (j & 31)) & 1u)) continue;
                        const int k = ord_key(lg[j * XS + e]);
                        if (bj == INT_MAX || k > key) {
                            key = k;
                            bj = j;
                        }
                    }
                    const int am = redux_argmax(key, bj);
                    a = am == INT_MAX ? -1 : am;
                } else {
                    a = select_sampled(lg + e, XS, A, p.mask ? mkc + e * W : nullptr, p.ctrl_tau, p.seed, p.ep0 + b,
                                       step);
                }
            }
            if (lane == 0) {
                act[e] = a;
                if (!teacher && r == 0 && e < nv) p.actions[(size_t)t * B + b] = a;
            }
        }
        if (t == 0) {  // the rest of the weights (W_a, W2, b2)
            w_rest = true;
            if (!wait_local(tc::smem_u32(&wbar[1]), 0, &wflag)) {
                if (tid == 0) report_status(p.status, WM_ERR_TIMEOUT);
                abort = true;
                break;
            }
        } else {
            __syncthreads();
        }
        // 4. the cell for the rank's units (a3, a4); h' into every CTA's next frame.  The last
        // warp meanwhile fetches the next step's mask words (the other buffer, last read by the
        // previous step's selection).
        if (last_thread && t + 1 < T) tc::mbar_arrive_expect_tx(MB_LG, in_lg);  // phase t + 1
        if (warp == nw - 1 && !teacher && p.mask && t + 1 < T) {
            uint32_t *mkn = mk + ((t + 1) & 1) * EB * W;
            for (int i = lane; i < EB * W; i += 32) {
                const int e = i / W;
                if (e < nv) cp4(mkn + i, p.mask + ((size_t)(t + 1) * B + b0 + e) * W + (i - e * W));
            }
            cp_commit();
        }
        for (int i = tid; i < EB * U; i += nt) {
            const int e = i / U, uu = i - e * U, u = u0 + uu;
            if (u >= H) continue;
            float hv = hs[i], cv = cs[i];
            if (!frz[e]) {
                const float *gr = g1 + e * G4;
                float gi = gr[uu], gf = gr[U + uu], gg = gr[2 * U + uu], go = gr[3 * U + uu];
                const int a = act[e];
                if (a >= 0) {
                    const float *wr = wa + a * G4;
                    gi += wr[uu];
                    gf += wr[U + uu];
                    gg += wr[2 * U + uu];
                    go += wr[3 * U + uu];
                }
                cv = sig_fast(gf) * cv + sig_fast(gi) * tanh_fast(gg);
                hv = sig_fast(go) * tanh_fast(cv);
                cs[i] = cv;
                hs[i] = hv;
            }
            xn[(Z + u) * XS + e] = rnd(hv);
            if (e < nv) {
                const size_t o = ((size_t)t * B + b0 + e) * H + u;
                if (p.h_seq) p.h_seq[o] = hv;
                if (p.c_seq) p.c_seq[o] = cv;
            }
        }
        __syncthreads();
        to_peers(xn + (Z + u0) * XS, nu * XS / 4, CL, r, MB_H);
        if (!wait_peers(CL, MB_H, t & 1, &wflag)) {
            if (tid == 0) report_status(p.status, WM_ERR_TIMEOUT);
            abort = true;
            break;
        }
        // 5. the rank's head columns (a5)
        if (last_thread && t + 1 < T) tc::mbar_arrive_expect_tx(MB_H, in_h);  // phase t + 1
        {
            const int ng = nt / S2, tiles = EG * CG2, gid = tid / S2, s = tid % S2;
            for (int base = 0; base < tiles; base += ng) {
                const int ti = base + gid;
                const bool on = ti < tiles;
                const int eg = on ? ti % EG : 0, cg = on ? ti / EG : 0;
                const float2 v2 = tile_dot<S2, XS>(xn + Z * XS, w2, g.NC2P, H, 4 * eg, 4 * cg, s, on);
                const float v[2] = {v2.x, v2.y};
                if (on && Fold<S2>::writer(s)) {
#pragma unroll
                    for (int j = 0; j < Fold<S2>::NV; ++j) {
                        const int o = Fold<S2>::out(s, j), e = 4 * eg + (o >> 2), c = 4 * cg + (o & 3);
                        if (c < g.NC2) hd[e * g.NC2P + c] = v[j] + b2[c];
                    }
                }
            }
        }
        __syncthreads();
        // 6. the rank's dims: the next latent (a6, a7) or the NLL (a9); z' into the next frame.
        // One warp per (episode, dim) item, lane k holding mixture component k (K <= 32).
        const int KD = K * DZ, X0 = 3 * KD;
        const float *puc = pu + (t & 1) * nsd, *pec = pe + (t & 1) * nsd;
        // the next step's Philox numbers, on the warps past the items (counted from the top)
        if (draw && t + 1 < T)
            for (int i = nt - 1 - tid; i >= 0 && i < nsd; i += nt) {
                const int e = i / DZ, d = d0 + (i - e * DZ);
                if (e >= nv || d >= Z) continue;
                const float2 ue = draw_dim(p.seed, p.ep0 + b0 + e, step + 1u, d);
                pu[((t + 1) & 1) * nsd + i] = ue.x;
                pe[((t + 1) & 1) * nsd + i] = ue.y;
            }
        for (int it = warp; it < nsd; it += nw) {
            const int e = it / DZ, dd = it - e * DZ, d = d0 + dd;
            if (d >= Z) continue;
            if (e >= nv) {
                if (lane == 0) xn[d * XS + e] = 0.f;
                continue;
            }
            const size_t b = (size_t)b0 + e, tb = (size_t)t * B + b;
            const float *row = hd + e * g.NC2P;
            const bool kv = lane < K;
            const float lgv = kv ? row[dd * K + lane] : -INFINITY;
            const float muv = kv ? row[KD + dd * K + lane] : 0.f, lsv = kv ? row[2 * KD + dd * K + lane] : 0.f;
            float *ms = p.mdn_seq ? p.mdn_seq + tb * M : nullptr;
            const bool fz = !teacher && frz[e];
            if (ms && kv) {
                ms[d * K + lane] = fz ? 0.f : lgv;
                ms[KZ + d * K + lane] = fz ? 0.f : muv;
                ms[2 * KZ + d * K + lane] = fz ? 0.f : lsv;
            }
            if (teacher) {
                const float x = p.z_seq[((size_t)(t + 1) * B + b) * Z + d];
                const float nll = nll_dim(lgv, muv, lsv, x, kv);
                if (lane == 0) {
                    nl[it] = nll;
                    xn[d * XS + e] = rnd(x);
                }
                continue;
            }
            float z;
            int kc;
            if (fz) {
                z = zs[it];
                kc = 255;
            } else if (!draw) {
                kc = redux_argmax(ord_key(lgv), kv ? lane : INT_MAX);  // lowest component on ties
                z = __shfl_sync(0xffffffffu, muv, kc);
            } else {
                // component by inverse CDF of softmax(logits / tau): the first k < K - 1 whose
                // cumulative weight exceeds u (u S against the unnormalised sums), then
                // z ~ N(mu, sigma^2).  The reductions and the prefix sum run over the KP lanes
                // of the components only.
                const float q = kv ? lgv * p.inv_tau : -INFINITY;
                float m = q;
                for (int o = KP >> 1; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
                const float ev = kv ? __expf(q - m) : 0.f;
                float S = ev, cum = ev;
                for (int o = KP >> 1; o; o >>= 1) S += __shfl_xor_sync(0xffffffffu, S, o);
                for (int o = 1; o < KP; o <<= 1) {
                    const float up = __shfl_up_sync(0xffffffffu, cum, o);
                    if (lane >= o) cum += up;
                }
                const unsigned hit = __ballot_sync(0xffffffffu, lane < K - 1 && puc[it] * S < cum);
                kc = hit ? __ffs(hit) - 1 : K - 1;
                const float mk_ = __shfl_sync(0xffffffffu, muv, kc), lk = __shfl_sync(0xffffffffu, lsv, kc);
                z = mk_ + __expf(lk) * p.sigma_scale * pec[it];
            }
            if (lane == 0) {
                if (!fz) zs[it] = z;
                xn[d * XS + e] = rnd(z);
                p.z_out[((size_t)(t + 1) * B + b) * Z + d] = z;
                if (p.comp_seq) p.comp_seq[tb * Z + d] = (uint8_t)kc;
            }
        }
        // reward, done and freezing of each episode (a8), in every CTA from the same bits
        if (!teacher && tid < nv) {
            const int e = tid;
            const size_t tb = (size_t)t * B + b0 + e;
            const float *row = hd + e * g.NC2P;
            int fz = frz[e];
            if (fz) {
                if (r == 0) {
                    p.rewards[tb] = 0.f;
                    p.done[tb] = 1;
                }
            } else {
                float rw = row[X0];
                const float dl = row[X0 + 1];
                const int a = act[e];
                const bool noop = p.noop_terminates && a == A - 1;
                if (p.shaped) {  // Eq. 2 on the predictions entering and leaving the step
                    const float rt = row[X0 + 2], mem = row[X0 + 3];
                    rw = a >= 0 ? p.alpha * (rts[e] - rt) + p.beta * (mems[e] - mem) : p.invalid_reward;
                    rts[e] = rt;
                    mems[e] = mem;
                }
                if (r == 0) {
                    p.rewards[tb] = rw;
                    p.done[tb] = (dl > 0.f || noop) ? 1 : 0;
                }
                fz = ((p.done_terminates && dl > 0.f) || noop) ? 1 : 0;
            }
            if (p.shaped && r == 0) {
                if (p.rt_seq) p.rt_seq[tb] = rts[e];
                if (p.mem_seq) p.mem_seq[tb] = mems[e];
            }
            frzn[e] = fz;
        }
        __syncthreads();
        if (tid < EB) {
            const int e = tid;
            if (teacher) {
                if (e < nv && t < len[e]) {
                    float part = 0.f;
                    for (int dd = 0; dd < nd; ++dd) part += nl[e * DZ + dd];
                    nacc[e] += (double)part;
                }
            } else {
                frz[e] = frzn[e];
            }
        }
        if (zx) {
            to_peers(xn + d0 * XS, nd * XS / 4, CL, r, MB_Z);
            if (!wait_peers(CL, MB_Z, t & 1, &wflag)) {
                if (tid == 0) report_status(p.status, WM_ERR_TIMEOUT);
                abort = true;
                break;
            }
        }
    }

    // ---- end of the call.  Nothing of this CTA's may still be in flight into its shared memory:
    // the second weight part (if no step waited for it) and the mask prefetches.
    if (!w_rest) wait_local(tc::smem_u32(&wbar[1]), 0, &wflag);
    cp_wait<0>();
    // every CTA's last writes (the NLL partials) are visible cluster-wide
    step_sync(CL);
    if (!abort && !teacher)
        for (int i = tid; i < EB * U; i += nt) {
            const int e = i / U, u = u0 + (i - e * U);
            if (e >= nv || u >= H) continue;
            const size_t o = ((size_t)b0 + e) * H + u;
            if (p.h_final) p.h_final[o] = hs[i];
            if (p.c_final) p.c_final[o] = cs[i];
        }
    if (teacher && !abort && r == 0 && tid < nv) {
        // each CTA holds the NLL of its dims; rank 0 adds them in rank order
        const uint32_t sa = tc::smem_u32(nacc + tid);
        double s = 0.0;
        for (int q = 0; q < CL; ++q) s += CL > 1 ? ld_cluster_f64(tc::map_rank(sa, (uint32_t)q)) : nacc[tid];
        p.nll[(size_t)b0 + tid] = (float)s;
    }
    step_sync(CL);  // no CTA leaves while a peer may still read its shared memory
}

// Packs rank blockIdx.x's weight image: the shared-memory layout [0, wend) of Geo, from the
// stepwise family's weights (zeros in the padding columns).
__global__ void k_small_pack(const Geo g, int Z, int A, int H, int K, int M, int NR, const float *__restrict__ Wg,
                             const float *__restrict__ Wa, const float *__restrict__ bg, const float *__restrict__ Wh,
                             const float *__restrict__ bh, float *img, size_t stride) {
    const int r = blockIdx.x, ldg = 4 * H + A, ldh = M + NR;
    float *o = img + (size_t)r * stride;
    for (int i = threadIdx.x; i < g.KX * g.NC1P; i += blockDim.x) {
        const int k = i / g.NC1P, col = col1(g, i - k * g.NC1P, r, H, A);
        o[g.w1 + i] = col >= 0 ? Wg[(size_t)k * ldg + col] : 0.f;
    }
    for (int c = threadIdx.x; c < g.NC1P; c += blockDim.x) {
        const int col = col1(g, c, r, H, A);
        o[g.b1 + c] = col >= 0 ? bg[col] : 0.f;
    }
    for (int i = threadIdx.x; i < A * g.G4; i += blockDim.x) {
        const int a = i / g.G4, col = col1(g, i - a * g.G4, r, H, A);
        o[g.wa + i] = col >= 0 ? Wa[(size_t)a * 4 * H + col] : 0.f;
    }
    for (int i = threadIdx.x; i < H * g.NC2P; i += blockDim.x) {
        const int k = i / g.NC2P, col = col2(g, i - k * g.NC2P, r, Z, K, M);
        o[g.w2 + i] = col >= 0 ? Wh[(size_t)k * ldh + col] : 0.f;
    }
    for (int c = threadIdx.x; c < g.NC2P; c += blockDim.x) {
        const int col = col2(g, c, r, Z, K, M);
        o[g.b2 + c] = col >= 0 ? bh[col] : 0.f;
    }
}

__global__ void k_small_copy(size_t n, const float *src, float *dst) {
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
        dst[i] = src ? src[i] : 0.f;
}

// Raises k_small<EB>'s dynamic shared-memory limit on the current device to at least
// `bytes`, never lowering it: handles of other models may launch the same kernel with more.
template <int EB>
cudaError_t smem_at_least(size_t bytes) {
    static std::mutex mu;
    static size_t cur[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(mu);
    if (dev >= 0 && dev < 64 && bytes <= cur[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(k_small<EB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_small<EB>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e == cudaSuccess && dev >= 0 && dev < 64) cur[dev] = bytes;
    return e;
}

// Estimated cycles of one step for a cluster of CL (16-episode tiles): the CTA's FMAs at about
// 60% of the FMA pipes' 128 per clock, plus the three cluster barriers and their exchanges.
double step_cost(const Geo &g, int H) {
    const double fma = 16.0 * ((double)g.NC1 * g.KX + (double)g.NC2 * H);
    return fma / 77.0 + (g.CL > 1 ? 1800.0 + 60.0 * g.CL : 300.0);
}

// Clusters of one tile size that can be resident at once (0: none).
template <int EB>
int max_clusters(const Geo &g) {
    if (smem_at_least<EB>(g.smem) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = g.CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(g.CL);
    lc.blockDim = dim3(g.nthreads);
    lc.dynamicSmemBytes = g.smem;
    lc.attrs = at;
    lc.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_small<EB>, &lc) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

// The tile size of a call of B episodes: the smallest whose tiles fit one wave of clusters,
// else 16.  Returns the slot (0: 16, 1: 8, 2: 4).
int pick_slot(const wm_handle *h, int B) {
    const int eb[3] = {16, 8, 4};
    for (int sl = 2; sl >= 1; --sl) {
        const int n = h->small.max_clusters_eb[sl];
        if (n > 0 && (B + eb[sl] - 1) / eb[sl] <= n) return sl;
    }
    return 0;
}

SmallParams base(const wm_handle *h, int B, int T, int slot) {
    const wm_config &c = h->cfg;
    SmallParams p{};
    memcpy(&p.g, h->small.geo[slot], sizeof(Geo));
    p.B = B; p.T = T; p.Z = c.z_dim; p.A = c.a_dim; p.H = c.h_dim; p.K = c.k_mix; p.M = h->M; p.NR = h->NR;
    p.round = c.precision == WM_BF16;
    p.seed = c.seed;
    p.ctrl_sample = c.ctrl_sample; p.ctrl_tau = c.ctrl_tau; p.mdn_tau = c.mdn_tau;
    p.inv_tau = c.mdn_tau > 0.f ? 1.f / c.mdn_tau : 0.f;
    p.sigma_scale = c.sigma_sqrt_tau && c.mdn_tau > 0.f ? sqrtf(c.mdn_tau) : 1.f;
    p.sigma_sqrt_tau = c.sigma_sqrt_tau; p.done_terminates = c.done_terminates;
    p.noop_terminates = c.noop_terminates;
    p.shaped = c.reward_mode == WM_REWARD_SHAPED;
    p.alpha = c.reward_alpha; p.beta = c.reward_beta; p.invalid_reward = c.invalid_reward;
    p.img = (const unsigned char *)h->small.img;
    p.img_stride = h->small.img_stride;
    p.status = h->status;
    p.test_wait = h->test_wait;
    h->test_wait = 0;
    return p;
}

template <int EB>
cudaError_t launch_eb(const wm_handle *h, const SmallParams &p, cudaStream_t s) {
    const Geo &g = p.g;
    cudaError_t e = smem_at_least<EB>(g.smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = g.CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(((p.B + EB - 1) / EB) * g.CL);
    lc.blockDim = dim3(g.nthreads);
    lc.dynamicSmemBytes = g.smem;
    lc.stream = s;
    lc.attrs = at;
    lc.numAttrs = 1;
    wm_ktime kt(h, WM_KERNEL_FUSED_SMALL, s);
    return cudaLaunchKernelEx(&lc, k_small<EB>, p);
}

cudaError_t launch(const wm_handle *h, const SmallParams &p, cudaStream_t s) {
    return p.g.EB == 4 ? launch_eb<4>(h, p, s) : p.g.EB == 8 ? launch_eb<8>(h, p, s) : launch_eb<16>(h, p, s);
}

}  // namespace

// ---------------------------------------------------------------------------
cudaError_t wm_small_prepare(wm_handle *h) {
    const wm_config &c = h->cfg;
    h->small.ok = 0;
    int dev = 0, optin = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
        cudaGetLastError();
        return cudaSuccess;
    }
    // the cluster size with the fewest estimated cycles per step among those whose 16-episode
    // tiles fit (the smaller tiles then fit too)
    Geo best{};
    double best_cost = 0.0;
    for (int CL = 1; CL <= 16; CL *= 2) {
        const Geo g = geometry_for<16>(h, CL);
        if (g.smem + 1024 > (size_t)optin) continue;
        const double cost = step_cost(g, c.h_dim);
        if (best.CL == 0 || cost < best_cost) {
            best = g;
            best_cost = cost;
        }
    }
    if (best.CL == 0) return cudaSuccess;
    const Geo gs[3] = {best, geometry_for<8>(h, best.CL), geometry_for<4>(h, best.CL)};
    const int n[3] = {max_clusters<16>(gs[0]), max_clusters<8>(gs[1]), max_clusters<4>(gs[2])};
    if (n[0] <= 0) return cudaSuccess;
    static_assert(sizeof(Geo) <= sizeof(h->small.geo[0]), "geometry record");
    for (int i = 0; i < 3; ++i) {
        memcpy(h->small.geo[i], &gs[i], sizeof(Geo));
        h->small.max_clusters_eb[i] = n[i];
    }
    h->small.cl = best.CL;
    h->small.img_stride = ((size_t)best.wend * 4 + 255) & ~(size_t)255;
    cudaError_t e = cudaMalloc(&h->small.img, h->small.img_stride * best.CL);
    if (e != cudaSuccess) return e;
    if ((e = wm_small_repack(h)) != cudaSuccess) return e;
    h->small.ok = 1;
    return cudaSuccess;
}

cudaError_t wm_small_repack(wm_handle *h) {
    if (!h->small.img) return cudaSuccess;
    const wm_config &c = h->cfg;
    Geo g;
    memcpy(&g, h->small.geo[0], sizeof(Geo));
    k_small_pack<<<g.CL, 256>>>(g, c.z_dim, c.a_dim, c.h_dim, c.k_mix, h->M, h->NR, h->step.Wg, h->step.Wa,
                                h->step.bg, h->step.Wh, h->step.bh, (float *)h->small.img, h->small.img_stride / 4);
    cudaError_t e = cudaGetLastError();
    return e != cudaSuccess ? e : cudaDeviceSynchronize();
}

void wm_small_free(wm_handle *h) {
    cudaFree(h->small.img);
    h->small.img = nullptr;
    h->small.ok = 0;
}

int wm_small_supported(const wm_handle *h, int B) {
    const wm_config &c = h->cfg;
    if (!h->small.ok || c.n_xfers > 0 || h->P > 1) return 0;
    const int tiles = (B + 15) / 16, m = h->small.max_clusters_eb[0];
    return (tiles + m - 1) / m <= 4;
}

int wm_small_cluster_size(const wm_handle *h) { return h->small.ok ? h->small.cl : 0; }

cudaError_t wm_small_rollout(const wm_handle *h, const wm_rollout_dev &a, cudaStream_t s) {
    h->last_launches = 0;
    if (a.B == 0) return cudaSuccess;
    const size_t nh = (size_t)a.B * h->cfg.h_dim;
    if (a.T == 0) {  // z_out[0] = z0, and the final state is the initial one
        const size_t nz = (size_t)a.B * h->cfg.z_dim;
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        const int gz = (int)((nz + 255) / 256 < 1024 ? (nz + 255) / 256 : 1024);
        const int gh = (int)((nh + 255) / 256 < 1024 ? (nh + 255) / 256 : 1024);
        k_small_copy<<<gz, 256, 0, s>>>(nz, a.z0, a.z_out);
        if (a.h_final) k_small_copy<<<gh, 256, 0, s>>>(nh, a.h0, a.h_final);
        if (a.c_final) k_small_copy<<<gh, 256, 0, s>>>(nh, a.c0, a.c_final);
        h->last_launches = 1 + (a.h_final ? 1 : 0) + (a.c_final ? 1 : 0);
        return cudaGetLastError();
    }
    SmallParams p = base(h, a.B, a.T, pick_slot(h, a.B));
    p.teacher = 0;
    p.ep0 = a.ep0; p.t0 = a.t0;
    p.z0 = a.z0; p.h0 = a.h0; p.c0 = a.c0; p.done0 = a.done0; p.mask = a.mask;
    p.z_out = a.z_out; p.actions = a.actions; p.rewards = a.rewards; p.done = a.done;
    p.h_final = a.h_final; p.c_final = a.c_final; p.h_seq = a.h_seq; p.c_seq = a.c_seq;
    p.mdn_seq = a.mdn_seq; p.comp_seq = a.comp_seq;
    p.rt0 = a.rt0; p.mem0 = a.mem0; p.rt_seq = a.rt_seq; p.mem_seq = a.mem_seq;
    cudaError_t e = launch(h, p, s);
    h->last_launches = 1;
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t wm_small_nll(const wm_handle *h, const wm_nll_dev &a, cudaStream_t s) {
    h->last_launches = 0;
    if (a.N == 0) return cudaSuccess;
    if (a.T == 0) return cudaMemsetAsync(a.nll, 0, (size_t)a.N * 4, s);
    SmallParams p = base(h, a.N, a.T, pick_slot(h, a.N));
    p.teacher = 1;
    p.z_seq = a.z_seq; p.act_in = a.actions; p.lengths = a.lengths;
    p.h_seq = a.h_seq; p.c_seq = a.c_seq; p.mdn_seq = a.mdn_seq;
    p.nll = a.nll;
    cudaError_t e = launch(h, p, s);
    h->last_launches = 1;
    return e != cudaSuccess ? e : cudaGetLastError();
}
