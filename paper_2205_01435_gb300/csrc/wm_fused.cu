// wm_fused.cu -- the fused kernel family: one launch runs all T dream steps.
//
// Layout of the work.  One thread-block cluster of CL = 16 CTAs owns a tile of
// 128 episodes (the M = 128 of a tcgen05 MMA; thread i of every CTA is episode
// i of the tile and TMEM lane i).  The weights are split by output column across
// the 16 CTAs and stay resident in shared memory for the whole rollout:
//   rank r owns hidden units [rU, rU+U)  -> 4U gate columns (i|f|g|o)   (a3)
//              actions [r*AC, r*AC+AC)   -> controller columns          (a1)
//              latent dims [r*ZD, r*ZD+ZD) -> 3*ZD*K mixture columns     (a5)
//   and every rank also computes the reward and done columns (2 columns), so
//   the done decision needs no exchange.
// Each CTA holds the full GEMM operand tile X = [z_t | h_t] (128 x (Z+H) bf16,
// K-major core-matrix layout).  Per step:
//   MMA1  X x W1_r -> TMEM (gate and controller pre-activations)
//   each CTA: masked local argmax over its actions; (value, index) partials are
//         written into every CTA (DSMEM)                               -- barrier 1
//   every CTA reduces the 16 partials (same order everywhere) -> a_t (a2);
//   gates + bias + W_a[a_t] row (shared-memory gather), LSTM cell with c kept
//         in registers (a4); h' (bf16) is written into every CTA's X    -- barrier 2
//   MMA2  X_h x W2_r -> TMEM (mixture head, reward, done)
//   per owned dim: temperature softmax, inverse-CDF component, Box-Muller
//         (a6, a7); z' (bf16) is written into every CTA's X; done/freeze (a8)
//                                                                       -- barrier 3
// In teacher-forced mode (a9) the actions and z come from the inputs, every CTA
// loads z_{t+1} itself, and each rank accumulates the NLL of its dims; a small
// kernel adds the 16 partials per sequence in a fixed order.
//
// Waits on MMA completion are bounded: on expiry the kernel records
// WM_ERR_TIMEOUT in the status word, stops issuing MMAs and waiting, and still
// runs every cluster barrier so that all CTAs finish.
#include <cuda_bf16.h>
#include <math.h>
#include <string.h>

#include <vector>

#include "tc_ptx.cuh"
#include "wm_device.cuh"
#include "wm_internal.h"

using namespace wmk;

namespace {

constexpr int CL = 16;     // CTAs per cluster
constexpr int TILE = 128;  // episodes per cluster = MMA M = threads per CTA
constexpr uint32_t WAIT_POLLS = 1u << 26;

template <int U_, int ZD_, int KM_>
struct Shape {
    static constexpr int U = U_, ZD = ZD_, KM = KM_;
    static constexpr int NG = 4 * U;                       // gate columns
    static constexpr int NA = 16;                          // controller columns (padded)
    static constexpr int N1 = NG + NA;                     // MMA1 N (rollout)
    static constexpr int NH = 3 * ZD * KM;                 // mixture-head columns
    static constexpr int N2 = (NH + 2 + 15) / 16 * 16;     // MMA2 N (+ reward, done)
    static_assert(N1 % 16 == 0 && N1 <= 256, "MMA1 N");
    static_assert(N2 % 16 == 0 && N2 <= 128, "MMA2 N");
};

// The one shape instantiated: Z = 32, H = 256, K = 5 (A = 16 * AC, AC <= 16).
using S0 = Shape<16, 2, 5>;

struct Geo {  // byte layout of a rank's weight image / of shared memory
    size_t w1, w2, wa, b1, b2, img;  // image sections (offsets) and total
    size_t x, part, smem;            // shared-memory extras and total
};

__host__ __device__ inline size_t a128(size_t x) { return (x + 127) & ~(size_t)127; }

template <class S>
__host__ __device__ Geo geometry(int Z, int A, int H) {
    Geo g{};
    const size_t K1 = Z + H;
    g.w1 = 0;
    g.w2 = a128(g.w1 + (size_t)S::N1 * K1 * 2);
    g.wa = a128(g.w2 + (size_t)S::N2 * H * 2);
    g.b1 = a128(g.wa + (size_t)A * S::NG * 2);
    g.b2 = a128(g.b1 + (size_t)S::N1 * 4);
    g.img = a128(g.b2 + (size_t)S::N2 * 4);
    g.x = (g.img + 1023) & ~(size_t)1023;
    g.part = a128(g.x + (size_t)TILE * K1 * 2);
    g.smem = a128(g.part + (size_t)CL * TILE * 8);
    return g;
}

struct FusedParams {
    int B, T, Z, A, H, AC;
    int teacher;
    unsigned long long ep0, seed;
    uint32_t t0;
    float mdn_tau;
    int sigma_sqrt_tau, done_terminates, noop_terminates;
    const unsigned char *img;
    size_t img_stride;
    const float *z0, *h0, *c0;
    const uint8_t *done0;
    const uint32_t *mask;
    float *z_out;
    int32_t *actions;
    float *rewards;
    uint8_t *done;
    float *h_final, *c_final, *h_seq, *c_seq, *mdn_seq;
    uint8_t *comp_seq;
    const float *z_seq;
    const int32_t *act_in, *lengths;
    float *nll_part;  // [CL, B]
    int *status;
};

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

// Write 8 consecutive K elements (one core-matrix row) of row r of the X tile.
__device__ __forceinline__ void x_store8(unsigned char *sx, int r, int k, const float *v) {
    uint4 q;
    q.x = pack_bf16x2(v[0], v[1]);
    q.y = pack_bf16x2(v[2], v[3]);
    q.z = pack_bf16x2(v[4], v[5]);
    q.w = pack_bf16x2(v[6], v[7]);
    *reinterpret_cast<uint4 *>(sx + tc::kmajor_offset(r, k, TILE)) = q;
}

template <class S>
__global__ void __launch_bounds__(TILE, 1) k_fused(FusedParams p) {
    extern __shared__ __align__(1024) unsigned char smem[];
    __shared__ __align__(8) uint64_t mbar[2];
    __shared__ uint32_t tmem_base;
    __shared__ int s_abort;

    const Geo g = geometry<S>(p.Z, p.A, p.H);
    const int tid = threadIdx.x, row = tid, warp = tid >> 5;
    const uint32_t rank = tc::cluster_rank();
    const int tile = blockIdx.x / CL;
    const int b = tile * TILE + row;
    const bool live = b < p.B;
    const int Z = p.Z, H = p.H, A = p.A, K1 = Z + H, KZ = S::KM * Z;
    const int U = S::U, NG = S::NG, NH = S::NH;
    const int W = (A + 31) >> 5;

    unsigned char *sW1 = smem + g.w1, *sW2 = smem + g.w2;
    const __nv_bfloat16 *sWa = reinterpret_cast<const __nv_bfloat16 *>(smem + g.wa);
    const float *sB1 = reinterpret_cast<const float *>(smem + g.b1);
    const float *sB2 = reinterpret_cast<const float *>(smem + g.b2);
    unsigned char *sX = smem + g.x;
    uint64_t *part = reinterpret_cast<uint64_t *>(smem + g.part);

    // ---- load this rank's weight image --------------------------------------
    {
        const uint4 *src = reinterpret_cast<const uint4 *>(p.img + rank * p.img_stride);
        uint4 *dst = reinterpret_cast<uint4 *>(smem);
        for (size_t i = tid; i < g.img / 16; i += TILE) dst[i] = src[i];
    }
    // ---- initial operand tile and register state -----------------------------
    float c[S::U], hs[S::U], zs[S::ZD];
    bool frozen = false;
    {
        const float *zsrc = p.teacher ? p.z_seq : p.z0;
        for (int k0 = 0; k0 < Z; k0 += 8) {
            float v[8];
            for (int j = 0; j < 8; ++j) v[j] = live ? zsrc[(size_t)b * Z + k0 + j] : 0.f;
            x_store8(sX, row, k0, v);
        }
        for (int k0 = 0; k0 < H; k0 += 8) {
            float v[8];
            for (int j = 0; j < 8; ++j) v[j] = (live && p.h0) ? p.h0[(size_t)b * H + k0 + j] : 0.f;
            x_store8(sX, row, Z + k0, v);
        }
#pragma unroll
        for (int j = 0; j < S::U; ++j) {
            const size_t i = (size_t)b * H + rank * U + j;
            c[j] = (live && p.c0) ? p.c0[i] : 0.f;
            hs[j] = (live && p.h0) ? p.h0[i] : 0.f;
        }
#pragma unroll
        for (int i = 0; i < S::ZD; ++i) zs[i] = live ? zsrc[(size_t)b * Z + rank * S::ZD + i] : 0.f;
        frozen = live && p.done0 && p.done0[b] != 0;
    }
    if (tid == 0) {
        tc::mbar_init(tc::smem_u32(&mbar[0]), 1);
        tc::mbar_init(tc::smem_u32(&mbar[1]), 1);
        tc::fence_mbar_init();
        s_abort = 0;
    }
    if (warp == 0) tc::tmem_alloc(tc::smem_u32(&tmem_base), 256);
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    tc::cluster_sync();  // every CTA of the cluster is resident before DSMEM traffic
    tc::fence_after_sync();
    const uint32_t tm = tmem_base;
    const uint32_t lane_base = (uint32_t)(32 * warp) << 16;
    const uint32_t x_u32 = tc::smem_u32(sX);
    const uint32_t part_u32 = tc::smem_u32(part);

    const int N1 = p.teacher ? S::NG : S::N1;
    const uint32_t idesc1 = tc::idesc_bf16_f32(128, p.teacher ? S::NG : S::N1);
    const uint32_t idesc2 = tc::idesc_bf16_f32(128, S::N2);
    const uint32_t lboX = TILE * 16, lbo1 = S::N1 * 16, lbo2 = S::N2 * 16;
    float nll_acc = 0.f;
    const int len = p.teacher ? (p.lengths ? min(max(p.lengths[live ? b : 0], 0), p.T) : p.T) : 0;
    const unsigned long long ep = p.ep0 + (unsigned long long)b;
    (void)N1;

    for (int t = 0; t < p.T; ++t) {
        const uint32_t step = p.t0 + (uint32_t)t;
        const size_t tb = (size_t)t * p.B + b;
        const uint32_t parity = (uint32_t)t & 1u;
        // ---------------- MMA1: gates (+ controller) -------------------------
        if (tid == 0 && !s_abort) {
            tc::fence_after_sync();
            for (int kb = 0; kb < K1 / 16; ++kb) {
                uint64_t da = tc::smem_desc(x_u32 + kb * 2 * lboX, lboX, 128);
                uint64_t db = tc::smem_desc(tc::smem_u32(sW1) + kb * 2 * lbo1, lbo1, 128);
                tc::mma_bf16(tm, da, db, idesc1, kb > 0);
            }
            tc::mma_commit(tc::smem_u32(&mbar[0]));
        }
        __syncwarp();
        if (!s_abort && !tc::mbar_wait_bounded(tc::smem_u32(&mbar[0]), parity, WAIT_POLLS)) {
            s_abort = 1;
            atomicExch(p.status, (int)WM_ERR_TIMEOUT);
        }
        __syncwarp();
        tc::fence_after_sync();
        float gv[S::NG];
#pragma unroll
        for (int c0 = 0; c0 < S::NG; c0 += 16) {
            uint32_t r[16];
            TC_LD16(tm + lane_base + c0, r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) gv[c0 + j] = __uint_as_float(r[j]);
        }
        if (!p.teacher) {
            uint32_t r[16];
            TC_LD16(tm + lane_base + S::NG, r);
            tc::tmem_ld_wait();
            // local masked argmax over this rank's actions (lowest index on ties)
            const int a0 = (int)rank * p.AC;
            float bv = -INFINITY;
            int bi = -1;
            const uint32_t *mw = (p.mask && live) ? p.mask + tb * W : nullptr;
            for (int j = 0; j < p.AC; ++j) {
                const int a = a0 + j;
                const bool ok = !mw || ((__ldg(mw + (a >> 5)) >> (a & 31)) & 1u);
                const float v = __uint_as_float(r[j]) + sB1[S::NG + j];
                if (ok && (bi < 0 || v > bv)) { bv = v; bi = a; }
            }
            const uint64_t rec = ((uint64_t)(uint32_t)bi << 32) | __float_as_uint(bv);
            const uint32_t slot = part_u32 + (rank * TILE + row) * 8;
#pragma unroll 4
            for (int dst = 0; dst < CL; ++dst) tc::st_cluster_u64(tc::map_rank(slot, dst), rec);
        }
        tc::fence_before_sync();
        tc::cluster_sync();  // barrier 1: partials visible, every MMA1 has drained X
        tc::fence_after_sync();

        // ---------------- action (a2) ----------------------------------------
        int a = -1;
        if (p.teacher) {
            if (live) {
                a = p.act_in[tb];
                if (a < 0 || a >= A) a = -1;
            }
        } else if (!frozen) {
            float bv = -INFINITY;
            for (int r = 0; r < CL; ++r) {
                const uint64_t rec = part[r * TILE + row];
                const int i = (int)(rec >> 32);
                const float v = __uint_as_float((uint32_t)rec);
                if (i >= 0 && (a < 0 || v > bv)) { bv = v; a = i; }
            }
        }
        if (!p.teacher && rank == 0 && live) p.actions[tb] = a;

        // ---------------- LSTM cell (a3, a4) ---------------------------------
        const __nv_bfloat16 *war = a >= 0 ? sWa + (size_t)a * NG : nullptr;
        float hn[S::U];
#pragma unroll
        for (int j = 0; j < S::U; ++j) {
            if (frozen) {
                hn[j] = hs[j];
                continue;
            }
            float gi = gv[j] + sB1[j], gf = gv[U + j] + sB1[U + j];
            float gg = gv[2 * U + j] + sB1[2 * U + j], go = gv[3 * U + j] + sB1[3 * U + j];
            if (war) {
                gi += __bfloat162float(war[j]);
                gf += __bfloat162float(war[U + j]);
                gg += __bfloat162float(war[2 * U + j]);
                go += __bfloat162float(war[3 * U + j]);
            }
            c[j] = sigmoidf_(gf) * c[j] + sigmoidf_(gi) * tanhf(gg);
            hn[j] = sigmoidf_(go) * tanhf(c[j]);
            hs[j] = hn[j];
        }
        if (live) {
            const size_t o = tb * H + rank * U;
            if (p.h_seq)
                for (int j = 0; j < S::U; ++j) p.h_seq[o + j] = hs[j];
            if (p.c_seq)
                for (int j = 0; j < S::U; ++j) p.c_seq[o + j] = c[j];
        }
        // broadcast h' (bf16) into every CTA's operand tile, U/8 core-matrix rows
#pragma unroll
        for (int q = 0; q < S::U / 8; ++q) {
            uint4 v;
            v.x = pack_bf16x2(hn[8 * q + 0], hn[8 * q + 1]);
            v.y = pack_bf16x2(hn[8 * q + 2], hn[8 * q + 3]);
            v.z = pack_bf16x2(hn[8 * q + 4], hn[8 * q + 5]);
            v.w = pack_bf16x2(hn[8 * q + 6], hn[8 * q + 7]);
            const uint32_t off = x_u32 + tc::kmajor_offset(row, Z + rank * U + 8 * q, TILE);
#pragma unroll 4
            for (int dst = 0; dst < CL; ++dst) tc::st_cluster_v4(tc::map_rank(off, dst), v);
        }
        tc::fence_proxy_async_cluster();
        tc::fence_before_sync();
        tc::cluster_sync();  // barrier 2: h' complete in every X
        tc::fence_after_sync();

        // ---------------- MMA2: heads (a5) -----------------------------------
        if (tid == 0 && !s_abort) {
            tc::fence_proxy_async_smem();
            tc::fence_after_sync();
            const uint32_t xh = x_u32 + (uint32_t)Z * 256u;  // Z/8 k-blocks of 128 rows
            for (int kb = 0; kb < H / 16; ++kb) {
                uint64_t da = tc::smem_desc(xh + kb * 2 * lboX, lboX, 128);
                uint64_t db = tc::smem_desc(tc::smem_u32(sW2) + kb * 2 * lbo2, lbo2, 128);
                tc::mma_bf16(tm + 128, da, db, idesc2, kb > 0);
            }
            tc::mma_commit(tc::smem_u32(&mbar[1]));
        }
        __syncwarp();
        if (!s_abort && !tc::mbar_wait_bounded(tc::smem_u32(&mbar[1]), parity, WAIT_POLLS)) {
            s_abort = 1;
            atomicExch(p.status, (int)WM_ERR_TIMEOUT);
        }
        __syncwarp();
        tc::fence_after_sync();
        float hv[S::N2];
#pragma unroll
        for (int c0 = 0; c0 < S::N2; c0 += 16) {
            uint32_t r[16];
            TC_LD16(tm + 128 + lane_base + c0, r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) hv[c0 + j] = __uint_as_float(r[j]) + sB2[c0 + j];
        }
        const float rew = hv[NH], dl = hv[NH + 1];

        // ---------------- mixture sample / NLL (a6, a7, a9) ------------------
        float zn[S::ZD];
        const int M = 3 * KZ;
#pragma unroll
        for (int i = 0; i < S::ZD; ++i) {
            const int d = rank * S::ZD + i;
            const float *lg = hv + i * S::KM, *mu = hv + S::ZD * S::KM + i * S::KM;
            const float *ls = hv + 2 * S::ZD * S::KM + i * S::KM;
            if (p.teacher) {
                const float x = live ? p.z_seq[((size_t)(t + 1) * p.B + b) * Z + d] : 0.f;
                float m = -INFINITY;
                for (int k = 0; k < S::KM; ++k) m = fmaxf(m, lg[k]);
                float s = 0.f;
                for (int k = 0; k < S::KM; ++k) s += expf(lg[k] - m);
                const float lse = m + logf(s);
                float lp[S::KM], tmax = -INFINITY;
                for (int k = 0; k < S::KM; ++k) {
                    const float zsc = (x - mu[k]) * expf(-ls[k]);
                    lp[k] = (lg[k] - lse) - 0.5f * zsc * zsc - ls[k] - 0.91893853320467274178f;
                    tmax = fmaxf(tmax, lp[k]);
                }
                float acc = 0.f;
                for (int k = 0; k < S::KM; ++k) acc += expf(lp[k] - tmax);
                if (t < len) nll_acc += -(tmax + logf(acc));
                zn[i] = x;
                continue;
            }
            if (frozen) {
                zn[i] = zs[i];
                continue;
            }
            int kc;
            float z;
            if (!(p.mdn_tau > 0.f)) {
                kc = 0;
                for (int k = 1; k < S::KM; ++k) if (lg[k] > lg[kc]) kc = k;
                z = mu[kc];
            } else {
                const float tau = p.mdn_tau;
                float m = -INFINITY;
                for (int k = 0; k < S::KM; ++k) m = fmaxf(m, lg[k] / tau);
                float pk[S::KM], s = 0.f;
                for (int k = 0; k < S::KM; ++k) { pk[k] = expf(lg[k] / tau - m); s += pk[k]; }
                const float u = uniform_for_dim(p.seed, ep, step, d);
                kc = S::KM - 1;
                float cum = 0.f;
                for (int k = 0; k < S::KM - 1; ++k) {
                    cum += pk[k] / s;
                    if (u < cum) { kc = k; break; }
                }
                const float eps = normal_for_dim(p.seed, ep, step, d);
                const float scale = p.sigma_sqrt_tau ? sqrtf(tau) : 1.f;
                z = mu[kc] + expf(ls[kc]) * scale * eps;
            }
            zn[i] = z;
            if (live && p.comp_seq) p.comp_seq[tb * Z + d] = (uint8_t)kc;
        }
        if (live) {
            if (!p.teacher) {
                for (int i = 0; i < S::ZD; ++i)
                    p.z_out[((size_t)(t + 1) * p.B + b) * Z + rank * S::ZD + i] = zn[i];
                if (frozen && p.comp_seq)
                    for (int i = 0; i < S::ZD; ++i) p.comp_seq[tb * Z + rank * S::ZD + i] = 255;
            }
            if (p.mdn_seq) {
                float *ms = p.mdn_seq + tb * M;
                for (int i = 0; i < S::ZD; ++i) {
                    const int d = rank * S::ZD + i;
                    for (int k = 0; k < S::KM; ++k) {
                        const bool z0 = frozen && !p.teacher;
                        ms[d * S::KM + k] = z0 ? 0.f : hv[i * S::KM + k];
                        ms[KZ + d * S::KM + k] = z0 ? 0.f : hv[S::ZD * S::KM + i * S::KM + k];
                        ms[2 * KZ + d * S::KM + k] = z0 ? 0.f : hv[2 * S::ZD * S::KM + i * S::KM + k];
                    }
                }
            }
            if (!p.teacher && rank == 0) {
                if (frozen) {
                    p.rewards[tb] = 0.f;
                    p.done[tb] = 1;
                } else {
                    const bool noop = p.noop_terminates && a == A - 1;
                    p.rewards[tb] = rew;
                    p.done[tb] = (dl > 0.f || noop) ? 1 : 0;
                }
            }
        }
        if (!p.teacher) {
            if (!frozen) {
                const bool noop = p.noop_terminates && a == A - 1;
                if ((p.done_terminates && dl > 0.f) || noop) frozen = true;
            }
            // broadcast z' (bf16) of the owned dims into every CTA's operand tile
            for (int i = 0; i < S::ZD; i += 2) {
                const int k = rank * S::ZD + i;
                const uint32_t v = pack_bf16x2(zn[i], i + 1 < S::ZD ? zn[i + 1] : 0.f);
                const uint32_t off = x_u32 + tc::kmajor_offset(row, k, TILE);
#pragma unroll 4
                for (int dst = 0; dst < CL; ++dst) tc::st_cluster_u32(tc::map_rank(off, dst), v);
            }
#pragma unroll
            for (int i = 0; i < S::ZD; ++i) zs[i] = zn[i];
        } else if (t + 1 < p.T) {
            // teacher: every CTA loads z_{t+1} itself into its own tile
            for (int k0 = 0; k0 < Z; k0 += 8) {
                float v[8];
                for (int j = 0; j < 8; ++j)
                    v[j] = live ? p.z_seq[((size_t)(t + 1) * p.B + b) * Z + k0 + j] : 0.f;
                x_store8(sX, row, k0, v);
            }
        }
        tc::fence_proxy_async_smem();
        tc::fence_proxy_async_cluster();
        tc::fence_before_sync();
        tc::cluster_sync();  // barrier 3: z' complete in every X
        tc::fence_after_sync();
        if (tid == 0) tc::fence_proxy_async_smem();
    }

    if (live) {
        const size_t o = (size_t)b * H + rank * U;
        if (p.h_final)
            for (int j = 0; j < S::U; ++j) p.h_final[o + j] = hs[j];
        if (p.c_final)
            for (int j = 0; j < S::U; ++j) p.c_final[o + j] = c[j];
        if (p.teacher) p.nll_part[(size_t)rank * p.B + b] = nll_acc;
    }
    tc::fence_before_sync();
    tc::cluster_sync();  // no CTA leaves while others may still write into it
    if (warp == 0) tc::tmem_dealloc(tm, 256);
}

// nll[n] = sum over the 16 rank partials, in rank order.
__global__ void k_nll_reduce(int N, const float *part, float *nll) {
    const int n = blockIdx.x * blockDim.x + threadIdx.x;
    if (n >= N) return;
    double s = 0.0;
    for (int r = 0; r < CL; ++r) s += (double)part[(size_t)r * N + n];
    nll[n] = (float)s;
}

inline float bf16r(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

template <class S>
bool shape_matches(const wm_config &c) {
    return c.h_dim == CL * S::U && c.z_dim == CL * S::ZD && c.k_mix == S::KM;
}

}  // namespace

// ---------------------------------------------------------------------------
int wm_fused_supported(const wm_handle *h, int B) {
    (void)B;
    const wm_config &c = h->cfg;
    if (!h->fused.ok) return 0;
    if (c.ctrl_sample && c.ctrl_tau > 0.f) return 0;  // masked argmax only
    return 1;
}

cudaError_t wm_fused_pack(wm_handle *h, const wm_weights *w) {
    const wm_config &c = h->cfg;
    h->fused.ok = 0;
    if (c.precision != WM_BF16 || !shape_matches<S0>(c) || c.a_dim % CL != 0 || c.a_dim / CL > S0::NA)
        return cudaSuccess;
    using S = S0;
    const int Z = c.z_dim, A = c.a_dim, H = c.h_dim, K = c.k_mix, AC = A / CL, U = S::U;
    const size_t K1 = Z + H, M = (size_t)3 * K * Z;
    const Geo g = geometry<S>(Z, A, H);
    int dev = 0, smem_optin = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if ((size_t)smem_optin < g.smem + 64) return cudaSuccess;

    std::vector<unsigned char> img(g.img * CL, 0);
    auto put_bf16 = [&](unsigned char *base, size_t off, float v) {
        __nv_bfloat16 q = __float2bfloat16_rn(v);
        memcpy(base + off, &q, 2);
    };
    auto host_kmajor = [](size_t r, size_t k, size_t R) {
        return ((k >> 3) * (R >> 3) + (r >> 3)) * 128 + (r & 7) * 16 + (k & 7) * 2;
    };
    for (int r = 0; r < CL; ++r) {
        unsigned char *base = img.data() + (size_t)r * g.img;
        float *b1 = reinterpret_cast<float *>(base + g.b1);
        float *b2 = reinterpret_cast<float *>(base + g.b2);
        // W1 rows: 4U gate columns, then AC controller columns
        for (int n = 0; n < S::N1; ++n) {
            if (n < S::NG) {
                const size_t col = (size_t)(n / U) * H + (size_t)r * U + (n % U);
                for (size_t k = 0; k < K1; ++k) {
                    const size_t src = k < (size_t)Z ? k : k + A;
                    put_bf16(base + g.w1, host_kmajor(n, k, S::N1), w->W_lstm[src * 4 * H + col]);
                }
                b1[n] = w->b_lstm[col];
                for (int a = 0; a < A; ++a)
                    put_bf16(base + g.wa, ((size_t)a * S::NG + n) * 2, w->W_lstm[(size_t)(Z + a) * 4 * H + col]);
            } else if (n - S::NG < AC) {
                const size_t act = (size_t)r * AC + (n - S::NG);
                for (size_t k = 0; k < K1; ++k)
                    put_bf16(base + g.w1, host_kmajor(n, k, S::N1), w->W_ctrl[k * A + act]);
                b1[n] = w->b_ctrl[act];
            }
        }
        // W2 rows: logit | mu | log sigma of the owned dims, then reward, done
        for (int n = 0; n < S::N2; ++n) {
            const float *colsrc = nullptr;
            size_t col = 0;
            float bias = 0.f;
            if (n < S::NH) {
                const int part = n / (S::ZD * S::KM), rem = n % (S::ZD * S::KM);
                const int i = rem / S::KM, kk = rem % S::KM;
                col = (size_t)part * K * Z + (size_t)(r * S::ZD + i) * K + kk;
                colsrc = w->W_mdn;
                bias = w->b_mdn[col];
            } else if (n == S::NH) {
                bias = w->b_rew;
            } else if (n == S::NH + 1) {
                bias = w->b_done;
            }
            for (int k = 0; k < H; ++k) {
                float v = 0.f;
                if (colsrc) v = colsrc[(size_t)k * M + col];
                else if (n == S::NH) v = w->w_rew[k];
                else if (n == S::NH + 1) v = w->w_done[k];
                put_bf16(base + g.w2, host_kmajor(n, k, S::N2), v);
            }
            b2[n] = bias;
        }
    }
    cudaError_t e = cudaMalloc(&h->fused.img, img.size());
    if (e != cudaSuccess) return e;
    e = cudaMemcpy(h->fused.img, img.data(), img.size(), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return e;
    h->fused.img_bytes = g.img;
    e = cudaFuncSetAttribute(k_fused<S>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)g.smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_fused<S>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return cudaSuccess;  // the family stays unavailable; stepwise serves the model
    }
    // can one 16-CTA cluster of this size be resident at all?
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(CL);
    lc.blockDim = dim3(TILE);
    lc.dynamicSmemBytes = g.smem;
    lc.attrs = at;
    lc.numAttrs = 1;
    int nclusters = 0;
    e = cudaOccupancyMaxActiveClusters(&nclusters, k_fused<S>, &lc);
    if (e != cudaSuccess || nclusters < 1) {
        cudaGetLastError();
        return cudaSuccess;
    }
    h->fused.cluster = CL;
    h->fused.max_clusters = nclusters;
    h->fused.ok = 1;
    (void)bf16r;
    return cudaSuccess;
}

void wm_fused_free(wm_handle *h) {
    cudaFree(h->fused.img);
    h->fused.img = nullptr;
}

static cudaError_t launch_fused(const wm_handle *h, FusedParams &p, cudaStream_t s) {
    using S = S0;
    const Geo g = geometry<S>(p.Z, p.A, p.H);
    const int nclusters = (p.B + TILE - 1) / TILE;
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(nclusters * CL);
    lc.blockDim = dim3(TILE);
    lc.dynamicSmemBytes = g.smem;
    lc.stream = s;
    lc.attrs = at;
    lc.numAttrs = 1;
    p.img = (const unsigned char *)h->fused.img;
    p.img_stride = h->fused.img_bytes;
    p.status = h->status;
    return cudaLaunchKernelEx(&lc, k_fused<S>, p);
}

static FusedParams base(const wm_handle *h, int B, int T) {
    const wm_config &c = h->cfg;
    FusedParams p{};
    p.B = B; p.T = T; p.Z = c.z_dim; p.A = c.a_dim; p.H = c.h_dim; p.AC = c.a_dim / CL;
    p.seed = c.seed; p.mdn_tau = c.mdn_tau; p.sigma_sqrt_tau = c.sigma_sqrt_tau;
    p.done_terminates = c.done_terminates; p.noop_terminates = c.noop_terminates;
    return p;
}

__global__ void k_copy_f32(size_t n, const float *src, float *dst) {
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
        dst[i] = src[i];
}

cudaError_t wm_fused_rollout(const wm_handle *h, const wm_rollout_dev &a, cudaStream_t s) {
    if (a.B == 0) { h->last_launches = 0; return cudaSuccess; }
    // z_out[0] = z0
    const size_t nz = (size_t)a.B * h->cfg.z_dim;
    k_copy_f32<<<(int)((nz + 255) / 256 < 1024 ? (nz + 255) / 256 : 1024), 256, 0, s>>>(nz, a.z0, a.z_out);
    h->last_launches = 1;
    if (a.T == 0) {
        const size_t nh = (size_t)a.B * h->cfg.h_dim;
        int grid = (int)((nh + 255) / 256 < 1024 ? (nh + 255) / 256 : 1024);
        if (a.h_final) {
            if (a.h0) k_copy_f32<<<grid, 256, 0, s>>>(nh, a.h0, a.h_final);
            else cudaMemsetAsync(a.h_final, 0, nh * 4, s);
        }
        if (a.c_final) {
            if (a.c0) k_copy_f32<<<grid, 256, 0, s>>>(nh, a.c0, a.c_final);
            else cudaMemsetAsync(a.c_final, 0, nh * 4, s);
        }
        return cudaGetLastError();
    }
    FusedParams p = base(h, a.B, a.T);
    p.teacher = 0;
    p.ep0 = a.ep0; p.t0 = a.t0;
    p.z0 = a.z0; p.h0 = a.h0; p.c0 = a.c0; p.done0 = a.done0; p.mask = a.mask;
    p.z_out = a.z_out; p.actions = a.actions; p.rewards = a.rewards; p.done = a.done;
    p.h_final = a.h_final; p.c_final = a.c_final; p.h_seq = a.h_seq; p.c_seq = a.c_seq;
    p.mdn_seq = a.mdn_seq; p.comp_seq = a.comp_seq;
    cudaError_t e = launch_fused(h, p, s);
    h->last_launches = 2;
    return e != cudaSuccess ? e : cudaGetLastError();
}

size_t wm_fused_nll_ws(const wm_handle *, int N) { return (size_t)CL * N * 4 + 256; }

cudaError_t wm_fused_nll(const wm_handle *h, const wm_nll_dev &a, void *ws, cudaStream_t s) {
    if (a.N == 0) { h->last_launches = 0; return cudaSuccess; }
    if (a.T == 0) {
        h->last_launches = 0;
        return cudaMemsetAsync(a.nll, 0, (size_t)a.N * 4, s);
    }
    FusedParams p = base(h, a.N, a.T);
    p.teacher = 1;
    p.z_seq = a.z_seq; p.act_in = a.actions; p.lengths = a.lengths;
    p.h_seq = a.h_seq; p.c_seq = a.c_seq; p.mdn_seq = a.mdn_seq;
    p.nll_part = (float *)ws;
    cudaError_t e = launch_fused(h, p, s);
    if (e != cudaSuccess) return e;
    k_nll_reduce<<<(a.N + 127) / 128, 128, 0, s>>>(a.N, p.nll_part, a.nll);
    h->last_launches = 2;
    return cudaGetLastError();
}
