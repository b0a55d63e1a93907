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
    static constexpr int WA_STRIDE = NG * 2 + 16;          // bytes per action row of W_a
    static_assert(N1 % 16 == 0 && N1 <= 256, "MMA1 N");
    static_assert(N2 % 16 == 0 && N2 <= 128, "MMA2 N");
};

// The one shape instantiated: Z = 32, H = 256, K = 5 (A = 16 * AC, AC <= 16).
using S0 = Shape<16, 2, 5>;
static_assert(S0::ZD == 2, "the z' exchange packs two bf16 dims per rank into one word");

struct Geo {  // byte layout of a rank's weight image / of shared memory
    size_t w1, w2, wa, b1, b2, img;  // image sections (offsets) and total
    size_t x, part, zst, smem;       // shared-memory extras and total
};

__host__ __device__ inline size_t a128(size_t x) { return (x + 127) & ~(size_t)127; }

template <class S>
__host__ __device__ Geo geometry(int Z, int A, int H) {
    Geo g{};
    const size_t K1 = Z + H;
    g.w1 = 0;
    g.w2 = a128(g.w1 + (size_t)S::N1 * K1 * 2);
    g.wa = a128(g.w2 + (size_t)S::N2 * H * 2);
    g.b1 = a128(g.wa + (size_t)A * S::WA_STRIDE);
    g.b2 = a128(g.b1 + (size_t)S::N1 * 4);
    g.img = a128(g.b2 + (size_t)S::N2 * 4);
    g.x = (g.img + 1023) & ~(size_t)1023;
    g.part = a128(g.x + (size_t)TILE * K1 * 2);
    g.zst = a128(g.part + (size_t)CL * TILE * 8);
    g.smem = a128(g.zst + (size_t)CL * TILE * 4);
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

constexpr int NT = 4 * TILE;  // 4 threads per episode row
constexpr int NGRP = NT / TILE;

// Push this CTA's block at shared address `src` (same offset in every CTA) to the
// 15 other CTAs of the cluster; lane 0 of warp w < nwarps serves peers w, w + nwarps, ...
__device__ __forceinline__ void push_to_peers(uint32_t src, uint32_t bytes, uint32_t mbar, uint32_t rank,
                                              int warp, int lane, int nwarps) {
    if (lane == 0 && warp < nwarps)
        for (int q = warp; q < CL; q += nwarps)
            if ((uint32_t)q != rank)
                tc::bulk_copy_to_peer(tc::map_rank(src, q), src, bytes, tc::map_rank(mbar, q));
}

// barrier over the first 12 warps (the sampling side); warps 12..15 may be issuing MMAs
__device__ __forceinline__ void sync_sampling_warps() { asm volatile("bar.sync 1, 384;" ::: "memory"); }

__device__ __forceinline__ float fast_sigmoid(float x) { return __fdividef(1.f, 1.f + __expf(-x)); }
__device__ __forceinline__ float fast_tanh(float x) { return 2.f * fast_sigmoid(2.f * x) - 1.f; }

// Thread roles.  row = 32*(warp%4) + lane is the episode (TMEM lane); grp = warp/4.
//   gates: group g owns hidden units [4g, 4g+4) of this rank (its 16 MMA1 columns
//          are i|f|g|o of those units); group 0 also owns the controller columns.
//   heads: group i < ZD owns latent dim rank*ZD + i (its 16 MMA2 columns are the
//          K logits, K means, K log-sigmas, then reward (group 0) / done (group 1)).
//   MMA issue: thread 0 issues MMA2; thread 384 issues MMA1 (so the h part of the
//          next step's MMA1 runs while the other warps sample).
template <class S>
__global__ void __launch_bounds__(NT, 1) k_fused(FusedParams p) {
    static_assert(S::U == 4 * NGRP && S::ZD == 2 && 3 * S::KM + 1 <= 16, "fused thread mapping");
    extern __shared__ __align__(1024) unsigned char smem[];
    // mbarriers: 0 MMA1 done, 1 MMA2 done, 2 partials in, 3 h' in, 4 z' in
    __shared__ __align__(8) uint64_t mbar[5];
    __shared__ uint32_t tmem_base;
    __shared__ int s_abort;
    __shared__ float s_done_logit[TILE];

    const Geo g = geometry<S>(p.Z, p.A, p.H);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int row = 32 * (warp & 3) + lane, grp = warp >> 2;
    const uint32_t rank = tc::cluster_rank();
    const int tile = blockIdx.x / CL;
    const int b = tile * TILE + row;
    const bool live = b < p.B;
    const int Z = p.Z, H = p.H, A = p.A, K1 = Z + H, KZ = S::KM * Z;
    const int U = S::U, NG = S::NG;
    const int W = (A + 31) >> 5;
    const int u0 = 4 * grp;                   // first owned unit (within this rank)
    const int dim = (int)rank * S::ZD + grp;  // owned latent dim (groups 0, 1)
    const bool has_dim = grp < S::ZD;
    const int MMA1_THREAD = 3 * TILE;         // warp 12, lane 0

    unsigned char *sW1 = smem + g.w1, *sW2 = smem + g.w2;
    const __nv_bfloat16 *sWa = reinterpret_cast<const __nv_bfloat16 *>(smem + g.wa);
    const float *sB1 = reinterpret_cast<const float *>(smem + g.b1);
    const float *sB2 = reinterpret_cast<const float *>(smem + g.b2);
    unsigned char *sX = smem + g.x;
    uint64_t *part = reinterpret_cast<uint64_t *>(smem + g.part);
    uint16_t *zst = reinterpret_cast<uint16_t *>(smem + g.zst);

    const uint32_t PART_BYTES = TILE * 8, H_BYTES = TILE * S::U * 2, Z_BYTES = TILE * 4;
    const uint32_t mb = tc::smem_u32(&mbar[0]);
    const uint32_t MB_MMA1 = mb, MB_MMA2 = mb + 8, MB_PART = mb + 16, MB_H = mb + 24, MB_Z = mb + 32;

    // ---- load this rank's weight image --------------------------------------
    {
        const uint4 *src = reinterpret_cast<const uint4 *>(p.img + rank * p.img_stride);
        uint4 *dst = reinterpret_cast<uint4 *>(smem);
        for (size_t i = tid; i < g.img / 16; i += NT) dst[i] = src[i];
    }
    // ---- initial operand tile and register state -----------------------------
    float c[4], hs[4], zs = 0.f;
    bool frozen = false;
    {
        const float *zsrc = p.teacher ? p.z_seq : p.z0;
        for (int k0 = 8 * grp; k0 < Z; k0 += 8 * NGRP) {
            float v[8];
            for (int j = 0; j < 8; ++j) v[j] = live ? zsrc[(size_t)b * Z + k0 + j] : 0.f;
            x_store8(sX, row, k0, v);
        }
        for (int k0 = 8 * grp; k0 < H; k0 += 8 * NGRP) {
            float v[8];
            for (int j = 0; j < 8; ++j) v[j] = (live && p.h0) ? p.h0[(size_t)b * H + k0 + j] : 0.f;
            x_store8(sX, row, Z + k0, v);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const size_t i = (size_t)b * H + rank * U + u0 + j;
            c[j] = (live && p.c0) ? p.c0[i] : 0.f;
            hs[j] = (live && p.h0) ? p.h0[i] : 0.f;
        }
        if (has_dim && live) zs = zsrc[(size_t)b * Z + dim];
        frozen = live && p.done0 && p.done0[b] != 0;
    }
    if (tid == 0) {
        for (int i = 0; i < 5; ++i) tc::mbar_init(mb + 8 * i, 1);
        tc::fence_mbar_init();
        // arm the exchange barriers for step 0
        tc::mbar_arrive_expect_tx(MB_PART, (CL - 1) * PART_BYTES);
        tc::mbar_arrive_expect_tx(MB_H, (CL - 1) * H_BYTES);
        tc::mbar_arrive_expect_tx(MB_Z, (CL - 1) * Z_BYTES);
        s_abort = 0;
    }
    if (warp == 0) tc::tmem_alloc(tc::smem_u32(&tmem_base), 256);
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    tc::cluster_sync();  // every CTA is resident (and armed) before any DSMEM traffic
    tc::fence_after_sync();
    const uint32_t tm = tmem_base;
    const uint32_t lane_base = (uint32_t)(32 * (warp & 3)) << 16;
    const uint32_t x_u32 = tc::smem_u32(sX);
    const uint32_t w1_u32 = tc::smem_u32(sW1), w2_u32 = tc::smem_u32(sW2);
    const uint32_t part_u32 = tc::smem_u32(part), zst_u32 = tc::smem_u32(zst);

    const uint32_t idesc1 = tc::idesc_bf16_f32(128, p.teacher ? S::NG : S::N1);
    const uint32_t idesc2 = tc::idesc_bf16_f32(128, S::N2);
    const uint32_t lboX = TILE * 16, lbo1 = S::N1 * 16, lbo2 = S::N2 * 16;
    // MMA1 over k-blocks [kb0, kb1) of 16: z part is [0, Z/16), h part [Z/16, K1/16).
    // Every step accumulates the h part first, then the z part.
    // (descriptor start addresses advance by 2 core matrices along K: 2*lbo bytes, >> 4)
    const uint64_t dX0 = tc::smem_desc(x_u32, lboX, 128), dW10 = tc::smem_desc(w1_u32, lbo1, 128);
    const uint64_t dW20 = tc::smem_desc(w2_u32, lbo2, 128);
    auto mma1 = [&](int kb0, int kb1, bool acc_first) {
        uint64_t da = dX0 + (uint64_t)kb0 * (2 * lboX >> 4), db = dW10 + (uint64_t)kb0 * (2 * lbo1 >> 4);
        for (int kb = kb0; kb < kb1; ++kb) {
            tc::mma_bf16(tm, da, db, idesc1, (kb > kb0 || acc_first) ? 1u : 0u);
            da += 2 * lboX >> 4;
            db += 2 * lbo1 >> 4;
        }
    };
    auto wait_bar = [&](uint32_t bar, uint32_t parity) {
        if (!s_abort && !tc::mbar_wait_bounded(bar, parity, WAIT_POLLS)) {
            s_abort = 1;
            atomicExch(p.status, (int)WM_ERR_TIMEOUT);
        }
        __syncwarp();
    };

    float nll_acc = 0.f;
    const int len = p.teacher ? (p.lengths ? min(max(p.lengths[live ? b : 0], 0), p.T) : p.T) : 0;
    const unsigned long long ep = p.ep0 + (unsigned long long)b;
    const int M = 3 * KZ;
    // the mask word holding this rank's actions, prefetched one step ahead
    const int a0 = (int)rank * p.AC;
    uint32_t mword = 0xFFFFFFFFu;
    if (!p.teacher && grp == 0 && p.mask && live && p.T > 0) mword = __ldg(p.mask + (size_t)b * W + (a0 >> 5));

    if (tid == MMA1_THREAD) {  // MMA1 of step 0
        tc::fence_after_sync();
        mma1(Z / 16, K1 / 16, false);
        mma1(0, Z / 16, true);
        tc::mma_commit(MB_MMA1);
    }

    for (int t = 0; t < p.T; ++t) {
        const uint32_t step = p.t0 + (uint32_t)t;
        const size_t tb = (size_t)t * p.B + b;
        const uint32_t parity = (uint32_t)t & 1u;
        const bool last = t + 1 == p.T;

        // ---------------- gates + controller pre-activations ------------------
        wait_bar(MB_MMA1, parity);
        tc::fence_after_sync();
        float gv[16];
        {
            uint32_t r[16];
            TC_LD16(tm + lane_base + 16 * grp, r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) gv[j] = __uint_as_float(r[j]);
        }
        if (grp == 0) {
            uint64_t rec = 0xFFFFFFFF00000000ull;  // index -1: nothing valid here
            if (!p.teacher) {
                uint32_t r[16];
                TC_LD16(tm + lane_base + S::NG, r);
                tc::tmem_ld_wait();
                // local masked argmax over this rank's actions (lowest index on ties)
                float bv = -INFINITY;
                int bi = -1;
                for (int j = 0; j < p.AC; ++j) {
                    const int a = a0 + j;
                    const bool ok = (mword >> (a & 31)) & 1u;
                    const float v = __uint_as_float(r[j]) + sB1[S::NG + j];
                    if (ok && (bi < 0 || v > bv)) { bv = v; bi = a; }
                }
                rec = ((uint64_t)(uint32_t)bi << 32) | __float_as_uint(bv);
                if (p.mask && live && !last)
                    mword = __ldg(p.mask + (tb + p.B) * W + (a0 >> 5));
            }
            // the partials exchange also tells every CTA that all MMA1 reads of X are done
            part[rank * TILE + row] = rec;
        }
        tc::fence_proxy_async_smem();
        tc::fence_before_sync();
        __syncthreads();
        push_to_peers(part_u32 + rank * PART_BYTES, PART_BYTES, MB_PART, rank, warp, lane, NT / 32);
        wait_bar(MB_PART, parity);
        if (tid == 0) tc::mbar_arrive_expect_tx(MB_PART, (CL - 1) * PART_BYTES);

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
                const uint64_t v64 = part[r * TILE + row];
                const int i = (int)(v64 >> 32);
                const float v = __uint_as_float((uint32_t)v64);
                if (i >= 0 && (a < 0 || v > bv)) { bv = v; a = i; }
            }
        }
        if (!p.teacher && rank == 0 && grp == 0 && live) p.actions[tb] = a;

        // ---------------- LSTM cell (a3, a4): 4 units per thread --------------
        float hn[4];
        {
            // W_a row of a_t: this group's 16 bf16 (i|f|g|o of 4 units) as two 16-byte loads
            float wa[16];
            if (a >= 0) {
                const uint4 *src = reinterpret_cast<const uint4 *>(
                    reinterpret_cast<const unsigned char *>(sWa) + (size_t)a * S::WA_STRIDE + 32 * grp);
                const uint4 q0 = src[0], q1 = src[1];
                const uint32_t wv[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const __nv_bfloat162 v2 = *reinterpret_cast<const __nv_bfloat162 *>(&wv[j]);
                    wa[2 * j] = __low2float(v2);
                    wa[2 * j + 1] = __high2float(v2);
                }
            } else {
#pragma unroll
                for (int j = 0; j < 16; ++j) wa[j] = 0.f;
            }
            const float *bb = sB1 + 16 * grp;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (frozen) {
                    hn[j] = hs[j];
                    continue;
                }
                const float gi = gv[j] + bb[j] + wa[j], gf = gv[4 + j] + bb[4 + j] + wa[4 + j];
                const float gg = gv[8 + j] + bb[8 + j] + wa[8 + j], go = gv[12 + j] + bb[12 + j] + wa[12 + j];
                c[j] = fast_sigmoid(gf) * c[j] + fast_sigmoid(gi) * fast_tanh(gg);
                hn[j] = fast_sigmoid(go) * fast_tanh(c[j]);
                hs[j] = hn[j];
            }
        }
        // h' (bf16) into this CTA's own tile; the rank's U/8 k-blocks are one contiguous block
        {
            uint2 v;
            v.x = pack_bf16x2(hn[0], hn[1]);
            v.y = pack_bf16x2(hn[2], hn[3]);
            *reinterpret_cast<uint2 *>(sX + tc::kmajor_offset(row, Z + rank * U + u0, TILE)) = v;
        }
        tc::fence_proxy_async_smem();
        tc::fence_before_sync();
        __syncthreads();
        const uint32_t hblk = x_u32 + tc::kmajor_offset(0, Z + rank * U, TILE);
        push_to_peers(hblk, H_BYTES, MB_H, rank, warp, lane, NT / 32);
        if (live) {
            const size_t o = tb * H + rank * U + u0;
            if (p.h_seq)
                for (int j = 0; j < 4; ++j) p.h_seq[o + j] = hs[j];
            if (p.c_seq)
                for (int j = 0; j < 4; ++j) p.c_seq[o + j] = c[j];
        }
        wait_bar(MB_H, parity);
        if (tid == 0) tc::mbar_arrive_expect_tx(MB_H, (CL - 1) * H_BYTES);

        // ---------------- MMA2: heads (a5); the h part of the next MMA1 ------
        if (tid == 0 && !s_abort) {
            tc::fence_after_sync();
            uint64_t da = dX0 + ((uint64_t)Z * 256u >> 4), db = dW20;  // X_h: Z/8 k-blocks in
            for (int kb = 0; kb < H / 16; ++kb) {
                tc::mma_bf16(tm + 128, da, db, idesc2, kb > 0);
                da += 2 * lboX >> 4;
                db += 2 * lbo2 >> 4;
            }
            tc::mma_commit(MB_MMA2);
        }
        wait_bar(MB_MMA2, parity);
        if (tid == MMA1_THREAD && !s_abort && !last) {
            // the h part of the next step's MMA1 (h_{t+1} is in X) runs while warps 0..11 sample
            tc::fence_after_sync();
            mma1(Z / 16, K1 / 16, false);
        }
        tc::fence_after_sync();
        float hv[16];
        {
            uint32_t r[16];
            TC_LD16(tm + 128 + lane_base + 16 * (has_dim ? grp : 0), r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) hv[j] = __uint_as_float(r[j]) + sB2[16 * (has_dim ? grp : 0) + j];
        }
        // reward is column 15 of group 0, the done logit column 15 of group 1
        const float rew = hv[15];

        // ---------------- mixture sample / NLL (a6, a7, a9): one dim per thread
        float zn = 0.f;
        int kc = 0;
        if (has_dim) {
            const float *lg = hv, *mu = hv + S::KM, *ls = hv + 2 * S::KM;
            if (p.teacher) {
                const float x = live ? p.z_seq[((size_t)(t + 1) * p.B + b) * Z + dim] : 0.f;
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
                zn = x;
            } else if (frozen) {
                zn = zs;
            } else if (!(p.mdn_tau > 0.f)) {
                for (int k = 1; k < S::KM; ++k) if (lg[k] > lg[kc]) kc = k;
                zn = mu[kc];
            } else {
                const float tau = p.mdn_tau;
                float m = -INFINITY;
                for (int k = 0; k < S::KM; ++k) m = fmaxf(m, lg[k] / tau);
                float pk[S::KM], s = 0.f;
                for (int k = 0; k < S::KM; ++k) { pk[k] = expf(lg[k] / tau - m); s += pk[k]; }
                const float u = uniform_for_dim(p.seed, ep, step, dim);
                kc = S::KM - 1;
                float cum = 0.f;
                for (int k = 0; k < S::KM - 1; ++k) {
                    cum += pk[k] / s;
                    if (u < cum) { kc = k; break; }
                }
                const float eps = normal_for_dim(p.seed, ep, step, dim);
                const float scale = p.sigma_sqrt_tau ? sqrtf(tau) : 1.f;
                zn = mu[kc] + expf(ls[kc]) * scale * eps;
            }
        }
        // ---------------- z' exchange, then the z part of the next MMA1 ------
        if (!p.teacher && has_dim) {
            __nv_bfloat16 zb = __float2bfloat16_rn(zn);
            zst[(rank * TILE + row) * 2 + grp] = *reinterpret_cast<uint16_t *>(&zb);
        }
        if (grp == 1) s_done_logit[row] = hv[15];
        tc::fence_proxy_async_smem();
        tc::fence_before_sync();
        float dl = 0.f;
        if (grp < 3) {
            sync_sampling_warps();  // z' staged, done logit published
            if (!last && !p.teacher)
                push_to_peers(zst_u32 + rank * Z_BYTES, Z_BYTES, MB_Z, rank, warp, lane, 12);
            dl = s_done_logit[row];
        }
        // outputs of this step (overlap the exchange)
        if (live) {
            if (has_dim) {
                if (!p.teacher) {
                    p.z_out[((size_t)(t + 1) * p.B + b) * Z + dim] = zn;
                    if (p.comp_seq) p.comp_seq[tb * Z + dim] = frozen ? (uint8_t)255 : (uint8_t)kc;
                }
                if (p.mdn_seq) {
                    float *ms = p.mdn_seq + tb * M;
                    const bool zero = frozen && !p.teacher;
                    for (int k = 0; k < S::KM; ++k) {
                        ms[dim * S::KM + k] = zero ? 0.f : hv[k];
                        ms[KZ + dim * S::KM + k] = zero ? 0.f : hv[S::KM + k];
                        ms[2 * KZ + dim * S::KM + k] = zero ? 0.f : hv[2 * S::KM + k];
                    }
                }
            }
            if (!p.teacher && rank == 0) {
                const bool noop = p.noop_terminates && a == A - 1;
                if (grp == 0) p.rewards[tb] = frozen ? 0.f : rew;
                if (grp == 1) p.done[tb] = (frozen || dl > 0.f || noop) ? 1 : 0;
            }
        }
        if (!last) {
            if (!p.teacher) {
                wait_bar(MB_Z, parity);
                if (tid == 0) tc::mbar_arrive_expect_tx(MB_Z, (CL - 1) * Z_BYTES);
                // z' of all ranks -> this CTA's operand tile; group g packs k-block g
                const uint32_t *zw = reinterpret_cast<const uint32_t *>(zst);
                for (int k0 = 8 * grp; k0 < Z; k0 += 8 * NGRP) {
                    uint4 q;
                    q.x = zw[(k0 / 2 + 0) * TILE + row];
                    q.y = zw[(k0 / 2 + 1) * TILE + row];
                    q.z = zw[(k0 / 2 + 2) * TILE + row];
                    q.w = zw[(k0 / 2 + 3) * TILE + row];
                    *reinterpret_cast<uint4 *>(sX + tc::kmajor_offset(row, k0, TILE)) = q;
                }
            } else {
                for (int k0 = 8 * grp; k0 < Z; k0 += 8 * NGRP) {
                    float v[8];
                    for (int j = 0; j < 8; ++j)
                        v[j] = live ? p.z_seq[((size_t)(t + 1) * p.B + b) * Z + k0 + j] : 0.f;
                    x_store8(sX, row, k0, v);
                }
            }
            tc::fence_proxy_async_smem();
            tc::fence_before_sync();
            __syncthreads();
            if (tid == MMA1_THREAD && !s_abort) {
                tc::fence_after_sync();
                mma1(0, Z / 16, true);  // accumulate onto the h part issued after MMA2
                tc::mma_commit(MB_MMA1);
            }
            if (!p.teacher) {  // freezing (a8), now that every group can read the done logit
                dl = s_done_logit[row];
                if (!frozen) {
                    const bool noop = p.noop_terminates && a == A - 1;
                    if ((p.done_terminates && dl > 0.f) || noop) frozen = true;
                }
                zs = zn;
            }
        }
    }

    if (live) {
        const size_t o = (size_t)b * H + rank * U + u0;
        if (p.h_final)
            for (int j = 0; j < 4; ++j) p.h_final[o + j] = hs[j];
        if (p.c_final)
            for (int j = 0; j < 4; ++j) p.c_final[o + j] = c[j];
        if (p.teacher && has_dim) p.nll_part[((size_t)rank * S::ZD + grp) * p.B + b] = nll_acc;
    }
    tc::fence_before_sync();
    tc::cluster_sync();  // no CTA leaves while others may still write into it
    if (warp == 0) tc::tmem_dealloc(tm, 256);
}

// nll[n] = sum over the 32 (rank, dim) partials, in a fixed order.
__global__ void k_nll_reduce(int N, int parts, const float *part, float *nll) {
    const int n = blockIdx.x * blockDim.x + threadIdx.x;
    if (n >= N) return;
    double s = 0.0;
    for (int r = 0; r < parts; ++r) s += (double)part[(size_t)r * N + n];
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
    if (c.precision != WM_BF16 || !shape_matches<S0>(c) || c.a_dim % CL != 0 || c.a_dim / CL > S0::NA ||
        32 % (c.a_dim / CL) != 0)  // a rank's actions must sit in one mask word
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
        // W1 rows: group gi (16 columns) = i|f|g|o of units 4gi..4gi+3, then the controller
        for (int n = 0; n < S::N1; ++n) {
            if (n < S::NG) {
                const int gi = n / 16, within = n % 16, gate = within / 4, j = within % 4;
                const size_t col = (size_t)gate * H + (size_t)r * U + 4 * gi + j;
                for (size_t k = 0; k < K1; ++k) {
                    const size_t src = k < (size_t)Z ? k : k + A;
                    put_bf16(base + g.w1, host_kmajor(n, k, S::N1), w->W_lstm[src * 4 * H + col]);
                }
                b1[n] = w->b_lstm[col];
                for (int a = 0; a < A; ++a)
                    put_bf16(base + g.wa, (size_t)a * S::WA_STRIDE + (size_t)n * 2, w->W_lstm[(size_t)(Z + a) * 4 * H + col]);
            } else if (n - S::NG < AC) {
                const size_t act = (size_t)r * AC + (n - S::NG);
                for (size_t k = 0; k < K1; ++k)
                    put_bf16(base + g.w1, host_kmajor(n, k, S::N1), w->W_ctrl[k * A + act]);
                b1[n] = w->b_ctrl[act];
            }
        }
        // W2 rows: 16 per owned dim i = [K logits | K means | K log-sigmas | pad...,
        // column 15: reward (i = 0) or done (i = 1)]
        for (int n = 0; n < S::N2; ++n) {
            const int i = n / 16, within = n % 16;
            const float *colsrc = nullptr;
            size_t col = 0;
            float bias = 0.f;
            int special = 0;  // 1 reward, 2 done
            if (within < 3 * S::KM) {
                const int part = within / S::KM, kk = within % S::KM;
                col = (size_t)part * K * Z + (size_t)(r * S::ZD + i) * K + kk;
                colsrc = w->W_mdn;
                bias = w->b_mdn[col];
            } else if (within == 15) {
                special = i == 0 ? 1 : 2;
                bias = special == 1 ? w->b_rew : w->b_done;
            }
            for (int k = 0; k < H; ++k) {
                float v = 0.f;
                if (colsrc) v = colsrc[(size_t)k * M + col];
                else if (special == 1) v = w->w_rew[k];
                else if (special == 2) v = w->w_done[k];
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
    lc.blockDim = dim3(NT);
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
    lc.blockDim = dim3(NT);
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

size_t wm_fused_nll_ws(const wm_handle *, int N) { return (size_t)CL * S0::ZD * N * 4 + 256; }

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
    k_nll_reduce<<<(a.N + 127) / 128, 128, 0, s>>>(a.N, CL * S0::ZD, p.nll_part, a.nll);
    h->last_launches = 2;
    return cudaGetLastError();
}
