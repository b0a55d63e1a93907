// wm_fused.cu -- the fused kernel family: one launch runs all T dream steps.
//
// Layout of the work.  One thread-block cluster of CL CTAs (CL = 16 or 8) owns a
// tile of 128 episodes (the M = 128 of a tcgen05 MMA; TMEM lane i = episode i of
// the tile).  The weights are split by output column across the CL CTAs:
//   rank r owns hidden units [rU, rU+U), U = H/CL -> 4U gate columns      (a3)
//              actions [r*AC, r*AC+AC), AC = A/CL -> controller columns   (a1)
//              latent dims [r*ZD, r*ZD+ZD), ZD = Z/CL -> 16 head columns
//              per dim (K logits, K means, K log-sigmas, one spare)       (a5)
//   and the spare columns of its first two dims carry the reward and done heads,
//   so every CTA knows the done decision without an exchange.
// Each CTA holds the full GEMM operand tile X = [z_t | h_t] (128 x (Z+H) bf16,
// K-major core-matrix layout), its gate/controller weights W1 and the biases.
// W_a (the action rows of the gate matrix, used by the cell update) and W2 (the
// head weights, used by MMA2) are needed at disjoint moments of a step, so they
// share one shared-memory buffer that TMA bulk loads refill from L2 each step
// while the exchanges run.  Per step:
//   MMA1  X x W1 -> TMEM: gate and controller pre-activations (the h part of it
//         was issued at the end of the previous step, the z part now)
//   masked local argmax over the rank's actions; (value, index) partials go to
//         every CTA                                                  (a2)
//   the CL partials are reduced in rank order -> a_t; gates + bias + the W_a
//         row, LSTM cell with c in registers; h' (bf16) goes into every CTA's X
//                                                                    (a3, a4)
//   MMA2  X_h x W2 -> TMEM: mixture head, reward, done
//   per owned dim: temperature softmax, inverse-CDF component, Box-Muller (a6,
//         a7); z' (bf16) goes to every CTA; done / freeze (a8)
// Exchanges: a CTA writes its slice into its own shared memory, then the TMA
// engine copies it into the same offset of every other CTA of the cluster
// (cp.async.bulk shared::cluster), completing on the receiver's mbarrier.  No
// cluster barrier runs inside the step loop: the data dependencies order every
// reuse of a buffer (the partials certify that every CTA's MMA1 has finished
// reading X before any h' lands in it; h' -> MMA2 -> z' certifies that the
// z staging area was consumed).
// Threads: 512 compute threads per CTA, 4 per episode row (TMEM lets warps w,
// w+4, w+8, w+12 read the same 32 lanes); group g = warp/4 owns U/4 hidden units
// and, if g < ZD, one latent dim.  A 17th warp issues every MMA and weight load,
// so the tensor core is fed while the compute warps work.
// In teacher-forced mode (a9) actions and z come from the inputs, every CTA
// loads z_{t+1} itself, and each latent dim keeps its NLL partial; a small
// kernel adds the partials per sequence in a fixed order.
//
// All waits are bounded: on expiry the kernel records WM_ERR_TIMEOUT in the
// status word, stops issuing MMAs and waiting, and still reaches the final
// cluster barrier, so that every CTA finishes.
#include <cuda_bf16.h>
#include <math.h>
#include <string.h>

#include <mutex>
#include <vector>

#include "tc_ptx.cuh"
#include "wm_device.cuh"
#include "wm_internal.h"

using namespace wmk;

namespace {

constexpr int TILE = 128;              // episodes per cluster = MMA M
constexpr int NT = 4 * TILE;           // compute threads per CTA: 4 per episode row
constexpr int NGRP = NT / TILE;        // thread groups per row
constexpr int NTHREADS = NT + 32;      // + one warp that issues MMAs and weight loads
constexpr int MMA_WARP = NT / 32;
constexpr uint32_t WAIT_POLLS = 1u << 26;
constexpr uint32_t D2_COL = 160;       // TMEM column of the MMA2 accumulator

template <int CL_, int U_, int ZD_, int KM_>
struct Shape {
    static constexpr int CL = CL_, U = U_, ZD = ZD_, KM = KM_;
    static constexpr int UG = U / NGRP;                    // units per thread
    static constexpr int NG = 4 * U;                       // gate columns
    static constexpr int NA = 16;                          // controller columns (padded)
    static constexpr int N1 = NG + NA;                     // MMA1 N (rollout)
    static constexpr int N2 = 16 * ZD;                     // MMA2 N
    static constexpr int WA_STRIDE = NG * 2 + 16;          // bytes per action row of W_a
    static_assert(UG == 4 || UG == 8, "4 or 8 units per thread");
    static_assert(ZD >= 2 && ZD <= NGRP && 3 * KM + 1 <= 16, "head column groups");
    static_assert(N1 % 16 == 0 && N1 <= (int)D2_COL && N2 <= 256 - (int)D2_COL, "TMEM columns");
};

// Z = 32, H = 256, K = 5: 16 CTAs of 16 units / 2 dims, or 8 CTAs of 32 units / 4 dims.
using S16 = Shape<16, 16, 2, 5>;
using S8 = Shape<8, 32, 4, 5>;

struct Geo {               // byte layout of a rank's weight image and of shared memory
    size_t w1, b1, b2;     // resident part (same offsets in the image and in smem)
    size_t iwa, iw2, img;  // streamed sections of the image, image size
    size_t buf, buf_bytes, x, part, zst, smem;
};

__host__ __device__ inline size_t a128(size_t x) { return (x + 127) & ~(size_t)127; }

template <class S>
__host__ __device__ Geo geometry(int Z, int A, int H) {
    Geo g{};
    const size_t K1 = Z + H;
    g.w1 = 0;
    g.b1 = a128(g.w1 + (size_t)S::N1 * K1 * 2);
    g.b2 = a128(g.b1 + (size_t)S::N1 * 4);
    g.iwa = a128(g.b2 + (size_t)S::N2 * 4);
    g.iw2 = a128(g.iwa + (size_t)A * S::WA_STRIDE);
    g.img = a128(g.iw2 + (size_t)S::N2 * H * 2);
    const size_t wa_bytes = (size_t)A * S::WA_STRIDE, w2_bytes = (size_t)S::N2 * H * 2;
    g.buf = g.iwa;
    g.buf_bytes = wa_bytes > w2_bytes ? wa_bytes : w2_bytes;
    g.x = (g.buf + g.buf_bytes + 1023) & ~(size_t)1023;
    g.part = a128(g.x + (size_t)TILE * K1 * 2);
    g.zst = a128(g.part + (size_t)S::CL * TILE * 8);
    g.smem = a128(g.zst + (size_t)S::CL * TILE * S::ZD * 2);
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
    float *nll_part;  // [Z, B]: one partial per latent dim
    int *status;
    // failure injection (wm_inject_wait_timeout): > 0 makes the kernel wait, before it issues
    // any MMA or copy of its own, on a barrier that nothing completes, at most this many polls
    uint32_t test_wait;
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

// Push this CTA's block at shared address `src` (same offset in every CTA) to the
// other CTAs of the cluster; lane 0 of warp w < nwarps serves peers w, w + nwarps, ...
template <int CL>
__device__ __forceinline__ void push_to_peers(uint32_t src, uint32_t bytes, uint32_t mbar, uint32_t rank,
                                              int warp, int lane, int nwarps) {
    if (lane == 0 && warp < nwarps)
        for (int q = warp; q < CL; q += nwarps)
            if ((uint32_t)q != rank)
                tc::bulk_copy_to_peer(tc::map_rank(src, q), src, bytes, tc::map_rank(mbar, q));
}

// barrier over the 16 compute warps (the MMA warp may still be issuing)
__device__ __forceinline__ void sync_compute_warps() { asm volatile("bar.sync 1, 512;" ::: "memory"); }

// Gate nonlinearities on the hardware tanh (one MUFU op each; relative error about
// 2^-11, far inside the bf16 path's tolerance): sigmoid(x) = (1 + tanh(x/2)) / 2.
__device__ __forceinline__ float fast_tanh(float x) {
    float y;
    asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float fast_sigmoid(float x) { return fmaf(0.5f, fast_tanh(0.5f * x), 0.5f); }

template <class S>
__global__ void __launch_bounds__(NTHREADS, 1) k_fused(FusedParams p) {
    constexpr int CL = S::CL, UG = S::UG, ZD = S::ZD, KM = S::KM;
    extern __shared__ __align__(1024) unsigned char smem[];
    // mbarriers: 0 MMA1 done, 1 MMA2 done, 2 partials in, 3 h' in, 4 z' in, 5 W_a in the
    // buffer, 6 never completed (the injected wait), 7 W2 in the buffer (compute threads)
    __shared__ __align__(8) uint64_t mbar[8];
    __shared__ uint32_t tmem_base;
    __shared__ int s_abort;
    __shared__ float s_done_logit[TILE];

    const Geo g = geometry<S>(p.Z, p.A, p.H);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool mma_warp = warp == MMA_WARP;
    const int row = 32 * (warp & 3) + lane, grp = mma_warp ? 0 : warp >> 2;
    const uint32_t rank = tc::cluster_rank();
    const int tile = blockIdx.x / CL;
    const int b = tile * TILE + row;
    const bool live = b < p.B && !mma_warp;
    const int Z = p.Z, H = p.H, A = p.A, K1 = Z + H, KZ = KM * Z;
    const int W = (A + 31) >> 5;
    const int u0 = UG * grp;               // first owned unit (within this rank)
    const int dim = (int)rank * ZD + grp;  // owned latent dim (groups < ZD)
    const bool has_dim = grp < ZD;

    unsigned char *sW1 = smem + g.w1, *sBuf = smem + g.buf;
    const float *sB1 = reinterpret_cast<const float *>(smem + g.b1);
    const float *sB2 = reinterpret_cast<const float *>(smem + g.b2);
    unsigned char *sX = smem + g.x;
    uint64_t *part = reinterpret_cast<uint64_t *>(smem + g.part);
    uint16_t *zst = reinterpret_cast<uint16_t *>(smem + g.zst);

    const uint32_t PART_BYTES = TILE * 8, H_BYTES = TILE * S::U * 2, Z_BYTES = TILE * ZD * 2;
    const uint32_t WA_BYTES = (uint32_t)A * S::WA_STRIDE, W2_BYTES = (uint32_t)S::N2 * H * 2;
    const uint32_t mb = tc::smem_u32(&mbar[0]);
    const uint32_t MB_MMA1 = mb, MB_MMA2 = mb + 8, MB_PART = mb + 16, MB_H = mb + 24, MB_Z = mb + 32,
                   MB_W = mb + 40, MB_NEVER = mb + 48, MB_W2 = mb + 56;
    const unsigned char *img = p.img + rank * p.img_stride;
    const uint32_t buf_u32 = tc::smem_u32(sBuf);

    // ---- resident part of this rank's weight image (W1, biases) ---------------
    {
        const uint4 *src = reinterpret_cast<const uint4 *>(img);
        uint4 *dst = reinterpret_cast<uint4 *>(smem);
        for (size_t i = tid; i < g.iwa / 16; i += NTHREADS) dst[i] = src[i];
    }
    // ---- initial operand tile and register state -----------------------------
    float c[UG], hs[UG], zs = 0.f;
    bool frozen = false;
    {
        const float *zsrc = p.teacher ? p.z_seq : p.z0;
        for (int k0 = 8 * grp; k0 < Z && !mma_warp; k0 += 8 * NGRP) {
            float v[8];
            for (int j = 0; j < 8; ++j) v[j] = live ? zsrc[(size_t)b * Z + k0 + j] : 0.f;
            x_store8(sX, row, k0, v);
        }
        for (int k0 = 8 * grp; k0 < H && !mma_warp; k0 += 8 * NGRP) {
            float v[8];
            for (int j = 0; j < 8; ++j) v[j] = (live && p.h0) ? p.h0[(size_t)b * H + k0 + j] : 0.f;
            x_store8(sX, row, Z + k0, v);
        }
#pragma unroll
        for (int j = 0; j < UG; ++j) {
            const size_t i = (size_t)b * H + rank * S::U + u0 + j;
            c[j] = (live && p.c0) ? p.c0[i] : 0.f;
            hs[j] = (live && p.h0) ? p.h0[i] : 0.f;
        }
        if (has_dim && live) zs = zsrc[(size_t)b * Z + dim];
        frozen = live && p.done0 && p.done0[b] != 0;
    }
    if (tid == 0) {
        for (int i = 0; i < 7; ++i) tc::mbar_init(mb + 8 * i, 1);
        tc::mbar_init(MB_W2, NT);  // every compute thread arrives once its part of W2 is stored
        tc::fence_mbar_init();
        // arm the exchange barriers for step 0; start the first W_a load
        tc::mbar_arrive_expect_tx(MB_PART, (CL - 1) * PART_BYTES);
        tc::mbar_arrive_expect_tx(MB_H, (CL - 1) * H_BYTES);
        tc::mbar_arrive_expect_tx(MB_Z, (CL - 1) * Z_BYTES);
        tc::mbar_arrive_expect_tx(MB_W, WA_BYTES);
        tc::bulk_load_global(buf_u32, img + g.iwa, WA_BYTES, MB_W);
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
    const uint32_t w1_u32 = tc::smem_u32(sW1);
    const uint32_t part_u32 = tc::smem_u32(part), zst_u32 = tc::smem_u32(zst);

    const uint32_t idesc1 = tc::idesc_bf16_f32(128, p.teacher ? S::NG : S::N1);
    const uint32_t idesc2 = tc::idesc_bf16_f32(128, S::N2);
    const uint32_t lboX = TILE * 16, lbo1 = S::N1 * 16, lbo2 = S::N2 * 16;
    // descriptor start addresses advance by 2 core matrices along K: 2*lbo bytes (>> 4)
    const uint64_t dX0 = tc::smem_desc(x_u32, lboX, 128), dW10 = tc::smem_desc(w1_u32, lbo1, 128);
    const uint64_t dW20 = tc::smem_desc(buf_u32, lbo2, 128);
    // MMA1 over k-blocks [kb0, kb1) of 16: z part is [0, Z/16), h part [Z/16, K1/16).
    // Every step accumulates the h part first, then the z part.
    auto mma1 = [&](int kb0, int kb1, bool acc_first) {
        uint64_t da = dX0 + (uint64_t)kb0 * (2 * lboX >> 4), db = dW10 + (uint64_t)kb0 * (2 * lbo1 >> 4);
        for (int kb = kb0; kb < kb1; ++kb) {
            tc::mma_bf16(tm, da, db, idesc1, (kb > kb0 || acc_first) ? 1u : 0u);
            da += 2 * lboX >> 4;
            db += 2 * lbo1 >> 4;
        }
    };
    // bounded waits: wait_one by a single thread, wait_bar by whole warps
    auto wait_one = [&](uint32_t bar, uint32_t parity) {
        if (!s_abort && !tc::mbar_wait_bounded(bar, parity, WAIT_POLLS)) {
            s_abort = 1;
            atomicExch(p.status, (int)WM_ERR_TIMEOUT);
        }
    };
    auto wait_bar = [&](uint32_t bar, uint32_t parity) {
        wait_one(bar, parity);
        __syncwarp();
    };
    const bool issuer = mma_warp && lane == 0;

    float nll_acc = 0.f;
    const int len_in = p.teacher && p.lengths ? p.lengths[live ? b : 0] : p.T;
    if (live && (len_in < 0 || len_in > p.T)) report_status(p.status, WM_ERR_INVALID_ARG);
    const int len = p.teacher ? min(max(len_in, 0), p.T) : 0;
    const unsigned long long ep = p.ep0 + (unsigned long long)b;
    const int M = 3 * KZ;
    // the mask word holding this rank's actions, prefetched one step ahead
    const int a0 = (int)rank * p.AC;
    uint32_t mword = 0xFFFFFFFFu;
    if (!p.teacher && grp == 0 && p.mask && live && p.T > 0) mword = __ldg(p.mask + (size_t)b * W + (a0 >> 5));

    // Injected wait (tests of the timeout path): one thread of every CTA waits on a barrier
    // that nothing completes, after the prologue's W_a load has landed and before any MMA or
    // exchange, so nothing of this kernel is in flight when it gives up.  Every CTA of the
    // cluster gives up the same way, records WM_ERR_TIMEOUT and skips all T steps; no CTA
    // then sends anything into another, and all of them still meet at the final cluster
    // barrier and free their TMEM.
    int t_end = p.T;
    if (p.test_wait) {
        if (tid == 0) {
            tc::mbar_wait_bounded(MB_W, 0, WAIT_POLLS);
            if (!tc::mbar_wait_bounded(MB_NEVER, 0, p.test_wait)) {
                s_abort = 1;
                atomicExch(p.status, (int)WM_ERR_TIMEOUT);
            }
        }
        __syncthreads();
        if (s_abort) t_end = 0;
    }

    if (issuer && t_end > 0) {  // MMA1 of step 0
        tc::fence_after_sync();
        mma1(Z / 16, K1 / 16, false);
        mma1(0, Z / 16, true);
        tc::mma_commit(MB_MMA1);
    }
    __syncwarp();  // the MMA warp reconverges before the next aligned barrier

    for (int t = 0; t < t_end; ++t) {
        const uint32_t step = p.t0 + (uint32_t)t;
        const size_t tb = (size_t)t * p.B + b;
        const uint32_t parity = (uint32_t)t & 1u;
        const bool last = t + 1 == p.T;

        // ---------------- gates + controller pre-activations ------------------
        float gv[4 * UG];
        uint32_t rc[16];  // controller columns (group 0)
        if (!mma_warp) {
            wait_bar(MB_MMA1, parity);
            tc::fence_after_sync();
            uint32_t rg[4 * UG];
            // all loads in flight before a single wait
#pragma unroll
            for (int c0 = 0; c0 < 4 * UG; c0 += 16) TC_LD16(tm + lane_base + 4 * UG * grp + c0, (rg + c0));
            if (grp == 0 && !p.teacher) TC_LD16(tm + lane_base + S::NG, rc);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 4 * UG; ++j) gv[j] = __uint_as_float(rg[j]);
        }
        if (grp == 0 && !mma_warp) {
            uint64_t rec = 0xFFFFFFFF00000000ull;  // index -1: nothing valid here
            if (!p.teacher) {
                // local masked argmax over this rank's actions (lowest index on ties); the
                // loop runs over the padded column count so that every register index is
                // static (a runtime bound put rc[] in local memory)
                float bv = -INFINITY;
                int bi = -1;
#pragma unroll
                for (int j = 0; j < S::NA; ++j) {
                    const int a = a0 + j;
                    const bool ok = j < p.AC && ((mword >> (a & 31)) & 1u);
                    const float v = __uint_as_float(rc[j]) + sB1[S::NG + j];
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
        push_to_peers<CL>(part_u32 + rank * PART_BYTES, PART_BYTES, MB_PART, rank, warp, lane, NT / 32);
        float hn[UG];
        int a = -1;
        if (!mma_warp) {
        wait_bar(MB_PART, parity);
        if (tid == 0) tc::mbar_arrive_expect_tx(MB_PART, (CL - 1) * PART_BYTES);

        // ---------------- action (a2) ----------------------------------------
        if (p.teacher) {
            if (live) {
                a = p.act_in[tb];
                if (a >= A) report_status(p.status, WM_ERR_INVALID_ARG);
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

        // ---------------- LSTM cell (a3, a4): UG units per thread -------------
        wait_bar(MB_W, parity);  // W_a is in the buffer (one load per step)
        {
            const float *bb = sB1 + 4 * UG * grp;
            const uint4 *src = reinterpret_cast<const uint4 *>(sBuf + (size_t)(a >= 0 ? a : 0) * S::WA_STRIDE +
                                                               8 * UG * grp);
#pragma unroll
            for (int q = 0; q < UG / 2; ++q) {  // 8 bf16 per 16-byte load
                const uint4 w4 = src[q];
                const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __nv_bfloat162 v2 = *reinterpret_cast<const __nv_bfloat162 *>(&wv[e]);
                    const int col = 8 * q + 2 * e;
                    const float w0 = a >= 0 ? __low2float(v2) : 0.f, w1 = a >= 0 ? __high2float(v2) : 0.f;
                    gv[col] += bb[col] + w0;
                    gv[col + 1] += bb[col + 1] + w1;
                }
            }
#pragma unroll
            for (int j = 0; j < UG; ++j) {
                if (frozen) {
                    hn[j] = hs[j];
                    continue;
                }
                const float gi = gv[j], gf = gv[UG + j], gg = gv[2 * UG + j], go = gv[3 * UG + j];
                c[j] = fast_sigmoid(gf) * c[j] + fast_sigmoid(gi) * fast_tanh(gg);
                hn[j] = fast_sigmoid(go) * fast_tanh(c[j]);
                hs[j] = hn[j];
            }
        }
        // h' (bf16) into this CTA's own tile; the rank's U/8 k-blocks are one contiguous block
        {
            unsigned char *dst = sX + tc::kmajor_offset(row, Z + rank * S::U + u0, TILE);
            uint32_t pk[UG / 2];
#pragma unroll
            for (int j = 0; j < UG / 2; ++j) pk[j] = pack_bf16x2(hn[2 * j], hn[2 * j + 1]);
            if constexpr (UG == 4) {
                *reinterpret_cast<uint2 *>(dst) = make_uint2(pk[0], pk[1]);
            } else {
                *reinterpret_cast<uint4 *>(dst) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
        }
        }  // !mma_warp
        tc::fence_proxy_async_smem();
        __syncthreads();  // every W_a read and h' write of this CTA is done
        const uint32_t hblk = x_u32 + tc::kmajor_offset(0, Z + rank * S::U, TILE);
        push_to_peers<CL>(hblk, H_BYTES, MB_H, rank, warp, lane, NT / 32);
        // W2 replaces W_a in the buffer while h' travels.  The compute threads copy it (L2 ->
        // registers -> shared memory): the TMA engine, which moves every exchange, is left to
        // the h' slices (with W2 in its queue too, MMA2 waited for both).
        if (!mma_warp) {
            const uint4 *src = reinterpret_cast<const uint4 *>(img + g.iw2);
            uint4 *dst = reinterpret_cast<uint4 *>(sBuf);
            constexpr int PER = (int)(S::N2 * 256 * 2 / 16 / NT);  // 16-byte chunks per thread (H = 256)
            static_assert(PER >= 1 && PER <= 8, "W2 chunks per thread");
            if ((int)(W2_BYTES / 16) == PER * NT) {
                uint4 v[PER];
#pragma unroll
                for (int i = 0; i < PER; ++i) v[i] = __ldg(src + tid + i * NT);
#pragma unroll
                for (int i = 0; i < PER; ++i) dst[tid + i * NT] = v[i];
            } else {
                for (int i = tid; i < (int)(W2_BYTES / 16); i += NT) dst[i] = __ldg(src + i);
            }
            tc::fence_proxy_async_smem();  // generic stores -> the MMA's reads
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(MB_W2) : "memory");
        }
        if (live) {
            const size_t o = tb * H + rank * S::U + u0;
            if (p.h_seq)
                for (int j = 0; j < UG; ++j) p.h_seq[o + j] = hs[j];
            if (p.c_seq)
                for (int j = 0; j < UG; ++j) p.c_seq[o + j] = c[j];
        }
        // this step's random numbers do not depend on the data: draw them while h' travels
        float u_dim = 0.f, eps_dim = 0.f;
        if (!mma_warp && has_dim && !p.teacher && !frozen && p.mdn_tau > 0.f) {
            u_dim = uniform_for_dim(p.seed, ep, step, dim);
            eps_dim = normal_for_dim(p.seed, ep, step, dim);
        }

        // ---------------- MMA2: heads (a5); then the h part of the next MMA1 ---
        if (issuer) {
            wait_one(MB_H, parity);  // h' of every rank is in X
            wait_one(MB_W2, parity);  // W2 is in the buffer
            if (!s_abort) {
                tc::fence_after_sync();
                uint64_t da = dX0 + ((uint64_t)Z * 256u >> 4), db = dW20;  // X_h: Z/8 k-blocks in
                for (int kb = 0; kb < H / 16; ++kb) {
                    tc::mma_bf16(tm + D2_COL, da, db, idesc2, kb > 0);
                    da += 2 * lboX >> 4;
                    db += 2 * lbo2 >> 4;
                }
                tc::mma_commit(MB_MMA2);
                // same issuing thread: runs after MMA2 and overlaps the sampling
                if (!last) mma1(Z / 16, K1 / 16, false);
            }
            if (!last) {  // W_a back into the buffer once MMA2 has read W2
                wait_one(MB_MMA2, parity);
                tc::mbar_arrive_expect_tx(MB_W, WA_BYTES);
                tc::bulk_load_global(buf_u32, img + g.iwa, WA_BYTES, MB_W);
            }
        }
        __syncwarp();
        float hv[16], zn = 0.f;
        int kc = 0;
        if (!mma_warp) {
        wait_bar(MB_H, parity);
        if (tid == 0) tc::mbar_arrive_expect_tx(MB_H, (CL - 1) * H_BYTES);
        wait_bar(MB_MMA2, parity);
        tc::fence_after_sync();
        {
            const int cg = has_dim ? grp : 0;
            uint32_t r[16];
            TC_LD16(tm + D2_COL + lane_base + 16 * cg, r);
            tc::tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < 16; ++j) hv[j] = __uint_as_float(r[j]) + sB2[16 * cg + j];
        }
        // reward is column 15 of group 0, the done logit column 15 of group 1
        const float rew = hv[15];

        // ---------------- mixture sample / NLL (a6, a7, a9): one dim per thread
        if (has_dim) {
            const float *lg = hv, *mu = hv + KM, *ls = hv + 2 * KM;
            if (p.teacher) {
                const float x = live ? p.z_seq[((size_t)(t + 1) * p.B + b) * Z + dim] : 0.f;
                float m = -INFINITY;
                for (int k = 0; k < KM; ++k) m = fmaxf(m, lg[k]);
                float s = 0.f;
                for (int k = 0; k < KM; ++k) s += expf(lg[k] - m);
                const float lse = m + logf(s);
                float lp[KM], tmax = -INFINITY;
                for (int k = 0; k < KM; ++k) {
                    const float zsc = (x - mu[k]) * expf(-ls[k]);
                    lp[k] = (lg[k] - lse) - 0.5f * zsc * zsc - ls[k] - 0.91893853320467274178f;
                    tmax = fmaxf(tmax, lp[k]);
                }
                float acc = 0.f;
                for (int k = 0; k < KM; ++k) acc += expf(lp[k] - tmax);
                if (t < len) nll_acc += -(tmax + logf(acc));
                zn = x;
            } else if (frozen) {
                zn = zs;
            } else if (!(p.mdn_tau > 0.f)) {
                float best = lg[0];
                zn = mu[0];
#pragma unroll
                for (int k = 1; k < KM; ++k)
                    if (lg[k] > best) { best = lg[k]; kc = k; zn = mu[k]; }
            } else {
                const float tau = p.mdn_tau;
                float m = -INFINITY;
                const float itau = __fdividef(1.f, tau);
                for (int k = 0; k < KM; ++k) m = fmaxf(m, lg[k] * itau);
                float pk[KM], s = 0.f;
                for (int k = 0; k < KM; ++k) { pk[k] = __expf(lg[k] * itau - m); s += pk[k]; }
                const float u = u_dim, is = __fdividef(1.f, s);
                // first k with u < C_k (else K-1), and its mu and log sigma by selects: every
                // register index static (mu[kc] with a runtime kc put hv[] in local memory)
                float cum = 0.f;
                uint32_t hit = 0u;
#pragma unroll
                for (int k = 0; k < KM - 1; ++k) {
                    cum += pk[k] * is;
                    hit |= (u < cum ? 1u : 0u) << k;
                }
                kc = hit ? __ffs(hit) - 1 : KM - 1;
                float muc = mu[0], lsc = ls[0];
#pragma unroll
                for (int k = 1; k < KM; ++k) {
                    muc = k == kc ? mu[k] : muc;
                    lsc = k == kc ? ls[k] : lsc;
                }
                const float scale = p.sigma_sqrt_tau ? sqrtf(tau) : 1.f;
                zn = muc + __expf(lsc) * scale * eps_dim;
            }
        }
        // ---------------- z' exchange, then the z part of the next MMA1 ------
        if (!p.teacher && has_dim) {
            __nv_bfloat16 zb = __float2bfloat16_rn(zn);
            zst[(rank * TILE + row) * ZD + grp] = *reinterpret_cast<uint16_t *>(&zb);
        }
        if (grp == 1) s_done_logit[row] = hv[15];
        tc::fence_proxy_async_smem();
        tc::fence_before_sync();
        sync_compute_warps();  // z' staged, done logit published
        if (!last && !p.teacher)
            push_to_peers<CL>(zst_u32 + rank * Z_BYTES, Z_BYTES, MB_Z, rank, warp, lane, NT / 32);
        const float dl = s_done_logit[row];
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
                    for (int k = 0; k < KM; ++k) {
                        ms[dim * KM + k] = zero ? 0.f : hv[k];
                        ms[KZ + dim * KM + k] = zero ? 0.f : hv[KM + k];
                        ms[2 * KZ + dim * KM + k] = zero ? 0.f : hv[2 * KM + k];
                    }
                }
            }
            if (!p.teacher && rank == 0) {
                const bool noop = p.noop_terminates && a == A - 1;
                if (grp == 0) p.rewards[tb] = frozen ? 0.f : rew;
                if (grp == 1) p.done[tb] = (frozen || dl > 0.f || noop) ? 1 : 0;
            }
        }
        }  // !mma_warp
        if (!last) {
            if (mma_warp) {
            } else if (!p.teacher) {
                wait_bar(MB_Z, parity);
                if (tid == 0) tc::mbar_arrive_expect_tx(MB_Z, (CL - 1) * Z_BYTES);
                // z' of all ranks -> this CTA's operand tile; group g packs k-blocks g, g+4, ...
                for (int k0 = 8 * grp; k0 < Z; k0 += 8 * NGRP) {
                    uint16_t v[8];
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const int d = k0 + j;
                        v[j] = zst[((d / ZD) * TILE + row) * ZD + d % ZD];
                    }
                    uint4 q;
                    q.x = v[0] | ((uint32_t)v[1] << 16);
                    q.y = v[2] | ((uint32_t)v[3] << 16);
                    q.z = v[4] | ((uint32_t)v[5] << 16);
                    q.w = v[6] | ((uint32_t)v[7] << 16);
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
            if (issuer && !s_abort) {
                tc::fence_after_sync();
                mma1(0, Z / 16, true);  // accumulate onto the h part issued after MMA2
                tc::mma_commit(MB_MMA1);
            }
            __syncwarp();
            if (!p.teacher && !mma_warp) {  // freezing (a8)
                const float dl = s_done_logit[row];
                if (!frozen) {
                    const bool noop = p.noop_terminates && a == A - 1;
                    if ((p.done_terminates && dl > 0.f) || noop) frozen = true;
                }
                zs = zn;
            }
        }
    }

    if (live) {
        const size_t o = (size_t)b * H + rank * S::U + u0;
        if (p.h_final)
            for (int j = 0; j < UG; ++j) p.h_final[o + j] = hs[j];
        if (p.c_final)
            for (int j = 0; j < UG; ++j) p.c_final[o + j] = c[j];
        if (p.teacher && has_dim) p.nll_part[(size_t)dim * p.B + b] = nll_acc;
    }
    tc::fence_before_sync();
    tc::cluster_sync();  // no CTA leaves while others may still write into it
    if (warp == 0) tc::tmem_dealloc(tm, 256);
}

// nll[n] = sum over the Z per-dim partials, in dim order.
__global__ void k_nll_reduce(int N, int parts, const float *part, float *nll) {
    const int n = blockIdx.x * blockDim.x + threadIdx.x;
    if (n >= N) return;
    double s = 0.0;
    for (int r = 0; r < parts; ++r) s += (double)part[(size_t)r * N + n];
    nll[n] = (float)s;
}

__global__ void k_copy_f32(size_t n, const float *src, float *dst) {
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
        dst[i] = src[i];
}

inline size_t host_kmajor(size_t r, size_t k, size_t R) {
    return ((k >> 3) * (R >> 3) + (r >> 3)) * 128 + (r & 7) * 16 + (k & 7) * 2;
}

inline void put_bf16(unsigned char *base, size_t off, float v) {
    __nv_bfloat16 q = __float2bfloat16_rn(v);
    memcpy(base + off, &q, 2);
}

template <class S>
bool shape_fits(const wm_config &c) {
    const int A = c.a_dim;
    return c.h_dim == S::CL * S::U && c.z_dim == S::CL * S::ZD && c.k_mix == S::KM && A % S::CL == 0 &&
           A / S::CL <= S::NA && 32 % (A / S::CL) == 0;  // a rank's actions sit in one mask word
}

// Builds the per-rank weight images of shape S; returns the device buffer (or null).
template <class S>
void *pack_images(const wm_config &c, const wm_weights *w, size_t *img_bytes, cudaError_t *err) {
    const int Z = c.z_dim, A = c.a_dim, H = c.h_dim, K = c.k_mix, AC = A / S::CL, U = S::U, UG = S::UG;
    const size_t K1 = Z + H, M = (size_t)3 * K * Z;
    const Geo g = geometry<S>(Z, A, H);
    std::vector<unsigned char> img(g.img * S::CL, 0);
    for (int r = 0; r < S::CL; ++r) {
        unsigned char *base = img.data() + (size_t)r * g.img;
        float *b1 = reinterpret_cast<float *>(base + g.b1);
        float *b2 = reinterpret_cast<float *>(base + g.b2);
        // W1 rows: group gi (4*UG columns) = i|f|g|o of units UG*gi.., then the controller
        for (int n = 0; n < S::N1; ++n) {
            if (n < S::NG) {
                const int gi = n / (4 * UG), within = n % (4 * UG), gate = within / UG, j = within % UG;
                const size_t col = (size_t)gate * H + (size_t)r * U + UG * gi + j;
                for (size_t k = 0; k < K1; ++k) {
                    const size_t src = k < (size_t)Z ? k : k + A;
                    put_bf16(base + g.w1, host_kmajor(n, k, S::N1), w->W_lstm[src * 4 * H + col]);
                }
                b1[n] = w->b_lstm[col];
                for (int a = 0; a < A; ++a)
                    put_bf16(base + g.iwa, (size_t)a * S::WA_STRIDE + (size_t)n * 2,
                             w->W_lstm[(size_t)(Z + a) * 4 * H + col]);
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
            } else if (within == 15 && i < 2) {
                special = i == 0 ? 1 : 2;
                bias = special == 1 ? w->b_rew : w->b_done;
            }
            for (int k = 0; k < H; ++k) {
                float v = 0.f;
                if (colsrc) v = colsrc[(size_t)k * M + col];
                else if (special == 1) v = w->w_rew[k];
                else if (special == 2) v = w->w_done[k];
                put_bf16(base + g.iw2, host_kmajor(n, k, S::N2), v);
            }
            b2[n] = bias;
        }
    }
    void *d = nullptr;
    *err = cudaMalloc(&d, img.size());
    if (*err != cudaSuccess) return nullptr;
    *err = cudaMemcpy(d, img.data(), img.size(), cudaMemcpyHostToDevice);
    if (*err != cudaSuccess) {
        cudaFree(d);
        return nullptr;
    }
    *img_bytes = g.img;
    return d;
}

// Raises k_fused<S>'s dynamic shared-memory limit on the current device to at least `bytes`,
// never lowering it: the geometry depends on A, and handles of other models may launch the
// same instantiation with more.
template <class S>
cudaError_t smem_at_least(size_t bytes) {
    static std::mutex mu;
    static size_t cur[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(mu);
    if (dev >= 0 && dev < 64 && bytes <= cur[dev]) return cudaSuccess;
    e = cudaFuncSetAttribute(k_fused<S>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess && dev >= 0 && dev < 64) cur[dev] = bytes;
    return e;
}

// How many clusters of shape S can be resident at once (0 if none).
template <class S>
int max_clusters(const wm_config &c) {
    const Geo g = geometry<S>(c.z_dim, c.a_dim, c.h_dim);
    int dev = 0, optin = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if ((size_t)optin < g.smem + 2048) return 0;
    if (smem_at_least<S>(g.smem) != cudaSuccess ||
        (S::CL > 8 && cudaFuncSetAttribute(k_fused<S>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                          cudaSuccess)) {
        cudaGetLastError();
        return 0;
    }
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = S::CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(S::CL);
    lc.blockDim = dim3(NTHREADS);
    lc.dynamicSmemBytes = g.smem;
    lc.attrs = at;
    lc.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, k_fused<S>, &lc) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

template <class S>
cudaError_t launch_fused(const wm_handle *h, int slot, FusedParams &p, cudaStream_t s) {
    const Geo g = geometry<S>(p.Z, p.A, p.H);
    const int nclusters = (p.B + TILE - 1) / TILE;
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = S::CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.gridDim = dim3(nclusters * S::CL);
    lc.blockDim = dim3(NTHREADS);
    lc.dynamicSmemBytes = g.smem;
    lc.stream = s;
    lc.attrs = at;
    lc.numAttrs = 1;
    p.img = (const unsigned char *)h->fused.img[slot];
    p.img_stride = h->fused.img_bytes[slot];
    p.AC = p.A / S::CL;
    p.status = h->status;
    const cudaError_t e = smem_at_least<S>(g.smem);
    if (e != cudaSuccess) return e;
    return cudaLaunchKernelEx(&lc, k_fused<S>, p);
}

// slot 0: 16-CTA clusters, slot 1: 8-CTA clusters.  Fewer waves wins; ties go to 16.
int choose_slot(const wm_handle *h, int B) {
    const int tiles = (B + TILE - 1) / TILE;
    const int m16 = h->fused.max_clusters[0], m8 = h->fused.max_clusters[1];
    if (h->fused.force_cluster == 8 && m8 > 0) return 1;
    if (h->fused.force_cluster == 16 && m16 > 0) return 0;
    if (m16 <= 0) return 1;
    if (m8 <= 0) return 0;
    const int w16 = (tiles + m16 - 1) / m16, w8 = (tiles + m8 - 1) / m8;
    return w8 < w16 ? 1 : 0;
}

cudaError_t launch_slot(const wm_handle *h, FusedParams &p, cudaStream_t s) {
    return choose_slot(h, p.B) == 0 ? launch_fused<S16>(h, 0, p, s) : launch_fused<S8>(h, 1, p, s);
}

FusedParams base_params(const wm_handle *h, int B, int T) {
    const wm_config &c = h->cfg;
    FusedParams p{};
    p.B = B; p.T = T; p.Z = c.z_dim; p.A = c.a_dim; p.H = c.h_dim;
    p.seed = c.seed; p.mdn_tau = c.mdn_tau; p.sigma_sqrt_tau = c.sigma_sqrt_tau;
    p.done_terminates = c.done_terminates; p.noop_terminates = c.noop_terminates;
    return p;
}

}  // namespace

// ---------------------------------------------------------------------------
// Whether the tcgen05 member takes the model: bf16, its shapes, masked argmax and the linear
// reward head.  The family's other member (wm_small.cu) takes small batches of the rest.
static int tc_member(const wm_handle *h) {
    const wm_config &c = h->cfg;
    if (!h->fused.ok) return 0;
    if (c.ctrl_sample && c.ctrl_tau > 0.f) return 0;  // masked argmax only
    if (c.reward_mode != WM_REWARD_HEAD) return 0;    // the linear reward head only
    return 1;
}

int wm_fused_supported(const wm_handle *h, int B) { return tc_member(h) || wm_small_supported(h, B); }

cudaError_t wm_fused_pack(wm_handle *h, const wm_weights *w) {
    const wm_config &c = h->cfg;
    h->fused.ok = 0;
    if (c.precision != WM_BF16 || !shape_fits<S16>(c) || !shape_fits<S8>(c)) return cudaSuccess;
    h->fused.max_clusters[0] = max_clusters<S16>(c);
    h->fused.max_clusters[1] = max_clusters<S8>(c);
    if (h->fused.max_clusters[0] <= 0 && h->fused.max_clusters[1] <= 0) return cudaSuccess;
    cudaError_t e = cudaSuccess;
    h->fused.img[0] = pack_images<S16>(c, w, &h->fused.img_bytes[0], &e);
    if (e != cudaSuccess) return e;
    h->fused.img[1] = pack_images<S8>(c, w, &h->fused.img_bytes[1], &e);
    if (e != cudaSuccess) return e;
    h->fused.ok = 1;
    return cudaSuccess;
}

void wm_fused_free(wm_handle *h) {
    for (int i = 0; i < 2; ++i) {
        cudaFree(h->fused.img[i]);
        h->fused.img[i] = nullptr;
    }
}

int wm_fused_cluster_size(const wm_handle *h, int B) { return choose_slot(h, B) == 0 ? S16::CL : S8::CL; }

cudaError_t wm_fused_rollout(const wm_handle *h, const wm_rollout_dev &a, cudaStream_t s) {
    if (!tc_member(h)) return wm_small_rollout(h, a, s);
    if (a.B == 0) { h->last_launches = 0; return cudaSuccess; }
    // z_out[0] = z0
    const size_t nz = (size_t)a.B * h->cfg.z_dim;
    {
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        k_copy_f32<<<(int)((nz + 255) / 256 < 1024 ? (nz + 255) / 256 : 1024), 256, 0, s>>>(nz, a.z0, a.z_out);
    }
    h->last_launches = 1;
    if (a.T == 0) {
        const size_t nh = (size_t)a.B * h->cfg.h_dim;
        int grid = (int)((nh + 255) / 256 < 1024 ? (nh + 255) / 256 : 1024);
        wm_ktime kt(h, WM_KERNEL_AUX, s);
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
    FusedParams p = base_params(h, a.B, a.T);
    p.teacher = 0;
    p.ep0 = a.ep0; p.t0 = a.t0;
    p.z0 = a.z0; p.h0 = a.h0; p.c0 = a.c0; p.done0 = a.done0; p.mask = a.mask;
    p.z_out = a.z_out; p.actions = a.actions; p.rewards = a.rewards; p.done = a.done;
    p.h_final = a.h_final; p.c_final = a.c_final; p.h_seq = a.h_seq; p.c_seq = a.c_seq;
    p.mdn_seq = a.mdn_seq; p.comp_seq = a.comp_seq;
    p.test_wait = h->test_wait;
    h->test_wait = 0;
    cudaError_t e;
    {
        wm_ktime kt(h, WM_KERNEL_FUSED, s);
        e = launch_slot(h, p, s);
    }
    h->last_launches = 2;
    return e != cudaSuccess ? e : cudaGetLastError();
}

size_t wm_fused_nll_ws(const wm_handle *h, int N) { return (size_t)h->cfg.z_dim * N * 4 + 256; }

cudaError_t wm_fused_nll(const wm_handle *h, const wm_nll_dev &a, void *ws, cudaStream_t s) {
    if (!tc_member(h)) return wm_small_nll(h, a, s);
    if (a.N == 0) { h->last_launches = 0; return cudaSuccess; }
    if (a.T == 0) {
        h->last_launches = 0;
        return cudaMemsetAsync(a.nll, 0, (size_t)a.N * 4, s);
    }
    FusedParams p = base_params(h, a.N, a.T);
    p.teacher = 1;
    p.z_seq = a.z_seq; p.act_in = a.actions; p.lengths = a.lengths;
    p.h_seq = a.h_seq; p.c_seq = a.c_seq; p.mdn_seq = a.mdn_seq;
    p.nll_part = (float *)ws;
    p.test_wait = h->test_wait;
    h->test_wait = 0;
    cudaError_t e;
    {
        wm_ktime kt(h, WM_KERNEL_FUSED, s);
        e = launch_slot(h, p, s);
    }
    if (e != cudaSuccess) return e;
    {
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        k_nll_reduce<<<(a.N + 127) / 128, 128, 0, s>>>(a.N, h->cfg.z_dim, p.nll_part, a.nll);
    }
    h->last_launches = 2;
    return cudaGetLastError();
}
