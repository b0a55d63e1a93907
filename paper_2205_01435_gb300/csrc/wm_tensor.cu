// wm_tensor.cu -- the tensor-core family for large batches: three persistent
// tcgen05 GEMMs per dream step, each with the step's math fused into its epilogue.
//
//   controller  [B, Z+H] x W_c^T [A, Z+H]   -> masked argmax / tempered draw    (a1, a2)
//   gates       [B, Z+H] x W_g^T [4H, Z+H]  -> + W_a[a_t] row, LSTM cell         (a3, a4)
//   heads       [B, H]   x W_h^T [Nh, H]    -> mixture sample (or NLL), reward,
//                                              done, freeze                       (a5..a9)
//
// Operands: bf16, K-major, loaded by TMA into 128-byte-swizzled shared-memory
// tiles (box 64 K x rows), consumed by tcgen05.mma.cta_group::2 (M = 256, a CTA
// pair per tile, each CTA holding 128 A rows and half of the B rows) with fp32
// accumulators in TMEM.  Each GEMM kernel is persistent (one CTA per SM, 256-row
// tiles in N-fastest order so that concurrently running pairs share the A rows in
// L2) and warp-specialised:
//   warp 0      TMA producer (both CTAs): a ring of STAGES stages of KPS k-steps,
//               one full and one empty mbarrier per stage,
//   warp 1      owns TMEM (512 columns, pair allocation); in the leader CTA it
//               issues the MMAs and commits once per stage; accumulators are
//               double-buffered when a tile is at most 256 columns wide, so the
//               epilogue of one tile overlaps the MMAs of the next,
//   warps 2..17 the epilogue: four warps per TMEM lane quadrant (one accumulator
//               row per thread), splitting the tile's columns.
// The operand X = [z_t | h_t] (bf16) is ping-ponged between two buffers: the
// gate epilogue writes h_{t+1} and the head epilogue z_{t+1} into the other one.
// The carried state c, h (fp32) lives in HBM.  All waits are bounded; on expiry a
// kernel records WM_ERR_TIMEOUT and stops waiting.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "tc_ptx.cuh"
#include "wm_device.cuh"
#include "wm_internal.h"

using namespace wmk;

namespace {

constexpr int BM = 128;          // rows per tile (MMA M)
constexpr int BK = 64;           // K per stage: one 128-byte swizzle row of bf16
constexpr int EPI_WARPS = 16;      // 4 per TMEM lane quadrant
constexpr int GEMM_THREADS = 64 + 32 * EPI_WARPS;
constexpr uint32_t POLLS = 1u << 26;
constexpr int HEAD_TILE = 240;   // head columns per tile (a multiple of 16 and of 24)

__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1u << 16;            // leading byte offset: unused for swizzled K-major
    d |= (uint64_t)(1024u >> 4) << 32;  // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1u << 46;            // descriptor version
    d |= (uint64_t)2u << 61;            // 128-byte swizzle
    return d;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint32_t mbar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        :: "r"(dst), "l"(map), "r"(x), "r"(y), "r"(mbar) : "memory");
}

// ---- CTA-pair (2-SM) forms: a pair computes a 256-row tile with one MMA stream issued
// by the leader CTA (cluster rank 0); each CTA holds its 128 rows of A and half of the B
// rows in its shared memory, and its 128 accumulator rows in its own TMEM.
__device__ __forceinline__ void tma_load_2sm(uint32_t dst, const CUtensorMap *map, int x, int y,
                                             uint32_t mbar_cluster) {  // completes on the leader's mbarrier
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        :: "r"(dst), "l"(map), "r"(x), "r"(y), "r"(mbar_cluster) : "memory");
}
__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.u32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate));
}
// arrive (once) on the mbarrier at this shared-memory offset in both CTAs of the pair when
// the leader's MMAs issued so far have completed
__device__ __forceinline__ void mma_commit_pair(uint32_t mbar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
        :: "r"(mbar), "h"((uint16_t)0x3) : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_saddr, uint32_t ncols) {  // a warp of each CTA
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" :: "r"(dst_saddr), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" :: "r"(taddr), "r"(ncols) : "memory");
}
// Relaxed: the epilogue's accumulator-empty arrive orders nothing in memory (the thread's
// TMEM loads have completed at tcgen05.wait::ld), and a release at cluster scope stalled
// the arriving thread for about 3K cycles per tile.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t mbar_cluster) {
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" :: "r"(mbar_cluster) : "memory");
}

// TMA store of a box from shared memory (bulk-group completion).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
                 :: "l"(map), "r"(x), "r"(y), "r"(src) : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// the shared-memory sources of this thread's committed stores have been read
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// ... and the stores are complete
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }


// Gate nonlinearities from the fast exponential (relative error ~1e-6).
// The cell's nonlinearities on the hardware tanh (tanh.approx.f32: one MUFU op, relative
// error about 2^-11); sigma(x) = (1 + tanh(x / 2)) / 2.
__device__ __forceinline__ float tanh_hw(float x) {
    float y;
    asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float sigmoid_hw(float x) { return fmaf(0.5f, tanh_hw(0.5f * x), 0.5f); }

struct GemmGrid {
    int m_tiles, n_tiles, k_steps;
    int a_col0;   // first K column of A (the heads read X from column Z)
    int *status;
    // B-operand rows per 256-row tile (controller population): tile m reads the B rows of
    // candidate ((ep0 + 256 m) / pop_E) mod pop_P, which start at row candidate * pop_rows
    unsigned long long ep0;
    int pop_P, pop_E, pop_rows;
    // failure injection (wm_inject_wait_timeout): > 0 makes the kernel wait, before it issues
    // any MMA or copy, on a barrier that nothing completes, at most this many polls
    uint32_t test_wait;
    // compacted live episodes: the rows to compute are *n_rows (written by the previous
    // kernel), not m_tiles * 256
    const int *n_rows;
};

// ---------------------------------------------------------------------------
// Epilogue parameters (device pointers; one step)
struct StepIO {
    int B, Z, A, H, K, T, t;
    uint32_t step;
    unsigned long long ep0, seed;
    int teacher, ctrl_sample, sigma_sqrt_tau, done_terminates, noop_terminates;
    int h32_mode;                   // when h (fp32) is stored: 0 never, 1 last step, 2 every step
    float ctrl_tau, mdn_tau;
    // state
    __nv_bfloat16 *x_cur, *x_next;  // [B, Z+H]
    __nv_bfloat16 *x_next_lo;       // fp32 path: the lo parts of x_next (else null)
    float *c, *h32;                 // [B, H]
    int32_t *act;                   // [B] the step's action
    const uint8_t *fz_cur;
    uint8_t *fz_next;
    // weights (packed orders, see wm_tc_pack)
    const float *b_ctrl, *b_gate, *b_head;
    const __nv_bfloat16 *wa;        // [A, 4H] gate-tile column order
    const __nv_bfloat16 *wa_lo;     // fp32 path: the lo parts of wa
    // head tiles
    int dims_per_tile, rd_tile, rd_col;  // reward / done columns: tile, first column
    // inputs / outputs
    const uint32_t *mask;           // [T, B, W] or null
    const int32_t *act_in;          // teacher: [T, B]
    const float *z_seq;             // teacher: [T+1, B, Z]
    // teacher: the head epilogue's targets, row e scores z_tgt[e]; nseq > 0: the rows are all
    // (step, sequence) pairs e = t nseq + n of a batched head GEMM (else the rows of step t)
    const float *z_tgt;
    int nseq;
    const int32_t *lengths;
    float *z_out;                   // [T+1, B, Z]
    int32_t *actions;
    float *rewards;
    uint8_t *done;
    float *h_seq, *c_seq, *mdn_seq;
    uint8_t *comp_seq;
    float *nll_part;                // [n_head_tiles, B]
    // shaped reward (Sec. 3.1.4, Eq. 2): columns rd_col + 2, + 3 predict runtime and memory
    // accesses; rt, mem carry each episode's last predictions
    int reward_mode;
    float alpha, beta, invalid_reward;
    const float *rt0, *mem0;
    float *rt, *mem, *rt_seq, *mem_seq;
    // controller population: episode e acts with candidate (e / pop_E) mod pop_P; b_ctrl is
    // [pop_P, A] (a 256-row tile belongs to one candidate)
    int pop_P, pop_E;
    float *logp_seq;                // log pi(a_t | z_t, h_t) of the action taken (optional)
    float *value_seq;               // value head at head column rd_col + nr - 1 (optional)
    int nr;                         // head columns from rd_col: reward, done (, rt, mem) (, value)
    // hierarchical action (n_xfers > 0): the controller GEMM writes its logits, a selection
    // kernel picks the xfer (act) and the location, whose action row n_xfers + location is
    // act2 (-1: none)
    int n_xfers;
    float *logits;                  // [B, A]
    const uint32_t *loc_mask;       // [T, B, NX, WL] or null
    int32_t *loc_actions;           // [T, B] optional
    int32_t *act2;                  // [B]
    // Compaction of the live episodes (rollouts whose episodes end): the step's GEMMs run
    // over the *n_rows live rows only, and row r holds episode rows[r].  Row-keyed: the
    // operands x, c, h32 and act, act2, logits, fz_cur, fz_next; episode-keyed: every [T, B]
    // input and output, rt, mem and the Philox counters.  Null: row b is episode b of B.
    const int32_t *rows;
    const int *n_rows;
    __device__ int live_rows() const { return n_rows ? *(volatile const int *)n_rows : B; }
    __device__ int ep_of(int r) const { return rows ? rows[r] : r; }
};

// Epilogue thread layout: 16 warps; warp w reads TMEM lanes 32*(w%4).. (the rows of
// quadrant w%4) and owns column group cg = (w-2)/4 of the tile.  The 4 groups of a
// quadrant cooperate through shared memory and a named barrier (ids 1..4).
//
// An epilogue may also stage data in a slab of shared memory per quadrant
// (QUAD_STAGE bytes, 1024-aligned): the quadrant's leader fills it by TMA
// (prefetch, signalled on the quadrant's mbarrier) and stores it back by TMA.
struct EpiCtx {
    int quad, cg, lane, row;
    float *red;  // [4 quad][4 group][32 lane][2] scratch for cross-group reductions
    unsigned char *stage;
    uint32_t stage_u, stage_bar, stage_phase;
    bool leader;        // lane 0 of the quadrant's first warp: issues the quadrant's TMA copies
    bool pending;       // leader: a prefetch not yet waited for (parity pending_phase)
    uint32_t pending_phase;
    const CUtensorMap *tm_c, *tm_xs, *tm_xs2;  // c; X_next (and its lo part, fp32 path)
    int *abort_flag, *status;
    __device__ void sync() const { asm volatile("bar.sync %0, 128;" :: "r"(1 + quad) : "memory"); }
    __device__ float *slot(int g) const { return red + ((quad * 4 + g) * 32 + lane) * 2; }
    __device__ void wait_stage() {
        if (!*abort_flag) {
            if (tc::mbar_wait_bounded(stage_bar, stage_phase, POLLS)) {
                pending = false;
            } else {
                *abort_flag = 1;
                atomicExch(status, (int)WM_ERR_TIMEOUT);
            }
        }
        stage_phase ^= 1u;
    }
    __device__ void note_prefetch() {
        pending = true;
        pending_phase = stage_phase;
    }
};

// ---- controller epilogue: A columns in TMEM, A/4 per column group ---------------
// Every thread of a warp issues the same TMEM loads (they are warp-collective);
// rows past B only skip their memory accesses.  The column group's columns are
// taken 16 at a time ("chunks"; A % 64 == 0 puts each chunk inside one mask word).
// The row's mask bits and frozen flag are loaded before the accumulator wait, and
// the bias is read from a copy in shared memory.  The tempered draw keeps each
// chunk's sum of weights, so only the chunk that holds the drawn point is read a
// third time.
struct EpiCtrl {
    static constexpr bool TMA_STAGE = false;
    static constexpr uint32_t QUAD_STAGE = 0;
    static constexpr int MAX_A = 512, NCH = MAX_A / 4 / 16;  // chunks per column group, at most
    static constexpr uint32_t RED_FLOATS = 4 * 4 * 32 * 2;
    // reductions | the bias, one copy per lane quadrant (a population's tiles change it)
    static constexpr uint32_t RED_BYTES = (RED_FLOATS + 4 * MAX_A) * 4;
    struct Pre {
        uint32_t bits[NCH];  // the chunk's 16 mask bits (0 for rows that do not act)
        bool live;           // a row of the batch whose episode is not frozen
        bool valid;          // a row of the batch
        int e;               // its episode
    };
    // once per CTA, by all 512 epilogue threads (e = 0..511), before the first tile: the
    // bias of a single controller into every quadrant's copy
    static __device__ void init(const StepIO &p, EpiCtx &x, int e) {
        if (p.pop_P > 1) return;
        for (int i = e; i < 4 * p.A; i += 32 * EPI_WARPS) x.red[RED_FLOATS + (i / p.A) * MAX_A + i % p.A] = p.b_ctrl[i % p.A];
    }
    static __device__ void prefetch(const StepIO &, int, int, EpiCtx &) {}
    static __device__ void pre(const StepIO &p, int m, int, EpiCtx &x, Pre &q) {
        const int b = m * BM + x.row;
        q.valid = b < p.live_rows();
        q.live = q.valid && !p.fz_cur[b];
        q.e = q.valid ? p.ep_of(b) : 0;
        const int A = p.A, W = (A + 31) >> 5, CW = A / 4, c_lo = x.cg * CW;
        const uint32_t *mw = (q.live && p.mask) ? p.mask + ((size_t)p.t * p.B + q.e) * W : nullptr;
#pragma unroll
        for (int k = 0; k < NCH; ++k) {
            const int c0 = c_lo + 16 * k;
            q.bits[k] = (!q.live || 16 * k >= CW) ? 0u : mw ? (mw[c0 >> 5] >> (c0 & 31)) & 0xFFFFu : 0xFFFFu;
        }
        if (p.pop_P > 1) {  // the tile's candidate's bias into the quadrant's copy (the previous
                            // tile's readers are past its closing barrier)
            const unsigned long long cand = ((p.ep0 + (unsigned long long)m * BM) / (unsigned long long)p.pop_E) %
                                            (unsigned long long)p.pop_P;
            const float *bc = p.b_ctrl + cand * p.A;
            float *bq = x.red + RED_FLOATS + x.quad * MAX_A;
            for (int i = x.cg * 32 + x.lane; i < A; i += 128) bq[i] = bc[i];
        }
    }
    // logits of chunk k (accumulator + bias)
    static __device__ __forceinline__ void chunk(uint32_t tacc, const float *bs, int c0, float (&v)[16]) {
        uint32_t r[16];
        TC_LD16(tacc + c0, r);
        const float4 *b4 = reinterpret_cast<const float4 *>(bs + c0);
        float bb[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float4 t = b4[i];
            bb[4 * i] = t.x; bb[4 * i + 1] = t.y; bb[4 * i + 2] = t.z; bb[4 * i + 3] = t.w;
        }
        tc::tmem_ld_wait();
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[j]) + bb[j];
    }
    // The per-column work is branch-free: each lane has its own mask bits, and a branch per
    // column splits the warp at every column (the mask is sparse).
    static __device__ __forceinline__ float ex2_approx(float x) {
        float y;
        asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
        return y;
    }
    // bit j of `bits` as an all-ones / all-zeros word
    static __device__ __forceinline__ uint32_t lane_mask(uint32_t bits, int j) { return 0u - ((bits >> j) & 1u); }
    static __device__ void run(const StepIO &p, uint32_t tacc, int m, int n, EpiCtx &x, const Pre &q, int, int) {
        (void)n;
        const int b = m * BM + x.row;
        const bool valid = q.valid, live = q.live;
        const int CW = p.A / 4, c_lo = x.cg * CW, nch = CW / 16;  // nch is warp-uniform
        const float *bs = x.red + RED_FLOATS + x.quad * MAX_A;
        if (p.pop_P > 1) x.sync();  // the quadrant's bias copy (pre) is complete
        // pass 1: masked argmax over this group's columns (lowest index on ties): per chunk,
        // the maximum of the valid logits, then the lowest valid column that attains it
        int a = -1, last_v = -1;
        float bv = -INFINITY;
#pragma unroll
        for (int k = 0; k < NCH; ++k) {
            if (k >= nch) break;
            const int c0 = c_lo + 16 * k;
            float v[16];
            chunk(tacc, bs, c0, v);
            const uint32_t bits = q.bits[k];
            float mx = -INFINITY;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                v[j] = __uint_as_float((__float_as_uint(v[j]) & lane_mask(bits, j)) |
                                       (0xff800000u & ~lane_mask(bits, j)));  // -inf where masked
                mx = fmaxf(mx, v[j]);
            }
            uint32_t eq = 0u;
#pragma unroll
            for (int j = 0; j < 16; ++j) eq |= (v[j] == mx ? 1u : 0u) << j;
            eq &= bits;
            const bool better = eq != 0u && (a < 0 || mx > bv);
            bv = better ? mx : bv;
            a = better ? c0 + __ffs(eq) - 1 : a;
            last_v = bits ? c0 + 31 - __clz(bits) : last_v;
        }
        float *my = x.slot(x.cg);
        my[0] = bv;
        my[1] = __int_as_float(a);
        x.sync();
        int ga = -1;
        float gbv = -INFINITY;
        for (int g = 0; g < 4; ++g) {  // groups in column order: ties keep the lower index
            const float *o = x.slot(g);
            const int i = __float_as_int(o[1]);
            if (i >= 0 && (ga < 0 || o[0] > gbv)) { gbv = o[0]; ga = i; }
        }
        const bool sampled = p.ctrl_sample && p.ctrl_tau > 0.f;         // uniform over the warp
        const bool want_lp = p.logp_seq != nullptr && p.ctrl_tau > 0.f;  // log pi(a) requested
        float logp = 0.f;
        if (sampled || want_lp) {
            const bool draw = live && ga >= 0;
            // weight of logit v: exp((v - max) / tau) = 2^(v * s - max * s), s = log2(e) / tau;
            // a masked column's weight is forced to +0 (its logit may exceed the maximum)
            const float sc = 1.4426950408889634f / p.ctrl_tau, off = -gbv * sc;
            // pass 2: the group's sum of tempered weights, chunk by chunk
            float cs[NCH], S = 0.f;
#pragma unroll
            for (int k = 0; k < NCH; ++k) {
                cs[k] = 0.f;
                if (k >= nch) continue;
                float v[16];
                chunk(tacc, bs, c_lo + 16 * k, v);
                const uint32_t bits = draw ? q.bits[k] : 0u;
                float sk = 0.f;
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    sk += __uint_as_float(__float_as_uint(ex2_approx(fmaf(v[j], sc, off))) & lane_mask(bits, j));
                cs[k] = sk;
                S += sk;
            }
            x.sync();  // everyone has read the argmax partials
            my[0] = S;
            my[1] = __int_as_float(last_v);
            x.sync();
            float total = 0.f, prefix = 0.f;
            int glast = -1;
            for (int g = 0; g < 4; ++g) {
                const float *o = x.slot(g);
                if (g < x.cg) prefix += o[0];
                total += o[0];
                glast = max(glast, __float_as_int(o[1]));
            }
            const float itau = 1.f / p.ctrl_tau, log_total = logf(total);
            if (!sampled) {
                logp = draw ? -log_total : 0.f;  // the argmax: its logit is the maximum
            } else {
                const float u = draw ? to_uniform(rng_draw(p.seed, p.ep0 + q.e, p.step, RNG_CONTROLLER, 0).x) : 0.f;
                const float target = u * total;
                // the group holding the drawn point; if rounding puts the target at or past the
                // total, the group holding the last valid action
                const bool mine = draw && ((target >= prefix && target < prefix + S) ||
                                           (target >= total && last_v == glast));
                // the chunk holding the drawn point (the group's last chunk with a valid
                // action if rounding carries the running sum past the target)
                int kc = -1, klast = -1;
                float base = prefix;
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    if (k >= nch || !mine) continue;
                    if (q.bits[k]) klast = k;
                    if (kc < 0) {
                        if (target < base + cs[k]) kc = k;
                        else base += cs[k];
                    }
                }
                if (mine && kc < 0) {
                    kc = klast;
                    base = prefix;
                    for (int k = 0; k < NCH; ++k)
                        if (k < klast) base += cs[k];
                }
                // pass 3: only chunks some row of the warp needs
                int chosen = -1;
                float lv = 0.f;  // the chosen column's logit
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    if (k >= nch) break;
                    if (!__any_sync(0xffffffffu, kc == k)) continue;
                    float v[16];
                    chunk(tacc, bs, c_lo + 16 * k, v);
                    if (kc != k) continue;
                    const uint32_t bits = q.bits[k];
                    float cum = base;
                    uint32_t hit = 0u;  // valid columns at which the running sum has passed the target
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        cum += __uint_as_float(__float_as_uint(ex2_approx(fmaf(v[j], sc, off))) & lane_mask(bits, j));
                        hit |= (target < cum ? 1u : 0u) << j;
                    }
                    hit &= bits;
                    // the first such column; rounding: the chunk's last valid action
                    const int jj = hit ? __ffs(hit) - 1 : (bits ? 31 - __clz(bits) : -1);
                    chosen = jj >= 0 ? c_lo + 16 * k + jj : -1;
#pragma unroll
                    for (int j = 0; j < 16; ++j) lv = j == jj ? v[j] : lv;
                }
                x.sync();  // everyone has read the sum partials
                my[0] = lv;
                my[1] = __int_as_float(chosen);
                x.sync();
                int pick = -1;
                float lvp = 0.f;
                for (int g = 0; g < 4; ++g) {
                    const int c = __float_as_int(x.slot(g)[1]);
                    if (c > pick) { pick = c; lvp = x.slot(g)[0]; }
                }
                if (draw) {
                    ga = pick >= 0 ? pick : glast;  // rounding past the last valid action
                    logp = pick >= 0 ? (lvp - gbv) * itau - log_total : 0.f;
                }
            }
        }
        x.sync();  // the scratch is reused by the next tile
        if (!valid || x.cg != 0) return;
        if (!live) ga = -1;
        p.act[b] = ga;
        const size_t tb = (size_t)p.t * p.B + q.e;
        p.actions[tb] = ga;
        if (p.logp_seq) p.logp_seq[tb] = ga >= 0 ? logp : 0.f;
    }
};


// ---- controller logits epilogue (hierarchical actions): every live row's A logits plus
// its candidate's bias to a [B, A] buffer; the two-stage choice is made by k_tc_select.
// Column group g stores its A/4 columns, 16 at a time (64 contiguous bytes per row).
struct EpiLogits {
    static constexpr bool TMA_STAGE = false;
    static constexpr uint32_t QUAD_STAGE = 0;
    static constexpr uint32_t RED_BYTES = 0;
    struct Pre {};
    static __device__ void init(const StepIO &, EpiCtx &, int) {}
    static __device__ void prefetch(const StepIO &, int, int, EpiCtx &) {}
    static __device__ void pre(const StepIO &, int, int, EpiCtx &, Pre &) {}
    static __device__ void run(const StepIO &p, uint32_t tacc, int m, int, EpiCtx &x, const Pre &, int, int) {
        const int b = m * BM + x.row;
        const int nrows = p.live_rows();
        const bool store = b < nrows && !p.fz_cur[b < nrows ? b : 0];  // frozen rows choose nothing
        const int CW = p.A / 4, c_lo = x.cg * CW, nch = CW / 16;  // nch is warp-uniform
        const unsigned long long cand =
            p.pop_P > 1 ? ((p.ep0 + (unsigned long long)m * BM) / (unsigned long long)p.pop_E) % (unsigned long long)p.pop_P
                        : 0ull;
        const float *bias = p.b_ctrl + cand * p.A;
        float *out = p.logits + (size_t)(b < p.B ? b : 0) * p.A;
        for (int k = 0; k < nch; ++k) {  // every lane issues the (warp-collective) TMEM loads
            const int c0 = c_lo + 16 * k;
            uint32_t r[16];
            TC_LD16(tacc + c0, r);
            tc::tmem_ld_wait();
            if (!store) continue;
            const float4 *b4 = reinterpret_cast<const float4 *>(bias + c0);
            float4 *o4 = reinterpret_cast<float4 *>(out + c0);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float4 t = b4[i];
                o4[i] = make_float4(__uint_as_float(r[4 * i]) + t.x, __uint_as_float(r[4 * i + 1]) + t.y,
                                    __uint_as_float(r[4 * i + 2]) + t.z, __uint_as_float(r[4 * i + 3]) + t.w);
            }
        }
    }
};

// The hierarchical choice (Sec. 3.1.3) from the stored logits, one warp per episode: the
// xfer among the first NX under the xfer mask, then (unless it is the NO-OP) the location
// among the other L under that xfer's location mask.
__global__ void __launch_bounds__(256) k_tc_select(StepIO p) {
    const int warp = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    if (warp >= p.live_rows()) return;
    const int b = warp, A = p.A, NX = p.n_xfers, L = A - NX, W = (A + 31) >> 5, WL = (L + 31) >> 5;
    const int e = p.ep_of(b);
    const size_t tb = (size_t)p.t * p.B + e;
    int x = -1, loc = -1;
    float lp = 0.f;
    if (!p.fz_cur[b]) {
        WarpSelect ws;
        ws.sample = p.ctrl_sample && p.ctrl_tau > 0.f;
        ws.tau = p.ctrl_tau;
        ws.want_lp = p.logp_seq != nullptr;
        ws.seed = p.seed;
        ws.episode = p.ep0 + e;
        ws.step = p.step;
        const float *l = p.logits + (size_t)b * A;
        const uint32_t *mw = p.mask ? p.mask + tb * W : nullptr;
        x = warp_select(ws, l, NX, mw, 0, &lp);
        if (x >= 0 && x != NX - 1) {
            const uint32_t *lmw = p.loc_mask ? p.loc_mask + (tb * NX + x) * WL : nullptr;
            float lpl = 0.f;
            loc = warp_select(ws, l + NX, L, lmw, 1, &lpl);
            lp += lpl;
        }
    }
    if (lane == 0) {
        p.act[b] = x;
        p.act2[b] = loc >= 0 ? NX + loc : -1;
        p.actions[tb] = x;
        if (p.loc_actions) p.loc_actions[tb] = loc;
        if (p.logp_seq) p.logp_seq[tb] = lp;
    }
}

// ---- gate epilogue: 64 units per tile, columns [i | f | g | o] x 64; 16 units per group
// The quadrant's c rows (32 x 64 fp32) and h' rows (32 x 64 bf16) go through
// shared memory in the 128-byte-swizzled layout of TMA boxes 128 bytes wide,
// so that every global access of the cell is a full-row TMA box instead of 32
// rows per instruction: c is loaded by TMA, updated in place and stored back by
// TMA; h' is stored by TMA into X_next.  The next tile's c is loaded as soon as
// the stores have read the slab.  (Separate in- and out-slabs, refilled
// mid-tile, measured slower: the extra quadrant barrier costs more than the
// load latency it hides.)  The cell is formed gate by gate over the thread's 16
// units, so that each gate's W_a segment is one 256-bit load.  TWO: a hierarchical action
// adds a second action row (the location's) to every gate.
// MODE 0: one action row, bf16 path.  MODE 1: two action rows (hierarchical action).
// MODE 2: the fp32 path: the action row is gathered as its bf16 hi and lo parts (the two-row
// machinery with the same action), the nonlinearities are the accurate ones, and h' is
// stored as bf16 hi and lo parts.
// UNITS: hidden units per tile (64: a 256-column tile; 32: a 128-column tile, for calls with
// few row tiles, where twice the tiles keep twice the CTA pairs busy and each tile's
// epilogue is half as long).  Each thread of a quadrant's 4 column groups takes UT units.
template <int MODE, int UNITS = 64>
struct EpiGatesT {
    static constexpr bool TWO = MODE != 0, F32 = MODE == 2;
    static constexpr int UT = UNITS / 4, WW = UT / 2;  // units per thread, W_a words per gate
    static_assert(UNITS == 64 || UNITS == 32, "gate tile of 64 or 32 units");
    static constexpr uint32_t C_SLAB = 32 * UNITS * 4;  // UNITS / 32 boxes of 32 fp32 x 32 rows
    static constexpr uint32_t X_SLAB = 32 * UNITS * 2;  // one box of UNITS bf16 x 32 rows
    static constexpr uint32_t QUAD_STAGE = C_SLAB + (F32 ? 2 : 1) * X_SLAB;  // c (in place) | h' out (| h' lo)
    static constexpr bool TMA_STAGE = true;
    static constexpr uint32_t RED_BYTES = 0;

    // byte offset of (row r, 16-byte chunk j) in a 128-byte-swizzled box
    static __device__ __forceinline__ uint32_t sw(int r, int j) { return r * 128 + ((j ^ (r & 7)) << 4); }
    // the h' slab: a 128-byte-swizzled box of 64 units, or a plain 64-byte-row box of 32
    static __device__ __forceinline__ uint32_t xsw(int r, int j) { return UNITS == 64 ? sw(r, j) : r * 64 + (j << 4); }

    // leader of a quadrant: TMA load of the c rows of 128-row block m, unit tile n
    static __device__ void prefetch(const StepIO &, int m, int n, EpiCtx &x) {
        x.note_prefetch();
        tc::mbar_arrive_expect_tx(x.stage_bar, C_SLAB);
        for (int bx = 0; bx < UNITS / 32; ++bx)
            tma_load_2d(x.stage_u + bx * 4096, x.tm_c, UNITS * n + 32 * bx, m * BM + 32 * x.quad, x.stage_bar);
    }

    struct Pre {
        uint32_t wi[WW], wg[WW];    // the W_a row segments of gates i and g (UT units, bf16)
        uint32_t wi2[WW], wg2[WW];  // TWO: the second action row's (F32: the lo parts)
        int a, a2;                // the action rows (-1: none)
        bool fz;                  // frozen episode
        int e;                    // the row's episode
    };
    static __device__ void init(const StepIO &, EpiCtx &, int) {}
    // one gate's W_a segment for the thread's 16 units: a single 32-byte sector, read with
    // one 256-bit load (half the L1 wavefronts of two 16-byte loads: each lane reads
    // another row, so every load instruction touches 32 lines)
    static __device__ __forceinline__ void ld_wa(const StepIO &p, int a, int n, int q, int gate, uint32_t (&w)[WW],
                                                 bool lo = false) {
        if (a < 0) {
#pragma unroll
            for (int i = 0; i < WW; ++i) w[i] = 0u;
            return;
        }
        const __nv_bfloat16 *src =
            (lo ? p.wa_lo : p.wa) + (size_t)a * 4 * p.H + 4 * UNITS * n + UNITS * gate + UT * q;
        if constexpr (WW == 8)
            asm volatile("ld.global.nc.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                         : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]), "=r"(w[7])
                         : "l"(src));
        else
            asm volatile("ld.global.nc.v4.b32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]) : "l"(src));
    }
    // before the accumulator wait: the row's action and the W_a segments of gates i and g
    // (L2 gathers), so that their latency overlaps the mainloop
    static __device__ void pre(const StepIO &p, int m, int n, EpiCtx &x, Pre &pr) {
        const int b = m * BM + x.row;
        const bool valid = b < p.live_rows();
        const int bb = valid ? b : 0;
        pr.fz = p.fz_cur[bb] != 0;
        pr.e = p.ep_of(bb);
        int a = p.act[bb];
        if (p.teacher) {
            a = p.act_in[(size_t)p.t * p.B + pr.e];
            if (a >= p.A && valid && n == 0 && x.cg == 0) report_status(x.status, WM_ERR_INVALID_ARG);
            if (a < 0 || a >= p.A) a = -1;
        }
        pr.a = (a >= 0 && a < p.A && !pr.fz) ? a : -1;
        ld_wa(p, pr.a, n, x.cg, 0, pr.wi);
        ld_wa(p, pr.a, n, x.cg, 2, pr.wg);
        if (TWO) {
            if (F32) {
                pr.a2 = pr.a;
            } else {
                const int a2 = p.act2[bb];
                pr.a2 = (a2 >= 0 && a2 < p.A && !pr.fz) ? a2 : -1;
            }
            ld_wa(p, pr.a2, n, x.cg, 0, pr.wi2, F32);
            ld_wa(p, pr.a2, n, x.cg, 2, pr.wg2, F32);
        }
    }
    // the cell's nonlinearities: the hardware tanh on the bf16 path; accurate ones on the
    // fp32 path (tanh.approx's relative error, about 2^-11, is above its tolerance)
    static __device__ __forceinline__ float sig_(float x) { return F32 ? fmaf(0.5f, tanhf(0.5f * x), 0.5f) : sigmoid_hw(x); }
    static __device__ __forceinline__ float tanh_(float x) { return F32 ? tanhf(x) : tanh_hw(x); }
    // pre-activations of one gate for the thread's 16 units: accumulator + bias + W_a[a]
    // (+ W_a[a2] when TWO)
    static __device__ __forceinline__ void gate_pre(uint32_t tacc, const float *bg, int gate, int ut,
                                                    const uint32_t (&w)[WW], const uint32_t (&w2)[WW],
                                                    float (&g)[UT]) {
#pragma unroll
        for (int h = 0; h < UT / 8; ++h) {  // 8 columns per TMEM load: fewer registers held
            uint32_t r[8];
            TC_LD8(tacc + UNITS * gate + ut + 8 * h, r);
            tc::tmem_ld_wait();
            // the bias is read after the wait (an L1 hit), so that it is not held across it
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                const float4 t = *reinterpret_cast<const float4 *>(bg + UNITS * gate + 8 * h + 4 * i);
                const float bv[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int k = 8 * h + 4 * i + 2 * e;  // unit (column) index in 0..UT-1
                    const __nv_bfloat162 v2 = *reinterpret_cast<const __nv_bfloat162 *>(&w[k / 2]);
                    g[k] = __uint_as_float(r[4 * i + 2 * e]) + bv[2 * e] + __low2float(v2);
                    g[k + 1] = __uint_as_float(r[4 * i + 2 * e + 1]) + bv[2 * e + 1] + __high2float(v2);
                    if (TWO) {
                        const __nv_bfloat162 u2 = *reinterpret_cast<const __nv_bfloat162 *>(&w2[k / 2]);
                        g[k] += __low2float(u2);
                        g[k + 1] += __high2float(u2);
                    }
                }
            }
        }
    }

    static __device__ void run(const StepIO &p, uint32_t tacc, int m, int n, EpiCtx &x, const Pre &pr, int next_m,
                               int next_n) {
        const int b = m * BM + x.row;
        const bool valid = b < p.live_rows();
        const int bb = valid ? b : 0;  // rows past the batch compute on row 0; TMA stores clip them
        const int H = p.H, r = x.lane, q = x.cg;
        const bool fz = pr.fz;
        const int ut = UT * q, u0 = UNITS * n + ut;  // the thread's first unit: in the tile, in H
        // gates f and o: loaded while i and g are computed
        uint32_t wf[WW], wo[WW], wf2[WW], wo2[WW];
        ld_wa(p, pr.a, n, q, 1, wf);
        ld_wa(p, pr.a, n, q, 3, wo);
        if (TWO) {
            ld_wa(p, pr.a2, n, q, 1, wf2, F32);
            ld_wa(p, pr.a2, n, q, 3, wo2, F32);
        }
        const float *bg = p.b_gate + 4 * UNITS * n + UT * q;
        const bool store_h32 = valid && !fz && (p.h32_mode == 2 || (p.h32_mode == 1 && p.t == p.T - 1));
        unsigned char *cs = x.stage, *xs = x.stage + C_SLAB;
        // the thread's UT c values: UT / 4 chunks of the swizzled box that holds units ut..
        const uint32_t cbox = (ut >> 5) * 4096, cch = (ut & 31) >> 2;
        // Every lane forms all four gates: the TMEM loads are warp-collective, and the rows
        // of a warp may be frozen or not; a frozen row keeps its c and its carried h.
        float cv[UT], hv[UT];
        {  // hv = sigma(i) * tanh(g), one gate's pre-activations live at a time
            float g[UT];
            gate_pre(tacc, bg, 0, ut, pr.wi, pr.wi2, g);
#pragma unroll
            for (int j = 0; j < UT; ++j) hv[j] = sig_(g[j]);
            gate_pre(tacc, bg, 2, ut, pr.wg, pr.wg2, g);
#pragma unroll
            for (int j = 0; j < UT; ++j) hv[j] *= tanh_(g[j]);
        }
        x.wait_stage();  // the quadrant's c rows have landed
#pragma unroll
        for (int i = 0; i < UT / 4; ++i) {
            const float4 t = *reinterpret_cast<const float4 *>(cs + cbox + sw(r, cch + i));
            cv[4 * i] = t.x; cv[4 * i + 1] = t.y; cv[4 * i + 2] = t.z; cv[4 * i + 3] = t.w;
        }
        {
            float g[UT];
            gate_pre(tacc, bg, 1, ut, wf, wf2, g);
            if (!fz) {
#pragma unroll
                for (int j = 0; j < UT; ++j) cv[j] = sig_(g[j]) * cv[j] + hv[j];
            }
            gate_pre(tacc, bg, 3, ut, wo, wo2, g);
#pragma unroll
            for (int j = 0; j < UT; ++j) hv[j] = sig_(g[j]) * tanh_(cv[j]);
        }
        if (fz) {  // frozen: h is the carried one
            const float4 *h4 = reinterpret_cast<const float4 *>(p.h32 + (size_t)bb * H + u0);
#pragma unroll
            for (int i = 0; i < UT / 4; ++i) {
                const float4 t = h4[i];
                hv[4 * i] = t.x; hv[4 * i + 1] = t.y; hv[4 * i + 2] = t.z; hv[4 * i + 3] = t.w;
            }
        }
#pragma unroll
        for (int i = 0; i < UT / 4; ++i)
            *reinterpret_cast<float4 *>(cs + cbox + sw(r, cch + i)) =
                make_float4(cv[4 * i], cv[4 * i + 1], cv[4 * i + 2], cv[4 * i + 3]);
#pragma unroll
        for (int i = 0; i < UT / 8; ++i) {
            uint32_t pk[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                __nv_bfloat162 v = __floats2bfloat162_rn(hv[8 * i + 2 * j], hv[8 * i + 2 * j + 1]);
                pk[j] = *reinterpret_cast<uint32_t *>(&v);
            }
            *reinterpret_cast<uint4 *>(xs + xsw(r, (ut >> 3) + i)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            if (F32) {  // the lo parts, h' - bf16(h')
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float a0 = hv[8 * i + 2 * j], a1 = hv[8 * i + 2 * j + 1];
                    __nv_bfloat162 hi2 = *reinterpret_cast<__nv_bfloat162 *>(&pk[j]);
                    __nv_bfloat162 v = __floats2bfloat162_rn(a0 - __low2float(hi2), a1 - __high2float(hi2));
                    pk[j] = *reinterpret_cast<uint32_t *>(&v);
                }
                *reinterpret_cast<uint4 *>(xs + X_SLAB + xsw(r, (ut >> 3) + i)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
        }
        if (store_h32) {
            float4 *h4 = reinterpret_cast<float4 *>(p.h32 + (size_t)b * H + u0);
#pragma unroll
            for (int i = 0; i < UT / 4; ++i) h4[i] = make_float4(hv[4 * i], hv[4 * i + 1], hv[4 * i + 2], hv[4 * i + 3]);
        }
        if (valid) {
            const size_t o = ((size_t)p.t * p.B + pr.e) * H + u0;
            if (p.h_seq)
                for (int j = 0; j < UT; ++j) p.h_seq[o + j] = hv[j];
            if (p.c_seq)
                for (int j = 0; j < UT; ++j) p.c_seq[o + j] = cv[j];
        }
        // the slab's generic-proxy reads and writes are ordered before the TMA (async-proxy)
        // stores and the refill by this fence and the barrier
        tc::fence_proxy_async_smem();
        x.sync();
        if (x.leader) {
            const int y = m * BM + 32 * x.quad;
            if (y < p.B) {  // rows past B are clipped by the stores; a slab wholly past B is skipped
                for (int bx = 0; bx < UNITS / 32; ++bx) tma_store_2d(x.tm_c, UNITS * n + 32 * bx, y, x.stage_u + 4096 * bx);
                tma_store_2d(x.tm_xs, p.Z + UNITS * n, y, x.stage_u + C_SLAB);
                if (F32) tma_store_2d(x.tm_xs2, p.Z + UNITS * n, y, x.stage_u + C_SLAB + X_SLAB);
                bulk_commit();
                bulk_wait_read();  // the slab may be refilled
            }
            if (next_m >= 0) prefetch(p, next_m, next_n, x);
        }
    }
};

using EpiGates = EpiGatesT<0>;
using EpiGates2 = EpiGatesT<1>;
using EpiGates32 = EpiGatesT<2>;
using EpiGatesN = EpiGatesT<0, 32>;  // 128-column tiles (few row tiles)
using EpiGates32N = EpiGatesT<2, 32>;  // the same, fp32 path (teacher-forced scoring)

// ---- head epilogue: dims_per_tile latent dims, DS columns each; reward / done -----
// Before the accumulator wait, the quadrant's 128 threads make the tile's random draws:
// thread (row, g) takes Philox blocks first + g, first + g + 4, ... (4 dims per block, so
// each block's two draws are made once per row) and leaves every (row, dim)'s uniform and
// Box-Muller normal in shared memory; the tile's bias is copied there too.  After the
// wait, column group g takes dims g, g + 4, ... (balanced: 10 dims go 3, 3, 2, 2).  The
// quadrant's z' values are staged in shared memory ([32 rows][33], conflict-free) and
// stored by all 128 threads in row-major order, so a warp's stores cover a few contiguous
// row segments instead of 32 rows.
struct EpiHeads {
    static constexpr bool TMA_STAGE = false;
    static constexpr int ZS_PITCH = 33;
    static constexpr uint32_t ZS_BYTES = 32 * ZS_PITCH * 4;  // [32 rows][<= 32 dims] floats
    static constexpr uint32_t ZS_ALIGNED = (ZS_BYTES + 15) & ~15u;
    static constexpr uint32_t US_OFF = ZS_ALIGNED, BIAS_OFF = 2 * ZS_ALIGNED;
    // normal draws, then z' | uniform draws | the tile's bias (+ 16 floats: a dim's six
    // float4 reads pass the tile's end by up to 16 when 3K < 24)
    static constexpr uint32_t QUAD_STAGE = BIAS_OFF + (HEAD_TILE + 16) * 4;
    static constexpr uint32_t RED_BYTES = 0;
    struct Pre {};
    static __device__ void init(const StepIO &, EpiCtx &, int) {}
    static __device__ void prefetch(const StepIO &, int, int, EpiCtx &) {}
    // the tile's HEAD_TILE bias values, by the quadrant's 128 threads (the previous tile's
    // readers are past its closing barrier)
    static __device__ void pre(const StepIO &p, int m, int n, EpiCtx &x, Pre &) {
        float *bq = reinterpret_cast<float *>(x.stage + BIAS_OFF);
        const float *bh = p.b_head + (size_t)n * HEAD_TILE;
        for (int i = x.cg * 32 + x.lane; i < HEAD_TILE; i += 128) bq[i] = bh[i];
        // the row's draws for the tile's dims (a5, a7): Philox blocks of 4 dims
        const int b0 = m * BM + x.row;
        const int b = b0 < p.live_rows() ? b0 : 0;
        if (p.teacher || !(p.mdn_tau > 0.f) || p.fz_cur[b]) return;
        const unsigned long long ep = p.ep0 + p.ep_of(b);
        const int d0 = n * p.dims_per_tile, nd = min(p.dims_per_tile, p.Z - d0);
        float *es = reinterpret_cast<float *>(x.stage), *us = reinterpret_cast<float *>(x.stage + US_OFF);
        for (int blk = (d0 >> 2) + x.cg; 4 * blk < d0 + nd; blk += 4) {
            const u32x4 ru = rng_draw(p.seed, ep, p.step, RNG_COMPONENT, (uint32_t)blk);
            const u32x4 rn = rng_draw(p.seed, ep, p.step, RNG_NORMAL, (uint32_t)blk);
            const int lo = max(d0, 4 * blk), hi = min(d0 + nd, 4 * blk + 4);
            for (int d = lo; d < hi; ++d) us[x.lane * ZS_PITCH + d - d0] = to_uniform(u32x4_get(ru, d & 3));
            for (int h = 0; h < 2; ++h) {  // the block's two Box-Muller pairs: dims da (cos), da + 1 (sin)
                const int da = 4 * blk + 2 * h;
                if (da + 1 < lo || da >= hi) continue;
                float c, sn;
                box_muller2(h ? rn.z : rn.x, h ? rn.w : rn.y, c, sn);
                if (da >= lo) es[x.lane * ZS_PITCH + da - d0] = c;
                if (da + 1 < hi) es[x.lane * ZS_PITCH + da + 1 - d0] = sn;
            }
        }
    }
    static __device__ void run(const StepIO &p, uint32_t tacc, int m, int n, EpiCtx &x, const Pre &, int, int) {
        const int b0 = m * BM + x.row;
        const int nrows = p.live_rows();
        const bool valid = b0 < nrows;
        const int b = valid ? b0 : 0;  // rows past the batch compute on row 0 and store nothing
        const int e = p.ep_of(b);     // the row's episode
        const int Z = p.Z, K = p.K, KZ = K * Z, M = 3 * KZ, KX = Z + p.H;
        const int DS = (3 * K + 7) & ~7;  // columns per latent dim (8-aligned TMEM loads)
        const bool fz = !p.teacher && p.fz_cur[b] != 0;
        const size_t tb = (size_t)p.t * p.B + e;
        const int d0 = n * p.dims_per_tile;
        const int nd = min(p.dims_per_tile, Z - d0);
        const float *bh = reinterpret_cast<const float *>(x.stage + BIAS_OFF);  // the tile's bias
        float *zs = reinterpret_cast<float *>(x.stage);  // the normal draws, then z'
        const float *us = reinterpret_cast<const float *>(x.stage + US_OFF);
        float nll = 0.f;
        x.sync();  // the quadrant's bias copy and draws are complete
        {
            for (int i = x.cg; i < nd; i += 4) {  // warp-uniform bounds
                const int d = d0 + i;
                float v[24];
                {
                    uint32_t r0[8], r1[8], r2[8];
                    TC_LD8(tacc + DS * i, r0);
                    TC_LD8(tacc + DS * i + 8, r1);
                    TC_LD8(tacc + DS * i + 16, r2);  // past the dim when 3K <= 16: unused
                    tc::tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        v[j] = __uint_as_float(r0[j]);
                        v[8 + j] = __uint_as_float(r1[j]);
                        v[16 + j] = __uint_as_float(r2[j]);
                    }
                }
                // columns of a dim are component-interleaved (logit, mu, log sigma) so that every
                // register index below is static: no local-memory arrays
                float lg[8], mu[8], ls[8];
                {
                    float bv[24];  // DS * i is a multiple of 8 floats: 16-byte aligned
                    const float4 *b4 = reinterpret_cast<const float4 *>(bh + DS * i);
#pragma unroll
                    for (int j = 0; j < 6; ++j) {
                        const float4 t = b4[j];
                        bv[4 * j] = t.x; bv[4 * j + 1] = t.y; bv[4 * j + 2] = t.z; bv[4 * j + 3] = t.w;
                    }
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        lg[k] = k < K ? v[3 * k] + bv[3 * k] : -INFINITY;
                        mu[k] = k < K ? v[3 * k + 1] + bv[3 * k + 1] : 0.f;
                        ls[k] = k < K ? v[3 * k + 2] + bv[3 * k + 2] : 0.f;
                    }
                }
                if (!valid) continue;
                if (p.mdn_seq) {
                    float *ms = p.mdn_seq + tb * M;
                    const bool zero = fz && !p.teacher;
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        if (k < K) {
                            ms[d * K + k] = zero ? 0.f : lg[k];
                            ms[KZ + d * K + k] = zero ? 0.f : mu[k];
                            ms[2 * KZ + d * K + k] = zero ? 0.f : ls[k];
                        }
                    }
                }
                float zn;
                if (p.teacher) {
                    const float xv = p.z_tgt[(size_t)e * Z + d];
                    float mx = -INFINITY;
#pragma unroll
                    for (int k = 0; k < 8; ++k) if (k < K) mx = fmaxf(mx, lg[k]);
                    float s = 0.f;
#pragma unroll
                    for (int k = 0; k < 8; ++k) if (k < K) s += expf(lg[k] - mx);
                    const float lse = mx + logf(s);
                    float lp[8], tmax = -INFINITY;
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        if (k < K) {
                            const float zsd = (xv - mu[k]) * expf(-ls[k]);
                            lp[k] = (lg[k] - lse) - 0.5f * zsd * zsd - ls[k] - 0.91893853320467274178f;
                            tmax = fmaxf(tmax, lp[k]);
                        }
                    }
                    float acc = 0.f;
#pragma unroll
                    for (int k = 0; k < 8; ++k) if (k < K) acc += expf(lp[k] - tmax);
                    nll += -(tmax + logf(acc));
                    zn = xv;
                } else if (fz) {
                    zn = p.z_out[tb * Z + d];
                    if (p.comp_seq) p.comp_seq[tb * Z + d] = 255;
                } else {
                    int kc = 0;
                    if (!(p.mdn_tau > 0.f)) {
                        float best = lg[0];
                        zn = mu[0];
#pragma unroll
                        for (int k = 1; k < 8; ++k)
                            if (k < K && lg[k] > best) { best = lg[k]; kc = k; zn = mu[k]; }
                    } else {
                        const float itau = __fdividef(1.f, p.mdn_tau);
                        float mx = -INFINITY;
#pragma unroll
                        for (int k = 0; k < 8; ++k) if (k < K) mx = fmaxf(mx, lg[k] * itau);
                        float pk[8], s = 0.f;
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            pk[k] = k < K ? __expf(lg[k] * itau - mx) : 0.f;
                            s += pk[k];
                        }
                        const float u = us[x.lane * ZS_PITCH + i], is = __fdividef(1.f, s);  // drawn in pre()
                        // first k with u < C_k (the last component when rounding leaves u >= C_{K-2}),
                        // from a compare mask: no per-lane branches
                        float cum = 0.f;
                        uint32_t hit = 0u;
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            if (k < K - 1) {  // uniform
                                cum += pk[k] * is;
                                hit |= (u < cum ? 1u : 0u) << k;
                            }
                        }
                        kc = hit ? __ffs(hit) - 1 : K - 1;
                        float muc = mu[0], lsc = ls[0];
#pragma unroll
                        for (int k = 1; k < 8; ++k) {
                            muc = (k < K && k == kc) ? mu[k] : muc;
                            lsc = (k < K && k == kc) ? ls[k] : lsc;
                        }
                        const float eps = zs[x.lane * ZS_PITCH + i];  // drawn in pre()
                        const float scale = p.sigma_sqrt_tau ? sqrtf(p.mdn_tau) : 1.f;
                        zn = muc + __expf(lsc) * scale * eps;
                    }
                    if (p.comp_seq) p.comp_seq[tb * Z + d] = (uint8_t)kc;
                }
                zs[x.lane * ZS_PITCH + i] = zn;
            }
        }
        if (p.teacher && valid) {
            const int sq = p.nseq ? e % p.nseq : e, tt = p.nseq ? e / p.nseq : p.t;  // sequence, step
            const int len = p.lengths ? p.lengths[sq] : p.T;
            if (tt == 0 && n == 0 && x.cg == 0 && (len < 0 || len > p.T))
                report_status(x.status, WM_ERR_INVALID_ARG);
            float *part = p.nll_part + ((size_t)n * 4 + x.cg) * p.B + e;
            if (p.nseq) *part = tt < len ? nll : 0.f;  // one row per (step, sequence)
            else if (tt < len) *part += nll;
        }
        if (n == p.rd_tile) {
            const bool shaped = p.reward_mode == WM_REWARD_SHAPED;  // uniform
            uint32_t r[2], q[2] = {0u, 0u};
            asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0, %1}, [%2];"
                         : "=r"(r[0]), "=r"(r[1]) : "r"(tacc + p.rd_col));
            if (shaped)
                asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0, %1}, [%2];"
                             : "=r"(q[0]), "=r"(q[1]) : "r"(tacc + p.rd_col + 2));
            uint32_t vr = 0u;
            if (p.value_seq)  // uniform
                asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];"
                             : "=r"(vr) : "r"(tacc + p.rd_col + p.nr - 1));
            tc::tmem_ld_wait();
            const float vq = __uint_as_float(vr);
            if (!p.teacher && valid && x.cg == 0) {
                float rew = __uint_as_float(r[0]) + bh[p.rd_col];
                const float dl = __uint_as_float(r[1]) + bh[p.rd_col + 1];
                const int a = p.act[b];
                const int noop_a = p.n_xfers > 0 ? p.n_xfers - 1 : p.A - 1;
                const bool noop = p.noop_terminates && a == noop_a;
                if (shaped) {
                    if (!fz) {  // Eq. 2 on the predictions entering and leaving the step
                        const float rt = __uint_as_float(q[0]) + bh[p.rd_col + 2];
                        const float mem = __uint_as_float(q[1]) + bh[p.rd_col + 3];
                        // valid: an action was taken (and, for an xfer, a location)
                        const bool ok = a >= 0 && (p.n_xfers == 0 || a == noop_a || p.act2[b] >= 0);
                        rew = ok ? p.alpha * (p.rt[e] - rt) + p.beta * (p.mem[e] - mem) : p.invalid_reward;
                        p.rt[e] = rt;
                        p.mem[e] = mem;
                    }
                    if (p.rt_seq) p.rt_seq[tb] = p.rt[e];
                    if (p.mem_seq) p.mem_seq[tb] = p.mem[e];
                }
                if (p.value_seq) p.value_seq[tb] = fz ? 0.f : vq + bh[p.rd_col + p.nr - 1];
                p.rewards[tb] = fz ? 0.f : rew;
                p.done[tb] = (fz || dl > 0.f || noop) ? 1 : 0;
                p.fz_next[b] = (fz || (p.done_terminates && dl > 0.f) || noop) ? 1 : 0;
            }
        }
        // the quadrant's 32 x nd block of z', stored row-major by its 128 threads
        x.sync();
        const int y0 = m * BM + 32 * x.quad, nrow = min(32, nrows - y0);
        for (int j = x.cg * 32 + x.lane; j < nrow * nd; j += 128) {
            const int rr = j / nd, i = j - rr * nd;
            const size_t bb = (size_t)(y0 + rr);
            const float zn = zs[rr * ZS_PITCH + i];
            if (!p.teacher) p.z_out[((size_t)(p.t + 1) * p.B + p.ep_of((int)bb)) * Z + d0 + i] = zn;
            if (p.x_next) {  // (a batched scoring GEMM has no next operand: the frames are staged)
                const __nv_bfloat16 zh = __float2bfloat16_rn(zn);
                p.x_next[bb * KX + d0 + i] = zh;
                if (p.x_next_lo) p.x_next_lo[bb * KX + d0 + i] = __float2bfloat16_rn(zn - __bfloat162float(zh));
            }
        }
        x.sync();  // the staging may be rewritten by the next tile
    }
};

// ---------------------------------------------------------------------------
// The persistent warp-specialised GEMM on CTA pairs.  A pair computes 256-row tiles of
// TILE_N = BN * NSUB columns with M = 256 tcgen05 MMAs (cta_group::2) issued by the leader
// CTA: each CTA loads its 128 rows of A and BN/2 rows of each BN-wide slice of B, and runs
// the epilogue on its own 128 accumulator rows.  (One M = 256 MMA does twice the work of an
// M = 128 one in about 0.6 of its time, per SM.)  A ring stage holds KPS k-steps of BK: the
// MMA thread waits for a stage once, issues all its MMAs back to back and commits once, to
// the stage's "empty" barrier: any wait or commit on the issuing thread lets the tensor
// pipe drain, and a pair's multicast commit costs more than one k-step's MMAs can hide.
// NP = 3: the fp32 path.  Each fp32 operand is split into bf16 parts x = x_hi + x_lo (x_hi =
// bf16(x), x_lo = bf16(x - x_hi)), and the accumulator takes three passes over K: A_hi B_hi,
// A_hi B_lo (tmB2) and A_lo B_hi (tmA2).  The dropped A_lo B_lo term and the parts'
// residuals are below 2^-16 of each product.
template <int BN, int NSUB, int STAGES, class Epi, int KPS = 1, int NP = 1>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmXs,
              const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
              const __grid_constant__ CUtensorMap tmXs2, GemmGrid g, StepIO io) {
    constexpr int TILE_N = BN * NSUB, BNH = BN / 2;
    constexpr uint32_t A_BYTES = BM * BK * 2, B_SUB = BNH * BK * 2, B_BYTES = B_SUB * NSUB;
    constexpr uint32_t KSTEP_BYTES = A_BYTES + B_BYTES, STAGE_BYTES = KPS * KSTEP_BYTES;  // per CTA
    constexpr int NACC = TILE_N <= 256 ? 2 : 1;
    constexpr uint32_t ACC_COLS = 256;
    static_assert(BN % 16 == 0 && BNH % 8 == 0 && BN <= 256 && TILE_N <= 512, "tile shape");
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    __shared__ __align__(8) uint64_t bar_full[STAGES], bar_empty[STAGES], bar_accf[2], bar_acce[2], bar_stage[4],
        bar_never;
    __shared__ uint32_t tmem_base;
    __shared__ int s_abort;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = tc::cluster_rank();  // 0: the pair's leader
    const int pair = (int)(blockIdx.x >> 1), npairs = (int)(gridDim.x >> 1);
    const uint32_t smem_u = tc::smem_u32(smem);
    auto full_b = [&](int s) { return tc::smem_u32(&bar_full[s]); };
    auto empty_b = [&](int s) { return tc::smem_u32(&bar_empty[s]); };

    if (tid == 0) {
        for (int s = 0; s < STAGES; ++s) tc::mbar_init(full_b(s), 1);             // the leader's: both CTAs' bytes
        for (int s = 0; s < STAGES; ++s) tc::mbar_init(empty_b(s), 1);            // the leader's commit, multicast
        for (int a = 0; a < 2; ++a) {
            tc::mbar_init(tc::smem_u32(&bar_accf[a]), 1);
            tc::mbar_init(tc::smem_u32(&bar_acce[a]), 2 * EPI_WARPS);  // the leader's: both CTAs' warps
        }
        for (int q = 0; q < 4; ++q) tc::mbar_init(tc::smem_u32(&bar_stage[q]), 1);
        tc::mbar_init(tc::smem_u32(&bar_never), 1);
        tc::fence_mbar_init();
        s_abort = 0;
    }
    if (warp == 1) tmem_alloc_pair(tc::smem_u32(&tmem_base), 512);
    tc::fence_before_sync();
    tc::cluster_sync();  // both CTAs' barriers exist before any cross-CTA arrive
    tc::fence_after_sync();
    const uint32_t tm = tmem_base;
    // Programmatic dependent launch (when the launch allows it): the set-up above may overlap
    // the previous kernel of the stream; every read of its outputs comes after this wait.
    // (It returns at once for a launch without programmatic serialization.)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    int m_tiles = g.m_tiles;  // 256-row tiles
    if (g.n_rows) m_tiles = (*(volatile const int *)g.n_rows + 2 * BM - 1) / (2 * BM);
    int ntiles = m_tiles * g.n_tiles;
    const int ksteps = NP * g.k_steps;  // k-steps per tile over all passes
    // Injected wait (tests of the timeout path): one thread of each CTA waits on a barrier
    // that nothing completes, before any MMA or copy is issued.  Both CTAs of every pair give
    // up the same way, record WM_ERR_TIMEOUT and take no tile, so nothing is in flight; the
    // set-up's TMEM is still freed at the end.
    if (g.test_wait) {
        if (tid == 0 && !tc::mbar_wait_bounded(tc::smem_u32(&bar_never), 0, g.test_wait)) {
            s_abort = 1;
            atomicExch(g.status, (int)WM_ERR_TIMEOUT);
        }
        __syncthreads();
        if (s_abort) ntiles = 0;
    }
    auto wait = [&](uint32_t bar, uint32_t parity) {
        if (!s_abort && !tc::mbar_wait_bounded(bar, parity, POLLS)) {
            s_abort = 1;
            atomicExch(g.status, (int)WM_ERR_TIMEOUT);
        }
    };

    if (warp == 0) {
        if (lane == 0) {  // ---- TMA producer (both CTAs)
            int stage = 0;
            uint32_t phase = 0;
            for (int tile = pair; tile < ntiles; tile += npairs) {
                const int m = tile / g.n_tiles, n = tile % g.n_tiles;
                const int brow = g.pop_P > 1 ? (int)(((g.ep0 + (unsigned long long)m * (2 * BM)) /
                                                      (unsigned long long)g.pop_E) % (unsigned long long)g.pop_P) * g.pop_rows
                                             : 0;
                for (int ks0 = 0; ks0 < ksteps; ks0 += KPS) {
                    const int nk = ksteps - ks0 < KPS ? ksteps - ks0 : KPS;  // k-steps in this stage
                    const uint32_t full_ldr = tc::map_rank(full_b(stage), 0);
                    wait(empty_b(stage), phase ^ 1u);  // the stage's previous MMAs are done
                    if (s_abort) break;
                    for (int h = 0; h < nk; ++h) {
                        int ks = ks0 + h;
                        const CUtensorMap *ma = &tmA, *mb = &tmB;
                        if (NP > 1) {  // pass 0: A_hi B_hi, 1: A_hi B_lo, 2: A_lo B_hi
                            const int pass = ks / g.k_steps;
                            ks -= pass * g.k_steps;
                            if (pass == 1) mb = &tmB2;
                            if (pass == 2) ma = &tmA2;
                        }
                        const uint32_t sa = smem_u + stage * STAGE_BYTES + h * KSTEP_BYTES;
                        if (h == 0 && rank == 0) tc::mbar_arrive_expect_tx(full_b(stage), 2 * nk * KSTEP_BYTES);
                        tma_load_2sm(sa, ma, g.a_col0 + ks * BK, (2 * m + (int)rank) * BM, full_ldr);
#pragma unroll
                        for (int s = 0; s < NSUB; ++s)
                            tma_load_2sm(sa + A_BYTES + s * B_SUB, mb, ks * BK,
                                         brow + n * TILE_N + s * BN + (int)rank * BNH, full_ldr);
                    }
                    if (s_abort) break;
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {  // ---- MMA issuer (the leader only)
            int stage = 0, acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            const uint32_t idesc = tc::idesc_bf16_f32(2 * BM, BN);
            for (int tile = pair; tile < ntiles; tile += npairs) {
                wait(tc::smem_u32(&bar_acce[acc]), acc_phase ^ 1u);
                tc::fence_after_sync();
                const uint32_t dcol = tm + acc * ACC_COLS;
                for (int ks0 = 0; ks0 < ksteps; ks0 += KPS) {
                    const int nk = ksteps - ks0 < KPS ? ksteps - ks0 : KPS;
                    wait(full_b(stage), phase);
                    if (s_abort) break;
                    tc::fence_after_sync();
                    // the issuing thread shares its SMSP with four epilogue warps: few instructions
                    // between MMAs (descriptors built once per k-step, stepped by 32 bytes = 2)
#pragma unroll
                    for (int h = 0; h < KPS; ++h) {
                        if (h >= nk) break;
                        const int ks = ks0 + h;
                        const uint32_t sa = smem_u + stage * STAGE_BYTES + h * KSTEP_BYTES;
                        const uint64_t da0 = desc_sw128(sa), db0 = desc_sw128(sa + A_BYTES);
#pragma unroll
                        for (int kk = 0; kk < BK / 16; ++kk) {
#pragma unroll
                            for (int s = 0; s < NSUB; ++s)
                                mma_bf16_pair(dcol + s * BN, da0 + 2 * kk, db0 + (s * B_SUB >> 4) + 2 * kk, idesc,
                                              (ks > 0 || kk > 0) ? 1u : 0u);
                        }
                    }
                    mma_commit_pair(empty_b(stage));  // both CTAs' stage is free once these are done
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                mma_commit_pair(tc::smem_u32(&bar_accf[acc]));
                if (NACC == 2) {
                    acc ^= 1;
                    if (acc == 0) acc_phase ^= 1u;
                } else {
                    acc_phase ^= 1u;
                }
            }
        }
    } else {  // ---- epilogue warps 2..17: 4 column groups per TMEM lane quadrant (both CTAs)
        const int quad = warp & 3;
        EpiCtx x;
        x.quad = quad;
        x.cg = (warp - 2) >> 2;
        x.lane = lane;
        x.row = 32 * quad + lane;
        x.red = reinterpret_cast<float *>(smem + STAGES * STAGE_BYTES + 4 * Epi::QUAD_STAGE);
        x.stage = smem + STAGES * STAGE_BYTES + quad * Epi::QUAD_STAGE;  // past the ring
        x.stage_u = tc::smem_u32(x.stage);
        x.stage_bar = tc::smem_u32(&bar_stage[quad]);
        x.stage_phase = 0;
        x.leader = x.cg == 0 && lane == 0;
        x.pending = false;
        x.pending_phase = 0;
        x.tm_c = &tmC;
        x.tm_xs = &tmXs;
        x.tm_xs2 = &tmXs2;
        x.abort_flag = &s_abort;
        x.status = g.status;
        int acc = 0;
        uint32_t acc_phase = 0;
        // this CTA's 128-row block of 256-row tile `tile`
        auto mblock = [&](int tile) { return 2 * (tile / g.n_tiles) + (int)rank; };
        Epi::init(io, x, tid - 64);
        asm volatile("bar.sync 5, %0;" :: "n"(32 * EPI_WARPS) : "memory");  // the epilogue warps' set-up is done
        if (Epi::TMA_STAGE && x.leader && pair < ntiles) Epi::prefetch(io, mblock(pair), pair % g.n_tiles, x);
        for (int tile = pair; tile < ntiles; tile += npairs) {
            const int mb = mblock(tile), n = tile % g.n_tiles;
            const int next = tile + npairs < ntiles ? tile + npairs : -1;
            typename Epi::Pre pr;
            Epi::pre(io, mb, n, x, pr);  // loads that do not need the accumulator
            wait(tc::smem_u32(&bar_accf[acc]), acc_phase);
            __syncwarp();
            tc::fence_after_sync();
            const uint32_t tacc = tm + ((uint32_t)(32 * quad) << 16) + acc * ACC_COLS;
            // always run: the epilogues use per-quadrant named barriers, so every thread of a
            // quadrant must take the same path (after an abort the results are just unused)
            Epi::run(io, tacc, mb, n, x, pr, next >= 0 ? mblock(next) : -1, next >= 0 ? next % g.n_tiles : 0);
            __syncwarp();
            tc::fence_before_sync();
            if (lane == 0) mbar_arrive_cluster(tc::map_rank(tc::smem_u32(&bar_acce[acc]), 0));
            if (NACC == 2) {
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1u;
            } else {
                acc_phase ^= 1u;
            }
        }
        if (Epi::TMA_STAGE && x.leader) {
            bulk_wait_all();  // the TMA stores have completed
            // after an abort a prefetch may still be in flight: let it land before the CTA exits
            if (x.pending) tc::mbar_wait_bounded(x.stage_bar, x.pending_phase, POLLS);
        }
    }
    __syncwarp();
    tc::fence_before_sync();
    // this CTA's work is done: the next kernel may be launched (its set-up then overlaps
    // the tail of this one; triggering at the start instead measured slower)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    tc::cluster_sync();  // the leader's MMAs into this CTA's TMEM and shared memory are done
    if (warp == 1) tmem_dealloc_pair(tm, 512);
}

// ---------------------------------------------------------------------------
__global__ void k_tc_init(StepIO p, const float *z0, const float *h0, const float *c0, const uint8_t *done0,
                          __nv_bfloat16 *x0, __nv_bfloat16 *x0_lo, uint8_t *fz0, uint8_t *fz1, int n_head_tiles,
                          int *dstep, int *cnt) {
    if (cnt && blockIdx.x == 0 && threadIdx.x < 4) cnt[threadIdx.x] = 0;
    const int KX = p.Z + p.H;
    const size_t nx = (size_t)p.B * KX;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < nx; i += (size_t)gridDim.x * blockDim.x) {
        const size_t b = i / KX, k = i % KX;
        float v;
        if (k < (size_t)p.Z) v = p.teacher ? p.z_seq[b * p.Z + k] : z0[b * p.Z + k];
        else v = h0 ? h0[b * p.H + (k - p.Z)] : 0.f;
        const __nv_bfloat16 vh = __float2bfloat16_rn(v);
        x0[i] = vh;
        if (x0_lo) x0_lo[i] = __float2bfloat16_rn(v - __bfloat162float(vh));
        if (k >= (size_t)p.Z) {
            const size_t j = b * p.H + (k - p.Z);
            p.h32[j] = h0 ? h0[j] : 0.f;
            p.c[j] = c0 ? c0[j] : 0.f;
        } else if (!p.teacher) {
            p.z_out[b * p.Z + k] = z0[b * p.Z + k];
        }
    }
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < (size_t)p.B; i += (size_t)gridDim.x * blockDim.x) {
        fz0[i] = fz1[i] = done0 ? (done0[i] != 0) : 0;
        // no action until a controller epilogue chooses one (a launch that gave up chooses none)
        p.act[i] = -1;
        if (p.act2) p.act2[i] = -1;
        if (dstep) dstep[i] = p.T;
        if (p.rt0) {
            p.rt[i] = p.rt0[i];
            p.mem[i] = p.mem0[i];
        }
        if (p.teacher)
            for (int t = 0; t < 4 * n_head_tiles; ++t) p.nll_part[(size_t)t * p.B + i] = 0.f;
    }
}

__global__ void k_tc_finish(int B, int H, const float *h32, const float *c, float *h_final, float *c_final,
                            const float *nll_part, int n_parts, float *nll) {
    const size_t n = (size_t)B * H;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        if (h_final) h_final[i] = h32[i];
        if (c_final) c_final[i] = c[i];
    }
    if (nll)
        for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < (size_t)B; i += (size_t)gridDim.x * blockDim.x) {
            double s = 0.0;
            for (int t = 0; t < n_parts; ++t) s += (double)nll_part[(size_t)t * B + i];
            nll[i] = (float)s;
        }
}

// ---------------------------------------------------------------------------
// Batched teacher-forced scoring: the operand rows of all T + 1 frames are staged at once
// (frame f, sequence n at row f N + n: z part from z_seq; the h part of frame f + 1 is
// written by step f's gate epilogue), the recurrence runs one gate GEMM per step, and one
// head GEMM then scores all N T (step, sequence) rows.
__global__ void k_tc_frames(int N, int T, int Z, int KX, const float *__restrict__ z_seq,
                            __nv_bfloat16 *__restrict__ x, __nv_bfloat16 *__restrict__ x_lo) {
    const size_t n = (size_t)T * N * Z;  // frames 1..T (frame 0 is the init kernel's)
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        const size_t r = (size_t)N + i / Z, k = i % Z;  // operand row, z column
        const float v = z_seq[r * Z + k];
        const __nv_bfloat16 vh = __float2bfloat16_rn(v);
        x[r * KX + k] = vh;
        if (x_lo) x_lo[r * KX + k] = __float2bfloat16_rn(v - __bfloat162float(vh));
    }
}

// nll[n] = sum over the head tiles' partials and the steps of sequence n (uncounted steps
// hold 0).  A warp per sequence: lane l adds the partials l, l + 32, ... of the sequence's
// parts x T values in fp64, then a shuffle tree of fixed shape combines the lanes, so the
// order, and the result, is the same every time.
__global__ void k_tc_nll_reduce(int N, int T, int parts, const float *__restrict__ part, float *__restrict__ nll) {
    const int lane = threadIdx.x & 31, nw = (int)((gridDim.x * blockDim.x) >> 5);
    const int total = parts * T;
    for (int n = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5); n < N; n += nw) {
        double s = 0.0;
        for (int i = lane; i < total; i += 32) s += (double)part[(size_t)i * N + n];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
        if (lane == 0) nll[n] = (float)s;
    }
}

// ---------------------------------------------------------------------------
// Compaction of the live episodes (rollouts whose episodes end: done head or NO-OP).
// Before step t's GEMMs, k_tc_compact packs the rows whose episode is still live after
// step t-1 into the first rows of the operand buffers, so that the three GEMMs of step t
// compute live episodes only, and writes step t's outputs of every frozen episode (the
// ones the GEMMs no longer see).  A row's arithmetic does not depend on its position in a
// tile, so the order in which blocks claim their output rows (an atomic per block) changes
// no result.  One block per 256 rows of step t-1, one warp per row copy.
struct CompactIO {
    int B, Z, H, KX, M, t;
    const int32_t *rows_in;           // [B] row -> episode at step t-1 (null: row b is episode b)
    const int *n_in;                  // rows of step t-1 (null: B)
    const uint8_t *dies;              // [B] row-keyed: the episode ended at step t-1 (at t = 0: done0)
    const __nv_bfloat16 *x_in;        // [B, KX] operands after step t-1
    __nv_bfloat16 *x_out;             // [B, KX] compacted
    const __nv_bfloat16 *x_in_lo;     // fp32 path: the lo parts (else null)
    __nv_bfloat16 *x_out_lo;
    const float *c_in, *h32;          // [B, H] row-keyed c, h after step t-1
    float *c_out;                     // [B, H] compacted c
    int32_t *rows_out;                // [B] row -> episode at step t
    int *n_out;                       // rows of step t (zero on entry)
    int *n_clear;                     // set to zero: the counter of step t + 1
    int T;
    int fill;                         // write the frozen episodes' step-t outputs now (else one
                                      // kernel writes every step's after the last step)
    int *dstep;                       // [B] first step at which the episode is frozen (T: never)
    int *dead_flag;                   // host-mapped: set to call_id once no episode is live
    int call_id;
    const int *n_prev2;               // rows of step t-2 (null at t < 2)
    float *hfin, *cfin;               // [B, H] an ended episode's h, c
    const float *rt, *mem;            // [B] carried predictions (shaped reward)
    float *z_out;                     // step t's outputs of frozen episodes
    int32_t *actions;
    float *rewards;
    uint8_t *done;
    float *h_seq, *c_seq, *mdn_seq;
    uint8_t *comp_seq;
    float *logp_seq, *value_seq, *rt_seq, *mem_seq;
    int32_t *loc_actions;
};

// Element k of frozen episode e's step-t outputs (k < fill_elems): z repeated (and component
// 255), h and c repeated, mixture outputs 0, then the scalars (no action, reward 0, done).
__device__ __forceinline__ int fill_elems(const CompactIO &q) {
    return q.Z + ((q.h_seq || q.c_seq) ? q.H : 0) + (q.mdn_seq ? q.M : 0) + 1;
}
__device__ void fill_elem(const CompactIO &q, int e, int k, const float *hs, const float *cs) {
    const size_t tb = (size_t)q.t * q.B + e;
    if (k < q.Z) {
        q.z_out[(tb + q.B) * q.Z + k] = q.z_out[tb * q.Z + k];
        if (q.comp_seq) q.comp_seq[tb * q.Z + k] = 255;
        return;
    }
    k -= q.Z;
    if (q.h_seq || q.c_seq) {
        if (k < q.H) {
            if (q.h_seq) q.h_seq[tb * q.H + k] = hs[k];
            if (q.c_seq) q.c_seq[tb * q.H + k] = cs[k];
            return;
        }
        k -= q.H;
    }
    if (q.mdn_seq) {
        if (k < q.M) {
            q.mdn_seq[tb * q.M + k] = 0.f;
            return;
        }
    }
    q.actions[tb] = -1;
    q.rewards[tb] = 0.f;
    q.done[tb] = 1;
    if (q.logp_seq) q.logp_seq[tb] = 0.f;
    if (q.value_seq) q.value_seq[tb] = 0.f;
    if (q.rt_seq) q.rt_seq[tb] = q.rt[e];
    if (q.mem_seq) q.mem_seq[tb] = q.mem[e];
    if (q.loc_actions) q.loc_actions[tb] = -1;
}

constexpr int CROWS = 8;          // rows of step t-1 per block: a warp per row
constexpr int CTHREADS = 32 * CROWS;

// A row's 16-byte chunks [0, n) from src to dst, by one warp: each lane loads up to 8 chunks
// before it stores any, so that the loads are in flight together (a load-then-store per
// chunk waits out the memory latency once per chunk).
__device__ __forceinline__ void warp_copy16(const uint4 *__restrict__ src, uint4 *__restrict__ dst, int n, int lane) {
    for (int base = 0; base < n; base += 256) {
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int k = base + 32 * u + lane;
            if (k < n) v[u] = src[k];
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int k = base + 32 * u + lane;
            if (k < n) dst[k] = v[u];
        }
    }
}

// Phase A (rows of step t-1, a warp per row): survivors' operand row (and its lo part) and c
// to their new row; ended episodes' h and c recorded, and, when outputs are staged step by
// step, their step-t outputs written.  Phase B (the whole grid): when staged, the step-t
// outputs of the episodes frozen before.
__global__ void __launch_bounds__(CTHREADS) k_tc_compact(CompactIO q) {
    asm volatile("griddepcontrol.wait;" ::: "memory");  // the previous step's outputs are complete
    __shared__ int s_pos[CROWS], s_e[CROWS];
    const int tid = (int)threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_in = q.n_in ? *(volatile const int *)q.n_in : q.B;
    const int r0 = (int)blockIdx.x * CROWS;
    if (r0 < n_in) {  // block-uniform
        const int nrow = min(CROWS, n_in - r0);
        if (warp == 0) {  // the block claims its output rows with one atomic
            const int r = r0 + lane;
            const bool in = lane < nrow;
            const bool keep = in && !(q.dies && q.dies[r]);
            const uint32_t bal = __ballot_sync(0xffffffffu, keep);
            int base = 0;
            if (lane == 0 && bal) base = atomicAdd(q.n_out, __popc(bal));
            base = __shfl_sync(0xffffffffu, base, 0);
            if (in) {
                const int e = q.rows_in ? q.rows_in[r] : r;
                const int pos = keep ? base + __popc(bal & ((1u << lane) - 1u)) : -1;
                s_e[lane] = e;
                s_pos[lane] = pos;
                if (keep) q.rows_out[pos] = e;
                else q.dstep[e] = q.t;
            }
        }
        __syncthreads();
        const int XC = q.KX / 8, CC = q.H / 4;  // 16-byte chunks per row
        if (warp < nrow) {
            const size_t rr = (size_t)(r0 + warp);
            const int pos = s_pos[warp];
            const uint4 *ci = reinterpret_cast<const uint4 *>(q.c_in) + rr * CC;
            if (pos >= 0) {
                warp_copy16(reinterpret_cast<const uint4 *>(q.x_in) + rr * XC,
                            reinterpret_cast<uint4 *>(q.x_out) + (size_t)pos * XC, XC, lane);
                if (q.x_in_lo)
                    warp_copy16(reinterpret_cast<const uint4 *>(q.x_in_lo) + rr * XC,
                                reinterpret_cast<uint4 *>(q.x_out_lo) + (size_t)pos * XC, XC, lane);
                warp_copy16(ci, reinterpret_cast<uint4 *>(q.c_out) + (size_t)pos * CC, CC, lane);
            } else {
                const size_t e = (size_t)s_e[warp];
                warp_copy16(reinterpret_cast<const uint4 *>(q.h32) + rr * CC, reinterpret_cast<uint4 *>(q.hfin) + e * CC,
                            CC, lane);
                warp_copy16(ci, reinterpret_cast<uint4 *>(q.cfin) + e * CC, CC, lane);
                if (q.fill) {  // its step-t outputs, from its row
                    const int fe = fill_elems(q);
                    for (int k = lane; k < fe; k += 32)
                        fill_elem(q, (int)e, k, q.h32 + rr * q.H, q.c_in + rr * q.H);
                }
            }
        }
    }
    // episodes frozen before this step's compaction stay frozen: their step-t outputs, over
    // the whole grid (an episode ending now reads dstep as T or t: either way it is not here)
    if (q.fill && q.t > 0) {
        const int fe = fill_elems(q);
        const size_t n = (size_t)q.B * fe, stride = (size_t)gridDim.x * CTHREADS;
        for (size_t i = (size_t)blockIdx.x * CTHREADS + tid; i < n; i += stride) {
            const int e = (int)(i / fe), k = (int)(i - (size_t)e * fe);
            if (q.dstep[e] >= q.t) continue;
            fill_elem(q, e, k, q.hfin + (size_t)e * q.H, q.cfin + (size_t)e * q.H);
        }
    }
    if (blockIdx.x == 0 && tid == 0) {
        *q.n_clear = 0;
        // every episode has ended (reported once, at the first step that sees it): the host
        // may stop issuing steps
        if (n_in == 0 && q.dead_flag && (!q.n_prev2 || *(volatile const int *)q.n_prev2 != 0))
            *(volatile int *)q.dead_flag = q.call_id;
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Every frozen episode's outputs of every step from the one at which it froze, after the
// last step (calls whose outputs are not staged step by step).  One warp per episode: each
// lane reads its z (and h, c) values once and writes them to every frozen step.
__global__ void k_tc_fill_frozen(CompactIO q) {
    const int lane = threadIdx.x & 31;
    const int nw = (int)((gridDim.x * blockDim.x) >> 5);
    for (int e = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5); e < q.B; e += nw) {
        const int d = q.dstep[e];
        if (d >= q.T) continue;  // warp-uniform
        const size_t B = (size_t)q.B;
        for (int k = lane; k < q.Z; k += 32) {
            const float v = q.z_out[((size_t)d * B + e) * q.Z + k];  // z of the step it froze at
            for (int t = d; t < q.T; ++t) {
                const size_t tb = (size_t)t * B + e;
                q.z_out[(tb + B) * q.Z + k] = v;
                if (q.comp_seq) q.comp_seq[tb * q.Z + k] = 255;
            }
        }
        if (q.h_seq || q.c_seq)
            for (int k = lane; k < q.H; k += 32) {
                const float hv = q.hfin[(size_t)e * q.H + k], cv = q.cfin[(size_t)e * q.H + k];
                for (int t = d; t < q.T; ++t) {
                    const size_t tb = (size_t)t * B + e;
                    if (q.h_seq) q.h_seq[tb * q.H + k] = hv;
                    if (q.c_seq) q.c_seq[tb * q.H + k] = cv;
                }
            }
        if (q.mdn_seq)
            for (int k = lane; k < q.M; k += 32)
                for (int t = d; t < q.T; ++t) q.mdn_seq[((size_t)t * B + e) * q.M + k] = 0.f;
        const float rt = q.rt_seq ? q.rt[e] : 0.f, mem = q.mem_seq ? q.mem[e] : 0.f;
        for (int t = d + lane; t < q.T; t += 32) {  // the scalars, a step per lane
            const size_t tb = (size_t)t * B + e;
            q.actions[tb] = -1;
            q.rewards[tb] = 0.f;
            q.done[tb] = 1;
            if (q.logp_seq) q.logp_seq[tb] = 0.f;
            if (q.value_seq) q.value_seq[tb] = 0.f;
            if (q.rt_seq) q.rt_seq[tb] = rt;
            if (q.mem_seq) q.mem_seq[tb] = mem;
            if (q.loc_actions) q.loc_actions[tb] = -1;
        }
    }
}

// h_final, c_final after a compacted rollout: the last step's rows, and the recorded state
// of the episodes frozen before it
__global__ void k_tc_finish_compact(int B, int H, int T, const int *dstep, const int32_t *rows, const int *n_rows,
                                    const float *h32, const float *c, const float *hfin, const float *cfin,
                                    float *h_final, float *c_final) {
    const int warp = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    const int nw = (int)((gridDim.x * blockDim.x) >> 5);
    const int n = *n_rows;
    // (the caller's arrays need only 4-byte alignment: element-wise copies)
    for (int r = warp; r < n; r += nw) {
        const int e = rows[r];
        for (int i = lane; i < H; i += 32) {
            if (h_final) h_final[(size_t)e * H + i] = h32[(size_t)r * H + i];
            if (c_final) c_final[(size_t)e * H + i] = c[(size_t)r * H + i];
        }
    }
    for (int e = warp; e < B; e += nw) {
        if (dstep[e] >= T) continue;  // live at the last step: one of its rows
        for (int i = lane; i < H; i += 32) {
            if (h_final) h_final[(size_t)e * H + i] = hfin[(size_t)e * H + i];
            if (c_final) c_final[(size_t)e * H + i] = cfin[(size_t)e * H + i];
        }
    }
}

// ---------------------------------------------------------------------------
typedef CUresult (*encode_fn_t)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

encode_fn_t get_encode() {
    static encode_fn_t fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            fn = (encode_fn_t)p;
    }
    return fn;
}

// 2-D map over a row-major [rows, cols] matrix of bf16 (or fp32), box = 128 bytes of a row x
// box_rows rows, 128-byte swizzle.  Rows past `rows` read as zero and are not written.
bool make_map(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows,
              bool fp32 = false) {
    encode_fn_t enc = get_encode();
    if (!enc) return false;
    const uint64_t es_bytes = fp32 ? 4 : 2;
    cuuint64_t dims[2] = {cols, rows}, strides[1] = {cols * es_bytes};
    cuuint32_t box[2] = {(cuuint32_t)(128 / es_bytes), box_rows}, es[2] = {1, 1};
    return enc(m, fp32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
               const_cast<void *>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same over bf16 with a box of 32 columns (64 bytes) x 32 rows, unswizzled: the h' slab
// of a 128-column gate tile.
bool make_map_x32(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols) {
    encode_fn_t enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {cols, rows}, strides[1] = {cols * 2};
    cuuint32_t box[2] = {32, 32}, es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int NSUB, int STAGES, class Epi, int KPS = 1>
size_t gemm_smem() {
    // per CTA: its A rows and half of each B slice per k-step
    return 1024 + (size_t)STAGES * KPS * (BM * BK * 2 + (size_t)(BN / 2) * NSUB * BK * 2) +
           4 * (size_t)Epi::QUAD_STAGE + Epi::RED_BYTES;
}

// The operand maps of one GEMM: A (and its lo part), B (and its lo part); the fp32 path's
// second maps are unused on the bf16 path (NP = 1).
struct OpMaps {
    const CUtensorMap *a, *b, *a2, *b2;
};

template <int BN, int NSUB, int STAGES, class Epi, int KPS = 1, int NP = 1>
cudaError_t launch_gemm(const OpMaps &op, const CUtensorMap &mc, const CUtensorMap &mxs, const CUtensorMap &mxs2,
                        GemmGrid g, const StepIO &io, int sms, cudaStream_t s, bool pdl) {
    const size_t smem = gemm_smem<BN, NSUB, STAGES, Epi, KPS>();
    auto kern = k_tc_gemm<BN, NSUB, STAGES, Epi, KPS, NP>;
    cudaLaunchConfig_t lc = {};
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;  // a CTA pair per 256-row tile
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.blockDim = dim3(GEMM_THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    lc.attrs = at;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    lc.numAttrs = 2;
    static int max_pairs = 0;  // pairs resident at once (the grid is persistent)
    if (!max_pairs) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        lc.gridDim = dim3(sms & ~1);
        int n = 0;
        e = cudaOccupancyMaxActiveClusters(&n, kern, &lc);
        if (e != cudaSuccess) return e;
        max_pairs = n > 0 ? n : 1;
    }
    const int tiles = g.m_tiles * g.n_tiles;
    const int pairs = tiles < max_pairs ? tiles : max_pairs;
    lc.gridDim = dim3(2 * pairs);
    return cudaLaunchKernelEx(&lc, kern, *op.a, *op.b, mc, mxs, *op.a2, *op.b2, mxs2, g, io);
}

inline size_t a256(size_t x) { return (x + 255) & ~(size_t)255; }

struct TcWs {
    __nv_bfloat16 *x[2];
    __nv_bfloat16 *x_lo[2];  // fp32 path: the lo parts of x
    float *c, *h32, *nll_part, *rt, *mem;
    float *logits;   // hierarchical action: [B, A]
    int32_t *act2;   // hierarchical action: the location's action row
    int32_t *act;
    uint8_t *fz[2];
    // compaction of live episodes (models whose episodes end)
    float *c2, *hfin, *cfin;
    int32_t *rows[2];
    int *cnt;        // [4] ring of per-step row counts
    int *dstep;      // [B] first step at which each episode is frozen
    // batched teacher-forced scoring
    __nv_bfloat16 *xall, *xall_lo;  // [(T+1) B, KX] the operand rows of every frame
    float *part;                    // [4 head tiles, T B] per-(step, sequence) partials
};

// models whose episodes can end get the compaction buffers (and use them when P = 1)
inline bool can_compact(const wm_config &c) { return c.done_terminates || c.noop_terminates; }

TcWs carve_ws(const wm_handle *h, int B, void *ws, int T_teacher = -1) {
    const wm_config &c = h->cfg;
    const size_t KX = (size_t)c.z_dim + c.h_dim, H = c.h_dim;
    char *p = (char *)ws;
    TcWs w{};
    for (int i = 0; i < 2; ++i) { w.x[i] = (__nv_bfloat16 *)p; p += a256((size_t)B * KX * 2); }
    if (c.precision == WM_FP32)
        for (int i = 0; i < 2; ++i) { w.x_lo[i] = (__nv_bfloat16 *)p; p += a256((size_t)B * KX * 2); }
    w.c = (float *)p; p += a256((size_t)B * H * 4);
    w.h32 = (float *)p; p += a256((size_t)B * H * 4);
    w.act = (int32_t *)p; p += a256((size_t)B * 4);
    for (int i = 0; i < 2; ++i) { w.fz[i] = (uint8_t *)p; p += a256((size_t)B); }
    w.rt = (float *)p; p += a256((size_t)B * 4);
    w.mem = (float *)p; p += a256((size_t)B * 4);
    if (c.n_xfers > 0) {
        w.logits = (float *)p; p += a256((size_t)B * c.a_dim * 4);
        w.act2 = (int32_t *)p; p += a256((size_t)B * 4);
    }
    if (can_compact(c)) {
        w.c2 = (float *)p; p += a256((size_t)B * H * 4);
        w.hfin = (float *)p; p += a256((size_t)B * H * 4);
        w.cfin = (float *)p; p += a256((size_t)B * H * 4);
        for (int i = 0; i < 2; ++i) { w.rows[i] = (int32_t *)p; p += a256((size_t)B * 4); }
        w.cnt = (int *)p; p += 256;
        w.dstep = (int *)p; p += a256((size_t)B * 4);
    }
    w.nll_part = (float *)p;
    p += a256((size_t)4 * h->tc.n_head_tiles * B * 4);
    if (T_teacher >= 0) {  // scoring: frame 0 is written by the init kernel even when T = 0
        const size_t rows = (size_t)(T_teacher + 1) * B;
        w.xall = (__nv_bfloat16 *)p; p += a256(rows * KX * 2);
        if (c.precision == WM_FP32) { w.xall_lo = (__nv_bfloat16 *)p; p += a256(rows * KX * 2); }
        w.part = (float *)p;
    }
    return w;
}

}  // namespace

// ---------------------------------------------------------------------------
// Host side: packing, support test, per-call orchestration.

int wm_tc_supported(const wm_handle *h) { return h->tc.ok; }

size_t wm_tc_ws(const wm_handle *h, int B, int T_teacher) {
    const wm_config &c = h->cfg;
    const size_t KX = (size_t)c.z_dim + c.h_dim, H = c.h_dim;
    const size_t rows = T_teacher >= 0 ? (size_t)(T_teacher + 1) * B : 0;
    const size_t teach = T_teacher >= 0 ? (c.precision == WM_FP32 ? 2 : 1) * a256(rows * KX * 2) +
                                              a256((size_t)4 * h->tc.n_head_tiles * T_teacher * B * 4)
                                        : 0;
    return teach + 2 * a256((size_t)B * KX * 2) + 2 * a256((size_t)B * H * 4) + a256((size_t)B * 4) + 2 * a256(B) +
           2 * a256((size_t)B * 4) + a256((size_t)4 * h->tc.n_head_tiles * B * 4) + 256 +
           (c.n_xfers > 0 ? a256((size_t)B * c.a_dim * 4) + a256((size_t)B * 4) : 0) +
           (can_compact(c) ? 3 * a256((size_t)B * H * 4) + 3 * a256((size_t)B * 4) + 256 : 0) +
           (c.precision == WM_FP32 ? 2 * a256((size_t)B * KX * 2) : 0);
}

cudaError_t wm_tc_pack(wm_handle *h, const wm_weights *w) {
    const wm_config &c = h->cfg;
    wm_tc_weights &T = h->tc;
    memset(&T, 0, sizeof(T));
    const int Z = c.z_dim, A = c.a_dim, H = c.h_dim, K = c.k_mix, KX = Z + H;
    // fp32 models: the split path (flat actions only: the gate epilogue's second-row slots
    // carry the action row's lo part)
    const bool f32 = c.precision == WM_FP32;
    if ((f32 && c.n_xfers > 0) || H % 64 != 0 || A % 64 != 0 || (A > 256 && A != 512) || K > 8 || Z % 8 != 0 ||
        !get_encode())
        return cudaSuccess;
    const int DS = (3 * K + 7) & ~7;  // head columns per latent dim
    const int dpt = HEAD_TILE / DS;
    int nht = (Z + dpt - 1) / dpt;
    const int last_dims = Z - (nht - 1) * dpt;
    int rd_tile = nht - 1, rd_col = DS * last_dims;
    if (rd_col + h->NR > HEAD_TILE) {  // reward / done (/ runtime / memory) get a tile of their own
        rd_tile = nht;
        rd_col = 0;
        ++nht;
    }
    T.dims_per_tile = dpt;
    T.n_head_tiles = nht;
    T.rd_tile = rd_tile;
    T.rd_col = rd_col;
    auto bf = [](float v) { return __float2bfloat16_rn(v); };
    // controller: W_c^T [A, KX]
    std::vector<__nv_bfloat16> wc((size_t)A * KX), wg((size_t)4 * H * KX), wa((size_t)A * 4 * H),
        wh((size_t)nht * HEAD_TILE * H, bf(0.f));
    std::vector<float> bc(A), bg(4 * H), bh((size_t)nht * HEAD_TILE, 0.f);
    for (int a = 0; a < A; ++a) {
        for (int k = 0; k < KX; ++k) wc[(size_t)a * KX + k] = bf(w->W_ctrl[(size_t)k * A + a]);
        bc[a] = w->b_ctrl[a];
    }
    // gates: row n = 256*j + 64*gate + u  <->  canonical column gate*H + 64*j + u
    for (int n = 0; n < 4 * H; ++n) {
        const int j = n / 256, gate = (n % 256) / 64, u = n % 64;
        const size_t col = (size_t)gate * H + 64 * j + u;
        for (int k = 0; k < KX; ++k) {
            const size_t src = k < Z ? k : k + A;
            wg[(size_t)n * KX + k] = bf(w->W_lstm[src * 4 * H + col]);
        }
        bg[n] = w->b_lstm[col];
        for (int a = 0; a < A; ++a) wa[(size_t)a * 4 * H + n] = bf(w->W_lstm[(size_t)(Z + a) * 4 * H + col]);
    }
    // heads: tile j, local dim i, component k, part p -> row j*240 + DS*i + 3k + p
    const size_t M = (size_t)3 * K * Z;
    for (int d = 0; d < Z; ++d)
        for (int part = 0; part < 3; ++part)
            for (int k = 0; k < K; ++k) {
                const size_t row = (size_t)(d / dpt) * HEAD_TILE + DS * (d % dpt) + 3 * k + part;
                const size_t col = (size_t)part * K * Z + (size_t)d * K + k;
                for (int i = 0; i < H; ++i) wh[row * H + i] = bf(w->W_mdn[(size_t)i * M + col]);
                bh[row] = w->b_mdn[col];
            }
    {
        const size_t rr = (size_t)rd_tile * HEAD_TILE + rd_col;
        for (int i = 0; i < H; ++i) {
            wh[rr * H + i] = bf(w->w_rew[i]);
            wh[(rr + 1) * H + i] = bf(w->w_done[i]);
        }
        bh[rr] = w->b_rew;
        bh[rr + 1] = w->b_done;
        if (c.reward_mode == WM_REWARD_SHAPED) {
            for (int i = 0; i < H; ++i) {
                wh[(rr + 2) * H + i] = bf(w->w_rt[i]);
                wh[(rr + 3) * H + i] = bf(w->w_mem[i]);
            }
            bh[rr + 2] = w->b_rt;
            bh[rr + 3] = w->b_mem;
        }
        if (c.value_head) {
            for (int i = 0; i < H; ++i) wh[(rr + h->NR - 1) * H + i] = bf(w->w_val[i]);
            bh[rr + h->NR - 1] = w->b_val;
        }
    }
    cudaError_t e;
    auto up = [&](void **dst, const void *src, size_t bytes) {
        cudaError_t r = cudaMalloc(dst, bytes);
        if (r == cudaSuccess) r = cudaMemcpy(*dst, src, bytes, cudaMemcpyHostToDevice);
        return r;
    };
    if (f32) {  // the lo parts: bf16(w - hi), from the same canonical values
        auto lo_of = [&](std::vector<__nv_bfloat16> &hi, auto canon) {
            std::vector<__nv_bfloat16> lo(hi.size());
            for (size_t i = 0; i < hi.size(); ++i) lo[i] = bf(canon(i) - __bfloat162float(hi[i]));
            return lo;
        };
        auto wc_lo = lo_of(wc, [&](size_t i) { const size_t a = i / KX, k = i % KX; return w->W_ctrl[k * A + a]; });
        auto wg_lo = lo_of(wg, [&](size_t i) {
            const size_t n = i / KX, k = i % KX;
            const size_t j = n / 256, gate = (n % 256) / 64, u = n % 64, col = gate * H + 64 * j + u;
            const size_t src = k < (size_t)Z ? k : k + A;
            return w->W_lstm[src * 4 * H + col];
        });
        auto wa_lo = lo_of(wa, [&](size_t i) {
            const size_t a = i / (4 * H), n = i % (4 * H);
            const size_t j = n / 256, gate = (n % 256) / 64, u = n % 64, col = gate * H + 64 * j + u;
            return w->W_lstm[(Z + a) * 4 * H + col];
        });
        std::vector<float> whf(wh.size(), 0.f);  // canonical values of the packed head rows
        for (int d = 0; d < Z; ++d)
            for (int part = 0; part < 3; ++part)
                for (int k = 0; k < K; ++k) {
                    const size_t row = (size_t)(d / dpt) * HEAD_TILE + DS * (d % dpt) + 3 * k + part;
                    const size_t col = (size_t)part * K * Z + (size_t)d * K + k;
                    for (int i = 0; i < H; ++i) whf[row * H + i] = w->W_mdn[(size_t)i * M + col];
                }
        {
            const size_t rr = (size_t)rd_tile * HEAD_TILE + rd_col;
            for (int i = 0; i < H; ++i) {
                whf[rr * H + i] = w->w_rew[i];
                whf[(rr + 1) * H + i] = w->w_done[i];
                if (c.reward_mode == WM_REWARD_SHAPED) {
                    whf[(rr + 2) * H + i] = w->w_rt[i];
                    whf[(rr + 3) * H + i] = w->w_mem[i];
                }
                if (c.value_head) whf[(rr + h->NR - 1) * H + i] = w->w_val[i];
            }
        }
        auto wh_lo = lo_of(wh, [&](size_t i) { return whf[i]; });
        if ((e = up(&T.wc_lo, wc_lo.data(), wc_lo.size() * 2)) != cudaSuccess) return e;
        if ((e = up(&T.wg_lo, wg_lo.data(), wg_lo.size() * 2)) != cudaSuccess) return e;
        if ((e = up(&T.wa_lo, wa_lo.data(), wa_lo.size() * 2)) != cudaSuccess) return e;
        if ((e = up(&T.wh_lo, wh_lo.data(), wh_lo.size() * 2)) != cudaSuccess) return e;
    }
    {  // 128-column gate tiles: row n = 128 j + 32 gate + u <-> column gate H + 32 j + u
        std::vector<__nv_bfloat16> wgn((size_t)4 * H * KX), wan((size_t)A * 4 * H);
        std::vector<__nv_bfloat16> wgnl(f32 ? wgn.size() : 0), wanl(f32 ? wan.size() : 0);
        std::vector<float> bgn(4 * H);
        auto lo = [&](float v, __nv_bfloat16 hi) { return bf(v - __bfloat162float(hi)); };
        for (int n = 0; n < 4 * H; ++n) {
            const int j = n / 128, gate = (n % 128) / 32, u = n % 32;
            const size_t col = (size_t)gate * H + 32 * j + u;
            for (int k = 0; k < KX; ++k) {
                const size_t src = k < Z ? k : k + A, i = (size_t)n * KX + k;
                const float v = w->W_lstm[src * 4 * H + col];
                wgn[i] = bf(v);
                if (f32) wgnl[i] = lo(v, wgn[i]);
            }
            bgn[n] = w->b_lstm[col];
            for (int a = 0; a < A; ++a) {
                const size_t i = (size_t)a * 4 * H + n;
                const float v = w->W_lstm[(size_t)(Z + a) * 4 * H + col];
                wan[i] = bf(v);
                if (f32) wanl[i] = lo(v, wan[i]);
            }
        }
        if ((e = up(&T.wg_n, wgn.data(), wgn.size() * 2)) != cudaSuccess) return e;
        if ((e = up(&T.wa_n, wan.data(), wan.size() * 2)) != cudaSuccess) return e;
        if ((e = up((void **)&T.bg_n, bgn.data(), bgn.size() * 4)) != cudaSuccess) return e;
        if (f32) {
            if ((e = up(&T.wg_n_lo, wgnl.data(), wgnl.size() * 2)) != cudaSuccess) return e;
            if ((e = up(&T.wa_n_lo, wanl.data(), wanl.size() * 2)) != cudaSuccess) return e;
        }
    }
    if ((e = up(&T.wc, wc.data(), wc.size() * 2)) != cudaSuccess) return e;
    if ((e = up(&T.wg, wg.data(), wg.size() * 2)) != cudaSuccess) return e;
    if ((e = up(&T.wa, wa.data(), wa.size() * 2)) != cudaSuccess) return e;
    if ((e = up(&T.wh, wh.data(), wh.size() * 2)) != cudaSuccess) return e;
    if ((e = up((void **)&T.bc, bc.data(), bc.size() * 4)) != cudaSuccess) return e;
    if ((e = up((void **)&T.bg, bg.data(), bg.size() * 4)) != cudaSuccess) return e;
    if ((e = up((void **)&T.bh, bh.data(), bh.size() * 4)) != cudaSuccess) return e;
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&T.sms, cudaDevAttrMultiProcessorCount, dev);
    T.ok = 1;
    return cudaSuccess;
}

int wm_tc_call_ok(const wm_handle *h, unsigned long long episode_offset) {
    // a 256-row tile must not straddle two candidates of a population
    return h->P <= 1 || (h->E % 256 == 0 && episode_offset % 256 == 0);
}

cudaError_t wm_tc_set_controllers(wm_handle *h, int P, const float *W_ctrl, const float *b_ctrl) {
    wm_tc_weights &T = h->tc;
    const wm_config &c = h->cfg;
    const int A = c.a_dim, KX = c.z_dim + c.h_dim;
    const bool f32 = c.precision == WM_FP32;
    std::vector<__nv_bfloat16> wc((size_t)P * A * KX), wcl(f32 ? wc.size() : 0);
    for (int g = 0; g < P; ++g)
        for (int a = 0; a < A; ++a)
            for (int k = 0; k < KX; ++k) {
                const size_t i = ((size_t)g * A + a) * KX + k;
                const float v = W_ctrl[((size_t)g * KX + k) * A + a];
                wc[i] = __float2bfloat16_rn(v);
                if (f32) wcl[i] = __float2bfloat16_rn(v - __bfloat162float(wc[i]));
            }
    cudaFree(T.wc);
    cudaFree(T.wc_lo);
    cudaFree(T.bc);
    T.wc = nullptr;
    T.wc_lo = nullptr;
    T.bc = nullptr;
    cudaError_t e = cudaMalloc(&T.wc, wc.size() * 2);
    if (e == cudaSuccess) e = cudaMemcpy(T.wc, wc.data(), wc.size() * 2, cudaMemcpyHostToDevice);
    if (e == cudaSuccess && f32) e = cudaMalloc(&T.wc_lo, wcl.size() * 2);
    if (e == cudaSuccess && f32) e = cudaMemcpy(T.wc_lo, wcl.data(), wcl.size() * 2, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMalloc((void **)&T.bc, (size_t)P * A * 4);
    if (e == cudaSuccess) e = cudaMemcpy(T.bc, b_ctrl, (size_t)P * A * 4, cudaMemcpyHostToDevice);
    return e;
}

void wm_tc_free(wm_handle *h) {
    wm_tc_weights &T = h->tc;
    cudaFree(T.wc); cudaFree(T.wg); cudaFree(T.wa); cudaFree(T.wh);
    cudaFree(T.wc_lo); cudaFree(T.wg_lo); cudaFree(T.wa_lo); cudaFree(T.wh_lo);
    cudaFree(T.wg_n); cudaFree(T.wa_n); cudaFree(T.bg_n); cudaFree(T.wg_n_lo); cudaFree(T.wa_n_lo);
    if (h->dead_host) cudaFreeHost(h->dead_host);
    h->dead_host = h->dead_dev = nullptr;
    for (cudaEvent_t ev : h->step_events) cudaEventDestroy(ev);
    h->step_events.clear();
    cudaFree(T.bc); cudaFree(T.bg); cudaFree(T.bh);
    memset(&T, 0, sizeof(T));
}

// One call: rollout (teacher = 0) or teacher-forced scoring (teacher = 1).
static cudaError_t tc_run(const wm_handle *h, int teacher, const wm_rollout_dev *ra, const wm_nll_dev *na,
                          void *ws, cudaStream_t s) {
    const wm_config &c = h->cfg;
    const wm_tc_weights &T = h->tc;
    const int B = teacher ? na->N : ra->B, Tn = teacher ? na->T : ra->T;
    const int Z = c.z_dim, A = c.a_dim, H = c.h_dim, KX = Z + H;
    if (B == 0) { h->last_launches = 0; return cudaSuccess; }
    TcWs w = carve_ws(h, B, ws, teacher ? Tn : -1);
    StepIO io{};
    io.B = B; io.Z = Z; io.A = A; io.H = H; io.K = c.k_mix; io.T = Tn;
    io.seed = c.seed; io.teacher = teacher;
    io.ctrl_sample = c.ctrl_sample; io.ctrl_tau = c.ctrl_tau; io.mdn_tau = c.mdn_tau;
    io.sigma_sqrt_tau = c.sigma_sqrt_tau; io.done_terminates = c.done_terminates;
    io.noop_terminates = c.noop_terminates;
    io.c = w.c; io.h32 = w.h32; io.act = w.act;
    io.b_ctrl = T.bc; io.b_gate = T.bg; io.b_head = T.bh;
    io.wa = (const __nv_bfloat16 *)T.wa;
    io.dims_per_tile = T.dims_per_tile; io.rd_tile = T.rd_tile; io.rd_col = T.rd_col;
    // h (fp32) is read back only by frozen episodes and for h_final: with no way to freeze
    // during the call it is needed after the last step only
    io.h32_mode = teacher ? 0 : (c.done_terminates || c.noop_terminates) ? 2 : 1;
    io.nll_part = w.nll_part;
    io.reward_mode = teacher ? WM_REWARD_HEAD : c.reward_mode;
    io.alpha = c.reward_alpha; io.beta = c.reward_beta; io.invalid_reward = c.invalid_reward;
    io.rt = w.rt; io.mem = w.mem;
    if (!teacher && c.reward_mode == WM_REWARD_SHAPED) {
        io.rt0 = ra->rt0; io.mem0 = ra->mem0; io.rt_seq = ra->rt_seq; io.mem_seq = ra->mem_seq;
    }
    io.pop_P = h->P; io.pop_E = h->E;
    io.nr = h->NR;
    const bool hier = !teacher && c.n_xfers > 0;
    io.n_xfers = hier ? c.n_xfers : 0;
    io.logits = w.logits;
    io.act2 = w.act2;
    if (hier) {
        io.loc_mask = ra->loc_mask;
        io.loc_actions = ra->loc_actions;
    }
    if (!teacher) {
        io.logp_seq = ra->logp_seq;
        io.value_seq = c.value_head ? ra->value_seq : nullptr;
    }
    if (teacher) {
        io.act_in = na->actions; io.z_seq = na->z_seq; io.lengths = na->lengths;
        io.h_seq = na->h_seq; io.c_seq = na->c_seq; io.mdn_seq = na->mdn_seq;
    } else {
        io.ep0 = ra->ep0;
        io.mask = ra->mask; io.z_out = ra->z_out; io.actions = ra->actions; io.rewards = ra->rewards;
        io.done = ra->done; io.h_seq = ra->h_seq; io.c_seq = ra->c_seq; io.mdn_seq = ra->mdn_seq;
        io.comp_seq = ra->comp_seq;
    }
    int launches = 0;
    const int init_grid = 1024;
    // Rollouts whose episodes end compact their live episodes before every step (one
    // controller per call: a population's tiles must stay whole).
    const bool compact = !teacher && can_compact(c) && h->P <= 1 && Tn > 0;
    io.fz_cur = w.fz[0];
    {
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        k_tc_init<<<init_grid, 256, 0, s>>>(io, teacher ? nullptr : ra->z0, teacher ? nullptr : ra->h0,
                                            teacher ? nullptr : ra->c0,
                                            (teacher || compact) ? nullptr : ra->done0,
                                            teacher ? w.xall : w.x[0], teacher ? w.xall_lo : w.x_lo[0], w.fz[0], w.fz[1],
                                            T.n_head_tiles, compact ? w.dstep : nullptr,
                                            compact ? w.cnt : nullptr);
    }
    ++launches;
    wm_step_stage *hooks = teacher ? nullptr : ra->stage;  // per-step staging of host arrays
    if (hooks) {
        cudaError_t he = hooks->after_init(s);
        if (he != cudaSuccess) return he;
    }
    const bool f32 = c.precision == WM_FP32;  // the split path: second operand maps and lo outputs
    CUtensorMap mx[2], mxs[2], mwc, mwg, mwh, mc, mc2, mxl[2], mxsl[2], mwcl, mwgl, mwhl;
    // B-operand boxes are half an instantiated BN (each CTA of a pair loads half the rows;
    // rows past A read as zero)
    const uint32_t ctrl_box = A > 128 ? 128u : 64u;
    if (!make_map(&mx[0], w.x[0], B, KX, BM) || !make_map(&mx[1], w.x[1], B, KX, BM) ||
        !make_map(&mxs[0], w.x[0], B, KX, 32) || !make_map(&mxs[1], w.x[1], B, KX, 32) ||
        !make_map(&mc, w.c, B, H, 32, true) || (compact && !make_map(&mc2, w.c2, B, H, 32, true)) ||
        !make_map(&mwc, T.wc, (uint64_t)h->P * A, KX, ctrl_box) || !make_map(&mwg, T.wg, 4 * H, KX, 128) ||
        !make_map(&mwh, T.wh, (uint64_t)T.n_head_tiles * HEAD_TILE, H, HEAD_TILE / 2))
        return cudaErrorInvalidValue;
    if (f32) {
        if (!make_map(&mxl[0], w.x_lo[0], B, KX, BM) || !make_map(&mxl[1], w.x_lo[1], B, KX, BM) ||
            !make_map(&mxsl[0], w.x_lo[0], B, KX, 32) || !make_map(&mxsl[1], w.x_lo[1], B, KX, 32) ||
            !make_map(&mwcl, T.wc_lo, (uint64_t)h->P * A, KX, ctrl_box) || !make_map(&mwgl, T.wg_lo, 4 * H, KX, 128) ||
            !make_map(&mwhl, T.wh_lo, (uint64_t)T.n_head_tiles * HEAD_TILE, H, HEAD_TILE / 2))
            return cudaErrorInvalidValue;
    } else {  // unused by the bf16 kernels
        mxl[0] = mx[0]; mxl[1] = mx[1]; mxsl[0] = mxs[0]; mxsl[1] = mxs[1];
        mwcl = mwc; mwgl = mwg; mwhl = mwh;
    }
    io.wa_lo = (const __nv_bfloat16 *)T.wa_lo;
    const int m_tiles = (B + 2 * BM - 1) / (2 * BM);  // 256-row tiles, one per CTA pair
    // Programmatic dependent launch hides the ~4 us between consecutive launches (a fifth of
    // a call at B = 8192), but made the long launches of B = 65536 3% slower: on below 32768.
    const bool pdl = B < 32768;
    // 128-column gate tiles when 256-column ones would leave most CTA pairs idle: few row
    // tiles, or compacted live rows (bf16, flat actions); on the fp32 path, scoring
    const int pairs = T.sms / 2;
    const bool narrow = !hier && T.wg_n &&
                        (f32 ? teacher && T.wg_n_lo : (compact || teacher || m_tiles * (H / 64) < pairs));
    CUtensorMap mwgn, mwgnl, mxsn[2];
    if (narrow && (!make_map(&mwgn, T.wg_n, 4 * H, KX, 64) || !make_map_x32(&mxsn[0], w.x[0], B, KX) ||
                   !make_map_x32(&mxsn[1], w.x[1], B, KX)))
        return cudaErrorInvalidValue;
    if (narrow && f32 && !make_map(&mwgnl, T.wg_n_lo, 4 * H, KX, 64)) return cudaErrorInvalidValue;
    StepIO gio_n;  // the gate launches' parameters with the 128-column packing
    if (teacher) {  // batched scoring: the recurrence step by step, then one head GEMM
        const size_t fr = (size_t)B * KX;  // elements of one frame of operand rows
        cudaError_t e = cudaSuccess;
        if (Tn > 0) {
            wm_ktime kt(h, WM_KERNEL_AUX, s);
            k_tc_frames<<<init_grid, 256, 0, s>>>(B, Tn, Z, KX, na->z_seq, w.xall, w.xall_lo);
            ++launches;
        }
        io.x_cur = io.x_next = io.x_next_lo = nullptr;
        for (int t = 0; t < Tn && e == cudaSuccess; ++t) {
            io.t = t;
            io.step = (uint32_t)t;
            // this step's operand rows (frame t) and where h' goes (frame t + 1)
            CUtensorMap ma, mal, ms, msl;
            if (!make_map(&ma, w.xall + t * fr, B, KX, BM) || !make_map(&ms, w.xall + (t + 1) * fr, B, KX, 32))
                return cudaErrorInvalidValue;
            if (f32) {
                if (!make_map(&mal, w.xall_lo + t * fr, B, KX, BM) || !make_map(&msl, w.xall_lo + (t + 1) * fr, B, KX, 32))
                    return cudaErrorInvalidValue;
            } else {
                mal = ma;
                msl = ms;
            }
            GemmGrid g2{m_tiles, H / 64, (KX + BK - 1) / BK, 0, h->status};
            if (t == 0) {  // an injected wait (wm_inject_wait_timeout) goes to the first GEMM
                g2.test_wait = h->test_wait;
                h->test_wait = 0;
            }
            const OpMaps opg{&ma, &mwg, &mal, &mwgl};
            if (narrow) {
                CUtensorMap msn, msnl;
                if (!make_map_x32(&msn, w.xall + (t + 1) * fr, B, KX)) return cudaErrorInvalidValue;
                if (f32 && !make_map_x32(&msnl, w.xall_lo + (t + 1) * fr, B, KX)) return cudaErrorInvalidValue;
                gio_n = io;
                gio_n.wa = (const __nv_bfloat16 *)T.wa_n;
                gio_n.b_gate = T.bg_n;
                GemmGrid g2n = g2;
                g2n.n_tiles = H / 32;
                wm_ktime kt(h, WM_KERNEL_TC_GATES, s);
                if (f32) {
                    gio_n.wa_lo = (const __nv_bfloat16 *)T.wa_n_lo;
                    const OpMaps opn{&ma, &mwgn, &mal, &mwgnl};
                    e = launch_gemm<128, 1, 3, EpiGates32N, 2, 3>(opn, mc, msn, msnl, g2n, gio_n, T.sms, s, pdl);
                } else {
                    const OpMaps opn{&ma, &mwgn, &ma, &mwgn};
                    e = launch_gemm<128, 1, 3, EpiGatesN, 2>(opn, mc, msn, msn, g2n, gio_n, T.sms, s, pdl);
                }
            } else {
                wm_ktime kt(h, WM_KERNEL_TC_GATES, s);
                if (f32) e = launch_gemm<256, 1, 2, EpiGates32, 2, 3>(opg, mc, ms, msl, g2, io, T.sms, s, pdl);
                else e = launch_gemm<256, 1, 2, EpiGates, 2>(opg, mc, ms, ms, g2, io, T.sms, s, pdl);
            }
            ++launches;
        }
        if (e != cudaSuccess) return e;
        const int parts = 4 * T.n_head_tiles;
        if (Tn > 0) {  // every (step, sequence) row: h_{t+1} of frame t + 1 against z_{t+1}
            CUtensorMap mh, mhl;
            const int rows = B * Tn;
            if (!make_map(&mh, w.xall + fr, (uint64_t)rows, KX, BM)) return cudaErrorInvalidValue;
            if (f32) {
                if (!make_map(&mhl, w.xall_lo + fr, (uint64_t)rows, KX, BM)) return cudaErrorInvalidValue;
            } else {
                mhl = mh;
            }
            StepIO hio = io;
            hio.B = rows;
            hio.t = 0;
            hio.nseq = B;
            hio.z_tgt = na->z_seq + (size_t)B * Z;
            hio.nll_part = w.part;
            const GemmGrid g3{(rows + 2 * BM - 1) / (2 * BM), T.n_head_tiles, (H + BK - 1) / BK, Z, h->status};
            const OpMaps oph{&mh, &mwh, &mhl, &mwhl};
            wm_ktime kt(h, WM_KERNEL_TC_HEADS, s);
            if (f32) e = launch_gemm<HEAD_TILE, 1, 3, EpiHeads, 2, 3>(oph, mc, mc, mc, g3, hio, T.sms, s, pdl);
            else e = launch_gemm<HEAD_TILE, 1, 3, EpiHeads, 2>(oph, mc, mc, mc, g3, hio, T.sms, s, pdl);
            ++launches;
            if (e != cudaSuccess) return e;
        }
        {
            wm_ktime kt(h, WM_KERNEL_AUX, s);
            k_tc_nll_reduce<<<(B + 7) / 8, 256, 0, s>>>(B, Tn, parts, w.part, na->nll);
        }
        ++launches;
        h->last_launches = launches;
        return cudaGetLastError();
    }
    float *cbuf[2] = {w.c, w.c2};
    const bool staged = hooks && hooks->stepping();  // host outputs copied step by step
    CompactIO q{};  // compaction: the fields that do not change from step to step
    // Early stop: once every episode has ended, the remaining steps would only launch empty
    // kernels; the compaction kernel then sets a host-mapped word to this call's number and
    // the host issues no further step.  To see it in time, the host keeps at most LOOKAHEAD
    // steps in flight (it waits for step t - LOOKAHEAD before issuing step t), so such a call
    // returns once its last step is issued, a few steps before the device finishes.  Where
    // the host stops depends on timing; the results do not.  Not with per-step staging or
    // during stream capture.
    constexpr int LOOKAHEAD = 4;
    bool early = false;
    if (compact && !staged) {
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (cudaStreamIsCapturing(s, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusNone) {
            if (!h->dead_host && cudaHostAlloc((void **)&h->dead_host, sizeof(int), cudaHostAllocMapped) == cudaSuccess) {
                *h->dead_host = 0;
                if (cudaHostGetDevicePointer((void **)&h->dead_dev, h->dead_host, 0) != cudaSuccess) {
                    cudaFreeHost(h->dead_host);
                    h->dead_host = h->dead_dev = nullptr;
                }
            }
            while (h->step_events.size() < (size_t)LOOKAHEAD) {
                cudaEvent_t ev = nullptr;
                if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) break;
                h->step_events.push_back(ev);
            }
            cudaGetLastError();
            early = h->dead_dev != nullptr && h->step_events.size() >= (size_t)LOOKAHEAD;
        }
    }
    if (compact) {
        q.dead_flag = early ? h->dead_dev : nullptr;
        q.call_id = ++h->call_seq;
        q.B = B; q.Z = Z; q.H = H; q.KX = KX; q.M = 3 * c.k_mix * Z; q.T = Tn;
        q.fill = staged;  // staged outputs leave step by step: fill each step's
        q.dstep = w.dstep; q.h32 = w.h32;
        q.hfin = w.hfin; q.cfin = w.cfin; q.rt = w.rt; q.mem = w.mem;
        q.z_out = ra->z_out; q.actions = ra->actions; q.rewards = ra->rewards; q.done = ra->done;
        q.h_seq = ra->h_seq; q.c_seq = ra->c_seq; q.mdn_seq = ra->mdn_seq; q.comp_seq = ra->comp_seq;
        q.logp_seq = io.logp_seq; q.value_seq = io.value_seq; q.rt_seq = io.rt_seq; q.mem_seq = io.mem_seq;
        q.loc_actions = io.loc_actions;
    }
    cudaError_t e = cudaSuccess;
    int t_end = Tn;  // steps issued
    for (int t = 0; t < Tn && e == cudaSuccess; ++t) {
        if (early && t >= LOOKAHEAD) {
            if ((e = cudaEventSynchronize(h->step_events[t % LOOKAHEAD])) != cudaSuccess) break;
            if (*(volatile int *)h->dead_host == q.call_id) {
                t_end = t;
                break;
            }
        }
        io.t = t;
        io.step = teacher ? (uint32_t)t : ra->t0 + (uint32_t)t;
        // operands: X ping-pongs between the two buffers; when compacting, the live rows are
        // packed from x[0] (written by the previous step) into x[1] (this step's operand), and
        // this step writes x[0] again; c alternates between its two buffers
        const int xa = compact ? 1 : (t & 1), xn = compact ? 0 : ((t + 1) & 1);
        io.x_cur = w.x[xa];
        io.x_next = w.x[xn];
        io.x_next_lo = w.x_lo[xn];
        io.fz_cur = w.fz[compact ? 0 : (t & 1)];
        io.fz_next = w.fz[compact ? 1 : ((t + 1) & 1)];
        const CUtensorMap &mC = (compact && ((t + 1) & 1)) ? mc2 : mc;
        if (hooks && (e = hooks->before_step(t, s)) != cudaSuccess) break;
        if (compact) {
            q.t = t;
            q.rows_in = t ? w.rows[(t - 1) & 1] : nullptr;
            q.n_in = t ? w.cnt + ((t - 1) & 3) : nullptr;
            q.dies = t ? w.fz[1] : ra->done0;
            q.x_in = w.x[0]; q.x_out = w.x[1];
            q.x_in_lo = w.x_lo[0]; q.x_out_lo = w.x_lo[1];
            q.c_in = cbuf[t & 1]; q.c_out = cbuf[(t + 1) & 1];
            q.rows_out = w.rows[t & 1]; q.n_out = w.cnt + (t & 3); q.n_clear = w.cnt + ((t + 1) & 3);
            q.n_prev2 = t >= 2 ? w.cnt + ((t - 2) & 3) : nullptr;
            io.rows = w.rows[t & 1];
            io.n_rows = w.cnt + (t & 3);
            io.c = cbuf[(t + 1) & 1];
            cudaLaunchConfig_t lc = {};
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
            at[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
            {  // a block per CROWS rows, and enough threads for the frozen episodes' outputs
                const size_t fe = q.fill ? (size_t)Z + ((q.h_seq || q.c_seq) ? H : 0) + (q.mdn_seq ? q.M : 0) + 1 : 0;
                const size_t rows_blocks = ((size_t)B + CROWS - 1) / CROWS;
                const size_t fill_blocks = std::min<size_t>(((size_t)B * fe + 4 * CTHREADS - 1) / (4 * CTHREADS),
                                                            (size_t)16 * T.sms);
                lc.gridDim = dim3((unsigned)std::max(rows_blocks, fill_blocks));
            }
            lc.blockDim = dim3(CTHREADS);
            lc.stream = s;
            lc.attrs = at;
            lc.numAttrs = 1;
            {
                wm_ktime kt(h, WM_KERNEL_AUX, s);
                e = cudaLaunchKernelEx(&lc, k_tc_compact, q);
            }
            ++launches;
            if (e != cudaSuccess) break;
        }
        // the controller's weight rows: the tile's candidate's, when there is a population
        GemmGrid g1{m_tiles, 1, (KX + BK - 1) / BK, 0, h->status, teacher ? 0ull : ra->ep0, h->P, h->E, A};
        g1.n_rows = io.n_rows;
        // an injected wait (wm_inject_wait_timeout) goes to the call's first GEMM launch
        uint32_t test_wait = 0;
        if (t == 0) {
            test_wait = h->test_wait;
            h->test_wait = 0;
        }
        if (!teacher) g1.test_wait = test_wait;
        const OpMaps opc{&mx[xa], &mwc, &mxl[xa], &mwcl}, opg{&mx[xa], &mwg, &mxl[xa], &mwgl},
            oph{&mx[xn], &mwh, &mxl[xn], &mwhl};
        if (!teacher && !hier) {
            wm_ktime kt(h, WM_KERNEL_TC_CTRL, s);
            if (f32) {
                if (A > 256) e = launch_gemm<256, 2, 2, EpiCtrl, 2, 3>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
                else if (A > 128) e = launch_gemm<256, 1, 3, EpiCtrl, 2, 3>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
                else e = launch_gemm<128, 1, 3, EpiCtrl, 2, 3>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
            } else {
                if (A > 256) e = launch_gemm<256, 2, 2, EpiCtrl, 2>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
                else if (A > 128) e = launch_gemm<256, 1, 3, EpiCtrl, 2>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
                else e = launch_gemm<128, 1, 3, EpiCtrl, 2>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
            }
            ++launches;
            if (e != cudaSuccess) break;
        } else if (hier) {  // the logits, then the two-stage choice (Sec. 3.1.3); bf16 models only
            {
                wm_ktime kt(h, WM_KERNEL_TC_CTRL, s);
                if (A > 256) e = launch_gemm<256, 2, 2, EpiLogits, 2>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
                else if (A > 128) e = launch_gemm<256, 1, 3, EpiLogits, 2>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
                else e = launch_gemm<128, 1, 3, EpiLogits, 2>(opc, mc, mc, mc, g1, io, T.sms, s, pdl);
            }
            ++launches;
            if (e != cudaSuccess) break;
            {
                wm_ktime kt(h, WM_KERNEL_AUX, s);
                k_tc_select<<<(unsigned)(((size_t)B * 32 + 255) / 256), 256, 0, s>>>(io);
            }
            ++launches;
        }
        GemmGrid g2{m_tiles, H / 64, (KX + BK - 1) / BK, 0, h->status};
        g2.n_rows = io.n_rows;
        if (teacher) g2.test_wait = test_wait;
        if (narrow) {
            gio_n = io;
            gio_n.wa = (const __nv_bfloat16 *)T.wa_n;
            gio_n.b_gate = T.bg_n;
            GemmGrid g2n = g2;
            g2n.n_tiles = H / 32;
            const OpMaps opn{&mx[xa], &mwgn, &mx[xa], &mwgn};
            wm_ktime kt(h, WM_KERNEL_TC_GATES, s);
            e = launch_gemm<128, 1, 3, EpiGatesN, 2>(opn, mC, mxsn[xn], mxsn[xn], g2n, gio_n, T.sms, s, pdl);
        } else {
            wm_ktime kt(h, WM_KERNEL_TC_GATES, s);
            if (f32) e = launch_gemm<256, 1, 2, EpiGates32, 2, 3>(opg, mC, mxs[xn], mxsl[xn], g2, io, T.sms, s, pdl);
            else if (hier) e = launch_gemm<256, 1, 2, EpiGates2, 2>(opg, mC, mxs[xn], mxs[xn], g2, io, T.sms, s, pdl);
            else e = launch_gemm<256, 1, 2, EpiGates, 2>(opg, mC, mxs[xn], mxs[xn], g2, io, T.sms, s, pdl);
        }
        ++launches;
        if (e != cudaSuccess) break;
        GemmGrid g3{m_tiles, T.n_head_tiles, (H + BK - 1) / BK, Z, h->status};
        g3.n_rows = io.n_rows;
        {
            wm_ktime kt(h, WM_KERNEL_TC_HEADS, s);
            if (f32) e = launch_gemm<HEAD_TILE, 1, 3, EpiHeads, 2, 3>(oph, mc, mc, mc, g3, io, T.sms, s, pdl);
            else e = launch_gemm<HEAD_TILE, 1, 3, EpiHeads, 2>(oph, mc, mc, mc, g3, io, T.sms, s, pdl);
        }
        ++launches;
        if (e == cudaSuccess && hooks) e = hooks->after_step(t, s);
        if (e == cudaSuccess && early) e = cudaEventRecord(h->step_events[t % LOOKAHEAD], s);
    }
    if (e != cudaSuccess) return e;
    if (compact) {
        if (!q.fill) {
            wm_ktime kt(h, WM_KERNEL_AUX, s);
            k_tc_fill_frozen<<<16 * T.sms, 256, 0, s>>>(q);
            ++launches;
        }
        if (ra->h_final || ra->c_final) {
            wm_ktime kt(h, WM_KERNEL_AUX, s);
            const int tl = t_end - 1;  // the last issued step
            k_tc_finish_compact<<<init_grid, 256, 0, s>>>(B, H, Tn, w.dstep, w.rows[tl & 1], w.cnt + (tl & 3),
                                                          w.h32, cbuf[Tn & 1], w.hfin, w.cfin, ra->h_final,
                                                          ra->c_final);
            ++launches;
        }
    } else {
        wm_ktime kt(h, WM_KERNEL_AUX, s);
        k_tc_finish<<<init_grid, 256, 0, s>>>(B, H, w.h32, w.c, teacher ? nullptr : ra->h_final,
                                              teacher ? nullptr : ra->c_final, w.nll_part, 4 * T.n_head_tiles,
                                              teacher ? na->nll : nullptr);
        ++launches;
    }
    h->last_launches = launches;
    return cudaGetLastError();
}

cudaError_t wm_tc_rollout(const wm_handle *h, const wm_rollout_dev &a, void *ws, cudaStream_t s) {
    return tc_run(h, 0, &a, nullptr, ws, s);
}

cudaError_t wm_tc_nll(const wm_handle *h, const wm_nll_dev &a, void *ws, cudaStream_t s) {
    return tc_run(h, 1, nullptr, &a, ws, s);
}
