/*
 * wm.h -- C ABI of the GB300 world-model "dream" engine.
 *
 * The engine runs batched rollouts inside the world model of RLFlow
 * (Mitchell et al., "RLFlow: Optimising Neural Network Subgraph
 * Transformation with World Models", SIGMOD'22) and scores teacher-forced
 * sequences under its mixture-density head.  The world model is an MDN-RNN
 * (Sec. 3.3.1 "Recurrent Neural Networks", Sec. 3.3.2 "MDN-RNN") driven by the
 * linear controller a_t = W_c [z_t, h_t] + b_c (Sec. 3.4 "Action Controller");
 * one wm_rollout step is the imagined-environment analogue of the Gym
 * step(action) -> (next_state, reward, terminal, info) of Sec. 3.1.1.
 *
 * Notation: B episodes, T steps, Z latent size, A actions, H LSTM hidden size,
 * K mixture components, M = 3*K*Z mixture-head outputs, W = ceil(A/32).
 *
 * Per episode and step t (all episodes independent):
 *   a1  l   = W_c^T [z_t; h_t] + b_c                               (Sec. 3.4)
 *   a2  l_j = -inf where action j is invalid (Sec. 3.1.3); a_t = lowest-index
 *       argmax, or a draw from softmax(l / ctrl_tau); -1 if nothing is valid
 *   a3  G   = W_lstm^T [z_t; onehot(a_t); h_t] + b_lstm, columns i|f|g|o
 *   a4  c'  = sig(f) c + sig(i) tanh(g);  h' = sig(o) tanh(c')       (Sec. 3.3.2)
 *   a5  [logit | mu | log sigma] = W_mdn^T h' + b_mdn;  r = w_rew.h' + b_rew;
 *       d = w_done.h' + b_done
 *   a6  pi_d = softmax(logit_d / mdn_tau) per latent dim d   (temperature eq., Sec. 3.3.2)
 *   a7  k ~ pi_d (inverse CDF on a Philox uniform), z'_d = mu_dk + sigma_dk eps_d
 *   a8  done = d > 0 (or NO-OP when noop_terminates); with done_terminates a
 *       done episode is frozen: later steps give a = -1, r = 0, done = 1 and
 *       repeat z, h, c.
 *   a9  (wm_mdn_nll) NLL_n = sum_{t<len_n} sum_d -log sum_k pi N(z_{t+1,d}; mu, sigma)
 *       with tau = 1 -- the world-model log-likelihood loss of Sec. 4.7.
 *
 * Random numbers: Philox-4x32-10 (Salmon et al., SC'11) with key = seed and
 * counter = (episode lo32, t0 + t, purpose << 24 | block, episode hi32), where
 * episode = episode_offset + b.  Purpose 0: component uniforms (4 dims per
 * block); 1: Box-Muller normals (4 dims per block); 2: controller uniform.
 * A uniform is (x >> 8) * 2^-24.  Results therefore do not depend on how the
 * episodes are split across calls or devices.
 *
 * Precision: WM_FP32 gives fp32-accurate results: the stepwise family computes
 * in fp32; the tensor-core family computes each contraction as three bf16
 * products of operands split into bf16 hi and lo parts (x = hi + lo), with fp32
 * accumulation (about 3e-6 relative error), and everything else in fp32.
 * WM_BF16 rounds every weight matrix to bf16 (RNE) at wm_create and rounds the
 * GEMM operands [z_t; h_t] and h' to bf16; biases, accumulation,
 * nonlinearities, state and sampling stay fp32.
 *
 * Memory: every array argument below may be device memory (cudaMalloc'd,
 * managed) or host memory (pinned or pageable); the library tells them apart
 * with cudaPointerGetAttributes.  Host arrays are staged through device
 * buffers owned by the handle.  In general they are copied whole on the call's
 * stream, inputs before the kernels and outputs after them.  When the call runs
 * step by step (wm_rollout on the tensor-core family, T > 1, a stream that is not
 * capturing), per-step slabs move on two copy streams owned by the handle
 * instead: the mask slab of step t goes up ahead of step t, and step t's output
 * slabs come down as soon as step t is done, overlapping the other steps.  A call
 * with a host output, or with per-step staging, returns only when every copy
 * touching the caller's arrays is complete (also when it returns an error).  All
 * arrays are dense, row-major, in the layouts given, and owned by the caller.
 *
 * Errors: argument errors are returned synchronously and leave outputs
 * untouched.  Device-side errors (a bounded wait that gave up) are recorded in
 * a device status word and returned by wm_sync.  wm_last_error gives a
 * message for the last failing call on a handle.
 *
 * Threading: a handle is not thread-safe; use one handle per host thread.
 * Calls on one handle must not overlap on the GPU (they share workspace):
 * issue them on one stream, or synchronise between streams.
 */
#ifndef WM_H
#define WM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    WM_OK = 0,
    WM_ERR_INVALID_ARG = 1,
    WM_ERR_CUDA = 2,
    WM_ERR_UNSUPPORTED = 3,
    WM_ERR_TIMEOUT = 4,
    WM_ERR_OOM = 5
} wm_status;

enum { WM_FP32 = 0, WM_BF16 = 1 };

/* Kernel family.  AUTO picks by batch size and model size; the others force
 * one (WM_ERR_UNSUPPORTED if it cannot run the model).
 *   STEPWISE  four SIMT launches per step; every model and option.
 *   FUSED     one launch for all T steps, in two members: a tcgen05 kernel for
 *             bf16 models with Z = 32, H = 256, K = 5, masked argmax and the
 *             linear reward head (one cluster per 128 episodes), and a small-batch
 *             fp32 SIMT kernel for the other models whose weights fit a cluster's
 *             shared memory (one cluster per 16 episodes; either precision,
 *             controller and reward), taken while the batch needs at most 4 waves
 *             of clusters.  Neither writes log-probs or values, takes a population
 *             or a hierarchical action.
 *   TENSOR    three tcgen05 GEMM launches per step (H % 64 == 0, A % 64 == 0). */
enum { WM_PATH_AUTO = 0, WM_PATH_STEPWISE = 1, WM_PATH_FUSED = 2, WM_PATH_TENSOR = 3 };

typedef struct {
    int z_dim, a_dim, h_dim, k_mix;   /* Z, A, H, K (K <= 32)                      */
    int precision;                    /* WM_FP32 or WM_BF16                        */
    float mdn_tau;                    /* >= 0; 0 = argmax component, z = mu        */
    int sigma_sqrt_tau;               /* 1: sigma scaled by sqrt(mdn_tau)          */
    int ctrl_sample;                  /* 0: masked argmax; 1: tempered draw        */
    float ctrl_tau;                   /* >= 0; 0 behaves as argmax                 */
    int done_terminates;              /* done head freezes the episode             */
    int noop_terminates;              /* action A-1 (NO-OP, Sec. 3.1.3) freezes it */
    unsigned long long seed;          /* Philox key                                */
    int path;                         /* WM_PATH_*                                 */
    int fused_cluster;                /* fused family, tcgen05 member: CTAs per
                                         cluster, 8 or 16; 0 = choose per call
                                         (fewest waves)                             */
    /* Reward (Sec. 3.1.4).  WM_REWARD_HEAD: r_t = w_rew . h' + b_rew.
     * WM_REWARD_SHAPED: two more linear heads on h' predict the graph's runtime
     * RT and memory accesses M, and r_t = alpha (RT_{t-1} - RT_t) +
     * beta (M_{t-1} - M_t) (Eq. 2; Eq. 1 is alpha = 1, beta = 0) when an action
     * was taken, invalid_reward when none was (a = -1).  Sec. 4.3 found
     * alpha = 0.8, beta = 0.2 best; Eq. 1 / 2 give -100 for an invalid action.
     * The stepwise and tensor-core families and the fused family's small-batch
     * member take it; the fused family's tcgen05 member does not. */
    int reward_mode;                  /* WM_REWARD_HEAD or WM_REWARD_SHAPED         */
    float reward_alpha, reward_beta;
    float invalid_reward;
    int value_head;                   /* 1: a value head V(h') = w_val . h' + b_val
                                         (a critic on the world model's state, for
                                         PPO-style training); stepwise and tensor
                                         families                                   */
    /* Hierarchical action (Sec. 3.1.3): n_xfers = NX > 0 splits the A controller
     * outputs into NX xfer logits (xfer NX-1 is the NO-OP) and L = A - NX location
     * logits.  The xfer is chosen among the valid ones (bits 0..NX-1 of the step's
     * mask words), then the location among the valid ones of the chosen xfer's
     * location mask (io.loc_mask); a tempered draw takes the controller uniform's
     * word 0 for the xfer and word 1 for the location.  The NO-OP takes no
     * location (and ends the episode with noop_terminates); an xfer with no valid
     * location gives location -1, an invalid action.  The LSTM input is
     * onehot(xfer) || onehot(location): action rows xfer and NX + location of
     * W_lstm.  0 = one flat action of A.  Stepwise and tensor-core families;
     * rollouts only (wm_mdn_nll returns WM_ERR_UNSUPPORTED).                  */
    int n_xfers;
} wm_config;

enum { WM_REWARD_HEAD = 0, WM_REWARD_SHAPED = 1 };

/* Canonical fp32 weights, row-major, HOST memory; copied (and packed) by
 * wm_create, so the caller may free them afterwards. */
typedef struct {
    const float *W_lstm;  /* [Z+A+H, 4H]: rows z | a | h; cols i | f | g | o      */
    const float *b_lstm;  /* [4H]                                                 */
    const float *W_mdn;   /* [H, 3KZ]: cols logit | mu | log sigma, index d*K + k  */
    const float *b_mdn;   /* [3KZ]                                                */
    const float *w_rew;   /* [H]                                                  */
    float b_rew;
    const float *w_done;  /* [H]                                                  */
    float b_done;
    const float *W_ctrl;  /* [Z+H, A]: rows z | h                                 */
    const float *b_ctrl;  /* [A]                                                  */
    const float *w_rt;    /* [H] predicted-runtime head (WM_REWARD_SHAPED only)   */
    float b_rt;
    const float *w_mem;   /* [H] predicted memory-access head (WM_REWARD_SHAPED)  */
    float b_mem;
    const float *w_val;   /* [H] value head (value_head only)                    */
    float b_val;
} wm_weights;

typedef struct wm_handle wm_handle;

/* Inputs and outputs of one wm_rollout call (see the memory rules above). */
typedef struct {
    const float *z0;             /* [B,Z]   required: z_{t0} of every episode        */
    const float *h0;             /* [B,H]   or NULL = zeros                          */
    const float *c0;             /* [B,H]   or NULL = zeros                          */
    const uint8_t *done0;        /* [B]     or NULL; nonzero = episode already frozen */
    const uint32_t *mask;        /* [T,B,W] or NULL = all valid; bit j of word w
                                    set = action 32w+j valid at that step            */
    float *z_out;                /* [T+1,B,Z] required; z_out[0] = z0                */
    int32_t *actions;            /* [T,B]   required; -1 = no action                 */
    float *rewards;              /* [T,B]   required                                 */
    uint8_t *done;               /* [T,B]   required                                 */
    float *h_final;              /* [B,H]   optional                                 */
    float *c_final;              /* [B,H]   optional                                 */
    float *h_seq;                /* [T,B,H] optional: h after each step              */
    float *c_seq;                /* [T,B,H] optional                                 */
    float *mdn_seq;              /* [T,B,M] optional: raw head outputs (0 if frozen) */
    uint8_t *comp_seq;           /* [T,B,Z] optional: chosen component (255 if frozen)*/
    /* WM_REWARD_SHAPED only (ignored otherwise): */
    const float *rt0, *mem0;     /* [B]     required: RT and M of each episode's graph
                                    entering the call (resume: the last rt_seq / mem_seq) */
    float *rt_seq, *mem_seq;     /* [T,B]   optional: RT_t, M_t after each step (frozen:
                                    repeated)                                          */
    float *logp_seq;             /* [T,B]   optional: log pi(a_t | z_t, h_t) of the action
                                    taken, pi = softmax(l / ctrl_tau) over the valid
                                    actions (Sec. 3.4); 0 if ctrl_tau = 0, no action was
                                    valid, or the episode is frozen                    */
    float *value_seq;            /* [T,B]   optional (value_head): V(h_{t+1}); 0 if frozen */
    /* hierarchical action (n_xfers > 0) only: */
    const uint32_t *loc_mask;    /* [T,B,NX,ceil(L/32)] or NULL = all valid: bit j of
                                    xfer x's words set = location j valid for x       */
    int32_t *loc_actions;        /* [T,B]   optional: the location taken (-1: none;
                                    `actions` holds the xfer)                         */
} wm_rollout_io;

/* Creates a world model on the current CUDA device from the weights of the
 * MDN-RNN (Sec. 3.3.1-3.3.2: the LSTM over [z_t, a_t] and the mixture head,
 * plus the reward and done heads) and of the linear controller
 * a_t = W_c [z_t, h_t] + b_c (Sec. 3.4).  Copies and packs the weights; the
 * handle owns that device memory until wm_destroy.  Returns
 * WM_ERR_INVALID_ARG for bad sizes (any dim <= 0, K > 32, negative
 * temperatures) or NULL weights (w_rt and w_mem are needed with
 * WM_REWARD_SHAPED only). */
wm_status wm_create(const wm_config *cfg, const wm_weights *weights, wm_handle **out);

/* Runs T dream steps (a1..a8 above) for B independent episodes, asynchronously
 * on cuda_stream (a cudaStream_t; NULL = legacy default stream).  Episode b is
 * keyed to Philox as episode_offset + b and its steps as t0 + t, so a rollout
 * split over calls (resume: pass z_out[T], h_final, c_final, done[T-1]) or over
 * devices (shard: episode_offset) reproduces the unsplit one bit for bit.
 * B = 0 or T = 0 are valid (T = 0 only copies z0 to z_out[0]).
 *
 * Models whose episodes end (done_terminates or noop_terminates) with one
 * controller: the tensor-core family packs the live episodes into the first
 * rows before every step and computes only those; a frozen episode's outputs
 * are written without computing it.  Once every episode has ended the call
 * issues no further step.  To notice that in time it keeps at most 4 steps in
 * flight, so it returns when its last step has been issued, a few steps before
 * the device has finished (not when per-step staging of host arrays or stream
 * capture is in use: then every step is issued).  Results are the same bit for
 * bit however far the host got. */
wm_status wm_rollout(wm_handle *h, int B, int T, unsigned long long episode_offset,
                     unsigned int t0, const wm_rollout_io *io, void *cuda_stream);

/* Teacher-forced scoring (a9) of a flat-action model: runs the LSTM over the given latents and
 * actions from h = c = 0 and returns the per-sequence mixture NLL in nats.
 *   z_seq   [T+1,N,Z] latents; step t reads z_seq[t] and scores z_seq[t+1]
 *   actions [T,N]     in [0,A) or negative for no action row
 *   lengths [N]       in [0,T], or NULL = T: only steps t < lengths[n] count
 *                     (Sec. 3.3.1 padding); the recurrence still runs all T
 *   nll     [N]       output
 *   h_seq, c_seq [T,N,H], mdn_seq [T,N,M]: optional per-step outputs.
 * An action >= A or a length outside [0,T] is an argument error.  On host
 * arrays it is returned by this call (outputs untouched); on device arrays the
 * kernels find it, record WM_ERR_INVALID_ARG in the status word (returned by
 * the next wm_sync) and go on with the action taken as no action and the
 * length clamped to [0,T]. */
wm_status wm_mdn_nll(wm_handle *h, int N, int T, const float *z_seq, const int32_t *actions,
                     const int32_t *lengths, float *nll, float *h_seq, float *c_seq,
                     float *mdn_seq, void *cuda_stream);

/* Gradients of the world model's training loss.  Output arrays (device or host
 * memory, overwritten, fp32) in the canonical layouts of wm_weights. */
typedef struct {
    float *W_lstm;   /* [Z+A+H, 4H] required */
    float *b_lstm;   /* [4H]        required */
    float *W_mdn;    /* [H, 3KZ]    required */
    float *b_mdn;    /* [3KZ]       required */
} wm_grads;

/* The world model's training step (Sec. 3.3.2: the MDN-RNN is trained by
 * backpropagation on minibatches of rollouts; Sec. 4.7: its loss is the
 * mixture log-likelihood): the teacher-forced loss sum_n NLL_n of wm_mdn_nll
 * and its gradient with respect to W_lstm, b_lstm, W_mdn and b_mdn, by
 * backpropagation through time.  Inputs as wm_mdn_nll (flat-action models);
 * nll [N] is optional.  The reward, done, runtime, memory and value heads are
 * not in the loss.  On the bf16 path the operand rounding is treated as the
 * identity in the backward pass, and the backward's GEMM operands are bf16
 * (fp32 accumulation); on the fp32 path the backward's batched GEMMs are
 * fp32-accurate (cuBLAS's fp32 emulation on the tensor cores, each operand
 * split into three bf16 parts; plain fp32 where the library lacks it), the
 * recurrence's dH = dG_t W_h^T takes each operand as two bf16 parts and
 * accumulates the three products hi.hi + hi.lo + lo.hi in fp32 (each product
 * within 3 * 2^-16 of the fp32 one at worst), all for finite inputs and weights
 * (non-finite values are not propagated as IEEE arithmetic would), and the
 * forward is fp32-accurate (see Precision above).  The forward runs on the
 * kernel family wm_mdn_nll would pick; the batched GEMMs of the backward
 * (gate activations over all N*T rows, the heads' and the recurrent input
 * gradients, the weight gradients) are cuBLAS calls, the rest (the mixture
 * NLL's gradient, the cell's backward step, the action-row and bias sums) are
 * the library's kernels.  Deterministic: every reduction has a fixed order.
 * Returns WM_ERR_UNSUPPORTED for hierarchical models. */
wm_status wm_mdn_nll_backward(wm_handle *h, int N, int T, const float *z_seq, const int32_t *actions,
                              const int32_t *lengths, float *nll, const wm_grads *grads,
                              void *cuda_stream);

/* wm_rollout without any device allocation.  The paper has no counterpart:
 * this entry point exists for callers that cannot call cudaMalloc/cudaFree
 * while they run -- work issued during CUDA stream capture, real-time loops
 * where an allocation (and the device-wide synchronisation cudaFree implies)
 * would stall other work, or hosts whose GPU memory belongs entirely to
 * another allocator.  wm_rollout may grow its per-handle workspace (and stage
 * host arrays) on demand; this call never does.
 *
 * Same arguments, results and Philox keying as wm_rollout, always on the
 * stepwise kernel family.  Differences:
 *   - every array must be device or managed memory (host memory is rejected
 *     with WM_ERR_INVALID_ARG, since it would need staging buffers);
 *   - its scratch (gate and head buffers, h, c, frozen flags) is a fixed
 *     WM_NOALLOC_SCRATCH_BYTES array inside the library, which every GPU that
 *     loads the library holds until the process exits; a batch whose scratch
 *     would exceed it is rejected with WM_ERR_INVALID_ARG (at Z=32, A=128,
 *     H=256, K=5 that allows about 1950 episodes);
 *   - all calls share that array, so calls that overlap on the GPU (on any
 *     handle of the process, on different streams) race and corrupt each
 *     other: serialise them.  Each call re-initialises the state it needs;
 *   - the first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress, with the handle's device made current) and
 *     caches it, so make that first call before any stream capture begins.
 * The handle itself (wm_create) still holds the packed weights allocated at
 * set-up time. */
#define WM_NOALLOC_SCRATCH_BYTES (16u << 20)
wm_status wm_rollout_noalloc(wm_handle *h, int B, int T, unsigned long long episode_offset,
                             unsigned int t0, const wm_rollout_io *io, void *cuda_stream);

/* Replaces the controller with a population of P candidates (Sec. 3.4: CMA-ES
 * searches over the controller's weights, evaluating each candidate by its
 * return in the world model).  Global episode e = episode_offset + b acts with
 * candidate (e / E) mod P, so a generation of P candidates x E episodes is one
 * wm_rollout of P*E episodes.  W_ctrl [P, Z+H, A] and b_ctrl [P, A] are host
 * fp32 arrays in the layout of wm_weights, copied and packed (P = 1 restores a
 * single controller).  The tensor-core family takes a population when E and
 * the call's episode_offset are multiples of 256 (its row tiles then belong to
 * one candidate); AUTO picks another family otherwise, and the fused family
 * takes none.  WM_ERR_INVALID_ARG for P < 1, E < 1 or NULL arrays. */
wm_status wm_set_controllers(wm_handle *h, int P, int E, const float *W_ctrl, const float *b_ctrl);

/* Discounted returns of a rollout (the objective of Sec. 3.1, discount gamma):
 * G_t = r_t + gamma G_{t+1}, from G_T = bootstrap[b] (NULL: 0); with
 * stop_at_done a step with done = 1 ends the sum (G_t = r_t).
 *   rewards, done [T,B] as wm_rollout wrote them; returns [T,B] out;
 *   fitness [P] optional out: each candidate's mean G_0 over this call's
 *   episodes (candidate of episode b: (episode_offset + b) / E mod P, the
 *   handle's population), summed in episode order (deterministic).
 * Arrays may be host or device memory, as for wm_rollout. */
wm_status wm_returns(wm_handle *h, int B, int T, unsigned long long episode_offset, float gamma,
                     int stop_at_done, const float *rewards, const uint8_t *done,
                     const float *bootstrap, float *returns, float *fitness, void *cuda_stream);

/* Failure injection for tests of the timeout path.  The paper has no
 * counterpart: every wait inside the fused and tensor-core kernels is bounded,
 * and this lets a test make one of them run out without faulting or hanging the
 * GPU.  With polls > 0, the next wm_rollout or wm_mdn_nll call that runs the
 * fused or the tensor-core family makes its first kernel launch wait, before
 * that kernel issues any MMA or copy, on a barrier that nothing completes, for
 * at most `polls` polls.  The wait then gives up the way a real bounded wait
 * does: the kernel records WM_ERR_TIMEOUT in the status word, skips its work and
 * frees what it holds, and the next wm_sync returns WM_ERR_TIMEOUT (and clears
 * it).  The outputs of that call are undefined; later calls are unaffected.
 * One shot: the call that consumes the setting clears it, and polls = 0 clears
 * it without a call.  The stepwise family has no waits and ignores it. */
wm_status wm_inject_wait_timeout(wm_handle *h, unsigned int polls);

/* Synchronises the device and returns the first device-side error since the
 * last wm_sync (WM_ERR_TIMEOUT if a bounded wait gave up), then clears it. */
wm_status wm_sync(wm_handle *h);

/* Message for the last failing call on h (never NULL; "" if none). */
const char *wm_last_error(const wm_handle *h);

/* Kernel family the last wm_rollout / wm_mdn_nll call ran (WM_PATH_*). */
int wm_last_path(const wm_handle *h);

/* Number of kernels the last wm_rollout / wm_mdn_nll call launched (staging
 * copies not counted). */
int wm_last_launches(const wm_handle *h);

/* Per-kernel timing.  The paper has no counterpart: this is instrumentation
 * that splits a call's device time by kernel.  While timing is enabled, every
 * kernel the handle launches is bracketed by two CUDA events recorded on the
 * call's stream (no synchronisation is added).  wm_kernel_time waits for the
 * events recorded so far, folds their elapsed times into per-class totals and
 * returns the totals (milliseconds, launches) since timing was last enabled.
 * Calls made during CUDA stream capture must not be timed. */
enum {
    WM_KERNEL_STEP_GEMM = 0,    /* stepwise: gate / controller and head GEMMs     */
    WM_KERNEL_STEP_CELL = 1,    /* stepwise: action selection and LSTM cell       */
    WM_KERNEL_STEP_SAMPLE = 2,  /* stepwise: mixture sampling or NLL              */
    WM_KERNEL_FUSED = 3,        /* fused: the single rollout / scoring kernel      */
    WM_KERNEL_TC_CTRL = 4,      /* tensor: controller GEMM with action selection   */
    WM_KERNEL_TC_GATES = 5,     /* tensor: gate GEMM with the LSTM cell            */
    WM_KERNEL_TC_HEADS = 6,     /* tensor: head GEMM with sampling or NLL          */
    WM_KERNEL_AUX = 7,          /* state set-up, finishing copies, reductions      */
    WM_KERNEL_BW = 8,           /* training step: the library's backward kernels    */
    WM_KERNEL_BW_GEMM = 9,      /* training step: its cuBLAS GEMMs                  */
    WM_KERNEL_FUSED_SMALL = 10, /* fused, small-batch member: the single kernel     */
    WM_KERNEL_CLASSES = 11
};

/* enable != 0 turns timing on and clears the totals; 0 turns it off (events
 * already recorded can still be read). */
wm_status wm_set_timing(wm_handle *h, int enable);

/* Totals of one class (WM_KERNEL_*) since timing was enabled.  Either output
 * may be NULL.  WM_ERR_CUDA if an event cannot be read. */
wm_status wm_kernel_time(wm_handle *h, int kernel_class, double *total_ms, long long *launches);

/* Frees everything the handle owns.  NULL is a no-op. */
void wm_destroy(wm_handle *h);

#ifdef __cplusplus
}
#endif
#endif /* WM_H */
