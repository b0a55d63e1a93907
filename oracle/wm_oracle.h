/*
 * wm_oracle.h -- plain, slow, obviously-correct CPU oracle for the RLFlow
 * world-model "dream" path (MDN-RNN world model + linear controller).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and
 * bench.py's cpu_baseline / reference arm may load or call this code.  The
 * CUDA product path shares no code, header, table or helper with it.
 *
 * Arithmetic is fp64 throughout.  Where a floating-point value decides an
 * integer (controller argmax, mixture-component choice, done threshold) the
 * deciding value is first rounded to fp32, the precision the kernels decide
 * in.  A "bf16" mode emulates the bf16 operand rounding points of the GPU
 * bf16 path (weights, and the GEMM A-operands [z_t; h_t] and h_{t+1}).
 *
 * Paper anchors (RLFlow, SIGMOD'22): MDN-RNN models P(z_{t+1}|a_t,z_t,h_t)
 * (Sec. 3.3.2); mixture weights = softmax(logits / tau) (Sec. 3.3.2, the
 * temperature equation); linear controller a_t = W_c[z_t,h_t] + b_c
 * (Sec. 3.4); invalid-action masking of the logits (Sec. 3.1.3); padding and
 * masking of sequences (Sec. 3.3.1); world-model log-likelihood loss
 * (Sec. 4.7).
 */
#ifndef WM_ORACLE_H
#define WM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
    int z_dim, a_dim, h_dim, k_mix;
    int bf16;             /* 1: emulate bf16 operand rounding              */
    double mdn_tau;       /* mixture temperature, >= 0                       */
    int sigma_sqrt_tau;   /* 1: sigma scaled by sqrt(tau)                    */
    int ctrl_sample;      /* 0: masked argmax, 1: tempered softmax sample    */
    double ctrl_tau;      /* controller temperature (sample mode), >= 0      */
    int done_terminates;  /* done head (logit > 0) freezes the episode       */
    int noop_terminates;  /* action a_dim-1 (NO-OP) freezes the episode      */
    uint64_t seed;        /* Philox key                                      */
    int nthreads;         /* OpenMP threads over episodes (<=0: 1)           */
    /* reward (Sec. 3.1.4): 0 = the linear reward head; 1 = Eq. 2 on the
     * predicted runtime and memory-access heads, alpha (RT_{t-1} - RT_t) +
     * beta (M_{t-1} - M_t) for a valid action, invalid_reward otherwise
     * (Eq. 1 is alpha = 1, beta = 0)                                       */
    int reward_mode;
    double reward_alpha, reward_beta, invalid_reward;
    /* controller population (Sec. 3.4, CMA-ES over controller weights):
     * pop_size P candidates; global episode e acts with candidate
     * (e / pop_group) mod P.  P <= 1: one controller.                     */
    int pop_size, pop_group;
    /* value head V(h') = w_val . h' + b_val (1 = on)                        */
    int value_head;
    /* hierarchical action (Sec. 3.1.3): n_xfers = NX > 0 splits the a_dim
     * controller outputs into NX xfer logits (the last one, NX - 1, is the
     * NO-OP) and L = a_dim - NX location logits; the xfer is chosen under the
     * step's xfer mask (bits 0..NX-1 of the mask words), then the location
     * under that xfer's location mask; the LSTM input is onehot(xfer) ||
     * onehot(location) (action rows xfer and NX + location).  0 = flat.     */
    int n_xfers;
    /* 1: carry the recurrent state, and take the fp32 path's GEMM operands,
     * in fp64 instead of rounding them to fp32 (a smooth model for the
     * finite-difference and autograd pins of the gradients only)           */
    int state64;
} orc_cfg;

typedef struct {
    const float *W_lstm;  /* [Z+A+H, 4H]  rows z | a | h, cols i | f | g | o  */
    const float *b_lstm;  /* [4H]                                            */
    const float *W_mdn;   /* [H, 3KZ]  cols logit | mu | logsigma, d*K+k      */
    const float *b_mdn;   /* [3KZ]                                           */
    const float *w_rew;   /* [H]                                             */
    float b_rew;
    const float *w_done;  /* [H]                                             */
    float b_done;
    const float *W_ctrl;  /* [P, Z+H, A]  (P = max(pop_size, 1))             */
    const float *b_ctrl;  /* [P, A]                                          */
    const float *w_rt;    /* [H] runtime head (reward_mode 1), else NULL     */
    float b_rt;
    const float *w_mem;   /* [H] memory-access head (reward_mode 1)          */
    float b_mem;
    const float *w_val;   /* [H] value head (value_head 1), else NULL        */
    float b_val;
} orc_weights;

/* Inputs and outputs of the optional parts of a rollout (NULL = not used).
 * Shaped reward (reward_mode 1): rt0, mem0 [B] are the predicted runtime and
 * memory accesses of each episode's current graph (required); rt_seq,
 * mem_seq [T,B] receive the predictions after each step. */
typedef struct {
    const float *rt0, *mem0;
    float *rt_seq, *mem_seq;
    /* logp_seq [T,B]: log pi(a_t | z_t, h_t) of the action taken under the
     * controller's masked softmax at temperature ctrl_tau (0 when ctrl_tau
     * is 0 or no action was valid); value_seq [T,B]: V(h_{t+1}) (value_head). */
    float *logp_seq, *value_seq;
    /* hierarchical action: loc_mask [T,B,NX,ceil(L/32)] (NULL = all valid);
     * loc_seq [T,B] the location taken (-1: none, e.g. NO-OP); loc_margin
     * [T,B] the location decision's margin (infinite when there is none). */
    const uint32_t *loc_mask;
    int32_t *loc_seq;
    float *loc_margin;
    const int32_t *loc_use;   /* orc_step only: [B] location override (< -1: none) */
} orc_ext;

/* ---- building blocks (exported so tests can pin each one) ---------------- */
void     orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
double   orc_uniform(uint32_t x);
void     orc_box_muller(uint32_t x1, uint32_t x2, double *e0, double *e1);
void     orc_draw(uint64_t seed, uint64_t episode, uint32_t step, uint32_t purpose,
                  uint32_t block, uint32_t out[4]);
float    orc_bf16(float x);
void     orc_lstm_cell(int H, const double *gates, const double *c_in,
                       double *c_out, double *h_out);
double   orc_mixture_nll_1d(int K, const double *logits, const double *mu,
                            const double *logsig, double x);
int      orc_sample_dim(int K, double tau, int sigma_sqrt_tau, const float *logits,
                        const double *mu, const double *logsig, double u, double eps,
                        double *z, double *margin);
int      orc_select_action(int A, const float *logits, const uint32_t *mask_words,
                           int ctrl_sample, double ctrl_tau, double u, double *margin);

/* ---- the two operations of the path --------------------------------------- */
int orc_rollout(const orc_cfg *cfg, const orc_weights *w, int B, int T,
                uint64_t episode_offset, uint32_t t0,
                const float *z0, const float *h0, const float *c0,
                const uint8_t *done0, const uint32_t *mask,
                float *z_out, int32_t *actions, float *rewards, uint8_t *done,
                float *h_final, float *c_final,
                float *h_seq, float *c_seq, float *mdn_seq, uint8_t *comp_seq,
                float *ctrl_margin, float *comp_margin, float *done_margin,
                const orc_ext *ext);

/* One dream step for B episodes started from a given state (z, h, c, frozen):
 * the step orc_rollout takes, for step-anchored comparisons.  episode[b] is the
 * global Philox episode index of row b, step the global step index; mask is
 * [B, ceil(A/32)] or NULL.  Optional overrides (NULL = none): a_use [B] is the
 * action row the LSTM takes (entries < -1: none), h_use [B,H] the h' the heads
 * read, k_use [B,Z] the components z_{t+1} is drawn from.  The outputs are the
 * oracle's own decisions and margins and the values downstream of the
 * overrides: action, ctrl_margin, reward, done, done_margin [B]; h_out, c_out
 * [B,H]; mdn_out [B,3KZ]; comp, comp_margin, z_next [B,Z].  ext (or NULL)
 * carries the optional parts for this one step, with T = 1: ext->rt0/mem0
 * are the predictions entering the step, ext->rt_seq/mem_seq [B] receive the
 * step's. */
int orc_step(const orc_cfg *cfg, const orc_weights *w, int B, const uint64_t *episode,
             uint32_t step, const float *z, const float *h, const float *c,
             const uint8_t *frozen, const uint32_t *mask,
             const int32_t *a_use, const float *h_use, const uint8_t *k_use,
             int32_t *action, float *ctrl_margin, float *h_out, float *c_out, float *mdn_out,
             float *reward, uint8_t *done, float *done_margin, uint8_t *comp,
             float *comp_margin, float *z_next, const orc_ext *ext);

/* Discounted returns of B rollouts of T steps (Sec. 3.1 objective):
 * G_t = r_t + gamma G_{t+1}, from G_T = bootstrap[b] (NULL: 0).  With
 * stop_at_done, a step with done_t = 1 ends the sum (G_t = r_t).  returns
 * [T,B] out.  If fitness is non-NULL, fitness[g] (g < P) is the mean G_0
 * over the call's episodes of candidate g ((episode_offset + b) / E mod P),
 * 0 for a candidate with no episode. */
int orc_returns(int B, int T, double gamma, int stop_at_done, const float *rewards,
                const uint8_t *done, const float *bootstrap, float *returns,
                uint64_t episode_offset, int P, int E, double *fitness);

int orc_mdn_nll(const orc_cfg *cfg, const orc_weights *w, int N, int T,
                const float *z_seq, const int32_t *actions, const int32_t *lengths,
                double *nll, float *h_seq, float *c_seq, float *mdn_seq);

/* Gradient of the teacher-forced loss sum_n NLL_n (the world model's training
 * objective, Sec. 4.7; trained by backpropagation, Sec. 3.3.2) with respect to
 * the MDN-RNN's parameters, by backpropagation through time: the mixture
 * NLL's gradient at each counted step, back through the heads and the LSTM.
 * Same inputs as orc_mdn_nll (flat actions).  Outputs (overwritten, fp64):
 * nll [N] (may be NULL), gW_lstm [Z+A+H, 4H], gb_lstm [4H], gW_mdn [H, 3KZ],
 * gb_mdn [3KZ].  With bf16 operand rounding (cfg->bf16) the rounding is
 * treated as the identity in the backward pass. */
int orc_mdn_nll_grad(const orc_cfg *cfg, const orc_weights *w, int N, int T,
                     const float *z_seq, const int32_t *actions, const int32_t *lengths,
                     double *nll, double *gW_lstm, double *gb_lstm, double *gW_mdn,
                     double *gb_mdn);

#ifdef __cplusplus
}
#endif
#endif
