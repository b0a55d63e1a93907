/*
 * wm_oracle.c -- plain CPU oracle for the RLFlow world-model dream path.
 *
 * TEST INFRASTRUCTURE ONLY (see wm_oracle.h).  Straight loops, fp64, no
 * blocking, fusion or reordering beyond the step order below:
 *
 *   for t = 0..T-1, for every episode independently:
 *     a1  controller logits   l = W_c^T [z_t; h_t] + b_c           (Sec. 3.4)
 *     a2  mask + select       invalid logits -> -inf; argmax or a
 *                             tempered-softmax draw                 (Sec. 3.1.3)
 *     a3  LSTM gates          G = W^T [z_t; onehot(a_t); h_t] + b   (Sec. 3.3.2)
 *     a4  cell update         c' = f c + i g, h' = o tanh(c')
 *     a5  heads               MDN params, reward, done logit on h'  (Sec. 3.3.2, 4.7)
 *     a6  mixture weights     log softmax(logit / tau)              (temperature eq.)
 *     a7  sample z_{t+1}      component by inverse CDF, then mu + sigma*eps
 *     a8  done / freeze       done = logit > 0; frozen episodes stay put
 *   a9  teacher-forced NLL  sum_t sum_d -log sum_k pi N(z_{t+1,d}; mu, sigma)  (Sec. 4.7)
 *
 * Readings where the paper is silent (all fixed here, mirrored by the kernels):
 *   - the state (z, h, c) is carried in fp32 between steps; inside a step the
 *     oracle computes in fp64;
 *   - per-latent-dim 1-D mixtures, K logits per dim (3KZ head outputs);
 *   - gate column order i,f,g,o, no implicit forget bias;
 *   - masked logits become -inf (the paper "zeroes" them, which could not keep
 *     a zeroed logit from winning an argmax);
 *   - ties: lowest index; inverse CDF: first k with u < C_k, else K-1;
 *   - tau = 0: argmax component, z = mu (the paper's "deterministic" limit);
 *   - reward / done are linear heads on h_{t+1}; done = (logit > 0).
 *
 * Random numbers: Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11),
 * key = (seed lo, seed hi), counter = (episode lo, step, purpose<<24 | block,
 * episode hi).  Purpose 0: component uniforms (4 dims per block); purpose 1:
 * normals by Box-Muller (4 dims per block, words (0,1) and (2,3) are pairs);
 * purpose 2: the controller's sampling uniform (word 0 of block 0).
 */
#include "wm_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#ifndef M_PI
#define M_PI 3.14159265358979323846
#endif

/* ------------------------------------------------------------------------- */
/* Philox-4x32-10, written from the round function of Salmon et al. (SC'11): */
/* two 32x32->64 multiplies per round on words 0 and 2, the high halves are   */
/* xored with the other words and the round key, the key is bumped by the     */
/* Weyl constants between rounds.                                             */
/* ------------------------------------------------------------------------- */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t n0 = hi1 ^ c1 ^ k0;
        uint32_t n1 = lo1;
        uint32_t n2 = hi0 ^ c3 ^ k1;
        uint32_t n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* u in [0,1): the top 24 bits scaled by 2^-24 (exact in fp32 and fp64). */
double orc_uniform(uint32_t x)
{
    return (double)(x >> 8) * (1.0 / 16777216.0);
}

/* Box-Muller (1958): r = sqrt(-2 ln(1-u1)), theta = 2 pi u2. */
void orc_box_muller(uint32_t x1, uint32_t x2, double *e0, double *e1)
{
    double u1 = orc_uniform(x1), u2 = orc_uniform(x2);
    double r = sqrt(-2.0 * log(1.0 - u1));
    double th = 2.0 * M_PI * u2;
    *e0 = r * cos(th);
    *e1 = r * sin(th);
}

void orc_draw(uint64_t seed, uint64_t episode, uint32_t step, uint32_t purpose,
              uint32_t block, uint32_t out[4])
{
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t ctr[4] = {(uint32_t)episode, step, (purpose << 24) | block,
                       (uint32_t)(episode >> 32)};
    orc_philox4x32_10(ctr, key, out);
}

/* fp32 -> bf16 round-to-nearest-even, returned widened to fp32. */
float orc_bf16(float x)
{
    uint32_t u;
    memcpy(&u, &x, 4);
    uint32_t r;
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu) != 0u) {
        r = 0x7FC00000u;                          /* canonical quiet NaN */
    } else {
        uint32_t lsb = (u >> 16) & 1u;
        r = ((u + 0x7FFFu + lsb) >> 16) << 16;   /* ties go to even */
    }
    float y;
    memcpy(&y, &r, 4);
    return y;
}

static double sigmoid(double v) { return 1.0 / (1.0 + exp(-v)); }

/* a4: gates = [i | f | g | o] pre-activations, each H long. */
void orc_lstm_cell(int H, const double *gates, const double *c_in,
                   double *c_out, double *h_out)
{
    for (int u = 0; u < H; ++u) {
        double ig = sigmoid(gates[u]);
        double fg = sigmoid(gates[H + u]);
        double gg = tanh(gates[2 * H + u]);
        double og = sigmoid(gates[3 * H + u]);
        double c = fg * c_in[u] + ig * gg;
        c_out[u] = c;
        h_out[u] = og * tanh(c);
    }
}

/* a9 for one latent dim: -log sum_k softmax(logits)_k N(x; mu_k, exp(logsig_k)). */
double orc_mixture_nll_1d(int K, const double *logits, const double *mu,
                          const double *logsig, double x)
{
    double lmax = -INFINITY;
    for (int k = 0; k < K; ++k) if (logits[k] > lmax) lmax = logits[k];
    double s = 0.0;
    for (int k = 0; k < K; ++k) s += exp(logits[k] - lmax);
    double logz = lmax + log(s);
    double terms[64];
    double tmax = -INFINITY;
    for (int k = 0; k < K; ++k) {
        double zsc = (x - mu[k]) * exp(-logsig[k]);
        double lp = (logits[k] - logz) - 0.5 * zsc * zsc - logsig[k] - 0.5 * log(2.0 * M_PI);
        terms[k] = lp;
        if (lp > tmax) tmax = lp;
    }
    double acc = 0.0;
    for (int k = 0; k < K; ++k) acc += exp(terms[k] - tmax);
    return -(tmax + log(acc));
}

/*
 * a6 + a7 for one latent dim.  logits are the fp32-rounded head outputs.
 * tau > 0: pi = softmax(logit / tau), k = first index with u < C_k (else K-1),
 *          z = mu_k + sigma_k * s * eps with s = sqrt(tau) if sigma_sqrt_tau.
 *          margin = min_k<K-1 |u - C_k|.
 * tau = 0: k = argmax logit (lowest index), z = mu_k; margin = top-2 gap.
 * Returns k.
 */
int orc_sample_dim(int K, double tau, int sigma_sqrt_tau, const float *logits,
                   const double *mu, const double *logsig, double u, double eps,
                   double *z, double *margin)
{
    if (tau <= 0.0) {
        int best = 0;
        for (int k = 1; k < K; ++k) if (logits[k] > logits[best]) best = k;
        double gap = INFINITY;
        for (int k = 0; k < K; ++k)
            if (k != best && (double)logits[best] - (double)logits[k] < gap)
                gap = (double)logits[best] - (double)logits[k];
        *z = mu[best];
        *margin = gap;
        return best;
    }
    double lmax = -INFINITY;
    for (int k = 0; k < K; ++k) if ((double)logits[k] / tau > lmax) lmax = (double)logits[k] / tau;
    double p[64], s = 0.0;
    for (int k = 0; k < K; ++k) { p[k] = exp((double)logits[k] / tau - lmax); s += p[k]; }
    int chosen = K - 1;
    double cum = 0.0, mg = INFINITY;
    for (int k = 0; k < K; ++k) {
        cum += p[k] / s;
        if (k < K - 1) {
            double d = fabs(u - cum);
            if (d < mg) mg = d;
        }
        if (chosen == K - 1 && k < K - 1 && u < cum) chosen = k;
    }
    double scale = sigma_sqrt_tau ? sqrt(tau) : 1.0;
    *z = mu[chosen] + exp(logsig[chosen]) * scale * eps;
    *margin = mg;
    return chosen;
}

static int bit_set(const uint32_t *words, int j)
{
    return (int)((words[j >> 5] >> (j & 31)) & 1u);
}

/*
 * a2: masked action choice.  mask_words == NULL means every action is valid.
 * argmax mode (ctrl_sample == 0 or ctrl_tau == 0): lowest index among the
 * valid maxima; margin = top-2 gap among valid logits.
 * sample mode: w_j = exp((l_j - l_max)/tau) on valid j, S = sum w, pick the
 * first valid j with u*S < cumsum_j (else the last valid one);
 * margin = min_j |u*S - cumsum_j| / S.
 * Returns -1 when no action is valid.
 */
int orc_select_action(int A, const float *logits, const uint32_t *mask_words,
                      int ctrl_sample, double ctrl_tau, double u, double *margin)
{
    int nvalid = 0, best = -1, last = -1;
    for (int j = 0; j < A; ++j) {
        if (mask_words && !bit_set(mask_words, j)) continue;
        ++nvalid;
        last = j;
        if (best < 0 || logits[j] > logits[best]) best = j;
    }
    *margin = INFINITY;
    if (nvalid == 0) return -1;
    if (!ctrl_sample || ctrl_tau <= 0.0) {
        double gap = INFINITY;
        for (int j = 0; j < A; ++j) {
            if (j == best || (mask_words && !bit_set(mask_words, j))) continue;
            double g = (double)logits[best] - (double)logits[j];
            if (g < gap) gap = g;
        }
        *margin = gap;
        return best;
    }
    double lmax = (double)logits[best];
    double S = 0.0;
    for (int j = 0; j < A; ++j) {
        if (mask_words && !bit_set(mask_words, j)) continue;
        S += exp(((double)logits[j] - lmax) / ctrl_tau);
    }
    double target = u * S, cum = 0.0, mg = INFINITY;
    int chosen = -1;
    for (int j = 0; j < A; ++j) {
        if (mask_words && !bit_set(mask_words, j)) continue;
        cum += exp(((double)logits[j] - lmax) / ctrl_tau);
        if (j != last) {
            double d = fabs(target - cum) / S;
            if (d < mg) mg = d;
        }
        if (chosen < 0 && target < cum) chosen = j;
    }
    if (chosen < 0) chosen = last;
    *margin = mg;
    return chosen;
}

/* ------------------------------------------------------------------------- */
/* Weights widened to fp64 (rounded to bf16 first in bf16 mode).             */
/* ------------------------------------------------------------------------- */
typedef struct {
    double *W_lstm, *b_lstm, *W_mdn, *b_mdn, *w_rew, *w_done, *W_ctrl, *b_ctrl, *w_rt, *w_mem,
        *w_val;
    double b_rew, b_done, b_rt, b_mem, b_val;
} wts64;

static double *widen(const float *src, size_t n, int round_bf16)
{
    double *dst = (double *)malloc(n * sizeof(double));
    if (!dst) return NULL;
    for (size_t i = 0; i < n; ++i) dst[i] = round_bf16 ? (double)orc_bf16(src[i]) : (double)src[i];
    return dst;
}

static void free_wts(wts64 *v)
{
    free(v->W_lstm); free(v->b_lstm); free(v->W_mdn); free(v->b_mdn);
    free(v->w_rew); free(v->w_done); free(v->W_ctrl); free(v->b_ctrl);
    free(v->w_rt); free(v->w_mem); free(v->w_val);
}

static int load_wts(const orc_cfg *cfg, const orc_weights *w, wts64 *v, int need_ctrl)
{
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, K = cfg->k_mix;
    const int rb = cfg->bf16;
    memset(v, 0, sizeof(*v));
    v->W_lstm = widen(w->W_lstm, (size_t)(Z + A + H) * 4 * H, rb);
    v->b_lstm = widen(w->b_lstm, (size_t)4 * H, 0);
    v->W_mdn = widen(w->W_mdn, (size_t)H * 3 * K * Z, rb);
    v->b_mdn = widen(w->b_mdn, (size_t)3 * K * Z, 0);
    v->w_rew = widen(w->w_rew, (size_t)H, rb);
    v->w_done = widen(w->w_done, (size_t)H, rb);
    v->b_rew = (double)w->b_rew;
    v->b_done = (double)w->b_done;
    if (need_ctrl) {
        const size_t P = cfg->pop_size > 1 ? (size_t)cfg->pop_size : 1;
        v->W_ctrl = widen(w->W_ctrl, P * (Z + H) * A, rb);
        v->b_ctrl = widen(w->b_ctrl, P * A, 0);
    }
    if (cfg->value_head) {
        if (!w->w_val) {
            free_wts(v);
            return -1;
        }
        v->w_val = widen(w->w_val, (size_t)H, rb);
        v->b_val = (double)w->b_val;
    }
    const int shaped = cfg->reward_mode == 1;
    if (shaped) {
        if (!w->w_rt || !w->w_mem) {
            free_wts(v);
            return -1;
        }
        v->w_rt = widen(w->w_rt, (size_t)H, rb);
        v->w_mem = widen(w->w_mem, (size_t)H, rb);
        v->b_rt = (double)w->b_rt;
        v->b_mem = (double)w->b_mem;
    }
    if (!v->W_lstm || !v->b_lstm || !v->W_mdn || !v->b_mdn || !v->w_rew || !v->w_done ||
        (need_ctrl && (!v->W_ctrl || !v->b_ctrl)) || (shaped && (!v->w_rt || !v->w_mem)) ||
        (cfg->value_head && !v->w_val)) {
        free_wts(v);
        return -1;
    }
    return 0;
}

/* GEMM A-operand: bf16-rounded through fp32 in bf16 mode, else fp32 value (unrounded
 * with state64, the smooth fp64 model the gradient pins differentiate). */
static double opnd(const orc_cfg *cfg, double v)
{
    float f = (float)v;
    if (cfg->bf16) return (double)orc_bf16(f);
    return cfg->state64 ? v : (double)f;
}

static int check_cfg(const orc_cfg *c)
{
    if (c->z_dim <= 0 || c->a_dim <= 0 || c->h_dim <= 0 || c->k_mix <= 0 || c->k_mix > 64) return -1;
    if (!(c->mdn_tau >= 0.0) || !(c->ctrl_tau >= 0.0)) return -1;
    if (c->reward_mode != 0 && c->reward_mode != 1) return -1;
    if (c->pop_size > 1 && c->pop_group < 1) return -1;
    if (c->n_xfers < 0 || c->n_xfers >= c->a_dim) return -1;
    return 0;
}

/* a3 + a4: one LSTM step for one episode.  x = [op(z); op(h)] of length Z+H; a, a2 are
 * the one-hot action rows taken (-1: none). */
static void lstm_step(const orc_cfg *cfg, const wts64 *v, const double *x, int a, int a2,
                      double *gates, double *c, double *h)
{
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, N4 = 4 * H;
    for (int n = 0; n < N4; ++n) {
        double g = v->b_lstm[n];
        for (int i = 0; i < Z; ++i) g += x[i] * v->W_lstm[(size_t)i * N4 + n];
        if (a >= 0) g += v->W_lstm[(size_t)(Z + a) * N4 + n];
        if (a2 >= 0) g += v->W_lstm[(size_t)(Z + a2) * N4 + n];
        for (int i = 0; i < H; ++i) g += x[Z + i] * v->W_lstm[(size_t)(Z + A + i) * N4 + n];
        gates[n] = g;
    }
    orc_lstm_cell(H, gates, c, c, h);
    /* the recurrent state is carried in fp32 between steps */
    if (!cfg->state64)
        for (int u = 0; u < H; ++u) {
            c[u] = (double)(float)c[u];
            h[u] = (double)(float)h[u];
        }
}

/* a5: MDN head outputs on y = op(h'). */
static void mdn_head(const orc_cfg *cfg, const wts64 *v, const double *y, double *mdn)
{
    const int H = cfg->h_dim, M = 3 * cfg->k_mix * cfg->z_dim;
    for (int m = 0; m < M; ++m) {
        double s = v->b_mdn[m];
        for (int i = 0; i < H; ++i) s += y[i] * v->W_mdn[(size_t)i * M + m];
        mdn[m] = s;
    }
}

#define INF_F ((float)INFINITY)

/* Per-episode work buffers of one step. */
typedef struct {
    double *x, *g, *y, *mdn, *znew;
    float *lg;
} step_buf;

static int buf_alloc(const orc_cfg *cfg, step_buf *sb)
{
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, K = cfg->k_mix;
    sb->x = malloc(sizeof(double) * (Z + H));
    sb->g = malloc(sizeof(double) * 4 * H);
    sb->y = malloc(sizeof(double) * H);
    sb->mdn = malloc(sizeof(double) * 3 * K * Z);
    sb->znew = malloc(sizeof(double) * Z);
    sb->lg = malloc(sizeof(float) * (A > K ? A : K));
    return (sb->x && sb->g && sb->y && sb->mdn && sb->znew && sb->lg) ? 0 : -1;
}

static void buf_free(step_buf *sb)
{
    free(sb->x); free(sb->g); free(sb->y); free(sb->mdn); free(sb->znew); free(sb->lg);
}

/*
 * One dream step (a1..a8) of one live episode e at global step s.  The state
 * z [Z], h [H], c [H] enters as fp32 values held in doubles and leaves as
 * (z_{t+1}, h', c'), again fp32 values.  mw: the step's mask words or NULL.
 *
 * Three optional overrides serve step-anchored checks, where the step is
 * replayed with another implementation's decisions so that every later value
 * stays comparable.  The oracle always reports its own decisions and margins;
 * an override only replaces what flows downstream of a decision:
 *   a_use (>= -1, or -2 for none) is the action row the LSTM takes (a3);
 *   h_use (or NULL) is the h' the heads read (a5..a7);
 *   k_use (or NULL) gives the component each dim's z_{t+1} is drawn from (a7).
 * The done flag is formed from the action actually taken.  With the shaped
 * reward (reward_mode 1) rt, mem hold the predicted runtime and memory
 * accesses entering the step (fp32 values) and leave with the step's; the
 * reward is Eq. 2 of Sec. 3.1.4 on them when the action taken is valid (a
 * row was taken, a >= 0), the invalid reward otherwise.  Returns 1 if the
 * episode freezes after this step (a8).
 */
static int step_episode(const orc_cfg *cfg, const wts64 *v, step_buf *sb, uint64_t e,
                        uint32_t s, double *z, double *h, double *c, double *rt, double *mem,
                        const uint32_t *mw, int a_use, const float *h_use, const uint8_t *k_use,
                        int32_t *action, float *ctrl_margin, float *reward, uint8_t *done,
                        float *done_margin, float *mdn_out, uint8_t *comp, float *comp_margin,
                        float *logp, float *value, const uint32_t *lmw, int l_use, int32_t *loc_out,
                        float *loc_margin)
{
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, K = cfg->k_mix;
    double *x = sb->x, *g = sb->g, *y = sb->y, *mdn = sb->mdn, *znew = sb->znew;
    float *lg = sb->lg;
    for (int i = 0; i < Z; ++i) x[i] = opnd(cfg, z[i]);
    for (int i = 0; i < H; ++i) x[Z + i] = opnd(cfg, h[i]);

    /* a1: controller logits of the episode's candidate, rounded to fp32 for the decision */
    const size_t cand = cfg->pop_size > 1 ? (size_t)((e / (uint64_t)cfg->pop_group) % (uint64_t)cfg->pop_size) : 0;
    const double *Wc = v->W_ctrl + cand * (size_t)(Z + H) * A, *bc = v->b_ctrl + cand * (size_t)A;
    for (int j = 0; j < A; ++j) {
        double l = bc[j];
        for (int i = 0; i < Z + H; ++i) l += x[i] * Wc[(size_t)i * A + j];
        lg[j] = (float)l;
    }
    /* a2: mask + select */
    double u_ctrl = 0.0;
    if (cfg->ctrl_sample && cfg->ctrl_tau > 0.0) {
        uint32_t r4[4];
        orc_draw(cfg->seed, e, s, 2u, 0u, r4);
        u_ctrl = orc_uniform(r4[0]);
    }
    double cm;
    /* hierarchical (Sec. 3.1.3): the xfer among the first NX logits, then the location
     * among the other L under the chosen xfer's location mask; flat: one choice of A */
    const int NX = cfg->n_xfers, hier = NX > 0, L = A - NX, WL = (L + 31) / 32;
    const int noop = hier ? NX - 1 : A - 1;
    int a = orc_select_action(hier ? NX : A, lg, mw, cfg->ctrl_sample, cfg->ctrl_tau, u_ctrl, &cm);
    int loc = -1;
    double lm = INFINITY;
    if (hier && a >= 0 && a != noop) {
        double u_loc = 0.0;
        if (cfg->ctrl_sample && cfg->ctrl_tau > 0.0) {
            uint32_t r4[4];
            orc_draw(cfg->seed, e, s, 2u, 0u, r4);
            u_loc = orc_uniform(r4[1]);
        }
        loc = orc_select_action(L, lg + NX, lmw ? lmw + (size_t)a * WL : NULL, cfg->ctrl_sample,
                                cfg->ctrl_tau, u_loc, &lm);
    }
    *action = a;
    if (ctrl_margin) *ctrl_margin = (float)cm;
    if (loc_out) *loc_out = loc;
    if (loc_margin) *loc_margin = (float)lm;
    if (a_use >= -1) a = a_use;
    if (hier && l_use >= -1) loc = l_use;
    if (hier && (a < 0 || a == noop)) loc = -1;
    /* log pi of the action taken, pi = softmax(l / ctrl_tau) over the valid actions; for a
     * hierarchical action log pi(xfer) + log pi(location | xfer) */
    if (logp) {
        double lp = 0.0;
        for (int part = 0; part < (hier ? 2 : 1); ++part) {
            const int choice = part ? loc : a;
            const int n0 = part ? NX : 0, n = hier ? (part ? L : NX) : A;
            const uint32_t *pm = part ? (lmw ? lmw + (size_t)a * WL : NULL) : mw;
            if (choice < 0 || !(cfg->ctrl_tau > 0.0)) continue;
            double lmax = -INFINITY, S = 0.0;
            for (int j = 0; j < n; ++j)
                if ((!pm || bit_set(pm, j)) && (double)lg[n0 + j] > lmax) lmax = (double)lg[n0 + j];
            for (int j = 0; j < n; ++j)
                if (!pm || bit_set(pm, j)) S += exp(((double)lg[n0 + j] - lmax) / cfg->ctrl_tau);
            lp += ((double)lg[n0 + choice] - lmax) / cfg->ctrl_tau - log(S);
        }
        *logp = (float)lp;
    }

    /* a3 + a4 */
    lstm_step(cfg, v, x, a, loc >= 0 ? NX + loc : -1, g, c, h);

    /* a5: heads on op(h') */
    for (int i = 0; i < H; ++i) y[i] = opnd(cfg, h_use ? (double)h_use[i] : h[i]);
    mdn_head(cfg, v, y, mdn);
    if (mdn_out) for (int m = 0; m < 3 * K * Z; ++m) mdn_out[m] = (float)mdn[m];
    double r = v->b_rew, dl = v->b_done;
    for (int i = 0; i < H; ++i) { r += y[i] * v->w_rew[i]; dl += y[i] * v->w_done[i]; }
    if (cfg->reward_mode == 1) {
        double rt_new = v->b_rt, mem_new = v->b_mem;
        for (int i = 0; i < H; ++i) { rt_new += y[i] * v->w_rt[i]; mem_new += y[i] * v->w_mem[i]; }
        rt_new = (double)(float)rt_new;   /* predictions are carried in fp32 */
        mem_new = (double)(float)mem_new;
        const int valid = a >= 0 && (!hier || a == noop || loc >= 0);
        r = valid ? cfg->reward_alpha * (*rt - rt_new) + cfg->reward_beta * (*mem - mem_new)
                  : cfg->invalid_reward;
        *rt = rt_new;
        *mem = mem_new;
    }
    *reward = (float)r;
    if (value) {
        double vv = v->b_val;
        for (int i = 0; i < H; ++i) vv += y[i] * v->w_val[i];
        *value = (float)vv;
    }
    float dlf = (float)dl;
    if (done_margin) *done_margin = fabsf(dlf);
    int is_noop = cfg->noop_terminates && a == noop;
    *done = (uint8_t)((dlf > 0.0f) || is_noop);

    /* a6 + a7: per-dim mixture sample */
    const double scale = cfg->sigma_sqrt_tau ? sqrt(cfg->mdn_tau) : 1.0;
    for (int d = 0; d < Z; ++d) {
        double u = 0.0, eps = 0.0;
        if (cfg->mdn_tau > 0.0) {
            uint32_t ru[4], rn[4];
            orc_draw(cfg->seed, e, s, 0u, (uint32_t)(d / 4), ru);
            u = orc_uniform(ru[d % 4]);
            orc_draw(cfg->seed, e, s, 1u, (uint32_t)(d / 4), rn);
            double e0, e1;
            int pair = (d % 4) / 2;
            orc_box_muller(rn[2 * pair], rn[2 * pair + 1], &e0, &e1);
            eps = (d % 2 == 0) ? e0 : e1;
        }
        for (int k = 0; k < K; ++k) lg[k] = (float)mdn[d * K + k];
        const double *mu = mdn + K * Z + d * K, *ls = mdn + 2 * K * Z + d * K;
        double zd, mg;
        int k = orc_sample_dim(K, cfg->mdn_tau, cfg->sigma_sqrt_tau, lg, mu, ls, u, eps, &zd, &mg);
        if (comp) comp[d] = (uint8_t)k;
        if (comp_margin) comp_margin[d] = (float)mg;
        if (k_use && k_use[d] != k) {
            int kf = k_use[d] < K ? k_use[d] : K - 1;
            zd = cfg->mdn_tau > 0.0 ? mu[kf] + exp(ls[kf]) * scale * eps : mu[kf];
        }
        znew[d] = zd;
    }
    for (int d = 0; d < Z; ++d) z[d] = (double)(float)znew[d];   /* fp32 latent state */
    /* a8 */
    return (cfg->done_terminates && dlf > 0.0f) || is_noop;
}

static int rollout_episode(const orc_cfg *cfg, const wts64 *v, int b, int B, int T,
                           uint64_t episode_offset, uint32_t t0,
                           const float *z0, const float *h0, const float *c0,
                           const uint8_t *done0, const uint32_t *mask,
                           float *z_out, int32_t *actions, float *rewards, uint8_t *done,
                           float *h_final, float *c_final,
                           float *h_seq, float *c_seq, float *mdn_seq, uint8_t *comp_seq,
                           float *ctrl_margin, float *comp_margin, float *done_margin,
                           const orc_ext *ext)
{
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, K = cfg->k_mix;
    const int M = 3 * K * Z, W = (A + 31) / 32;
    const uint64_t e = episode_offset + (uint64_t)b;
    const int shaped = cfg->reward_mode == 1;
    double rt = shaped ? (double)ext->rt0[b] : 0.0, mem = shaped ? (double)ext->mem0[b] : 0.0;
    double *z = malloc(sizeof(double) * Z), *h = malloc(sizeof(double) * H);
    double *c = malloc(sizeof(double) * H);
    step_buf sb;
    int ok = buf_alloc(cfg, &sb) == 0 && z && h && c;
    if (!ok) {
        free(z); free(h); free(c); buf_free(&sb);
        return -1;
    }
    for (int i = 0; i < Z; ++i) z[i] = z0[(size_t)b * Z + i];
    for (int i = 0; i < H; ++i) {
        h[i] = h0 ? h0[(size_t)b * H + i] : 0.0;
        c[i] = c0 ? c0[(size_t)b * H + i] : 0.0;
    }
    int frozen = done0 ? (done0[b] != 0) : 0;
    for (int i = 0; i < Z; ++i) z_out[(size_t)b * Z + i] = (float)z[i];

    for (int t = 0; t < T; ++t) {
        const uint32_t s = t0 + (uint32_t)t;
        const size_t tb = (size_t)t * B + b;
        float *lp_out = ext && ext->logp_seq ? ext->logp_seq + tb : NULL;
        float *v_out = ext && ext->value_seq && cfg->value_head ? ext->value_seq + tb : NULL;
        const int NX = cfg->n_xfers, WL = (A - NX + 31) / 32;
        const uint32_t *lmw = NX > 0 && ext && ext->loc_mask ? ext->loc_mask + tb * NX * WL : NULL;
        int32_t *loc_out = NX > 0 && ext && ext->loc_seq ? ext->loc_seq + tb : NULL;
        float *lm_out = NX > 0 && ext && ext->loc_margin ? ext->loc_margin + tb : NULL;
        if (frozen) {
            actions[tb] = -1; rewards[tb] = 0.0f; done[tb] = 1;
            if (lp_out) *lp_out = 0.0f;
            if (v_out) *v_out = 0.0f;
            if (loc_out) *loc_out = -1;
            if (lm_out) *lm_out = INF_F;
            if (mdn_seq) for (int m = 0; m < M; ++m) mdn_seq[tb * M + m] = 0.0f;
            if (comp_seq) for (int d = 0; d < Z; ++d) comp_seq[tb * Z + d] = 255;
            if (ctrl_margin) ctrl_margin[tb] = INF_F;
            if (done_margin) done_margin[tb] = INF_F;
            if (comp_margin) for (int d = 0; d < Z; ++d) comp_margin[tb * Z + d] = INF_F;
        } else {
            frozen = step_episode(cfg, v, &sb, e, s, z, h, c, &rt, &mem,
                                  mask ? mask + tb * W : NULL, -2, NULL, NULL, &actions[tb],
                                  ctrl_margin ? &ctrl_margin[tb] : NULL, &rewards[tb], &done[tb],
                                  done_margin ? &done_margin[tb] : NULL,
                                  mdn_seq ? mdn_seq + tb * M : NULL,
                                  comp_seq ? comp_seq + tb * Z : NULL,
                                  comp_margin ? comp_margin + tb * Z : NULL, lp_out, v_out, lmw, -2,
                                  loc_out, lm_out);
        }
        for (int i = 0; i < Z; ++i) z_out[((size_t)(t + 1) * B + b) * Z + i] = (float)z[i];
        if (h_seq) for (int i = 0; i < H; ++i) h_seq[tb * H + i] = (float)h[i];
        if (c_seq) for (int i = 0; i < H; ++i) c_seq[tb * H + i] = (float)c[i];
        if (shaped && ext->rt_seq) ext->rt_seq[tb] = (float)rt;
        if (shaped && ext->mem_seq) ext->mem_seq[tb] = (float)mem;
    }
    if (h_final) for (int i = 0; i < H; ++i) h_final[(size_t)b * H + i] = (float)h[i];
    if (c_final) for (int i = 0; i < H; ++i) c_final[(size_t)b * H + i] = (float)c[i];
    free(z); free(h); free(c); buf_free(&sb);
    return 0;
}

int orc_rollout(const orc_cfg *cfg, const orc_weights *w, int B, int T,
                uint64_t episode_offset, uint32_t t0,
                const float *z0, const float *h0, const float *c0,
                const uint8_t *done0, const uint32_t *mask,
                float *z_out, int32_t *actions, float *rewards, uint8_t *done,
                float *h_final, float *c_final,
                float *h_seq, float *c_seq, float *mdn_seq, uint8_t *comp_seq,
                float *ctrl_margin, float *comp_margin, float *done_margin,
                const orc_ext *ext)
{
    if (check_cfg(cfg) || B < 0 || T < 0 || !z0 || !z_out || !actions || !rewards || !done)
        return -1;
    if (cfg->reward_mode == 1 && (!ext || !ext->rt0 || !ext->mem0)) return -1;
    wts64 v;
    if (load_wts(cfg, w, &v, 1)) return -2;
    int bad = 0;
    int nt = cfg->nthreads > 0 ? cfg->nthreads : 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt) reduction(| : bad)
    for (int b = 0; b < B; ++b) {
        bad |= rollout_episode(cfg, &v, b, B, T, episode_offset, t0, z0, h0, c0, done0, mask,
                               z_out, actions, rewards, done, h_final, c_final,
                               h_seq, c_seq, mdn_seq, comp_seq,
                               ctrl_margin, comp_margin, done_margin, ext) ? 1 : 0;
    }
    free_wts(&v);
    return bad ? -2 : 0;
}

/*
 * One dream step for B episodes from a given state: the step of orc_rollout,
 * started from (z, h, c, frozen) instead of the previous step's results.
 * episode[b] is episode b's global Philox index, step the global step index.
 * The overrides a_use / h_use / k_use (see step_episode) may be NULL; a_use
 * entries below -1 mean "no override" for that episode.  A frozen episode
 * gives the frozen row (a = -1, r = 0, done = 1, state repeated, mdn 0,
 * components 255, infinite margins).
 */
int orc_step(const orc_cfg *cfg, const orc_weights *w, int B, const uint64_t *episode,
             uint32_t step, const float *z, const float *h, const float *c,
             const uint8_t *frozen, const uint32_t *mask,
             const int32_t *a_use, const float *h_use, const uint8_t *k_use,
             int32_t *action, float *ctrl_margin, float *h_out, float *c_out, float *mdn_out,
             float *reward, uint8_t *done, float *done_margin, uint8_t *comp,
             float *comp_margin, float *z_next, const orc_ext *ext)
{
    if (check_cfg(cfg) || B < 0 || !episode || !z || !h || !c || !action || !ctrl_margin ||
        !h_out || !c_out || !mdn_out || !reward || !done || !done_margin || !comp ||
        !comp_margin || !z_next)
        return -1;
    const int shaped = cfg->reward_mode == 1;
    if (shaped && (!ext || !ext->rt0 || !ext->mem0)) return -1;
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, K = cfg->k_mix;
    const int M = 3 * K * Z, W = (A + 31) / 32;
    wts64 v;
    if (load_wts(cfg, w, &v, 1)) return -2;
    int bad = 0;
    int nt = cfg->nthreads > 0 ? cfg->nthreads : 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt) reduction(| : bad)
    for (int b = 0; b < B; ++b) {
        double *zs = malloc(sizeof(double) * Z), *hs = malloc(sizeof(double) * H);
        double *cs = malloc(sizeof(double) * H);
        step_buf sb;
        if (buf_alloc(cfg, &sb) || !zs || !hs || !cs) {
            free(zs); free(hs); free(cs); buf_free(&sb);
            bad |= 1;
            continue;
        }
        for (int i = 0; i < Z; ++i) zs[i] = z[(size_t)b * Z + i];
        for (int i = 0; i < H; ++i) { hs[i] = h[(size_t)b * H + i]; cs[i] = c[(size_t)b * H + i]; }
        double rt = shaped ? (double)ext->rt0[b] : 0.0, mem = shaped ? (double)ext->mem0[b] : 0.0;
        float *lp_out = ext && ext->logp_seq ? ext->logp_seq + b : NULL;
        float *v_out = ext && ext->value_seq && cfg->value_head ? ext->value_seq + b : NULL;
        const int NX = cfg->n_xfers, WL = (A - NX + 31) / 32;
        const uint32_t *lmw = NX > 0 && ext && ext->loc_mask ? ext->loc_mask + (size_t)b * NX * WL : NULL;
        int32_t *loc_out = NX > 0 && ext && ext->loc_seq ? ext->loc_seq + b : NULL;
        float *lm_out = NX > 0 && ext && ext->loc_margin ? ext->loc_margin + b : NULL;
        const int l_use = NX > 0 && ext && ext->loc_use ? ext->loc_use[b] : -2;
        if (frozen && frozen[b]) {
            action[b] = -1; ctrl_margin[b] = INF_F; reward[b] = 0.0f; done[b] = 1;
            if (lp_out) *lp_out = 0.0f;
            if (v_out) *v_out = 0.0f;
            if (loc_out) *loc_out = -1;
            if (lm_out) *lm_out = INF_F;
            done_margin[b] = INF_F;
            for (int m = 0; m < M; ++m) mdn_out[(size_t)b * M + m] = 0.0f;
            for (int d = 0; d < Z; ++d) {
                comp[(size_t)b * Z + d] = 255;
                comp_margin[(size_t)b * Z + d] = INF_F;
            }
        } else {
            step_episode(cfg, &v, &sb, episode[b], step, zs, hs, cs, &rt, &mem,
                         mask ? mask + (size_t)b * W : NULL,
                         a_use ? a_use[b] : -2, h_use ? h_use + (size_t)b * H : NULL,
                         k_use ? k_use + (size_t)b * Z : NULL,
                         &action[b], &ctrl_margin[b], &reward[b], &done[b], &done_margin[b],
                         mdn_out + (size_t)b * M, comp + (size_t)b * Z,
                         comp_margin + (size_t)b * Z, lp_out, v_out, lmw, l_use, loc_out, lm_out);
        }
        for (int i = 0; i < Z; ++i) z_next[(size_t)b * Z + i] = (float)zs[i];
        for (int i = 0; i < H; ++i) {
            h_out[(size_t)b * H + i] = (float)hs[i];
            c_out[(size_t)b * H + i] = (float)cs[i];
        }
        if (shaped && ext->rt_seq) ext->rt_seq[b] = (float)rt;
        if (shaped && ext->mem_seq) ext->mem_seq[b] = (float)mem;
        free(zs); free(hs); free(cs); buf_free(&sb);
    }
    free_wts(&v);
    return bad ? -2 : 0;
}

int orc_returns(int B, int T, double gamma, int stop_at_done, const float *rewards,
                const uint8_t *done, const float *bootstrap, float *returns,
                uint64_t episode_offset, int P, int E, double *fitness)
{
    if (B < 0 || T < 0 || !rewards || !done || !returns) return -1;
    if (fitness && (P < 1 || E < 1)) return -1;
    double *g0 = malloc(sizeof(double) * (B > 0 ? B : 1));
    if (!g0) return -2;
    for (int b = 0; b < B; ++b) {
        double G = bootstrap ? (double)bootstrap[b] : 0.0;
        for (int t = T - 1; t >= 0; --t) {
            const size_t tb = (size_t)t * B + b;
            if (stop_at_done && done[tb]) G = 0.0;
            G = (double)rewards[tb] + gamma * G;
            returns[tb] = (float)G;
        }
        g0[b] = T > 0 ? G : (bootstrap ? (double)bootstrap[b] : 0.0);
    }
    if (fitness) {
        for (int g = 0; g < P; ++g) {
            double sum = 0.0;
            long n = 0;
            for (int b = 0; b < B; ++b) {
                const uint64_t e = episode_offset + (uint64_t)b;
                if ((int)((e / (uint64_t)E) % (uint64_t)P) != g) continue;
                sum += g0[b];
                ++n;
            }
            fitness[g] = n ? sum / (double)n : 0.0;
        }
    }
    free(g0);
    return 0;
}

static int nll_sequence(const orc_cfg *cfg, const wts64 *v, int n, int N, int T,
                        const float *z_seq, const int32_t *actions, int len,
                        double *nll, float *h_seq, float *c_seq, float *mdn_seq)
{
    const int Z = cfg->z_dim, H = cfg->h_dim, K = cfg->k_mix, M = 3 * K * Z;
    double *h = calloc((size_t)H, sizeof(double)), *c = calloc((size_t)H, sizeof(double));
    double *x = malloc(sizeof(double) * (Z + H)), *g = malloc(sizeof(double) * 4 * H);
    double *y = malloc(sizeof(double) * H), *mdn = malloc(sizeof(double) * M);
    if (!h || !c || !x || !g || !y || !mdn) {
        free(h); free(c); free(x); free(g); free(y); free(mdn);
        return -1;
    }
    double total = 0.0;
    for (int t = 0; t < T; ++t) {
        const size_t tn = (size_t)t * N + n;
        for (int i = 0; i < Z; ++i) x[i] = opnd(cfg, z_seq[tn * Z + i]);
        for (int i = 0; i < H; ++i) x[Z + i] = opnd(cfg, h[i]);
        lstm_step(cfg, v, x, actions[tn], -1, g, c, h);
        for (int i = 0; i < H; ++i) y[i] = opnd(cfg, h[i]);
        mdn_head(cfg, v, y, mdn);
        if (h_seq) for (int i = 0; i < H; ++i) h_seq[tn * H + i] = (float)h[i];
        if (c_seq) for (int i = 0; i < H; ++i) c_seq[tn * H + i] = (float)c[i];
        if (mdn_seq) for (int m = 0; m < M; ++m) mdn_seq[tn * M + m] = (float)mdn[m];
        if (t < len) {
            const float *target = z_seq + ((size_t)(t + 1) * N + n) * Z;
            for (int d = 0; d < Z; ++d)
                total += orc_mixture_nll_1d(K, mdn + d * K, mdn + K * Z + d * K,
                                            mdn + 2 * K * Z + d * K, (double)target[d]);
        }
    }
    nll[n] = total;
    free(h); free(c); free(x); free(g); free(y); free(mdn);
    return 0;
}

/* d NLL / d [logit | mu | log sigma] of one latent dim's mixture (K components) at
 * target x, with responsibilities g_k = pi_k N_k / sum_j pi_j N_j:
 *   d/d logit_k = pi_k - g_k,  d/d mu_k = -g_k (x - mu_k) / sigma_k^2,
 *   d/d log sigma_k = g_k (1 - ((x - mu_k) / sigma_k)^2).  Returns the NLL. */
static double mixture_nll_grad_1d(int K, const double *lg, const double *mu, const double *ls, double x,
                                  double *dlg, double *dmu, double *dls)
{
    double lmax = -INFINITY, s = 0.0, terms[64], tmax = -INFINITY, acc = 0.0;
    for (int k = 0; k < K; ++k) if (lg[k] > lmax) lmax = lg[k];
    for (int k = 0; k < K; ++k) s += exp(lg[k] - lmax);
    const double logz = lmax + log(s);
    for (int k = 0; k < K; ++k) {
        const double zs = (x - mu[k]) * exp(-ls[k]);
        terms[k] = (lg[k] - logz) - 0.5 * zs * zs - ls[k] - 0.5 * log(2.0 * M_PI);
        if (terms[k] > tmax) tmax = terms[k];
    }
    for (int k = 0; k < K; ++k) acc += exp(terms[k] - tmax);
    const double lse = tmax + log(acc);
    for (int k = 0; k < K; ++k) {
        const double pi = exp(lg[k] - logz), gam = exp(terms[k] - lse);
        const double zs = (x - mu[k]) * exp(-ls[k]);
        dlg[k] = pi - gam;
        dmu[k] = -gam * zs * exp(-ls[k]);
        dls[k] = gam * (1.0 - zs * zs);
    }
    return -lse;
}

/* BPTT of one sequence; gradients are added to the per-thread accumulators. */
static int grad_sequence(const orc_cfg *cfg, const wts64 *v, int n, int N, int T, const float *z_seq,
                         const int32_t *actions, int len, double *nll_out, double *gW, double *gb,
                         double *gWm, double *gbm)
{
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, K = cfg->k_mix, M = 3 * K * Z;
    const int KX = Z + H, N4 = 4 * H;
    /* forward, keeping every step's operands, gate activations, cell and head outputs */
    double *X = malloc(sizeof(double) * (size_t)T * KX), *act = malloc(sizeof(double) * (size_t)T * N4);
    double *C = malloc(sizeof(double) * (size_t)(T + 1) * H), *Y = malloc(sizeof(double) * (size_t)T * H);
    double *MD = malloc(sizeof(double) * (size_t)T * M), *h = calloc((size_t)H, sizeof(double));
    double *g = malloc(sizeof(double) * N4), *dmd = malloc(sizeof(double) * M);
    double *dh = malloc(sizeof(double) * H), *dhn = calloc((size_t)H, sizeof(double));
    double *dcn = calloc((size_t)H, sizeof(double)), *dG = malloc(sizeof(double) * N4);
    if (!X || !act || !C || !Y || !MD || !h || !g || !dmd || !dh || !dhn || !dcn || !dG) {
        free(X); free(act); free(C); free(Y); free(MD); free(h); free(g); free(dmd); free(dh);
        free(dhn); free(dcn); free(dG);
        return -1;
    }
    for (int u = 0; u < H; ++u) C[u] = 0.0;  /* c_0 */
    double total = 0.0;
    for (int t = 0; t < T; ++t) {
        const size_t tn = (size_t)t * N + n;
        double *x = X + (size_t)t * KX, *c = C + (size_t)(t + 1) * H;
        for (int i = 0; i < Z; ++i) x[i] = opnd(cfg, z_seq[tn * Z + i]);
        for (int i = 0; i < H; ++i) x[Z + i] = opnd(cfg, h[i]);
        for (int u = 0; u < H; ++u) c[u] = C[(size_t)t * H + u];
        lstm_step(cfg, v, x, actions[tn], -1, g, c, h);
        double *ac = act + (size_t)t * N4;
        for (int u = 0; u < H; ++u) {  /* i, f, g, o from the pre-activations */
            ac[u] = 1.0 / (1.0 + exp(-g[u]));
            ac[H + u] = 1.0 / (1.0 + exp(-g[H + u]));
            ac[2 * H + u] = tanh(g[2 * H + u]);
            ac[3 * H + u] = 1.0 / (1.0 + exp(-g[3 * H + u]));
        }
        double *y = Y + (size_t)t * H, *md = MD + (size_t)t * M;
        for (int i = 0; i < H; ++i) y[i] = opnd(cfg, h[i]);
        mdn_head(cfg, v, y, md);
    }
    /* backward through time */
    for (int t = T - 1; t >= 0; --t) {
        const size_t tn = (size_t)t * N + n;
        const double *md = MD + (size_t)t * M, *y = Y + (size_t)t * H, *x = X + (size_t)t * KX;
        const double *ac = act + (size_t)t * N4, *c = C + (size_t)(t + 1) * H, *cp = C + (size_t)t * H;
        for (int m = 0; m < M; ++m) dmd[m] = 0.0;
        if (t < len) {
            const float *target = z_seq + ((size_t)(t + 1) * N + n) * Z;
            for (int d = 0; d < Z; ++d)
                total += mixture_nll_grad_1d(K, md + d * K, md + K * Z + d * K, md + 2 * K * Z + d * K,
                                             (double)target[d], dmd + d * K, dmd + K * Z + d * K,
                                             dmd + 2 * K * Z + d * K);
        }
        /* heads: mdn = W_mdn^T y + b_mdn */
        for (int i = 0; i < H; ++i) {
            double s = 0.0;
            for (int m = 0; m < M; ++m) {
                gWm[(size_t)i * M + m] += y[i] * dmd[m];
                s += v->W_mdn[(size_t)i * M + m] * dmd[m];
            }
            dh[i] = s + dhn[i];
        }
        for (int m = 0; m < M; ++m) gbm[m] += dmd[m];
        /* cell: c = f c_prev + i g, h = o tanh(c) */
        for (int u = 0; u < H; ++u) {
            const double ig = ac[u], fg = ac[H + u], gg = ac[2 * H + u], og = ac[3 * H + u];
            const double tc = tanh(c[u]);
            const double dc = dh[u] * og * (1.0 - tc * tc) + dcn[u];
            dG[u] = dc * gg * ig * (1.0 - ig);
            dG[H + u] = dc * cp[u] * fg * (1.0 - fg);
            dG[2 * H + u] = dc * ig * (1.0 - gg * gg);
            dG[3 * H + u] = dh[u] * tc * og * (1.0 - og);
            dcn[u] = dc * fg;
        }
        /* gates: G = W^T [x_z; onehot(a); x_h] + b */
        const int a = actions[tn];
        for (int k = 0; k < N4; ++k) gb[k] += dG[k];
        for (int i = 0; i < Z; ++i)
            for (int k = 0; k < N4; ++k) gW[(size_t)i * N4 + k] += x[i] * dG[k];
        if (a >= 0)
            for (int k = 0; k < N4; ++k) gW[(size_t)(Z + a) * N4 + k] += dG[k];
        for (int i = 0; i < H; ++i) {
            double s = 0.0;
            for (int k = 0; k < N4; ++k) {
                gW[(size_t)(Z + A + i) * N4 + k] += x[Z + i] * dG[k];
                s += v->W_lstm[(size_t)(Z + A + i) * N4 + k] * dG[k];
            }
            dhn[i] = s;
        }
    }
    if (nll_out) nll_out[n] = total;
    free(X); free(act); free(C); free(Y); free(MD); free(h); free(g); free(dmd); free(dh);
    free(dhn); free(dcn); free(dG);
    return 0;
}

int orc_mdn_nll_grad(const orc_cfg *cfg, const orc_weights *w, int N, int T,
                     const float *z_seq, const int32_t *actions, const int32_t *lengths,
                     double *nll, double *gW_lstm, double *gb_lstm, double *gW_mdn,
                     double *gb_mdn)
{
    if (check_cfg(cfg) || N < 0 || T < 0 || !z_seq || !actions || !gW_lstm || !gb_lstm ||
        !gW_mdn || !gb_mdn)
        return -1;
    for (size_t i = 0; i < (size_t)N * T; ++i)
        if (actions[i] >= cfg->a_dim) return -1;
    if (lengths)
        for (int n = 0; n < N; ++n)
            if (lengths[n] < 0 || lengths[n] > T) return -1;
    const int Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, M = 3 * cfg->k_mix * Z;
    const size_t nW = (size_t)(Z + A + H) * 4 * H, nb = (size_t)4 * H, nWm = (size_t)H * M;
    const size_t per = nW + nb + nWm + (size_t)M;
    wts64 v;
    if (load_wts(cfg, w, &v, 0)) return -2;
    int nt = cfg->nthreads > 0 ? cfg->nthreads : 1;
    if (nt > N && N > 0) nt = N;
    if (nt < 1) nt = 1;
    /* one accumulator per thread; sequence n goes to thread n % nt, partials summed in
     * thread order (deterministic for a given thread count) */
    double *acc = calloc((size_t)nt * per, sizeof(double));
    if (!acc) { free_wts(&v); return -2; }
    int bad = 0;
#pragma omp parallel for schedule(static, 1) num_threads(nt) reduction(| : bad)
    for (int r = 0; r < nt; ++r) {
        double *a = acc + (size_t)r * per;
        for (int n = r; n < N; n += nt) {
            const int len = lengths ? lengths[n] : T;
            bad |= grad_sequence(cfg, &v, n, N, T, z_seq, actions, len, nll, a, a + nW, a + nW + nb,
                                 a + nW + nb + nWm) ? 1 : 0;
        }
    }
    for (size_t i = 0; i < nW; ++i) { double s = 0; for (int r = 0; r < nt; ++r) s += acc[(size_t)r * per + i]; gW_lstm[i] = s; }
    for (size_t i = 0; i < nb; ++i) { double s = 0; for (int r = 0; r < nt; ++r) s += acc[(size_t)r * per + nW + i]; gb_lstm[i] = s; }
    for (size_t i = 0; i < nWm; ++i) { double s = 0; for (int r = 0; r < nt; ++r) s += acc[(size_t)r * per + nW + nb + i]; gW_mdn[i] = s; }
    for (size_t i = 0; i < (size_t)M; ++i) { double s = 0; for (int r = 0; r < nt; ++r) s += acc[(size_t)r * per + nW + nb + nWm + i]; gb_mdn[i] = s; }
    free(acc);
    free_wts(&v);
    return bad ? -2 : 0;
}

int orc_mdn_nll(const orc_cfg *cfg, const orc_weights *w, int N, int T,
                const float *z_seq, const int32_t *actions, const int32_t *lengths,
                double *nll, float *h_seq, float *c_seq, float *mdn_seq)
{
    if (check_cfg(cfg) || N < 0 || T < 0 || !z_seq || !actions || !nll) return -1;
    for (size_t i = 0; i < (size_t)N * T; ++i)
        if (actions[i] >= cfg->a_dim) return -1;
    if (lengths)
        for (int n = 0; n < N; ++n)
            if (lengths[n] < 0 || lengths[n] > T) return -1;
    wts64 v;
    if (load_wts(cfg, w, &v, 0)) return -2;
    int bad = 0;
    int nt = cfg->nthreads > 0 ? cfg->nthreads : 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nt) reduction(| : bad)
    for (int n = 0; n < N; ++n) {
        int len = lengths ? lengths[n] : T;
        bad |= nll_sequence(cfg, &v, n, N, T, z_seq, actions, len, nll, h_seq, c_seq, mdn_seq) ? 1 : 0;
    }
    free_wts(&v);
    return bad ? -2 : 0;
}
