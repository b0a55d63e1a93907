// wm_internal.h -- handle layout and kernel-family launchers behind the C ABI
// of include/wm.h.  Not part of the public interface.
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "wm.h"

// Device pointers of one rollout call (after host arrays were staged).
// Per-step staging of caller host arrays, for families that launch step by step: the
// family calls these around its launches on stream s so that step t's inputs arrive
// and its outputs leave on copy streams while other steps compute.
struct wm_step_stage {
    virtual cudaError_t after_init(cudaStream_t s) = 0;        // the init kernel is enqueued
    virtual cudaError_t before_step(int t, cudaStream_t s) = 0;  // before step t's first launch
    virtual cudaError_t after_step(int t, cudaStream_t s) = 0;   // after step t's last launch
    virtual bool stepping() const = 0;  // whether outputs leave step by step (after_step copies)
    virtual ~wm_step_stage() {}
};

struct wm_rollout_dev {
    wm_step_stage *stage = nullptr;  // null: the arrays are whole on the device
    int B, T;
    unsigned long long ep0;
    unsigned int t0;
    const float *z0, *h0, *c0;
    const uint8_t *done0;
    const uint32_t *mask;
    float *z_out;
    int32_t *actions;
    float *rewards;
    uint8_t *done;
    float *h_final, *c_final, *h_seq, *c_seq, *mdn_seq;
    uint8_t *comp_seq;
    const float *rt0, *mem0;   // shaped reward: predictions entering the call
    float *rt_seq, *mem_seq;   // shaped reward: predictions after each step (optional)
    float *logp_seq;           // log-prob of the action taken (optional)
    float *value_seq;          // value head V(h_{t+1}) (optional)
    const uint32_t *loc_mask;  // hierarchical action: [T, B, NX, WL] location masks (or null)
    int32_t *loc_actions;      // hierarchical action: the location taken (optional)
};

// Device pointers of one teacher-forced scoring call.
struct wm_nll_dev {
    int N, T;
    const float *z_seq;
    const int32_t *actions;
    const int32_t *lengths;
    float *nll, *h_seq, *c_seq, *mdn_seq;
};

// Weights of the stepwise (SIMT) family: fp32 values (bf16-rounded in WM_BF16).
struct wm_step_weights {
    float *Wg;   // [Z+H, 4H+A]  rows z | h; cols gates i|f|g|o then controller
    float *Wa;   // [A, 4H]      action rows of the gate matrix
    float *bg;   // [4H+A]       gate bias then controller bias
    float *Wh;   // [H, M+NR]    mixture head, reward, done (+ runtime, memory) (+ value)
    float *bh;   // [M+NR]
    float *Wp;   // [P, Z+H, A]  controller candidates (P > 1 only; else in Wg)
    float *bp;   // [P, A]
};

// Weights of the fused single-launch family: per cluster size (slot 0: 16 CTAs,
// slot 1: 8 CTAs) one bf16 image per cluster rank, laid out as in wm_fused.cu.
struct wm_fused_weights {
    void *img[2];
    size_t img_bytes[2];   // bytes per rank image
    int max_clusters[2];   // clusters of that size that can be resident at once
    int force_cluster;     // 0 = choose per call, else 8 or 16
    int ok;                // 1 if the model fits this family
};

// The fused family's small-batch member (wm_small.cu): it reads the stepwise weights;
// this records the cluster size chosen for the model and its shared-memory geometry.
struct wm_small_cfg {
    int ok;                  // 1 if the model's per-CTA columns fit a cluster's shared memory
    int cl;                  // CTAs per cluster (1, 2, 4, 8 or 16)
    int max_clusters_eb[3];  // clusters resident at once, per tile size (16, 8, 4 episodes)
    alignas(8) unsigned char geo[3][256];  // wm_small.cu's geometry record per tile size
    void *img;               // per-rank weight images (the shared-memory layout), cl of them
    size_t img_stride;       // bytes between two ranks' images
};

// Weights of the tensor-core family (bf16, K-major; orders in wm_tensor.cu).
struct wm_tc_weights {
    void *wc, *wg, *wa, *wh;  // W_c^T [P*A, Z+H], W_g^T [4H, Z+H], W_a [A, 4H], W_h^T [tiles*240, H]
    // fp32 path: the weights are the bf16 sums hi + lo; these are the lo parts (else null)
    void *wc_lo, *wg_lo, *wa_lo, *wh_lo;
    // the gate weights, action rows and bias packed again for 128-column tiles (32 units x
    // i|f|g|o per tile), for calls with few row tiles; the fp32 path's lo parts of the first two
    void *wg_n, *wa_n;
    void *wg_n_lo, *wa_n_lo;
    float *bg_n;
    float *bc, *bg, *bh;
    int dims_per_tile, n_head_tiles, rd_tile, rd_col;  // reward, done (, runtime, memory) columns
    int sms;
    int ok;
};

// Per-kernel timing (wm_set_timing): event pairs recorded on the launching
// stream, folded into per-class totals when read.
struct wm_timer {
    struct Rec {
        int cls;
        cudaEvent_t a, b;
    };
    bool on = false;
    std::vector<Rec> pending;
    std::vector<cudaEvent_t> spare;
    double ms[WM_KERNEL_CLASSES] = {};
    long long launches[WM_KERNEL_CLASSES] = {};
};

// A canonical host copy of the weights (the layouts of wm_weights).
struct wm_host_weights {
    std::vector<float> W_lstm, b_lstm, W_mdn, b_mdn, w_rew, w_done, W_ctrl, b_ctrl, w_rt, w_mem, w_val;
    float b_rew = 0.f, b_done = 0.f, b_rt = 0.f, b_mem = 0.f, b_val = 0.f;
    wm_weights view() const {
        auto p = [](const std::vector<float> &v) { return v.empty() ? nullptr : v.data(); };
        wm_weights w{};
        w.W_lstm = p(W_lstm); w.b_lstm = p(b_lstm); w.W_mdn = p(W_mdn); w.b_mdn = p(b_mdn);
        w.w_rew = p(w_rew); w.b_rew = b_rew; w.w_done = p(w_done); w.b_done = b_done;
        w.W_ctrl = p(W_ctrl); w.b_ctrl = p(b_ctrl); w.w_rt = p(w_rt); w.b_rt = b_rt;
        w.w_mem = p(w_mem); w.b_mem = b_mem; w.w_val = p(w_val); w.b_val = b_val;
        return w;
    }
};

struct wm_handle {
    wm_config cfg;
    int device;
    int M;                       // 3 K Z
    int NR;                      // head columns after the mixture: reward, done (+ runtime,
                                 // memory when shaped) (+ value when value_head), in that order
    int P = 1, E = 1;            // controller population: candidate of episode e = (e / E) mod P
    wm_host_weights host;        // canonical host copy (repacks the fused family's images
                                 // when the controller changes)
    wm_step_weights step;
    wm_fused_weights fused;
    wm_small_cfg small;
    wm_tc_weights tc;
    void *ws = nullptr;          // workspace (grows on demand)
    size_t ws_bytes = 0;
    void *stage = nullptr;       // staging for host arrays (grows on demand)
    size_t stage_bytes = 0;
    cudaStream_t copy_in = nullptr, copy_out = nullptr;  // per-step staging copies (lazy)
    std::vector<cudaEvent_t> events;                       // per-step staging events (grows)
    int *status = nullptr;       // device status word (WM_ERR_TIMEOUT etc.)
    // tensor family, compacted rollouts: a host-mapped word the compaction kernel sets to the
    // call's sequence number once no episode is live, so that the host stops issuing steps
    mutable int *dead_host = nullptr;
    mutable int *dead_dev = nullptr;
    mutable int call_seq = 0;
    mutable std::vector<cudaEvent_t> step_events;  // the early stop's step events (lazy)
    mutable uint32_t test_wait = 0;  // wm_inject_wait_timeout: polls of the next call's injected
                                     // wait (consumed by that call's first fused / GEMM launch)
    int last_path = 0;
    mutable int last_launches = 0;   // kernels launched by the last call
    mutable wm_timer timer;
    std::string err;
    // the training step (wm_backward.cu): cuBLAS handle, copies of its GEMMs' weights (bf16 for
    // the bf16 path; W_mdn packed without the reward and done columns for the fp32 path), and its
    // workspace (all created on first use)
    void *cublas = nullptr;
    void *bw_wzh = nullptr, *bw_wm = nullptr;
    void *bw_w3 = nullptr;  // fp32 path: W_h as bf16 rows [hi | lo | hi] for the recurrence GEMM
    void *bws = nullptr;
    size_t bws_bytes = 0;
};

// Brackets the kernel launches of its scope with CUDA events on stream s when
// timing is on for h; does nothing otherwise.
class wm_ktime {
  public:
    wm_ktime(const wm_handle *h, int cls, cudaStream_t s);
    ~wm_ktime();
    wm_ktime(const wm_ktime &) = delete;
    wm_ktime &operator=(const wm_ktime &) = delete;

  private:
    wm_timer *t_;
    int cls_;
    cudaStream_t s_;
    cudaEvent_t a_ = nullptr;
};

// ---- tensor-core family (wm_tensor.cu) ----------------------------------------
int wm_tc_supported(const wm_handle *h);
// workspace of a call of B rows; T_teacher >= 0: teacher-forced scoring of T_teacher steps
// (its operand rows of all T_teacher + 1 frames), -1: a rollout
size_t wm_tc_ws(const wm_handle *h, int B, int T_teacher = -1);
cudaError_t wm_tc_pack(wm_handle *h, const wm_weights *w);
void wm_tc_free(wm_handle *h);
cudaError_t wm_tc_rollout(const wm_handle *h, const wm_rollout_dev &a, void *ws, cudaStream_t s);
cudaError_t wm_tc_nll(const wm_handle *h, const wm_nll_dev &a, void *ws, cudaStream_t s);
cudaError_t wm_tc_set_controllers(wm_handle *h, int P, const float *W_ctrl, const float *b_ctrl);
// whether the tensor family can run a rollout call starting at this episode (population tiles)
int wm_tc_call_ok(const wm_handle *h, unsigned long long episode_offset);

// ---- the fused family's small-batch member (wm_small.cu) ----------------------
cudaError_t wm_small_prepare(wm_handle *h);
cudaError_t wm_small_repack(wm_handle *h);  // after the stepwise weights changed
void wm_small_free(wm_handle *h);
int wm_small_supported(const wm_handle *h, int B);
int wm_small_cluster_size(const wm_handle *h);
cudaError_t wm_small_rollout(const wm_handle *h, const wm_rollout_dev &a, cudaStream_t s);
cudaError_t wm_small_nll(const wm_handle *h, const wm_nll_dev &a, cudaStream_t s);

// ---- the training step (wm_backward.cu) -----------------------------------------
size_t wm_bw_ws(const wm_handle *h, int N, int T);
void wm_bw_carve(const wm_handle *h, int N, int T, void *base, float **hs, float **cs, float **md, float **nll,
                 void **tail);
cudaError_t wm_bw_prepare(wm_handle *h);
void wm_bw_free(wm_handle *h);
cudaError_t wm_bw_launch(const wm_handle *h, int N, int T, const float *z_seq, const int32_t *actions,
                         const int32_t *lengths, const wm_grads &g, const float *hs, const float *cs,
                         const float *md, void *tail, cudaStream_t s);

// ---- discounted returns (wm_returns.cu) ----------------------------------------
cudaError_t wm_returns_launch(const wm_handle *h, int B, int T, unsigned long long ep0, float gamma,
                              int stop_at_done, const float *rewards, const uint8_t *done,
                              const float *bootstrap, float *returns, float *fitness, void *ws,
                              cudaStream_t s);
size_t wm_returns_ws(const wm_handle *h, int B);

// ---- stepwise family (wm_step.cu) -------------------------------------------
size_t wm_step_rollout_ws(const wm_handle *h, int B);
size_t wm_step_nll_ws(const wm_handle *h, int N);
cudaError_t wm_step_rollout(const wm_handle *h, const wm_rollout_dev &a, void *ws, cudaStream_t s);
cudaError_t wm_step_nll(const wm_handle *h, const wm_nll_dev &a, void *ws, cudaStream_t s);
