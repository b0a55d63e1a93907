// wm_api.cu -- the C ABI of include/wm.h: argument checks, weight packing,
// host<->device staging of caller arrays, and dispatch to a kernel family.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdio.h>
#include <string.h>

#include <new>
#include <string>
#include <vector>

#include "wm_internal.h"

// ---- kernel families implemented in other translation units ---------------
int wm_fused_supported(const wm_handle *h, int B);
cudaError_t wm_fused_pack(wm_handle *h, const wm_weights *w);
void wm_fused_free(wm_handle *h);
cudaError_t wm_fused_rollout(const wm_handle *h, const wm_rollout_dev &a, cudaStream_t s);
cudaError_t wm_fused_nll(const wm_handle *h, const wm_nll_dev &a, void *ws, cudaStream_t s);
size_t wm_fused_nll_ws(const wm_handle *h, int N);

namespace {

wm_status fail(wm_handle *h, wm_status st, const std::string &msg) {
    if (h) h->err = msg;
    return st;
}

wm_status cuda_fail(wm_handle *h, cudaError_t e, const char *where) {
    std::string m = std::string(where) + ": " + cudaGetErrorString(e);
    return fail(h, e == cudaErrorMemoryAllocation ? WM_ERR_OOM : WM_ERR_CUDA, m);
}

bool is_host_ptr(const void *p) {
    cudaPointerAttributes at;
    cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return true;
    }
    return at.type == cudaMemoryTypeHost || at.type == cudaMemoryTypeUnregistered;
}

float bf16_round_host(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

cudaError_t grow(void **buf, size_t *have, size_t need) {
    if (need <= *have) return cudaSuccess;
    if (*buf) {
        cudaError_t e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return e;
        cudaFree(*buf);
        *buf = nullptr;
        *have = 0;
    }
    size_t n = need + need / 8;
    cudaError_t e = cudaMalloc(buf, n);
    if (e != cudaSuccess) return e;
    *have = n;
    return cudaSuccess;
}

template <class T>
cudaError_t upload(T **dst, const std::vector<T> &src) {
    cudaError_t e = cudaMalloc((void **)dst, src.size() * sizeof(T));
    if (e != cudaSuccess) return e;
    return cudaMemcpy(*dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice);
}

// One caller array that may need staging.
// How a staged array meets the steps of a call.
enum StageKind {
    WHOLE = 0,    // copied whole: inputs before the call, outputs after it
    STEP_IN = 1,  // input; slab t is first read by step t
    STEP_OUT = 2, // output; slab t is final after step t
    TRAJ_OUT = 3, // output of T + 1 slabs; slab 0 is final after the init kernel, slab t + 1 after step t
};

struct Stage {
    void **dev;        // where the device pointer goes
    const void *user;  // caller pointer
    size_t bytes;
    bool out;
    size_t off;
    int kind;
    size_t slab;       // bytes per step (per-step kinds)
};

// Copies caller host arrays through the handle's staging buffer.  With per-step
// staging on (a family that launches step by step, pinned or pageable host memory,
// a stream that is not capturing), step t's input slabs go up on copy_in ahead of the
// steps and its output slabs come down on copy_out as soon as step t is done, so the
// copies overlap the computation; otherwise everything is copied whole around the call.
// Either way a call with host arrays returns once every copy is complete.
struct Stager : wm_step_stage {
    std::vector<Stage> items;
    size_t total = 0;
    bool any_host = false, any_host_out = false;
    bool stepped = false;
    int T = 0;
    wm_handle *h = nullptr;
    cudaEvent_t *ev = nullptr;  // [0]: start, [1]: init done, [2 + t]: step t's inputs, [2 + T + t]: step t done
    void add(void **dev, const void *user, size_t bytes, bool out, int kind = WHOLE, size_t slab = 0) {
        *dev = const_cast<void *>(user);
        if (!user || bytes == 0 || !is_host_ptr(user)) return;
        items.push_back({dev, user, bytes, out, total, kind, slab});
        total += (bytes + 255) & ~(size_t)255;
        any_host = true;
        if (out) any_host_out = true;
    }
    cudaError_t copy_slab(const Stage &it, size_t i, cudaStream_t s) {
        const size_t o = i * it.slab;
        if (it.out)
            return cudaMemcpyAsync((char *)const_cast<void *>(it.user) + o, (char *)*it.dev + o, it.slab,
                                   cudaMemcpyDeviceToHost, s);
        return cudaMemcpyAsync((char *)*it.dev + o, (const char *)it.user + o, it.slab, cudaMemcpyHostToDevice, s);
    }
    // step_wise: the family will call the wm_step_stage hooks
    cudaError_t begin(wm_handle *hd, int steps, bool step_wise, cudaStream_t s) {
        if (items.empty()) return cudaSuccess;
        h = hd;
        T = steps;
        cudaError_t e = grow(&h->stage, &h->stage_bytes, total);
        if (e != cudaSuccess) return e;
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if ((e = cudaStreamIsCapturing(s, &cs)) != cudaSuccess) return e;
        stepped = step_wise && T > 1 && cs == cudaStreamCaptureStatusNone;
        if (stepped) {
            if (!h->copy_in && (e = cudaStreamCreateWithFlags(&h->copy_in, cudaStreamNonBlocking)) != cudaSuccess)
                return e;
            if (!h->copy_out && (e = cudaStreamCreateWithFlags(&h->copy_out, cudaStreamNonBlocking)) != cudaSuccess)
                return e;
            const size_t need = 2 + 2 * (size_t)T;
            while (h->events.size() < need) {
                cudaEvent_t x;
                if ((e = cudaEventCreateWithFlags(&x, cudaEventDisableTiming)) != cudaSuccess) return e;
                h->events.push_back(x);
            }
            ev = h->events.data();
        }
        for (auto &it : items) {
            *it.dev = (char *)h->stage + it.off;
            if (it.out) continue;
            if (!stepped || it.kind == WHOLE) {
                e = cudaMemcpyAsync(*it.dev, it.user, it.bytes, cudaMemcpyHostToDevice, s);
                if (e != cudaSuccess) return e;
            }
        }
        if (!stepped) return cudaSuccess;
        // the copy streams start after the stream's earlier work (the staging buffer's
        // previous users); step inputs go up in step order
        if ((e = cudaEventRecord(ev[0], s)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(h->copy_in, ev[0], 0)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(h->copy_out, ev[0], 0)) != cudaSuccess) return e;
        for (int t = 0; t < T; ++t) {
            for (auto &it : items)
                if (it.kind == STEP_IN && (e = copy_slab(it, (size_t)t, h->copy_in)) != cudaSuccess) return e;
            if ((e = cudaEventRecord(ev[2 + t], h->copy_in)) != cudaSuccess) return e;
        }
        return cudaSuccess;
    }
    bool stepping() const override { return stepped; }
    cudaError_t after_init(cudaStream_t s) override {
        if (!stepped) return cudaSuccess;
        cudaError_t e = cudaEventRecord(ev[1], s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(h->copy_out, ev[1], 0);
        for (auto &it : items)
            if (e == cudaSuccess && it.kind == TRAJ_OUT) e = copy_slab(it, 0, h->copy_out);
        return e;
    }
    cudaError_t before_step(int t, cudaStream_t s) override {
        return stepped ? cudaStreamWaitEvent(s, ev[2 + t], 0) : cudaSuccess;
    }
    cudaError_t after_step(int t, cudaStream_t s) override {
        if (!stepped) return cudaSuccess;
        cudaEvent_t done = ev[2 + T + t];
        cudaError_t e = cudaEventRecord(done, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(h->copy_out, done, 0);
        for (auto &it : items) {
            if (e != cudaSuccess) break;
            if (it.kind == STEP_OUT) e = copy_slab(it, (size_t)t, h->copy_out);
            else if (it.kind == TRAJ_OUT) e = copy_slab(it, (size_t)t + 1, h->copy_out);
        }
        return e;
    }
    cudaError_t end(cudaStream_t s) {
        for (auto &it : items) {
            if (!it.out || (stepped && it.kind != WHOLE)) continue;
            cudaError_t e = cudaMemcpyAsync(const_cast<void *>(it.user), *it.dev, it.bytes,
                                            cudaMemcpyDeviceToHost, s);
            if (e != cudaSuccess) return e;
        }
        if (stepped) {
            cudaError_t e = cudaStreamSynchronize(h->copy_in);
            if (e == cudaSuccess) e = cudaStreamSynchronize(h->copy_out);
            if (e != cudaSuccess) return e;
        }
        if (any_host_out || stepped) return cudaStreamSynchronize(s);
        return cudaSuccess;
    }
    // an early return (an error) still waits for the copies that touch the caller's arrays
    ~Stager() {
        if (stepped && h) {
            cudaStreamSynchronize(h->copy_in);
            cudaStreamSynchronize(h->copy_out);
        }
    }
};

bool valid_cfg(const wm_config *c) {
    return c && c->z_dim > 0 && c->a_dim > 0 && c->h_dim > 0 && c->k_mix > 0 && c->k_mix <= 32 &&
           (c->precision == WM_FP32 || c->precision == WM_BF16) && c->mdn_tau >= 0.f &&
           c->ctrl_tau >= 0.f && c->path >= WM_PATH_AUTO && c->path <= WM_PATH_TENSOR &&
           c->z_dim <= 4096 && c->a_dim <= 65536 && c->h_dim <= 16384 &&
           (c->fused_cluster == 0 || c->fused_cluster == 8 || c->fused_cluster == 16) &&
           (c->reward_mode == WM_REWARD_HEAD || c->reward_mode == WM_REWARD_SHAPED) &&
           c->n_xfers >= 0 && c->n_xfers < c->a_dim;
}

cudaError_t pack_step(wm_handle *h, const wm_weights *w) {
    const wm_config &c = h->cfg;
    const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M, N1 = 4 * H + A, NR = h->NR;
    const bool rb = c.precision == WM_BF16;
    auto wv = [&](float x) { return rb ? bf16_round_host(x) : x; };
    std::vector<float> Wg((Z + H) * N1), Wa(A * 4 * H), bg(N1), Wh(H * (M + NR)), bh(M + NR);
    for (size_t r = 0; r < Z + H; ++r) {
        const size_t src = r < Z ? r : r + A;  // skip the action rows
        for (size_t n = 0; n < 4 * H; ++n) Wg[r * N1 + n] = wv(w->W_lstm[src * 4 * H + n]);
        for (size_t j = 0; j < A; ++j) Wg[r * N1 + 4 * H + j] = wv(w->W_ctrl[r * A + j]);
    }
    for (size_t a = 0; a < A; ++a)
        for (size_t n = 0; n < 4 * H; ++n) Wa[a * 4 * H + n] = wv(w->W_lstm[(Z + a) * 4 * H + n]);
    for (size_t n = 0; n < 4 * H; ++n) bg[n] = w->b_lstm[n];
    for (size_t j = 0; j < A; ++j) bg[4 * H + j] = w->b_ctrl[j];
    for (size_t i = 0; i < H; ++i) {
        for (size_t m = 0; m < M; ++m) Wh[i * (M + NR) + m] = wv(w->W_mdn[i * M + m]);
        Wh[i * (M + NR) + M] = wv(w->w_rew[i]);
        Wh[i * (M + NR) + M + 1] = wv(w->w_done[i]);
        if (c.reward_mode == WM_REWARD_SHAPED) {
            Wh[i * (M + NR) + M + 2] = wv(w->w_rt[i]);
            Wh[i * (M + NR) + M + 3] = wv(w->w_mem[i]);
        }
        if (c.value_head) Wh[i * (M + NR) + M + NR - 1] = wv(w->w_val[i]);
    }
    for (size_t m = 0; m < M; ++m) bh[m] = w->b_mdn[m];
    bh[M] = w->b_rew;
    bh[M + 1] = w->b_done;
    if (c.reward_mode == WM_REWARD_SHAPED) {
        bh[M + 2] = w->b_rt;
        bh[M + 3] = w->b_mem;
    }
    if (c.value_head) bh[M + NR - 1] = w->b_val;
    cudaError_t e;
    if ((e = upload(&h->step.Wg, Wg)) != cudaSuccess) return e;
    if ((e = upload(&h->step.Wa, Wa)) != cudaSuccess) return e;
    if ((e = upload(&h->step.bg, bg)) != cudaSuccess) return e;
    if ((e = upload(&h->step.Wh, Wh)) != cudaSuccess) return e;
    return upload(&h->step.bh, bh);
}

// AUTO: the fused single-launch family when one of its members takes the model and the
// batch (its tcgen05 member up to B = 2048; its small-batch member while the batch needs at
// most 4 waves of 16-episode clusters), else the tensor-core family for large bf16 batches
// and for fp32 models of any batch (its three-pass split beat the stepwise fp32 SIMT family
// 2x even at B = 16), the stepwise family otherwise.  fused_ok / tc_ok: whether this call's
// options allow those families.
int pick_path(const wm_handle *h, int B, bool fused_ok = true, bool tc_ok = true) {
    const int p = h->cfg.path;
    if (p != WM_PATH_AUTO) return p;
    const bool fu = fused_ok && wm_fused_supported(h, B), tc = tc_ok && wm_tc_supported(h);
    if (fu && B <= 2048) return WM_PATH_FUSED;
    if (tc && (B >= 256 || h->cfg.precision == WM_FP32)) return WM_PATH_TENSOR;
    if (fu) return WM_PATH_FUSED;
    return WM_PATH_STEPWISE;
}

template <class T>
std::vector<T> host_vec(const T *p, size_t n) {
    return p ? std::vector<T>(p, p + n) : std::vector<T>();
}

}  // namespace

extern "C" {

wm_status wm_create(const wm_config *cfg, const wm_weights *w, wm_handle **out) {
    if (!out) return WM_ERR_INVALID_ARG;
    *out = nullptr;
    if (!valid_cfg(cfg)) return WM_ERR_INVALID_ARG;
    if (!w || !w->W_lstm || !w->b_lstm || !w->W_mdn || !w->b_mdn || !w->w_rew || !w->w_done ||
        !w->W_ctrl || !w->b_ctrl)
        return WM_ERR_INVALID_ARG;
    if (cfg->reward_mode == WM_REWARD_SHAPED && (!w->w_rt || !w->w_mem)) return WM_ERR_INVALID_ARG;
    if (cfg->value_head && !w->w_val) return WM_ERR_INVALID_ARG;
    wm_handle *h = new (std::nothrow) wm_handle();
    if (!h) return WM_ERR_OOM;
    h->cfg = *cfg;
    h->M = 3 * cfg->k_mix * cfg->z_dim;
    h->NR = 2 + (cfg->reward_mode == WM_REWARD_SHAPED ? 2 : 0) + (cfg->value_head ? 1 : 0);
    {
        const size_t Z = cfg->z_dim, A = cfg->a_dim, H = cfg->h_dim, M = h->M;
        wm_host_weights &hw = h->host;
        hw.W_lstm = host_vec(w->W_lstm, (Z + A + H) * 4 * H);
        hw.b_lstm = host_vec(w->b_lstm, 4 * H);
        hw.W_mdn = host_vec(w->W_mdn, H * M);
        hw.b_mdn = host_vec(w->b_mdn, M);
        hw.w_rew = host_vec(w->w_rew, H);
        hw.w_done = host_vec(w->w_done, H);
        hw.W_ctrl = host_vec(w->W_ctrl, (Z + H) * A);
        hw.b_ctrl = host_vec(w->b_ctrl, A);
        if (cfg->reward_mode == WM_REWARD_SHAPED) {
            hw.w_rt = host_vec(w->w_rt, H);
            hw.w_mem = host_vec(w->w_mem, H);
        }
        if (cfg->value_head) hw.w_val = host_vec(w->w_val, H);
        hw.b_rew = w->b_rew; hw.b_done = w->b_done; hw.b_rt = w->b_rt; hw.b_mem = w->b_mem;
        hw.b_val = w->b_val;
    }
    memset(&h->step, 0, sizeof(h->step));
    memset(&h->fused, 0, sizeof(h->fused));
    memset(&h->small, 0, sizeof(h->small));
    memset(&h->tc, 0, sizeof(h->tc));
    cudaError_t e = cudaGetDevice(&h->device);
    if (e == cudaSuccess) e = pack_step(h, w);
    h->fused.force_cluster = cfg->fused_cluster;
    if (e == cudaSuccess) e = wm_fused_pack(h, w);
    if (e == cudaSuccess) e = wm_small_prepare(h);
    if (e == cudaSuccess) e = wm_tc_pack(h, w);
    if (e == cudaSuccess) e = cudaMalloc((void **)&h->status, sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(h->status, 0, sizeof(int));
    if (e != cudaSuccess) {
        wm_status st = e == cudaErrorMemoryAllocation ? WM_ERR_OOM : WM_ERR_CUDA;
        cudaGetLastError();
        wm_destroy(h);
        return st;
    }
    *out = h;
    return WM_OK;
}

void wm_destroy(wm_handle *h) {
    if (!h) return;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    cudaDeviceSynchronize();
    cudaFree(h->step.Wg);
    cudaFree(h->step.Wa);
    cudaFree(h->step.bg);
    cudaFree(h->step.Wh);
    cudaFree(h->step.bh);
    cudaFree(h->step.Wp);
    cudaFree(h->step.bp);
    wm_fused_free(h);
    wm_small_free(h);
    wm_tc_free(h);
    wm_bw_free(h);
    cudaFree(h->ws);
    cudaFree(h->stage);
    cudaFree(h->status);
    for (auto &r : h->timer.pending) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
    }
    for (cudaEvent_t ev : h->timer.spare) cudaEventDestroy(ev);
    for (cudaEvent_t ev : h->events) cudaEventDestroy(ev);
    if (h->copy_in) cudaStreamDestroy(h->copy_in);
    if (h->copy_out) cudaStreamDestroy(h->copy_out);
    if (prev >= 0) cudaSetDevice(prev);
    delete h;
}

// ---- per-kernel timing --------------------------------------------------------
static cudaEvent_t timer_event(wm_timer &t) {
    if (!t.spare.empty()) {
        cudaEvent_t ev = t.spare.back();
        t.spare.pop_back();
        return ev;
    }
    cudaEvent_t ev = nullptr;
    if (cudaEventCreate(&ev) != cudaSuccess) return nullptr;
    return ev;
}

wm_ktime::wm_ktime(const wm_handle *h, int cls, cudaStream_t s) : t_(nullptr), cls_(cls), s_(s) {
    if (!h || !h->timer.on) return;
    t_ = &h->timer;
    a_ = timer_event(*t_);
    if (a_ && cudaEventRecord(a_, s_) != cudaSuccess) {
        t_->spare.push_back(a_);
        a_ = nullptr;
    }
}

wm_ktime::~wm_ktime() {
    if (!t_ || !a_) return;
    cudaEvent_t b = timer_event(*t_);
    if (b && cudaEventRecord(b, s_) == cudaSuccess) {
        t_->pending.push_back({cls_, a_, b});
        return;
    }
    t_->spare.push_back(a_);
    if (b) t_->spare.push_back(b);
}

wm_status wm_set_timing(wm_handle *h, int enable) {
    if (!h) return WM_ERR_INVALID_ARG;
    wm_timer &t = h->timer;
    if (enable) {
        for (auto &r : t.pending) {  // discard what was recorded before
            cudaEventSynchronize(r.b);
            t.spare.push_back(r.a);
            t.spare.push_back(r.b);
        }
        t.pending.clear();
        for (int i = 0; i < WM_KERNEL_CLASSES; ++i) {
            t.ms[i] = 0.0;
            t.launches[i] = 0;
        }
    }
    t.on = enable != 0;
    return WM_OK;
}

wm_status wm_kernel_time(wm_handle *h, int kernel_class, double *total_ms, long long *launches) {
    if (!h) return WM_ERR_INVALID_ARG;
    if (kernel_class < 0 || kernel_class >= WM_KERNEL_CLASSES)
        return fail(h, WM_ERR_INVALID_ARG, "kernel class out of range");
    wm_timer &t = h->timer;
    cudaError_t err = cudaSuccess;
    for (auto &r : t.pending) {
        float ms = 0.f;
        cudaError_t e = cudaEventSynchronize(r.b);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, r.a, r.b);
        if (e == cudaSuccess) {
            t.ms[r.cls] += ms;
            t.launches[r.cls] += 1;
        } else if (err == cudaSuccess) {
            err = e;
        }
        t.spare.push_back(r.a);
        t.spare.push_back(r.b);
    }
    t.pending.clear();
    if (err != cudaSuccess) return cuda_fail(h, err, "wm_kernel_time");
    if (total_ms) *total_ms = t.ms[kernel_class];
    if (launches) *launches = t.launches[kernel_class];
    return WM_OK;
}

wm_status wm_inject_wait_timeout(wm_handle *h, unsigned int polls) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->test_wait = polls;
    return WM_OK;
}

const char *wm_last_error(const wm_handle *h) { return h ? h->err.c_str() : "null handle"; }

int wm_last_path(const wm_handle *h) { return h ? h->last_path : 0; }

int wm_last_launches(const wm_handle *h) { return h ? h->last_launches : 0; }

wm_status wm_sync(wm_handle *h) {
    if (!h) return WM_ERR_INVALID_ARG;
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(h, e, "wm_sync");
    int st = 0;
    e = cudaMemcpy(&st, h->status, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(h, e, "wm_sync status");
    if (st != 0) {
        cudaMemset(h->status, 0, sizeof(int));
        return fail(h, (wm_status)st, "device-side error reported by a kernel");
    }
    return WM_OK;
}

wm_status wm_rollout(wm_handle *h, int B, int T, unsigned long long episode_offset, unsigned int t0,
                     const wm_rollout_io *io, void *cuda_stream) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->err.clear();
    if (!io) return fail(h, WM_ERR_INVALID_ARG, "io is NULL");
    if (B < 0 || T < 0 || B > (1 << 22)) return fail(h, WM_ERR_INVALID_ARG, "B must be in [0, 2^22], T >= 0");
    if (B > 0 && (!io->z0 || !io->z_out || (T > 0 && (!io->actions || !io->rewards || !io->done))))
        return fail(h, WM_ERR_INVALID_ARG, "z0, z_out, actions, rewards and done are required");
    if ((unsigned long long)t0 + (unsigned long long)T > 0x100000000ull)
        return fail(h, WM_ERR_INVALID_ARG, "t0 + T overflows the 32-bit Philox step counter");
    const wm_config &c = h->cfg;
    const bool shaped = c.reward_mode == WM_REWARD_SHAPED;
    if (shaped && B > 0 && (!io->rt0 || !io->mem0))
        return fail(h, WM_ERR_INVALID_ARG, "the shaped reward needs rt0 and mem0");
    const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M, W = (A + 31) / 32;
    const size_t b = (size_t)B, t = (size_t)T;
    cudaStream_t s = (cudaStream_t)cuda_stream;
    cudaError_t e = cudaSetDevice(h->device);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");

    wm_rollout_dev a{};
    a.B = B; a.T = T; a.ep0 = episode_offset; a.t0 = t0;
    Stager st;
    st.add((void **)&a.z0, io->z0, b * Z * 4, false);
    st.add((void **)&a.h0, io->h0, b * H * 4, false);
    st.add((void **)&a.c0, io->c0, b * H * 4, false);
    st.add((void **)&a.done0, io->done0, b, false);
    st.add((void **)&a.mask, io->mask, t * b * W * 4, false, STEP_IN, b * W * 4);
    st.add((void **)&a.z_out, io->z_out, (t + 1) * b * Z * 4, true, TRAJ_OUT, b * Z * 4);
    st.add((void **)&a.actions, io->actions, t * b * 4, true, STEP_OUT, b * 4);
    st.add((void **)&a.rewards, io->rewards, t * b * 4, true, STEP_OUT, b * 4);
    st.add((void **)&a.done, io->done, t * b, true, STEP_OUT, b);
    st.add((void **)&a.h_final, io->h_final, b * H * 4, true);
    st.add((void **)&a.c_final, io->c_final, b * H * 4, true);
    st.add((void **)&a.h_seq, io->h_seq, t * b * H * 4, true, STEP_OUT, b * H * 4);
    st.add((void **)&a.c_seq, io->c_seq, t * b * H * 4, true, STEP_OUT, b * H * 4);
    st.add((void **)&a.mdn_seq, io->mdn_seq, t * b * M * 4, true, STEP_OUT, b * M * 4);
    st.add((void **)&a.comp_seq, io->comp_seq, t * b * Z, true, STEP_OUT, b * Z);
    st.add((void **)&a.logp_seq, io->logp_seq, t * b * 4, true, STEP_OUT, b * 4);
    if (c.n_xfers > 0) {
        const size_t WL = (A - c.n_xfers + 31) / 32, NX = c.n_xfers;
        st.add((void **)&a.loc_mask, io->loc_mask, t * b * NX * WL * 4, false, STEP_IN, b * NX * WL * 4);
        st.add((void **)&a.loc_actions, io->loc_actions, t * b * 4, true, STEP_OUT, b * 4);
    }
    if (c.value_head) st.add((void **)&a.value_seq, io->value_seq, t * b * 4, true, STEP_OUT, b * 4);
    if (shaped) {
        st.add((void **)&a.rt0, io->rt0, b * 4, false);
        st.add((void **)&a.mem0, io->mem0, b * 4, false);
        st.add((void **)&a.rt_seq, io->rt_seq, t * b * 4, true, STEP_OUT, b * 4);
        st.add((void **)&a.mem_seq, io->mem_seq, t * b * 4, true, STEP_OUT, b * 4);
    }

    // the fused family writes no log-probs or values and has one controller; the tensor
    // family needs a population's candidates aligned to its 256-row tiles
    const bool fused_ok = !io->logp_seq && !(c.value_head && io->value_seq) && h->P == 1 && c.n_xfers == 0;
    const bool tc_ok = wm_tc_call_ok(h, episode_offset) != 0;
    int path = pick_path(h, B, fused_ok, tc_ok);
    if (path == WM_PATH_FUSED && !(fused_ok && wm_fused_supported(h, B)))
        return fail(h, WM_ERR_UNSUPPORTED, "the fused family does not take this model / batch / outputs");
    if (path == WM_PATH_TENSOR && !(tc_ok && wm_tc_supported(h)))
        return fail(h, WM_ERR_UNSUPPORTED, "the tensor family does not take this model / call");

    size_t need = path == WM_PATH_STEPWISE ? wm_step_rollout_ws(h, B) : path == WM_PATH_TENSOR ? wm_tc_ws(h, B) : 0;
    if (need) {
        e = grow(&h->ws, &h->ws_bytes, need);
        if (e != cudaSuccess) return cuda_fail(h, e, "workspace");
    }
    // the tensor family launches step by step: its host arrays are staged per step
    if ((e = st.begin(h, T, path == WM_PATH_TENSOR && B > 0, s)) != cudaSuccess) return cuda_fail(h, e, "staging inputs");
    a.stage = &st;
    if (path == WM_PATH_FUSED)
        e = wm_fused_rollout(h, a, s);
    else if (path == WM_PATH_TENSOR)
        e = wm_tc_rollout(h, a, h->ws, s);
    else
        e = wm_step_rollout(h, a, h->ws, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "rollout launch");
    h->last_path = path;
    if (path == WM_PATH_STEPWISE)
        h->last_launches = B == 0 ? 0 : 1 + (h->P > 1 ? 5 : 4) * T + ((a.h_final || a.c_final) ? 1 : 0);
    if ((e = st.end(s)) != cudaSuccess) return cuda_fail(h, e, "staging outputs");
    return WM_OK;
}

wm_status wm_set_controllers(wm_handle *h, int P, int E, const float *W_ctrl, const float *b_ctrl) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->err.clear();
    if (P < 1 || E < 1 || !W_ctrl || !b_ctrl) return fail(h, WM_ERR_INVALID_ARG, "P, E >= 1 and arrays required");
    const wm_config &c = h->cfg;
    const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, KX = Z + H, N1 = 4 * H + A;
    cudaError_t e = cudaSetDevice(h->device);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
    e = cudaDeviceSynchronize();  // earlier calls may still read the controller weights
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaDeviceSynchronize");
    const bool rb = c.precision == WM_BF16;
    auto wv = [&](float x) { return rb ? bf16_round_host(x) : x; };
    // stepwise: candidate 0 in the controller columns of the combined GEMM matrix, and all
    // candidates in Wp / bp when there is more than one
    std::vector<float> w0(KX * A);
    for (size_t i = 0; i < KX * A; ++i) w0[i] = wv(W_ctrl[i]);
    e = cudaMemcpy2D(h->step.Wg + 4 * H, N1 * 4, w0.data(), A * 4, A * 4, KX, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(h->step.bg + 4 * H, b_ctrl, A * 4, cudaMemcpyHostToDevice);
    cudaFree(h->step.Wp);
    cudaFree(h->step.bp);
    h->step.Wp = h->step.bp = nullptr;
    if (e == cudaSuccess && P > 1) {
        std::vector<float> wp((size_t)P * KX * A), bpv(b_ctrl, b_ctrl + (size_t)P * A);
        for (size_t i = 0; i < wp.size(); ++i) wp[i] = wv(W_ctrl[i]);
        e = upload(&h->step.Wp, wp);
        if (e == cudaSuccess) e = upload(&h->step.bp, bpv);
    }
    if (e == cudaSuccess && h->tc.ok) e = wm_tc_set_controllers(h, P, W_ctrl, b_ctrl);
    // the fused family packs the controller into its per-rank images: repack them
    if (e == cudaSuccess && P == 1) {
        h->host.W_ctrl.assign(W_ctrl, W_ctrl + KX * A);
        h->host.b_ctrl.assign(b_ctrl, b_ctrl + A);
        wm_fused_free(h);
        const wm_weights hv = h->host.view();
        e = wm_fused_pack(h, &hv);
        if (e == cudaSuccess) e = wm_small_repack(h);
    }
    if (e != cudaSuccess) return cuda_fail(h, e, "wm_set_controllers");
    h->P = P;
    h->E = E;
    return WM_OK;
}

wm_status wm_returns(wm_handle *h, int B, int T, unsigned long long episode_offset, float gamma,
                     int stop_at_done, const float *rewards, const uint8_t *done, const float *bootstrap,
                     float *returns, float *fitness, void *cuda_stream) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->err.clear();
    if (B < 0 || T < 0 || B > (1 << 22)) return fail(h, WM_ERR_INVALID_ARG, "B must be in [0, 2^22], T >= 0");
    if (B > 0 && T > 0 && (!rewards || !done || !returns))
        return fail(h, WM_ERR_INVALID_ARG, "rewards, done and returns are required");
    if (!(gamma >= 0.f && gamma <= 1.f)) return fail(h, WM_ERR_INVALID_ARG, "gamma must be in [0, 1]");
    cudaStream_t s = (cudaStream_t)cuda_stream;
    cudaError_t e = cudaSetDevice(h->device);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
    const size_t b = (size_t)B, t = (size_t)T;
    const float *r = rewards, *bs = bootstrap;
    const uint8_t *d = done;
    float *ret = returns, *fit = fitness;
    Stager st;
    st.add((void **)&r, rewards, t * b * 4, false);
    st.add((void **)&d, done, t * b, false);
    st.add((void **)&bs, bootstrap, b * 4, false);
    st.add((void **)&ret, returns, t * b * 4, true);
    st.add((void **)&fit, fitness, (size_t)h->P * 4, true);
    e = grow(&h->ws, &h->ws_bytes, wm_returns_ws(h, B));
    if (e != cudaSuccess) return cuda_fail(h, e, "workspace");
    if ((e = st.begin(h, T, false, s)) != cudaSuccess) return cuda_fail(h, e, "staging inputs");
    e = wm_returns_launch(h, B, T, episode_offset, gamma, stop_at_done, r, d, bs, ret, fit, h->ws, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "returns launch");
    if ((e = st.end(s)) != cudaSuccess) return cuda_fail(h, e, "staging outputs");
    return WM_OK;
}

wm_status wm_mdn_nll_backward(wm_handle *h, int N, int T, const float *z_seq, const int32_t *actions,
                              const int32_t *lengths, float *nll, const wm_grads *grads, void *cuda_stream) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->err.clear();
    const wm_config &c = h->cfg;
    if (c.n_xfers > 0) return fail(h, WM_ERR_UNSUPPORTED, "the training step takes flat-action models only");
    if (N < 0 || T < 0 || N > (1 << 22)) return fail(h, WM_ERR_INVALID_ARG, "N must be in [0, 2^22], T >= 0");
    if (!grads || !grads->W_lstm || !grads->b_lstm || !grads->W_mdn || !grads->b_mdn)
        return fail(h, WM_ERR_INVALID_ARG, "all four gradient arrays are required");
    if (N > 0 && T > 0 && (!z_seq || !actions)) return fail(h, WM_ERR_INVALID_ARG, "z_seq and actions are required");
    const size_t Z = c.z_dim, A = c.a_dim, H = c.h_dim, M = h->M, n = (size_t)N, t = (size_t)T;
    if (actions && is_host_ptr(actions))
        for (size_t i = 0; i < n * t; ++i)
            if (actions[i] >= c.a_dim) return fail(h, WM_ERR_INVALID_ARG, "action index >= A");
    if (lengths && is_host_ptr(lengths))
        for (size_t i = 0; i < n; ++i)
            if (lengths[i] < 0 || lengths[i] > T) return fail(h, WM_ERR_INVALID_ARG, "length outside [0, T]");
    cudaStream_t s = (cudaStream_t)cuda_stream;
    cudaError_t e = cudaSetDevice(h->device);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");
    if ((e = wm_bw_prepare(h)) != cudaSuccess) return cuda_fail(h, e, "training-step set-up (cuBLAS)");

    const float *zs = z_seq;
    const int32_t *ac = actions, *ln = lengths;
    float *nl = nll;
    wm_grads g = *grads;
    Stager st;
    st.add((void **)&zs, z_seq, (t + 1) * n * Z * 4, false);
    st.add((void **)&ac, actions, t * n * 4, false);
    st.add((void **)&ln, lengths, n * 4, false);
    st.add((void **)&nl, nll, n * 4, true);
    st.add((void **)&g.W_lstm, grads->W_lstm, (Z + A + H) * 4 * H * 4, true);
    st.add((void **)&g.b_lstm, grads->b_lstm, 4 * H * 4, true);
    st.add((void **)&g.W_mdn, grads->W_mdn, H * M * 4, true);
    st.add((void **)&g.b_mdn, grads->b_mdn, M * 4, true);

    // the forward: the teacher-forced pass, keeping h, c and the head outputs of every row
    const int path = pick_path(h, N);
    if (path == WM_PATH_FUSED && !wm_fused_supported(h, N))
        return fail(h, WM_ERR_UNSUPPORTED, "the fused family does not take this model / batch");
    if (path == WM_PATH_TENSOR && !wm_tc_supported(h))
        return fail(h, WM_ERR_UNSUPPORTED, "the tensor family does not take this model");
    size_t need = path == WM_PATH_FUSED ? wm_fused_nll_ws(h, N) : path == WM_PATH_TENSOR ? wm_tc_ws(h, N, T)
                                                                                      : wm_step_nll_ws(h, N);
    if ((e = grow(&h->ws, &h->ws_bytes, need)) != cudaSuccess) return cuda_fail(h, e, "workspace");
    if ((e = grow(&h->bws, &h->bws_bytes, wm_bw_ws(h, N, T))) != cudaSuccess)
        return cuda_fail(h, e, "training-step workspace");
    if ((e = st.begin(h, T, false, s)) != cudaSuccess) return cuda_fail(h, e, "staging inputs");
    wm_nll_dev a{};
    a.N = N; a.T = T; a.z_seq = zs; a.actions = ac; a.lengths = ln;
    float *nll_ws;
    void *tail;
    wm_bw_carve(h, N, T, h->bws, &a.h_seq, &a.c_seq, &a.mdn_seq, &nll_ws, &tail);
    a.nll = nl ? nl : nll_ws;
    int fwd_launches = 0;
    if (N > 0 && T > 0) {
        if (path == WM_PATH_FUSED) e = wm_fused_nll(h, a, h->ws, s);
        else if (path == WM_PATH_TENSOR) e = wm_tc_nll(h, a, h->ws, s);
        else e = wm_step_nll(h, a, h->ws, s);
        if (e != cudaSuccess) return cuda_fail(h, e, "training-step forward");
        fwd_launches = path == WM_PATH_STEPWISE ? 2 + 4 * T : h->last_launches;
    } else if (nl && N > 0) {
        if ((e = cudaMemsetAsync(nl, 0, n * 4, s)) != cudaSuccess) return cuda_fail(h, e, "nll");
    }
    h->last_path = path;
    h->last_launches = fwd_launches;
    e = wm_bw_launch(h, N, T, zs, ac, ln, g, a.h_seq, a.c_seq, a.mdn_seq, tail, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "training-step backward");
    if ((e = st.end(s)) != cudaSuccess) return cuda_fail(h, e, "staging outputs");
    return WM_OK;
}

wm_status wm_mdn_nll(wm_handle *h, int N, int T, const float *z_seq, const int32_t *actions,
                     const int32_t *lengths, float *nll, float *h_seq, float *c_seq, float *mdn_seq,
                     void *cuda_stream) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->err.clear();
    if (N < 0 || T < 0 || N > (1 << 22)) return fail(h, WM_ERR_INVALID_ARG, "N must be in [0, 2^22], T >= 0");
    if (N > 0 && (!z_seq || !nll || (T > 0 && !actions)))
        return fail(h, WM_ERR_INVALID_ARG, "z_seq, actions and nll are required");
    const wm_config &c = h->cfg;
    if (c.n_xfers > 0)
        return fail(h, WM_ERR_UNSUPPORTED, "teacher-forced scoring takes flat-action models only");
    const size_t Z = c.z_dim, H = c.h_dim, M = h->M, n = (size_t)N, t = (size_t)T;
    if (actions && is_host_ptr(actions))
        for (size_t i = 0; i < n * t; ++i)
            if (actions[i] >= c.a_dim) return fail(h, WM_ERR_INVALID_ARG, "action index >= A");
    if (lengths && is_host_ptr(lengths))
        for (size_t i = 0; i < n; ++i)
            if (lengths[i] < 0 || lengths[i] > T) return fail(h, WM_ERR_INVALID_ARG, "length outside [0, T]");
    cudaStream_t s = (cudaStream_t)cuda_stream;
    cudaError_t e = cudaSetDevice(h->device);
    if (e != cudaSuccess) return cuda_fail(h, e, "cudaSetDevice");

    wm_nll_dev a{};
    a.N = N; a.T = T;
    Stager st;
    st.add((void **)&a.z_seq, z_seq, (t + 1) * n * Z * 4, false);
    st.add((void **)&a.actions, actions, t * n * 4, false);
    st.add((void **)&a.lengths, lengths, n * 4, false);
    st.add((void **)&a.nll, nll, n * 4, true);
    st.add((void **)&a.h_seq, h_seq, t * n * H * 4, true);
    st.add((void **)&a.c_seq, c_seq, t * n * H * 4, true);
    st.add((void **)&a.mdn_seq, mdn_seq, t * n * M * 4, true);

    int path = pick_path(h, N);
    if (path == WM_PATH_FUSED && !wm_fused_supported(h, N))
        return fail(h, WM_ERR_UNSUPPORTED, "the fused family does not take this model / batch");
    if (path == WM_PATH_TENSOR && !wm_tc_supported(h))
        return fail(h, WM_ERR_UNSUPPORTED, "the tensor family does not take this model");
    size_t need = path == WM_PATH_FUSED ? wm_fused_nll_ws(h, N) : path == WM_PATH_TENSOR ? wm_tc_ws(h, N, T)
                                                                                      : wm_step_nll_ws(h, N);
    e = grow(&h->ws, &h->ws_bytes, need);
    if (e != cudaSuccess) return cuda_fail(h, e, "workspace");
    if ((e = st.begin(h, T, false, s)) != cudaSuccess) return cuda_fail(h, e, "staging inputs");
    if (path == WM_PATH_FUSED)
        e = wm_fused_nll(h, a, h->ws, s);
    else if (path == WM_PATH_TENSOR)
        e = wm_tc_nll(h, a, h->ws, s);
    else
        e = wm_step_nll(h, a, h->ws, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "nll launch");
    h->last_path = path;
    if (path == WM_PATH_STEPWISE) h->last_launches = N == 0 ? 0 : 2 + 4 * T;
    if ((e = st.end(s)) != cudaSuccess) return cuda_fail(h, e, "staging outputs");
    return WM_OK;
}

}  // extern "C"
