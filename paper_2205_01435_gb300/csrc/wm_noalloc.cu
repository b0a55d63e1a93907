// wm_noalloc.cu -- wm_rollout_noalloc: the stepwise dream rollout running on a
// fixed scratch area that is part of the library image, so the call itself
// never allocates device memory.
//
// Who needs it: callers that must not call cudaMalloc / cudaFree while they
// run -- code issued during CUDA stream capture, real-time loops where an
// allocation (and the device-wide synchronisation cudaFree implies) would
// stall other work, and hosts whose memory is entirely owned by another
// allocator.  wm_rollout grows a per-handle workspace on demand (which can
// synchronise the device and allocate); this entry point uses
// g_wm_noalloc_scratch below instead.
//
// The scratch array is a file-scope __device__ variable: every GPU that loads
// this library holds WM_NOALLOC_SCRATCH_BYTES of it until the process exits.
// All calls share it, so two calls that overlap on the GPU race on it.  Each
// call re-initialises the parts that must start from a known value (the
// recurrent state h, c and the frozen flags, in k_init_state) before use; the
// rest is fully written before it is read.
#include <mutex>

#include "wm_internal.h"

static __device__ __align__(256) unsigned char g_wm_noalloc_scratch[WM_NOALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
void *g_scratch_ptr[kMaxDevices];  // device address of the array, per device

// In host code g_wm_noalloc_scratch names a host-side stand-in, not the device
// array, so the address kernels need is looked up once per device (with that
// device current) and cached.
cudaError_t scratch_for_device(int dev, void **out) {
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_setup_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_wm_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return cudaSuccess;
}

bool device_accessible(const void *p) {
    if (!p) return true;
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

wm_status fail(wm_handle *h, wm_status st, const char *msg) {
    h->err = msg;
    return st;
}

}  // namespace

extern "C" wm_status wm_rollout_noalloc(wm_handle *h, int B, int T, unsigned long long episode_offset,
                                        unsigned int t0, const wm_rollout_io *io, void *cuda_stream) {
    if (!h) return WM_ERR_INVALID_ARG;
    h->err.clear();
    if (!io) return fail(h, WM_ERR_INVALID_ARG, "io is NULL");
    if (B < 0 || T < 0) return fail(h, WM_ERR_INVALID_ARG, "B and T must be >= 0");
    if (B > 0 && (!io->z0 || !io->z_out || (T > 0 && (!io->actions || !io->rewards || !io->done))))
        return fail(h, WM_ERR_INVALID_ARG, "z0, z_out, actions, rewards and done are required");
    if ((unsigned long long)t0 + (unsigned long long)T > 0x100000000ull)
        return fail(h, WM_ERR_INVALID_ARG, "t0 + T overflows the 32-bit Philox step counter");
    const size_t need = wm_step_rollout_ws(h, B);
    if (need > (size_t)WM_NOALLOC_SCRATCH_BYTES)
        return fail(h, WM_ERR_INVALID_ARG,
                    "batch too large for wm_rollout_noalloc: its scratch exceeds "
                    "WM_NOALLOC_SCRATCH_BYTES (use a smaller B, or wm_rollout)");
    const bool shaped = h->cfg.reward_mode == WM_REWARD_SHAPED;
    if (shaped && B > 0 && (!io->rt0 || !io->mem0))
        return fail(h, WM_ERR_INVALID_ARG, "the shaped reward needs rt0 and mem0");
    const void *ptrs[] = {io->z0, io->h0, io->c0, io->done0, io->mask, io->z_out, io->actions,
                          io->rewards, io->done, io->h_final, io->c_final, io->h_seq, io->c_seq,
                          io->mdn_seq, io->comp_seq, shaped ? io->rt0 : nullptr,
                          shaped ? io->mem0 : nullptr, shaped ? io->rt_seq : nullptr,
                          shaped ? io->mem_seq : nullptr, io->logp_seq,
                          h->cfg.value_head ? io->value_seq : nullptr,
                          h->cfg.n_xfers > 0 ? io->loc_mask : nullptr,
                          h->cfg.n_xfers > 0 ? io->loc_actions : nullptr};
    for (const void *p : ptrs)
        if (!device_accessible(p))
            return fail(h, WM_ERR_INVALID_ARG,
                        "wm_rollout_noalloc takes device (or managed) memory only: host arrays "
                        "would need staging buffers");
    cudaError_t e = cudaSetDevice(h->device);
    void *scratch = nullptr;
    if (e == cudaSuccess) e = scratch_for_device(h->device, &scratch);
    if (e != cudaSuccess) return fail(h, WM_ERR_CUDA, "scratch set-up (cudaGetSymbolAddress) failed");

    wm_rollout_dev a{};
    a.B = B; a.T = T; a.ep0 = episode_offset; a.t0 = t0;
    a.z0 = io->z0; a.h0 = io->h0; a.c0 = io->c0; a.done0 = io->done0; a.mask = io->mask;
    a.z_out = io->z_out; a.actions = io->actions; a.rewards = io->rewards; a.done = io->done;
    a.h_final = io->h_final; a.c_final = io->c_final; a.h_seq = io->h_seq; a.c_seq = io->c_seq;
    a.mdn_seq = io->mdn_seq; a.comp_seq = io->comp_seq;
    if (shaped) {
        a.rt0 = io->rt0; a.mem0 = io->mem0; a.rt_seq = io->rt_seq; a.mem_seq = io->mem_seq;
    }
    a.logp_seq = io->logp_seq;
    a.value_seq = h->cfg.value_head ? io->value_seq : nullptr;
    if (h->cfg.n_xfers > 0) {
        a.loc_mask = io->loc_mask;
        a.loc_actions = io->loc_actions;
    }
    e = wm_step_rollout(h, a, scratch, (cudaStream_t)cuda_stream);
    if (e != cudaSuccess) return fail(h, WM_ERR_CUDA, "wm_rollout_noalloc launch failed");
    h->last_path = WM_PATH_STEPWISE;
    h->last_launches = B == 0 ? 0 : 1 + (h->P > 1 ? 5 : 4) * T + ((a.h_final || a.c_final) ? 1 : 0);
    return WM_OK;
}
