// wm_fused.cu -- single-launch fused family (placeholder until the kernel lands).
#include "wm_internal.h"

int wm_fused_supported(const wm_handle *, int) { return 0; }
cudaError_t wm_fused_pack(wm_handle *h, const wm_weights *) { h->fused.ok = 0; return cudaSuccess; }
void wm_fused_free(wm_handle *) {}
cudaError_t wm_fused_rollout(const wm_handle *, const wm_rollout_dev &, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t wm_fused_nll(const wm_handle *, const wm_nll_dev &, void *, cudaStream_t) { return cudaErrorNotSupported; }
size_t wm_fused_nll_ws(const wm_handle *, int) { return 0; }
