"""wm_rollout_noalloc, the entry point for callers that cannot allocate device
memory while they run (stream capture, real-time loops, hosts whose GPU memory
belongs to another allocator): it must give the same results as wm_rollout on
two calls in a row, reject batches whose scratch would not fit its fixed array,
and reject host arrays.  This file is named so that pytest collects it last."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

TOL = 1e-4  # the fp32-path value tolerance of the parity tests


@pytest.fixture(scope="module")
def wm():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2205_01435_gb300 as pkg
    return pkg.load()


def _outputs(B, T, cfg, dev="cuda"):
    Z, H, K = cfg["z_dim"], cfg["h_dim"], cfg["k_mix"]
    return {"z_out": torch.empty((T + 1, B, Z), device=dev),
            "actions": torch.empty((T, B), dtype=torch.int32, device=dev),
            "rewards": torch.empty((T, B), device=dev),
            "done": torch.empty((T, B), dtype=torch.uint8, device=dev),
            "h_final": torch.empty((B, H), device=dev), "c_final": torch.empty((B, H), device=dev),
            "h_seq": torch.empty((T, B, H), device=dev), "c_seq": torch.empty((T, B, H), device=dev),
            "mdn_seq": torch.empty((T, B, 3 * K * Z), device=dev),
            "comp_seq": torch.empty((T, B, Z), dtype=torch.uint8, device=dev)}


def _compare(ref: dict, got: dict):
    for k in ("actions", "done", "comp_seq"):
        assert torch.equal(ref[k], got[k]), k
    for k in ("z_out", "rewards", "h_final", "c_final", "h_seq", "c_seq", "mdn_seq"):
        assert float((ref[k] - got[k]).abs().max()) <= TOL, k


def test_noalloc_matches_wm_rollout_on_two_calls(wm):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32")
    cfg = dict(cfg, done_terminates=1, path="stepwise")
    m = wm.WorldModel(cfg, w)
    stream = torch.cuda.current_stream().cuda_stream
    calls = [
        dict(B=B, T=T, ep=0, t0=0, z0=z0, mask=mask, h0=None, c0=None, done0=None),
        # second call: other episodes, a resumed state and some already-frozen episodes,
        # so stale scratch from the first call would show
        dict(B=11, T=7, ep=1000, t0=5, z0=synth.z0(11, cfg["z_dim"], seed=8),
             mask=synth.mask(7, 11, cfg["a_dim"], 0.5, seed=8),
             h0=np.random.default_rng(8).standard_normal((11, cfg["h_dim"])).astype(np.float32),
             c0=np.random.default_rng(9).standard_normal((11, cfg["h_dim"])).astype(np.float32),
             done0=(np.arange(11) % 4 == 0).astype(np.uint8)),
    ]
    for c in calls:
        io_in = {k: (None if c[k] is None else torch.from_numpy(np.ascontiguousarray(c[k])).cuda())
                 for k in ("z0", "mask", "h0", "c0", "done0")}
        ref = _outputs(c["B"], c["T"], cfg)
        got = _outputs(c["B"], c["T"], cfg)
        for v in got.values():
            v.fill_(7)  # garbage the entry point must overwrite
        wm.wm_rollout(m.h, c["B"], c["T"], c["ep"], c["t0"], dict(io_in, **ref), stream)
        wm.wm_rollout_noalloc(m.h, c["B"], c["T"], c["ep"], c["t0"], dict(io_in, **got), stream)
        torch.cuda.synchronize()
        assert m.last_path == "stepwise"
        _compare(ref, got)


def test_noalloc_rejects_oversize_and_host_arrays(wm):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("small_bf16", B=4096, T=2)
    m = wm.WorldModel(cfg, w)
    out = _outputs(4096, 2, cfg)
    io = dict(z0=torch.from_numpy(z0).cuda(), mask=torch.from_numpy(mask).cuda(), **out)
    with pytest.raises(wm.WMError) as ei:
        wm.wm_rollout_noalloc(m.h, 4096, 2, 0, 0, io)
    assert ei.value.status == wm.WM_ERR_INVALID_ARG
    host = dict(io, z0=torch.from_numpy(z0[:8]))
    with pytest.raises(wm.WMError) as ei:
        wm.wm_rollout_noalloc(m.h, 8, 2, 0, 0, host)
    assert ei.value.status == wm.WM_ERR_INVALID_ARG
