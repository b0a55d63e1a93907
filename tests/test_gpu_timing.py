"""Per-kernel timing (wm_set_timing / wm_kernel_time): every launch of a call is
counted once under its kernel class, and the per-class device times add up to
no more than the call's own event-timed duration."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

CASES = [  # workload, path, B, T, classes the call must launch
    ("tiny_fp32", "stepwise", 16, 5, {"step_gemm", "step_cell", "step_sample", "aux"}),
    ("small_bf16", "fused", 256, 6, {"fused", "aux"}),
    ("tiny_fp32", "fused", 16, 5, {"fused_small"}),
    ("mid_bf16", "tensor", 384, 4, {"tc_ctrl", "tc_gates", "tc_heads", "aux"}),
]


@pytest.mark.parametrize("name,path,B,T,classes", CASES)
def test_kernel_times_cover_every_launch(name, path, B, T, classes):
    import paper_2205_01435_gb300 as pkg
    wm = pkg.load()
    cfg, w, z0, mask, _, _ = synth.rollout_inputs(name, B=B, T=T)
    cfg["path"] = path
    model = wm.WorldModel(cfg, w)
    z0d = torch.from_numpy(z0).cuda()
    md = torch.from_numpy(mask).cuda()
    model.rollout(z0d, T, md)  # untimed: workspace growth, first-launch set-up
    torch.cuda.synchronize()
    assert model.kernel_times() == {}  # timing is off by default
    model.set_timing(True)
    s = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    model.rollout(z0d, T, md)
    b.record(s)
    torch.cuda.synchronize()
    assert model.last_path == path
    kt = model.kernel_times()
    assert set(kt) == classes, kt
    assert sum(n for _, n in kt.values()) == model.last_launches
    assert all(ms > 0 for ms, _ in kt.values())
    assert sum(ms for ms, _ in kt.values()) <= a.elapsed_time(b) * 1.01 + 0.01
    # reading folds the events in once; a second read returns the same totals
    assert model.kernel_times() == kt
    model.set_timing(False)
    model.rollout(z0d, T, md)
    torch.cuda.synchronize()
    assert model.kernel_times() == kt  # nothing recorded while off
    model.set_timing(True)  # re-enabling clears the totals
    assert model.kernel_times() == {}
    model.close()
