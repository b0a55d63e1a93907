"""The timeout path of the fused and tensor-core kernels.

Every wait inside those kernels is bounded; when one gives up, the kernel records
WM_ERR_TIMEOUT in the device status word, stops issuing work, lets nothing of its own
stay in flight and frees its TMEM, and wm_sync reports it.  wm_inject_wait_timeout
makes the next call's first kernel wait on a barrier that nothing completes (before
it issues any MMA or copy), so the path runs without faulting or hanging the GPU.
After the failed call the handle must be usable: the status clears on wm_sync and the
next call matches the oracle."""
import numpy as np
import pytest
import torch

import synth
from parity import check_rollout, check_teacher

pytestmark = pytest.mark.gpu

WM_ERR_TIMEOUT = 4
POLLS = 1 << 12


@pytest.fixture(scope="module")
def wm():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2205_01435_gb300 as pkg
    return pkg.load()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _expect_timeout(wm, m):
    with pytest.raises(wm.WMError) as e:
        m.sync()
    assert e.value.status == WM_ERR_TIMEOUT
    m.sync()  # the status word was cleared


@pytest.mark.parametrize("name,path,B,T", [("small_bf16", "fused", 256, 4), ("tiny_fp32", "fused", 40, 4),
                                            ("small_bf16", "tensor", 300, 3)])
def test_rollout_wait_runs_out_then_recovers(wm, orc, name, path, B, T):
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name, B=B, T=T)
    m = wm.WorldModel(dict(cfg, path=path), w)
    zc, mc = _cuda(z0), _cuda(mask)
    m.inject_wait_timeout(POLLS)
    m.rollout(zc, T, mask=mc)
    assert m.last_path == path
    _expect_timeout(wm, m)
    # one shot: the next call runs normally and matches the oracle
    g = m.rollout(zc, T, mask=mc, want_seq=True)
    m.sync()
    r = check_rollout(g, cfg, w, z0, mask, orc=orc)
    assert r["compared"] == B * T
    # polls = 0 clears a pending injection without a call
    m.inject_wait_timeout(POLLS)
    m.inject_wait_timeout(0)
    g2 = m.rollout(zc, T, mask=mc, want_seq=True)
    m.sync()
    for k in ("z", "actions", "rewards", "done"):
        assert torch.equal(g[k], g2[k]), k
    m.close()


@pytest.mark.parametrize("name,path", [("small_bf16", "fused"), ("tiny_fp32", "fused"),
                                       ("small_bf16", "tensor")])
def test_scoring_wait_runs_out_then_recovers(wm, orc, name, path):
    cfg = synth.model_config(name)
    w = synth.weights(cfg)
    N, T = 200, 5
    zs, acts, _ = synth.teacher_inputs(N, T, cfg["z_dim"], cfg["a_dim"], seed=5)
    m = wm.WorldModel(dict(cfg, path=path), w)
    m.inject_wait_timeout(POLLS)
    m.mdn_nll(_cuda(zs), _cuda(acts))
    assert m.last_path == path
    _expect_timeout(wm, m)
    g = m.mdn_nll(_cuda(zs), _cuda(acts), want_seq=True)
    m.sync()
    o = orc.mdn_nll(cfg, w, zs, acts, want_seq=True)
    check_teacher({k: v.cpu().numpy() for k, v in g.items()}, o, cfg["precision"])
    m.close()


def test_stepwise_ignores_the_injection(wm, orc):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32")
    m = wm.WorldModel(dict(cfg, path="stepwise"), w)
    m.inject_wait_timeout(POLLS)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    m.sync()  # no status: the stepwise family has no waits
    check_rollout(g, cfg, w, z0, mask, orc=orc)
    m.close()
