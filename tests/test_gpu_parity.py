"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs and Philox noise.  Rules and tolerances: tests/parity.py."""
import os

import numpy as np
import pytest
import torch

import synth
from parity import check_free_running, check_rollout, check_teacher, np_

pytestmark = pytest.mark.gpu
NT = os.cpu_count() or 1


@pytest.fixture(scope="module")
def wm():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2205_01435_gb300 as pkg
    return pkg.load()


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _spread(B, n):
    """n episode indices spread over [0, B), always including the first and last."""
    if n >= B:
        return np.arange(B)
    return np.unique(np.linspace(0, B - 1, n).round().astype(np.int64))


def _sub(g, idx):
    """The batch columns idx of a rollout's outputs (as numpy)."""
    return {k: (np_(v)[idx] if k in ("h_final", "c_final") else np_(v)[:, idx])
            for k, v in g.items() if v is not None}


PATHS_SMALL = ["stepwise", "auto"]


# ------------------------------------------------------------------ teacher-forced
TEACHER = [("tiny_fp32", None, 16, 20), ("small_bf16", None, 64, 50), ("mid_bf16", None, 32, 40),
           ("nll", "fp32", 512, 128), ("nll", "bf16", 512, 128), ("large_bf16", None, 8, 12)]


@pytest.mark.parametrize("name,prec,N,T", TEACHER)
@pytest.mark.parametrize("path", PATHS_SMALL)
def test_teacher_forced_parity(wm, orc, name, prec, N, T, path):
    cfg = synth.model_config(name)
    if prec:
        cfg["precision"] = prec
    w = synth.weights(cfg)
    zs, acts, _ = synth.teacher_inputs(N, T, cfg["z_dim"], cfg["a_dim"], seed=3)
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.mdn_nll(_cuda(zs), _cuda(acts), want_seq=True)
    torch.cuda.synchronize()
    idx = _spread(N, 96)
    o = orc.mdn_nll(cfg, w, zs[:, idx], acts[:, idx], want_seq=True, nthreads=NT)
    gs = {k: np_(v)[:, idx] if k != "nll" else np_(v)[idx] for k, v in g.items()}
    check_teacher(gs, o, cfg["precision"])
    if cfg["precision"] == "bf16":
        # the bf16 path also stays within 2e-2 of the plain fp32 oracle
        o32 = orc.mdn_nll(dict(cfg, precision="fp32"), w, zs[:, idx], acts[:, idx],
                          want_seq=True, nthreads=NT)
        for k in ("h_seq", "c_seq", "mdn_seq"):
            assert float(np.abs(gs[k] - o32[k]).max()) <= 2e-2


def test_teacher_forced_ragged_lengths_and_no_action(wm, orc):
    cfg = dict(synth.model_config("tiny_fp32"), z_dim=7, a_dim=45, h_dim=40, k_mix=3)
    w = synth.weights(cfg, seed=4)
    zs, acts, lens = synth.teacher_inputs(37, 9, 7, 45, seed=4, ragged=True)
    acts[::3, ::2] = -1
    lens[0], lens[1] = 0, 9
    for path in PATHS_SMALL:
        m = wm.WorldModel(dict(cfg, path=path), w)
        g = m.mdn_nll(_cuda(zs), _cuda(acts), lengths=_cuda(lens), want_seq=True)
        o = orc.mdn_nll(cfg, w, zs, acts, lengths=lens, want_seq=True)
        check_teacher({k: np_(v) for k, v in g.items()}, o, "fp32")


# ------------------------------------------------------------------ free-running rollouts
@pytest.mark.parametrize("path", PATHS_SMALL + ["tensor"])
def test_rollout_tiny_full(wm, orc, path):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32")
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    torch.cuda.synchronize()
    if path == "tensor":
        assert m.last_path == "tensor"
    r = check_rollout(g, cfg, w, z0, mask, orc=orc)
    assert r["compared"] == B * T
    # the fp32 path also follows the oracle's own free-running trajectory
    o = orc.rollout(cfg, w, z0, mask, T, want_seq=True)
    fr = check_free_running(g, o, cfg)
    assert fr["diverged"] <= 2, fr


@pytest.mark.parametrize("path", PATHS_SMALL)
def test_rollout_small_bf16(wm, orc, path):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("small_bf16")
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    torch.cuda.synchronize()
    idx = _spread(B, 48)
    r = check_rollout(_sub(g, idx), cfg, w, z0[idx], mask[:, idx], episodes=idx, orc=orc)
    assert r["compared"] == len(idx) * T


def _rollout_sampled(wm, orc, name, n_oracle, path="auto"):
    """Full-size GPU rollout; the sampled episodes are re-run alone on the GPU (bit-exact
    against the full batch, since episodes are independent) to get their per-step
    sequences, then compared with the oracle."""
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name)
    m = wm.WorldModel(dict(cfg, path=path), w)
    comp = torch.empty((T, B, cfg["z_dim"]), dtype=torch.uint8, device="cuda")
    full = m.rollout(_cuda(z0), T, mask=_cuda(mask), out={"comp_seq": comp})
    torch.cuda.synchronize()
    idx = _spread(B, n_oracle)
    parts = []
    for b in idx:
        one = m.rollout(_cuda(z0[b:b + 1]), T, mask=_cuda(mask[:, b:b + 1]), episode_offset=int(b),
                        want_seq=True)
        for k in ("z", "actions", "rewards", "done", "comp_seq"):
            assert torch.equal(one[k][:, 0], full[k][:, int(b)]), (k, int(b))
        parts.append({k: np_(v) for k, v in one.items()})
    assert m.last_path == path  # the re-runs used the same kernel family as the full batch
    g = {k: np.concatenate([p[k] for p in parts], axis=0 if k in ("h_final", "c_final") else 1)
         for k in parts[0]}
    r = check_rollout(g, cfg, w, z0[idx], mask[:, idx], episodes=idx, orc=orc)
    # every live step of every sampled episode is compared
    assert r["compared"] + r["frozen_steps"] == len(idx) * T
    return r


@pytest.mark.parametrize("path", ["tensor", "stepwise"])
def test_rollout_mid_bf16_sampled(wm, orc, path):
    r = _rollout_sampled(wm, orc, "mid_bf16", 24, path=path)
    print("mid_bf16 parity:", path, r)


@pytest.mark.parametrize("path", ["tensor", "stepwise"])
def test_rollout_large_bf16_sampled(wm, orc, path):
    r = _rollout_sampled(wm, orc, "large_bf16", 24, path=path)
    print("large_bf16 parity:", path, r)


# ------------------------------------------------------------------ edge cases
@pytest.mark.parametrize("path", PATHS_SMALL)
def test_ragged_shapes_and_flags(wm, orc, path):
    cfg = dict(synth.model_config("tiny_fp32"), z_dim=5, a_dim=33, h_dim=24, k_mix=3,
               noop_terminates=1, done_terminates=1)
    w = synth.weights(cfg, seed=9, std=0.3)
    B, T = 37, 7
    z0 = synth.z0(B, 5, seed=9)
    mask = synth.mask(T, B, 33, 0.4, seed=9)
    mask[2, 5] = 0  # all masked at one step
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=123456789012, t0=77,
                  want_seq=True)
    check_rollout(g, cfg, w, z0, mask, episodes=123456789012 + np.arange(B), t0=77, orc=orc)
    o = orc.rollout(cfg, w, z0, mask, T, episode_offset=123456789012, t0=77, want_seq=True)
    check_free_running(g, o, cfg)


@pytest.mark.parametrize("tau,sq", [(0.0, 0), (0.5, 1), (1.7, 0)])
def test_mixture_temperature(wm, orc, tau, sq):
    cfg = dict(synth.model_config("tiny_fp32"), mdn_tau=tau, sigma_sqrt_tau=sq)
    cfg2, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32", T=8)
    m = wm.WorldModel(dict(cfg, path="auto"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    check_rollout(g, cfg, w, z0, mask, orc=orc)
    o = orc.rollout(cfg, w, z0, mask, T, want_seq=True)
    check_free_running(g, o, cfg)


def test_sampled_controller(wm, orc):
    cfg = dict(synth.model_config("tiny_fp32"), ctrl_sample=1, ctrl_tau=0.8)
    _, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32")
    for path in PATHS_SMALL:
        m = wm.WorldModel(dict(cfg, path=path), w)
        g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
        check_rollout(g, cfg, w, z0, mask, orc=orc)
        o = orc.rollout(cfg, w, z0, mask, T, want_seq=True)
        check_free_running(g, o, cfg)


def test_empty_and_zero_length(wm):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32")
    m = wm.WorldModel(cfg, w)
    g = m.rollout(_cuda(z0[:0]), T, mask=_cuda(mask[:, :0]))
    assert g["z"].shape == (T + 1, 0, cfg["z_dim"])
    h0 = torch.randn(B, cfg["h_dim"], device="cuda")
    g = m.rollout(_cuda(z0), 0, h0=h0)
    torch.cuda.synchronize()
    assert torch.equal(g["z"][0].cpu(), torch.from_numpy(z0))
    assert torch.equal(g["h_final"], h0)
    n = m.mdn_nll(_cuda(np.zeros((1, 0, cfg["z_dim"]), np.float32)),
                  _cuda(np.zeros((0, 0), np.int32)))
    assert n["nll"].numel() == 0


@pytest.mark.parametrize("path,name", [("fused", "small_bf16"), ("fused", "tiny_fp32"),
                                       ("tensor", "small_bf16")])
def test_empty_and_zero_length_on_each_family(wm, path, name):
    """B = 0, T = 0 (state passes through unchanged) and N = 0 / T = 0 scoring on both
    members of the fused family and on the tensor-core family."""
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name, B=40, T=3)
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.rollout(_cuda(z0[:0]), T, mask=_cuda(mask[:, :0]))
    torch.cuda.synchronize()
    assert g["z"].shape == (T + 1, 0, cfg["z_dim"])
    h0 = torch.randn(B, cfg["h_dim"], device="cuda")
    c0 = torch.randn(B, cfg["h_dim"], device="cuda")
    g = m.rollout(_cuda(z0), 0, h0=h0, c0=c0)
    torch.cuda.synchronize()
    assert torch.equal(g["z"][0].cpu(), torch.from_numpy(z0))
    assert torch.equal(g["h_final"], h0) and torch.equal(g["c_final"], c0)
    zs = np.zeros((1, 4, cfg["z_dim"]), np.float32)
    n = m.mdn_nll(_cuda(zs), _cuda(np.zeros((0, 4), np.int32)))
    torch.cuda.synchronize()
    assert torch.equal(n["nll"].cpu(), torch.zeros(4))
    m.sync()


def test_invalid_arguments(wm):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("tiny_fp32")
    m = wm.WorldModel(cfg, w)
    with pytest.raises(wm.WMError) as ei:
        wm.wm_rollout(m.h, -1, T, 0, 0, {"z0": _cuda(z0)})
    assert ei.value.status == wm.WM_ERR_INVALID_ARG
    with pytest.raises(wm.WMError):
        wm.wm_rollout(m.h, B, T, 0, 0, {"z0": _cuda(z0)})  # outputs missing
    zs, acts, _ = synth.teacher_inputs(4, 3, cfg["z_dim"], cfg["a_dim"])
    acts[0, 0] = cfg["a_dim"]
    with pytest.raises(wm.WMError):
        m.mdn_nll(torch.from_numpy(zs), torch.from_numpy(acts))  # host actions are checked


@pytest.mark.parametrize("path,name", [("stepwise", "small_bf16"), ("fused", "small_bf16"),
                                       ("fused", "tiny_fp32"), ("tensor", "small_bf16")])
def test_device_teacher_inputs_out_of_range_are_reported(wm, orc, path, name):
    """On device arrays an action >= A or a length outside [0, T] is found by the kernels:
    wm_sync reports WM_ERR_INVALID_ARG once, the action counts as no action, the length is
    clamped, and the next call runs clean."""
    cfg = synth.model_config(name)
    w = synth.weights(cfg, seed=12)
    N, T = 40, 5
    zs, acts, _ = synth.teacher_inputs(N, T, cfg["z_dim"], cfg["a_dim"], seed=12)
    m = wm.WorldModel(dict(cfg, path=path), w)
    for bad_action in (True, False):
        a2, lens = acts.copy(), np.full(N, T, np.int32)
        if bad_action:
            a2[1, 3] = cfg["a_dim"] + 7
        else:
            lens[5] = T + 2
        g = m.mdn_nll(_cuda(zs), _cuda(a2), lengths=_cuda(lens))
        with pytest.raises(wm.WMError) as ei:
            m.sync()
        assert ei.value.status == wm.WM_ERR_INVALID_ARG
        assert m.last_path == path
        fixed_a = np.where(a2 >= cfg["a_dim"], -1, a2)
        o = orc.mdn_nll(cfg, w, zs, fixed_a, lengths=np.clip(lens, 0, T))
        check_teacher({"nll": g["nll"]}, o, cfg["precision"])
        m.mdn_nll(_cuda(zs), _cuda(acts))
        m.sync()  # the status was cleared


# ------------------------------------------------------------------ invariants of the GPU path
@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_sharding_is_bit_exact(wm, name):
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name, T=12)
    m = wm.WorldModel(cfg, w)
    zc, mc = _cuda(z0), _cuda(mask)
    full = m.rollout(zc, T, mask=mc)
    cut = B // 3
    lo = m.rollout(zc[:cut].contiguous(), T, mask=mc[:, :cut].contiguous())
    hi = m.rollout(zc[cut:].contiguous(), T, mask=mc[:, cut:].contiguous(), episode_offset=cut)
    for k in ("z", "actions", "rewards", "done"):
        assert torch.equal(torch.cat([lo[k], hi[k]], 1), full[k]), k


@pytest.mark.parametrize("name,path", [("tiny_fp32", "auto"), ("small_bf16", "auto"),
                                       ("small_bf16", "tensor")])  # tensor: compacted live episodes
def test_resume_is_bit_exact(wm, name, path):
    cfg, w, z0, mask, B, T = synth.rollout_inputs(name, T=10)
    cfg["done_terminates"] = 1
    m = wm.WorldModel(dict(cfg, path=path), w)
    zc, mc = _cuda(z0), _cuda(mask)
    full = m.rollout(zc, T, mask=mc)
    a = m.rollout(zc, 4, mask=mc[:4].contiguous())
    b = m.rollout(a["z"][4].contiguous(), T - 4, mask=mc[4:].contiguous(), t0=4,
                  h0=a["h_final"], c0=a["c_final"], done0=a["done"][3].contiguous())
    assert torch.equal(torch.cat([a["z"], b["z"][1:]]), full["z"])
    for k in ("actions", "rewards", "done"):
        assert torch.equal(torch.cat([a[k], b[k]]), full[k]), k


@pytest.mark.parametrize("kind", ["pinned", "pageable"])
@pytest.mark.parametrize("path,B,T,seq,done", [("auto", None, 6, False, 0),  # fused: copied whole around the call
                                               ("tensor", 700, 6, True, 0),   # per-step staging, every output kind
                                               ("tensor", 700, 6, True, 1),   # ... with compacted live episodes
                                               ("tensor", 700, 1, False, 0)])  # one step: copied whole
def test_host_buffers_match_device_buffers(wm, kind, path, B, T, seq, done):
    cfg, w, z0, mask, B, T = synth.rollout_inputs("small_bf16", B=B, T=T)
    cfg["done_terminates"] = done
    m = wm.WorldModel(dict(cfg, path=path), w)
    dev = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=seq)
    zh, mh = torch.from_numpy(z0), torch.from_numpy(mask)
    if kind == "pinned":
        zh, mh = zh.pin_memory(), mh.pin_memory()
    keys = ["z", "actions", "rewards", "done", "h_final", "c_final"]
    if seq:
        keys += ["h_seq", "c_seq", "mdn_seq", "comp_seq"]
    for _ in range(2):  # the second call reuses the staging buffer and its events
        host = m.rollout(zh, T, mask=mh, want_seq=seq)  # outputs allocated on the host, call syncs
        if path == "tensor":
            assert m.last_path == "tensor"
        for k in keys:
            assert not host[k].is_cuda
            assert torch.equal(host[k], dev[k].cpu()), k


# ------------------------------------------------------------------ the fused single-launch family
@pytest.mark.parametrize("cluster", [16, 8])
@pytest.mark.parametrize("flags", [dict(), dict(done_terminates=1, noop_terminates=1),
                                   dict(mdn_tau=0.0), dict(mdn_tau=0.5, sigma_sqrt_tau=1)])
def test_fused_against_oracle(wm, orc, flags, cluster):
    """Two clusters (the second one partly filled), resumed state, offsets, flags."""
    cfg = dict(synth.model_config("small_bf16"), fused_cluster=cluster, **flags)
    w = synth.weights(cfg, seed=5)
    B, T = 200, 9
    z0 = synth.z0(B, cfg["z_dim"], seed=5)
    mask = synth.mask(T, B, cfg["a_dim"], 0.3, seed=5)
    mask[3, 17] = 0  # no valid action for one episode at one step
    rng = np.random.default_rng(5)
    h0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    done0 = (np.arange(B) % 37 == 0).astype(np.uint8)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=77, t0=3, h0=_cuda(h0),
                  c0=_cuda(c0), done0=_cuda(done0), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    r = check_rollout(g, cfg, w, z0, mask, episodes=77 + np.arange(B), t0=3, h0=h0, c0=c0,
                      done0=done0, orc=orc)
    print("fused", cluster, flags, r)


@pytest.mark.parametrize("cluster", [16, 8])
def test_fused_teacher_forced_ragged(wm, orc, cluster):
    cfg = dict(synth.model_config("small_bf16"), fused_cluster=cluster)
    w = synth.weights(cfg, seed=6)
    zs, acts, lens = synth.teacher_inputs(300, 11, cfg["z_dim"], cfg["a_dim"], seed=6, ragged=True)
    acts[2, ::5] = -1
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.mdn_nll(_cuda(zs), _cuda(acts), lengths=_cuda(lens), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    o = orc.mdn_nll(cfg, w, zs, acts, lengths=lens, want_seq=True, nthreads=NT)
    check_teacher({k: np_(v) for k, v in g.items()}, o, "bf16")


def test_fused_matches_stepwise_closely(wm):
    """Same model through both families: equal decisions and close values until an
    episode's first near-tie flip (the two families round differently)."""
    cfg, w, z0, mask, B, T = synth.rollout_inputs("small_bf16", T=20)
    a = wm.WorldModel(dict(cfg, path="fused"), w).rollout(_cuda(z0), T, mask=_cuda(mask))
    b = wm.WorldModel(dict(cfg, path="stepwise"), w).rollout(_cuda(z0), T, mask=_cuda(mask))
    torch.cuda.synchronize()
    act_eq = (a["actions"] == b["actions"]).cpu().numpy()             # [T, B]
    z_eq = ((a["z"][1:] - b["z"][1:]).abs().amax(-1) < 2e-2).cpu().numpy()
    ok = np.cumprod(act_eq & z_eq, axis=0)                           # 1 until first divergence
    assert ok.mean() > 0.95, ok.mean()


# ------------------------------------------------------------------ the fused family's small-batch member
SMALL_CASES = [
    ("fp32", dict()),
    ("fp32", dict(done_terminates=1, noop_terminates=1)),
    ("fp32", dict(ctrl_sample=1, ctrl_tau=0.7, mdn_tau=0.5, sigma_sqrt_tau=1)),
    ("fp32", dict(mdn_tau=0.0)),
    ("fp32", dict(reward_mode=1, done_terminates=1)),
    ("bf16", dict(ctrl_sample=1, ctrl_tau=1.0)),  # bf16, a controller the tcgen05 member does not take
]


@pytest.mark.parametrize("prec,flags", SMALL_CASES)
def test_fused_small_against_oracle(wm, orc, prec, flags):
    """The single-launch fp32 SIMT member on the tiny model: 13 clusters of 16 episodes (the
    last one partly filled), resumed state, frozen episodes, offsets, every flag; one launch."""
    cfg = dict(synth.model_config("tiny_fp32"), precision=prec, **flags)
    w = synth.weights(cfg, seed=21)
    B, T = 200, 9
    z0 = synth.z0(B, cfg["z_dim"], seed=21)
    mask = synth.mask(T, B, cfg["a_dim"], 0.5, seed=21)
    mask[3, 17] = 0  # no valid action for one episode at one step
    rng = np.random.default_rng(21)
    h0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    done0 = (np.arange(B) % 37 == 0).astype(np.uint8)
    extra, okw = {}, {}
    if flags.get("reward_mode") == 1:
        rt0, mem0 = synth.shaping_state(B, seed=21)
        extra = dict(rt0=_cuda(rt0), mem0=_cuda(mem0))
        okw = dict(rt0=rt0, mem0=mem0)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=91, t0=5, h0=_cuda(h0), c0=_cuda(c0),
                  done0=_cuda(done0), want_seq=True, **extra)
    torch.cuda.synchronize()
    assert m.last_path == "fused" and m.last_launches == 1
    assert int(g["actions"][3, 17]) == -1 or bool(done0[17])
    r = check_rollout(g, cfg, w, z0, mask, episodes=91 + np.arange(B), t0=5, h0=h0, c0=c0,
                      done0=done0, orc=orc, **okw)
    assert r["compared"] + r["frozen_steps"] == B * T
    print("fused small", prec, flags, r)
    # AUTO takes the same member for this batch: the same bits
    ga = wm.WorldModel(dict(cfg, path="auto"), w).rollout(
        _cuda(z0), T, mask=_cuda(mask), episode_offset=91, t0=5, h0=_cuda(h0), c0=_cuda(c0),
        done0=_cuda(done0), **extra)
    for k in ("z", "actions", "rewards", "done"):
        assert torch.equal(ga[k], g[k]), k


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_fused_small_teacher_forced_ragged(wm, orc, prec):
    """Scoring on the small-batch member: ragged lengths, no-action steps, a partial tile."""
    cfg = dict(synth.model_config("tiny_fp32"), precision=prec, ctrl_sample=1)
    w = synth.weights(cfg, seed=22)
    zs, acts, lens = synth.teacher_inputs(45, 13, cfg["z_dim"], cfg["a_dim"], seed=22, ragged=True)
    acts[4, ::3] = -1
    lens[0], lens[1] = 0, 13
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.mdn_nll(_cuda(zs), _cuda(acts), lengths=_cuda(lens), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused" and m.last_launches == 1
    o = orc.mdn_nll(cfg, w, zs, acts, lengths=lens, want_seq=True, nthreads=NT)
    check_teacher({k: np_(v) for k, v in g.items()}, o, prec)


def test_fused_small_scores_a_shaped_reward_model(wm, orc):
    """Scoring ignores the reward heads: a model with the runtime / memory heads of Eq. 2 scores
    on the small-batch member (no runtime / memory inputs) as on the stepwise family."""
    cfg = dict(synth.model_config("tiny_fp32"), reward_mode=1)
    w = synth.weights(cfg, seed=24)
    zs, acts, lens = synth.teacher_inputs(21, 6, cfg["z_dim"], cfg["a_dim"], seed=24, ragged=True)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.mdn_nll(_cuda(zs), _cuda(acts), lengths=_cuda(lens), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    o = orc.mdn_nll(cfg, w, zs, acts, lengths=lens, want_seq=True)
    check_teacher({k: np_(v) for k, v in g.items()}, o, "fp32")


@pytest.mark.parametrize("K,tau", [(1, 1.0), (32, 1.0), (32, 0.0), (7, 0.4)])
def test_fused_small_mixture_sizes(wm, orc, K, tau):
    """The mixture's warp reductions over K component lanes at the edges: one component (no
    reduction level), a full warp of 32, an odd K; argmax (tau = 0) and tempered draws."""
    cfg = dict(synth.model_config("tiny_fp32"), z_dim=6, a_dim=40, h_dim=48, k_mix=K, mdn_tau=tau,
               done_terminates=1)
    w = synth.weights(cfg, seed=25, std=0.2)
    B, T = 21, 7
    z0 = synth.z0(B, 6, seed=25)
    mask = synth.mask(T, B, 40, 0.5, seed=25)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    r = check_rollout(g, cfg, w, z0, mask, orc=orc)
    assert r["compared"] + r["frozen_steps"] == B * T
    zs, acts, lens = synth.teacher_inputs(B, T, 6, 40, seed=25, ragged=True)
    gn = m.mdn_nll(_cuda(zs), _cuda(acts), lengths=_cuda(lens), want_seq=True)
    torch.cuda.synchronize()
    o = orc.mdn_nll(cfg, w, zs, acts, lengths=lens, want_seq=True)
    check_teacher({k: np_(v) for k, v in gn.items()}, o, "fp32")


def test_fused_small_odd_shapes(wm, orc):
    """A model whose sizes divide nothing (Z=7, A=45, H=40, K=3): ranks own ragged slices of
    units, actions and dims, and some own none."""
    cfg = dict(synth.model_config("tiny_fp32"), z_dim=7, a_dim=45, h_dim=40, k_mix=3,
               done_terminates=1, noop_terminates=1, ctrl_sample=1, ctrl_tau=0.9)
    w = synth.weights(cfg, seed=23, std=0.3)
    B, T = 53, 11
    z0 = synth.z0(B, 7, seed=23)
    mask = synth.mask(T, B, 45, 0.4, seed=23)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=5, want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    r = check_rollout(g, cfg, w, z0, mask, episodes=5 + np.arange(B), orc=orc)
    assert r["compared"] + r["frozen_steps"] == B * T


def test_fused_small_bf16_sampled_controller(wm, orc):
    """The small bf16 model with a tempered-draw controller, which the tcgen05 member does not
    take: the fused family runs it on the small-batch member (bf16-rounded operands)."""
    cfg, w, z0, mask, B, T = synth.rollout_inputs("small_bf16", B=100, T=10)
    cfg.update(ctrl_sample=1, ctrl_tau=0.9)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused" and m.last_launches == 1
    r = check_rollout(g, cfg, w, z0, mask, orc=orc)
    assert r["compared"] == B * T


def test_fused_small_at_the_wave_limit(wm, orc):
    """The largest batch AUTO gives the small-batch member (at most 4 waves of 16-episode
    clusters, several tiles per SM over the call): parity on a spread of its episodes."""
    cfg, w, z0, mask, _, T = synth.rollout_inputs("tiny_fp32", B=1, T=6)
    m = wm.WorldModel(dict(cfg, path="auto"), w)
    nmax = None
    for B in range(16 * 64, 0, -16):  # find the limit by asking for the path
        zb = synth.z0(B, cfg["z_dim"], seed=31)
        mb = synth.mask(T, B, cfg["a_dim"], 0.5, seed=31)
        m.rollout(_cuda(zb), 1, mask=_cuda(mb[:1]))
        if m.last_path == "fused":
            nmax = B
            break
    assert nmax is not None and nmax >= 16 * 4, nmax
    z0 = synth.z0(nmax, cfg["z_dim"], seed=31)
    mask = synth.mask(T, nmax, cfg["a_dim"], 0.5, seed=31)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    idx = _spread(nmax, 40)
    r = check_rollout(_sub(g, idx), cfg, w, z0[idx], mask[:, idx], episodes=idx, orc=orc)
    assert r["compared"] == len(idx) * T


# ------------------------------------------------------------------ the tensor-core family
@pytest.mark.parametrize("name,flags", [("mid_bf16", dict()), ("large_bf16", dict()),
                                        ("small_bf16", dict(mdn_tau=0.0)),
                                        ("small_bf16", dict(mdn_tau=0.6, sigma_sqrt_tau=1,
                                                            noop_terminates=1, done_terminates=1)),
                                        ("mid_bf16", dict(ctrl_sample=1, ctrl_tau=0.7)),
                                        # column groups starting mid-word of the action mask
                                        ("small_bf16", dict(a_dim=192, ctrl_sample=1, ctrl_tau=0.8)),
                                        ("small_bf16", dict(a_dim=64)),
                                        # an odd number of k-steps in the head GEMM (H / 64 = 5)
                                        ("small_bf16", dict(h_dim=320)),
                                        # fp32: three bf16 passes over K (hi/lo split operands)
                                        ("tiny_fp32", dict()),
                                        ("tiny_fp32", dict(ctrl_sample=1, ctrl_tau=0.8, done_terminates=1,
                                                           noop_terminates=1, mdn_tau=0.7)),
                                        ("mid_bf16", dict(precision="fp32", k_mix=5))])
def test_tensor_against_oracle(wm, orc, name, flags):
    """Two row tiles (the second partly filled), resumed state, offsets, flags."""
    cfg = dict(synth.model_config(name), **flags)
    w = synth.weights(cfg, seed=7)
    B, T = 200, 6
    z0 = synth.z0(B, cfg["z_dim"], seed=7)
    mask = synth.mask(T, B, cfg["a_dim"], synth.WORKLOADS[name]["mask_density"], seed=7)
    mask[2, 9] = 0
    rng = np.random.default_rng(7)
    h0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    done0 = (np.arange(B) % 41 == 0).astype(np.uint8)
    m = wm.WorldModel(dict(cfg, path="tensor"), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=99, t0=11, h0=_cuda(h0),
                  c0=_cuda(c0), done0=_cuda(done0), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "tensor"
    r = check_rollout(g, cfg, w, z0, mask, episodes=99 + np.arange(B), t0=11, h0=h0, c0=c0,
                      done0=done0, orc=orc)
    print("tensor", name, flags, r)


@pytest.mark.parametrize("name,prec,N,T", [("mid_bf16", None, 300, 9), ("nll", "bf16", 512, 128),
                                           ("large_bf16", None, 130, 5), ("nll", "fp32", 512, 128),
                                           ("tiny_fp32", None, 300, 20)])
def test_tensor_teacher_forced(wm, orc, name, prec, N, T):
    cfg = synth.model_config(name)
    if prec:
        cfg["precision"] = prec
    w = synth.weights(cfg, seed=8)
    zs, acts, lens = synth.teacher_inputs(N, T, cfg["z_dim"], cfg["a_dim"], seed=8, ragged=True)
    acts[1, ::7] = -1
    m = wm.WorldModel(dict(cfg, path="tensor"), w)
    g = m.mdn_nll(_cuda(zs), _cuda(acts), lengths=_cuda(lens), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "tensor"
    idx = _spread(N, 96)
    o = orc.mdn_nll(cfg, w, zs[:, idx], acts[:, idx], lengths=lens[idx], want_seq=True, nthreads=NT)
    gs = {k: np_(v)[:, idx] if k != "nll" else np_(v)[idx] for k, v in g.items()}
    check_teacher(gs, o, "bf16")


@pytest.mark.parametrize("name,T,B,flags", [("large_bf16", 4, None, {}), ("mid_bf16", 8, None, {}),
                                            # odd k-step counts: gates (Z + H) / 64 = 6, heads H / 64 = 5
                                            ("small_bf16", 4, 16384, dict(h_dim=320))])
def test_tensor_full_batch_is_deterministic(wm, name, T, B, flags):
    """Repeated full-batch calls are bit-identical (the persistent kernels' shared-memory
    staging and operand ring have no race: a missing ordering there shows up as run-to-run
    differences).  Each CTA pair runs several tiles, so every ring slot is reused."""
    cfg, _, z0, mask, B, T = synth.rollout_inputs(name, B=B, T=T)
    cfg = dict(cfg, **flags)
    w = synth.weights(cfg, seed=3)
    m = wm.WorldModel(dict(cfg, path="tensor"), w)
    zc, mc = _cuda(z0), _cuda(mask)
    first = m.rollout(zc, T, mask=mc)
    for _ in range(2):
        again = m.rollout(zc, T, mask=mc)
        torch.cuda.synchronize()
        for k in ("z", "actions", "rewards", "done", "h_final", "c_final"):
            assert torch.equal(first[k], again[k]), k
    m.sync()


# ------------------------------------------------------------------ shaped reward (Eq. 1 / Eq. 2)
@pytest.mark.parametrize("path,name,flags", [("stepwise", "tiny_fp32", dict(done_terminates=1)),
                                             ("auto", "small_bf16", dict()),
                                             ("tensor", "small_bf16", dict(done_terminates=1)),
                                             ("tensor", "large_bf16", dict()),
                                             ("stepwise", "mid_bf16", dict(reward_alpha=1.0, reward_beta=0.0))])
def test_shaped_reward_against_oracle(wm, orc, path, name, flags):
    """Eq. 2 on the predicted runtime / memory heads, with an invalid step (-100), resumed
    state, offsets and frozen episodes."""
    cfg = dict(synth.model_config(name), reward_mode=1, **flags)
    w = synth.weights(cfg, seed=13)
    B, T = (16, 12) if name == "tiny_fp32" else (200, 6)
    z0 = synth.z0(B, cfg["z_dim"], seed=13)
    mask = synth.mask(T, B, cfg["a_dim"], synth.WORKLOADS[name]["mask_density"], seed=13)
    mask[0, 9] = 0  # no valid action at the first step (episode 9 is live then)
    rng = np.random.default_rng(13)
    h0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((B, cfg["h_dim"]))).astype(np.float32)
    done0 = (np.arange(B) % 37 == 5).astype(np.uint8)
    rt0, mem0 = synth.shaping_state(B, seed=13)
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=55, t0=4, h0=_cuda(h0), c0=_cuda(c0),
                  done0=_cuda(done0), rt0=_cuda(rt0), mem0=_cuda(mem0), want_seq=True)
    torch.cuda.synchronize()
    assert path == "auto" or m.last_path == path  # AUTO: the fused family's small-batch member
    assert int(g["actions"][0, 9]) == -1 and float(g["rewards"][0, 9]) == -100.0
    r = check_rollout(g, cfg, w, z0, mask, episodes=55 + np.arange(B), t0=4, h0=h0, c0=c0,
                      done0=done0, orc=orc, rt0=rt0, mem0=mem0)
    print("shaped", path, name, flags, r)
    # resumed in two calls: bit for bit the same
    a = m.rollout(_cuda(z0), 3, mask=_cuda(mask[:3]), episode_offset=55, t0=4, h0=_cuda(h0),
                  c0=_cuda(c0), done0=_cuda(done0), rt0=_cuda(rt0), mem0=_cuda(mem0), want_seq=True)
    d0b = torch.maximum(a["done"][2], _cuda(done0)) if cfg.get("done_terminates") else _cuda(done0)
    b = m.rollout(a["z"][3].contiguous(), T - 3, mask=_cuda(mask[3:]), episode_offset=55, t0=7,
                  h0=a["h_final"], c0=a["c_final"], done0=d0b,
                  rt0=a["rt_seq"][2].contiguous(), mem0=a["mem_seq"][2].contiguous(), want_seq=True)
    for k in ("rewards", "rt_seq", "mem_seq", "actions"):
        assert torch.equal(torch.cat([a[k], b[k]]), g[k]), k


# ------------------------------------------------------------------ population, log-probs, values, returns
@pytest.mark.parametrize("path,name,P,E,off,flags", [
    ("tensor", "small_bf16", 3, 256, 512, dict(ctrl_sample=1, ctrl_tau=0.8)),
    ("tensor", "mid_bf16", 2, 256, 0, dict(done_terminates=1)),
    ("stepwise", "tiny_fp32", 3, 5, 7, dict(ctrl_sample=1, ctrl_tau=1.2)),
    ("auto", "small_bf16", 4, 100, 0, dict()),  # E not a multiple of 256: not the tensor family
])
def test_population_logp_value_against_oracle(wm, orc, path, name, P, E, off, flags):
    """A population of controllers (episode e -> candidate (e / E) mod P), the log-prob of
    each action taken and the value head, step-anchored against the oracle."""
    cfg = dict(synth.model_config(name), value_head=1, **flags)
    w = synth.weights(cfg, seed=14)
    Wp, bp = synth.population(cfg, P, seed=14)
    B, T = (768, 5) if name != "tiny_fp32" else (16, 10)
    z0 = synth.z0(B, cfg["z_dim"], seed=14)
    mask = synth.mask(T, B, cfg["a_dim"], synth.WORKLOADS[name]["mask_density"], seed=14)
    m = wm.WorldModel(dict(cfg, path=path), w)
    m.set_controllers(Wp, bp, pop_group=E)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=off, want_seq=True, want_logp=True)
    torch.cuda.synchronize()
    if path != "auto":
        assert m.last_path == path
    else:
        assert m.last_path == "stepwise"
    ocfg = dict(cfg, pop_size=P, pop_group=E)
    r = check_rollout(g, ocfg, dict(w, W_ctrl=Wp, b_ctrl=bp), z0, mask, episodes=off + np.arange(B),
                      orc=orc)
    print("population", path, name, P, E, r)
    # every candidate acted
    cands = ((off + np.arange(B)) // E) % P
    assert len(set(cands.tolist())) == P
    # back to a single controller: the call matches the base model again
    m.set_controllers(w["W_ctrl"][None], w["b_ctrl"][None], pop_group=1)
    g1 = m.rollout(_cuda(z0[:300]), 3, mask=_cuda(mask[:3, :300]), want_seq=True, want_logp=True)
    check_rollout(g1, cfg, w, z0[:300], mask[:3, :300], orc=orc)


def test_fused_family_takes_a_new_single_controller(wm, orc):
    """wm_set_controllers with P = 1 repacks the fused family's images."""
    cfg = synth.model_config("small_bf16")
    w = synth.weights(cfg, seed=15)
    Wp, bp = synth.population(cfg, 1, seed=16)
    B, T = 200, 4
    z0 = synth.z0(B, cfg["z_dim"], seed=15)
    mask = synth.mask(T, B, cfg["a_dim"], 0.3, seed=15)
    m = wm.WorldModel(dict(cfg, path="fused"), w)
    m.set_controllers(Wp, bp)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), want_seq=True)
    torch.cuda.synchronize()
    assert m.last_path == "fused"
    check_rollout(g, cfg, dict(w, W_ctrl=Wp[0], b_ctrl=bp[0]), z0, mask, orc=orc)
    with pytest.raises(wm.WMError):  # the fused family writes no log-probs
        m.rollout(_cuda(z0), T, mask=_cuda(mask), want_logp=True)


@pytest.mark.parametrize("host", [False, True])
def test_returns_and_fitness_match_oracle(wm, orc, host):
    """wm_returns: G_t = r_t + gamma G_{t+1} (done ends the sum), bit for bit the oracle's
    fp64 recursion; fitness = each candidate's mean G_0."""
    cfg, w, z0, mask, B, T = synth.rollout_inputs("mid_bf16", B=1000, T=30)
    P, E, off = 5, 7, 3
    m = wm.WorldModel(dict(cfg, value_head=1), w)
    Wp, bp = synth.population(cfg, P, seed=17)
    m.set_controllers(Wp, bp, pop_group=E)
    g = m.rollout(_cuda(z0), T, mask=_cuda(mask), episode_offset=off)
    gamma = float(np.float32(0.97))
    boot = torch.randn(B, device="cuda")
    args = (g["rewards"], g["done"], gamma)
    if host:
        args = (g["rewards"].cpu(), g["done"].cpu(), gamma)
        boot = boot.cpu()
    res = m.returns(*args, bootstrap=boot, episode_offset=off, want_fitness=True)
    torch.cuda.synchronize()
    o = orc.returns(np_(g["rewards"]), np_(g["done"]), gamma, stop_at_done=True, bootstrap=np_(boot),
                    episode_offset=off, pop_size=P, pop_group=E)
    assert np.array_equal(np_(res["returns"]), o["returns"])
    np.testing.assert_allclose(np_(res["fitness"]), o["fitness"], rtol=1e-6)


# ------------------------------------------------------------------ hierarchical (xfer, location) action
@pytest.mark.parametrize("path,name,NX,flags", [
    ("stepwise", "tiny_fp32", 16, dict(ctrl_sample=1, ctrl_tau=0.9, noop_terminates=1)),
    ("tensor", "small_bf16", 32, dict(ctrl_sample=1, ctrl_tau=1.0)),
    # 55 transformations + NO-OP and the paper's 200 location slots
    ("tensor", "mid_bf16", 56, dict(done_terminates=1, noop_terminates=1, reward_mode=1)),
    ("tensor", "large_bf16", 112, dict(value_head=1)),
    ("auto", "small_bf16", 32, dict()),
])
def test_hierarchical_action_against_oracle(wm, orc, path, name, NX, flags):
    """Sec. 3.1.3: the xfer under the xfer mask, then the location under that xfer's location
    mask; the LSTM takes both one-hot rows.  Step-anchored against the oracle; AUTO never
    routes it to the fused family, and teacher-forced scoring declines it."""
    cfg = dict(synth.model_config(name), n_xfers=NX, **flags)
    w = synth.weights(cfg, seed=18)
    A = cfg["a_dim"]
    B, T = (16, 10) if name == "tiny_fp32" else (600, 5)
    z0 = synth.z0(B, cfg["z_dim"], seed=18)
    xm, lm = synth.hier_masks(T, B, NX, A - NX, 0.5, seed=18)
    sh = {}
    if cfg.get("reward_mode"):
        rt0, mem0 = synth.shaping_state(B, seed=18)
        sh = dict(rt0=rt0, mem0=mem0)
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.rollout(_cuda(z0), T, mask=_cuda(xm), loc_mask=_cuda(lm), episode_offset=33, t0=2,
                  want_seq=True, want_logp=True, **{k: _cuda(v) for k, v in sh.items()})
    torch.cuda.synchronize()
    assert m.last_path != "fused" and (path == "auto" or m.last_path == path)
    r = check_rollout(g, cfg, w, z0, xm, episodes=33 + np.arange(B), t0=2, loc_mask=lm, orc=orc, **sh)
    print("hierarchical", path, name, NX, flags, r)
    locs = np_(g["loc_actions"])
    assert (locs >= 0).any() and (np_(g["actions"]) == NX - 1).any() or name == "large_bf16"
    if path == "tensor" and name == "small_bf16":
        # host arrays (the location masks staged per step) give the same bits
        hz, hx, hl = (torch.from_numpy(a).pin_memory() for a in (z0, xm, lm))
        gh = m.rollout(hz, T, mask=hx, loc_mask=hl, episode_offset=33, t0=2, want_seq=True, want_logp=True)
        for k in ("actions", "loc_actions", "z", "rewards", "logp_seq"):
            assert torch.equal(gh[k], g[k].cpu()), k
    zs, acts, _ = synth.teacher_inputs(4, 3, cfg["z_dim"], A)
    with pytest.raises(wm.WMError) as ei:
        m.mdn_nll(_cuda(zs), _cuda(acts))
    assert ei.value.status == wm.WM_ERR_UNSUPPORTED


# ------------------------------------------------------------------ the training step (BPTT)
GRAD_KEYS = ("W_lstm", "b_lstm", "W_mdn", "b_mdn")
# relative Frobenius error of each gradient block: fp32 ~ 100 fp32 roundoffs; bf16 ~ 4 bf16
# roundoffs (2^-9 each: the backward's GEMM operands are rounded to bf16 once)
GRAD_TOL = {"fp32": 1e-5, "bf16": 1e-2}


def _grad_err(g, o):
    out = {}
    for k in GRAD_KEYS:
        a, b = np_(g[k]).astype(np.float64), np.asarray(o[k], np.float64)
        out[k] = float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))
    return out


@pytest.mark.parametrize("name,prec,path,N,T", [("tiny_fp32", "fp32", "stepwise", 37, 9),
                                                ("tiny_fp32", "fp32", "fused", 37, 9),  # small-batch member's forward
                                                ("small_bf16", "bf16", "auto", 64, 12),
                                                ("nll", "bf16", "tensor", 300, 10),
                                                ("nll", "fp32", "stepwise", 64, 16),
                                                ("nll", "fp32", "tensor", 300, 10)])
def test_training_step_gradient_against_oracle(wm, orc, name, prec, path, N, T):
    """wm_mdn_nll_backward against the oracle's fp64 BPTT, ragged lengths and no-action rows."""
    cfg = dict(synth.model_config(name), precision=prec)
    if name == "tiny_fp32":
        cfg.update(z_dim=7, a_dim=45, h_dim=40, k_mix=3)
    w = synth.weights(cfg, seed=19)
    zs, acts, lens = synth.teacher_inputs(N, T, cfg["z_dim"], cfg["a_dim"], seed=19, ragged=True)
    acts[1, ::5] = -1
    lens[0], lens[1] = 0, T
    m = wm.WorldModel(dict(cfg, path=path), w)
    g = m.mdn_nll_backward(_cuda(zs), _cuda(acts), lengths=_cuda(lens))
    torch.cuda.synchronize()
    o = orc.mdn_nll_grad(cfg, w, zs, acts, lens, nthreads=NT)
    err = _grad_err(g, o)
    print("gradient", name, prec, m.last_path, err)
    for k, e in err.items():
        assert e <= GRAD_TOL[prec], (k, e)
    rel = np.abs(np_(g["nll"]) - o["nll"]) / np.maximum(np.abs(o["nll"]), 1e-12)
    assert np.all(rel[o["nll"] != 0] <= 1e-3) and np.all(np_(g["nll"])[o["nll"] == 0] == 0)
    # deterministic, and host arrays give the same bits
    g2 = m.mdn_nll_backward(_cuda(zs), _cuda(acts), lengths=_cuda(lens))
    gh = m.mdn_nll_backward(torch.from_numpy(zs), torch.from_numpy(acts), lengths=torch.from_numpy(lens))
    for k in GRAD_KEYS + ("nll",):
        assert torch.equal(g[k], g2[k]) and torch.equal(g[k].cpu(), gh[k]), k


def test_training_step_full_size(wm, orc):
    """The nll workload at full size (512 sequences x 128 steps, bf16, tensor forward): the
    gradient is additive over sequences (two halves sum to the whole), and 16 sequences
    against the oracle."""
    cfg = dict(synth.model_config("nll"), precision="bf16")
    w = synth.weights(cfg, seed=20)
    N, T = 512, 128
    zs, acts, lens = synth.teacher_inputs(N, T, cfg["z_dim"], cfg["a_dim"], seed=20, ragged=True)
    m = wm.WorldModel(dict(cfg, path="tensor"), w)
    zc, ac, lc = _cuda(zs), _cuda(acts), _cuda(lens)
    full = m.mdn_nll_backward(zc, ac, lengths=lc)
    a = m.mdn_nll_backward(zc[:, :256].contiguous(), ac[:, :256].contiguous(), lengths=lc[:256].contiguous())
    b = m.mdn_nll_backward(zc[:, 256:].contiguous(), ac[:, 256:].contiguous(), lengths=lc[256:].contiguous())
    torch.cuda.synchronize()
    assert m.last_path == "tensor"
    err = _grad_err(full, {k: np_(a[k]).astype(np.float64) + np_(b[k]) for k in GRAD_KEYS})
    print("additivity", err)
    for k, e in err.items():
        assert e <= 1e-5, (k, e)  # the same bf16 products, summed in another order
    sub = m.mdn_nll_backward(zc[:, :16].contiguous(), ac[:, :16].contiguous(), lengths=lc[:16].contiguous())
    o = orc.mdn_nll_grad(cfg, w, zs[:, :16], acts[:, :16], lens[:16], nthreads=NT)
    err = _grad_err(sub, o)
    print("full-T subset vs oracle", err)
    for k, e in err.items():
        assert e <= GRAD_TOL["bf16"], (k, e)


def test_tensor_compaction_when_every_episode_ends_early(wm, orc):
    """Compacted rollouts whose episodes all end within the first steps: the host may stop
    issuing steps once the device reports no live episode (when it does depends on timing),
    and every later step's outputs are the frozen ones.  Two calls in a row: the second must
    not see the first's report."""
    cfg = dict(synth.model_config("mid_bf16"), done_terminates=1)
    w = synth.weights(cfg, seed=12)
    w["b_done"] = np.float32(3.0)  # done logits well above 0: almost every episode ends at once
    B, T = 300, 40
    z0 = synth.z0(B, cfg["z_dim"], seed=12)
    mask = synth.mask(T, B, cfg["a_dim"], 0.2, seed=12)
    done0 = (np.arange(B) % 7 == 3).astype(np.uint8)
    m = wm.WorldModel(dict(cfg, path="tensor"), w)
    outs = []
    for _ in range(2):
        g = m.rollout(_cuda(z0), T, mask=_cuda(mask), done0=_cuda(done0), want_seq=True)
        m.sync()
        assert m.last_path == "tensor"
        outs.append(g)
    r = check_rollout(outs[0], cfg, w, z0, mask, done0=done0, orc=orc)
    assert r["frozen_steps"] > 0.9 * B * T, r
    for k in ("z", "actions", "rewards", "done", "h_seq", "c_seq", "mdn_seq", "comp_seq", "h_final",
              "c_final"):
        assert torch.equal(outs[0][k], outs[1][k]), k
