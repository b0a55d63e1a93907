"""Pins of the oracle's parts beyond the basic dream step (no GPU needed):
the shaped reward of Sec. 3.1.4 (Eq. 1 and Eq. 2 on the predicted runtime and
memory-access heads)."""
import numpy as np
import pytest

import synth


def _cfg(Z, A, H, K, **kw):
    c = dict(z_dim=Z, a_dim=A, h_dim=H, k_mix=K, precision="fp32", mdn_tau=1.0,
             sigma_sqrt_tau=0, ctrl_sample=0, ctrl_tau=1.0, done_terminates=0,
             noop_terminates=0, seed=0, reward_mode=1, reward_alpha=0.8, reward_beta=0.2,
             invalid_reward=-100.0)
    c.update(kw)
    return c


def _shaped_case(seed=51, **kw):
    Z, A, H, K, B, T = 4, 10, 16, 2, 6, 7
    cfg = _cfg(Z, A, H, K, **kw)
    w = synth.weights(cfg, seed=seed, std=0.4)
    z0 = synth.z0(B, Z, seed=seed)
    mk = synth.mask(T, B, A, 0.6, seed=seed)
    rt0, mem0 = synth.shaping_state(B, seed=seed)
    return cfg, w, z0, mk, rt0, mem0, B, T


# ----------------------------------------------------------------------------- Eq. 1 / Eq. 2
def test_eq1_rewards_telescope(orc):
    """Eq. 1 (alpha = 1, beta = 0): the rewards of a run of valid actions sum to the
    runtime entering the run minus the runtime after it."""
    cfg, w, z0, mk, rt0, mem0, B, T = _shaped_case(reward_alpha=1.0, reward_beta=0.0)
    mk[:] = 0xFFFFFFFF  # every action valid
    o = orc.rollout(cfg, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0)
    np.testing.assert_allclose(o["rewards"].astype(np.float64).sum(0),
                               rt0.astype(np.float64) - o["rt_seq"][-1], atol=1e-5)
    # and Eq. 2 with both weights: alpha * (RT drop) + beta * (M drop) over the run
    cfg2 = dict(cfg, reward_alpha=0.8, reward_beta=0.2)
    o2 = orc.rollout(cfg2, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0)
    ref = 0.8 * (rt0 - o2["rt_seq"][-1].astype(np.float64)) + 0.2 * (mem0 - o2["mem_seq"][-1].astype(np.float64))
    np.testing.assert_allclose(o2["rewards"].astype(np.float64).sum(0), ref, atol=1e-5)


def test_constant_heads_closed_form(orc):
    """Zero head weights: RT_t = b_rt, M_t = b_mem for every t, so only the first step
    rewards alpha (rt0 - b_rt) + beta (mem0 - b_mem); the rest are exactly 0."""
    cfg, w, z0, mk, rt0, mem0, B, T = _shaped_case()
    mk[:] = 0xFFFFFFFF
    w["w_rt"][:] = 0
    w["w_mem"][:] = 0
    w["b_rt"], w["b_mem"] = 0.75, -0.25
    o = orc.rollout(cfg, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0)
    ref0 = 0.8 * (rt0.astype(np.float64) - 0.75) + 0.2 * (mem0.astype(np.float64) + 0.25)
    np.testing.assert_allclose(o["rewards"][0], ref0, rtol=1e-6, atol=1e-7)
    assert np.all(o["rewards"][1:] == 0.0)
    assert np.all(o["rt_seq"] == np.float32(0.75)) and np.all(o["mem_seq"] == np.float32(-0.25))


def test_heads_are_linear_in_h(orc):
    """RT_t = w_rt . h_{t+1} + b_rt and M_t likewise (numpy on the rollout's own h)."""
    cfg, w, z0, mk, rt0, mem0, B, T = _shaped_case()
    o = orc.rollout(cfg, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0)
    h = o["h_seq"].astype(np.float64)
    np.testing.assert_allclose(o["rt_seq"], h @ w["w_rt"].astype(np.float64) + w["b_rt"], atol=1e-6)
    np.testing.assert_allclose(o["mem_seq"], h @ w["w_mem"].astype(np.float64) + w["b_mem"], atol=1e-6)


def test_invalid_action_reward(orc):
    """No valid action (a = -1): the reward is the invalid reward; the predictions still
    move with the world model's state."""
    cfg, w, z0, mk, rt0, mem0, B, T = _shaped_case(invalid_reward=-100.0)
    mk[3, 2] = 0
    mk[0, 5] = 0
    o = orc.rollout(cfg, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0)
    assert o["actions"][3, 2] == -1 and o["rewards"][3, 2] == np.float32(-100.0)
    assert o["actions"][0, 5] == -1 and o["rewards"][0, 5] == np.float32(-100.0)
    ok = o["actions"] >= 0
    assert np.all(o["rewards"][ok] != -100.0)
    # the step after an invalid one measures from the prediction the invalid step made
    r = 0.8 * (o["rt_seq"][3, 2].astype(np.float64) - o["rt_seq"][4, 2]) + \
        0.2 * (o["mem_seq"][3, 2].astype(np.float64) - o["mem_seq"][4, 2])
    assert o["rewards"][4, 2] == pytest.approx(r, abs=1e-6)


def test_frozen_and_resume(orc):
    """A frozen episode earns 0 and keeps its predictions; a run split in two (resuming
    with the last predictions) reproduces the unsplit one bit for bit."""
    cfg, w, z0, mk, rt0, mem0, B, T = _shaped_case(done_terminates=1)
    w["w_done"][:] = 0
    w["b_done"] = -1.0
    done0 = (np.arange(B) == 1).astype(np.uint8)
    full = orc.rollout(cfg, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0, done0=done0)
    assert np.all(full["rewards"][:, 1] == 0) and np.all(full["rt_seq"][:, 1] == rt0[1])
    a = orc.rollout(cfg, w, z0, mk[:3], 3, want_seq=True, rt0=rt0, mem0=mem0, done0=done0)
    b = orc.rollout(cfg, w, a["z"][-1], mk[3:], T - 3, t0=3, h0=a["h_final"], c0=a["c_final"],
                    done0=np.maximum(a["done"][-1], done0), want_seq=True,
                    rt0=a["rt_seq"][-1], mem0=a["mem_seq"][-1])
    for k in ("rewards", "rt_seq", "mem_seq", "actions"):
        assert np.array_equal(np.concatenate([a[k], b[k]]), full[k]), k


def test_step_carries_the_predictions(orc):
    """orc_step from a shaped rollout's own state and predictions reproduces its step."""
    cfg, w, z0, mk, rt0, mem0, B, T = _shaped_case(precision="bf16")
    o = orc.rollout(cfg, w, z0, mk, T, want_seq=True, rt0=rt0, mem0=mem0)
    for t in range(T):
        h = np.zeros((B, 16), np.float32) if t == 0 else o["h_seq"][t - 1]
        c = np.zeros((B, 16), np.float32) if t == 0 else o["c_seq"][t - 1]
        rp = rt0 if t == 0 else o["rt_seq"][t - 1]
        mp = mem0 if t == 0 else o["mem_seq"][t - 1]
        s = orc.step(cfg, w, np.arange(B), t, o["z"][t], h, c, mask=mk[t], rt=rp, mem=mp)
        assert np.array_equal(s["reward"], o["rewards"][t])
        assert np.array_equal(s["rt"], o["rt_seq"][t]) and np.array_equal(s["mem"], o["mem_seq"][t])
