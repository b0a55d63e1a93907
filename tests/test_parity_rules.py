"""The step-anchored parity checker on CPU: the oracle's own trajectory passes with
no flips, a trajectory that breaks an exact tie the other way passes with one
excused flip, and each planted mistake (a decision or value outside the rules)
fails.  Every 'GPU' trajectory here is made by the oracle."""
import numpy as np
import pytest

import synth
from parity import check_free_running, check_rollout

SEQ = ("z", "actions", "rewards", "done", "h_seq", "c_seq", "mdn_seq", "comp_seq")


def _case(orc, precision="fp32", **flags):
    cfg = dict(synth.model_config("tiny_fp32"), z_dim=6, a_dim=20, h_dim=24, k_mix=3,
               precision=precision, **flags)
    w = synth.weights(cfg, seed=41, std=0.3)
    B, T = 7, 6
    z0 = synth.z0(B, 6, seed=41)
    mask = synth.mask(T, B, 20, 0.5, seed=41)
    rng = np.random.default_rng(41)
    h0 = (0.3 * rng.standard_normal((B, 24))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((B, 24))).astype(np.float32)
    done0 = (np.arange(B) == 5).astype(np.uint8)
    kw = dict(episode_offset=300, t0=9, h0=h0, c0=c0, done0=done0)
    ck = dict(episodes=300 + np.arange(B), t0=9, h0=h0, c0=c0, done0=done0, orc=orc)
    keys = SEQ + ("h_final", "c_final")
    if cfg.get("reward_mode"):
        rt0, mem0 = synth.shaping_state(B, seed=41)
        kw.update(rt0=rt0, mem0=mem0)
        ck.update(rt0=rt0, mem0=mem0)
        keys += ("rt_seq", "mem_seq")
    if cfg.get("n_xfers"):
        mask, lm = synth.hier_masks(T, B, cfg["n_xfers"], 20 - cfg["n_xfers"], 0.6, seed=41)
        kw.update(loc_mask=lm)
        ck.update(loc_mask=lm)
    o = orc.rollout(cfg, w, z0, mask, T, want_seq=True, **kw)
    if cfg.get("n_xfers"):
        o["loc_actions"] = o["loc_seq"]
        keys += ("loc_actions",)
    g = {k: o[k].copy() for k in keys}
    return cfg, w, z0, mask, g, o, ck


@pytest.mark.parametrize("precision,flags", [("fp32", {}), ("bf16", {}),
                                             ("fp32", dict(done_terminates=1, noop_terminates=1)),
                                             ("fp32", dict(ctrl_sample=1, ctrl_tau=0.8)),
                                             ("bf16", dict(reward_mode=1, done_terminates=1)),
                                             ("fp32", dict(n_xfers=7, noop_terminates=1, ctrl_sample=1,
                                                           ctrl_tau=0.9))])
def test_oracle_trajectory_passes_without_flips(orc, precision, flags):
    cfg, w, z0, mask, g, o, ck = _case(orc, precision, **flags)
    r = check_rollout(g, cfg, w, z0, mask, **ck)
    assert r["flips"] == 0 and r["worst"] == 0.0
    T, B = g["actions"].shape
    assert r["compared"] + r["frozen_steps"] == T * B
    assert check_free_running(g, o, cfg)["diverged"] == 0


def test_tie_broken_the_other_way_is_one_excused_flip(orc):
    """Zero controller weights and two equal biases: the oracle takes the lower index;
    a trajectory that takes the higher one at one step (and follows it through) passes,
    with exactly one excused action flip."""
    cfg = dict(synth.model_config("tiny_fp32"), z_dim=4, a_dim=8, h_dim=12, k_mix=2)
    w = synth.weights(cfg, seed=42, std=0.3)
    w["W_ctrl"][:] = 0
    w["b_ctrl"][:] = 0
    w["b_ctrl"][[2, 5]] = 1.0
    B, T = 3, 4
    z0 = synth.z0(B, 4, seed=42)
    ep = np.arange(B)
    z, h, c = z0, np.zeros((B, 12), np.float32), np.zeros((B, 12), np.float32)
    g = {k: [] for k in SEQ}
    g["z"].append(z0)
    for t in range(T):
        s = orc.step(cfg, w, ep, t, z, h, c)
        a = s["action"].copy()
        if t == 2:
            a[1] = 5  # the tie partner
            s = orc.step(cfg, w, ep, t, z, h, c, a_use=a)
        for key, v in (("actions", a), ("rewards", s["reward"]), ("done", s["done"]),
                       ("h_seq", s["h"]), ("c_seq", s["c"]), ("mdn_seq", s["mdn"]),
                       ("comp_seq", s["comp"]), ("z", s["z_next"])):
            g[key].append(v)
        z, h, c = s["z_next"], s["h"], s["c"]
    g = {k: np.stack(v) for k, v in g.items()}
    r = check_rollout(g, cfg, w, z0, None, orc=orc)
    assert r["flips"] == 1 and r["kinds"]["action"] == 1 and r["flip_margins"] == [0.0]


def _planted(orc, how):
    shaped = how in ("shaped_reward", "runtime")
    cfg, w, z0, mask, g, o, ck = _case(orc, "fp32", done_terminates=1, reward_mode=int(shaped))
    T, B = g["actions"].shape
    live = np.argwhere(o["done"] == 0)
    t, b = (int(x) for x in live[len(live) // 2])
    if how == "action":
        valid = np.unpackbits(mask[t, b].view(np.uint8), bitorder="little")[:20].astype(bool)
        other = [j for j in np.nonzero(valid)[0] if j != g["actions"][t, b]]
        assert o["ctrl_margin"][t, b] > 1e-3
        g["actions"][t, b] = other[0]
    elif how == "component":
        d = int(np.argmax(o["comp_margin"][t, b]))
        assert o["comp_margin"][t, b, d] > 1e-4
        g["comp_seq"][t, b, d] = (g["comp_seq"][t, b, d] + 1) % 3
    elif how == "done":
        assert o["done_margin"][t, b] > 1e-4
        g["done"][t, b] = 1 - g["done"][t, b]
    elif how == "z":
        g["z"][t + 1, b, 2] += 5e-4
    elif how == "h":
        g["h_seq"][t, b, 7] -= 5e-4
    elif how == "mdn":
        g["mdn_seq"][t, b, 11] += 5e-4
    elif how == "reward":
        g["rewards"][t, b] += 5e-4
    elif how == "frozen_z":
        fb = 5  # frozen from the start (done0)
        g["z"][t + 1, fb, 0] += 1e-6
    elif how == "shaped_reward":
        g["rewards"][t, b] += 5e-4
    elif how == "runtime":
        g["rt_seq"][t, b] -= 5e-4
    return cfg, w, z0, mask, g, ck


@pytest.mark.parametrize("how", ["action", "component", "done", "z", "h", "mdn", "reward",
                                 "frozen_z", "shaped_reward", "runtime"])
def test_planted_mistakes_fail(orc, how):
    cfg, w, z0, mask, g, ck = _planted(orc, how)
    with pytest.raises(AssertionError):
        check_rollout(g, cfg, w, z0, mask, **ck)
