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


# ----------------------------------------------------------------------------- population (Sec. 3.4)
def test_population_equals_single_controller_runs(orc):
    """Episode e acts with candidate (e / E) mod P: a population rollout equals, episode by
    episode, a one-controller rollout with that candidate's weights."""
    Z, A, H, K, B, T, P, E = 4, 12, 16, 2, 11, 5, 3, 2
    cfg = _cfg(Z, A, H, K, reward_mode=0, ctrl_sample=1, ctrl_tau=0.9, pop_size=P, pop_group=E)
    w = synth.weights(cfg, seed=52, std=0.4)
    Wp, bp = synth.population(cfg, P, seed=52, std=0.4)
    wp = dict(w, W_ctrl=Wp, b_ctrl=bp)
    z0 = synth.z0(B, Z, seed=52)
    mk = synth.mask(T, B, A, 0.6, seed=52)
    off = 5
    o = orc.rollout(cfg, wp, z0, mk, T, episode_offset=off, want_seq=True)
    single = dict(cfg, pop_size=0)
    seen = set()
    for b in range(B):
        g = ((off + b) // E) % P
        seen.add(g)
        one = orc.rollout(single, dict(w, W_ctrl=Wp[g], b_ctrl=bp[g]), z0[b:b + 1], mk[:, b:b + 1], T,
                          episode_offset=off + b, want_seq=True)
        for k in ("actions", "z", "rewards", "logp_seq", "h_seq"):
            assert np.array_equal(o[k][:, b], one[k][:, 0]), (k, b)
    assert seen == set(range(P))


# ----------------------------------------------------------------------------- log-prob, value
def test_logp_matches_torch_categorical(orc):
    """logp_seq = log softmax(l / tau)[a] over the valid actions (torch Categorical on the
    logits rebuilt from the rollout's own state)."""
    import torch
    Z, A, H, K, B, T = 5, 14, 16, 2, 6, 5
    for sample, tau in ((1, 0.7), (0, 1.3)):
        cfg = _cfg(Z, A, H, K, reward_mode=0, ctrl_sample=sample, ctrl_tau=tau)
        w = synth.weights(cfg, seed=53, std=0.5)
        z0 = synth.z0(B, Z, seed=53)
        mk = synth.mask(T, B, A, 0.5, seed=53)
        mk[1, 2] = 0
        o = orc.rollout(cfg, w, z0, mk, T, want_seq=True)
        for t in range(T):
            h = np.zeros((B, H)) if t == 0 else o["h_seq"][t - 1].astype(np.float64)
            lg = (np.concatenate([o["z"][t].astype(np.float64), h], 1) @ w["W_ctrl"].astype(np.float64)
                  + w["b_ctrl"]).astype(np.float32).astype(np.float64)
            valid = np.unpackbits(mk[t].view(np.uint8), axis=1, bitorder="little")[:, :A].astype(bool)
            for b in range(B):
                a = int(o["actions"][t, b])
                if a < 0:
                    assert o["logp_seq"][t, b] == 0.0
                    continue
                d = torch.distributions.Categorical(
                    logits=torch.from_numpy(np.where(valid[b], lg[b] / tau, -np.inf)))
                assert o["logp_seq"][t, b] == pytest.approx(float(d.log_prob(torch.tensor(a))), abs=2e-6)


def test_logp_normalises_over_valid_actions(orc):
    """Forcing each valid action in turn, exp(logp) sums to 1 (and tau = 0 gives 0)."""
    Z, A, H, K, B = 4, 9, 12, 2, 5
    cfg = _cfg(Z, A, H, K, reward_mode=0, ctrl_sample=1, ctrl_tau=0.6)
    w = synth.weights(cfg, seed=54, std=0.6)
    rng = np.random.default_rng(54)
    z = rng.standard_normal((B, Z)).astype(np.float32)
    h = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    c = np.zeros((B, H), np.float32)
    mk = synth.mask(1, B, A, 0.6, seed=54)[0]
    valid = np.unpackbits(mk.view(np.uint8), axis=1, bitorder="little")[:, :A].astype(bool)
    total = np.zeros(B)
    for j in range(A):
        s = orc.step(cfg, w, np.arange(B), 0, z, h, c, mask=mk, a_use=np.full(B, j))
        total += np.where(valid[:, j], np.exp(s["logp"].astype(np.float64)), 0.0)
    np.testing.assert_allclose(total[valid.any(1)], 1.0, atol=1e-5)
    s0 = orc.step(dict(cfg, ctrl_tau=0.0), w, np.arange(B), 0, z, h, c, mask=mk)
    assert np.all(s0["logp"] == 0.0)


def test_value_head_is_linear_in_h(orc):
    Z, A, H, K, B, T = 4, 8, 16, 2, 5, 4
    cfg = _cfg(Z, A, H, K, reward_mode=0, value_head=1, done_terminates=1)
    w = synth.weights(cfg, seed=55, std=0.4)
    z0 = synth.z0(B, Z, seed=55)
    o = orc.rollout(cfg, w, z0, None, T, want_seq=True)
    ref = o["h_seq"].astype(np.float64) @ w["w_val"].astype(np.float64) + w["b_val"]
    live = np.ones((T, B), bool)
    live[1:] = np.cumsum(o["done"], 0)[:-1] == 0
    np.testing.assert_allclose(o["value_seq"][live], ref[live], atol=1e-6)
    assert np.all(o["value_seq"][~live] == 0)


# ----------------------------------------------------------------------------- returns, fitness
def test_returns_closed_forms(orc):
    T, B, gamma = 6, 4, 0.9
    r = np.full((T, B), 2.0, np.float32)
    d = np.zeros((T, B), np.uint8)
    boot = np.array([0.0, 1.0, -3.0, 10.0], np.float32)
    out = orc.returns(r, d, gamma, bootstrap=boot)["returns"]
    for t in range(T):
        n = T - t
        ref = 2.0 * (1 - gamma**n) / (1 - gamma) + gamma**n * boot.astype(np.float64)
        np.testing.assert_allclose(out[t], ref, rtol=1e-6)
    # a done step ends the sum: G_t = r_t there, and nothing after it leaks back
    d[2, 1] = 1
    r2 = r.copy()
    r2[3:, 1] = 1000.0
    out2 = orc.returns(r2, d, gamma, bootstrap=boot)["returns"]
    assert out2[2, 1] == np.float32(2.0)
    assert out2[0, 1] == pytest.approx(2.0 + gamma * 2.0 + gamma**2 * 2.0, rel=1e-6)
    # without stop_at_done the done flag is ignored
    out3 = orc.returns(r2, d, gamma, stop_at_done=False)["returns"]
    assert out3[2, 1] > 100


def test_fitness_is_mean_return_per_candidate(orc):
    T, B, P, E, off = 3, 13, 3, 2, 7
    rng = np.random.default_rng(56)
    r = rng.standard_normal((T, B)).astype(np.float32)
    d = np.zeros((T, B), np.uint8)
    out = orc.returns(r, d, 0.5, episode_offset=off, pop_size=P, pop_group=E)
    g0 = out["returns"][0].astype(np.float64)
    for g in range(P):
        sel = [b for b in range(B) if ((off + b) // E) % P == g]
        assert out["fitness"][g] == pytest.approx(g0[sel].mean(), rel=1e-6)


# ----------------------------------------------------------------------------- hierarchical action (Sec. 3.1.3)
def _hier_case(seed=57, **kw):
    NX, L = 6, 11
    Z, A, H, K, B, T = 4, NX + L, 16, 2, 9, 6
    kw.setdefault("reward_mode", 0)
    cfg = _cfg(Z, A, H, K, n_xfers=NX, **kw)
    w = synth.weights(cfg, seed=seed, std=0.5)
    z0 = synth.z0(B, Z, seed=seed)
    xm, lm = synth.hier_masks(T, B, NX, L, 0.6, seed=seed)
    return cfg, w, z0, xm, lm, NX, L, B, T


def test_hier_argmax_is_two_masked_argmaxes(orc):
    """Argmax mode: the xfer is the masked argmax of the first NX logits, the location the
    masked argmax of the other L under the chosen xfer's location mask (numpy, on logits
    rebuilt from the rollout's own state); NO-OP takes no location."""
    cfg, w, z0, xm, lm, NX, L, B, T = _hier_case()
    o = orc.rollout(cfg, w, z0, xm, T, want_seq=True, loc_mask=lm)
    Z, H = cfg["z_dim"], cfg["h_dim"]
    checked = 0
    for t in range(T):
        h = np.zeros((B, H)) if t == 0 else o["h_seq"][t - 1].astype(np.float64)
        lg = (np.concatenate([o["z"][t].astype(np.float64), h], 1) @ w["W_ctrl"].astype(np.float64)
              + w["b_ctrl"]).astype(np.float32)
        vx = np.unpackbits(xm[t].view(np.uint8), axis=1, bitorder="little")[:, :NX].astype(bool)
        for b in range(B):
            x = int(o["actions"][t, b])
            assert x == int(np.argmax(np.where(vx[b], lg[b, :NX], -np.inf)))
            loc = int(o["loc_seq"][t, b])
            if x == NX - 1:
                assert loc == -1
                continue
            vl = np.unpackbits(lm[t, b, x].view(np.uint8), bitorder="little")[:L].astype(bool)
            assert vl.any() and vl[loc]
            assert loc == int(np.argmax(np.where(vl, lg[b, NX:], -np.inf)))
            checked += 1
    assert checked > B * T // 3


def test_hier_lstm_takes_both_rows(orc):
    """h' = LSTMCell([z, onehot(xfer), onehot(location)], (h, c)) with the action rows of
    W_lstm (torch, forced choices)."""
    import torch
    cfg, w, z0, xm, lm, NX, L, B, T = _hier_case()
    Z, A, H = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"]
    rng = np.random.default_rng(58)
    h = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    c = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    xs = rng.integers(0, NX - 1, B).astype(np.int32)
    ls = rng.integers(0, L, B).astype(np.int32)
    ls[2] = -1
    s = orc.step(cfg, w, np.arange(B), 0, z0, h, c, mask=xm[0], loc_mask=lm[0], a_use=xs, loc_use=ls)
    cell = torch.nn.LSTMCell(Z + A, H, dtype=torch.float64)
    Wl = torch.from_numpy(w["W_lstm"]).double()
    with torch.no_grad():
        cell.weight_ih.copy_(Wl[:Z + A].T)
        cell.weight_hh.copy_(Wl[Z + A:].T)
        cell.bias_ih.copy_(torch.from_numpy(w["b_lstm"]).double())
        cell.bias_hh.zero_()
        oh = torch.zeros(B, A, dtype=torch.float64)
        oh[np.arange(B), xs] = 1.0
        ok = ls >= 0
        oh[np.nonzero(ok)[0], NX + ls[ok]] = 1.0
        hr, cr = cell(torch.cat([torch.from_numpy(z0).double(), oh], 1),
                      (torch.from_numpy(h).double(), torch.from_numpy(c).double()))
    np.testing.assert_allclose(s["h"], hr.numpy(), atol=2e-6)
    np.testing.assert_allclose(s["c"], cr.numpy(), atol=2e-6)


def test_hier_logp_normalises_over_joint_actions(orc):
    """exp(logp) summed over every valid (xfer, location) pair and the NO-OP is 1."""
    cfg, w, z0, xm, lm, NX, L, B, T = _hier_case(ctrl_sample=1, ctrl_tau=0.8)
    rng = np.random.default_rng(59)
    h = (0.5 * rng.standard_normal((B, 16))).astype(np.float32)
    c = np.zeros((B, 16), np.float32)
    vx = np.unpackbits(xm[0].view(np.uint8), axis=1, bitorder="little")[:, :NX].astype(bool)
    total = np.zeros(B)
    for x in range(NX):
        for loc in ([-1] if x == NX - 1 else range(L)):
            s = orc.step(cfg, w, np.arange(B), 0, z0, h, c, mask=xm[0], loc_mask=lm[0],
                         a_use=np.full(B, x), loc_use=np.full(B, loc))
            ok = vx[:, x].copy()
            if loc >= 0:
                ok &= np.array([bool((lm[0, b, x, loc // 32] >> (loc % 32)) & 1) for b in range(B)])
            total += np.where(ok, np.exp(s["logp"].astype(np.float64)), 0.0)
    np.testing.assert_allclose(total, 1.0, atol=1e-5)


def test_hier_sampled_frequencies(orc):
    """Sampled mode: over many episodes (independent Philox streams) from one state, the
    (xfer, location) frequencies follow pi(xfer) pi(location | xfer) (chi-square)."""
    from scipy import stats
    NX, L = 4, 5
    Z, A, H, K, B = 3, NX + L, 8, 2, 6000
    cfg = _cfg(Z, A, H, K, reward_mode=0, n_xfers=NX, ctrl_sample=1, ctrl_tau=1.0)
    w = synth.weights(cfg, seed=60, std=0.6)
    z = np.tile(synth.z0(1, Z, seed=60), (B, 1))
    h = np.zeros((B, H), np.float32)
    xm = synth.pack_mask(np.tile(np.array([[1, 0, 1, 1] + [0] * L], bool), (B, 1)))
    locs = np.zeros((NX, L), bool)
    locs[0, :3] = True
    locs[2, :5] = True
    lm = np.tile(synth.pack_mask(locs)[None], (B, 1, 1))
    s = orc.step(cfg, w, np.arange(B), 0, z, h, h, mask=xm, loc_mask=lm)
    lg = (np.concatenate([z[0].astype(np.float64), h[0]]) @ w["W_ctrl"].astype(np.float64)
          + w["b_ctrl"]).astype(np.float32).astype(np.float64)
    px = np.where([1, 0, 1, 1], np.exp(lg[:NX]), 0.0)
    px /= px.sum()
    cells, probs = [], []
    for x in (0, 2):
        pl = np.where(locs[x], np.exp(lg[NX:]), 0.0)
        pl /= pl.sum()
        for loc in np.nonzero(locs[x])[0]:
            cells.append((x, loc))
            probs.append(px[x] * pl[loc])
    cells.append((3, -1))
    probs.append(px[3])
    counts = [int(np.sum((s["action"] == x) & (s["loc"] == loc))) for x, loc in cells]
    assert sum(counts) == B
    assert stats.chisquare(counts, np.array(probs) * B).pvalue > 1e-4


def test_hier_noop_terminates_and_invalid(orc):
    cfg, w, z0, xm, lm, NX, L, B, T = _hier_case(noop_terminates=1, reward_mode=1)
    w["b_ctrl"][:] = 0
    w["W_ctrl"][:] = 0
    w["b_ctrl"][NX - 1] = 5.0  # NO-OP wins wherever it is valid
    rt0, mem0 = synth.shaping_state(B, seed=57)
    o = orc.rollout(cfg, w, z0, xm, T, want_seq=True, loc_mask=lm, rt0=rt0, mem0=mem0)
    assert np.all(o["actions"][0] == NX - 1) and np.all(o["loc_seq"][0] == -1)
    assert np.all(o["done"] == 1) and np.all(o["actions"][1:] == -1)
    assert np.all(o["rewards"][0] != -100.0)  # the NO-OP is a valid action
    # an xfer whose location mask is empty: the location is -1, the action invalid (-100)
    cfg2 = dict(cfg, noop_terminates=0)
    w2 = dict(w, b_ctrl=np.zeros(NX + L, np.float32))
    w2["b_ctrl"][0] = 5.0
    xm2 = xm.copy()
    xm2[:] = 1  # xfer 0 valid everywhere ...
    lm2 = lm.copy()
    lm2[:, :, 0, :] = 0  # ... but with no location
    o2 = orc.rollout(cfg2, w2, z0, xm2, T, want_seq=True, loc_mask=lm2, rt0=rt0, mem0=mem0)
    assert np.all(o2["actions"] == 0) and np.all(o2["loc_seq"] == -1)
    assert np.all(o2["rewards"] == np.float32(-100.0))


# ----------------------------------------------------------------------------- BPTT gradient (Sec. 3.3.2, Sec. 4.7)
def _grad_case(seed=61, precision="fp32", **kw):
    Z, A, H, K, N, T = 3, 5, 6, 2, 4, 5
    cfg = _cfg(Z, A, H, K, reward_mode=0, precision=precision, **kw)
    w = synth.weights(cfg, seed=seed, std=0.4)
    zs, acts, lens = synth.teacher_inputs(N, T, Z, A, seed=seed, ragged=True)
    acts[1, 2] = -1
    lens[0] = T
    return cfg, w, zs, acts, lens


def test_grad_matches_central_differences(orc):
    """Every parameter block against central differences of sum_n NLL_n (state carried in
    fp64, so the loss is smooth to the last bit; the step is the fp32 weights' own)."""
    cfg, w, zs, acts, lens = _grad_case(state64=1)
    g = orc.mdn_nll_grad(cfg, w, zs, acts, lens)
    loss = lambda ww: orc.mdn_nll(cfg, ww, zs, acts, lengths=lens)["nll"].sum()
    assert np.allclose(g["nll"], orc.mdn_nll(cfg, w, zs, acts, lengths=lens)["nll"], rtol=1e-12)
    rng = np.random.default_rng(61)
    Z, A = cfg["z_dim"], cfg["a_dim"]
    picks = {"W_lstm": [(0, 3), (Z + 1, 7), (Z + acts[0, 1], 2), (Z + A + 2, 20), (Z + A + 5, 23)],
             "b_lstm": [(5,), (12,), (19,)], "W_mdn": [(0, 0), (3, 11), (5, 17)], "b_mdn": [(2,), (9,), (16,)]}
    for name, idxs in picks.items():
        for idx in idxs:
            wp, wm = {k: (np.array(v, copy=True) if isinstance(v, np.ndarray) else v) for k, v in w.items()}, \
                     {k: (np.array(v, copy=True) if isinstance(v, np.ndarray) else v) for k, v in w.items()}
            x0 = float(w[name][idx])
            xp, xm = np.float32(x0 + 1e-3), np.float32(x0 - 1e-3)
            wp[name][idx], wm[name][idx] = xp, xm
            fd = (loss(wp) - loss(wm)) / (float(xp) - float(xm))
            assert g[name][idx] == pytest.approx(fd, rel=2e-5, abs=2e-7), (name, idx, g[name][idx], fd)


def _torch_loss(cfg, w, zs, acts, lens, bf16=False):
    """sum_n NLL_n in torch fp64 (LSTMCell + MixtureSameFamily), for autograd; bf16 rounds the
    weights and the GEMM operands with a straight-through gradient."""
    import torch
    from torch.distributions import Categorical, MixtureSameFamily, Normal
    Z, A, H, K = (cfg[k] for k in ("z_dim", "a_dim", "h_dim", "k_mix"))
    rnd = (lambda x: x + (x.to(torch.bfloat16).double() - x).detach()) if bf16 else (lambda x: x)
    wr = (lambda a: torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).double()) if bf16 else \
         (lambda a: torch.from_numpy(np.asarray(a, np.float32)).double())
    P = {"W_lstm": wr(w["W_lstm"]).requires_grad_(), "b_lstm": torch.from_numpy(w["b_lstm"]).double().requires_grad_(),
         "W_mdn": wr(w["W_mdn"]).requires_grad_(), "b_mdn": torch.from_numpy(w["b_mdn"]).double().requires_grad_()}
    T, N = acts.shape
    h = torch.zeros(N, H, dtype=torch.float64)
    c = torch.zeros(N, H, dtype=torch.float64)
    total = 0.0
    for t in range(T):
        x = torch.cat([rnd(torch.from_numpy(zs[t]).double()), rnd(h)], 1)
        Wz, Wa, Wh = P["W_lstm"][:Z], P["W_lstm"][Z:Z + A], P["W_lstm"][Z + A:]
        oh = torch.zeros(N, A, dtype=torch.float64)
        ok = acts[t] >= 0
        oh[np.nonzero(ok)[0], acts[t][ok]] = 1.0
        G = x[:, :Z] @ Wz + oh @ Wa + x[:, Z:] @ Wh + P["b_lstm"]
        i, f, g, o = G[:, :H].sigmoid(), G[:, H:2 * H].sigmoid(), G[:, 2 * H:3 * H].tanh(), G[:, 3 * H:].sigmoid()
        c = f * c + i * g
        h = o * c.tanh()
        md = (rnd(h) @ P["W_mdn"] + P["b_mdn"]).view(N, 3, Z, K)
        mix = MixtureSameFamily(Categorical(logits=md[:, 0]), Normal(md[:, 1], md[:, 2].exp()))
        lp = mix.log_prob(torch.from_numpy(zs[t + 1]).double()).sum(1)
        total = total - (lp * torch.from_numpy((t < lens).astype(np.float64))).sum()
    total.backward()
    return total, P


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_grad_matches_torch_autograd(orc, precision):
    """fp32: torch autograd through LSTMCell-style gates and MixtureSameFamily (fp64, state
    in fp64); bf16: the same with bf16 weights and straight-through operand rounding."""
    Z, A, H, K, N, T = 5, 7, 12, 3, 6, 6
    cfg = _cfg(Z, A, H, K, reward_mode=0, precision=precision, state64=1)
    w = synth.weights(cfg, seed=62, std=0.4)
    zs, acts, lens = synth.teacher_inputs(N, T, Z, A, seed=62, ragged=True)
    acts[2, 3] = -1
    g = orc.mdn_nll_grad(cfg, w, zs, acts, lens, nthreads=3)
    total, P = _torch_loss(cfg, w, zs, acts, lens, bf16=(precision == "bf16"))
    assert g["nll"].sum() == pytest.approx(float(total), rel=1e-10)
    for k in P:
        np.testing.assert_allclose(g[k], P[k].grad.numpy(), rtol=1e-8, atol=1e-10, err_msg=k)


def test_grad_is_additive_over_sequences(orc):
    """The gradient of a batch is the sum of its sequences' gradients (any split)."""
    cfg, w, zs, acts, lens = _grad_case(seed=63)
    full = orc.mdn_nll_grad(cfg, w, zs, acts, lens, nthreads=2)
    a = orc.mdn_nll_grad(cfg, w, zs[:, :1], acts[:, :1], lens[:1])
    b = orc.mdn_nll_grad(cfg, w, zs[:, 1:], acts[:, 1:], lens[1:])
    for k in ("W_lstm", "b_lstm", "W_mdn", "b_mdn"):
        np.testing.assert_allclose(full[k], a[k] + b[k], rtol=1e-12, atol=1e-15)
    # padding: a zero-length sequence contributes nothing
    l0 = lens.copy()
    l0[:] = 0
    z = orc.mdn_nll_grad(cfg, w, zs, acts, l0)
    assert all(np.all(z[k] == 0) for k in ("W_lstm", "b_lstm", "W_mdn", "b_mdn"))
