"""Pins of the oracle's decision margins and of its one-step entry point (no GPU needed).

The margins (controller top-2 gap, sampled-action and mixture-component CDF
distances, |done logit|) decide which GPU decision flips the parity checks
excuse, so each is pinned to a characterisation other than its formula: the
distance, found by bisection on the oracle's own decision function, from the
input to the nearest point where that decision changes.  ``orc_step`` (one
dream step from a given state, with optional overrides of the action, h' and
components) is pinned to ``orc_rollout`` bit for bit and to torch / numpy for
what each override must change.
"""
import math

import numpy as np
import pytest
import torch

import synth


def _cfg(Z, A, H, K, **kw):
    c = dict(z_dim=Z, a_dim=A, h_dim=H, k_mix=K, precision="fp32", mdn_tau=1.0,
             sigma_sqrt_tau=0, ctrl_sample=0, ctrl_tau=1.0, done_terminates=0,
             noop_terminates=0, seed=0)
    c.update(kw)
    return c


def _bisect(f, lo, hi, iters=80):
    """f(lo) != f(hi): the point where f changes, to ~2^-80 of the bracket."""
    flo = f(lo)
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if f(mid) == flo:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def _u_boundaries(decide, grid=1 << 14):
    """Every u in (0, 1) where decide(u) changes (grid scan, then bisection)."""
    us = (np.arange(grid) + 0.5) / grid
    ds = [decide(float(u)) for u in us]
    out = []
    for i in range(grid - 1):
        if ds[i] != ds[i + 1]:
            out.append(_bisect(decide, float(us[i]), float(us[i + 1]), iters=60))
    # the ends of [0, 1): a change inside the first or last half cell
    if decide(0.0) != ds[0]:
        out.append(_bisect(decide, 0.0, float(us[0]), iters=60))
    if decide(1.0 - 2.0**-40) != ds[-1]:
        out.append(_bisect(decide, float(us[-1]), 1.0 - 2.0**-40, iters=60))
    return out


def _argmax_margin_brute(decide, logits, valid):
    """Smallest raise of one valid non-chosen logit that changes the decision."""
    base = decide(logits)
    best = math.inf
    for j in np.nonzero(valid)[0]:
        if j == base:
            continue

        def raised(d, j=j):
            lg = logits.astype(np.float64).copy()
            lg[j] += d
            return decide(lg.astype(np.float32))
        hi = 1.0
        while raised(hi) == base:
            hi *= 2.0
        best = min(best, _bisect(raised, 0.0, hi, iters=60))
    return best


# ----------------------------------------------------------------------------- controller margin
def test_argmax_margin_is_distance_to_decision_change(orc):
    rng = np.random.default_rng(31)
    for trial in range(60):
        A = int(rng.integers(2, 40))
        lg = rng.standard_normal(A).astype(np.float32)
        valid = rng.random(A) < 0.6
        valid[rng.integers(A)] = True
        mw = synth.pack_mask(valid[None])[0]
        a, m = orc.select_action(lg, mw)
        if valid.sum() == 1:
            assert a == int(np.nonzero(valid)[0][0]) and m == math.inf
            continue
        ref = _argmax_margin_brute(lambda x: orc.select_action(x, mw)[0], lg, valid)
        assert m == pytest.approx(ref, abs=1e-6), (trial, m, ref)


def test_argmax_margin_ties_and_edges(orc):
    # an exact tie among valid maxima: margin 0, lowest index chosen
    lg = np.array([0.5, 2.0, -1.0, 2.0, 1.9], np.float32)
    a, m = orc.select_action(lg, None)
    assert a == 1 and m == 0.0
    # masking the tie partner away leaves the gap to the next valid logit (2.0 - 1.9)
    mw = synth.pack_mask(np.array([[1, 1, 1, 0, 1]], bool))[0]
    a, m = orc.select_action(lg, mw)
    assert a == 1 and m == pytest.approx(0.1, abs=1e-6)
    # a single valid action can never flip; no valid action gives -1
    mw = synth.pack_mask(np.array([[0, 0, 1, 0, 0]], bool))[0]
    assert orc.select_action(lg, mw) == (2, math.inf)
    mw = synth.pack_mask(np.zeros((1, 5), bool))[0]
    assert orc.select_action(lg, mw) == (-1, math.inf)
    # temperature 0 in sample mode behaves as argmax (same margin)
    assert orc.select_action(lg, None, ctrl_sample=1, ctrl_tau=0.0, u=0.3) == (1, 0.0)


def test_sampled_action_margin_is_distance_to_decision_change(orc):
    rng = np.random.default_rng(32)
    for trial in range(16):
        A = int(rng.integers(2, 14))
        tau = float(rng.uniform(0.6, 1.6))
        lg = rng.standard_normal(A).astype(np.float32)
        valid = rng.random(A) < 0.7
        valid[rng.integers(A)] = True
        mw = synth.pack_mask(valid[None])[0]
        bounds = _u_boundaries(lambda u: orc.select_action(lg, mw, 1, tau, u)[0])
        assert len(bounds) == int(valid.sum()) - 1
        for u in rng.random(6):
            _, m = orc.select_action(lg, mw, 1, tau, float(u))
            ref = min((abs(float(u) - b) for b in bounds), default=math.inf)
            assert m == pytest.approx(ref, abs=1e-9), (trial, u, m, ref)
    # u exactly on a boundary: margin 0 (two equal weights put a boundary at 1/2)
    lg = np.zeros(2, np.float32)
    a, m = orc.select_action(lg, None, 1, 1.0, 0.5)
    assert a == 1 and m == 0.0


# ----------------------------------------------------------------------------- component margin
def test_component_margin_is_distance_to_decision_change(orc):
    rng = np.random.default_rng(33)
    for trial in range(16):
        K = int(rng.integers(2, 9))
        tau = float(rng.choice([0.5, 1.0, 1.7]))
        lg = rng.standard_normal(K).astype(np.float32)
        mu, ls = rng.standard_normal(K), 0.3 * rng.standard_normal(K)
        bounds = _u_boundaries(lambda u: orc.sample_dim(lg, mu, ls, u, 0.0, tau)[0])
        assert len(bounds) == K - 1
        for u in rng.random(6):
            _, _, m = orc.sample_dim(lg, mu, ls, float(u), 0.0, tau)
            ref = min(abs(float(u) - b) for b in bounds)
            assert m == pytest.approx(ref, abs=1e-9), (trial, u, m, ref)
    # u on a boundary (equal logits: C_0 = 1/2 exactly): margin 0, the next component;
    # K = 1 has no boundary at all
    k, _, m = orc.sample_dim(np.zeros(2, np.float32), np.zeros(2), np.zeros(2), 0.5, 0.0)
    assert k == 1 and m == 0.0
    assert orc.sample_dim(np.zeros(1, np.float32), np.zeros(1), np.zeros(1), 0.4, 0.0)[2] == math.inf


def test_component_margin_at_zero_temperature_is_argmax_gap(orc):
    rng = np.random.default_rng(34)
    for _ in range(30):
        K = int(rng.integers(2, 9))
        lg = rng.standard_normal(K).astype(np.float32)
        mu, ls = rng.standard_normal(K), np.zeros(K)
        k, z, m = orc.sample_dim(lg, mu, ls, 0.3, 0.0, tau=0.0)
        ref = _argmax_margin_brute(lambda x: orc.sample_dim(x, mu, ls, 0.3, 0.0, tau=0.0)[0],
                                   lg, np.ones(K, bool))
        assert m == pytest.approx(ref, abs=1e-6) and z == mu[k]


# ----------------------------------------------------------------------------- margins in a rollout
def test_rollout_margins_match_brute_force(orc):
    """The margins a rollout reports are those of its own decisions: the controller's
    logits rebuilt from its state, the component uniforms from its Philox stream."""
    Z, A, H, K, B, T = 6, 20, 16, 3, 5, 4
    cfg = _cfg(Z, A, H, K, done_terminates=0)
    w = synth.weights(cfg, seed=35, std=0.5)
    z0 = synth.z0(B, Z, seed=35)
    mk = synth.mask(T, B, A, 0.5, seed=35)
    out = orc.rollout(cfg, w, z0, mk, T, want_seq=True)
    Wc = w["W_ctrl"].astype(np.float64)
    for t in range(T):
        for b in range(B):
            h = np.zeros(H) if t == 0 else out["h_seq"][t - 1, b].astype(np.float64)
            lg = (np.concatenate([out["z"][t, b].astype(np.float64), h]) @ Wc
                  + w["b_ctrl"]).astype(np.float32)
            valid = np.unpackbits(mk[t, b].view(np.uint8), bitorder="little")[:A].astype(bool)
            ref = _argmax_margin_brute(lambda x: orc.select_action(x, mk[t, b])[0], lg, valid)
            assert out["ctrl_margin"][t, b] == pytest.approx(ref, rel=1e-5, abs=1e-6)
            for d in range(0, Z, 2):
                u = orc.uniform(int(orc.draw(0, b, t, 0, d // 4)[d % 4]))
                m = out["mdn_seq"][t, b]
                lgk, mu, ls = m[d * K:(d + 1) * K], m[K * Z + d * K:], m[2 * K * Z + d * K:]
                bounds = _u_boundaries(
                    lambda uu: orc.sample_dim(lgk, mu[:K], ls[:K], uu, 0.0)[0], grid=1 << 12)
                ref = min(abs(u - x) for x in bounds)
                assert out["comp_margin"][t, b, d] == pytest.approx(ref, rel=1e-5, abs=1e-7)


def test_done_margin_is_distance_to_done_flip(orc):
    """|done logit| is how far b_done must move before the done flag flips."""
    Z, A, H, K, B = 4, 8, 12, 2, 6
    cfg = _cfg(Z, A, H, K)
    w = synth.weights(cfg, seed=36, std=0.4)
    rng = np.random.default_rng(36)
    z = rng.standard_normal((B, Z)).astype(np.float32)
    h = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    c = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    ep = np.arange(B)
    base = orc.step(cfg, w, ep, 0, z, h, c)

    def done_with(shift, b):
        w2 = dict(w, b_done=float(np.float32(w["b_done"] + shift)))
        return int(orc.step(cfg, w2, ep[b:b + 1], 0, z[b:b + 1], h[b:b + 1], c[b:b + 1])["done"][0])

    for b in range(B):
        sgn = -1.0 if base["done"][b] else 1.0
        ref = _bisect(lambda s: done_with(sgn * s, b), 0.0, 4.0, iters=50)
        assert base["done_margin"][b] == pytest.approx(ref, abs=2e-6)


# ----------------------------------------------------------------------------- orc_step
def _frozen_before(out, t, cfg, done0=None):
    B = out["actions"].shape[1]
    f = np.zeros(B, bool) if done0 is None else done0.astype(bool).copy()
    A = cfg["a_dim"]
    for s in range(t):
        if cfg["done_terminates"]:
            f |= out["done"][s] == 1
        if cfg["noop_terminates"]:
            f |= out["actions"][s] == A - 1
    return f


@pytest.mark.parametrize("flags", [dict(), dict(done_terminates=1, noop_terminates=1),
                                   dict(ctrl_sample=1, ctrl_tau=0.7, mdn_tau=0.0),
                                   dict(precision="bf16", mdn_tau=0.5, sigma_sqrt_tau=1)])
def test_step_replays_rollout_bit_for_bit(orc, flags):
    """Started from a rollout's own state, orc_step reproduces every output of that
    rollout's step exactly, with and without overrides equal to its own decisions."""
    Z, A, H, K, B, T = 5, 12, 16, 3, 9, 6
    cfg = _cfg(Z, A, H, K, **flags)
    w = synth.weights(cfg, seed=37, std=0.4)
    z0 = synth.z0(B, Z, seed=37)
    mk = synth.mask(T, B, A, 0.5, seed=37)
    rng = np.random.default_rng(37)
    h0 = (0.3 * rng.standard_normal((B, H))).astype(np.float32)
    c0 = (0.3 * rng.standard_normal((B, H))).astype(np.float32)
    done0 = (np.arange(B) == 4).astype(np.uint8)
    off, t0 = 1000, 17
    out = orc.rollout(cfg, w, z0, mk, T, episode_offset=off, t0=t0, h0=h0, c0=c0, done0=done0,
                      want_seq=True)
    ep = off + np.arange(B)
    for t in range(T):
        h = h0 if t == 0 else out["h_seq"][t - 1]
        c = c0 if t == 0 else out["c_seq"][t - 1]
        fr = _frozen_before(out, t, cfg, done0)
        for over in (False, True):
            kw = {}
            if over:
                kw = dict(a_use=out["actions"][t], h_use=out["h_seq"][t], k_use=out["comp_seq"][t])
            s = orc.step(cfg, w, ep, t0 + t, out["z"][t], h, c, frozen=fr, mask=mk[t], **kw)
            assert np.array_equal(s["action"], out["actions"][t])
            assert np.array_equal(s["ctrl_margin"], out["ctrl_margin"][t])
            assert np.array_equal(s["h"], out["h_seq"][t])
            assert np.array_equal(s["c"], out["c_seq"][t])
            assert np.array_equal(s["mdn"], out["mdn_seq"][t])
            assert np.array_equal(s["reward"], out["rewards"][t])
            assert np.array_equal(s["done"], out["done"][t])
            assert np.array_equal(s["done_margin"], out["done_margin"][t])
            assert np.array_equal(s["comp"], out["comp_seq"][t])
            assert np.array_equal(s["comp_margin"], out["comp_margin"][t])
            assert np.array_equal(s["z_next"], out["z"][t + 1])


def test_step_overrides_change_only_what_follows_them(orc):
    """a_use drives the LSTM (torch LSTMCell with that one-hot row), h_use drives the heads
    (torch linear), k_use picks the component z is drawn from (mu_k + sigma_k eps)."""
    Z, A, H, K, B = 4, 10, 12, 3, 7
    cfg = _cfg(Z, A, H, K)
    w = synth.weights(cfg, seed=38, std=0.4)
    rng = np.random.default_rng(38)
    z = rng.standard_normal((B, Z)).astype(np.float32)
    h = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    c = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    ep = 50 + np.arange(B)
    base = orc.step(cfg, w, ep, 3, z, h, c)
    a_use = (base["action"] + 1) % A
    a_use[0] = -1
    hu = (0.5 * rng.standard_normal((B, H))).astype(np.float32)
    ku = ((base["comp"].astype(np.int64) + 1) % K).astype(np.uint8)
    s = orc.step(cfg, w, ep, 3, z, h, c, a_use=a_use, h_use=hu, k_use=ku)
    # decisions and margins stay the oracle's own
    assert np.array_equal(s["action"], base["action"])
    assert np.array_equal(s["ctrl_margin"], base["ctrl_margin"])
    # LSTM with the forced action row
    Wl = torch.from_numpy(w["W_lstm"]).double()
    cell = torch.nn.LSTMCell(Z + A, H, dtype=torch.float64)
    with torch.no_grad():
        cell.weight_ih.copy_(Wl[:Z + A].T)
        cell.weight_hh.copy_(Wl[Z + A:].T)
        cell.bias_ih.copy_(torch.from_numpy(w["b_lstm"]).double())
        cell.bias_hh.zero_()
        oh = torch.zeros(B, A, dtype=torch.float64)
        ok = a_use >= 0
        oh[np.nonzero(ok)[0], a_use[ok]] = 1.0
        hr, cr = cell(torch.cat([torch.from_numpy(z).double(), oh], 1),
                      (torch.from_numpy(h).double(), torch.from_numpy(c).double()))
    np.testing.assert_allclose(s["h"], hr.numpy(), atol=2e-6, rtol=0)
    np.testing.assert_allclose(s["c"], cr.numpy(), atol=2e-6, rtol=0)
    # heads read h_use
    hu64 = torch.from_numpy(hu).double()
    mdn = torch.nn.functional.linear(hu64, torch.from_numpy(w["W_mdn"]).double().T,
                                     torch.from_numpy(w["b_mdn"]).double()).numpy()
    np.testing.assert_allclose(s["mdn"], mdn, atol=1e-5, rtol=1e-6)
    np.testing.assert_allclose(s["reward"], hu.astype(np.float64) @ w["w_rew"] + w["b_rew"], atol=1e-6)
    # z drawn from the forced component with the step's own normal
    for b in range(B):
        for d in range(Z):
            r = orc.draw(0, int(ep[b]), 3, 1, d // 4)
            p = (d % 4) // 2
            e0, e1 = orc.box_muller(int(r[2 * p]), int(r[2 * p + 1]))
            eps = e0 if d % 2 == 0 else e1
            k = int(ku[b, d])
            ref = mdn[b, K * Z + d * K + k] + math.exp(mdn[b, 2 * K * Z + d * K + k]) * eps
            assert s["z_next"][b, d] == pytest.approx(ref, abs=1e-5)
    # the done flag follows the action taken (NO-OP forced on episode 1)
    cfg2 = dict(cfg, noop_terminates=1)
    a2 = base["action"].copy()
    a2[1] = A - 1
    s2 = orc.step(cfg2, w, ep, 3, z, h, c, a_use=a2)
    assert s2["done"][1] == 1


def test_step_frozen_rows(orc):
    Z, A, H, K, B = 3, 6, 8, 2, 4
    cfg = _cfg(Z, A, H, K)
    w = synth.weights(cfg, seed=39)
    rng = np.random.default_rng(39)
    z = rng.standard_normal((B, Z)).astype(np.float32)
    h = rng.standard_normal((B, H)).astype(np.float32)
    c = rng.standard_normal((B, H)).astype(np.float32)
    fr = np.array([1, 0, 1, 0], np.uint8)
    s = orc.step(cfg, w, np.arange(B), 0, z, h, c, frozen=fr)
    for b in (0, 2):
        assert s["action"][b] == -1 and s["reward"][b] == 0 and s["done"][b] == 1
        assert np.array_equal(s["z_next"][b], z[b]) and np.array_equal(s["h"][b], h[b])
        assert np.array_equal(s["c"][b], c[b]) and np.all(s["mdn"][b] == 0)
        assert np.all(s["comp"][b] == 255) and s["ctrl_margin"][b] == np.inf
    assert np.all(s["action"][[1, 3]] >= 0)
