"""Pins of the CPU oracle to things other than itself (no GPU needed).

Each test ties one piece of the oracle to a published value, a closed form, a
library routine that computes the same thing independently, brute force on a
tiny input, or a statistical law -- chosen so that a dropped term, a wrong
sign or index, or a transposed operand fails at least one of them.
"""
import math
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _zero_weights(Z, A, H, K):
    return {"W_lstm": np.zeros((Z + A + H, 4 * H), np.float32), "b_lstm": np.zeros(4 * H, np.float32),
            "W_mdn": np.zeros((H, 3 * K * Z), np.float32), "b_mdn": np.zeros(3 * K * Z, np.float32),
            "w_rew": np.zeros(H, np.float32), "b_rew": 0.0, "w_done": np.zeros(H, np.float32),
            "b_done": 0.0, "W_ctrl": np.zeros((Z + H, A), np.float32),
            "b_ctrl": np.zeros(A, np.float32)}


def _cfg(Z, A, H, K, **kw):
    c = dict(z_dim=Z, a_dim=A, h_dim=H, k_mix=K, precision="fp32", mdn_tau=1.0,
             sigma_sqrt_tau=0, ctrl_sample=0, ctrl_tau=1.0, done_terminates=0,
             noop_terminates=0, seed=0)
    c.update(kw)
    return c


# ----------------------------------------------------------------------------- Philox
def test_philox_known_answer_vectors(orc):
    """Published Philox-4x32-10 known-answer vectors (Salmon et al., SC'11)."""
    n = 0
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            v = [int(x, 16) for x in line.split()]
            out = orc.philox4x32_10(v[0:4], v[4:6])
            assert [int(x) for x in out] == v[6:10]
            n += 1
    assert n == 3


_TRITON_SCRIPT = r"""
import os, sys
os.environ["TRITON_INTERPRET"] = "1"
import numpy as np, torch, triton, triton.language as tl
@triton.jit
def k(out_ptr, seed, c_ptr):
    i = tl.arange(0, 4)
    c0 = tl.load(c_ptr + 0 + i * 0); c1 = tl.load(c_ptr + 1 + i * 0)
    c2 = tl.load(c_ptr + 2 + i * 0); c3 = tl.load(c_ptr + 3 + i * 0)
    a, b, c, d = tl.philox(seed, c0, c1, c2, c3, 10)
    tl.store(out_ptr + i * 4 + 0, a); tl.store(out_ptr + i * 4 + 1, b)
    tl.store(out_ptr + i * 4 + 2, c); tl.store(out_ptr + i * 4 + 3, d)
rows = np.loadtxt(sys.argv[1], dtype=np.uint64).reshape(-1, 6)
for r in rows:
    out = torch.zeros(16, dtype=torch.uint32)
    c = torch.from_numpy(r[:4].astype(np.uint32).view(np.int32).copy()).view(torch.uint32)
    k[(1,)](out, int(r[4]) | (int(r[5]) << 32), c)
    print(" ".join(str(int(v) & 0xffffffff) for v in out[:4]))
"""


def test_philox_matches_independent_library(orc, tmp_path):
    """Random counters and keys against Triton's own Philox, run in its CPU interpreter."""
    pytest.importorskip("triton")
    rng = np.random.default_rng(7)
    rows = rng.integers(0, 2**32, size=(24, 6), dtype=np.uint64)
    np.savetxt(tmp_path / "in.txt", rows, fmt="%d")
    script = tmp_path / "tri.py"
    script.write_text(_TRITON_SCRIPT)
    env = dict(os.environ, TRITON_INTERPRET="1")
    res = subprocess.run([sys.executable, str(script), str(tmp_path / "in.txt")], env=env,
                         capture_output=True, text=True, timeout=600)
    if res.returncode != 0:
        pytest.skip("triton interpreter unavailable: " + res.stderr.strip().splitlines()[-1])
    got = [list(map(int, ln.split())) for ln in res.stdout.strip().splitlines()]
    for r, ref in zip(rows, got):
        out = orc.philox4x32_10([int(x) for x in r[:4]], [int(r[4]), int(r[5])])
        assert [int(x) for x in out] == ref


def test_draw_counter_layout(orc):
    """Counter = (episode lo, step, purpose<<24 | block, episode hi); key = seed (lo, hi)."""
    seed, ep, step, purpose, block = 0x0123456789ABCDEF, 0x1_0000_0005, 77, 3, 9
    out = orc.draw(seed, ep, step, purpose, block)
    ref = orc.philox4x32_10([ep & 0xFFFFFFFF, step, (purpose << 24) | block, ep >> 32],
                            [seed & 0xFFFFFFFF, seed >> 32])
    assert list(out) == list(ref)


# ----------------------------------------------------------------------------- uniforms / normals
def test_uniform_closed_forms(orc):
    assert orc.uniform(0) == 0.0
    assert orc.uniform(0xFF) == 0.0
    assert orc.uniform(0x100) == 2.0**-24
    assert orc.uniform(0xFFFFFFFF) == 1.0 - 2.0**-24
    xs = np.random.default_rng(1).integers(0, 2**32, 2000, dtype=np.uint64)
    us = np.array([orc.uniform(int(x)) for x in xs])
    assert np.all(us.astype(np.float32).astype(np.float64) == us)  # exact in fp32
    assert np.all((us >= 0) & (us < 1))


def test_box_muller_closed_forms_and_law(orc):
    from scipy import stats
    # u1 = 0 -> radius 0
    assert orc.box_muller(0, 12345 << 8) == (0.0, 0.0)
    # u2 = 0 -> angle 0: (r, 0);  u2 = 1/4 -> (0, r)
    x1 = 0x80000000  # u1 = 1/2
    r = math.sqrt(-2.0 * math.log(0.5))
    e0, e1 = orc.box_muller(x1, 0)
    assert e0 == pytest.approx(r, abs=1e-15) and e1 == 0.0
    e0, e1 = orc.box_muller(x1, 0x40000000)
    assert e0 == pytest.approx(0.0, abs=1e-15) and e1 == pytest.approx(r, abs=1e-15)
    # the law: Philox-driven normals are N(0,1) (KS test against scipy)
    eps = []
    for i in range(4000):
        w = orc.draw(0, i, 0, 1, 0)
        a, b = orc.box_muller(int(w[0]), int(w[1]))
        c, d = orc.box_muller(int(w[2]), int(w[3]))
        eps += [a, b, c, d]
    eps = np.array(eps)
    assert stats.kstest(eps, "norm").pvalue > 1e-3
    assert abs(eps.mean()) < 5 / math.sqrt(len(eps))
    assert abs(eps.var() - 1.0) < 5 * math.sqrt(2.0 / len(eps))


# ----------------------------------------------------------------------------- bf16
def test_bf16_round_matches_torch(orc):
    rng = np.random.default_rng(3)
    bits = list(rng.integers(0, 2**32, 20000, dtype=np.uint64))
    special = [0x00000000, 0x80000000, 0x3F808000, 0x3F818000, 0x3F80FFFF, 0x3F817FFF,
               0x7F7FFFFF, 0xFF7FFFFF, 0x7F800000, 0xFF800000, 0x00000001, 0x00008000,
               0x00018000, 0x807FFFFF, 0x7F7F8000, 0x7F7F7FFF, 0x7FC00000, 0x7F800001, 0xFFFFFFFF]
    bits = np.array([int(b) for b in bits] + special, dtype=np.uint64).astype(np.uint32)
    xs = bits.view(np.float32)
    ref = torch.from_numpy(xs.copy()).to(torch.bfloat16).to(torch.float32).numpy()
    got = orc.bf16_array(xs)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan].view(np.uint32), ref[~nan].view(np.uint32))


# ----------------------------------------------------------------------------- LSTM (a3, a4)
def _torch_lstm_reference(cfg, w, z_seq, acts, round_bf16=False):
    """torch.nn.LSTMCell (float64) with W_ih = [W_z; W_a]^T, W_hh = W_h^T, b_ih = b, b_hh = 0."""
    Z, A, H = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"]
    Wl = torch.from_numpy(w["W_lstm"]).double()
    if round_bf16:
        Wl = Wl.to(torch.bfloat16).double()
    cell = torch.nn.LSTMCell(Z + A, H).double()
    with torch.no_grad():
        cell.weight_ih.copy_(Wl[:Z + A].T)
        cell.weight_hh.copy_(Wl[Z + A:].T)
        cell.bias_ih.copy_(torch.from_numpy(w["b_lstm"]).double())
        cell.bias_hh.zero_()
    T, N = acts.shape
    h = torch.zeros(N, H, dtype=torch.float64)
    c = torch.zeros(N, H, dtype=torch.float64)
    hs, cs = [], []
    for t in range(T):
        z = torch.from_numpy(z_seq[t]).double()
        hin = h.float().double()
        if round_bf16:
            z = z.to(torch.bfloat16).double()
            hin = h.float().to(torch.bfloat16).double()
        a = torch.from_numpy(acts[t]).long()
        onehot = torch.zeros(N, A, dtype=torch.float64)
        ok = a >= 0
        onehot[ok.nonzero()[:, 0], a[ok]] = 1.0
        with torch.no_grad():
            h, c = cell(torch.cat([z, onehot], 1), (hin, c))
        hs.append(h.clone())
        cs.append(c.clone())
    return torch.stack(hs).numpy(), torch.stack(cs).numpy()


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_lstm_matches_torch_lstmcell(orc, precision):
    cfg = _cfg(8, 12, 16, 3, precision=precision)
    w = synth.weights(cfg, seed=5, std=0.3)
    zs, acts, _ = synth.teacher_inputs(6, 5, 8, 12, seed=5)
    acts[2, 1] = -1  # no action row
    out = orc.mdn_nll(cfg, w, zs, acts, want_seq=True)
    hr, cr = _torch_lstm_reference(cfg, w, zs, acts, round_bf16=(precision == "bf16"))
    np.testing.assert_allclose(out["h_seq"], hr, atol=2e-6, rtol=0)
    np.testing.assert_allclose(out["c_seq"], cr, atol=2e-6, rtol=0)


def test_lstm_zero_weights_closed_form(orc):
    """Zero weights: i = f = o = 1/2, g = 0, so c_t = c_0 2^-t and h_t = tanh(c_t)/2."""
    Z, A, H, K, B, T = 4, 8, 16, 2, 3, 7
    cfg = _cfg(Z, A, H, K)
    w = _zero_weights(Z, A, H, K)
    rng = np.random.default_rng(0)
    c0 = rng.standard_normal((B, H)).astype(np.float32)
    h0 = rng.standard_normal((B, H)).astype(np.float32)
    z0 = rng.standard_normal((B, Z)).astype(np.float32)
    out = orc.rollout(cfg, w, z0, None, T, h0=h0, c0=c0, want_seq=True)
    for t in range(T):
        ct = c0.astype(np.float64) * 2.0 ** -(t + 1)
        np.testing.assert_allclose(out["c_seq"][t], ct, rtol=1e-6, atol=0)
        np.testing.assert_allclose(out["h_seq"][t], 0.5 * np.tanh(ct), rtol=1e-6, atol=1e-12)
    # all logits equal -> lowest valid index; zero MDN -> pi uniform, mu 0, sigma 1 -> z = eps
    assert np.all(out["actions"] == 0)
    for t in range(T):
        for b in range(B):
            w1 = orc.draw(0, b, t, 1, 0)
            e0, e1 = orc.box_muller(int(w1[0]), int(w1[1]))
            e2, e3 = orc.box_muller(int(w1[2]), int(w1[3]))
            np.testing.assert_allclose(out["z"][t + 1, b], [e0, e1, e2, e3], rtol=1e-6, atol=1e-7)
    assert np.all(out["rewards"] == 0.0) and np.all(out["done"] == 0)


def test_zero_weight_rollout_with_mask_offset_and_resume(orc):
    """The same closed form over a whole call with a mask, an episode offset, a resumed step
    and a seed: every step's action is the lowest valid index of that step's mask row (equal
    logits, ties to the lowest index), and z_{t+1} is the episode's own normals for its
    absolute step (counter: episode_offset + b, t0 + t; block d / 4, pair (d mod 4) / 2),
    whatever component is drawn (uniform weights, mu = 0, sigma = 1)."""
    Z, A, H, K, B, T = 6, 40, 8, 3, 5, 6
    off, t0, seed = 1000, 17, 9
    cfg = _cfg(Z, A, H, K, seed=seed)
    w = _zero_weights(Z, A, H, K)
    rng = np.random.default_rng(5)
    valid = rng.random((T, B, A)) < 0.15
    valid[..., A - 1] |= ~valid.any(axis=-1)  # at least one valid action per (t, b)
    valid[2, 1, :] = False
    valid[2, 1, 37] = True  # the only valid action sits in the second mask word
    mask = synth.pack_mask(valid)
    c0 = rng.standard_normal((B, H)).astype(np.float32)
    h0 = rng.standard_normal((B, H)).astype(np.float32)
    z0 = rng.standard_normal((B, Z)).astype(np.float32)
    out = orc.rollout(cfg, w, z0, mask, T, episode_offset=off, t0=t0, h0=h0, c0=c0, want_seq=True)
    np.testing.assert_array_equal(out["actions"], valid.argmax(axis=-1))
    assert out["actions"][2, 1] == 37
    for t in range(T):
        ct = c0.astype(np.float64) * 2.0 ** -(t + 1)
        np.testing.assert_allclose(out["c_seq"][t], ct, rtol=1e-6, atol=0)
        np.testing.assert_allclose(out["h_seq"][t], 0.5 * np.tanh(ct), rtol=1e-6, atol=1e-12)
        for b in range(B):
            want = []
            for d in range(Z):
                r = orc.draw(seed, off + b, t0 + t, 1, d // 4)
                pair = (d % 4) // 2
                e0, e1 = orc.box_muller(int(r[2 * pair]), int(r[2 * pair + 1]))
                want.append(e0 if d % 2 == 0 else e1)
            np.testing.assert_allclose(out["z"][t + 1, b], want, rtol=1e-6, atol=1e-7)
    np.testing.assert_array_equal(out["z"][0], z0)
    assert np.all(out["rewards"] == 0.0) and np.all(out["done"] == 0)


# ----------------------------------------------------------------------------- heads (a5)
@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_mdn_head_matches_torch_linear(orc, precision):
    cfg = _cfg(4, 6, 16, 3, precision=precision)
    w = synth.weights(cfg, seed=11, std=0.3)
    zs, acts, _ = synth.teacher_inputs(5, 4, 4, 6, seed=11)
    out = orc.mdn_nll(cfg, w, zs, acts, want_seq=True)
    h = torch.from_numpy(out["h_seq"]).double()
    Wm = torch.from_numpy(w["W_mdn"]).double()
    if precision == "bf16":
        h = h.to(torch.bfloat16).double()
        Wm = Wm.to(torch.bfloat16).double()
    ref = torch.nn.functional.linear(h, Wm.T, torch.from_numpy(w["b_mdn"]).double()).numpy()
    np.testing.assert_allclose(out["mdn_seq"], ref, atol=1e-5, rtol=1e-6)


def test_reward_and_done_heads_via_rollout(orc):
    """r_t = w_r . h_{t+1} + b_r;  done_t = (w_d . h_{t+1} + b_d > 0)."""
    cfg = _cfg(4, 8, 16, 2)
    w = synth.weights(cfg, seed=2, std=0.4)
    z0 = synth.z0(6, 4, seed=2)
    out = orc.rollout(cfg, w, z0, None, 5, want_seq=True)
    h = out["h_seq"].astype(np.float64)
    r = h @ w["w_rew"].astype(np.float64) + w["b_rew"]
    dl = h @ w["w_done"].astype(np.float64) + w["b_done"]
    np.testing.assert_allclose(out["rewards"], r, atol=1e-6)
    clear = np.abs(dl) > 1e-5
    assert np.array_equal(out["done"][clear], (dl > 0)[clear].astype(np.uint8))


# ----------------------------------------------------------------------------- NLL (a9)
def test_nll_matches_torch_mixture_same_family(orc):
    from torch.distributions import Categorical, MixtureSameFamily, Normal
    Z, A, H, K, N, T = 5, 7, 12, 4, 6, 5
    cfg = _cfg(Z, A, H, K)
    w = synth.weights(cfg, seed=4, std=0.4)
    zs, acts, _ = synth.teacher_inputs(N, T, Z, A, seed=4)
    out = orc.mdn_nll(cfg, w, zs, acts, want_seq=True)
    mdn = torch.from_numpy(out["mdn_seq"]).double().view(T, N, 3, Z, K)
    mix = MixtureSameFamily(Categorical(logits=mdn[:, :, 0]),
                            Normal(mdn[:, :, 1], mdn[:, :, 2].exp()))
    lp = mix.log_prob(torch.from_numpy(zs[1:]).double())  # [T, N, Z]
    ref = -lp.sum(dim=(0, 2)).numpy()
    np.testing.assert_allclose(out["nll"], ref, rtol=1e-5)


def test_nll_k1_is_single_gaussian(orc):
    from torch.distributions import Normal
    Z, A, H, N, T = 6, 5, 10, 4, 3
    cfg = _cfg(Z, A, H, 1)
    w = synth.weights(cfg, seed=8, std=0.4)
    zs, acts, _ = synth.teacher_inputs(N, T, Z, A, seed=8)
    out = orc.mdn_nll(cfg, w, zs, acts, want_seq=True)
    mdn = torch.from_numpy(out["mdn_seq"]).double().view(T, N, 3, Z)
    lp = Normal(mdn[:, :, 1], mdn[:, :, 2].exp()).log_prob(torch.from_numpy(zs[1:]).double())
    np.testing.assert_allclose(out["nll"], -lp.sum(dim=(0, 2)).numpy(), rtol=1e-5)


def test_nll_zero_weights_closed_form(orc):
    """Zero head weights: pi = 1/K, mu = 0, sigma = 1 -> each dim costs ln(2 pi)/2 + z^2/2."""
    Z, A, H, K, N, T = 5, 4, 8, 3, 7, 6
    cfg = _cfg(Z, A, H, K)
    w = _zero_weights(Z, A, H, K)
    zs, acts, _ = synth.teacher_inputs(N, T, Z, A, seed=1)
    out = orc.mdn_nll(cfg, w, zs, acts)
    ref = (0.5 * math.log(2 * math.pi) * T * Z
           + 0.5 * (zs[1:].astype(np.float64) ** 2).sum(axis=(0, 2)))
    np.testing.assert_allclose(out["nll"], ref, rtol=1e-12)


def test_nll_lengths_mask_the_padding(orc):
    """lengths[n] = L sums exactly the first L steps; L = 0 gives 0."""
    Z, A, H, K, N, T = 3, 4, 8, 2, 3, 6
    cfg = _cfg(Z, A, H, K)
    w = synth.weights(cfg, seed=9, std=0.4)
    zs, acts, _ = synth.teacher_inputs(N, T, Z, A, seed=9)
    per = []
    for L in range(T + 1):
        per.append(orc.mdn_nll(cfg, w, zs, acts, lengths=np.full(N, L))["nll"])
    per = np.array(per)
    assert np.all(per[0] == 0.0)
    full = orc.mdn_nll(cfg, w, zs, acts, want_seq=True)
    mdn = full["mdn_seq"].astype(np.float64)
    for L in range(1, T + 1):
        t = L - 1
        step = sum(orc.mixture_nll_1d(mdn[t, n, d * K:(d + 1) * K],
                                      mdn[t, n, K * Z + d * K:K * Z + (d + 1) * K],
                                      mdn[t, n, 2 * K * Z + d * K:2 * K * Z + (d + 1) * K],
                                      zs[t + 1, n, d]) for d in range(Z) for n in [0])
        assert per[L, 0] - per[L - 1, 0] == pytest.approx(step, rel=1e-5, abs=1e-6)
    mixed = orc.mdn_nll(cfg, w, zs, acts, lengths=np.array([0, 3, 6]))["nll"]
    np.testing.assert_allclose(mixed, [per[0, 0], per[3, 1], per[6, 2]], rtol=1e-12)


def test_mixture_density_integrates_to_one(orc):
    from scipy import integrate
    rng = np.random.default_rng(12)
    for K in (1, 2, 3, 5):
        lg = rng.standard_normal(K) * 1.5
        mu = rng.standard_normal(K) * 2.0
        ls = rng.standard_normal(K) * 0.5
        smax = float(np.exp(ls).max())
        lo, hi = float(mu.min()) - 12 * smax, float(mu.max()) + 12 * smax
        val, _ = integrate.quad(lambda x: math.exp(-orc.mixture_nll_1d(lg, mu, ls, x)), lo, hi,
                                limit=400, points=list(mu))
        assert val == pytest.approx(1.0, abs=1e-8)
        # direct long-double sum, no log-sum-exp
        for x in (-1.3, 0.0, 0.7, 2.9):
            p = np.exp(np.longdouble(lg) - np.longdouble(lg).max())
            p = p / p.sum()
            s = np.exp(np.longdouble(ls))
            dens = (p * np.exp(-0.5 * ((np.longdouble(x) - mu) / s) ** 2)
                    / (s * np.sqrt(2 * np.longdouble(math.pi)))).sum()
            assert orc.mixture_nll_1d(lg, mu, ls, x) == pytest.approx(float(-np.log(dens)), rel=1e-12)


# ----------------------------------------------------------------------------- sampling (a6, a7)
def _mixture_rollout(orc, logits, mu, logsig, tau=1.0, sqrt_tau=0, B=3000, Z=8, seed=3):
    K = len(logits)
    cfg = _cfg(Z, 4, 8, K, mdn_tau=tau, sigma_sqrt_tau=sqrt_tau, seed=seed)
    w = _zero_weights(Z, 4, 8, K)
    b = np.zeros((3, Z, K), np.float32)
    b[0] = logits
    b[1] = mu
    b[2] = logsig
    w["b_mdn"] = b.reshape(-1)
    z0 = np.zeros((B, Z), np.float32)
    return orc.rollout(cfg, w, z0, None, 1, want_seq=True)


@pytest.mark.parametrize("tau", [1.0, 0.5, 2.0])
def test_component_frequencies_chi2(orc, tau):
    from scipy import stats
    logits = np.array([0.3, -1.0, 1.2, 0.0, -0.4], np.float32)
    out = _mixture_rollout(orc, logits, np.zeros(5), np.zeros(5), tau=tau)
    comp = out["comp_seq"][0].ravel()
    p = np.exp(logits.astype(np.float64) / tau)
    p /= p.sum()
    counts = np.bincount(comp, minlength=5)
    assert stats.chisquare(counts, p * counts.sum()).pvalue > 1e-4


def test_mixture_moments(orc):
    logits = np.array([0.5, -0.5, 0.1], np.float32)
    mu = np.array([-2.0, 1.0, 3.0], np.float32)
    logsig = np.array([-0.5, 0.2, -1.0], np.float32)
    for sqrt_tau, tau in ((0, 1.0), (1, 0.6)):
        out = _mixture_rollout(orc, logits, mu, logsig, tau=tau, sqrt_tau=sqrt_tau)
        z = out["z"][1].ravel().astype(np.float64)
        p = np.exp(logits.astype(np.float64) / tau)
        p /= p.sum()
        s = np.exp(logsig.astype(np.float64)) * (math.sqrt(tau) if sqrt_tau else 1.0)
        mean = (p * mu).sum()
        var = (p * (s**2 + mu.astype(np.float64) ** 2)).sum() - mean**2
        n = len(z)
        assert abs(z.mean() - mean) < 5 * math.sqrt(var / n)
        assert abs(z.var() - var) < 0.05 * var


def test_tau_zero_is_deterministic_argmax(orc):
    logits = np.array([0.3, 1.7, 1.7, -2.0], np.float32)  # tie: lowest index wins
    mu = np.array([5.0, -1.25, 4.0, 0.0], np.float32)
    out = _mixture_rollout(orc, logits, mu, np.zeros(4), tau=0.0, B=10)
    assert np.all(out["comp_seq"][0] == 1)
    assert np.all(out["z"][1] == np.float32(-1.25))


def test_component_inverse_cdf_boundaries(orc):
    """First k with u < C_k; u beyond the last cumulative weight falls in K-1."""
    lg = np.log(np.array([0.25, 0.25, 0.5], np.float32))
    mu = np.array([0.0, 1.0, 2.0])
    for u, k in ((0.0, 0), (0.2499, 0), (0.25, 1), (0.4999, 1), (0.5, 2), (0.999999, 2)):
        got, z, _ = orc.sample_dim(lg, mu, np.zeros(3), u, 0.0)
        assert got == k and z == mu[k]


# ----------------------------------------------------------------------------- controller (a1, a2)
def test_masked_argmax_brute_force(orc):
    rng = np.random.default_rng(21)
    for trial in range(300):
        A = int(rng.integers(1, 90))
        lg = rng.standard_normal(A).astype(np.float32)
        if trial % 3 == 0:
            lg = np.round(lg)  # many exact ties
        valid = rng.random(A) < rng.uniform(0.05, 1.0)
        mw = synth.pack_mask(valid[None])[0]
        a, _ = orc.select_action(lg, mw)
        if not valid.any():
            assert a == -1
            continue
        ref = int(np.argmax(np.where(valid, lg, -np.inf)))  # numpy: first maximum
        assert a == ref and valid[a]


def test_sampled_action_frequencies(orc):
    from scipy import stats
    A, tau = 10, 0.7
    lg = np.linspace(-1, 1, A).astype(np.float32)
    valid = np.array([1, 0, 1, 1, 0, 1, 1, 1, 0, 1], bool)
    mw = synth.pack_mask(valid[None])[0]
    n = 20000
    counts = np.zeros(A)
    for i in range(n):
        u = (i + 0.5) / n  # stratified: frequencies follow the CDF exactly
        a, _ = orc.select_action(lg, mw, ctrl_sample=1, ctrl_tau=tau, u=u)
        counts[a] += 1
    p = np.where(valid, np.exp(lg.astype(np.float64) / tau), 0.0)
    p /= p.sum()
    assert np.all(counts[~valid] == 0)
    np.testing.assert_allclose(counts / n, p, atol=2.0 / n)
    # and with Philox uniforms
    counts = np.zeros(A)
    for i in range(4000):
        u = orc.uniform(int(orc.draw(0, i, 0, 2, 0)[0]))
        counts[orc.select_action(lg, mw, 1, tau, u)[0]] += 1
    assert stats.chisquare(counts[valid], p[valid] * 4000).pvalue > 1e-4


def test_controller_is_linear_in_z_and_h(orc):
    """Actions equal a numpy masked argmax of W_c^T [z_t; h_t] + b_c (clear gaps only)."""
    Z, A, H, K, B, T = 6, 20, 16, 2, 12, 6
    cfg = _cfg(Z, A, H, K)
    w = synth.weights(cfg, seed=13, std=0.5)
    z0 = synth.z0(B, Z, seed=13)
    m = synth.mask(T, B, A, 0.4, seed=13)
    out = orc.rollout(cfg, w, z0, m, T, want_seq=True)
    checked = 0
    for t in range(T):
        h = np.zeros((B, H)) if t == 0 else out["h_seq"][t - 1].astype(np.float64)
        x = np.concatenate([out["z"][t].astype(np.float64), h], 1)
        lg = x @ w["W_ctrl"].astype(np.float64) + w["b_ctrl"]
        bits = np.unpackbits(m[t].view(np.uint8), axis=1, bitorder="little")[:, :A].astype(bool)
        ml = np.where(bits, lg, -np.inf)
        srt = np.sort(ml, axis=1)
        for b in range(B):
            if srt[b, -1] - srt[b, -2] > 1e-4:
                assert out["actions"][t, b] == int(np.argmax(ml[b]))
                checked += 1
    assert checked > 0.9 * B * T


# ----------------------------------------------------------------------------- invariants
def test_rollout_sharding_is_bit_exact(orc):
    cfg, w, z0, m, B, T = synth.rollout_inputs("tiny_fp32", B=8, T=6)
    full = orc.rollout(cfg, w, z0, m, T)
    lo = orc.rollout(cfg, w, z0[:3], m[:, :3], T, episode_offset=0)
    hi = orc.rollout(cfg, w, z0[3:], m[:, 3:], T, episode_offset=3)
    for k in ("z", "actions", "rewards", "done"):
        assert np.array_equal(np.concatenate([lo[k], hi[k]], axis=1), full[k])


def test_rollout_resume_is_bit_exact(orc):
    cfg, w, z0, m, B, T = synth.rollout_inputs("tiny_fp32", B=5, T=8)
    cfg["done_terminates"] = 1
    full = orc.rollout(cfg, w, z0, m, T)
    a = orc.rollout(cfg, w, z0, m[:3], 3)
    done_at = a["done"][-1]
    b = orc.rollout(cfg, w, a["z"][-1], m[3:], T - 3, t0=3, h0=a["h_final"], c0=a["c_final"],
                    done0=done_at)
    assert np.array_equal(np.concatenate([a["z"], b["z"][1:]]), full["z"])
    for k in ("actions", "rewards", "done"):
        assert np.array_equal(np.concatenate([a[k], b[k]]), full[k])


def test_done_freezes_episode(orc):
    cfg = _cfg(4, 8, 8, 2, done_terminates=1)
    w = synth.weights(cfg, seed=1, std=0.3)
    w["w_done"][:] = 0
    w["b_done"] = 1.0  # done at the first step
    z0 = synth.z0(3, 4, seed=1)
    out = orc.rollout(cfg, w, z0, None, 4, want_seq=True)
    assert np.all(out["done"] == 1)
    assert np.all(out["actions"][1:] == -1) and np.all(out["rewards"][1:] == 0)
    assert np.all(out["z"][2:] == out["z"][1])
    assert np.all(out["h_seq"][1:] == out["h_seq"][0])
    assert np.all(out["comp_seq"][1:] == 255) and np.all(out["mdn_seq"][1:] == 0)
    # without done_terminates the done flag is only reported
    cfg["done_terminates"] = 0
    out2 = orc.rollout(cfg, w, z0, None, 4)
    assert np.all(out2["done"] == 1) and np.all(out2["actions"] >= 0)


def test_noop_terminates(orc):
    cfg = _cfg(4, 8, 8, 2, noop_terminates=1)
    w = _zero_weights(4, 8, 8, 2)
    w["b_ctrl"][-1] = 1.0  # NO-OP (last action) wins
    out = orc.rollout(cfg, w, np.zeros((2, 4), np.float32), None, 3)
    assert list(out["actions"][:, 0]) == [7, -1, -1]
    assert list(out["done"][:, 0]) == [1, 1, 1]


def test_no_valid_action(orc):
    cfg = _cfg(4, 40, 8, 2)
    w = synth.weights(cfg, seed=3)
    m = np.zeros((2, 2, 2), np.uint32)
    m[1, 1, 1] = 1 << 3  # only action 35 valid for episode 1 at t=1
    out = orc.rollout(cfg, w, synth.z0(2, 4), m, 2)
    assert list(out["actions"][0]) == [-1, -1] and list(out["actions"][1]) == [-1, 35]


def test_synthetic_inputs_are_seeded_and_prefix_stable():
    cfg, w, z0, m, B, T = synth.rollout_inputs("tiny_fp32")
    cfg2, w2, z02, m2, _, _ = synth.rollout_inputs("tiny_fp32")
    assert np.array_equal(z0, z02) and np.array_equal(m, m2)
    assert all(np.array_equal(np.asarray(w[k]), np.asarray(w2[k])) for k in w)
    small = synth.rollout_inputs("tiny_fp32", B=5)
    assert np.array_equal(small[2], z0[:5]) and np.array_equal(small[3], m[:, :5])
    dens = np.unpackbits(m.view(np.uint8)).mean()
    assert abs(dens - 0.5) < 0.02
