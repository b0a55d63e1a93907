"""Comparison rules shared by the GPU parity tests.

Free-running rollouts are checked step by step against the oracle started from
the GPU's own state (step-anchored parity).  For every step t of every checked
episode, the oracle replays the step from the state the GPU entered it with
(z_t, h_{t-1}, c_{t-1} and whether the episode was frozen), so every step is
compared, however far the two trajectories would have drifted apart if each
had run on its own:

  * decisions (action, done, mixture component of every latent dim) must equal
    the oracle's, except where the oracle's own margin puts it within a hair
    of the decision boundary:
      - controller argmax: top-2 logit gap < 1e-3;
      - sampled controller action: |u*S - cumsum| / S < 1e-4;
      - mixture component: |u - C_k| < 1e-4 for the nearest cumulative weight;
      - done: |done logit| < 1e-4;
    such excused flips must be < 0.1% of the draws;
  * values (h', c', head outputs, reward, z_{t+1}) must be within max-abs 1e-4
    (fp32 path) or 2e-2 (bf16 path) of the oracle's.  The bf16 path is held to
    2e-2 of both the bf16-emulating oracle and the plain fp32 oracle.

To keep every value comparable after an excused flip, the replay takes the
GPU's decisions downstream of the oracle's own: its action row into the LSTM,
its h' into the heads (the second state point inside a step) and its
components into z_{t+1}.  The oracle still reports its own decisions, and each
GPU decision is checked against them.  The teacher-forced check compares the
GPU's whole chain with the oracle's directly.
"""
from __future__ import annotations

import os

import numpy as np

TOL = {"fp32": 1e-4, "bf16": 2e-2}
CTRL_GAP, CTRL_SAMPLE_GAP, COMP_GAP, DONE_GAP = 1e-3, 1e-4, 1e-4, 1e-4
NT = os.cpu_count() or 1


def np_(x):
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return x.detach().cpu().numpy()
    except ImportError:
        pass
    return np.asarray(x)


def check_rollout(g: dict, cfg: dict, weights: dict, z0, mask=None, episodes=None, t0: int = 0,
                  h0=None, c0=None, done0=None, orc=None, nthreads: int = NT, rt0=None,
                  mem0=None, loc_mask=None) -> dict:
    """Step-anchored parity of a GPU rollout of B episodes.

    g: the GPU's outputs with their per-step sequences (z, actions, rewards, done,
    h_seq, c_seq, mdn_seq, comp_seq; optional h_final, c_final), batch axis = the
    checked episodes.  z0, mask [T, B, W], h0, c0, done0: the inputs of those
    episodes.  episodes: their global Philox indices (default 0..B-1); t0: the
    global index of step 0.  With the shaped reward, rt0 / mem0 are the predictions
    entering the call and g carries rt_seq / mem_seq; with a hierarchical action, loc_mask
    [T, B, NX, WL] are the location masks and g carries loc_actions."""
    if orc is None:
        import oracle as orc
    prec = cfg.get("precision", "fp32")
    tol = TOL[prec]
    sampled = bool(cfg.get("ctrl_sample", 0)) and cfg.get("ctrl_tau", 1.0) > 0
    ctrl_thr = CTRL_SAMPLE_GAP if sampled else CTRL_GAP
    Z, A, H, K = (int(cfg[k]) for k in ("z_dim", "a_dim", "h_dim", "k_mix"))
    ga, gd, gr = np_(g["actions"]), np_(g["done"]), np_(g["rewards"])
    gz, gh, gc = np_(g["z"]), np_(g["h_seq"]), np_(g["c_seq"])
    gm, gk = np_(g["mdn_seq"]), np_(g["comp_seq"])
    T, B = ga.shape
    ep = np.arange(B, dtype=np.uint64) if episodes is None else np.asarray(episodes, np.uint64)
    assert np.array_equal(gz[0], np.asarray(z0, np.float32)), "z_out[0] must be z0"
    h = np.zeros((B, H), np.float32) if h0 is None else np.asarray(h0, np.float32)
    c = np.zeros((B, H), np.float32) if c0 is None else np.asarray(c0, np.float32)
    frozen = np.zeros(B, bool) if done0 is None else np.asarray(done0).astype(bool)
    shaped = int(cfg.get("reward_mode", 0)) == 1
    g_lp = np_(g["logp_seq"]) if g.get("logp_seq") is not None else None
    hier = int(cfg.get("n_xfers", 0)) > 0
    g_loc = np_(g["loc_actions"]) if hier else None
    g_v = np_(g["value_seq"]) if g.get("value_seq") is not None else None
    if shaped:
        rt, mem = np.asarray(rt0, np.float32), np.asarray(mem0, np.float32)
        g_rt, g_mem = np_(g["rt_seq"]), np_(g["mem_seq"])
    refs = [(cfg, tol)]
    if prec == "bf16":
        refs.append((dict(cfg, precision="fp32"), TOL["bf16"]))
    st = {"flips": 0, "draws": 0, "compared": 0, "frozen_steps": 0, "worst": 0.0,
          "kinds": {"action": 0, "done": 0, "component": 0}, "flip_margins": []}

    def flip(kind, margin):
        st["flips"] += 1
        st["kinds"][kind] += 1
        st["flip_margins"].append(float(margin))

    last = None
    for t in range(T):
        mk = None if mask is None else np.asarray(mask)[t]
        for ri, (rcfg, rtol) in enumerate(refs):
            sk = dict(rt=rt, mem=mem) if shaped else {}
            if hier:
                sk.update(loc_use=g_loc[t], loc_mask=None if loc_mask is None else np.asarray(loc_mask)[t])
            s = orc.step(rcfg, weights, ep, t0 + t, gz[t], h, c, frozen=frozen, mask=mk,
                         a_use=ga[t], h_use=gh[t], k_use=gk[t], nthreads=nthreads, **sk)
            if ri == 0:
                last = s
            live = ~frozen
            where = f"t={t}"
            # values downstream of the shared decisions
            vals = [("h", gh[t], s["h"]), ("c", gc[t], s["c"]), ("mdn", gm[t], s["mdn"]),
                    ("reward", gr[t], s["reward"]), ("z", gz[t + 1], s["z_next"])]
            if shaped:
                vals += [("rt", g_rt[t], s["rt"]), ("mem", g_mem[t], s["mem"])]
            if g_lp is not None:
                vals.append(("logp", g_lp[t], s["logp"]))
            if g_v is not None:
                vals.append(("value", g_v[t], s["value"]))
            for key, gv, ov in vals:
                e = np.abs(gv.astype(np.float64) - ov.astype(np.float64))
                e = e.reshape(B, -1).max(axis=1) if e.ndim > 1 else e
                bad = np.nonzero(live & (e > rtol))[0]
                assert not len(bad), (f"{key} {where} episodes {ep[bad][:8]} err {e[bad][:8]} "
                                      f"(tol {rtol}, {rcfg['precision']} oracle)")
                if ri == 0 and live.any():
                    st["worst"] = max(st["worst"], float(e[live].max()))
            if ri:
                continue
            # frozen rows are exact copies
            fz = np.nonzero(frozen)[0]
            if len(fz):
                assert np.all(ga[t, fz] == -1) and np.all(gd[t, fz] == 1), where
                assert np.all(gr[t, fz] == 0) and np.all(gk[t, fz] == 255), where
                assert np.array_equal(gz[t + 1, fz], gz[t, fz]), where
                assert np.array_equal(gh[t, fz], h[fz]) and np.array_equal(gc[t, fz], c[fz]), where
                assert np.all(gm[t, fz] == 0), where
                if shaped:
                    assert np.array_equal(g_rt[t, fz], rt[fz]) and np.array_equal(g_mem[t, fz], mem[fz]), where
                if g_lp is not None:
                    assert np.all(g_lp[t, fz] == 0), where
                if g_v is not None:
                    assert np.all(g_v[t, fz] == 0), where
                if hier:
                    assert np.all(g_loc[t, fz] == -1), where
                st["frozen_steps"] += len(fz)
            # decisions: equal, or excused by the oracle's own margin
            nl = int(live.sum())
            st["draws"] += nl * (Z + 2)
            st["compared"] += nl
            for b in np.nonzero(live & (ga[t] != s["action"]))[0]:
                m = s["ctrl_margin"][b]
                assert m < ctrl_thr, (f"action {where} episode {ep[b]}: gpu {ga[t, b]} oracle "
                                      f"{s['action'][b]} margin {m}")
                flip("action", m)
            if hier:  # the location: a second decision (counted with the action's draws)
                for b in np.nonzero(live & (g_loc[t] != s["loc"]))[0]:
                    m = s["loc_margin"][b]
                    assert m < ctrl_thr, (f"location {where} episode {ep[b]}: gpu {g_loc[t, b]} "
                                          f"oracle {s['loc'][b]} margin {m}")
                    flip("action", m)
            for b in np.nonzero(live & (gd[t] != s["done"]))[0]:
                m = s["done_margin"][b]
                assert m < DONE_GAP, (f"done {where} episode {ep[b]}: gpu {gd[t, b]} oracle "
                                      f"{s['done'][b]} margin {m}")
                flip("done", m)
            bb, dd = np.nonzero(live[:, None] & (gk[t] != s["comp"]))
            for b, d in zip(bb, dd):
                m = s["comp_margin"][b, d]
                assert m < COMP_GAP, (f"component {where} episode {ep[b]} dim {d}: gpu "
                                      f"{gk[t, b, d]} oracle {s['comp'][b, d]} margin {m}")
                flip("component", m)
        # the state the GPU carries into the next step
        h, c = gh[t], gc[t]
        if shaped:
            rt, mem = g_rt[t], g_mem[t]
        if cfg.get("done_terminates"):
            frozen = frozen | (gd[t] == 1)
        if cfg.get("noop_terminates"):
            frozen = frozen | (ga[t] == (int(cfg["n_xfers"]) - 1 if hier else A - 1))
    if T > 0 and g.get("h_final") is not None:
        for key, gv in (("h_final", g["h_final"]), ("c_final", g["c_final"])):
            e = float(np.abs(np_(gv).astype(np.float64)
                             - last[key[0]].astype(np.float64)).max()) if B else 0.0
            assert e <= tol, f"{key} err {e}"
    f, d = st["flips"], st["draws"]
    assert f <= max(1, 0.001 * d), f"{f} excused flips in {d} draws: {st['kinds']}"
    return st


def check_free_running(g: dict, o: dict, cfg: dict) -> dict:
    """Compare a GPU rollout with the oracle's own free-running rollout o of the same
    episodes, up to each episode's first decision mismatch, which must be excused by
    the oracle's margin (after it the two trajectories legitimately differ).  Returns
    how many (episode, step) pairs were compared before the first mismatch."""
    tol = TOL[cfg.get("precision", "fp32")]
    sampled = bool(cfg.get("ctrl_sample", 0)) and cfg.get("ctrl_tau", 1.0) > 0
    ctrl_thr = CTRL_SAMPLE_GAP if sampled else CTRL_GAP
    ga, gd, gr, gz = (np_(g[k]) for k in ("actions", "done", "rewards", "z"))
    gk = np_(g["comp_seq"]) if g.get("comp_seq") is not None else None
    T, B = ga.shape
    st = {"compared": 0, "diverged": 0}
    for b in range(B):
        for t in range(T):
            if ga[t, b] != o["actions"][t, b]:
                assert o["ctrl_margin"][t, b] < ctrl_thr, (t, b, o["ctrl_margin"][t, b])
                st["diverged"] += 1
                break
            if gd[t, b] != o["done"][t, b]:
                assert o["done_margin"][t, b] < DONE_GAP, (t, b, o["done_margin"][t, b])
                st["diverged"] += 1
                break
            if gk is not None and not np.array_equal(gk[t, b], o["comp_seq"][t, b]):
                dd = np.nonzero(gk[t, b] != o["comp_seq"][t, b])[0]
                assert np.all(o["comp_margin"][t, b, dd] < COMP_GAP), (t, b, dd)
                st["diverged"] += 1
                break
            assert abs(float(gr[t, b]) - float(o["rewards"][t, b])) <= tol, (t, b)
            e = float(np.abs(gz[t + 1, b] - o["z"][t + 1, b]).max())
            assert e <= tol, (t, b, e)
            st["compared"] += 1
    return st


def check_teacher(g: dict, o: dict, precision: str, nll_rtol: float = 1e-3):
    tol = TOL[precision]
    out = {}
    for k in ("h_seq", "c_seq", "mdn_seq"):
        if g.get(k) is not None:
            e = float(np.abs(np_(g[k]) - o[k]).max())
            out[k] = e
            assert e <= tol, f"{k} max-abs err {e} > {tol}"
    gn = np_(g["nll"]).astype(np.float64)
    on = o["nll"]
    rel = np.abs(gn - on) / np.maximum(np.abs(on), 1e-12)
    zero = on == 0
    assert np.all(gn[zero] == 0)
    out["nll_rel"] = float(rel[~zero].max()) if (~zero).any() else 0.0
    assert out["nll_rel"] <= nll_rtol, f"nll rel err {out['nll_rel']}"
    return out
