"""Plain CPU oracle for the RLFlow world-model dream path (ctypes over wm_oracle.c).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s ``cpu_baseline`` leg / ``--impl reference`` arm may import this
package.  It shares no code with the CUDA product path
(``paper_2205_01435_gb300``) and never imports it.

Every function follows the paper's statement of the world model (RLFlow,
SIGMOD'22): the MDN-RNN that models P(z_{t+1} | a_t, z_t, h_t) (Sec. 3.3.2),
the temperature softmax of the mixture weights (Sec. 3.3.2), the linear
controller a_t = W_c [z_t, h_t] + b_c (Sec. 3.4), invalid-action masking
(Sec. 3.1.3) and the world-model log-likelihood loss (Sec. 4.7).  The
arithmetic lives in ``wm_oracle.c``; this module only marshals arguments.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "wm_oracle.c")
_HDR = os.path.join(_HERE, "wm_oracle.h")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile wm_oracle.c into liboracle.so (plain C11, -O2, OpenMP over episodes)."""
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < newest:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
             "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


class _Cfg(C.Structure):
    _fields_ = [("z_dim", C.c_int), ("a_dim", C.c_int), ("h_dim", C.c_int), ("k_mix", C.c_int),
                ("bf16", C.c_int), ("mdn_tau", C.c_double), ("sigma_sqrt_tau", C.c_int),
                ("ctrl_sample", C.c_int), ("ctrl_tau", C.c_double),
                ("done_terminates", C.c_int), ("noop_terminates", C.c_int),
                ("seed", C.c_uint64), ("nthreads", C.c_int), ("reward_mode", C.c_int),
                ("reward_alpha", C.c_double), ("reward_beta", C.c_double),
                ("invalid_reward", C.c_double), ("pop_size", C.c_int), ("pop_group", C.c_int),
                ("value_head", C.c_int), ("n_xfers", C.c_int), ("state64", C.c_int)]


class _W(C.Structure):
    _fields_ = [("W_lstm", C.c_void_p), ("b_lstm", C.c_void_p), ("W_mdn", C.c_void_p),
                ("b_mdn", C.c_void_p), ("w_rew", C.c_void_p), ("b_rew", C.c_float),
                ("w_done", C.c_void_p), ("b_done", C.c_float), ("W_ctrl", C.c_void_p),
                ("b_ctrl", C.c_void_p), ("w_rt", C.c_void_p), ("b_rt", C.c_float),
                ("w_mem", C.c_void_p), ("b_mem", C.c_float), ("w_val", C.c_void_p),
                ("b_val", C.c_float)]


class _Ext(C.Structure):
    _fields_ = [("rt0", C.c_void_p), ("mem0", C.c_void_p), ("rt_seq", C.c_void_p),
                ("mem_seq", C.c_void_p), ("logp_seq", C.c_void_p), ("value_seq", C.c_void_p),
                ("loc_mask", C.c_void_p), ("loc_seq", C.c_void_p), ("loc_margin", C.c_void_p),
                ("loc_use", C.c_void_p)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P = C.c_void_p
            lib.orc_philox4x32_10.argtypes = [P, P, P]
            lib.orc_uniform.argtypes = [C.c_uint32]
            lib.orc_uniform.restype = C.c_double
            lib.orc_box_muller.argtypes = [C.c_uint32, C.c_uint32, P, P]
            lib.orc_draw.argtypes = [C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint32, P]
            lib.orc_bf16.argtypes = [C.c_float]
            lib.orc_bf16.restype = C.c_float
            lib.orc_lstm_cell.argtypes = [C.c_int, P, P, P, P]
            lib.orc_mixture_nll_1d.argtypes = [C.c_int, P, P, P, C.c_double]
            lib.orc_mixture_nll_1d.restype = C.c_double
            lib.orc_sample_dim.argtypes = [C.c_int, C.c_double, C.c_int, P, P, P, C.c_double,
                                           C.c_double, P, P]
            lib.orc_sample_dim.restype = C.c_int
            lib.orc_select_action.argtypes = [C.c_int, P, P, C.c_int, C.c_double, C.c_double, P]
            lib.orc_select_action.restype = C.c_int
            lib.orc_rollout.argtypes = [P, P, C.c_int, C.c_int, C.c_uint64, C.c_uint32] + [P] * 19
            lib.orc_rollout.restype = C.c_int
            lib.orc_step.argtypes = [P, P, C.c_int, P, C.c_uint32] + [P] * 20
            lib.orc_step.restype = C.c_int
            lib.orc_returns.argtypes = [C.c_int, C.c_int, C.c_double, C.c_int, P, P, P, P,
                                        C.c_uint64, C.c_int, C.c_int, P]
            lib.orc_returns.restype = C.c_int
            lib.orc_mdn_nll_grad.argtypes = [P, P, C.c_int, C.c_int] + [P] * 8
            lib.orc_mdn_nll_grad.restype = C.c_int
            lib.orc_mdn_nll.argtypes = [P, P, C.c_int, C.c_int] + [P] * 7
            lib.orc_mdn_nll.restype = C.c_int
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _cfg(cfg: dict, nthreads: int) -> _Cfg:
    return _Cfg(int(cfg["z_dim"]), int(cfg["a_dim"]), int(cfg["h_dim"]), int(cfg["k_mix"]),
                1 if cfg.get("precision", "fp32") == "bf16" else 0,
                float(cfg.get("mdn_tau", 1.0)), int(cfg.get("sigma_sqrt_tau", 0)),
                int(cfg.get("ctrl_sample", 0)), float(cfg.get("ctrl_tau", 1.0)),
                int(cfg.get("done_terminates", 0)), int(cfg.get("noop_terminates", 0)),
                int(cfg.get("seed", 0)) & 0xFFFFFFFFFFFFFFFF, int(nthreads),
                int(cfg.get("reward_mode", 0)), float(cfg.get("reward_alpha", 0.8)),
                float(cfg.get("reward_beta", 0.2)), float(cfg.get("invalid_reward", -100.0)),
                int(cfg.get("pop_size", 0)), int(cfg.get("pop_group", 1)),
                int(cfg.get("value_head", 0)), int(cfg.get("n_xfers", 0)),
                int(cfg.get("state64", 0)))


class _Weights:
    """Keeps the contiguous fp32 arrays alive while the C struct points at them."""

    def __init__(self, w: dict):
        self.arrs = {k: _f32(w[k]) for k in ("W_lstm", "b_lstm", "W_mdn", "b_mdn", "w_rew",
                                               "w_done", "W_ctrl", "b_ctrl", "w_rt", "w_mem",
                                               "w_val") if w.get(k) is not None}
        a = self.arrs
        self.s = _W(_ptr(a["W_lstm"]), _ptr(a["b_lstm"]), _ptr(a["W_mdn"]), _ptr(a["b_mdn"]),
                    _ptr(a["w_rew"]), float(w["b_rew"]), _ptr(a["w_done"]), float(w["b_done"]),
                    _ptr(a["W_ctrl"]), _ptr(a["b_ctrl"]), _ptr(a.get("w_rt")),
                    float(w.get("b_rt", 0.0)), _ptr(a.get("w_mem")), float(w.get("b_mem", 0.0)),
                    _ptr(a.get("w_val")), float(w.get("b_val", 0.0)))


class _ExtArgs:
    """The optional parts of a call (shaped-reward state, log-probs, values); keeps the
    arrays alive."""

    def __init__(self, cfg: dict, B: int, T: int, rt0=None, mem0=None, loc_mask=None, loc_use=None):
        self.out = {"logp_seq": np.zeros((T, B), np.float32)}
        NX = int(cfg.get("n_xfers", 0))
        lm = lu = None
        if NX > 0:
            WL = (int(cfg["a_dim"]) - NX + 31) // 32
            if loc_mask is not None:
                lm = np.ascontiguousarray(loc_mask, dtype=np.uint32).reshape(T, B, NX, WL)
            if loc_use is not None:
                lu = np.ascontiguousarray(loc_use, dtype=np.int32).reshape(B)
            self.out.update(loc_seq=np.zeros((T, B), np.int32), loc_margin=np.zeros((T, B), np.float32))
        r = m = None
        if int(cfg.get("reward_mode", 0)) == 1:
            if rt0 is None or mem0 is None:
                raise ValueError("the shaped reward needs rt0 and mem0")
            r, m = _f32(rt0).reshape(B), _f32(mem0).reshape(B)
            self.out.update(rt_seq=np.zeros((T, B), np.float32), mem_seq=np.zeros((T, B), np.float32))
        if int(cfg.get("value_head", 0)):
            self.out["value_seq"] = np.zeros((T, B), np.float32)
        self.keep = [r, m, lm, lu]
        o = self.out
        self.s = _Ext(_ptr(r), _ptr(m), _ptr(o.get("rt_seq")), _ptr(o.get("mem_seq")),
                      _ptr(o["logp_seq"]), _ptr(o.get("value_seq")), _ptr(lm),
                      _ptr(o.get("loc_seq")), _ptr(o.get("loc_margin")), _ptr(lu))

    def ref(self):
        return C.byref(self.s)


# ---------------------------------------------------------------- building blocks
def philox4x32_10(ctr, key) -> np.ndarray:
    """Philox-4x32-10 block function (Salmon et al., SC'11)."""
    lib = _load()
    c = np.asarray(ctr, dtype=np.uint32).copy()
    k = np.asarray(key, dtype=np.uint32).copy()
    out = np.zeros(4, dtype=np.uint32)
    lib.orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def draw(seed: int, episode: int, step: int, purpose: int, block: int) -> np.ndarray:
    lib = _load()
    out = np.zeros(4, dtype=np.uint32)
    lib.orc_draw(seed, episode, step, purpose, block, _ptr(out))
    return out


def uniform(x: int) -> float:
    return _load().orc_uniform(int(x) & 0xFFFFFFFF)


def box_muller(x1: int, x2: int):
    e0, e1 = C.c_double(), C.c_double()
    _load().orc_box_muller(x1, x2, C.byref(e0), C.byref(e1))
    return e0.value, e1.value


def bf16(x: float) -> float:
    return _load().orc_bf16(float(x))


def bf16_array(x) -> np.ndarray:
    lib = _load()
    x = np.asarray(x, dtype=np.float32).ravel()
    return np.array([lib.orc_bf16(float(v)) for v in x], dtype=np.float32)


def lstm_cell(gates, c_in):
    gates = np.ascontiguousarray(gates, dtype=np.float64)
    c_in = np.ascontiguousarray(c_in, dtype=np.float64)
    H = c_in.shape[0]
    c_out = np.zeros(H)
    h_out = np.zeros(H)
    _load().orc_lstm_cell(H, _ptr(gates), _ptr(c_in), _ptr(c_out), _ptr(h_out))
    return c_out, h_out


def mixture_nll_1d(logits, mu, logsig, x: float) -> float:
    lg = np.ascontiguousarray(logits, dtype=np.float64)
    m = np.ascontiguousarray(mu, dtype=np.float64)
    s = np.ascontiguousarray(logsig, dtype=np.float64)
    return _load().orc_mixture_nll_1d(lg.shape[0], _ptr(lg), _ptr(m), _ptr(s), float(x))


def sample_dim(logits, mu, logsig, u: float, eps: float, tau: float = 1.0,
               sigma_sqrt_tau: int = 0):
    lg = np.ascontiguousarray(logits, dtype=np.float32)
    m = np.ascontiguousarray(mu, dtype=np.float64)
    s = np.ascontiguousarray(logsig, dtype=np.float64)
    z, mg = C.c_double(), C.c_double()
    k = _load().orc_sample_dim(lg.shape[0], float(tau), int(sigma_sqrt_tau), _ptr(lg), _ptr(m),
                               _ptr(s), float(u), float(eps), C.byref(z), C.byref(mg))
    return k, z.value, mg.value


def select_action(logits, mask_words=None, ctrl_sample: int = 0, ctrl_tau: float = 1.0,
                  u: float = 0.0):
    lg = np.ascontiguousarray(logits, dtype=np.float32)
    mw = None if mask_words is None else np.ascontiguousarray(mask_words, dtype=np.uint32)
    mg = C.c_double()
    a = _load().orc_select_action(lg.shape[0], _ptr(lg), _ptr(mw), int(ctrl_sample),
                                  float(ctrl_tau), float(u), C.byref(mg))
    return a, mg.value


# ---------------------------------------------------------------- the path
def rollout(cfg: dict, weights: dict, z0, mask=None, T: int = 1, episode_offset: int = 0,
            t0: int = 0, h0=None, c0=None, done0=None, want_seq: bool = False,
            nthreads: int = 1, rt0=None, mem0=None, loc_mask=None) -> dict:
    """Free-running dream rollout of B = len(z0) episodes for T steps (a1..a8).
    With the shaped reward (reward_mode 1), rt0 / mem0 [B] are the predictions of the
    current graphs and the result carries rt_seq / mem_seq [T, B]."""
    lib = _load()
    Z, A, H, K = (int(cfg[k]) for k in ("z_dim", "a_dim", "h_dim", "k_mix"))
    z0 = _f32(z0).reshape(-1, Z)
    B = z0.shape[0]
    W = (A + 31) // 32
    h0 = None if h0 is None else _f32(h0).reshape(B, H)
    c0 = None if c0 is None else _f32(c0).reshape(B, H)
    d0 = None if done0 is None else np.ascontiguousarray(done0, dtype=np.uint8).reshape(B)
    mk = None if mask is None else np.ascontiguousarray(mask, dtype=np.uint32).reshape(T, B, W)
    out = {
        "z": np.zeros((T + 1, B, Z), np.float32), "actions": np.zeros((T, B), np.int32),
        "rewards": np.zeros((T, B), np.float32), "done": np.zeros((T, B), np.uint8),
        "h_final": np.zeros((B, H), np.float32), "c_final": np.zeros((B, H), np.float32),
        "ctrl_margin": np.zeros((T, B), np.float32), "comp_margin": np.zeros((T, B, Z), np.float32),
        "done_margin": np.zeros((T, B), np.float32),
    }
    if want_seq:
        out.update(h_seq=np.zeros((T, B, H), np.float32), c_seq=np.zeros((T, B, H), np.float32),
                   mdn_seq=np.zeros((T, B, 3 * K * Z), np.float32),
                   comp_seq=np.zeros((T, B, Z), np.uint8))
    w = _Weights(weights)
    cs = _cfg(cfg, nthreads)
    ext = _ExtArgs(cfg, B, T, rt0, mem0, loc_mask)
    out.update(ext.out)
    rc = lib.orc_rollout(C.byref(cs), C.byref(w.s), B, T, int(episode_offset), int(t0),
                         _ptr(z0), _ptr(h0), _ptr(c0), _ptr(d0), _ptr(mk),
                         _ptr(out["z"]), _ptr(out["actions"]), _ptr(out["rewards"]),
                         _ptr(out["done"]), _ptr(out["h_final"]), _ptr(out["c_final"]),
                         _ptr(out.get("h_seq")), _ptr(out.get("c_seq")), _ptr(out.get("mdn_seq")),
                         _ptr(out.get("comp_seq")), _ptr(out["ctrl_margin"]),
                         _ptr(out["comp_margin"]), _ptr(out["done_margin"]), ext.ref())
    if rc != 0:
        raise ValueError(f"orc_rollout failed ({rc})")
    return out


def step(cfg: dict, weights: dict, episodes, step_index: int, z, h, c, frozen=None, mask=None,
         a_use=None, h_use=None, k_use=None, nthreads: int = 1, rt=None, mem=None,
         loc_mask=None, loc_use=None) -> dict:
    """One dream step (a1..a8) of B = len(episodes) episodes started from the state
    (z [B,Z], h [B,H], c [B,H], frozen [B]); episodes are global Philox indices.
    a_use / h_use / k_use replace what flows downstream of the action, h' and
    component decisions (the returned decisions and margins are the oracle's own).
    With the shaped reward, rt / mem [B] are the predictions entering the step and the
    result carries the step's as "rt" / "mem"."""
    lib = _load()
    Z, A, H, K = (int(cfg[k]) for k in ("z_dim", "a_dim", "h_dim", "k_mix"))
    ep = np.ascontiguousarray(episodes, dtype=np.uint64).reshape(-1)
    B = ep.shape[0]
    W = (A + 31) // 32
    z, h, c = _f32(z).reshape(B, Z), _f32(h).reshape(B, H), _f32(c).reshape(B, H)
    fz = None if frozen is None else np.ascontiguousarray(frozen, dtype=np.uint8).reshape(B)
    mk = None if mask is None else np.ascontiguousarray(mask, dtype=np.uint32).reshape(B, W)
    au = None if a_use is None else np.ascontiguousarray(a_use, dtype=np.int32).reshape(B)
    hu = None if h_use is None else _f32(h_use).reshape(B, H)
    ku = None if k_use is None else np.ascontiguousarray(k_use, dtype=np.uint8).reshape(B, Z)
    out = {"action": np.zeros(B, np.int32), "ctrl_margin": np.zeros(B, np.float32),
           "h": np.zeros((B, H), np.float32), "c": np.zeros((B, H), np.float32),
           "mdn": np.zeros((B, 3 * K * Z), np.float32), "reward": np.zeros(B, np.float32),
           "done": np.zeros(B, np.uint8), "done_margin": np.zeros(B, np.float32),
           "comp": np.zeros((B, Z), np.uint8), "comp_margin": np.zeros((B, Z), np.float32),
           "z_next": np.zeros((B, Z), np.float32)}
    w = _Weights(weights)
    cs = _cfg(cfg, nthreads)
    ext = _ExtArgs(cfg, B, 1, rt, mem, loc_mask, loc_use)
    rc = lib.orc_step(C.byref(cs), C.byref(w.s), B, _ptr(ep), int(step_index) & 0xFFFFFFFF,
                      _ptr(z), _ptr(h), _ptr(c), _ptr(fz), _ptr(mk), _ptr(au), _ptr(hu), _ptr(ku),
                      _ptr(out["action"]), _ptr(out["ctrl_margin"]), _ptr(out["h"]), _ptr(out["c"]),
                      _ptr(out["mdn"]), _ptr(out["reward"]), _ptr(out["done"]),
                      _ptr(out["done_margin"]), _ptr(out["comp"]), _ptr(out["comp_margin"]),
                      _ptr(out["z_next"]), ext.ref())
    if rc != 0:
        raise ValueError(f"orc_step failed ({rc})")
    if "rt_seq" in ext.out:
        out["rt"], out["mem"] = ext.out["rt_seq"][0], ext.out["mem_seq"][0]
    out["logp"] = ext.out["logp_seq"][0]
    if "loc_seq" in ext.out:
        out["loc"], out["loc_margin"] = ext.out["loc_seq"][0], ext.out["loc_margin"][0]
    if "value_seq" in ext.out:
        out["value"] = ext.out["value_seq"][0]
    return out


def returns(rewards, done, gamma: float, stop_at_done: bool = True, bootstrap=None,
            episode_offset: int = 0, pop_size: int = 0, pop_group: int = 1) -> dict:
    """Discounted returns G_t = r_t + gamma G_{t+1} of [T, B] rollouts (from bootstrap [B],
    else 0; a done step ends the sum when stop_at_done) and, with a population, each
    candidate's mean G_0 ("fitness")."""
    lib = _load()
    r = _f32(rewards)
    T, B = r.shape
    d = np.ascontiguousarray(done, dtype=np.uint8).reshape(T, B)
    bs = None if bootstrap is None else _f32(bootstrap).reshape(B)
    out = {"returns": np.zeros((T, B), np.float32)}
    fit = None
    if pop_size >= 1:
        fit = np.zeros(pop_size, np.float64)
        out["fitness"] = fit
    rc = lib.orc_returns(B, T, float(gamma), int(bool(stop_at_done)), _ptr(r), _ptr(d), _ptr(bs),
                         _ptr(out["returns"]), int(episode_offset), int(max(pop_size, 1)),
                         int(pop_group), _ptr(fit))
    if rc != 0:
        raise ValueError(f"orc_returns failed ({rc})")
    return out


def mdn_nll_grad(cfg: dict, weights: dict, z_seq, actions, lengths=None, nthreads: int = 1) -> dict:
    """Gradient of sum_n NLL_n with respect to W_lstm, b_lstm, W_mdn, b_mdn (BPTT, fp64),
    plus the per-sequence NLL."""
    lib = _load()
    Z, A, H, K = (int(cfg[k]) for k in ("z_dim", "a_dim", "h_dim", "k_mix"))
    z_seq = _f32(z_seq)
    T, N = z_seq.shape[0] - 1, z_seq.shape[1]
    act = np.ascontiguousarray(actions, dtype=np.int32).reshape(T, N)
    ln = None if lengths is None else np.ascontiguousarray(lengths, dtype=np.int32).reshape(N)
    M = 3 * K * Z
    out = {"nll": np.zeros(N), "W_lstm": np.zeros((Z + A + H, 4 * H)), "b_lstm": np.zeros(4 * H),
           "W_mdn": np.zeros((H, M)), "b_mdn": np.zeros(M)}
    w = _Weights(weights)
    cs = _cfg(cfg, nthreads)
    rc = lib.orc_mdn_nll_grad(C.byref(cs), C.byref(w.s), N, T, _ptr(z_seq), _ptr(act), _ptr(ln),
                              _ptr(out["nll"]), _ptr(out["W_lstm"]), _ptr(out["b_lstm"]),
                              _ptr(out["W_mdn"]), _ptr(out["b_mdn"]))
    if rc != 0:
        raise ValueError(f"orc_mdn_nll_grad failed ({rc})")
    return out


def mdn_nll(cfg: dict, weights: dict, z_seq, actions, lengths=None, want_seq: bool = False,
            nthreads: int = 1) -> dict:
    """Teacher-forced per-sequence mixture NLL in nats (a9)."""
    lib = _load()
    Z, H, K = int(cfg["z_dim"]), int(cfg["h_dim"]), int(cfg["k_mix"])
    z_seq = _f32(z_seq)
    T = z_seq.shape[0] - 1
    N = z_seq.shape[1]
    act = np.ascontiguousarray(actions, dtype=np.int32).reshape(T, N)
    ln = None if lengths is None else np.ascontiguousarray(lengths, dtype=np.int32).reshape(N)
    out = {"nll": np.zeros(N, np.float64)}
    if want_seq:
        out.update(h_seq=np.zeros((T, N, H), np.float32), c_seq=np.zeros((T, N, H), np.float32),
                   mdn_seq=np.zeros((T, N, 3 * K * Z), np.float32))
    w = _Weights(weights)
    cs = _cfg(cfg, nthreads)
    rc = lib.orc_mdn_nll(C.byref(cs), C.byref(w.s), N, T, _ptr(z_seq), _ptr(act), _ptr(ln),
                         _ptr(out["nll"]), _ptr(out.get("h_seq")), _ptr(out.get("c_seq")),
                         _ptr(out.get("mdn_seq")))
    if rc != 0:
        raise ValueError(f"orc_mdn_nll failed ({rc})")
    return out
