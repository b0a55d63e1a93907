"""Thin Python binding of the C ABI in include/wm.h (ctypes, argument marshalling only).

Every step of the dream path runs in the CUDA kernels of ``libwm.so``; this
module only turns torch tensors into pointers and the call's stream.  There is
no CPU fallback: if ``libwm.so`` is missing, importing the binding fails.

Names mirror the C entry points: ``wm_create``, ``wm_rollout``, ``wm_mdn_nll``,
``wm_sync``, ``wm_destroy``, ``wm_last_error``, ``wm_last_path``, ``wm_last_launches``,
``wm_set_timing``, ``wm_kernel_time``, ``wm_set_controllers``, ``wm_returns``.  The
``WorldModel`` class wraps them for convenience.
"""
from __future__ import annotations

import ctypes as C
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libwm.so")

WM_OK, WM_ERR_INVALID_ARG, WM_ERR_CUDA, WM_ERR_UNSUPPORTED, WM_ERR_TIMEOUT, WM_ERR_OOM = range(6)
WM_FP32, WM_BF16 = 0, 1
PATHS = {"auto": 0, "stepwise": 1, "fused": 2, "tensor": 3}
PATH_NAMES = {v: k for k, v in PATHS.items()}
KERNEL_CLASSES = ("step_gemm", "step_cell", "step_sample", "fused", "tc_ctrl", "tc_gates",
                  "tc_heads", "aux", "bw", "bw_gemm", "fused_small")  # WM_KERNEL_* in order


class WMError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"wm status {status}: {msg}")
        self.status = status


class wm_config(C.Structure):
    _fields_ = [("z_dim", C.c_int), ("a_dim", C.c_int), ("h_dim", C.c_int), ("k_mix", C.c_int),
                ("precision", C.c_int), ("mdn_tau", C.c_float), ("sigma_sqrt_tau", C.c_int),
                ("ctrl_sample", C.c_int), ("ctrl_tau", C.c_float), ("done_terminates", C.c_int),
                ("noop_terminates", C.c_int), ("seed", C.c_ulonglong), ("path", C.c_int),
                ("fused_cluster", C.c_int), ("reward_mode", C.c_int), ("reward_alpha", C.c_float),
                ("reward_beta", C.c_float), ("invalid_reward", C.c_float), ("value_head", C.c_int),
                ("n_xfers", C.c_int)]


class wm_weights(C.Structure):
    _fields_ = [("W_lstm", C.c_void_p), ("b_lstm", C.c_void_p), ("W_mdn", C.c_void_p),
                ("b_mdn", C.c_void_p), ("w_rew", C.c_void_p), ("b_rew", C.c_float),
                ("w_done", C.c_void_p), ("b_done", C.c_float), ("W_ctrl", C.c_void_p),
                ("b_ctrl", C.c_void_p), ("w_rt", C.c_void_p), ("b_rt", C.c_float),
                ("w_mem", C.c_void_p), ("b_mem", C.c_float), ("w_val", C.c_void_p),
                ("b_val", C.c_float)]


class wm_rollout_io(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "z0", "h0", "c0", "done0", "mask", "z_out", "actions", "rewards", "done", "h_final",
        "c_final", "h_seq", "c_seq", "mdn_seq", "comp_seq", "rt0", "mem0", "rt_seq", "mem_seq",
        "logp_seq", "value_seq", "loc_mask", "loc_actions")]


class wm_grads(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("W_lstm", "b_lstm", "W_mdn", "b_mdn")]


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"{_LIB_PATH} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'` (no CPU fallback)")
    lib = C.CDLL(_LIB_PATH)
    P = C.c_void_p
    lib.wm_create.argtypes = [C.POINTER(wm_config), C.POINTER(wm_weights), C.POINTER(P)]
    lib.wm_create.restype = C.c_int
    lib.wm_rollout.argtypes = [P, C.c_int, C.c_int, C.c_ulonglong, C.c_uint,
                               C.POINTER(wm_rollout_io), P]
    lib.wm_rollout.restype = C.c_int
    lib.wm_rollout_noalloc.argtypes = [P, C.c_int, C.c_int, C.c_ulonglong, C.c_uint,
                                       C.POINTER(wm_rollout_io), P]
    lib.wm_rollout_noalloc.restype = C.c_int
    lib.wm_set_controllers.argtypes = [P, C.c_int, C.c_int, P, P]
    lib.wm_set_controllers.restype = C.c_int
    lib.wm_returns.argtypes = [P, C.c_int, C.c_int, C.c_ulonglong, C.c_float, C.c_int, P, P, P, P, P, P]
    lib.wm_returns.restype = C.c_int
    lib.wm_mdn_nll_backward.argtypes = [P, C.c_int, C.c_int, P, P, P, P, C.POINTER(wm_grads), P]
    lib.wm_mdn_nll_backward.restype = C.c_int
    lib.wm_mdn_nll.argtypes = [P, C.c_int, C.c_int] + [P] * 7 + [P]
    lib.wm_mdn_nll.restype = C.c_int
    lib.wm_inject_wait_timeout.argtypes = [P, C.c_uint]
    lib.wm_inject_wait_timeout.restype = C.c_int
    lib.wm_sync.argtypes = [P]
    lib.wm_sync.restype = C.c_int
    lib.wm_last_error.argtypes = [P]
    lib.wm_last_error.restype = C.c_char_p
    lib.wm_last_path.argtypes = [P]
    lib.wm_last_path.restype = C.c_int
    lib.wm_last_launches.argtypes = [P]
    lib.wm_last_launches.restype = C.c_int
    lib.wm_set_timing.argtypes = [P, C.c_int]
    lib.wm_set_timing.restype = C.c_int
    lib.wm_kernel_time.argtypes = [P, C.c_int, C.POINTER(C.c_double), C.POINTER(C.c_longlong)]
    lib.wm_kernel_time.restype = C.c_int
    lib.wm_destroy.argtypes = [P]
    lib.wm_destroy.restype = None
    return lib


_lib = _load()


def lib_path() -> str:
    return _LIB_PATH


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        if not t.is_contiguous():
            raise ValueError("tensors passed to the engine must be contiguous")
        return C.c_void_p(t.data_ptr())
    return C.c_void_p(int(t))


def _check(h, st: int, what: str):
    if st != WM_OK:
        msg = _lib.wm_last_error(h).decode() if h else ""
        raise WMError(st, f"{what}: {msg}")


# ------------------------------------------------------------------ the C names
def wm_create(cfg: dict, weights: dict):
    """wm_create: copies + packs the fp32 host weights onto the current CUDA device."""
    c = wm_config(int(cfg["z_dim"]), int(cfg["a_dim"]), int(cfg["h_dim"]), int(cfg["k_mix"]),
                  WM_BF16 if cfg.get("precision", "fp32") == "bf16" else WM_FP32,
                  float(cfg.get("mdn_tau", 1.0)), int(cfg.get("sigma_sqrt_tau", 0)),
                  int(cfg.get("ctrl_sample", 0)), float(cfg.get("ctrl_tau", 1.0)),
                  int(cfg.get("done_terminates", 0)), int(cfg.get("noop_terminates", 0)),
                  int(cfg.get("seed", 0)) & 0xFFFFFFFFFFFFFFFF,
                  PATHS[cfg.get("path", "auto")] if isinstance(cfg.get("path", "auto"), str)
                  else int(cfg["path"]), int(cfg.get("fused_cluster", 0)),
                  int(cfg.get("reward_mode", 0)), float(cfg.get("reward_alpha", 0.8)),
                  float(cfg.get("reward_beta", 0.2)), float(cfg.get("invalid_reward", -100.0)),
                  int(cfg.get("value_head", 0)), int(cfg.get("n_xfers", 0)))
    keep = {k: torch.as_tensor(weights[k], dtype=torch.float32).contiguous().cpu()
            for k in ("W_lstm", "b_lstm", "W_mdn", "b_mdn", "w_rew", "w_done", "W_ctrl", "b_ctrl",
                      "w_rt", "w_mem", "w_val") if weights.get(k) is not None}
    w = wm_weights(_ptr(keep["W_lstm"]), _ptr(keep["b_lstm"]), _ptr(keep["W_mdn"]),
                   _ptr(keep["b_mdn"]), _ptr(keep["w_rew"]), float(weights["b_rew"]),
                   _ptr(keep["w_done"]), float(weights["b_done"]), _ptr(keep["W_ctrl"]),
                   _ptr(keep["b_ctrl"]), _ptr(keep.get("w_rt")), float(weights.get("b_rt", 0.0)),
                   _ptr(keep.get("w_mem")), float(weights.get("b_mem", 0.0)), _ptr(keep.get("w_val")),
                   float(weights.get("b_val", 0.0)))
    h = C.c_void_p()
    st = _lib.wm_create(C.byref(c), C.byref(w), C.byref(h))
    if st != WM_OK:
        raise WMError(st, "wm_create failed (invalid sizes or CUDA error)")
    return h


def wm_rollout(h, B: int, T: int, episode_offset: int, t0: int, io: dict, stream: int = 0):
    s = wm_rollout_io(*[_ptr(io.get(n)) for n, _ in wm_rollout_io._fields_])
    _check(h, _lib.wm_rollout(h, B, T, episode_offset, t0, C.byref(s), C.c_void_p(stream)),
           "wm_rollout")


def wm_rollout_noalloc(h, B: int, T: int, episode_offset: int, t0: int, io: dict,
                       stream: int = 0):
    """wm_rollout_noalloc: device arrays only; scratch from the library's fixed array."""
    s = wm_rollout_io(*[_ptr(io.get(n)) for n, _ in wm_rollout_io._fields_])
    _check(h, _lib.wm_rollout_noalloc(h, B, T, episode_offset, t0, C.byref(s),
                                      C.c_void_p(stream)), "wm_rollout_noalloc")


def wm_mdn_nll(h, N: int, T: int, z_seq, actions, lengths, nll, h_seq=None, c_seq=None,
               mdn_seq=None, stream: int = 0):
    _check(h, _lib.wm_mdn_nll(h, N, T, _ptr(z_seq), _ptr(actions), _ptr(lengths), _ptr(nll),
                              _ptr(h_seq), _ptr(c_seq), _ptr(mdn_seq), C.c_void_p(stream)),
           "wm_mdn_nll")


def wm_set_controllers(h, W_ctrl, b_ctrl, pop_group: int):
    """wm_set_controllers: P = W_ctrl.shape[0] candidates (host fp32 [P, Z+H, A], [P, A])."""
    W = torch.as_tensor(W_ctrl, dtype=torch.float32).contiguous().cpu()
    b = torch.as_tensor(b_ctrl, dtype=torch.float32).contiguous().cpu()
    _check(h, _lib.wm_set_controllers(h, int(W.shape[0]), int(pop_group), _ptr(W), _ptr(b)),
           "wm_set_controllers")


def wm_returns(h, B: int, T: int, episode_offset: int, gamma: float, stop_at_done: bool, rewards,
               done, bootstrap, returns, fitness=None, stream: int = 0):
    _check(h, _lib.wm_returns(h, B, T, episode_offset, float(gamma), int(bool(stop_at_done)),
                              _ptr(rewards), _ptr(done), _ptr(bootstrap), _ptr(returns),
                              _ptr(fitness), C.c_void_p(stream)), "wm_returns")


def wm_mdn_nll_backward(h, N: int, T: int, z_seq, actions, lengths, nll, grads: dict, stream: int = 0):
    g = wm_grads(*[_ptr(grads.get(n)) for n, _ in wm_grads._fields_])
    _check(h, _lib.wm_mdn_nll_backward(h, N, T, _ptr(z_seq), _ptr(actions), _ptr(lengths), _ptr(nll),
                                       C.byref(g), C.c_void_p(stream)), "wm_mdn_nll_backward")


def wm_inject_wait_timeout(h, polls: int):
    _check(h, _lib.wm_inject_wait_timeout(h, int(polls)), "wm_inject_wait_timeout")


def wm_sync(h):
    _check(h, _lib.wm_sync(h), "wm_sync")


def wm_last_path(h) -> str:
    return PATH_NAMES.get(_lib.wm_last_path(h), "?")


def wm_last_launches(h) -> int:
    return int(_lib.wm_last_launches(h))


def wm_set_timing(h, enable: bool):
    _check(h, _lib.wm_set_timing(h, int(bool(enable))), "wm_set_timing")


def wm_kernel_time(h, kernel_class: int) -> tuple[float, int]:
    """(total milliseconds, launches) of one WM_KERNEL_* class since timing was enabled."""
    ms, n = C.c_double(0.0), C.c_longlong(0)
    _check(h, _lib.wm_kernel_time(h, int(kernel_class), C.byref(ms), C.byref(n)), "wm_kernel_time")
    return float(ms.value), int(n.value)


def wm_destroy(h):
    _lib.wm_destroy(h)


# ------------------------------------------------------------------ convenience wrapper
class WorldModel:
    """Owns one wm_handle on one CUDA device."""

    def __init__(self, cfg: dict, weights: dict, device: int | torch.device | None = None):
        self.cfg = dict(cfg)
        self.Z, self.A, self.H, self.K = (int(cfg[k]) for k in ("z_dim", "a_dim", "h_dim", "k_mix"))
        self.M = 3 * self.K * self.Z
        self.device = torch.device("cuda", torch.cuda.current_device() if device is None
                                   else torch.device("cuda", device).index if isinstance(device, int)
                                   else torch.device(device).index)
        with torch.cuda.device(self.device):
            self.h = wm_create(cfg, weights)

    def close(self):
        if getattr(self, "h", None):
            wm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _stream(self, stream):
        if stream is not None:
            return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
        return torch.cuda.current_stream(self.device).cuda_stream

    def _alloc(self, like: torch.Tensor, shape, dtype):
        if like.is_cuda:
            return torch.empty(shape, dtype=dtype, device=like.device)
        return torch.empty(shape, dtype=dtype, pin_memory=like.is_pinned())

    def rollout(self, z0: torch.Tensor, T: int, mask: torch.Tensor | None = None,
                episode_offset: int = 0, t0: int = 0, h0=None, c0=None, done0=None,
                want_final: bool = True, want_seq: bool = False, out: dict | None = None,
                stream=None, rt0=None, mem0=None, want_logp: bool = False, loc_mask=None) -> dict:
        """wm_rollout on B = z0.shape[0] episodes; returns the output tensors (device of z0).
        With the shaped reward, rt0 / mem0 are required and rt_seq / mem_seq are returned;
        want_logp adds logp_seq, and a value head adds value_seq."""
        B = int(z0.shape[0])
        o = dict(out or {})
        for name, shape, dt in (("z", (T + 1, B, self.Z), torch.float32),
                                ("actions", (T, B), torch.int32),
                                ("rewards", (T, B), torch.float32),
                                ("done", (T, B), torch.uint8)):
            if name not in o:
                o[name] = self._alloc(z0, shape, dt)
        if want_final:
            for name in ("h_final", "c_final"):
                if name not in o:
                    o[name] = self._alloc(z0, (B, self.H), torch.float32)
        if want_seq:
            o.setdefault("h_seq", self._alloc(z0, (T, B, self.H), torch.float32))
            o.setdefault("c_seq", self._alloc(z0, (T, B, self.H), torch.float32))
            o.setdefault("mdn_seq", self._alloc(z0, (T, B, self.M), torch.float32))
            o.setdefault("comp_seq", self._alloc(z0, (T, B, self.Z), torch.uint8))
        if int(self.cfg.get("reward_mode", 0)) == 1:
            o.setdefault("rt_seq", self._alloc(z0, (T, B), torch.float32))
            o.setdefault("mem_seq", self._alloc(z0, (T, B), torch.float32))
        if want_logp:
            o.setdefault("logp_seq", self._alloc(z0, (T, B), torch.float32))
        if int(self.cfg.get("value_head", 0)):
            o.setdefault("value_seq", self._alloc(z0, (T, B), torch.float32))
        if int(self.cfg.get("n_xfers", 0)) > 0:
            o.setdefault("loc_actions", self._alloc(z0, (T, B), torch.int32))
        io = {"z0": z0, "h0": h0, "c0": c0, "done0": done0, "mask": mask, "z_out": o["z"],
              "actions": o["actions"], "rewards": o["rewards"], "done": o["done"],
              "h_final": o.get("h_final"), "c_final": o.get("c_final"), "h_seq": o.get("h_seq"),
              "c_seq": o.get("c_seq"), "mdn_seq": o.get("mdn_seq"), "comp_seq": o.get("comp_seq"),
              "rt0": rt0, "mem0": mem0, "rt_seq": o.get("rt_seq"), "mem_seq": o.get("mem_seq"),
              "logp_seq": o.get("logp_seq"), "value_seq": o.get("value_seq"), "loc_mask": loc_mask,
              "loc_actions": o.get("loc_actions")}
        with torch.cuda.device(self.device):
            wm_rollout(self.h, B, T, episode_offset, t0, io, self._stream(stream))
        return o

    def mdn_nll(self, z_seq: torch.Tensor, actions: torch.Tensor, lengths=None,
                want_seq: bool = False, stream=None) -> dict:
        T = int(z_seq.shape[0]) - 1
        N = int(z_seq.shape[1])
        o = {"nll": self._alloc(z_seq, (N,), torch.float32)}
        if want_seq:
            o["h_seq"] = self._alloc(z_seq, (T, N, self.H), torch.float32)
            o["c_seq"] = self._alloc(z_seq, (T, N, self.H), torch.float32)
            o["mdn_seq"] = self._alloc(z_seq, (T, N, self.M), torch.float32)
        with torch.cuda.device(self.device):
            wm_mdn_nll(self.h, N, T, z_seq, actions, lengths, o["nll"], o.get("h_seq"),
                       o.get("c_seq"), o.get("mdn_seq"), self._stream(stream))
        return o

    def set_controllers(self, W_ctrl, b_ctrl, pop_group: int = 1):
        """A population of W_ctrl.shape[0] controllers; episode e acts with candidate
        (e / pop_group) mod P."""
        with torch.cuda.device(self.device):
            wm_set_controllers(self.h, W_ctrl, b_ctrl, pop_group)
        self.P = int(torch.as_tensor(W_ctrl).shape[0])

    def returns(self, rewards: torch.Tensor, done: torch.Tensor, gamma: float,
                stop_at_done: bool = True, bootstrap=None, episode_offset: int = 0,
                want_fitness: bool = False, stream=None) -> dict:
        """wm_returns: discounted returns [T, B] (and each candidate's mean G_0)."""
        T, B = int(rewards.shape[0]), int(rewards.shape[1])
        o = {"returns": self._alloc(rewards, (T, B), torch.float32)}
        if want_fitness:
            o["fitness"] = self._alloc(rewards, (getattr(self, "P", 1),), torch.float32)
        with torch.cuda.device(self.device):
            wm_returns(self.h, B, T, episode_offset, gamma, stop_at_done, rewards, done, bootstrap,
                       o["returns"], o.get("fitness"), self._stream(stream))
        return o

    def mdn_nll_backward(self, z_seq: torch.Tensor, actions: torch.Tensor, lengths=None,
                         stream=None) -> dict:
        """wm_mdn_nll_backward: the per-sequence NLL and the gradient of their sum with respect
        to W_lstm, b_lstm, W_mdn, b_mdn (arrays on z_seq's device)."""
        T = int(z_seq.shape[0]) - 1
        N = int(z_seq.shape[1])
        Z, A, H, M = self.Z, self.A, self.H, self.M
        o = {"nll": self._alloc(z_seq, (N,), torch.float32),
             "W_lstm": self._alloc(z_seq, (Z + A + H, 4 * H), torch.float32),
             "b_lstm": self._alloc(z_seq, (4 * H,), torch.float32),
             "W_mdn": self._alloc(z_seq, (H, M), torch.float32),
             "b_mdn": self._alloc(z_seq, (M,), torch.float32)}
        with torch.cuda.device(self.device):
            wm_mdn_nll_backward(self.h, N, T, z_seq, actions, lengths, o["nll"], o, self._stream(stream))
        return o

    def sync(self):
        wm_sync(self.h)

    def inject_wait_timeout(self, polls: int):
        """Make the next fused / tensor-core call's first kernel give up on a wait that
        nothing completes, after at most `polls` polls (tests of the timeout path)."""
        wm_inject_wait_timeout(self.h, polls)

    @property
    def last_path(self) -> str:
        return wm_last_path(self.h)

    @property
    def last_launches(self) -> int:
        return wm_last_launches(self.h)

    def set_timing(self, enable: bool = True):
        """Bracket every kernel of later calls with CUDA events (clears the totals)."""
        wm_set_timing(self.h, enable)

    def kernel_times(self) -> dict:
        """{class name: (total ms, launches)} for the classes that launched since set_timing."""
        out = {}
        for i, name in enumerate(KERNEL_CLASSES):
            ms, n = wm_kernel_time(self.h, i)
            if n:
                out[name] = (ms, n)
        return out
