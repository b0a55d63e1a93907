"""Seeded synthetic inputs for the world-model dream path.

This module is shared by the oracle tests, the GPU parity tests, ``bench.py``
and ``__graft_entry__.smoke()``.  It holds none of the method's arithmetic:
it only draws the inputs (weights, initial latents, action masks, teacher
sequences) from numpy's PCG64 generator, one independent stream per tensor.

The paper's graphs, GNN latents, TASO environment and trained weights are not
available, so these stand in for them.  Recipe (per workload below):

* every weight and bias ~ N(0, 0.05^2) (fp32);
* z_0 ~ N(0, 1);
* action masks: each (step, episode, action) bit valid with probability
  ``mask_density``, independently; packed little-endian into uint32 words
  ([T, B, ceil(A/32)], bit j of word w = action 32*w + j);
* teacher-forced sequences: z ~ N(0, 1) for all T+1 frames, actions uniform
  on [0, A);
* shaped-reward state: the predicted runtime and memory accesses of each
  episode's current graph ~ N(0, 0.5^2).

Sharding: a run over S shards of B episodes (one shard per GPU) draws shard
r's z_0 and masks from streams of their own; shard 0's are exactly the
unsharded workload's.  The global batch is the concatenation of the shards,
global episode r*B + b being episode b of shard r (its Philox episode index).

The five workloads follow the world-model hyper-parameters the paper uses
(256 hidden units, a handful of Gaussians, Sec. 4.7) scaled to the regimes
that matter on one GPU.
"""
from __future__ import annotations

import numpy as np

WORKLOADS = {
    # tiny CPU-checkable rollout, fp32 path
    "tiny_fp32": dict(B=16, T=20, z_dim=32, a_dim=64, h_dim=256, k_mix=5, precision="fp32",
                      mask_density=0.5),
    # small-batch latency regime, bf16 operands / fp32 state
    "small_bf16": dict(B=1024, T=50, z_dim=32, a_dim=128, h_dim=256, k_mix=5, precision="bf16",
                       mask_density=0.3),
    # mid regime, done head ends episodes
    "mid_bf16": dict(B=8192, T=100, z_dim=64, a_dim=256, h_dim=512, k_mix=8, precision="bf16",
                     mask_density=0.2, done_terminates=1),
    # teacher-forced MDN NLL scoring (fp32 and bf16)
    "nll": dict(N=512, T=128, z_dim=64, a_dim=256, h_dim=512, k_mix=5, precision="fp32"),
    # large-batch tensor-core regime, sampled controller at temperature 1
    "large_bf16": dict(B=65536, T=64, z_dim=128, a_dim=512, h_dim=1024, k_mix=8,
                       precision="bf16", mask_density=0.1, ctrl_sample=1, ctrl_tau=1.0),
}

_STREAM = {"W_lstm": 1, "b_lstm": 2, "W_mdn": 3, "b_mdn": 4, "w_rew": 5, "b_rew": 6,
           "w_done": 7, "b_done": 8, "W_ctrl": 9, "b_ctrl": 10, "w_rt": 11, "b_rt": 12,
           "w_mem": 13, "b_mem": 14, "W_pop": 15, "b_pop": 16, "w_val": 17, "b_val": 18,
           "hier": 27,
           "z0": 20, "mask": 21, "zseq": 22, "actions": 23, "lengths": 24, "rt0": 25, "mem0": 26}


def _rng(seed: int, stream: int, sub: int = 0) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(seed), int(stream), int(sub)]))


def _shard_rng(seed: int, stream: int, sub: int, shard: int) -> np.random.Generator:
    """Shard 0 uses the unsharded streams; shard r > 0 a disjoint family of its own."""
    if shard == 0:
        return _rng(seed, stream, sub)
    return _rng(seed, 1000 + stream, int(shard) * 65536 + sub)


def model_config(name: str, **over) -> dict:
    """The wm_config-style dict of a workload (sizes, precision, flags)."""
    w = dict(WORKLOADS[name])
    w.update(over)
    cfg = dict(z_dim=w["z_dim"], a_dim=w["a_dim"], h_dim=w["h_dim"], k_mix=w["k_mix"],
               precision=w.get("precision", "fp32"), mdn_tau=w.get("mdn_tau", 1.0),
               sigma_sqrt_tau=w.get("sigma_sqrt_tau", 0), ctrl_sample=w.get("ctrl_sample", 0),
               ctrl_tau=w.get("ctrl_tau", 1.0), done_terminates=w.get("done_terminates", 0),
               noop_terminates=w.get("noop_terminates", 0), seed=w.get("seed", 0),
               reward_mode=w.get("reward_mode", 0), reward_alpha=w.get("reward_alpha", 0.8),
               reward_beta=w.get("reward_beta", 0.2), invalid_reward=w.get("invalid_reward", -100.0),
               pop_size=w.get("pop_size", 0), pop_group=w.get("pop_group", 1),
               value_head=w.get("value_head", 0), n_xfers=w.get("n_xfers", 0))
    return cfg


def weights(cfg: dict, seed: int = 0, std: float = 0.05) -> dict:
    """All world-model and controller parameters ~ N(0, std^2), canonical fp32 layout."""
    Z, A, H, K = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"], cfg["k_mix"]
    shapes = {"W_lstm": (Z + A + H, 4 * H), "b_lstm": (4 * H,), "W_mdn": (H, 3 * K * Z),
              "b_mdn": (3 * K * Z,), "w_rew": (H,), "b_rew": (), "w_done": (H,), "b_done": (),
              "W_ctrl": (Z + H, A), "b_ctrl": (A,), "w_rt": (H,), "b_rt": (), "w_mem": (H,),
              "b_mem": (), "w_val": (H,), "b_val": ()}
    out = {}
    for name, shp in shapes.items():
        v = _rng(seed, _STREAM[name]).standard_normal(shp, dtype=np.float32) * np.float32(std)
        out[name] = float(v) if shp == () else np.ascontiguousarray(v, dtype=np.float32)
    return out


def population(cfg: dict, P: int, seed: int = 0, std: float = 0.05):
    """(W_ctrl [P, Z+H, A], b_ctrl [P, A]): P controller candidates, each ~ N(0, std^2)
    from a stream of its own (one generation of a controller search)."""
    Z, A, H = cfg["z_dim"], cfg["a_dim"], cfg["h_dim"]
    W = np.stack([_rng(seed, _STREAM["W_pop"], g).standard_normal((Z + H, A), dtype=np.float32)
                  for g in range(P)]) * np.float32(std)
    b = np.stack([_rng(seed, _STREAM["b_pop"], g).standard_normal(A, dtype=np.float32)
                  for g in range(P)]) * np.float32(std)
    return np.ascontiguousarray(W, np.float32), np.ascontiguousarray(b, np.float32)


def shaping_state(B: int, seed: int = 0, shard: int = 0):
    """(rt0, mem0) [B]: the predicted runtime and memory accesses of each episode's
    current graph, for the shaped reward; ~ N(0, 0.5^2), the scale of the random-init
    heads' outputs."""
    rt = _shard_rng(seed, _STREAM["rt0"], 0, shard).standard_normal(B, dtype=np.float32) * np.float32(0.5)
    mem = _shard_rng(seed, _STREAM["mem0"], 0, shard).standard_normal(B, dtype=np.float32) * np.float32(0.5)
    return rt, mem


def z0(B: int, Z: int, seed: int = 0, shard: int = 0) -> np.ndarray:
    return _shard_rng(seed, _STREAM["z0"], 0, shard).standard_normal((B, Z), dtype=np.float32)


def pack_mask(valid: np.ndarray) -> np.ndarray:
    """bool [..., A] -> uint32 [..., ceil(A/32)], little-endian bit order."""
    A = valid.shape[-1]
    W = (A + 31) // 32
    pad = W * 32 - A
    v = valid
    if pad:
        v = np.concatenate([v, np.zeros(v.shape[:-1] + (pad,), dtype=bool)], axis=-1)
    by = np.packbits(v.astype(np.uint8), axis=-1, bitorder="little")
    return np.ascontiguousarray(by).view("<u4").astype(np.uint32, copy=False)


def mask(T: int, B: int, A: int, density: float, seed: int = 0, shard: int = 0) -> np.ndarray:
    """Bernoulli(density) valid-action bits, packed [T, B, ceil(A/32)] uint32."""
    W = (A + 31) // 32
    out = np.empty((T, B, W), dtype=np.uint32)
    thr = np.float32(density)
    for t in range(T):
        r = _shard_rng(seed, _STREAM["mask"], t, shard)
        out[t] = pack_mask(r.random((B, A), dtype=np.float32) < thr)
    return out


def hier_masks(T: int, B: int, NX: int, L: int, density: float, seed: int = 0, shard: int = 0):
    """Masks of the hierarchical action (Sec. 3.1.3): (xfer mask [T, B, ceil((NX+L)/32)],
    location masks [T, B, NX, ceil(L/32)]).  Each (step, episode, xfer) has a count of valid
    locations, a prefix of the L location slots (the environment lists a graph's locations
    first and marks the rest of the slots invalid): 0 with probability 1 - density, else
    uniform on [1, L].  An xfer is valid iff it has a location; the NO-OP (xfer NX - 1)
    is always valid and has none."""
    A = NX + L
    W, WL = (A + 31) // 32, (L + 31) // 32
    xm = np.empty((T, B, W), dtype=np.uint32)
    lm = np.empty((T, B, NX, WL), dtype=np.uint32)
    for t in range(T):
        r = _shard_rng(seed, _STREAM["hier"], t, shard)
        n = r.integers(1, L + 1, size=(B, NX), dtype=np.int32)
        n = np.where(r.random((B, NX), dtype=np.float32) < np.float32(density), n, 0)
        n[:, NX - 1] = 0
        valid_x = n > 0
        valid_x[:, NX - 1] = True
        xm[t] = pack_mask(np.concatenate([valid_x, np.zeros((B, L), bool)], axis=1))
        lm[t] = pack_mask(np.arange(L)[None, None, :] < n[:, :, None])
    return xm, lm


def teacher_inputs(N: int, T: int, Z: int, A: int, seed: int = 0, ragged: bool = False):
    """(z_seq [T+1,N,Z], actions [T,N], lengths [N] or None) for teacher-forced scoring."""
    zs = _rng(seed, _STREAM["zseq"]).standard_normal((T + 1, N, Z), dtype=np.float32)
    acts = _rng(seed, _STREAM["actions"]).integers(0, A, size=(T, N), dtype=np.int32)
    lens = None
    if ragged:
        lens = _rng(seed, _STREAM["lengths"]).integers(0, T + 1, size=N, dtype=np.int32)
    return zs, acts, lens


def rollout_inputs(name: str, seed: int = 0, B: int | None = None, T: int | None = None,
                   shard: int = 0):
    """(cfg, weights, z0, mask, B, T) for a rollout workload; `shard` picks the shard's
    episodes (the weights are the same for every shard)."""
    w = WORKLOADS[name]
    cfg = model_config(name)
    B = w["B"] if B is None else B
    T = w["T"] if T is None else T
    wts = weights(cfg, seed)
    z = z0(B, cfg["z_dim"], seed, shard)
    m = mask(T, B, cfg["a_dim"], w["mask_density"], seed, shard)
    return cfg, wts, z, m, B, T
