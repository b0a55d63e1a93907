"""The multi-GPU path's host logic on CPU: two `gloo` ranks (world_size 2).

Each rank runs shard r of the global batch (its own inputs, Philox episodes r*B + b) with
no data-path collective; the shards' results must be bit-identical to one unsharded run
over the concatenated inputs, and the timing reduction must give every rank the slowest
rank's time.  The oracle stands in for the GPU kernels here (it computes the same steps)."""
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
B, T = 6, 5


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, out_dir: str) -> None:
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    import oracle
    import synth

    dist.init_process_group("gloo", rank=rank, world_size=world)
    cfg, w, z0, mask, b, t = synth.rollout_inputs("tiny_fp32", B=B, T=T, shard=rank)
    out = oracle.rollout(cfg, w, z0, mask, t, episode_offset=rank * b, nthreads=1)
    slowest = bench.max_over_ranks(1.5 + rank, world)
    gathered = [None] * world
    dist.all_gather_object(gathered, out)
    if rank == 0:
        np.savez(os.path.join(out_dir, "shards.npz"), slowest=slowest,
                 **{f"{k}_{r}": v for r, o in enumerate(gathered) for k, v in o.items()})
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_bit_exactly(tmp_path, orc):
    import multiprocessing as mp

    ctx = mp.get_context("spawn")
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0, p.exitcode
    got = np.load(tmp_path / "shards.npz")
    assert float(got["slowest"]) == 2.5  # rank 1's 2.5 s, on rank 0

    import synth
    parts = [synth.rollout_inputs("tiny_fp32", B=B, T=T, shard=r) for r in range(2)]
    cfg, w = parts[0][0], parts[0][1]
    z0 = np.concatenate([p[2] for p in parts], axis=0)
    mask = np.concatenate([p[3] for p in parts], axis=1)
    whole = orc.rollout(cfg, w, z0, mask, T, episode_offset=0, nthreads=1)
    for k, v in whole.items():
        ax = 0 if k in ("h_final", "c_final") else 1
        cat = np.concatenate([got[f"{k}_0"], got[f"{k}_1"]], axis=ax)
        assert np.array_equal(cat, v), k


def test_shard_zero_is_the_unsharded_workload_and_shards_differ():
    import synth
    a = synth.rollout_inputs("tiny_fp32")
    b = synth.rollout_inputs("tiny_fp32", shard=0)
    c = synth.rollout_inputs("tiny_fp32", shard=1)
    assert np.array_equal(a[2], b[2]) and np.array_equal(a[3], b[3])
    assert not np.array_equal(a[2], c[2]) and not np.array_equal(a[3], c[3])
    for k in a[1]:
        assert np.array_equal(np.asarray(a[1][k]), np.asarray(c[1][k]))  # one model


def test_reference_arm_runs_on_rank_zero_only():
    env = dict(os.environ, WORLD_SIZE="2", RANK="1", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--gpus", "2", "--steps", "1", "--warmup", "3"],
                       capture_output=True, text=True, env=env, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""
