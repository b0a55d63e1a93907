"""The bench's host-side arithmetic on CPU: the algorithmic FLOP counts its roofline
divides by, the lookup of committed DRAM traffic by kernel source hash, and the count of
(episode, step) pairs a done-terminating rollout executes."""
import hashlib
import json
import os

import numpy as np
import pytest

import bench
import synth

# Per (episode, step) FLOPs of the three contractions (controller [Z+H]x[Z+H, A], gates
# [Z+H]x[Z+H, 4H], heads [H]x[H, 3KZ] plus reward and done), from the workload table's
# dimensions: 2 (Z+H) A + 2 (Z+H) 4H + 2 H (3KZ + 2).
EXPECTED_MFLOP = {"tiny_fp32": 0.873472, "small_bf16": 0.910336, "mid_bf16": 4.22912, "large_bf16": 16.912384}


@pytest.mark.parametrize("name", sorted(EXPECTED_MFLOP))
def test_flops_per_env_step(name):
    cfg = synth.model_config(name)
    assert bench.flops_per_env_step(cfg) == pytest.approx(EXPECTED_MFLOP[name] * 1e6, rel=1e-12)


def test_kernel_flops_add_up_to_the_step():
    cfg = synth.model_config("large_bf16")
    B = 65536
    parts = sum(bench.kernel_flops(c, cfg, B, 64, 1) for c in ("tc_ctrl", "tc_gates", "tc_heads"))
    assert parts == pytest.approx(bench.flops_per_env_step(cfg) * B, rel=1e-12)
    # the gate GEMM of one step at B = 65536: 65536 x 1152 x 4096 multiply-adds
    assert bench.kernel_flops("tc_gates", cfg, B, 64, 1) == 2 * 65536 * 1152 * 4096


def test_nll_flops_have_no_controller():
    cfg = synth.model_config("nll")
    Z, H, K = cfg["z_dim"], cfg["h_dim"], cfg["k_mix"]
    assert bench.nll_flops_per_step(cfg) == 2 * ((Z + H) * 4 * H + H * (3 * K * Z + 2))
    assert bench.kernel_flops("fused", dict(cfg, teacher=True), 10, 3, 1) == bench.nll_flops_per_step(cfg) * 30


def test_traffic_is_read_only_for_the_captured_source(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2205_01435_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "k.cu").write_text("__global__ void k() {}\n")
    sha = hashlib.sha256((csrc / "k.cu").read_bytes()).hexdigest()[:16]
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(
        {"k/w": {"source_sha": sha, "dram_bytes_per_launch": 1234}}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.kernel_source_sha("k.cu") == sha
    assert bench.ncu_traffic("k/w", sha) == 1234
    assert bench.ncu_traffic("k/other", sha) is None
    # the source changed since the capture: no traffic figure
    (csrc / "k.cu").write_text("__global__ void k() { }\n")
    assert bench.ncu_traffic("k/w", bench.kernel_source_sha("k.cu")) is None
    os.remove(tmp_path / "profiles" / "traffic.json")
    assert bench.ncu_traffic("k/w", sha) is None


def test_committed_traffic_entries_are_well_formed():
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as f:
        d = json.load(f)
    for key, e in d.items():
        assert "/" in key
        assert len(e["source_sha"]) == 16
        # read and write are averages over the captured launches, each truncated to bytes
        assert abs(e["dram_bytes_per_launch"] - e["dram_read_bytes"] - e["dram_write_bytes"]) <= 2
        assert "--clock-control none" in e["command"]


def test_counted_steps_stop_after_done():
    done = np.array([[0, 1, 0], [1, 0, 0], [0, 1, 0], [0, 0, 0]], dtype=np.uint8)  # [T=4, B=3]
    # episode 0 ends at t=1 (live at 0, 1), episode 1 at t=0 (live at 0), episode 2 never
    assert bench.counted_steps({"done_terminates": 1}, done) == 2 + 1 + 4
    assert bench.counted_steps({"noop_terminates": 1}, done) == 7
    assert bench.counted_steps({}, done) == 12


def test_oracle_sample_is_bounded():
    for name in ("tiny_fp32", "large_bf16"):
        w = synth.WORKLOADS[name]
        assert 8 <= bench.oracle_episodes(name, 1.0) <= w["B"]
        assert bench.oracle_episodes(name, 1e30) == w["B"]
