"""Host-side logic of bench.py that runs without a GPU: the max-over-ranks
timing of a multi-process run (two gloo ranks on the CPU), the reference arm
under torchrun (rank 0 alone prints), and the unit counts the metrics use."""
from __future__ import annotations

import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workload as wk  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, values, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out[rank] = bench.max_over_ranks(values[rank], world, "cpu")
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_two_gloo_ranks():
    import torch.multiprocessing as mp
    port = _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        procs = [ctx.Process(target=_rank_main, args=(r, 2, port, [1.5, 4.25], out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        assert dict(out) == {0: 4.25, 1: 4.25}


def test_max_over_ranks_single_rank_is_identity():
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5


def test_reference_arm_under_torchrun_prints_once():
    """Two ranks: rank 0 times the oracle and prints one JSON line, rank 1
    exits 0 without output."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={port}", os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3", "--config", "4"]
    res = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0


def test_search_children_counts_roots_then_frontiers():
    torch = pytest.importorskip("torch")
    trace_n = torch.tensor([[3, 7, 0], [1, 0, 0]], dtype=torch.int32)
    # iteration 0 expands each root; iteration i > 0 the frontier left by i - 1
    assert bench.search_children(trace_n) == 5 * (2 + 3 + 7 + 1 + 0)


def test_valid_anchor_rules_by_hand():
    wl = wk.Workload(0, "t", 1, 4, 6, 2, 2, ((1, 1),), 0.1, 0.1, 0.1, 0.1, 0, 0)
    rules = wk.empty_rules(1, 2)
    rules["h"], rules["w"] = [[1, 2]], [[1, 3]]
    # 1x1: 4 rotations x 24 anchors; 2x3 on a 4x6 board: rotations 0, 2 have
    # (4-2+1) x (6-3+1) anchors, rotations 1, 3 (3x2) have (4-3+1) x (6-2+1)
    assert bench.valid_anchor_rules(wl, rules) == 4 * 24 + 2 * 12 + 2 * 10


def test_profile_traffic_follows_the_kernel_source(tmp_path, monkeypatch):
    """The bench line reports a profile's DRAM traffic only while the kernel
    source hashes to the value recorded with the capture."""
    import hashlib
    from types import SimpleNamespace

    src = tmp_path / "kernel.cu"
    src.write_text("__global__ void k() {}\n")
    digest = hashlib.sha256(src.read_bytes()).hexdigest()
    monkeypatch.setattr(bench, "PROFILE_DIR", str(tmp_path))
    wl = SimpleNamespace(name="toy")
    prof = tmp_path / "k_toy.md"
    prof.write_text(f"kernel_source_sha256: {digest[:16]}\ndram_bytes_per_launch: 12345\n")
    assert bench.profile_traffic("k", wl, str(src)) == 12345.0
    src.write_text("__global__ void k() { /* changed */ }\n")
    assert bench.profile_traffic("k", wl, str(src)) is None
    assert bench.profile_traffic("missing", wl, str(src)) is None


def test_committed_profiles_name_their_kernel_sources():
    """Every committed profile with a traffic figure records a source hash."""
    import glob
    import re
    for path in glob.glob(os.path.join(bench.PROFILE_DIR, "*.md")):
        text = open(path).read()
        if "dram_bytes_per_launch:" in text:
            assert re.search(r"kernel_source_sha256:\s*[0-9a-f]{16}", text), path


def test_row_basis_ops_by_hand():
    """One op per (rule rotation, input or output entry, valid anchor row)."""
    wl = wk.Workload(0, "t", 1, 4, 6, 2, 2, ((1, 1),), 0.1, 0.1, 0.1, 0.1, 0, 0)
    rules = wk.empty_rules(1, 2)
    rules["h"], rules["w"] = [[1, 2]], [[1, 3]]
    rules["present"][0, 0, 0] = 0b11      # 2 input entries
    rules["set"][0, 0, 0] = 0b01          # 1 output entry
    rules["absent"][0, 1, 5] = 0b10       # 1 input entry
    rules["clear"][0, 1, 0] = 0b11        # 2 output entries
    # rule 0, 1x1: 4 rotations x 4 rows x 3 entries; rule 1, 2x3: rotations 0, 2
    # have 4 - 2 + 1 = 3 rows, rotations 1, 3 (3x2) have 4 - 3 + 1 = 2 rows, x 3 entries
    assert bench.row_basis_ops(wl, rules) == 4 * 4 * 3 + (2 * 3 + 2 * 2) * 3


def test_trajectory_bytes_and_default_workload():
    wl3 = wk.WORKLOADS[3]
    assert bench.traj_bytes_per_env_step(wl3) == 16 * 16 * 2 + 4 + 1
    import argparse  # noqa: F401
    # the default benchmark line is the largest single-GPU workload (config 3)
    src = open(os.path.join(ROOT, "bench.py")).read()
    assert '"--config", type=int, default=3' in src


def test_search_workload_names_its_base_game_rules():
    d = bench.config_dict(wk.WORKLOADS[4])
    assert "move and eat rules" in d["workload"]
    assert "far exceed L2" in bench.config_dict(wk.WORKLOADS[3])["l2"]


def test_single_step_actions_match_the_rollout_draw():
    """The single-step benchmark's actions are the fused rollout's on-device
    draws (SplitMix64 counter, stream 4), recomputed independently here."""
    a = wk.actions(7, 3, 4)
    M = (1 << 64) - 1

    def mix(z):
        z = ((z ^ (z >> 30)) * 0xbf58476d1ce4e5b9) & M
        z = ((z ^ (z >> 27)) * 0x94d049bb133111eb) & M
        return z ^ (z >> 31)
    for s in range(4):
        for e in range(3):
            z = mix((7 + 0x9E3779B97F4A7C15 * 5) & M)
            z = mix(z ^ e)
            d = mix(z ^ s)
            assert a[s, e] == ((d >> 32) * 5) >> 32
