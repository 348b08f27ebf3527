"""Benchmark: batched Autoverse environment steps on one GB300 (per process).

Default workload (config 3, the RL training shape): 16,384 envs, 16x16 boards,
10 tile channels, 12 rules per env of 1x2 / 1x3 / 3x3 in 4 rotations each,
2000 fused steps per launch (av_rollout) writing the observation, reward and
done flag of every step (16.9 GB per launch), done at no goal tile or t = 200
with auto-reset.  One benchmark step = one launch = 16,384 x 2000 env-steps.
The line also carries an `extra` entry for the 64x64 workload (config 5).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--config 1|2|3|4|5|6] [--single-step] [--seed S]

Prints one JSON line.  Under torchrun (N > 1) every rank runs its own replica
of the workload (envs never interact: no data-path collective); the timing is
the max over ranks and `value` counts the env-steps of all ranks.

--single-step times av_step (one launch per step) on the workload's shape.
--impl reference times the CPU oracle (the slow, literal restatement of the
paper's rule semantics) on this machine's host cores, on a bounded sample of
the same workload; only rank 0 runs it.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workload as wk  # noqa: E402

PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
KERNEL_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "kernels.cuh")
PROFILE_DIR = os.path.join(ROOT, "profiles")
# rollout kernel launched for each av_rollout_path value
KERNEL_NAMES = {1: "rollout_kernel", 2: "rollout_fast_kernel", 3: "rollout_env_warp_kernel",
                4: "rollout_variant_kernel", 5: "rollout_band_kernel", 6: "rollout_memo_kernel",
                7: "step_warp_kernel"}
VARIANT_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "k_variant.cu")
MEMO_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "k_memo_impl.cuh")
BAND_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "k_band.cu")
STEP_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "k_step.cu")


def bench_variant(wl) -> dict:
    """Variant semantics of the --variant runs: every rule applied at most once
    per step, chosen by random index values; rule r inhibits rule r + 1."""
    R = wl.n_rules
    return dict(random_keys=1, key_seed=12345, limit=[1] * R,
                inhibit=[1 << ((r + 1) % R) for r in range(R)])
SM_COUNT_GB300 = 152
# 32-bit integer instructions issued per SM per clock: 4 schedulers x 32 lanes.
# The committed probe (--int-probe) reaches 113-114 of them for IADD3, SHF and
# IMAD chains and 76 for LOP3 on GB300.
INT_LANES_PER_SM = 128
PROBE_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "probe", "int_issue_probe.cu")


# ------------------------------------------------------------ workload
def workload_for(key: int) -> wk.Workload:
    return wk.WORKLOADS[key]


def algorithmic_ops(wl: wk.Workload, rules: np.ndarray) -> float:
    """Full-evaluation 32-bit word ops for one env-step, averaged over envs.

    Every rule rotation tests each of its input terms (a present or absent
    (position, channel) entry) at each valid anchor, and ORs each of its
    output entries (set or clear, per position and channel) at each valid
    anchor: one 32-bit op handles 32 anchors.  Rotation keeps the term and
    output counts; a 90-degree turn swaps h and w for the anchor count.
    """
    h = rules["h"].astype(np.int64)
    w = rules["w"].astype(np.int64)

    def popc(a):
        a = a.astype(np.uint64)
        c = np.zeros(a.shape, np.int64)
        for b in range(32):
            c += ((a >> np.uint64(b)) & np.uint64(1)).astype(np.int64)
        return c

    terms = popc(rules["present"]).sum(-1) + popc(rules["absent"]).sum(-1)
    outs = popc(rules["set"]).sum(-1) + popc(rules["clear"]).sum(-1)
    va = np.clip(wl.H - h + 1, 0, None) * np.clip(wl.W - w + 1, 0, None)
    vb = np.clip(wl.H - w + 1, 0, None) * np.clip(wl.W - h + 1, 0, None)
    anchors = 2 * va + 2 * vb  # rotations 0, 2 and 1, 3
    per_table = ((terms + outs) * anchors).sum(-1) / 32.0
    return float(per_table.mean())


# --------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples every 25 ms; stats over those taken inside the timed
    window (between mark_start and mark_end)."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.rows = []
        self.t0 = self.t1 = None

    def start(self, wait_s: float = 5.0):
        import threading
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "25"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return

        def reader():
            for line in self.proc.stdout:
                r = [x.strip() for x in line.split(",")]
                if len(r) >= 9:
                    self.rows.append((self._when(r[0]), r))

        threading.Thread(target=reader, daemon=True).start()
        end = time.time() + wait_s
        while not self.rows and time.time() < end:  # sampling has begun
            time.sleep(0.01)

    @staticmethod
    def _when(stamp: str) -> float | None:
        import datetime
        try:
            return datetime.datetime.strptime(stamp, "%Y/%m/%d %H:%M:%S.%f").timestamp()
        except ValueError:
            return None

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()
        end = self.t1 + 0.2
        while time.time() < end and not any(t and t >= self.t1 for t, _ in self.rows[-3:]):
            time.sleep(0.01)

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        inside = [r for t, r in self.rows if t is not None and self.t0 is not None
                  and self.t0 <= t <= self.t1]
        rows = inside or [r for _, r in self.rows]
        if not rows:
            return None
        mhz = [float(r[1]) for r in rows]
        mx = max(float(r[2]) for r in rows)
        reasons = set()
        for r in rows:
            for name, col in (("hw_slowdown", 5), ("hw_thermal_slowdown", 6),
                              ("sw_thermal_slowdown", 7), ("sw_power_cap", 8)):
                if r[col].strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(rows), "samples_in_timed_region": len(inside),
                "power_w_max": max(float(r[3]) for r in rows)}


def valid_anchor_rules(wl: wk.Workload, rules: np.ndarray) -> float:
    """Valid (anchor, rule rotation) pairs per env-step, averaged over envs."""
    h = rules["h"].astype(np.int64)
    w = rules["w"].astype(np.int64)
    va = np.clip(wl.H - h + 1, 0, None) * np.clip(wl.W - w + 1, 0, None)
    vb = np.clip(wl.H - w + 1, 0, None) * np.clip(wl.W - h + 1, 0, None)
    return float((2 * va + 2 * vb).sum(-1).mean())


def max_over_ranks(x: float, world: int, device) -> float:
    """The largest x over the ranks of the default process group (x itself
    with one rank).  `device` is where the reduction runs: the rank's GPU
    under NCCL, the CPU under gloo."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def measured_peaks() -> dict:
    try:
        return json.load(open(PEAKS_FILE))
    except (OSError, ValueError):
        return {}


def profile_path(kernel: str, wl) -> str:
    return os.path.join(PROFILE_DIR, f"{kernel}_{wl.name}.md")


def source_digest(src) -> str:
    """sha256 of a kernel's source: one file, or several read in order."""
    h = hashlib.sha256()
    for path in ((src,) if isinstance(src, str) else src):
        h.update(open(path, "rb").read())
    return h.hexdigest()


def profile_traffic(kernel: str, wl, src=KERNEL_SRC) -> float | None:
    """DRAM bytes per launch from the committed ncu summary of this kernel on
    this workload, if it was taken on the current kernel source `src` (a path,
    or a tuple of paths hashed together)."""
    return profile_field(kernel, wl, "dram_bytes_per_launch", src)


def cpu_baseline(wl, rules, cum, cfg, seed, budget_s: float = 12.0, variant=None) -> dict:
    """The oracle as it stands, all host cores, on a bounded sample of envs
    (variant: the variant semantics of the run, as keyword arguments)."""
    import oracle
    ov = oracle.make_variant(**variant) if variant else None
    threads = os.cpu_count() or 1
    s = wk.seeds(seed)
    n = max(threads, 8)
    steps = wl.steps
    while True:
        ids = np.arange(n)
        g = oracle.reset(cfg, cum, s["reset"], ids)
        t0 = time.perf_counter()
        oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), steps, s["actions"], env_ids=ids,
                       threads=threads, variant=ov)
        dt = time.perf_counter() - t0
        if dt > budget_s / 4 or n >= wl.batch:
            break
        n = min(wl.batch, int(n * max(2.0, budget_s / 4 / max(dt, 1e-3))))
    # The same oracle on one thread, over about one core's share of the sample.
    m = max(1, n // threads)
    ids1 = np.arange(m)
    g1 = oracle.reset(cfg, cum, s["reset"], ids1)
    t0 = time.perf_counter()
    oracle.rollout(cfg, rules, g1, g1, np.zeros(m, np.int32), steps, s["actions"], env_ids=ids1,
                   threads=1, variant=ov)
    dt1 = time.perf_counter() - t0
    return {"value": n * steps / dt, "unit": "env-steps/s", "cores": threads, "kind": "oracle",
            "sample": f"{n} of {wl.batch} envs x {steps} fused steps (envs are independent)",
            "seconds": dt,
            "one_thread": {"value": m * steps / dt1, "cores": 1,
                           "sample": f"{m} of {wl.batch} envs x {steps} fused steps"}}


# ------------------------------------------------------------ reference
def run_reference(args, wl):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    _, rules, cum = wk.make(wl, args.seed)
    fields = wk.config_fields(wl)
    cfg = oracle.make_cfg(**fields)
    threads = os.cpu_count() or 1
    s = wk.seeds(args.seed)
    n = max(threads, 16)
    ids = np.arange(n)
    ov = oracle.make_variant(**bench_variant(wl)) if args.variant else None
    g = oracle.reset(cfg, cum, s["reset"], ids)
    for _ in range(args.warmup):
        oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), 50, s["actions"], env_ids=ids,
                       threads=threads, variant=ov)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), wl.steps, s["actions"],
                       env_ids=ids, threads=threads, variant=ov)
        times.append(time.perf_counter() - t0)
    mean = sum(times) / len(times)
    value = n * wl.steps / mean
    line = {
        "impl": "reference", "metric": "env-steps/s", "value": value, "unit": "env-steps/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
        "data": "synthetic",
        "config": dict(config_dict(wl, sample=n), **({"workload": VariantName(wl).name,
                                                       "variant": bench_variant(wl)} if args.variant else {})),
        "cpu_baseline": {"value": value, "unit": "env-steps/s", "cores": threads,
                         "kind": "oracle",
                         "sample": f"{n} of {wl.batch} envs x {wl.steps} fused steps per step"},
        "e2e": {"value": value, "unit": "env-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def config_dict(wl, sample=None):
    full = wk.WORKLOADS[wl.key]
    name = wl.name if (wl.batch, wl.steps) == (full.batch, full.steps) else \
        f"{wl.name}, smaller case: {wl.batch} envs x {wl.steps} steps"
    if wl.base_game:
        name += " (rules 0-1 of each table: the maze game's 1x2 move and eat rules, not random 3x3)"
    l2 = "flushed (256 MiB write) between timed launches"
    if wl.trajectory:
        gb = wl.batch * wl.steps * traj_bytes_per_env_step(wl) / 1e9
        l2 = f"trajectory outputs ({gb:.1f} GB per launch) far exceed L2; also flushed (256 MiB write)" \
             " between timed launches"
    d = {"workload": name, "batch": wl.batch, "H": wl.H,
         "W": wl.W, "tile_channels": wl.C, "rules": wl.n_rules, "rotations": 4,
         "pattern_sizes": [f"{h}x{w}" for h, w in wl.shapes],
         "fused_steps_per_launch": wl.steps, "per_env_rules": bool(wl.rules_per_env),
         "trajectory_outputs": wl.trajectory,
         "l2": l2, "parallelism": "replicas"}
    if wl.max_steps or wl.auto_reset:
        d["done"] = f"no goal tile left or t = {wl.max_steps}" + (", auto-reset" if wl.auto_reset else "")
    if sample:
        d["sample_envs"] = sample
    return d


# ------------------------------------------------------------------ ours
def popcount(a: np.ndarray) -> np.ndarray:
    a = a.astype(np.uint64)
    c = np.zeros(a.shape, np.int64)
    for b in range(32):
        c += ((a >> np.uint64(b)) & np.uint64(1)).astype(np.int64)
    return c


def row_basis_ops(wl: wk.Workload, rules: np.ndarray) -> float:
    """Full-evaluation op count of one env-step on the basis the hot-path scope
    table uses: every rule rotation tests each input term (a present or absent
    (position, channel) entry) and ORs each output entry once per valid anchor
    ROW (one op per row of anchors), averaged over the environments' tables."""
    h = rules["h"].astype(np.int64)
    w = rules["w"].astype(np.int64)
    entries = (popcount(rules["present"]).sum(-1) + popcount(rules["absent"]).sum(-1) +
               popcount(rules["set"]).sum(-1) + popcount(rules["clear"]).sum(-1))
    rows_a = np.clip(wl.H - h + 1, 0, None) * (wl.W - w + 1 > 0)  # rotations 0, 2
    rows_b = np.clip(wl.H - w + 1, 0, None) * (wl.W - h + 1 > 0)  # rotations 1, 3
    return float((entries * (2 * rows_a + 2 * rows_b)).sum(-1).mean())


def traj_bytes_per_env_step(wl: wk.Workload) -> int:
    """Algorithmic HBM bytes of one env-step of a trajectory rollout: the
    observation (the board's canonical bytes), the int32 reward, the done byte."""
    return wl.H * wl.W * wl.cell_bytes + 4 + 1


def profile_field(kernel: str, wl, field: str, src=KERNEL_SRC) -> float | None:
    """A machine-readable figure of the committed ncu summary of this kernel on
    this workload, if the summary was taken on the current kernel source."""
    try:
        text = open(profile_path(kernel, wl)).read()
    except OSError:
        return None
    m = re.search(r"kernel_source_sha256:\s*([0-9a-f]{16,64})", text)
    t = re.search(field + r":\s*([0-9.eE+]+)", text)
    if not m or not t:
        return None
    return float(t.group(1)) if source_digest(src).startswith(m.group(1)) else None


def kernel_source(path: int, av):
    """The source of the rollout kernel for an av_rollout_path (or
    av_step_path) value: its file, or its files hashed together."""
    if path == av.AV_PATH_MEMO:
        return (MEMO_SRC, KERNEL_SRC)
    if path == av.AV_PATH_STEP:
        return (STEP_SRC, KERNEL_SRC)
    if path == av.AV_PATH_VARIANT:
        return VARIANT_SRC
    if path == av.AV_PATH_BAND:
        return BAND_SRC
    return KERNEL_SRC


def measure_activity(av, fields, rules, cum, wl, seed, dev, budget_bytes: int = 2 << 30) -> dict:
    """How much the rules do on this workload, counted on the GPU by the library
    itself (outside any timed region): one launch from the reset boards with the
    timed launches' first action seed, on a copy of the rule tables whose
    rewards are all 1, so that a step's reward is its number of rule
    applications ((rule, rotation, anchor) matches).  Envs beyond what a
    `budget_bytes` trajectory holds are left out (the first envs are kept)."""
    import torch
    per_env = wl.steps * wl.H * wl.W * wl.cell_bytes
    n = max(1, min(wl.batch, budget_bytes // max(per_env, 1)))
    r1 = rules.copy()
    r1["reward"] = 1
    if wl.rules_per_env:
        r1 = r1[:n]
    f = dict(fields, batch=n)
    c1 = cum[:n] if (cum is not None and cum.ndim == 2 and cum.shape[0] == wl.batch) else cum
    e = av.Env(f, r1, c1, device=dev)
    s = wk.seeds(seed)
    g0 = e.reset(s["reset"]).clone()
    res = e.rollout(wl.steps, s["actions"], trajectory=True)
    obs = res["obs"]
    prev = torch.cat([g0[None], obs[:-1]], 0)
    changed = (obs != prev).flatten(2).any(-1)
    matches = res["rew"].double()
    out = {"applications_per_env_step": float(matches.mean()),
           "match_step_frac": float((res["rew"] > 0).double().mean()),
           "board_change_frac": float(changed.double().mean()),
           "done_frac": float(res["done"].double().mean()),
           "source": f"library, first launch from the reset boards, {n} of {wl.batch} envs x"
                     f" {wl.steps} steps, rewards set to 1 on a copy of the tables"}
    e.close()
    return out


def time_rollout(args, wl, rank, world, dev, steps, warmup, e2e: bool):
    """Times `steps` av_rollout launches of workload wl (after `warmup`), L2
    flushed between launches outside the events.  Returns the measurements and
    the handle's setup (rules, cum, fields, seed, env)."""
    import torch

    import paper_2407_04221_gb300 as av
    seed = args.seed + 1000 * rank
    _, rules, cum = wk.make(wl, seed)
    fields = wk.config_fields(wl)
    env = av.Env(fields, rules, cum, device=dev)
    std_path = av.av_rollout_path(env.h)
    if args.variant:
        av.av_set_variant(env.h, **bench_variant(wl))
    s = wk.seeds(seed)
    g0 = env.reset(s["reset"])
    stream = torch.cuda.current_stream(dev)
    traj = None
    if wl.trajectory:
        traj = (env.boards(wl.steps, wl.batch),
                torch.zeros(wl.steps, wl.batch, dtype=torch.int32, device=dev),
                torch.zeros(wl.steps, wl.batch, dtype=torch.uint8, device=dev))
    rew_sum = torch.zeros(wl.batch, dtype=torch.int32, device=dev)
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)

    def launch(i):
        obs, rew, done = traj if traj else (None, None, None)
        av.av_rollout(env.h, wl.steps, s["actions"] + 7919 * i, obs, rew, done, rew_sum, stream)

    for i in range(warmup):
        launch(i)
    torch.cuda.synchronize(dev)
    env.sync()

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    sampler = ClockSampler(torch.cuda.current_device() if world == 1 else local_index(dev))
    sampler.start()
    barrier()
    sampler.mark_start()
    t_wall = time.perf_counter()
    for i in range(steps):
        flush.fill_(i & 0xff)  # evict L2 between timed launches (outside the events)
        starts[i].record(stream)
        launch(warmup + i)
        ends[i].record(stream)
    barrier()
    wall = time.perf_counter() - t_wall
    sampler.mark_end()
    clocks = sampler.stop()
    env.sync()
    ms = [a.elapsed_time(b) for a, b in zip(starts, ends)]
    kernel_ms = sum(ms) / len(ms)
    total_ms = max_over_ranks(sum(ms), world, dev)
    out = dict(rules=rules, cum=cum, fields=fields, seed=seed, env=env, std_path=std_path,
               path=av.av_rollout_path(env.h),
               kernel_ms=kernel_ms, total_ms=total_ms, wall=wall, clocks=clocks, g0=g0)
    if e2e:
        # the same launch through host buffers (pinned), copies timed
        host_in = g0.cpu().pin_memory()
        host_out = torch.empty(wl.batch, dtype=torch.int32).pin_memory()
        dev_in = torch.empty_like(g0)
        e2e_steps = max(3, min(steps, 20))
        barrier()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(e2e_steps):
            dev_in.copy_(host_in, non_blocking=True)
            av.av_set_state(env.h, dev_in, None, False, stream)
            launch(10_000 + i)
            host_out.copy_(rew_sum, non_blocking=True)
        e1.record(stream)
        barrier()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)
        out["e2e"] = {"value": wl.batch * wl.steps * world / (e2e_ms / 1e3), "unit": "env-steps/s",
                      "h2d_bytes_per_step": int(host_in.numel() * host_in.element_size()),
                      "d2h_bytes_per_step": int(host_out.numel() * host_out.element_size())}
    del traj, flush
    return out


def local_index(dev) -> int:
    return dev.index if dev.index is not None else 0


def rollout_roofline(av, wl, m, sm_mhz) -> dict:
    """Roofline of the rollout kernel that ran: HBM for trajectory workloads
    (the observation stream), integer issue otherwise."""
    peaks = measured_peaks()
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    path = av.av_rollout_path(m["env"].h)
    kernel = KERNEL_NAMES[path]
    if path == av.AV_PATH_VARIANT and wl.key in (1, 2):
        kernel = "rollout_variant_warp_kernel"  # variants on the one-warp layout
    pw = VariantName(wl) if path == av.AV_PATH_VARIANT else wl
    src = kernel_source(path, av)
    env_steps = wl.batch * wl.steps
    kernel_s = m["kernel_ms"] / 1e3
    ops = row_basis_ops(wl, m["rules"])
    peak_ops = SM_COUNT_GB300 * INT_LANES_PER_SM * sm_max * 1e6 / 1e9  # Gop/s
    inst = profile_field(kernel, pw, "warp_instructions_per_launch", src)
    clock = (sm_mhz or sm_max) * 1e6
    alu = {"achieved": ops * env_steps / kernel_s / 1e9, "peak": peak_ops, "unit": "Gop/s",
           "frac": ops * env_steps / kernel_s / 1e9 / peak_ops, "ops_per_env_step": ops,
           "ops_basis": "full evaluation, one op per (rule rotation, input or output entry,"
                        " valid anchor row); the kernels evaluate far less (early exit, and"
                        " the memoising rollout evaluates a (board, action) pair once), so this"
                        " ratio is a full-evaluation equivalent, not a utilisation",
           "peak_from": f"{SM_COUNT_GB300} SMs x {INT_LANES_PER_SM} int32 lanes/clk"
                        f" x {sm_max:.0f} MHz (sm_max_mhz of measured peaks); the LOP3 issue"
                        " probe measured 76 of the 128 lanes/clk",
           "issue_util": (inst / (SM_COUNT_GB300 * 4 * clock * kernel_s)) if inst else None,
           "issue_util_basis": "ncu warp instructions of one launch (committed profile, scaled to"
                               " this launch by env-steps) / (152 SMs x 4 schedulers x median SM"
                               " clock x launch time)"}
    if wl.batch == 1:
        alu["note"] = ("one environment: the launch is bound by the latency of one CTA, so the"
                       " fraction says nothing about the kernel's use of the GPU")
    if wl.trajectory:
        bpes = traj_bytes_per_env_step(wl)
        peak = float(peaks.get("hbm_gbs", 6723.0))
        achieved = bpes * env_steps / kernel_s / 1e9
        return {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": profile_traffic(kernel, pw, src),
                "kernel": kernel, "bytes_per_env_step": bpes,
                "bytes_basis": "observation (board bytes) + int32 reward + done byte per env-step"
                               " (boards in and out once per launch not counted)",
                "peak_from": "hbm_gbs of measured peaks (copy bandwidth)", "alu": alu}
    out = {"bound": "alu", "achieved": alu["achieved"], "peak": peak_ops, "unit": "Gop/s",
           "frac": alu["frac"], "traffic": profile_traffic(kernel, pw, src), "kernel": kernel,
           "ops_per_env_step": ops, "ops_basis": alu["ops_basis"], "peak_from": alu["peak_from"],
           "issue_util": alu["issue_util"], "issue_util_basis": alu["issue_util_basis"]}
    if "note" in alu:
        out["note"] = alu["note"]
    return out


def run_ours(args, wl):
    import torch

    import paper_2407_04221_gb300 as av

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    m = time_rollout(args, wl, rank, world, dev, args.steps, args.warmup, e2e=True)
    value = wl.batch * wl.steps * args.steps * world / (m["total_ms"] / 1e3)
    activity = None
    if rank == 0 and not args.variant:
        activity = measure_activity(av, m["fields"], m["rules"], m["cum"], wl, m["seed"], dev)
    extra = {}
    if world == 1 and args.extra and wl.key == 3 and args.batch == 0 and args.fused_steps == 0:
        wl5 = workload_for(5)
        m5 = time_rollout(args, wl5, rank, world, dev, min(args.steps, 10), 3, e2e=False)
        v5 = wl5.batch * wl5.steps * min(args.steps, 10) / (m5["total_ms"] / 1e3)
        sm5 = (m5["clocks"] or {}).get("sm_mhz")
        extra[wl5.name] = {
            "value": v5, "unit": "env-steps/s", "steps": min(args.steps, 10), "warmup": 3,
            "ms_per_step": m5["total_ms"] / min(args.steps, 10),
            "config": config_dict(wl5),
            "cell_rule_updates_per_s": v5 * wl5.H * wl5.W * wl5.n_rules * 4,
            "roofline": rollout_roofline(av, wl5, m5, sm5),
            "activity": measure_activity(av, m5["fields"], m5["rules"], m5["cum"], wl5, m5["seed"], dev),
            "clocks": m5["clocks"]}
        m5["env"].close()

    if rank == 0:
        sm_mhz = (m["clocks"] or {}).get("sm_mhz")
        line = {
            "metric": "env-steps/s", "value": value, "unit": "env-steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": m["total_ms"] / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
            "data": "synthetic",
            "config": dict(config_dict(wl), **({"workload": VariantName(wl).name,
                                                "variant": bench_variant(wl)} if args.variant else {})),
            "cell_rule_updates_per_s": value * wl.H * wl.W * wl.n_rules * 4,
            "valid_anchor_rule_tests_per_s": value * valid_anchor_rules(wl, m["rules"]),
            "e2e": m["e2e"],
            "roofline": rollout_roofline(av, wl, m, sm_mhz),
            "gpu_launches": args.steps * (2 if m["path"] == av.AV_PATH_MEMO else 1),
            "wall_s_timed_region": m["wall"],
        }
        if activity:
            line["activity"] = activity
        if m["clocks"]:
            line["clocks"] = m["clocks"]
        if world == 1 and not args.no_cpu_baseline:
            import oracle
            cfg = oracle.make_cfg(**m["fields"])
            line["cpu_baseline"] = cpu_baseline(wl, m["rules"], m["cum"], cfg, m["seed"],
                                                variant=bench_variant(wl) if args.variant else None)
        if extra:
            line["extra"] = extra
        print(json.dumps(line))
    m["env"].close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def run_single_step(args, wl):
    """One benchmark step = one av_step over the workload's batch: one kernel
    launch, the boards read and written once, obs / reward / done written to
    caller buffers, actions read from a device buffer (seeded, uniform 0..4,
    a new row each step).  L2 flushed between timed launches."""
    import torch

    import paper_2407_04221_gb300 as av
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    seed = args.seed + 1000 * rank
    _, rules, cum = wk.make(wl, seed)
    fields = wk.config_fields(wl)
    env = av.Env(fields, rules, cum, device=dev)
    s = wk.seeds(seed)
    env.reset(s["reset"])
    n_act = args.warmup + args.steps
    acts = torch.from_numpy(wk.actions(s["actions"], wl.batch, n_act)).to(dev)  # [n_act][B] uint8
    obs = env.boards(wl.batch)
    rew = torch.zeros(wl.batch, dtype=torch.int32, device=dev)
    done = torch.zeros(wl.batch, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
    for i in range(args.warmup):
        av.av_step(env.h, acts[i], obs, rew, done, stream)
    torch.cuda.synchronize(dev)
    env.sync()

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(torch.cuda.current_device() if world == 1 else local)
    sampler.start()
    barrier()
    sampler.mark_start()
    t_wall = time.perf_counter()
    for i in range(args.steps):
        flush.fill_(i & 0xff)
        starts[i].record(stream)
        av.av_step(env.h, acts[args.warmup + i], obs, rew, done, stream)
        ends[i].record(stream)
    barrier()
    wall = time.perf_counter() - t_wall
    sampler.mark_end()
    clocks = sampler.stop()
    env.sync()
    ms = [a.elapsed_time(b) for a, b in zip(starts, ends)]
    kernel_ms = sum(ms) / len(ms)
    total_ms = max_over_ranks(sum(ms), world, dev)
    value = wl.batch * args.steps * world / (total_ms / 1e3)

    # e2e: actions in from pinned host memory, rewards and done flags back
    host_a = acts[: min(20, n_act)].cpu().pin_memory()
    host_r = torch.empty(wl.batch, dtype=torch.int32).pin_memory()
    host_d = torch.empty(wl.batch, dtype=torch.uint8).pin_memory()
    dev_a = torch.empty_like(acts[0])
    e2e_steps = max(3, min(args.steps, host_a.shape[0]))
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(e2e_steps):
        dev_a.copy_(host_a[i], non_blocking=True)
        av.av_step(env.h, dev_a, obs, rew, done, stream)
        host_r.copy_(rew, non_blocking=True)
        host_d.copy_(done, non_blocking=True)
    e1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)

    if rank == 0:
        peaks = measured_peaks()
        path = av.av_step_path(env.h)
        kernel = KERNEL_NAMES[path]
        src = kernel_source(path, av)
        sw = SingleStepName(wl)
        board = wl.H * wl.W * wl.cell_bytes
        bpes = 2 * board + 1 + 4 + 1
        peak = float(peaks.get("hbm_gbs", 6723.0))
        achieved = bpes * wl.batch / (kernel_ms / 1e3) / 1e9
        traffic = profile_traffic(kernel, sw, src)
        inst = profile_field(kernel, sw, "warp_instructions_per_launch", src)
        clock = float((clocks or {}).get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)) * 1e6
        line = {
            "metric": "env-steps/s", "value": value, "unit": "env-steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32",
            "data": "synthetic",
            "config": dict(config_dict(wl), workload=sw.name, fused_steps_per_launch=1,
                           actions="seeded uniform 0..4 from a device buffer, one row per step",
                           l2="flushed (256 MiB write) between timed launches"),
            "e2e": {"value": wl.batch * world / (e2e_ms / 1e3), "unit": "env-steps/s",
                    "h2d_bytes_per_step": wl.batch, "d2h_bytes_per_step": 5 * wl.batch},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic, "kernel": kernel,
                         "bytes_per_env_step": bpes,
                         "bytes_basis": "board in + observation out + action + int32 reward + done"
                                        " byte; the handle's own copy of the board written back and"
                                        " the env's rule table (per-env tables, read every launch)"
                                        " are extra traffic, counted in `traffic`",
                         "traffic_per_env_step": traffic / wl.batch if traffic else None,
                         "peak_from": "hbm_gbs of measured peaks (copy bandwidth)",
                         "issue_util": (inst / (SM_COUNT_GB300 * 4 * clock * kernel_ms / 1e3))
                                       if inst else None,
                         "issue_util_basis": "ncu warp instructions of one launch (committed"
                                             " profile) / (152 SMs x 4 schedulers x median SM"
                                             " clock x launch time): the step's limiter"},
            "gpu_launches": args.steps,
            "wall_s_timed_region": wall,
        }
        if clocks:
            line["clocks"] = clocks
        print(json.dumps(line))
    env.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


class SingleStepName:
    """Profile naming for single-step launches of a workload."""
    def __init__(self, wl):
        self.name = f"{wl.name.replace('-traj', '')}-step"


# ------------------------------------------------------------ search (config 4)
def search_ops_per_child(wl, rules) -> float:
    """Full-evaluation ops of one child's step plus its FNV-1a-64 hash: per
    board byte one 64-bit xor and one 64-bit multiply, counted as 2 + 4
    32-bit operations."""
    return algorithmic_ops(wl, rules) + 6.0 * wl.H * wl.W * wl.cell_bytes


def search_children(trace_n) -> int:
    """Children generated by one search: 5 per parent expanded.  The root is
    the only parent of iteration 0; later iterations expand the frontier the
    previous one selected."""
    import torch
    n = trace_n.to(torch.int64)
    parents = n.shape[0] + int(n[:, :-1].sum())
    return 5 * parents


def run_search(args, wl):
    """One benchmark step = one full search per env (Env.search: iterations of
    av_expand + av_select from the reset boards); env-steps count children."""
    import torch

    import paper_2407_04221_gb300 as av

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    seed = args.seed + 1000 * rank
    _, rules, cum = wk.make(wl, seed)
    fields = wk.config_fields(wl)
    k, iters = wl.frontier, wl.iterations
    env = av.Env(fields, rules, cum, device=dev, search_capacity=1 + k * iters)
    s = wk.seeds(seed)
    roots = env.reset(s["reset"]).clone()
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        res = env.search(roots, iters, k)
    torch.cuda.synchronize(dev)
    env.sync()
    children = search_children(res["trace_n"])  # the same every step: same roots, same rules

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(torch.cuda.current_device() if world == 1 else local)
    sampler.start()
    barrier()
    sampler.mark_start()
    t_wall = time.perf_counter()
    for i in range(args.steps):
        flush.fill_(i & 0xff)
        starts[i].record(stream)
        env.search(roots, iters, k)
        ends[i].record(stream)
    barrier()
    wall = time.perf_counter() - t_wall
    sampler.mark_end()
    clocks = sampler.stop()
    env.sync()
    total_ms = sum(a.elapsed_time(b) for a, b in zip(starts, ends))
    total_ms = max_over_ranks(total_ms, world, dev)
    value = children * args.steps * world / (total_ms / 1e3)

    # ---- the expand kernel alone: events around each av_expand of one search
    # (the same calls, in the same order, as Env.search)
    i32, u8 = torch.int32, torch.uint8
    front, nxt = env.boards(wl.batch, k), env.boards(wl.batch, k)
    cum_, ncum = (torch.zeros(wl.batch, k, dtype=i32, device=dev) for _ in range(2))
    hsh, nhsh = (torch.zeros(wl.batch, k, dtype=torch.int64, device=dev) for _ in range(2))
    live, nlive = (torch.zeros(wl.batch, k, dtype=u8, device=dev) for _ in range(2))
    n = torch.ones(wl.batch, dtype=i32, device=dev)
    nn = torch.zeros_like(n)
    front[:, 0].copy_(roots)
    rh = torch.zeros(wl.batch, dtype=torch.int64, device=dev)
    rl = torch.zeros(wl.batch, dtype=u8, device=dev)
    av.av_search_init(env.h, roots, rh, rl)
    hsh[:, 0].copy_(rh)
    live[:, 0].copy_(rl)
    ch = env.boards(wl.batch, k, 5)
    rw = torch.zeros(wl.batch, k, 5, dtype=i32, device=dev)
    dn = torch.zeros(wl.batch, k, 5, dtype=u8, device=dev)
    chh = torch.zeros(wl.batch, k, 5, dtype=torch.int64, device=dev)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(iters)]
    parents = []
    for it in range(iters):
        parents.append(n.clone())
        ev[it][0].record(stream)
        av.av_expand(env.h, front, k, ch, rw, dn, chh, n)
        ev[it][1].record(stream)
        av.av_select(env.h, k, n, cum_, live, ch, rw, dn, chh, k, nxt, ncum, nhsh, nlive, nn)
        front, nxt, cum_, ncum, hsh, nhsh = nxt, front, ncum, cum_, nhsh, hsh
        live, nlive, n, nn = nlive, live, nn, n
    torch.cuda.synchronize(dev)
    env.sync()
    exp_ms = sum(a.elapsed_time(b) for a, b in ev)
    exp_children = 5 * int(sum(int(p.sum()) for p in parents))

    # ---- e2e: roots from pinned host memory, best cumulative reward back
    host_roots = roots.cpu().pin_memory()
    host_best = torch.empty(wl.batch, iters, dtype=torch.int32).pin_memory()
    dev_roots = torch.empty_like(roots)
    e2e_steps = max(3, min(args.steps, 10))
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        dev_roots.copy_(host_roots, non_blocking=True)
        r = env.search(dev_roots, iters, k)
        host_best.copy_(r["trace_best"], non_blocking=True)
    e1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)
    e2e_value = children * world / (e2e_ms / 1e3)

    if rank == 0:
        peaks = measured_peaks()
        sm_max = float(peaks.get("sm_max_mhz", 2070.0))
        peak_ops = SM_COUNT_GB300 * INT_LANES_PER_SM * sm_max * 1e6 / 1e9
        ops = search_ops_per_child(wl, rules)
        achieved = ops * exp_children / (exp_ms / 1e3) / 1e9
        kernel = "expand_warp_kernel" if wl.H * wl.W <= 512 else "expand_kernel"
        line = {
            "metric": "env-steps/s", "value": value, "unit": "env-steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8",
            "data": "synthetic",
            "config": dict(config_dict(wl), frontier=k, iterations=iters,
                           children_per_step=children,
                           rules_note="rules 0-1 of every table are the maze game's move and"
                                      " eat rules, the rest random"),
            "e2e": {"value": e2e_value, "unit": "env-steps/s",
                    "h2d_bytes_per_step": int(host_roots.numel() * host_roots.element_size()),
                    "d2h_bytes_per_step": int(host_best.numel() * host_best.element_size())},
            "roofline": {"bound": "alu", "achieved": achieved, "peak": peak_ops,
                         "unit": "Gop/s", "frac": achieved / peak_ops,
                         "traffic": profile_traffic(kernel, wl), "kernel": kernel,
                         "ops_per_child": ops,
                         "ops_basis": "full evaluation of the child's step (as for rollouts)"
                                      " plus FNV-1a-64 over the child's board, 6 ops per byte",
                         "kernel_ms_per_search": exp_ms,
                         "peak_from": f"{SM_COUNT_GB300} SMs x {INT_LANES_PER_SM} int32 lanes/clk"
                                      f" x {sm_max:.0f} MHz (sm_max_mhz of measured peaks)"},
            "gpu_launches": args.steps * (1 + 2 * iters),
            "wall_s_timed_region": wall,
        }
        if clocks:
            line["clocks"] = clocks
        if world == 1 and not args.no_cpu_baseline:
            import oracle
            cfg = oracle.make_cfg(**fields)
            line["cpu_baseline"] = search_cpu_baseline(wl, rules, cum, cfg, seed)
        print(json.dumps(line))
    env.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def search_cpu_baseline(wl, rules, cum, cfg, seed, budget_s: float = 12.0) -> dict:
    """The oracle's search, all host cores, on a bounded sample of envs."""
    import oracle
    threads = os.cpu_count() or 1
    s = wk.seeds(seed)
    n = min(wl.batch, max(threads, 4))
    while True:
        ids = np.arange(n)
        roots = oracle.reset(cfg, cum, s["reset"], ids)
        t0 = time.perf_counter()
        ref = oracle.search(cfg, rules, roots, wl.iterations, wl.frontier, env_ids=ids,
                            threads=threads)
        dt = time.perf_counter() - t0
        if dt > budget_s / 4 or n >= wl.batch:
            break
        n = min(wl.batch, int(n * max(2.0, budget_s / 4 / max(dt, 1e-3))))
    children = 5 * (n + int(ref["trace_n"][:, :-1].sum()))
    # The same search on one thread, over about one core's share of the sample.
    m = max(1, n // threads)
    ids1 = np.arange(m)
    roots1 = oracle.reset(cfg, cum, s["reset"], ids1)
    t0 = time.perf_counter()
    one = oracle.search(cfg, rules, roots1, wl.iterations, wl.frontier, env_ids=ids1, threads=1)
    dt1 = time.perf_counter() - t0
    children1 = 5 * (m + int(one["trace_n"][:, :-1].sum()))
    return {"value": children / dt, "unit": "env-steps/s", "cores": threads, "kind": "oracle",
            "sample": f"{n} of {wl.batch} envs, full search ({wl.iterations} iterations,"
                      f" frontier {wl.frontier})", "seconds": dt,
            "one_thread": {"value": children1 / dt1, "cores": 1,
                           "sample": f"{m} of {wl.batch} envs, full search"}}


def run_search_reference(args, wl):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    _, rules, cum = wk.make(wl, args.seed)
    fields = wk.config_fields(wl)
    cfg = oracle.make_cfg(**fields)
    threads = os.cpu_count() or 1
    s = wk.seeds(args.seed)
    n = min(wl.batch, max(threads, 4))
    ids = np.arange(n)
    roots = oracle.reset(cfg, cum, s["reset"], ids)
    for _ in range(args.warmup):
        oracle.search(cfg, rules, roots, 2, wl.frontier, env_ids=ids, threads=threads)
    times, children = [], 0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        ref = oracle.search(cfg, rules, roots, wl.iterations, wl.frontier, env_ids=ids,
                            threads=threads)
        times.append(time.perf_counter() - t0)
        children = 5 * (n + int(ref["trace_n"][:, :-1].sum()))
    mean = sum(times) / len(times)
    value = children / mean
    line = {
        "impl": "reference", "metric": "env-steps/s", "value": value, "unit": "env-steps/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8",
        "data": "synthetic", "config": dict(config_dict(wl, sample=n), frontier=wl.frontier,
                                            iterations=wl.iterations),
        "cpu_baseline": {"value": value, "unit": "env-steps/s", "cores": threads,
                         "kind": "oracle",
                         "sample": f"{n} of {wl.batch} envs, full search per step"},
        "e2e": {"value": value, "unit": "env-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ------------------------------------------------- policy observation
OBSERVE_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "k_observe.cu")
OBSERVE_ROLLOUT_STEPS = 60  # boards observed after this many random steps (multi-hot cells)


class ObserveWorkload:
    """Player-centred patches (av_observe) of the 16,384 boards of the
    training shape (16 x 16, C = 10) for one window width."""

    def __init__(self, base: wk.Workload, window: int):
        self.base, self.window = base, window
        self.name = f"observe-w{window}-grid{base.H}-b{base.batch}-c{base.C}"

    def bytes_per_obs(self) -> int:
        b = self.base
        return b.H * b.W * b.cell_bytes + self.window * self.window * b.C

    def config(self, sample=None) -> dict:
        b = self.base
        d = {"workload": self.name, "batch": b.batch, "H": b.H, "W": b.W, "tile_channels": b.C,
             "window": self.window, "obs_layout": "uint8 [B][window][window][C], channels last",
             "boards": f"reset, then {OBSERVE_ROLLOUT_STEPS} random-action steps of the"
                       f" {b.n_rules}-rule tables",
             "l2": "flushed (256 MiB write) between timed launches", "parallelism": "replicas"}
        if sample:
            d["sample_envs"] = sample
        return d


def observe_boards(wl: ObserveWorkload, seed: int, env=None):
    """(env, boards after the warm-up rollout) for the observation benchmark."""
    s = wk.seeds(seed)
    env.reset(s["reset"])
    env.rollout(OBSERVE_ROLLOUT_STEPS, s["actions"])
    g, _ = env.get_state()
    return g


def observe_cpu_baseline(cfg, boards_np, window, budget_s: float = 4.0) -> dict:
    """The oracle's observation (one thread), repeated over the whole batch."""
    import oracle
    t0 = time.perf_counter()
    reps = 0
    while True:
        oracle.observe(cfg, boards_np, window)
        reps += 1
        dt = time.perf_counter() - t0
        if dt > budget_s:
            break
    n = boards_np.shape[0]
    return {"value": reps * n / dt, "unit": "observations/s", "cores": 1, "kind": "oracle",
            "sample": f"all {n} boards x {reps} passes", "seconds": dt}


def run_observe(args, wl: ObserveWorkload):
    """One benchmark step = one av_observe launch over every board."""
    import torch

    import paper_2407_04221_gb300 as av

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    seed = args.seed + 1000 * rank
    base = wl.base
    _, rules, cum = wk.make(base, seed)
    fields = wk.config_fields(base)
    env = av.Env(fields, rules, cum, device=dev)
    boards = observe_boards(wl, seed, env)
    B, w = base.batch, wl.window
    obs = torch.empty(B, w, w, base.C, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        av.av_observe(env.h, None, w, obs, None, stream)
    torch.cuda.synchronize(dev)
    env.sync()

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(torch.cuda.current_device() if world == 1 else local)
    sampler.start()
    barrier()
    sampler.mark_start()
    t_wall = time.perf_counter()
    for i in range(args.steps):
        flush.fill_(i & 0xff)
        starts[i].record(stream)
        av.av_observe(env.h, None, w, obs, None, stream)
        ends[i].record(stream)
    barrier()
    wall = time.perf_counter() - t_wall
    sampler.mark_end()
    clocks = sampler.stop()
    env.sync()
    ms = [a.elapsed_time(b) for a, b in zip(starts, ends)]
    kernel_ms = sum(ms) / len(ms)
    total_ms = max_over_ranks(sum(ms), world, dev)
    value = B * args.steps * world / (total_ms / 1e3)

    # ---- e2e: boards from pinned host memory in, observations to pinned host memory out
    host_in = boards.cpu().pin_memory()
    host_out = torch.empty(obs.shape, dtype=torch.uint8).pin_memory()
    dev_in = torch.empty_like(boards)
    e2e_steps = max(3, min(args.steps, 10))
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(e2e_steps):
        dev_in.copy_(host_in, non_blocking=True)
        av.av_observe(env.h, dev_in, w, obs, None, stream)
        host_out.copy_(obs, non_blocking=True)
    e1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)
    e2e_value = B * world / (e2e_ms / 1e3)

    if rank == 0:
        peaks = measured_peaks()
        peak = float(peaks.get("hbm_gbs", 6800.0))
        per_obs = wl.bytes_per_obs()
        achieved = per_obs * B / (kernel_ms / 1e3) / 1e9
        line = {
            "metric": "observations/s", "value": value, "unit": "observations/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": total_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "u8", "data": "synthetic", "config": wl.config(),
            "e2e": {"value": e2e_value, "unit": "observations/s",
                    "h2d_bytes_per_step": int(host_in.numel() * host_in.element_size()),
                    "d2h_bytes_per_step": int(host_out.numel())},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak,
                         "traffic": profile_traffic("observe_kernel", wl, OBSERVE_SRC),
                         "kernel": "observe_kernel", "bytes_per_obs": per_obs,
                         "bytes_basis": "board read once (H*W cell bytes) + patch written once"
                                        " (window^2 * C bytes)",
                         "peak_from": "hbm_gbs of measured peaks" if "hbm_gbs" in peaks
                                      else "fallback 6800 GB/s"},
            "gpu_launches": args.steps,
            "wall_s_timed_region": wall,
        }
        if clocks:
            line["clocks"] = clocks
        if world == 1 and not args.no_cpu_baseline:
            import oracle
            line["cpu_baseline"] = observe_cpu_baseline(oracle.make_cfg(**fields),
                                                        gpu_boards_np(boards), w)
        print(json.dumps(line))
    env.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def gpu_boards_np(t) -> np.ndarray:
    a = t.cpu().numpy()
    return a.view(np.uint16) if a.dtype == np.int16 else a


def run_observe_reference(args, wl: ObserveWorkload):
    """The oracle's observation on the host, on the same boards (made by the
    oracle's own rollout of the same seeds), one thread."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    base = wl.base
    _, rules, cum = wk.make(base, args.seed)
    cfg = oracle.make_cfg(**wk.config_fields(base))
    s = wk.seeds(args.seed)
    n = min(base.batch, 2048)
    ids = np.arange(n)
    g = oracle.reset(cfg, cum, s["reset"], ids)
    g = oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), OBSERVE_ROLLOUT_STEPS,
                       s["actions"], env_ids=ids)["grids"]
    for _ in range(args.warmup):
        oracle.observe(cfg, g[:64], wl.window)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.observe(cfg, g, wl.window)
        times.append(time.perf_counter() - t0)
    mean = sum(times) / len(times)
    value = n / mean
    line = {
        "impl": "reference", "metric": "observations/s", "value": value,
        "unit": "observations/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": mean * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u8", "data": "synthetic", "config": wl.config(sample=n),
        "cpu_baseline": {"value": value, "unit": "observations/s", "cores": 1, "kind": "oracle",
                         "sample": f"{n} of {base.batch} boards per step"},
        "e2e": {"value": value, "unit": "observations/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------- mutation
MUTATE_SRC = os.path.join(ROOT, "paper_2407_04221_gb300", "csrc", "k_mutate.cu")
MIX64_OPS = 20  # 32-bit operations of one SplitMix64 finaliser (3 xor-shifts, 2 64-bit multiplies, input xor)


class VariantName:
    """Name of a rollout workload run under the benchmark's variant semantics."""

    def __init__(self, wl):
        self.name = f"{wl.name}-variant"


class MutateName:
    """Name of the mutation workload (for its profile summary)."""

    def __init__(self, wl):
        self.name = f"mutate-grid{wl.H}-b{wl.batch}-c{wl.C}-r{wl.n_rules}"


def mutation_rates(wl) -> dict:
    """Rates of the mutation benchmark: about ten map bits per board, one in
    eight rule entries, one in four rewards; every rule slot mutable."""
    bits = wl.H * wl.W * wl.C
    return dict(p_map=max(1, (10 << 24) // bits), map_channels=(1 << wl.C) - 1, p_rule=1 << 21,
                p_reward=1 << 22, reward_min=wl.reward_lo, reward_max=wl.reward_hi,
                mutable_rules=(1 << wl.n_rules) - 1)


def mutation_draws(wl, rules) -> float:
    """Counter draws (one mix each) per environment of one av_mutate call,
    averaged over the tables, plus the three-mix prefixes per stream."""
    cells = wl.H * wl.W * wl.C + 2
    entries = (rules["h"].astype(np.int64) * rules["w"]).sum(axis=1).mean()
    rule_draws = entries * (2 * wl.C + 1) + 4 + 2 + wl.n_rules * (1 + 0.25)
    return float(cells + rule_draws)


def run_mutate(args, wl):
    """One benchmark step = one av_mutate call over every map and rule table
    of the 16,384-env training shape."""
    import torch

    import paper_2407_04221_gb300 as av

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    seed = args.seed + 1000 * rank
    _, rules, cum = wk.make(wl, seed)
    fields = wk.config_fields(wl)
    import oracle
    cfg = oracle.make_cfg(**fields)
    env = av.Env(fields, rules, cum, device=dev)
    maps0 = env.reset(wk.seeds(seed)["reset"])
    env.close()
    B, R = wl.batch, wl.n_rules
    maps = maps0.clone()
    rules_dev = torch.from_numpy(np.ascontiguousarray(rules).view(np.uint8).reshape(B, R, 408).copy()).to(dev)
    rates = mutation_rates(wl)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)

    def launch(i):
        av.av_mutate(B, wl.H, wl.W, wl.C, R, rates, seed * 7919 + i, maps, rules_dev, stream)

    for i in range(args.warmup):
        launch(i)
    torch.cuda.synchronize(dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(torch.cuda.current_device() if world == 1 else local)
    sampler.start()
    barrier()
    sampler.mark_start()
    t_wall = time.perf_counter()
    for i in range(args.steps):
        flush.fill_(i & 0xff)
        starts[i].record(stream)
        launch(args.warmup + i)
        ends[i].record(stream)
    barrier()
    wall = time.perf_counter() - t_wall
    sampler.mark_end()
    clocks = sampler.stop()
    ms = [a.elapsed_time(b) for a, b in zip(starts, ends)]
    kernel_ms = sum(ms) / len(ms)
    total_ms = max_over_ranks(sum(ms), world, dev)
    value = B * args.steps * world / (total_ms / 1e3)

    # ---- e2e: maps and tables from pinned host memory, mutated copies back
    h_maps = maps0.cpu().pin_memory()
    h_rules = rules_dev.cpu().pin_memory()
    o_maps = torch.empty_like(h_maps).pin_memory()
    o_rules = torch.empty_like(h_rules).pin_memory()
    e2e_steps = max(3, min(args.steps, 20))
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(e2e_steps):
        maps.copy_(h_maps, non_blocking=True)
        rules_dev.copy_(h_rules, non_blocking=True)
        launch(50_000 + i)
        o_maps.copy_(maps, non_blocking=True)
        o_rules.copy_(rules_dev, non_blocking=True)
    e1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world, dev)
    e2e_value = B * world / (e2e_ms / 1e3)

    if rank == 0:
        peaks = measured_peaks()
        sm_max = float(peaks.get("sm_max_mhz", 2070.0))
        peak_ops = SM_COUNT_GB300 * INT_LANES_PER_SM * sm_max * 1e6 / 1e9
        ops = mutation_draws(wl, rules) * MIX64_OPS
        achieved = ops * B / (kernel_ms / 1e3) / 1e9
        nbytes = 2 * (wl.H * wl.W * wl.cell_bytes + R * 408)
        hbm = float(peaks.get("hbm_gbs", 6800.0))
        line = {
            "metric": "env-mutations/s", "value": value, "unit": "env-mutations/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": total_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "u64", "data": "synthetic",
            "config": {"workload": MutateName(wl).name, "batch": B, "H": wl.H,
                       "W": wl.W, "tile_channels": wl.C, "rules": R, "rates": rates,
                       "l2": "flushed (256 MiB write) between timed launches",
                       "parallelism": "replicas"},
            "e2e": {"value": e2e_value, "unit": "env-mutations/s",
                    "h2d_bytes_per_step": int(h_maps.numel() * h_maps.element_size() + h_rules.numel()),
                    "d2h_bytes_per_step": int(o_maps.numel() * o_maps.element_size() + o_rules.numel())},
            "roofline": {"bound": "alu", "achieved": achieved, "peak": peak_ops, "unit": "Gop/s",
                         "frac": achieved / peak_ops,
                         "traffic": profile_traffic("mutate_kernels", MutateName(wl), MUTATE_SRC),
                         "kernel": "mutate_maps_kernel + mutate_rules_kernel",
                         "ops_per_env": ops,
                         "ops_basis": f"one SplitMix64 mix ({MIX64_OPS} 32-bit ops) per decision"
                                      " (map bit, rule entry channel, reward) plus the per-stream"
                                      " prefixes",
                         "hbm_frac": nbytes * B / (kernel_ms / 1e3) / 1e9 / hbm,
                         "bytes_per_env": nbytes,
                         "peak_from": f"{SM_COUNT_GB300} SMs x {INT_LANES_PER_SM} int32 lanes/clk"
                                      f" x {sm_max:.0f} MHz (sm_max_mhz of measured peaks)"},
            "gpu_launches": 2 * args.steps,
            "wall_s_timed_region": wall,
        }
        if clocks:
            line["clocks"] = clocks
        if world == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = mutate_cpu_baseline(wl, rules, maps0, rates, seed)
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def mutate_cpu_baseline(wl, rules, maps0, rates, seed, budget_s: float = 3.0) -> dict:
    """The oracle's mutation, one thread, on a sample of environments."""
    import oracle
    m = maps0.cpu().numpy()
    m = m.view(np.uint16) if m.dtype == np.int16 else m
    n = 256
    ids = np.arange(n, dtype=np.int32)
    reps, t0 = 0, time.perf_counter()
    while True:
        oracle.mutate(wl.H, wl.W, wl.C, rates, seed, m[:n], rules[:n], env_ids=ids)
        reps += 1
        dt = time.perf_counter() - t0
        if dt > budget_s:
            break
    return {"value": reps * n / dt, "unit": "env-mutations/s", "cores": 1, "kind": "oracle",
            "sample": f"{n} of {wl.batch} envs x {reps} passes", "seconds": dt}


def run_mutate_reference(args, wl):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    _, rules, cum = wk.make(wl, args.seed)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    n = 1024
    maps = oracle.reset(cfg, cum, wk.seeds(args.seed)["reset"], range(n))
    rates = mutation_rates(wl)
    ids = np.arange(n, dtype=np.int32)
    for _ in range(args.warmup):
        oracle.mutate(wl.H, wl.W, wl.C, rates, 1, maps[:64], rules[:64], env_ids=ids[:64])
    times = []
    for i in range(args.steps):
        t0 = time.perf_counter()
        oracle.mutate(wl.H, wl.W, wl.C, rates, i, maps, rules[:n], env_ids=ids)
        times.append(time.perf_counter() - t0)
    mean = sum(times) / len(times)
    value = n / mean
    line = {
        "impl": "reference", "metric": "env-mutations/s", "value": value,
        "unit": "env-mutations/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": mean * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": {"workload": f"mutate-grid{wl.H}-b{wl.batch}-c{wl.C}-r{wl.n_rules}",
                   "sample_envs": n, "rates": rates},
        "cpu_baseline": {"value": value, "unit": "env-mutations/s", "cores": 1, "kind": "oracle",
                         "sample": f"{n} of {wl.batch} envs per step"},
        "e2e": {"value": value, "unit": "env-mutations/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def run_int_probe() -> int:
    """Build and run the integer-issue probe (needs nvcc and a GPU)."""
    import tempfile
    nvcc = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "int_issue_probe")
        subprocess.check_call([nvcc if os.path.exists(nvcc) else "nvcc", "-O3", "-gencode",
                               "arch=compute_103a,code=sm_103a", "-o", exe, PROBE_SRC])
        return subprocess.call([exe])


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--config", type=int, default=3, choices=(1, 2, 3, 4, 5, 6))
    ap.add_argument("--no-extra", dest="extra", action="store_false",
                    help="config 3 only: skip the extra line for the 64x64 workload (config 5)")
    ap.add_argument("--single-step", action="store_true",
                    help="time av_step (one launch per step, obs / reward / done written) on the"
                         " workload's shape instead of fused rollouts")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="run a smaller case of the workload (profiling): this many envs")
    ap.add_argument("--fused-steps", type=int, default=0,
                    help="run a smaller case of the workload (profiling): steps per launch")
    ap.add_argument("--int-probe", action="store_true", help="measure integer issue rate and exit")
    ap.add_argument("--observe", type=int, default=0, metavar="WINDOW",
                    help="time av_observe (player-centred patches of this width) on the"
                         " 16,384-env training shape instead of a rollout")
    ap.add_argument("--variant", action="store_true",
                    help="run the rollout under variant semantics (apply once by random index,"
                         " rule r inhibits rule r + 1)")
    ap.add_argument("--mutate", action="store_true",
                    help="time av_mutate (maps and rule tables) on the 16,384-env training shape")
    args = ap.parse_args(argv)
    if args.int_probe:
        return run_int_probe()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.mutate:
        base = workload_for(3)
        if args.batch > 0:
            base = base.scaled(batch=args.batch)
        return run_mutate_reference(args, base) if args.impl == "reference" else run_mutate(args, base)
    if args.observe:
        base = workload_for(3)
        if args.batch > 0:
            base = base.scaled(batch=args.batch)
        owl = ObserveWorkload(base, args.observe)
        return run_observe_reference(args, owl) if args.impl == "reference" else run_observe(args, owl)
    wl = workload_for(args.config)
    if args.batch > 0:
        wl = wl.scaled(batch=args.batch)
    if args.fused_steps > 0 and not wl.frontier:
        wl = wl.scaled(steps=args.fused_steps)
    if wl.frontier:
        return run_search_reference(args, wl) if args.impl == "reference" else run_search(args, wl)
    if args.impl == "reference":
        return run_reference(args, wl)
    if args.single_step:
        return run_single_step(args, wl)
    return run_ours(args, wl)


if __name__ == "__main__":
    sys.exit(main())
