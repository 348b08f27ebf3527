"""CUDA path (through the C-ABI) against the CPU oracle, bit-exact.

Boards, rewards, done flags, step counters and hashes are integers, so every
comparison is exact.  Small cases compare every element; full-size workloads
(the launch configurations the benchmark times) compare every env on the
GPU side against the oracle on a sample of envs, which is exact because envs
never interact.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests import golden_io
from tests.gpu_helpers import make, sample_envs, to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()  # fail loudly if the library is missing


# ------------------------------------------------------------ fixtures
@pytest.mark.parametrize("path", golden_io.all_fixtures(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_golden_fixture_step(path):
    import paper_2407_04221_gb300 as av
    fx = golden_io.load(path)
    env = av.Env(fx.cfg_fields(), fx.rules)
    g = to_dev(fx.before[None])
    env.set_state(g, set_as_init=True)
    obs, rew, done = env.step(to_dev(np.array([fx.action], np.uint8)))
    np.testing.assert_array_equal(to_np(obs)[0], fx.after)
    assert int(rew[0]) == fx.reward
    assert int(done[0]) == fx.done
    env.sync()
    env.close()


# --------------------------------------------------------------- reset
@pytest.mark.parametrize("key", [1, 2, 3, 5])
def test_reset_matches_oracle(key):
    wl = wk.WORKLOADS[key]
    env, cfg, rules, cum = make(wl, 0)
    seed = wk.seeds(0)["reset"]
    g = to_np(env.reset(seed))
    ids = np.arange(wl.batch) if wl.batch <= 4096 else sample_envs(wl.batch, 512)
    np.testing.assert_array_equal(g[ids], oracle.reset(cfg, cum, seed, ids))
    state, t = env.get_state()
    np.testing.assert_array_equal(to_np(state), g)
    assert int(t.abs().sum()) == 0
    env.close()


# -------------------------------------------------------------- rollout
def _oracle_rollout(cfg, rules, g0, ids, n_steps, seed, t0=None, trajectory=True):
    t0 = np.zeros(len(ids), np.int32) if t0 is None else t0[ids]
    return oracle.rollout(cfg, rules, g0[ids], g0[ids], t0, n_steps, seed, env_ids=ids,
                          trajectory=trajectory)


@pytest.mark.parametrize("key,batch,steps", [(1, 1, 100), (2, 37, 80), (3, 45, 260), (4, 5, 40),
                                             (5, 3, 30)])
def test_rollout_small_full_compare(key, batch, steps):
    wl = wk.WORKLOADS[key].scaled(batch=batch)
    env, cfg, rules, cum = make(wl, key)
    s = wk.seeds(key)
    g0 = to_np(env.reset(s["reset"]))
    res = env.rollout(steps, s["actions"], trajectory=True)
    ref = _oracle_rollout(cfg, rules, g0, np.arange(batch), steps, s["actions"])
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    np.testing.assert_array_equal(to_np(res["rew_sum"]), ref["rew_sum"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(g), ref["grids"])
    np.testing.assert_array_equal(to_np(t), ref["t"])
    env.sync()
    env.close()


@pytest.mark.parametrize("key,n_sample,steps", [(2, 64, 200), (5, 6, 40), (6, 2, 10)])
def test_full_size_with_firing_rules(key, n_sample, steps):
    """The full batch and board of the 1024-env, 64 x 64 and 256 x 256
    workloads, with rule entries sparse enough (3 % present, 2 % absent per
    window cell and channel) that rules match and boards change on most steps:
    the workloads' own random rules almost never match, so this is the
    full-size check of the match and apply path on those launch shapes (the
    memoising, block and band kernels)."""
    wl = wk.WORKLOADS[key].scaled(p_present=0.03, p_absent=0.02)
    env, cfg, rules, cum = make(wl, 7)
    s = wk.seeds(7)
    g0 = to_np(env.reset(s["reset"]))
    ids = sample_envs(wl.batch, n_sample, seed=key + 10)
    res = env.rollout(steps, s["actions"], trajectory=True)
    ref = _oracle_rollout(cfg, rules, g0, ids, steps, s["actions"], trajectory=True)
    idt = torch.from_numpy(ids).cuda()
    np.testing.assert_array_equal(to_np(res["obs"].index_select(1, idt)), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"].index_select(1, idt)), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"].index_select(1, idt)), ref["done"])
    np.testing.assert_array_equal(to_np(res["rew_sum"])[ids], ref["rew_sum"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(g)[ids], ref["grids"])
    np.testing.assert_array_equal(to_np(t)[ids], ref["t"])
    prev = np.concatenate([g0[ids][None], ref["obs"][:-1]], 0)
    assert (ref["obs"] != prev).reshape(steps, len(ids), -1).any(-1).mean() > 0.5  # boards change
    assert (ref["rew"] != 0).mean() > 0.5  # and matches pay
    env.sync()
    env.close()


@pytest.mark.parametrize("key,n_sample", [(2, 96), (3, 24), (5, 6)])
def test_rollout_full_size_sampled(key, n_sample):
    """The benchmark's launch configuration: full batch, full fused length."""
    wl = wk.WORKLOADS[key]
    env, cfg, rules, cum = make(wl, 0)
    s = wk.seeds(0)
    g0 = to_np(env.reset(s["reset"]))
    ids = sample_envs(wl.batch, n_sample, seed=key)
    res = env.rollout(wl.steps, s["actions"], trajectory=wl.trajectory)
    ref = _oracle_rollout(cfg, rules, g0, ids, wl.steps, s["actions"], trajectory=wl.trajectory)
    np.testing.assert_array_equal(to_np(res["rew_sum"])[ids], ref["rew_sum"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(g)[ids], ref["grids"])
    np.testing.assert_array_equal(to_np(t)[ids], ref["t"])
    if wl.trajectory:
        idt = torch.from_numpy(ids).cuda()
        np.testing.assert_array_equal(to_np(res["obs"].index_select(1, idt)), ref["obs"])
        np.testing.assert_array_equal(to_np(res["rew"].index_select(1, idt)), ref["rew"])
        np.testing.assert_array_equal(to_np(res["done"].index_select(1, idt)), ref["done"])
        assert ref["done"].any()  # auto-reset is exercised
    env.sync()
    env.close()


def test_rollout_continues_across_calls():
    wl = wk.WORKLOADS[3].scaled(batch=20)
    env, cfg, rules, cum = make(wl, 9)
    g0 = to_np(env.reset(109))
    a = env.rollout(150, 7)
    b = env.rollout(150, 8)
    ids = np.arange(20)
    r1 = _oracle_rollout(cfg, rules, g0, ids, 150, 7, trajectory=False)
    r2 = oracle.rollout(cfg, rules, r1["grids"], g0, r1["t"], 150, 8, trajectory=False)
    np.testing.assert_array_equal(to_np(a["rew_sum"]), r1["rew_sum"])
    np.testing.assert_array_equal(to_np(b["rew_sum"]), r2["rew_sum"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(g), r2["grids"])
    np.testing.assert_array_equal(to_np(t), r2["t"])
    env.close()


# ----------------------------------------------------------------- step
@pytest.mark.parametrize("key", [2, 3, 5])
def test_step_random_actions(key):
    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[key].scaled(batch=33 if key != 5 else 4, max_steps=6, auto_reset=1)
    env, cfg, rules, cum = make(wl, 3)
    # one warp per environment for 16 x 16 boards, the block kernel for 64 x 64
    assert av.av_step_path(env.h) == (av.AV_PATH_BLOCK if key == 5 else av.AV_PATH_STEP)
    g0 = to_np(env.reset(77))
    rng = np.random.default_rng(key)
    cur, t = g0.copy(), np.zeros(wl.batch, np.int32)
    for _ in range(9):
        acts = rng.integers(0, 5, wl.batch).astype(np.uint8)
        obs, rew, done = env.step(to_dev(acts))
        cur, t, erew, edone = oracle.step(cfg, rules, cur, g0, t, acts)
        np.testing.assert_array_equal(to_np(obs), cur)
        np.testing.assert_array_equal(to_np(rew), erew)
        np.testing.assert_array_equal(to_np(done), edone)
    assert av.av_warnings(env.h) == 0
    acts = np.full(wl.batch, 7, np.uint8)  # out of range -> no-op, warning bit
    obs, rew, done = env.step(to_dev(acts))
    cur2, t2, erew, edone = oracle.step(cfg, rules, cur, g0, t, acts)
    np.testing.assert_array_equal(to_np(obs), cur2)
    assert av.av_warnings(env.h) == av.AV_WARN_ACTION
    env.close()


# --------------------------------------------------------------- edges
@pytest.mark.parametrize("H,W,C,shapes,R", [
    (1, 1, 1, ((1, 1),), 2),
    (3, 5, 2, ((1, 2), (2, 3)), 3),
    (7, 9, 3, ((3, 3), (5, 5), (1, 4)), 4),      # ragged: 63 cells; rules wider than the board
    (5, 5, 16, ((5, 5), (4, 2)), 2),            # uint16 cells, 17 channels
    (64, 3, 5, ((3, 3), (2, 5)), 3),            # tall and thin
    (2, 64, 9, ((1, 5), (2, 2)), 3),            # short and wide, 2-byte cells
    (33, 33, 8, ((5, 5), (3, 1)), 5),           # rows straddle 32-bit words
    (64, 64, 4, ((5, 5),), 1),
    (64, 64, 16, ((5, 5), (3, 3), (1, 2)), 64),  # the largest board, channels and rules in one CTA
])
def test_edge_shapes(H, W, C, shapes, R):
    wl = wk.Workload(0, "edge", 3, H, W, C, R, shapes, 0.12, 0.08, 0.2, 0.2, -2, 2,
                     steps=12, max_steps=5, auto_reset=1)
    _, rules, _ = wk.make(wl, 5)
    g0 = wk.random_grids(3, 3, H, W, C, density=0.4)
    if C > 2:
        g0[:, H // 2, W // 2] |= 1 << 2
    env, cfg, _, _ = make(wl, 0, rules=rules, cum=None)
    env.set_state(to_dev(g0), set_as_init=True)
    res = env.rollout(12, 99, trajectory=True)
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(3), 12, 99, trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    env.close()


@pytest.mark.parametrize("H,W,C,shapes,R,per_env", [
    (1, 1, 1, ((1, 1),), 2, 1),
    (3, 5, 2, ((1, 2), (2, 3)), 3, 1),
    (7, 9, 3, ((3, 3), (5, 5), (1, 4)), 4, 0),   # ragged, rules wider than the board, one shared table
    (5, 5, 16, ((5, 5), (4, 2)), 2, 1),          # two-byte cells, 17 channels
    (20, 21, 5, ((3, 3), (2, 5)), 6, 1),         # 420 cells: two anchor words per lane
    (16, 32, 10, ((3, 3), (1, 3)), 12, 1),       # 512 cells, the largest board of the one-warp step
    (2, 64, 9, ((1, 5), (2, 2)), 3, 0),
    (16, 16, 4, ((3, 3),), 0, 1),                # no rules
])
def test_step_edge_shapes(H, W, C, shapes, R, per_env):
    """av_step on its one-warp kernel over ragged and edge board shapes, one and
    two anchor words per lane, shared and per-environment tables, no rules:
    six steps of random actions with auto-reset, against the oracle."""
    import paper_2407_04221_gb300 as av
    n = 19
    wl = wk.Workload(0, "edge-step", n, H, W, C, R, shapes, 0.1, 0.06, 0.2, 0.2, -2, 2,
                     max_steps=4, auto_reset=1, rules_per_env=per_env)
    _, rules, _ = wk.make(wl, 6)
    g0 = wk.random_grids(11, n, H, W, C, density=0.4)
    if C > 2:
        g0[:, H // 2, W // 2] |= 1 << 2
    env, cfg, _, _ = make(wl, 0, rules=rules, cum=None)
    assert av.av_step_path(env.h) == av.AV_PATH_STEP
    env.set_state(to_dev(g0), set_as_init=True)
    cur, t = g0.copy(), np.zeros(n, np.int32)
    rng = np.random.default_rng(H * 100 + W)
    for _ in range(6):
        acts = rng.integers(0, 5, n).astype(np.uint8)
        obs, rew, done = env.step(to_dev(acts))
        cur, t, erew, edone = oracle.step(cfg, rules, cur, g0, t, acts)
        np.testing.assert_array_equal(to_np(obs), cur)
        np.testing.assert_array_equal(to_np(rew), erew)
        np.testing.assert_array_equal(to_np(done), edone)
    g, tt = env.get_state()
    np.testing.assert_array_equal(to_np(g), cur)
    np.testing.assert_array_equal(to_np(tt), t)
    env.close()


def test_shared_rules_and_zero_rules():
    wl = wk.WORKLOADS[1].scaled(batch=40)  # one shared table, 40 envs
    env, cfg, rules, cum = make(wl, 2)
    g0 = to_np(env.reset(5))
    res = env.rollout(50, 6, trajectory=True)
    ref = _oracle_rollout(cfg, rules, g0, np.arange(40), 50, 6)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    env.close()
    wl0 = wl.scaled(n_rules=0)
    env0, cfg0, _, _ = make(wl0, 0, rules=wk.empty_rules(1, 0), cum=cum)
    g0 = to_np(env0.reset(5))
    res = env0.rollout(5, 6, trajectory=True)
    assert (to_np(res["obs"]) == g0[None]).all() and int(res["rew_sum"].abs().sum()) == 0
    env0.close()


def test_dense_matches_stress_apply():
    """Rules with few terms match almost everywhere: many atomics per step."""
    wl = wk.Workload(0, "dense", 16, 16, 16, 4, 6, ((1, 1), (2, 2), (3, 3)), 0.03, 0.03, 0.3,
                     0.3, -3, 3, steps=20)
    _, rules, _ = wk.make(wl, 8)
    g0 = wk.random_grids(4, 16, 16, 16, 4, density=0.5)
    env, cfg, _, _ = make(wl, 0, rules=rules)
    env.set_state(to_dev(g0), set_as_init=True)
    res = env.rollout(20, 3, trajectory=True)
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(16), 20, 3, trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    assert np.abs(ref["rew"]).sum() > 1000
    env.close()


# ------------------------------------------------- both kernel paths
_PATH_IDS = {"block": 1, "fast": 2, "fast8": 2, "warp": 3, "memo": 6}

@pytest.mark.parametrize("path", ["block", "fast", "fast8", "warp", "memo"])
@pytest.mark.parametrize("key,batch,steps", [(1, 3, 60), (2, 9, 70), (3, 7, 230), (4, 4, 30)])
def test_both_kernel_paths_rollout(monkeypatch, path, key, batch, steps):
    import paper_2407_04221_gb300 as av
    monkeypatch.setenv("AV_KERNEL_PATH", path.rstrip("8"))
    if path.endswith("8"):
        monkeypatch.setenv("AV_FAST_WARPS", "8")
    wl = wk.WORKLOADS[key].scaled(batch=batch)
    env, cfg, rules, cum = make(wl, 11 + key)
    assert av.av_rollout_path(env.h) == _PATH_IDS[path]
    s = wk.seeds(11 + key)
    g0 = to_np(env.reset(s["reset"]))
    res = env.rollout(steps, s["actions"], trajectory=True)
    ref = _oracle_rollout(cfg, rules, g0, np.arange(batch), steps, s["actions"])
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(t), ref["t"])
    env.close()


@pytest.mark.parametrize("path", ["block", "fast", "fast8", "warp", "memo"])
@pytest.mark.parametrize("H,W,C,shapes,R", [
    (1, 1, 1, ((1, 1),), 2),
    (7, 9, 3, ((3, 3), (5, 5), (1, 4)), 4),
    (5, 5, 16, ((5, 5), (4, 2)), 2),
    (2, 64, 9, ((1, 5), (2, 2)), 3),
    (20, 21, 6, ((3, 3), (2, 4)), 9),  # 420 cells: two anchor words per lane
    (16, 16, 5, ((1, 1), (1, 2)), 40),  # many rules: several per warp
    (16, 16, 5, ((1, 1), (1, 2)), 16),  # the most rules one warp per environment holds
    (12, 16, 4, ((2, 2), (1, 3)), 11),
    (16, 16, 8, ((3, 3), (1, 2), (5, 5)), 64),  # the most rules a table holds
])
def test_both_kernel_paths_edges(monkeypatch, path, H, W, C, shapes, R):
    import paper_2407_04221_gb300 as av
    monkeypatch.setenv("AV_KERNEL_PATH", path.rstrip("8"))
    if path.endswith("8"):
        monkeypatch.setenv("AV_FAST_WARPS", "8")
    wl = wk.Workload(0, "edge", 5, H, W, C, R, shapes, 0.1, 0.06, 0.2, 0.2, -2, 2,
                     steps=15, max_steps=6, auto_reset=1)
    _, rules, _ = wk.make(wl, 21)
    g0 = wk.random_grids(9, 5, H, W, C, density=0.45)
    if C > 2:
        g0[:, H // 2, W // 2] |= 1 << 2
    env, cfg, _, _ = make(wl, 0, rules=rules, cum=None)
    # one warp per environment holds at most 16 rules; beyond that the fast kernel runs
    want = av.AV_PATH_FAST if path == "warp" and R > 16 else _PATH_IDS[path]
    assert av.av_rollout_path(env.h) == want
    env.set_state(to_dev(g0), set_as_init=True)
    res = env.rollout(15, 123, trajectory=True)
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(5), 15, 123, trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    env.close()


# ------------------------------------- launch lengths around the action ring
@pytest.mark.parametrize("path", ["block", "fast", "warp", "memo"])
def test_launch_lengths_and_continuation(monkeypatch, path):
    """Rollouts of 0 and 1 steps, lengths around the 128-step refill of the
    pre-drawn actions, and launches that continue one another, each compared
    with the oracle run for the total length (trajectories and auto-reset on,
    so resets fall inside and across launches)."""
    import paper_2407_04221_gb300 as av
    monkeypatch.setenv("AV_KERNEL_PATH", path)
    wl = wk.WORKLOADS[3].scaled(batch=6, max_steps=37)
    env, cfg, rules, cum = make(wl, 31)
    assert av.av_rollout_path(env.h) == _PATH_IDS[path]
    s = wk.seeds(31)
    g0 = to_np(env.reset(s["reset"]))
    ids = np.arange(wl.batch)
    lengths = [0, 1, 127, 128, 129, 255, 257]
    t0 = np.zeros(wl.batch, np.int32)
    g = g0
    for n, seed in zip(lengths, range(900, 900 + len(lengths))):
        res = env.rollout(n, seed, trajectory=True)
        ref = oracle.rollout(cfg, rules, g, g0, t0, n, seed, env_ids=ids, trajectory=True)
        if n:
            np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
            np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
            np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
        got, t = env.get_state()
        np.testing.assert_array_equal(to_np(got), ref["grids"])
        np.testing.assert_array_equal(to_np(t), ref["t"])
        g, t0 = ref["grids"], ref["t"]
    env.close()


def test_destroyed_handle_is_refused():
    """After av_destroy every call on the handle returns AV_ESTATE (the handle
    is not alive any more), a second av_destroy included."""
    import ctypes

    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[2].scaled(batch=4)
    env, cfg, rules, cum = make(wl, 0)
    env.reset(5)
    h = env.h
    lib = av.load()
    assert lib.av_destroy(h) == av.AV_OK
    env.h = None
    acts = to_dev(np.zeros(4, np.uint8))
    assert lib.av_step(h, ctypes.c_void_p(acts.data_ptr()), None, None, None, 0) == av.AV_ESTATE
    assert lib.av_rollout(h, 3, 1, None, None, None, None, 0) == av.AV_ESTATE
    assert lib.av_sync(h) == av.AV_ESTATE
    assert lib.av_destroy(h) == av.AV_ESTATE
