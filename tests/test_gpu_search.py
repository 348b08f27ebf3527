"""Tree-search expansion and greedy best-first selection: CUDA path vs oracle.

Parents come from oracle rollouts (never from the CUDA path).  Children,
rewards, done flags and FNV-1a hashes are compared exactly; the search loop is
compared on its final frontier (size, boards, cumulative rewards, hashes,
liveness) and per-iteration traces.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests.gpu_helpers import make, sample_envs, to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _parents(wl, cfg, rules, cum, F, seed):
    ids = np.arange(wl.batch)
    g0 = oracle.reset(cfg, cum, seed, ids)
    res = oracle.rollout(cfg, rules, g0, g0, np.zeros(wl.batch), F, seed + 1, trajectory=True)
    return np.ascontiguousarray(res["obs"].transpose(1, 0, 2, 3))  # [B, F, H, W]


@pytest.mark.parametrize("key,batch,F", [(4, 64, 256), (3, 6, 17), (5, 2, 3)])
def test_expand_matches_oracle(key, batch, F):
    wl = wk.WORKLOADS[key].scaled(batch=batch)
    env, cfg, rules, cum = make(wl, 1)
    parents = _parents(wl, cfg, rules, cum, F, 41)
    ch, rew, done, hsh = env.expand(to_dev(parents))
    ech, erew, edone, ehsh = oracle.expand(cfg, rules, parents)
    np.testing.assert_array_equal(to_np(ch), ech)
    np.testing.assert_array_equal(to_np(rew), erew)
    np.testing.assert_array_equal(to_np(done), edone)
    np.testing.assert_array_equal(to_np(hsh, "hash"), ehsh)
    env.sync()
    env.close()


def test_expand_skips_parents_beyond_count():
    wl = wk.WORKLOADS[4].scaled(batch=4)
    env, cfg, rules, cum = make(wl, 2)
    parents = _parents(wl, cfg, rules, cum, 8, 5)
    n_parent = np.array([0, 3, 8, 1], np.int32)
    ch, rew, done, hsh = env.expand(to_dev(parents), to_dev(n_parent))
    ech, erew, edone, ehsh = oracle.expand(cfg, rules, parents)
    rew, hsh = to_np(rew), to_np(hsh, "hash")
    for b in range(4):
        n = n_parent[b]
        np.testing.assert_array_equal(rew[b, :n], erew[b, :n])
        np.testing.assert_array_equal(hsh[b, :n], ehsh[b, :n])
        assert (hsh[b, n:] == 0).all()  # untouched (zero-initialised) slots
    env.close()


def _compare_search(gpu, ref, ids):
    n = to_np(gpu["n"])[ids]
    np.testing.assert_array_equal(n, ref["n"])
    tn = to_np(gpu["trace_n"])[ids]
    np.testing.assert_array_equal(tn, ref["trace_n"])
    tb = to_np(gpu["trace_best"])[ids]
    np.testing.assert_array_equal(np.where(tn > 0, tb, 0), np.where(tn > 0, ref["trace_best"], 0))
    cum, hsh = to_np(gpu["cum"])[ids], to_np(gpu["hash"], "hash")[ids]
    live, grids = to_np(gpu["live"])[ids], to_np(gpu["grids"])[ids]
    for i in range(len(ids)):
        m = n[i]
        np.testing.assert_array_equal(cum[i, :m], ref["cum"][i, :m])
        np.testing.assert_array_equal(hsh[i, :m], ref["hash"][i, :m])
        np.testing.assert_array_equal(live[i, :m], 1 - ref["done"][i, :m])
        np.testing.assert_array_equal(grids[i, :m], ref["grids"][i, :m])


@pytest.mark.parametrize("batch,k,iters", [(6, 16, 12), (3, 40, 8)])
def test_search_small_full_compare(batch, k, iters):
    wl = wk.WORKLOADS[4].scaled(batch=batch)
    env, cfg, rules, cum = make(wl, 3, search_capacity=1 + k * iters)
    roots = env.reset(wk.seeds(3)["reset"])
    gpu = env.search(roots, iters, k)
    ref = oracle.search(cfg, rules, to_np(roots), iters, k)
    _compare_search(gpu, ref, np.arange(batch))
    env.sync()
    env.close()


def test_search_full_size_sampled():
    wl = wk.WORKLOADS[4]
    k, iters = wl.frontier, wl.iterations
    env, cfg, rules, cum = make(wl, 0, search_capacity=1 + k * iters)
    roots = env.reset(wk.seeds(0)["reset"])
    gpu = env.search(roots, iters, k)
    ids = sample_envs(wl.batch, 4, seed=4)
    ref = oracle.search(cfg, rules, to_np(roots)[ids], iters, k, env_ids=ids)
    _compare_search(gpu, ref, ids)
    assert (to_np(gpu["trace_n"])[:, 0] > 0).any()
    env.sync()
    env.close()


def _maze(batch, capacity):
    """The paper's base maze game (Sec. 2.2.1): move and eat rules, an open
    16x16 board with border walls, one player and one food tile per env."""
    from tests import golden_io
    import paper_2407_04221_gb300 as av
    fx = golden_io.load(golden_io.GOLDEN_DIR + "/03_eat_food.txt")
    fields = dict(fx.cfg_fields(), batch=batch, H=16, W=16)
    env = av.Env(fields, fx.rules, search_capacity=capacity)
    g = np.full((batch, 16, 16), 1, np.uint8)  # floor
    g[:, 0, :] = g[:, -1, :] = g[:, :, 0] = g[:, :, -1] = 2  # walls
    for b in range(batch):
        g[b, 2 + b % 5, 3] |= 4  # player
        g[b, 11, 12 - b % 7] = 8  # food
    return env, oracle.make_cfg(**fields), fx.rules, g


def test_search_maze_reaches_food():
    env, cfg, rules, g = _maze(7, 1 + 12 * 64)
    roots = to_dev(g)
    gpu = env.search(roots, 12, 64)
    ref = oracle.search(cfg, rules, g, 12, 64)
    _compare_search(gpu, ref, np.arange(7))
    assert (ref["trace_best"].max(axis=1) == 1).any()  # some beam eats the food
    env.close()


def test_visited_overflow_reports_device_error():
    import paper_2407_04221_gb300 as av
    env, cfg, rules, g = _maze(2, 10)  # far too small: 1 + 4 + 8 > 10 after two rounds
    env.search(to_dev(g), 4, 8)
    with pytest.raises(av.AvError) as ei:
        env.sync()
    assert ei.value.status == av.AV_EDEVICE
    env.sync()  # the status is cleared once reported
    env.close()


@pytest.mark.parametrize("path", ["block", "default"])
def test_expand_both_kernel_paths(monkeypatch, path):
    monkeypatch.setenv("AV_KERNEL_PATH", path)
    wl = wk.WORKLOADS[3].scaled(batch=5)
    env, cfg, rules, cum = make(wl, 6)
    parents = _parents(wl, cfg, rules, cum, 11, 17)
    ch, rew, done, hsh = env.expand(to_dev(parents))
    ech, erew, edone, ehsh = oracle.expand(cfg, rules, parents)
    np.testing.assert_array_equal(to_np(ch), ech)
    np.testing.assert_array_equal(to_np(rew), erew)
    np.testing.assert_array_equal(to_np(done), edone)
    np.testing.assert_array_equal(to_np(hsh, "hash"), ehsh)
    env.close()
