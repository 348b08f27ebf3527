"""The memoising rollout's remembered outcomes, against the oracle, bit-exact.

The memoising rollout (AV_PATH_MEMO) evaluates each (board, action) pair once
and repeats the outcome while the board stays; it also keeps the board before
the current one with its outcomes, so a board that comes back is not evaluated
again.  These rollouts are built to walk every branch of that bookkeeping:
boards that oscillate between two states every step (floor and wall tiles
trading places), a player that moves on top of the oscillation (so the
oscillation's states differ with each position), boards that come back after
more than one step, goal tiles whose removal ends the episode (auto-reset to a
board that may equal the current one), and the step limit.  Every comparison
covers the observation, reward and done trajectories and the final state, for
one, two and four warps per environment, boards of one and of two plane words
per lane, one- and two-byte cells.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests.gpu_helpers import to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

E, Wl, P, G = 1 << wk.CH_EMPTY, 1 << wk.CH_WALL, 1 << wk.CH_PLAYER, 1 << wk.CH_GOAL


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()


def _rules(C, goal_eater: bool):
    """Floor and wall trade places everywhere every step (two 1x1 rules, in
    parallel: period 2); the maze game's move rule; optionally a rule that eats
    the goal tile under the player after a push (the episode then ends)."""
    n = 4 if goal_eater else 3
    r = wk.empty_rules(1, n)
    for j, (src, dst, rew) in enumerate(((E, Wl, 1), (Wl, E, -2))):
        r[0, j]["h"], r[0, j]["w"], r[0, j]["reward"] = 1, 1, rew
        r[0, j]["present"][0] = src
        r[0, j]["absent"][0] = P  # the player's cell stays floor
        r[0, j]["clear"][0], r[0, j]["set"][0] = src, dst
    r[0, 2] = wk.base_game_rules(C)[0]
    if goal_eater:
        F = 1 << C
        r[0, 3]["h"], r[0, 3]["w"], r[0, 3]["reward"] = 1, 2, 5
        r[0, 3]["present"][0], r[0, 3]["present"][1] = P | G, F
        r[0, 3]["clear"][0] = G
    return r


def _boards(n, H, W, C, seed, goals: bool):
    rng = np.random.default_rng(seed)
    dt = np.uint8 if C <= 8 else np.uint16
    g = np.where(rng.random((n, H, W)) < 0.5, E, Wl).astype(dt)
    ys, xs = rng.integers(0, H, n), rng.integers(0, W, n)
    g[np.arange(n), ys, xs] = E | P
    if goals:
        g[np.arange(n), ys, xs] |= G  # the player stands on a goal tile
    return g


def _fields(n, H, W, C, R, max_steps, auto_reset, ch_goal):
    return dict(batch=n, H=H, W=W, C=C, n_rules=R, rules_per_env=0, max_steps=max_steps,
                auto_reset=auto_reset, ch_player=wk.CH_PLAYER, ch_goal=ch_goal,
                ch_empty=wk.CH_EMPTY, ch_wall=wk.CH_WALL, border_wall=0, cum_per_env=0)


@pytest.mark.parametrize("warps", ["1", "2", "4"])
@pytest.mark.parametrize("H,W,C", [(8, 8, 4), (16, 16, 10), (20, 21, 5)])
@pytest.mark.parametrize("goals", [False, True])
def test_oscillating_boards(monkeypatch, warps, H, W, C, goals):
    import paper_2407_04221_gb300 as av
    monkeypatch.setenv("AV_MEMO_WARPS", warps)
    n, steps = 24, 150
    rules = _rules(C, goals)
    fields = _fields(n, H, W, C, rules.shape[1], 37 if goals else 0, 1 if goals else 0,
                     wk.CH_GOAL if goals else -1)
    env = av.Env(fields, rules)
    assert av.av_rollout_path(env.h) == av.AV_PATH_MEMO
    g0 = _boards(n, H, W, C, 7 + H, goals)
    env.set_state(to_dev(g0), set_as_init=True)
    res = env.rollout(steps, 31, trajectory=True)
    cfg = oracle.make_cfg(**fields)
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(n, np.int32), steps, 31, trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    np.testing.assert_array_equal(to_np(res["rew_sum"]), ref["rew_sum"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(g), ref["grids"])
    np.testing.assert_array_equal(to_np(t), ref["t"])
    # the bookkeeping was exercised: boards came back, and (with goals) episodes ended
    obs = ref["obs"]
    back = (obs[2:] == obs[:-2]).reshape(steps - 2, n, -1).all(-1) & \
        (obs[2:] != obs[1:-1]).reshape(steps - 2, n, -1).any(-1)
    assert back.mean() > 0.15
    if goals:
        assert ref["done"].any()
    env.close()


@pytest.mark.parametrize("warps", ["1", "2", "4"])
def test_training_shape_busy_envs(monkeypatch, warps):
    """The trajectory workload's environments that change their board on most
    steps (found with the oracle on 512 environments), 600 steps each."""
    import paper_2407_04221_gb300 as av
    monkeypatch.setenv("AV_MEMO_WARPS", warps)
    wl = wk.WORKLOADS[3].scaled(batch=512)
    _, rules, cum = wk.make(wl, 4)
    fields = wk.config_fields(wl)
    cfg = oracle.make_cfg(**fields)
    s = wk.seeds(4)
    ids = np.arange(512)
    g0 = oracle.reset(cfg, cum, s["reset"], ids)
    probe = oracle.rollout(cfg, rules, g0, g0, np.zeros(512, np.int32), 60, s["actions"], env_ids=ids,
                           trajectory=True)
    prev = np.concatenate([g0[None], probe["obs"][:-1]], 0)
    busy = np.argsort(-(probe["obs"] != prev).reshape(60, 512, -1).any(-1).mean(0))[:16]
    sel = np.sort(busy)
    f = dict(fields, batch=len(sel))
    env = av.Env(f, rules[sel], cum[sel] if cum.ndim == 2 else cum)
    env.set_state(to_dev(g0[sel]), set_as_init=True)
    res = env.rollout(600, 77, trajectory=True)
    cf2 = oracle.make_cfg(**f)
    ref = oracle.rollout(cf2, rules[sel], g0[sel], g0[sel], np.zeros(len(sel), np.int32), 600, 77,
                         trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    env.close()
