"""Boards larger than one CTA's shared memory (more than 4096 cells, up to
256 x 256): the band-streamed step through the C-ABI against the CPU oracle,
bit-exact -- rollouts with trajectories on square, wide, tall and ragged
boards with one- and two-byte cells, rule sets dense enough that windows and
writes cross band boundaries every step, done / auto-reset, single steps, the
256 x 256 workload, and the calls such boards do not support."""
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
    import paper_2407_04221_gb300 as av
    av.load()


# dense 5 x 5 rules: few terms per rule, so matches (and writes reaching four
# rows below their anchors) are common
DENSE = wk.WORKLOADS[5].scaled(p_present=0.03, p_absent=0.03, p_set=0.15, p_clear=0.15)

CASES = {
    "256x256-c16": (wk.WORKLOADS[6], dict(batch=3)),
    "100x70-c10-reset": (wk.WORKLOADS[3], dict(batch=5, H=100, W=70)),
    "65x65-c8": (wk.WORKLOADS[2], dict(batch=4, H=65, W=65)),
    "256x17-c10": (wk.WORKLOADS[3], dict(batch=3, H=256, W=17)),
    "17x256-c16-dense": (DENSE, dict(batch=3, H=17, W=256)),
    "96x96-c16-dense": (DENSE, dict(batch=3, H=96, W=96)),
    "200x33-c8": (wk.WORKLOADS[2], dict(batch=4, H=200, W=33)),
    "256x256-c16-r64-dense": (DENSE, dict(batch=2, H=256, W=256, n_rules=64)),  # every limit at once
}


def _one_channel_rules():
    """Two hand-made rules on one tile channel: a lit cell goes dark, and a
    dark cell left of a lit one lights up (both every step, in parallel)."""
    r = wk.empty_rules(1, 2)
    r[0, 0]["h"], r[0, 0]["w"], r[0, 0]["reward"] = 1, 1, 1
    r[0, 0]["present"][0], r[0, 0]["clear"][0] = 1, 1
    r[0, 1]["h"], r[0, 1]["w"], r[0, 1]["reward"] = 1, 2, -1
    r[0, 1]["absent"][0], r[0, 1]["present"][1], r[0, 1]["set"][0] = 1, 1, 1
    return r


def test_one_channel_256x256():
    """C = 1 (no player, no goal): the smallest cell and the largest board."""
    import paper_2407_04221_gb300 as av
    fields = dict(batch=2, H=256, W=256, C=1, n_rules=2, rules_per_env=0, max_steps=0, auto_reset=0,
                  ch_player=-1, ch_goal=-1, ch_empty=-1, ch_wall=-1, border_wall=0, cum_per_env=0)
    rules = _one_channel_rules()
    g0 = wk.random_grids(4, 2, 256, 256, 1, density=0.3)
    env = av.Env(fields, rules)
    assert av.av_rollout_path(env.h) == av.AV_PATH_BAND
    env.set_state(to_dev(g0), set_as_init=True)
    res = env.rollout(10, 5, trajectory=True)
    cfg = oracle.make_cfg(**fields)
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(2, np.int32), 10, 5, trajectory=True)
    assert (ref["obs"][0] != g0).any()
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    env.close()


@pytest.mark.parametrize("case", list(CASES))
def test_rollout_with_trajectory(case):
    import paper_2407_04221_gb300 as av
    base, kw = CASES[case]
    wl = base.scaled(**kw)
    env, cfg, rules, cum = make(wl, 3)
    assert av.av_rollout_path(env.h) == av.AV_PATH_BAND
    s = wk.seeds(3)
    g0 = to_np(env.reset(s["reset"]))
    np.testing.assert_array_equal(g0, oracle.reset(cfg, cum, s["reset"], range(wl.batch)))
    steps = 12
    res = env.rollout(steps, s["actions"], trajectory=True)
    g, t = env.get_state()
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(wl.batch, np.int32), steps, s["actions"],
                         trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    np.testing.assert_array_equal(to_np(g), ref["grids"])
    np.testing.assert_array_equal(to_np(t), ref["t"])
    env.sync()
    env.close()


def test_boards_change_across_bands():
    """The dense rule set changes boards every step, near band edges too."""
    wl = DENSE.scaled(batch=2, H=96, W=96)
    _, rules, cum = wk.make(wl, 3)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    g0 = oracle.reset(cfg, cum, 103, range(2))
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(2, np.int32), 4, 203, trajectory=True)
    changed = ref["obs"][0] != g0
    assert changed.sum() > 200 and changed.any(axis=(0, 2)).sum() > 60  # many cells, most rows


def test_single_steps_and_continuation():
    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[3].scaled(batch=4, H=80, W=90, max_steps=5)
    env, cfg, rules, cum = make(wl, 4)
    g0 = to_np(env.reset(104))
    cur, t = g0.copy(), np.zeros(4, np.int32)
    rng = np.random.default_rng(0)
    for s in range(8):  # crosses max_steps: done and auto-reset
        a = rng.integers(0, 5, 4).astype(np.uint8)
        obs, rew, done = env.step(to_dev(a))
        cur, t, rew_o, done_o = oracle.step(cfg, rules, cur, g0, t, a)
        np.testing.assert_array_equal(to_np(obs), cur)
        np.testing.assert_array_equal(to_np(rew), rew_o)
        np.testing.assert_array_equal(to_np(done), done_o)
    res = env.rollout(7, 204)  # a rollout continuing from the stepped state
    g, tt = env.get_state()
    ref = oracle.rollout(cfg, rules, cur, g0, t, 7, 204)
    np.testing.assert_array_equal(to_np(g), ref["grids"])
    np.testing.assert_array_equal(to_np(tt), ref["t"])
    np.testing.assert_array_equal(to_np(res["rew_sum"]), ref["rew_sum"])
    env.close()


def test_full_workload_sampled():
    wl = wk.WORKLOADS[6]
    env, cfg, rules, cum = make(wl, 0)
    s = wk.seeds(0)
    g0 = to_np(env.reset(s["reset"]))
    res = env.rollout(wl.steps, s["actions"])
    g, _ = env.get_state()
    ids = sample_envs(wl.batch, 6, seed=2)
    ref = oracle.rollout(cfg, rules, g0[ids], g0[ids], np.zeros(len(ids), np.int32), wl.steps,
                         s["actions"], env_ids=ids)
    np.testing.assert_array_equal(to_np(g)[ids], ref["grids"])
    np.testing.assert_array_equal(to_np(res["rew_sum"])[ids], ref["rew_sum"])
    env.sync()
    env.close()


def test_unsupported_calls_on_large_boards():
    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[2].scaled(batch=2, H=65, W=65)
    env, cfg, rules, cum = make(wl, 0, search_capacity=16)
    parents = env.boards(2, 1)
    for call in (lambda: env.expand(parents),
                 lambda: av.av_search_init(env.h, env.boards(2),
                                           torch.zeros(2, dtype=torch.int64, device="cuda"),
                                           torch.zeros(2, dtype=torch.uint8, device="cuda")),
                 lambda: av.av_set_variant(env.h, limit=[1])):
        with pytest.raises(av.AvError) as ei:
            call()
        assert ei.value.status == av.AV_EINVAL
    env.close()


@pytest.mark.parametrize("H,W,C,window", [(256, 256, 16, 31), (256, 256, 10, 127), (100, 70, 8, 20),
                                          (65, 65, 3, 5)])
def test_observation_of_large_boards(H, W, C, window):
    """Boards too large to stage in shared memory are observed from global
    memory: players anywhere, none, or several."""
    import paper_2407_04221_gb300 as av
    rng = np.random.default_rng(H + W + C)
    B = 5
    boards = rng.integers(0, 1 << C, size=(B, H, W)).astype(oracle.cell_dtype(C))
    boards &= ~np.array(1 << 2, boards.dtype)
    for b in range(B):
        for _ in range(b % 3):
            boards[b, rng.integers(H), rng.integers(W)] |= 1 << 2
    fields = dict(batch=B, H=H, W=W, C=C, n_rules=0, rules_per_env=0, max_steps=0, auto_reset=0,
                  ch_player=2, ch_goal=-1, ch_empty=-1, ch_wall=-1, border_wall=0, cum_per_env=0)
    env = av.Env(fields, np.zeros(0, np.uint8))
    env.set_state(to_dev(boards))
    obs, pyx = env.observe(window)
    want, want_pyx = oracle.observe(oracle.make_cfg(**fields), boards, window)
    np.testing.assert_array_equal(to_np(obs), want)
    np.testing.assert_array_equal(to_np(pyx), want_pyx)
    env.close()


def test_remembered_steps_on_large_boards():
    """The maze game (move and eat rules) on 72 x 72 boards: a push into a wall
    leaves the board as it is (the band kernel remembers that action's outcome
    and skips the bands next time), a move or a meal changes it (everything
    remembered is dropped).  Trajectories against the oracle, bit-exact."""
    import paper_2407_04221_gb300 as av
    H = W = 72
    C, n, steps = 4, 6, 60
    rules = wk.base_game_rules(C)[None]
    fields = dict(batch=n, H=H, W=W, C=C, n_rules=2, rules_per_env=0, max_steps=25, auto_reset=1,
                  ch_player=2, ch_goal=3, ch_empty=0, ch_wall=1, border_wall=0, cum_per_env=0)
    rng = np.random.default_rng(72)
    g = np.where(rng.random((n, H, W)) < 0.3, 2, 1).astype(np.uint8)  # walls and floor
    g[:, rng.random((H, W)) < 0.02] = 8  # food
    for e in range(n):
        y, x = 10 + 7 * e, 20 + 3 * e
        g[e, y, x] = 1 | 4
    env = av.Env(fields, rules)
    assert av.av_rollout_path(env.h) == av.AV_PATH_BAND
    env.set_state(to_dev(g), set_as_init=True)
    res = env.rollout(steps, 5, trajectory=True)
    cfg = oracle.make_cfg(**fields)
    ref = oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), steps, 5, trajectory=True)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    obs = ref["obs"]
    moved = (obs[1:] != obs[:-1]).reshape(steps - 1, n, -1).any(-1)
    assert 0.1 < moved.mean() < 0.95  # both kinds of step occur
    env.close()
