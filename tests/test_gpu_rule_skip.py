"""Rules that survive their leading present terms but whose tile terms pass
nowhere on the board are skipped by the one-warp kernels until the board
changes, and for the others only anchors that pass every tile term go on to
the remaining terms (the result is the same: only force terms change while
the board stays).  These rollouts are built so that such rules turn live
again: a rule that needs the player beside a food tile (dead until a move
brings the player there) and one with an absent force term (whose test must
ignore the force of the step it is made in).  Every path, and the variant
kernels, against the oracle, bit-exact, on a board of one plane word per lane
(with the tile masks kept in registers) and one of two (without)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests.gpu_helpers import to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

E, Wl, P, G = 1 << wk.CH_EMPTY, 1 << wk.CH_WALL, 1 << wk.CH_PLAYER, 1 << wk.CH_GOAL
C = 4
F = 1 << C
B = 48
# (H, W, copies of the three rules): 54 cells and 3 rules; 384 cells (two
# plane words per lane) and 6 rules
SHAPES = {"6x9-r3": (6, 9, 1), "16x24-r6": (16, 24, 2)}


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()


def _rules(copies):
    """Move; beside food and not pushing into it (an absent force term); beside
    a cell that is neither floor, wall nor player (food), no output.  Food is
    never eaten, so pushing into it leaves the board as it is and the force
    term alone decides the second rule.  Copies carry other rewards."""
    r = wk.empty_rules(1, 3 * copies)
    for i in range(copies):
        j = 3 * i
        r[0, j] = wk.base_game_rules(C)[0]
        r[0, j + 1]["h"], r[0, j + 1]["w"], r[0, j + 1]["reward"] = 1, 2, 3 + 10 * i
        r[0, j + 1]["present"][0], r[0, j + 1]["present"][1], r[0, j + 1]["absent"][1] = P, G, F
        r[0, j + 2]["h"], r[0, j + 2]["w"], r[0, j + 2]["reward"] = 1, 2, 2 + 10 * i
        r[0, j + 2]["present"][0], r[0, j + 2]["absent"][1] = P, E | Wl | P
    return r


def _boards(H, W, seed):
    rng = np.random.default_rng(seed)
    g = np.full((B, H, W), E, np.uint8)
    g[:, 0, :] = g[:, -1, :] = g[:, :, 0] = g[:, :, -1] = Wl
    inner = g[:, 1:-1, 1:-1]
    inner[rng.random(inner.shape) < 0.2] = G
    for b in range(B):
        ys, xs = np.nonzero(g[b] == E)
        k = rng.integers(len(ys))
        g[b, ys[k], xs[k]] |= P
    return g


def _fields(H, W, R):
    return dict(batch=B, H=H, W=W, C=C, n_rules=R, rules_per_env=0, max_steps=0, auto_reset=0,
                ch_player=wk.CH_PLAYER, ch_goal=wk.CH_GOAL, ch_empty=wk.CH_EMPTY, ch_wall=wk.CH_WALL,
                border_wall=1, cum_per_env=0)


def _check(env, shape, variant, steps=200, action_seed=11):
    H, W, copies = SHAPES[shape]
    rules, g0 = _rules(copies), _boards(H, W, 4)
    env.set_state(to_dev(g0), set_as_init=True)
    res = env.rollout(steps, action_seed, trajectory=True)
    cfg = oracle.make_cfg(**_fields(H, W, 3 * copies))
    ref = oracle.rollout(cfg, rules, g0, g0, np.zeros(B, np.int32), steps, action_seed,
                         trajectory=True, variant=variant)
    # the scenario does what it is for: rewards come and go as the player
    # moves, and the force rule is blocked in steps that change nothing
    per_env = (ref["rew"] > 0).sum(axis=0)
    assert ((per_env > 0) & (per_env < steps)).sum() > B // 2
    if variant is None and copies == 1:
        still = (ref["obs"][1:] == ref["obs"][:-1]).all(axis=(2, 3))
        assert (still & (ref["rew"][1:] == 2)).any() and (still & (ref["rew"][1:] == 5)).any()
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    g, t = env.get_state()
    np.testing.assert_array_equal(to_np(g), ref["grids"])


@pytest.mark.parametrize("shape", list(SHAPES))
@pytest.mark.parametrize("path", ["warp", "fast", "block", "memo", "default"])
def test_standard(path, shape, monkeypatch):
    import paper_2407_04221_gb300 as av
    if path != "default":
        monkeypatch.setenv("AV_KERNEL_PATH", path)
    H, W, copies = SHAPES[shape]
    env = av.Env(_fields(H, W, 3 * copies), _rules(copies))
    if path == "warp":
        assert av.av_rollout_path(env.h) == av.AV_PATH_WARP
    if path == "memo":
        assert av.av_rollout_path(env.h) == av.AV_PATH_MEMO
    _check(env, shape, None)
    env.sync()
    env.close()


@pytest.mark.parametrize("shape", list(SHAPES))
@pytest.mark.parametrize("path", ["warp", "block"])
@pytest.mark.parametrize("random_keys", [0, 1])
def test_variant(path, random_keys, shape, monkeypatch):
    import paper_2407_04221_gb300 as av
    monkeypatch.setenv("AV_KERNEL_PATH", path)
    H, W, copies = SHAPES[shape]
    R = 3 * copies
    env = av.Env(_fields(H, W, R), _rules(copies))
    limit = [(0, 1, 2)[r % 3] for r in range(R)]
    inhibit = [(1 << (r + 1)) if r % 3 == 1 else 0 for r in range(R)]
    v = dict(random_keys=random_keys, key_seed=9, limit=limit, inhibit=inhibit)
    av.av_set_variant(env.h, **v)
    assert av.av_rollout_path(env.h) == av.AV_PATH_VARIANT
    _check(env, shape, oracle.make_variant(**v))
    env.sync()
    env.close()
