"""Every 3 x 3 board with two tile channels, through every step kernel.

All 4^9 = 262,144 boards of a 3 x 3 grid whose cells hold any subset of two
tile channels (channel 0 the player, channel 1 the goal), each stepped with
each of the five actions by `av_step` on every kernel (the one-warp step
kernel that `av_step` takes by default, and every rollout kernel forced by
AV_KERNEL_PATH), compared with
the oracle element by element: boards, rewards and done flags.  The rule
tables are the ones whose oracle step is pinned against the convolution
formulation of Sec. 2.1 (Eq. 1 and Eq. 3) on the same enumeration in
`test_oracle_pins.py`: patterns of 1 x 1 up to 3 x 3 with dense present and
absent entries, so matches, conflicting writes, rotations and the VALID
anchors at every edge of the board occur in large numbers.  The variant
kernels run under a neutral variant (every rule limited to 255 applications
per step, more than a 3 x 3 board can hold), which takes them without
changing the result.
"""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests.gpu_helpers import to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

PATHS = ["step", "block", "fast", "fast8", "warp", "memo", "variant-warp", "variant-block"]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()


def _all_3x3_boards_c2():
    vals = np.arange(4 ** 9, dtype=np.int64)
    digits = (vals[:, None] // (4 ** np.arange(9))[None, :]) % 4
    return digits.reshape(-1, 3, 3).astype(np.uint8)


_EXPECTED = {}


def _expected(rule_seed):
    """Oracle results for every board and action (computed once per table)."""
    if rule_seed not in _EXPECTED:
        boards = _all_3x3_boards_c2()
        wl, fields = _workload()
        rules = wk.make_rules(wl, rule_seed)
        cfg = oracle.make_cfg(**fields)
        n = len(boards)
        per_action = []
        for a in range(5):
            acts = np.full(n, a, np.uint8)
            got, _, rew, done = oracle.step(cfg, rules, boards, boards, np.zeros(n, np.int32), acts)
            per_action.append((got, rew, done))
        _EXPECTED[rule_seed] = (boards, rules, fields, per_action)
    return _EXPECTED[rule_seed]


def _workload():
    wl = wk.Workload(0, "bf", 1, 3, 3, 2, 4, ((1, 1), (1, 2), (2, 2), (2, 3), (3, 3)),
                     0.25, 0.2, 0.25, 0.25, -3, 3, rules_per_env=0)
    fields = dict(batch=4 ** 9, H=3, W=3, C=2, n_rules=4, rules_per_env=0, max_steps=0,
                  auto_reset=0, ch_player=0, ch_goal=1, ch_empty=-1, ch_wall=-1, border_wall=0,
                  cum_per_env=0)
    return wl, fields


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("rule_seed", [11, 12])
def test_every_3x3_board_every_action(monkeypatch, path, rule_seed):
    import paper_2407_04221_gb300 as av
    boards, rules, fields, per_action = _expected(rule_seed)
    kernel = path.split("-")[-1]
    if kernel != "step":
        monkeypatch.setenv("AV_KERNEL_PATH", kernel.rstrip("8"))
    if kernel.endswith("8"):
        monkeypatch.setenv("AV_FAST_WARPS", "8")
    env = av.Env(fields, rules)
    if kernel == "step":
        assert av.av_step_path(env.h) == av.AV_PATH_STEP
    elif path.startswith("variant"):
        av.av_set_variant(env.h, random_keys=0, limit=[255] * 4, inhibit=[0] * 4)
        assert av.av_rollout_path(env.h) == av.AV_PATH_VARIANT
    else:
        want = {"block": av.AV_PATH_BLOCK, "fast": av.AV_PATH_FAST, "fast8": av.AV_PATH_FAST,
                "warp": av.AV_PATH_WARP, "memo": av.AV_PATH_MEMO}[kernel]
        assert av.av_rollout_path(env.h) == want
    n = len(boards)
    dev_boards = to_dev(boards)
    for a in range(5):
        env.set_state(dev_boards, set_as_init=True)
        obs, rew, done = env.step(to_dev(np.full(n, a, np.uint8)))
        exp_g, exp_r, exp_d = per_action[a]
        np.testing.assert_array_equal(to_np(obs), exp_g, err_msg=f"boards, action {a}")
        np.testing.assert_array_equal(to_np(rew), exp_r, err_msg=f"rewards, action {a}")
        np.testing.assert_array_equal(to_np(done), exp_d, err_msg=f"done flags, action {a}")
    env.sync()
    env.close()


def test_enumeration_is_dense():
    """The tables really exercise the step: most boards see a match, many
    change, and rewards of both signs occur (checked on the oracle side)."""
    for seed in (11, 12):
        boards, _, _, per_action = _expected(seed)
        got, rew, _ = per_action[1]
        assert (rew != 0).mean() > 0.3
        assert (got != boards).any(axis=(1, 2)).mean() > 0.2
