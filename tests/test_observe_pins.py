"""Pins of the oracle's policy observation (Sec. 3.2; Sec. 4, Tables 1 and 2):
hand-worked fixtures, an independent numpy formulation (pad the board with
zeros, slice the window), the full-board window, and the rule encoding decoded
back into its records."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests import golden_obs


def _bits(cells: np.ndarray, C: int) -> np.ndarray:
    """Cell words [..] -> channel bytes [.., C] (byte c = bit c)."""
    return ((cells.astype(np.int64)[..., None] >> np.arange(C)) & 1).astype(np.uint8)


@pytest.mark.parametrize("path", golden_obs.patch_fixtures(), ids=lambda p: p.split("/")[-1])
def test_patch_fixture(path):
    fx = golden_obs.load_patch(path)
    cfg = oracle.make_cfg(**fx.cfg_fields())
    obs, pyx = oracle.observe(cfg, fx.board[None], fx.window)
    assert fx.cite
    assert tuple(pyx[0]) == fx.player
    np.testing.assert_array_equal(obs[0], _bits(fx.patch, fx.C))


def numpy_patch(board: np.ndarray, C: int, ch_player: int, window: int) -> np.ndarray:
    """The patch by library routines: channel bytes, np.pad by `window` zeros
    on every side, then a slice starting window/2 before the first player."""
    bits = _bits(board, C)
    players = np.argwhere(bits[..., ch_player])  # row-major order
    if len(players) == 0:
        return np.zeros((window, window, C), np.uint8)
    py, px = players[0]
    padded = np.pad(bits, ((window, window), (window, window), (0, 0)))
    top, left = py - window // 2 + window, px - window // 2 + window
    return padded[top:top + window, left:left + window]


@pytest.mark.parametrize("H,W,C", [(16, 16, 8), (16, 16, 10), (7, 9, 4), (1, 1, 1), (64, 3, 16),
                                   (2, 64, 5), (33, 33, 12)])
def test_patch_against_numpy_padding(H, W, C):
    rng = np.random.default_rng(H * 1000 + W * 10 + C)
    ch_player = C // 2
    cfg = oracle.make_cfg(batch=1, H=H, W=W, C=C, n_rules=0, rules_per_env=0, max_steps=0,
                          auto_reset=0, ch_player=ch_player, ch_goal=-1, ch_empty=-1, ch_wall=-1,
                          border_wall=0, cum_per_env=0)
    n = 12
    boards = rng.integers(0, 1 << C, size=(n, H, W)).astype(oracle.cell_dtype(C))
    boards &= ~np.array(1 << ch_player, boards.dtype)
    for b in range(n):  # 0, 1 or 2 players
        for _ in range(b % 3):
            boards[b, rng.integers(H), rng.integers(W)] |= 1 << ch_player
    for window in (1, 2, 3, 4, 5, 10, 20, 31, 32, 127):
        obs, pyx = oracle.observe(cfg, boards, window)
        for b in range(n):
            np.testing.assert_array_equal(obs[b], numpy_patch(boards[b], C, ch_player, window),
                                          err_msg=f"board {b} window {window}")
            players = np.argwhere((boards[b] >> ch_player) & 1)
            want = tuple(players[0]) if len(players) else (-1, -1)
            assert tuple(pyx[b]) == want


def test_full_width_window_holds_the_whole_board():
    """A patch 2*16 - 1 = 31 wide (Table 1's largest) holds every cell of a
    16 x 16 board exactly once, at (15 - py + y, 15 - px + x), whatever the
    player's position."""
    H = W = 16
    C = 8
    wl = wk.WORKLOADS[2].scaled(batch=32)
    _, _, cum = wk.make(wl, 0)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    boards = oracle.reset(cfg, cum, 100, range(32))
    obs, pyx = oracle.observe(cfg, boards, 31)
    for b in range(32):
        py, px = pyx[b]
        assert boards[b, py, px] & (1 << wk.CH_PLAYER)
        assert int(obs[b].sum()) == int(_bits(boards[b], C).sum())
        np.testing.assert_array_equal(obs[b, 15 - py:15 - py + H, 15 - px:15 - px + W],
                                      _bits(boards[b], C))


@pytest.mark.parametrize("path", golden_obs.rule_fixtures(), ids=lambda p: p.split("/")[-1])
def test_rule_fixture(path):
    fx = golden_obs.load_rules(path)
    assert fx.cite
    cfg = oracle.make_cfg(batch=1, H=4, W=4, C=fx.C, n_rules=fx.rules.shape[1], rules_per_env=0,
                          max_steps=0, auto_reset=0, ch_player=-1, ch_goal=-1, ch_empty=-1,
                          ch_wall=-1, border_wall=0, cum_per_env=0)
    bits, rew = oracle.rule_obs(cfg, fx.rules)
    np.testing.assert_array_equal(bits, fx.bits)
    np.testing.assert_array_equal(rew, fx.rewards)


@pytest.mark.parametrize("key", [3, 5])
def test_rule_encoding_decodes_to_the_records(key):
    """Reading the planes back as bit masks gives the records' present,
    absent, set and clear words at every entry, and zeros outside h x w."""
    wl = wk.WORKLOADS[key].scaled(batch=6)
    _, rules, _ = wk.make(wl, 1)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    bits, rew = oracle.rule_obs(cfg, rules)
    NCH = wl.C + 1
    weights = (1 << np.arange(NCH)).astype(np.int64)
    masks = (bits.astype(np.int64) * weights).sum(-1)  # [T, R, 4, 5, 5]
    np.testing.assert_array_equal(rew, rules["reward"])
    for t in range(rules.shape[0]):
        for r in range(rules.shape[1]):
            rec = rules[t, r]
            h, w = int(rec["h"]), int(rec["w"])
            for p, field in enumerate(golden_obs.PLANES):
                frame = np.zeros((5, 5), np.int64)
                frame[:h, :w] = rec[field][:h * w].reshape(h, w)
                np.testing.assert_array_equal(masks[t, r, p], frame)
