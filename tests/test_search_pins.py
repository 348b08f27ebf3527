"""Pins of the oracle's expansion and search (Sec. 2.2.1: the environment as
its own forward model for best-first search; equal states keep the shallower
node, and of equal states the higher reward): children equal to the pinned
standard step, hashes equal to the pinned FNV-1a of the children's bytes, and
closed forms of the search itself -- on an open floor the frontier after d
iterations is exactly the ring of cells at Manhattan distance d (breadth-first
layers), in a corridor of food the best reward after d iterations is the food
within d cells -- plus the frontier's order and distinctness."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk

E, Wl, P, G = 1 << wk.CH_EMPTY, 1 << wk.CH_WALL, 1 << wk.CH_PLAYER, 1 << wk.CH_GOAL


def _fields(B, H, W, C=4, R=2):
    return dict(batch=B, H=H, W=W, C=C, n_rules=R, rules_per_env=1, max_steps=0, auto_reset=0,
                ch_player=wk.CH_PLAYER, ch_goal=wk.CH_GOAL, ch_empty=wk.CH_EMPTY, ch_wall=wk.CH_WALL,
                border_wall=1, cum_per_env=0)


def _walled(H, W):
    g = np.full((H, W), E, np.uint8)
    g[0, :] = g[-1, :] = g[:, 0] = g[:, -1] = Wl
    return g


@pytest.mark.parametrize("key", [4, 2, 3])
def test_expand_children_are_steps_and_hashes_are_fnv(key):
    wl = wk.WORKLOADS[key].scaled(batch=4)
    _, rules, cum = wk.make(wl, 6)
    cfg = oracle.make_cfg(**dict(wk.config_fields(wl), max_steps=0, auto_reset=0))
    g0 = oracle.reset(cfg, cum, 106, range(4))
    parents = np.stack([g0, g0 | wk.random_grids(2, 4, wl.H, wl.W, wl.C, density=0.1)], axis=1)
    kids, rew, done, hsh = oracle.expand(cfg, rules, parents)
    for f in range(2):
        for a in range(5):
            out, _, r, _ = oracle.step(cfg, rules, parents[:, f], parents[:, f], np.zeros(4, np.int32),
                                       np.full(4, a, np.uint8))
            np.testing.assert_array_equal(kids[:, f, a], out)
            np.testing.assert_array_equal(rew[:, f, a], r)
            no_goal = ((out.astype(np.int64) >> wk.CH_GOAL) & 1).sum(axis=(1, 2)) == 0
            np.testing.assert_array_equal(done[:, f, a].astype(bool), no_goal)
            for b in range(4):
                assert int(hsh[b, f, a]) == oracle.fnv1a64(out[b].tobytes())


def test_open_floor_search_is_breadth_first():
    """Only the move rule, an open floor, a beam wider than any layer: the
    states are the player's cells, and iteration d keeps exactly the cells at
    Manhattan distance d from the start that no earlier iteration reached."""
    H = W = 13
    g = _walled(H, W)
    y0, x0 = 6, 4
    g[y0, x0] |= P
    g[0, 0] |= G  # a goal out of reach keeps every node live (no goal = done)
    rules = wk.empty_rules(1, 1)
    rules[0, 0] = wk.base_game_rules(4)[0]  # move
    cfg = oracle.make_cfg(**_fields(1, H, W, R=1))
    iters = 10
    res = oracle.search(cfg, rules, g[None], iters, 256)
    ys, xs = np.mgrid[1:H - 1, 1:W - 1]
    dist = np.abs(ys - y0) + np.abs(xs - x0)
    want = [int((dist == d).sum()) for d in range(1, iters + 1)]
    np.testing.assert_array_equal(res["trace_n"][0], want)
    n = int(res["n"][0])
    pos = sorted((int(np.argwhere((res["grids"][0, i] & P) != 0)[0][0]), int(np.argwhere((res["grids"][0, i] & P) != 0)[0][1]))
                 for i in range(n))
    assert pos == sorted((int(y), int(x)) for y, x in zip(ys[dist == iters], xs[dist == iters]))
    assert (res["cum"][0, :n] == 0).all()
    assert int(res["n_visited"][0]) == 1 + sum(want)


def test_food_corridor_best_reward():
    """A corridor with food at known distances right of the player: after d
    iterations the best cumulative reward in the beam is the food within d cells
    (moving onto food eats it, reward 1; Sec. 2.2.1).  Eating the last food
    ends the episode (no goal left): that node stays in the beam of its iteration
    but is not expanded, so one iteration later no node holds all the food."""
    W = 14
    g = _walled(3, W)
    g[1, 1] |= P
    food = [3, 4, 8, 12]
    for x in food:
        g[1, x] = G
    rules = wk.base_game_rules(4)[None]
    cfg = oracle.make_cfg(**_fields(1, 3, W))
    last = food[-1] - 1  # iterations to reach the last food
    res = oracle.search(cfg, rules, g[None], last, 64)
    want = [sum(1 for x in food if x - 1 <= d) for d in range(1, last + 1)]
    np.testing.assert_array_equal(res["trace_best"][0], want)
    n = int(res["n"][0])
    best = [i for i in range(n) if res["cum"][0, i] == len(food)]
    assert len(best) == 1 and res["done"][0, best[0]] == 1
    assert (res["done"][0, :n] == (res["cum"][0, :n] == len(food))).all()
    more = oracle.search(cfg, rules, g[None], last + 1, 64)
    assert more["trace_best"][0, -1] == len(food) - 1


@pytest.mark.parametrize("seed", [0, 1])
def test_frontier_sorted_distinct_and_hashed(seed):
    wl = wk.WORKLOADS[4].scaled(batch=3)
    _, rules, cum = wk.make(wl, seed)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    roots = oracle.reset(cfg, cum, 100 + seed, range(3))
    res = oracle.search(cfg, rules, roots, 12, 32)
    for b in range(3):
        n = int(res["n"][b])
        assert n > 0
        cum_b, h_b = res["cum"][b, :n], res["hash"][b, :n]
        keys = list(zip((-cum_b).tolist(), h_b.tolist()))
        assert keys == sorted(keys)          # (cum desc, hash asc)
        assert len(set(h_b.tolist())) == n   # one node per state
        for i in range(n):
            assert int(h_b[i]) == oracle.fnv1a64(res["grids"][b, i].tobytes())
