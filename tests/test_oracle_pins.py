"""Pins of the CPU oracle against things other than itself.

* hand-worked one-step fixtures (tests/golden), each citing its passage;
* published test vectors of SplitMix64 and FNV-1a 64;
* brute force over every 3x3 board with two tile types, against the paper's
  convolution formulation written with torch CPU library routines
  (conv2d for the matching convolution, conv_transpose2d for the output
  write, numpy.rot90 for rotations);
* invariants: no-op rules are the identity, a single mover conserves tile
  counts, rotating the board commutes with the step, rule order does not
  matter, seeds reproduce trajectories;
* initial-map distribution checks (the initialiser is build-defined: these
  are its only pins).
"""
from __future__ import annotations

import itertools

import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

import oracle
import workload as wk
from tests import golden_io


# ----------------------------------------------------------------- fixtures
@pytest.mark.parametrize("path", golden_io.all_fixtures(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_golden_fixture(path):
    fx = golden_io.load(path)
    assert fx.cite, "every fixture cites its passage"
    cfg = oracle.make_cfg(**fx.cfg_fields())
    g = fx.before[None]
    out, t, rew, done = oracle.step(cfg, fx.rules, g, g, np.zeros(1), np.array([fx.action]))
    np.testing.assert_array_equal(out[0], fx.after)
    assert int(rew[0]) == fx.reward
    assert int(done[0]) == fx.done
    assert int(t[0]) == 1


def test_fixture_shuffled_rule_order_same():
    fx = golden_io.load(golden_io.GOLDEN_DIR + "/06_conflict.txt")
    cfg = oracle.make_cfg(**fx.cfg_fields())
    g = fx.before[None]
    perm = fx.rules[:, ::-1].copy()
    a = oracle.step(cfg, fx.rules, g, g, np.zeros(1), np.zeros(1))
    b = oracle.step(cfg, perm, g, g, np.zeros(1), np.zeros(1))
    np.testing.assert_array_equal(a[0], b[0])


# ------------------------------------------------------------ test vectors
def test_splitmix64_published_sequence():
    # splitmix64.c (Vigna): state += 0x9e3779b97f4a7c15; output = mix(state).
    # Published first outputs for seed 1234567.
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423,
              4593380528125082431, 16408922859458223821]
    x = 1234567
    got = []
    L = oracle.lib()
    for _ in range(5):
        x = (x + 0x9E3779B97F4A7C15) % (1 << 64)
        got.append(int(L.or_mix64(x)))
    assert got == expect


def test_fnv1a64_published_vectors():
    assert oracle.fnv1a64(b"") == 0xCBF29CE484222325
    assert oracle.fnv1a64(b"a") == 0xAF63DC4C8601EC8C
    assert oracle.fnv1a64(b"foobar") == 0x85944171F73967E8


def test_grid_hash_canonical_bytes():
    # 2x3 board, C=4: one byte per cell, row-major.  Bits above C are dropped.
    g = np.array([[1, 2, 4], [8, 0, 0x31]], np.uint8)
    assert oracle.grid_hash(g, 4) == oracle.fnv1a64(bytes([1, 2, 4, 8, 0, 1]))
    # C=10: two little-endian bytes per cell
    g16 = np.array([[0x0201, 0x0003]], np.uint16)
    assert oracle.grid_hash(g16, 10) == oracle.fnv1a64(bytes([1, 2, 3, 0]))


def test_draw_matches_generator_definition():
    # The generator module and the oracle implement the same published keyed
    # draw independently.
    for seed, stream, a, b, c in [(0, 1, 0, 0, 0), (7, 4, 1023, 0, 999), (2**63, 6, 5, 7, 12345)]:
        assert oracle.draw(seed, stream, a, b, c) == int(wk.draw(seed, stream, a, b, c))


# --------------------------------------------------------------- rotations
def test_rotation_matches_numpy_rot90():
    wl = wk.WORKLOADS[3]
    rules = wk.make_rules(wl, 3)
    for rec in rules[:4].reshape(-1):
        h, w = int(rec["h"]), int(rec["w"])
        base = [rec[f][: h * w].reshape(h, w) for f in ("present", "absent", "set", "clear")]
        for j in range(4):
            rh, rw, *arrs = oracle.rotate(rec, j)
            for a, b in zip(arrs, base):
                np.testing.assert_array_equal(a, np.rot90(b, j))
            assert (rh, rw) == np.rot90(base[0], j).shape


# ------------------------------------------------ brute force vs convolution
def conv_formulation(boards, rule_table, C, ch_player, actions):
    """The paper's eqs. 1/3 with torch library routines.

    boards [N,H,W] int cell words, rule_table [R] RULE_DTYPE.  Returns
    (next boards, rewards).  Written independently of the oracle: force by
    shifting the player plane, matching by conv2d with +1/-1 weights and
    ReLU(conv - #present + 1), writes by conv_transpose2d of the binary
    activations, summed as target-minus-current changes and clamped.
    """
    N, H, W = boards.shape
    NCH = C + 1
    x = torch.zeros(N, NCH, H, W, dtype=torch.float64)
    b = torch.from_numpy(boards.astype(np.int64))
    for c in range(C):
        x[:, c] = ((b >> c) & 1).double()
    # force: next to each player cell in the action's direction
    if ch_player >= 0:
        pl = x[:, ch_player]
        force = torch.zeros(N, H, W, dtype=torch.float64)
        a = torch.from_numpy(np.asarray(actions, np.int64))
        up = torch.zeros_like(pl); up[:, :-1] = pl[:, 1:]
        down = torch.zeros_like(pl); down[:, 1:] = pl[:, :-1]
        right = torch.zeros_like(pl); right[:, :, 1:] = pl[:, :, :-1]
        left = torch.zeros_like(pl); left[:, :, :-1] = pl[:, :, 1:]
        for code, f in ((1, up), (2, right), (3, down), (4, left)):
            force += f * (a == code).double()[:, None, None]
        x[:, C] = (force > 0).double()
    setd = torch.zeros(N, C, H, W, dtype=torch.float64)
    clrd = torch.zeros(N, C, H, W, dtype=torch.float64)
    reward = torch.zeros(N, dtype=torch.float64)
    for rec in rule_table:
        h, w = int(rec["h"]), int(rec["w"])
        pres = rec["present"][: h * w].reshape(h, w)
        absn = rec["absent"][: h * w].reshape(h, w)
        sets = rec["set"][: h * w].reshape(h, w)
        clrs = rec["clear"][: h * w].reshape(h, w)
        for j in range(4):
            P, A = np.rot90(pres, j), np.rot90(absn, j)
            S, Cl = np.rot90(sets, j), np.rot90(clrs, j)
            hh, ww = P.shape
            if hh > H or ww > W:
                continue
            KI = torch.zeros(1, NCH, hh, ww, dtype=torch.float64)
            KS = torch.zeros(1, C, hh, ww, dtype=torch.float64)
            KC = torch.zeros(1, C, hh, ww, dtype=torch.float64)
            for c in range(NCH):
                KI[0, c] = torch.from_numpy(((P >> c) & 1).astype(np.float64) - ((A >> c) & 1))
            for c in range(C):
                KS[0, c] = torch.from_numpy(((S >> c) & 1).astype(np.float64))
                KC[0, c] = torch.from_numpy(((Cl >> c) & 1).astype(np.float64))
            n_present = float(sum(bin(int(v)).count("1") for v in P.reshape(-1)))
            B = torch.relu(Fnn.conv2d(x, KI) - n_present + 1.0)  # eq. 1
            reward += float(rec["reward"]) * B.sum(dim=(1, 2, 3))
            setd += Fnn.conv_transpose2d(B, KS)
            clrd += Fnn.conv_transpose2d(B, KC)
    D = x[:, :C]
    nxt = torch.clamp(D + setd * (1 - D) - clrd * D, 0, 1)  # eq. 3, clamped
    out = torch.zeros(N, H, W, dtype=torch.int64)
    for c in range(C):
        out |= nxt[:, c].round().long() << c
    return out.numpy(), reward.round().long().numpy()


def _all_3x3_boards_c2():
    vals = np.arange(4 ** 9, dtype=np.int64)
    digits = (vals[:, None] // (4 ** np.arange(9))[None, :]) % 4
    return digits.reshape(-1, 3, 3).astype(np.uint8)


@pytest.mark.parametrize("rule_seed", [11, 12])
def test_bruteforce_all_3x3_boards_against_convolution(rule_seed):
    C = 2
    boards = _all_3x3_boards_c2()
    wl = wk.Workload(0, "bf", 1, 3, 3, C, 4, ((1, 1), (1, 2), (2, 2), (2, 3), (3, 3)),
                     0.25, 0.2, 0.25, 0.25, -3, 3, rules_per_env=0)
    rules = wk.make_rules(wl, rule_seed)
    fields = dict(batch=len(boards), H=3, W=3, C=C, n_rules=4, rules_per_env=0, max_steps=0,
                  auto_reset=0, ch_player=0, ch_goal=1, ch_empty=-1, ch_wall=-1, border_wall=0,
                  cum_per_env=0)
    cfg = oracle.make_cfg(**fields)
    n = len(boards)
    for a in range(5):
        acts = np.full(n, a, np.uint8)
        got, _, rew, done = oracle.step(cfg, rules, boards, boards, np.zeros(n, np.int32), acts)
        exp, exp_rew = conv_formulation(boards, rules[0], C, 0, acts)
        np.testing.assert_array_equal(got.astype(np.int64), exp)
        np.testing.assert_array_equal(rew.astype(np.int64), exp_rew)
        np.testing.assert_array_equal(done, ((got >> 1) & 1).sum(axis=(1, 2)) == 0)


@pytest.mark.parametrize("key", [1, 2, 3, 6])
def test_random_16x16_against_convolution(key):
    """Random boards of the workloads' sizes (16 x 16, and 256 x 256)."""
    n = 6 if key != 6 else 2
    wl = wk.WORKLOADS[key].scaled(batch=n)
    rules = wk.make_rules(wl.scaled(rules_per_env=0), 40 + key)
    g = wk.random_grids(5 + key, n, wl.H, wl.W, wl.C, density=0.35)
    g[:, 3, 4] |= 1 << wk.CH_PLAYER
    fields = dict(wk.config_fields(wl), batch=n, rules_per_env=0, max_steps=0, auto_reset=0)
    cfg = oracle.make_cfg(**fields)
    acts = np.arange(n, dtype=np.uint8) % 5 + (key == 6)
    got, _, rew, _ = oracle.step(cfg, rules, g, g, np.zeros(n, np.int32), acts)
    exp, exp_rew = conv_formulation(g, rules[0], wl.C, wk.CH_PLAYER, acts)
    np.testing.assert_array_equal(got.astype(np.int64), exp)
    np.testing.assert_array_equal(rew.astype(np.int64), exp_rew)


def test_conflict_closed_form_equals_sum_then_clamp_bruteforce():
    # For one bit: D in {0,1}; any multiset of writes, each either "set" or
    # "clear" expressed as (target - D).  Sum then clamp equals
    # D ? !anyCLR : anySET.
    for D in (0, 1):
        for n_set, n_clr in itertools.product(range(4), range(4)):
            s = D + n_set * (1 - D) + n_clr * (0 - D)
            clamped = min(1, max(0, s))
            closed = (1 if n_clr == 0 else 0) if D else (1 if n_set > 0 else 0)
            assert clamped == closed


# --------------------------------------------------------------- invariants
def _cfg(wl, **kw):
    return oracle.make_cfg(**dict(wk.config_fields(wl), **kw))


def test_noop_rules_identity_and_reward():
    wl = wk.WORKLOADS[2].scaled(batch=8)
    _, rules, cum = wk.make(wl, 3)
    rules = rules.copy()
    rules["set"] = 0
    rules["clear"] = 0
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 103, range(8))
    for a in range(5):
        out, _, _, _ = oracle.step(cfg, rules, g, g, np.zeros(8), np.full(8, a))
        np.testing.assert_array_equal(out, g)
    # rules with no input terms match at every valid anchor, 4 rotations each
    empty = wk.empty_rules(8, 8)
    empty["h"], empty["w"] = 3, 3
    empty["reward"] = np.arange(8)[None, :] - 3
    out, _, rew, _ = oracle.step(cfg, empty, g, g, np.zeros(8), np.zeros(8))
    np.testing.assert_array_equal(out, g)
    assert (rew == sum(r - 3 for r in range(8)) * 14 * 14 * 4).all()


def test_single_mover_conserves_counts():
    fx = golden_io.load(golden_io.GOLDEN_DIR + "/03_eat_food.txt")
    rules = fx.rules[:, :1]  # move only
    H = W = 12
    n = 16
    g = wk.random_grids(77, n, H, W, 4, density=0.25)
    g &= ~np.uint8(1 << 2)  # no player bits
    g[:, :, :] = np.where(g & 2, 2, 1).astype(np.uint8)  # wall or floor
    g[:, 5, 5] = 1 | 4  # one player on floor
    fields = dict(batch=n, H=H, W=W, C=4, n_rules=1, rules_per_env=0, max_steps=0, auto_reset=0,
                  ch_player=2, ch_goal=-1, ch_empty=0, ch_wall=1, border_wall=0, cum_per_env=0)
    cfg = oracle.make_cfg(**fields)
    res = oracle.rollout(cfg, rules, g, g, np.zeros(n), 200, 9, trajectory=True)
    obs = res["obs"]
    for c in range(4):
        cnt = ((obs >> c) & 1).sum(axis=(2, 3))
        assert (cnt == ((g >> c) & 1).sum(axis=(1, 2))[None, :]).all()
    moved = (obs[-1] != g).any(axis=(1, 2))
    assert moved.sum() >= n // 2  # the player does move


ROT_ACTION = {0: 0, 1: 4, 2: 1, 3: 2, 4: 3}  # action after a CCW quarter turn


@pytest.mark.parametrize("key", [2, 3, 6])
def test_rotation_commutes_with_step(key):
    wl = wk.WORKLOADS[key].scaled(batch=10 if key != 6 else 2)
    _, rules, cum = wk.make(wl, 21)
    cfg = _cfg(wl)
    n = wl.batch
    g = oracle.reset(cfg, cum, 121, range(n))
    g = g | wk.random_grids(8, n, wl.H, wl.W, wl.C, density=0.08)
    for a in range(5):
        acts = np.full(n, a, np.uint8)
        out, _, rew, _ = oracle.step(cfg, rules, g, g, np.zeros(n), acts)
        g_rot = np.ascontiguousarray(np.rot90(g, 1, axes=(1, 2)))
        acts_rot = np.full(n, ROT_ACTION[a], np.uint8)
        out_rot, _, rew_rot, _ = oracle.step(cfg, rules, g_rot, g_rot, np.zeros(n), acts_rot)
        np.testing.assert_array_equal(out_rot, np.rot90(out, 1, axes=(1, 2)))
        np.testing.assert_array_equal(rew_rot, rew)


def test_rule_order_independence_random():
    wl = wk.WORKLOADS[3].scaled(batch=12)
    _, rules, cum = wk.make(wl, 5)
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 105, range(12))
    g = g | wk.random_grids(3, 12, wl.H, wl.W, wl.C, density=0.1)
    perm = rules[:, np.random.default_rng(0).permutation(wl.n_rules)].copy()
    for a in range(5):
        x = oracle.step(cfg, rules, g, g, np.zeros(12), np.full(12, a))
        y = oracle.step(cfg, perm, g, g, np.zeros(12), np.full(12, a))
        for u, v in zip(x, y):
            np.testing.assert_array_equal(u, v)


def test_same_seed_same_trajectory_and_threads_agree():
    wl = wk.WORKLOADS[3].scaled(batch=24)
    _, rules, cum = wk.make(wl, 2)
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 102, range(24))
    t0 = np.zeros(24, np.int32)
    a = oracle.rollout(cfg, rules, g, g, t0, 300, 202, trajectory=True, threads=1)
    b = oracle.rollout(cfg, rules, g, g, t0, 300, 202, trajectory=True, threads=8)
    for k in a:
        np.testing.assert_array_equal(a[k], b[k])
    c = oracle.rollout(cfg, rules, g, g, t0, 300, 203, trajectory=True)
    assert (c["obs"] != a["obs"]).any()
    # auto-reset: t restarts, and a done step returns the env's own initial map
    d = a["done"].astype(bool)
    assert d.any()
    s, e = np.argwhere(d)[0]
    np.testing.assert_array_equal(a["obs"][s, e], g[e])


def test_rollout_equals_repeated_steps():
    wl = wk.WORKLOADS[3].scaled(batch=8)
    _, rules, cum = wk.make(wl, 4)
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 104, range(8))
    res = oracle.rollout(cfg, rules, g, g, np.zeros(8), 40, 204, trajectory=True)
    cur, t = g.copy(), np.zeros(8, np.int32)
    for s in range(40):
        acts = np.array([int(wk.uniform_int(wk.draw(204, 4, e, 0, s), 5)) for e in range(8)])
        cur, t, rew, done = oracle.step(cfg, rules, cur, g, t, acts)
        np.testing.assert_array_equal(cur, res["obs"][s])
        np.testing.assert_array_equal(rew, res["rew"][s])
        np.testing.assert_array_equal(done, res["done"][s])
    np.testing.assert_array_equal(t, res["t"])


def test_max_steps_done_and_reset():
    wl = wk.WORKLOADS[3].scaled(batch=4, max_steps=7)
    _, rules, cum = wk.make(wl, 6)
    rules = rules.copy()
    rules["set"] = 0
    rules["clear"] = 0  # frozen boards keep their goals
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 106, range(4))
    g[:, 2, 2] |= 1 << wk.CH_GOAL
    res = oracle.rollout(cfg, rules, g, g, np.zeros(4), 21, 1, trajectory=True)
    assert (res["done"][6::7] == 1).all() and res["done"].sum() == 3 * 4
    assert (res["t"] == 0).all()


# ------------------------------------------------------------ initial maps
def test_reset_distribution_and_single_player():
    wl = wk.WORKLOADS[2].scaled(batch=400)
    _, _, cum = wk.make(wl, 0)
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 100, range(400)).astype(np.int64)
    players = ((g >> wk.CH_PLAYER) & 1).sum(axis=(1, 2))
    assert (players == 1).all()
    pl = (g >> wk.CH_PLAYER) & 1
    has_floor = (((g >> wk.CH_EMPTY) & 1).sum(axis=(1, 2)) > 0)
    on_floor = (((g >> wk.CH_EMPTY) & 1) * pl).sum(axis=(1, 2)) == 1
    assert (on_floor | ~has_floor).all()  # the player sits on floor when there is any
    assert has_floor.mean() > 0.9
    assert (g[:, 0, :] == 1 << wk.CH_WALL).all() and (g[:, :, -1] == 1 << wk.CH_WALL).all()
    inner = g[:, 1:-1, 1:-1] & ~(1 << wk.CH_PLAYER)
    # every interior cell is exactly one type
    assert (np.array([bin(int(v)).count("1") for v in inner.reshape(-1)[:5000]]) == 1).all()
    n = inner.shape[1] * inner.shape[2]
    prev = np.zeros(400)
    for t in range(wl.C):
        p = (cum[:, t].astype(np.float64) - prev) / 2 ** 24
        prev = cum[:, t].astype(np.float64)
        cnt = ((inner >> t) & 1).sum(axis=(1, 2))
        mu, sd = n * p, np.sqrt(n * p * (1 - p)) + 1e-9
        z = (cnt.sum() - mu.sum()) / np.sqrt((sd ** 2).sum() + 1e-9)
        assert abs(z) < 4, (t, z)
    assert (cum[:, wk.CH_PLAYER] == cum[:, wk.CH_PLAYER - 1]).all()


def test_reset_maze_probabilities():
    wl = wk.WORKLOADS[1].scaled(batch=1500)
    _, _, cum = wk.make(wl, 0)
    cfg = _cfg(wl)
    g = oracle.reset(cfg, cum, 100, range(1500)).astype(np.int64)
    inner = g[:, 1:-1, 1:-1]
    n = inner.size
    for ch, p in ((0, 0.7), (1, 0.25), (3, 0.05)):
        cnt = ((inner >> ch) & 1).sum()
        assert abs(cnt - n * p) < 4 * np.sqrt(n * p * (1 - p)), ch
