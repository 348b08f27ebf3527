"""Pins of the oracle's variant semantics (Sec. 2.1, "Possible extensions":
apply a rule once or a fixed number of times, choosing the tiles by the
maximum over an ordered or random index channel; let rules inhibit others):
hand-worked fixtures, the neutral variant equal to the standard step, and
rewards that follow from each rule's raw match count -- counted independently
by the standard step on a one-rule table -- under limits and inhibition."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests import golden_io


def _variant_of(fx):
    v = fx.variant
    R = fx.rules.shape[1]
    return oracle.make_variant(random_keys=v["index"] == "random",
                               limit=[v["limit"].get(r, 0) for r in range(R)],
                               inhibit=[v["inhibit"].get(r, 0) for r in range(R)])


@pytest.mark.parametrize("path", golden_io.variant_fixtures(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_variant_fixture(path):
    fx = golden_io.load(path)
    assert fx.cite
    cfg = oracle.make_cfg(**fx.cfg_fields())
    g = fx.before[None]
    out, t, rew, done = oracle.step(cfg, fx.rules, g, g, np.zeros(1, np.int32),
                                    np.array([fx.action], np.uint8), variant=_variant_of(fx))
    np.testing.assert_array_equal(out[0], fx.after)
    assert int(rew[0]) == fx.reward
    assert int(done[0]) == fx.done


def _state(key, n=24, steps=0, seed=0):
    wl = wk.WORKLOADS[key].scaled(batch=n)
    _, rules, cum = wk.make(wl, seed)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    g = oracle.reset(cfg, cum, 100, range(n))
    if steps:
        g = oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), steps, 200)["grids"]
    return wl, cfg, rules, g


def _raw_counts(cfg, rules, g, actions):
    """Matches of each rule (all rotations and anchors) on each board: the
    standard step on a one-rule table with reward 1 and no outputs."""
    n, R = rules.shape
    counts = np.zeros((n, R), np.int64)
    c1 = oracle.make_cfg(**{f: getattr(cfg, f) for f in oracle.FIELDS})
    c1.n_rules = 1
    for r in range(R):
        one = rules[:, r:r + 1].copy()
        one["reward"] = 1
        one["set"] = 0
        one["clear"] = 0
        _, _, rew, _ = oracle.step(c1, one, g, g, np.zeros(n, np.int32), actions)
        counts[:, r] = rew
    return counts


@pytest.mark.parametrize("key,steps", [(2, 0), (3, 40), (1, 10)])
def test_neutral_variant_is_the_standard_step(key, steps):
    wl, cfg, rules, g = _state(key, steps=steps)
    n = g.shape[0]
    v = oracle.make_variant(random_keys=1, key_seed=9)
    a = oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), 30, 201, trajectory=True)
    b = oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), 30, 201, trajectory=True, variant=v)
    for k in ("grids", "rew", "done", "obs", "t"):
        np.testing.assert_array_equal(a[k], b[k])


@pytest.mark.parametrize("key,steps,random_keys", [(3, 40, 0), (3, 40, 1), (3, 5, 1)])
@pytest.mark.parametrize("k", [1, 2, 5])
def test_limited_reward_follows_raw_counts(key, steps, random_keys, k):
    wl, cfg, rules, g = _state(key, steps=steps)
    n, R = g.shape[0], wl.n_rules
    tab = rules if rules.shape[0] == n else np.repeat(rules, n, axis=0)
    cfg.rules_per_env = 1
    actions = np.arange(n, dtype=np.uint8) % 5
    counts = _raw_counts(cfg, tab, g, actions)
    v = oracle.make_variant(random_keys=random_keys, key_seed=5, limit=[k] * R)
    _, _, rew, _ = oracle.step(cfg, tab, g, g, np.zeros(n, np.int32), actions, variant=v)
    want = (np.minimum(counts, k) * tab["reward"].astype(np.int64)).sum(axis=1)
    np.testing.assert_array_equal(rew, want)
    assert (counts > k).any()  # the limit binds somewhere


def test_inhibited_reward_follows_raw_counts():
    wl, cfg, rules, g = _state(3, n=40, steps=40)
    n, R = g.shape[0], wl.n_rules
    actions = np.arange(n, dtype=np.uint8) % 5
    counts = _raw_counts(cfg, rules, g, actions)
    rng = np.random.default_rng(3)
    inhibit = [int(rng.integers(0, 1 << R)) & ~(1 << r) for r in range(R)]
    v = oracle.make_variant(inhibit=inhibit)
    _, _, rew, _ = oracle.step(cfg, rules, g, g, np.zeros(n, np.int32), actions, variant=v)
    for e in range(n):
        sup = 0
        for r in range(R):
            if counts[e, r] > 0:
                sup |= inhibit[r]
        want = sum(int(counts[e, r]) * int(rules[e, r]["reward"]) for r in range(R) if not (sup >> r) & 1)
        assert int(rew[e]) == want, e


def test_random_keys_spread_the_single_application():
    """Apply once with random keys: over many step counters the applied
    anchor is spread evenly over the rule's matches (chi-square)."""
    fx = golden_io.load(golden_io.variant_fixtures()[0])  # 'grow' on three floor cells
    cfg = oracle.make_cfg(**fx.cfg_fields())
    v = oracle.make_variant(random_keys=1, key_seed=11, limit=[1])
    g = fx.before[None]
    hits = {}
    T = 600
    for t in range(T):
        out, _, rew, _ = oracle.step(cfg, fx.rules, g, g, np.array([t], np.int32),
                                     np.zeros(1, np.uint8), variant=v)
        changed = tuple(map(tuple, np.argwhere(out[0] != g[0])))
        assert len(changed) == 1 and int(rew[0]) == 2
        hits[changed[0]] = hits.get(changed[0], 0) + 1
    assert set(hits) == {(0, 0), (1, 1), (2, 0)}
    obs = np.array(list(hits.values()), float)
    assert (((obs - T / 3) ** 2) / (T / 3)).sum() < 20  # 2 dof, far tail


def test_rollout_equals_repeated_variant_steps():
    wl, cfg, rules, g = _state(3, n=8, steps=20)
    n, R = g.shape[0], wl.n_rules
    v = oracle.make_variant(random_keys=1, key_seed=4, limit=[1, 2, 0, 3] * 3,
                            inhibit=[0b10, 0, 0b1000, 0] + [0] * 8)
    res = oracle.rollout(cfg, rules, g, g, np.zeros(n, np.int32), 12, 300, trajectory=True, variant=v)
    cur, t = g.copy(), np.zeros(n, np.int32)
    for s in range(12):
        a = np.array([wk.uniform_int(wk.draw(300, 4, e, 0, s), 5) for e in range(n)], np.uint8)
        cur, t, rew, done = oracle.step(cfg, rules, cur, g, t, a, variant=v)
        np.testing.assert_array_equal(cur, res["obs"][s])
        np.testing.assert_array_equal(rew, res["rew"][s])
