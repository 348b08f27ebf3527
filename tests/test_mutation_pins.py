"""Pins of the oracle's mutation operators (Sec. 3.1.1: map bits flipped at
random, tiles of the mutable rules' input and output patterns changed,
rewards changed): closed forms at rates 0 and 1, rates and choices within
statistical bounds, validity of the mutated records, and independence of
each environment's mutation from the rest of the batch.  Which counter draw
decides which bit is build-defined (like the initial maps) and is not pinned
beyond these properties."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk

ONE = 1 << 24


def _mut(**kw):
    m = dict(p_map=0, map_channels=0xFFFF, p_rule=0, p_reward=0, reward_min=-3, reward_max=3,
             mutable_rules=(1 << 64) - 1)
    m.update(kw)
    return m


def _batch(key=3, n=24, seed=0):
    wl = wk.WORKLOADS[key].scaled(batch=n)
    _, rules, cum = wk.make(wl, seed)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    maps = oracle.reset(cfg, cum, 100, range(n))
    return wl, maps, rules


def _states(one, two):
    """Per (entry, channel) ternary state of a pair of mask arrays [..., 25] -> [..., 25, 32]."""
    bits = np.arange(32, dtype=np.uint64)
    o = (one.astype(np.uint64)[..., None] >> bits) & 1
    t = (two.astype(np.uint64)[..., None] >> bits) & 1
    return (o + 2 * t).astype(np.int64)


def test_rate_zero_is_the_identity():
    wl, maps, rules = _batch()
    m2, r2 = oracle.mutate(wl.H, wl.W, wl.C, _mut(), 5, maps, rules)
    np.testing.assert_array_equal(m2, maps)
    assert r2.tobytes() == rules.tobytes()


@pytest.mark.parametrize("channels", [0xFFFF, 0b101, 1 << 2])
def test_map_rate_one_flips_every_chosen_bit(channels):
    wl, maps, rules = _batch()
    m2, _ = oracle.mutate(wl.H, wl.W, wl.C, _mut(p_map=ONE, map_channels=channels), 5, maps, None)
    mask = channels & ((1 << wl.C) - 1)
    np.testing.assert_array_equal(m2, maps ^ np.array(mask, maps.dtype))


def test_rule_rate_one_changes_every_entry_of_mutable_rules_only():
    wl, maps, rules = _batch(key=5, n=6)
    mutable = 0b1011_0110
    _, r2 = oracle.mutate(wl.H, wl.W, wl.C, _mut(p_rule=ONE, mutable_rules=mutable), 9, None, rules)
    C = wl.C
    for t in range(rules.shape[0]):
        for r in range(rules.shape[1]):
            a, b = rules[t, r], r2[t, r]
            assert (a["h"], a["w"]) == (b["h"], b["w"])
            if not (mutable >> r) & 1:
                assert a.tobytes() == b.tobytes()
                continue
            n_e = int(a["h"]) * int(a["w"])
            si, so = _states(a["present"], a["absent"]), _states(b["present"], b["absent"])
            assert (si[:n_e, :C + 1] != so[:n_e, :C + 1]).all()      # every input entry changed
            assert (so[:, C + 1:] == 0).all() and (so[n_e:] == 0).all()
            si, so = _states(a["set"], a["clear"]), _states(b["set"], b["clear"])
            assert (si[:n_e, :C] != so[:n_e, :C]).all()              # every output entry changed
            assert (so[:, C:] == 0).all() and (so[n_e:] == 0).all()
            assert a["reward"] == b["reward"]                        # p_reward = 0


def _binom_ok(k, n, p, z=5.0):
    return abs(k - n * p) <= z * np.sqrt(n * p * (1 - p)) + 1


def test_rates_and_choices_within_statistical_bounds():
    wl, maps, rules = _batch(n=64)
    C = wl.C
    m2, r2 = oracle.mutate(wl.H, wl.W, wl.C, _mut(p_map=ONE // 8, p_rule=ONE // 4), 11, maps, rules)
    flips = int(np.unpackbits((maps ^ m2).view(np.uint8)).sum())
    assert _binom_ok(flips, maps.size * C, 1 / 8)
    changed = toward_next = total = 0
    for t in range(rules.shape[0]):
        for r in range(rules.shape[1]):
            a, b = rules[t, r], r2[t, r]
            n_e = int(a["h"]) * int(a["w"])
            for one, two, nch in (("present", "absent", C + 1), ("set", "clear", C)):
                s0 = _states(a[one], a[two])[:n_e, :nch]
                s1 = _states(b[one], b[two])[:n_e, :nch]
                total += s0.size
                ch = s0 != s1
                changed += int(ch.sum())
                toward_next += int((s1[ch] == (s0[ch] + 1) % 3).sum())
    assert _binom_ok(changed, total, 1 / 4)
    assert _binom_ok(toward_next, changed, 1 / 2)


def test_reward_redraw_stays_in_range_and_covers_it():
    wl, maps, rules = _batch(n=200)
    _, r2 = oracle.mutate(wl.H, wl.W, wl.C, _mut(p_reward=ONE, reward_min=-5, reward_max=7), 3,
                          None, rules)
    rew = r2["reward"].reshape(-1)
    assert rew.min() >= -5 and rew.max() <= 7
    counts = np.bincount(rew + 5, minlength=13)
    assert (counts > 0).all()
    expect = rew.size / 13
    assert ((counts - expect) ** 2 / expect).sum() < 60  # chi-square, 12 dof, far tail
    _, r3 = oracle.mutate(wl.H, wl.W, wl.C, _mut(p_reward=ONE // 2, reward_min=-5, reward_max=7), 3,
                          None, rules)
    kept = int((r3["reward"] == rules["reward"]).sum())
    n = rules["reward"].size
    # kept: not redrawn (1/2) or redrawn to the same value (1/2 x ~1/13)
    assert _binom_ok(kept, n, 0.5 + 0.5 / 13)


def test_mutated_records_are_valid_and_masks_disjoint():
    wl, maps, rules = _batch(key=5, n=8)
    _, r2 = oracle.mutate(wl.H, wl.W, wl.C, _mut(p_rule=ONE // 3, p_reward=ONE // 2), 17, None, rules)
    assert ((r2["present"] & r2["absent"]) == 0).all()
    assert ((r2["set"] & r2["clear"]) == 0).all()
    assert ((r2["set"] | r2["clear"]) >> wl.C == 0).all()
    assert ((r2["present"] | r2["absent"]) >> (wl.C + 1) == 0).all()


def test_each_env_independent_of_the_batch_and_seeded():
    wl, maps, rules = _batch(n=40)
    mut = _mut(p_map=ONE // 16, p_rule=ONE // 8, p_reward=ONE // 4)
    full_m, full_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 21, maps, rules)
    ids = np.array([3, 17, 39, 0], np.int32)
    sub_m, sub_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 21, maps[ids], rules[ids], env_ids=ids)
    np.testing.assert_array_equal(sub_m, full_m[ids])
    assert sub_r.tobytes() == full_r[ids].tobytes()
    again_m, again_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 21, maps, rules)
    np.testing.assert_array_equal(again_m, full_m)
    other_m, _ = oracle.mutate(wl.H, wl.W, wl.C, mut, 22, maps, rules)
    assert (other_m != full_m).any()
