"""Mutation operators (Sec. 3.1.1) through the C-ABI against the CPU oracle,
bit-exact: maps and packed rule records after av_mutate, for every workload
shape (one- and two-byte cells, 1x2 to 5x5 patterns, shared and per-env
tables), the full 16,384-env batch on sampled envs, single operators, and an
evolution step end to end (mutate, build a handle from the offspring, roll
out)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests.gpu_helpers import sample_envs, to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ONE = 1 << 24


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()


def _mut(**kw):
    m = dict(p_map=ONE // 64, map_channels=0xFFFF, p_rule=ONE // 8, p_reward=ONE // 4,
             reward_min=-3, reward_max=3, mutable_rules=(1 << 64) - 1)
    m.update(kw)
    return m


def _rules_dev(rules):
    B, R = rules.shape
    return torch.from_numpy(np.ascontiguousarray(rules).view(np.uint8).reshape(B, R, 408).copy()).cuda()


def _rules_host(t, B, R):
    return t.cpu().numpy().reshape(-1).view(wk.RULE_DTYPE).reshape(B, R)


def _inputs(key, batch, seed=0):
    wl = wk.WORKLOADS[key].scaled(batch=batch)
    _, rules, cum = wk.make(wl, seed)
    if rules.shape[0] == 1 and batch > 1:  # shared table: one per env for mutation
        rules = np.repeat(rules, batch, axis=0)
    cfg = oracle.make_cfg(**wk.config_fields(wl))
    maps = oracle.reset(cfg, cum, 100, range(batch))
    return wl, maps, rules


@pytest.mark.parametrize("key", [1, 2, 3, 4, 5])
def test_every_workload_shape(key):
    import paper_2407_04221_gb300 as av
    wl, maps, rules = _inputs(key, 37)
    mut = _mut(mutable_rules=0b1111_1111_1100 if key != 1 else 0b110)
    dm, dr = to_dev(maps), _rules_dev(rules)
    av.av_mutate(37, wl.H, wl.W, wl.C, rules.shape[1], mut, 77, dm, dr)
    want_m, want_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 77, maps, rules)
    np.testing.assert_array_equal(to_np(dm), want_m)
    assert _rules_host(dr, 37, rules.shape[1]).tobytes() == want_r.tobytes()


@pytest.mark.parametrize("which", ["map", "rule", "reward", "all_rate_one"])
def test_single_operators(which):
    import paper_2407_04221_gb300 as av
    wl, maps, rules = _inputs(5, 9)
    mut = {"map": _mut(p_rule=0, p_reward=0, map_channels=0b1010_0000_0101),
           "rule": _mut(p_map=0, p_reward=0, p_rule=ONE // 3),
           "reward": _mut(p_map=0, p_rule=0, p_reward=ONE // 2, reward_min=-100000, reward_max=2**31 - 1),
           "all_rate_one": _mut(p_map=ONE, p_rule=ONE, p_reward=ONE)}[which]
    dm, dr = to_dev(maps), _rules_dev(rules)
    av.av_mutate(9, wl.H, wl.W, wl.C, rules.shape[1], mut, 5, dm, dr)
    want_m, want_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 5, maps, rules)
    np.testing.assert_array_equal(to_np(dm), want_m)
    assert _rules_host(dr, 9, rules.shape[1]).tobytes() == want_r.tobytes()


def test_full_batch_sampled():
    import paper_2407_04221_gb300 as av
    wl, maps, rules = _inputs(3, 16384)
    mut = _mut()
    dm, dr = to_dev(maps), _rules_dev(rules)
    av.av_mutate(16384, wl.H, wl.W, wl.C, rules.shape[1], mut, 2024, dm, dr)
    ids = sample_envs(16384, 256, seed=1).astype(np.int32)
    want_m, want_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 2024, maps[ids], rules[ids], env_ids=ids)
    np.testing.assert_array_equal(to_np(dm)[ids], want_m)
    assert _rules_host(dr, 16384, rules.shape[1])[ids].tobytes() == want_r.tobytes()


def test_evolution_step_end_to_end():
    """Offspring (mutated copies of parents) become a new handle whose
    rollout matches the oracle's on the same offspring."""
    import paper_2407_04221_gb300 as av
    wl, maps, rules = _inputs(2, 64)
    parents = np.arange(64) // 2  # two offspring per parent
    dm, dr = to_dev(maps[parents]), _rules_dev(rules[parents])
    mut = _mut(mutable_rules=0b1111_1100)
    av.av_mutate(64, wl.H, wl.W, wl.C, wl.n_rules, mut, 31, dm, dr)
    kids_r = _rules_host(dr, 64, wl.n_rules).copy()
    kids_m = to_np(dm)
    want_m, want_r = oracle.mutate(wl.H, wl.W, wl.C, mut, 31, maps[parents], rules[parents])
    np.testing.assert_array_equal(kids_m, want_m)
    assert kids_r.tobytes() == want_r.tobytes()
    fields = dict(wk.config_fields(wl), batch=64)
    env = av.Env(fields, kids_r)
    env.set_state(to_dev(kids_m), set_as_init=True)
    res = env.rollout(50, 200)
    cfg = oracle.make_cfg(**fields)
    ref = oracle.rollout(cfg, kids_r, kids_m, kids_m, np.zeros(64, np.int32), 50, 200)
    g, _ = env.get_state()
    np.testing.assert_array_equal(to_np(g), ref["grids"])
    np.testing.assert_array_equal(to_np(res["rew_sum"]), ref["rew_sum"])
    env.close()


def test_rejects_bad_rates():
    import paper_2407_04221_gb300 as av
    for bad in (_mut(p_map=ONE + 1), _mut(p_rule=ONE + 1), _mut(reward_min=1, reward_max=0)):
        with pytest.raises(av.AvError) as ei:
            av.av_mutate(1, 16, 16, 8, 8, bad, 0, None, None)
        assert ei.value.status == av.AV_EINVAL
