"""Variant rule semantics (Sec. 2.1, "Possible extensions": apply limits chosen
by the largest keys of an ordered or random index channel; inhibition masks)
through the C-ABI against the CPU oracle, bit-exact: the hand-worked fixtures,
rollouts with trajectories on every workload shape under random limits and
masks in both key modes, the full 16,384-env training shape on sampled envs,
single steps against fused rollouts, and the handle's path and errors."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests import golden_io
from tests.gpu_helpers import make, sample_envs, to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()


def _random_variant(R, seed, random_keys):
    rng = np.random.default_rng(seed)
    limit = [int(x) for x in rng.choice([0, 1, 2, 3, 7], size=R)]
    inhibit = [int(rng.integers(0, 1 << R)) if rng.random() < 0.3 else 0 for _ in range(R)]
    return dict(random_keys=random_keys, key_seed=seed * 7 + 1, limit=limit, inhibit=inhibit)


@pytest.mark.parametrize("path", golden_io.variant_fixtures(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_variant_fixture(path):
    import paper_2407_04221_gb300 as av
    fx = golden_io.load(path)
    R = fx.rules.shape[1]
    env = av.Env(fx.cfg_fields(), fx.rules)
    av.av_set_variant(env.h, random_keys=fx.variant["index"] == "random",
                      limit=[fx.variant["limit"].get(r, 0) for r in range(R)],
                      inhibit=[fx.variant["inhibit"].get(r, 0) for r in range(R)])
    assert av.av_rollout_path(env.h) == av.AV_PATH_VARIANT
    env.set_state(to_dev(fx.before[None]), set_as_init=True)
    obs, rew, done = env.step(to_dev(np.array([fx.action], np.uint8)))
    np.testing.assert_array_equal(to_np(obs)[0], fx.after)
    assert int(rew[0]) == fx.reward
    assert int(done[0]) == fx.done
    env.close()


@pytest.mark.parametrize("key", [1, 2, 3, 4, 5])
@pytest.mark.parametrize("random_keys", [0, 1])
@pytest.mark.parametrize("kernel", ["default", "warp", "block"])
def test_rollout_every_shape(key, random_keys, kernel, monkeypatch):
    """Both variant kernels (one warp per environment, one CTA per
    environment) on every shape the first supports."""
    import paper_2407_04221_gb300 as av
    if kernel != "default":
        if key == 5 and kernel == "warp":
            pytest.skip("64 x 64 boards take the CTA-per-environment kernel")
        monkeypatch.setenv("AV_KERNEL_PATH", kernel)
    n = 24 if key != 5 else 8
    steps = 40 if key != 5 else 12
    wl = wk.WORKLOADS[key].scaled(batch=n)
    env, cfg, rules, cum = make(wl, 1)
    v = _random_variant(wl.n_rules, 10 * key + random_keys, random_keys)
    av.av_set_variant(env.h, **v)
    s = wk.seeds(1)
    g0 = to_np(env.reset(s["reset"]))
    # boards after some standard steps make more rules match
    av.av_set_variant(env.h, clear=True)
    env.rollout(20, 77)
    av.av_set_variant(env.h, **v)
    g1, t1 = env.get_state()
    res = env.rollout(steps, s["actions"], trajectory=True)
    g2, t2 = env.get_state()
    ov = oracle.make_variant(**v)
    ref = oracle.rollout(cfg, rules, to_np(g1), g0, to_np(t1), steps, s["actions"], trajectory=True,
                         variant=ov)
    np.testing.assert_array_equal(to_np(res["obs"]), ref["obs"])
    np.testing.assert_array_equal(to_np(res["rew"]), ref["rew"])
    np.testing.assert_array_equal(to_np(res["done"]), ref["done"])
    np.testing.assert_array_equal(to_np(g2), ref["grids"])
    np.testing.assert_array_equal(to_np(t2), ref["t"])
    env.sync()
    env.close()


def test_full_training_shape_sampled():
    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[3]
    env, cfg, rules, cum = make(wl, 0)
    v = _random_variant(wl.n_rules, 5, 1)
    s = wk.seeds(0)
    g0 = to_np(env.reset(s["reset"]))
    av.av_set_variant(env.h, **v)
    res = env.rollout(120, s["actions"])
    g, t = env.get_state()
    ids = sample_envs(wl.batch, 256, seed=3)
    ref = oracle.rollout(cfg, rules, g0[ids], g0[ids], np.zeros(len(ids), np.int32), 120, s["actions"],
                         env_ids=ids, variant=oracle.make_variant(**v))
    np.testing.assert_array_equal(to_np(g)[ids], ref["grids"])
    np.testing.assert_array_equal(to_np(res["rew_sum"])[ids], ref["rew_sum"])
    np.testing.assert_array_equal(to_np(t)[ids], ref["t"])
    env.sync()
    env.close()


def test_steps_equal_fused_rollout():
    """av_step repeated with the rollout's own actions equals av_rollout: the
    random keys follow the env's step counter, not the call."""
    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[3].scaled(batch=16)
    env, cfg, rules, cum = make(wl, 2)
    v = _random_variant(wl.n_rules, 9, 1)
    av.av_set_variant(env.h, **v)
    g0 = env.reset(100)
    res = env.rollout(25, 300, trajectory=True)
    env.set_state(g0, set_as_init=True)
    for s in range(25):
        a = np.array([wk.uniform_int(wk.draw(300, 4, e, 0, s), 5) for e in range(16)], np.uint8)
        obs, rew, done = env.step(to_dev(a))
        np.testing.assert_array_equal(to_np(obs), to_np(res["obs"][s]))
        np.testing.assert_array_equal(to_np(rew), to_np(res["rew"][s]))
    env.close()


def test_path_neutral_and_errors():
    import paper_2407_04221_gb300 as av
    wl = wk.WORKLOADS[2].scaled(batch=4)
    env, cfg, rules, cum = make(wl, 0)
    std = av.av_rollout_path(env.h)
    av.av_set_variant(env.h, limit=[0] * 8, inhibit=[0] * 8)  # neutral: the standard step
    assert av.av_rollout_path(env.h) == std
    av.av_set_variant(env.h, limit=[1] + [0] * 7)
    assert av.av_rollout_path(env.h) == av.AV_PATH_VARIANT
    parents = env.boards(4, 2)
    with pytest.raises(av.AvError) as ei:
        env.expand(parents)
    assert ei.value.status == av.AV_ESTATE
    av.av_set_variant(env.h, clear=True)
    assert av.av_rollout_path(env.h) == std
    for bad in (dict(limit=[256]), dict(limit=[-1]), dict(limit=[0] * 8 + [1]),
                dict(inhibit=[1 << 8]), dict(random_keys=2)):
        with pytest.raises(av.AvError) as ei:
            av.av_set_variant(env.h, **bad)
        assert ei.value.status == av.AV_EINVAL, bad
    env.close()
