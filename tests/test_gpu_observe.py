"""Policy observation (Sec. 3.2; Sec. 4, Tables 1 and 2) through the C-ABI
against the CPU oracle, bit-exact: player-centred patches of every width from
1 to 127 (one and several row slabs per patch), boards with no, one or two
players, cell words of one and two bytes, patches starting at every byte
alignment, the full-size training shape, and the binary rule encoding."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import workload as wk
from tests import golden_obs
from tests.gpu_helpers import make, sample_envs, to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2407_04221_gb300 as av
    av.load()


def _fields(B, H, W, C, ch_player):
    return dict(batch=B, H=H, W=W, C=C, n_rules=0, rules_per_env=0, max_steps=0, auto_reset=0,
                ch_player=ch_player, ch_goal=-1, ch_empty=-1, ch_wall=-1, border_wall=0,
                cum_per_env=0)


def _random_boards(rng, B, H, W, C, ch_player):
    boards = rng.integers(0, 1 << C, size=(B, H, W)).astype(oracle.cell_dtype(C))
    boards &= ~np.array(1 << ch_player, boards.dtype)
    for b in range(B):  # 0, 1 or 2 players
        for _ in range(b % 3):
            boards[b, rng.integers(H), rng.integers(W)] |= 1 << ch_player
    return boards


@pytest.mark.parametrize("path", golden_obs.patch_fixtures(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_patch_fixture(path):
    import paper_2407_04221_gb300 as av
    fx = golden_obs.load_patch(path)
    env = av.Env(fx.cfg_fields(), np.zeros(0, np.uint8))
    env.set_state(to_dev(fx.board[None]))
    obs, pyx = env.observe(fx.window)
    want = ((fx.patch.astype(np.int64)[..., None] >> np.arange(fx.C)) & 1).astype(np.uint8)
    np.testing.assert_array_equal(to_np(obs)[0], want)
    assert tuple(to_np(pyx)[0]) == fx.player
    env.close()


@pytest.mark.parametrize("H,W,C", [(16, 16, 8), (16, 16, 10), (7, 9, 4), (1, 1, 1), (64, 3, 16),
                                   (2, 64, 5), (33, 33, 12), (64, 64, 16)])
def test_random_boards_every_window(H, W, C):
    import paper_2407_04221_gb300 as av
    rng = np.random.default_rng(H * 1000 + W * 10 + C)
    B = 37  # odd, so consecutive patches start at many byte alignments
    ch_player = C // 2
    boards = _random_boards(rng, B, H, W, C, ch_player)
    fields = _fields(B, H, W, C, ch_player)
    env = av.Env(fields, np.zeros(0, np.uint8))
    env.set_state(to_dev(boards))
    cfg = oracle.make_cfg(**fields)
    for window in (1, 2, 3, 4, 5, 10, 20, 31, 32, 63, 127):
        obs, pyx = env.observe(window)
        want, want_pyx = oracle.observe(cfg, boards, window)
        np.testing.assert_array_equal(to_np(obs), want, err_msg=f"window {window}")
        np.testing.assert_array_equal(to_np(pyx), want_pyx)
    env.sync()
    env.close()


@pytest.mark.parametrize("B,H,W,C,window", [
    (5000, 7, 9, 5, 3),       # 63-byte boards: plain loads; ~2 envs per CTA
    (6000, 16, 16, 8, 31),    # 256-byte boards: asynchronous 16-byte copies
    (700, 33, 33, 12, 127),   # seven row slabs per patch, several patches per CTA
])
def test_many_envs_per_cta(B, H, W, C, window):
    """More environments than resident CTAs: each CTA runs several patches
    through its two board buffers and two staging slabs."""
    import paper_2407_04221_gb300 as av
    rng = np.random.default_rng(B + window)
    boards = _random_boards(rng, B, H, W, C, 0)
    fields = _fields(B, H, W, C, 0)
    env = av.Env(fields, np.zeros(0, np.uint8))
    env.set_state(to_dev(boards))
    obs, pyx = env.observe(window)
    want, want_pyx = oracle.observe(oracle.make_cfg(**fields), boards, window)
    np.testing.assert_array_equal(to_np(obs), want)
    np.testing.assert_array_equal(to_np(pyx), want_pyx)
    env.sync()
    env.close()


@pytest.mark.parametrize("offset", list(range(16)))
def test_any_output_alignment_and_no_stray_writes(offset):
    """Patches written at every byte offset from a 16-byte boundary; the bytes
    around the output stay untouched."""
    import paper_2407_04221_gb300 as av
    rng = np.random.default_rng(offset)
    B, H, W, C, window = 5, 16, 16, 10, 31
    boards = _random_boards(rng, B, H, W, C, 2)
    fields = _fields(B, H, W, C, 2)
    env = av.Env(fields, np.zeros(0, np.uint8))
    env.set_state(to_dev(boards))
    n = B * window * window * C
    raw = torch.full((n + 64,), 0xAB, dtype=torch.uint8, device="cuda")
    out = raw[16 + offset:16 + offset + n].view(B, window, window, C)
    av.av_observe(env.h, None, window, out)
    want, _ = oracle.observe(oracle.make_cfg(**fields), boards, window)
    got = to_np(raw)
    np.testing.assert_array_equal(got[16 + offset:16 + offset + n].reshape(want.shape), want)
    assert (got[:16 + offset] == 0xAB).all() and (got[16 + offset + n:] == 0xAB).all()
    env.close()


def test_bits_above_c_are_not_observed():
    """Cell words may carry bits at or above C (uint8 cells with C < 8): they
    are not tiles and never reach the patch."""
    import paper_2407_04221_gb300 as av
    rng = np.random.default_rng(11)
    B, H, W, C = 7, 16, 16, 3
    boards = rng.integers(0, 256, size=(B, H, W)).astype(np.uint8)
    fields = _fields(B, H, W, C, 1)
    env = av.Env(fields, np.zeros(0, np.uint8))
    obs, pyx = env.observe(31, grids=to_dev(boards))
    want, want_pyx = oracle.observe(oracle.make_cfg(**fields), boards, 31)
    np.testing.assert_array_equal(to_np(obs), want)
    np.testing.assert_array_equal(to_np(pyx), want_pyx)
    env.close()


def test_given_boards_and_errors():
    """`grids` observes caller boards without touching the handle's state; a
    configuration without a player channel is AV_ESTATE; bad windows AV_EINVAL."""
    import paper_2407_04221_gb300 as av
    rng = np.random.default_rng(7)
    B, H, W, C = 9, 12, 10, 6
    fields = _fields(B, H, W, C, 1)
    cur = _random_boards(rng, B, H, W, C, 1)
    other = _random_boards(rng, B, H, W, C, 1)
    env = av.Env(fields, np.zeros(0, np.uint8))
    env.set_state(to_dev(cur))
    obs, pyx = env.observe(5, grids=to_dev(other))
    want, want_pyx = oracle.observe(oracle.make_cfg(**fields), other, 5)
    np.testing.assert_array_equal(to_np(obs), want)
    np.testing.assert_array_equal(to_np(pyx), want_pyx)
    state, _ = env.get_state()
    np.testing.assert_array_equal(to_np(state), cur)
    for bad in (0, av.AV_MAX_WINDOW + 1):
        with pytest.raises(av.AvError) as ei:
            av.av_observe(env.h, None, bad, obs)
        assert ei.value.status == av.AV_EINVAL
    env.close()
    env = av.Env(_fields(B, H, W, C, -1), np.zeros(0, np.uint8))
    with pytest.raises(av.AvError) as ei:
        env.observe(5)
    assert ei.value.status == av.AV_ESTATE
    env.close()


@pytest.mark.parametrize("window", [5, 10, 20, 31])
def test_full_size_training_shape(window):
    """The 16,384-env training shape (16 x 16, C = 10, two-byte cells) after
    a 60-step rollout (multi-hot cells, moved or vanished players), every
    Table 1 width; oracle on a sample of envs (envs are independent)."""
    wl = wk.WORKLOADS[3]
    env, cfg, rules, cum = make(wl, 0)
    s = wk.seeds(0)
    env.reset(s["reset"])
    env.rollout(60, s["actions"])
    boards, _ = env.get_state()
    obs, pyx = env.observe(window)
    ids = sample_envs(wl.batch, 512, seed=window)
    b = to_np(boards)[ids]
    want, want_pyx = oracle.observe(cfg, b, window)
    np.testing.assert_array_equal(to_np(obs)[ids], want)
    np.testing.assert_array_equal(to_np(pyx)[ids], want_pyx)
    env.sync()
    env.close()


@pytest.mark.parametrize("key,per_env", [(3, True), (5, True), (1, False)])
def test_rule_encoding(key, per_env):
    wl = wk.WORKLOADS[key].scaled(batch=64)
    env, cfg, rules, cum = make(wl, 2)
    bits, rew = env.rule_obs()
    want, want_rew = oracle.rule_obs(cfg, rules)
    assert bool(int(wk.config_fields(wl)["rules_per_env"])) == per_env
    np.testing.assert_array_equal(to_np(bits), want)
    np.testing.assert_array_equal(to_np(rew), want_rew)
    env.close()


@pytest.mark.parametrize("path", golden_obs.rule_fixtures(), ids=lambda p: p.rsplit("/", 1)[-1])
def test_rule_fixture(path):
    import paper_2407_04221_gb300 as av
    fx = golden_obs.load_rules(path)
    fields = _fields(1, 4, 4, fx.C, -1)
    fields["n_rules"] = fx.rules.shape[1]
    env = av.Env(fields, fx.rules)
    bits, rew = env.rule_obs()
    np.testing.assert_array_equal(to_np(bits), fx.bits)
    np.testing.assert_array_equal(to_np(rew), fx.rewards)
    env.close()
