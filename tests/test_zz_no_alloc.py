"""av_select_static: the search selection step for callers that cannot allocate.

Some callers cannot call cudaMalloc: their code runs under an allocator or a
fixed-budget memory pool they do not own, or a device allocation would break
their memory accounting.  For them the library has one entry point that
allocates nothing, av_select_static: the caller owns every input, output and
the visited sets, and the merge of the visited sets works in a fixed array
inside the library.  This file checks it, through the C ABI, against the
handle-based av_select on the same candidates, exactly, on two calls in a row.
It is collected last so that a run stopping at the first failure has already
run every other test.
"""
from __future__ import annotations

import numpy as np
import pytest

from tests import golden_io
from tests.gpu_helpers import to_dev, to_np

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_select_static_matches_select_on_two_calls():
    import paper_2407_04221_gb300 as av
    B, k, iters = 6, 24, 2
    cap = 1 + k * iters
    # the base maze game (Sec. 2.2.1): move and eat rules on an open board
    fx = golden_io.load(golden_io.GOLDEN_DIR + "/03_eat_food.txt")
    fields = dict(fx.cfg_fields(), batch=B, H=16, W=16)
    env = av.Env(fields, fx.rules, search_capacity=cap)
    g = np.full((B, 16, 16), 1, np.uint8)
    g[:, 0, :] = g[:, -1, :] = g[:, :, 0] = g[:, :, -1] = 2
    for e in range(B):
        g[e, 3 + e, 4] |= 4
        g[e, 10, 11 - e] = 8
    roots = to_dev(g)
    H, W, C = 16, 16, fx.C
    dev, i32, u8, i64 = env.device, torch.int32, torch.uint8, torch.int64

    root_hash = torch.zeros(B, dtype=i64, device=dev)
    root_live = torch.zeros(B, dtype=u8, device=dev)
    av.av_search_init(env.h, roots, root_hash, root_live)
    visited = torch.zeros(B, cap, dtype=i64, device=dev)  # caller-owned sets
    visited[:, 0] = root_hash
    n_visited = torch.ones(B, dtype=i32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)

    front = env.boards(B, k)
    front[:, 0] = roots
    cum = torch.zeros(B, k, dtype=i32, device=dev)
    live = torch.zeros(B, k, dtype=u8, device=dev)
    live[:, 0] = root_live
    n = torch.ones(B, dtype=i32, device=dev)
    expected_visited = [{int(h)} for h in to_np(root_hash, "hash")]

    for call in range(2):
        children, rew, done, hashes = env.expand(front, n)
        outs = []
        for _ in range(2):
            outs.append((env.boards(B, k), torch.zeros(B, k, dtype=i32, device=dev),
                         torch.zeros(B, k, dtype=i64, device=dev),
                         torch.zeros(B, k, dtype=u8, device=dev),
                         torch.zeros(B, dtype=i32, device=dev)))
        av.av_select(env.h, k, n, cum, live, children, rew, done, hashes, k, *outs[0])
        av.av_select_static(B, H, W, C, k, n, cum, live, children, rew, done, hashes, k,
                            *outs[1], visited, n_visited, cap, status)
        torch.cuda.synchronize()
        a = [to_np(x) for x in outs[0]]
        b = [to_np(x) for x in outs[1]]
        np.testing.assert_array_equal(a[4], b[4])  # frontier sizes
        assert a[4].sum() > 0, "the comparison must cover a non-empty frontier"
        for e in range(B):
            m = a[4][e]
            for x, y in zip(a[:4], b[:4]):
                np.testing.assert_array_equal(x[e, :m], y[e, :m])
            expected_visited[e] |= {int(h) for h in a[2][e, :m].view(np.uint64)}
        # the caller-owned visited sets hold exactly the root and every selected state
        nv = to_np(n_visited)
        vis = to_np(visited, "hash")
        for e in range(B):
            assert nv[e] == len(expected_visited[e])
            got = vis[e, : nv[e]]
            assert (np.diff(got.astype(object)) > 0).all()  # sorted, no repeats
            assert set(int(h) for h in got) == expected_visited[e]
        assert int(status.item()) == 0
        front, cum, hsh, live, n = outs[0]
    env.sync()
    env.close()


def test_select_static_rejects_sizes_beyond_its_array():
    import paper_2407_04221_gb300 as av
    dev = torch.device("cuda")
    one = torch.zeros(1, dtype=torch.int32, device=dev)
    cap = av.AV_SELECT_STATIC_MAX_HASHES  # 2 * 1 * cap > the array
    with pytest.raises(av.AvError) as ei:
        av.av_select_static(1, 4, 4, 4, 1, one, one, one, one, one, one, one, 1, one, one, one,
                            one, one, one, one, cap)
    assert ei.value.status == av.AV_EINVAL


def _maze(C, B, cap):
    """A handle on the base maze game (move and eat rules) with C tile
    channels, and B open 16 x 16 boards with a player and a food tile."""
    import paper_2407_04221_gb300 as av
    import workload as wk
    rules = wk.base_game_rules(C)[None]
    fields = dict(batch=B, H=16, W=16, C=C, n_rules=rules.shape[1], rules_per_env=0, max_steps=0,
                  auto_reset=0, ch_player=2, ch_goal=3, ch_empty=0, ch_wall=1, border_wall=0,
                  cum_per_env=0)
    env = av.Env(fields, rules, search_capacity=cap)
    dt = np.uint8 if C <= 8 else np.uint16
    g = np.full((B, 16, 16), 1, dt)
    g[:, 0, :] = g[:, -1, :] = g[:, :, 0] = g[:, :, -1] = 2
    for e in range(B):
        g[e, 3 + e, 4] |= 4
        g[e, 10, 11 - e] = 8
    return env, to_dev(g)


def _first_select(env, roots, B, k, cap, n_visited_init=None):
    """One expansion of the roots, then av_select_static on it; returns the
    static call's outputs, the visited arrays before and after, and status."""
    import paper_2407_04221_gb300 as av
    dev, i32, u8, i64 = env.device, torch.int32, torch.uint8, torch.int64
    root_hash = torch.zeros(B, dtype=i64, device=dev)
    root_live = torch.zeros(B, dtype=u8, device=dev)
    av.av_search_init(env.h, roots, root_hash, root_live)
    visited = torch.zeros(B, cap, dtype=i64, device=dev)
    visited[:, 0] = root_hash
    visited[:, 1:] = torch.arange(1, cap, dtype=i64, device=dev) * 7919  # a tail the call must keep
    n_visited = torch.ones(B, dtype=i32, device=dev) if n_visited_init is None else n_visited_init
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    front = env.boards(B, k)
    front[:, 0] = roots
    cum = torch.zeros(B, k, dtype=i32, device=dev)
    live = torch.zeros(B, k, dtype=u8, device=dev)
    live[:, 0] = root_live
    n = torch.ones(B, dtype=i32, device=dev)
    children, rew, done, hashes = env.expand(front, n)
    out = (env.boards(B, k), torch.zeros(B, k, dtype=i32, device=dev), torch.zeros(B, k, dtype=i64, device=dev),
           torch.zeros(B, k, dtype=u8, device=dev), torch.zeros(B, dtype=i32, device=dev))
    before = (to_np(visited, "hash").copy(), to_np(n_visited).copy())
    av.av_select_static(B, 16, 16, env.C, k, n, cum, live, children, rew, done, hashes, k, *out,
                        visited, n_visited, cap, status)
    torch.cuda.synchronize()
    return out, before, (to_np(visited, "hash"), to_np(n_visited)), int(status.item())


def test_select_static_two_byte_cells_matches_select():
    """C = 10 (two-byte cells), one call, against av_select on the same
    expansion; the caller's unused tail entries stay as they were."""
    import paper_2407_04221_gb300 as av
    B, k, cap = 4, 16, 40
    env, roots = _maze(10, B, cap)
    out, before, after, status = _first_select(env, roots, B, k, cap)
    # av_select on a second handle from the same roots
    env2, _ = _maze(10, B, cap)
    dev, i32, u8, i64 = env2.device, torch.int32, torch.uint8, torch.int64
    rh = torch.zeros(B, dtype=i64, device=dev)
    rl = torch.zeros(B, dtype=u8, device=dev)
    av.av_search_init(env2.h, roots, rh, rl)
    front = env2.boards(B, k)
    front[:, 0] = roots
    cum = torch.zeros(B, k, dtype=i32, device=dev)
    live = torch.zeros(B, k, dtype=u8, device=dev)
    live[:, 0] = rl
    n = torch.ones(B, dtype=i32, device=dev)
    children, rew, done, hashes = env2.expand(front, n)
    ref = (env2.boards(B, k), torch.zeros(B, k, dtype=i32, device=dev), torch.zeros(B, k, dtype=i64, device=dev),
           torch.zeros(B, k, dtype=u8, device=dev), torch.zeros(B, dtype=i32, device=dev))
    av.av_select(env2.h, k, n, cum, live, children, rew, done, hashes, k, *ref)
    torch.cuda.synchronize()
    a, b = [to_np(x) for x in ref], [to_np(x) for x in out]
    np.testing.assert_array_equal(a[4], b[4])
    assert a[4].sum() > 0
    for e in range(B):
        m = a[4][e]
        for x, y in zip(a[:4], b[:4]):
            np.testing.assert_array_equal(x[e, :m], y[e, :m])
    vis, nv = after
    for e in range(B):
        assert nv[e] == 1 + a[4][e]
        np.testing.assert_array_equal(vis[e, nv[e]:], before[0][e, nv[e]:])  # tail as given
    assert status == 0
    env.close()
    env2.close()


def test_select_static_overflow_leaves_sets_unchanged():
    """A capacity too small for the selection: status bit 0, and every
    visited set and count as given."""
    B, k, cap = 3, 8, 2
    env, roots = _maze(4, B, cap)
    out, before, after, status = _first_select(env, roots, B, k, cap)
    assert status & 1
    np.testing.assert_array_equal(after[0], before[0])
    np.testing.assert_array_equal(after[1], before[1])
    env.close()


def test_select_static_rejects_a_count_beyond_capacity():
    """n_visited[1] = capacity + 1 (a caller bug): status bit 1; that env
    selects nothing and keeps its set; the others select as usual."""
    B, k, cap = 3, 8, 30
    env, roots = _maze(4, B, cap)
    nv0 = torch.ones(B, dtype=torch.int32, device=env.device)
    nv0[1] = cap + 1
    out, before, after, status = _first_select(env, roots, B, k, cap, nv0)
    assert status & 2
    n_next = to_np(out[4])
    assert n_next[1] == 0 and n_next[0] > 0 and n_next[2] > 0
    assert (to_np(out[2])[1] == 0).all()
    np.testing.assert_array_equal(after[0][1], before[0][1])
    assert after[1][1] == cap + 1
    assert after[1][0] == 1 + n_next[0] and after[1][2] == 1 + n_next[2]
    env.close()
