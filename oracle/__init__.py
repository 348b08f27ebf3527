"""ctypes loader for the CPU oracle (``oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by the tests, by ``__graft_entry__.smoke``
and by the benchmark's CPU-baseline / reference leg.  The product path (the
CUDA library and its Python binding) never imports this package.

Grids crossing this boundary are canonical numpy arrays ``[..., H, W]`` of
cell words (uint8 when C <= 8, else uint16, tile bits only).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None

FIELDS = ("batch", "H", "W", "C", "n_rules", "rules_per_env", "max_steps", "auto_reset",
          "ch_player", "ch_goal", "ch_empty", "ch_wall", "border_wall", "cum_per_env")


class OrVariant(ctypes.Structure):
    _fields_ = [("random_keys", ctypes.c_int32), ("_pad", ctypes.c_int32),
                ("key_seed", ctypes.c_uint64), ("limit", ctypes.c_int32 * 64),
                ("inhibit", ctypes.c_uint64 * 64)]


def make_variant(random_keys=0, key_seed=0, limit=None, inhibit=None) -> OrVariant:
    """Variant semantics: limit[r] matches per step (0 = all) chosen by
    largest key, inhibit[r] = bit mask of the rules a match of r suppresses."""
    v = OrVariant()
    v.random_keys = int(random_keys)
    v.key_seed = int(key_seed) & (2**64 - 1)
    for r, k in enumerate(limit or []):
        v.limit[r] = int(k)
    for r, m in enumerate(inhibit or []):
        v.inhibit[r] = int(m)
    return v


class OrMutation(ctypes.Structure):
    _fields_ = [("p_map", ctypes.c_uint32), ("map_channels", ctypes.c_uint32),
                ("p_rule", ctypes.c_uint32), ("p_reward", ctypes.c_uint32),
                ("reward_min", ctypes.c_int32), ("reward_max", ctypes.c_int32),
                ("mutable_rules", ctypes.c_uint64)]


class OrCfg(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int32) for f in FIELDS]


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so next to it (plain gcc, -O2)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-Wall", "-shared", "-fPIC", "-pthread",
                               _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        u64, i32, vp = ctypes.c_uint64, ctypes.c_int32, ctypes.c_void_p
        L.or_mix64.restype = u64
        L.or_mix64.argtypes = [u64]
        L.or_draw.restype = u64
        L.or_draw.argtypes = [u64, u64, u64, u64, u64]
        L.or_fnv1a64.restype = u64
        L.or_fnv1a64.argtypes = [vp, ctypes.c_int64]
        L.or_grid_hash.restype = u64
        L.or_grid_hash.argtypes = [vp, i32, i32, i32]
        L.or_rotate.restype = None
        L.or_rotate.argtypes = [vp, i32, vp, vp, vp, vp, vp]
        L.or_reset.restype = i32
        L.or_reset.argtypes = [vp, vp, u64, i32, vp]
        L.or_step_batch.restype = i32
        L.or_step_batch.argtypes = [vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, i32]
        L.or_rollout.restype = i32
        L.or_rollout.argtypes = [vp, vp, i32, vp, vp, vp, vp, i32, u64, vp, vp, vp, vp, i32]
        L.or_expand.restype = i32
        L.or_expand.argtypes = [vp, vp, i32, vp, vp, i32, vp, vp, vp, vp, i32]
        L.or_search.restype = i32
        L.or_search.argtypes = [vp, vp, i32, vp, vp, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, i32]
        L.or_observe.restype = i32
        L.or_observe.argtypes = [vp, i32, vp, i32, vp, vp]
        L.or_rule_obs.restype = i32
        L.or_rule_obs.argtypes = [vp, vp, i32, vp, vp]
        L.or_step_batch_v.restype = i32
        L.or_step_batch_v.argtypes = [vp, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, i32]
        L.or_rollout_v.restype = i32
        L.or_rollout_v.argtypes = [vp, vp, vp, i32, vp, vp, vp, vp, i32, u64, vp, vp, vp, vp, i32]
        L.or_mutate.restype = i32
        L.or_mutate.argtypes = [i32, vp, i32, i32, i32, i32, vp, u64, vp, vp]
        _lib = L
    return _lib


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def make_cfg(**fields) -> OrCfg:
    return OrCfg(*[int(fields[f]) for f in FIELDS])


def cell_dtype(C: int):
    return np.uint8 if C <= 8 else np.uint16


def _rules_buf(rules: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(rules).view(np.uint8).reshape(-1)


def _ids(env_ids, n):
    if env_ids is None:
        return None
    a = np.ascontiguousarray(env_ids, dtype=np.int32)
    assert a.shape == (n,)
    return a


def draw(seed, stream, a, b, c) -> int:
    return int(lib().or_draw(seed, stream, a, b, c))


def fnv1a64(data: bytes) -> int:
    buf = np.frombuffer(data, dtype=np.uint8) if data else np.zeros(1, np.uint8)
    return int(lib().or_fnv1a64(_p(buf), len(data)))


def grid_hash(grid: np.ndarray, C: int) -> int:
    g = np.ascontiguousarray(grid, dtype=cell_dtype(C))
    H, W = g.shape
    return int(lib().or_grid_hash(_p(g), H, W, C))


def rotate(rule_record: np.ndarray, j: int):
    """Rotation j (CCW quarter turns) of one packed record -> (h, w, P, A, S, Cl)."""
    rec = np.ascontiguousarray(rule_record).view(np.uint8).reshape(-1)
    hw = np.zeros(2, np.int32)
    arrs = [np.zeros(25, np.uint32) for _ in range(4)]
    lib().or_rotate(_p(rec), j, _p(hw), *[_p(a) for a in arrs])
    h, w = int(hw[0]), int(hw[1])
    return (h, w) + tuple(a[: h * w].reshape(h, w) for a in arrs)


def reset(cfg: OrCfg, cum: np.ndarray, seed: int, envs) -> np.ndarray:
    envs = list(envs)
    cum = np.ascontiguousarray(cum, dtype=np.uint32)
    out = np.zeros((len(envs), cfg.H, cfg.W), dtype=cell_dtype(cfg.C))
    L = lib()
    for i, e in enumerate(envs):
        rc = L.or_reset(ctypes.byref(cfg), _p(cum), seed, int(e), _p(out[i]))
        assert rc == 0
    return out


def step(cfg: OrCfg, rules, grids, inits, t, actions, env_ids=None, threads=None, variant=None):
    """One step of n envs -> (grids, t, rewards, dones); variant: OrVariant or None."""
    grids = np.ascontiguousarray(grids, dtype=cell_dtype(cfg.C))
    n = grids.shape[0]
    inits = np.ascontiguousarray(inits, dtype=cell_dtype(cfg.C))
    t = np.ascontiguousarray(t, dtype=np.int32)
    actions = np.ascontiguousarray(actions, dtype=np.uint8)
    out = np.zeros_like(grids)
    t_out = np.zeros(n, np.int32)
    rew = np.zeros(n, np.int32)
    done = np.zeros(n, np.uint8)
    rb = _rules_buf(rules)
    ids = _ids(env_ids, n)
    rc = lib().or_step_batch_v(ctypes.byref(cfg), _p(rb), None if variant is None else ctypes.byref(variant),
                               n, _p(ids), _p(grids), _p(inits), _p(t), _p(actions), _p(out),
                               _p(t_out), _p(rew), _p(done), threads or default_threads())
    assert rc == 0, rc
    return out, t_out, rew, done


def rollout(cfg: OrCfg, rules, grids, inits, t, n_steps, action_seed, env_ids=None,
            trajectory=False, threads=None, variant=None):
    """Fused rollout -> dict(grids, t, rew_sum[, obs, rew, done])."""
    grids = np.array(grids, dtype=cell_dtype(cfg.C), copy=True, order="C")
    n = grids.shape[0]
    inits = np.ascontiguousarray(inits, dtype=cell_dtype(cfg.C))
    t = np.array(t, dtype=np.int32, copy=True)
    rew_sum = np.zeros(n, np.int32)
    obs = rew = done = None
    if trajectory:
        obs = np.zeros((n_steps,) + grids.shape, dtype=grids.dtype)
        rew = np.zeros((n_steps, n), np.int32)
        done = np.zeros((n_steps, n), np.uint8)
    rb = _rules_buf(rules)
    ids = _ids(env_ids, n)
    rc = lib().or_rollout_v(ctypes.byref(cfg), _p(rb), None if variant is None else ctypes.byref(variant),
                            n, _p(ids), _p(grids), _p(inits), _p(t), int(n_steps), int(action_seed),
                            _p(obs), _p(rew), _p(done), _p(rew_sum), threads or default_threads())
    assert rc == 0, rc
    res = dict(grids=grids, t=t, rew_sum=rew_sum)
    if trajectory:
        res.update(obs=obs, rew=rew, done=done)
    return res


def expand(cfg: OrCfg, rules, parents, env_ids=None, threads=None):
    """parents [n, F, H, W] -> (children [n,F,5,H,W], rewards, done, hashes)."""
    parents = np.ascontiguousarray(parents, dtype=cell_dtype(cfg.C))
    n, F = parents.shape[:2]
    children = np.zeros((n, F, 5, cfg.H, cfg.W), dtype=parents.dtype)
    rew = np.zeros((n, F, 5), np.int32)
    done = np.zeros((n, F, 5), np.uint8)
    hashes = np.zeros((n, F, 5), np.uint64)
    rb = _rules_buf(rules)
    rc = lib().or_expand(ctypes.byref(cfg), _p(rb), n, _p(_ids(env_ids, n)), _p(parents), F,
                         _p(children), _p(rew), _p(done), _p(hashes), threads or default_threads())
    assert rc == 0, rc
    return children, rew, done, hashes


def search(cfg: OrCfg, rules, roots, iterations, k, env_ids=None, threads=None):
    """Greedy best-first beam search from roots [n, H, W]."""
    roots = np.ascontiguousarray(roots, dtype=cell_dtype(cfg.C))
    n = roots.shape[0]
    fg = np.zeros((n, k, cfg.H, cfg.W), dtype=roots.dtype)
    fc = np.zeros((n, k), np.int32)
    fh = np.zeros((n, k), np.uint64)
    fd = np.zeros((n, k), np.uint8)
    nf = np.zeros(n, np.int32)
    tn = np.zeros((n, max(iterations, 1)), np.int32)
    tb = np.zeros((n, max(iterations, 1)), np.int32)
    nv = np.zeros(n, np.int32)
    rb = _rules_buf(rules)
    rc = lib().or_search(ctypes.byref(cfg), _p(rb), n, _p(_ids(env_ids, n)), _p(roots),
                         int(iterations), int(k), _p(fg), _p(fc), _p(fh), _p(fd), _p(nf), _p(tn),
                         _p(tb), _p(nv), threads or default_threads())
    assert rc == 0, rc
    return dict(grids=fg, cum=fc, hash=fh, done=fd, n=nf, trace_n=tn[:, :iterations],
                trace_best=tb[:, :iterations], n_visited=nv)


def observe(cfg: OrCfg, grids, window: int):
    """Player-centred patches of boards [n, H, W] -> (obs [n, window, window, C] uint8,
    player_yx [n, 2] int32, (-1, -1) where no player is on the board)."""
    grids = np.ascontiguousarray(grids, dtype=cell_dtype(cfg.C))
    n = grids.shape[0]
    obs = np.zeros((n, window, window, cfg.C), np.uint8)
    pyx = np.zeros((n, 2), np.int32)
    rc = lib().or_observe(ctypes.byref(cfg), n, _p(grids), int(window), _p(obs), _p(pyx))
    assert rc == 0, rc
    return obs, pyx


def rule_obs(cfg: OrCfg, rules):
    """Binary form of rule tables [T, R] records -> (bits [T, R, 4, 5, 5, C+1] uint8,
    reward [T, R] int32)."""
    rb = _rules_buf(rules)
    T = rb.size // (408 * max(cfg.n_rules, 1)) if cfg.n_rules else 0
    bits = np.zeros((T, cfg.n_rules, 4, 5, 5, cfg.C + 1), np.uint8)
    rew = np.zeros((T, cfg.n_rules), np.int32)
    rc = lib().or_rule_obs(ctypes.byref(cfg), _p(rb), T, _p(bits), _p(rew))
    assert rc == 0, rc
    return bits, rew


def mutate(H: int, W: int, C: int, mutation: dict, seed: int, maps=None, rules=None,
           env_ids=None):
    """Mutation operators of the evolution loop: returns mutated copies of
    maps [n, H, W] and rule tables [n, R] (either may be None).  mutation:
    p_map, map_channels, p_rule, p_reward (24-bit thresholds), reward_min,
    reward_max, mutable_rules (bit mask over rule slots)."""
    m = OrMutation(**{k: int(mutation[k]) for k, _ in OrMutation._fields_})
    n = maps.shape[0] if maps is not None else rules.shape[0]
    mp = None if maps is None else np.array(maps, dtype=cell_dtype(C), copy=True, order="C")
    rl = None if rules is None else np.array(rules, copy=True, order="C")
    R = 0 if rl is None else rl.shape[1]
    rb = None if rl is None else rl.view(np.uint8).reshape(-1)
    rc = lib().or_mutate(n, _p(_ids(env_ids, n)), H, W, C, R, ctypes.byref(m), int(seed) & (2**64 - 1),
                         _p(mp), _p(rb))
    assert rc == 0, rc
    return mp, rl
