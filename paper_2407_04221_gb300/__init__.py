"""Python binding of libautoverse.so (batched Autoverse rewrite-rule engine).

Argument marshalling only: every step of the path runs in the CUDA library.
torch is used for device memory and streams; tensors are passed by pointer.
The functions keep the C names (``av_create``, ``av_step`` ...); ``Env`` is a
small convenience wrapper that owns a handle.

If the library has not been built, importing works but every call raises
RuntimeError: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libautoverse.so")

AV_OK, AV_EINVAL, AV_ENOMEM, AV_ECUDA, AV_ESTATE, AV_EDEVICE = 0, -1, -2, -3, -4, -5
AV_WARN_ACTION = 1
AV_PATH_BLOCK, AV_PATH_FAST, AV_PATH_WARP = 1, 2, 3
RULE_BYTES = 408
EXPORTS = ("av_create", "av_destroy", "av_reset", "av_set_state", "av_get_state", "av_step",
           "av_rollout", "av_expand", "av_search_init", "av_select", "av_select_static", "av_sync",
           "av_warnings", "av_rollout_path", "av_step_path", "av_observe", "av_rule_obs", "av_mutate", "av_set_variant", "av_strerror",
           "av_last_error")
AV_MAX_WINDOW = 127
AV_MAX_LIMIT = 255
AV_PATH_VARIANT = 4
AV_PATH_BAND = 5
AV_PATH_MEMO = 6
AV_PATH_STEP = 7
AV_MAX_SMEM_CELLS = 4096
AV_SELECT_STATIC_MAX_HASHES = 1 << 21


class AvConfig(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("H", ctypes.c_int32), ("W", ctypes.c_int32),
                ("C", ctypes.c_int32), ("n_rules", ctypes.c_int32),
                ("rules_per_env", ctypes.c_int32), ("max_steps", ctypes.c_int32),
                ("auto_reset", ctypes.c_int32), ("ch_player", ctypes.c_int32),
                ("ch_goal", ctypes.c_int32), ("ch_empty", ctypes.c_int32),
                ("ch_wall", ctypes.c_int32), ("border_wall", ctypes.c_int32),
                ("cum_per_env", ctypes.c_int32), ("init_cum", ctypes.c_void_p),
                ("search_capacity", ctypes.c_int32)]


class AvVariant(ctypes.Structure):
    _fields_ = [("random_keys", ctypes.c_int32), ("_pad", ctypes.c_int32),
                ("key_seed", ctypes.c_uint64), ("limit", ctypes.c_int32 * 64),
                ("inhibit", ctypes.c_uint64 * 64)]


class AvMutation(ctypes.Structure):
    _fields_ = [("p_map", ctypes.c_uint32), ("map_channels", ctypes.c_uint32),
                ("p_rule", ctypes.c_uint32), ("p_reward", ctypes.c_uint32),
                ("reward_min", ctypes.c_int32), ("reward_max", ctypes.c_int32),
                ("mutable_rules", ctypes.c_uint64)]


class AvError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn} failed: status {status} ({msg})")
        self.status = status


_lib = None


def load() -> ctypes.CDLL:
    """Load the in-tree library; raise if it is missing (no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, u64, up = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64, ctypes.c_size_t
    sig = {
        "av_create": [ctypes.POINTER(AvConfig), vp, ctypes.POINTER(vp)],
        "av_destroy": [vp],
        "av_reset": [vp, u64, vp, up],
        "av_set_state": [vp, vp, vp, ctypes.c_int, up],
        "av_get_state": [vp, vp, vp, up],
        "av_step": [vp, vp, vp, vp, vp, up],
        "av_rollout": [vp, i32, u64, vp, vp, vp, vp, up],
        "av_expand": [vp, vp, i32, vp, vp, vp, vp, vp, up],
        "av_search_init": [vp, vp, vp, vp, up],
        "av_select": [vp, i32, vp, vp, vp, vp, vp, vp, vp, i32, vp, vp, vp, vp, vp, up],
        "av_select_static": [i32, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, i32, vp, vp, vp,
                             vp, vp, vp, vp, i32, vp, up],
        "av_sync": [vp],
        "av_warnings": [vp, ctypes.POINTER(ctypes.c_uint32)],
        "av_rollout_path": [vp, ctypes.POINTER(ctypes.c_int32)],
        "av_step_path": [vp, ctypes.POINTER(ctypes.c_int32)],
        "av_observe": [vp, vp, i32, vp, vp, up],
        "av_rule_obs": [vp, vp, vp, up],
        "av_mutate": [i32, i32, i32, i32, i32, ctypes.POINTER(AvMutation), u64, vp, vp, up],
        "av_set_variant": [vp, ctypes.POINTER(AvVariant)],
    }
    for name, args in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    L.av_strerror.argtypes = [ctypes.c_int]
    L.av_strerror.restype = ctypes.c_char_p
    L.av_last_error.argtypes = [vp]
    L.av_last_error.restype = ctypes.c_char_p
    _lib = L
    return L


def _ptr(x):
    """Device pointer of a torch tensor (or None / int passthrough)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not x.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(stream) if isinstance(stream, int) else stream.cuda_stream


def _check(h, fn, rc):
    if rc != AV_OK:
        L = load()
        msg = (L.av_last_error(h) or b"").decode() if h else ""
        raise AvError(fn, rc, msg or L.av_strerror(rc).decode())


def av_strerror(status: int) -> str:
    return load().av_strerror(status).decode()


def av_create(cfg: dict, rules, init_cum=None, search_capacity: int = 0):
    """cfg: the int fields of av_config; rules: buffer of packed 408-byte
    records ([B][R] or [R]); init_cum: uint32 array or None.  -> handle."""
    L = load()
    c = AvConfig()
    for name, _ in AvConfig._fields_:
        if name not in ("init_cum", "search_capacity"):
            setattr(c, name, int(cfg[name]))
    c.search_capacity = int(search_capacity)
    if isinstance(rules, (bytes, bytearray, memoryview)):
        rb = np.frombuffer(rules, dtype=np.uint8)
    else:
        a = np.ascontiguousarray(rules)
        rb = a.reshape(-1).view(np.uint8) if a.size else np.zeros(0, np.uint8)
    if rb.size % RULE_BYTES:
        raise ValueError("rules must be packed 408-byte records")
    cum = None
    if init_cum is not None:
        cum = np.ascontiguousarray(init_cum, dtype=np.uint32)
        c.init_cum = cum.ctypes.data
    h = ctypes.c_void_p()
    rc = L.av_create(ctypes.byref(c), rb.ctypes.data if rb.size else None, ctypes.byref(h))
    _check(None, "av_create", rc)
    return h


def av_destroy(h):
    _check(None, "av_destroy", load().av_destroy(h))


def av_reset(h, seed: int, obs=None, stream=None):
    _check(h, "av_reset", load().av_reset(h, int(seed) & (2**64 - 1), _ptr(obs), _stream(stream)))


def av_set_state(h, grids, t=None, set_as_init: bool = False, stream=None):
    _check(h, "av_set_state", load().av_set_state(h, _ptr(grids), _ptr(t), int(bool(set_as_init)),
                                                  _stream(stream)))


def av_get_state(h, grids, t=None, stream=None):
    _check(h, "av_get_state", load().av_get_state(h, _ptr(grids), _ptr(t), _stream(stream)))


def av_step(h, actions, obs=None, reward=None, done=None, stream=None):
    _check(h, "av_step", load().av_step(h, _ptr(actions), _ptr(obs), _ptr(reward), _ptr(done),
                                        _stream(stream)))


def av_rollout(h, n_steps: int, action_seed: int, obs_traj=None, rew_traj=None, done_traj=None,
               rew_sum=None, stream=None):
    _check(h, "av_rollout", load().av_rollout(h, int(n_steps), int(action_seed) & (2**64 - 1),
                                              _ptr(obs_traj), _ptr(rew_traj), _ptr(done_traj),
                                              _ptr(rew_sum), _stream(stream)))


def av_expand(h, parents, F: int, children, rewards, done, hashes, n_parent=None, stream=None):
    _check(h, "av_expand", load().av_expand(h, _ptr(parents), int(F), _ptr(n_parent),
                                            _ptr(children), _ptr(rewards), _ptr(done),
                                            _ptr(hashes), _stream(stream)))


def av_search_init(h, roots, root_hash, root_live, stream=None):
    _check(h, "av_search_init", load().av_search_init(h, _ptr(roots), _ptr(root_hash),
                                                      _ptr(root_live), _stream(stream)))


def av_select(h, F, n_parent, parent_cum, parent_live, cand_grids, cand_reward, cand_done,
              cand_hash, k, next_grids, next_cum, next_hash, next_live, n_next, stream=None):
    rc = load().av_select(h, int(F), _ptr(n_parent), _ptr(parent_cum), _ptr(parent_live),
                          _ptr(cand_grids), _ptr(cand_reward), _ptr(cand_done), _ptr(cand_hash),
                          int(k), _ptr(next_grids), _ptr(next_cum), _ptr(next_hash),
                          _ptr(next_live), _ptr(n_next), _stream(stream))
    _check(h, "av_select", rc)


def av_select_static(batch, H, W, C, F, n_parent, parent_cum, parent_live, cand_grids,
                     cand_reward, cand_done, cand_hash, k, next_grids, next_cum, next_hash,
                     next_live, n_next, visited, n_visited, capacity, status=None, stream=None):
    """av_select without a handle or any device allocation: the caller owns
    the visited sets (visited [batch, capacity] uint64, n_visited [batch]);
    the library's fixed working array holds the merge.  See the C header for
    the size limit and for why overlapping calls must be serialised."""
    rc = load().av_select_static(int(batch), int(H), int(W), int(C), int(F), _ptr(n_parent),
                                 _ptr(parent_cum), _ptr(parent_live), _ptr(cand_grids),
                                 _ptr(cand_reward), _ptr(cand_done), _ptr(cand_hash), int(k),
                                 _ptr(next_grids), _ptr(next_cum), _ptr(next_hash), _ptr(next_live),
                                 _ptr(n_next), _ptr(visited), _ptr(n_visited), int(capacity),
                                 _ptr(status), _stream(stream))
    _check(None, "av_select_static", rc)


def av_sync(h):
    _check(h, "av_sync", load().av_sync(h))


def av_warnings(h) -> int:
    bits = ctypes.c_uint32()
    _check(h, "av_warnings", load().av_warnings(h, ctypes.byref(bits)))
    return int(bits.value)


def av_rollout_path(h) -> int:
    path = ctypes.c_int32()
    _check(h, "av_rollout_path", load().av_rollout_path(h, ctypes.byref(path)))
    return int(path.value)


def av_step_path(h) -> int:
    path = ctypes.c_int32()
    _check(h, "av_step_path", load().av_step_path(h, ctypes.byref(path)))
    return int(path.value)


def av_observe(h, grids, window: int, obs, player_yx=None, stream=None):
    """Player-centred patches (Sec. 3.2): obs [B, window, window, C] uint8;
    grids None observes the handle's current boards."""
    _check(h, "av_observe", load().av_observe(h, _ptr(grids), int(window), _ptr(obs),
                                              _ptr(player_yx), _stream(stream)))


def av_rule_obs(h, bits, reward=None, stream=None):
    """Binary form of the rule tables: bits [T, R, 4, 5, 5, C+1] uint8, reward [T, R]."""
    _check(h, "av_rule_obs", load().av_rule_obs(h, _ptr(bits), _ptr(reward), _stream(stream)))


def av_set_variant(h, random_keys=0, key_seed=0, limit=None, inhibit=None, clear=False):
    """Variant semantics for av_step / av_rollout (Sec. 2.1, possible
    extensions): limit[r] applications per step by largest key (ordered or
    random index channel), inhibit[r] = mask of rules a match of r suppresses.
    clear=True restores the standard step."""
    L = load()
    if clear:
        _check(h, "av_set_variant", L.av_set_variant(h, None))
        return
    v = AvVariant()
    v.random_keys = int(random_keys)
    v.key_seed = int(key_seed) & (2**64 - 1)
    for r, k in enumerate(limit or []):
        v.limit[r] = int(k)
    for r, m in enumerate(inhibit or []):
        v.inhibit[r] = int(m)
    _check(h, "av_set_variant", L.av_set_variant(h, ctypes.byref(v)))


def av_mutate(batch, H, W, C, n_rules, mutation: dict, seed: int, maps=None, rules=None,
              stream=None):
    """Mutation operators (Sec. 3.1.1), in place on device tensors: maps
    [batch, H, W] cell words, rules [batch, n_rules, 408] uint8 packed records
    (either may be None).  mutation: p_map, map_channels, p_rule, p_reward
    (rates x 2^24), reward_min, reward_max, mutable_rules (bit mask)."""
    m = AvMutation(**{k: int(mutation[k]) for k, _ in AvMutation._fields_})
    rc = load().av_mutate(int(batch), int(H), int(W), int(C), int(n_rules), ctypes.byref(m),
                          int(seed) & (2**64 - 1), _ptr(maps), _ptr(rules), _stream(stream))
    _check(None, "av_mutate", rc)


class Env:
    """Owns one handle; allocates output tensors on demand (torch, cuda)."""

    def __init__(self, cfg: dict, rules, init_cum=None, search_capacity: int = 0, device=None):
        import torch
        self.cfg = dict(cfg)
        self.B, self.H, self.W, self.C = (int(cfg[k]) for k in ("batch", "H", "W", "C"))
        self.device = torch.device(device or "cuda")
        self.cell_dtype = torch.uint8 if self.C <= 8 else torch.int16
        self.h = av_create(cfg, rules, init_cum, search_capacity)

    def close(self):
        if self.h is not None:
            av_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def boards(self, *lead):
        import torch
        return torch.zeros(*lead, self.H, self.W, dtype=self.cell_dtype, device=self.device)

    def reset(self, seed: int, stream=None):
        obs = self.boards(self.B)
        av_reset(self.h, seed, obs, stream)
        return obs

    def get_state(self, stream=None):
        import torch
        g = self.boards(self.B)
        t = torch.zeros(self.B, dtype=torch.int32, device=self.device)
        av_get_state(self.h, g, t, stream)
        return g, t

    def set_state(self, grids, t=None, set_as_init=False, stream=None):
        av_set_state(self.h, grids, t, set_as_init, stream)

    def step(self, actions, stream=None):
        import torch
        obs = self.boards(self.B)
        rew = torch.zeros(self.B, dtype=torch.int32, device=self.device)
        done = torch.zeros(self.B, dtype=torch.uint8, device=self.device)
        av_step(self.h, actions, obs, rew, done, stream)
        return obs, rew, done

    def rollout(self, n_steps: int, action_seed: int, trajectory: bool = False, stream=None):
        import torch
        rew_sum = torch.zeros(self.B, dtype=torch.int32, device=self.device)
        obs = rew = done = None
        if trajectory:
            obs = self.boards(n_steps, self.B)
            rew = torch.zeros(n_steps, self.B, dtype=torch.int32, device=self.device)
            done = torch.zeros(n_steps, self.B, dtype=torch.uint8, device=self.device)
        av_rollout(self.h, n_steps, action_seed, obs, rew, done, rew_sum, stream)
        return dict(rew_sum=rew_sum, obs=obs, rew=rew, done=done)

    def expand(self, parents, n_parent=None, stream=None):
        import torch
        F = parents.shape[1]
        children = self.boards(self.B, F, 5)
        rew = torch.zeros(self.B, F, 5, dtype=torch.int32, device=self.device)
        done = torch.zeros(self.B, F, 5, dtype=torch.uint8, device=self.device)
        hashes = torch.zeros(self.B, F, 5, dtype=torch.int64, device=self.device)
        av_expand(self.h, parents, F, children, rew, done, hashes, n_parent, stream)
        return children, rew, done, hashes

    def search(self, roots, iterations: int, k: int, stream=None):
        """Greedy best-first beam search (Sec. 2.2.1) from roots [B,H,W]:
        `iterations` rounds of av_expand + av_select, frontier kept on the
        device.  The handle needs search_capacity >= 1 + iterations * k.
        Returns the final frontier and per-iteration frontier size / best
        cumulative reward (INT32_MIN when empty)."""
        import torch
        dev, B = self.device, self.B
        i32, u8 = torch.int32, torch.uint8
        front = self.boards(B, k)
        nxt = self.boards(B, k)
        cum = torch.zeros(B, k, dtype=i32, device=dev)
        ncum = torch.zeros_like(cum)
        hsh = torch.zeros(B, k, dtype=torch.int64, device=dev)
        nhsh = torch.zeros_like(hsh)
        live = torch.zeros(B, k, dtype=u8, device=dev)
        nlive = torch.zeros_like(live)
        n = torch.ones(B, dtype=i32, device=dev)
        nn = torch.zeros_like(n)
        front[:, 0].copy_(roots)
        root_hash = torch.zeros(B, dtype=torch.int64, device=dev)
        root_live = torch.zeros(B, dtype=u8, device=dev)
        av_search_init(self.h, roots, root_hash, root_live, stream)
        hsh[:, 0].copy_(root_hash)
        live[:, 0].copy_(root_live)
        children = self.boards(B, k, 5)
        rew = torch.zeros(B, k, 5, dtype=i32, device=dev)
        done = torch.zeros(B, k, 5, dtype=u8, device=dev)
        chash = torch.zeros(B, k, 5, dtype=torch.int64, device=dev)
        trace_n = torch.zeros(B, iterations, dtype=i32, device=dev)
        trace_best = torch.zeros(B, iterations, dtype=i32, device=dev)
        for it in range(iterations):
            av_expand(self.h, front, k, children, rew, done, chash, n, stream)
            av_select(self.h, k, n, cum, live, children, rew, done, chash, k, nxt, ncum, nhsh,
                      nlive, nn, stream)
            front, nxt = nxt, front
            cum, ncum = ncum, cum
            hsh, nhsh = nhsh, hsh
            live, nlive = nlive, live
            n, nn = nn, n
            trace_n[:, it].copy_(n)
            trace_best[:, it].copy_(cum[:, 0])
        return dict(grids=front, cum=cum, hash=hsh, live=live, n=n, trace_n=trace_n,
                    trace_best=trace_best)

    def observe(self, window: int, grids=None, stream=None):
        """Player-centred patches of the current boards (or of `grids`
        [B, H, W]) -> (obs [B, window, window, C] uint8, player_yx [B, 2])."""
        import torch
        obs = torch.empty(self.B, window, window, self.C, dtype=torch.uint8, device=self.device)
        pyx = torch.empty(self.B, 2, dtype=torch.int32, device=self.device)
        av_observe(self.h, grids, window, obs, pyx, stream)
        return obs, pyx

    def rule_obs(self, stream=None):
        """-> (bits [T, R, 4, 5, 5, C+1] uint8, reward [T, R] int32), T = B
        with per-env rules, else 1."""
        import torch
        T = self.B if int(self.cfg["rules_per_env"]) else 1
        R = int(self.cfg["n_rules"])
        bits = torch.empty(T, R, 4, 5, 5, self.C + 1, dtype=torch.uint8, device=self.device)
        rew = torch.empty(T, R, dtype=torch.int32, device=self.device)
        av_rule_obs(self.h, bits, rew, stream)
        return bits, rew

    def sync(self):
        av_sync(self.h)
