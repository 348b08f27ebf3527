"""Seeded synthetic inputs for the Autoverse batched step.

This module produces the *inputs* shared by the CUDA library and by the CPU
oracle: the packed rewrite-rule tables and the initial-map type thresholds of
the five benchmark workloads.  It holds none of the step's arithmetic (no
matching, no rotation, no rule application, no hashing).

Everything is integer-only and counter-based, so that any platform regenerates
the same bytes from the same seed.  The generator is SplitMix64's output
finaliser (Vigna, ``splitmix64.c``, public domain: xor-shift 30, multiply by
0xbf58476d1ce4e5b9, xor-shift 27, multiply by 0x94d049bb133111eb, xor-shift
31), keyed as

    draw(seed, stream, a, b, c) =
        mix(mix(mix(seed + 0x9E3779B97F4A7C15 * (stream + 1)) ^ a) ^ (b << 32 | c))

Streams used here: 3 (Dirichlet type thresholds), 5 (pattern size), 6 (input
pattern entries), 7 (output pattern entries), 8 (reward).  Streams 1, 2 and 4
(initial cells, player cell, actions) are drawn by the library and the oracle
themselves, each from its own implementation of the same definition.

Rule semantics follow the paper's rewrite rules (Sec. 2.1, Fig. 2a): an input
pattern I over the c tile channels of an n x m patch, an output pattern O and a
reward.  Input entries are ternary per (position, channel) -- present, absent
or don't-care -- and span the tile channels plus the transient "force"
channel (index C) through which a player action enters the grid (Sec. 2.1).
Output entries are set / clear / unchanged per (position, tile channel).
"""
from __future__ import annotations

import dataclasses

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15
ONE24 = 1 << 24

#: Packed rule record: 408 bytes, little-endian.  Bit ``c`` of each mask word
#: refers to tile channel ``c`` (c < C); bit C is the force channel.  Entry
#: (i, k) of an h x w pattern sits at index i * w + k.
RULE_DTYPE = np.dtype(
    [
        ("h", "<u1"),
        ("w", "<u1"),
        ("pad", "<u1", (2,)),
        ("reward", "<i4"),
        ("present", "<u4", (25,)),
        ("absent", "<u4", (25,)),
        ("set", "<u4", (25,)),
        ("clear", "<u4", (25,)),
    ]
)
assert RULE_DTYPE.itemsize == 408

# Role channels of the base maze game (Sec. 2.2.1): empty floor, wall, player,
# goal ("food").  Further channels are extra tile types.
CH_EMPTY, CH_WALL, CH_PLAYER, CH_GOAL = 0, 1, 2, 3


def thr24(p: float) -> int:
    """Probability -> 24-bit integer threshold (round half up)."""
    return int(p * ONE24 + 0.5)


# --------------------------------------------------------------------------
# counter-based generator
# --------------------------------------------------------------------------
_C1 = np.uint64(0xBF58476D1CE4E5B9)
_C2 = np.uint64(0x94D049BB133111EB)


def _mix(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _C1
        z = (z ^ (z >> np.uint64(27))) * _C2
    return z ^ (z >> np.uint64(31))


def draw(seed: int, stream: int, a, b, c) -> np.ndarray:
    """Vectorised counter draw; a, b, c broadcast as unsigned 64-bit."""
    base = np.uint64((seed + GOLDEN * (stream + 1)) & MASK64)
    a = np.asarray(a, dtype=np.uint64)
    b = np.asarray(b, dtype=np.uint64)
    c = np.asarray(c, dtype=np.uint64)
    z = _mix(np.asarray(base, dtype=np.uint64))
    z = _mix(z ^ a)
    return _mix(z ^ ((b << np.uint64(32)) | c))


def uniform_int(d: np.ndarray, n: int) -> np.ndarray:
    """Uniform integer in [0, n) from a 64-bit draw: ((d >> 32) * n) >> 32."""
    return ((d >> np.uint64(32)) * np.uint64(n)) >> np.uint64(32)


def u24(d: np.ndarray) -> np.ndarray:
    return (d >> np.uint64(40)).astype(np.int64)


# --------------------------------------------------------------------------
# workload definitions
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload: sizes, rule distribution and run length."""

    key: int
    name: str
    batch: int
    H: int
    W: int
    C: int
    n_rules: int
    shapes: tuple  # base (h, w) pattern sizes, chosen uniformly per rule
    p_present: float
    p_absent: float
    p_set: float
    p_clear: float
    reward_lo: int
    reward_hi: int
    steps: int = 0  # fused steps per rollout launch
    max_steps: int = 0
    auto_reset: int = 0
    rules_per_env: int = 1
    border_wall: int = 1
    init: str = "dirichlet"  # or "maze": fixed empty/wall/goal mix
    trajectory: bool = False  # rollout also writes obs/reward/done per step
    frontier: int = 0  # search: nodes kept per env (top-k)
    iterations: int = 0  # search: expand+select iterations
    base_game: bool = False  # rules 0 and 1 of every table: the maze game's move and eat

    @property
    def nch(self) -> int:
        return self.C + 1

    @property
    def cell_bytes(self) -> int:
        return 1 if self.C <= 8 else 2

    def scaled(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    1: Workload(1, "maze16-b1-c4-r3", 1, 16, 16, 4, 3, ((3, 3),), 0.15, 0.15, 0.1, 0.1,
                -3, 3, steps=100, rules_per_env=0, init="maze"),
    2: Workload(2, "grid16-b1024-c8-r8", 1024, 16, 16, 8, 8, ((3, 3),), 0.15, 0.15, 0.1,
                0.1, -3, 3, steps=1000),
    3: Workload(3, "grid16-b16384-c10-r12-traj", 16384, 16, 16, 10, 12,
                ((1, 2), (1, 3), (3, 3)), 0.15, 0.15, 0.1, 0.1, -3, 3, steps=2000,
                max_steps=200, auto_reset=1, trajectory=True),
    4: Workload(4, "search16-b64-f256-c8-r8", 64, 16, 16, 8, 8, ((3, 3),), 0.15, 0.15,
                0.1, 0.1, -3, 3, init="maze", frontier=256, iterations=50, base_game=True),
    5: Workload(5, "grid64-b4096-c16-r24", 4096, 64, 64, 16, 24, ((3, 3), (5, 5)), 0.1,
                0.1, 0.1, 0.1, -5, 5, steps=500),
    # boards larger than one CTA's shared memory (the band-streamed rollout)
    6: Workload(6, "grid256-b256-c16-r24", 256, 256, 256, 16, 24, ((3, 3), (5, 5)), 0.1,
                0.1, 0.1, 0.1, -5, 5, steps=50),
}


def seeds(seed: int) -> dict:
    """Seed convention: s -> rules and thresholds, s+100 -> reset, s+200 -> actions."""
    return {"rules": seed, "reset": seed + 100, "actions": seed + 200}


# --------------------------------------------------------------------------
# generators
# --------------------------------------------------------------------------
def make_rules(wl: Workload, seed: int, env_chunk: int = 2048) -> np.ndarray:
    """Rule tables, shape [n_tables, R] of RULE_DTYPE (n_tables = B or 1)."""
    n_tab = wl.batch if wl.rules_per_env else 1
    R, NCH, C = wl.n_rules, wl.nch, wl.C
    out = np.zeros((n_tab, R), dtype=RULE_DTYPE)
    tp, ta = thr24(wl.p_present), thr24(wl.p_present + wl.p_absent)
    ts, tc = thr24(wl.p_set), thr24(wl.p_set + wl.p_clear)
    span = wl.reward_hi - wl.reward_lo + 1
    pos = np.arange(25, dtype=np.uint64)
    for e0 in range(0, n_tab, env_chunk):
        e1 = min(n_tab, e0 + env_chunk)
        env = np.arange(e0, e1, dtype=np.uint64)[:, None]
        rr = np.arange(R, dtype=np.uint64)[None, :]
        shape_idx = uniform_int(draw(seed, 5, env, rr, 0), len(wl.shapes)).astype(np.int64)
        hs = np.array([s[0] for s in wl.shapes])[shape_idx]
        ws = np.array([s[1] for s in wl.shapes])[shape_idx]
        rew = wl.reward_lo + uniform_int(draw(seed, 8, env, rr, 0), span).astype(np.int64)
        blk = out[e0:e1]
        blk["h"] = hs
        blk["w"] = ws
        blk["reward"] = rew
        valid = pos[None, None, :].astype(np.int64) < (hs * ws)[:, :, None]  # [E,R,25]
        present = np.zeros((e1 - e0, R, 25), dtype=np.uint32)
        absent = np.zeros_like(present)
        setm = np.zeros_like(present)
        clrm = np.zeros_like(present)
        e3, r3, p3 = env[:, :, None], rr[:, :, None], pos[None, None, :]
        for ch in range(NCH):
            u = u24(draw(seed, 6, e3, r3, p3 * np.uint64(32) + np.uint64(ch)))
            bit = np.uint32(1 << ch)
            present |= np.where(valid & (u < tp), bit, np.uint32(0)).astype(np.uint32)
            absent |= np.where(valid & (u >= tp) & (u < ta), bit, np.uint32(0)).astype(np.uint32)
        for ch in range(C):
            u = u24(draw(seed, 7, e3, r3, p3 * np.uint64(32) + np.uint64(ch)))
            bit = np.uint32(1 << ch)
            setm |= np.where(valid & (u < ts), bit, np.uint32(0)).astype(np.uint32)
            clrm |= np.where(valid & (u >= ts) & (u < tc), bit, np.uint32(0)).astype(np.uint32)
        blk["present"] = present
        blk["absent"] = absent
        blk["set"] = setm
        blk["clear"] = clrm
    if wl.base_game and R >= 2:
        out[:, 0:2] = base_game_rules(C)
    return out


def base_game_rules(C: int) -> np.ndarray:
    """The maze game every evolved environment starts from (Sec. 2.2.1): the
    player moves onto floor where it pushes the force tile (Sec. 2.1, movement
    paragraph), and moving onto a food tile eats it for a reward of 1."""
    r = np.zeros(2, dtype=RULE_DTYPE)
    P, E, G, F = 1 << CH_PLAYER, 1 << CH_EMPTY, 1 << CH_GOAL, 1 << C
    for j in range(2):
        r[j]["h"], r[j]["w"] = 1, 2
        r[j]["present"][0] = P
        r[j]["clear"][0] = P
    r[0]["present"][1] = F | E  # move: player, then force on floor
    r[0]["set"][1] = P
    r[1]["present"][1] = F | G  # eat: player, then force on food
    r[1]["set"][1] = P | E
    r[1]["clear"][1] = G
    r[1]["reward"] = 1
    return r


def make_init_cum(wl: Workload, seed: int) -> np.ndarray:
    """Cumulative 24-bit type thresholds, shape [n, C] uint32 (n = B or 1).

    A cell draws u in [0, 2^24) and takes the first type t with u < cum[t];
    cum[C-1] = 2^24.  The player type has zero width: the player is placed
    separately.  "maze": empty 0.7 / wall 0.25 / goal 0.05.  "dirichlet":
    per env, Dirichlet(1) over the non-player types as the spacings of sorted
    uniform 24-bit draws (exact integer arithmetic).
    """
    C = wl.C
    if wl.init == "maze":
        probs = {CH_EMPTY: 0.7, CH_WALL: 0.25, CH_GOAL: 0.05}
        cum = np.zeros((1, C), dtype=np.uint32)
        acc = 0.0
        for t in range(C):
            acc += probs.get(t, 0.0)
            cum[0, t] = thr24(acc)
        cum[0, C - 1] = ONE24
        return cum
    kinds = [t for t in range(C) if t != CH_PLAYER]
    K = len(kinds)
    n = wl.batch
    env = np.arange(n, dtype=np.uint64)[:, None]
    k = np.arange(max(K - 1, 0), dtype=np.uint64)[None, :]
    u = np.sort(u24(draw(seed, 3, env, 0, k)), axis=1) if K > 1 else np.zeros((n, 0), np.int64)
    cum_np = np.concatenate([u, np.full((n, 1), ONE24, dtype=np.int64)], axis=1)
    cum = np.zeros((n, C), dtype=np.uint32)
    j = 0
    prev = np.zeros(n, dtype=np.int64)
    for t in range(C):
        if t == CH_PLAYER:
            cum[:, t] = prev
        else:
            cum[:, t] = cum_np[:, j]
            prev = cum_np[:, j]
            j += 1
    cum[:, C - 1] = ONE24
    return cum


def actions(seed: int, batch: int, n_steps: int) -> np.ndarray:
    """Actions [n_steps][batch] uint8 in 0..4 for step-by-step runs: step s of
    env e takes uniform_int(draw(seed, 4, e, 0, s), 5), the same action a fused
    rollout with action seed `seed` draws on the device."""
    e = np.arange(batch, dtype=np.uint64)[None, :]
    st = np.arange(n_steps, dtype=np.uint64)[:, None]
    return uniform_int(draw(seed, 4, e, np.uint64(0), st), 5).astype(np.uint8)


def config_fields(wl: Workload) -> dict:
    """Scalar fields of the library's / oracle's configuration structs."""
    def role(ch):
        return ch if ch < wl.C else -1

    return dict(
        batch=wl.batch, H=wl.H, W=wl.W, C=wl.C, n_rules=wl.n_rules,
        rules_per_env=wl.rules_per_env, max_steps=wl.max_steps, auto_reset=wl.auto_reset,
        ch_player=role(CH_PLAYER), ch_goal=role(CH_GOAL), ch_empty=role(CH_EMPTY),
        ch_wall=role(CH_WALL), border_wall=wl.border_wall,
        cum_per_env=0 if wl.init == "maze" else 1,
    )


def make(wl_or_key, seed: int = 0):
    """(workload, rules [n,R] RULE_DTYPE, init_cum [n,C] uint32)."""
    wl = WORKLOADS[wl_or_key] if isinstance(wl_or_key, int) else wl_or_key
    s = seeds(seed)["rules"]
    return wl, make_rules(wl, s), make_init_cum(wl, s)


def empty_rules(n_tab: int, R: int) -> np.ndarray:
    return np.zeros((n_tab, R), dtype=RULE_DTYPE)


def random_grids(rng_seed: int, n: int, H: int, W: int, C: int, density: float = 0.3,
                 stream: int = 9) -> np.ndarray:
    """Multi-hot random grids [n, H, W] (uint8 if C <= 8 else uint16), for tests."""
    env = np.arange(n, dtype=np.uint64)[:, None, None, None]
    y = np.arange(H, dtype=np.uint64)[None, :, None, None]
    x = np.arange(W, dtype=np.uint64)[None, None, :, None]
    ch = np.arange(C, dtype=np.uint64)[None, None, None, :]
    u = u24(draw(rng_seed, stream, env, y, x * np.uint64(32) + ch))
    bits = (u < thr24(density)).astype(np.uint32) << ch.astype(np.uint32)
    g = bits.sum(axis=3).astype(np.uint32)
    return g.astype(np.uint8 if C <= 8 else np.uint16)
