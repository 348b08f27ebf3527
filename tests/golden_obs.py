"""Reader for the hand-worked observation fixtures in tests/golden/observe/.

Patch fixtures (obs_*.txt):

    # comments; '# cite:' lines name the passage the case follows
    channels: E W P G          names of tile channels 0..C-1
    roles: player=P
    window: <int>
    board:
      <H lines of W cells>     cell: letters of its channels, '.' = no bits
    player: <y> <x>            (-1 -1: no player on the board)
    patch:
      <window lines of window cells>   '.' = zero (padding or an empty cell)

Rule-encoding fixtures (rules_*.txt): 'channels:', then rule blocks in the
step fixtures' format, then

    bits:
      <rule> <plane> <row> <col> <channel>   one line per 1 of the encoding;
                                             plane present|absent|set|clear,
                                             channel a name or F (force)
    rewards: <one int per rule>
"""
from __future__ import annotations

import dataclasses
import os

import numpy as np

import workload as wk
from tests.golden_io import _cell, _in_entry, _out_entry

OBS_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "observe")
PLANES = ("present", "absent", "set", "clear")


@dataclasses.dataclass
class PatchFixture:
    name: str
    cite: str
    C: int
    ch_player: int
    window: int
    board: np.ndarray   # [H, W] cell words
    player: tuple
    patch: np.ndarray   # [window, window] cell words

    def cfg_fields(self) -> dict:
        H, W = self.board.shape
        return dict(batch=1, H=H, W=W, C=self.C, n_rules=0, rules_per_env=0, max_steps=0,
                    auto_reset=0, ch_player=self.ch_player, ch_goal=-1, ch_empty=-1,
                    ch_wall=-1, border_wall=0, cum_per_env=0)


@dataclasses.dataclass
class RuleFixture:
    name: str
    cite: str
    C: int
    rules: np.ndarray   # [1, R] RULE_DTYPE
    bits: np.ndarray    # [1, R, 4, 5, 5, C+1] uint8, the expected encoding
    rewards: np.ndarray  # [1, R] int32


def _split(path):
    lines = [ln.rstrip("\n") for ln in open(path)]
    cite = " ".join(ln.split(":", 1)[1].strip() for ln in lines if ln.startswith("# cite:"))
    body = [ln.strip() for ln in lines if ln.strip() and not ln.startswith("#")]
    return cite, body


def _block(body, i):
    rows = []
    while i < len(body) and ":" not in body[i] and not body[i].startswith("rule"):
        rows.append(body[i].split())
        i += 1
    return rows, i


def load_patch(path: str) -> PatchFixture:
    cite, body = _split(path)
    names, roles, window, player = {}, {}, 0, None
    board = patch = None
    i = 0
    while i < len(body):
        ln = body[i]
        key = ln.split(":", 1)[0]
        if key == "channels":
            names = {nm: c for c, nm in enumerate(ln.split(":", 1)[1].split())}
            i += 1
        elif key == "roles":
            roles = {k: names[v] for k, v in (kv.split("=") for kv in ln.split(":", 1)[1].split())}
            i += 1
        elif key == "window":
            window = int(ln.split(":")[1])
            i += 1
        elif key == "player":
            player = tuple(int(v) for v in ln.split(":")[1].split())
            i += 1
        elif key in ("board", "patch"):
            rows, i = _block(body, i + 1)
            g = np.array([[_cell(t, names) for t in r] for r in rows], dtype=np.uint16)
            if key == "board":
                board = g
            else:
                patch = g
        else:
            raise ValueError(f"{path}: cannot parse line {ln!r}")
    C = len(names)
    dt = np.uint8 if C <= 8 else np.uint16
    return PatchFixture(os.path.basename(path), cite, C, roles["player"], window,
                        board.astype(dt), player, patch.astype(dt))


def load_rules(path: str) -> RuleFixture:
    cite, body = _split(path)
    names, recs, ones, rewards = {}, [], [], []
    i = 0
    while i < len(body):
        ln = body[i]
        if ln.startswith("channels:"):
            names = {nm: c for c, nm in enumerate(ln.split(":", 1)[1].split())}
            i += 1
        elif ln.startswith("rule"):
            _, _, rew, size = ln.split()
            h, w = (int(v) for v in size.split("=")[1].split("x"))
            rec = np.zeros((), dtype=wk.RULE_DTYPE)
            rec["h"], rec["w"], rec["reward"] = h, w, int(rew.split("=")[1])
            C = len(names)
            assert body[i + 1] == "in:" and body[i + 2 + h] == "out:" and body[i + 3 + 2 * h] == "end"
            for r in range(h):
                for k, tok in enumerate(body[i + 2 + r].split()):
                    rec["present"][r * w + k], rec["absent"][r * w + k] = _in_entry(tok, names, C)
                for k, tok in enumerate(body[i + 3 + h + r].split()):
                    rec["set"][r * w + k], rec["clear"][r * w + k] = _out_entry(tok, names)
            recs.append(rec)
            i += 4 + 2 * h
        elif ln.startswith("bits:"):
            rows, i = _block(body, i + 1)
            ones = rows
        elif ln.startswith("rewards:"):
            rewards = [int(v) for v in ln.split(":")[1].split()]
            i += 1
        else:
            raise ValueError(f"{path}: cannot parse line {ln!r}")
    C = len(names)
    R = len(recs)
    rules = np.zeros((1, R), dtype=wk.RULE_DTYPE)
    for r, rec in enumerate(recs):
        rules[0, r] = rec
    bits = np.zeros((1, R, 4, 5, 5, C + 1), np.uint8)
    for rule, plane, row, col, ch in ones:
        c = C if ch == "F" else names[ch]
        bits[0, int(rule), PLANES.index(plane), int(row), int(col), c] = 1
    return RuleFixture(os.path.basename(path), cite, C, rules, bits,
                       np.array([rewards], np.int32))


def patch_fixtures():
    return sorted(os.path.join(OBS_DIR, f) for f in os.listdir(OBS_DIR) if f.startswith("obs_"))


def rule_fixtures():
    return sorted(os.path.join(OBS_DIR, f) for f in os.listdir(OBS_DIR) if f.startswith("rules_"))
