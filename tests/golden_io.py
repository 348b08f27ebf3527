"""Reader for the hand-worked fixtures in tests/golden/*.txt.

Fixture format (one step of one env):

    # comment lines; a '# cite:' line names the passage the case follows
    channels: E W P G          names of tile channels 0..C-1 (force is 'F')
    roles: player=P goal=G empty=E wall=W
    rule <name> reward=<int> size=<h>x<w>  (variant fixtures add 'limit: <rule> <k>',
                               'inhibit: <rule> <rule>', 'index: ordered|random')
    in:
      <h lines of w entries>   entry: letters = present channels, '!X' = X absent,
                               'F' = force present, '.' = don't care
    out:
      <h lines of w entries>   entry: '+X' set X, '-X' clear X, '.' = unchanged
    end
    action: <0..4>
    before:
      <H lines of W cells>     cell: letters of its channels, '.' = no bits
    after:
      <H lines of W cells>
    reward: <int>
    done: <0|1>
"""
from __future__ import annotations

import dataclasses
import os
import re

import numpy as np

import workload as wk

GOLDEN_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@dataclasses.dataclass
class Fixture:
    name: str
    cite: str
    C: int
    roles: dict
    rules: np.ndarray  # [1, R] RULE_DTYPE
    action: int
    before: np.ndarray
    after: np.ndarray
    reward: int
    done: int
    variant: dict = dataclasses.field(default_factory=dict)  # limit {r: k}, inhibit {r: mask}, index

    def cfg_fields(self) -> dict:
        H, W = self.before.shape
        return dict(batch=1, H=H, W=W, C=self.C, n_rules=self.rules.shape[1], rules_per_env=0,
                    max_steps=0, auto_reset=0, ch_player=self.roles.get("player", -1),
                    ch_goal=self.roles.get("goal", -1), ch_empty=self.roles.get("empty", -1),
                    ch_wall=self.roles.get("wall", -1), border_wall=0, cum_per_env=0)


def _cell(tok: str, names: dict) -> int:
    if tok == ".":
        return 0
    v = 0
    for ch in tok:
        v |= 1 << names[ch]
    return v


def _in_entry(tok: str, names: dict, C: int):
    pres = absn = 0
    if tok == ".":
        return 0, 0
    i = 0
    while i < len(tok):
        if tok[i] == "!":
            absn |= 1 << (C if tok[i + 1] == "F" else names[tok[i + 1]])
            i += 2
        else:
            pres |= 1 << (C if tok[i] == "F" else names[tok[i]])
            i += 1
    return pres, absn


def _out_entry(tok: str, names: dict):
    s = c = 0
    if tok == ".":
        return 0, 0
    for sign, ch in re.findall(r"([+-])([A-Z])", tok):
        if sign == "+":
            s |= 1 << names[ch]
        else:
            c |= 1 << names[ch]
    return s, c


def load(path: str) -> Fixture:
    lines = [ln.rstrip("\n") for ln in open(path)]
    cite = " ".join(ln.split(":", 1)[1].strip() for ln in lines if ln.startswith("# cite:"))
    body = [ln.strip() for ln in lines if ln.strip() and not ln.startswith("#")]
    names, roles, rules = {}, {}, []
    variant = {"limit": {}, "inhibit": {}, "index": "ordered"}
    action = reward = done = 0
    before = after = None
    i = 0

    def grid_block(start):
        rows = []
        j = start
        while j < len(body) and not re.match(r"^[a-z_]+:", body[j]) and not body[j].startswith("rule"):
            rows.append(body[j].split())
            j += 1
        return rows, j

    while i < len(body):
        ln = body[i]
        if ln.startswith("channels:"):
            for c, nm in enumerate(ln.split(":", 1)[1].split()):
                names[nm] = c
            i += 1
        elif ln.startswith("roles:"):
            for kv in ln.split(":", 1)[1].split():
                k, v = kv.split("=")
                roles[k] = names[v]
            i += 1
        elif ln.startswith("rule"):
            m = re.match(r"rule (\S+) reward=(-?\d+) size=(\d+)x(\d+)", ln)
            h, w = int(m.group(3)), int(m.group(4))
            rec = np.zeros((), dtype=wk.RULE_DTYPE)
            rec["h"], rec["w"], rec["reward"] = h, w, int(m.group(2))
            assert body[i + 1] == "in:"
            C = len(names)
            for r in range(h):
                toks = body[i + 2 + r].split()
                assert len(toks) == w, ln
                for k, tok in enumerate(toks):
                    p, a = _in_entry(tok, names, C)
                    rec["present"][r * w + k], rec["absent"][r * w + k] = p, a
            assert body[i + 2 + h] == "out:"
            for r in range(h):
                toks = body[i + 3 + h + r].split()
                assert len(toks) == w, ln
                for k, tok in enumerate(toks):
                    s, c = _out_entry(tok, names)
                    rec["set"][r * w + k], rec["clear"][r * w + k] = s, c
            assert body[i + 3 + 2 * h] == "end"
            rules.append(rec)
            i += 4 + 2 * h
        elif ln.startswith("limit:"):
            r, k = (int(v) for v in ln.split(":")[1].split())
            variant["limit"][r] = k
            i += 1
        elif ln.startswith("inhibit:"):
            r, q = (int(v) for v in ln.split(":")[1].split())
            variant["inhibit"][r] = variant["inhibit"].get(r, 0) | (1 << q)
            i += 1
        elif ln.startswith("index:"):
            variant["index"] = ln.split(":")[1].strip()
            i += 1
        elif ln.startswith("action:"):
            action = int(ln.split(":")[1])
            i += 1
        elif ln.startswith("reward:"):
            reward = int(ln.split(":")[1])
            i += 1
        elif ln.startswith("done:"):
            done = int(ln.split(":")[1])
            i += 1
        elif ln.startswith("before:") or ln.startswith("after:"):
            rows, j = grid_block(i + 1)
            g = np.array([[_cell(t, names) for t in r] for r in rows], dtype=np.uint16)
            if ln.startswith("before:"):
                before = g
            else:
                after = g
            i = j
        else:
            raise ValueError(f"{path}: cannot parse line {ln!r}")
    C = len(names)
    dt = np.uint8 if C <= 8 else np.uint16
    rt = np.zeros((1, len(rules)), dtype=wk.RULE_DTYPE)
    for r, rec in enumerate(rules):
        rt[0, r] = rec
    return Fixture(os.path.basename(path), cite, C, roles, rt, action, before.astype(dt),
                   after.astype(dt), reward, done, variant)


def variant_fixtures():
    d = os.path.join(GOLDEN_DIR, "variant")
    return sorted(os.path.join(d, f) for f in os.listdir(d) if f.endswith(".txt"))


def all_fixtures():
    return sorted(os.path.join(GOLDEN_DIR, f) for f in os.listdir(GOLDEN_DIR) if f.endswith(".txt"))
