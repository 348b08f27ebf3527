"""Shared helpers for the GPU parity tests (CUDA path via the C-ABI vs oracle)."""
from __future__ import annotations

import numpy as np

import oracle
import workload as wk


def to_np(t, C=None):
    a = t.detach().cpu().numpy()
    if a.dtype == np.int16:
        a = a.view(np.uint16)
    if a.dtype == np.int64 and C == "hash":
        a = a.view(np.uint64)
    return a


def to_dev(a, device="cuda"):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    if a.dtype == np.uint64:
        a = a.view(np.int64)
    return torch.from_numpy(a).to(device)


def make(wl: wk.Workload, seed: int, search_capacity: int = 0, rules=None, cum=None):
    """(Env, oracle cfg, rules, cum) for a workload."""
    import paper_2407_04221_gb300 as av
    if rules is None:
        _, rules, cum = wk.make(wl, seed)
    fields = wk.config_fields(wl)
    env = av.Env(fields, rules, cum, search_capacity=search_capacity)
    return env, oracle.make_cfg(**fields), rules, cum


def sample_envs(B: int, n: int, seed: int = 0) -> np.ndarray:
    """n env indices spread over [0, B), always including the first and last."""
    if n >= B:
        return np.arange(B)
    rng = np.random.default_rng(seed)
    mid = rng.choice(np.arange(1, B - 1), size=n - 2, replace=False)
    return np.sort(np.concatenate([[0, B - 1], mid]))
