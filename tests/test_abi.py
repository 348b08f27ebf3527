"""The C-ABI library loads and exports every entry point its header declares.

No compute call is made here (no GPU needed): only host-side argument checks
that return before any CUDA work.
"""
from __future__ import annotations

import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "autoverse.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:int|const char \*)\s*(av_\w+)\s*\(", text, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    from paper_2407_04221_gb300 import build
    build.build()
    import paper_2407_04221_gb300 as av
    return av.load()


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("av_create", "av_destroy", "av_reset", "av_step", "av_rollout", "av_expand",
              "av_select", "av_sync"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    import paper_2407_04221_gb300 as av
    names = declared_functions()
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    assert set(names) == set(av.EXPORTS)


def test_rule_record_size_matches_header():
    import workload as wk
    assert wk.RULE_DTYPE.itemsize == 408
    text = open(HEADER).read()
    assert "uint32_t present[25], absent[25], set[25], clear[25];" in text


def test_host_side_argument_checks(lib):
    import paper_2407_04221_gb300 as av
    assert lib.av_destroy(None) == av.AV_EINVAL
    assert lib.av_sync(None) == av.AV_EINVAL
    assert lib.av_create(None, None, None) == av.AV_EINVAL
    assert lib.av_rollout_path(None, None) == av.AV_EINVAL
    assert lib.av_observe(None, None, 5, None, None, 0) == av.AV_EINVAL
    assert lib.av_rule_obs(None, None, None, 0) == av.AV_EINVAL
    assert lib.av_mutate(1, 16, 16, 8, 8, None, 0, None, None, 0) == av.AV_EINVAL
    assert lib.av_set_variant(None, None) == av.AV_EINVAL
    m = av.AvMutation(p_map=(1 << 24) + 1)
    assert lib.av_mutate(1, 16, 16, 8, 8, ctypes.byref(m), 0, None, None, 0) == av.AV_EINVAL
    m = av.AvMutation(reward_min=2, reward_max=1)
    assert lib.av_mutate(1, 16, 16, 8, 8, ctypes.byref(m), 0, None, None, 0) == av.AV_EINVAL
    m = av.AvMutation()
    assert lib.av_mutate(1, 257, 16, 8, 8, ctypes.byref(m), 0, None, None, 0) == av.AV_EINVAL
    assert av.av_strerror(av.AV_EINVAL) == "invalid argument"
    base = dict(batch=1, H=16, W=16, C=4, n_rules=0, rules_per_env=0, max_steps=0, auto_reset=0,
                ch_player=2, ch_goal=3, ch_empty=0, ch_wall=1, border_wall=1, cum_per_env=0)
    bad = [dict(batch=0), dict(H=257), dict(W=0), dict(C=17), dict(C=0), dict(n_rules=65),
           dict(ch_goal=4), dict(ch_player=-2), dict(rules_per_env=2), dict(max_steps=-1)]
    for b in bad:
        with pytest.raises(av.AvError) as ei:
            av.av_create(dict(base, **b), np.zeros(0, np.uint8))
        assert ei.value.status == av.AV_EINVAL, b
    # malformed rule records are rejected before any device work
    import workload as wk
    r = wk.empty_rules(1, 1)
    r["h"], r["w"] = 3, 3
    r["present"][0, 0, 9] = 1  # entry outside the 3x3 window
    with pytest.raises(av.AvError):
        av.av_create(dict(base, n_rules=1), r)
    r = wk.empty_rules(1, 1)
    r["h"], r["w"] = 6, 1
    with pytest.raises(av.AvError):
        av.av_create(dict(base, n_rules=1), r)
    r = wk.empty_rules(1, 1)
    r["h"], r["w"] = 1, 1
    r["set"][0, 0, 0] = 1 << 4  # writes the force channel
    with pytest.raises(av.AvError):
        av.av_create(dict(base, n_rules=1), r)


def test_missing_library_fails_loudly(tmp_path, monkeypatch):
    import paper_2407_04221_gb300 as av
    monkeypatch.setattr(av, "_lib", None)
    monkeypatch.setattr(av, "LIB_PATH", str(tmp_path / "absent.so"))
    with pytest.raises(RuntimeError, match="missing"):
        av.load()


def test_allocation_failure_gives_enomem(lib, monkeypatch):
    """AV_FAIL_ALLOC makes av_create's device allocations fail: AV_ENOMEM, and
    no handle (the refusal comes before any device memory is touched)."""
    import paper_2407_04221_gb300 as av
    import workload as wk
    monkeypatch.setenv("AV_FAIL_ALLOC", "1")
    fields = dict(batch=4, H=16, W=16, C=4, n_rules=2, rules_per_env=0, max_steps=0, auto_reset=0,
                  ch_player=2, ch_goal=3, ch_empty=0, ch_wall=1, border_wall=1, cum_per_env=0)
    cfg = av.AvConfig(**{k: v for k, v in fields.items()})
    rules = np.ascontiguousarray(wk.base_game_rules(4))
    h = ctypes.c_void_p()
    rc = lib.av_create(ctypes.byref(cfg), rules.ctypes.data_as(ctypes.c_void_p), ctypes.byref(h))
    assert rc == av.AV_ENOMEM
    assert h.value is None


def test_calls_on_a_handle_that_is_not_alive(lib):
    """A pointer that av_create never returned (or that av_destroy already
    took) is refused with AV_ESTATE, without being dereferenced."""
    import paper_2407_04221_gb300 as av
    fake = ctypes.c_void_p(0x1000)
    assert lib.av_destroy(fake) == av.AV_ESTATE
    assert lib.av_sync(fake) == av.AV_ESTATE
    assert lib.av_step(fake, fake, None, None, None, 0) == av.AV_ESTATE
    assert lib.av_rollout(fake, 1, 0, None, None, None, None, 0) == av.AV_ESTATE
    assert lib.av_set_variant(fake, None) == av.AV_ESTATE
    path = ctypes.c_int32()
    assert lib.av_rollout_path(fake, ctypes.byref(path)) == av.AV_ESTATE
    assert b"not a live handle" in lib.av_last_error(fake)
