"""The C-ABI library loads, exports every entry point include/adt.h declares,
and its host-only parts (argument checks that return before any launch, the
depth / width controller) behave as specified.  No GPU is used here."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import oracle
from paper_2512_21857_gb300 import binding as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2512_21857_gb300 import build
    build.build()
    return B.lib()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "adt.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(adt_[a-z_0-9]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 17
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (adt_\w+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert hasattr(lib, n)
    assert set(B.EXPORTED) <= set(names)


def test_version_and_status_names(lib):
    assert B.adt_version() >= 100
    assert lib.adt_status_string(1) == b"ADT_ERR_INVALID_ARG"
    assert lib.adt_status_string(99) == b"ADT_ERR_UNKNOWN"


def test_invalid_arguments_rejected_before_launch(lib):
    f = ctypes.c_void_p(16)  # never dereferenced: every call below fails its host checks first
    # null pointers
    assert lib.adt_tree_attn(None, f, f, f, 0, 0, f, f, f, f, 1, 1, 1, 64, 1, 1, 1.0, f, None, f, 0, None) == 1
    # head_dim outside {64, 128} -> unsupported
    assert lib.adt_tree_attn(f, f, f, f, 0, 0, f, f, f, f, 1, 1, 1, 96, 1, 1, 1.0, f, None, f, 0, None) == 2
    # more than 256 nodes per tree -> unsupported
    assert lib.adt_tree_attn(f, f, f, f, 0, 0, f, f, f, f, 1, 1, 1, 64, 257, 1, 1.0, f, None, f, 0, None) == 2
    # H not a multiple of Hkv
    assert lib.adt_tree_attn(f, f, f, f, 0, 0, f, f, f, f, 1, 3, 2, 64, 8, 1, 1.0, f, None, f, 0, None) == 1
    # expand: k_child > 64, k_keep > F*k, ld not a multiple of 4
    assert lib.adt_tree_expand(f, 100, f, None, 2, 100, 65, 1, 1.0, 0, f, f, f, f, f, None, None, f, 1 << 20, None) == 1
    assert lib.adt_tree_expand(f, 100, f, None, 2, 100, 4, 9, 1.0, 0, f, f, f, f, f, None, None, f, 1 << 20, None) == 1
    assert lib.adt_tree_expand(f, 102, f, None, 2, 100, 4, 2, 1.0, 0, f, f, f, f, f, None, None, f, 1 << 20, None) == 1
    # rerank: more nodes than candidates + 1
    assert lib.adt_tree_rerank(f, f, f, 5, f, 7, f, f, None, None, f, 1 << 20, None) == 1
    # accept: SPEC without uniforms / bad mode
    assert lib.adt_tree_accept(f, 128, f, 128, None, f, f, f, 1, 100, 8, None, None, 1, 1.0, f, 8, f, f, None, 0, None) == 1
    assert lib.adt_tree_accept(f, 128, None, 0, None, f, f, f, 1, 100, 8, None, None, 7, 1.0, f, 8, f, f, None, 0, None) == 1
    # compact: kv_len_out aliasing kv_len, unaligned stride
    assert lib.adt_kv_compact(f, f, f, f, f, f, f, f, 8, f, 1, 2, 64, 2, 100, 64, 64, 64, 64, None) == 1
    assert lib.adt_kv_compact(f, f, f, None, f, f, f, f, 8, f, 1, 2, 64, 2, 100, 65, 64, 64, 64, None) == 1
    # in-place compact: more than 256 staged path rows -> unsupported; kv_len_out aliasing kv_len
    assert lib.adt_kv_compact_inplace(f, f, f, None, f, f, 257, f, 1, 2, 64, 2, 300, 64, 64, 64, None) == 2
    assert lib.adt_kv_compact_inplace(f, f, f, f, f, f, 8, f, 1, 2, 64, 2, 300, 64, 64, 64, None) == 1


def _run_both(params, grid, accepts):
    ctl_c = B.Controller(*grid, **params)
    op = dict(params)
    ctl_o = oracle.Controller(oracle.CtrlParams(**op), *grid)
    pos_c = pos_o = 0
    for a in accepts:
        if pos_c >= grid[0] * grid[1]:
            break
        dc, kc = ctl_c.next(pos_c)
        do, ko = ctl_o.next(pos_o)
        assert (dc, kc) == (do, ko)
        a = min(a, dc)
        pos_c = ctl_c.update(pos_c, a)
        pos_o = ctl_o.update(pos_o, a)
        assert pos_c == pos_o
    for p in range(grid[0] * grid[1]):
        assert ctl_c.get(p) == (ctl_o.d_grid[p], ctl_o.k_grid[p])


@pytest.mark.parametrize("init_mode", [0, 1, 2, 3])
@pytest.mark.parametrize("preset", ["anole", "llamagen", "c4"])
def test_controller_matches_oracle_bit_exactly(lib, init_mode, preset):
    params = {
        "anole": dict(beta=1.0, l_d=1, l_k=3, d_lo=1, d_hi=9, k_lo=4, k_hi=13),
        "llamagen": dict(beta=1.0, l_d=1, l_k=10, d_lo=1, d_hi=9, k_lo=4, k_hi=39),
        "c4": dict(beta=1.0, l_d=1, l_k=3, d_lo=2, d_hi=10, k_lo=1, k_hi=8, d0=5, k0=4),
    }[preset]
    params = dict(params, init_mode=init_mode, seed=1234 + init_mode)
    g = np.random.default_rng(init_mode * 7 + len(preset))
    accepts = g.integers(0, 10, size=400).tolist()
    _run_both(params, (48, 48), accepts)
    _run_both(dict(params, clamp_k_always=False, k_cap=64), (24, 24), accepts)
    _run_both(dict(params, fix_d=1, fix_k=25 if preset == "llamagen" else 0), (8, 8), accepts)
    _run_both(dict(params, beta=0.5), (8, 8), accepts)
    if init_mode == 3:
        for delta in (1, 3, 5):
            _run_both(dict(params, flock_delta=delta), (24, 24), accepts)


def test_controller_hand_traces_through_abi(lib, golden_dir):
    import json
    g = json.load(open(os.path.join(golden_dir, "controller_traces.json")))
    for c in g["cases"]:
        ctl = B.Controller(*c["grid"], **c["params"])
        pos = 0
        for a, dk, p in zip(c["accept"], c["expected_dk"], c["expected_pos"]):
            assert pos == p
            assert list(ctl.next(pos)) == dk, c["name"]
            pos = ctl.update(pos, a)


def test_controller_rejects_bad_input(lib):
    with pytest.raises(B.AdtError):
        B.Controller(4, 4, d_lo=3, d_hi=2)
    with pytest.raises(B.AdtError):
        B.Controller(4, 4, init_mode=B.INIT_TOKENFLOCK, flock_delta=0)
    c = B.Controller(4, 4)
    with pytest.raises(B.AdtError):
        c.update(0, 1)  # update before next
    d, k = c.next(0)
    with pytest.raises(B.AdtError):
        c.update(0, d + 1)
    with pytest.raises(B.AdtError):
        c.next(16)


def test_guidance_entry_points_check_their_extra_arguments(lib):
    f = ctypes.c_void_p(16)
    ws = ctypes.c_void_p(256)
    # expand: no unconditional rows / non-finite scale
    assert lib.adt_tree_expand_cfg(f, None, 100, 3.0, f, None, 2, 100, 4, 2, 1.0, 0, f, f, f, f, f, None, None, ws,
                                   1 << 20, None) == 1
    assert lib.adt_tree_expand_cfg(f, f, 100, float("inf"), f, None, 2, 100, 4, 2, 1.0, 0, f, f, f, f, f, None, None,
                                   ws, 1 << 20, None) == 1
    # accept: no unconditional target; SPEC without unconditional draft
    assert lib.adt_tree_accept_cfg(f, None, 128, None, None, 0, None, 3.0, f, f, f, 1, 100, 8, None, None, 0, 1.0, f,
                                   8, f, f, None, 0, None) == 1
    assert lib.adt_tree_accept_cfg(f, f, 128, f, None, 128, None, 3.0, f, f, f, 1, 100, 8, f, f, 1, 1.0, f, 8, f, f,
                                   None, 0, None) == 1


def test_controller_checkpoint_resume(lib):
    """A controller saved mid-image and loaded again makes the same choices
    as the one that kept running."""
    params = dict(beta=1.0, l_d=1, l_k=3, d_lo=1, d_hi=9, k_lo=4, k_hi=13, init_mode=B.INIT_TOKENFLOCK, seed=5)
    g = np.random.default_rng(9)
    accepts = g.integers(0, 10, size=200).tolist()
    a = B.Controller(24, 24, **params)
    pos = 0
    for x in accepts[:60]:
        d, _ = a.next(pos)
        pos = a.update(pos, min(x, d))
    state = a.save()
    b = B.Controller.load(state)
    pos_a = pos_b = pos
    for x in accepts[60:]:
        if pos_a >= 24 * 24:
            break
        da = a.next(pos_a)
        assert b.next(pos_b) == da
        pos_a = a.update(pos_a, min(x, da[0]))
        pos_b = b.update(pos_b, min(x, da[0]))
    for p in range(24 * 24):
        assert a.get(p) == b.get(p)
    # short or foreign buffers are rejected
    with pytest.raises(B.AdtError):
        B.Controller.load(state[:40])
    with pytest.raises(B.AdtError):
        B.Controller.load(b"\0" * len(state))
