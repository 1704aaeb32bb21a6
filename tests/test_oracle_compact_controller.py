"""Pins of the oracle's K/V commit (accepted nodes join the prefix, Sec. 3.1)
and of the depth / width controller (Sec. 4.1, Eq. 2, end of Sec. 4.2)."""
import json
import os

import numpy as np
import pytest

import oracle


def test_compact_brute_force_gather():
    layers, B, Hkv, Lmax, D = 3, 2, 2, 12, 4
    g = np.random.default_rng(0)
    kc = g.standard_normal((layers, B, Hkv, Lmax, D))
    vc = g.standard_normal((layers, B, Hkv, Lmax, D))
    kt = g.standard_normal((layers, 9, Hkv, D))
    vt = g.standard_normal((layers, 9, Hkv, D))
    offs = [0, 5, 9]
    kv_len = [4, 7]
    paths = [[0, 2, 4], [0]]
    k2, v2, nl = oracle.kv_compact(kc, vc, kv_len, kt, vt, offs, paths)
    assert nl.tolist() == [7, 8]
    for l in range(layers):
        for h in range(Hkv):
            assert (k2[l, 0, h, 4] == kt[l, 0, h]).all()
            assert (k2[l, 0, h, 5] == kt[l, 2, h]).all()
            assert (v2[l, 0, h, 6] == vt[l, 4, h]).all()
            assert (k2[l, 1, h, 7] == kt[l, 5, h]).all()  # a = 0: only the root is appended
    untouched = np.ones_like(kc, bool)
    untouched[:, 0, :, 4:7] = False
    untouched[:, 1, :, 7] = False
    assert (k2[untouched] == kc[untouched]).all() and (v2[untouched] == vc[untouched]).all()


def test_compact_overflow_rejected():
    z = np.zeros((1, 1, 1, 3, 2))
    zt = np.zeros((1, 3, 1, 2))
    with pytest.raises(ValueError):
        oracle.kv_compact(z, z, [2], zt, zt, [0, 3], [[0, 1]])


def test_splitmix64_published_vectors(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "splitmix64.json")))
    for c in g["cases"]:
        state, outs = c["seed"], []
        for _ in range(3):
            outs.append(oracle.splitmix64(state))
            state = (state + 0x9E3779B97F4A7C15) & ((1 << 64) - 1)
        if "outputs_hex" in c:
            assert [f"{o:016x}" for o in outs] == c["outputs_hex"]
        else:
            assert [str(o) for o in outs] == c["outputs_dec"]


def test_controller_hand_traces(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "controller_traces.json")))
    for c in g["cases"]:
        ctl = oracle.Controller(oracle.CtrlParams(**c["params"]), *c["grid"])
        pos, got, gp = 0, [], []
        for a in c["accept"]:
            gp.append(pos)
            got.append(list(ctl.next(pos)))
            pos = ctl.update(pos, a)
        assert got == c["expected_dk"], c["name"]
        assert gp == c["expected_pos"], c["name"]


def test_controller_random_init_in_range_and_seeded():
    P = oracle.anole_params(init_mode=oracle.INIT_RANDOM, seed=99)
    a = oracle.Controller(P, 8, 8)
    b = oracle.Controller(P, 8, 8)
    for pos in range(0, 60, 3):
        da, ka = a.next(pos)
        db, kb = b.next(pos)
        assert (da, ka) == (db, kb)
        assert 1 <= da <= 9 and 4 <= ka <= 13
        a.update(pos, min(2, da))
        b.update(pos, min(2, db))
    # the first draw follows SplitMix64 with counter 0 / 1
    c = oracle.Controller(P, 8, 8)
    assert c.next(0) == (1 + oracle.counter_draw(99, 0) % 9, 4 + oracle.counter_draw(99, 1) % 10)


def test_controller_fixed_init_ablation():
    """Table 3 ablations: d~ or k~ held fixed, Eq. 2 still applied."""
    P = oracle.llamagen_params(fix_d=1, fix_k=25, d0=3, k0=10)
    c = oracle.Controller(P, 4, 4)
    assert c.next(0) == (1, 25)
    p = c.update(0, 1)           # alpha = 1 -> deeper, narrower
    assert c.next(p) == (2, 15)
    p = c.update(p, 0)           # alpha = 0 -> shallower, wider
    assert c.next(p) == (1, 35)


def test_controller_rejects_bad_accept_len():
    c = oracle.Controller(oracle.anole_params(), 2, 2)
    c.next(0)
    with pytest.raises(ValueError):
        c.update(0, 6)
