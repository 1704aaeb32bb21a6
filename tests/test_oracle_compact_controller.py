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


def test_compact_inplace_hazard_path_brute_force():
    """Tree in the cache tail, path [0, 2, 5]: row L + 2 is the destination
    of entry 2 and the source of entry 1; every destination must get the
    value its source had before the call."""
    layers, B, Hkv, Lmax, D = 2, 1, 2, 16, 3
    g = np.random.default_rng(1)
    kc = g.standard_normal((layers, B, Hkv, Lmax, D))
    vc = g.standard_normal((layers, B, Hkv, Lmax, D))
    L = 4
    k2, v2, nl = oracle.kv_compact_inplace(kc, vc, [L], [[0, 2, 5]])
    assert nl.tolist() == [7]
    assert (k2[:, 0, :, L] == kc[:, 0, :, L]).all()          # the root stays
    assert (k2[:, 0, :, L + 1] == kc[:, 0, :, L + 2]).all()  # old row L + 2, before it is overwritten
    assert (k2[:, 0, :, L + 2] == kc[:, 0, :, L + 5]).all()
    assert (v2[:, 0, :, L + 2] == vc[:, 0, :, L + 5]).all()
    rest = np.ones(Lmax, bool)
    rest[L + 1:L + 3] = False
    assert (k2[:, :, :, rest] == kc[:, :, :, rest]).all()


def test_compact_inplace_equals_out_of_place_from_the_tail():
    """The same commit through a separate tree buffer copied from the
    cache tail gives the same cache."""
    layers, B, Hkv, Lmax, D = 3, 2, 2, 20, 4
    g = np.random.default_rng(2)
    kc = g.standard_normal((layers, B, Hkv, Lmax, D))
    vc = g.standard_normal((layers, B, Hkv, Lmax, D))
    kv_len, sizes = [3, 9], [7, 6]
    offs = np.concatenate([[0], np.cumsum(sizes)])
    kt = np.concatenate([kc[:, b, :, kv_len[b]:kv_len[b] + sizes[b]].transpose(0, 2, 1, 3) for b in range(B)], 1)
    vt = np.concatenate([vc[:, b, :, kv_len[b]:kv_len[b] + sizes[b]].transpose(0, 2, 1, 3) for b in range(B)], 1)
    paths = [[0, 1, 3, 6], [0, 4, 5]]
    a = oracle.kv_compact_inplace(kc, vc, kv_len, paths)
    b = oracle.kv_compact(kc, vc, kv_len, kt, vt, offs, paths)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    # a = 0: nothing moves
    same = oracle.kv_compact_inplace(kc, vc, kv_len, [[0], [0]])
    assert np.array_equal(same[0], kc) and np.array_equal(same[1], vc) and same[2].tolist() == [4, 10]


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


def test_tokenflock_hand_examples():
    """TokenFlock (Table 3's alternative initialisation): Omega = generated
    positions before (i, j) within distance delta; weights delta + 1 - dy,
    normalised; the means rounded half up."""
    P = oracle.CtrlParams(init_mode=oracle.INIT_TOKENFLOCK, flock_delta=1)
    c = oracle.Controller(P, 3, 4)
    # (1, 1) with delta 1: left neighbour (1, 0) weight 2, (0, 1) above weight 1
    c.d_grid[:5] = [9, 3, 9, 9, 6]
    c.k_grid[:5] = [13, 10, 13, 13, 4]
    assert c._flock(5) == (5, 6)          # (2*6 + 3) / 3, (2*4 + 10) / 3
    # delta 2 at (0, 2): (0, 0) and (0, 1), both weight 3: means 4.5 and 11.5 round up
    c2 = oracle.Controller(oracle.CtrlParams(init_mode=oracle.INIT_TOKENFLOCK, flock_delta=2), 2, 8)
    c2.d_grid[:2] = [4, 5]
    c2.k_grid[:2] = [10, 13]
    assert c2._flock(2) == (5, 12)
    # delta 2 at (2, 2) of a 4 x 5 grid: same row (2,0),(2,1) weight 3; row 1
    # columns 1..3 weight 2; (0, 2) weight 1 -> sum of weights 13
    c3 = oracle.Controller(oracle.CtrlParams(init_mode=oracle.INIT_TOKENFLOCK, flock_delta=2), 4, 5)
    d = [1, 2, 3, 4, 5, 6, 7, 8, 9, 1, 2, 3]
    c3.d_grid[:12] = d
    c3.k_grid[:12] = [4] * 12
    num = 3 * d[10] + 3 * d[11] + 2 * (d[6] + d[7] + d[8]) + 1 * d[2]   # = 6 + 9 + 48 + 3 = 66
    assert num == 66 and c3._flock(12) == (5, 4)                        # 66 / 13 = 5.08 -> 5
    # nothing generated before: (d0, k0)
    assert oracle.Controller(P, 3, 4)._flock(0) is None


def test_tokenflock_trace():
    P = oracle.anole_params(init_mode=oracle.INIT_TOKENFLOCK, flock_delta=2)
    c = oracle.Controller(P, 4, 8)
    assert c.next(0) == (5, 10)           # first tree: (d0, k0), no adaptation
    assert c.update(0, 2) == 3            # alpha = 2/5 < beta
    # Omega of (0, 3): (0, 1) and (0, 2), both (5, 10) -> (5, 10); alpha < 1 -> (4, 13)
    assert c.next(3) == (4, 13)
    assert c.update(3, 4) == 8            # alpha = 1 >= beta; positions 3..7 hold (4, 13)
    # Omega of (1, 0): (0, 0) .. (0, 2)? distance <= 2 -> (0, 0) w 2, (0, 1) w 2, and
    # (0, 2) is at distance sqrt(5) > 2: mean of (5, 10) twice = (5, 10); alpha >= 1 -> (6, 7)
    assert c.next(8) == (6, 7)
