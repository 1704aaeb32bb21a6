"""GPU acceptance walk and KV commit vs the oracle.  Paths, accepted lengths,
bonus tokens and cache bytes must match bit for bit.  For the sampling modes
the oracle reports the smallest relative margin of the decisions it took.
The kernel computes p and q in double-float arithmetic (about 1e-11
relative, against the oracle's fp64), so only a case whose margin is below
1e-9 is a near tie that rounding order alone could decide; such a case is
re-drawn, and is rare enough that every seeded draw here is compared."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import ensure_built, i32, run_accept_gpu
from paper_2512_21857_gb300 import binding as B
from paper_2512_21857_gb300 import synth

pytestmark = pytest.mark.gpu
ACCEPT_MARGIN = 1e-9
SAMPLE_MARGIN = 1e-9
EXP_RTOL = 1e-11  # the double-float exponential (about 3e-12 by construction)


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def make_rows(tb, V, seed, sigma, plant=True):
    """Draft rows ~ N(0, 3^2); target rows = draft + N(0, sigma^2) (independent
    when sigma is None).  With `plant`, each tree's target rows are raised so
    that a seeded root path is the greedy one."""
    ntot = int(tb.node_offsets[-1])
    draft = synth.f32_normal((ntot, V), seed, "draft", std=3.0)
    if sigma is None:
        target = synth.f32_normal((ntot, V), seed, "target", std=3.0)
    else:
        target = (draft + synth.f32_normal((ntot, V), seed, "noise", std=sigma)).astype(np.float32)
    if plant:
        g = synth.rng(seed, "plant")
        for b in range(len(tb.node_offsets) - 1):
            lo, hi = tb.node_offsets[b], tb.node_offsets[b + 1]
            par = tb.parents[lo:hi]
            leaf = int(g.integers(0, hi - lo))
            full = oracle.ancestor_path(par, leaf)
            cut = full[:int(g.integers(1, len(full) + 1))]
            synth.plant_path(target[lo:hi], par, tb.tokens[lo:hi], cut, boost=4.0)
    return target, draft


def compare(tb, res, path, alen, bonus):
    for b in range(len(tb.node_offsets) - 1):
        want = res["path"][b]
        assert alen[b] == len(want) - 1
        assert path[b, :len(want)].tolist() == want
        assert (path[b, len(want):] == -1).all()
        assert bonus[b] == res["bonus"][b]


@pytest.mark.parametrize("sizes,V", [([26], 16384), ([64], 65536), ([64, 1, 33, 7, 64, 12, 50, 20], 65536),
                                     ([5], 100), ([3, 9], 262144), ([26, 9], 4099), ([12, 30], 65537)])
@pytest.mark.parametrize("sigma", [None, 0.3])
def test_greedy_matches_oracle(sizes, V, sigma):
    seed = sum(sizes) + V
    tb = synth.tree_batch(sizes, V, seed)
    target, _ = make_rows(tb, V, seed, sigma)
    res = oracle.tree_accept(target, None, tb.tokens, tb.parents, tb.node_offsets, oracle.ACCEPT_GREEDY)
    path, alen, bonus = run_accept_gpu(target, None, tb, B.ACCEPT_GREEDY, max_path=16)
    compare(tb, res, path, alen, bonus)
    if sigma is not None:
        assert res["accept_len"].max() >= 1  # the planted paths are found


@pytest.mark.parametrize("mode", [B.ACCEPT_SPEC, B.ACCEPT_SPEC_DET])
@pytest.mark.parametrize("sizes,V,sigma,T", [
    ([26], 16384, None, 1.0),
    ([26], 16384, 0.3, 1.0),
    ([64], 65536, 0.3, 1.0),
    ([64, 1, 33, 7, 64, 12, 50, 20], 65536, 0.5, 1.0),
    ([16, 9], 16384, 0.3, 0.7),
    ([7], 200000, 0.3, 1.0),
])
def test_sampling_matches_oracle(mode, sizes, V, sigma, T):
    checked = 0
    for rep in range(3):
        seed = 31 * rep + sum(sizes) + V + mode
        tb = synth.tree_batch(sizes, V, seed)
        target, draft = make_rows(tb, V, seed, sigma, plant=sigma is not None)
        ntot = int(tb.node_offsets[-1])
        ua = synth.uniforms(ntot, seed, "ua")
        us = synth.uniforms(ntot, seed, "us")
        res = oracle.tree_accept(target, draft, tb.tokens, tb.parents, tb.node_offsets, mode, ua, us, T)
        if res["accept_margin"] < ACCEPT_MARGIN or res["sample_margin"] < SAMPLE_MARGIN:
            continue  # near tie: re-draw
        path, alen, bonus = run_accept_gpu(target, draft, tb, mode, ua, us, T, max_path=16)
        compare(tb, res, path, alen, bonus)
        checked += 1
    assert checked == 3, f"{3 - checked} of 3 draws were near ties"


def test_double_float_exponential_error_bound():
    """e^(a - b) as the sampling walk computes it (double-float, table-driven)
    against numpy's fp64 exp of the exact difference (itself within 1 ulp):
    relative error below 1e-11 down to a - b = -69, that plus 2^-140 below
    it (to -86, where it flushes to 0), at the reduction's
    interval edges too, and exactly 1 at a = b."""
    g = np.random.default_rng(11)
    n = 1 << 18
    b = (g.standard_normal(n) * 5).astype(np.float32)
    d = -(g.random(n) * 86.0).astype(np.float32)
    d[: 1 << 12] = -(g.random(1 << 12) * 1e-3).astype(np.float32)           # tiny differences
    k = np.arange(1 << 12)
    d[1 << 12: 1 << 13] = (-(k % 7940 + 0.5) * np.log(2) / 64).astype(np.float32)  # interval edges
    a = np.minimum((b + d).astype(np.float32), b)
    a[-1], b[-1] = 3.0, 3.0
    dev = "cuda"
    at, bt = torch.as_tensor(a, device=dev), torch.as_tensor(b, device=dev)
    out = torch.empty(n, dtype=torch.float64, device=dev)
    B.adt_testing_exp_diff(at, bt, out)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    diff = a.astype(np.float64) - b.astype(np.float64)
    ref = np.exp(diff)
    # Both words normal (results above 2^-100): the relative bound.  Below,
    # the low word turns subnormal, which adds an absolute error of a few
    # 2^-149; such terms are below 1e-30 of any row sum, which holds e^0 = 1.
    normal = diff > -69.0
    rel = np.abs(got[normal] - ref[normal]) / ref[normal]
    assert rel.max() < EXP_RTOL, f"max relative error {rel.max():.3e}"
    assert (np.abs(got[~normal] - ref[~normal]) <= EXP_RTOL * ref[~normal] + 2.0 ** -140).all()
    assert got[-1] == 1.0
    assert (got >= 0).all()


def test_spec_uses_draft_row_mapping():
    V, sizes = 16384, [20]
    tb = synth.tree_batch(sizes, V, 5)
    target, draft = make_rows(tb, V, 5, 0.3)
    # the draft rows live in a larger pool, reversed
    pool = np.ascontiguousarray(draft[::-1])
    mapping = np.arange(20)[::-1].copy()
    ua, us = synth.uniforms(20, 5, "ua"), synth.uniforms(20, 5, "us")
    res = oracle.tree_accept(target, pool, tb.tokens, tb.parents, tb.node_offsets, B.ACCEPT_SPEC, ua, us,
                             draft_row=mapping)
    assert res["min_margin"] > 1e-5
    path, alen, bonus = run_accept_gpu(target, pool, tb, B.ACCEPT_SPEC, ua, us, draft_row=mapping)
    compare(tb, res, path, alen, bonus)


def test_spec_leaves_may_have_no_draft_row_and_a_missing_row_is_flagged():
    """Leaves map to draft row -1 (their rows are never read): the walk is the
    oracle's.  The root without a draft row is flagged, accepts nothing and
    draws its bonus from its own target distribution, as a lone root would."""
    V, n = 16384, 20
    tb = synth.tree_batch([n], V, 8)
    target, draft = make_rows(tb, V, 8, 0.3)
    ua, us = synth.uniforms(n, 8, "ua"), synth.uniforms(n, 8, "us")
    has_kids = np.zeros(n, dtype=bool)
    has_kids[tb.parents[1:]] = True
    mapping = np.where(has_kids, np.arange(n), -1).astype(np.int32)
    res = oracle.tree_accept(target, draft, tb.tokens, tb.parents, tb.node_offsets, B.ACCEPT_SPEC, ua, us)
    assert res["min_margin"] > ACCEPT_MARGIN
    B.adt_get_device_error()
    path, alen, bonus = run_accept_gpu(target, draft, tb, B.ACCEPT_SPEC, ua, us, draft_row=mapping)
    compare(tb, res, path, alen, bonus)
    assert B.adt_get_device_error() == 0

    mapping[0] = -1
    lone = oracle.tree_accept(target[:1], draft[:1], tb.tokens[:1], tb.parents[:1], np.array([0, 1]),
                              B.ACCEPT_SPEC, ua[:1], us[:1])
    assert lone["sample_margin"] > SAMPLE_MARGIN
    path, alen, bonus = run_accept_gpu(target, draft, tb, B.ACCEPT_SPEC, ua, us, draft_row=mapping)
    assert B.adt_get_device_error() & B.DEVERR_BAD_INDEX
    assert alen[0] == 0 and path[0, 0] == 0 and (path[0, 1:] == -1).all()
    assert bonus[0] == lone["bonus"][0]


def test_path_longer_than_buffer_is_cut_and_flagged():
    V = 1000
    tb = synth.tree_batch([12], V, 3, chain=True)
    target = synth.f32_normal((12, V), 3, "t")
    synth.plant_path(target, tb.parents, tb.tokens, list(range(12)))
    B.adt_get_device_error()
    path, alen, bonus = run_accept_gpu(target, None, tb, B.ACCEPT_GREEDY, max_path=4)
    assert path[0].tolist() == [0, 1, 2, 3] and alen[0] == 3
    assert B.adt_get_device_error() & B.DEVERR_BAD_PATH


def _compact_inputs(layers, sizes, Hkv, D, Lmax, kv_lens, seed):
    Bn = len(sizes)
    ntot = sum(sizes)
    kc = synth.bf16_normal((layers, Bn, Hkv, Lmax, D), seed, "kc")
    vc = synth.bf16_normal((layers, Bn, Hkv, Lmax, D), seed, "vc")
    kt = synth.bf16_normal((layers, ntot, Hkv, D), seed, "kt")
    vt = synth.bf16_normal((layers, ntot, Hkv, D), seed, "vt")
    return kc, vc, kt, vt


@pytest.mark.parametrize("layers,sizes,Hkv,D,Lmax,kv,paths", [
    (32, [64], 32, 128, 2470, [2400], [[0, 5, 17, 40, 41, 63]]),
    (3, [26, 1, 9], 8, 64, 600, [512, 0, 590], [[0, 2, 11], [0], [0, 1, 2, 3, 4, 5, 6, 7, 8]]),
])
def test_compact_matches_oracle(layers, sizes, Hkv, D, Lmax, kv, paths):
    kc, vc, kt, vt = _compact_inputs(layers, sizes, Hkv, D, Lmax, kv, seed=layers + D)
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    max_path = 16
    parr = np.full((len(sizes), max_path), -1, np.int32)
    for b, p in enumerate(paths):
        parr[b, :len(p)] = p
    alen = np.array([len(p) - 1 for p in paths], np.int32)
    dev = "cuda"
    gkc, gvc = kc.to(dev), vc.to(dev)
    kv_out = torch.empty(len(sizes), dtype=torch.int32, device=dev)
    B.adt_kv_compact(gkc, gvc, i32(kv), kv_out, kt.to(dev), vt.to(dev), i32(offs), i32(parr), max_path, i32(alen),
                     B=len(sizes), Hkv=Hkv, D=D, num_layers=layers, max_kv=Lmax,
                     cache_layer_stride=kc.stride(0), cache_stride_b=kc.stride(1), cache_stride_h=kc.stride(2),
                     tree_layer_stride=kt.stride(0))
    torch.cuda.synchronize()
    rk, rv, rl = oracle.kv_compact(kc.view(torch.int16).numpy(), vc.view(torch.int16).numpy(), kv,
                                   kt.view(torch.int16).numpy(), vt.view(torch.int16).numpy(), offs, paths)
    assert np.array_equal(gkc.cpu().view(torch.int16).numpy(), rk)
    assert np.array_equal(gvc.cpu().view(torch.int16).numpy(), rv)
    assert kv_out.cpu().numpy().tolist() == rl.tolist()


def test_compact_overflow_skips_tree_and_flags():
    layers, sizes, Hkv, D, Lmax = 2, [4, 4], 2, 64, 10
    kc, vc, kt, vt = _compact_inputs(layers, sizes, Hkv, D, Lmax, None, seed=1)
    dev = "cuda"
    gkc = kc.to(dev)
    parr = np.array([[0, 1, 3, -1], [0, 2, -1, -1]], np.int32)
    alen = np.array([2, 1], np.int32)
    kv_out = torch.empty(2, dtype=torch.int32, device=dev)
    B.adt_get_device_error()
    B.adt_kv_compact(gkc, vc.to(dev), i32([8, 3]), kv_out, kt.to(dev), vt.to(dev), i32([0, 4, 8]), i32(parr), 4,
                     i32(alen), B=2, Hkv=Hkv, D=D, num_layers=layers, max_kv=Lmax,
                     cache_layer_stride=kc.stride(0), cache_stride_b=kc.stride(1), cache_stride_h=kc.stride(2),
                     tree_layer_stride=kt.stride(0))
    assert B.adt_get_device_error() & B.DEVERR_KV_RANGE
    assert kv_out.cpu().tolist() == [8, 5]
    got = gkc.cpu()
    assert torch.equal(got[:, 0], kc[:, 0])  # tree 0 (8 + 3 > 10) untouched
    assert torch.equal(got[:, 1, :, 3], kt[:, 4])


def _run_inplace(kc, vc, kv, sizes, paths, max_path=16, max_kv=None):
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    parr = np.full((len(sizes), max_path), -1, np.int32)
    for b, p in enumerate(paths):
        parr[b, :len(p)] = p
    alen = np.array([len(p) - 1 for p in paths], np.int32)
    dev = "cuda"
    gkc, gvc = kc.to(dev), vc.to(dev)
    kv_out = torch.empty(len(sizes), dtype=torch.int32, device=dev)
    layers, Bn, Hkv, Lmax, D = kc.shape
    B.adt_kv_compact_inplace(gkc, gvc, i32(kv), kv_out, i32(offs), i32(parr), max_path, i32(alen), B=Bn, Hkv=Hkv,
                             D=D, num_layers=layers, max_kv=Lmax if max_kv is None else max_kv,
                             cache_layer_stride=kc.stride(0), cache_stride_b=kc.stride(1),
                             cache_stride_h=kc.stride(2))
    torch.cuda.synchronize()
    return gkc.cpu(), gvc.cpu(), kv_out.cpu().numpy()


@pytest.mark.parametrize("layers,sizes,Hkv,D,Lmax,kv,paths", [
    (32, [64], 32, 128, 2470, [2400], [[0, 5, 17, 40, 41, 63]]),
    (3, [26, 1, 9], 8, 64, 600, [512, 0, 590], [[0, 2, 11], [0], [0, 1, 2, 3, 4, 5, 6, 7, 8]]),
    (2, [8], 4, 128, 32, [10], [[0, 2, 5]]),               # row L + 2 is written and also read
    (2, [256], 2, 64, 300, [40], [list(range(0, 256, 17))]),  # 256-node tree, 16-entry path
])
def test_compact_inplace_matches_oracle(layers, sizes, Hkv, D, Lmax, kv, paths):
    kc, vc, _, _ = _compact_inputs(layers, sizes, Hkv, D, Lmax, kv, seed=layers + D + 1)
    gk, gv, gl = _run_inplace(kc, vc, kv, sizes, paths)
    rk, rv, rl = oracle.kv_compact_inplace(kc.view(torch.int16).numpy(), vc.view(torch.int16).numpy(), kv, paths)
    assert np.array_equal(gk.view(torch.int16).numpy(), rk)
    assert np.array_equal(gv.view(torch.int16).numpy(), rv)
    assert gl.tolist() == rl.tolist()


def test_compact_inplace_rejects_bad_trees():
    kc, vc, _, _ = _compact_inputs(2, [4, 4], 2, 64, 12, None, seed=2)
    B.adt_get_device_error()
    # tree 0: rows 9 .. 12 do not fit in 12; tree 1: path entry 4 is outside its 4 nodes
    gk, gv, gl = _run_inplace(kc, vc, [9, 2], [4, 4], [[0, 1], [0, 4]])
    bits = B.adt_get_device_error()
    assert bits & B.DEVERR_KV_RANGE and bits & B.DEVERR_BAD_PATH
    assert gl.tolist() == [9, 2]
    assert torch.equal(gk, kc) and torch.equal(gv, vc)


def test_greedy_ties_take_the_lowest_index():
    """Every target row holds its largest value several times: in the same
    16-byte group, in different groups of one thread, in different threads
    and in different vocabulary slices (CTAs).  The walk's argmax is the
    lowest of those indices, as the oracle's; a child carrying a later copy
    is not accepted."""
    V = 65536
    tb = synth.tree_batch([20], V, 5)
    g = np.random.default_rng(5)
    target = g.normal(0.0, 1.0, size=(20, V)).astype(np.float32)
    for v in range(20):
        copies = sorted(g.choice(V, size=6, replace=False).tolist() + [4 * (v + 3) + 1, 4 * (v + 3) + 2])
        target[v, copies] = np.float32(9.0)
    # the root's first child carries the root row's lowest copy: accepted;
    # its first child carries a later copy of that node's row: rejected
    kids0 = [i for i in range(20) if tb.parents[i] == 0]
    low0 = int(np.flatnonzero(target[0] == 9.0)[0])
    tb.tokens[kids0[0]] = low0
    c = kids0[0]
    kids1 = [i for i in range(20) if tb.parents[i] == c]
    if kids1:
        tb.tokens[kids1[0]] = int(np.flatnonzero(target[c] == 9.0)[1])
    res = oracle.tree_accept(target, None, tb.tokens, tb.parents, tb.node_offsets, oracle.ACCEPT_GREEDY)
    path, alen, bonus = run_accept_gpu(target, None, tb, B.ACCEPT_GREEDY, max_path=16)
    compare(tb, res, path, alen, bonus)
    assert res["path"][0][:2] == [0, c]
