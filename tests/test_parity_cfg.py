"""Classifier-free guidance fused into expansion and acceptance (p and q
under CFG, Sec. 3.1 under Eq. 1; guidance scale 3.0, Sec. 5.1): the GPU
entry points read the conditional and unconditional rows and combine them on
the fly; the oracle combines first (oracle.cfg_logits) and then runs its
usual definitions.  Same bars as the plain entry points: tokens, parents,
paths bit-exact, log-probabilities and scores within 5e-5."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import ensure_built, f32, f32_rows, i32
from paper_2512_21857_gb300 import binding as B
from paper_2512_21857_gb300 import synth
from test_parity_accept_compact import ACCEPT_MARGIN, SAMPLE_MARGIN, compare
from test_parity_expand_rerank import check_expand

pytestmark = pytest.mark.gpu
SCALE = 3.0


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def run_expand_cfg(cond, uncond, fscore, fid, k, keep, T=1.0, base=0):
    F, V = cond.shape
    dev = "cuda"
    ws = B.zeroed_workspace(B.adt_tree_expand_workspace_size(F, V, k))
    ld = (V + 3) // 4 * 4
    pc = torch.zeros((F, ld), dtype=torch.float32, device=dev)
    pu = torch.zeros((F, ld), dtype=torch.float32, device=dev)
    pc[:, :V] = f32(cond)
    pu[:, :V] = f32(uncond)
    out = dict(child_token=torch.empty(F * k, dtype=torch.int32, device=dev),
               child_logp=torch.empty(F * k, dtype=torch.float32, device=dev),
               child_score=torch.empty(F * k, dtype=torch.float32, device=dev),
               child_parent=torch.empty(F * k, dtype=torch.int32, device=dev))
    keep_idx = torch.empty(keep, dtype=torch.int32, device=dev)
    ns = torch.empty(keep, dtype=torch.float32, device=dev)
    nid = torch.empty(keep, dtype=torch.int32, device=dev)
    B.adt_tree_expand_cfg(pc[:, :V], pu[:, :V], f32(fscore), None if fid is None else i32(fid), cfg_scale=SCALE, F=F,
                          V=V, k_child=k, k_keep=keep, temperature=T, child_id_base=base, keep_idx=keep_idx,
                          next_score=ns, next_id=nid, workspace=ws, **out)
    torch.cuda.synchronize()
    res = {kk: v.cpu().numpy() for kk, v in out.items()}
    res.update(keep_idx=keep_idx.cpu().numpy(), next_score=ns.cpu().numpy(), next_id=nid.cpu().numpy())
    assert int(ws[:16640].cpu().sum()) == 0
    return res


@pytest.mark.parametrize("F,V,k,keep,T", [(1, 65536, 8, 8, 1.0), (8, 65536, 8, 8, 1.0), (13, 16384, 13, 13, 0.7),
                                          (3, 4099, 5, 7, 1.0), (4, 100, 64, 100, 1.0)])
def test_expand_cfg_matches_oracle(F, V, k, keep, T):
    seed = 7000 + F * 10 + V
    cond = synth.f32_normal((F, V), seed, "cond", std=3.0)
    uncond = synth.f32_normal((F, V), seed, "uncond", std=3.0)
    fscore = synth.f32_normal((F,), seed, "fs", std=1.0) - 2.0
    fid = np.arange(F, dtype=np.int32) * 2
    got = run_expand_cfg(cond, uncond, fscore, fid, k, keep, T, base=5)
    ref = oracle.tree_expand(oracle.cfg_logits(cond, uncond, SCALE), fscore, k, keep, temperature=T, frontier_id=fid,
                             child_id_base=5)
    check_expand(got, ref, keep)
    # guidance changed the selection (the test would not see a missing combine otherwise)
    plain = oracle.tree_expand(cond, fscore, k, keep, temperature=T, frontier_id=fid, child_id_base=5)
    assert not np.array_equal(plain["child_token"], ref["child_token"])


def run_accept_cfg(tc, tu, dc, du, tb, mode, ua=None, us=None, T=1.0, max_path=16):
    dev = "cuda"
    Bn = len(tb.node_offsets) - 1
    path = torch.empty((Bn, max_path), dtype=torch.int32, device=dev)
    alen = torch.empty(Bn, dtype=torch.int32, device=dev)
    bonus = torch.empty(Bn, dtype=torch.int32, device=dev)
    opt = lambda x: None if x is None else f32(x)  # noqa: E731
    rows_ = lambda x: None if x is None else f32_rows(x)  # noqa: E731
    B.adt_tree_accept_cfg(rows_(tc), rows_(tu), rows_(dc), rows_(du), i32(tb.tokens), i32(tb.parents),
                          i32(tb.node_offsets), cfg_scale=SCALE, B=Bn, V=tc.shape[1],
                          max_nodes=int(np.diff(tb.node_offsets).max()),
                          mode=mode, u_accept=opt(ua), u_sample=opt(us), temperature=T, path=path,
                          max_path=max_path, accept_len=alen, bonus_token=bonus)
    torch.cuda.synchronize()
    return path.cpu().numpy(), alen.cpu().numpy(), bonus.cpu().numpy()


def rows(tb, V, seed, plant):
    ntot = int(tb.node_offsets[-1])
    dc = synth.f32_normal((ntot, V), seed, "dc", std=3.0)
    du = synth.f32_normal((ntot, V), seed, "du", std=3.0)
    tc = (dc + synth.f32_normal((ntot, V), seed, "nc", std=0.3)).astype(np.float32)
    tu = (du + synth.f32_normal((ntot, V), seed, "nu", std=0.3)).astype(np.float32)
    if plant:  # raise conditional target entries so that a seeded path is the guided greedy one
        g = synth.rng(seed, "plant")
        for b in range(len(tb.node_offsets) - 1):
            lo, hi = tb.node_offsets[b], tb.node_offsets[b + 1]
            par = tb.parents[lo:hi]
            full = oracle.ancestor_path(par, int(g.integers(0, hi - lo)))
            synth.plant_path(tc[lo:hi], par, tb.tokens[lo:hi], full[:int(g.integers(1, len(full) + 1))], boost=8.0)
    return tc, tu, dc, du


@pytest.mark.parametrize("sizes,V", [([26], 16384), ([64, 1, 33, 7], 65536), ([9, 4], 4099)])
def test_accept_cfg_greedy_matches_oracle(sizes, V):
    seed = 900 + sum(sizes)
    tb = synth.tree_batch(sizes, V, seed)
    tc, tu, _, _ = rows(tb, V, seed, plant=True)
    res = oracle.tree_accept(oracle.cfg_logits(tc, tu, SCALE), None, tb.tokens, tb.parents, tb.node_offsets,
                             oracle.ACCEPT_GREEDY)
    compare(tb, res, *run_accept_cfg(tc, tu, None, None, tb, B.ACCEPT_GREEDY))
    assert res["accept_len"].max() >= 1


@pytest.mark.parametrize("mode", [B.ACCEPT_SPEC, B.ACCEPT_SPEC_DET])
@pytest.mark.parametrize("sizes,V,T", [([26], 16384, 1.0), ([64, 12, 50], 65536, 1.0), ([16, 9], 16384, 0.7)])
def test_accept_cfg_sampling_matches_oracle(mode, sizes, V, T):
    checked = 0
    for rep in range(3):
        seed = 41 * rep + sum(sizes) + V + mode
        tb = synth.tree_batch(sizes, V, seed)
        tc, tu, dc, du = rows(tb, V, seed, plant=True)
        ntot = int(tb.node_offsets[-1])
        ua, us = synth.uniforms(ntot, seed, "ua"), synth.uniforms(ntot, seed, "us")
        res = oracle.tree_accept(oracle.cfg_logits(tc, tu, SCALE), oracle.cfg_logits(dc, du, SCALE), tb.tokens,
                                 tb.parents, tb.node_offsets, mode, ua, us, T)
        if res["accept_margin"] < ACCEPT_MARGIN or res["sample_margin"] < SAMPLE_MARGIN:
            continue  # near tie: re-draw
        compare(tb, res, *run_accept_cfg(tc, tu, dc, du, tb, mode, ua, us, T))
        checked += 1
    assert checked >= 2
