"""GPU draft-tree expansion and rerank vs the oracle.  Token ids, parents,
candidate indices and depths must match bit for bit; log-probabilities and
scores (fp32 outputs of an fp64 formula with fp32 exponentials inside the
normaliser) within 5e-5.  Where the oracle's own selection has a near tie
(score gap < 1e-5), the GPU selection is checked for validity instead."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import ensure_built, f32, grow_candidates_gpu, i32
from paper_2512_21857_gb300 import binding as B
from paper_2512_21857_gb300 import synth

pytestmark = pytest.mark.gpu
TOL = 5e-5
TIE = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def run_expand(logits, fscore, fid, k, keep, T=1.0, base=0, ws=None):
    F, V = logits.shape
    dev = "cuda"
    if ws is None:
        ws = B.zeroed_workspace(B.adt_tree_expand_workspace_size(F, V, k))
    out = dict(child_token=torch.empty(F * k, dtype=torch.int32, device=dev),
               child_logp=torch.empty(F * k, dtype=torch.float32, device=dev),
               child_score=torch.empty(F * k, dtype=torch.float32, device=dev),
               child_parent=torch.empty(F * k, dtype=torch.int32, device=dev))
    keep_idx = torch.empty(keep, dtype=torch.int32, device=dev)
    ns = torch.empty(keep, dtype=torch.float32, device=dev)
    nid = torch.empty(keep, dtype=torch.int32, device=dev)
    ld = (V + 3) // 4 * 4  # rows padded to a multiple of 4 floats, as the ABI requires
    padded = torch.zeros((F, ld), dtype=torch.float32, device=dev)
    padded[:, :V] = f32(logits)
    B.adt_tree_expand(padded[:, :V], f32(fscore), None if fid is None else i32(fid), F=F, V=V, k_child=k,
                      k_keep=keep, temperature=T, child_id_base=base, keep_idx=keep_idx, next_score=ns,
                      next_id=nid, workspace=ws, **out)
    torch.cuda.synchronize()
    res = {kk: v.cpu().numpy() for kk, v in out.items()}
    res.update(keep_idx=keep_idx.cpu().numpy(), next_score=ns.cpu().numpy(), next_id=nid.cpu().numpy())
    # the completion counters (start of the workspace) are back at zero
    assert int(ws[:16640].cpu().sum()) == 0
    return res, ws


def near_tie(scores, count):
    s = np.sort(np.asarray(scores, np.float64))[::-1][:count + 1]
    return len(s) > 1 and np.min(np.abs(np.diff(s))) < TIE


def check_expand(got, ref, k_keep):
    assert np.array_equal(got["child_token"], ref["child_token"])
    assert np.array_equal(got["child_parent"], ref["child_parent"])
    assert np.abs(got["child_logp"] - ref["child_logp"]).max() <= TOL
    assert np.abs(got["child_score"] - ref["child_score"]).max() <= TOL
    if near_tie(ref["child_score"], k_keep):
        # valid selection w.r.t. the GPU's own scores
        order = sorted(range(len(got["child_score"])), key=lambda c: (-float(got["child_score"][c]), c))
        assert got["keep_idx"].tolist() == order[:k_keep]
    else:
        assert np.array_equal(got["keep_idx"], ref["keep_idx"])
        assert np.array_equal(got["next_id"], ref["next_id"])
    assert np.array_equal(got["next_score"], got["child_score"][got["keep_idx"]])


@pytest.mark.parametrize("F,V,k,keep,T", [
    (1, 65536, 8, 8, 1.0),       # first layer of the 7B-shape tree
    (8, 65536, 8, 8, 1.0),       # later layers
    (13, 16384, 13, 13, 1.0),    # Anole width bound
    (39, 16384, 39, 39, 1.0),    # LlamaGen width bound
    (4, 100, 64, 100, 1.0),      # k > chunk rows, k_keep > 64
    (3, 4099, 5, 7, 0.7),        # ragged last chunk, temperature
    (2, 7, 7, 14, 1.0),          # V == k
])
def test_expand_matches_oracle(F, V, k, keep, T):
    seed = F * 1000 + V
    logits = synth.f32_normal((F, V), seed, "logits", std=3.0)
    fscore = synth.f32_normal((F,), seed, "fs", std=1.0) - 2.0
    fid = np.arange(F, dtype=np.int32) * 3 + 1
    got, _ = run_expand(logits, fscore, fid, k, keep, T, base=17)
    ref = oracle.tree_expand(logits, fscore, k, keep, temperature=T, frontier_id=fid, child_id_base=17)
    check_expand(got, ref, keep)


def test_expand_ties_take_lowest_index():
    V = 20000
    logits = np.zeros((2, V), np.float32)
    logits[0, 5000:5003] = 1.0      # three-way tie at the top
    logits[0, 17] = -0.0            # -0.0 equals +0.0
    logits[1, :] = np.float32(2.5)  # a row of ties: lowest indices win
    fscore = np.array([0.0, -1.0], np.float32)
    got, _ = run_expand(logits, fscore, None, 6, 5)
    ref = oracle.tree_expand(logits, fscore, 6, 5)
    assert got["child_token"][:6].tolist() == [5000, 5001, 5002, 0, 1, 2]
    assert got["child_token"][6:].tolist() == [0, 1, 2, 3, 4, 5]
    check_expand(got, ref, 5)


def test_expand_shared_workspace_across_shapes_and_repeats():
    """One workspace serves calls of different F in any order (a step's
    first layer has F = 1, later ones F = k), repeatedly."""
    V = 65536
    ws = B.zeroed_workspace(B.adt_tree_expand_workspace_size(8, V, 8))
    rows1 = synth.f32_normal((1, V), 11, "a")
    rows8 = synth.f32_normal((8, V), 11, "b")
    ref1 = oracle.tree_expand(rows1, np.zeros(1, np.float32), 8, 8)
    ref8 = oracle.tree_expand(rows8, np.zeros(8, np.float32), 8, 8)
    for _ in range(3):
        g1, _ = run_expand(rows1, np.zeros(1, np.float32), None, 8, 8, ws=ws)
        check_expand(g1, ref1, 8)
        g8, _ = run_expand(rows8, np.zeros(8, np.float32), None, 8, 8, ws=ws)
        check_expand(g8, ref8, 8)


def _oracle_grow(draft_rows, k, depth, root_token, n_nodes):
    tok, sc, par = [], [], []
    fscore = np.zeros(1, np.float32)
    fid = np.array([-1], np.int32)
    ties = False
    for d in range(depth):
        F = len(fscore)
        res = oracle.tree_expand(draft_rows[d][:F], fscore, k, min(k, F * k), frontier_id=fid,
                                 child_id_base=len(tok))
        ties |= near_tie(res["child_score"], min(k, F * k))
        tok += res["child_token"].tolist()
        sc += res["child_score"].tolist()
        par += res["child_parent"].tolist()
        fscore, fid = res["next_score"], res["next_id"]
    n = min(n_nodes, len(tok) + 1)
    ties |= near_tie(sc, n - 1)
    tree = oracle.tree_rerank(tok, np.array(sc, np.float32), par, root_token, n)
    return tree, np.array(tok), np.array(sc, np.float32), np.array(par), ties


@pytest.mark.parametrize("V,k,depth,n", [(65536, 8, 6, 64), (16384, 10, 5, 64), (16384, 4, 9, 30),
                                         (1000, 3, 2, 12)])
def test_grown_tree_matches_oracle(V, k, depth, n):
    """d-hat expand calls chained on the device, then the final rerank: the
    draft phase of one ADT-Tree step (Sec. 3.1, Fig. 5, Eq. 4)."""
    seed = V + k * 10 + depth
    rows = [synth.f32_normal((k, V), seed, f"draft{d}", std=3.0) for d in range(depth)]
    g = grow_candidates_gpu(rows, k, depth, 4242, n)
    tree, tok, sc, par, ties = _oracle_grow(rows, k, depth, 4242, n)
    assert not ties, "near tie in the seeded draft rows: pick another seed"
    assert np.array_equal(g["pool_token"], tok)
    assert np.array_equal(g["pool_parent"], par)
    assert np.abs(g["pool_score"] - sc).max() <= TOL
    for key in ("tokens", "parents", "cand_index", "depth"):
        assert np.array_equal(g["tree"][key], tree[key]), key


def _random_pool(C, seed):
    """A valid depth-major candidate pool: parents precede children and a
    child's score never exceeds its parent's."""
    g = np.random.default_rng(seed)
    tok = g.integers(0, 50000, C).astype(np.int32)
    par = np.full(C, -1, np.int32)
    sc = np.zeros(C, np.float32)
    layer_start, layer = 0, 0
    i = 0
    while i < C:
        width = int(g.integers(1, 40))
        prev = list(range(layer_start, i)) if layer else []
        start = i
        for _ in range(width):
            if i >= C:
                break
            if prev:
                p = int(g.choice(prev))
                par[i] = p
                sc[i] = np.float32(sc[p] - np.float32(abs(g.standard_normal()) + 1e-3))
            else:
                sc[i] = np.float32(-abs(g.standard_normal()))
            i += 1
        layer_start, layer = start, layer + 1
    return tok, sc, par


@pytest.mark.parametrize("C,n", [(328, 64), (1534, 64), (5000, 4096), (9, 10), (70, 1),
                                 (64, 65), (100, 65), (1024, 64), (600, 200), (63, 64), (1024, 1025)])
@pytest.mark.parametrize("flat", [False, True])
def test_rerank_matches_oracle(C, n, flat):
    """Small pools select by a bound when n - 1 <= 64 and C >= 64, by full
    ranking otherwise; pools past 1024 candidates take the radix kernel.
    flat: every score equal, so the candidate index alone decides."""
    tok, sc, par = _random_pool(C, seed=C + n)
    if flat:
        sc = np.zeros_like(sc)
    dev = "cuda"
    res = dict(tokens=torch.empty(n, dtype=torch.int32, device=dev),
               parents=torch.empty(n, dtype=torch.int32, device=dev),
               cand_index=torch.empty(n, dtype=torch.int32, device=dev),
               depth=torch.empty(n, dtype=torch.int32, device=dev))
    ws = B.zeroed_workspace(B.adt_tree_rerank_workspace_size(C))
    B.adt_tree_rerank(i32(tok), f32(sc), i32(par), C, i32([7]), n, workspace=ws, **res)
    torch.cuda.synchronize()
    ref = oracle.tree_rerank(tok, sc, par, 7, n)
    for key in res:
        assert np.array_equal(res[key].cpu().numpy(), ref[key]), key


def test_expand_masked_vocabulary_few_finite_values_per_cta():
    """Logits -inf (a masked vocabulary) except one or two per eighth of the
    row: every CTA of the row holds fewer than k finite values, so its bound
    falls to -inf and the overflow path ranks its whole share; the k
    children are the row's finite logits, best first."""
    V, F, k = 65536, 2, 8
    g = np.random.default_rng(3)
    logits = np.full((F, V), -np.inf, np.float32)
    for r in range(F):
        for c in range(8):
            pos = g.choice(8192, size=1 + (c % 2), replace=False) + 8192 * c
            logits[r, pos] = g.normal(0.0, 3.0, size=len(pos)).astype(np.float32)
    fscore = np.array([-0.5, -1.5], np.float32)
    got, _ = run_expand(logits, fscore, None, k, 8)
    ref = oracle.tree_expand(logits, fscore, k, 8)
    assert np.isfinite(ref["child_score"]).all()
    check_expand(got, ref, 8)


def test_expand_finite_values_held_by_one_thread():
    """The only finite logits sit where one thread holds them (indices 0-3
    and 1024 of an 1100-wide row, one CTA): fewer than k lanes have a finite
    maximum, the bound is -inf, and every logit of the share is a candidate
    without overflowing the candidate buffer."""
    F, k = 3, 5
    for V in (1100,):
        logits = np.full((F, V), -np.inf, np.float32)
        g = np.random.default_rng(V)
        for r in range(F):
            logits[r, [0, 1, 2, 3, 1024]] = g.normal(0.0, 2.0, size=5).astype(np.float32)
        fscore = np.zeros(F, np.float32)
        got, _ = run_expand(logits, fscore, None, k, 5)
        ref = oracle.tree_expand(logits, fscore, k, 5)
        assert np.isfinite(ref["child_score"]).all()
        check_expand(got, ref, 5)


@pytest.mark.parametrize("n_top", [64, 65, 200, 1024])
def test_expand_many_values_at_the_bound(n_top):
    """n_top copies of the row's largest value spread over one CTA's eighth
    of the row: at least k of that CTA's warp maxima are that value, so its
    bound equals it and exactly n_top values are candidates.  Up to 64 they
    are ranked by groups of 16 threads, beyond that by a warp per key (1024:
    the candidate buffer's capacity).  The row's children are the k copies
    of lowest index."""
    V, F, k = 65536, 2, 8
    g = np.random.default_rng(n_top)
    logits = g.normal(0.0, 1.0, size=(F, V)).astype(np.float32)
    pos = np.sort(g.choice(8192, size=n_top, replace=False)) + 8192 * 3
    assert len(set((pos % 1024) // 32)) >= k  # copies in at least k warps of that CTA
    logits[0, pos] = np.float32(7.0)
    fscore = np.array([-1.0, -0.25], np.float32)
    got, _ = run_expand(logits, fscore, None, k, 8)
    ref = oracle.tree_expand(logits, fscore, k, 8)
    assert got["child_token"][:k].tolist() == pos[:k].tolist()
    check_expand(got, ref, 8)


def test_expand_without_next_frontier():
    """keep_idx, next_score and next_id NULL (a tree's last layer): the
    children are the oracle's, and the shared workspace's counter stays at
    zero for the next call, which selects a frontier as usual."""
    F, V, k = 8, 65536, 8
    logits = synth.f32_normal((F, V), 77, "logits", std=3.0)
    fscore = synth.f32_normal((F,), 77, "fs", std=1.0) - 2.0
    ref = oracle.tree_expand(logits, fscore, k, k)
    dev = "cuda"
    ws = B.zeroed_workspace(B.adt_tree_expand_workspace_size(F, V, k))
    out = dict(child_token=torch.empty(F * k, dtype=torch.int32, device=dev),
               child_logp=torch.empty(F * k, dtype=torch.float32, device=dev),
               child_score=torch.empty(F * k, dtype=torch.float32, device=dev),
               child_parent=torch.empty(F * k, dtype=torch.int32, device=dev))
    B.adt_tree_expand(f32(logits), f32(fscore), None, F=F, V=V, k_child=k, k_keep=k, keep_idx=None,
                      workspace=ws, **out)
    torch.cuda.synchronize()
    assert np.array_equal(out["child_token"].cpu().numpy(), ref["child_token"])
    assert np.array_equal(out["child_parent"].cpu().numpy(), ref["child_parent"])
    assert np.abs(out["child_score"].cpu().numpy() - ref["child_score"]).max() <= TOL
    assert int(ws[:16640].cpu().sum()) == 0
    got, _ = run_expand(logits, fscore, None, k, k, ws=ws)
    check_expand(got, ref, k)
    with pytest.raises(B.AdtError):
        B.adt_tree_expand(f32(logits), f32(fscore), None, F=F, V=V, k_child=k, k_keep=k, keep_idx=None,
                          next_score=torch.empty(k, dtype=torch.float32, device=dev), workspace=ws, **out)
