"""Pins of the oracle's draft-tree expansion and final rerank (Sec. 3.1,
Eq. 4, Fig. 5): hand-derived fixtures, another library's sort and
logsumexp, closed forms (uniform row -> -ln V) and invariants."""
import json
import math
import os

import numpy as np
import pytest
from scipy.special import logsumexp

import oracle
from paper_2512_21857_gb300 import synth


def test_expand_golden(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "expand_small.json")))
    res = oracle.tree_expand(np.array(g["logits"], np.float32), np.array(g["frontier_score"], np.float32),
                             g["k_child"], g["k_keep"])
    assert res["child_token"].tolist() == g["expected_child_token"]
    assert res["keep_idx"].tolist() == g["expected_keep_idx"]
    assert np.allclose(res["child_logp"][5:], g["expected_row1_logp"], atol=1e-6)
    lse0 = math.log(sum(math.exp(v) for v in g["expected_row0_lse_terms"]))
    assert abs(res["lse"][0] - lse0) < 1e-12
    assert res["child_parent"].tolist() == [0] * 5 + [1] * 5


@pytest.mark.parametrize("V,k,T", [(50, 7, 1.0), (1000, 64, 1.0), (16384, 8, 1.0), (300, 13, 0.7)])
def test_expand_topk_matches_stable_argsort_and_scipy_lse(V, k, T):
    F = 5
    logits = synth.f32_normal((F, V), 3, "lg")
    logits[1, 10:20] = logits[1, 10]  # a block of ties
    logits[2, :] = np.round(logits[2, :])  # many ties
    ps = synth.f32_normal((F,), 3, "ps", std=1.0) - 5
    res = oracle.tree_expand(logits, ps, k, min(F * k, 9), temperature=T)
    for r in range(F):
        x = (logits[r] / np.float32(T)).astype(np.float32) if T != 1.0 else logits[r]
        order = np.argsort(-x.astype(np.float64), kind="stable")[:k]
        assert res["child_token"][r * k:(r + 1) * k].tolist() == order.tolist()
        lse = logsumexp(x.astype(np.float64))
        assert abs(res["lse"][r] - lse) < 1e-12 * max(1, abs(lse))
        lp = x[order].astype(np.float64) - lse
        np.testing.assert_array_equal(res["child_logp"][r * k:(r + 1) * k], lp.astype(np.float32))
    # next frontier = brute-force best by (score desc, index asc)
    cands = sorted(range(F * k), key=lambda c: (-float(res["child_score"][c]), c))
    assert res["keep_idx"].tolist() == cands[:len(res["keep_idx"])]


def test_expand_probabilities_sum_to_one_and_scores_decrease():
    V = 37
    logits = synth.f32_normal((3, V), 9, "lg")
    ps = np.array([0.0, -1.5, -3.25], np.float32)
    res = oracle.tree_expand(logits, ps, V, 3)
    for r in range(3):
        lp = res["child_logp"][r * V:(r + 1) * V].astype(np.float64)
        assert abs(math.fsum(np.exp(lp)) - 1.0) < 1e-6
        assert (lp <= 0).all()
        assert (res["child_score"][r * V:(r + 1) * V] <= ps[r]).all()


def test_expand_uniform_row_closed_form():
    V = 1024
    res = oracle.tree_expand(np.full((1, V), 3.5, np.float32), np.zeros(1, np.float32), 4, 2)
    assert res["child_token"].tolist() == [0, 1, 2, 3]
    assert res["keep_idx"].tolist() == [0, 1]
    assert np.allclose(res["child_logp"], -math.log(V), atol=1e-6)


def test_expand_temperature_scaling_is_exact():
    """logits * 2 at T = 2 equals logits at T = 1 (x*2/2 is exact in fp32)."""
    lg = synth.f32_normal((4, 500), 4, "lg")
    ps = np.zeros(4, np.float32)
    a = oracle.tree_expand(lg, ps, 6, 5, temperature=1.0)
    b = oracle.tree_expand(lg * np.float32(2), ps, 6, 5, temperature=2.0)
    for key in ("child_token", "child_logp", "child_score", "keep_idx"):
        np.testing.assert_array_equal(a[key], b[key])


def test_rerank_golden(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "rerank_small.json")))
    res = oracle.tree_rerank(g["cand_token"], np.array(g["cand_score"], np.float32), g["cand_parent"],
                             g["root_token"], g["n_nodes"])
    assert res["tokens"].tolist() == g["expected_tokens"]
    assert res["parents"].tolist() == g["expected_parents"]
    assert res["cand_index"].tolist() == g["expected_cand_index"]
    assert res["depth"].tolist() == g["expected_depth"]


def _grow(V, k, depth, seed, row_std=3.0):
    """Run the oracle expansion layer by layer on random draft rows;
    returns the candidate pool (token, score, parent) in depth-major order."""
    tok, sc, par = [], [], []
    fscore = np.zeros(1, np.float32)
    fid = np.array([-1], np.int32)
    for d in range(depth):
        lg = synth.f32_normal((len(fscore), V), seed, f"draft{d}", std=row_std)
        res = oracle.tree_expand(lg, fscore, k, k, frontier_id=fid, child_id_base=len(tok))
        tok += res["child_token"].tolist()
        sc += res["child_score"].tolist()
        par += res["child_parent"].tolist()
        fscore, fid = res["next_score"], res["next_id"]
    return np.array(tok, np.int32), np.array(sc, np.float32), np.array(par, np.int32)


@pytest.mark.parametrize("V,k,depth,n", [(64, 3, 4, 12), (500, 8, 6, 64), (100, 2, 5, 11)])
def test_rerank_is_top_scores_and_ancestor_closed(V, k, depth, n):
    tok, sc, par = _grow(V, k, depth, seed=21)
    res = oracle.tree_rerank(tok, sc, par, 9, n)
    chosen = sorted(range(len(sc)), key=lambda c: (-float(sc[c]), c))[:n - 1]
    assert res["cand_index"][1:].tolist() == sorted(chosen)
    for i in range(1, n):
        p = res["parents"][i]
        assert 0 <= p < i
        c = res["cand_index"][i]
        assert res["tokens"][i] == tok[c]
        assert (p == 0 and par[c] == -1) or res["cand_index"][p] == par[c]
        assert res["depth"][i] == res["depth"][p] + 1


def test_rerank_child_tied_with_parent_keeps_parent():
    # a one-hot-like row: log q(top) rounds to 0, so the child ties its parent
    lg = np.zeros((1, 8), np.float32)
    lg[0, 5] = 1000.0
    r1 = oracle.tree_expand(lg, np.zeros(1, np.float32), 2, 1, frontier_id=np.array([-1]))
    assert r1["child_logp"][0] == 0.0
    r2 = oracle.tree_expand(lg, r1["next_score"], 2, 1, frontier_id=r1["next_id"], child_id_base=2)
    tok = np.concatenate([r1["child_token"], r2["child_token"]])
    sc = np.concatenate([r1["child_score"], r2["child_score"]])
    par = np.concatenate([r1["child_parent"], r2["child_parent"]])
    assert sc[0] == sc[2] == 0.0
    res = oracle.tree_rerank(tok, sc, par, 1, 3)
    assert res["cand_index"].tolist() == [-1, 0, 2]
    assert res["parents"].tolist() == [-1, 0, 1]
