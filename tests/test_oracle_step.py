"""Pins of the oracle's whole-step composition (oracle/step.py) to worked
examples: the layer-wise draft growth of Sec. 3.1 / Fig. 5 with the final
top-N selection of Eq. 4, and one verify step over two images whose every
output can be written down by hand."""
import json
import math
import os

import numpy as np

from oracle.step import draft_tree, verify_step
import oracle


def _rows(spec, V):
    """Rows of a fixture layer: {token: logit} dicts, 0 elsewhere."""
    out = np.zeros((len(spec), V), np.float32)
    for r, d in enumerate(spec):
        for tok, val in d.items():
            out[r, int(tok)] = val
    return out


def test_draft_tree_golden(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "draft_tree_small.json")))
    V = g["V"]
    rows = [_rows(g["rows"][f"layer{d}"], V) for d in range(g["depth"])]
    assert [len(r) for r in rows] == g["expected_frontier_sizes"]
    t = draft_tree(rows, g["k"], g["depth"], g["root_token"], g["n_nodes"])
    assert t["pool_token"].tolist() == g["expected_pool_token"]
    assert t["pool_parent"].tolist() == g["expected_pool_parent"]
    assert np.abs(t["pool_score"] - np.array(g["expected_pool_score"])).max() < 2e-6
    assert t["tokens"].tolist() == g["expected_tokens"]
    assert t["parents"].tolist() == g["expected_parents"]
    assert t["cand_index"].tolist() == g["expected_cand_index"]
    assert t["depth"].tolist() == g["expected_depth"]


def test_draft_tree_golden_fails_with_frontier_rows_swapped(golden_dir):
    """The next layer's rows follow the frontier's best-first order: fed in
    candidate order (c2's row before c4's), the tree comes out different,
    so the fixture tells the two readings apart."""
    g = json.load(open(os.path.join(golden_dir, "draft_tree_small.json")))
    V = g["V"]
    rows = [_rows(g["rows"][f"layer{d}"], V) for d in range(g["depth"])]
    rows[2] = rows[2][::-1].copy()
    t = draft_tree(rows, g["k"], g["depth"], g["root_token"], g["n_nodes"])
    got = (t["tokens"].tolist(), t["parents"].tolist(), t["cand_index"].tolist())
    assert got != (g["expected_tokens"], g["expected_parents"], g["expected_cand_index"])


def test_verify_step_worked_example():
    """Two images, depth 1, width 2 (trees: root + its two best tokens),
    one layer, one head of dimension 2 with q = 0, so that every node's
    attention output is the mean of the values it sees and its lse is the
    log of their count; greedy acceptance of a planted path; the commit of
    the accepted rows after each prefix.  Expected values worked by hand."""
    V = 4
    rows0 = [np.array([[0.0, 3.0, 1.0, 2.0]], np.float32)]   # image 0: tokens 1 then 3
    rows1 = [np.array([[1.0, 0.0, 0.5, 0.0]], np.float32)]   # image 1: tokens 0 then 2
    q = np.zeros((1, 6, 1, 2))
    v_cache = np.zeros((1, 2, 1, 4, 2))
    v_cache[0, 0, 0, 0] = (1, 0)
    v_cache[0, 0, 0, 1] = (0, 1)
    v_cache[0, 1, 0, 0] = (2, 2)
    k_cache = v_cache.copy()
    v_tree = np.array([(0, 0), (3, 0), (0, 3), (4, 4), (1, -1), (-1, 1)], float).reshape(1, 6, 1, 2)
    k_tree = v_tree.copy()
    target = np.zeros((6, V), np.float32)
    target[0, 3] = 5.0   # image 0 root: argmax 3 = node 2's token -> accepted
    target[2, 1] = 4.0   # node 2 (a leaf): bonus 1
    target[3, 1] = 7.0   # image 1 root: argmax 1, no child holds it -> bonus 1
    res = verify_step([rows0, rows1], [2, 2], [1, 1], [0, 2], 3, q, k_cache, v_cache, [2, 1], k_tree, v_tree,
                      target, np.zeros(6, np.float32), np.zeros(6, np.float32), oracle.ACCEPT_GREEDY)
    assert res["node_offsets"].tolist() == [0, 3, 6]
    assert res["tokens"].tolist() == [0, 1, 3, 2, 0, 2]
    assert res["parents"].tolist() == [-1, 0, 0, -1, 0, 0]
    out, lse = res["attn"][0]
    want = np.array([(1 / 3, 1 / 3), (1.0, 0.25), (0.25, 1.0), (3.0, 3.0), (7 / 3, 5 / 3), (5 / 3, 7 / 3)])
    assert np.abs(out[:, 0, :] - want).max() < 1e-12
    assert np.abs(lse[:, 0] - np.log([3, 4, 4, 2, 3, 3])).max() < 1e-12
    acc = res["accept"]
    assert acc["path"] == [[0, 2], [0]]
    assert acc["accept_len"].tolist() == [1, 0]
    assert acc["bonus"].tolist() == [1, 1]
    assert res["kv_len"].tolist() == [4, 2]
    vc = res["v_cache"][0, :, 0]
    assert vc[0].tolist() == [[1, 0], [0, 1], [0, 0], [0, 3]]
    assert vc[1].tolist() == [[2, 2], [4, 4], [0, 0], [0, 0]]
    assert np.array_equal(res["k_cache"], res["v_cache"])
    assert math.isclose(float(lse[0, 0]), math.log(3))
