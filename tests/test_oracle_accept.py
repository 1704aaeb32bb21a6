"""Pins of the oracle's acceptance walk (Sec. 3.1, Eq. 1; T in {0, 1},
Sec. 5.1): hand-derived fixtures, planted greedy paths, an independent
networkx walk, and the losslessness the paper claims (Sec. 5.1, 5.2: the
generation distribution is unchanged), checked by chi-square tests."""
import json
import os

import networkx as nx
import numpy as np
import pytest
from scipy.stats import chisquare

import oracle
from paper_2512_21857_gb300 import synth


def _rows(p):
    return np.log(np.asarray(p, np.float64)).astype(np.float32)


def test_accept_golden(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "accept_small.json")))
    for c in g["cases"]:
        n = len(c["parents"])
        res = oracle.tree_accept(_rows(c["target_p"]), None if c["draft_p"] is None else _rows(c["draft_p"]),
                                 c["tokens"], c["parents"], [0, n], c["mode"],
                                 np.array(c["u_accept"], np.float32), np.array(c["u_sample"], np.float32))
        assert res["path"][0] == c["expected_path"], c["name"]
        assert res["accept_len"][0] == len(c["expected_path"]) - 1
        assert res["bonus"][0] == c["expected_bonus"], c["name"]
        assert res["min_margin"] > 1e-3


@pytest.mark.parametrize("seed", range(6))
def test_greedy_planted_path(seed):
    V, n = 300, 26
    parents = synth.random_tree(n, seed, "t")
    tokens = synth.tree_tokens(parents, V, seed)
    target = synth.f32_normal((n, V), seed, "target")
    # plant a root-to-leaf path (or a prefix of one) chosen from the seed
    g = synth.rng(seed, "plant")
    leaf = int(g.integers(1, n))
    full = oracle.ancestor_path(parents, leaf)
    a = int(g.integers(0, len(full)))
    planted = full[:a + 1]
    # make sure the node where the walk stops does not by chance point at a child
    stop = planted[-1]
    kids = oracle.children(parents, stop)
    row = target[stop]
    for c in kids:
        row[tokens[c]] = row.min() - 1
    synth.plant_path(target, parents, tokens, planted)
    res = oracle.tree_accept(target, None, tokens, parents, [0, n], oracle.ACCEPT_GREEDY)
    assert res["path"][0] == planted
    assert res["accept_len"][0] == a
    assert res["bonus"][0] == int(np.argmax(target[planted[-1]]))


@pytest.mark.parametrize("seed", range(4))
def test_greedy_equals_independent_argmax_walk(seed):
    V, sizes = 40, [7, 16, 1, 33]
    tb = synth.tree_batch(sizes, V, seed)
    ntot = int(tb.node_offsets[-1])
    draft = synth.f32_normal((ntot, V), seed, "d")
    target = draft + synth.f32_normal((ntot, V), seed, "noise", std=0.3)  # correlated: paths get accepted
    res = oracle.tree_accept(target, None, tb.tokens, tb.parents, tb.node_offsets, oracle.ACCEPT_GREEDY)
    for b in range(len(sizes)):
        lo, hi = tb.node_offsets[b], tb.node_offsets[b + 1]
        G = nx.DiGraph()
        G.add_nodes_from(range(hi - lo))
        G.add_edges_from((int(tb.parents[lo + t]), t) for t in range(1, hi - lo))
        v, path = 0, [0]
        while True:
            g = int(np.argmax(target[lo + v]))
            m = [c for c in sorted(G.successors(v)) if tb.tokens[lo + c] == g]
            if not m:
                break
            v = m[0]
            path.append(v)
        assert res["path"][b] == path
        assert res["bonus"][b] == int(np.argmax(target[lo + v]))
        assert res["accept_len"][b] == len(path) - 1


@pytest.mark.parametrize("mode", [oracle.ACCEPT_GREEDY, oracle.ACCEPT_SPEC, oracle.ACCEPT_SPEC_DET])
def test_accept_len_never_exceeds_depth(mode):
    V = 16
    for seed in range(10):
        tb = synth.tree_batch([26, 9], V, seed)
        ntot = int(tb.node_offsets[-1])
        draft = synth.f32_normal((ntot, V), seed, "d", std=1.0)
        target = draft + synth.f32_normal((ntot, V), seed, "n", std=0.2)
        res = oracle.tree_accept(target, draft, tb.tokens, tb.parents, tb.node_offsets, mode,
                                 synth.uniforms(ntot, seed, "ua"), synth.uniforms(ntot, seed, "us"))
        for b in range(2):
            lo = tb.node_offsets[b]
            par = tb.parents[lo:tb.node_offsets[b + 1]]
            depth = max(len(oracle.ancestor_path(par, t)) - 1 for t in range(len(par)))
            assert 0 <= res["accept_len"][b] <= depth
            path = res["path"][b]
            for x, y in zip(path[:-1], path[1:]):
                assert par[y] == x
            assert 0 <= res["bonus"][b] < V


def _first_two_tokens(res, tokens, lo=0):
    path = res["path"][0]
    seq = [int(tokens[lo + c]) for c in path[1:]] + [int(res["bonus"][0])]
    return seq


@pytest.mark.slow
@pytest.mark.parametrize("mode", [oracle.ACCEPT_SPEC_DET, oracle.ACCEPT_SPEC])
def test_losslessness_chi_square(mode):
    """The first emitted token must follow p(root), and the second, given
    that the first was a drafted child x, must follow p(child x) (Sec. 5.1:
    the acceptance conditions are not relaxed, so the output distribution
    is the target's).  SPEC needs children drawn without replacement from
    q; SPEC_DET holds for any fixed candidates."""
    V = 5
    parents = np.array([-1, 0, 0, 0, 1, 1], np.int32)
    tp = np.array([[0.05, 0.3, 0.25, 0.1, 0.3],
                   [0.4, 0.1, 0.2, 0.2, 0.1],
                   [0.2, 0.2, 0.2, 0.2, 0.2],
                   [0.1, 0.1, 0.1, 0.1, 0.6],
                   [0.2, 0.2, 0.2, 0.2, 0.2],
                   [0.2, 0.2, 0.2, 0.2, 0.2]])
    qp = np.array([[0.4, 0.1, 0.1, 0.3, 0.1],
                   [0.1, 0.2, 0.5, 0.1, 0.1],
                   [0.2] * 5, [0.2] * 5, [0.2] * 5, [0.2] * 5])
    target, draft = _rows(tp), _rows(qp)
    g = np.random.default_rng(1234 + mode)
    n_draws = 30000
    first = np.zeros(V)
    second = {}
    fixed_tokens = np.array([0, 3, 1, 4, 0, 2], np.int32)
    for _ in range(n_draws):
        tokens = fixed_tokens.copy()
        if mode == oracle.ACCEPT_SPEC:
            tokens[1:4] = g.choice(V, 3, replace=False, p=qp[0])
            tokens[4:6] = g.choice(V, 2, replace=False, p=qp[1])
        ua = g.integers(0, 1 << 24, 6) * 2.0 ** -24
        us = g.integers(0, 1 << 24, 6) * 2.0 ** -24
        res = oracle.tree_accept(target, draft, tokens, parents, [0, 6], mode, ua, us)
        seq = _first_two_tokens(res, tokens)
        first[seq[0]] += 1
        if len(seq) > 1 and res["path"][0][1] == 1:  # the first token is node 1's, so p(node 1) follows
            second.setdefault(0, np.zeros(V))[seq[1]] += 1
    assert chisquare(first, tp[0] * n_draws).pvalue > 1e-3
    h = second[0]
    assert h.sum() > 2000
    assert chisquare(h, tp[1] * h.sum()).pvalue > 1e-3


def test_wrong_rule_is_detected_by_the_chi_square():
    """Sanity of the statistical pin: accepting with u < p(x) but without
    renormalising the residual shifts the first-token law far enough that
    the same chi-square test rejects it."""
    V = 5
    p = np.array([0.05, 0.3, 0.25, 0.1, 0.3])
    cand = [0, 3, 1]
    g = np.random.default_rng(7)
    hist = np.zeros(V)
    n = 30000
    for _ in range(n):
        out = None
        for x in cand:
            if g.random() < p[x]:  # no renormalisation after rejections
                out = x
                break
        if out is None:
            r = p.copy()
            r[cand] = 0
            out = int(np.searchsorted(np.cumsum(r / r.sum()), g.random(), side="right"))
        hist[out] += 1
    assert chisquare(hist, p * n).pvalue < 1e-6


def test_inverse_cdf_edges():
    p = np.array([0.0, 0.5, 0.0, 0.5, 0.0])
    assert oracle.sample_inverse_cdf(p, 0.0)[0] == 1
    assert oracle.sample_inverse_cdf(p, 0.49)[0] == 1
    assert oracle.sample_inverse_cdf(p, 0.5)[0] == 3
    assert oracle.sample_inverse_cdf(p, 1.0 - 2 ** -24)[0] == 3
