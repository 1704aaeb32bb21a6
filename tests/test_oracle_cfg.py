"""Pins of the oracle's classifier-free-guidance combine (p and q under CFG,
Sec. 3.1 under Eq. 1; guidance scale 3.0, Sec. 5.1), checked against values
fixed by arithmetic rather than by the formula's own code."""
import numpy as np

import oracle


def test_scale_zero_returns_the_unconditional_row_exactly():
    g = np.random.default_rng(1)
    c = g.standard_normal(1000).astype(np.float32) * 3
    u = g.standard_normal(1000).astype(np.float32) * 3
    assert np.array_equal(oracle.cfg_logits(c, u, 0.0), u)


def test_hand_values():
    # u + 3 (c - u) with small integers: 1 + 3*2 = 7, 1 + 3*(-3) = -8, 1 + 3*4 = 13, -2 + 3*0 = -2
    c = np.array([3, -2, 5, -2], np.float32)
    u = np.array([1, 1, 1, -2], np.float32)
    assert oracle.cfg_logits(c, u, 3.0).tolist() == [7.0, -8.0, 13.0, -2.0]
    # scale 1 on exactly representable values gives the conditional row
    assert oracle.cfg_logits(c, u, 1.0).tolist() == c.tolist()


def test_exact_on_dyadic_values():
    # multiples of 1/16 in [-8, 8): c - u, 3 (c - u) and the sum are exact in
    # fp32, so the result equals the fp64 extrapolation
    g = np.random.default_rng(2)
    c = (g.integers(-128, 128, 500) / 16.0).astype(np.float32)
    u = (g.integers(-128, 128, 500) / 16.0).astype(np.float32)
    want = u.astype(np.float64) + 3.0 * (c.astype(np.float64) - u.astype(np.float64))
    assert np.array_equal(oracle.cfg_logits(c, u, 3.0).astype(np.float64), want)


def test_guidance_reorders_the_top_k():
    # the conditional leader is also favoured by the unconditional branch,
    # so guidance (which amplifies cond - uncond) promotes the second token
    c = np.array([5.0, 4.5, 0.0, -1.0], np.float32)
    u = np.array([5.0, 2.0, 0.0, -1.0], np.float32)
    l = oracle.cfg_logits(c, u, 3.0)
    assert l.tolist() == [5.0, 9.5, 0.0, -1.0]
    res = oracle.tree_expand(l[None, :], np.zeros(1, np.float32), 2, 2)
    assert res["child_token"].tolist() == [1, 0]
