"""Pins of the oracle's tree attention against things other than itself:
torch's scaled_dot_product_attention (fp64, CPU) with a mask built from
networkx's ancestor sets, closed forms and invariants (Sec. 3.1)."""
import math

import networkx as nx
import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2512_21857_gb300 import synth


def _inputs(sizes, L, H, Hkv, D, seed, chain=False, lmax_extra=3):
    B = len(sizes)
    tb = synth.tree_batch(sizes, 100, seed, chain=chain)
    ntot = int(tb.node_offsets[-1])
    q = synth.bf16_normal((ntot, H, D), seed, "q").double().numpy()
    kc = synth.bf16_normal((B, Hkv, max(L) + lmax_extra, D), seed, "kc").double().numpy()
    vc = synth.bf16_normal((B, Hkv, max(L) + lmax_extra, D), seed, "vc").double().numpy()
    kt = synth.bf16_normal((ntot, Hkv, D), seed, "kt").double().numpy()
    vt = synth.bf16_normal((ntot, Hkv, D), seed, "vt").double().numpy()
    return tb, q, kc, vc, kt, vt


def _sdpa_reference(tb, q, kc, vc, kt, vt, kv_len, scale):
    """Each tree as one SDPA call: keys = prefix + all tree nodes, boolean
    mask = prefix visible, tree node j visible to t iff j == t or j is an
    ancestor of t (networkx)."""
    ntot, H, D = q.shape
    Hkv = kt.shape[1]
    out = np.zeros_like(q)
    for b in range(len(tb.node_offsets) - 1):
        lo, hi = int(tb.node_offsets[b]), int(tb.node_offsets[b + 1])
        n, L = hi - lo, int(kv_len[b])
        G = nx.DiGraph()
        G.add_nodes_from(range(n))
        G.add_edges_from((int(tb.parents[lo + t]), t) for t in range(1, n))
        mask = torch.zeros(n, L + n, dtype=torch.bool)
        mask[:, :L] = True
        for t in range(n):
            mask[t, L + t] = True
            for a in nx.ancestors(G, t):
                mask[t, L + a] = True
        rep = H // Hkv
        K = np.concatenate([kc[b, :, :L], kt[lo:hi].transpose(1, 0, 2)], axis=1)  # [Hkv, L+n, D]
        Vv = np.concatenate([vc[b, :, :L], vt[lo:hi].transpose(1, 0, 2)], axis=1)
        K = torch.from_numpy(np.repeat(K, rep, axis=0))[None]
        Vv = torch.from_numpy(np.repeat(Vv, rep, axis=0))[None]
        Q = torch.from_numpy(q[lo:hi].transpose(1, 0, 2).copy())[None]
        o = F.scaled_dot_product_attention(Q, K, Vv, attn_mask=mask, scale=scale)
        out[lo:hi] = o[0].numpy().transpose(1, 0, 2)
    return out


@pytest.mark.parametrize("sizes,L,H,Hkv,D,chain", [
    ([7], [5], 2, 2, 16, True),             # chain tree = causal attention over prefix + chain
    ([1], [9], 3, 3, 8, False),             # single node = ordinary decode attention
    ([26], [40], 2, 2, 16, False),          # random layered tree
    ([5, 1, 9], [0, 7, 3], 4, 2, 8, False),  # ragged batch, L = 0, grouped kv heads
])
def test_attention_matches_sdpa_with_networkx_mask(sizes, L, H, Hkv, D, chain):
    tb, q, kc, vc, kt, vt = _inputs(sizes, L, H, Hkv, D, seed=3, chain=chain)
    scale = 1.0 / math.sqrt(D)
    out, lse = oracle.tree_attention(q, kc, vc, L, kt, vt, tb.parents, tb.node_offsets, scale)
    ref = _sdpa_reference(tb, q, kc, vc, kt, vt, L, scale)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_chain_equals_causal_sdpa():
    """Chain tree of n nodes over prefix L: bottom-right aligned causal mask."""
    n, L, H, D = 6, 4, 2, 8
    tb, q, kc, vc, kt, vt = _inputs([n], [L], H, H, D, seed=5, chain=True, lmax_extra=0)
    out, _ = oracle.tree_attention(q, kc, vc, [L], kt, vt, tb.parents, tb.node_offsets, 0.3)
    K = torch.from_numpy(np.concatenate([kc[0], kt.transpose(1, 0, 2)], axis=1))[None]
    Vv = torch.from_numpy(np.concatenate([vc[0], vt.transpose(1, 0, 2)], axis=1))[None]
    Q = torch.from_numpy(q.transpose(1, 0, 2).copy())[None]
    causal = torch.ones(n, L + n, dtype=torch.bool).tril(diagonal=L)
    ref = F.scaled_dot_product_attention(Q, K, Vv, attn_mask=causal, scale=0.3)[0].numpy()
    np.testing.assert_allclose(out, ref.transpose(1, 0, 2), atol=1e-12)


def test_empty_prefix_root_returns_its_own_value():
    tb, q, kc, vc, kt, vt = _inputs([4], [0], 2, 2, 8, seed=7)
    out, lse = oracle.tree_attention(q, kc, vc, [0], kt, vt, tb.parents, tb.node_offsets, 0.5)
    np.testing.assert_array_equal(out[0], vt[0])
    np.testing.assert_allclose(lse[0], 0.5 * np.einsum("hd,hd->h", q[0], kt[0]), atol=1e-12)


def test_equal_keys_give_mean_of_visible_values():
    """All keys equal -> uniform softmax -> mean of the values the node sees
    (prefix + its ancestors + itself); a wrong key set changes the mean."""
    n, L, H, D = 16, 5, 2, 4
    tb, q, kc, vc, kt, vt = _inputs([n], [L], H, H, D, seed=11)
    kc[:] = 0.25
    kt[:] = 0.25
    out, lse = oracle.tree_attention(q, kc, vc, [L], kt, vt, tb.parents, tb.node_offsets, 1.0)
    G = nx.DiGraph((int(tb.parents[t]), t) for t in range(1, n))
    for t in range(n):
        vis = sorted((nx.ancestors(G, t) if t in G else set()) | {t})
        expect = np.concatenate([vc[0, :, :L], vt[vis].transpose(1, 0, 2)], axis=1).mean(axis=1)
        np.testing.assert_allclose(out[t], expect, atol=1e-12)
        np.testing.assert_allclose(lse[t], 0.25 * q[t].sum(axis=-1) + math.log(L + len(vis)), atol=1e-12)


def test_sibling_relabelling_permutes_outputs():
    # root 0, children 1 and 2; 3 under 1; 4 under 2.  Swap the subtrees of 1 and 2.
    parents = np.array([-1, 0, 0, 1, 2], np.int32)
    perm = np.array([0, 2, 1, 4, 3])          # new node i is old node perm[i]
    new_parents = np.array([-1, 0, 0, 1, 2], np.int32)  # same shape after the swap
    _, q, kc, vc, kt, vt = _inputs([5], [6], 2, 2, 8, seed=13)
    offs = np.array([0, 5])
    out, lse = oracle.tree_attention(q, kc, vc, [6], kt, vt, parents, offs, 0.4)
    out2, lse2 = oracle.tree_attention(q[perm], kc, vc, [6], kt[perm], vt[perm], new_parents, offs, 0.4)
    np.testing.assert_array_equal(out2, out[perm])
    np.testing.assert_array_equal(lse2, lse[perm])


def test_lse_matches_scipy_logsumexp():
    from scipy.special import logsumexp
    tb, q, kc, vc, kt, vt = _inputs([9], [12], 2, 2, 8, seed=17)
    out, lse = oracle.tree_attention(q, kc, vc, [12], kt, vt, tb.parents, tb.node_offsets, 0.35)
    G = nx.DiGraph((int(tb.parents[t]), t) for t in range(1, 9))
    for t in range(9):
        vis = sorted((nx.ancestors(G, t) if t in G else set()) | {t})
        for h in range(2):
            K = np.concatenate([kc[0, h, :12], kt[vis, h]], axis=0)
            assert abs(lse[t, h] - logsumexp(0.35 * (K @ q[t, h]))) < 1e-12


def test_bad_parents_rejected():
    _, q, kc, vc, kt, vt = _inputs([3], [2], 1, 1, 4, seed=1)
    with pytest.raises(ValueError):
        oracle.tree_attention(q, kc, vc, [2], kt, vt, [-1, 2, 0], [0, 3], 1.0)
    with pytest.raises(ValueError):
        oracle.tree_attention(q, kc, vc, [2], kt, vt, [0, 0, 1], [0, 3], 1.0)
