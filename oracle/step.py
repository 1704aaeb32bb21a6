"""The oracle's whole verify step: the oracle functions composed in the
order of Sec. 3.1 / Fig. 5 (draft layers, rerank, target attention per
layer, acceptance walk, KV commit), for one image at a time.

TEST INFRASTRUCTURE: only tests, smoke() and bench's CPU legs call it.
"""
from __future__ import annotations

import numpy as np

from .tree_verify import kv_compact, tree_accept, tree_attention, tree_expand, tree_rerank


def draft_tree(draft_rows, k: int, depth: int, root_token: int, n_nodes: int):
    """draft_rows[d] holds the draft rows of layer d's frontier (F_0 = 1)."""
    tok, sc, par = [], [], []
    fscore = np.zeros(1, np.float32)
    fid = np.array([-1], np.int32)
    for d in range(depth):
        F = len(fscore)
        res = tree_expand(np.asarray(draft_rows[d][:F], np.float32), fscore, k, min(k, F * k), frontier_id=fid,
                          child_id_base=len(tok))
        tok += res["child_token"].tolist()
        sc += res["child_score"].tolist()
        par += res["child_parent"].tolist()
        fscore, fid = res["next_score"], res["next_id"]
    n = min(n_nodes, len(tok) + 1)
    tree = tree_rerank(tok, np.array(sc, np.float32), par, root_token, n)
    tree["pool_token"] = np.array(tok, np.int32)
    tree["pool_score"] = np.array(sc, np.float32)
    tree["pool_parent"] = np.array(par, np.int32)
    return tree


def verify_step(draft_rows_per_image, widths, depths, root_tokens, n_nodes, q, k_cache, v_cache, kv_len,
                k_tree, v_tree, target, u_accept, u_sample, mode, temperature=1.0, layers=None):
    """Returns dict(trees, node_offsets, attn [layers] (out, lse), accept, k_cache', v_cache', kv_len').

    q: [layers, Ntot, H, D]; caches [layers, B, Hkv, Lmax, D]; k_tree/v_tree
    [layers, Ntot, Hkv, D]; target [Ntot, V]; all as float64/float32 arrays.
    ``layers`` restricts the attention to a subset (compact still covers all).
    """
    Bn = len(widths)
    trees = [draft_tree(draft_rows_per_image[b], widths[b], depths[b], root_tokens[b], n_nodes)
             for b in range(Bn)]
    offs = np.concatenate([[0], np.cumsum([len(t["tokens"]) for t in trees])]).astype(np.int64)
    parents = np.concatenate([t["parents"] for t in trees])
    tokens = np.concatenate([t["tokens"] for t in trees])
    L = q.shape[0]
    attn = {}
    D = q.shape[3]
    for layer in (range(L) if layers is None else layers):
        attn[layer] = tree_attention(q[layer], k_cache[layer], v_cache[layer], kv_len, k_tree[layer],
                                     v_tree[layer], parents, offs, 1.0 / np.sqrt(D))
    acc = tree_accept(target, None, tokens, parents, offs, mode, u_accept, u_sample, temperature)
    kc, vc, new_len = kv_compact(k_cache, v_cache, kv_len, k_tree, v_tree, offs, acc["path"])
    return dict(trees=trees, node_offsets=offs, parents=parents, tokens=tokens, attn=attn, accept=acc,
                k_cache=kc, v_cache=vc, kv_len=new_len)
