"""Plain CPU oracle for the data-parallel verify path of ADT-Tree.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import or run
anything under ``oracle/``.  The product path (the CUDA library and its
binding) never calls it and shares no code with it.

Everything here is the slow, literal definition: one node at a time, fp64
arithmetic on inputs widened exactly from their stored types (bf16 / fp32),
library primitives (matmul, sort, exp) used only as single steps.  Each
function names the passage of the paper it follows.

Notation (Sec. 3.1): a draft tree has N nodes; node 0 is the root, i.e. the
last committed token whose K/V is produced in the same verify pass; every
other node t has a parent parents[t] < t.  ans(t) is the root-to-t path.

Decisions that turn floating point into an integer (accept / reject, the
index an inverse-CDF draw lands on, a top-k membership) are made here in
fp64.  Each call can report the smallest relative margin of the decisions it
took, so a parity test can tell a genuine disagreement from a near-tie where
rounding order alone decides.
"""
from __future__ import annotations

import math

import numpy as np

ACCEPT_GREEDY = 0
ACCEPT_SPEC = 1
ACCEPT_SPEC_DET = 2


# ----------------------------------------------------------------------------
# Tree structure (Sec. 3.1: "ancestor sequence ... based on the tree mask")
# ----------------------------------------------------------------------------

def check_parents(parents) -> None:
    """A tree is valid iff node 0 is the only root and every parent precedes
    its child (then the parent pointers form a tree rooted at node 0)."""
    parents = [int(p) for p in parents]
    if len(parents) == 0:
        raise ValueError("empty tree")
    if parents[0] != -1:
        raise ValueError("node 0 must be the root (parent -1)")
    for i in range(1, len(parents)):
        if not (0 <= parents[i] < i):
            raise ValueError(f"parents[{i}]={parents[i]} must be in [0, {i})")


def ancestor_path(parents, t: int) -> list[int]:
    """ans(t) together with t itself, root first (Sec. 3.1)."""
    path = []
    j = int(t)
    while j >= 0:
        path.append(j)
        j = int(parents[j])
    return path[::-1]


def children(parents, v: int) -> list[int]:
    """Children of v in ascending node index (the rerank order, Sec. 4.2)."""
    return [c for c in range(len(parents)) if int(parents[c]) == v]


# ----------------------------------------------------------------------------
# Tree attention (Sec. 3.1: the target verifies all L draft tokens in one pass,
# each node conditioned on the prefix s_{1:t} and its ancestors ans(t))
# ----------------------------------------------------------------------------

def tree_attention(q, k_cache, v_cache, kv_len, k_tree, v_tree, parents, node_offsets,
                   scale: float):
    """Exact tree-masked attention, one (node, head) at a time.

    q:        [Ntot, H, D]     queries of all tree nodes (RoPE already applied)
    k_cache:  [B, Hkv, Lmax, D] prefix keys; only the first kv_len[b] are valid
    v_cache:  [B, Hkv, Lmax, D]
    k_tree:   [Ntot, Hkv, D]   keys / values of the tree nodes themselves
    parents:  [Ntot]           tree-local parent index, -1 at each root
    node_offsets: [B+1]        tree b owns global nodes node_offsets[b] .. [b+1]-1
    Query head h reads kv head h // (H // Hkv).

    Node t of tree b attends to keys [prefix_0 .. prefix_{L_b-1}] followed by
    the tree keys of ans(t) and t (root first): o = softmax(scale * K q) V.
    Returns (out [Ntot, H, D], lse [Ntot, H]) in fp64, lse in natural log.
    """
    q = np.asarray(q, dtype=np.float64)
    k_cache = np.asarray(k_cache, dtype=np.float64)
    v_cache = np.asarray(v_cache, dtype=np.float64)
    k_tree = np.asarray(k_tree, dtype=np.float64)
    v_tree = np.asarray(v_tree, dtype=np.float64)
    ntot, H, D = q.shape
    Hkv = k_tree.shape[1]
    if H % Hkv:
        raise ValueError("H must be a multiple of Hkv")
    group = H // Hkv
    out = np.zeros((ntot, H, D))
    lse = np.zeros((ntot, H))
    B = len(node_offsets) - 1
    for b in range(B):
        lo, hi = int(node_offsets[b]), int(node_offsets[b + 1])
        par = [int(p) for p in parents[lo:hi]]
        if hi == lo:
            continue
        check_parents(par)
        L = int(kv_len[b])
        for t in range(hi - lo):
            path = [lo + j for j in ancestor_path(par, t)]
            for h in range(H):
                g = h // group
                keys = np.concatenate([k_cache[b, g, :L], k_tree[path, g]], axis=0)
                vals = np.concatenate([v_cache[b, g, :L], v_tree[path, g]], axis=0)
                s = scale * (keys @ q[lo + t, h])
                m = s.max()
                w = np.exp(s - m)
                denom = w.sum()
                out[lo + t, h] = (w @ vals) / denom
                lse[lo + t, h] = m + math.log(denom)
    return out, lse


# ----------------------------------------------------------------------------
# Draft-tree expansion (Sec. 3.1 last paragraph; Sec. 4.2, Fig. 5 and the
# EAGLE-2 node score, Eq. 4)
# ----------------------------------------------------------------------------

def cfg_logits(cond, uncond, scale: float) -> np.ndarray:
    """Classifier-free guidance on logits.  The paper computes both p and q
    under CFG (Sec. 3.1, under Eq. 1) with guidance scale 3.0 (Sec. 5.1) but
    prints no formula; the standard combine is taken:
        l = l_uncond + s * (l_cond - l_uncond),
    each operation (difference, product, sum) rounded to fp32 as written.
    The result then goes through the usual definitions (expansion, walk)."""
    c = np.asarray(cond, dtype=np.float32)
    u = np.asarray(uncond, dtype=np.float32)
    s = np.float32(scale)
    d = (c - u).astype(np.float32)
    return (u + (s * d).astype(np.float32)).astype(np.float32)


def _tempered(row32, temperature: float) -> np.ndarray:
    """Row / T in fp32 (the stored type), -0.0 canonicalised to +0.0."""
    x = np.asarray(row32, dtype=np.float32)
    if temperature != 1.0:
        x = (x / np.float32(temperature)).astype(np.float32)
    x = x.copy()
    x[x == 0] = np.float32(0.0)
    return x


def log_softmax_normaliser(x32) -> float:
    """log sum_j exp(x_j) in fp64, shifted by the maximum."""
    x = np.asarray(x32, dtype=np.float64)
    m = x.max()
    return float(m + math.log(math.fsum(np.exp(x - m))))


def tree_expand(logits, frontier_score, k_child: int, k_keep: int, temperature: float = 1.0,
                frontier_id=None, child_id_base: int = 0):
    """One layer of dynamic draft-tree growth.

    For each frontier row r (a node selected at the previous depth) the draft
    distribution q(. | ans(r)) = softmax(logits[r] / T) proposes its top
    ``k_child`` tokens (largest logit first, lowest token id on ties).  Each
    child's confidence c = q(token) enters the path confidence P_v as a
    product (Sec. 3.1, Eq. 4); it is carried in the log domain:
        child_logp  = log q(token) = x_token - log sum exp(x)
        child_score = frontier_score[r] + child_logp
    The ``k_keep`` children with the highest score (lowest candidate index on
    ties; candidate index = r * k_child + rank) form the next frontier.

    Returns a dict of numpy arrays: child_token, child_logp, child_score
    (fp32, rounded once from fp64), child_parent (frontier_id[r], or r),
    keep_idx (local candidate indices, best first), next_score, next_id
    (= child_id_base + keep_idx), lse (fp64 per row).
    """
    logits = np.asarray(logits, dtype=np.float32)
    F, V = logits.shape
    if not (1 <= k_child <= V):
        raise ValueError("1 <= k_child <= V")
    if not (1 <= k_keep <= F * k_child):
        raise ValueError("1 <= k_keep <= F * k_child")
    child_token = np.zeros(F * k_child, np.int32)
    child_logp = np.zeros(F * k_child, np.float32)
    child_score = np.zeros(F * k_child, np.float32)
    child_parent = np.zeros(F * k_child, np.int32)
    lses = np.zeros(F)
    for r in range(F):
        x = _tempered(logits[r], temperature)
        if np.isnan(x).any():
            raise ValueError("NaN logits are outside the domain")
        order = np.lexsort((np.arange(V), -x.astype(np.float64)))[:k_child]
        lse = log_softmax_normaliser(x)
        lses[r] = lse
        for j, tok in enumerate(order):
            lp = float(x[tok]) - lse
            child_token[r * k_child + j] = tok
            child_logp[r * k_child + j] = np.float32(lp)
            child_score[r * k_child + j] = np.float32(float(np.float32(frontier_score[r])) + lp)
            child_parent[r * k_child + j] = r if frontier_id is None else int(frontier_id[r])
    keep = np.lexsort((np.arange(F * k_child), -child_score.astype(np.float64)))[:k_keep]
    keep = keep.astype(np.int32)
    return dict(child_token=child_token, child_logp=child_logp, child_score=child_score,
                child_parent=child_parent, keep_idx=keep, next_score=child_score[keep].copy(),
                next_id=(child_id_base + keep).astype(np.int32), lse=lses)


def tree_rerank(cand_token, cand_score, cand_parent, root_token: int, n_nodes: int):
    """Final draft tree: the n_nodes-1 candidates with the highest score
    (Eq. 4: "the top-N nodes with the highest scores ... form the final draft
    tree"), lowest candidate index on ties, plus the root as node 0.

    Candidates are numbered depth-major (a layer's candidates follow all of
    the previous layer's), and a child's score never exceeds its parent's
    (log q <= 0), so the chosen set contains every chosen node's parent.
    Nodes are emitted in ascending candidate index, hence parents[i] < i.
    Returns dict(tokens, parents, cand_index (-1 at the root), depth).
    """
    cand_score = np.asarray(cand_score, dtype=np.float32)
    C = len(cand_score)
    need = n_nodes - 1
    if need < 0 or need > C:
        raise ValueError("need 1 <= n_nodes <= C + 1")
    order = np.lexsort((np.arange(C), -cand_score.astype(np.float64)))[:need]
    sel = np.sort(order)
    node_of = {int(c): i + 1 for i, c in enumerate(sel)}
    tokens = [int(root_token)] + [int(cand_token[c]) for c in sel]
    parents = [-1]
    for c in sel:
        pc = int(cand_parent[c])
        if pc < 0:
            parents.append(0)
        elif pc in node_of:
            parents.append(node_of[pc])
        else:
            raise ValueError(f"candidate {c} chosen without its parent {pc}")
    depth = [0] * n_nodes
    for i in range(1, n_nodes):
        depth[i] = depth[parents[i]] + 1
    return dict(tokens=np.asarray(tokens, np.int32), parents=np.asarray(parents, np.int32),
                cand_index=np.asarray([-1] + [int(c) for c in sel], np.int32),
                depth=np.asarray(depth, np.int32))


# ----------------------------------------------------------------------------
# Acceptance (Sec. 3.1, Eq. 1; greedy T = 0 and sampling T = 1, Sec. 5.1)
# ----------------------------------------------------------------------------

def softmax64(row32, temperature: float) -> np.ndarray:
    """softmax(row / T): row / T rounded to fp32 (as stored), then fp64."""
    x = _tempered(row32, temperature).astype(np.float64)
    e = np.exp(x - x.max())
    return e / e.sum()


def argmax_lowest(row32) -> int:
    """Largest entry, lowest index among equal entries (-0.0 == +0.0)."""
    x = np.asarray(row32, dtype=np.float32).astype(np.float64)
    return int(np.argmax(x))


def sample_inverse_cdf(p: np.ndarray, u: float):
    """Smallest t with sum_{j<=t} p_j > u * sum_j p_j (index order, fp64);
    the last index with p_t > 0 if rounding leaves none.  Returns (t, margin)."""
    c = np.cumsum(p)
    total = c[-1]
    target = float(u) * total
    t = int(np.searchsorted(c, target, side="right"))
    if t >= len(p):
        t = int(np.nonzero(p > 0)[0][-1])
    lo = c[t - 1] if t > 0 else 0.0
    margin = min(abs(c[t] - target), abs(target - lo)) / max(total, 1e-300)
    return t, margin


def tree_accept(target_logits, draft_logits, tokens, parents, node_offsets, mode: int,
                u_accept=None, u_sample=None, temperature: float = 1.0, draft_row=None):
    """Walk each tree from the root and emit the accepted path.

    GREEDY (T = 0): a child is accepted iff its token is the target's argmax at
    the parent; the bonus token is the argmax at the last accepted node.

    SPEC: Eq. 1, r = min(1, p(x)/q(x)), tested as u * q(x) < p(x), extended to
    several siblings by recursive rejection sampling: children are tried in
    ascending index; after a rejection of token x the target becomes the
    residual p <- max(0, p - q) / sum (kept as is when that sum is 0) and the
    draft drops x: q(x) <- 0, q <- q / sum (all zero when nothing is left).

    SPEC_DET: the same with a deterministic proposal (q = 1 on the candidate):
    accept iff u < p(x); after a rejection p(x) <- 0 and p is renormalised.

    When no child is accepted (or the node is a leaf) the bonus token is drawn
    from the current p by inverse CDF with u_sample[v].  p and q are
    softmax(row / T) of the rows of the node being expanded; draft rows are
    draft_logits[draft_row[v]] (identity when draft_row is None).

    Returns dict(path [B][*] tree-local node lists, accept_len [B],
    bonus [B], accept_margin, sample_margin, min_margin): the smallest
    relative margin of the accept tests, of the inverse-CDF draws, and of
    both (inf for GREEDY, whose decisions are exact comparisons).
    """
    tokens = [int(t) for t in tokens]
    B = len(node_offsets) - 1
    paths, acc, bonus = [], [], []
    acc_margin = math.inf
    smp_margin = math.inf
    for b in range(B):
        lo, hi = int(node_offsets[b]), int(node_offsets[b + 1])
        par = [int(p) for p in parents[lo:hi]]
        check_parents(par)
        v = 0
        path = [0]
        while True:
            kids = children(par, v)
            gv = lo + v
            if mode == ACCEPT_GREEDY:
                g = argmax_lowest(target_logits[gv])
                nxt = next((c for c in kids if tokens[lo + c] == g), None)
                if nxt is None:
                    bonus.append(g)
                    break
                path.append(nxt)
                v = nxt
                continue
            p = softmax64(target_logits[gv], temperature)
            q = None
            if mode == ACCEPT_SPEC and kids:
                drow = gv if draft_row is None else int(draft_row[gv])
                q = softmax64(draft_logits[drow], temperature)
            nxt = None
            for c in kids:
                x = tokens[lo + c]
                u = float(u_accept[lo + c])
                if mode == ACCEPT_SPEC_DET:
                    lhs, rhs = u, p[x]
                else:
                    lhs, rhs = u * q[x], p[x]
                scale = max(abs(lhs), abs(rhs))
                if scale > 0:
                    acc_margin = min(acc_margin, abs(lhs - rhs) / scale)
                if lhs < rhs:
                    nxt = c
                    break
                if mode == ACCEPT_SPEC_DET:
                    r = p.copy()
                    r[x] = 0.0
                else:
                    r = np.maximum(p - q, 0.0)
                s = r.sum()
                if s > 0:
                    p = r / s
                if mode == ACCEPT_SPEC:
                    q = q.copy()
                    q[x] = 0.0
                    qs = q.sum()
                    q = q / qs if qs > 0 else np.zeros_like(q)
            if nxt is None:
                t, m = sample_inverse_cdf(p, float(u_sample[gv]))
                smp_margin = min(smp_margin, m)
                bonus.append(t)
                break
            path.append(nxt)
            v = nxt
        paths.append(path)
        acc.append(len(path) - 1)
    return dict(path=paths, accept_len=np.asarray(acc, np.int32),
                bonus=np.asarray(bonus, np.int32), accept_margin=acc_margin,
                sample_margin=smp_margin, min_margin=min(acc_margin, smp_margin))


# ----------------------------------------------------------------------------
# KV commit of the accepted path (Sec. 3.1: accepted draft tokens extend the
# prefix, so their keys / values join the cache)
# ----------------------------------------------------------------------------

def kv_compact(k_cache, v_cache, kv_len, k_tree, v_tree, node_offsets, paths):
    """For every layer l, tree b and i in 0..a_b (root included):
        cache[l, b, :, kv_len[b] + i, :] <- tree[l, node_offsets[b] + path_b[i], :, :]
    k_cache: [layers, B, Hkv, Lmax, D]; k_tree: [layers, Ntot, Hkv, D].
    Returns (k_cache', v_cache', kv_len') as new arrays."""
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    new_len = np.array(kv_len, dtype=np.int64, copy=True)
    Lmax = kc.shape[3]
    for b, path in enumerate(paths):
        base = int(kv_len[b])
        if base + len(path) > Lmax:
            raise ValueError("cache overflow")
        for i, node in enumerate(path):
            src = int(node_offsets[b]) + int(node)
            kc[:, b, :, base + i, :] = k_tree[:, src, :, :]
            vc[:, b, :, base + i, :] = v_tree[:, src, :, :]
        new_len[b] = base + len(path)
    return kc, vc, new_len


def kv_compact_inplace(k_cache, v_cache, kv_len, paths):
    """The cache holds tree b's K/V in its tail: row kv_len[b] + t is node t.
    For every layer l, tree b and i in 0..a_b, computed from the cache as it
    was before (Sec. 3.1: the accepted tokens extend the prefix):
        cache'[l, b, :, kv_len[b] + i, :] = cache[l, b, :, kv_len[b] + path_b[i], :]
    Returns (k_cache', v_cache', kv_len') as new arrays."""
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    new_len = np.array(kv_len, dtype=np.int64, copy=True)
    for b, path in enumerate(paths):
        base = int(kv_len[b])
        for i, node in enumerate(path):
            kc[:, b, :, base + i, :] = k_cache[:, b, :, base + int(node), :]
            vc[:, b, :, base + i, :] = v_cache[:, b, :, base + int(node), :]
        new_len[b] = base + len(path)
    return kc, vc, new_len
