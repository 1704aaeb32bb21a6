"""Seeded synthetic inputs for the tree-verify path.

This module only draws inputs: random numbers, random tree shapes and
planted target rows.  It holds none of the method's arithmetic (no softmax,
no attention, no top-k, no acceptance rule), so both the CUDA path and the
CPU oracle can take their inputs from here without sharing any logic.

The workloads stand in for the paper's evaluation sets (MS-COCO / Parti
prompts / ImageNet, Sec. 5.1), which are not available: shapes follow the
7B-class models (Anole / Lumina-mGPT: 32 layers, 32 heads x 128) and the
LlamaGen-XL class (36 layers, 20 heads x 64, 24x24 latent grid, Sec. 5.1).
"""
from __future__ import annotations

import zlib
from dataclasses import dataclass

import numpy as np
import torch

BASE_SEED = 20251221


def rng(seed: int, name: str) -> np.random.Generator:
    """PCG64 stream for (seed, name); the name keeps sub-streams independent."""
    return np.random.Generator(np.random.PCG64([seed, zlib.crc32(name.encode())]))


def bf16_normal(shape, seed: int, name: str, std: float = 1.0) -> torch.Tensor:
    """N(0, std^2) drawn in fp32, rounded to bf16 (round-to-nearest-even)."""
    x = rng(seed, name).standard_normal(size=shape, dtype=np.float32) * np.float32(std)
    return torch.from_numpy(x).to(torch.bfloat16)


def f32_normal(shape, seed: int, name: str, std: float = 3.0) -> np.ndarray:
    return (rng(seed, name).standard_normal(size=shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def uniforms(n: int, seed: int, name: str) -> np.ndarray:
    """fp32 uniforms k * 2^-24, k in [0, 2^24): exact in fp32 and fp64, always < 1."""
    k = rng(seed, name).integers(0, 1 << 24, size=n, dtype=np.int64)
    return (k.astype(np.float64) * 2.0 ** -24).astype(np.float32)


def random_tree(n_nodes: int, seed: int, name: str = "tree", max_depth: int = 6,
                max_children: int = 4) -> np.ndarray:
    """Layered draft-tree shape: node 0 is the root, parents[i] < i.

    Layer sizes are drawn so that every node has at most ``max_children``
    children and the depth is at most ``max_depth``; each node picks its
    parent uniformly from the previous layer among parents with room left.
    Nodes of a layer are ordered by parent, as a depth-major rerank emits them.
    """
    if n_nodes < 1:
        raise ValueError("n_nodes >= 1")
    g = rng(seed, name)
    parents = [-1]
    prev = [0]
    remaining = n_nodes - 1
    depth = 0
    while remaining > 0:
        depth += 1
        cap = len(prev) * max_children
        layers_left = max_depth - depth + 1
        if layers_left <= 0:
            raise ValueError("tree does not fit in max_depth with max_children")
        hi = min(cap, remaining)

        def fits(s: int) -> bool:  # can layers after this one hold the rest?
            room_after, width = 0, s
            for _ in range(layers_left - 1):
                width *= max_children
                room_after += width
            return remaining - s <= room_after

        lo = next((s for s in range(1, hi + 1) if fits(s)), None)
        if lo is None:
            raise ValueError("tree does not fit in max_depth with max_children")
        size = int(g.integers(lo, hi + 1))
        room = {p: max_children for p in prev}
        chosen = []
        for _ in range(size):
            cands = [p for p in prev if room[p] > 0]
            p = cands[int(g.integers(0, len(cands)))]
            room[p] -= 1
            chosen.append(p)
        chosen.sort()
        base = len(parents)
        parents.extend(chosen)
        prev = list(range(base, base + size))
        remaining -= size
    return np.asarray(parents, dtype=np.int32)


def chain_tree(n_nodes: int) -> np.ndarray:
    return np.arange(-1, n_nodes - 1, dtype=np.int32)


def tree_tokens(parents: np.ndarray, vocab: int, seed: int, name: str = "tokens") -> np.ndarray:
    """Token per node; siblings always hold distinct tokens."""
    g = rng(seed, name)
    n = len(parents)
    tokens = np.zeros(n, dtype=np.int32)
    tokens[0] = int(g.integers(0, vocab))
    for p in sorted(set(int(x) for x in parents[1:])):
        kids = [i for i in range(n) if parents[i] == p]
        tokens[kids] = g.choice(vocab, size=len(kids), replace=False)
    return tokens


def plant_path(target: np.ndarray, parents: np.ndarray, tokens: np.ndarray, path_nodes,
               boost: float = 50.0) -> None:
    """Raise the target row of each node on ``path_nodes`` (root-first) so that
    its largest entry is the token of the next node on the path.  The last node
    keeps its row, so the walk stops there.  Modifies ``target`` in place."""
    for v, c in zip(path_nodes[:-1], path_nodes[1:]):
        row = target[v]
        row[tokens[c]] = row.max() + np.float32(boost)


@dataclass
class TreeBatch:
    """B trees packed back to back (node_offsets), with per-node tokens."""
    parents: np.ndarray       # int32 [Ntot], tree-local parent, -1 at each root
    tokens: np.ndarray        # int32 [Ntot]
    node_offsets: np.ndarray  # int32 [B+1]


def tree_batch(sizes, vocab: int, seed: int, max_depth: int = 6, max_children: int = 4,
               chain: bool = False) -> TreeBatch:
    par, tok, offs = [], [], [0]
    for b, n in enumerate(sizes):
        p = chain_tree(n) if chain else random_tree(n, seed, f"tree{b}", max_depth, max_children)
        t = tree_tokens(p, vocab, seed, f"tokens{b}")
        par.append(p)
        tok.append(t)
        offs.append(offs[-1] + n)
    return TreeBatch(np.concatenate(par).astype(np.int32), np.concatenate(tok).astype(np.int32),
                     np.asarray(offs, dtype=np.int32))


def acceptance_map(h: int, w: int, seed: int, n_blobs: int = 6, lo: float = 0.15,
                   hi: float = 0.9) -> np.ndarray:
    """Smooth per-position acceptance-rate map in [lo, hi] made of Gaussian blobs:
    high in 'simple' regions, low in 'complex' ones (Sec. 3.2 observation)."""
    g = rng(seed, "alpha_map")
    yy, xx = np.mgrid[0:h, 0:w].astype(np.float64)
    acc = np.zeros((h, w))
    for _ in range(n_blobs):
        cy, cx = g.uniform(0, h), g.uniform(0, w)
        s = g.uniform(0.1, 0.3) * max(h, w)
        amp = g.uniform(-1.0, 1.0)
        acc += amp * np.exp(-((yy - cy) ** 2 + (xx - cx) ** 2) / (2 * s * s))
    acc = (acc - acc.min()) / max(acc.max() - acc.min(), 1e-12)
    return lo + (hi - lo) * acc


def step_inputs(layers, H, Hkv, D, V, kv_len, depth, width, n_nodes, lmax, seed, logit_std=3.0):
    """Host inputs of one verify step (all seeded): caches and tree
    projections bf16 ~ N(0, 1); draft rows per image and layer fp32
    ~ N(0, logit_std^2); target rows ~ N(0, logit_std^2); uniforms; root
    tokens.  n_nodes[b] is the tree size of image b."""
    Bn = len(kv_len)
    ntot = int(sum(n_nodes))
    out = dict(
        k_cache=bf16_normal((layers, Bn, Hkv, lmax, D), seed, "k_cache"),
        v_cache=bf16_normal((layers, Bn, Hkv, lmax, D), seed, "v_cache"),
        q=bf16_normal((layers, ntot, H, D), seed, "q"),
        k_tree=bf16_normal((layers, ntot, Hkv, D), seed, "k_tree"),
        v_tree=bf16_normal((layers, ntot, Hkv, D), seed, "v_tree"),
        draft_rows=[f32_normal((depth[b], width[b], V), seed, f"draft{b}", std=logit_std) for b in range(Bn)],
        target=f32_normal((ntot, V), seed, "target", std=logit_std),
        u_accept=uniforms(ntot, seed, "u_accept"),
        u_sample=uniforms(ntot, seed, "u_sample"),
        root_token=rng(seed, "root").integers(0, V, size=Bn).astype(np.int32),
    )
    return out
