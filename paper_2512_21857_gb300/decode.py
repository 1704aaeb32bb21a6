"""End-to-end synthetic decode loop: a random-init decoder-only target, an
EAGLE-style one-layer draft head, and ADT-Tree's per-step draft trees
(Sec. 3.1 draft-then-verify, Sec. 4 depth / width control), generating an
image-token grid in raster order.

The library does every step of the verify path: tree attention for the
prompt, the draft head and the target (`adt_tree_attn`), draft-tree growth
(`adt_tree_expand`) and the final top-N (`adt_tree_rerank`), the acceptance
walk (`adt_tree_accept`), the K/V commits (`adt_kv_compact`) and the depth /
width controller (`adt_ctrl_*`).  The dense parts of the two networks
(embeddings, RMSNorm, the Q/K/V/O and SwiGLU projections, rotary position
embedding, the LM head) are plain torch around it: the model, not the
method.

Draft head (EAGLE's feature-level draft): node u with token x_u and parent
feature f (the target's last hidden state before the final norm for the
tree root's parent, the draft's own output otherwise) enters as
fc([embed(x_u), f]); one decoder layer attends to the draft cache and u's
ancestors; its output is u's feature, and the shared final norm and LM head
turn it into the logits of u's children.  The tokens a verify step commits
are run through the draft head again with the target's true features at the
start of the next step (the draft cache holds only those).

Tree node t of a step sits at position kv_len + depth(t); node 0 (the root)
is the last emitted token, whose K/V the step computes and commits.
"""
from __future__ import annotations

import math
import time
from dataclasses import dataclass, field

import torch

from . import binding as B


@dataclass
class ModelShape:
    layers: int = 32
    hidden: int = 4096
    heads: int = 32
    kv_heads: int = 32
    head_dim: int = 128
    ffn: int = 11008
    vocab: int = 65536
    rope_theta: float = 10000.0
    eps: float = 1e-5
    init_std: float = 0.02
    lm_std: float = 0.0        # LM head init std (0: init_std)
    dtype: torch.dtype = torch.bfloat16  # weights and residual stream (the caches and attention stay bf16)


def _rms_norm(x, w, eps):
    xf = x.float()
    return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + eps) * w.float()).to(x.dtype)


def _rope(x, pos, theta):
    """Rotary embedding (rotate-half form) of x [N, heads, D] at positions pos [N]."""
    D = x.shape[-1]
    inv = theta ** (-torch.arange(0, D, 2, device=x.device, dtype=torch.float32) / D)
    ang = pos.float()[:, None] * inv[None, :]
    cos, sin = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    xf = x.float()
    x1, x2 = xf[..., : D // 2], xf[..., D // 2:]
    return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], -1).to(x.dtype)


class DecoderWeights:
    """Random-init weights of `layers` decoder layers (bf16), plus (when
    `lm` is set) embedding, final norm and LM head."""

    def __init__(self, shape: ModelShape, layers: int, seed: int, device, lm=True, draft_fc=False):
        g = torch.Generator(device=device).manual_seed(seed)  # drawn on the device: 7B weights in seconds
        s = shape
        std = s.init_std
        bf = dict(dtype=s.dtype)

        def rnd(*size, scale=std):
            return (torch.randn(*size, generator=g, device=device) * scale).to(**bf)

        qkv = (s.heads + 2 * s.kv_heads) * s.head_dim
        self.layers = [dict(ln1=torch.ones(s.hidden, device=device, **bf), wqkv=rnd(s.hidden, qkv),
                            wo=rnd(s.heads * s.head_dim, s.hidden), ln2=torch.ones(s.hidden, device=device, **bf),
                            wgu=rnd(s.hidden, 2 * s.ffn), wd=rnd(s.ffn, s.hidden))
                       for _ in range(layers)]
        if lm:
            self.embed = rnd(s.vocab, s.hidden, scale=1.0)
            self.norm = torch.ones(s.hidden, device=device, **bf)
            self.lm_head = rnd(s.hidden, s.vocab, scale=s.lm_std or std)
        if draft_fc:
            self.fc = rnd(2 * s.hidden, s.hidden)


def lm_logits(weights: DecoderWeights, h, eps):
    """fp32 logits of hidden states h: final RMSNorm, then the LM head in
    fp32 (bf16 logits tie too often for a greedy argmax)."""
    if getattr(weights, "lm_head32", None) is None:
        weights.lm_head32 = weights.lm_head.float()  # the same tensor when the weights are fp32
    return _rms_norm(h, weights.norm, eps).float() @ weights.lm_head32


class TreeModel:
    """The decoder stack over a batch of trees: dense parts in torch,
    attention through adt_tree_attn over each image's cache and tree."""

    def __init__(self, shape: ModelShape, weights: DecoderWeights, batch: int, lmax: int, max_nodes: int,
                 device):
        s = self.s = shape
        self.w = weights
        self.lmax = lmax
        self.max_nodes = max_nodes
        L = len(weights.layers)
        bf = dict(dtype=torch.bfloat16, device=device)
        self.k_cache = torch.zeros((L, batch, s.kv_heads, lmax, s.head_dim), **bf)
        self.v_cache = torch.zeros((L, batch, s.kv_heads, lmax, s.head_dim), **bf)
        self.ws = B.zeroed_workspace(B.adt_tree_attn_workspace_size(batch, s.heads, s.head_dim, max_nodes, lmax),
                                     device)
        self.device = device
        self.graphs_enabled = False
        self._graphs = {}

    def forward(self, x, pos, parents, node_offsets, kv_len, batch, image=None):
        """x [N, hidden] (bf16) for the nodes of `batch` trees (of image
        `image` alone when given: its cache slice, batch 1); returns the final
        hidden states [N, hidden] and each layer's tree K/V ([layers, N,
        kv_heads, D]) for the commit."""
        s = self.s
        N = x.shape[0]
        L = len(self.w.layers)
        k_tree = torch.empty((L, N, s.kv_heads, s.head_dim), dtype=torch.bfloat16, device=self.device)
        v_tree = torch.empty_like(k_tree)
        out = torch.empty((N, s.heads, s.head_dim), dtype=torch.bfloat16, device=self.device)
        hq, hk = s.heads * s.head_dim, s.kv_heads * s.head_dim
        sl = slice(None) if image is None else slice(image, image + 1)
        for li, lw in enumerate(self.w.layers):
            h = _rms_norm(x, lw["ln1"], s.eps)
            qkv = h @ lw["wqkv"]
            q = _rope(qkv[:, :hq].view(N, s.heads, s.head_dim), pos, s.rope_theta).to(torch.bfloat16).contiguous()
            k_tree[li] = _rope(qkv[:, hq:hq + hk].view(N, s.kv_heads, s.head_dim), pos, s.rope_theta)
            v_tree[li] = qkv[:, hq + hk:].view(N, s.kv_heads, s.head_dim)
            B.adt_tree_attn(q, self.k_cache[li, sl], self.v_cache[li, sl], kv_len, k_tree[li], v_tree[li], parents,
                            node_offsets, B=batch, H=s.heads, Hkv=s.kv_heads, D=s.head_dim,
                            max_nodes=self.max_nodes, max_kv=self.lmax, softmax_scale=s.head_dim ** -0.5, out=out,
                            workspace=self.ws, cache_stride_b=self.k_cache.stride(1),
                            cache_stride_h=self.k_cache.stride(2))
            x = x + out.view(N, hq).to(x.dtype) @ lw["wo"]
            h = _rms_norm(x, lw["ln2"], s.eps)
            gu = h @ lw["wgu"]
            x = x + (torch.nn.functional.silu(gu[:, : s.ffn].float()) * gu[:, s.ffn:].float()).to(x.dtype) @ lw["wd"]
        return x, k_tree, v_tree

    def run(self, x, pos, parents, node_offsets, kv_len, batch, image=None):
        """forward() through a CUDA graph captured once per (nodes, batch,
        image): the stack's few hundred launches replay without host work.
        The outputs are the graph's own buffers, rewritten by the next replay
        of the same shape: copy what must outlive it."""
        if not self.graphs_enabled:
            return self.forward(x, pos, parents, node_offsets, kv_len, batch, image)
        key = (x.shape[0], batch, image)
        g = self._graphs.get(key)
        if g is None:
            ins = [t.clone() for t in (x, pos, parents, node_offsets, kv_len)]
            side = torch.cuda.Stream()
            side.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(side):
                self.forward(*ins, batch, image)  # warm-up outside the capture
            torch.cuda.current_stream().wait_stream(side)
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                outs = self.forward(*ins, batch, image)
            g = self._graphs[key] = (graph, ins, outs)
        graph, ins, outs = g
        for dst, src in zip(ins, (x, pos, parents, node_offsets, kv_len)):
            dst.copy_(src)
        graph.replay()
        return outs

    def commit(self, k_tree, v_tree, kv_len, kv_len_out, node_offsets, path, max_path, accept_len, batch):
        B.adt_kv_compact(self.k_cache, self.v_cache, kv_len, kv_len_out, k_tree, v_tree, node_offsets, path,
                         max_path, accept_len, B=batch, Hkv=self.s.kv_heads, D=self.s.head_dim,
                         num_layers=len(self.w.layers), max_kv=self.lmax,
                         cache_layer_stride=self.k_cache.stride(0), cache_stride_b=self.k_cache.stride(1),
                         cache_stride_h=self.k_cache.stride(2), tree_layer_stride=k_tree.stride(0))


    def commit_one(self, b, k_tree, v_tree, kv_len, kv_len_out, offs, path, max_path, accept_len):
        B.adt_kv_compact(self.k_cache[:, b:b + 1], self.v_cache[:, b:b + 1], kv_len, kv_len_out, k_tree, v_tree, offs,
                         path, max_path, accept_len, B=1, Hkv=self.s.kv_heads, D=self.s.head_dim,
                         num_layers=len(self.w.layers), max_kv=self.lmax, cache_layer_stride=self.k_cache.stride(0),
                         cache_stride_b=self.k_cache.stride(1), cache_stride_h=self.k_cache.stride(2),
                         tree_layer_stride=k_tree.stride(0))


def _chain(n, device):
    return torch.arange(-1, n - 1, dtype=torch.int32, device=device)


@dataclass
class DecodeStats:
    tokens: int = 0
    steps: int = 0
    accepted: int = 0          # accepted draft tokens (the bonus tokens not counted)
    accept_hist: dict = field(default_factory=dict)  # accepted length -> (image, step) count
    seconds: float = 0.0
    depth_sum: int = 0
    batch: int = 1

    @property
    def tau(self):
        """Mean tokens emitted per image and verify step (accepted + bonus)."""
        return self.tokens / max(self.steps * self.batch, 1)

    @property
    def mean_depth(self):
        return self.depth_sum / max(self.steps, 1)


class Decoder:
    """Target + draft head + controller for `batch` images of grid_h x grid_w
    tokens after a prompt (the same prompt for every image)."""

    def __init__(self, shape: ModelShape, *, batch=1, grid=(48, 48), prompt_len=16, seed=2025, device="cuda",
                 max_nodes=64, ctrl_params=None, draft_equals_target=False, target=None, graphs=False):
        s = self.s = shape
        self.batch, self.grid, self.prompt_len = batch, grid, prompt_len
        self.device = device
        self.max_nodes = max_nodes
        n_img = grid[0] * grid[1]
        self.lmax = prompt_len + n_img + 16
        tw = target if target is not None else DecoderWeights(s, s.layers, seed, device)
        self.target_w = tw
        self.target = TreeModel(s, tw, batch, self.lmax, max_nodes, device)
        # draft head: fc + one layer, sharing the target's embedding, norm and LM head
        if draft_equals_target:
            # a draft that reproduces a one-layer target exactly: fc passes the
            # embedding through, and the layer is the target's
            dw = DecoderWeights(s, 0, seed + 1, device, lm=False, draft_fc=True)
            dw.layers = tw.layers[:1]
            eye = torch.eye(s.hidden, dtype=s.dtype, device=device)
            dw.fc = torch.cat([eye, torch.zeros_like(eye)], 0)
        else:
            dw = DecoderWeights(s, 1, seed + 1, device, lm=False, draft_fc=True)
        self.draft_w = dw
        self.draft = TreeModel(s, dw, batch, self.lmax, 256, device)
        self.target.graphs_enabled = self.draft.graphs_enabled = graphs
        self.ctrl_params = dict(ctrl_params or {})
        self.ctrl_params.setdefault("d_lo", 1)
        self.ctrl_params.setdefault("d_hi", 9)
        self.k_max = self.ctrl_params.get("k_hi", 13)
        self.ws_expand = B.zeroed_workspace(B.adt_tree_expand_workspace_size(self.k_max, s.vocab, self.k_max), device)
        self.ws_rerank = B.zeroed_workspace(B.adt_tree_rerank_workspace_size(self._pool_cap()), device)

    def _pool_cap(self):
        d, k = self.ctrl_params["d_hi"], self.k_max
        return k + (d - 1) * k * k

    # ------------------------------------------------------------------ helpers
    def _embed(self, tokens):
        return self.target_w.embed[tokens.long()]

    def _logits(self, h):
        return lm_logits(self.target_w, h, self.s.eps)

    def _i32(self, x):
        return torch.as_tensor(x, dtype=torch.int32, device=self.device)

    # ------------------------------------------------------------------ prompt
    def prefill(self, prompt):
        """Target and draft caches for prompt[:-1] (chains from position 0);
        returns the per-image state of the first step."""
        s, dev, Bn = self.s, self.device, self.batch
        P = len(prompt)
        if not 2 <= P <= self.max_nodes + 1:
            raise ValueError("prompt of 2 .. max_nodes + 1 tokens (the prefill is one tree)")
        n = P - 1
        tok = self._i32(list(prompt[:-1]) * Bn)
        par = torch.cat([_chain(n, dev)] * Bn)
        offs = self._i32([b * n for b in range(Bn + 1)])
        zero = self._i32([0] * Bn)
        pos = torch.arange(n, device=dev, dtype=torch.int32).repeat(Bn)
        h, kt, vt = self.target.run(self._embed(tok), pos, par, offs, zero, Bn)
        path = torch.arange(n, dtype=torch.int32, device=dev).repeat(Bn, 1).contiguous()
        alen = self._i32([n - 1] * Bn)
        kv_out = torch.empty(Bn, dtype=torch.int32, device=dev)
        self.target.commit(kt, vt, zero, kv_out, offs, path, n, alen, Bn)
        feats = h.view(Bn, n, s.hidden)
        zf = torch.zeros(s.hidden, dtype=s.dtype, device=dev)
        state = []
        for b in range(Bn):
            # the draft catches up on prompt[:-1]: parent features f_{t-1} (zeros for t = 0)
            pf = torch.cat([zf[None], feats[b, :-1]], 0)
            state.append(dict(kv=n, dkv=0, root=int(prompt[-1]), root_pf=feats[b, -1].clone(),
                              catch_tok=list(prompt[:-1]),
                              catch_pf=pf, pos=0))
        return state

    # ------------------------------------------------------------------ draft
    def _draft_image(self, b, st, depth, width):
        """Grows image b's candidate pool: `depth` expand calls fed by the
        draft head; commits the catch-up tokens' draft K/V.  Returns the pool
        (tokens, scores, parents) as device tensors."""
        s, dev = self.s, self.device
        m = len(st["catch_tok"])
        C = width + (depth - 1) * width * width
        pool_tok = torch.empty(C, dtype=torch.int32, device=dev)
        pool_sc = torch.empty(C, dtype=torch.float32, device=dev)
        pool_lp = torch.empty(C, dtype=torch.float32, device=dev)
        pool_par = torch.empty(C, dtype=torch.int32, device=dev)
        # draft tree: catch-up chain (m nodes), the root (node m), then the kept nodes of each depth
        tok = torch.cat([self._i32(st["catch_tok"]), self._i32([st["root"]])])
        par = _chain(m + 1, dev)
        pf = torch.cat([st["catch_pf"], st["root_pf"][None]], 0)
        dep = torch.arange(m + 1, device=dev, dtype=torch.int32)
        pool2node = torch.full((C,), -1, dtype=torch.int64, device=dev)
        fscore = torch.zeros(1, dtype=torch.float32, device=dev)
        fid = torch.full((1,), -1, dtype=torch.int32, device=dev)
        front = torch.tensor([m], dtype=torch.int64, device=dev)  # draft-tree nodes of the frontier
        dkv = self._i32([st["dkv"]])
        base = 0
        kt = vt = None
        for d in range(depth):
            n = tok.numel()
            x = torch.cat([self._embed(tok), pf], 1) @ self.draft_w.fc
            offs = self._i32([0, n])
            h, kt, vt = self.draft.run(x, st["dkv"] + dep, par, offs, dkv, 1, image=b)
            logits = self._logits(h[front]).contiguous()
            F = front.numel()
            keep = torch.empty(width, dtype=torch.int32, device=dev)
            nsc = torch.empty(width, dtype=torch.float32, device=dev)
            nid = torch.empty(width, dtype=torch.int32, device=dev)
            last = d + 1 == depth  # no next frontier after the last layer
            B.adt_tree_expand(logits, fscore, fid, F=F, V=s.vocab, k_child=width, k_keep=width, child_id_base=base,
                              child_token=pool_tok[base:base + F * width], child_logp=pool_lp[base:base + F * width],
                              child_score=pool_sc[base:base + F * width],
                              child_parent=pool_par[base:base + F * width], keep_idx=None if last else keep,
                              next_score=None if last else nsc, next_id=None if last else nid,
                              workspace=self.ws_expand)
            if d + 1 < depth:
                # the kept candidates join the draft tree (their parents: frontier nodes)
                kept = nid.long()
                ppool = pool_par[kept].long()
                pnode = torch.where(ppool < 0, torch.full_like(ppool, m), pool2node[ppool.clamp(min=0)])
                new = torch.arange(n, n + width, device=dev)
                pool2node[kept] = new
                tok = torch.cat([tok, pool_tok[kept]])
                par = torch.cat([par, pnode.to(torch.int32)])
                pf = torch.cat([pf, h[pnode]], 0)
                dep = torch.cat([dep, dep[pnode] + 1])
                front = new
            fscore, fid = nsc, nid
            base += F * width
        # commit the catch-up chain's draft K/V (not the root's: it is caught up next step)
        path = torch.arange(m, dtype=torch.int32, device=dev)[None].contiguous()
        alen = self._i32([m - 1])
        out = torch.empty(1, dtype=torch.int32, device=dev)
        self.draft.commit_one(b, kt, vt, dkv, out, self._i32([0, kt.shape[1]]), path, m, alen)
        st["dkv"] += m
        return pool_tok, pool_sc, pool_par, C

    # ------------------------------------------------------------------ one step
    def step(self, state, ctrls):
        s, dev, Bn = self.s, self.device, self.batch
        n_img = self.grid[0] * self.grid[1]
        dk = [c.next(min(st["pos"], n_img - 1)) for c, st in zip(ctrls, state)]
        trees = []
        for b, (st, (d, k)) in enumerate(zip(state, dk)):
            pool_tok, pool_sc, pool_par, C = self._draft_image(b, st, d, k)
            n = min(self.max_nodes, C + 1)
            t = dict(tokens=torch.empty(n, dtype=torch.int32, device=dev),
                     parents=torch.empty(n, dtype=torch.int32, device=dev),
                     cand=torch.empty(n, dtype=torch.int32, device=dev),
                     depth=torch.empty(n, dtype=torch.int32, device=dev))
            B.adt_tree_rerank(pool_tok, pool_sc, pool_par, C, self._i32([st["root"]]), n, tokens=t["tokens"],
                              parents=t["parents"], cand_index=t["cand"], depth=t["depth"],
                              workspace=self.ws_rerank)
            trees.append(t)
        sizes = [t["tokens"].numel() for t in trees]
        offs_l = [0]
        for n in sizes:
            offs_l.append(offs_l[-1] + n)
        offs = self._i32(offs_l)
        tok = torch.cat([t["tokens"] for t in trees])
        par = torch.cat([t["parents"] for t in trees])
        kv = self._i32([st["kv"] for st in state])
        pos = torch.cat([t["depth"] + st["kv"] for t, st in zip(trees, state)])
        h, kt, vt = self.target.run(self._embed(tok), pos, par, offs, kv, Bn)
        logits = self._logits(h).contiguous()
        max_path = max(d for d, _ in dk) + 1
        path = torch.full((Bn, max_path), -1, dtype=torch.int32, device=dev)
        alen = torch.empty(Bn, dtype=torch.int32, device=dev)
        bonus = torch.empty(Bn, dtype=torch.int32, device=dev)
        B.adt_tree_accept(logits, None, tok, par, offs, B=Bn, V=s.vocab, max_nodes=max(sizes),
                          mode=B.ACCEPT_GREEDY, path=path, max_path=max_path, accept_len=alen, bonus_token=bonus)
        kv_out = torch.empty(Bn, dtype=torch.int32, device=dev)
        self.target.commit(kt, vt, kv, kv_out, offs, path, max_path, alen, Bn)
        # one host read per step: the path decides the next trees
        path_h, alen_h, bonus_h = path.cpu().tolist(), alen.cpu().tolist(), bonus.cpu().tolist()
        emitted = []
        for b, st in enumerate(state):
            a = alen_h[b]
            nodes = path_h[b][:a + 1]
            glob = [offs_l[b] + v for v in nodes]
            toks = tok[glob].tolist()
            new = toks[1:] + [bonus_h[b]]
            new = new[: max(0, n_img - st["pos"])]
            emitted.append(new)
            if st["pos"] < n_img:
                ctrls[b].update(st["pos"], min(a, dk[b][0]))
            # the next step's draft catch-up: this step's path with the true features
            idx = torch.tensor(glob, device=dev)
            st["catch_tok"] = toks
            st["catch_pf"] = torch.cat([st["root_pf"][None], h[idx[:-1]]], 0)
            st["root"] = bonus_h[b]
            st["root_pf"] = h[idx[-1]].clone()
            st["kv"] += a + 1
            st["pos"] += len(new)
        return emitted, dk, alen_h

    def generate(self, prompt, ctrl_params=None):
        """Decodes grid_h * grid_w tokens per image.  Returns (tokens per
        image, DecodeStats)."""
        n_img = self.grid[0] * self.grid[1]
        params = dict(self.ctrl_params)
        if ctrl_params:
            params.update(ctrl_params)
        ctrls = [B.Controller(*self.grid, **dict(params, seed=params.get("seed", 0) + b)) for b in range(self.batch)]
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        state = self.prefill(prompt)
        out = [[] for _ in range(self.batch)]
        stats = DecodeStats(batch=self.batch)
        while any(st["pos"] < n_img for st in state):
            emitted, dk, alen = self.step(state, ctrls)
            stats.steps += 1
            stats.depth_sum += sum(d for d, _ in dk) // self.batch
            for b in range(self.batch):
                out[b] += emitted[b]
                stats.accepted += alen[b]
                stats.accept_hist[alen[b]] = stats.accept_hist.get(alen[b], 0) + 1
        torch.cuda.synchronize()
        stats.seconds = time.perf_counter() - t0
        stats.tokens = sum(len(o) for o in out)
        return out, stats




class DenseModel:
    """The same decoder stack as TreeModel for vanilla decoding, without the
    library: a plain KV cache tensor written by indexing, and attention by
    torch's scaled_dot_product_attention (in fp32 by default) over the cache
    with a causal mask.  Every image holds the same number of tokens (they
    advance in lockstep), so one start position serves the batch.  The
    shapes are static (attention always spans the whole cache, masked), so
    a step can be captured in a CUDA graph."""

    def __init__(self, shape: ModelShape, weights: DecoderWeights, batch: int, lmax: int, device,
                 attn_dtype=torch.float32):
        s = self.s = shape
        self.w = weights
        self.lmax = lmax
        self.batch = batch
        self.attn_dtype = attn_dtype
        L = len(weights.layers)
        bf = dict(dtype=torch.bfloat16, device=device)
        self.k_cache = torch.zeros((L, batch, s.kv_heads, lmax, s.head_dim), **bf)
        self.v_cache = torch.zeros((L, batch, s.kv_heads, lmax, s.head_dim), **bf)
        self.keys = torch.arange(lmax, device=device)
        self.device = device

    def forward(self, x, start):
        """x [batch, n, hidden]: n new tokens per image at positions start ..
        start + n - 1 (start: a 0-d int64 device tensor).  Writes their K/V
        into the cache and returns the final hidden states [batch, n, hidden]."""
        s = self.s
        Bn, n, _ = x.shape
        hq, hk = s.heads * s.head_dim, s.kv_heads * s.head_dim
        pos = start + torch.arange(n, device=self.device)
        rows = pos.repeat(Bn)
        visible = self.keys[None, :] <= pos[:, None]          # [n, lmax]: causal over the cache
        group = s.heads // s.kv_heads
        for li, lw in enumerate(self.w.layers):
            h = _rms_norm(x, lw["ln1"], s.eps).view(Bn * n, -1)
            qkv = h @ lw["wqkv"]
            q = _rope(qkv[:, :hq].view(Bn * n, s.heads, s.head_dim), rows, s.rope_theta).to(torch.bfloat16)
            k = _rope(qkv[:, hq:hq + hk].view(Bn * n, s.kv_heads, s.head_dim), rows, s.rope_theta).to(torch.bfloat16)
            v = qkv[:, hq + hk:].view(Bn * n, s.kv_heads, s.head_dim).to(torch.bfloat16)
            self.k_cache[li].index_copy_(2, pos, k.view(Bn, n, s.kv_heads, s.head_dim).transpose(1, 2))
            self.v_cache[li].index_copy_(2, pos, v.view(Bn, n, s.kv_heads, s.head_dim).transpose(1, 2))
            kc = self.k_cache[li].to(self.attn_dtype)
            vc = self.v_cache[li].to(self.attn_dtype)
            if group > 1:
                kc = kc.repeat_interleave(group, dim=1)
                vc = vc.repeat_interleave(group, dim=1)
            qh = q.view(Bn, n, s.heads, s.head_dim).transpose(1, 2).to(self.attn_dtype)
            o = torch.nn.functional.scaled_dot_product_attention(qh, kc, vc, attn_mask=visible,
                                                                 scale=s.head_dim ** -0.5)
            o = o.transpose(1, 2).reshape(Bn * n, hq).to(torch.bfloat16)
            xf = x.view(Bn * n, -1) + o.to(x.dtype) @ lw["wo"]
            h = _rms_norm(xf, lw["ln2"], s.eps)
            gu = h @ lw["wgu"]
            xf = xf + (torch.nn.functional.silu(gu[:, : s.ffn].float()) * gu[:, s.ffn:].float()).to(x.dtype) @ lw["wd"]
            x = xf.view(Bn, n, -1)
        return x


def greedy_decode(shape: ModelShape, weights: DecoderWeights, prompt, n_tokens, device="cuda", batch=1,
                  return_margins=False, graphs=False, attn_dtype=torch.float32, forced=None, stats=None):
    """Vanilla greedy decoding with the same target, one token per step,
    through DenseModel: none of the library's entry points (neither its
    attention nor its KV commit) is on this path, so it is an independent
    reference for the tree decoder's output (greedy verification is
    lossless).  Returns the tokens (and, with return_margins, the top-1
    minus top-2 logit gap of every decision over the standard deviation of
    that logit row).  With graphs, each step replays one CUDA graph.

    forced (a [batch][n_tokens] token list) teacher-forces the sequence: step
    i still returns the target's greedy choice, but the token fed to step
    i + 1 is forced[b][i], so every position of another decoder's output can
    be checked against the target's choice given that output's own prefix.
    stats (a dict), if given, receives the seconds of the token loop alone
    (after the prefill and any graph capture)."""
    if not 2 <= len(prompt) <= 257:
        raise ValueError("prompt of 2 .. 257 tokens")
    P = len(prompt)
    model = DenseModel(shape, weights, batch, P + n_tokens + 16, device, attn_dtype)
    dev = device
    tok = torch.tensor(list(prompt[:-1]), dtype=torch.long, device=dev)
    model.forward(weights.embed[tok][None].expand(batch, -1, -1).contiguous(),
                  torch.zeros((), dtype=torch.long, device=dev))
    start = torch.full((), P - 1, dtype=torch.long, device=dev)
    root = torch.full((batch,), int(prompt[-1]), dtype=torch.long, device=dev)

    def one_step():
        h = model.forward(weights.embed[root][:, None, :], start)
        logits = lm_logits(weights, h[:, 0], shape.eps)
        top2 = torch.topk(logits, 2, dim=-1)
        return top2.indices[:, 0], (top2.values[:, 0] - top2.values[:, 1]) / logits.std(dim=-1)

    graph = None
    if graphs:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        saved = [model.k_cache.clone(), model.v_cache.clone()]
        with torch.cuda.stream(side):
            one_step()  # warm-up outside the capture (it writes a cache row that is restored below)
        torch.cuda.current_stream().wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            g_next, g_margin = one_step()
        model.k_cache.copy_(saved[0])
        model.v_cache.copy_(saved[1])
    feed = None if forced is None else torch.tensor(forced, dtype=torch.long, device=dev)
    out, margins = [], []
    if str(dev).startswith("cuda"):
        torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(n_tokens):
        if graph is not None:
            graph.replay()
            nxt, margin = g_next.clone(), g_margin.clone()
        else:
            nxt, margin = one_step()
        out.append(nxt)
        margins.append(margin)
        root.copy_(nxt if feed is None else feed[:, i])
        start += 1
    toks = torch.stack(out, 1).cpu().tolist()
    if stats is not None:  # (the .cpu() above waited for the device)
        stats["seconds"] = time.perf_counter() - t0
    if return_margins:
        return toks, torch.stack(margins, 1).cpu().tolist()
    return toks


def tokens_per_second(stats: DecodeStats):
    return stats.tokens / stats.seconds if stats.seconds > 0 else math.nan
