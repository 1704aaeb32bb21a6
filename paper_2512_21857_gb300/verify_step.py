"""One ADT-Tree verify step on the GPU, launched through the C ABI.

A step, for each image b of a batch (Sec. 3.1, Fig. 5, Eq. 4):
  1. d_b calls of adt_tree_expand grow the draft tree layer by layer from the
     draft rows of the current frontier (row f of layer d is the draft
     distribution of frontier node f; layer 0 has the root only);
  2. adt_tree_rerank keeps the n_b - 1 best candidates plus the root;
  3. for every transformer layer, adt_tree_attn attends the n_b nodes over
     the prefix KV cache and their ancestors;
  4. adt_tree_accept walks each tree (greedy or speculative sampling);
  5. adt_kv_compact commits the accepted path's K/V for all layers.
Tree shapes (d_b, k_b) are host decisions (the controller, Sec. 4), so all
launch shapes are known on the host and the whole step can be captured in a
CUDA graph.  The images' draft phases (1-2) are independent chains of small,
latency-bound launches: with more than one image each chain runs on its own
stream, forked from the step's stream and joined back to it (in a captured
graph, parallel branches).  This module only allocates device memory
(torch) and issues the library calls; every computation runs in the
library's kernels.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import binding as B


@dataclass
class StepShape:
    layers: int
    H: int
    Hkv: int
    D: int
    V: int
    kv_len: list          # prefix length per image
    depth: list           # d_b per image (number of expand calls)
    width: list           # k_b per image (children per node = frontier size)
    max_nodes: int = 64   # tree size cap (root included)
    lmax: int = 0         # cache capacity per image (default: max kv_len + max_nodes)
    mode: int = B.ACCEPT_GREEDY
    temperature: float = 1.0

    @property
    def batch(self):
        return len(self.kv_len)

    def candidates(self, b):
        k, d = self.width[b], self.depth[b]
        return k + (d - 1) * k * k  # C_S of Eq. 6

    def nodes(self, b):
        return min(self.max_nodes, self.candidates(b) + 1)


class TreeVerifyStep:
    """Persistent buffers and the launch sequence of one verify step."""

    # Per-step inputs (what the model produces for each step); the KV cache
    # persists across steps.
    STEP_INPUTS = ("q", "k_tree", "v_tree", "target", "u_accept", "u_sample", "root_token", "draft_rows")

    def __init__(self, shape: StepShape, device="cuda", keep_layer_outputs=False, input_slots=1):
        s = self.shape = shape
        self.device = device
        Bn = s.batch
        self.n = [s.nodes(b) for b in range(Bn)]
        offs = [0]
        for n in self.n:
            offs.append(offs[-1] + n)
        self.ntot = offs[-1]
        self.lmax = s.lmax or (max(s.kv_len) + s.max_nodes)
        self.max_path = max(s.depth) + 1
        dev = device
        i32 = dict(dtype=torch.int32, device=dev)
        f32 = dict(dtype=torch.float32, device=dev)
        bf16 = dict(dtype=torch.bfloat16, device=dev)
        # model-side tensors (inputs of the step)
        self.k_cache = torch.zeros((s.layers, Bn, s.Hkv, self.lmax, s.D), **bf16)
        self.v_cache = torch.zeros((s.layers, Bn, s.Hkv, self.lmax, s.D), **bf16)
        # per-step inputs: `input_slots` copies, so that the inputs of the next
        # step can be copied in while this one computes (use_slot picks one)
        self._slots = [dict(q=torch.zeros((s.layers, self.ntot, s.H, s.D), **bf16),
                            k_tree=torch.zeros((s.layers, self.ntot, s.Hkv, s.D), **bf16),
                            v_tree=torch.zeros((s.layers, self.ntot, s.Hkv, s.D), **bf16),
                            draft_rows=[torch.zeros((s.depth[b], s.width[b], s.V), **f32) for b in range(Bn)],
                            target=torch.zeros((self.ntot, s.V), **f32),
                            u_accept=torch.zeros(self.ntot, **f32),
                            u_sample=torch.zeros(self.ntot, **f32),
                            root_token=torch.zeros(Bn, **i32))
                       for _ in range(input_slots)]
        self.use_slot(0)
        self.kv_len = torch.tensor(s.kv_len, **i32)
        self.node_offsets = torch.tensor(offs, **i32)
        # intermediate and output buffers
        kmax = max(s.width)
        self.pool_tok = [torch.zeros(s.candidates(b), **i32) for b in range(Bn)]
        self.pool_score = [torch.zeros(s.candidates(b), **f32) for b in range(Bn)]
        self.pool_logp = [torch.zeros(s.candidates(b), **f32) for b in range(Bn)]
        self.pool_par = [torch.zeros(s.candidates(b), **i32) for b in range(Bn)]
        # per image: the two alternating frontiers and the kept indices, so
        # that the images' draft chains can run concurrently
        self.front_score = [torch.zeros((2, kmax), **f32) for _ in range(Bn)]
        self.front_id = [torch.full((2, kmax), -1, **i32) for _ in range(Bn)]
        self.root_score = torch.zeros(1, **f32)
        self.root_id = torch.full((1,), -1, **i32)
        self.keep_idx = [torch.zeros(kmax, **i32) for _ in range(Bn)]
        self.tokens = torch.zeros(self.ntot, **i32)
        self.parents = torch.zeros(self.ntot, **i32)
        self.cand_index = torch.zeros(self.ntot, **i32)
        self.node_depth = torch.zeros(self.ntot, **i32)
        # attention output: one buffer reused by every layer, or one per layer
        self.keep_layer_outputs = keep_layer_outputs
        self.attn_out = torch.zeros(((s.layers if keep_layer_outputs else 1), self.ntot, s.H, s.D), **bf16)
        self.path = torch.zeros((Bn, self.max_path), **i32)
        self.accept_len = torch.zeros(Bn, **i32)
        self.bonus = torch.zeros(Bn, **i32)
        self.kv_len_out = torch.zeros(Bn, **i32)
        # workspaces (zero-filled once; the library leaves its counters at
        # zero); one expand and one rerank workspace per image's draft chain
        self.ws_expand = [B.zeroed_workspace(max(B.adt_tree_expand_workspace_size(kmax, s.V, kmax), 16), dev)
                          for _ in range(Bn)]
        self.ws_rerank = [B.zeroed_workspace(B.adt_tree_rerank_workspace_size(s.candidates(b)), dev)
                          for b in range(Bn)]
        self.draft_streams = [torch.cuda.Stream(device=dev) for _ in range(Bn)] if Bn > 1 else []
        self.ws_attn = B.zeroed_workspace(
            B.adt_tree_attn_workspace_size(Bn, s.H, s.D, s.max_nodes, self.lmax), dev)

    def use_slot(self, i):
        """Points the step's per-step input attributes at input slot i; the
        launches that follow (and graphs captured from them) read that slot."""
        self.slot = i
        for name, t in self._slots[i].items():
            setattr(self, name, t)

    def step_input_tensors(self):
        """The current slot's per-step input tensors, in a fixed order."""
        return [self.q, self.k_tree, self.v_tree, self.target, self.u_accept, self.u_sample,
                self.root_token] + list(self.draft_rows)

    # -------------------------------------------------------------- phases
    def launch_draft_image(self, b, stream=None, rerank=True):
        """Expand d_b layers and rerank (unless `rerank` is false), for image b."""
        s = self.shape
        k = s.width[b]
        base = 0
        fscore, fid = self.root_score, self.root_id
        rows = self.draft_rows[b]
        front_score, front_id, keep = self.front_score[b], self.front_id[b], self.keep_idx[b]
        for d in range(s.depth[b]):
            F = 1 if d == 0 else k
            nxt = d % 2
            last = d == s.depth[b] - 1  # the tree's last layer: no next frontier
            B.adt_tree_expand(rows[d, :F], fscore, fid, F=F, V=s.V, k_child=k, k_keep=k,
                              temperature=1.0, child_id_base=base,
                              child_token=self.pool_tok[b][base:base + F * k],
                              child_logp=self.pool_logp[b][base:base + F * k],
                              child_score=self.pool_score[b][base:base + F * k],
                              child_parent=self.pool_par[b][base:base + F * k],
                              keep_idx=None if last else keep[:k],
                              next_score=None if last else front_score[nxt, :k],
                              next_id=None if last else front_id[nxt, :k], workspace=self.ws_expand[b],
                              stream=stream)
            fscore, fid = front_score[nxt, :k], front_id[nxt, :k]
            base += F * k
        if not rerank:
            return
        lo, hi = int(self.node_offsets_host(b)), int(self.node_offsets_host(b + 1))
        B.adt_tree_rerank(self.pool_tok[b], self.pool_score[b], self.pool_par[b], base,
                          self.root_token[b:b + 1], hi - lo, tokens=self.tokens[lo:hi],
                          parents=self.parents[lo:hi], cand_index=self.cand_index[lo:hi],
                          depth=self.node_depth[lo:hi], workspace=self.ws_rerank[b], stream=stream)

    def launch_draft(self, stream=None):
        """Expand d_b layers and rerank, for every image: one chain, or with
        several images one chain per image on its own stream, forked from
        `stream` and joined back to it."""
        if self.shape.batch == 1:
            self.launch_draft_image(0, stream)
            return
        main = stream if stream is not None else torch.cuda.current_stream()
        fork = torch.cuda.Event()
        fork.record(main)
        for b, sb in enumerate(self.draft_streams):
            sb.wait_event(fork)
            self.launch_draft_image(b, sb)
            join = torch.cuda.Event()
            join.record(sb)
            main.wait_event(join)

    def node_offsets_host(self, i):
        return sum(self.n[:i])

    def launch_attention(self, layer, stream=None):
        s = self.shape
        kc = self.k_cache[layer]
        B.adt_tree_attn(self.q[layer], kc, self.v_cache[layer], self.kv_len, self.k_tree[layer],
                        self.v_tree[layer], self.parents, self.node_offsets, B=s.batch, H=s.H, Hkv=s.Hkv,
                        D=s.D, max_nodes=s.max_nodes, max_kv=self.lmax, softmax_scale=s.D ** -0.5,
                        out=self.attn_out[layer if self.keep_layer_outputs else 0], lse=None,
                        workspace=self.ws_attn, stream=stream)

    def launch_verify(self, stream=None):
        s = self.shape
        B.adt_tree_accept(self.target, None, self.tokens, self.parents, self.node_offsets, B=s.batch, V=s.V,
                          max_nodes=max(self.n), mode=s.mode, u_accept=self.u_accept, u_sample=self.u_sample,
                          temperature=s.temperature, path=self.path, max_path=self.max_path,
                          accept_len=self.accept_len, bonus_token=self.bonus, stream=stream)
        B.adt_kv_compact(self.k_cache, self.v_cache, self.kv_len, self.kv_len_out, self.k_tree, self.v_tree,
                         self.node_offsets, self.path, self.max_path, self.accept_len, B=s.batch, Hkv=s.Hkv,
                         D=s.D, num_layers=s.layers, max_kv=self.lmax,
                         cache_layer_stride=self.k_cache.stride(0), cache_stride_b=self.k_cache.stride(1),
                         cache_stride_h=self.k_cache.stride(2), tree_layer_stride=self.k_tree.stride(0),
                         stream=stream)

    def launch(self, stream=None):
        """The whole step: draft growth, attention over every layer, accept, commit."""
        self.launch_draft(stream)
        for layer in range(self.shape.layers):
            self.launch_attention(layer, stream)
        self.launch_verify(stream)

    def load_inputs(self, inp):
        """Copies a dict of host inputs (see synth.step_inputs) into the step's
        device buffers."""
        for name in ("k_cache", "v_cache", "q", "k_tree", "v_tree", "target", "u_accept", "u_sample",
                     "root_token"):
            if name in inp:
                getattr(self, name).copy_(torch.as_tensor(inp[name]))
        if "draft_rows" in inp:
            for b, rows in enumerate(inp["draft_rows"]):
                self.draft_rows[b].copy_(torch.as_tensor(rows))

    def kernel_launches_per_step(self):
        s = self.shape
        return sum(s.depth) + s.batch + s.layers + 2

    def algorithmic_bytes(self):
        """Bytes the step must move at minimum (reads + writes)."""
        s = self.shape
        bf = 2
        attn = 0
        for b in range(s.batch):
            n = self.n[b]
            attn += 2 * s.kv_len[b] * s.Hkv * s.D * bf          # prefix K and V
            attn += 2 * n * s.Hkv * s.D * bf                    # tree K and V
            attn += 2 * n * s.H * s.D * bf                      # Q in, O out
        return dict(attention_per_layer=attn, attention=attn * s.layers)
