"""Shared builders for the GPU parity tests: seeded inputs from synth, the
library call through the binding, and the oracle on the same inputs."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2512_21857_gb300 import binding as B
from paper_2512_21857_gb300 import synth

# Attention: |gpu - oracle| <= ATOL + OUT_RTOL |oracle| elementwise, and
# max |gpu - oracle| / max |oracle| <= NORM_RTOL.  ATOL covers the outputs
# of long prefixes (|o| ~ 0.02-0.1); the output is bf16, whose rounding alone
# is up to half an ulp, 2^-9 |o|, which exceeds ATOL / 2 once |o| > 2.5 (rows
# that see few keys, short prefixes): OUT_RTOL adds that half ulp.
ATOL = 1e-2
OUT_RTOL = 2.0 ** -9
NORM_RTOL = 2e-2
# lse: the log of the normaliser the kernel applies, the sum of the
# probabilities as rounded to bf16 for the PV product; each rounding is
# within a relative 2^-9, so the sum (and its log) is within 2^-9 of the
# exact one, plus fp32 accumulation and exponential error: bound 2^-8.
LSE_ATOL = 2.0 ** -8


def ensure_built():
    from paper_2512_21857_gb300 import build
    build.build()
    B.lib()


def i32(x, dev="cuda"):
    return torch.as_tensor(np.asarray(x, dtype=np.int32), device=dev)


def f32(x, dev="cuda"):
    return torch.as_tensor(np.asarray(x, dtype=np.float32), device=dev)


def f32_rows(x, dev="cuda"):
    """A [rows][V] fp32 array on the device with its rows padded to a multiple
    of 4 floats (the row stride the ABI requires); the [:, :V] view."""
    x = np.asarray(x, dtype=np.float32)
    ld = (x.shape[1] + 3) // 4 * 4
    t = torch.zeros((x.shape[0], ld), dtype=torch.float32, device=dev)
    t[:, :x.shape[1]] = torch.as_tensor(x, device=dev)
    return t[:, :x.shape[1]]


class AttnCase:
    """Inputs of one adt_tree_attn call: B trees of the given sizes, prefix
    lengths, heads and head dim."""

    def __init__(self, sizes, kv_lens, H, Hkv, D, seed, chain=False, lmax=None, max_depth=6, max_children=4):
        self.sizes, self.kv_lens, self.H, self.Hkv, self.D = list(sizes), list(kv_lens), H, Hkv, D
        self.B = len(sizes)
        self.tb = synth.tree_batch(sizes, 1000, seed, chain=chain, max_depth=max_depth, max_children=max_children)
        ntot = int(self.tb.node_offsets[-1])
        self.ntot = ntot
        self.lmax = lmax if lmax is not None else max(max(kv_lens), 1) + 8
        self.q = synth.bf16_normal((ntot, H, D), seed, "q")
        self.kc = synth.bf16_normal((self.B, Hkv, self.lmax, D), seed, "kc")
        self.vc = synth.bf16_normal((self.B, Hkv, self.lmax, D), seed, "vc")
        self.kt = synth.bf16_normal((ntot, Hkv, D), seed, "kt")
        self.vt = synth.bf16_normal((ntot, Hkv, D), seed, "vt")
        self.scale = 1.0 / math.sqrt(D)

    def run_gpu(self, max_nodes=None, max_kv=None, ws=None):
        dev = "cuda"
        max_nodes = max_nodes or max(self.sizes)
        max_kv = max(self.kv_lens) if max_kv is None else max_kv
        out = torch.empty((self.ntot, self.H, self.D), dtype=torch.bfloat16, device=dev)
        lse = torch.empty((self.ntot, self.H), dtype=torch.float32, device=dev)
        if ws is None:
            ws = B.zeroed_workspace(B.adt_tree_attn_workspace_size(self.B, self.H, self.D, max_nodes, max_kv))
        kc, vc = self.kc.to(dev), self.vc.to(dev)
        B.adt_tree_attn(self.q.to(dev), kc, vc, i32(self.kv_lens), self.kt.to(dev), self.vt.to(dev),
                        i32(self.tb.parents), i32(self.tb.node_offsets), B=self.B, H=self.H, Hkv=self.Hkv, D=self.D,
                        max_nodes=max_nodes, max_kv=max_kv, softmax_scale=self.scale, out=out, lse=lse,
                        workspace=ws)
        torch.cuda.synchronize()
        return out.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64), ws

    def run_oracle(self):
        return oracle.tree_attention(self.q.double().numpy(), self.kc.double().numpy(), self.vc.double().numpy(),
                                     self.kv_lens, self.kt.double().numpy(), self.vt.double().numpy(),
                                     self.tb.parents, self.tb.node_offsets, self.scale)


def assert_attention_close(got, ref):
    err = np.abs(got - ref)
    excess = err - (ATOL + OUT_RTOL * np.abs(ref))
    assert excess.max() <= 0, f"max abs err {err.max():.3e}, max excess over the bound {excess.max():.3e}"
    assert err.max() / max(np.abs(ref).max(), 1e-30) <= NORM_RTOL, "normwise error"


def grow_candidates_gpu(draft_rows, k, depth, root_token, n_nodes, temperature=1.0):
    """Runs adt_tree_expand depth times (frontier chained on the device) and
    adt_tree_rerank; draft_rows[d] holds the rows of depth d (F_d x V).
    Returns dict of numpy arrays: per-call expand outputs and the tree."""
    dev = "cuda"
    V = draft_rows[0].shape[1]
    pool_tok, pool_score, pool_par = [], [], []
    calls = []
    fscore = torch.zeros(1, dtype=torch.float32, device=dev)
    fid = torch.full((1,), -1, dtype=torch.int32, device=dev)
    base = 0
    for d in range(depth):
        F = int(fscore.numel())
        lg = torch.as_tensor(draft_rows[d][:F], device=dev).contiguous()
        ws = B.zeroed_workspace(B.adt_tree_expand_workspace_size(F, V, k))
        out = dict(child_token=torch.empty(F * k, dtype=torch.int32, device=dev),
                   child_logp=torch.empty(F * k, dtype=torch.float32, device=dev),
                   child_score=torch.empty(F * k, dtype=torch.float32, device=dev),
                   child_parent=torch.empty(F * k, dtype=torch.int32, device=dev))
        keep = min(k, F * k)
        keep_idx = torch.empty(keep, dtype=torch.int32, device=dev)
        nscore = torch.empty(keep, dtype=torch.float32, device=dev)
        nid = torch.empty(keep, dtype=torch.int32, device=dev)
        B.adt_tree_expand(lg, fscore, fid, F=F, V=V, k_child=k, k_keep=keep, temperature=temperature,
                          child_id_base=base, keep_idx=keep_idx, next_score=nscore, next_id=nid, workspace=ws,
                          **out)
        calls.append({kk: v.cpu().numpy() for kk, v in out.items()} | dict(
            keep_idx=keep_idx.cpu().numpy(), next_score=nscore.cpu().numpy(), next_id=nid.cpu().numpy(),
            frontier_score=fscore.cpu().numpy(), frontier_id=fid.cpu().numpy(), logits=draft_rows[d][:F]))
        pool_tok.append(out["child_token"])
        pool_score.append(out["child_score"])
        pool_par.append(out["child_parent"])
        base += F * k
        fscore, fid = nscore, nid
    tok = torch.cat(pool_tok)
    sc = torch.cat(pool_score)
    par = torch.cat(pool_par)
    C = int(tok.numel())
    n = min(n_nodes, C + 1)
    res = dict(tokens=torch.empty(n, dtype=torch.int32, device=dev),
               parents=torch.empty(n, dtype=torch.int32, device=dev),
               cand_index=torch.empty(n, dtype=torch.int32, device=dev),
               depth=torch.empty(n, dtype=torch.int32, device=dev))
    ws = B.zeroed_workspace(B.adt_tree_rerank_workspace_size(C))
    B.adt_tree_rerank(tok, sc, par, C, i32([root_token]), n, workspace=ws, **res)
    torch.cuda.synchronize()
    return dict(calls=calls, pool_token=tok.cpu().numpy(), pool_score=sc.cpu().numpy(),
                pool_parent=par.cpu().numpy(), tree={kk: v.cpu().numpy() for kk, v in res.items()})


def run_accept_gpu(target, draft, tb, mode, ua=None, us=None, temperature=1.0, max_path=16, draft_row=None):
    dev = "cuda"
    Bn = len(tb.node_offsets) - 1
    sizes = np.diff(tb.node_offsets)
    V = target.shape[1]
    path = torch.empty((Bn, max_path), dtype=torch.int32, device=dev)
    alen = torch.empty(Bn, dtype=torch.int32, device=dev)
    bonus = torch.empty(Bn, dtype=torch.int32, device=dev)
    B.adt_tree_accept(f32_rows(target), None if draft is None else f32_rows(draft), i32(tb.tokens), i32(tb.parents),
                      i32(tb.node_offsets), B=Bn, V=V, max_nodes=int(sizes.max()), mode=mode,
                      u_accept=None if ua is None else f32(ua), u_sample=None if us is None else f32(us),
                      temperature=temperature, path=path, max_path=max_path, accept_len=alen, bonus_token=bonus,
                      draft_row=None if draft_row is None else i32(draft_row))
    torch.cuda.synchronize()
    return path.cpu().numpy(), alen.cpu().numpy(), bonus.cpu().numpy()
