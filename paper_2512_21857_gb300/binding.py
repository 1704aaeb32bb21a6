"""Thin Python binding of libadt (ctypes): argument marshalling only.

Each function has the name of the C entry point it calls and takes torch
tensors in place of raw pointers; every step of the computation runs in the
library's CUDA kernels.  A non-OK status raises AdtError.  The library must
have been built (``python -m paper_2512_21857_gb300.build``); importing a
missing library raises instead of falling back to anything else.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libadt.so")

ADT_OK = 0
STATUS_NAMES = {0: "ADT_OK", 1: "ADT_ERR_INVALID_ARG", 2: "ADT_ERR_UNSUPPORTED", 3: "ADT_ERR_CUDA",
                4: "ADT_ERR_TIMEOUT", 5: "ADT_ERR_WORKSPACE", 6: "ADT_ERR_DEVICE"}
ACCEPT_GREEDY, ACCEPT_SPEC, ACCEPT_SPEC_DET = 0, 1, 2
INIT_HORIZONTAL, INIT_VERTICAL, INIT_RANDOM, INIT_TOKENFLOCK = 0, 1, 2, 3
DEVERR_BAD_TREE, DEVERR_KV_RANGE, DEVERR_BAD_PATH, DEVERR_TIMEOUT, DEVERR_BAD_INDEX = 1, 2, 4, 8, 16

EXPORTED = [
    "adt_version", "adt_get_device_error", "adt_status_string", "adt_testing_set_wait_limit", "adt_testing_exp_diff",
    "adt_tree_attn_workspace_size", "adt_tree_attn", "adt_tree_attn_noalloc",
    "adt_tree_expand_workspace_size", "adt_tree_expand", "adt_tree_expand_cfg",
    "adt_tree_rerank_workspace_size", "adt_tree_rerank",
    "adt_tree_accept_workspace_size", "adt_tree_accept", "adt_tree_accept_cfg",
    "adt_kv_compact", "adt_kv_compact_inplace",
    "adt_ctrl_create", "adt_ctrl_destroy", "adt_ctrl_next", "adt_ctrl_update", "adt_ctrl_get",
    "adt_ctrl_state_size", "adt_ctrl_save", "adt_ctrl_load",
]


class AdtError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}")
        self.status = status


class CtrlParams(ctypes.Structure):
    _fields_ = [("beta", ctypes.c_double), ("l_d", ctypes.c_int32), ("l_k", ctypes.c_int32),
                ("d_lo", ctypes.c_int32), ("d_hi", ctypes.c_int32), ("k_lo", ctypes.c_int32),
                ("k_hi", ctypes.c_int32), ("init_mode", ctypes.c_int32), ("d0", ctypes.c_int32),
                ("k0", ctypes.c_int32), ("clamp_k_always", ctypes.c_int32), ("k_cap", ctypes.c_int32),
                ("fix_d", ctypes.c_int32), ("fix_k", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("flock_delta", ctypes.c_int32)]


_P, _I32, _I64, _F32, _SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
_SIGS = {
    "adt_version": ([], _I32),
    "adt_get_device_error": ([_P, ctypes.POINTER(ctypes.c_uint32)], _I32),
    "adt_status_string": ([_I32], ctypes.c_char_p),
    "adt_testing_set_wait_limit": ([ctypes.c_uint32], _I32),
    "adt_testing_exp_diff": ([_P, _P, _I32, _P, _P], _I32),
    "adt_tree_attn_workspace_size": ([_I32] * 5, _SZ),
    "adt_tree_attn": ([_P, _P, _P, _P, _I64, _I64, _P, _P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _F32,
                       _P, _P, _P, _SZ, _P], _I32),
    "adt_tree_attn_noalloc": ([_P, _P, _P, _P, _I64, _I64, _P, _P, _P, _P, _I32, _I32, _I32, _I32, _I32, _I32,
                               _F32, _P, _P, _P], _I32),
    "adt_tree_expand_workspace_size": ([_I32] * 3, _SZ),
    "adt_tree_expand": ([_P, _I64, _P, _P, _I32, _I32, _I32, _I32, _F32, _I32, _P, _P, _P, _P, _P, _P, _P,
                         _P, _SZ, _P], _I32),
    "adt_tree_expand_cfg": ([_P, _P, _I64, _F32, _P, _P, _I32, _I32, _I32, _I32, _F32, _I32, _P, _P, _P, _P, _P,
                             _P, _P, _P, _SZ, _P], _I32),
    "adt_tree_rerank_workspace_size": ([_I32], _SZ),
    "adt_tree_rerank": ([_P, _P, _P, _I32, _P, _I32, _P, _P, _P, _P, _P, _SZ, _P], _I32),
    "adt_tree_accept_workspace_size": ([_I32, _I32], _SZ),
    "adt_tree_accept": ([_P, _I64, _P, _I64, _P, _P, _P, _P, _I32, _I32, _I32, _P, _P, _I32, _F32, _P, _I32,
                         _P, _P, _P, _SZ, _P], _I32),
    "adt_tree_accept_cfg": ([_P, _P, _I64, _P, _P, _I64, _P, _F32, _P, _P, _P, _I32, _I32, _I32, _P, _P, _I32,
                             _F32, _P, _I32, _P, _P, _P, _SZ, _P], _I32),
    "adt_kv_compact": ([_P, _P, _P, _P, _P, _P, _P, _P, _I32, _P, _I32, _I32, _I32, _I32, _I32, _I64, _I64,
                        _I64, _I64, _P], _I32),
    "adt_kv_compact_inplace": ([_P, _P, _P, _P, _P, _P, _I32, _P, _I32, _I32, _I32, _I32, _I32, _I64, _I64, _I64,
                                _P], _I32),
    "adt_ctrl_create": ([ctypes.POINTER(CtrlParams), _I32, _I32, ctypes.POINTER(_P)], _I32),
    "adt_ctrl_destroy": ([_P], None),
    "adt_ctrl_state_size": ([_P], _SZ),
    "adt_ctrl_save": ([_P, _P, _SZ], _I32),
    "adt_ctrl_load": ([_P, _SZ, ctypes.POINTER(_P)], _I32),
    "adt_ctrl_next": ([_P, _I32, ctypes.POINTER(_I32), ctypes.POINTER(_I32)], _I32),
    "adt_ctrl_update": ([_P, _I32, _I32, ctypes.POINTER(_I32)], _I32),
    "adt_ctrl_get": ([_P, _I32, ctypes.POINTER(_I32), ctypes.POINTER(_I32)], _I32),
}

_LIB = None


def lib() -> ctypes.CDLL:
    """Loads libadt.so (once).  Raises if it has not been built."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2512_21857_gb300.build`")
        so = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGS.items():
            fn = getattr(so, name)
            fn.argtypes = args
            fn.restype = res
        _LIB = so
    return _LIB


def _check(status: int, where: str) -> None:
    if status != ADT_OK:
        raise AdtError(status, where)


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _expect(t, dtype, name):
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: expected a contiguous tensor")


def zeroed_workspace(nbytes: int, device=None) -> torch.Tensor:
    """A zero-filled byte buffer usable as a workspace (counters start at 0)."""
    return torch.zeros(max(int(nbytes), 16), dtype=torch.uint8, device=device or "cuda")


# ----------------------------------------------------------------------------- queries

def adt_version() -> int:
    return lib().adt_version()


def adt_get_device_error(stream=None) -> int:
    bits = ctypes.c_uint32(0)
    lib().adt_get_device_error(_stream(stream), ctypes.byref(bits))
    return int(bits.value)


def adt_testing_set_wait_limit(polls: int) -> None:
    """Testing hook: polls before adt_tree_attn's pipeline waits give up (0 = default)."""
    _check(lib().adt_testing_set_wait_limit(int(polls)), "adt_testing_set_wait_limit")


def adt_testing_exp_diff(a, b, out, stream=None) -> None:
    """Testing hook: out = e^(a - b) in the acceptance walk's double-float arithmetic."""
    _check(lib().adt_testing_exp_diff(_ptr(a), _ptr(b), int(a.numel()), _ptr(out), _stream(stream)),
           "adt_testing_exp_diff")


def adt_tree_attn_workspace_size(B, H, D, max_nodes, max_kv) -> int:
    return int(lib().adt_tree_attn_workspace_size(B, H, D, max_nodes, max_kv))


def adt_tree_expand_workspace_size(F, V, k_child) -> int:
    return int(lib().adt_tree_expand_workspace_size(F, V, k_child))


def adt_tree_rerank_workspace_size(C) -> int:
    return int(lib().adt_tree_rerank_workspace_size(C))


def adt_tree_accept_workspace_size(B, V) -> int:
    return int(lib().adt_tree_accept_workspace_size(B, V))


# ----------------------------------------------------------------------------- kernels

def adt_tree_attn(q, k_cache, v_cache, kv_len, k_tree, v_tree, parents, node_offsets, *, B, H, Hkv, D,
                  max_nodes, max_kv, softmax_scale, out, lse=None, workspace, cache_stride_b=None,
                  cache_stride_h=None, stream=None) -> None:
    """q, k_tree, v_tree, out: bf16 [Ntot, *, D]; caches bf16 with (b, g, pos, d) strides."""
    for t, n in ((q, "q"), (k_tree, "k_tree"), (v_tree, "v_tree"), (out, "out")):
        _expect(t, torch.bfloat16, n)
    for t, n in ((kv_len, "kv_len"), (parents, "parents"), (node_offsets, "node_offsets")):
        _expect(t, torch.int32, n)
    if k_cache.dtype != torch.bfloat16 or v_cache.dtype != torch.bfloat16:
        raise TypeError("caches must be bf16")
    if k_cache.stride() != v_cache.stride():
        raise ValueError("k_cache and v_cache must share strides")
    sb = k_cache.stride(0) if cache_stride_b is None else cache_stride_b
    sh = k_cache.stride(1) if cache_stride_h is None else cache_stride_h
    if lse is not None:
        _expect(lse, torch.float32, "lse")
    st = lib().adt_tree_attn(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(kv_len), sb, sh, _ptr(k_tree),
                             _ptr(v_tree), _ptr(parents), _ptr(node_offsets), B, H, Hkv, D, max_nodes, max_kv,
                             float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace),
                             workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "adt_tree_attn")


def adt_tree_expand(logits, frontier_score, frontier_id, *, F, V, k_child, k_keep, temperature=1.0,
                    child_id_base=0, child_token, child_logp, child_score, child_parent, keep_idx,
                    next_score=None, next_id=None, workspace, ld=None, stream=None) -> None:
    _expect(frontier_score, torch.float32, "frontier_score")
    if logits.dtype != torch.float32 or logits.stride(-1) != 1:
        raise TypeError("logits: fp32 rows with unit inner stride")
    if logits.dim() != 2:
        raise ValueError("logits: [F, V] rows")
    ld = logits.stride(0) if ld is None else ld
    st = lib().adt_tree_expand(_ptr(logits), ld, _ptr(frontier_score), _ptr(frontier_id), F, V, k_child, k_keep,
                               float(temperature), int(child_id_base), _ptr(child_token), _ptr(child_logp),
                               _ptr(child_score), _ptr(child_parent), _ptr(keep_idx), _ptr(next_score),
                               _ptr(next_id), _ptr(workspace), workspace.numel() * workspace.element_size(),
                               _stream(stream))
    _check(st, "adt_tree_expand")


def adt_tree_expand_cfg(logits_cond, logits_uncond, frontier_score, frontier_id, *, cfg_scale, F, V, k_child,
                        k_keep, temperature=1.0, child_id_base=0, child_token, child_logp, child_score,
                        child_parent, keep_idx, next_score=None, next_id=None, workspace, stream=None) -> None:
    """adt_tree_expand on uncond + cfg_scale * (cond - uncond); both [F, V] rows share one row stride."""
    _expect(frontier_score, torch.float32, "frontier_score")
    for t in (logits_cond, logits_uncond):
        if t.dtype != torch.float32 or t.dim() != 2 or t.stride(-1) != 1:
            raise TypeError("logits: fp32 [F, V] rows with unit inner stride")
    if logits_cond.stride(0) != logits_uncond.stride(0):
        raise ValueError("conditional and unconditional rows must share a row stride")
    st = lib().adt_tree_expand_cfg(_ptr(logits_cond), _ptr(logits_uncond), logits_cond.stride(0), float(cfg_scale),
                                   _ptr(frontier_score), _ptr(frontier_id), F, V, k_child, k_keep,
                                   float(temperature), int(child_id_base), _ptr(child_token), _ptr(child_logp),
                                   _ptr(child_score), _ptr(child_parent), _ptr(keep_idx), _ptr(next_score),
                                   _ptr(next_id), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                   _stream(stream))
    _check(st, "adt_tree_expand_cfg")


def adt_tree_rerank(cand_token, cand_score, cand_parent, C, root_token, n_nodes, *, tokens, parents,
                    cand_index=None, depth=None, workspace, stream=None) -> None:
    st = lib().adt_tree_rerank(_ptr(cand_token), _ptr(cand_score), _ptr(cand_parent), int(C), _ptr(root_token),
                               int(n_nodes), _ptr(tokens), _ptr(parents), _ptr(cand_index), _ptr(depth),
                               _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream))
    _check(st, "adt_tree_rerank")


def adt_tree_accept(target_logits, draft_logits, tokens, parents, node_offsets, *, B, V, max_nodes, mode,
                    u_accept=None, u_sample=None, temperature=1.0, path, max_path, accept_len, bonus_token,
                    draft_row=None, workspace=None, stream=None) -> None:
    ldt = target_logits.stride(0)
    ldd = draft_logits.stride(0) if draft_logits is not None else 0
    ws = workspace
    st = lib().adt_tree_accept(_ptr(target_logits), ldt, _ptr(draft_logits), ldd, _ptr(draft_row), _ptr(tokens),
                               _ptr(parents), _ptr(node_offsets), B, V, max_nodes, _ptr(u_accept),
                               _ptr(u_sample), int(mode), float(temperature), _ptr(path), int(max_path),
                               _ptr(accept_len), _ptr(bonus_token), _ptr(ws),
                               0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))
    _check(st, "adt_tree_accept")


def adt_tree_accept_cfg(target_cond, target_uncond, draft_cond, draft_uncond, tokens, parents, node_offsets, *,
                        cfg_scale, B, V, max_nodes, mode, u_accept=None, u_sample=None, temperature=1.0, path,
                        max_path, accept_len, bonus_token, draft_row=None, stream=None) -> None:
    """adt_tree_accept with every target / draft row formed as uncond + cfg_scale * (cond - uncond)."""
    if target_cond.stride(0) != target_uncond.stride(0):
        raise ValueError("conditional and unconditional target rows must share a row stride")
    ldd = draft_cond.stride(0) if draft_cond is not None else 0
    if draft_cond is not None and draft_uncond is not None and draft_uncond.stride(0) != ldd:
        raise ValueError("conditional and unconditional draft rows must share a row stride")
    st = lib().adt_tree_accept_cfg(_ptr(target_cond), _ptr(target_uncond), target_cond.stride(0), _ptr(draft_cond),
                                   _ptr(draft_uncond), ldd, _ptr(draft_row), float(cfg_scale), _ptr(tokens),
                                   _ptr(parents), _ptr(node_offsets), B, V, max_nodes, _ptr(u_accept),
                                   _ptr(u_sample), int(mode), float(temperature), _ptr(path), int(max_path),
                                   _ptr(accept_len), _ptr(bonus_token), None, 0, _stream(stream))
    _check(st, "adt_tree_accept_cfg")


def adt_kv_compact(k_cache, v_cache, kv_len, kv_len_out, k_tree, v_tree, node_offsets, path, max_path,
                   accept_len, *, B, Hkv, D, num_layers, max_kv, cache_layer_stride, cache_stride_b,
                   cache_stride_h, tree_layer_stride, stream=None) -> None:
    st = lib().adt_kv_compact(_ptr(k_cache), _ptr(v_cache), _ptr(kv_len), _ptr(kv_len_out), _ptr(k_tree),
                              _ptr(v_tree), _ptr(node_offsets), _ptr(path), int(max_path), _ptr(accept_len),
                              B, Hkv, D, num_layers, max_kv, cache_layer_stride, cache_stride_b, cache_stride_h,
                              tree_layer_stride, _stream(stream))
    _check(st, "adt_kv_compact")


def adt_kv_compact_inplace(k_cache, v_cache, kv_len, kv_len_out, node_offsets, path, max_path, accept_len, *, B,
                           Hkv, D, num_layers, max_kv, cache_layer_stride, cache_stride_b, cache_stride_h,
                           stream=None) -> None:
    st = lib().adt_kv_compact_inplace(_ptr(k_cache), _ptr(v_cache), _ptr(kv_len), _ptr(kv_len_out),
                                      _ptr(node_offsets), _ptr(path), int(max_path), _ptr(accept_len), B, Hkv, D,
                                      num_layers, max_kv, cache_layer_stride, cache_stride_b, cache_stride_h,
                                      _stream(stream))
    _check(st, "adt_kv_compact_inplace")


# ----------------------------------------------------------------------------- controller

class Controller:
    """Host depth / width controller (adt_ctrl_*); one per image."""

    def __init__(self, grid_h, grid_w, *, beta=1.0, l_d=1, l_k=3, d_lo=1, d_hi=9, k_lo=4, k_hi=13,
                 init_mode=INIT_HORIZONTAL, d0=5, k0=10, clamp_k_always=True, k_cap=64, fix_d=0, fix_k=0,
                 seed=0, flock_delta=2):
        self._p = CtrlParams(beta, l_d, l_k, d_lo, d_hi, k_lo, k_hi, init_mode, d0, k0, int(bool(clamp_k_always)),
                             k_cap, fix_d, fix_k, seed, flock_delta)
        h = ctypes.c_void_p()
        _check(lib().adt_ctrl_create(ctypes.byref(self._p), grid_h, grid_w, ctypes.byref(h)), "adt_ctrl_create")
        self._h = h

    def next(self, pos):
        d, k = ctypes.c_int32(), ctypes.c_int32()
        _check(lib().adt_ctrl_next(self._h, pos, ctypes.byref(d), ctypes.byref(k)), "adt_ctrl_next")
        return d.value, k.value

    def update(self, pos, accept_len):
        nxt = ctypes.c_int32()
        _check(lib().adt_ctrl_update(self._h, pos, accept_len, ctypes.byref(nxt)), "adt_ctrl_update")
        return nxt.value

    def get(self, pos):
        d, k = ctypes.c_int32(), ctypes.c_int32()
        _check(lib().adt_ctrl_get(self._h, pos, ctypes.byref(d), ctypes.byref(k)), "adt_ctrl_get")
        return d.value, k.value

    def save(self) -> bytes:
        """The controller's state as bytes (checkpoint)."""
        n = int(lib().adt_ctrl_state_size(self._h))
        buf = ctypes.create_string_buffer(n)
        _check(lib().adt_ctrl_save(self._h, buf, n), "adt_ctrl_save")
        return buf.raw

    @classmethod
    def load(cls, state: bytes) -> "Controller":
        """A controller resumed from save()'s bytes."""
        h = ctypes.c_void_p()
        _check(lib().adt_ctrl_load(state, len(state), ctypes.byref(h)), "adt_ctrl_load")
        obj = cls.__new__(cls)
        obj._h = h
        return obj

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and _LIB is not None:
            _LIB.adt_ctrl_destroy(h)
            self._h = None
