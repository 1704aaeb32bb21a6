"""adt_tree_attn_noalloc, the tree-attention entry point for callers that
cannot allocate device memory themselves (a plugin whose host engine owns
all device allocations, or a latency-critical thread that must not call
cudaMalloc).  Its scratch is a fixed per-device static array; these tests
call it through the C ABI and compare it with adt_tree_attn, which takes a
caller-provided workspace.

Kept in a file collected last so that, if it fails, a run that stops at the
first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_cases import LSE_ATOL, AttnCase, assert_attention_close, ensure_built, i32
from paper_2512_21857_gb300 import binding as B

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def call_noalloc(case, out, lse, max_nodes, max_kv):
    dev = "cuda"
    kc, vc = case.kc.to(dev), case.vc.to(dev)
    q, kt, vt = case.q.to(dev), case.kt.to(dev), case.vt.to(dev)
    kv, par, offs = i32(case.kv_lens), i32(case.tb.parents), i32(case.tb.node_offsets)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    st = B.lib().adt_tree_attn_noalloc(_ptr(q), _ptr(kc), _ptr(vc), _ptr(kv), kc.stride(0), kc.stride(1), _ptr(kt),
                                       _ptr(vt), _ptr(par), _ptr(offs), case.B, case.H, case.Hkv, case.D, max_nodes,
                                       max_kv, float(case.scale), _ptr(out), _ptr(lse), stream)
    torch.cuda.synchronize()
    return st


@pytest.mark.parametrize("sizes,kv,H,Hkv,D", [
    ([64], [2400], 32, 32, 128),          # 7B-shape layer (fewer splits fit in the scratch)
    ([26, 5, 64], [512, 0, 700], 8, 4, 64),  # ragged batch, grouped heads
])
def test_noalloc_matches_workspace_entry_point_on_two_calls(sizes, kv, H, Hkv, D):
    case = AttnCase(sizes, kv, H, Hkv, D, seed=600 + sum(sizes))
    max_nodes, max_kv = max(sizes), max(kv)
    want, want_lse, _ = case.run_gpu(max_nodes=max_nodes, max_kv=max_kv)
    for _ in range(2):  # the second call finds the first call's contents in the shared scratch
        out = torch.full((case.ntot, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((case.ntot, H), float("nan"), dtype=torch.float32, device="cuda")
        assert call_noalloc(case, out, lse, max_nodes, max_kv) == B.ADT_OK
        got = out.float().cpu().numpy().astype(np.float64)
        assert_attention_close(got, want)
        assert np.abs(lse.cpu().numpy() - want_lse).max() < LSE_ATOL
    assert B.adt_get_device_error() == 0


def test_noalloc_rejects_a_shape_beyond_its_scratch():
    # 64 trees x 64 heads x 64 rows x (128 + 2) x 4 bytes of partials > 8 MiB even unsplit
    t = torch.zeros(64, dtype=torch.int32, device="cuda")
    p = _ptr(t)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    sh, sb = 100 * 128, 64 * 100 * 128  # strides of a [64][64][100][128] cache
    st = B.lib().adt_tree_attn_noalloc(p, p, p, p, sb, sh, p, p, p, p, 64, 64, 64, 128, 64, 100, 0.1, p, None, stream)
    assert st == 5  # ADT_ERR_WORKSPACE, nothing launched
