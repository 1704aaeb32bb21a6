"""adt_tree_attn_noalloc, the tree-attention entry point for callers that
cannot allocate device memory themselves (a plugin whose host engine owns
all device allocations, or a latency-critical thread that must not call
cudaMalloc).  Its scratch is a fixed per-device static array; these tests
call it through the C ABI and compare it with adt_tree_attn, which takes a
caller-provided workspace, and with the oracle.

Kept in a file collected last so that, if it fails, a run that stops at the
first failure has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_cases import LSE_ATOL, AttnCase, assert_attention_close, ensure_built
from gpu_cases import i32
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


C4_KV = [751, 1596, 1444, 640, 1427, 1245, 2352, 1248]
C4_SIZES = [64, 64, 64, 27, 23, 7, 64, 64]  # the ragged batch bench step's trees


@pytest.mark.parametrize("sizes,kv,H,Hkv,D", [
    ([64], [2400], 32, 32, 128),          # 7B-shape layer: 4 splits merge on chip, no scratch
    ([26, 5, 64], [512, 0, 700], 8, 4, 64),  # ragged batch, grouped heads
    ([40], [2400], 2, 2, 128),            # 20 splits merge through the static array
    ([100], [2400], 2, 2, 128),           # two query tiles, the same merge through the array
    ([64], [9728], 2, 2, 128),            # 76 splits' partials exceed the array: cut to 63 splits
    (C4_SIZES, C4_KV, 32, 32, 128),       # 8 trees x 32 heads: one split, no scratch
])
def test_noalloc_matches_workspace_entry_point_on_two_calls(sizes, kv, H, Hkv, D):
    case = AttnCase(sizes, kv, H, Hkv, D, seed=600 + sum(sizes), max_depth=10, max_children=8)
    max_nodes, max_kv = max(sizes), max(kv)
    want, want_lse, _ = case.run_gpu(max_nodes=max_nodes, max_kv=max_kv)
    ref, ref_lse = case.run_oracle()
    for _ in range(2):  # the second call finds the first call's contents in the shared scratch
        out = torch.full((case.ntot, H, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((case.ntot, H), float("nan"), dtype=torch.float32, device="cuda")
        assert call_noalloc(case, out, lse, max_nodes, max_kv) == B.ADT_OK
        got = out.float().cpu().numpy().astype(np.float64)
        got_lse = lse.cpu().numpy()
        assert_attention_close(got, want)
        assert np.abs(got_lse - want_lse).max() < LSE_ATOL
        assert_attention_close(got, ref)
        assert np.abs(got_lse - ref_lse).max() < LSE_ATOL
    assert B.adt_get_device_error() == 0


def test_noalloc_rejects_a_shape_beyond_its_limits():
    # 1024 trees x 65 heads: more (tree, head) pairs than the call handles
    t = torch.zeros(64, dtype=torch.int32, device="cuda")
    p = _ptr(t)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    sh, sb = 100 * 128, 65 * 100 * 128  # strides of a [1024][65][100][128] cache
    st = B.lib().adt_tree_attn_noalloc(p, p, p, p, sb, sh, p, p, p, p, 1024, 65, 65, 128, 64, 100, 0.1, p, None,
                                       stream)
    assert st == 1  # ADT_ERR_INVALID_ARG, nothing launched
    torch.cuda.synchronize()
    assert B.adt_get_device_error() == 0
