"""GPU tree attention vs the oracle, element by element (tolerance: 1e-2
plus half a bf16 ulp of the reference elementwise, and 2e-2 normwise, on
bf16 inputs), over the workload shapes of the 7B-class and LlamaGen-class
models and the edge cases."""
import numpy as np
import pytest

from gpu_cases import LSE_ATOL, AttnCase, assert_attention_close, ensure_built

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


CASES = [
    # sizes, kv_lens, H, Hkv, D
    ([26], [512], 8, 8, 64),              # single verify step, batch 1, 26-node tree
    ([64], [696], 20, 20, 64),            # LlamaGen-XL-shaped layer, 64 nodes, 120 + 576 prefix
    ([16], [120], 20, 20, 64),            # LlamaGen-XL, text prefix only
    ([33, 7, 1, 64], [63, 64, 65, 0], 4, 4, 128),  # ragged batch, tile edges, empty prefix
    ([12, 5], [700, 1], 8, 2, 128),       # grouped kv heads
    ([1], [300], 4, 4, 64),               # single node = ordinary decode attention
    ([40], [2400], 2, 2, 128),            # few heads, long prefix: 20 splits merge through the workspace
    ([64, 9], [4000, 3000], 2, 1, 64),    # the same with grouped heads, two trees
]


@pytest.mark.parametrize("sizes,kv,H,Hkv,D", CASES)
def test_attention_matches_oracle(sizes, kv, H, Hkv, D):
    case = AttnCase(sizes, kv, H, Hkv, D, seed=101 + sum(sizes))
    got, lse, _ = case.run_gpu()
    ref, ref_lse = case.run_oracle()
    assert_attention_close(got, ref)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


# Trees of more than 64 nodes (width bound 39 for LlamaGen-class drafts):
# 64-row query tiles, each seeing the tree units up to its own.
LARGE_CASES = [
    # sizes, kv_lens, H, Hkv, D
    ([256], [600], 8, 8, 128),                  # four full query tiles
    ([100], [2400], 16, 16, 128),               # second tile partial, long prefix
    ([65], [0], 4, 4, 64),                      # one node in the second tile, empty prefix
    ([200, 7, 129], [700, 64, 1], 8, 2, 128),   # ragged batch across tile counts, grouped kv heads
    ([192], [696], 20, 20, 64),                 # LlamaGen-XL-shaped layer, three tiles
]


@pytest.mark.parametrize("sizes,kv,H,Hkv,D", LARGE_CASES)
def test_large_tree_matches_oracle(sizes, kv, H, Hkv, D):
    case = AttnCase(sizes, kv, H, Hkv, D, seed=301 + sum(sizes), max_depth=10, max_children=39)
    got, lse, _ = case.run_gpu(max_nodes=max(sizes))
    ref, ref_lse = case.run_oracle()
    assert_attention_close(got, ref)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


@pytest.mark.parametrize("chain", [True, False])
def test_256_node_extremes(chain):
    """A 256-node chain (every mask word full below the diagonal) and a
    256-node star (each node sees the root and itself)."""
    case = AttnCase([256], [130], 4, 4, 128, seed=9, chain=chain, max_depth=1, max_children=255)
    got, _, _ = case.run_gpu(max_nodes=256)
    ref, _ = case.run_oracle()
    assert_attention_close(got, ref)


def test_chain_tree_matches_oracle():
    case = AttnCase([64], [257], 4, 4, 128, seed=7, chain=True)
    got, _, _ = case.run_gpu()
    ref, _ = case.run_oracle()
    assert_attention_close(got, ref)


def test_7b_shape_one_layer_full_size():
    """KV 2400, 32 heads x 128, 64-node tree: the launch configuration the
    benchmark times (one layer; every layer is the same call)."""
    case = AttnCase([64], [2400], 32, 32, 128, seed=2024, lmax=2400 + 64)
    got, lse, _ = case.run_gpu(max_kv=2400 + 64)
    ref, ref_lse = case.run_oracle()
    assert_attention_close(got, ref)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


@pytest.mark.parametrize("sizes,kv,H,D", [
    ([64], [16384], 8, 128),        # 19 splits of 7 chunks each, merged through the workspace
    ([64, 40], [8192, 7000], 32, 128),  # 2 splits per head: 33-chunk pipelines, many barrier phases
])
def test_long_prefixes(sizes, kv, H, D):
    case = AttnCase(sizes, kv, H, H, D, seed=17 + len(sizes), lmax=max(kv) + 8)
    got, lse, _ = case.run_gpu(max_nodes=64, max_kv=max(kv) + 8)
    ref, ref_lse = case.run_oracle()
    assert_attention_close(got, ref)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


@pytest.mark.parametrize("nb", [2, 32, 33])
def test_tree_order_by_prefix_length(nb):
    """Launches of 2-32 trees hand their slots to the trees by decreasing
    prefix length (ties to the lower index); 33 trees keep tree order.
    Prefix lengths repeat, so ties occur; every tree's output is checked."""
    g = np.random.default_rng(nb)
    kv = g.choice([0, 1, 63, 64, 65, 200, 200, 333], size=nb).tolist()
    sizes = g.integers(1, 21, size=nb).tolist()
    case = AttnCase(sizes, kv, 2, 2, 64, seed=700 + nb, lmax=max(kv) + 8)
    got, lse, _ = case.run_gpu(max_nodes=max(sizes), max_kv=max(kv) + 8)
    ref, ref_lse = case.run_oracle()
    assert_attention_close(got, ref)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


def test_batch_of_eight_ragged_prefixes():
    g = np.random.default_rng(5)
    kv = g.integers(600, 2401, size=8).tolist()
    sizes = g.integers(8, 65, size=8).tolist()
    case = AttnCase(sizes, kv, 8, 8, 128, seed=77, max_depth=10, max_children=8, lmax=2400 + 8)
    got, _, _ = case.run_gpu(max_nodes=64, max_kv=2400)
    ref, _ = case.run_oracle()
    assert_attention_close(got, ref)


def test_ragged_batch_bench_launch():
    """The launch the ragged 8-image benchmark times, at its exact shape: 8
    trees (the sizes its depths and widths give), 32 heads x 128, its prefix
    lengths.  256 (tree, head) pairs take one split each (256 CTAs on the
    GPU's SMs, no merge) and the launch slots go to the trees longest prefix
    first."""
    kv = [751, 1596, 1444, 640, 1427, 1245, 2352, 1248]
    sizes = [64, 64, 64, 27, 23, 7, 64, 64]
    case = AttnCase(sizes, kv, 32, 32, 128, seed=88, max_depth=10, max_children=8, lmax=2352 + 64)
    got, lse, _ = case.run_gpu(max_nodes=64, max_kv=2352 + 64)
    ref, ref_lse = case.run_oracle()
    assert_attention_close(got, ref)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


def test_workspace_reuse_and_repeat_is_deterministic():
    case = AttnCase([26], [512], 8, 8, 64, seed=3)
    a, la, ws = case.run_gpu()
    b, lb, _ = case.run_gpu()
    assert np.array_equal(a, b) and np.array_equal(la, lb)
    # the ticket counters (start of the workspace) are back at zero after every call
    assert int(ws[:65536 * 4].cpu().sum()) == 0


def test_shared_workspace_across_shapes():
    """One workspace, sized for the largest call, serves calls of different
    shapes in any order."""
    from paper_2512_21857_gb300 import binding as B
    big = AttnCase([64, 30], [2400, 900], 8, 8, 128, seed=41)
    small = AttnCase([9], [100], 2, 2, 128, seed=42)
    ws = B.zeroed_workspace(B.adt_tree_attn_workspace_size(2, 8, 128, 64, 2400))
    ref_big, _ = big.run_oracle()
    ref_small, _ = small.run_oracle()
    for _ in range(2):
        for case, ref in ((small, ref_small), (big, ref_big)):
            got, _, _ = case.run_gpu(ws=ws)
            assert_attention_close(got, ref)


def test_bad_tree_sets_device_error():
    from paper_2512_21857_gb300 import binding as B
    case = AttnCase([5], [10], 2, 2, 64, seed=1)
    case.tb.parents[3] = 4  # parent after child
    B.adt_get_device_error()
    case.run_gpu()
    bits = B.adt_get_device_error()
    assert bits & B.DEVERR_BAD_TREE
    assert B.adt_get_device_error() == 0


@pytest.mark.parametrize("scale", [1e5, 1e-6])
def test_value_range_extremes(scale):
    """V around 4 * scale: the splits' partial rows (averages of V rows) lie
    far outside the fp16 range the cluster merge moves them in (above 65504,
    or in its subnormals), so the kernel's power-of-two scaling of each row
    decides the result.  Outputs scale with V, so they are compared after
    dividing by `scale`.  The 7B launch shape: 4 splits per head, merged in
    the cluster."""
    import torch
    case = AttnCase([64], [2400], 32, 32, 128, seed=31, lmax=2400 + 64)
    case.vc = ((case.vc.float() + 4.0) * scale).to(torch.bfloat16)
    case.vt = ((case.vt.float() + 4.0) * scale).to(torch.bfloat16)
    got, lse, _ = case.run_gpu(max_kv=2400 + 64)
    ref, ref_lse = case.run_oracle()
    assert np.isfinite(got).all()
    assert_attention_close(got / scale, ref / scale)
    assert np.abs(lse - ref_lse).max() < LSE_ATOL


def test_zero_and_mixed_magnitude_values():
    """V all zero (every partial row's largest magnitude is 0: outputs
    exactly 0), then V rows whose magnitudes differ by 2^40 between heads and
    between halves of the prefix, so that the splits of one head stage rows
    at very different scales: the cluster merge must combine them by their
    weights alone.  The 7B launch shape (4 splits per head)."""
    import torch
    case = AttnCase([64], [2400], 32, 32, 128, seed=32, lmax=2400 + 64)
    vc, vt = case.vc.clone(), case.vt.clone()
    case.vc = torch.zeros_like(vc)
    case.vt = torch.zeros_like(vt)
    got, _, _ = case.run_gpu(max_kv=2400 + 64)
    assert not got.any()
    scale_h = (2.0 ** (torch.arange(32) % 5 * 10 - 20)).view(1, 32, 1, 1)   # per head: 2^-20 .. 2^20
    scale_pos = torch.where(torch.arange(2400 + 64) < 1200, 1.0, 2.0 ** -20).view(1, 1, -1, 1)
    case.vc = (vc.float() * scale_h * scale_pos).to(torch.bfloat16)
    case.vt = (vt.float() * scale_h.view(1, 32, 1)).to(torch.bfloat16)
    got, _, _ = case.run_gpu(max_kv=2400 + 64)
    ref, _ = case.run_oracle()
    s = scale_h.view(32, 1).numpy().astype(np.float64)
    for h in range(32):
        assert_attention_close(got[:, h] / s[h], ref[:, h] / s[h])
