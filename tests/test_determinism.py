"""Replays of the benchmark's whole verify step (32 layers at the 7B shape:
32 heads x 128, KV 2400, a 64-node tree grown from a 65,536-word draft,
greedy walk, KV commit) are bit-identical.  Every step of the path hands
data between roles and CTAs (TMA copies into rings, tensor-core products,
cluster merges through distributed shared memory, completion tickets); a
consumer that ran ahead of its producer would show as outputs that differ
from one replay to the next.  The outputs compared after every replay:
the tree (tokens, parents), every layer's attention, the path, its length,
the bonus token, the new cache length and both caches."""
import pytest
import torch

from gpu_cases import ensure_built
from paper_2512_21857_gb300 import binding as B
from paper_2512_21857_gb300.verify_step import StepShape, TreeVerifyStep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def _fill(step, seed):
    """Seeded inputs drawn on the device: bf16 ~ N(0, 1) caches and
    projections, fp32 ~ N(0, 3^2) logits, 24-bit uniforms, a random root."""
    g = torch.Generator(device=step.device)
    g.manual_seed(seed)

    def normal_(t, std=1.0):
        t.copy_((torch.randn(t.shape, generator=g, device=step.device) * std).to(t.dtype))

    for name in ("k_cache", "v_cache", "q", "k_tree", "v_tree"):
        normal_(getattr(step, name))
    for rows in step.draft_rows:
        normal_(rows, 3.0)
    normal_(step.target, 3.0)
    for t in (step.u_accept, step.u_sample):
        t.copy_(torch.randint(0, 1 << 24, t.shape, generator=g, device=step.device).float() * 2.0 ** -24)
    step.root_token.copy_(torch.randint(0, step.shape.V, step.root_token.shape, generator=g, device=step.device))


@pytest.mark.parametrize("plant", [0, 3])
def test_7b_step_replays_are_bit_identical(plant):
    shape = StepShape(layers=32, H=32, Hkv=32, D=128, V=65536, kv_len=[2400], depth=[6], width=[8], max_nodes=64,
                      mode=B.ACCEPT_GREEDY)
    step = TreeVerifyStep(shape, keep_layer_outputs=True)
    _fill(step, 11 + plant)
    s = torch.cuda.Stream()
    B.adt_get_device_error()
    with torch.cuda.stream(s):
        step.launch(s)
    torch.cuda.synchronize()
    if plant:
        # Raise the target rows along the root-first path to the deepest
        # node, so that the greedy walk accepts `plant` nodes (the tree is
        # the same every replay: the draft inputs do not change).
        parents, tokens = step.parents.cpu().tolist(), step.tokens.cpu().tolist()
        deepest = max(range(len(parents)), key=lambda i: (step.node_depth[i].item(), -i))
        path = [deepest]
        while parents[path[-1]] >= 0:
            path.append(parents[path[-1]])
        path = path[::-1][:plant + 1]
        assert len(path) == plant + 1
        for v, c in zip(path[:-1], path[1:]):
            row = step.target[v]
            row[tokens[c]] = row.max() + 50.0
    outs = ("tokens", "parents", "attn_out", "path", "accept_len", "bonus", "kv_len_out", "k_cache", "v_cache")
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            step.launch(s)
        g.replay()
    torch.cuda.synchronize()
    assert B.adt_get_device_error() == 0
    assert int(step.accept_len[0]) == plant
    first = {name: getattr(step, name).clone() for name in outs}
    for rep in range(20):
        with torch.cuda.stream(s):
            g.replay()
        torch.cuda.synchronize()
        for name in outs:
            assert torch.equal(getattr(step, name), first[name]), f"replay {rep}: {name} differs"
    assert B.adt_get_device_error() == 0


def test_ragged_batch_step_replays_are_bit_identical():
    """The ragged eight-image batch at the 7B head shape (prefixes 640-2352,
    per-image depth and width, each image's draft chain on its own stream,
    one split per (tree, head) in longest-prefix-first slot order), four
    layers: 21 graph replays give bit-identical outputs."""
    kv = [751, 1596, 1444, 640, 1427, 1245, 2352, 1248]
    shape = StepShape(layers=4, H=32, Hkv=32, D=128, V=65536, kv_len=kv, depth=[4, 7, 8, 7, 6, 6, 7, 6],
                      width=[6, 8, 4, 2, 2, 1, 6, 4], max_nodes=64, mode=B.ACCEPT_GREEDY)
    step = TreeVerifyStep(shape, keep_layer_outputs=True)
    _fill(step, 23)
    s = torch.cuda.Stream()
    B.adt_get_device_error()
    with torch.cuda.stream(s):
        step.launch(s)
    torch.cuda.synchronize()
    outs = ("tokens", "parents", "attn_out", "path", "accept_len", "bonus", "kv_len_out", "k_cache", "v_cache")
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            step.launch(s)
        g.replay()
    torch.cuda.synchronize()
    assert B.adt_get_device_error() == 0
    first = {name: getattr(step, name).clone() for name in outs}
    for rep in range(20):
        with torch.cuda.stream(s):
            g.replay()
        torch.cuda.synchronize()
        for name in outs:
            assert torch.equal(getattr(step, name), first[name]), f"replay {rep}: {name} differs"
    assert B.adt_get_device_error() == 0
