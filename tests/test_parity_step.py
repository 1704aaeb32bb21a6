"""A whole verify step (draft growth, rerank, tree attention per layer,
acceptance walk, KV commit) through TreeVerifyStep, against the oracle's
composition of the same steps, repeated with the same buffers (the
benchmark's replay pattern) and captured in a CUDA graph."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_attention_close, ensure_built
from oracle.step import draft_tree
from paper_2512_21857_gb300 import binding as B
from paper_2512_21857_gb300 import synth
from paper_2512_21857_gb300.verify_step import StepShape, TreeVerifyStep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()


def _setup(layers, H, D, V, L, depth, width, nmax, mode, seed, plant):
    shape = StepShape(layers=layers, H=H, Hkv=H, D=D, V=V, kv_len=[L], depth=[depth], width=[width],
                      max_nodes=nmax, mode=mode)
    step = TreeVerifyStep(shape, keep_layer_outputs=True)
    inp = synth.step_inputs(layers, H, H, D, V, [L], [depth], [width], step.n, step.lmax, seed)
    tree = draft_tree(inp["draft_rows"][0], width, depth, int(inp["root_token"][0]), nmax)
    if plant:
        deepest = int(np.argmax(tree["depth"]))
        synth.plant_path(inp["target"], tree["parents"], tree["tokens"],
                         oracle.ancestor_path(tree["parents"], deepest)[:plant])
    step.load_inputs(inp)
    return step, inp, tree


def _check(step, inp, tree, mode, layers):
    n = len(tree["tokens"])
    assert np.array_equal(step.tokens.cpu().numpy(), tree["tokens"])
    assert np.array_equal(step.parents.cpu().numpy(), tree["parents"])
    assert np.array_equal(step.cand_index.cpu().numpy(), tree["cand_index"])
    offs = [0, n]
    for layer in layers:
        ref, _ = oracle.tree_attention(inp["q"][layer].double().numpy(), inp["k_cache"][layer].double().numpy(),
                                       inp["v_cache"][layer].double().numpy(), step.shape.kv_len,
                                       inp["k_tree"][layer].double().numpy(), inp["v_tree"][layer].double().numpy(),
                                       tree["parents"], offs, step.shape.D ** -0.5)
        assert_attention_close(step.attn_out[layer].double().cpu().numpy(), ref)
    acc = oracle.tree_accept(inp["target"], None, tree["tokens"], tree["parents"], offs, mode, inp["u_accept"],
                             inp["u_sample"])
    assert acc["accept_margin"] > 1e-5 and acc["sample_margin"] > 1e-7
    a = int(acc["accept_len"][0])
    assert int(step.accept_len[0]) == a
    assert step.path[0, :a + 1].cpu().tolist() == acc["path"][0]
    assert int(step.bonus[0]) == int(acc["bonus"][0])
    kc, vc, kl = oracle.kv_compact(inp["k_cache"].view(torch.int16).numpy(), inp["v_cache"].view(torch.int16).numpy(),
                                   step.shape.kv_len, inp["k_tree"].view(torch.int16).numpy(),
                                   inp["v_tree"].view(torch.int16).numpy(), offs, acc["path"])
    assert np.array_equal(step.k_cache.cpu().view(torch.int16).numpy(), kc)
    assert np.array_equal(step.v_cache.cpu().view(torch.int16).numpy(), vc)
    assert int(step.kv_len_out[0]) == int(kl[0])
    return a


@pytest.mark.parametrize("mode,plant", [(B.ACCEPT_GREEDY, 4), (B.ACCEPT_SPEC_DET, 0)])
def test_step_7b_shape_two_layers_repeated_and_graphed(mode, plant):
    step, inp, tree = _setup(2, 32, 128, 65536, 2400, 6, 8, 64, mode, seed=99 + mode, plant=plant)
    B.adt_get_device_error()
    for _ in range(3):  # eager, same buffers: the committed cache rows are rewritten with the same bytes
        step.launch()
        torch.cuda.synchronize()
        a = _check(step, inp, tree, mode, layers=[0, 1])
    if mode == B.ACCEPT_GREEDY:
        assert a >= 3
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            step.launch(s)
        for _ in range(3):
            g.replay()
    torch.cuda.synchronize()
    _check(step, inp, tree, mode, layers=[0, 1])
    assert B.adt_get_device_error() == 0


def test_step_llamagen_shape():
    step, inp, tree = _setup(2, 20, 64, 16384, 696, 5, 10, 64, B.ACCEPT_GREEDY, seed=5, plant=3)
    step.launch()
    torch.cuda.synchronize()
    assert _check(step, inp, tree, B.ACCEPT_GREEDY, layers=[0, 1]) >= 2


@pytest.mark.parametrize("mode,plant", [(B.ACCEPT_GREEDY, 3), (B.ACCEPT_SPEC_DET, 0)])
def test_step_llamagen_width_39_tree_of_256(mode, plant):
    """LlamaGen-class width bound (k = 39, Sec. 5.1): 39 + 4 * 39^2
    candidates, the 255 best kept, so attention runs four query tiles."""
    step, inp, tree = _setup(2, 20, 64, 16384, 696, 5, 39, 256, mode, seed=12 + mode, plant=plant)
    assert len(tree["tokens"]) == 256
    step.launch()
    torch.cuda.synchronize()
    a = _check(step, inp, tree, mode, layers=[0, 1])
    if mode == B.ACCEPT_GREEDY:
        assert a >= 2


def test_ragged_batch_graph_replay_equals_eager():
    """Eight images of different depth, width and prefix length: each image's
    draft chain runs on its own stream, forked from the step's stream and
    joined before attention.  The grown trees match the oracle; a captured
    graph of the step, replayed over zeroed outputs, reproduces the eager
    step bit for bit (trees, attention of every layer, acceptance, cache)."""
    kv = [751, 1596, 1444, 640, 1427, 1245, 2352, 1248]
    depth, width = [4, 7, 8, 7, 6, 6, 7, 6], [6, 8, 4, 2, 2, 1, 6, 4]
    layers, H, D, V = 2, 8, 128, 16384
    shape = StepShape(layers=layers, H=H, Hkv=H, D=D, V=V, kv_len=kv, depth=depth, width=width, max_nodes=64)
    step = TreeVerifyStep(shape, keep_layer_outputs=True)
    inp = synth.step_inputs(layers, H, H, D, V, kv, depth, width, step.n, step.lmax, 31)
    step.load_inputs(inp)
    B.adt_get_device_error()
    step.launch()
    torch.cuda.synchronize()
    assert B.adt_get_device_error() == 0
    trees = [draft_tree(inp["draft_rows"][b], width[b], depth[b], int(inp["root_token"][b]), step.n[b])
             for b in range(len(kv))]
    assert np.array_equal(step.tokens.cpu().numpy(), np.concatenate([t["tokens"] for t in trees]))
    assert np.array_equal(step.parents.cpu().numpy(), np.concatenate([t["parents"] for t in trees]))
    outs = ("tokens", "parents", "cand_index", "attn_out", "path", "accept_len", "bonus", "kv_len_out")
    eager = {name: getattr(step, name).clone() for name in outs}
    eager_k, eager_v = step.k_cache.clone(), step.v_cache.clone()

    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            step.launch(s)
    torch.cuda.synchronize()
    for name in outs:
        getattr(step, name).zero_()
    with torch.cuda.stream(s):
        g.replay()
    torch.cuda.synchronize()
    assert B.adt_get_device_error() == 0
    for name in outs:
        assert torch.equal(getattr(step, name), eager[name]), name
    assert torch.equal(step.k_cache.view(torch.int16), eager_k.view(torch.int16))
    assert torch.equal(step.v_cache.view(torch.int16), eager_v.view(torch.int16))
