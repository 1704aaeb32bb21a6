"""The ragged, controller-driven batch (the adjacency-adaptive sweep): 8
images with prefix lengths of 600-2400 keys at head_dim 128, three verify
steps in a row, each image's tree depth and width chosen every step by the
depth / width controller (horizontal-adjacency init, Eq. 2 bisection, the
clamps of Sec. 4.2) from a seeded acceptance-rate map.  Each step is checked
against the oracle on the same inputs: the grown trees, tree attention of
every image and head, the acceptance walk, the KV commit; the C controller
against the oracle controller.  The next step starts from the committed
cache and the new prefix lengths, as a decode loop would."""
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

GRID = (48, 48)
# d in [2, 10], k in [1, 8], beta = 1, l_d = 1, l_k = 3
PARAMS = dict(beta=1.0, l_d=1, l_k=3, d_lo=2, d_hi=10, k_lo=1, k_hi=8, d0=5, k0=4)


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy()


@pytest.mark.parametrize("init_mode", [B.INIT_HORIZONTAL, B.INIT_TOKENFLOCK])
def test_ragged_batch_three_controller_steps(init_mode):
    ensure_built()
    nb, layers, H, D, V, steps, seed = 8, 2, 8, 128, 16384, 3, 404
    g = synth.rng(seed, "batch_controller")
    kv = [int(x) for x in g.integers(600, 2401, size=nb)]
    pos = [int(x) for x in g.integers(0, GRID[0] * GRID[1] - 100, size=nb)]
    amap = synth.acceptance_map(*GRID, seed).ravel()
    lmax = 2400 + steps * 11 + 64
    ctl_c = [B.Controller(*GRID, **PARAMS, init_mode=init_mode, seed=seed + b) for b in range(nb)]
    ctl_o = [oracle.Controller(oracle.CtrlParams(**PARAMS, init_mode=init_mode, seed=seed + b), *GRID)
             for b in range(nb)]
    kc = vc = None  # the committed caches (bf16 bits), carried to the next step
    seen_dk, seen_a = set(), []
    B.adt_get_device_error()
    for t in range(steps):
        dk = [c.next(p) for c, p in zip(ctl_c, pos)]
        assert dk == [c.next(p) for c, p in zip(ctl_o, pos)]
        depth, width = [d for d, _ in dk], [k for _, k in dk]
        seen_dk.update(dk)
        shape = StepShape(layers=layers, H=H, Hkv=H, D=D, V=V, kv_len=kv, depth=depth, width=width, max_nodes=64,
                          lmax=lmax, mode=B.ACCEPT_GREEDY)
        step = TreeVerifyStep(shape, keep_layer_outputs=True)
        inp = synth.step_inputs(layers, H, H, D, V, kv, depth, width, step.n, lmax, seed + 100 * t)
        if kc is not None:
            inp["k_cache"] = torch.from_numpy(kc).view(torch.bfloat16)
            inp["v_cache"] = torch.from_numpy(vc).view(torch.bfloat16)
        trees = [draft_tree(inp["draft_rows"][b], width[b], depth[b], int(inp["root_token"][b]), step.n[b])
                 for b in range(nb)]
        offs = np.concatenate([[0], np.cumsum(step.n)]).astype(np.int64)
        # per image, accept levels while a draw falls under the map's rate at
        # the image's position, and plant that path in the target rows
        for b, tr in enumerate(trees):
            a = 0
            while a < int(tr["depth"].max()) and g.random() < amap[pos[b]]:
                a += 1
            if a:
                path = oracle.ancestor_path(tr["parents"], int(np.argmax(tr["depth"])))[:a + 1]
                synth.plant_path(inp["target"][offs[b]:offs[b + 1]], tr["parents"], tr["tokens"], path)
        step.load_inputs(inp)
        step.launch()
        torch.cuda.synchronize()
        assert B.adt_get_device_error() == 0

        parents = np.concatenate([tr["parents"] for tr in trees])
        tokens = np.concatenate([tr["tokens"] for tr in trees])
        assert np.array_equal(step.tokens.cpu().numpy(), tokens)
        assert np.array_equal(step.parents.cpu().numpy(), parents)
        for layer in ([0, 1] if t == 0 else [t % layers]):
            ref, _ = oracle.tree_attention(inp["q"][layer].double().numpy(), inp["k_cache"][layer].double().numpy(),
                                           inp["v_cache"][layer].double().numpy(), kv,
                                           inp["k_tree"][layer].double().numpy(),
                                           inp["v_tree"][layer].double().numpy(), parents, offs, D ** -0.5)
            assert_attention_close(step.attn_out[layer].double().cpu().numpy(), ref)
        acc = oracle.tree_accept(inp["target"], None, tokens, parents, offs, oracle.ACCEPT_GREEDY,
                                 inp["u_accept"], inp["u_sample"])
        assert acc["accept_margin"] > 1e-5
        alen = [int(x) for x in acc["accept_len"]]
        seen_a += alen
        assert step.accept_len.cpu().tolist() == alen
        assert step.bonus.cpu().tolist() == [int(x) for x in acc["bonus"]]
        for b in range(nb):
            assert step.path[b, :alen[b] + 1].cpu().tolist() == list(acc["path"][b])
        kc, vc, kl = oracle.kv_compact(_bits(inp["k_cache"]), _bits(inp["v_cache"]), kv, _bits(inp["k_tree"]),
                                       _bits(inp["v_tree"]), offs, acc["path"])
        assert np.array_equal(_bits(step.k_cache), kc)
        assert np.array_equal(_bits(step.v_cache), vc)
        kv = [int(x) for x in kl]
        assert step.kv_len_out.cpu().tolist() == kv
        new_pos = [c.update(p, a) for c, p, a in zip(ctl_c, pos, alen)]
        assert new_pos == [c.update(p, a) for c, p, a in zip(ctl_o, pos, alen)]
        pos = new_pos
    print("depth/width seen:", sorted(seen_dk), "accept lengths:", seen_a)
    # the sweep is not degenerate: trees differ between images and steps, and paths get accepted
    assert len(seen_dk) >= 3 and max(seen_a) >= 2
