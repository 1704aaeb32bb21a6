"""CPU oracle for the ADT-Tree verify path.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline legs of ``bench.py``; never by the library itself.
"""
from .tree_verify import (ACCEPT_GREEDY, ACCEPT_SPEC, ACCEPT_SPEC_DET, ancestor_path,  # noqa: F401
                          argmax_lowest, cfg_logits, check_parents, children, kv_compact, kv_compact_inplace,
                          sample_inverse_cdf,
                          softmax64, tree_accept, tree_attention, tree_expand, tree_rerank)
from .controller import (INIT_HORIZONTAL, INIT_RANDOM, INIT_TOKENFLOCK, INIT_VERTICAL, Controller,  # noqa: F401
                         CtrlParams, anole_params, counter_draw, llamagen_params, splitmix64)
