"""CPU oracle of the dMoE MoE-layer forward — test infrastructure only.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference legs of
``bench.py`` import this package. The CUDA library never does, and this package imports
nothing of the library. Every function is pinned by the ``-m "not gpu"`` tests in
``tests/test_oracle_pins.py`` (hand-worked Algorithm 1 cases, closed forms, brute force,
invariants).
"""
from .dmoe_oracle import *  # noqa: F401,F403
from .dmoe_oracle import (ROUTE_BLOCK, ROUTE_TOKEN, Coreset, Dispatch, Routing,  # noqa: F401
                          aggregate, bf16_bits_to_f64, dispatch, gates_for, layer_forward,
                          mask_outside, moe_forward_given_routing, normalize, renormalize,
                          route, route_block, route_token, router_logits, router_scores,
                          silu, sort_desc, swiglu_ffn, top_p, topk_desc, topk_margins,
                          topk_mask)
