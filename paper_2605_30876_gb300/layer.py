"""A resident MoE layer: device weights, workspace and output buffers around
dmoe_layer_forward (argument marshalling only; the forward runs in libdmoe's kernels)."""
from __future__ import annotations

from typing import Dict, Optional

import torch

from . import (DMOE_ROUTE_BLOCK, LayerDesc, alloc_workspace, dmoe_layer_forward,
               dmoe_router_prepare, make_desc)

WEIGHT_KEYS = ("w_r", "bias", "w_gate", "w_up", "w_down", "ws_gate", "ws_up", "ws_down")


class MoELayer:
    """One MoE layer with its weights resident in HBM.

    weights: dict with w_r fp32 [d,E], bias fp32 [E] (or None), w_gate/w_up bf16 [E,I,d],
    w_down bf16 [E,d,I] and, with a shared expert, ws_gate/ws_up bf16 [I_s,d],
    ws_down bf16 [d,I_s] (None otherwise).
    """

    def __init__(self, desc: LayerDesc, weights: Dict[str, Optional[torch.Tensor]],
                 device="cuda", workspace: Optional[torch.Tensor] = None):
        self.desc = desc
        self.w = {k: weights.get(k) for k in WEIGHT_KEYS}
        self.device = torch.device(device)
        T, k, E, d = desc.T, desc.top_k, desc.n_experts, desc.d_model
        self.ws = workspace if workspace is not None else alloc_workspace(desc, self.device)
        self.y = torch.empty((T, d), dtype=torch.bfloat16, device=self.device)
        self.topk_idx = torch.empty((T, k), dtype=torch.int32, device=self.device)
        self.topk_gate = torch.empty((T, k), dtype=torch.float32, device=self.device)
        self.n_unique = torch.zeros(1, dtype=torch.int32, device=self.device)
        self.unique_ids = torch.empty(E, dtype=torch.int32, device=self.device)
        # the router weight's tensor-core split, once (the forwards on this workspace then
        # skip it); prepare() again after changing w_r in place
        self.prepare()

    def prepare(self, stream=None) -> None:
        dmoe_router_prepare(self.desc, self.w["w_r"], self.ws, stream=stream)

    @classmethod
    def from_shape(cls, shape, weights, device="cuda", workspace=None) -> "MoELayer":
        desc = make_desc(shape.d_model, shape.n_experts, shape.top_k, shape.d_ff,
                         shape.d_ff_shared, shape.block_size, shape.n_blocks,
                         getattr(shape, "mode", DMOE_ROUTE_BLOCK), getattr(shape, "top_p", 0.0),
                         getattr(shape, "block_top_k", 0))
        return cls(desc, weights, device, workspace)

    def forward(self, x: torch.Tensor, y: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        out = self.y if y is None else y
        w = self.w
        dmoe_layer_forward(self.desc, x, w["w_r"], w["bias"], w["w_gate"], w["w_up"], w["w_down"],
                           w["ws_gate"], w["ws_up"], w["ws_down"], out, self.topk_idx,
                           self.topk_gate, self.n_unique, self.unique_ids, workspace=self.ws,
                           stream=stream)
        return out
