"""Seeded synthetic inputs for the block-routed MoE-layer forward.

This module is shared by the CUDA path's tests/bench and by the CPU oracle. It holds
no arithmetic of the method itself: it only draws random tensors with the shapes and
distributions of the workloads below and rounds them to the storage types.

Workload shapes (one MoE layer of a block-diffusion decoding step):

* ``tiny``       d=256,  E=16,  top-2, I=128, no shared expert, 2 sequences x 1 block of 8
* ``layer``      d=2048, E=256, top-8, I=512, one shared expert (I_s=512),
                 1 sequence x 1 block of 32 tokens, Zipf-like router bias 0.5*ln(1/rank)
* ``layer_b8``   the ``layer`` shape, 8 sequences x 1 block of 32 (256 tokens)
* ``sweep``      the ``layer`` shape, block size in {4,8,16,32,64} x batch in {1,4,16,32},
                 bias scale in {0, 0.5, 1.0}
* ``stack20``    20 layers of the ``layer`` shape, 64 sequences x 1 block of 32 (2048 tokens)

Distributions: x ~ N(0,1) bf16; expert weights ~ N(0, 0.02^2) bf16 (0.02 is the standard
deviation); router weight W_r ~ N(0, 1/d) fp32; router bias b_e = s * ln(1/rank_e) with
rank a seeded permutation of 1..E (s = bias scale; s = 0 gives b = 0).

Random numbers come from ``torch.Generator`` (CPU: mt19937, CUDA: Philox) seeded from
(seed, tensor tag); the rank permutation comes from NumPy's PCG64. Generating on the
device is much faster for the 1.6 GB-per-layer weight sets; the same seed gives
different (equally distributed) numbers on CPU and CUDA, so a parity test always draws
once and hands the same tensors to both sides.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Iterator, Optional

import numpy as np
import torch

ROUTE_TOKEN = 0
ROUTE_BLOCK = 1

_TAGS = {"x": 1, "w_r": 2, "w_gate": 3, "w_up": 4, "w_down": 5,
         "ws_gate": 6, "ws_up": 7, "ws_down": 8, "perm": 9}

EXPERT_STD = 0.02


@dataclasses.dataclass(frozen=True)
class MoEShape:
    """One MoE layer and one decoding-step batch.

    d_model: hidden size d; n_experts: routed experts E; top_k: experts per token k;
    d_ff: expert SwiGLU intermediate I; d_ff_shared: shared-expert intermediate (0 = none);
    block_size: diffusion block size B; n_blocks: blocks per forward (one per sequence);
    mode: ROUTE_BLOCK or ROUTE_TOKEN; top_p: coreset threshold p (0 => coreset of size k,
    i.e. block top-k; >= 1 => every expert with a nonzero block score);
    bias_scale: s in b_e = s * ln(1/rank_e); block_top_k: block mode, the k of TopKMask and
    of the coreset floor when every token keeps only top_k < block_top_k members of its
    coreset (0 = top_k).
    """
    d_model: int
    n_experts: int
    top_k: int
    d_ff: int
    d_ff_shared: int
    block_size: int
    n_blocks: int
    mode: int = ROUTE_BLOCK
    top_p: float = 0.0
    bias_scale: float = 0.0
    block_top_k: int = 0

    @property
    def T(self) -> int:
        return self.block_size * self.n_blocks

    def with_(self, **kw) -> "MoEShape":
        return dataclasses.replace(self, **kw)

    def expert_bytes(self) -> int:
        """bf16 bytes of one routed expert (gate, up and down)."""
        return 3 * self.d_model * self.d_ff * 2

    def shared_bytes(self) -> int:
        return 3 * self.d_model * self.d_ff_shared * 2


TINY = MoEShape(d_model=256, n_experts=16, top_k=2, d_ff=128, d_ff_shared=0,
                block_size=8, n_blocks=2, mode=ROUTE_BLOCK, top_p=0.0, bias_scale=0.0)
LAYER = MoEShape(d_model=2048, n_experts=256, top_k=8, d_ff=512, d_ff_shared=512,
                 block_size=32, n_blocks=1, mode=ROUTE_BLOCK, top_p=0.0, bias_scale=0.5)
LAYER_B8 = LAYER.with_(n_blocks=8)
STACK20 = LAYER.with_(n_blocks=64)
STACK20_LAYERS = 20

SWEEP_BLOCK_SIZES = (4, 8, 16, 32, 64)
SWEEP_BATCHES = (1, 4, 16, 32)
SWEEP_BIAS_SCALES = (0.0, 0.5, 1.0)


def sweep_shapes(mode: int = ROUTE_BLOCK, top_p: float = 0.0) -> Iterator[MoEShape]:
    """The block-size x batch x bias-scale grid on the ``layer`` shape."""
    for s in SWEEP_BIAS_SCALES:
        for bsz in SWEEP_BLOCK_SIZES:
            for nb in SWEEP_BATCHES:
                yield LAYER.with_(block_size=bsz, n_blocks=nb, bias_scale=s,
                                  mode=mode, top_p=top_p)


def _gen(device, seed: int, tag: str, layer: int = 0) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((seed * 1_000_003 + layer * 7919 + _TAGS[tag]) & 0x7FFF_FFFF_FFFF_FFFF)
    return g


def _normal(shape, std, device, seed, tag, layer=0, dtype=torch.bfloat16):
    g = _gen(device, seed, tag, layer)
    t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)  # round-to-nearest-even for bf16


def router_bias(n_experts: int, scale: float, seed: int, layer: int = 0) -> np.ndarray:
    """b_e = scale * ln(1/rank_e), rank = seeded permutation of 1..E (Zipf-like popularity)."""
    rng = np.random.default_rng([seed, layer, _TAGS["perm"]])
    rank = rng.permutation(n_experts) + 1
    return (scale * np.log(1.0 / rank.astype(np.float64))).astype(np.float32)


def layer_inputs(shape: MoEShape, seed: int = 0, device="cpu", layer: int = 0,
                 with_weights: bool = True) -> Dict[str, Optional[torch.Tensor]]:
    """All tensors of one MoE-layer forward, on ``device``.

    Returns x [T,d] bf16, w_r [d,E] fp32, bias [E] fp32, w_gate/w_up [E,I,d] bf16,
    w_down [E,d,I] bf16 and, when d_ff_shared > 0, ws_gate/ws_up [I_s,d], ws_down [d,I_s]
    bf16 (else None). Expert weights are skipped when ``with_weights`` is False.
    """
    d, E, I, Is, T = shape.d_model, shape.n_experts, shape.d_ff, shape.d_ff_shared, shape.T
    out: Dict[str, Optional[torch.Tensor]] = {}
    out["x"] = _normal((T, d), 1.0, device, seed, "x", layer)
    out["w_r"] = _normal((d, E), 1.0 / math.sqrt(d), device, seed, "w_r", layer,
                         dtype=torch.float32)
    out["bias"] = torch.from_numpy(router_bias(E, shape.bias_scale, seed, layer)).to(device)
    if with_weights:
        out["w_gate"] = _normal((E, I, d), EXPERT_STD, device, seed, "w_gate", layer)
        out["w_up"] = _normal((E, I, d), EXPERT_STD, device, seed, "w_up", layer)
        out["w_down"] = _normal((E, d, I), EXPERT_STD, device, seed, "w_down", layer)
        if Is > 0:
            out["ws_gate"] = _normal((Is, d), EXPERT_STD, device, seed, "ws_gate", layer)
            out["ws_up"] = _normal((Is, d), EXPERT_STD, device, seed, "ws_up", layer)
            out["ws_down"] = _normal((d, Is), EXPERT_STD, device, seed, "ws_down", layer)
        else:
            out["ws_gate"] = out["ws_up"] = out["ws_down"] = None
    return out


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw bf16 bit patterns of a tensor as a host uint16 array (no arithmetic)."""
    assert t.dtype == torch.bfloat16
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def to_numpy(inputs: Dict[str, Optional[torch.Tensor]]) -> Dict[str, Optional[np.ndarray]]:
    """Host copies for the oracle: bf16 tensors as uint16 bit patterns, fp32 as float32."""
    res: Dict[str, Optional[np.ndarray]] = {}
    for k, v in inputs.items():
        if v is None:
            res[k] = None
        elif v.dtype == torch.bfloat16:
            res[k] = bf16_bits(v)
        else:
            res[k] = v.detach().cpu().numpy()
    return res
