"""GPU parity of the expert execution and of the whole layer against the CPU oracle: the
GPU's bf16 y against the oracle's float64 y on the GPU's own selection (rel-L2 <= 1e-2,
max-abs <= 3e-2), through dmoe_moe_forward and dmoe_layer_forward."""
import numpy as np
import pytest
import torch

import oracle as O
from dmoe_synth import LAYER, LAYER_B8, ROUTE_BLOCK, ROUTE_TOKEN, STACK20, TINY
from tests import parity as P

pytestmark = pytest.mark.gpu

LAYER_CASES = {
    "tiny_block_p0": TINY,
    "tiny_block_p06": TINY.with_(top_p=0.6),
    "tiny_token": TINY.with_(mode=ROUTE_TOKEN),
    "tiny_shared": TINY.with_(d_ff_shared=256, top_p=0.6),
    "layer_block_p0": LAYER,
    "layer_block_p06": LAYER.with_(top_p=0.6),
    "layer_token": LAYER.with_(mode=ROUTE_TOKEN),
    "layer_noshared": LAYER.with_(d_ff_shared=0, top_p=0.6),
    "layer_b8_block_p0": LAYER_B8,
    "layer_b8_token": LAYER_B8.with_(mode=ROUTE_TOKEN),
    "ragged_T60_k1": TINY.with_(block_size=12, n_blocks=5, top_k=1, top_p=0.5, d_ff_shared=128),
    "E8_k3_d128": TINY.with_(n_experts=8, top_k=3, top_p=0.7, d_model=128, d_ff=256),
    "T300_multi_ntile": LAYER.with_(block_size=60, n_blocks=5, top_p=0.0),
    "wide_ff_I1024": TINY.with_(d_model=512, d_ff=1024, d_ff_shared=384, n_blocks=3, top_p=0.6),
    # block top-k at decode sizes: the expert launch starts on the published coresets
    "decode_B16x4_p0": LAYER.with_(block_size=16, n_blocks=4),
    "decode_B1x40_p0": LAYER.with_(block_size=1, n_blocks=40, bias_scale=0.0),
}
SAMPLED = {"T300_multi_ntile"}


def _tokens(shape, name):
    if name in SAMPLED:
        rng = np.random.default_rng(1)
        t = np.sort(rng.choice(shape.T, 48, replace=False))
        return np.unique(np.concatenate([t, [0, shape.T - 1]]))
    return None


@pytest.mark.parametrize("name", list(LAYER_CASES))
def test_layer_forward_matches_oracle(name):
    shape = LAYER_CASES[name]
    m = P.dm()
    dev, host = P.make(shape, seed=3)
    from paper_2605_30876_gb300.layer import MoELayer
    layer = MoELayer.from_shape(shape, dev)
    y = layer.forward(dev["x"]).clone()
    st, info = m.dmoe_get_device_error(layer.ws)
    assert st == 0, info
    idx = layer.topk_idx.cpu().numpy()
    orc = P.oracle_routing(shape, host)
    g = dict(idx=idx, gate=layer.topk_gate.cpu().numpy())
    # selection valid and equal to the oracle's where unambiguous
    for t in range(shape.T):
        if orc.set_margin[t] >= P.DELTA and (shape.mode == ROUTE_TOKEN or
                                             orc.coreset_margin[t // shape.block_size] >= P.DELTA):
            assert set(idx[t].tolist()) == set(orc.idx[t].tolist())
    np.testing.assert_allclose(g["gate"], O.gates_for(orc.scores, idx), atol=P.GATE_ATOL)
    assert int(layer.n_unique.item()) == len(np.unique(idx))
    tokens = _tokens(shape, name)
    ref = P.oracle_output(host, idx, orc.scores, tokens=tokens)
    P.check_output(y, ref, tokens=tokens, label=name)
    # deterministic: a second call gives the same bits
    y2 = layer.forward(dev["x"])
    assert torch.equal(y, y2)


@pytest.mark.parametrize("name", ["tiny_block_p06", "layer_block_p06", "layer_token"])
def test_moe_forward_on_injected_oracle_routing(name):
    """dmoe_dispatch + dmoe_moe_forward on the oracle's own routing (ids and gates)."""
    shape = LAYER_CASES[name]
    m = P.dm()
    dev, host = P.make(shape, seed=5)
    orc = P.oracle_routing(shape, host)
    desc = P.desc_of(shape)
    idx_t = torch.from_numpy(orc.idx).cuda()
    gate_t = torch.from_numpy(orc.gate.astype(np.float32)).cuda()
    out, ws = P.gpu_dispatch(shape, idx_t)
    y = torch.empty((shape.T, shape.d_model), dtype=torch.bfloat16, device="cuda")
    m.dmoe_moe_forward(desc, dev["x"], dev["w_gate"], dev["w_up"], dev["w_down"], dev["ws_gate"],
                       dev["ws_up"], dev["ws_down"], gate_t, out["n_unique"], out["unique_ids"],
                       out["offsets"], out["rows"], out["pos"], y, workspace=ws)
    st, info = m.dmoe_get_device_error(ws)
    assert st == 0, info
    ref = O.moe_forward_given_routing(host["x"], host["w_gate"], host["w_up"], host["w_down"],
                                      orc.idx, orc.gate, host["ws_gate"], host["ws_up"],
                                      host["ws_down"])
    P.check_output(y, ref, label=name)


def test_stack_shape_layer_sampled():
    """One layer of the 2048-token stack shape (64 blocks of 32): routing parity on all
    tokens, outputs on sampled tokens (the oracle is slow at this size)."""
    shape = STACK20
    dev, host = P.make(shape, seed=11)
    from paper_2605_30876_gb300.layer import MoELayer
    layer = MoELayer.from_shape(shape, dev)
    y = layer.forward(dev["x"])
    st, info = P.dm().dmoe_get_device_error(layer.ws)
    assert st == 0, info
    idx = layer.topk_idx.cpu().numpy()
    orc = P.oracle_routing(shape, host)
    tokens = np.unique(np.concatenate([np.random.default_rng(2).choice(shape.T, 40, replace=False),
                                       [0, shape.T - 1]]))
    ref = P.oracle_output(host, idx, orc.scores, tokens=tokens)
    P.check_output(y, ref, tokens=tokens, label="stack_T2048")


def test_identical_experts_give_plain_ffn():
    """All routed experts equal: whatever the routing, y = FFN(x) + shared(x) (gates sum to 1)."""
    shape = LAYER.with_(top_p=0.6)
    dev, host = P.make(shape, seed=7)
    for k_ in ("w_gate", "w_up", "w_down"):
        dev[k_] = dev[k_][:1].expand_as(dev[k_]).contiguous()
    host = {k_: (v if k_ not in ("w_gate", "w_up", "w_down") else None) for k_, v in host.items()}
    from dmoe_synth import to_numpy
    w1 = to_numpy({k_: dev[k_][:1] for k_ in ("w_gate", "w_up", "w_down")})
    from paper_2605_30876_gb300.layer import MoELayer
    y = MoELayer.from_shape(shape, dev).forward(dev["x"])
    x = O.bf16_bits_to_f64(host["x"])
    ref = O.swiglu_ffn(x, O.bf16_bits_to_f64(w1["w_gate"][0]), O.bf16_bits_to_f64(w1["w_up"][0]),
                       O.bf16_bits_to_f64(w1["w_down"][0]))
    ref += O.swiglu_ffn(x, O.bf16_bits_to_f64(host["ws_gate"]), O.bf16_bits_to_f64(host["ws_up"]),
                        O.bf16_bits_to_f64(host["ws_down"]))
    P.check_output(y, ref, label="identical_experts")
