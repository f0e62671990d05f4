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
    # fewer experts per token inside the coreset; the Top-4 token baseline
    "layer_fewer_k4_of8_p0": LAYER.with_(top_k=4, block_top_k=8),
    "layer_fewer_k2_of8_p06": LAYER.with_(top_k=2, block_top_k=8, top_p=0.6),
    "layer_b8_fewer_k4_of8": LAYER_B8.with_(top_k=4, block_top_k=8),
    "tiny_fewer_k1_of2_shared": TINY.with_(top_k=1, block_top_k=2, d_ff_shared=128),
    "layer_token_top4": LAYER.with_(mode=ROUTE_TOKEN, top_k=4),
    # the paper's top-p sweep ends beside p = 0.6 (Table 3: p_test 0.4 ... 0.8)
    "layer_block_p04": LAYER.with_(top_p=0.4),
    "layer_block_p08": LAYER.with_(top_p=0.8),
    # block top-k on the general path (the expert launch plans from the published coresets
    # and does the dispatch): no shared expert, k not a multiple of three, fewer experts;
    # 20 blocks of 16 (ragged token tiles), skewed bias, k = 6
    "spec_b8x16_noshared_k4_E64": LAYER.with_(block_size=16, n_blocks=8, d_ff_shared=0,
                                              top_k=4, n_experts=64),
    "spec_b20x16_k6_bias1": LAYER.with_(block_size=16, n_blocks=20, top_k=6, bias_scale=1.0),
    # decode size, the coresets published as masks (the expert launch streams their union):
    # two blocks at p = 0.4, and k = 1 of 8 over blocks of 4 tokens (at most 4 of a block's
    # 8 coreset members are kept: the others take no rows from the dispatch)
    "decode_masks_b2_p04": LAYER.with_(n_blocks=2, top_p=0.4),
    "decode_masks_k1_of8": LAYER.with_(block_size=4, n_blocks=2, top_k=1, block_top_k=8),
    # the block-size x batch x bias grid: its smallest corner, uniform router bias
    "sweep_B4x1_bias0_block": LAYER.with_(block_size=4, n_blocks=1, bias_scale=0.0),
    "sweep_B4x1_bias0_token": LAYER.with_(block_size=4, n_blocks=1, bias_scale=0.0,
                                          mode=ROUTE_TOKEN),
}
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
    ref = P.oracle_output(host, idx, orc.scores)
    P.check_output(y, ref, label=name)
    # deterministic: a second call gives the same bits
    y2 = layer.forward(dev["x"])
    assert torch.equal(y, y2)


@pytest.mark.parametrize("name", ["tiny_block_p06", "layer_block_p06", "layer_token",
                                  "layer_b8_block_p0", "T300_multi_ntile"])
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


def test_router_prepare_skips_only_a_matching_split():
    """dmoe_router_prepare (the tensor-core router's split of W_r, once): the prepared
    forward equals an unprepared one bit for bit; a call with another W_r on the prepared
    workspace splits that one, and a later call with the first W_r splits it again."""
    shape = LAYER_B8
    m = P.dm()
    dev, _ = P.make(shape, seed=3)
    from paper_2605_30876_gb300.layer import MoELayer
    layer = MoELayer.from_shape(shape, dev)   # prepares its workspace
    y_prep = layer.forward(dev["x"]).clone()

    def fwd(w_r, ws):
        y = torch.empty_like(y_prep)
        m.dmoe_layer_forward(layer.desc, dev["x"], w_r, dev["bias"], dev["w_gate"], dev["w_up"],
                             dev["w_down"], dev["ws_gate"], dev["ws_up"], dev["ws_down"], y,
                             None, None, None, None, workspace=ws)
        st, info = m.dmoe_get_device_error(ws)
        assert st == 0, info
        return y

    assert torch.equal(fwd(dev["w_r"], m.alloc_workspace(layer.desc)), y_prep)
    w_r2 = dev["w_r"].flip(1).contiguous()   # the experts' router columns reversed
    y_b = fwd(w_r2, layer.ws)
    assert torch.equal(y_b, fwd(w_r2, m.alloc_workspace(layer.desc)))
    assert not torch.equal(y_b, y_prep)
    assert torch.equal(layer.forward(dev["x"]), y_prep)


def test_stack_shape_layer_all_tokens():
    """One layer of the 2048-token stack shape (64 blocks of 32): routing parity and outputs
    on every token."""
    shape = STACK20
    dev, host = P.make(shape, seed=11)
    from paper_2605_30876_gb300.layer import MoELayer
    layer = MoELayer.from_shape(shape, dev)
    y = layer.forward(dev["x"])
    st, info = P.dm().dmoe_get_device_error(layer.ws)
    assert st == 0, info
    idx = layer.topk_idx.cpu().numpy()
    orc = P.oracle_routing(shape, host)
    ref = P.oracle_output(host, idx, orc.scores)
    P.check_output(y, ref, label="stack_T2048")


# Large forwards: routing and outputs of every token against the oracle.
LARGE_CASES = {
    # the 2048-token stack layer with token routing (the general expert launch at its
    # heaviest, every expert unique)
    "stack_T2048_token": STACK20.with_(mode=ROUTE_TOKEN),
    # the block-size x batch x bias grid's largest corner, most skewed router bias
    "sweep_B64x32_bias1_block": LAYER.with_(block_size=64, n_blocks=32, bias_scale=1.0),
    "sweep_B64x32_bias1_token": LAYER.with_(block_size=64, n_blocks=32, bias_scale=1.0,
                                            mode=ROUTE_TOKEN),
}


@pytest.mark.parametrize("name", list(LARGE_CASES))
def test_large_forward_all_tokens(name):
    shape = LARGE_CASES[name]
    m = P.dm()
    from dmoe_synth import layer_inputs
    from paper_2605_30876_gb300.layer import MoELayer
    dev = layer_inputs(shape, seed=13, device="cuda")
    layer = MoELayer.from_shape(shape, dev)
    y = layer.forward(dev["x"]).clone()
    st, info = m.dmoe_get_device_error(layer.ws)
    assert st == 0, info
    host = P.lazy_host(dev)
    idx = layer.topk_idx.cpu().numpy()
    orc = P.oracle_routing(shape, host)
    near = 0
    for t in range(shape.T):
        if orc.set_margin[t] >= P.DELTA and (shape.mode == ROUTE_TOKEN or
                                             orc.coreset_margin[t // shape.block_size] >= P.DELTA):
            assert set(idx[t].tolist()) == set(orc.idx[t].tolist()), t
        else:
            near += 1
    np.testing.assert_allclose(layer.topk_gate.cpu().numpy(), O.gates_for(orc.scores, idx),
                               atol=P.GATE_ATOL)
    assert int(layer.n_unique.item()) == len(np.unique(idx))
    ref = P.oracle_output(host, idx, orc.scores)
    r, mx = P.check_output(y, ref, label=name)
    print(f"{name}: unique {int(layer.n_unique.item())}, near-tie tokens {near}, "
          f"all {shape.T} tokens: rel-L2 {r:.2e} max-abs {mx:.2e}")


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


_ExpertRows = P.ExpertRows


def _rms_norm(x: torch.Tensor) -> torch.Tensor:
    """Row-wise RMS normalisation (no weight), rounded to bf16: each stack layer's input."""
    xf = x.double()
    return (xf / xf.pow(2).mean(-1, keepdim=True).sqrt()).to(torch.bfloat16)


def test_stack20_end_to_end():
    """The 20-layer residual stack of 64 blocks of 32 tokens, block top-k, separate seeded
    weights per layer, each layer fed the RMS-normalised stream: u_l = bf16(x_l / rms(x_l)),
    x_{l+1} = bf16(x_l + y_l(u_l)). Two sampled blocks: every layer's output against the
    oracle fed the GPU's u_l and evaluated on the GPU's routing (teacher-forced, the one-layer
    bounds), and the oracle's own free-running stack against the GPU's final x (reported; a
    loose bound, since a near-tie routing decision may flip)."""
    from dmoe_synth import STACK20_LAYERS, bf16_bits, layer_inputs
    from paper_2605_30876_gb300.layer import MoELayer
    shape = STACK20
    L = STACK20_LAYERS
    weights = [layer_inputs(shape, seed=500 + l, device="cuda", layer=l) for l in range(L)]
    x0 = layer_inputs(shape, seed=499, device="cuda", with_weights=False)["x"]
    layers = [MoELayer.from_shape(shape, w) for w in weights]
    xs, us, ys = [x0], [], []
    for l in range(L):
        u = _rms_norm(xs[l])
        y = layers[l].forward(u).clone()
        st, info = P.dm().dmoe_get_device_error(layers[l].ws)
        assert st == 0, info
        us.append(u)
        ys.append(y)
        xs.append(torch.add(xs[l], y))
    B = shape.block_size
    blocks = (0, 37)
    tokens = np.concatenate([np.arange(b * B, (b + 1) * B) for b in blocks])
    tok_t = torch.from_numpy(tokens).cuda()
    x_free = x0[tok_t].cpu()
    diverged = 0   # (layer, token) pairs where the free-running oracle routes differently
    for l in range(L):
        w = weights[l]
        host = {"x": bf16_bits(us[l][tok_t]), "w_r": w["w_r"].cpu().numpy(),
                "bias": w["bias"].cpu().numpy(), "w_gate": _ExpertRows(w["w_gate"]),
                "w_up": _ExpertRows(w["w_up"]), "w_down": _ExpertRows(w["w_down"]),
                "ws_gate": bf16_bits(w["ws_gate"]), "ws_up": bf16_bits(w["ws_up"]),
                "ws_down": bf16_bits(w["ws_down"])}
        # teacher-forced: this layer on the GPU's input and routing
        orc = O.route(host["x"], host["w_r"], host["bias"], shape.top_k, shape.mode, B,
                      shape.top_p)
        idx = layers[l].topk_idx[tok_t].cpu().numpy()
        ref = P.oracle_output(host, idx, orc.scores)
        r_l, m_l = P.check_output(ys[l][tok_t], ref, label=f"stack layer {l}")
        print(f"stack layer {l:2d}: rel-L2 {r_l:.2e}  max-abs {m_l:.2e}")
        # free-running: the oracle's own routing on its own stream
        free = dict(host, x=bf16_bits(_rms_norm(x_free)))
        r = O.route(free["x"], free["w_r"], free["bias"], shape.top_k, shape.mode, B,
                    shape.top_p)
        yf = O.moe_forward_given_routing(free["x"], free["w_gate"], free["w_up"], free["w_down"],
                                         r.idx, r.gate, free["ws_gate"], free["ws_up"],
                                         free["ws_down"])
        diverged += sum(set(r.idx[t].tolist()) != set(idx[t].tolist()) for t in range(len(tokens)))
        x_free = (x_free.double() + torch.from_numpy(yf)).to(torch.bfloat16)
    final = xs[L][tok_t].double().cpu().numpy()
    err = P.rel_l2(final, x_free.double().numpy())
    print(f"stack20 end-to-end rel-L2 on blocks {blocks}: {err:.3e}; free-running routing "
          f"differs from the GPU's at {diverged} of {L * len(tokens)} (layer, token) pairs")
    # reported figure: once a near-tie flips a block's coreset the two streams carry different
    # experts' outputs from there on; the bound only rules out a systematic drift
    assert err < 0.25


def test_decode_masks_case_has_unkept_coreset_members():
    """The k = 1 of 8 case above streams coreset members that no token keeps (their groups
    take no rows from the dispatch): the oracle's coresets' union is larger than its set of
    routed experts, so the output parity case exercises that path."""
    shape = LAYER_CASES["decode_masks_k1_of8"]
    dev, host = P.make(shape, seed=3)
    orc = P.oracle_routing(shape, host)
    union = set(np.concatenate([np.asarray(c) for c in orc.coresets]).tolist())
    routed = set(np.unique(orc.idx).tolist())
    assert routed <= union and len(union) > len(routed), (len(union), len(routed))

