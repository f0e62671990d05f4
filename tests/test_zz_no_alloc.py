"""dmoe_router_no_alloc: the router entry point that takes no workspace, for callers that
may not allocate device memory (allocator callbacks, plugin hosts that own every device
allocation, loops that must never enter an allocator). It keeps its scratch in a fixed
static device array of the library.

Called through the C ABI twice in a row on the same inputs, it must give what dmoe_router
(with a caller-allocated workspace) gives, within the parity tolerances of the other
tests, and the oracle's routing. Its fault record, which lives in the static array, must be
readable through dmoe_router_no_alloc_device_error. This file is collected last so that a
stop-at-first-failure run has run every other test before it; it also passes on its own in
a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from dmoe_synth import LAYER, LAYER_B8, ROUTE_TOKEN, TINY, layer_inputs, to_numpy
from tests import parity as P

pytestmark = pytest.mark.gpu

# scratch of the router at E = 256, k = 8 (the header's formula): 1169 tokens fit in 4 MiB
MAX_T_E256_K8 = 1169


def _lib():
    m = P.dm()
    return m, m._lib.dmoe_router_no_alloc


def _outputs(shape):
    T, k, E, nb = shape.T, shape.top_k, shape.n_experts, shape.n_blocks
    return dict(idx=torch.full((T, k), -7, dtype=torch.int32, device="cuda"),
                gate=torch.full((T, k), -7.0, dtype=torch.float32, device="cuda"),
                coreset=torch.full((nb, E), -7, dtype=torch.int32, device="cuda"),
                coreset_size=torch.full((nb,), -7, dtype=torch.int32, device="cuda"),
                probs=torch.full((T, E), -7.0, dtype=torch.float32, device="cuda"))


def _no_alloc_call(m, fn, shape, dev, out, with_probs=True):
    desc = P.desc_of(shape)
    st = fn(ctypes.byref(desc), dev["x"].data_ptr(), dev["w_r"].data_ptr(),
            dev["bias"].data_ptr(), out["idx"].data_ptr(), out["gate"].data_ptr(),
            out["coreset"].data_ptr(), out["coreset_size"].data_ptr(),
            out["probs"].data_ptr() if with_probs else None,
            torch.cuda.current_stream().cuda_stream)
    return st


SHAPES = {
    "layer_block_p06": LAYER.with_(top_p=0.6),
    "layer_block_p0": LAYER,
    "tiny_token": TINY.with_(mode=ROUTE_TOKEN),
    # more than 64 tokens: the tiled logits launch, the softmax launch, the block launch
    "layer_b8_block_p0": LAYER_B8,
    "layer_b8_token": LAYER_B8.with_(mode=ROUTE_TOKEN),
    # d not a multiple of 256: the FFMA logits kernel split over d
    "d384_block_p06": LAYER.with_(d_model=384, top_p=0.6),
    # the largest token count whose scratch fits the 4 MiB array at E = 256, k = 8
    "max_tokens_1169": LAYER.with_(block_size=167, n_blocks=7, top_p=0.6),
}


def _same_logits_path(shape) -> bool:
    """dmoe_router computes the logits of 128 or more tokens (d % 64 == 0, E % 32 == 0) on
    tcgen05 from a split of W_r kept in its workspace; the no-alloc call has no room for that
    split and keeps the mma.sync logits, so the two differ there by rounding order only."""
    T = shape.n_blocks * shape.block_size
    tc = T >= 128 and shape.d_model % 64 == 0 and shape.n_experts % 32 == 0
    return not tc


@pytest.mark.parametrize("name", list(SHAPES))
def test_no_alloc_router_matches_workspace_router(name):
    shape = SHAPES[name]
    m, fn = _lib()
    dev = layer_inputs(shape, seed=21, device="cuda", with_weights=False)
    ref = P.gpu_router(shape, dev)               # dmoe_router with a torch workspace
    orc = P.oracle_routing(shape, to_numpy(dev))
    same = _same_logits_path(shape)
    for call in range(2):                        # two calls in a row share the array
        out = _outputs(shape)
        st = _no_alloc_call(m, fn, shape, dev, out, with_probs=(call == 0))
        assert st == 0, m.dmoe_status_string(st)
        st, info = m.dmoe_router_no_alloc_device_error()
        assert st == 0 and info == (0, 0, 0), (st, info)
        got = {k: v.cpu().numpy() for k, v in out.items()}
        if same:
            assert np.array_equal(got["idx"], ref["idx"])
            np.testing.assert_allclose(got["gate"], ref["gate"], rtol=0, atol=P.GATE_ATOL)
            assert np.array_equal(got["coreset"], ref["coreset"])
            assert np.array_equal(got["coreset_size"], ref["coreset_size"])
        if call == 0:
            if same:
                np.testing.assert_allclose(got["probs"], ref["probs"], rtol=1e-6, atol=1e-8)
            else:   # the scores' tolerance against the oracle
                np.testing.assert_allclose(got["probs"], ref["probs"], rtol=1e-5, atol=1e-7)
        # the oracle's routing, under the same rules as dmoe_router's parity test (the
        # scores are checked on the call that asked for them)
        if call == 0:
            stats = P.check_routing(shape, got, orc)
            print(f"{name}: {stats}")
        else:
            assert np.array_equal(got["coreset_size"], first["coreset_size"])
            assert np.array_equal(got["idx"], first["idx"])
        first = got


def test_no_alloc_router_size_limit():
    """One token past the documented limit is refused before anything is launched."""
    m, fn = _lib()
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    p = dummy.data_ptr()
    for shape in (LAYER.with_(block_size=117, n_blocks=10, top_p=0.6),   # 1170 tokens
                  LAYER.with_(block_size=64, n_blocks=64)):              # 4096 tokens
        desc = P.desc_of(shape)
        st = fn(ctypes.byref(desc), p, p, None, p, p, None, None, None,
                torch.cuda.current_stream().cuda_stream)
        assert st == 2, shape                            # DMOE_ERR_UNSUPPORTED
        assert b"static buffer" in m._lib.dmoe_last_error_message()
    assert SHAPES["max_tokens_1169"].T == MAX_T_E256_K8


def test_no_alloc_fault_record_is_readable():
    """A fault recorded on the device into the static array's record is reported (and
    cleared) by dmoe_router_no_alloc_device_error. The fault is a real device-side check:
    the dispatch kernel, given the static array as its workspace, meets an expert id out of
    range. Afterwards the record is clear and the router runs normally."""
    m, fn = _lib()
    ptr, nbytes = m.dmoe_no_alloc_scratch()
    assert ptr != 0 and ptr % 256 == 0 and nbytes == 4 << 20
    shape = TINY
    desc = P.desc_of(shape)
    assert m.dmoe_workspace_size(desc) <= nbytes
    T, k, E = shape.T, shape.top_k, shape.n_experts
    idx = torch.arange(T * k, dtype=torch.int32, device="cuda").reshape(T, k) % E
    idx[3, 1] = E                                    # out of range: recorded, not trapped
    outs = [torch.zeros(n, dtype=torch.int32, device="cuda") for n in (1, E, E + 1, T * k, T * k)]
    st = m._lib.dmoe_dispatch(ctypes.byref(desc), idx.data_ptr(), *[o.data_ptr() for o in outs],
                              ptr, nbytes, torch.cuda.current_stream().cuda_stream)
    assert st == 0, m.dmoe_status_string(st)
    st, info = m.dmoe_router_no_alloc_device_error()
    assert st == 5, (st, info)                       # DMOE_ERR_DEVICE
    assert info[0] == 2 and info[1] == 3 and info[2] == 3 * k + 1   # expert id, dispatch, slot
    st, info = m.dmoe_router_no_alloc_device_error()
    assert st == 0 and info == (0, 0, 0), (st, info)
    # the router still works on the same array, twice
    dev = layer_inputs(shape, seed=4, device="cuda", with_weights=False)
    ref = P.gpu_router(shape, dev)
    for _ in range(2):
        out = _outputs(shape)
        assert _no_alloc_call(m, fn, shape, dev, out) == 0
        st, info = m.dmoe_router_no_alloc_device_error()
        assert st == 0, (st, info)
        assert np.array_equal(out["idx"].cpu().numpy(), ref["idx"])
