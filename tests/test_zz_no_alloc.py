"""dmoe_router_no_alloc: the router entry point that takes no workspace, for callers that
may not allocate device memory (allocator callbacks, plugin hosts that own every device
allocation, loops that must never enter an allocator). It keeps its scratch in a fixed
static device array of the library.

Called through the C ABI twice in a row on the same inputs, it must give what dmoe_router
(with a caller-allocated workspace) gives, within the parity tolerances of the other
tests. This file is collected last so that a stop-at-first-failure run has run every other
test before it; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from dmoe_synth import LAYER, ROUTE_TOKEN, TINY, layer_inputs
from tests import parity as P

pytestmark = pytest.mark.gpu


def _lib():
    m = P.dm()
    lib = m._lib
    fn = lib.dmoe_router_no_alloc
    Vp = ctypes.c_void_p
    fn.argtypes = [ctypes.POINTER(m.LayerDesc), Vp, Vp, Vp, Vp, Vp, Vp, Vp, Vp, Vp]
    fn.restype = ctypes.c_int
    return m, fn


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


@pytest.mark.parametrize("shape", [LAYER.with_(top_p=0.6), LAYER,
                                   TINY.with_(mode=ROUTE_TOKEN)],
                         ids=["layer_block_p06", "layer_block_p0", "tiny_token"])
def test_no_alloc_router_matches_workspace_router(shape):
    m, fn = _lib()
    dev = layer_inputs(shape, seed=21, device="cuda", with_weights=False)
    ref = P.gpu_router(shape, dev)               # dmoe_router with a torch workspace
    for call in range(2):                        # two calls in a row share the array
        out = _outputs(shape)
        st = _no_alloc_call(m, fn, shape, dev, out, with_probs=(call == 0))
        assert st == 0, m.dmoe_status_string(st)
        torch.cuda.synchronize()
        got = {k: v.cpu().numpy() for k, v in out.items()}
        assert np.array_equal(got["idx"], ref["idx"])
        np.testing.assert_allclose(got["gate"], ref["gate"], rtol=0, atol=P.GATE_ATOL)
        assert np.array_equal(got["coreset"], ref["coreset"])
        assert np.array_equal(got["coreset_size"], ref["coreset_size"])
        if call == 0:
            np.testing.assert_allclose(got["probs"], ref["probs"], rtol=1e-6, atol=1e-8)


def test_no_alloc_router_rejects_oversized_shapes():
    m, fn = _lib()
    shape = LAYER.with_(block_size=64, n_blocks=64)     # 4096 tokens: 12 MiB of scratch
    desc = P.desc_of(shape)
    dummy = torch.zeros(16, dtype=torch.int32, device="cuda")
    p = dummy.data_ptr()
    st = fn(ctypes.byref(desc), p, p, None, p, p, None, None, None,
            torch.cuda.current_stream().cuda_stream)
    assert st == 2                                      # DMOE_ERR_UNSUPPORTED
    assert b"static buffer" in m._lib.dmoe_last_error_message()
