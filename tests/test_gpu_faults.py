"""Failure detection without a GPU fault: a bounded device-side wait that runs out.

dmoe_set_debug_hold makes every down tile of the decode-size expert launch wait for more
gate/up tiles than its group has (a count nothing will reach). The wait gives up after its
1 s limit: the kernel records DMOE_ERR_TIMEOUT in the workspace, lets its in-flight copies
land, frees its tensor memory and exits; no trap, no unbounded wait. dmoe_get_device_error
reports the timeout and clears it (with the hold), and the next call on the same workspace
is a normal, parity-checked forward."""
import time

import numpy as np
import pytest

from dmoe_synth import ROUTE_TOKEN, TINY
from tests import parity as P

pytestmark = pytest.mark.gpu

TIMEOUT = 6          # DMOE_ERR_TIMEOUT
ERR_TIMEOUT = 1      # the record's code for a bounded wait that ran out


@pytest.mark.parametrize("shape", [TINY, TINY.with_(mode=ROUTE_TOKEN)], ids=["block", "token"])
def test_bounded_wait_times_out_and_the_workspace_recovers(shape):
    m = P.dm()
    from paper_2605_30876_gb300.layer import MoELayer
    dev, host = P.make(shape, seed=3)
    layer = MoELayer.from_shape(shape, dev)
    layer.forward(dev["x"])
    assert m.dmoe_get_device_error(layer.ws)[0] == 0
    m.dmoe_set_debug_hold(layer.ws, 1 << 20)
    t0 = time.time()
    layer.forward(dev["x"])
    st, info = m.dmoe_get_device_error(layer.ws)
    elapsed = time.time() - t0
    assert st == TIMEOUT, (st, info)
    assert info[0] == ERR_TIMEOUT and info[1] in (4, 5), info     # gate/up or down stage
    assert 0.5 < elapsed < 60, elapsed
    # the record (and the hold with it) is clear; the same workspace gives a normal forward
    assert m.dmoe_get_device_error(layer.ws) == (0, (0, 0, 0))
    y = layer.forward(dev["x"]).clone()
    st, info = m.dmoe_get_device_error(layer.ws)
    assert st == 0, info
    idx = layer.topk_idx.cpu().numpy()
    orc = P.oracle_routing(shape, host)
    ref = P.oracle_output(host, idx, orc.scores)
    P.check_output(y, ref, label="after timeout")


def test_debug_hold_argument_checks():
    m = P.dm()
    import torch
    ws = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(m.DmoeError):
        m.dmoe_set_debug_hold(ws, -1)
    m.dmoe_set_debug_hold(ws, 0)
    assert np.all(ws.cpu().numpy() == 0)
