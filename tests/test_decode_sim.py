"""The decoding-step harness of bench.py (--decode-sim): a synthetic block-diffusion loop
around the MoE stack that records the unique-expert count U of every layer at every step
(§3, Table 1: U varies across decoding steps, reported as its coefficient of variation).

GPU test: a two-layer, one-block run at a small shape. The U the harness records at each
step must be the number of distinct experts in that step's routing (read back from the
layers' outputs), and its CV must be sigma / mu over the recorded steps. CPU test: the CV
helper on hand values."""
import numpy as np
import pytest
import torch

import bench
from dmoe_synth import ROUTE_TOKEN, TINY


def test_unique_count_cv_hand_values():
    # layer 0: U = 2, 4, 6 -> mean 4, population sigma sqrt(8/3); layer 1 constant -> 0
    U = np.array([[2, 8], [4, 8], [6, 8]], dtype=np.float64)
    cv = bench.unique_count_cv(U)
    assert cv[0] == pytest.approx(np.sqrt(8.0 / 3.0) / 4.0, rel=1e-12)
    assert cv[1] == 0.0


@pytest.mark.gpu
def test_decode_sim_records_the_library_unique_counts():
    import paper_2605_30876_gb300 as dm
    from paper_2605_30876_gb300.layer import MoELayer
    shape = TINY.with_(n_blocks=1, block_size=8)
    modes = [("block_p0", shape), ("token", shape.with_(mode=ROUTE_TOKEN))]
    seen = {}

    def on_step(name, step, layers):
        seen.setdefault(name, []).append(
            [len(np.unique(L.topk_idx.cpu().numpy())) for L in layers])

    recs = bench.decode_sim(torch, dm, MoELayer, shape, n_layers=2, n_blocks=1, vocab=512,
                            ctx=64, head_dim=128, seed=0, modes=modes, on_step=on_step)
    assert [r["routing"] for r in recs] == ["block_p0", "token"]
    for r in recs:
        U = r["U"]
        assert U.shape[1] == 2 and U.shape[0] >= 1
        assert U.shape[0] == len(seen[r["routing"]])
        # the harness's U is the library's n_unique, which equals the distinct routed ids
        assert np.array_equal(U, np.asarray(seen[r["routing"]], np.float64))
        # the CV is sigma / mu over the recorded steps
        cv = bench.unique_count_cv(U)
        np.testing.assert_allclose(cv, U.std(0) / U.mean(0), rtol=1e-12)
        # every step unmasks at least one position, and the block of 8 ends
        assert r["tokens_per_step"].sum() == shape.block_size
        assert np.all(r["t_step"] > 0) and np.all(r["t_moe"] > 0)
    # block top-k with one block per forward: exactly k experts in every layer at every step
    assert np.all(recs[0]["U"] == shape.top_k)
    assert np.all(recs[1]["U"] >= shape.top_k)
