"""The C ABI without a GPU: the library loads, exports every call include/dmoe.h declares,
sizes its workspace, and rejects bad arguments on the host before launching anything."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dmoe.h")


@pytest.fixture(scope="module")
def dm():
    import paper_2605_30876_gb300 as dm
    return dm


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dmoe_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(dm):
    lib = ctypes.CDLL(dm.LIB_PATH)
    names = declared_functions()
    assert len(names) >= 9
    for n in names:
        assert hasattr(lib, n), n


def test_abi_version_and_status_strings(dm):
    assert dm.dmoe_abi_version() == 2
    for s in range(7):
        assert dm.dmoe_status_string(s).startswith("DMOE_")


def _desc(dm, **kw):
    base = dict(d_model=2048, n_experts=256, top_k=8, d_ff=512, d_ff_shared=512, block_size=32,
                n_blocks=1, mode=dm.DMOE_ROUTE_BLOCK, top_p=0.0)
    base.update(kw)
    return dm.make_desc(**base)


def test_workspace_size_grows_with_tokens(dm):
    a = dm.dmoe_workspace_size(_desc(dm))
    b = dm.dmoe_workspace_size(_desc(dm, n_blocks=8))
    assert 0 < a < b
    # the split-K partials and scatter rows dominate; bounded well below the weights
    assert b < 64 * 2 ** 20


@pytest.mark.parametrize("kw,status", [
    (dict(top_k=0), 1), (dict(top_k=300), 1), (dict(n_experts=12), 2), (dict(n_experts=512), 2),
    (dict(top_k=17, n_experts=64), 2), (dict(d_model=200), 2), (dict(d_ff=100), 2),
    (dict(d_ff_shared=-1), 1), (dict(d_ff_shared=96), 2), (dict(block_size=0), 1),
    (dict(n_blocks=200), 2), (dict(mode=7), 1), (dict(top_p=-0.5), 1),
    (dict(top_p=float("nan")), 1), (dict(block_top_k=-1), 1), (dict(block_top_k=4), 1),
    (dict(block_top_k=17), 2), (dict(n_experts=16, top_k=2, block_top_k=24), 1),
])
def test_invalid_desc_is_rejected(dm, kw, status):
    with pytest.raises(dm.DmoeError) as ei:
        dm.dmoe_workspace_size(_desc(dm, **kw))
    assert ei.value.status == status


def test_block_top_k_accepted_and_struct_layout(dm):
    # block_top_k = 0 (= top_k), = top_k, and above top_k are valid
    for kw in (dict(), dict(block_top_k=8), dict(top_k=4, block_top_k=8),
               dict(top_k=1, block_top_k=16), dict(mode=dm.DMOE_ROUTE_TOKEN, top_k=4)):
        assert dm.dmoe_workspace_size(_desc(dm, **kw)) > 0
    # the C struct: nine 4-byte fields, block_top_k last
    assert ctypes.sizeof(dm.LayerDesc) == 40
    assert dm.LayerDesc.block_top_k.offset == 36


def test_null_and_misaligned_pointers_are_rejected_before_launch(dm):
    lib = dm._lib
    desc = _desc(dm)
    n = dm.dmoe_workspace_size(desc)
    fake = 1 << 40       # aligned, never dereferenced: the checks return first
    P = ctypes.c_void_p
    # null x
    st = lib.dmoe_router(ctypes.byref(desc), None, P(fake), None, P(fake), P(fake), None, None,
                         None, P(fake), n, None)
    assert st == 1
    # misaligned topk_idx
    st = lib.dmoe_router(ctypes.byref(desc), P(fake), P(fake), None, P(fake + 4), P(fake), None,
                         None, None, P(fake), n, None)
    assert st == 1
    # workspace too small
    st = lib.dmoe_router(ctypes.byref(desc), P(fake), P(fake), None, P(fake), P(fake), None,
                         None, None, P(fake), n - 1, None)
    assert st == 3
    # workspace not 256-B aligned
    st = lib.dmoe_dispatch(ctypes.byref(desc), P(fake), P(fake), P(fake), P(fake), P(fake),
                           P(fake), P(fake + 16), n, None)
    assert st == 1
    # shared expert declared but its weights missing
    st = lib.dmoe_moe_forward(ctypes.byref(desc), *([P(fake)] * 4), None, None, None,
                              *([P(fake)] * 7), P(fake), n, None)
    assert st == 1
    st = lib.dmoe_layer_forward(None, *([P(fake)] * 14), P(fake), n, None)
    assert st == 1
    # router preparation: misaligned W_r, workspace too small
    st = lib.dmoe_router_prepare(ctypes.byref(desc), P(fake + 4), P(fake), n, None)
    assert st == 1
    st = lib.dmoe_router_prepare(ctypes.byref(desc), P(fake), P(fake), n - 1, None)
    assert st == 3


def test_layer_forward_launch_count(dm):
    # decode-size forward: one routing launch (dispatch fused), the expert launch, the combine
    assert dm.dmoe_layer_forward_launches(_desc(dm)) == 3
    # 2048 tokens, block top-k: split of W_r, logits, softmax / top-k, Algorithm 1 (which
    # publishes the coresets); experts (which do the dispatch), combine
    assert dm.dmoe_layer_forward_launches(_desc(dm, n_blocks=64)) == 6
    # with p > 0 (a token keeps part of the coreset): dispatch (count, place with the
    # gather) before the experts
    assert dm.dmoe_layer_forward_launches(_desc(dm, n_blocks=64, top_p=0.6)) == 8
    assert dm.dmoe_layer_forward_launches(_desc(dm, n_blocks=64, mode=dm.DMOE_ROUTE_TOKEN)) == 7
    assert dm.dmoe_layer_forward_launches(_desc(dm, top_k=0)) == -1
