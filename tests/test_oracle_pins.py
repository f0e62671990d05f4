"""Pins of the CPU oracle against what Algorithm 1 (§4.2) and the mathematics fix.

Each test targets a plausible mistake: a dropped or extra term, a wrong sign, an index or
tie-break error, a transposed operand. None of them compares the oracle with itself.
"""
import itertools
import math

import numpy as np
import pytest

import oracle as O
from dmoe_synth import MoEShape, ROUTE_BLOCK, ROUTE_TOKEN, TINY, layer_inputs, to_numpy

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def f32(a):
    return np.asarray(a, np.float32)


def bits_of(a):
    """float values exactly representable in bf16 -> bf16 bit patterns (test helper)."""
    u = np.asarray(a, np.float32).view(np.uint32)
    assert np.all((u & 0xFFFF) == 0), "value not exact in bf16"
    return (u >> 16).astype(np.uint16)


# ------------------------------------------------------------------------------------
# Hand-worked case, derived from Algorithm 1 by hand (the paper prints no example).
# E=4, k=2, one block of B=2 tokens:
#   s_1 = [.5, .3, .15, .05]  -> TopKMask -> [.5, .3, 0, 0]
#   s_2 = [.1, .4, .2, .3]    -> TopKMask -> [0, .4, 0, .3]
#   S = [.5, .7, 0, .3], S~ = S/1.5 = [1/3, 7/15, 0, 1/5], sorted order 1, 0, 3, 2
#   p=0.6: running sums 7/15 < .6 <= 12/15 -> C = {1, 0}
#          R_1 = (0, 1), g = (.5/.8, .3/.8) = (.625, .375)
#          R_2 = (1, 0), g = (.4/.5, .1/.5) = (.8, .2);   unique experts {0, 1}
#   p=0.9: 12/15 < .9 <= 15/15 -> C = {1, 0, 3}; R_2 = (1, 3), g = (4/7, 3/7)  (= token routing)
#   p=0:   C has the floor size k=2 -> {1, 0}
#   token routing: R_1 = (0, 1), R_2 = (1, 3); unique {0, 1, 3}
# ------------------------------------------------------------------------------------
S_HAND = f32([[0.5, 0.3, 0.15, 0.05], [0.1, 0.4, 0.2, 0.3]])


def test_hand_case_block_p06():
    r = O.route_block(S_HAND, k=2, block_size=2, p=0.6)
    assert list(r.coresets[0]) == [1, 0]
    assert r.idx.tolist() == [[0, 1], [1, 0]]
    np.testing.assert_allclose(r.gate, [[0.625, 0.375], [0.8, 0.2]], rtol=1e-6)
    assert sorted(set(r.idx.ravel().tolist())) == [0, 1]


def test_hand_case_block_p09_equals_token():
    r = O.route_block(S_HAND, k=2, block_size=2, p=0.9)
    assert list(r.coresets[0]) == [1, 0, 3]
    assert r.idx.tolist() == [[0, 1], [1, 3]]
    np.testing.assert_allclose(r.gate[1], [4 / 7, 3 / 7], rtol=1e-6)
    t = O.route_token(S_HAND, 2)
    assert t.idx.tolist() == r.idx.tolist()
    assert sorted(set(t.idx.ravel().tolist())) == [0, 1, 3]


def test_hand_case_block_p0_floor():
    r = O.route_block(S_HAND, k=2, block_size=2, p=0.0)
    assert list(r.coresets[0]) == [1, 0]
    assert r.idx.tolist() == [[0, 1], [1, 0]]


def test_hand_case_aggregate_and_normalize():
    S = O.aggregate(S_HAND, 2)
    np.testing.assert_allclose(S, [0.5, 0.7, 0.0, 0.3], rtol=1e-7)
    np.testing.assert_allclose(O.normalize(S), [1 / 3, 7 / 15, 0.0, 1 / 5], rtol=1e-6)


def test_hand_case_through_router():
    """x_i one-hot, W_r row i = ln s_i, b = 0: the logits are ln s_i, the softmax gives s_i
    back, and routing must reproduce the hand case. A transposed W_r or x fails here."""
    d, E = 5, 4
    x = np.zeros((2, d), np.float32)
    x[0, 0] = 1.0
    x[1, 3] = 1.0
    w_r = np.full((d, E), 7.0, np.float32)      # rows not selected by x must not matter
    w_r[0] = np.log(S_HAND[0])
    w_r[3] = np.log(S_HAND[1])
    s = O.router_scores(O.router_logits(bits_of(x), w_r, np.zeros(E, np.float32)))
    np.testing.assert_allclose(s, S_HAND, rtol=1e-6)
    r = O.route(bits_of(x), w_r, None, 2, ROUTE_BLOCK, 2, 0.6)
    assert r.idx.tolist() == [[0, 1], [1, 0]]


# ------------------------------------------------------------------------------------
# Fewer experts per token (App. A): TopKMask and the floor at k_mask, final TopK at k.
# Hand case, S_HAND with k_mask = 3, k = 2, p = 0:
#   TopKMask(s_1, 3) = [.5, .3, .15, 0], TopKMask(s_2, 3) = [0, .4, .2, .3]
#   S = [.5, .7, .35, .3] -> sorted order 1, 0, 2, 3 -> floor 3: C = {1, 0, 2}
#   R_1 = (0, 1), g = (.625, .375); R_2 inside {1, 0, 2} = (1, 2), g = (2/3, 1/3)
#   (with TopKMask at k = 2 the coreset would be {1, 0} and R_2 = (1, 0); token routing
#   gives R_2 = (1, 3): the case separates all three)
# k_mask = 2, k = 1: p = 0 -> C = {1, 0}, R_1 = (0,), R_2 = (1,), gates 1;
#                    p = .9 -> C = {1, 0, 3}, the same R (the coreset only grows)
# ------------------------------------------------------------------------------------
def test_hand_case_fewer_experts_k_mask3_k2():
    r = O.route_block(S_HAND, k=2, block_size=2, p=0.0, k_mask=3)
    assert list(r.coresets[0]) == [1, 0, 2]
    assert r.idx.tolist() == [[0, 1], [1, 2]]
    np.testing.assert_allclose(r.gate, [[0.625, 0.375], [2 / 3, 1 / 3]], rtol=1e-6)


@pytest.mark.parametrize("p,core", [(0.0, [1, 0]), (0.9, [1, 0, 3])])
def test_hand_case_fewer_experts_k1(p, core):
    r = O.route_block(S_HAND, k=1, block_size=2, p=p, k_mask=2)
    assert list(r.coresets[0]) == core
    assert r.idx.tolist() == [[0], [1]]
    np.testing.assert_allclose(r.gate, [[1.0], [1.0]], rtol=0)


def test_near_tie_mask_flip_lists_the_other_coreset():
    """k = 1, p = 0, B = 2: token 1 ties experts 0 and 1 exactly; TopKMask keeps 0 (lower
    index), S = [.4, 0, .35, 0], C = {0}. Keeping 1 instead gives S = [0, .4, .35, 0] and
    C = {1}: the block's margin is 0 and {1} is listed as the alternative. A third token
    pattern with no tie leaves the margin at the boundary gap and lists nothing."""
    s = f32([[0.4, 0.4, 0.1, 0.1], [0.1, 0.3, 0.35, 0.25]])
    r = O.route_block(s, k=1, block_size=2, p=0.0)
    assert list(r.coresets[0]) == [0]
    assert r.coreset_margin[0] == 0.0
    assert [a.tolist() for a in r.coreset_alts[0]] == [[1]]
    s2 = f32([[0.5, 0.3, 0.1, 0.1], [0.1, 0.3, 0.35, 0.25]])
    r2 = O.route_block(s2, k=1, block_size=2, p=0.0)
    assert r2.coreset_alts[0] == []
    np.testing.assert_allclose(r2.coreset_margin[0], (0.5 - 0.35) / 0.85, rtol=1e-6)


def test_near_tie_boundary_and_p_crossing_alternatives():
    """S~ with an exact tie at the floor boundary lists the swapped coreset; p set exactly on
    a running sum lists the coreset with one expert more."""
    C = O.top_p(f32([0.4, 0.3, 0.3, 0.0]), 0.0, 2)
    assert C.ids.tolist() == [0, 1] and C.margin == 0.0
    assert [a.tolist() for a in C.alts] == [[0, 2]]
    St = f32([0.5, 0.25, 0.25, 0.0])               # running sums .5, .75, 1 exact in fp32
    C = O.top_p(St, 0.75, 1)
    assert C.ids.tolist() == [0, 1] and C.margin == 0.0
    assert [a.tolist() for a in C.alts] == [[0, 2], [0, 1, 2]]


@pytest.mark.parametrize("E,km,k,p", [(8, 3, 2, 0.0), (8, 4, 1, 0.5), (10, 4, 3, 0.8),
                                      (6, 5, 2, 1.0)])
def test_fewer_experts_brute_force(E, km, k, p):
    """R_i is the k-subset of the coreset with the largest score sum (brute force over
    all subsets), listed by descending score; the coreset is the k_mask one."""
    rng = np.random.default_rng(100 + E + km)
    B, nb = 4, 3
    s = f32(rng.dirichlet(np.ones(E), size=B * nb))
    r = O.route_block(s, k, B, p, k_mask=km)
    full = O.route_block(s, km, B, p)
    for b in range(nb):
        assert np.array_equal(r.coresets[b], full.coresets[b])   # the coreset uses k_mask
        C = r.coresets[b].tolist()
        assert len(C) >= km
        for i in range(b * B, (b + 1) * B):
            best = max(itertools.combinations(C, k), key=lambda c: s[i, list(c)].astype(float).sum())
            assert set(r.idx[i].tolist()) == set(best)
            v = s[i, r.idx[i]]
            assert all(v[j] > v[j + 1] for j in range(k - 1))
            assert abs(r.gate[i].sum() - 1.0) <= 1e-12


@pytest.mark.parametrize("p", [0.0, 0.6])
def test_fewer_experts_is_prefix_of_full_routing(p):
    """Inside one coreset TopK(., k) is the first k of TopK(., k_mask): the same ids in
    the same order, gates renormalised over the k."""
    shape = TINY.with_(top_k=4, n_blocks=4, bias_scale=0.5)
    s = _scores(shape, 21)
    full = O.route_block(s, 4, shape.block_size, p)
    for k in (1, 2, 3):
        r = O.route_block(s, k, shape.block_size, p, k_mask=4)
        assert np.array_equal(r.idx, full.idx[:, :k])
        w = s[np.arange(shape.T)[:, None], full.idx[:, :k]].astype(np.float64)
        np.testing.assert_allclose(r.gate, w / w.sum(1, keepdims=True), rtol=1e-12)


# ------------------------------------------------------------------------------------
# Router closed forms
# ------------------------------------------------------------------------------------
def test_softmax_closed_form():
    L = f32([[0.0, math.log(2.0), math.log(3.0)]])
    np.testing.assert_allclose(O.router_scores(L), [[1 / 6, 2 / 6, 3 / 6]], rtol=1e-6)


def test_softmax_shift_invariance_and_bias_sign():
    rng = np.random.default_rng(1)
    L = f32(rng.standard_normal((3, 7)))
    np.testing.assert_allclose(O.router_scores(L), O.router_scores(L + f32(5.0)), rtol=1e-6)
    # a positive bias on one expert raises its score (catches a sign error on b)
    x = bits_of(np.eye(3, 4, dtype=np.float32))
    w = f32(rng.standard_normal((4, 7)))
    b = np.zeros(7, np.float32)
    b[2] = 3.0
    s0 = O.router_scores(O.router_logits(x, w, None))
    s1 = O.router_scores(O.router_logits(x, w, b))
    assert np.all(s1[:, 2] > s0[:, 2])
    np.testing.assert_allclose(s1.sum(1), 1.0, rtol=1e-6)


def test_router_logits_closed_form():
    # x = [1, 2, 0] (exact in bf16), W_r [3, 2]: logits = [1*1 + 2*3, 1*2 + 2*4] + b
    x = bits_of([[1.0, 2.0, 0.0]])
    w = f32([[1.0, 2.0], [3.0, 4.0], [100.0, -100.0]])
    L = O.router_logits(x, w, f32([0.5, -0.5]))
    np.testing.assert_array_equal(L, f32([[7.5, 9.5]]))


# ------------------------------------------------------------------------------------
# Brute force
# ------------------------------------------------------------------------------------
@pytest.mark.parametrize("E,k", [(16, 2), (10, 3), (7, 1)])
def test_topk_brute_force(E, k):
    rng = np.random.default_rng(E * 10 + k)
    for _ in range(40):
        v = f32(rng.random(E))
        v[rng.integers(E)] = v[rng.integers(E)]        # plant a tie now and then
        best = max(itertools.combinations(range(E), k),
                   key=lambda c: (sum(float(v[i]) for i in c), [-i for i in c]))
        got = O.topk_desc(v, k)
        assert sorted(got.tolist()) == sorted(best)
        assert all(v[got[j]] >= v[got[j + 1]] for j in range(k - 1))


def test_topk_tie_goes_to_lower_index():
    assert O.topk_desc(f32([0.2, 0.5, 0.5, 0.1]), 1).tolist() == [1]
    assert O.topk_desc(f32([0.3, 0.3, 0.3]), 2).tolist() == [0, 1]



def test_topk_margins_hand_values():
    """TopK margins (reading R11): v = [.5, .3, .29, .1], k = 2 -> the set decision is .30
    vs .29 (margin .01), the slot order .5 vs .3 (margin .2). A margin that is always 0
    would turn every token ambiguous; one taken from the wrong end would hide near ties."""
    sm, om = O.topk_margins(np.array([0.5, 0.3, 0.29, 0.1]), 2)
    assert sm == pytest.approx(0.01, abs=1e-15)
    assert om == pytest.approx(0.2, abs=1e-15)
    # the same values permuted: margins depend on values, not positions
    sm2, om2 = O.topk_margins(np.array([0.1, 0.29, 0.5, 0.3]), 2)
    assert (sm2, om2) == (sm, om)
    # k = 3: set .29 vs .1 = .19, order min(.5 - .3, .3 - .29) = .01
    sm3, om3 = O.topk_margins(np.array([0.5, 0.3, 0.29, 0.1]), 3)
    assert sm3 == pytest.approx(0.19, abs=1e-15) and om3 == pytest.approx(0.01, abs=1e-15)
    # k = 1: no order decision; no (k+1)-th finite candidate -> infinite set margin
    assert O.topk_margins(np.array([0.7, 0.2]), 1) == (pytest.approx(0.5), float("inf"))
    assert O.topk_margins(np.array([0.7, -np.inf, -np.inf]), 1)[0] == float("inf")
    # inside a coreset (MaskOutside fills -inf): only the members compete
    sC = O.mask_outside(f32([0.5, 0.3, 0.29, 0.1]), np.array([0, 3, 1]))
    sm4, om4 = O.topk_margins(sC, 2)
    assert sm4 == pytest.approx(float(f32(0.3)) - float(f32(0.1)), abs=1e-12)
    assert om4 == pytest.approx(float(f32(0.5)) - float(f32(0.3)), abs=1e-12)


def test_topk_margins_order_margin_alone_can_be_near():
    """A token whose set is clear but whose first two slots nearly tie: the order margin is
    below 1e-5 while the set margin is large, so the parity check may accept either slot
    order but must still demand the same set."""
    v = np.array([0.4, 0.4 - 4e-6, 0.1, 0.05])
    sm, om = O.topk_margins(v, 2)
    assert sm == pytest.approx(0.4 - 4e-6 - 0.1, abs=1e-15)
    assert om == pytest.approx(4e-6, abs=1e-15)
    assert om < O.NEAR_TIE <= sm


def test_gates_for_hand_values():
    """R8 gates of a given selection, by hand: token 0 routed to (2, 0) with s = [.5, .2,
    .3] -> (.3/.8, .5/.8) = (.375, .625); token 1 routed to (1, 2) with s = [.1, .6, .3] ->
    (.6/.9, .3/.9). A transposed token index or a sum over the wrong row fails here."""
    s = f32([[0.5, 0.2, 0.3], [0.1, 0.6, 0.3]])
    idx = np.array([[2, 0], [1, 2]], np.int32)
    g = O.gates_for(s, idx)
    s64 = s.astype(np.float64)
    exp0 = [s64[0, 2] / (s64[0, 2] + s64[0, 0]), s64[0, 0] / (s64[0, 2] + s64[0, 0])]
    exp1 = [s64[1, 1] / (s64[1, 1] + s64[1, 2]), s64[1, 2] / (s64[1, 1] + s64[1, 2])]
    np.testing.assert_allclose(g, [exp0, exp1], rtol=0, atol=1e-15)
    np.testing.assert_allclose(g, [[0.375, 0.625], [2 / 3, 1 / 3]], rtol=0, atol=1e-7)
    assert g.dtype == np.float64 and np.allclose(g.sum(axis=1), 1.0, atol=1e-15)
    # the hand case of Algorithm 1 above: p = 0.6 gates through gates_for
    r = O.route_block(S_HAND, 2, 2, 0.6)
    np.testing.assert_allclose(O.gates_for(S_HAND, r.idx), [[0.625, 0.375], [0.8, 0.2]],
                               rtol=0, atol=1e-7)

@pytest.mark.parametrize("E", [5, 8, 10])
def test_top_p_brute_force(E):
    """The p rule takes the fewest experts whose normalised mass reaches p (checked against
    every subset), and the floor raises that count to k."""
    rng = np.random.default_rng(E)
    for trial in range(30):
        raw = rng.random(E) ** 3
        raw[rng.random(E) < 0.2] = 0.0
        if np.count_nonzero(raw) < 3:
            continue
        St = O.normalize(raw)
        for p in (0.3, 0.5, 0.6, 0.8, 0.95):
            for k in (1, 2, 3):
                C = O.top_p(St, p, k)
                if C.margin < 1e-5:
                    continue
                best = None
                for m in range(1, E + 1):
                    if any(sum(float(St[i]) for i in c) >= p
                           for c in itertools.combinations(range(E), m)):
                        best = m
                        break
                assert C.m_p == best
                assert len(C.ids) == max(best, k)
                # the chosen prefix is a heaviest subset of its size
                heaviest = max(sum(float(St[i]) for i in c)
                               for c in itertools.combinations(range(E), len(C.ids)))
                assert abs(sum(float(St[i]) for i in C.ids) - heaviest) < 1e-6


def test_top_p_p_ge_1_takes_all_nonzero():
    St = O.normalize(f32([0.5, 0.0, 0.25, 0.25]))
    assert sorted(O.top_p(St, 1.0, 1).ids.tolist()) == [0, 2, 3]


# ------------------------------------------------------------------------------------
# Invariants of Algorithm 1 on seeded random inputs
# ------------------------------------------------------------------------------------
def _scores(shape, seed):
    inp = to_numpy(layer_inputs(shape, seed=seed, with_weights=False))
    return O.router_scores(O.router_logits(inp["x"], inp["w_r"], inp["bias"]))


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_block_size_one_equals_token_routing(seed):
    shape = TINY.with_(block_size=1, n_blocks=16)
    s = _scores(shape, seed)
    tok = O.route_token(s, shape.top_k)
    for p in (0.0, 0.3, 0.6, 1.0):
        blk = O.route_block(s, shape.top_k, 1, p)
        assert np.array_equal(blk.idx, tok.idx)
        np.testing.assert_allclose(blk.gate, tok.gate, rtol=1e-12)


@pytest.mark.parametrize("seed", [0, 3])
def test_p_one_equals_token_routing(seed):
    shape = TINY.with_(block_size=8, n_blocks=4)
    s = _scores(shape, seed)
    assert np.array_equal(O.route_block(s, shape.top_k, 8, 1.0).idx,
                          O.route_token(s, shape.top_k).idx)


@pytest.mark.parametrize("shape", [TINY, TINY.with_(top_k=4, block_size=16, n_blocks=3,
                                                     bias_scale=1.0)])
def test_p_zero_block_top_k(shape):
    s = _scores(shape, 5)
    k, B = shape.top_k, shape.block_size
    r = O.route_block(s, k, B, 0.0)
    for b in range(shape.n_blocks):
        sets = {tuple(sorted(r.idx[i].tolist())) for i in range(b * B, (b + 1) * B)}
        assert len(sets) == 1                       # the whole block shares one group
        assert len(set(r.idx[b * B:(b + 1) * B].ravel().tolist())) == k
        assert sorted(r.coresets[b].tolist()) == sorted(sets.pop())


@pytest.mark.parametrize("p", [0.0, 0.4, 0.6, 0.8, 1.0])
def test_routing_invariants(p):
    shape = TINY.with_(n_blocks=6, bias_scale=0.5)
    s = _scores(shape, 11)
    k, B = shape.top_k, shape.block_size
    r = O.route_block(s, k, B, p)
    assert r.idx.shape == (shape.T, k)
    for t in range(shape.T):
        row = r.idx[t].tolist()
        assert len(set(row)) == k                     # k distinct experts per token
        assert set(row) <= set(r.coresets[t // B].tolist())   # R_i inside the coreset
        vals = s[t, r.idx[t]]
        assert all(vals[j] >= vals[j + 1] for j in range(k - 1))
        assert abs(r.gate[t].sum() - 1.0) <= 1e-12
        assert np.all(r.gate[t] > 0)
    U = len(set(r.idx.ravel().tolist()))
    assert k <= U <= min(shape.n_experts, shape.n_blocks * len(r.coresets[0]) * 99)


def test_coreset_size_grows_with_p():
    shape = TINY.with_(n_blocks=5, bias_scale=0.5)
    s = _scores(shape, 4)
    prev = None
    for p in (0.0, 0.2, 0.4, 0.6, 0.8, 0.95, 1.0):
        sizes = [len(c) for c in O.route_block(s, shape.top_k, shape.block_size, p).coresets]
        if prev is not None:
            assert all(a >= b for a, b in zip(sizes, prev))
        prev = sizes


def test_identical_tokens_block_equals_token_topk():
    s = np.repeat(_scores(TINY.with_(n_blocks=1, block_size=1), 2), 8, axis=0)
    r = O.route_block(s, 2, 8, 0.6)
    t = O.route_token(s, 2)
    assert np.array_equal(r.idx, t.idx)


# ------------------------------------------------------------------------------------
# Dispatch
# ------------------------------------------------------------------------------------
def test_dispatch_hand_case():
    idx = np.array([[2, 0], [0, 1], [2, 1]], np.int32)
    d = O.dispatch(idx)
    assert d.unique_ids.tolist() == [0, 1, 2]
    assert d.offsets.tolist() == [0, 2, 4, 6]
    assert d.rows.tolist() == [1, 2, 3, 5, 0, 4]
    assert d.pos.tolist() == [4, 0, 1, 2, 5, 3]


def test_dispatch_invariants():
    rng = np.random.default_rng(7)
    T, k, E = 50, 4, 23
    idx = np.stack([rng.choice(E, k, replace=False) for _ in range(T)]).astype(np.int32)
    d = O.dispatch(idx)
    assert np.array_equal(d.unique_ids, np.unique(idx))
    assert sorted(d.rows.tolist()) == list(range(T * k))
    assert d.offsets[0] == 0 and d.offsets[-1] == T * k
    for u, e in enumerate(d.unique_ids):
        seg = d.rows[d.offsets[u]:d.offsets[u + 1]]
        assert np.all(idx.ravel()[seg] == e)
        assert np.all(np.diff(seg // k) > 0)          # tokens ascending within an expert
    assert np.array_equal(d.rows[d.pos], np.arange(T * k))


# ------------------------------------------------------------------------------------
# Expert execution
# ------------------------------------------------------------------------------------
SILU2 = 1.7615941559557646      # silu(2) = 2 / (1 + e^-2)


def test_swiglu_closed_form():
    """x = e_1, d=4, I=2. g = W_gate[:,1] = [2, 0], u = W_up[:,1] = [.5, 3];
    h = [silu(2)*.5, silu(0)*3] = [silu(2)/2, 0]; y = W_down h."""
    d, I = 4, 2
    x = np.zeros((1, d))
    x[0, 1] = 1.0
    wg = np.zeros((I, d))
    wg[:, 1] = [2.0, 0.0]
    wg[:, 0] = [50.0, -50.0]                 # a transposed operand would pick these up
    wu = np.zeros((I, d))
    wu[:, 1] = [0.5, 3.0]
    wd = np.array([[1.0, 0.0], [0.0, 1.0], [1.0, 1.0], [2.0, -1.0]])
    y = O.swiglu_ffn(x, wg, wu, wd)
    h0 = SILU2 * 0.5
    np.testing.assert_allclose(y, [[h0, 0.0, h0, 2 * h0]], rtol=1e-14)


def _tiny_layer(seed=0, **kw):
    shape = TINY.with_(**kw)
    return shape, to_numpy(layer_inputs(shape, seed=seed))


def test_single_expert_k1_is_plain_ffn():
    shape, inp = _tiny_layer(n_experts=1, top_k=1, n_blocks=1)
    y, r, _ = O.layer_forward(inp, 1, ROUTE_BLOCK, shape.block_size, 0.6)
    assert np.all(r.idx == 0) and np.allclose(r.gate, 1.0)
    x = O.bf16_bits_to_f64(inp["x"])
    ref = O.swiglu_ffn(x, O.bf16_bits_to_f64(inp["w_gate"][0]), O.bf16_bits_to_f64(inp["w_up"][0]),
                       O.bf16_bits_to_f64(inp["w_down"][0]))
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-15)


def test_identical_experts_any_routing():
    """All experts equal: gates sum to one, so y = FFN(x) whatever the routing."""
    shape, inp = _tiny_layer(seed=3)
    for key in ("w_gate", "w_up", "w_down"):
        inp[key] = np.repeat(inp[key][:1], shape.n_experts, axis=0)
    x = O.bf16_bits_to_f64(inp["x"])
    ref = O.swiglu_ffn(x, O.bf16_bits_to_f64(inp["w_gate"][0]), O.bf16_bits_to_f64(inp["w_up"][0]),
                       O.bf16_bits_to_f64(inp["w_down"][0]))
    for mode in (ROUTE_TOKEN, ROUTE_BLOCK):
        y, _, _ = O.layer_forward(inp, shape.top_k, mode, shape.block_size, 0.6)
        np.testing.assert_allclose(y, ref, rtol=1e-10, atol=1e-13)


def test_expert_permutation_invariance():
    """Relabelling experts (weights, router columns and bias together; new expert j is old
    expert perm[j]) maps the selected ids through perm and leaves y unchanged."""
    shape, inp = _tiny_layer(seed=4, bias_scale=0.5)
    perm = np.random.default_rng(9).permutation(shape.n_experts)
    inp2 = dict(inp)
    inp2["w_r"] = inp["w_r"][:, perm]
    inp2["bias"] = inp["bias"][perm]
    for key in ("w_gate", "w_up", "w_down"):
        inp2[key] = inp[key][perm]
    for mode, p in ((ROUTE_TOKEN, 0.0), (ROUTE_BLOCK, 0.6), (ROUTE_BLOCK, 0.0)):
        y1, r1, _ = O.layer_forward(inp, shape.top_k, mode, shape.block_size, p)
        y2, r2, _ = O.layer_forward(inp2, shape.top_k, mode, shape.block_size, p)
        assert np.array_equal(np.sort(r1.idx, 1), np.sort(perm[r2.idx], 1))
        np.testing.assert_allclose(y1, y2, rtol=1e-10, atol=1e-13)


def test_shared_only_when_routed_weights_zero():
    shape, inp = _tiny_layer(seed=5, d_ff_shared=64)
    for key in ("w_gate", "w_up", "w_down"):
        inp[key] = np.zeros_like(inp[key])
    y, _, _ = O.layer_forward(inp, shape.top_k, ROUTE_BLOCK, shape.block_size, 0.6)
    x = O.bf16_bits_to_f64(inp["x"])
    ref = O.swiglu_ffn(x, O.bf16_bits_to_f64(inp["ws_gate"]), O.bf16_bits_to_f64(inp["ws_up"]),
                       O.bf16_bits_to_f64(inp["ws_down"]))
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-15)
    assert np.abs(ref).max() > 1e-3


def test_gate_weighted_combine_two_experts():
    """Two experts whose outputs differ by a known factor: expert 1 = 2 x expert 0 through
    W_down, so y = (g0 + 2 g1) * FFN_0(x) for a token routed to both."""
    shape, inp = _tiny_layer(seed=6, n_experts=2, top_k=2, n_blocks=1)
    inp["w_gate"][1] = inp["w_gate"][0]
    inp["w_up"][1] = inp["w_up"][0]
    wd0 = O.bf16_bits_to_f64(inp["w_down"][0])
    inp["w_down"][1] = bits_of((2.0 * wd0).astype(np.float32))
    y, r, _ = O.layer_forward(inp, 2, ROUTE_TOKEN, shape.block_size, 0.0)
    x = O.bf16_bits_to_f64(inp["x"])
    f0 = O.swiglu_ffn(x, O.bf16_bits_to_f64(inp["w_gate"][0]), O.bf16_bits_to_f64(inp["w_up"][0]), wd0)
    g = np.zeros((shape.T, 2))
    for t in range(shape.T):
        for j in range(2):
            g[t, r.idx[t, j]] = r.gate[t, j]
    np.testing.assert_allclose(y, (g[:, :1] + 2 * g[:, 1:]) * f0, rtol=1e-10, atol=1e-13)
