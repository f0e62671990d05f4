"""CPU oracle of the dMoE MoE-layer forward (arXiv 2605.30876, "dLLMs with Learnable Block Experts").

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline /
reference legs of ``bench.py`` may import this module. The CUDA library
(``paper_2605_30876_gb300``) never imports it, and this module imports nothing of the
library: the two share only the seeded input generator ``dmoe_synth``.

Plain, slow NumPy in float64, written step by step after Algorithm 1 (Block-Level Expert
Routing) and the prose of §4.2, so that each step can be checked against the paper by eye.
The parts the paper leaves open are fixed by the readings below; each function names the
reading it implements.

Readings (the paper is silent or ambiguous here):
  R1  router:   s_i = softmax(t_i W_r + b) over the |E| experts; logits are summed in
                float64 and rounded once to fp32, the softmax is taken in float64 from the
                fp32 logits and rounded to fp32 (the router works in fp32).
  R2  TopKMask: keeps the k largest score *values* of s_i and zeroes the rest.
  R3  aggregation: the operator of §4.2 is the sum (Algorithm 1 adds the masked scores).
  R4  Normalize: L1 normalisation, S~ = S / sum_e S[e].
  R5  Top-P:    sort S~ descending (equal values: lower expert index first); the coreset is
                the shortest prefix whose running fp32 sum, in sorted order, reaches p (the
                crossing element is included). Zero-score experts are never added by the p
                rule. p >= 1 selects every expert with a nonzero block score.
  R6  floor:    a coreset shorter than k is extended along the sorted order to k entries,
                so every token keeps exactly k experts (p = 0 gives |C| = k: "block top-k").
  R7  MaskOutside fills -inf; TopK breaks ties towards the lower expert index and lists
                the k experts by descending score.
  R8  gates:    g_ij = s_i[R_ij] / sum_j s_i[R_ij] (they sum to 1); the shared expert is
                ungated (weight 1).
  R9  dispatch: unique experts ascending; the expert->(token, slot) list is ordered by
                expert, then token; rows hold t*k + slot; pos is its inverse.
  R10 expert:   SwiGLU, y_e(x) = W_down (silu(W_gate x) * (W_up x)), fp64 throughout, with
                the intermediate kept unrounded. Token-level routing (the "Original"
                baseline of §5.1) is R_i = TopK(s_i, k) with the same gates.
  R17 fewer experts per token (the direction App. A names, not evaluated in the paper):
                Algorithm 1 runs with k_mask in TopKMask and in the floor, and the final
                TopK inside the coreset keeps k < k_mask experts per token, gates R8 over
                those k. k_mask = k is Algorithm 1 itself.

Decisions (a top-k, the coreset boundary) are taken on fp32 values, as the router's
fp32 output is the input of Algorithm 1. Each decision also reports a *margin*: how far
the decision is from flipping, in the units of the compared quantity. A decision with a
margin below NEAR_TIE = 1e-5 may legitimately come out either way on the GPU; for a block
whose coreset decision is that close, the coresets that one such flip reaches are listed
too (Routing.coreset_alts), so that a GPU result can be checked against them.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np

F32 = np.float32
F64 = np.float64

ROUTE_TOKEN = 0
ROUTE_BLOCK = 1
NEAR_TIE = 1e-5        # decisions closer than this may come out either way on the GPU


# ----------------------------------------------------------------------------------------
# storage conversion
# ----------------------------------------------------------------------------------------
def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64. Exact: a bf16 value is the upper half of an
    IEEE binary32 word."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(F64)


# ----------------------------------------------------------------------------------------
# router (§4.2, s_i = Router(t_i); reading R1)
# ----------------------------------------------------------------------------------------
def router_logits(x_bits: np.ndarray, w_r: np.ndarray, bias: Optional[np.ndarray]) -> np.ndarray:
    """Router logits t_i W_r + b for every token: [T,d] bf16 x [d,E] fp32 (+ [E]) -> [T,E] fp32.
    Products and sums in float64, one rounding to fp32 at the end (R1)."""
    L = bf16_bits_to_f64(x_bits) @ np.asarray(w_r, F64)
    if bias is not None:
        L = L + np.asarray(bias, F64)[None, :]
    return L.astype(F32)


def router_scores(logits32: np.ndarray) -> np.ndarray:
    """Token-level expert scores s_i (§4.2): softmax over the experts of each row, taken in
    float64 from the fp32 logits (max-subtracted) and rounded to fp32 (R1)."""
    z = np.asarray(logits32, F32).astype(F64)
    z = z - z.max(axis=-1, keepdims=True)
    e = np.exp(z)
    s = e / e.sum(axis=-1, keepdims=True)
    return s.astype(F32)


# ----------------------------------------------------------------------------------------
# top-k helpers (reading R7)
# ----------------------------------------------------------------------------------------
def sort_desc(v: np.ndarray) -> np.ndarray:
    """All indices of v ordered by value, largest first; equal values keep the lower index
    first (stable sort of -v)."""
    return np.argsort(-np.asarray(v, F64), kind="stable")


def topk_desc(v: np.ndarray, k: int) -> np.ndarray:
    """TopK: the k largest entries, largest first, ties towards the lower index (R7)."""
    return sort_desc(v)[:k]


def topk_margins(v: np.ndarray, k: int) -> (float, float):
    """(set margin, order margin) of TopK(v, k): the gap between the k-th and (k+1)-th
    largest finite values (inf if there is no (k+1)-th candidate), and the smallest gap
    between consecutive entries of the top k."""
    v64 = np.asarray(v, F64)
    order = sort_desc(v64)
    vals = v64[order]
    finite = np.isfinite(vals)
    n_cand = int(finite.sum())
    set_margin = float(vals[k - 1] - vals[k]) if n_cand > k else float("inf")
    if k > 1:
        order_margin = float(np.min(vals[: k - 1] - vals[1:k]))
    else:
        order_margin = float("inf")
    return set_margin, order_margin


def topk_mask(s: np.ndarray, k: int) -> np.ndarray:
    """TopKMask(s_i, k) of Algorithm 1 (R2): keep the k largest scores, zero elsewhere."""
    keep = topk_desc(s, k)
    out = np.zeros_like(np.asarray(s, F32))
    out[keep] = np.asarray(s, F32)[keep]
    return out


def renormalize(s: np.ndarray, R: np.ndarray) -> np.ndarray:
    """Gate weights over the routed set R_i (R8): s_i[R] / sum s_i[R], in float64."""
    v = np.asarray(s, F32)[R].astype(F64)
    return v / v.sum()


# ----------------------------------------------------------------------------------------
# block-level routing (Algorithm 1, §4.2)
# ----------------------------------------------------------------------------------------
def aggregate(s_block: np.ndarray, k: int) -> np.ndarray:
    """S_block of Algorithm 1: start from zero and add TopKMask(s_i, k) for every token i of
    the block (R2, R3). float64 sum of the fp32 masked scores."""
    S = np.zeros(s_block.shape[1], F64)
    for i in range(s_block.shape[0]):
        S = S + topk_mask(s_block[i], k).astype(F64)
    return S


def normalize(S: np.ndarray) -> np.ndarray:
    """Normalize(S_block) of Algorithm 1 (R4): L1 normalisation, rounded to fp32 because the
    coreset decision that follows is taken in fp32."""
    S = np.asarray(S, F64)
    return (S / S.sum()).astype(F32)


@dataclasses.dataclass
class Coreset:
    ids: np.ndarray       # int32, sorted by S~ descending (ties: lower index first)
    m_p: int              # length of the prefix the p rule alone selects
    margin: float         # distance of the decision from flipping (see coreset_margin)
    alts: List[np.ndarray] = dataclasses.field(default_factory=list)
    # the coresets one flip of a decision closer than NEAR_TIE reaches (see coreset_margin)


def top_p(S_tilde: np.ndarray, p: float, k: int) -> Coreset:
    """C = TopP(S~_block, p) of Algorithm 1 with the readings R5 and R6.

    Sort descending; the p rule takes the shortest prefix whose running fp32 sum reaches
    fp32(p) (p >= 1: every nonzero entry); the floor extends it to k entries."""
    St = np.asarray(S_tilde, F32)
    order = sort_desc(St)
    vals = St[order]
    nnz = int(np.count_nonzero(vals > 0))
    if p >= 1.0:
        m = nnz
        cum = None
    else:
        cum = np.cumsum(vals, dtype=F32)          # sequential fp32 running sum
        hit = np.nonzero(cum >= F32(p))[0]
        m = int(hit[0]) + 1 if hit.size else nnz
        m = min(m, nnz)
    size = max(m, k)
    ids = order[:size].astype(np.int32)
    C = Coreset(ids=ids, m_p=m, margin=coreset_margin(vals, cum, p, m, k, size))
    # one flip of a near decision: the boundary pair swapped, one expert more (the sum
    # falls just short of p) or one fewer (the sum reaches p one step earlier)
    v = np.asarray(vals, F64)
    if size < v.size and v[size - 1] - v[size] < NEAR_TIE:
        C.alts.append(np.concatenate([order[:size - 1], order[size:size + 1]]).astype(np.int32))
    if cum is not None and p > 0.0 and m >= k:
        pp = float(F32(p))
        if float(cum[m - 1]) - pp < NEAR_TIE and size < v.size and v[size] > 0:
            C.alts.append(order[:size + 1].astype(np.int32))
        if m > k and m >= 2 and pp - float(cum[m - 2]) < NEAR_TIE:
            C.alts.append(order[:size - 1].astype(np.int32))
    return C


def coreset_margin(vals: np.ndarray, cum: Optional[np.ndarray], p: float, m: int, k: int,
                   size: int) -> float:
    """How far the coreset decision is from flipping.

    * boundary gap: S~ of the last member minus S~ of the first non-member (a near tie
      there can swap which expert is in);
    * p crossing: when the p rule set the size (m >= k), the running sum at the crossing
      minus p (a GPU sum just below p would take one more expert) and, when m > k, p minus
      the running sum one step earlier (one expert fewer)."""
    v = np.asarray(vals, F64)
    margin = float("inf")
    if size < v.size:
        margin = min(margin, float(v[size - 1] - v[size]))
    if cum is not None and p > 0.0 and m >= k:
        pp = float(F32(p))
        margin = min(margin, float(cum[m - 1]) - pp)
        if m > k and m >= 2:
            margin = min(margin, pp - float(cum[m - 2]))
    return margin


def mask_outside(s: np.ndarray, C: np.ndarray) -> np.ndarray:
    """MaskOutside(s_i, C) of Algorithm 1 (R7): -inf for experts outside the coreset."""
    out = np.full(np.asarray(s).shape, -np.inf, F64)
    out[C] = np.asarray(s, F32)[C].astype(F64)
    return out


# ----------------------------------------------------------------------------------------
# full routing of one forward
# ----------------------------------------------------------------------------------------
@dataclasses.dataclass
class Routing:
    idx: np.ndarray                 # int32 [T,k] routed experts R_i, by descending s_i
    gate: np.ndarray                # float64 [T,k] renormalised gates
    coresets: List[np.ndarray]      # per block: coreset ids (block mode), [] in token mode
    set_margin: np.ndarray          # float64 [T]: margin of the set decision of token i
    order_margin: np.ndarray        # float64 [T]: margin of the slot order of token i
    coreset_margin: np.ndarray      # float64 [n_blocks] (inf in token mode)
    scores: np.ndarray              # fp32 [T,E] router scores s_i
    coreset_alts: List[List[np.ndarray]] = dataclasses.field(default_factory=list)
    # per block: the coresets one near-tie flip reaches ([] per block in token mode)


def topk_in_coreset(s_i: np.ndarray, C: np.ndarray, k: int):
    """MaskOutside then TopK for one token (R7): (R_i, set margin, order margin)."""
    sC = mask_outside(s_i, C)
    sm, om = topk_margins(sC, k)
    return topk_desc(sC, k), sm, om


def route_token(s: np.ndarray, k: int) -> Routing:
    """Token-level routing (the "Original" baseline, §5.1): R_i = TopK(s_i, k), gates R8."""
    T = s.shape[0]
    idx = np.zeros((T, k), np.int32)
    gate = np.zeros((T, k), F64)
    sm = np.zeros(T, F64)
    om = np.zeros(T, F64)
    for i in range(T):
        R = topk_desc(s[i], k)
        idx[i] = R
        gate[i] = renormalize(s[i], R)
        sm[i], om[i] = topk_margins(s[i], k)
    return Routing(idx, gate, [], sm, om, np.zeros(0), s)


def route_block(s: np.ndarray, k: int, block_size: int, p: float,
                k_mask: Optional[int] = None) -> Routing:
    """Algorithm 1 applied to every block of ``block_size`` consecutive tokens; blocks are
    routed independently. Returns R_i for every token with the R8 gates.

    ``k_mask`` (default k) is the k of TopKMask and of the floor (R6); the final TopK keeps
    k <= k_mask members of the coreset per token (R17: App. A's "fewer experts for each
    token"). The block's margin also covers the TopKMask decisions of its tokens that
    matter: where swapping a token's k_mask-th and (k_mask+1)-th experts in its mask would
    change the coreset, that token's set margin bounds the block's margin."""
    T, E = s.shape
    assert T % block_size == 0
    km = k if k_mask is None or k_mask <= 0 else int(k_mask)
    assert 1 <= k <= km <= E
    nb = T // block_size
    idx = np.zeros((T, k), np.int32)
    gate = np.zeros((T, k), F64)
    sm = np.zeros(T, F64)
    om = np.zeros(T, F64)
    cm = np.zeros(nb, F64)
    coresets, alts = [], []
    for b in range(nb):
        rows = slice(b * block_size, (b + 1) * block_size)
        S = aggregate(s[rows], km)                    # Algorithm 1: S_block
        S_tilde = normalize(S)                        # Algorithm 1: Normalize
        C = top_p(S_tilde, p, km)                     # Algorithm 1: TopP (+ floor)
        coresets.append(C.ids)
        cm[b] = min(C.margin, mask_flip_margin(s[rows], S, km, p, C, C.margin))
        alts.append(C.alts)
        for i in range(b * block_size, (b + 1) * block_size):
            R, sm[i], om[i] = topk_in_coreset(s[i], C.ids, k)   # MaskOutside, TopK
            idx[i] = R
            gate[i] = renormalize(s[i], R)
    return Routing(idx, gate, coresets, sm, om, cm, s, alts)


def mask_flip_margin(s_block: np.ndarray, S: np.ndarray, k: int, p: float, C: Coreset,
                     bound: float) -> float:
    """Smallest TopKMask set margin (gap between a token's k-th and (k+1)-th score) among
    the block's tokens whose flip at that boundary changes the coreset as a set; only
    margins below ``bound`` or NEAR_TIE are examined (larger ones cannot lower the block's
    margin). The coreset such a flip closer than NEAR_TIE reaches joins C.alts."""
    out = float("inf")
    core = set(C.ids.tolist())
    for i in range(s_block.shape[0]):
        sm, _ = topk_margins(s_block[i], k)
        if not (sm < min(bound, out) or sm < NEAR_TIE):
            continue
        order = sort_desc(np.asarray(s_block[i], F64))
        a, c = int(order[k - 1]), int(order[k])      # the k-th and the first left out
        v = np.asarray(s_block[i], F32).astype(F64)
        S_alt = np.array(S, F64)
        S_alt[a] -= v[a]
        S_alt[c] += v[c]
        alt = top_p(normalize(S_alt), p, k)
        if set(alt.ids.tolist()) != core:
            out = min(out, sm)
            if sm < NEAR_TIE:
                C.alts.append(alt.ids)
    return out


def route(x_bits, w_r, bias, k: int, mode: int, block_size: int, p: float,
          k_mask: Optional[int] = None) -> Routing:
    """Router (R1) followed by token-level or block-level routing (k_mask: see route_block;
    ignored in token mode)."""
    s = router_scores(router_logits(x_bits, w_r, bias))
    if mode == ROUTE_TOKEN:
        return route_token(s, k)
    return route_block(s, k, block_size, p, k_mask)


# ----------------------------------------------------------------------------------------
# dispatch (reading R9): the unique experts of one forward and the expert -> token list
# ----------------------------------------------------------------------------------------
@dataclasses.dataclass
class Dispatch:
    unique_ids: np.ndarray   # int32 [U], ascending
    offsets: np.ndarray      # int32 [U+1]
    rows: np.ndarray         # int32 [T*k], t*k + slot, ordered by (expert, token)
    pos: np.ndarray          # int32 [T*k], pos[t*k+slot] = r with rows[r] = t*k+slot


def dispatch(idx: np.ndarray) -> Dispatch:
    T, k = idx.shape
    unique = sorted(set(int(e) for e in idx.ravel()))
    per_expert: Dict[int, List[int]] = {e: [] for e in unique}
    for t in range(T):               # token order, so each list is ordered by token
        for j in range(k):
            per_expert[int(idx[t, j])].append(t * k + j)
    rows: List[int] = []
    offsets = [0]
    for e in unique:
        rows.extend(per_expert[e])
        offsets.append(len(rows))
    rows_a = np.asarray(rows, np.int32)
    pos = np.empty(T * k, np.int32)
    pos[rows_a] = np.arange(T * k, dtype=np.int32)
    return Dispatch(np.asarray(unique, np.int32), np.asarray(offsets, np.int32), rows_a, pos)


# ----------------------------------------------------------------------------------------
# expert execution (reading R10)
# ----------------------------------------------------------------------------------------
def silu(z: np.ndarray) -> np.ndarray:
    return z / (1.0 + np.exp(-z))


def swiglu_ffn(x64: np.ndarray, wg64: np.ndarray, wu64: np.ndarray, wd64: np.ndarray) -> np.ndarray:
    """One SwiGLU expert on rows x [n,d]: W_down (silu(W_gate x) * (W_up x)).
    wg, wu: [I,d]; wd: [d,I]; float64, intermediate unrounded."""
    g = x64 @ wg64.T
    u = x64 @ wu64.T
    return (silu(g) * u) @ wd64.T


def moe_forward_given_routing(x_bits, w_gate, w_up, w_down, idx, gate,
                              ws_gate=None, ws_up=None, ws_down=None,
                              tokens: Optional[Sequence[int]] = None) -> np.ndarray:
    """y_t = sum_j g_tj * Expert_{R_tj}(x_t) + Shared(x_t) for the tokens in ``tokens``
    (all tokens by default); float64 [len(tokens), d]. Weight tensors are bf16 bit
    patterns: w_gate/w_up [E,I,d], w_down [E,d,I]; the shared expert [I_s,d],[I_s,d],[d,I_s]."""
    T = x_bits.shape[0]
    tok = np.arange(T) if tokens is None else np.asarray(tokens)
    x = bf16_bits_to_f64(x_bits[tok])
    sel = np.asarray(idx)[tok]
    g = np.asarray(gate, F64)[tok]
    y = np.zeros((len(tok), x.shape[1]), F64)
    for e in sorted(set(int(v) for v in sel.ravel())):
        rr, jj = np.nonzero(sel == e)
        ye = swiglu_ffn(x[rr], bf16_bits_to_f64(w_gate[e]), bf16_bits_to_f64(w_up[e]),
                        bf16_bits_to_f64(w_down[e]))
        y[rr] += g[rr, jj][:, None] * ye
    if ws_gate is not None:
        y += swiglu_ffn(x, bf16_bits_to_f64(ws_gate), bf16_bits_to_f64(ws_up),
                        bf16_bits_to_f64(ws_down))
    return y


def gates_for(scores32: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """R8 gates of a given selection (used to evaluate a selection made elsewhere)."""
    T, k = idx.shape
    out = np.zeros((T, k), F64)
    for t in range(T):
        out[t] = renormalize(scores32[t], idx[t])
    return out


def layer_forward(inp: Dict[str, np.ndarray], k: int, mode: int, block_size: int, p: float):
    """Router, routing, dispatch and expert execution of one MoE layer.
    Returns (y float64 [T,d], Routing, Dispatch)."""
    r = route(inp["x"], inp["w_r"], inp.get("bias"), k, mode, block_size, p)
    dsp = dispatch(r.idx)
    y = moe_forward_given_routing(inp["x"], inp["w_gate"], inp["w_up"], inp["w_down"],
                                  r.idx, r.gate, inp.get("ws_gate"), inp.get("ws_up"),
                                  inp.get("ws_down"))
    return y, r, dsp
