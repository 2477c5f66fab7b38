"""Plain CPU oracle for one XShare MoE layer forward (arxiv 2602.07265).

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously-correct
restatement of the method that the CUDA library is checked against.  Only the
tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import it.  It shares no code with the CUDA path and imports nothing from the
product package.

What it computes, in the paper's order and notation:

* Router logits  h = W_g x                                 (Sec. 2.2)
* Dense softmax gating scores g_ij over all N experts      (Sec. 2.2, Sec. 3.1;
  dense reading, see ``softmax_scores``)
* Warm-up set S_0 = union of per-token top-k0              (Sec. 3.4, Algorithm 2)
* Column scores scores[j] = sum_i g_ij                      (Algorithm 1, Eq. 2)
* Budgeted selection:
    - BATCH  : Algorithm 2 with Algorithm 1 in fixed-budget form
    - HIER   : Algorithm 4 calling Algorithm 3 per request, Eq. 3-4
    - GROUP  : Algorithm 6 calling Algorithm 5, Eq. 5
    - THRESH : Algorithm 2 with Algorithm 1 in its threshold form (tau)
    - TOPK   : S = E, i.e. plain top-k routing (Sec. 2.2)
* Refinement: each token routed to Top k(G_i, S) with renormalised weights
                                                            (Sec. 2.2, Algorithms 2/4/6)
* Permutation of (token, slot) pairs by expert (counting sort, stable)
* Expert FFN E_i(x) = W_down (silu(W_gate x) * (W_up x)) over the pairs, and the
  weighted combine y = sum_i g_i(x) E_i(x) + sum_j E^s_j(x)   (Sec. 2.1)
* A stack of L residual MoE layers with the global budget split m_l = K / L
                                                            (Eq. 1, Sec. 3.2)
* Expert parallelism: the experts partitioned into G contiguous groups, one
  per device, each device computing its group's pairs    (Sec. 5)

Precision.  Selection is decided on fp32 scores (the precision the kernels
decide in): softmax is evaluated in fp64 and rounded to fp32 once, column sums
use the canonical fp32 order defined in ``canonical_column_sum``, the
renormalised weights are fp32.  Router logits and the expert FFN are fp64.

Readings of the paper where it is silent or ambiguous are stated at each
function; every one of them is listed in the design notes of the repository.
"""

from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence, Set, Tuple

import numpy as np

MODE_TOPK = 0
MODE_BATCH = 1
MODE_GROUP = 2
MODE_HIER = 3
MODE_THRESH = 4

MODE_NAMES = {MODE_TOPK: "topk", MODE_BATCH: "batch", MODE_GROUP: "group", MODE_HIER: "hier",
              MODE_THRESH: "thresh"}

# Width of one chunk of the canonical column sum (one warp of 32 lanes).
CHUNK = 32


# --------------------------------------------------------------------------
# Number formats
# --------------------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Widen raw bf16 bit patterns (uint16) to float64 exactly.

    A bf16 value is the upper 16 bits of an IEEE binary32 value, so shifting
    the pattern left by 16 gives the fp32 number, which fp64 holds exactly.
    """
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float64 values to bf16 (8 significant bits, fp32's exponent range),
    to nearest with ties to even, in one step.  Returns uint16 bit patterns.

    x = m 2^e with 0.5 <= |m| < 1; the bf16 quantum at that binade is
    2^(e - 8), or 2^-133 below the normal range (e < -125).  np.rint rounds
    half to even.  Values beyond bf16's range are not expected here.
    """
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)
    q = np.maximum(e, -125) - 8
    r = np.ldexp(np.rint(np.ldexp(x, -q)), q)
    return (r.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


# --------------------------------------------------------------------------
# Sec. 2.2: router logits and gating scores
# --------------------------------------------------------------------------

def router_logits(x_bits: np.ndarray, W_g: np.ndarray) -> np.ndarray:
    """h(x) = W_g x for every token (Sec. 2.2), in fp64.

    x_bits: [B, d] uint16 bf16 patterns; W_g: [N, d] float32.  Returns [B, N]
    float64.  The bf16 inputs and fp32 weights are widened exactly; the dot
    products use fp64 arithmetic.
    """
    x = bf16_bits_to_f64(x_bits)
    W = np.asarray(W_g, dtype=np.float32).astype(np.float64)
    return x @ W.T


def softmax_scores(h: np.ndarray) -> np.ndarray:
    """Gating scores g_ij = exp(h_ij) / sum_j' exp(h_ij') over ALL N experts.

    Reading of Sec. 2.2 / Sec. 3.1: the scores G_i that the selection step sums
    are the dense softmax over the full expert set, not the top-k-masked ones;
    only dense scores make "top-k within S" (the refinement step) meaningful.
    Evaluated in fp64 (row maximum subtracted first), then rounded once to
    fp32, the precision in which every selection decision is taken.
    """
    h = np.asarray(h, dtype=np.float64)
    z = h - h.max(axis=1, keepdims=True)
    e = np.exp(z)
    return (e / e.sum(axis=1, keepdims=True)).astype(np.float32)


# --------------------------------------------------------------------------
# Total order used by every top-k / argmax of the method
# --------------------------------------------------------------------------

def ranked(values: np.ndarray, candidates: Sequence[int]) -> List[int]:
    """Candidates sorted best-first: larger value first, ties to the lower index.

    The paper does not say how ties break; the lower expert index wins
    everywhere.  Values are fp32 and compared exactly.
    """
    return sorted(candidates, key=lambda j: (-float(values[j]), j))


def top(values: np.ndarray, count: int, candidates: Sequence[int]) -> List[int]:
    """Top `count` of `candidates` under the total order (fewer if not enough)."""
    if count <= 0:
        return []
    return ranked(values, candidates)[:count]


# --------------------------------------------------------------------------
# Algorithm 1 / Eq. 2: column scores
# --------------------------------------------------------------------------

def canonical_column_sum(p: np.ndarray, rows: Sequence[int]) -> np.ndarray:
    """scores[j] = sum over the given rows i of g_ij, in the canonical fp32 order.

    The paper does not fix a summation order.  Selection compares these sums,
    so the order is fixed here and the kernels follow the same one:

    * the rows are taken in the given order and split into chunks of 32,
      the last chunk padded with zeros;
    * inside a chunk of values v[0..31] a halving tree is applied:
      for o = 16, 8, 4, 2, 1: v[l] <- v[l] + v[l + o] for every l < o;
      the chunk's sum is v[0];
    * chunk sums are added left to right to an accumulator that starts at 0.

    Every addition is one fp32 addition rounded to nearest.  Returns [N] float32.
    """
    p = np.asarray(p, dtype=np.float32)
    N = p.shape[1]
    rows = list(rows)
    acc = np.zeros(N, dtype=np.float32)
    for c0 in range(0, len(rows), CHUNK):
        chunk_rows = rows[c0:c0 + CHUNK]
        v = np.zeros((CHUNK, N), dtype=np.float32)
        v[:len(chunk_rows)] = p[chunk_rows]
        o = CHUNK // 2
        while o >= 1:
            v[:o] = v[:o] + v[o:2 * o]
            o //= 2
        acc = acc + v[0]
    return acc


# --------------------------------------------------------------------------
# Warm-up initialisation (Sec. 3.4)
# --------------------------------------------------------------------------

def warmup_set(p: np.ndarray, k0: int, tokens: Sequence[int]) -> Set[int]:
    """S_0 = union over the given tokens of Top k0(G_i, E) (Algorithms 2, 3, 6)."""
    N = p.shape[1]
    S0: Set[int] = set()
    for i in tokens:
        S0.update(top(p[i], k0, range(N)))
    return S0


# --------------------------------------------------------------------------
# Selection algorithms
# --------------------------------------------------------------------------

def candidates(scores: np.ndarray, S: Set[int], positive_only: bool,
               pool: Optional[Sequence[int]] = None) -> List[int]:
    """Experts of `pool` (all of E by default) outside S that may be added.

    With `positive_only` (the sparse-score reading of Sec. 2.2, where g is 0
    outside each token's top-k) an expert whose column score is 0 has no gain
    and is never added.
    """
    pool = range(scores.shape[0]) if pool is None else pool
    return [e for e in pool if e not in S and (not positive_only or scores[e] > 0)]


def greedy_select_budget(scores: np.ndarray, m: int, S0: Set[int],
                         positive_only: bool = False) -> Set[int]:
    """Algorithm 1 in the fixed-budget form used in practice (Sec. 3.4).

    Starting from S_0, repeatedly add argmax_{e in E \\ S} scores[e], m times
    (or until E is exhausted).  Reading: the budget m counts experts added
    beyond S_0, as Algorithm 3 writes explicitly (S_0 union Top m_r).
    By Proposition 1 the marginal gain of e is scores[e] whatever S is, so the
    argmax is taken over the precomputed column scores.
    """
    S = set(S0)
    for _ in range(m):
        rest = candidates(scores, S, positive_only)
        if not rest:
            break
        S.add(ranked(scores, rest)[0])
    return S


def expert_tree_sum(values: np.ndarray, members: Set[int]) -> np.float32:
    """f(S) = sum of values[j] over j in S, in a fixed fp32 order.

    The values of the members are placed at their expert index in a vector of
    zeros whose length is a power of two >= N, and a halving tree is applied
    (for o = len/2, ..., 1: v[l] <- v[l] + v[l + o] for l < o); the sum is
    v[0].  Because x + 0 = x exactly, the padded length does not change the
    result.  Every addition is one fp32 addition rounded to nearest.
    """
    values = np.asarray(values, dtype=np.float32)
    L = 1
    while L < values.shape[0]:
        L *= 2
    v = np.zeros(L, dtype=np.float32)
    for j in members:
        v[j] = values[j]
    o = L // 2
    while o >= 1:
        v[:o] = v[:o] + v[o:2 * o]
        o //= 2
    return np.float32(v[0])


def greedy_select_threshold(scores: np.ndarray, tau: float, S0: Set[int],
                            positive_only: bool = False) -> Set[int]:
    """Algorithm 1 in its threshold form: experts are added until they cover
    a fraction tau of the batch's score mass.

    Starting from S_0, while f(S) < tau * f(E), the expert of E \\ S with the
    largest score is added (Algorithm 1's condition names P for G, read as the
    scores G).  Selection also ends when E \\ S is empty.

    Precision.  f(E) and f(S_0) are `expert_tree_sum`s; the target is the
    fp32 product tau * f(E) rounded once.  When e is added, f(S) becomes the
    fp32 sum f(S) + scores[e]: by Proposition 1 the gain of adding e is
    exactly scores[e], whatever S is.
    """
    scores = np.asarray(scores, dtype=np.float32)
    N = scores.shape[0]
    S = set(S0)
    target = np.float32(np.float32(tau) * expert_tree_sum(scores, set(range(N))))
    f = expert_tree_sum(scores, S)
    while f < target:
        rest = candidates(scores, S, positive_only)
        if not rest:
            break
        e = ranked(scores, rest)[0]
        S.add(e)
        f = np.float32(f + scores[e])
    return S


def select_threshold(p: np.ndarray, tau: float, k0: int,
                     gs: Optional[np.ndarray] = None) -> Tuple[Set[int], Set[int]]:
    """Algorithm 2 with GreedySelect in its threshold form: warm-up S_0, then
    add experts until they cover a fraction tau of the batch's score mass.
    With `gs` (sparse scores) the column scores are taken from gs."""
    B = p.shape[0]
    S0 = warmup_set(p, k0, range(B))
    scores = canonical_column_sum(p if gs is None else gs, range(B))
    return greedy_select_threshold(scores, tau, S0, gs is not None), S0


def select_batch(p: np.ndarray, m: int, k0: int,
                 gs: Optional[np.ndarray] = None) -> Tuple[Set[int], Set[int]]:
    """Algorithm 2: warm-up S_0, then GreedySelect with budget m.  Returns (S, S_0).
    With `gs` (sparse scores) the column scores are taken from gs."""
    B = p.shape[0]
    S0 = warmup_set(p, k0, range(B))
    scores = canonical_column_sum(p if gs is None else gs, range(B))
    return greedy_select_budget(scores, m, S0, gs is not None), S0


def per_request_select(p: np.ndarray, tokens: Sequence[int], m_r: int, k0: int,
                       gs: Optional[np.ndarray] = None) -> Set[int]:
    """Algorithm 3 for one request r with tokens T_r.

    S_0 = union of Top k0 over T_r; scores[j] = sum over T_r of g_xj (Eq. 3);
    S_r = S_0 union Top m_r(scores, E \\ S_0).  With `gs` (sparse scores) the
    request's column scores are taken from gs.
    """
    S0 = warmup_set(p, k0, tokens)
    scores = canonical_column_sum(p if gs is None else gs, tokens)
    rest = candidates(scores, S0, gs is not None)
    return S0 | set(top(scores, m_r, rest))


def select_hier(p: np.ndarray, m: int, m_r: int, k0: int, tokens_per_request: int,
                gs: Optional[np.ndarray] = None) -> Tuple[Set[int], Set[int]]:
    """Algorithm 4: union of per-request selections, then GreedySelect(m).

    Requests are contiguous runs of `tokens_per_request` = 1 + L_s tokens
    (Sec. 4.1).  Returns (S_batch, union of the S_r before the batch step).
    """
    B = p.shape[0]
    T = tokens_per_request
    S_b: Set[int] = set()
    for r in range(B // T):
        S_b |= per_request_select(p, range(r * T, (r + 1) * T), m_r, k0, gs)
    scores = canonical_column_sum(p if gs is None else gs, range(B))
    return greedy_select_budget(scores, m, S_b, gs is not None), S_b


def group_of(e: int, N: int, G: int) -> int:
    """Index of the group E_g holding expert e: G contiguous ranges of N/G."""
    return e // (N // G)


def gpu_aware_greedy(scores: np.ndarray, G: int, m_g: int, S0: Set[int],
                     positive_only: bool = False) -> Set[int]:
    """Algorithm 5 (Sec. 5.1): greedy selection with a per-group budget m_g
    over the G contiguous expert groups E_g.

    By Proposition 1 the marginal gain of adding expert e is its column score
    scores[e], whatever has been selected, so the order in which a group
    receives experts is known in advance: its candidates E_g \ S_0 (with a
    positive score when positive_only) ranked by score.  Selection proceeds in
    rounds; round r gives every group that still has an r-th candidate that
    expert.  Rounds are whole (every group gets its turn in each), and a new
    round starts while |S| < m_g * G and some group still has candidates.
    Readings: |S| may therefore end above m_g * G by up to G - 1; S_0 is kept
    even where it exceeds a group's share; selection stops when every group is
    exhausted.
    """
    N = scores.shape[0]
    size = N // G
    order = [ranked(scores, candidates(scores, set(S0), positive_only,
                                       range(g * size, (g + 1) * size)))
             for g in range(G)]
    S = set(S0)
    r = 0
    while len(S) < m_g * G and any(r < len(o) for o in order):
        for o in order:
            if r < len(o):
                S.add(o[r])
        r += 1
    return S


def select_group(p: np.ndarray, G: int, m_g: int, k0: int,
                 gs: Optional[np.ndarray] = None) -> Tuple[Set[int], Set[int]]:
    """Algorithm 6: warm-up S_0 over the batch, then Algorithm 5.  Returns (S, S_0).
    With `gs` (sparse scores) the column scores are taken from gs."""
    B = p.shape[0]
    S0 = warmup_set(p, k0, range(B))
    scores = canonical_column_sum(p if gs is None else gs, range(B))
    return gpu_aware_greedy(scores, G, m_g, S0, gs is not None), S0


def topk_gating(p: np.ndarray, k: int) -> np.ndarray:
    """Sec. 2.2's gating values: g_ij = exp(h_j) / sum_{T_i} exp(h) for j in
    T_i = Top k(G_i, E), and 0 outside T_i (the sparse reading of the scores
    that Sec. 3 sums).

    exp(h_j) / sum_T exp(h) = p_j / sum_T p for the dense softmax p, so each
    row is computed from p as the standard top-k routing weights are: D = fp32
    sum of p over T_i in rank order, one fp32 division per expert; if D = 0
    each of the k experts gets 1/k.  Returns [B, N] float32.
    """
    p = np.asarray(p, dtype=np.float32)
    B, N = p.shape
    g = np.zeros((B, N), dtype=np.float32)
    for i in range(B):
        T = top(p[i], k, range(N))
        D = np.float32(0.0)
        for j in T:
            D = np.float32(D + p[i, j])
        for j in T:
            g[i, j] = np.float32(p[i, j] / D) if D > 0 else np.float32(1.0) / np.float32(len(T))
    return g


# --------------------------------------------------------------------------
# Refinement (Sec. 3.4) with renormalised weights (Sec. 2.2)
# --------------------------------------------------------------------------

def refine(p: np.ndarray, S: Set[int], k: int) -> Tuple[np.ndarray, np.ndarray]:
    """Route every token to Top k(G_i, S) and renormalise.

    k' = min(k, |S|) experts per token, listed best-first; slots k'..k-1 hold
    id -1 and weight 0 (reading for |S| < k).  The weight of a routed expert
    follows Sec. 2.2 restricted to the routed set T':
        g_bar = exp(h_e) / sum_{j in T'} exp(h_j) = g_e / sum_{j in T'} g_j,
    with the denominator D the fp32 sum of the k' scores in slot order and one
    fp32 division.  If D is 0 (every score underflowed) each weight is 1/k'.
    Returns ids [B, k] int32 and weights [B, k] float32.
    """
    p = np.asarray(p, dtype=np.float32)
    B = p.shape[0]
    kp = min(k, len(S))
    cands = sorted(S)
    ids = np.full((B, k), -1, dtype=np.int32)
    w = np.zeros((B, k), dtype=np.float32)
    for i in range(B):
        chosen = top(p[i], kp, cands)
        D = np.float32(0.0)
        for e in chosen:
            D = np.float32(D + p[i, e])
        for s, e in enumerate(chosen):
            ids[i, s] = e
            if D > 0:
                w[i, s] = np.float32(p[i, e] / D)
            else:
                w[i, s] = np.float32(np.float32(1.0) / np.float32(kp))
    return ids, w


# --------------------------------------------------------------------------
# Token permutation
# --------------------------------------------------------------------------

def permute(ids: np.ndarray, N: int) -> Dict[str, np.ndarray]:
    """Counting sort of the (token, slot) pairs by expert.

    Pair id = t * k + slot.  counts[e] = pairs routed to e; offsets = exclusive
    prefix of counts (length N + 1); perm lists pair ids grouped by expert in
    ascending expert order and, inside an expert, in ascending (token, slot)
    order; used = experts with at least one pair, ascending.
    """
    B, k = ids.shape
    counts = np.zeros(N, dtype=np.int32)
    for t in range(B):
        for s in range(k):
            e = int(ids[t, s])
            if e >= 0:
                counts[e] += 1
    offsets = np.zeros(N + 1, dtype=np.int32)
    for e in range(N):
        offsets[e + 1] = offsets[e] + counts[e]
    fill = offsets[:N].copy()
    perm = np.zeros(int(offsets[N]), dtype=np.int32)
    for t in range(B):
        for s in range(k):
            e = int(ids[t, s])
            if e >= 0:
                perm[fill[e]] = t * k + s
                fill[e] += 1
    used = np.array([e for e in range(N) if counts[e] > 0], dtype=np.int32)
    return {"counts": counts, "offsets": offsets, "perm": perm, "used": used}


# --------------------------------------------------------------------------
# Full routing step
# --------------------------------------------------------------------------

def route(p: np.ndarray, k: int, budget: int, mode: int, k0: int = 0, m_r: int = 0,
          tokens_per_request: int = 1, n_groups: int = 1, m_g: int = 0,
          tau: float = 0.0, sparse_scores: int = 0) -> Dict[str, object]:
    """Batch-aware selection and refinement on fp32 gating scores p [B, N].

    mode TOPK : S = E (standard top-k routing, the paper's baseline)
    mode BATCH: Algorithm 2 with budget m = `budget`, warm-up k0
    mode HIER : Algorithm 4 with batch budget m = `budget`, per-request m_r, k0
    mode GROUP: Algorithm 6 with G = n_groups contiguous groups, per-group m_g, k0
    mode THRESH: Algorithm 2 with Algorithm 1's threshold tau (fp32), k0; no budget
    With `sparse_scores` the column scores of every selection step sum Sec.
    2.2's top-k-masked g instead of the dense softmax, and experts with a zero
    column score are never added; warm-up and refinement use the dense scores.
    Returns the selected mask, the routing, the permutation and the statistics
    |S|, |U|, |union of plain top-k| and max_g |S intersect E_g|.
    """
    p = np.asarray(p, dtype=np.float32)
    B, N = p.shape
    gs = topk_gating(p, k) if sparse_scores and mode != MODE_TOPK else None
    if mode == MODE_TOPK:
        S = set(range(N))
    elif mode == MODE_BATCH:
        S, _ = select_batch(p, budget, k0, gs)
    elif mode == MODE_HIER:
        S, _ = select_hier(p, budget, m_r, k0, tokens_per_request, gs)
    elif mode == MODE_GROUP:
        S, _ = select_group(p, n_groups, m_g, k0, gs)
    elif mode == MODE_THRESH:
        S, _ = select_threshold(p, tau, k0, gs)
    else:
        raise ValueError(f"unknown mode {mode}")
    ids, w = refine(p, S, k)
    perm = permute(ids, N)
    union = warmup_set(p, k, range(B))
    G = n_groups if n_groups >= 1 else 1
    loads = [0] * G
    for e in S:
        loads[group_of(e, N, G)] += 1
    mask = np.zeros(N, dtype=np.uint8)
    for e in S:
        mask[e] = 1
    return {
        "mask": mask, "ids": ids, "w": w, **perm,
        "n_selected": len(S), "n_used": int(len(perm["used"])),
        "union_topk": len(union), "max_group_load": max(loads),
    }


# --------------------------------------------------------------------------
# Sec. 2.1: expert FFN and weighted combine
# --------------------------------------------------------------------------

def silu(z: np.ndarray) -> np.ndarray:
    """silu(z) = z / (1 + exp(-z)), fp64."""
    return z / (1.0 + np.exp(-z))


def expert_ffn(x_rows: np.ndarray, Wgate_e: np.ndarray, Wup_e: np.ndarray,
               Wdown_e: np.ndarray) -> np.ndarray:
    """SwiGLU expert E_e(x) = W_down (silu(W_gate x) * (W_up x)) for a stack of x rows.

    x_rows [n, d] float64; Wgate_e, Wup_e: [F, d] uint16 bf16 patterns;
    Wdown_e: [d, F] uint16.  fp64 throughout.  Returns [n, d] float64.
    """
    g = x_rows @ bf16_bits_to_f64(Wgate_e).T
    u = x_rows @ bf16_bits_to_f64(Wup_e).T
    a = silu(g) * u
    return a @ bf16_bits_to_f64(Wdown_e).T


def combine(ids: np.ndarray, w: np.ndarray, expert_out: Dict[Tuple[int, int], np.ndarray],
            tokens: Sequence[int], d: int) -> np.ndarray:
    """Routed part of the layer output, y_t = sum over slots of w_ts * E_{ids_ts}(x_t).

    `expert_out[(t, s)]` is the expert output for pair (t, s).  Slots with id -1
    contribute nothing.  fp64, weights widened from fp32.  Returns [len(tokens), d].
    """
    y = np.zeros((len(tokens), d), dtype=np.float64)
    for r, t in enumerate(tokens):
        for s in range(ids.shape[1]):
            if ids[t, s] >= 0:
                y[r] += float(w[t, s]) * expert_out[(t, s)]
    return y


def moe_ffn_combine(x_bits: np.ndarray, ids: np.ndarray, w: np.ndarray,
                    get_expert, tokens: Optional[Sequence[int]] = None) -> np.ndarray:
    """Expert FFN over the routed pairs of `tokens` and the weighted combine.

    get_expert(e) -> (Wgate_e [F, d], Wup_e [F, d], Wdown_e [d, F]) as uint16
    bf16 patterns; only experts some listed token is routed to are requested,
    one at a time.  Returns y [len(tokens), d] float64 (all tokens by default).
    """
    B, k = ids.shape
    d = x_bits.shape[1]
    if tokens is None:
        tokens = list(range(B))
    x = bf16_bits_to_f64(x_bits)
    pairs_of: Dict[int, List[Tuple[int, int]]] = {}
    for t in tokens:
        for s in range(k):
            e = int(ids[t, s])
            if e >= 0:
                pairs_of.setdefault(e, []).append((t, s))
    out: Dict[Tuple[int, int], np.ndarray] = {}
    for e in sorted(pairs_of):
        Wg, Wu, Wd = get_expert(e)
        pairs = pairs_of[e]
        o = expert_ffn(x[[t for t, _ in pairs]], Wg, Wu, Wd)
        for r, ts in enumerate(pairs):
            out[ts] = o[r]
    return combine(ids, w, out, tokens, d)


def shared_experts_out(x_bits: np.ndarray, get_shared, n_shared: int,
                       tokens: Sequence[int]) -> np.ndarray:
    """Sum over the shared experts of E^s_j(x_t) (Sec. 2.1, second term), fp64.

    get_shared(j) -> (Wgate [F, d], Wup [F, d], Wdown [d, F]) uint16 bf16 patterns.
    """
    x = bf16_bits_to_f64(x_bits)[list(tokens)]
    out = np.zeros((len(tokens), x.shape[1]), dtype=np.float64)
    for j in range(n_shared):
        Wg, Wu, Wd = get_shared(j)
        out += expert_ffn(x, Wg, Wu, Wd)
    return out


def moe_forward(x_bits: np.ndarray, W_g: np.ndarray, get_expert, k: int, budget: int,
                mode: int, tokens: Optional[Sequence[int]] = None, get_shared=None,
                n_shared: int = 0, **params) -> Dict[str, object]:
    """One MoE layer forward: router, dense softmax, selection, refinement,
    permutation, expert FFN over the routed pairs and weighted combine, plus
    the shared experts when given (Sec. 2.1):
        y = sum_i g_i(x) E_i(x) + sum_j E^s_j(x).

    Returns the routing dictionary of `route` plus "h" (fp64 logits), "p" (fp32
    scores) and "y" (fp64 output for `tokens`, all by default).
    """
    h = router_logits(x_bits, W_g)
    p = softmax_scores(h)
    r = route(p, k, budget, mode, **params)
    r["h"] = h
    r["p"] = p
    toks = list(range(x_bits.shape[0])) if tokens is None else list(tokens)
    y = moe_ffn_combine(x_bits, r["ids"], r["w"], get_expert, toks)
    if n_shared:
        y = y + shared_experts_out(x_bits, get_shared, n_shared, toks)
    r["y"] = y
    return r


# --------------------------------------------------------------------------
# Sec. 5: expert parallelism (experts partitioned over G devices)
# --------------------------------------------------------------------------

def expert_group_range(N: int, G: int, g: int) -> Tuple[int, int]:
    """E_g = experts [g N/G, (g+1) N/G): G contiguous groups of N/G (N % G == 0),
    the same partition as the groups of Algorithm 5."""
    if N % G != 0 or not 0 <= g < G:
        raise ValueError("need N % G == 0 and 0 <= g < G")
    return g * (N // G), (g + 1) * (N // G)


def moe_forward_ep_rank(x_bits: np.ndarray, W_g: np.ndarray, get_local_expert, k: int,
                        budget: int, mode: int, G: int, g: int, get_shared=None,
                        n_shared: int = 0, **params) -> Dict[str, object]:
    """Device g's part of an expert-parallel layer forward (Sec. 5).

    Every device holds the whole batch and the router, so the routing (router,
    softmax, selection, refinement, permutation) is the one of `route`, the
    same on every device.  Device g holds only the experts of E_g
    (get_local_expert(e) for e in E_g) and computes the expert outputs of the
    (token, slot) pairs routed to them; device 0 also computes the shared
    experts.  They are returned as rows of an exchange matrix in the
    permutation's order: row offsets[e] + i is the i-th pair of expert e
    (perm), row n_pairs + j B + t is token t through shared expert j; rows of
    other devices' experts are zero.  Summing the devices' matrices gives every
    row from exactly one device.  Returns the routing dictionary plus "h", "p"
    and "out" [n_pairs + n_shared B, d] float64.
    """
    h = router_logits(x_bits, W_g)
    p = softmax_scores(h)
    r = route(p, k, budget, mode, **params)
    r["h"] = h
    r["p"] = p
    B, d = x_bits.shape
    N = np.asarray(W_g).shape[0]
    lo, hi = expert_group_range(N, G, g)
    n_pairs = len(r["perm"])
    out = np.zeros((n_pairs + n_shared * B, d), dtype=np.float64)
    x = bf16_bits_to_f64(x_bits)
    for e in range(lo, hi):
        a, b = int(r["offsets"][e]), int(r["offsets"][e + 1])
        if b > a:
            tokens = [int(q) // k for q in r["perm"][a:b]]
            Wg, Wu, Wd = get_local_expert(e)
            out[a:b] = expert_ffn(x[tokens], Wg, Wu, Wd)
    if g == 0:
        for j in range(n_shared):
            Sg, Su, Sd = get_shared(j)
            out[n_pairs + j * B:n_pairs + (j + 1) * B] = expert_ffn(x, Sg, Su, Sd)
    r["out"] = out
    return r


def ep_combine(r: Dict[str, object], out: np.ndarray, n_shared: int = 0) -> np.ndarray:
    """The layer output from the summed exchange rows (Sec. 2.1): y_t = sum over
    slots, in slot order, of w_ts times the row of pair (t, s), plus the sum
    over shared experts j, in order, of row n_pairs + j B + t.  fp64."""
    ids, w, perm = r["ids"], r["w"], r["perm"]
    B, k = ids.shape
    n_pairs = len(perm)
    row_of = {int(q): i for i, q in enumerate(perm)}
    y = np.zeros((B, out.shape[1]), dtype=np.float64)
    for t in range(B):
        for s in range(k):
            if ids[t, s] >= 0:
                y[t] += float(w[t, s]) * out[row_of[t * k + s]]
    if n_shared:
        sh = np.zeros_like(y)
        for j in range(n_shared):
            sh += out[n_pairs + j * B:n_pairs + (j + 1) * B]
        y = y + sh
    return y


# --------------------------------------------------------------------------
# Eq. 1 at the system level: a stack of L MoE layers under a global budget
# --------------------------------------------------------------------------

def layer_budgets(K: int, L: int) -> List[int]:
    """Uniform split m_l = K / L of the global budget K (Sec. 3.2, Eq. 1).

    Reading: K is split into integers that sum to K, the first K mod L
    layers taking one more: m_l = floor(K / L) + (1 if l < K mod L else 0).
    """
    return [K // L + (1 if l < K % L else 0) for l in range(L)]


def moe_stack_forward(x_bits: np.ndarray, layers: Sequence[dict], k: int, K: int, mode: int,
                      stats: Optional[list] = None, **params) -> List[np.ndarray]:
    """L residual MoE layers, x_{l+1} = x_l + MoE_l(x_l), each with budget m_l.

    layers[l] = {"W_g": [N, d] fp32, "get_expert": e -> bf16 patterns,
    optional "get_shared", "n_shared"}.  Each layer runs `moe_forward` on
    all tokens with budget layer_budgets(K, L)[l] (the modes that take no
    budget ignore it); the sum x_l + MoE_l(x_l) is formed in fp64 and rounded
    once to bf16, the precision activations have between layers.  Returns the
    bf16 patterns of x_1 .. x_L; with `stats` (a list) each layer's routing
    dictionary is appended to it.
    """
    budgets = layer_budgets(K, len(layers))
    outs = []
    x = np.asarray(x_bits, dtype=np.uint16)
    for l, layer in enumerate(layers):
        r = moe_forward(x, layer["W_g"], layer["get_expert"], k, budgets[l], mode,
                        get_shared=layer.get("get_shared"), n_shared=layer.get("n_shared", 0),
                        **params)
        x = f64_to_bf16_bits(bf16_bits_to_f64(x) + r["y"])
        outs.append(x)
        if stats is not None:
            stats.append(r)
    return outs


def expected_union_size(N: int, k: int, B: int) -> float:
    """Closed form E[N_a] = N (1 - (1 - k/N)^B) of Sec. 1 for uniform routing."""
    return N * (1.0 - (1.0 - k / N) ** B)


__all__ = [n for n in dir() if not n.startswith("_")]
