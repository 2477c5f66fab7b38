"""Plant plausible mistakes in the oracle (on the CPU) and check that a pin fails.

Each mutation replaces one oracle function with a subtly wrong version (a
wrong order, a dropped term, a wrong index, a swapped operand).  The oracle
module looks its helpers up at call time, so patching the module attribute
changes every internal use.  A mutation counts as caught when any pin raises.
"""
import numpy as np
import pytest

import oracle_pins as P
from oracle import xshare_oracle as O


def _ranked_ascending(values, candidates):
    return sorted(candidates, key=lambda j: (float(values[j]), j))


def _ranked_high_index_ties(values, candidates):
    return sorted(candidates, key=lambda j: (-float(values[j]), -j))


def _colsum_sequential(p, rows):
    p = np.asarray(p, dtype=np.float32)
    acc = np.zeros(p.shape[1], dtype=np.float32)
    for i in rows:
        acc = acc + p[i]
    return acc


def _colsum_drop_last_chunk(p, rows):
    rows = list(rows)
    if len(rows) > 32:
        rows = rows[:(len(rows) // 32) * 32]
    return _orig["canonical_column_sum"](p, rows)


def _colsum_adjacent_tree(p, rows):
    p = np.asarray(p, dtype=np.float32)
    rows = list(rows)
    acc = np.zeros(p.shape[1], dtype=np.float32)
    for c0 in range(0, len(rows), 32):
        v = np.zeros((32, p.shape[1]), dtype=np.float32)
        v[:len(rows[c0:c0 + 32])] = p[rows[c0:c0 + 32]]
        while v.shape[0] > 1:
            v = v[0::2] + v[1::2]
        acc = acc + v[0]
    return acc


def _greedy_total_cap(scores, m, S0):
    S = set(S0)
    N = scores.shape[0]
    while len(S) < m:
        rest = [e for e in range(N) if e not in S]
        if not rest:
            break
        S.add(O.ranked(scores, rest)[0])
    return S


def _greedy_off_by_one(scores, m, S0):
    return _orig["greedy_select_budget"](scores, max(m - 1, 0), S0)


def _warmup_uses_k0_plus_one(p, k0, tokens):
    return _orig["warmup_set"](p, k0 + 1 if k0 > 0 else 0, tokens)


def _refine_no_renorm(p, S, k):
    ids, w = _orig["refine"](p, S, k)
    for i in range(ids.shape[0]):
        for s in range(k):
            if ids[i, s] >= 0:
                w[i, s] = p[i, ids[i, s]]
    return ids, w


def _refine_over_all_experts(p, S, k):
    return _orig["refine"](p, set(range(p.shape[1])), k)


def _permute_unstable(ids, N):
    r = _orig["permute"](ids, N)
    perm = r["perm"].copy()
    off = r["offsets"]
    for e in range(N):
        perm[off[e]:off[e + 1]] = perm[off[e]:off[e + 1]][::-1]
    r["perm"] = perm
    return r


def _group_strict_cap(scores, G, m_g, S0):
    N = scores.shape[0]
    size = N // G
    S = set(S0)
    while len(S) < m_g * G:
        added = False
        for g in range(G):
            if len(S) >= m_g * G:
                break
            rest = [e for e in range(g * size, (g + 1) * size) if e not in S]
            if rest:
                S.add(O.ranked(scores, rest)[0])
                added = True
        if not added:
            break
    return S


def _request_uses_batch_scores(p, tokens, m_r, k0):
    N = p.shape[1]
    S0 = O.warmup_set(p, k0, tokens)
    scores = O.canonical_column_sum(p, range(p.shape[0]))
    rest = [e for e in range(N) if e not in S0]
    return S0 | set(O.top(scores, m_r, rest))


def _softmax_unnormalised(h):
    h = np.asarray(h, dtype=np.float64)
    return np.exp(h - h.max(axis=1, keepdims=True)).astype(np.float32)


def _silu_wrong_sign(z):
    return z / (1.0 + np.exp(z))


def _ffn_swapped_gate_up(x_rows, Wg, Wu, Wd):
    return _orig["expert_ffn"](x_rows, Wu, Wg, Wd)


def _ffn_drops_up(x_rows, Wg, Wu, Wd):
    g = x_rows @ O.bf16_bits_to_f64(Wg).T
    return O.silu(g) @ O.bf16_bits_to_f64(Wd).T


def _combine_unweighted(ids, w, expert_out, tokens, d):
    return _orig["combine"](ids, np.where(ids >= 0, 1.0, 0.0).astype(np.float32), expert_out, tokens, d)


def _router_transposed_input(x_bits, W_g):
    x = O.bf16_bits_to_f64(x_bits)
    W = np.asarray(W_g, dtype=np.float64)
    return (x[::-1] @ W.T)


def _shared_dropped(x_bits, get_shared, n_shared, tokens):
    return np.zeros((len(list(tokens)), x_bits.shape[1]))


def _shared_first_only(x_bits, get_shared, n_shared, tokens):
    return _orig["shared_experts_out"](x_bits, get_shared, min(n_shared, 1), tokens)


def _threshold_non_strict(scores, tau, S0):
    scores = np.asarray(scores, dtype=np.float32)
    N = scores.shape[0]
    S = set(S0)
    target = np.float32(np.float32(tau) * O.expert_tree_sum(scores, set(range(N))))
    f = O.expert_tree_sum(scores, S)
    while f <= target and len(S) < N:
        e = O.ranked(scores, [j for j in range(N) if j not in S])[0]
        S.add(e)
        f = np.float32(f + scores[e])
    return S


def _threshold_ignores_s0_mass(scores, tau, S0):
    scores = np.asarray(scores, dtype=np.float32)
    N = scores.shape[0]
    S = set(S0)
    target = np.float32(np.float32(tau) * O.expert_tree_sum(scores, set(range(N))))
    f = np.float32(0.0)
    while f < target and len(S) < N:
        e = O.ranked(scores, [j for j in range(N) if j not in S])[0]
        S.add(e)
        f = np.float32(f + scores[e])
    return S


def _tree_sum_left_to_right(values, members):
    acc = np.float32(0.0)
    for j in sorted(members):
        acc = np.float32(acc + np.float32(values[j]))
    return acc


def _budgets_floor(K, L):
    return [K // L] * L


def _bf16_truncate(x):
    x = np.asarray(x, dtype=np.float64)
    return (x.astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def _bf16_via_fp32(x):
    x = np.asarray(x, dtype=np.float64).astype(np.float32)
    return _orig["f64_to_bf16_bits"](x.astype(np.float64))


def _gating_unnormalised(p, k):
    p = np.asarray(p, dtype=np.float32)
    g = np.zeros_like(p)
    for i in range(p.shape[0]):
        for j in O.top(p[i], k, range(p.shape[1])):
            g[i, j] = p[i, j]
    return g


def _candidates_allow_zero(scores, S, positive_only, pool=None):
    return _orig["candidates"](scores, S, False, pool)


def _group_range_shifted(N, G, g):
    lo, hi = _orig["expert_group_range"](N, G, g)
    return lo + 1, min(hi + 1, N)


def _ep_combine_shared_first(r, out, n_shared=0):
    ids, w, perm = r["ids"], r["w"], r["perm"]
    B, k = ids.shape
    n_pairs = len(perm)
    row_of = {int(q): i for i, q in enumerate(perm)}
    y = np.zeros((B, out.shape[1]))
    for t in range(B):
        for j in range(n_shared):
            y[t] += out[n_pairs + j * B + t]
        for s in range(k):
            if ids[t, s] >= 0:
                y[t] += float(w[t, s]) * out[row_of[t * k + s]]
    return y


def _closed_form_wrong(N, k, B):
    return N * (1.0 - (1.0 - k / N) ** (B - 1))


MUTATIONS = {
    "ranked ascending": ("ranked", _ranked_ascending),
    "ties to higher index": ("ranked", _ranked_high_index_ties),
    "column sum sequential": ("canonical_column_sum", _colsum_sequential),
    "column sum drops last chunk": ("canonical_column_sum", _colsum_drop_last_chunk),
    "column sum adjacent-pair tree": ("canonical_column_sum", _colsum_adjacent_tree),
    "budget caps |S| instead of adding": ("greedy_select_budget", _greedy_total_cap),
    "budget off by one": ("greedy_select_budget", _greedy_off_by_one),
    "warm-up uses k0+1": ("warmup_set", _warmup_uses_k0_plus_one),
    "refine without renormalising": ("refine", _refine_no_renorm),
    "refine ignores S": ("refine", _refine_over_all_experts),
    "permutation not stable": ("permute", _permute_unstable),
    "group greedy stops mid-round": ("gpu_aware_greedy", _group_strict_cap),
    "per-request step uses batch scores": ("per_request_select", _request_uses_batch_scores),
    "softmax not normalised": ("softmax_scores", _softmax_unnormalised),
    "silu wrong sign": ("silu", _silu_wrong_sign),
    "gate and up swapped": ("expert_ffn", _ffn_swapped_gate_up),
    "up projection dropped": ("expert_ffn", _ffn_drops_up),
    "combine ignores weights": ("combine", _combine_unweighted),
    "router rows misindexed": ("router_logits", _router_transposed_input),
    "closed form exponent": ("expected_union_size", _closed_form_wrong),
    "shared experts dropped": ("shared_experts_out", _shared_dropped),
    "only the first shared expert": ("shared_experts_out", _shared_first_only),
    "threshold loop runs while f <= target": ("greedy_select_threshold", _threshold_non_strict),
    "threshold ignores the warm-up mass": ("greedy_select_threshold", _threshold_ignores_s0_mass),
    "expert sum left to right": ("expert_tree_sum", _tree_sum_left_to_right),
    "budget split drops the remainder": ("layer_budgets", _budgets_floor),
    "bf16 by truncation": ("f64_to_bf16_bits", _bf16_truncate),
    "bf16 rounded through fp32": ("f64_to_bf16_bits", _bf16_via_fp32),
    "sparse gating not renormalised": ("topk_gating", _gating_unnormalised),
    "sparse selection adds zero-gain experts": ("candidates", _candidates_allow_zero),
    "device owns the wrong expert group": ("expert_group_range", _group_range_shifted),
    "combine adds the shared experts first": ("ep_combine", _ep_combine_shared_first),
}

_orig = {name: getattr(O, name) for name, _ in MUTATIONS.values()}


@pytest.mark.parametrize("label", sorted(MUTATIONS))
def test_mutation_is_caught(label, monkeypatch):
    name, fn = MUTATIONS[label]
    monkeypatch.setattr(O, name, fn)
    failures = []
    for check in P.ALL_CHECKS:
        if check is P.check_union_statistics:
            continue   # slowest pin; every mutation here is caught by a faster one
        try:
            check(O)
        except Exception as exc:  # noqa: BLE001 - any failure counts as caught
            failures.append((check.__name__, type(exc).__name__))
            break
    assert failures, f"mutation '{label}' was not caught by any pin"
