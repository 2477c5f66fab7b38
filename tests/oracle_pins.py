"""Pins of the CPU oracle to facts outside itself.

Each ``check_*`` function takes the oracle module and raises AssertionError if
the oracle disagrees with what the paper or the mathematics fixes:

* the closed form E[N_a] = N(1-(1-k/N)^B) of Sec. 1, statistically, and the
  two values the paper prints for it (golden fixture);
* Corollary 1 (greedy is optimal for the modular objective of Eq. 2), and the
  same for Algorithm 3's per-request step, by brute force on tiny N;
* the balance claim of Sec. 5.1 for Algorithm 5 and the round structure of
  its pseudocode;
* the refinement invariants of Sec. 3.4 and the renormalised weights of
  Sec. 2.2;
* special cases that reduce to library routines: budget = N is plain top-k
  (numpy lexsort), softmax / router / SwiGLU against torch float64, the
  permutation against Python's sorted;
* the canonical column-sum order on a hand-derived fixture, and its error
  against the exact sum;
* Algorithm 1's threshold form on a hand-derived fixture, and by brute force:
  the smallest superset of S_0 covering a fraction tau of the score mass;
* the layer stack of Eq. 1: the budget split, bf16 rounding against torch and
  hand-derived double-rounding cases, the residual identity, budget = N per
  layer as a plain top-k stack;
* the sparse-score reading of Sec. 2.2: the gating rows are the plain top-k
  routing weights, a hand-derived example, S inside the union of the top-k
  sets, greedy optimality by brute force, and budget = N as plain top-k.

`test_oracle_pins.py` runs them on the oracle; `test_oracle_mutations.py`
plants mistakes in the oracle and checks that some pin fails.
"""

from __future__ import annotations

import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import torch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- helpers

def lexsort_top(values: np.ndarray, count: int, candidates) -> list:
    """Top `count` candidates by (value desc, index asc) using numpy's lexsort."""
    c = np.asarray(sorted(candidates), dtype=np.int64)
    if count <= 0 or c.size == 0:
        return []
    v = np.asarray(values, dtype=np.float64)[c]
    order = np.lexsort((c, -v))
    return [int(x) for x in c[order][:count]]


def exact_colsum(p: np.ndarray, rows) -> list:
    """Exact (rational) column sums of fp32 values."""
    rows = list(rows)
    return [sum((Fraction(float(p[i, j])) for i in rows), Fraction(0)) for j in range(p.shape[1])]


def quantised_scores(rng, B, N, levels=4096) -> np.ndarray:
    """Scores that are multiples of 2^-12, so small column sums are exact in fp32."""
    return (rng.integers(1, levels, size=(B, N)).astype(np.float64) / 4096.0).astype(np.float32)


def distinct_colsums(p, rows) -> bool:
    s = exact_colsum(p, rows)
    return len(set(s)) == len(s)


def mask_to_set(mask) -> set:
    return {int(j) for j in np.nonzero(np.asarray(mask))[0]}


def bf16_round(x: torch.Tensor) -> torch.Tensor:
    return x.to(torch.bfloat16)


def bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


# ---------------------------------------------------------------- Sec. 1

def check_closed_form_golden(O):
    with open(os.path.join(GOLDEN, "union_closed_form.json")) as f:
        g = json.load(f)
    for c in g["cases"]:
        val = O.expected_union_size(c["N"], c["k"], c["B"])
        closed = c["N"] * (1 - (1 - c["k"] / c["N"]) ** c["B"])
        assert abs(val - closed) < 1e-9
        assert abs(val - c["printed"]) < 0.5, (c, val)


def check_union_statistics(O, trials=(( 64, 8, 8, 600), (256, 8, 8, 200), (256, 8, 32, 60))):
    """Under iid continuous logits each token's top-k is a uniform k-subset, so the
    union size of plain top-k routing has mean N(1-(1-k/N)^B) exactly (Sec. 1)."""
    rng = np.random.default_rng(1234)
    for N, k, B, n in trials:
        sizes = []
        for _ in range(n):
            h = rng.standard_normal((B, N))
            p = O.softmax_scores(h)
            sizes.append(O.route(p, k, 0, O.MODE_TOPK)["union_topk"])
        sizes = np.asarray(sizes, dtype=np.float64)
        mean, se = sizes.mean(), sizes.std(ddof=1) / math.sqrt(n)
        closed = N * (1 - (1 - k / N) ** B)
        assert abs(mean - closed) <= 4 * se + 1e-9, (N, k, B, mean, closed, se)


# ---------------------------------------------------------------- Eq. 2, Corollary 1

def check_greedy_bruteforce(O, cases=40):
    """Algorithm 2's selection maximises f(S) = sum_{j in S} sum_i g_ij over all
    supersets of S_0 with |S| = |S_0| + min(m, N - |S_0|)."""
    rng = np.random.default_rng(7)
    done = 0
    while done < cases:
        N = int(rng.integers(4, 11))
        B = int(rng.integers(1, 7))
        k = int(rng.integers(1, N + 1))
        k0 = int(rng.integers(0, 3))
        m = int(rng.integers(0, N + 1))
        p = quantised_scores(rng, B, N)
        S0 = set()
        for i in range(B):
            S0 |= set(lexsort_top(p[i], k0, range(N)))
        col = exact_colsum(p, range(B))
        r = O.route(p, k, m, O.MODE_BATCH, k0=k0)
        S = mask_to_set(r["mask"])
        size = len(S0) + min(m, N - len(S0))
        assert S0 <= S and len(S) == size, (S0, S, size)
        rest = [j for j in range(N) if j not in S0]
        best = max(sum((col[j] for j in c), Fraction(0))
                   for c in itertools.combinations(rest, size - len(S0)))
        got = sum((col[j] for j in S - S0), Fraction(0))
        assert got == best, (got, best)
        # among equal-score experts the lower index is preferred
        for j in S - S0:
            for q in rest:
                if q not in S:
                    assert col[q] < col[j] or (col[q] == col[j] and q > j), (q, j)
        done += 1


def check_hier_bruteforce(O, cases=25):
    """Algorithm 3: S_r maximises the per-request proxy (Eq. 3) over supersets of
    the request's warm-up set; Algorithm 4's batch step maximises Eq. 4 given
    the union of the S_r."""
    rng = np.random.default_rng(11)
    done = 0
    while done < cases:
        N = int(rng.integers(4, 10))
        T = int(rng.integers(1, 4))
        R = int(rng.integers(1, 4))
        B = R * T
        k = int(rng.integers(1, N + 1))
        k0 = int(rng.integers(0, 2))
        m_r = int(rng.integers(0, N))
        m = int(rng.integers(0, N))
        p = quantised_scores(rng, B, N)
        if not all(distinct_colsums(p, range(r * T, (r + 1) * T)) for r in range(R)):
            continue
        if not distinct_colsums(p, range(B)):
            continue
        Sb = set()
        for r in range(R):
            toks = range(r * T, (r + 1) * T)
            S0r = set()
            for i in toks:
                S0r |= set(lexsort_top(p[i], k0, range(N)))
            col = exact_colsum(p, toks)
            rest = [j for j in range(N) if j not in S0r]
            add = min(m_r, len(rest))
            best = max(itertools.combinations(rest, add),
                       key=lambda c: sum((col[j] for j in c), Fraction(0)))
            Sb |= S0r | set(best)
        col = exact_colsum(p, range(B))
        rest = [j for j in range(N) if j not in Sb]
        add = min(m, len(rest))
        best = max(itertools.combinations(rest, add),
                   key=lambda c: sum((col[j] for j in c), Fraction(0)))
        expect = Sb | set(best)
        r_ = O.route(p, k, m, O.MODE_HIER, k0=k0, m_r=m_r, tokens_per_request=T)
        assert mask_to_set(r_["mask"]) == expect, (mask_to_set(r_["mask"]), expect)
        done += 1


def check_hier_single_request_is_batch(O, cases=20):
    """Algorithm 4 with one request and m = 0 is Algorithm 2 with budget m_r."""
    rng = np.random.default_rng(5)
    for _ in range(cases):
        N = int(rng.integers(8, 40)); B = int(rng.integers(1, 40)); k = int(rng.integers(1, 9))
        k0 = int(rng.integers(0, 3)); m_r = int(rng.integers(0, N))
        p = (np.exp(rng.standard_normal((B, N))) / N).astype(np.float32)
        a = O.route(p, k, 0, O.MODE_HIER, k0=k0, m_r=m_r, tokens_per_request=B)
        b = O.route(p, k, m_r, O.MODE_BATCH, k0=k0)
        assert np.array_equal(a["mask"], b["mask"])
        assert np.array_equal(a["ids"], b["ids"]) and np.array_equal(a["w"], b["w"])


# ---------------------------------------------------------------- Sec. 5, Algorithm 5

def check_group(O, cases=30):
    """Algorithm 5/6: S_0 kept; every group that is not exhausted receives the same
    number R of additions, its top-R remaining experts by column score; R is the
    smallest round count reaching |S| >= m_g G (or every group is exhausted).
    With S_0 empty, MaxLoad(S) <= ceil(|S| / G) (Sec. 5.1)."""
    rng = np.random.default_rng(3)
    for c in range(cases):
        G = int(rng.choice([1, 2, 4, 8]))
        size = int(rng.integers(1, 9))
        N = G * size
        B = int(rng.integers(1, 40))
        k = int(rng.integers(1, min(N, 8) + 1))
        k0 = 0 if c % 2 == 0 else int(rng.integers(1, 3))
        m_g = int(rng.integers(0, size + 2))
        p = quantised_scores(rng, B, N) if c % 3 == 0 else \
            (np.exp(rng.standard_normal((B, N))) / N).astype(np.float32)
        r = O.route(p, k, 0, O.MODE_GROUP, k0=k0, n_groups=G, m_g=m_g)
        S = mask_to_set(r["mask"])
        S0 = set()
        for i in range(B):
            S0 |= set(lexsort_top(p[i], k0, range(N)))
        assert S0 <= S
        col = np.asarray(O.canonical_column_sum(p, range(B)), dtype=np.float64)
        avail = [[e for e in range(g * size, (g + 1) * size) if e not in S0] for g in range(G)]
        R = 0
        def total(R):
            return len(S0) + sum(min(R, len(a)) for a in avail)
        max_avail = max(len(a) for a in avail)
        while total(R) < m_g * G and R < max_avail:
            R += 1
        expect = set(S0)
        for a in avail:
            expect |= set(lexsort_top(col, min(R, len(a)), a))
        assert S == expect, (S, expect)
        loads = [len([e for e in S if e // size == g]) for g in range(G)]
        assert r["max_group_load"] == max(loads)
        if k0 == 0:
            assert max(loads) <= math.ceil(len(S) / G)


# ---------------------------------------------------------------- refinement, Sec. 2.2

def check_refine_invariants(O, cases=30):
    rng = np.random.default_rng(9)
    for c in range(cases):
        N = int(rng.integers(2, 70)); B = int(rng.integers(1, 50)); k = int(rng.integers(1, min(N, 16) + 1))
        mode = int(rng.integers(0, 4))
        T = int(rng.choice([t for t in (1, 2, 4) if B % t == 0]))
        G = int(rng.choice([g for g in (1, 2, 4) if N % g == 0]))
        kw = dict(k0=int(rng.integers(0, 3)), m_r=int(rng.integers(0, 6)), tokens_per_request=T,
                  n_groups=G, m_g=int(rng.integers(0, 4)))
        ties = c % 3 == 0
        p = (np.round(np.exp(rng.standard_normal((B, N))) * 4) / 4 / N if ties
             else np.exp(rng.standard_normal((B, N))) / N).astype(np.float32)
        m = int(rng.integers(0, N + 1))
        r = O.route(p, k, m, mode, **kw)
        S = mask_to_set(r["mask"])
        assert r["n_selected"] == len(S)
        kp = min(k, len(S))
        for i in range(B):
            ids = [int(e) for e in r["ids"][i]]
            w = r["w"][i]
            sel = ids[:kp]
            assert all(e == -1 for e in ids[kp:]) and np.all(w[kp:] == 0)
            assert len(set(sel)) == kp and set(sel) <= S
            assert sel == lexsort_top(p[i], kp, S)
            if kp:
                D = sum(float(p[i, e]) for e in sel)
                assert abs(float(np.sum(w[:kp], dtype=np.float64)) - 1.0) <= 1e-6 * max(1, kp)
                if D > 0:
                    ref = np.array([float(p[i, e]) / D for e in sel])
                    assert np.allclose(w[:kp], ref, rtol=2e-6, atol=0)


def check_zero_scores(O):
    """A token whose scores are all zero gets equal weights 1/k'."""
    p = np.zeros((3, 10), dtype=np.float32)
    p[1] = np.linspace(0.1, 1.0, 10, dtype=np.float32)
    r = O.route(p, 4, 10, O.MODE_BATCH)
    assert list(r["ids"][0]) == [0, 1, 2, 3]
    assert np.all(r["w"][0] == np.float32(0.25))
    assert list(r["ids"][1]) == [9, 8, 7, 6]


def check_budget_n_is_topk(O, cases=20):
    """With S = E the refinement is the standard top-k routing of Sec. 2.2:
    ids are the top-k of g_i and the weights are exp(h_i)/sum_T exp(h_j)."""
    rng = np.random.default_rng(21)
    for c in range(cases):
        N = int(rng.integers(2, 80)); B = int(rng.integers(1, 40)); k = int(rng.integers(1, min(N, 16) + 1))
        h = rng.standard_normal((B, N)) * 2
        if c % 2:
            h = np.round(h * 2) / 2   # many tied logits
        p = O.softmax_scores(h)
        k0 = int(rng.integers(0, 3))
        rb = O.route(p, k, N, O.MODE_BATCH, k0=k0)
        rt = O.route(p, k, 0, O.MODE_TOPK)
        rh = O.route(p, k, 0, O.MODE_HIER, k0=k0, m_r=N, tokens_per_request=1)
        rg = O.route(p, k, 0, O.MODE_GROUP, n_groups=1, m_g=N)
        for r in (rb, rt, rh, rg):
            assert r["n_selected"] == N
            assert np.array_equal(r["ids"], rt["ids"]) and np.array_equal(r["w"], rt["w"])
        for i in range(B):
            ref_ids = lexsort_top(p[i], k, range(N))
            assert [int(e) for e in rt["ids"][i]] == ref_ids
            z = np.exp(h[i, ref_ids] - h[i, ref_ids].max())
            ref_w = z / z.sum()
            assert np.allclose(rt["w"][i], ref_w, rtol=3e-6, atol=1e-12)


# ---------------------------------------------------------------- permutation

def check_permutation(O, cases=20):
    rng = np.random.default_rng(4)
    for _ in range(cases):
        N = int(rng.integers(1, 40)); B = int(rng.integers(1, 30)); k = int(rng.integers(1, 9))
        ids = rng.integers(-1, N, size=(B, k)).astype(np.int32)
        r = O.permute(ids, N)
        pairs = sorted((int(ids[t, s]), t, s) for t in range(B) for s in range(k) if ids[t, s] >= 0)
        assert [int(q) for q in r["perm"]] == [t * k + s for _, t, s in pairs]
        cnt = np.bincount([e for e, _, _ in pairs], minlength=N) if pairs else np.zeros(N, int)
        assert np.array_equal(r["counts"], cnt)
        assert np.array_equal(r["offsets"], np.concatenate([[0], np.cumsum(cnt)]))
        assert [int(e) for e in r["used"]] == [e for e in range(N) if cnt[e] > 0]


# ---------------------------------------------------------------- numerics vs torch

def check_router_softmax(O, cases=6):
    g = torch.Generator().manual_seed(3)
    for _ in range(cases):
        B, N, d = int(torch.randint(1, 20, (1,), generator=g)), int(torch.randint(2, 70, (1,), generator=g)), 64
        x = bf16_round(torch.randn(B, d, generator=g) * 2)
        W = torch.randn(N, d, generator=g) / 8
        h = O.router_logits(bits(x), W.numpy())
        ref_h = x.to(torch.float64) @ W.to(torch.float64).T
        assert np.allclose(h, ref_h.numpy(), rtol=1e-12, atol=1e-12)
        p = O.softmax_scores(h)
        ref_p = torch.softmax(ref_h, dim=1).numpy()
        assert p.dtype == np.float32
        assert np.allclose(p, ref_p, rtol=1.2e-7, atol=0)
        assert np.allclose(p.astype(np.float64).sum(axis=1), 1.0, atol=N * 6e-8)


def check_expert_ffn(O):
    g = torch.Generator().manual_seed(8)
    n, d, F = 5, 48, 32
    x = bf16_round(torch.randn(n, d, generator=g))
    Wg = bf16_round(torch.randn(F, d, generator=g) * 0.1)
    Wu = bf16_round(torch.randn(F, d, generator=g) * 0.1)
    Wd = bf16_round(torch.randn(d, F, generator=g) * 0.1)
    out = O.expert_ffn(x.to(torch.float64).numpy(), bits(Wg), bits(Wu), bits(Wd))
    X = x.to(torch.float64)
    ref = (torch.nn.functional.silu(X @ Wg.to(torch.float64).T) * (X @ Wu.to(torch.float64).T)) \
        @ Wd.to(torch.float64).T
    assert np.allclose(out, ref.numpy(), rtol=1e-12, atol=1e-13)


def check_layer_single_token(O):
    """One token with S = E: y = sum over its top-k of g_bar_i E_i(x) (Sec. 2.1-2.2)."""
    g = torch.Generator().manual_seed(12)
    N, k, d, F = 12, 3, 40, 24
    x = bf16_round(torch.randn(1, d, generator=g))
    W_g = torch.randn(N, d, generator=g) / math.sqrt(d)
    Wg = bf16_round(torch.randn(N, F, d, generator=g) * 0.1)
    Wu = bf16_round(torch.randn(N, F, d, generator=g) * 0.1)
    Wd = bf16_round(torch.randn(N, d, F, generator=g) * 0.1)
    get = lambda e: (bits(Wg[e]), bits(Wu[e]), bits(Wd[e]))
    r = O.moe_forward(bits(x), W_g.numpy(), get, k, 0, O.MODE_TOPK)
    X = x.to(torch.float64)
    h = X @ W_g.to(torch.float64).T
    val, idx = torch.topk(h[0], k)
    gbar = torch.softmax(val, dim=0)
    y = torch.zeros(d, dtype=torch.float64)
    for wgt, e in zip(gbar, idx):
        a = torch.nn.functional.silu(X[0] @ Wg[e].to(torch.float64).T) * (X[0] @ Wu[e].to(torch.float64).T)
        y += wgt * (a @ Wd[e].to(torch.float64).T)
    assert [int(e) for e in r["ids"][0]] == [int(e) for e in idx]
    assert np.allclose(r["y"][0], y.numpy(), rtol=1e-5, atol=1e-7 * float(y.abs().max()))


def check_shared_experts(O):
    """With shared experts, y = sum_i g_i E_i(x) + sum_j E^s_j(x) (Sec. 2.1):
    the layer output minus the routed-only output equals the shared experts'
    SwiGLU outputs computed with torch, for every token."""
    g = torch.Generator().manual_seed(14)
    N, k, d, F, B, Ns = 10, 2, 24, 16, 5, 2
    x = bf16_round(torch.randn(B, d, generator=g))
    W_g = torch.randn(N, d, generator=g) / math.sqrt(d)
    Wg = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
    Wu = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
    Wd = bf16_round(torch.randn(N, d, F, generator=g) * 0.2)
    Sg = bf16_round(torch.randn(Ns, F, d, generator=g) * 0.2)
    Su = bf16_round(torch.randn(Ns, F, d, generator=g) * 0.2)
    Sd = bf16_round(torch.randn(Ns, d, F, generator=g) * 0.2)
    get = lambda e: (bits(Wg[e]), bits(Wu[e]), bits(Wd[e]))
    gets = lambda j: (bits(Sg[j]), bits(Su[j]), bits(Sd[j]))
    routed = O.moe_forward(bits(x), W_g.numpy(), get, k, 3, O.MODE_BATCH)["y"]
    full = O.moe_forward(bits(x), W_g.numpy(), get, k, 3, O.MODE_BATCH, get_shared=gets,
                         n_shared=Ns)["y"]
    X = x.to(torch.float64)
    ref = torch.zeros(B, d, dtype=torch.float64)
    for j in range(Ns):
        ref += (torch.nn.functional.silu(X @ Sg[j].to(torch.float64).T) *
                (X @ Su[j].to(torch.float64).T)) @ Sd[j].to(torch.float64).T
    assert np.allclose(full - routed, ref.numpy(), rtol=1e-10, atol=1e-12)
    sub = O.moe_forward(bits(x), W_g.numpy(), get, k, 3, O.MODE_BATCH, tokens=[4, 0],
                        get_shared=gets, n_shared=Ns)["y"]
    assert np.allclose(sub, full[[4, 0]], rtol=1e-12, atol=1e-14)


def check_combine_multi_token(O):
    """y for several tokens equals per-token sums of w * E_e(x) (Sec. 2.1) computed
    with torch, for a routing with padding slots."""
    g = torch.Generator().manual_seed(13)
    N, k, d, F, B = 6, 3, 16, 8, 4
    x = bf16_round(torch.randn(B, d, generator=g))
    Wg = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
    Wu = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
    Wd = bf16_round(torch.randn(N, d, F, generator=g) * 0.2)
    ids = np.array([[0, 3, -1], [5, 0, 1], [2, -1, -1], [4, 5, 3]], dtype=np.int32)
    w = np.array([[0.7, 0.3, 0], [0.5, 0.25, 0.25], [1, 0, 0], [0.2, 0.3, 0.5]], dtype=np.float32)
    get = lambda e: (bits(Wg[e]), bits(Wu[e]), bits(Wd[e]))
    y = O.moe_ffn_combine(bits(x), ids, w, get)
    X = x.to(torch.float64)
    for t in range(B):
        ref = torch.zeros(d, dtype=torch.float64)
        for s in range(k):
            e = int(ids[t, s])
            if e < 0:
                continue
            a = torch.nn.functional.silu(X[t] @ Wg[e].to(torch.float64).T) * (X[t] @ Wu[e].to(torch.float64).T)
            ref += float(w[t, s]) * (a @ Wd[e].to(torch.float64).T)
        assert np.allclose(y[t], ref.numpy(), rtol=1e-12, atol=1e-14)
    sub = O.moe_ffn_combine(bits(x), ids, w, get, tokens=[3, 1])
    assert np.allclose(sub, y[[3, 1]], rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------- canonical column sum

def check_canonical_sum_golden(O):
    with open(os.path.join(GOLDEN, "canonical_sum.json")) as f:
        g = json.load(f)
    for col in g["columns"]:
        rows = np.zeros((col["rows"], 1), dtype=np.uint32)
        for key, val in col["rows_hex"].items():
            lo, _, hi = key.partition("-")
            rows[int(lo):int(hi or lo) + 1] = int(val, 16)
        p = rows.view(np.float32)
        got = O.canonical_column_sum(p, range(col["rows"])).view(np.uint32)[0]
        assert int(got) == int(col["expected_hex"], 16), (col["describe"], hex(int(got)))


def check_canonical_sum_bound(O, cases=20):
    """|canonical - exact| <= (5 + chunks) u sum|p|, u = 2^-24 (depth-5 tree per
    chunk plus one accumulation per chunk)."""
    rng = np.random.default_rng(17)
    for _ in range(cases):
        B = int(rng.integers(1, 150)); N = int(rng.integers(1, 10))
        p = (np.exp(rng.standard_normal((B, N)) * 3) / N).astype(np.float32)
        rows = list(rng.permutation(B)) if rng.integers(2) else list(range(B))
        got = O.canonical_column_sum(p, rows)
        ex = exact_colsum(p, rows)
        chunks = (len(rows) + 31) // 32
        for j in range(N):
            bound = (5 + chunks) * 2.0 ** -24 * float(ex[j]) * 1.0000001
            assert abs(Fraction(float(got[j])) - ex[j]) <= Fraction(bound), (B, j)


# ---------------------------------------------------------------- Algorithm 1, threshold form

def check_threshold_golden(O):
    """Hand-derived threshold selections and expert-order sums (fixture)."""
    with open(os.path.join(GOLDEN, "threshold_example.json")) as f:
        g = json.load(f)
    p = np.array(g["p"], dtype=np.float32)
    for c in g["cases"]:
        r = O.route(p, 2, 0, O.MODE_THRESH, k0=c["k0"], tau=c["tau"])
        assert sorted(mask_to_set(r["mask"])) == c["S"], (c, sorted(mask_to_set(r["mask"])))
    t = g["tree_sum"]
    v = np.array([int(h, 16) for h in t["values_hex"]], dtype=np.uint32).view(np.float32)
    got = np.float32(O.expert_tree_sum(v, set(range(v.shape[0])))).view(np.uint32)
    assert got == int(t["expected_hex"], 16), hex(int(got))
    got = np.float32(O.expert_tree_sum(v, set(t["subset"]["members"]))).view(np.uint32)
    assert got == int(t["subset"]["expected_hex"], 16), hex(int(got))


def check_threshold_bruteforce(O, cases=40):
    """With exact sums, the threshold selection is S_0 alone if f(S_0) already
    reaches tau f(E); otherwise a superset of S_0 reaching tau f(E) (or all of
    E) such that no superset of S_0 with one expert fewer reaches it, and with
    the largest f among the supersets of its size (Corollary 1)."""
    rng = np.random.default_rng(21)
    done = 0
    while done < cases:
        N = int(rng.integers(3, 10))
        B = int(rng.integers(1, 6))
        k0 = int(rng.integers(0, 3))
        tau = float(rng.integers(0, 33)) / 32.0
        p = quantised_scores(rng, B, N)
        col = exact_colsum(p, range(B))
        total = sum(col, Fraction(0))
        target = Fraction(tau) * total
        if Fraction(float(np.float32(np.float32(tau) * np.float32(float(total))))) != target:
            continue   # keep to cases whose target is exact in fp32
        S0 = set()
        for i in range(B):
            S0 |= set(lexsort_top(p[i], k0, range(N)))
        S = mask_to_set(O.route(p, 1, 0, O.MODE_THRESH, k0=k0, tau=tau)["mask"])
        f = lambda A: sum((col[j] for j in A), Fraction(0))
        assert S0 <= S
        rest = [j for j in range(N) if j not in S0]
        if f(S0) >= target:
            assert S == S0
        else:
            assert f(S) >= target or len(S) == N
            fewer = len(S) - len(S0) - 1
            for c in itertools.combinations(rest, fewer):
                assert f(S0 | set(c)) < target, (S0, c, target)
            best = max(f(S0 | set(c)) for c in itertools.combinations(rest, len(S) - len(S0)))
            assert f(S) == best
        done += 1


def check_threshold_consistency(O):
    """On softmax scores: the threshold selection equals the fixed-budget one
    with m = |S| - |S_0| (one greedy order), and grows with tau."""
    rng = np.random.default_rng(5)
    for trial in range(6):
        B, N = int(rng.integers(1, 40)), int(rng.integers(8, 80))
        h = rng.standard_normal((B, N)) * 1.5
        p = (np.exp(h) / np.exp(h).sum(axis=1, keepdims=True)).astype(np.float32)
        k0 = trial % 3
        prev = None
        for tau in (0.0, 0.2, 0.45, 0.7, 0.9, 1.0):
            S = mask_to_set(O.route(p, 2, 0, O.MODE_THRESH, k0=k0, tau=tau)["mask"])
            S0 = O.warmup_set(p, k0, range(B))
            Sb = mask_to_set(O.route(p, 2, len(S) - len(S0), O.MODE_BATCH, k0=k0)["mask"])
            assert S == Sb, (tau, len(S), len(Sb))
            if prev is not None:
                assert prev <= S
            prev = S


# ---------------------------------------------------------------- Eq. 1: layer stack

def check_bf16_rounding(O):
    """Round-to-nearest-even to bf16: equals torch's fp32 -> bf16 on fp32 values
    (ties and subnormals included), and rounds fp64 values once (hand-derived
    cases where rounding through fp32 first would differ)."""
    rng = np.random.default_rng(3)
    v = (rng.standard_normal(20000) * np.exp(rng.uniform(-40, 40, 20000))).astype(np.float32)
    base = torch.from_numpy(v).to(torch.bfloat16).to(torch.float32).numpy()
    ties = (base.astype(np.float64) * (1 + 2.0 ** -8)).astype(np.float32)   # halfway points
    sub = (rng.standard_normal(2000) * 2.0 ** -130).astype(np.float32)
    for vals in (v, ties, sub):
        want = torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        got = O.f64_to_bf16_bits(vals.astype(np.float64))
        assert np.array_equal(got, want)
    # 1 + 2^-8 + 2^-30: above the tie between 1 and 1 + 2^-7 -> 1 + 2^-7 (0x3f81);
    # through fp32 first it becomes the tie 1 + 2^-8 and then 1.0 (even).
    # -(1 + 3 * 2^-8 - 2^-40): below the tie between 1 + 2^-7 and 1 + 2^-6 -> 0xbf81.
    got = O.f64_to_bf16_bits(np.array([1 + 2.0 ** -8 + 2.0 ** -30, -(1 + 3 * 2.0 ** -8 - 2.0 ** -40)]))
    assert list(got) == [0x3F81, 0xBF81], [hex(int(g)) for g in got]


def check_layer_budgets(O):
    """m_l = K / L (Sec. 3.2): integers summing to K that differ by at most one,
    larger first."""
    assert O.layer_budgets(10, 4) == [3, 3, 2, 2]
    assert O.layer_budgets(24 * 58, 58) == [24] * 58
    assert O.layer_budgets(3, 5) == [1, 1, 1, 0, 0]
    for K in range(0, 60):
        for L in range(1, 9):
            m = O.layer_budgets(K, L)
            assert sum(m) == K and max(m) - min(m) <= 1 and m == sorted(m, reverse=True)


def _tiny_stack(seed, L, N, d, F, zero=False):
    g = torch.Generator().manual_seed(seed)
    layers = []
    for _ in range(L):
        Wg = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
        Wu = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
        Wd = bf16_round(torch.randn(N, d, F, generator=g) * (0.0 if zero else 0.2))
        W_g = (torch.randn(N, d, generator=g) / math.sqrt(d)).numpy()
        layers.append({"W_g": W_g, "get_expert": (lambda e, Wg=Wg, Wu=Wu, Wd=Wd:
                                                  (bits(Wg[e]), bits(Wu[e]), bits(Wd[e])))})
    return layers


def check_stack_invariants(O):
    """Residual identity with zero expert outputs; each layer gets budget m_l
    (|S_l| = m_l with k0 = 0); budget N in every layer is a plain top-k stack."""
    B, N, d, F, k, L = 6, 8, 16, 8, 2, 3
    x = bits(bf16_round(torch.randn(B, d, generator=torch.Generator().manual_seed(1))))
    zero = _tiny_stack(2, L, N, d, F, zero=True)
    outs = O.moe_stack_forward(x, zero, k, 7, O.MODE_BATCH)
    assert all(np.array_equal(o, x) for o in outs)
    layers = _tiny_stack(3, L, N, d, F)
    st = []
    O.moe_stack_forward(x, layers, k, 7, O.MODE_BATCH, stats=st)
    assert [r["n_selected"] for r in st] == O.layer_budgets(7, L) == [3, 2, 2]
    a = O.moe_stack_forward(x, layers, k, N * L, O.MODE_BATCH)
    b = O.moe_stack_forward(x, layers, k, 0, O.MODE_TOPK)
    assert all(np.array_equal(p, q) for p, q in zip(a, b))
    assert not np.array_equal(a[-1], x)


# ---------------------------------------------------------------- Sec. 2.2: sparse gating scores

def check_topk_gating(O):
    """Sec. 2.2's g has k nonzeros per token, proportional to p on the token's
    top-k and summing to 1; they equal plain top-k routing's weights; and a
    hand-derived example."""
    rng = np.random.default_rng(8)
    p = W_softmax(rng, 20, 40)
    for k in (1, 3, 8):
        g = O.topk_gating(p, k)
        r = O.route(p, k, 0, O.MODE_TOPK)
        assert np.all((g > 0).sum(axis=1) == k)
        for i in range(p.shape[0]):
            nz = sorted(np.nonzero(g[i])[0].tolist())
            assert nz == sorted(lexsort_top(p[i], k, range(p.shape[1])))
            assert np.array_equal(g[i, r["ids"][i]], r["w"][i])     # same fp32 values
            assert abs(float(np.sum(g[i].astype(np.float64))) - 1.0) < 1e-6
    # p = [0.5, 0.25, 0.125, 0.125], k = 2: T = {0, 1}, D = 0.75,
    # g = [fp32(0.5/0.75), fp32(0.25/0.75), 0, 0] = [0x3f2aaaab, 0x3eaaaaab, 0, 0]
    g = O.topk_gating(np.array([[0.5, 0.25, 0.125, 0.125]], dtype=np.float32), 2)
    assert [hex(int(v)) for v in g[0].view(np.uint32)] == ["0x3f2aaaab", "0x3eaaaaab", "0x0", "0x0"]


def W_softmax(rng, B, N, scale=1.5):
    h = rng.standard_normal((B, N)) * scale
    return (np.exp(h) / np.exp(h).sum(axis=1, keepdims=True)).astype(np.float32)


def check_sparse_selection(O, cases=30):
    """With sparse scores: S is S_0 plus only experts some token ranks in its
    top-k; |S| = |S_0| + min(m, available); among supersets of S_0 of that
    size S maximises the sparse objective (brute force); budget N gives plain
    top-k routing exactly."""
    rng = np.random.default_rng(17)
    done = 0
    while done < cases:
        N = int(rng.integers(4, 10))
        B = int(rng.integers(1, 6))
        k = int(rng.integers(1, min(N, 4) + 1))
        k0 = int(rng.integers(0, k + 1))
        m = int(rng.integers(0, N + 1))
        p = quantised_scores(rng, B, N)
        g = O.topk_gating(p, k)
        union = set()
        for i in range(B):
            union |= set(lexsort_top(p[i], k, range(N)))
        S0 = set()
        for i in range(B):
            S0 |= set(lexsort_top(p[i], k0, range(N)))
        S = mask_to_set(O.route(p, k, m, O.MODE_BATCH, k0=k0, sparse_scores=1)["mask"])
        assert S0 <= S <= (S0 | union)
        avail = [j for j in union if j not in S0]
        assert len(S) == len(S0) + min(m, len(avail))
        col = exact_colsum(g, range(B))
        best = max(sum((col[j] for j in c), Fraction(0))
                   for c in itertools.combinations(avail, len(S) - len(S0)))
        assert sum((col[j] for j in S - S0), Fraction(0)) == best
        done += 1
    for trial in range(5):
        B, N, k = 12, 24, 4
        p = W_softmax(rng, B, N)
        a = O.route(p, k, N, O.MODE_BATCH, k0=1, sparse_scores=1)
        b = O.route(p, k, 0, O.MODE_TOPK)
        assert np.array_equal(a["ids"], b["ids"]) and np.array_equal(a["w"], b["w"])
        assert a["n_selected"] == b["union_topk"]
        for mode, prm in ((O.MODE_GROUP, dict(n_groups=4, m_g=N)),
                          (O.MODE_HIER, dict(m_r=N, tokens_per_request=3))):
            c = O.route(p, k, N, mode, k0=1, sparse_scores=1, **prm)
            assert mask_to_set(c["mask"]) == mask_to_set(a["mask"]), mode
        # tau = 1 stops once the running fp32 sum reaches f(E): never beyond the union
        c = O.route(p, k, 0, O.MODE_THRESH, k0=1, sparse_scores=1, tau=1.0)
        assert mask_to_set(c["mask"]) <= mask_to_set(a["mask"])


def check_expert_parallel(O):
    """Sec. 5, experts split over G devices: device g's exchange rows hold, at
    row offsets[e] + i, the SwiGLU output (torch float64) of the i-th pair of
    each of its experts e, and at n_pairs + j B + t (device 0 only) token t
    through shared expert j; all other rows are zero.  The rows of all
    devices, summed, combine to the one-device layer output exactly."""
    g = torch.Generator().manual_seed(21)
    N, k, d, F, B, Ns = 8, 2, 16, 8, 5, 1
    x = bf16_round(torch.randn(B, d, generator=g))
    W_g = torch.randn(N, d, generator=g) / math.sqrt(d)
    Wg = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
    Wu = bf16_round(torch.randn(N, F, d, generator=g) * 0.2)
    Wd = bf16_round(torch.randn(N, d, F, generator=g) * 0.2)
    Sg = bf16_round(torch.randn(Ns, F, d, generator=g) * 0.2)
    Su = bf16_round(torch.randn(Ns, F, d, generator=g) * 0.2)
    Sd = bf16_round(torch.randn(Ns, d, F, generator=g) * 0.2)
    get = lambda e: (bits(Wg[e]), bits(Wu[e]), bits(Wd[e]))
    gets = lambda j: (bits(Sg[j]), bits(Su[j]), bits(Sd[j]))
    X = x.to(torch.float64)

    def swiglu(t, Wg_, Wu_, Wd_):
        a = torch.nn.functional.silu(X[t] @ Wg_.to(torch.float64).T) * (X[t] @ Wu_.to(torch.float64).T)
        return (a @ Wd_.to(torch.float64).T).numpy()

    ref = O.moe_forward(bits(x), W_g.numpy(), get, k, 3, O.MODE_BATCH, get_shared=gets, n_shared=Ns)
    for G in (2, 4):
        total = 0
        for dev in range(G):
            lo, hi = (N // G) * dev, (N // G) * (dev + 1)
            r = O.moe_forward_ep_rank(bits(x), W_g.numpy(), get, k, 3, O.MODE_BATCH, G, dev,
                                      get_shared=gets, n_shared=Ns)
            n_pairs = len(r["perm"])
            for row in range(r["out"].shape[0]):
                if row < n_pairs:
                    q = int(r["perm"][row])
                    e = int(r["ids"][q // k, q % k])
                    want = swiglu(q // k, Wg[e], Wu[e], Wd[e]) if lo <= e < hi else np.zeros(d)
                else:
                    t = (row - n_pairs) % B
                    want = swiglu(t, Sg[0], Su[0], Sd[0]) if dev == 0 else np.zeros(d)
                assert np.allclose(r["out"][row], want, rtol=1e-12, atol=1e-14), (G, dev, row)
            total = total + r["out"]
        assert np.array_equal(O.ep_combine(ref, total, Ns), ref["y"])


ALL_CHECKS = [
    check_closed_form_golden, check_union_statistics, check_greedy_bruteforce,
    check_hier_bruteforce, check_hier_single_request_is_batch, check_group,
    check_refine_invariants, check_zero_scores, check_budget_n_is_topk, check_permutation,
    check_router_softmax, check_expert_ffn, check_layer_single_token, check_shared_experts,
    check_combine_multi_token, check_canonical_sum_golden, check_canonical_sum_bound,
    check_threshold_golden, check_threshold_bruteforce, check_threshold_consistency,
    check_bf16_rounding, check_layer_budgets, check_stack_invariants,
    check_topk_gating, check_sparse_selection, check_expert_parallel,
]
