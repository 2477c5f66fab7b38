"""GPU parity of xshare_route (steps a3-a7) against the oracle, through the C ABI.

Scores are produced on the CPU (the oracle's softmax of seeded router inputs,
or seeded synthetic score matrices), fed to both sides, and every integer
output must match bit for bit: the selected mask, the top-k ids, the
permutation, the counts and offsets and the statistics.  The fp32 weights are
computed by the same sequence of correctly rounded fp32 operations on both
sides, so they must match bit for bit too.
"""
import numpy as np
import pytest
import torch

from oracle import xshare_oracle as O
from paper_2602_07265_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare
    return xshare


def gpu_route(X, p: np.ndarray, k: int, budget: int, mode: int, **params):
    B, N = p.shape
    dev = torch.device("cuda")
    prm = X.route_params(**{**dict(k0=0, m_r=0, tokens_per_request=1, n_groups=1, m_g=0, tau=0.0,
                                   sparse_scores=0), **params})
    ws = torch.empty(X.xshare_workspace_size(B, N, k, 0, 0, mode, prm), dtype=torch.uint8, device=dev)
    scores = torch.from_numpy(np.ascontiguousarray(p)).to(dev)
    out = dict(
        mask=torch.full((N,), 7, dtype=torch.uint8, device=dev),
        ids=torch.full((B, k), 99, dtype=torch.int32, device=dev),
        w=torch.full((B, k), 9.0, dtype=torch.float32, device=dev),
        stats=torch.full((8,), -5, dtype=torch.int32, device=dev),
        counts=torch.full((N,), -1, dtype=torch.int32, device=dev),
        offsets=torch.full((N + 1,), -1, dtype=torch.int32, device=dev),
        perm=torch.full((B * k,), -1, dtype=torch.int32, device=dev),
    )
    X.xshare_route(scores, k, budget, mode, prm, out["mask"], out["ids"], out["w"], ws,
                   stats=out["stats"], expert_counts=out["counts"],
                   expert_offsets=out["offsets"], perm=out["perm"])
    torch.cuda.synchronize()
    r = {name: t.cpu().numpy() for name, t in out.items()}
    r["stats"] = X.stats_dict(out["stats"])
    return r


def assert_route_equal(g, ref, k):
    assert np.array_equal(g["mask"], ref["mask"]), "selected set"
    assert np.array_equal(g["ids"], ref["ids"]), "top-k ids"
    assert np.array_equal(g["w"].view(np.uint32), ref["w"].view(np.uint32)), "weights (bits)"
    assert np.array_equal(g["counts"], ref["counts"]), "counts"
    assert np.array_equal(g["offsets"], ref["offsets"]), "offsets"
    P = int(ref["offsets"][-1])
    assert np.array_equal(g["perm"][:P], ref["perm"]), "permutation"
    s = g["stats"]
    assert s["status"] == 0
    assert s["n_selected"] == ref["n_selected"]
    assert s["n_used"] == ref["n_used"]
    assert s["union_topk"] == ref["union_topk"]
    assert s["max_group_load"] == ref["max_group_load"]
    assert s["n_pairs"] == P


def oracle_scores(w: W.Workload, seed: int) -> np.ndarray:
    x, W_g = W.router_inputs(w, seed)
    return O.softmax_scores(O.router_logits(W.bf16_bits(x), W_g.numpy()))


def check(X, p, k, budget, mode, **params):
    full = dict(k0=0, m_r=0, tokens_per_request=1, n_groups=1, m_g=0, tau=0.0, sparse_scores=0)
    full.update(params)
    ref = O.route(p, k, budget, mode, **full)
    g = gpu_route(X, p, k, budget, mode, **full)
    assert_route_equal(g, ref, k)
    return ref


# ---- the five workloads, their own mode, seeds 0-2 ----
WL_CASES = [
    (W.TINY, {}), (W.TINY.with_(k0=1), {}),
    (W.OLMOE.with_(B=8, budget=16), {}), (W.OLMOE.with_(B=16, budget=24, k0=1), {}),
    (W.OLMOE.with_(B=32, budget=32), {}), (W.OLMOE.with_(B=64, budget=48, k0=1), {}),
    (W.QWEN3, {}), (W.QWEN3.with_(m_r=5), {}), (W.QWEN3.with_(k0=2), {}),
    (W.QWEN3.with_(k0=0, budget=16), {}), (W.QWEN3.with_(B=16), {}), (W.QWEN3.with_(B=64), {}),
    (W.DSR1.with_(B=8), {}), (W.DSR1, {}), (W.DSR1.with_(B=128, budget=64), {}),
    (W.DSR1.with_(k0=0, budget=32), {}),
    (W.DSR1_GROUP, {}), (W.DSR1_GROUP.with_(k0=0), {}), (W.DSR1_GROUP.with_(k0=0, m_g=8), {}),
    (W.DSR1_GROUP.with_(k0=0, m_g=16), {}),
]


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("case", range(len(WL_CASES)))
def test_workload_route_parity(X, case, seed):
    w, _ = WL_CASES[case]
    p = oracle_scores(w, seed)
    check(X, p, w.k, w.budget, w.mode, **w.params())


@pytest.mark.parametrize("name", ["tiny", "olmoe", "qwen3", "dsr1"])
def test_plain_topk_and_batch_on_workloads(X, name):
    w = W.WORKLOADS[name]
    p = oracle_scores(w, 0)
    ref = check(X, p, w.k, 0, W.MODE_TOPK)
    assert ref["n_selected"] == w.N
    for m in (16, 24, 32, 48, 64, 128):
        check(X, p, w.k, m, W.MODE_BATCH, k0=1)


# ---- edge cases ----
@pytest.mark.parametrize("B,N,k,budget,mode,params,ties", [
    (1, 64, 8, 24, W.MODE_BATCH, dict(k0=1), False),            # one token
    (32, 64, 1, 4, W.MODE_BATCH, dict(k0=0), False),            # k = 1
    (32, 64, 8, 3, W.MODE_BATCH, dict(k0=0), False),            # |S| < k
    (32, 64, 8, 0, W.MODE_BATCH, dict(k0=0), False),            # S empty: no routing at all
    (32, 64, 8, 0, W.MODE_BATCH, dict(k0=1), False),            # warm-up only (paper's (0,1))
    (32, 64, 8, 24, W.MODE_BATCH, dict(k0=0), True),            # tie-heavy scores
    (40, 50, 8, 20, W.MODE_BATCH, dict(k0=2), False),           # N not a multiple of 32
    (40, 50, 8, 20, W.MODE_TOPK, {}, True),
    (33, 1000, 16, 100, W.MODE_BATCH, dict(k0=16), False),       # large N, k = k0 = 16
    (64, 1024, 8, 0, W.MODE_HIER, dict(k0=1, m_r=4, tokens_per_request=4), False),
    (96, 1024, 8, 0, W.MODE_GROUP, dict(k0=0, n_groups=64, m_g=2), True),
    (256, 128, 8, 8, W.MODE_HIER, dict(k0=1, m_r=200, tokens_per_request=4), False),  # m_r > N
    (128, 64, 8, 0, W.MODE_HIER, dict(k0=0, m_r=6, tokens_per_request=64), False),   # 2 chunks/request
    (96, 64, 8, 4, W.MODE_HIER, dict(k0=2, m_r=3, tokens_per_request=32), True),
    (16, 64, 8, 0, W.MODE_HIER, dict(k0=0, m_r=3, tokens_per_request=1), False),
    (96, 128, 8, 2, W.MODE_HIER, dict(k0=1, m_r=3, tokens_per_request=3), False),  # straddles chunks
    (120, 128, 8, 0, W.MODE_HIER, dict(k0=1, m_r=4, tokens_per_request=8), True),  # 8 | 32
    (144, 64, 4, 5, W.MODE_HIER, dict(k0=2, m_r=2, tokens_per_request=48), False),  # 48 > 32
    (65, 256, 8, 24, W.MODE_BATCH, dict(k0=1), False),                          # 3 chunks, ragged
    # chunk counts around the refinement kernel (3 to 9 chunks)
    (257, 256, 8, 24, W.MODE_BATCH, dict(k0=1), False),                         # 9 chunks, ragged
    (200, 128, 8, 0, W.MODE_THRESH, dict(k0=1, tau=0.6), False),                # 7 chunks, THRESH
    (160, 64, 8, 0, W.MODE_TOPK, {}, True),                                     # 5 chunks, top-k
    (100, 64, 8, 3, W.MODE_BATCH, dict(k0=0), False),                           # 4 chunks, |S| < k
    (96, 64, 8, 0, W.MODE_BATCH, dict(k0=0), False),                            # 3 chunks, S empty
    (64, 256, 8, 0, W.MODE_GROUP, dict(k0=1, n_groups=8, m_g=5), False),        # 2 chunks (fused)
    (256, 256, 8, 0, W.MODE_GROUP, dict(k0=0, n_groups=1, m_g=24), False),     # G = 1 is BATCH
    (256, 256, 8, 0, W.MODE_GROUP, dict(k0=1, n_groups=256, m_g=1), False),    # singleton groups
    (256, 256, 8, 0, W.MODE_GROUP, dict(k0=3, n_groups=8, m_g=2), False),      # S_0 beyond m_g G
    (64, 256, 8, 0, W.MODE_GROUP, dict(k0=0, n_groups=8, m_g=40), True),       # groups exhausted
    (2048, 256, 8, 32, W.MODE_BATCH, dict(k0=1), False),                       # large B
    (8192, 64, 2, 8, W.MODE_BATCH, dict(k0=0), True),                          # B at the limit
    (37, 96, 5, 11, W.MODE_BATCH, dict(k0=3, n_groups=3), False),              # ragged, group stat
])
def test_route_edge_cases(X, B, N, k, budget, mode, params, ties):
    p = W.random_scores(B, N, seed=B * 7 + N, ties=ties)
    check(X, p, k, budget, mode, **params)


def tied_boundary_scores(B, N, tied, high, seed):
    """Scores whose column sums put a group of equal columns (`tied`, equal
    entries in every row) right at the budget boundary, below the `high`
    columns and above all the others; the per-token ranking ties too."""
    rng = np.random.default_rng(seed)
    p = (rng.uniform(0.5, 1.0, size=(B, N)) / (4.0 * N)).astype(np.float32)
    p[:, high] = (rng.uniform(4.0, 8.0, size=(B, len(high))) / N).astype(np.float32)
    p[:, tied] = np.float32(2.0 / N)
    return p


@pytest.mark.parametrize("k0,budget", [(0, 10), (0, 7), (1, 7), (0, 16)])
def test_batch_ties_at_the_budget_boundary(X, k0, budget):
    """BATCH takes the budget best columns in (score descending, index
    ascending) order: with ten equal columns at the boundary the lowest
    indices win, across the lanes and slots of the warp's candidate lists
    (indices 3 .. 63 and, for N = 256, beyond 128)."""
    for N, tied, high in ((64, [3, 17, 20, 33, 40, 41, 50, 58, 61, 63], [0, 9, 30, 31, 45, 60]),
                          (256, [5, 37, 70, 99, 130, 131, 160, 200, 201, 255], [1, 2, 64, 128, 190, 254])):
        p = tied_boundary_scores(32, N, tied, high, seed=N + budget)
        ref = check(X, p, 8, budget, W.MODE_BATCH, k0=k0)
        sel = set(np.flatnonzero(ref["mask"]).tolist())
        assert set(high) <= sel or k0 > 0


@pytest.mark.parametrize("B,N,budget,k0", [(32, 256, 24, 1), (64, 256, 40, 0), (96, 1024, 60, 2)])
def test_refinement_over_a_short_selected_list_with_ties(X, B, N, budget, k0):
    """Refinement over a compact list of S (|S| <= 128 with N >= 256):
    per-token ties broken by the lower expert index, as over all N."""
    p = W.random_scores(B, N, seed=B + N + budget, ties=True)
    check(X, p, 8, budget, W.MODE_BATCH, k0=k0)


def test_zero_rows_get_equal_weights(X):
    p = W.random_scores(12, 64, seed=3)
    p[[0, 5, 11]] = 0.0
    check(X, p, 8, 16, W.MODE_BATCH, k0=1)


def test_hier_one_request_is_batch(X):
    p = W.random_scores(32, 128, seed=9)
    a = gpu_route(X, p, 8, 0, W.MODE_HIER, k0=1, m_r=20, tokens_per_request=32)
    b = gpu_route(X, p, 8, 20, W.MODE_BATCH, k0=1)
    for key in ("mask", "ids", "w", "perm"):
        assert np.array_equal(a[key], b[key]), key


def test_selection_activates_fewer_experts_than_topk(X):
    """At equal budget the selected set is smaller than the plain top-k union
    (the paper's premise, Sec. 1 / Sec. 3)."""
    w = W.DSR1
    p = oracle_scores(w, 0)
    g = gpu_route(X, p, w.k, w.budget, w.mode, **w.params())
    assert g["stats"]["n_used"] <= g["stats"]["n_selected"] < g["stats"]["union_topk"]


def test_repeatable(X):
    p = W.random_scores(64, 256, seed=1, ties=True)
    a = gpu_route(X, p, 8, 32, W.MODE_BATCH, k0=1)
    b = gpu_route(X, p, 8, 32, W.MODE_BATCH, k0=1)
    for key in ("mask", "ids", "w", "perm", "counts"):
        assert np.array_equal(a[key], b[key]), key


# ---- Algorithm 1 in its threshold form ----
TAUS = [0.0, 0.25, 0.5, 0.8, 0.95, 1.0]


@pytest.mark.parametrize("tau", TAUS)
@pytest.mark.parametrize("name", ["tiny", "olmoe", "qwen3", "dsr1", "dsr1_group"])
def test_threshold_route_parity(X, name, tau):
    w = W.WORKLOADS[name]
    for k0, seed in ((0, 0), (1, 1)):
        p = oracle_scores(w, seed)
        check(X, p, w.k, 0, W.MODE_THRESH, k0=k0, tau=tau,
              n_groups=w.n_groups)


@pytest.mark.parametrize("B,N,k,k0,tau,ties", [
    (1, 64, 8, 0, 0.5, False),
    (32, 50, 8, 1, 0.6, False),        # N not a multiple of 32
    (40, 1000, 16, 2, 0.7, False),     # 32 candidates per lane
    (96, 1024, 8, 0, 0.99, True),      # tie-heavy, nearly all the mass
    (64, 256, 8, 0, 1.0, True),        # tau = 1: every expert
    (2048, 256, 8, 1, 0.4, False),     # many chunks
    (8192, 64, 2, 0, 0.3, True),       # B at the limit
    (33, 128, 4, 4, 0.0, False),       # tau = 0: the warm-up set alone
])
def test_threshold_edge_cases(X, B, N, k, k0, tau, ties):
    p = W.random_scores(B, N, seed=B + N + k0, ties=ties)
    check(X, p, k, 0, W.MODE_THRESH, k0=k0, tau=tau)


def test_threshold_tau_grid_bit_exact(X):
    """Many tau values on one score matrix: every |S| from the warm-up set to
    N is met, so each stopping point is compared."""
    p = W.random_scores(48, 128, seed=11)
    sizes = set()
    for i in range(41):
        ref = check(X, p, 8, 0, W.MODE_THRESH, k0=1, tau=i / 40.0)
        sizes.add(ref["n_selected"])
    assert len(sizes) > 20


def test_threshold_zero_scores(X):
    p = W.random_scores(16, 64, seed=2)
    p[:, 10:] = 0.0
    check(X, p, 8, 0, W.MODE_THRESH, k0=0, tau=1.0)
    p[:] = 0.0
    check(X, p, 8, 0, W.MODE_THRESH, k0=0, tau=0.5)


# ---- sparse-score reading (Sec. 2.2's top-k-masked g in the column sums) ----
@pytest.mark.parametrize("case", range(len(WL_CASES)))
def test_sparse_scores_route_parity(X, case):
    w, _ = WL_CASES[case]
    p = oracle_scores(w, 5)
    ref = check(X, p, w.k, w.budget, w.mode, **{**w.params(), "sparse_scores": 1})
    assert ref["n_selected"] <= ref["union_topk"] + len(O.warmup_set(p, w.k0, range(w.B)))


@pytest.mark.parametrize("B,N,k,budget,mode,params", [
    (32, 64, 8, 64, W.MODE_BATCH, dict(k0=1)),                         # budget beyond the union
    (33, 1000, 16, 100, W.MODE_BATCH, dict(k0=16)),
    (96, 128, 8, 2, W.MODE_HIER, dict(k0=1, m_r=3, tokens_per_request=3)),   # straddling requests
    (144, 64, 4, 5, W.MODE_HIER, dict(k0=2, m_r=2, tokens_per_request=48)),
    (256, 256, 8, 0, W.MODE_GROUP, dict(k0=1, n_groups=8, m_g=40)),     # groups run out of gain
    (64, 256, 8, 0, W.MODE_THRESH, dict(k0=1, tau=0.9)),
    (2048, 256, 8, 32, W.MODE_BATCH, dict(k0=1)),
    (40, 50, 8, 20, W.MODE_BATCH, dict(k0=0)),
])
def test_sparse_scores_edge_cases(X, B, N, k, budget, mode, params):
    for ties in (False, True):
        p = W.random_scores(B, N, seed=B + 3 * N, ties=ties)
        check(X, p, k, budget, mode, sparse_scores=1, **params)


def test_sparse_budget_n_is_plain_topk(X):
    p = W.random_scores(64, 128, seed=4)
    a = gpu_route(X, p, 8, 128, W.MODE_BATCH, k0=1, sparse_scores=1)
    b = gpu_route(X, p, 8, 0, W.MODE_TOPK)
    assert np.array_equal(a["ids"], b["ids"]) and np.array_equal(a["w"], b["w"])
    assert a["stats"]["n_selected"] == b["stats"]["union_topk"]
