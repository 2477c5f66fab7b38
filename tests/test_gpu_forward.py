"""GPU parity of xshare_moe_forward (steps a1-a9) against the oracle, through the C ABI.

Inputs are seeded and synthetic (paper_2602_07265_gb300.workloads); the
oracle computes everything itself from the same inputs (router in fp64,
softmax rounded once to fp32, selection on its own fp32 scores, FFN in fp64).

Checks:
* scores: |p_gpu - p_ref| <= P_RTOL * p_ref elementwise (fp32 router and
  softmax vs fp64; see P_RTOL);
* selection: the mask and the top-k ids equal the oracle's, provided the
  oracle's decision is robust to perturbing its scores by the scores
  tolerance (checked, never assumed);
* output: max|y - y_ref| / max|y_ref| <= 2e-2 and ||y - y_ref||_F / ||y_ref||_F
  <= 1e-2 (bf16 output of an fp32-accumulated path with a bf16 activation).
At the DeepSeek-R1 shapes up to B = 128 every token is compared; at B = 256
the first 128 tokens (one full 128-row FFN tile's worth).  Each comparison
records whether the near-tie rule (below) had to drop tokens; a last test in
this file bounds how often that happened.
"""
import numpy as np
import pytest
import torch

from oracle import xshare_oracle as O
from paper_2602_07265_gb300 import workloads as W

pytestmark = pytest.mark.gpu

# Relative tolerance on the fp32 softmax scores.  h = W_g x is accumulated in
# fp32 over d terms in a fixed order: each lane adds d/128 float4 steps, then
# a 5-level butterfly.  With |x_c w_c| ~ 0.02 and partial sums ~ 0.3, the
# rounding error of h is a few 1e-7 absolute; a softmax score's relative error
# is at most |dh_j| + |d logsumexp| plus a few ulps of expf and the division.
P_RTOL = 2e-5
MAX_REL = 2e-2
FRO_REL = 1e-2


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare
    return xshare


_weights_cache = {}


def device_weights(w: W.Workload, seed: int):
    key = (w.N, w.d, w.F, seed)
    if key not in _weights_cache:
        _weights_cache.clear()
        torch.cuda.empty_cache()
        _weights_cache[key] = W.expert_weights(w, seed, device="cuda")
    return _weights_cache[key]


def gpu_forward(X, w: W.Workload, x, W_g, weights, shared=None):
    dev = torch.device("cuda")
    Wg, Wu, Wd = weights
    prm = X.route_params(**w.params())
    n_shared = 0 if shared is None else shared[0].shape[0]
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, n_shared),
                     dtype=torch.uint8, device=dev)
    out = dict(
        y=torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev),
        p=torch.empty(w.B, w.N, dtype=torch.float32, device=dev),
        mask=torch.empty(w.N, dtype=torch.uint8, device=dev),
        ids=torch.empty(w.B, w.k, dtype=torch.int32, device=dev),
        w=torch.empty(w.B, w.k, dtype=torch.float32, device=dev),
        stats=torch.zeros(8, dtype=torch.int32, device=dev),
    )
    X.xshare_moe_forward(x.to(dev), W_g.to(dev), Wg, Wu, Wd, w.k, w.budget, w.mode, prm,
                         out["y"], ws, scores_out=out["p"], sel_mask=out["mask"],
                         topk_ids=out["ids"], topk_w=out["w"], stats=out["stats"],
                         shared=shared)
    torch.cuda.synchronize()
    r = {name: t.cpu() for name, t in out.items()}
    r["stats"] = X.stats_dict(out["stats"])
    r["y"] = r["y"].float().numpy().astype(np.float64)
    for name in ("p", "mask", "ids", "w"):
        r[name] = r[name].numpy()
    return r


def robust_selection(p, w: W.Workload, rtol: float, trials: int = 6) -> bool:
    """True if the oracle's routing is unchanged when its scores move by up to rtol
    (random relative perturbations, including the all-up / all-down extremes)."""
    base = O.route(p, w.k, w.budget, w.mode, **w.params())
    rng = np.random.default_rng(0)
    for i in range(trials):
        if i < 2:
            f = 1.0 + rtol * (1 if i == 0 else -1) * np.sign(rng.standard_normal(p.shape))
        else:
            f = 1.0 + rtol * rng.uniform(-1, 1, size=p.shape)
        q = (p.astype(np.float64) * f).astype(np.float32)
        r = O.route(q, w.k, w.budget, w.mode, **w.params())
        if not (np.array_equal(r["mask"], base["mask"]) and np.array_equal(r["ids"], base["ids"])):
            return False
    return True


# One entry per compare() call: (case label, tokens dropped by the near-tie rule).
NEAR_TIE_LOG = []
# At most this fraction of the compared cases may fall back to the near-tie
# rule (routing differing from the oracle's on a near-tie of its fp32 scores).
NEAR_TIE_MAX_FRACTION = 0.05


def compare(w, g, x, W_g, weights, tokens=None, shared=None):
    """Check a GPU forward against the oracle; returns (ref, max_rel, fro, n_tokens_compared).

    The GPU decides its selection on its own fp32 scores, which differ from
    the oracle's by rounding (|dp| / p <= P_RTOL, checked).  Its mask and ids
    must equal the oracle's unless the oracle's own decision flips under a
    perturbation of the size actually observed (a near-tie); then y is
    compared on every token whose routing (ids) is identical."""
    Wg, Wu, Wd = weights
    xb = W.bf16_bits(x)

    def get(e):
        return W.bf16_bits(Wg[e]), W.bf16_bits(Wu[e]), W.bf16_bits(Wd[e])

    extra = {}
    if shared is not None:
        Sg, Su, Sd = shared
        extra = dict(n_shared=Sg.shape[0], get_shared=lambda j: (
            W.bf16_bits(Sg[j]), W.bf16_bits(Su[j]), W.bf16_bits(Sd[j])))
    ref = O.moe_forward(xb, W_g.numpy(), get, w.k, w.budget, w.mode, tokens=tokens,
                        **extra, **w.params())
    rel = np.abs(g["p"].astype(np.float64) - ref["p"]) / ref["p"].astype(np.float64)
    assert rel.max() <= P_RTOL, f"scores: max relative error {rel.max():.3e}"
    toks = list(range(w.B)) if tokens is None else list(tokens)
    same_mask = np.array_equal(g["mask"], ref["mask"])
    same_row = np.all(g["ids"] == ref["ids"], axis=1)
    if not (same_mask and same_row.all()):
        eps = max(4 * float(rel.max()), 1e-6)
        assert not robust_selection(ref["p"], w, eps), \
            "routing differs from the oracle's although its decision is not near a tie"
    keep = [i for i, t in enumerate(toks) if same_row[t]]
    dropped = len(toks) - len(keep)
    NEAR_TIE_LOG.append((f"{w.name} B={w.B} mode={w.mode}", dropped, same_mask))
    print(f"[{w.name} B={w.B} mode={w.mode}] p_rel_max={rel.max():.2e} same_mask={same_mask} "
          f"same_rows={int(same_row.sum())}/{w.B} compared={len(keep)}/{len(toks)}"
          + (f" NEAR-TIE FALLBACK: {dropped} token(s) dropped" if dropped or not same_mask else ""))
    assert len(keep) >= max(1, (3 * len(toks)) // 4), "too few tokens with identical routing"
    rows = [toks[i] for i in keep]
    assert np.allclose(g["w"][rows], ref["w"][rows], rtol=4 * P_RTOL, atol=0), "weights"
    s = g["stats"]
    assert s["status"] == 0
    if same_mask and same_row.all():
        for key in ("n_selected", "n_used", "max_group_load"):
            assert s[key] == ref[key], key
        # the plain top-k union depends on every token's k-th/(k+1)-th gap over E
        assert abs(s["union_topk"] - ref["union_topk"]) <= 1
    yg = g["y"][rows]
    yr = ref["y"][keep]
    if np.abs(yr).max() == 0:
        assert np.all(yg == 0)
        return ref, 0.0, 0.0, len(keep)
    max_rel = np.abs(yg - yr).max() / np.abs(yr).max()
    fro = np.linalg.norm(yg - yr) / np.linalg.norm(yr)
    print(f"    y: max_rel={max_rel:.3e} fro={fro:.3e}")
    assert max_rel <= MAX_REL and fro <= FRO_REL, (max_rel, fro)
    return ref, max_rel, fro, len(keep)


SMALL = [
    W.TINY, W.TINY.with_(k0=1), W.TINY.with_(mode=W.MODE_TOPK),
    W.OLMOE.with_(B=8, budget=16), W.OLMOE.with_(B=32, budget=24, k0=1),
    W.OLMOE.with_(B=64, budget=48), W.OLMOE.with_(B=16, mode=W.MODE_TOPK),
    W.QWEN3, W.QWEN3.with_(B=16, m_r=5), W.QWEN3.with_(k0=0, budget=16),
    W.QWEN3.with_(mode=W.MODE_TOPK),
    W.TINY.with_(mode=W.MODE_THRESH, tau=0.5, k0=1), W.OLMOE.with_(mode=W.MODE_THRESH, tau=0.7),
    W.OLMOE.with_(B=32, budget=24, sparse_scores=1), W.QWEN3.with_(sparse_scores=1),
]


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("case", range(len(SMALL)))
def test_forward_parity_small(X, case, seed):
    w = SMALL[case]
    x, W_g = W.router_inputs(w, seed)
    weights = device_weights(w, seed)
    g = gpu_forward(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights)


FULL_SIZE = [
    W.DSR1.with_(B=8), W.DSR1, W.DSR1.with_(B=128, budget=64), W.DSR1.with_(k0=0, budget=32),
    W.DSR1_GROUP, W.DSR1_GROUP.with_(k0=0, m_g=8), W.DSR1.with_(mode=W.MODE_THRESH, tau=0.5),
    W.DSR1.with_(budget=40, sparse_scores=1),
]


def full_size_tokens(w):
    """Every token up to B = 128; beyond, the first 128 (a full FFN tile's rows)."""
    return None if w.B <= 128 else list(range(128))


@pytest.mark.parametrize("w", FULL_SIZE,
                         ids=lambda w: f"{w.name}-B{w.B}-m{w.budget}-k0{w.k0}-mg{w.m_g}-mode{w.mode}"
                                       f"-s{w.sparse_scores}")
def test_forward_parity_full_size(X, w):
    """DeepSeek-R1-shaped layers at full size (d = 7168, F = 2048: 112 K-steps of
    64 in gate/up, 32 in down, split across CTAs by the stream-K schedule),
    compared with the oracle token by token."""
    x, W_g = W.router_inputs(w, 0)
    weights = device_weights(w, 0)
    g = gpu_forward(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights, tokens=full_size_tokens(w))


def gpu_forward_packed(X, w: W.Workload, x, W_g, weights):
    """xshare_moe_forward_packed (the path bench.py times) with the same outputs
    as gpu_forward."""
    dev = torch.device("cuda")
    pk = X.Packed(*weights)
    prm = X.route_params(**w.params())
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, 0),
                     dtype=torch.uint8, device=dev)
    out = dict(
        y=torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev),
        p=torch.empty(w.B, w.N, dtype=torch.float32, device=dev),
        mask=torch.empty(w.N, dtype=torch.uint8, device=dev),
        ids=torch.empty(w.B, w.k, dtype=torch.int32, device=dev),
        w=torch.empty(w.B, w.k, dtype=torch.float32, device=dev),
        stats=torch.zeros(8, dtype=torch.int32, device=dev),
    )
    X.xshare_moe_forward_packed(x.to(dev), W_g.to(dev), pk, w.k, w.budget, w.mode, prm,
                                out["y"], ws, scores_out=out["p"], sel_mask=out["mask"],
                                topk_ids=out["ids"], topk_w=out["w"], stats=out["stats"])
    torch.cuda.synchronize()
    del pk
    r = {name: t.cpu() for name, t in out.items()}
    r["stats"] = X.stats_dict(out["stats"])
    r["y"] = r["y"].float().numpy().astype(np.float64)
    for name in ("p", "mask", "ids", "w"):
        r[name] = r[name].numpy()
    return r


@pytest.mark.parametrize("w", [W.DSR1, W.DSR1.with_(B=8)], ids=lambda w: f"{w.name}-B{w.B}")
def test_forward_packed_parity_full_size(X, w):
    """The benchmarked path itself, xshare_moe_forward_packed on packed expert
    weights at the DeepSeek-R1 shape, against the oracle on every token."""
    x, W_g = W.router_inputs(w, 1)
    weights = device_weights(w, 1)
    g = gpu_forward_packed(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights)


@pytest.mark.parametrize("budget,k0", [(0, 0), (3, 0), (0, 1)])
def test_forward_small_selected_set(X, budget, k0):
    """|S| = 0 (no routed expert: y = 0), |S| < k, and warm-up only."""
    w = W.TINY.with_(budget=budget, k0=k0)
    x, W_g = W.router_inputs(w, 5)
    weights = device_weights(w, 0)
    g = gpu_forward(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights)
    if budget == 0 and k0 == 0:
        assert np.all(g["y"] == 0) and g["stats"]["n_pairs"] == 0


def test_forward_single_token(X):
    w = W.OLMOE.with_(B=1, budget=8, k0=1)
    x, W_g = W.router_inputs(w, 3)
    weights = device_weights(w, 3)
    g = gpu_forward(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights)


def test_forward_expert_with_many_tokens(X):
    """Tiles of more than 128 tokens of one expert (popular experts at B = 512)."""
    w = W.QWEN3.with_(B=512, k0=0, m_r=1, budget=0, tokens_per_request=512)
    x, W_g = W.router_inputs(w, 1)
    weights = device_weights(w, 1)
    g = gpu_forward(X, w, x, W_g, weights)
    assert max(np.bincount(g["ids"][g["ids"] >= 0])) > 128
    compare(w, g, x, W_g, weights, tokens=[0, 5, 100, 511])


@pytest.mark.parametrize("w", [
    # 2 used experts x 1 row block x 112 K steps over 28 CTAs of 8 steps: every
    # gate/up unit is cut into 14 pieces (a CTA's range lies inside one unit).
    W.TINY.with_(N=8, k=2, d=7168, F=128, B=5, budget=2, k0=0),
    # 3 used experts: gate/up units of 112 steps cut into about 4 pieces,
    # down units of 32 steps into 2.
    W.TINY.with_(N=8, k=2, d=7168, F=2048, B=7, budget=3, k0=0),
], ids=["units-cut-14-ways", "units-cut-2-to-4-ways"])
def test_forward_units_cut_across_ctas(X, w):
    """FFN units whose K steps are spread over many CTAs: each CTA does the
    pieces it shares with its neighbours first, the last piece to arrive adds
    them all (in CTA order).  Every token against the oracle; the packed path
    gives the same bits, and so does a second call."""
    x, W_g = W.router_inputs(w, 4)
    weights = device_weights(w, 4)
    g = gpu_forward(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights)
    g2 = gpu_forward_packed(X, w, x, W_g, weights)
    assert np.array_equal(g["y"], g2["y"])
    g3 = gpu_forward(X, w, x, W_g, weights)
    assert np.array_equal(g["y"], g3["y"])


def test_forward_deterministic(X):
    w = W.OLMOE.with_(B=32, budget=24, k0=1)
    x, W_g = W.router_inputs(w, 0)
    weights = device_weights(w, 0)
    a = gpu_forward(X, w, x, W_g, weights)
    b = gpu_forward(X, w, x, W_g, weights)
    assert np.array_equal(a["y"], b["y"]) and np.array_equal(a["p"], b["p"])


# ---- shared experts (Sec. 2.1: y = sum_i g_i E_i(x) + sum_j E^s_j(x)) ----
SHARED = [
    (W.TINY, 1), (W.TINY, 2), (W.TINY.with_(mode=W.MODE_TOPK), 1),
    (W.OLMOE.with_(B=32, budget=24, k0=1), 1), (W.QWEN3, 1), (W.QWEN3.with_(B=200), 2),
    (W.TINY.with_(B=1, budget=4, k0=1), 3),
]


@pytest.mark.parametrize("case", range(len(SHARED)))
def test_forward_shared_experts_small(X, case):
    w, ns = SHARED[case]
    x, W_g = W.router_inputs(w, 4)
    weights = device_weights(w, 4)
    shared = W.shared_expert_weights(w, ns, 4)
    g = gpu_forward(X, w, x, W_g, weights, shared=shared)
    compare(w, g, x, W_g, weights, shared=shared)


def test_forward_shared_experts_empty_selection(X):
    """|S| = 0: no routed expert, y is the shared experts' output alone."""
    w = W.TINY.with_(budget=0, k0=0)
    x, W_g = W.router_inputs(w, 6)
    weights = device_weights(w, 0)
    shared = W.shared_expert_weights(w, 1, 6)
    g = gpu_forward(X, w, x, W_g, weights, shared=shared)
    assert g["stats"]["n_pairs"] == 0 and np.abs(g["y"]).max() > 0
    compare(w, g, x, W_g, weights, shared=shared)


def test_forward_shared_experts_full_size_sampled(X):
    """DeepSeek-R1 layer with its one shared expert, sampled tokens."""
    w = W.DSR1
    x, W_g = W.router_inputs(w, 0)
    weights = device_weights(w, 0)
    shared = W.shared_expert_weights(w, 1, 0)
    g = gpu_forward(X, w, x, W_g, weights, shared=shared)
    compare(w, g, x, W_g, weights, tokens=[0, 13, 31], shared=shared)
    # The routed part is unchanged by adding the shared expert.
    g0 = gpu_forward(X, w, x, W_g, weights)
    assert np.array_equal(g0["ids"], g["ids"]) and np.array_equal(g0["p"], g["p"])
    assert not np.array_equal(g0["y"], g["y"])


# ---- router logits on every path (CUDA cores below 64 tokens: whole-d blocks
# below d = 4096, d-sliced blocks from it; tensor cores from 64 tokens) ----
# Below 64 tokens: one or two token blocks, ragged expert blocks (N = 100),
# every cluster split of d (d = 128: 1; 512: 4; 2048 and 7168: 8 or 4) and the
# unsplit grid of N = 1024.  The d-sliced router: 1, 2 and 4 token groups per
# lane (B = 1, 13, 37, 63), ragged expert blocks (N = 100, 250), ragged
# slices (d = 4224 = 66 columns of 64), 1 to 128 expert blocks and 2, 4 and 8
# slices (d = 16384).
@pytest.mark.parametrize("w", [
    W.TINY.with_(d=4096, F=128, B=1, budget=8), W.TINY.with_(N=100, d=4224, F=128, B=13),
    W.TINY.with_(N=250, d=4096, F=128, B=37, budget=24),
    W.TINY.with_(N=8, k=4, d=8192, F=128, B=63, budget=4),
    W.TINY.with_(N=1024, k=16, d=4096, F=128, B=20, budget=64),
    W.TINY.with_(N=32, d=16384, F=128, B=9, budget=8), W.DSR1.with_(B=8),
    W.TINY.with_(B=1, budget=8), W.TINY.with_(B=33), W.TINY.with_(N=100, B=40),
    W.TINY.with_(d=128, F=128, B=20, budget=8), W.TINY.with_(N=1024, k=16, budget=64, B=16),
    W.TINY.with_(B=63), W.TINY.with_(B=64), W.TINY.with_(B=65, budget=16),
    W.OLMOE.with_(B=8, budget=16), W.OLMOE.with_(B=200), W.QWEN3.with_(B=48),
    W.QWEN3.with_(B=1000, tokens_per_request=8),
    W.DSR1, W.DSR1.with_(B=256, budget=40),
], ids=lambda w: f"{w.name}-N{w.N}-d{w.d}-B{w.B}")
def test_router_scores_both_paths(X, w):
    """The dense scores from the router and softmax are within P_RTOL of the
    oracle's (fp64 logits, fp32 softmax), elementwise, and repeat bit for bit."""
    x, W_g = W.router_inputs(w, 2)
    weights = device_weights(w, 2)
    a = gpu_forward(X, w, x, W_g, weights)
    b = gpu_forward(X, w, x, W_g, weights)
    assert np.array_equal(a["p"], b["p"]) and np.array_equal(a["y"], b["y"])
    assert a["stats"]["status"] == 0
    ref = O.softmax_scores(O.router_logits(W.bf16_bits(x), W_g.numpy()))
    rel = np.abs(a["p"].astype(np.float64) - ref) / ref.astype(np.float64)
    print(f"[{w.name} B={w.B}] router+softmax max rel {rel.max():.2e}")
    assert rel.max() <= P_RTOL


# ---- limits: the largest batch and expert count, the smallest d and F ----
@pytest.mark.parametrize("w,tokens", [
    (W.TINY.with_(B=8192, budget=24, k0=1), [0, 4095, 8191]),           # B at the limit
    (W.TINY.with_(N=1024, k=16, budget=64, k0=2, B=96), None),           # N and k at the limit
    (W.TINY.with_(d=128, F=128, B=80, budget=8), None),                  # smallest d and F
    (W.TINY.with_(N=1000, k=8, budget=40, B=130, n_groups=8), None),    # N not a multiple of 32
])
def test_forward_limits(X, w, tokens):
    x, W_g = W.router_inputs(w, 7)
    weights = device_weights(w, 7)
    g = gpu_forward(X, w, x, W_g, weights)
    compare(w, g, x, W_g, weights, tokens=tokens)


def test_zz_near_tie_fallback_rate():
    """The near-tie rule of compare() is a rare exception, not a way around
    the comparison: it may fire on at most NEAR_TIE_MAX_FRACTION of the cases
    this file compared (run after them: pytest keeps the file order)."""
    if len(NEAR_TIE_LOG) < 20:
        pytest.skip("needs the other forward parity tests of this file in the same run")
    fired = [(c, n) for c, n, same_mask in NEAR_TIE_LOG if n or not same_mask]
    print(f"near-tie fallback fired on {len(fired)} of {len(NEAR_TIE_LOG)} compared cases: {fired}")
    assert len(fired) <= NEAR_TIE_MAX_FRACTION * len(NEAR_TIE_LOG), fired
