"""Randomised parity: seeded random layer shapes and selection settings,
through the C ABI, against the oracle.

Each case draws N (1 .. 1024), k, B (1 .. 300), d and F (multiples of 128, at
most 512 so that the oracle stays quick), a mode with random parameters
(k0, budget, m_r and request length, groups and m_g, tau, sparse scores),
and shared experts.  Two checks per case:

* selection from identical scores: xshare_route on the oracle's own fp32
  scores equals oracle.route bit for bit (mask, ids, weight bits, counts,
  offsets, permutation, statistics);
* the whole forward (xshare_moe_forward_packed) against the oracle with the
  forward tolerances of test_gpu_forward.compare.
"""
import numpy as np
import pytest
import torch

from oracle import xshare_oracle as O
from paper_2602_07265_gb300 import workloads as W
from test_gpu_forward import compare

pytestmark = pytest.mark.gpu

N_CASES = 40


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare
    return xshare


def random_case(i: int):
    rng = np.random.default_rng(1000 + i)
    N = int(rng.choice([8, 17, 32, 64, 100, 128, 200, 256, 512, 1000, 1024]))
    k = int(rng.integers(1, min(16, N) + 1))
    mode = int(rng.choice([W.MODE_TOPK, W.MODE_BATCH, W.MODE_GROUP, W.MODE_HIER, W.MODE_THRESH]))
    T = int(rng.choice([1, 2, 4, 8, 16, 32, 64])) if mode == W.MODE_HIER else 1
    B = int(rng.integers(1, 300))
    B = max(T, B - B % T)
    divisors = [g for g in (1, 2, 4, 8, 16) if N % g == 0]
    kw = dict(
        name="random", N=N, k=k, d=int(rng.choice([128, 256, 512])),
        F=int(rng.choice([128, 256, 384])), B=B, mode=mode,
        budget=int(rng.integers(0, N + 1)), k0=int(rng.integers(0, min(16, N, 3) + 1)),
        m_r=int(rng.integers(0, 8)), tokens_per_request=T,
        n_groups=int(rng.choice(divisors)), m_g=int(rng.integers(0, N // 4 + 2)),
        tau=float(rng.choice([0.0, 0.2, 0.5, 0.8, 1.0])),
        sparse_scores=int(mode != W.MODE_TOPK and rng.random() < 0.25),
        x_kind=str(rng.choice(["iid", "request", "domains"])))
    n_shared = int(rng.choice([0, 0, 0, 1, 2]))
    return W.Workload(**kw), n_shared


@pytest.mark.parametrize("i", range(N_CASES))
def test_random_layer(X, i):
    w, ns = random_case(i)
    dev = torch.device("cuda")
    print(f"case {i}: N={w.N} k={w.k} B={w.B} d={w.d} F={w.F} mode={w.mode} m={w.budget} "
          f"k0={w.k0} m_r={w.m_r} T={w.tokens_per_request} G={w.n_groups} m_g={w.m_g} "
          f"tau={w.tau} sparse={w.sparse_scores} shared={ns}")
    x, W_g = W.router_inputs(w, i)
    prm = X.route_params(**w.params())

    # Selection from the oracle's own scores: bit-exact.
    p = O.softmax_scores(O.router_logits(W.bf16_bits(x), W_g.numpy()))
    ref = O.route(p, w.k, w.budget, w.mode, **w.params())
    out = dict(mask=torch.empty(w.N, dtype=torch.uint8, device=dev),
               ids=torch.empty(w.B, w.k, dtype=torch.int32, device=dev),
               w=torch.empty(w.B, w.k, dtype=torch.float32, device=dev),
               stats=torch.zeros(8, dtype=torch.int32, device=dev),
               counts=torch.empty(w.N, dtype=torch.int32, device=dev),
               offsets=torch.empty(w.N + 1, dtype=torch.int32, device=dev),
               perm=torch.empty(w.B * w.k, dtype=torch.int32, device=dev))
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, 0, 0, w.mode, prm), dtype=torch.uint8,
                     device=dev)
    X.xshare_route(torch.from_numpy(p).to(dev), w.k, w.budget, w.mode, prm, out["mask"], out["ids"],
                   out["w"], ws, stats=out["stats"], expert_counts=out["counts"],
                   expert_offsets=out["offsets"], perm=out["perm"])
    torch.cuda.synchronize()
    assert np.array_equal(out["mask"].cpu().numpy(), ref["mask"])
    assert np.array_equal(out["ids"].cpu().numpy(), ref["ids"])
    assert np.array_equal(out["w"].cpu().numpy().view(np.uint32), ref["w"].view(np.uint32))
    assert np.array_equal(out["counts"].cpu().numpy(), ref["counts"])
    assert np.array_equal(out["offsets"].cpu().numpy(), ref["offsets"])
    n_pairs = len(ref["perm"])
    assert np.array_equal(out["perm"][:n_pairs].cpu().numpy(), ref["perm"])
    st = X.stats_dict(out["stats"])
    for key in ("n_selected", "n_used", "union_topk", "max_group_load"):
        assert st[key] == ref[key], key
    assert st["n_pairs"] == n_pairs and st["status"] == 0

    # The whole layer on packed weights against the oracle.
    weights = W.expert_weights(w, i, device="cuda")
    pk = X.Packed(*weights)
    sh_w = W.shared_expert_weights(w, ns, i) if ns else None
    shared = X.Packed(*sh_w) if ns else None
    wsf = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, ns),
                      dtype=torch.uint8, device=dev)
    g = dict(y=torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev),
             p=torch.empty(w.B, w.N, dtype=torch.float32, device=dev),
             mask=torch.empty(w.N, dtype=torch.uint8, device=dev),
             ids=torch.empty(w.B, w.k, dtype=torch.int32, device=dev),
             w=torch.empty(w.B, w.k, dtype=torch.float32, device=dev),
             stats=torch.zeros(8, dtype=torch.int32, device=dev))
    X.xshare_moe_forward_packed(x.to(dev), W_g.to(dev), pk, w.k, w.budget, w.mode, prm, g["y"], wsf,
                                shared=shared, scores_out=g["p"], sel_mask=g["mask"],
                                topk_ids=g["ids"], topk_w=g["w"], stats=g["stats"])
    torch.cuda.synchronize()
    r = {name: t.cpu() for name, t in g.items()}
    r["stats"] = X.stats_dict(g["stats"])
    r["y"] = r["y"].float().numpy().astype(np.float64)
    for name in ("p", "mask", "ids", "w"):
        r[name] = r[name].numpy()
    compare(w, r, x, W_g, weights, shared=sh_w)
