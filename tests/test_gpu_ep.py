"""Expert parallelism (Sec. 5) through the C ABI, on one GPU: G logical ranks
run one after another, each with its own workspace and only its own experts'
packed weights; the exchange is the sum of their exchange buffers (what an
all-reduce over G GPUs computes); rank 0's workspace then runs the combine.

Checks, per case:
* every rank's routing (mask, ids, weights, statistics) equals the one-GPU
  forward's: the routing is replicated, not sharded;
* every exchange row is non-zero on at most one rank, and the rows a rank
  fills are exactly those of its expert group's pairs (and the shared rows
  on rank 0);
* y after the exchange and combine equals the oracle on every token (the
  first 128 at B = 256) within the forward's tolerance, and equals the
  one-GPU packed forward within one bf16 rounding step (a rank's FFN splits
  a unit's K range by its own schedule);
* with G = 1 it is the one-GPU forward, bit for bit.
"""
import numpy as np
import pytest
import torch

from oracle import xshare_oracle as O
from paper_2602_07265_gb300 import workloads as W
from test_gpu_forward import compare, device_weights, full_size_tokens

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def X():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare
    return xshare


def _outs(w, dev):
    return dict(mask=torch.empty(w.N, dtype=torch.uint8, device=dev),
                ids=torch.empty(w.B, w.k, dtype=torch.int32, device=dev),
                w=torch.empty(w.B, w.k, dtype=torch.float32, device=dev),
                stats=torch.zeros(8, dtype=torch.int32, device=dev))


def run_ep(X, w, x, W_g, pk, G, shared=None):
    """The G ranks in sequence; returns (y, per-rank outputs, per-rank exchange buffers)."""
    dev = torch.device("cuda")
    prm = X.route_params(**w.params())
    ns = shared.n if shared is not None else 0
    xd, Wgd = x.to(dev), W_g.to(dev)
    ranks, bufs, wss = [], [], []
    for g in range(G):
        ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, ns),
                         dtype=torch.uint8, device=dev)
        o = _outs(w, dev)
        local = pk.experts(g * (w.N // G), (g + 1) * (w.N // G))
        X.xshare_moe_forward_ep(xd, Wgd, local, w.k, w.budget, w.mode, prm, G, g, ws,
                                shared=shared, sel_mask=o["mask"], topk_ids=o["ids"],
                                topk_w=o["w"], stats=o["stats"])
        bufs.append(X.ep_exchange_buffer(ws, w.B, w.N, w.k, w.d, w.F, w.mode, prm, ns))
        ranks.append(o)
        wss.append(ws)
    torch.cuda.synchronize()
    snap = [b.clone() for b in bufs]
    total = snap[0].clone()
    for b in snap[1:]:
        total += b
    bufs[0].copy_(total)
    y = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    X.xshare_ep_combine(wss[0], w.B, w.N, w.k, w.d, w.F, w.mode, prm, y, ns)
    torch.cuda.synchronize()
    return y, ranks, [b.view(-1, w.d).cpu().numpy() for b in snap]


def run_one_gpu(X, w, x, W_g, pk, shared=None):
    dev = torch.device("cuda")
    prm = X.route_params(**w.params())
    ns = shared.n if shared is not None else 0
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, ns),
                     dtype=torch.uint8, device=dev)
    o = _outs(w, dev)
    o["y"] = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    o["p"] = torch.empty(w.B, w.N, dtype=torch.float32, device=dev)
    X.xshare_moe_forward_packed(x.to(dev), W_g.to(dev), pk, w.k, w.budget, w.mode, prm, o["y"],
                                ws, shared=shared, scores_out=o["p"], sel_mask=o["mask"],
                                topk_ids=o["ids"], topk_w=o["w"], stats=o["stats"])
    torch.cuda.synchronize()
    return o


CASES = [
    (W.TINY, 2, 0), (W.TINY, 64, 1), (W.TINY.with_(k0=1), 4, 2),
    (W.OLMOE.with_(B=32, budget=24), 8, 0),
    (W.QWEN3.with_(B=64), 4, 1),
    (W.DSR1, 8, 1),
    (W.DSR1_GROUP, 8, 0),
]


@pytest.mark.parametrize("case", range(len(CASES)),
                         ids=lambda i: f"{CASES[i][0].name}-B{CASES[i][0].B}-G{CASES[i][1]}-s{CASES[i][2]}")
def test_ep_matches_one_gpu_and_oracle(X, case):
    w, G, ns = CASES[case]
    x, W_g = W.router_inputs(w, 4)
    weights = device_weights(w, 4)
    pk = X.Packed(*weights)
    sh_w = W.shared_expert_weights(w, ns, 4) if ns else None
    shared = X.Packed(*sh_w) if ns else None
    one = run_one_gpu(X, w, x, W_g, pk, shared)
    y, ranks, bufs = run_ep(X, w, x, W_g, pk, G, shared)

    # Replicated routing.
    for o in ranks:
        for key in ("mask", "ids", "stats"):
            assert torch.equal(o[key], one[key]), key
        assert torch.equal(o["w"].view(torch.int32), one["w"].view(torch.int32))
    st = X.stats_dict(one["stats"])
    assert st["status"] == 0

    # Row ownership: the pairs of rank g's experts (and the shared rows on rank 0).
    ids = one["ids"].cpu().numpy()
    r = O.permute(ids, w.N)
    n_pairs = len(r["perm"])
    nz = np.stack([np.any(b != 0, axis=1) for b in bufs])
    assert nz.sum(axis=0).max() <= 1, "an exchange row computed by two ranks"
    for g in range(G):
        lo, hi = r["offsets"][g * (w.N // G)], r["offsets"][(g + 1) * (w.N // G)]
        own = np.zeros(nz.shape[1], dtype=bool)
        own[lo:hi] = True
        if g == 0:
            own[n_pairs:n_pairs + ns * w.B] = True
        assert not np.any(nz[g] & ~own), f"rank {g} wrote rows of another group"
        assert np.all(nz[g][own]), f"rank {g} left rows of its group empty"

    # Against the oracle and the one-GPU forward.
    g_out = {"y": y.float().cpu().numpy().astype(np.float64), "p": one["p"].cpu().numpy(),
             "mask": one["mask"].cpu().numpy(), "ids": ids, "w": one["w"].cpu().numpy(),
             "stats": st}
    compare(w, g_out, x, W_g, weights, tokens=full_size_tokens(w), shared=sh_w)
    y1 = one["y"].float()
    diff = (y.float() - y1).abs()
    scale = y1.abs().max().item()
    same = (y.view(torch.int16) == one["y"].view(torch.int16)).float().mean().item()
    print(f"    ep vs one GPU: max|dy|/max|y| = {diff.max().item() / scale:.2e}, identical {same:.4f}")
    assert diff.max().item() <= 2 ** -7 * scale


def test_ep_single_rank_is_the_forward(X):
    """G = 1: one rank holds every expert; the result is the one-GPU forward's bits."""
    w = W.OLMOE.with_(B=32, budget=24, k0=1)
    x, W_g = W.router_inputs(w, 2)
    pk = X.Packed(*device_weights(w, 2))
    one = run_one_gpu(X, w, x, W_g, pk)
    y, _, _ = run_ep(X, w, x, W_g, pk, 1)
    assert torch.equal(y.view(torch.int16), one["y"].view(torch.int16))
