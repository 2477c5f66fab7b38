"""Packed expert weights (xshare_pack_experts, xshare_moe_forward_packed).

The packed layout is checked byte for byte against a torch restatement of
it, and the forward on packed weights must equal the forward on the
unpacked matrices bit for bit (same arithmetic in the same order; only the
way the weights reach shared memory differs).
"""
import numpy as np
import pytest
import torch

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


def packed_reference(W0, W1=None):
    """[n, M, K] bf16 -> 128 x 64 tiles, rows at 128 B, 16-byte chunk c of row r
    at chunk position c ^ (r % 8); blocks (e, mt, kk), with W1's tile after
    W0's when given."""
    n, M, K = W0.shape
    mats = [m.view(torch.int16) for m in ([W0] if W1 is None else [W0, W1])]  # bits, not values
    t = torch.stack([m.view(n, M // 128, 128, K // 64, 8, 8) for m in mats], dim=0)
    # t[w, e, mt, r, kk, c, b] -> blocks [e, mt, kk, w, r, c', b]
    t = t.permute(1, 2, 4, 0, 3, 5, 6).contiguous()
    r = torch.arange(128, device=W0.device).view(128, 1)
    c = torch.arange(8, device=W0.device).view(1, 8)
    src = (c ^ (r % 8))                       # position c' holds chunk c' ^ (r % 8)
    idx = src.view(1, 1, 1, 1, 128, 8, 1).expand_as(t)
    out = torch.gather(t, 5, idx)
    return out.view(torch.uint8).reshape(-1)


def test_pack_layout(X):
    w = W.TINY.with_(N=3, d=256, F=384)
    Wg, Wu, Wd = W.expert_weights(w, 1, device="cuda")
    pk = X.Packed(Wg, Wu, Wd)
    torch.cuda.synchronize()
    assert torch.equal(pk.gate_up, packed_reference(Wg, Wu))
    assert torch.equal(pk.down, packed_reference(Wd))


_cache = {}


def weights(w, seed):
    key = (w.N, w.d, w.F, seed)
    if key not in _cache:
        _cache.clear()
        torch.cuda.empty_cache()
        Wg, Wu, Wd = W.expert_weights(w, seed, device="cuda")
        _cache[key] = (Wg, Wu, Wd, X_packed(Wg, Wu, Wd))
    return _cache[key]


def X_packed(Wg, Wu, Wd):
    from paper_2602_07265_gb300 import xshare
    return xshare.Packed(Wg, Wu, Wd)


def run_both(X, w, seed, n_shared=0):
    dev = torch.device("cuda")
    Wg, Wu, Wd, pk = weights(w, seed)
    shared = W.shared_expert_weights(w, n_shared, seed, device="cuda") if n_shared else None
    pshared = X.Packed(*shared) if shared is not None else None
    x, W_g = W.router_inputs(w, seed)
    x, W_g = x.to(dev), W_g.to(dev)
    prm = X.route_params(**w.params())
    outs = []
    for packed in (False, True):
        ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm, n_shared),
                         dtype=torch.uint8, device=dev)
        o = dict(y=torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev),
                 p=torch.empty(w.B, w.N, dtype=torch.float32, device=dev),
                 mask=torch.empty(w.N, dtype=torch.uint8, device=dev),
                 ids=torch.empty(w.B, w.k, dtype=torch.int32, device=dev),
                 w=torch.empty(w.B, w.k, dtype=torch.float32, device=dev),
                 stats=torch.zeros(8, dtype=torch.int32, device=dev))
        kw = dict(scores_out=o["p"], sel_mask=o["mask"], topk_ids=o["ids"], topk_w=o["w"],
                  stats=o["stats"])
        if packed:
            X.xshare_moe_forward_packed(x, W_g, pk, w.k, w.budget, w.mode, prm, o["y"], ws,
                                        shared=pshared, **kw)
        else:
            X.xshare_moe_forward(x, W_g, Wg, Wu, Wd, w.k, w.budget, w.mode, prm, o["y"], ws,
                                 shared=shared, **kw)
        torch.cuda.synchronize()
        outs.append({k: v.cpu() for k, v in o.items()})
    return outs


@pytest.mark.parametrize("w,n_shared", [
    (W.TINY, 0), (W.TINY.with_(k0=1), 2), (W.OLMOE.with_(B=32, budget=24), 0),
    (W.QWEN3, 1), (W.DSR1_GROUP.with_(F=256), 0), (W.DSR1, 0), (W.DSR1, 1),
], ids=lambda v: str(v) if isinstance(v, int) else f"{v.name}-B{v.B}-F{v.F}")
def test_packed_forward_is_bit_identical(X, w, n_shared):
    a, b = run_both(X, w, 3, n_shared)
    assert a["stats"][5] == 0 and b["stats"][5] == 0
    for key in ("p", "mask", "ids", "w", "stats"):
        assert torch.equal(a[key], b[key]), key
    assert torch.equal(a["y"].view(torch.int16), b["y"].view(torch.int16)), "y"


def test_packed_stack_matches_unpacked(X):
    w = W.OLMOE.with_(B=64, budget=16)
    dev = torch.device("cuda")
    sets = [W.expert_weights(w, s, device="cuda", down_std=W.STACK_DOWN_STD) for s in (1, 2)]
    packs = [X.Packed(*ws) for ws in sets]
    routers = [W.router_inputs(w, 100 + l)[1].to(dev) for l in range(4)]
    plain = [(routers[l],) + tuple(sets[l % 2]) for l in range(4)]
    packed = [(routers[l], packs[l % 2]) for l in range(4)]
    x = W.router_inputs(w, 9)[0].to(dev)
    prm = X.route_params(**w.params())
    res = []
    for layers in (plain, packed):
        ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm),
                         dtype=torch.uint8, device=dev)
        h = torch.empty(4, w.B, w.d, dtype=torch.bfloat16, device=dev)
        g = X.StackGraph(x, layers, w.k, 4 * w.budget, w.mode, prm, h, ws)
        g.launch()
        torch.cuda.synchronize()
        g.close()
        res.append(h.cpu())
    assert torch.equal(res[0].view(torch.int16), res[1].view(torch.int16))
