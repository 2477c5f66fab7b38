"""The forward calls inside CUDA graphs and on concurrent streams.

* A torch CUDA graph capturing copy-in + xshare_moe_forward_packed replays to
  the same bits as the direct call, for two different inputs.
* Two forwards with separate workspaces on two streams, launched without
  ordering between them, give the results each gives alone.
"""
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


def setup(X, w, seed):
    dev = torch.device("cuda")
    Wg, Wu, Wd = W.expert_weights(w, seed, device="cuda")
    pk = X.Packed(Wg, Wu, Wd)
    _, W_g = W.router_inputs(w, seed)
    prm = X.route_params(**w.params())
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm),
                     dtype=torch.uint8, device=dev)
    return pk, W_g.to(dev), prm, ws


@pytest.mark.parametrize("w", [W.OLMOE.with_(B=32, budget=24, k0=1), W.QWEN3],
                         ids=lambda w: f"{w.name}-B{w.B}")
def test_forward_captured_in_a_graph(X, w):
    dev = torch.device("cuda")
    pk, W_g, prm, ws = setup(X, w, 1)
    xs = [W.router_inputs(w, s)[0].to(dev) for s in (3, 4)]
    x_in = torch.empty_like(xs[0])
    y = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    st = torch.zeros(X.STATS_WORDS, dtype=torch.int32, device=dev)
    direct = []
    for x in xs:
        X.xshare_moe_forward_packed(x, W_g, pk, w.k, w.budget, w.mode, prm, y, ws, stats=st)
        torch.cuda.synchronize()
        direct.append((y.clone(), st.clone()))
    src = torch.empty_like(xs[0])
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        x_in.copy_(src)
        X.xshare_moe_forward_packed(x_in, W_g, pk, w.k, w.budget, w.mode, prm, y, ws, stats=st)
    for x, (yd, sd) in zip(xs, direct):
        src.copy_(x)
        y.fill_(0)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(y.view(torch.int16), yd.view(torch.int16))
        assert torch.equal(st, sd) and int(st[5]) == 0


def test_two_streams_with_separate_workspaces(X):
    w = W.DSR1.with_(N=64, B=64, budget=16)
    dev = torch.device("cuda")
    pk, W_g, prm, _ = setup(X, w, 2)
    xs = [W.router_inputs(w, s)[0].to(dev) for s in (5, 6)]
    wss = [torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm),
                       dtype=torch.uint8, device=dev) for _ in range(2)]
    ys = [torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev) for _ in range(2)]
    alone = []
    for x, ws, y in zip(xs, wss, ys):
        X.xshare_moe_forward_packed(x, W_g, pk, w.k, w.budget, w.mode, prm, y, ws)
        torch.cuda.synchronize()
        alone.append(y.clone())
    streams = [torch.cuda.Stream() for _ in range(2)]
    for rep in range(3):
        for y in ys:
            y.fill_(0)
        torch.cuda.synchronize()
        for x, ws, y, s in zip(xs, wss, ys, streams):
            X.xshare_moe_forward_packed(x, W_g, pk, w.k, w.budget, w.mode, prm, y, ws, stream=s)
        torch.cuda.synchronize()
        for y, ya in zip(ys, alone):
            assert torch.equal(y.view(torch.int16), ya.view(torch.int16))
