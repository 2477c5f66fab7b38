"""xshare_route_static, the workspace-free variant of xshare_route.

It exists for callers that are not allowed to allocate device memory: a
plugin whose host program owns all GPU memory through its own allocator, or
a serving loop that must not call cudaMalloc after start-up because that can
stall the whole device.  Its scratch is a fixed array in the library's own
device memory instead of a caller workspace.

This file is named so that pytest collects it last.  The first test runs
the entry point on several problems in a row (each runs over whatever the
one before left in the shared array), among them problems at the size limit
(B = 1024 tokens, N = 1024 experts, k = 16, which reach the far ends of
every scratch region), and requires every output to equal xshare_route's
bit for bit, the bar the other routing tests use.  The second compares it
with the CPU oracle directly.  They must pass alone in a fresh process and
after the other tests.
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


def _outputs(B, N, k, dev):
    return dict(mask=torch.full((N,), 5, dtype=torch.uint8, device=dev),
                ids=torch.full((B, k), 77, dtype=torch.int32, device=dev),
                w=torch.full((B, k), 3.0, dtype=torch.float32, device=dev),
                stats=torch.full((8,), -9, dtype=torch.int32, device=dev),
                counts=torch.full((N,), -1, dtype=torch.int32, device=dev),
                offsets=torch.full((N + 1,), -1, dtype=torch.int32, device=dev),
                perm=torch.full((B * k,), -1, dtype=torch.int32, device=dev))


def test_route_static_matches_route_twice(X):
    dev = torch.device("cuda")
    cases = [
        (W.random_scores(256, 256, seed=41), 8, 24, W.MODE_HIER,
         X.route_params(k0=1, m_r=4, tokens_per_request=4)),
        (W.random_scores(32, 64, seed=42, ties=True), 8, 12, W.MODE_BATCH,
         X.route_params(k0=1)),
        (W.random_scores(96, 128, seed=43), 8, 0, W.MODE_THRESH,
         X.route_params(k0=1, tau=0.6)),
        # At the limit: B = 1024, N = 1024, k = 16, GROUP (Algorithms 5-6).
        (W.random_scores(1024, 1024, seed=44), 16, 0, W.MODE_GROUP,
         X.route_params(k0=0, n_groups=8, m_g=12)),
        # B = 1024 with few experts (every token shares them), tie-heavy.
        (W.random_scores(1024, 48, seed=45, ties=True), 6, 10, W.MODE_BATCH,
         X.route_params(k0=2)),
        # B = 1024, N = 1024, k = 16 with a warm-up set and HIER requests of 8.
        (W.random_scores(1024, 1024, seed=46), 16, 32, W.MODE_HIER,
         X.route_params(k0=1, m_r=2, tokens_per_request=8)),
    ]
    for p, k, budget, mode, prm in cases:
        B, N = p.shape
        scores = torch.from_numpy(p).to(dev)
        ref = _outputs(B, N, k, dev)
        ws = torch.empty(X.xshare_workspace_size(B, N, k, 0, 0, mode, prm), dtype=torch.uint8, device=dev)
        X.xshare_route(scores, k, budget, mode, prm, ref["mask"], ref["ids"], ref["w"], ws,
                       stats=ref["stats"], expert_counts=ref["counts"],
                       expert_offsets=ref["offsets"], perm=ref["perm"])
        got = _outputs(B, N, k, dev)
        X.xshare_route_static(scores, k, budget, mode, prm, got["mask"], got["ids"], got["w"],
                              stats=got["stats"], expert_counts=got["counts"],
                              expert_offsets=got["offsets"], perm=got["perm"])
        torch.cuda.synchronize()
        n_pairs = int(ref["stats"][4].item())
        for key in ("mask", "ids", "w", "stats", "counts", "offsets"):
            a, b = ref[key].cpu().numpy(), got[key].cpu().numpy()
            assert np.array_equal(a.view(np.uint8), b.view(np.uint8)), key
        assert torch.equal(ref["perm"][:n_pairs].cpu(), got["perm"][:n_pairs].cpu())
        assert int(got["stats"][5].item()) == 0


@pytest.mark.parametrize("wl", [W.DSR1, W.DSR1_GROUP.with_(B=1024)], ids=lambda w: f"{w.name}-B{w.B}")
def test_route_static_matches_oracle(X, wl):
    """Softmax scores the oracle computed from a seeded DeepSeek-R1-shaped
    batch, routed by xshare_route_static and by the oracle: mask, ids,
    weights (fp32 bits), counts, offsets, permutation and statistics equal."""
    dev = torch.device("cuda")
    x, W_g = W.router_inputs(wl, 3)
    p = O.softmax_scores(O.router_logits(W.bf16_bits(x), W_g.numpy()))
    ref = O.route(p, wl.k, wl.budget, wl.mode, **wl.params())
    B, N, k = wl.B, wl.N, wl.k
    got = _outputs(B, N, k, dev)
    X.xshare_route_static(torch.from_numpy(p).to(dev), k, wl.budget, wl.mode,
                          X.route_params(**wl.params()), got["mask"], got["ids"], got["w"],
                          stats=got["stats"], expert_counts=got["counts"],
                          expert_offsets=got["offsets"], perm=got["perm"])
    torch.cuda.synchronize()
    assert np.array_equal(got["mask"].cpu().numpy(), ref["mask"])
    assert np.array_equal(got["ids"].cpu().numpy(), ref["ids"])
    assert np.array_equal(got["w"].cpu().numpy().view(np.uint32), ref["w"].view(np.uint32))
    assert np.array_equal(got["counts"].cpu().numpy(), ref["counts"])
    assert np.array_equal(got["offsets"].cpu().numpy(), ref["offsets"])
    n_pairs = len(ref["perm"])
    assert np.array_equal(got["perm"][:n_pairs].cpu().numpy(), ref["perm"])
    st = X.stats_dict(got["stats"])
    for key in ("n_selected", "n_used", "union_topk", "max_group_load"):
        assert st[key] == ref[key], key
    assert st["n_pairs"] == n_pairs and st["status"] == 0


def test_route_static_rejects_large_batches(X):
    dev = torch.device("cuda")
    B, N, k = X.STATIC_MAX_B + 1, 64, 4
    scores = torch.ones(B, N, dtype=torch.float32, device=dev)
    out = _outputs(B, N, k, dev)
    with pytest.raises(X.XShareError) as e:
        X.xshare_route_static(scores, k, 8, W.MODE_BATCH, X.route_params(), out["mask"],
                              out["ids"], out["w"])
    assert e.value.code == -1
