"""xshare_route_static, the workspace-free variant of xshare_route.

It exists for callers that are not allowed to allocate device memory: a
plugin whose host program owns all GPU memory through its own allocator, or
a serving loop that must not call cudaMalloc after start-up because that can
stall the whole device.  Its scratch is a fixed array in the library's own
device memory instead of a caller workspace.

This file is named so that pytest collects it last.  The test runs the new
entry point twice in a row, on two different problems (the second smaller,
so it runs over whatever the first left in the shared array), and requires
every output to equal xshare_route's bit for bit, the bar the other routing
tests use.  It must pass alone in a fresh process and after the other tests.
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


def test_route_static_rejects_large_batches(X):
    dev = torch.device("cuda")
    B, N, k = X.STATIC_MAX_B + 1, 64, 4
    scores = torch.ones(B, N, dtype=torch.float32, device=dev)
    out = _outputs(B, N, k, dev)
    with pytest.raises(X.XShareError) as e:
        X.xshare_route_static(scores, k, 8, W.MODE_BATCH, X.route_params(), out["mask"],
                              out["ids"], out["w"])
    assert e.value.code == -1
