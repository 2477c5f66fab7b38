"""Failure reporting on the GPU without faulting it.

Every pipeline wait inside the library's kernels is bounded in time; when a
wait runs out, the kernel records XS_DEV_TIMEOUT in xs_stats.status and
returns.  The self-test kernel makes such a wait run out (it waits on a
barrier nothing arrives at) and this test checks the status, the time waited
and that the context still runs a full forward afterwards.
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


def test_bounded_wait_reports_timeout_and_context_survives(X):
    dev = torch.device("cuda")
    st = torch.zeros(X.STATS_WORDS, dtype=torch.int32, device=dev)
    X.xshare_selftest_wait_timeout(st, 50_000_000)   # 50 ms
    torch.cuda.synchronize()
    s = st.cpu().tolist()
    assert s[5] == X.XS_DEV_TIMEOUT
    assert 50 <= s[6] < 2000   # milliseconds actually waited
    # the context is still usable: a normal forward runs and reports no error
    w = W.TINY
    x, W_g = W.router_inputs(w, 0)
    Wg, Wu, Wd = W.expert_weights(w, 0, device="cuda")
    prm = X.route_params(**w.params())
    ws = torch.empty(X.xshare_workspace_size(w.B, w.N, w.k, w.d, w.F, w.mode, prm),
                     dtype=torch.uint8, device=dev)
    y = torch.empty(w.B, w.d, dtype=torch.bfloat16, device=dev)
    st2 = torch.full((X.STATS_WORDS,), -1, dtype=torch.int32, device=dev)
    X.xshare_moe_forward(x.to(dev), W_g.to(dev), Wg, Wu, Wd, w.k, w.budget, w.mode, prm, y, ws,
                         stats=st2)
    torch.cuda.synchronize()
    assert X.stats_dict(st2)["status"] == 0
    assert torch.isfinite(y.float()).all()


def test_selftest_rejects_bad_budget(X):
    st = torch.zeros(X.STATS_WORDS, dtype=torch.int32, device="cuda")
    with pytest.raises(X.XShareError):
        X.xshare_selftest_wait_timeout(st, 0)
    with pytest.raises(X.XShareError):
        X.xshare_selftest_wait_timeout(st, 3_000_000_000)
