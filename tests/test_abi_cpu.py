"""The C-ABI library builds, loads and exports every declared entry point;
host-side argument checks reject bad calls before anything is launched.
No compute runs here (no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "xshare.h")


@pytest.fixture(scope="module")
def X():
    from paper_2602_07265_gb300 import _build
    _build.build()
    from paper_2602_07265_gb300 import xshare
    return xshare


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(xshare_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    assert declared_functions() == ["xshare_ep_combine", "xshare_ep_exchange_buffer",
                                    "xshare_moe_forward", "xshare_moe_forward_ep",
                                    "xshare_moe_forward_packed",
                                    "xshare_moe_forward_profiled", "xshare_pack_experts",
                                    "xshare_route", "xshare_route_static",
                                    "xshare_selftest_wait_timeout", "xshare_stack_forward",
                                    "xshare_stack_graph_create", "xshare_stack_graph_destroy",
                                    "xshare_stack_graph_launch", "xshare_stage_name",
                                    "xshare_strerror",
                                    "xshare_workspace_size"]


def test_stage_names(X):
    assert X.STAGE_NAMES == ["router", "select", "refine", "gather", "ffn_gate_up", "ffn_down",
                             "combine"]
    assert X.LIB.xshare_stage_name(7) == b""


def test_library_exports_every_declared_symbol(X):
    from paper_2602_07265_gb300 import _build
    out = subprocess.run(["nm", "-D", "--defined-only", _build.LIB], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (\w+)$", out, flags=re.M))
    for name in declared_functions():
        assert name in exported, name
        assert getattr(X.LIB, name) is not None


def test_strerror_covers_codes(X):
    for code in (0, -1, -2, -3, -4, -5, -6, -7, 1):
        s = X.xshare_strerror(code)
        assert s and "unknown" not in s
    assert "unknown" in X.xshare_strerror(12345)


def _route_rc(X, B=8, N=16, k=4, budget=4, mode=1, prm=None, scores=1 << 20, mask=1 << 20,
              ids=1 << 20, w=1 << 20, ws=1 << 20, ws_bytes=1 << 20):
    prm = prm or X.route_params()
    return X.LIB.xshare_route(scores, B, N, k, budget, mode, ctypes.byref(prm), mask, ids, w,
                              None, None, None, None, ws, ws_bytes, None)


@pytest.mark.parametrize("kw,code", [
    (dict(B=0), -1), (dict(B=8193), -1), (dict(N=0), -1), (dict(N=1025), -1),
    (dict(k=0), -1), (dict(k=17), -1), (dict(N=4, k=5), -1),
    (dict(mode=5), -2), (dict(mode=-1), -2), (dict(budget=-1), -2),
    (dict(scores=None), -3), (dict(mask=None), -3), (dict(ids=None), -3), (dict(w=None), -3),
    (dict(scores=(1 << 20) + 4), -5),
    (dict(ws=None), -4), (dict(ws=(1 << 20) + 16), -4),
])
def test_route_rejects_bad_arguments(X, kw, code):
    assert _route_rc(X, **kw) == code


@pytest.mark.parametrize("prm,mode,code", [
    (dict(k0=-1), 1, -2), (dict(k0=17), 1, -2), (dict(m_r=-1), 3, -2), (dict(m_g=-1), 2, -2),
    (dict(n_groups=0), 2, -2), (dict(n_groups=3), 2, -2), (dict(n_groups=32), 2, -2),
    (dict(tokens_per_request=0), 3, -2), (dict(tokens_per_request=3), 3, -2),
    (dict(tokens_per_request=16), 3, -2),
    (dict(tau=-0.1), 4, -2), (dict(tau=1.5), 4, -2), (dict(tau=float("nan")), 4, -2),
    (dict(), 5, -2), (dict(sparse_scores=2), 1, -2), (dict(sparse_scores=-1), 1, -2),
])
def test_route_rejects_bad_params(X, prm, mode, code):
    assert _route_rc(X, mode=mode, prm=X.route_params(**prm)) == code


def test_forward_rejects_bad_shapes(X):
    prm = X.route_params()
    P = 1 << 20
    def rc(d, F, x=P, y=P, shared=None):
        sh = ctypes.byref(shared) if shared is not None else None
        return X.LIB.xshare_moe_forward(x, P, P, P, P, 4, d, F, 16, 2, 2, 1, ctypes.byref(prm),
                                        sh, y, None, None, None, None, None, P, 1 << 20, None)
    assert rc(100, 256) == -1
    assert rc(256, 64) == -1
    assert rc(0, 256) == -1
    assert rc(256, 256, x=None) == -3
    assert rc(256, 256, y=P + 8) == -5
    assert rc(256, 256, shared=X.SharedExperts(P, P, P, 9)) == -2
    assert rc(256, 256, shared=X.SharedExperts(P, P, P, -1)) == -2
    assert rc(256, 256, shared=X.SharedExperts(P, None, P, 1)) == -3
    assert rc(256, 256, shared=X.SharedExperts(P, P, P + 2, 1)) == -5


def test_workspace_size_rejects_invalid(X):
    prm = X.route_params()
    assert X.xshare_workspace_size(0, 16, 4, 0, 0, 1, prm) == 0
    assert X.xshare_workspace_size(8, 16, 4, 100, 256, 1, prm) == 0
    assert X.xshare_workspace_size(8, 16, 4, 256, 256, 1, prm, 9) == 0
    assert X.xshare_workspace_size(8, 16, 4, 0, 0, 1, prm, 1) == 0  # routing alone has none


def test_stack_rejects_bad_arguments(X):
    prm = X.route_params()
    P = 1 << 20
    lay = (X.Layer * 2)()
    for l in range(2):
        lay[l].W_g = lay[l].W_gate = lay[l].W_up = lay[l].W_down = P
    def rc(L=2, x=P, h=P << 4, d=256, F=256, K=8, layers=lay):
        return X.LIB.xshare_stack_forward(x, layers, L, 4, d, F, 16, 2, K, 1, ctypes.byref(prm),
                                          h, None, P, 1 << 20, None)
    assert rc(L=0) == -1
    assert rc(K=-1) == -2
    assert rc(x=None) == -3
    assert rc(layers=None) == -3
    assert rc(h=P) == -2            # output overlaps the input
    assert rc(d=100) == -1
    lay[1].W_up = None               # a later layer is checked before anything runs
    assert rc() == -3
    lay[1].W_up = P
    out = ctypes.c_void_p(7)
    assert X.LIB.xshare_stack_graph_create(P, lay, 0, 4, 256, 256, 16, 2, 8, 1,
                                           ctypes.byref(prm), P << 4, None, P, 1 << 20,
                                           ctypes.byref(out)) == -1
    assert not out.value
    assert X.LIB.xshare_stack_graph_launch(None, None) == -3
    X.LIB.xshare_stack_graph_destroy(None)


def test_route_static_rejects_sparse_scores(X):
    P = 1 << 20
    prm = X.route_params(sparse_scores=1)
    assert X.LIB.xshare_route_static(P, 8, 16, 4, 4, 1, ctypes.byref(prm), P, P, P, None, None,
                                     None, None, None) == -2


def test_packed_entry_points_reject_bad_arguments(X):
    P = 1 << 20
    assert X.LIB.xshare_pack_experts(P, P, P, 0, 256, 256, P, P, None) == -1
    assert X.LIB.xshare_pack_experts(P, P, P, 4, 100, 256, P, P, None) == -1
    assert X.LIB.xshare_pack_experts(P, None, P, 4, 256, 256, P, P, None) == -3
    assert X.LIB.xshare_pack_experts(P, P, P, 4, 256, 256, P + 8, P, None) == -5
    prm = X.route_params()
    ex = X.PackedExperts(P, P, 16)
    def rc(ex=ex, sh=None, ev=None):
        return X.LIB.xshare_moe_forward_packed(P, P, ctypes.byref(ex) if ex is not None else None,
                                               4, 256, 256, 16, 2, 2, 1, ctypes.byref(prm),
                                               ctypes.byref(sh) if sh is not None else None,
                                               P, None, None, None, None, None, P, 1 << 20, None, ev)
    assert rc(ex=None) == -3
    assert rc(ex=X.PackedExperts(P, P, 15)) == -1          # count must equal N
    assert rc(ex=X.PackedExperts(P, None, 16)) == -3
    assert rc(ex=X.PackedExperts(P + 4, P, 16)) == -5
    assert rc(sh=X.PackedExperts(P, P, 9)) == -2
    assert rc(sh=X.PackedExperts(None, P, 1)) == -3


def test_ep_entry_points_reject_bad_arguments(X):
    """Expert-parallel calls: n_ranks and rank, N % n_ranks, the local expert
    count, NULL outputs; all checked before anything touches a GPU."""
    prm = X.route_params()
    ws = ctypes.c_void_p(256)  # never dereferenced: every call below fails its checks first
    pk = X.PackedExperts(16, 16, 32)

    def fwd(n_ranks, rank, N=64, local=pk):
        return X.LIB.xshare_moe_forward_ep(16, 16, ctypes.byref(local) if local else None, 32, 512,
                                           256, N, 8, 24, 1, ctypes.byref(prm), None, n_ranks,
                                           rank, None, None, None, None, ws, 1 << 30, None)
    assert fwd(0, 0) == -2          # n_ranks < 1
    assert fwd(2, 2) == -2          # rank >= n_ranks
    assert fwd(2, -1) == -2         # rank < 0
    assert fwd(3, 0) == -2          # N % n_ranks != 0
    assert fwd(2, 0, local=None) == -3
    assert fwd(2, 0, local=X.PackedExperts(16, 16, 16)) == -1   # N / n_ranks = 32 experts expected
    buf, count = ctypes.c_void_p(), ctypes.c_size_t()
    assert X.LIB.xshare_ep_exchange_buffer(ws, 32, 64, 8, 512, 256, 1, ctypes.byref(prm), 0,
                                           None, ctypes.byref(count)) == -3
    assert X.LIB.xshare_ep_exchange_buffer(ws, 32, 64, 8, 500, 256, 1, ctypes.byref(prm), 0,
                                           ctypes.byref(buf), ctypes.byref(count)) == -1
    assert X.LIB.xshare_ep_combine(ws, 32, 64, 8, 512, 256, 1, ctypes.byref(prm), 0, None,
                                   None) == -3
    assert X.LIB.xshare_ep_combine(ws, 32, 64, 8, 512, 256, 1, ctypes.byref(prm), 0, 18,
                                   None) == -5
