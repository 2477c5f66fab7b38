"""The oracle's C-ABI-shaped entry points: same parameter lists as the header,
same results as the oracle functions they wrap."""
import inspect
import os
import re

import numpy as np
import torch

from oracle import abi as A
from oracle import xshare_oracle as O

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "xshare.h")


def header_params(name):
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    m = re.search(r"\b" + name + r"\s*\(([^;]*?)\)\s*;", text, flags=re.S)
    params = [re.split(r"[\s\*]+", p.strip())[-1] for p in m.group(1).split(",")]
    return [p for p in params if p not in ("workspace", "ws_bytes", "stream")]


def test_parameter_lists_follow_the_header():
    assert list(inspect.signature(A.oracle_route).parameters) == header_params("xshare_route")
    assert list(inspect.signature(A.oracle_moe_forward).parameters) == \
        header_params("xshare_moe_forward")


def test_route_and_forward_write_the_oracle_results():
    rng = np.random.default_rng(3)
    B, N, k, d, F = 6, 16, 2, 128, 128
    h = rng.standard_normal((B, N))
    p = (np.exp(h) / np.exp(h).sum(1, keepdims=True)).astype(np.float32)
    prm = dict(k0=1)
    out = dict(sel_mask=np.zeros(N, np.uint8), topk_ids=np.zeros((B, k), np.int32),
               topk_w=np.zeros((B, k), np.float32), stats=np.zeros(8, np.int32),
               expert_counts=np.zeros(N, np.int32), expert_offsets=np.zeros(N + 1, np.int32),
               perm=np.full(B * k, -1, np.int32))
    assert A.oracle_route(p, B, N, k, 3, O.MODE_BATCH, prm, **out) == 0
    r = O.route(p, k, 3, O.MODE_BATCH, k0=1)
    assert np.array_equal(out["sel_mask"], r["mask"]) and np.array_equal(out["topk_ids"], r["ids"])
    assert out["stats"][0] == r["n_selected"] and np.array_equal(out["perm"], r["perm"])
    assert A.oracle_route(p, B, N, 17, 3, O.MODE_BATCH, prm, **out) == A.XS_ERR_SHAPE
    assert A.oracle_route(p, B, N, k, -1, O.MODE_BATCH, prm, **out) == A.XS_ERR_PARAM

    g = torch.Generator().manual_seed(2)
    bits = lambda t: t.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    x = bits(torch.randn(B, d, generator=g))
    W_g = (torch.randn(N, d, generator=g) / d ** 0.5).numpy()
    Wg, Wu = bits(torch.randn(N, F, d, generator=g) * 0.05), bits(torch.randn(N, F, d, generator=g) * 0.05)
    Wd = bits(torch.randn(N, d, F, generator=g) * 0.05)
    y = np.zeros((B, d), np.uint16)
    assert A.oracle_moe_forward(x, W_g, Wg, Wu, Wd, B, d, F, N, k, 3, O.MODE_BATCH, prm, None, y) == 0
    ref = O.moe_forward(x, W_g, lambda e: (Wg[e], Wu[e], Wd[e]), k, 3, O.MODE_BATCH, k0=1)
    assert np.array_equal(y, O.f64_to_bf16_bits(ref["y"]))
