"""The oracle behind the parameter lists of the C ABI (include/xshare.h).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``.  ``oracle_route`` and
``oracle_moe_forward`` take the arguments of ``xshare_route`` and
``xshare_moe_forward`` in the same order, with host numpy arrays where the
library takes device pointers and without the workspace and stream, and
write their results into the given output arrays, so a test can hand both
sides one argument list.  The arithmetic is ``xshare_oracle``'s; this module
only unpacks arguments and packs results.

Layouts follow the header: scores [B, N] fp32; sel_mask [N] uint8; topk_ids
[B, k] int32; topk_w [B, k] fp32; stats int32[8] (n_selected, n_used,
union_topk, max_group_load, n_pairs, status, 0, 0); expert_counts [N],
expert_offsets [N + 1], perm [B k] int32; x [B, d], W_gate / W_up [N, F, d],
W_down [N, d, F] and y [B, d] as uint16 bf16 patterns; W_g [N, d] fp32.
``prm`` is a mapping or object with the fields of xs_route_params.  Returns
0, or the header's negative code for the argument errors it checks.
"""

from __future__ import annotations

from typing import Optional

import numpy as np

from . import xshare_oracle as O

XS_OK, XS_ERR_SHAPE, XS_ERR_PARAM, XS_ERR_NULL = 0, -1, -2, -3
_FIELDS = ("k0", "m_r", "tokens_per_request", "n_groups", "m_g", "tau", "sparse_scores")


def _params(prm) -> dict:
    if isinstance(prm, dict):
        return {f: prm.get(f, 0 if f != "tokens_per_request" else 1) for f in _FIELDS}
    return {f: getattr(prm, f) for f in _FIELDS}


def _check(B, N, k, budget, mode, p) -> int:
    if B < 1 or B > 8192 or N < 1 or N > 1024 or k < 1 or k > 16 or k > N:
        return XS_ERR_SHAPE
    if mode not in (O.MODE_TOPK, O.MODE_BATCH, O.MODE_GROUP, O.MODE_HIER, O.MODE_THRESH):
        return XS_ERR_PARAM
    if budget < 0 or p["k0"] < 0 or p["k0"] > 16 or p["m_r"] < 0 or p["m_g"] < 0:
        return XS_ERR_PARAM
    G = p["n_groups"]
    if G < 0 or (G > 0 and (G > N or N % G)) or (mode == O.MODE_GROUP and G < 1):
        return XS_ERR_PARAM
    T = p["tokens_per_request"]
    if mode == O.MODE_HIER and (T < 1 or T > B or B % T):
        return XS_ERR_PARAM
    if mode == O.MODE_THRESH and not (0.0 <= p["tau"] <= 1.0):
        return XS_ERR_PARAM
    if p["sparse_scores"] not in (0, 1):
        return XS_ERR_PARAM
    return XS_OK


def _route_kwargs(p) -> dict:
    return dict(k0=0 if p["k0"] is None else p["k0"], m_r=p["m_r"],
                tokens_per_request=max(1, p["tokens_per_request"]), n_groups=max(1, p["n_groups"]),
                m_g=p["m_g"], tau=p["tau"], sparse_scores=p["sparse_scores"])


def _write_route(r, k, sel_mask, topk_ids, topk_w, stats, expert_counts, expert_offsets, perm):
    sel_mask[...] = r["mask"]
    topk_ids[...] = r["ids"]
    topk_w[...] = r["w"]
    if stats is not None:
        stats[...] = [r["n_selected"], r["n_used"], r["union_topk"], r["max_group_load"],
                      int(r["offsets"][-1]), 0, 0, 0]
    if expert_counts is not None:
        expert_counts[...] = r["counts"]
    if expert_offsets is not None:
        expert_offsets[...] = r["offsets"]
    if perm is not None:
        perm.reshape(-1)[:len(r["perm"])] = r["perm"]


def oracle_route(scores: np.ndarray, B: int, N: int, k: int, budget: int, mode: int, prm,
                 sel_mask: np.ndarray, topk_ids: np.ndarray, topk_w: np.ndarray,
                 stats: Optional[np.ndarray] = None, expert_counts: Optional[np.ndarray] = None,
                 expert_offsets: Optional[np.ndarray] = None,
                 perm: Optional[np.ndarray] = None) -> int:
    """xshare_route's arguments, host arrays (selection and refinement, Sec. 3-5)."""
    p = _params(prm)
    rc = _check(B, N, k, budget, mode, p)
    if rc != XS_OK:
        return rc
    if scores is None or sel_mask is None or topk_ids is None or topk_w is None:
        return XS_ERR_NULL
    kw = _route_kwargs(p)
    if mode == O.MODE_TOPK:
        kw["k0"] = 0
    r = O.route(np.asarray(scores, dtype=np.float32).reshape(B, N), k, budget, mode, **kw)
    _write_route(r, k, sel_mask, topk_ids, topk_w, stats, expert_counts, expert_offsets, perm)
    return XS_OK


def oracle_moe_forward(x: np.ndarray, W_g: np.ndarray, W_gate: np.ndarray, W_up: np.ndarray,
                       W_down: np.ndarray, B: int, d: int, F: int, N: int, k: int, budget: int,
                       mode: int, prm, shared, y: np.ndarray,
                       scores_out: Optional[np.ndarray] = None,
                       sel_mask: Optional[np.ndarray] = None,
                       topk_ids: Optional[np.ndarray] = None,
                       topk_w: Optional[np.ndarray] = None,
                       stats: Optional[np.ndarray] = None) -> int:
    """xshare_moe_forward's arguments, host arrays (the layer of Sec. 2.1).

    ``shared`` is None or (S_gate [n, F, d], S_up [n, F, d], S_down [n, d, F])
    bf16 patterns.  y receives the bf16 rounding of the fp64 result.
    """
    p = _params(prm)
    rc = _check(B, N, k, budget, mode, p)
    if rc != XS_OK:
        return rc
    if d < 128 or F < 128 or d % 128 or F % 128:
        return XS_ERR_SHAPE
    if any(a is None for a in (x, W_g, W_gate, W_up, W_down, y)):
        return XS_ERR_NULL
    kw = _route_kwargs(p)
    if mode == O.MODE_TOPK:
        kw["k0"] = 0
    get = lambda e: (W_gate[e], W_up[e], W_down[e])
    extra = {}
    if shared is not None:
        Sg, Su, Sd = shared
        extra = dict(n_shared=Sg.shape[0], get_shared=lambda j: (Sg[j], Su[j], Sd[j]))
    r = O.moe_forward(np.asarray(x, dtype=np.uint16).reshape(B, d), np.asarray(W_g).reshape(N, d),
                      get, k, budget, mode, **extra, **kw)
    y[...] = O.f64_to_bf16_bits(r["y"]).reshape(y.shape)
    if scores_out is not None:
        scores_out[...] = r["p"]
    if sel_mask is not None:
        sel_mask[...] = r["mask"]
    if topk_ids is not None:
        topk_ids[...] = r["ids"]
    if topk_w is not None:
        topk_w[...] = r["w"]
    if stats is not None:
        stats[...] = [r["n_selected"], r["n_used"], r["union_topk"], r["max_group_load"],
                      int(r["offsets"][-1]), 0, 0, 0]
    return XS_OK
