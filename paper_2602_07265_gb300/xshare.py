"""ctypes binding of libxshare.so (include/xshare.h).

Argument marshalling only: each function checks tensor devices, dtypes and
contiguity, passes raw pointers and the current CUDA stream to the C ABI and
raises `XShareError` on a non-zero return code.  Every step of the layer runs
in the library's CUDA kernels; there is no other code path.  Importing this
module loads the library and raises if it has not been built.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from . import _build

MODE_TOPK, MODE_BATCH, MODE_GROUP, MODE_HIER, MODE_THRESH = 0, 1, 2, 3, 4
MODES = {"topk": MODE_TOPK, "batch": MODE_BATCH, "group": MODE_GROUP, "hier": MODE_HIER}

XS_DEV_OK, XS_DEV_TIMEOUT = 0, 1
STATS_FIELDS = ("n_selected", "n_used", "union_topk", "max_group_load", "n_pairs", "status")
STATS_WORDS = 8


class XShareError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: xshare error {code}: {xshare_strerror(code)}")


class RouteParams(ctypes.Structure):
    """xs_route_params."""
    _fields_ = [("k0", ctypes.c_int32), ("m_r", ctypes.c_int32),
                ("tokens_per_request", ctypes.c_int32), ("n_groups", ctypes.c_int32),
                ("m_g", ctypes.c_int32), ("tau", ctypes.c_float),
                ("sparse_scores", ctypes.c_int32)]


class SharedExperts(ctypes.Structure):
    """xs_shared_experts (device pointers and count)."""
    _fields_ = [("W_gate", ctypes.c_void_p), ("W_up", ctypes.c_void_p),
                ("W_down", ctypes.c_void_p), ("n_shared", ctypes.c_int32)]


MAX_SHARED = 8


class PackedExperts(ctypes.Structure):
    """xs_packed_experts (device pointers and count)."""
    _fields_ = [("gate_up", ctypes.c_void_p), ("down", ctypes.c_void_p), ("n", ctypes.c_int32)]


class Layer(ctypes.Structure):
    """xs_layer (device pointers; `shared`, `packed`, `packed_shared` may be NULL)."""
    _fields_ = [("W_g", ctypes.c_void_p), ("W_gate", ctypes.c_void_p),
                ("W_up", ctypes.c_void_p), ("W_down", ctypes.c_void_p),
                ("shared", ctypes.POINTER(SharedExperts)),
                ("packed", ctypes.POINTER(PackedExperts)),
                ("packed_shared", ctypes.POINTER(PackedExperts))]


def route_params(k0: int = 0, m_r: int = 0, tokens_per_request: int = 1, n_groups: int = 1,
                 m_g: int = 0, tau: float = 0.0, sparse_scores: int = 0) -> RouteParams:
    return RouteParams(k0, m_r, tokens_per_request, n_groups, m_g, tau, sparse_scores)


def _load() -> ctypes.CDLL:
    path = _build.LIB
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build() "
                           "(there is no fallback implementation)")
    lib = ctypes.CDLL(path)
    P, I, Z = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    PR = ctypes.POINTER(RouteParams)
    PS = ctypes.POINTER(SharedExperts)
    lib.xshare_workspace_size.argtypes = [I, I, I, I, I, I, PR, I]
    lib.xshare_workspace_size.restype = Z
    lib.xshare_route.argtypes = [P, I, I, I, I, I, PR, P, P, P, P, P, P, P, P, Z, P]
    lib.xshare_route.restype = I
    lib.xshare_moe_forward.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, PR, PS,
                                       P, P, P, P, P, P, P, Z, P]
    lib.xshare_moe_forward.restype = I
    lib.xshare_route_static.argtypes = [P, I, I, I, I, I, PR, P, P, P, P, P, P, P, P]
    lib.xshare_route_static.restype = I
    lib.xshare_moe_forward_profiled.argtypes = lib.xshare_moe_forward.argtypes + [P]
    lib.xshare_moe_forward_profiled.restype = I
    PP = ctypes.POINTER(PackedExperts)
    lib.xshare_pack_experts.argtypes = [P, P, P, I, I, I, P, P, P]
    lib.xshare_pack_experts.restype = I
    lib.xshare_moe_forward_packed.argtypes = [P, P, PP, I, I, I, I, I, I, I, PR, PP,
                                              P, P, P, P, P, P, P, Z, P, P]
    lib.xshare_moe_forward_packed.restype = I
    lib.xshare_moe_forward_ep.argtypes = [P, P, PP, I, I, I, I, I, I, I, PR, PP, I, I,
                                          P, P, P, P, P, Z, P]
    lib.xshare_moe_forward_ep.restype = I
    lib.xshare_ep_exchange_buffer.argtypes = [P, I, I, I, I, I, I, PR, I, ctypes.POINTER(P),
                                              ctypes.POINTER(Z)]
    lib.xshare_ep_exchange_buffer.restype = I
    lib.xshare_ep_combine.argtypes = [P, I, I, I, I, I, I, PR, I, P, P]
    lib.xshare_ep_combine.restype = I
    PL = ctypes.POINTER(Layer)
    lib.xshare_stack_forward.argtypes = [P, PL, I, I, I, I, I, I, I, I, PR, P, P, P, Z, P]
    lib.xshare_stack_forward.restype = I
    lib.xshare_stack_graph_create.argtypes = [P, PL, I, I, I, I, I, I, I, I, PR, P, P, P, Z,
                                              ctypes.POINTER(P)]
    lib.xshare_stack_graph_create.restype = I
    lib.xshare_stack_graph_launch.argtypes = [P, P]
    lib.xshare_stack_graph_launch.restype = I
    lib.xshare_stack_graph_destroy.argtypes = [P]
    lib.xshare_stack_graph_destroy.restype = None
    lib.xshare_selftest_wait_timeout.argtypes = [P, ctypes.c_uint64, P]
    lib.xshare_selftest_wait_timeout.restype = I
    lib.xshare_stage_name.argtypes = [I]
    lib.xshare_stage_name.restype = ctypes.c_char_p
    lib.xshare_strerror.argtypes = [I]
    lib.xshare_strerror.restype = ctypes.c_char_p
    return lib


LIB = _load()

N_STAGES = 7
STAGE_NAMES = [LIB.xshare_stage_name(i).decode() for i in range(N_STAGES)]


def xshare_strerror(code: int) -> str:
    return LIB.xshare_strerror(int(code)).decode()


def _ptr(t: Optional[torch.Tensor], dtype, name: str, numel: Optional[int] = None) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.device.index != torch.cuda.current_device():
        # The library launches on the current device.
        raise ValueError(f"{name} is on {t.device}, the current device is "
                         f"cuda:{torch.cuda.current_device()}")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} has {t.numel()} elements, needs {numel}")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check(rc: int, where: str):
    if rc != 0:
        raise XShareError(rc, where)


def xshare_workspace_size(B: int, N: int, k: int, d: int, F: int, mode: int,
                          params: RouteParams, n_shared: int = 0) -> int:
    """Bytes of workspace for these sizes (d = F = 0 for xshare_route); 0 if invalid."""
    return int(LIB.xshare_workspace_size(B, N, k, d, F, mode, ctypes.byref(params), n_shared))


def xshare_route(scores: torch.Tensor, k: int, budget: int, mode: int, params: RouteParams,
                 sel_mask: torch.Tensor, topk_ids: torch.Tensor, topk_w: torch.Tensor,
                 workspace: torch.Tensor, stats: Optional[torch.Tensor] = None,
                 expert_counts: Optional[torch.Tensor] = None,
                 expert_offsets: Optional[torch.Tensor] = None,
                 perm: Optional[torch.Tensor] = None, stream=None) -> None:
    """Selection + refinement (+ permutation) on fp32 scores [B, N]; see xshare.h."""
    B, N = scores.shape
    rc = LIB.xshare_route(
        _ptr(scores, torch.float32, "scores"), B, N, k, budget, mode, ctypes.byref(params),
        _ptr(sel_mask, torch.uint8, "sel_mask", N), _ptr(topk_ids, torch.int32, "topk_ids", B * k),
        _ptr(topk_w, torch.float32, "topk_w", B * k), _ptr(stats, torch.int32, "stats", STATS_WORDS),
        _ptr(expert_counts, torch.int32, "expert_counts", N),
        _ptr(expert_offsets, torch.int32, "expert_offsets", N + 1),
        _ptr(perm, torch.int32, "perm", B * k),
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream))
    _check(rc, "xshare_route")


STATIC_MAX_B = 1024


def xshare_route_static(scores: torch.Tensor, k: int, budget: int, mode: int,
                        params: RouteParams, sel_mask: torch.Tensor, topk_ids: torch.Tensor,
                        topk_w: torch.Tensor, stats: Optional[torch.Tensor] = None,
                        expert_counts: Optional[torch.Tensor] = None,
                        expert_offsets: Optional[torch.Tensor] = None,
                        perm: Optional[torch.Tensor] = None, stream=None) -> None:
    """xshare_route without a workspace, for callers that may not allocate
    device memory (B <= STATIC_MAX_B; see xshare.h)."""
    B, N = scores.shape
    rc = LIB.xshare_route_static(
        _ptr(scores, torch.float32, "scores"), B, N, k, budget, mode, ctypes.byref(params),
        _ptr(sel_mask, torch.uint8, "sel_mask", N), _ptr(topk_ids, torch.int32, "topk_ids", B * k),
        _ptr(topk_w, torch.float32, "topk_w", B * k), _ptr(stats, torch.int32, "stats", STATS_WORDS),
        _ptr(expert_counts, torch.int32, "expert_counts", N),
        _ptr(expert_offsets, torch.int32, "expert_offsets", N + 1),
        _ptr(perm, torch.int32, "perm", B * k), _stream(stream))
    _check(rc, "xshare_route_static")


def xshare_moe_forward(x: torch.Tensor, W_g: torch.Tensor, W_gate: torch.Tensor,
                       W_up: torch.Tensor, W_down: torch.Tensor, k: int, budget: int, mode: int,
                       params: RouteParams, y: torch.Tensor, workspace: torch.Tensor,
                       scores_out: Optional[torch.Tensor] = None,
                       sel_mask: Optional[torch.Tensor] = None,
                       topk_ids: Optional[torch.Tensor] = None,
                       topk_w: Optional[torch.Tensor] = None,
                       stats: Optional[torch.Tensor] = None, stream=None,
                       stage_events: Optional[list] = None,
                       shared: Optional[tuple] = None) -> None:
    """One MoE-layer forward into y [B, d] bf16; see xshare.h.

    `shared` = (S_gate [Ns, F, d], S_up [Ns, F, d], S_down [Ns, d, F]) bf16
    adds the shared experts.  With `stage_events` (XS_N_STAGES + 1
    torch.cuda.Event objects) the profiled entry point records them between
    the kernel launches."""
    B, d = x.shape
    N = W_g.shape[0]
    F = W_gate.shape[1]
    if W_g.shape[1] != d or tuple(W_gate.shape) != (N, F, d) or tuple(W_up.shape) != (N, F, d) \
            or tuple(W_down.shape) != (N, d, F) or tuple(y.shape) != (B, d):
        raise ValueError("inconsistent shapes: x [B,d], W_g [N,d], W_gate/W_up [N,F,d], "
                         "W_down [N,d,F], y [B,d]")
    sh = None
    if shared is not None:
        S_gate, S_up, S_down = shared
        Ns = S_gate.shape[0]
        if tuple(S_gate.shape) != (Ns, F, d) or tuple(S_up.shape) != (Ns, F, d) \
                or tuple(S_down.shape) != (Ns, d, F):
            raise ValueError("inconsistent shared-expert shapes: [Ns,F,d], [Ns,F,d], [Ns,d,F]")
        sh = SharedExperts(_ptr(S_gate, torch.bfloat16, "S_gate"),
                           _ptr(S_up, torch.bfloat16, "S_up"),
                           _ptr(S_down, torch.bfloat16, "S_down"), Ns)
    args = [
        _ptr(x, torch.bfloat16, "x"), _ptr(W_g, torch.float32, "W_g"),
        _ptr(W_gate, torch.bfloat16, "W_gate"), _ptr(W_up, torch.bfloat16, "W_up"),
        _ptr(W_down, torch.bfloat16, "W_down"), B, d, F, N, k, budget, mode,
        ctypes.byref(params), ctypes.byref(sh) if sh is not None else None,
        _ptr(y, torch.bfloat16, "y"),
        _ptr(scores_out, torch.float32, "scores_out", B * N),
        _ptr(sel_mask, torch.uint8, "sel_mask", N), _ptr(topk_ids, torch.int32, "topk_ids", B * k),
        _ptr(topk_w, torch.float32, "topk_w", B * k), _ptr(stats, torch.int32, "stats", STATS_WORDS),
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)]
    if stage_events is None:
        _check(LIB.xshare_moe_forward(*args), "xshare_moe_forward")
        return
    if len(stage_events) != N_STAGES + 1:
        raise ValueError(f"stage_events needs {N_STAGES + 1} events")
    handles = (ctypes.c_void_p * (N_STAGES + 1))()
    for i, ev in enumerate(stage_events):
        if not ev.cuda_event:
            ev.record()   # torch creates the CUDA event lazily
        handles[i] = ev.cuda_event
    _check(LIB.xshare_moe_forward_profiled(*args, handles), "xshare_moe_forward_profiled")


class Packed:
    """Packed expert weights (xshare_pack_experts) on the device: gate_up and
    down byte buffers plus the expert count, d and F."""

    def __init__(self, W_gate: torch.Tensor, W_up: torch.Tensor, W_down: torch.Tensor, stream=None):
        n, F, d = W_gate.shape
        if tuple(W_up.shape) != (n, F, d) or tuple(W_down.shape) != (n, d, F):
            raise ValueError("W_gate, W_up [n, F, d] and W_down [n, d, F]")
        self.n, self.d, self.F = n, d, F
        self.gate_up = torch.empty(n * F * d * 2 * 2, dtype=torch.uint8, device=W_gate.device)
        self.down = torch.empty(n * d * F * 2, dtype=torch.uint8, device=W_gate.device)
        _check(LIB.xshare_pack_experts(_ptr(W_gate, torch.bfloat16, "W_gate"),
                                       _ptr(W_up, torch.bfloat16, "W_up"),
                                       _ptr(W_down, torch.bfloat16, "W_down"), n, d, F,
                                       self.gate_up.data_ptr(), self.down.data_ptr(),
                                       _stream(stream)), "xshare_pack_experts")

    def struct(self) -> PackedExperts:
        return PackedExperts(self.gate_up.data_ptr(), self.down.data_ptr(), self.n)

    def experts(self, lo: int, hi: int) -> "Packed":
        """Experts lo .. hi-1 as packed weights of their own (views of these
        buffers: the packed layout keeps each expert's tiles contiguous)."""
        if not 0 <= lo < hi <= self.n:
            raise ValueError(f"expert range [{lo}, {hi}) outside [0, {self.n})")
        v = Packed.__new__(Packed)
        v.n, v.d, v.F = hi - lo, self.d, self.F
        gu, dn = self.F * self.d * 2 * 2, self.d * self.F * 2
        v.gate_up = self.gate_up[lo * gu:hi * gu]
        v.down = self.down[lo * dn:hi * dn]
        return v


def xshare_moe_forward_packed(x: torch.Tensor, W_g: torch.Tensor, experts: Packed, k: int,
                              budget: int, mode: int, params: RouteParams, y: torch.Tensor,
                              workspace: torch.Tensor, shared: Optional[Packed] = None,
                              scores_out: Optional[torch.Tensor] = None,
                              sel_mask: Optional[torch.Tensor] = None,
                              topk_ids: Optional[torch.Tensor] = None,
                              topk_w: Optional[torch.Tensor] = None,
                              stats: Optional[torch.Tensor] = None, stream=None,
                              stage_events: Optional[list] = None) -> None:
    """xshare_moe_forward on packed expert weights; see xshare.h."""
    B, d = x.shape
    N = W_g.shape[0]
    if experts.n != N or experts.d != d or tuple(y.shape) != (B, d) or W_g.shape[1] != d:
        raise ValueError("inconsistent shapes")
    ex = experts.struct()
    sh = shared.struct() if shared is not None else None
    handles = None
    if stage_events is not None:
        if len(stage_events) != N_STAGES + 1:
            raise ValueError(f"stage_events needs {N_STAGES + 1} events")
        handles = (ctypes.c_void_p * (N_STAGES + 1))()
        for i, ev in enumerate(stage_events):
            if not ev.cuda_event:
                ev.record()
            handles[i] = ev.cuda_event
    rc = LIB.xshare_moe_forward_packed(
        _ptr(x, torch.bfloat16, "x"), _ptr(W_g, torch.float32, "W_g"), ctypes.byref(ex), B, d,
        experts.F, N, k, budget, mode, ctypes.byref(params),
        ctypes.byref(sh) if sh is not None else None, _ptr(y, torch.bfloat16, "y"),
        _ptr(scores_out, torch.float32, "scores_out", B * N),
        _ptr(sel_mask, torch.uint8, "sel_mask", N), _ptr(topk_ids, torch.int32, "topk_ids", B * k),
        _ptr(topk_w, torch.float32, "topk_w", B * k), _ptr(stats, torch.int32, "stats", STATS_WORDS),
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream), handles)
    _check(rc, "xshare_moe_forward_packed")


def xshare_moe_forward_ep(x: torch.Tensor, W_g: torch.Tensor, local_experts: Packed, k: int,
                          budget: int, mode: int, params: RouteParams, n_ranks: int, rank: int,
                          workspace: torch.Tensor, shared: Optional[Packed] = None,
                          sel_mask: Optional[torch.Tensor] = None,
                          topk_ids: Optional[torch.Tensor] = None,
                          topk_w: Optional[torch.Tensor] = None,
                          stats: Optional[torch.Tensor] = None, stream=None) -> None:
    """This rank's part of an expert-parallel layer forward (routing of the
    whole batch, the FFN of expert group `rank`); see xshare.h."""
    B, d = x.shape
    N = W_g.shape[0]
    if local_experts.n * n_ranks != N or local_experts.d != d or W_g.shape[1] != d:
        raise ValueError("inconsistent shapes")
    ex = local_experts.struct()
    sh = shared.struct() if shared is not None else None
    rc = LIB.xshare_moe_forward_ep(
        _ptr(x, torch.bfloat16, "x"), _ptr(W_g, torch.float32, "W_g"), ctypes.byref(ex), B, d,
        local_experts.F, N, k, budget, mode, ctypes.byref(params),
        ctypes.byref(sh) if sh is not None else None, n_ranks, rank,
        _ptr(sel_mask, torch.uint8, "sel_mask", N), _ptr(topk_ids, torch.int32, "topk_ids", B * k),
        _ptr(topk_w, torch.float32, "topk_w", B * k), _ptr(stats, torch.int32, "stats", STATS_WORDS),
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream))
    _check(rc, "xshare_moe_forward_ep")


def ep_exchange_buffer(workspace: torch.Tensor, B: int, N: int, k: int, d: int, F: int, mode: int,
                       params: RouteParams, n_shared: int = 0) -> torch.Tensor:
    """The exchange buffer of an expert-parallel forward: an fp32 view of the
    workspace (xshare_ep_exchange_buffer)."""
    buf, count = ctypes.c_void_p(), ctypes.c_size_t()
    _check(LIB.xshare_ep_exchange_buffer(_ptr(workspace, torch.uint8, "workspace"), B, N, k, d, F,
                                         mode, ctypes.byref(params), n_shared, ctypes.byref(buf),
                                         ctypes.byref(count)), "xshare_ep_exchange_buffer")
    off = buf.value - workspace.data_ptr()
    if off < 0 or off + 4 * count.value > workspace.numel():
        raise XShareError(-4, "ep_exchange_buffer")
    return workspace[off:off + 4 * count.value].view(torch.float32)


def xshare_ep_combine(workspace: torch.Tensor, B: int, N: int, k: int, d: int, F: int, mode: int,
                      params: RouteParams, y: torch.Tensor, n_shared: int = 0, stream=None) -> None:
    """The weighted combine after the exchange; see xshare.h."""
    if tuple(y.shape) != (B, d):
        raise ValueError("y must be [B, d]")
    _check(LIB.xshare_ep_combine(_ptr(workspace, torch.uint8, "workspace"), B, N, k, d, F, mode,
                                 ctypes.byref(params), n_shared, _ptr(y, torch.bfloat16, "y"),
                                 _stream(stream)), "xshare_ep_combine")


def ep_layer_forward(x: torch.Tensor, W_g: torch.Tensor, local_experts: Packed, k: int,
                     budget: int, mode: int, params: RouteParams, y: torch.Tensor,
                     workspace: torch.Tensor, group=None, shared: Optional[Packed] = None,
                     stats: Optional[torch.Tensor] = None, n_shared: int = 0) -> None:
    """One expert-parallel layer forward over the ranks of a torch.distributed
    process group (one GPU per rank): this rank's forward, an in-place sum
    all-reduce of the exchange buffers, the combine."""
    import torch.distributed as dist
    n_ranks = dist.get_world_size(group)
    rank = dist.get_rank(group)
    B, d = x.shape
    N = W_g.shape[0]
    xshare_moe_forward_ep(x, W_g, local_experts, k, budget, mode, params, n_ranks, rank, workspace,
                          shared=shared, stats=stats)
    buf = ep_exchange_buffer(workspace, B, N, k, d, local_experts.F, mode, params, n_shared)
    dist.all_reduce(buf, op=dist.ReduceOp.SUM, group=group)
    xshare_ep_combine(workspace, B, N, k, d, local_experts.F, mode, params, y, n_shared)


def _stack_args(x, layers, k, K_total, mode, params, h_out, workspace, stats):
    """Marshals a layer stack: `layers` is a list of (W_g, W_gate, W_up, W_down)
    or (W_g, W_gate, W_up, W_down, (S_gate, S_up, S_down)) tensors, or of
    (W_g, Packed[, Packed shared]) for packed expert weights."""
    B, d = x.shape
    L = len(layers)
    if L < 1:
        raise ValueError("at least one layer")
    first = layers[0][1]
    N, F = (first.n, first.F) if isinstance(first, Packed) else (first.shape[0], first.shape[1])
    arr = (Layer * L)()
    keep = []
    for l, lay in enumerate(layers):
        W_g = lay[0]
        if W_g.shape != (N, d):
            raise ValueError(f"layer {l}: W_g must be [N, d]")
        arr[l].W_g = _ptr(W_g, torch.float32, "W_g")
        if isinstance(lay[1], Packed):
            pk = lay[1].struct()
            keep.append(pk)
            arr[l].packed = ctypes.pointer(pk)
            if len(lay) > 2 and lay[2] is not None:
                ps = lay[2].struct()
                keep.append(ps)
                arr[l].packed_shared = ctypes.pointer(ps)
            continue
        Wg, Wu, Wd = lay[1:4]
        if tuple(Wg.shape) != (N, F, d) or tuple(Wu.shape) != (N, F, d) or tuple(Wd.shape) != (N, d, F):
            raise ValueError(f"layer {l}: inconsistent shapes")
        arr[l].W_gate = _ptr(Wg, torch.bfloat16, "W_gate")
        arr[l].W_up = _ptr(Wu, torch.bfloat16, "W_up")
        arr[l].W_down = _ptr(Wd, torch.bfloat16, "W_down")
        if len(lay) > 4 and lay[4] is not None:
            Sg, Su, Sd = lay[4]
            sh = SharedExperts(_ptr(Sg, torch.bfloat16, "S_gate"), _ptr(Su, torch.bfloat16, "S_up"),
                               _ptr(Sd, torch.bfloat16, "S_down"), Sg.shape[0])
            keep.append(sh)
            arr[l].shared = ctypes.pointer(sh)
    if tuple(h_out.shape) != (L, B, d):
        raise ValueError("h_out must be [L, B, d]")
    args = [_ptr(x, torch.bfloat16, "x"), arr, L, B, d, F, N, k, K_total, mode,
            ctypes.byref(params), _ptr(h_out, torch.bfloat16, "h_out"),
            _ptr(stats, torch.int32, "stats", L * STATS_WORDS),
            _ptr(workspace, torch.uint8, "workspace"), workspace.numel()]
    return args, keep


def xshare_stack_forward(x: torch.Tensor, layers: list, k: int, K_total: int, mode: int,
                         params: RouteParams, h_out: torch.Tensor, workspace: torch.Tensor,
                         stats: Optional[torch.Tensor] = None, stream=None) -> None:
    """L residual MoE layers under the global budget K_total into h_out [L, B, d]; see xshare.h."""
    args, keep = _stack_args(x, layers, k, K_total, mode, params, h_out, workspace, stats)
    _check(LIB.xshare_stack_forward(*args, _stream(stream)), "xshare_stack_forward")
    del keep


class StackGraph:
    """xshare_stack_graph_create / _launch / _destroy.  Keeps references to the
    tensors it was captured with, which replays read and write."""

    def __init__(self, x, layers, k, K_total, mode, params, h_out, workspace, stats=None):
        self._args, self._keep = _stack_args(x, layers, k, K_total, mode, params, h_out,
                                             workspace, stats)
        self._tensors = (x, layers, h_out, workspace, stats, params)
        self._handle = ctypes.c_void_p()
        _check(LIB.xshare_stack_graph_create(*self._args, ctypes.byref(self._handle)),
               "xshare_stack_graph_create")

    def launch(self, stream=None) -> None:
        _check(LIB.xshare_stack_graph_launch(self._handle, _stream(stream)),
               "xshare_stack_graph_launch")

    def close(self) -> None:
        if self._handle:
            LIB.xshare_stack_graph_destroy(self._handle)
            self._handle = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass


def xshare_selftest_wait_timeout(stats: torch.Tensor, budget_ns: int, stream=None) -> None:
    """Run the bounded-wait self-test kernel; see xshare.h."""
    _check(LIB.xshare_selftest_wait_timeout(_ptr(stats, torch.int32, "stats", STATS_WORDS),
                                            int(budget_ns), _stream(stream)),
           "xshare_selftest_wait_timeout")


def stats_dict(stats: torch.Tensor) -> dict:
    """Host view of an xs_stats tensor (copies to the host, so it synchronises)."""
    v = stats.cpu().tolist()
    return {name: int(v[i]) for i, name in enumerate(STATS_FIELDS)}
