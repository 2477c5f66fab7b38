"""Seeded synthetic workloads shaped like the paper's MoE layers.

This module only draws random numbers: it holds none of the method's
arithmetic, so both the CUDA path and the CPU oracle can be fed from it.

Shapes follow the MoE layers the paper evaluates or cites (DeepSeek-R1,
Sec. 1 and App. A; a Qwen3-MoE-like layer for speculative verify batches,
Sec. 4; an OLMoE-like layer for plain decode batches, Sec. 3).  None of the
paper's models, weights or datasets are used: router inputs are drawn so that
the token-to-token correlation structure the method exploits is present
(independent tokens; tokens of one request sharing a request-level component,
Sec. 4 / Assumption 2; requests drawn from a few latent domains, Sec. 6.3).

Distributions (second parameter of N(., .) is a standard deviation):
  x     : bf16, see `x_kind` below
  W_g   : fp32, N(0, 1/sqrt(d)), so a logit has variance |x|^2 / d
  W_gate, W_up [N, F, d], W_down [N, d, F]: bf16, N(0, 0.02); shared experts alike
"""

from __future__ import annotations

import dataclasses
from typing import Dict, Optional, Tuple

import numpy as np
import torch

MODE_TOPK, MODE_BATCH, MODE_GROUP, MODE_HIER, MODE_THRESH = 0, 1, 2, 3, 4
MODES = {"topk": MODE_TOPK, "batch": MODE_BATCH, "group": MODE_GROUP, "hier": MODE_HIER,
         "thresh": MODE_THRESH}

EXPERT_STD = 0.02
# Layer stacks add each layer's output to the residual stream x.  A SwiGLU
# expert's output grows with |x|^2, so at N(0, 0.02) a DeepSeek-R1-sized layer
# returns about |x| itself and a stack's activations explode within a few
# layers.  Stacks therefore draw W_down with a ten times smaller deviation:
# a layer then adds roughly a tenth of |x|, and |x| stays near 1 over tens of
# layers (there is no normalisation between layers).
STACK_DOWN_STD = 0.002


@dataclasses.dataclass(frozen=True)
class Workload:
    """One MoE layer shape plus the selection settings it is run with."""
    name: str
    N: int              # routed experts
    k: int              # top-k per token
    d: int              # model dimension
    F: int              # SwiGLU hidden dimension (d_ff)
    B: int              # tokens in the batch
    mode: int           # MODE_*
    budget: int = 0     # m: experts added by the batch-level greedy step
    k0: int = 0         # warm-up top-k0
    m_r: int = 0        # per-request budget (HIER)
    tokens_per_request: int = 1   # 1 + L_s
    n_groups: int = 1   # G (GROUP)
    m_g: int = 0        # per-group budget (GROUP)
    tau: float = 0.0    # covered score-mass fraction (THRESH)
    sparse_scores: int = 0  # column scores from the top-k-masked gating values
    x_kind: str = "iid"  # "iid" | "request" | "domains"
    n_domains: int = 4
    domain_std: float = 1.5
    request_std: float = 1.0
    token_std: float = 0.5

    def params(self) -> Dict[str, int]:
        return dict(k0=self.k0, m_r=self.m_r, tokens_per_request=self.tokens_per_request,
                    n_groups=self.n_groups, m_g=self.m_g, tau=self.tau,
                    sparse_scores=self.sparse_scores)

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def expert_bytes(self) -> int:
        """bf16 bytes of one expert's three matrices."""
        return 6 * self.d * self.F


# The five layer shapes.  Sweeps vary B, budget, k0, m_r, m_g with `with_`.
TINY = Workload("tiny", N=64, k=8, d=512, F=256, B=32, mode=MODE_BATCH, budget=24, k0=0)
OLMOE = Workload("olmoe", N=64, k=8, d=2048, F=1024, B=32, mode=MODE_BATCH, budget=24, k0=0)
QWEN3 = Workload("qwen3", N=128, k=8, d=2048, F=768, B=256, mode=MODE_HIER, budget=0, k0=1,
                 m_r=4, tokens_per_request=4, x_kind="request")
DSR1 = Workload("dsr1", N=256, k=8, d=7168, F=2048, B=32, mode=MODE_BATCH, budget=24, k0=1,
                x_kind="domains")
DSR1_GROUP = Workload("dsr1_group", N=256, k=8, d=7168, F=2048, B=256, mode=MODE_GROUP,
                      k0=1, n_groups=8, m_g=5, tokens_per_request=4, x_kind="domains")

WORKLOADS = {w.name: w for w in (TINY, OLMOE, QWEN3, DSR1, DSR1_GROUP)}


def _gen(seed: int, stream: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed) * 1_000_003 + int(stream))
    return g


def router_inputs(w: Workload, seed: int = 0) -> Tuple[torch.Tensor, torch.Tensor]:
    """x [B, d] bf16 and W_g [N, d] fp32 on the CPU.

    x_kind:
      "iid"     : x_t ~ N(0, I_d) independently per token.
      "request" : requests are runs of `tokens_per_request` tokens;
                  x_t = a_r + token_std * z_t with a_r ~ N(0, request_std^2 I),
                  z_t ~ N(0, I): a request-level logit component N(0, 1) plus
                  per-token logit noise of std 0.5 under W_g ~ N(0, 1/sqrt(d)).
      "domains" : n_domains latent domains u_c ~ N(0, domain_std^2 I); each
                  request draws its domain uniformly; x_t = u_{c(r)} + z_t.
    """
    g = _gen(seed, 1)
    B, d, N = w.B, w.d, w.N
    W_g = torch.randn(N, d, generator=g, dtype=torch.float32) / float(np.sqrt(d))
    z = torch.randn(B, d, generator=g, dtype=torch.float32)
    T = max(1, w.tokens_per_request)
    R = (B + T - 1) // T
    req = torch.arange(B) // T
    if w.x_kind == "iid":
        x = z
    elif w.x_kind == "request":
        a = torch.randn(R, d, generator=g, dtype=torch.float32) * w.request_std
        x = a[req] + w.token_std * z
    elif w.x_kind == "domains":
        u = torch.randn(w.n_domains, d, generator=g, dtype=torch.float32) * w.domain_std
        dom = torch.randint(0, w.n_domains, (R,), generator=g)
        x = u[dom[req]] + z
    else:
        raise ValueError(w.x_kind)
    return x.to(torch.bfloat16), W_g


def batch_stream(w: Workload, seed: int, count: int) -> list:
    """`count` independent router-input batches (seeds seed, seed+1, ...) for
    rotating inputs between timed steps."""
    return [router_inputs(w, seed + i)[0] for i in range(count)]


def expert_weights(w: Workload, seed: int = 0, device: str = "cuda",
                   experts: Optional[list] = None, f_rows: Optional[int] = None,
                   down_std: float = EXPERT_STD) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """W_gate [N, F, d], W_up [N, F, d], W_down [N, d, F], bf16, N(0, 0.02)
    (W_down N(0, down_std)).

    Drawn expert by expert from a generator on `device`, so that peak
    temporary memory stays at one fp32 expert matrix.  With `experts` given
    (CPU only), only those experts are drawn and the tensors are
    [len(experts), ...]; each expert's values then depend on (seed, e) only.
    With `f_rows` (CPU only) only the first f_rows hidden units are drawn
    (W_gate, W_up [., f_rows, d], W_down [., d, f_rows]).
    """
    N, d = w.N, w.d
    F = w.F if f_rows is None else int(f_rows)
    ids = list(range(N)) if experts is None else list(experts)
    n = len(ids)
    Wg = torch.empty(n, F, d, dtype=torch.bfloat16, device=device)
    Wu = torch.empty(n, F, d, dtype=torch.bfloat16, device=device)
    Wd = torch.empty(n, d, F, dtype=torch.bfloat16, device=device)
    if device == "cpu" or experts is not None or f_rows is not None:
        for i, e in enumerate(ids):
            g = _gen(seed, 1000 + e)
            for t, shape, std in ((Wg, (F, d), EXPERT_STD), (Wu, (F, d), EXPERT_STD),
                                  (Wd, (d, F), down_std)):
                t[i].copy_(torch.randn(*shape, generator=g) * std)
    else:
        g = torch.Generator(device=device)
        g.manual_seed(int(seed) * 1_000_003 + 7)
        for i in range(n):
            for t, shape, std in ((Wg, (F, d), EXPERT_STD), (Wu, (F, d), EXPERT_STD),
                                  (Wd, (d, F), down_std)):
                t[i].copy_(torch.randn(*shape, generator=g, device=device) * std)
    return Wg, Wu, Wd


def shared_expert_weights(w: Workload, n_shared: int, seed: int = 0, device: str = "cuda",
                          down_std: float = EXPERT_STD
                          ) -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """Shared experts [n_shared, F, d], [n_shared, F, d], [n_shared, d, F], bf16,
    N(0, 0.02) (W_down N(0, down_std)), from a seed stream apart from the
    routed experts'."""
    return expert_weights(w.with_(N=n_shared), seed + 7_777_777, device=device, down_std=down_std)


def random_scores(B: int, N: int, seed: int, ties: bool = False) -> np.ndarray:
    """A [B, N] float32 matrix of positive scores for exercising selection alone.

    Draws exp(N(0, 1)) values (the unnormalised shape of softmax scores);
    with `ties` they are quantised to multiples of 1/8 so that equal column
    scores and equal per-token scores are common.
    """
    rng = np.random.default_rng(seed)
    v = np.exp(rng.standard_normal((B, N))) / N
    if ties:
        v = np.round(v * 8.0 * N) / (8.0 * N)
    return v.astype(np.float32)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw uint16 patterns of a bf16 tensor (copied to the host)."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
