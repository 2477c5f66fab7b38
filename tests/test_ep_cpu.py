"""Expert parallelism (Sec. 5) on the CPU: the oracle's per-device forward,
the exchange as a sum over devices and the combine reproduce the one-device
layer forward exactly.

* In one process: G = 1, 2, 4 and N devices (one expert each), BATCH and
  GROUP selection, with and without shared experts.
* Over two gloo ranks (world size 2, separate processes): each rank draws
  only its own experts' weights, the exchange is torch.distributed's
  all_reduce, and both ranks end with the one-device output, bit for bit
  (fp64: every exchange row is non-zero on exactly one rank, so the sum is
  exact).
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

from oracle import xshare_oracle as O
from paper_2602_07265_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CASES = [
    (W.TINY, 0),
    (W.TINY.with_(k0=1, budget=16), 2),
    (W.TINY.with_(mode=W.MODE_GROUP, n_groups=4, m_g=5, k0=1), 1),
    (W.TINY.with_(B=7, budget=3), 0),
]


def _inputs(w, seed, n_shared):
    x, W_g = W.router_inputs(w, seed)
    Wg, Wu, Wd = W.expert_weights(w, seed, device="cpu", experts=list(range(w.N)))
    experts = {e: (W.bf16_bits(Wg[e]), W.bf16_bits(Wu[e]), W.bf16_bits(Wd[e])) for e in range(w.N)}
    shared = []
    if n_shared:
        Sg, Su, Sd = W.shared_expert_weights(w, n_shared, seed, device="cpu")
        shared = [(W.bf16_bits(Sg[j]), W.bf16_bits(Su[j]), W.bf16_bits(Sd[j])) for j in range(n_shared)]
    return W.bf16_bits(x), W_g.numpy(), experts, shared


@pytest.mark.parametrize("case", range(len(CASES)))
@pytest.mark.parametrize("G", [1, 2, 4, 64])
def test_ep_oracle_equals_one_device(case, G):
    w, ns = CASES[case]
    xb, Wg, experts, shared = _inputs(w, 3, ns)
    extra = dict(get_shared=shared.__getitem__, n_shared=ns) if ns else {}
    ref = O.moe_forward(xb, Wg, experts.__getitem__, w.k, w.budget, w.mode, **extra, **w.params())
    total = None
    for g in range(G):
        lo, hi = O.expert_group_range(w.N, G, g)

        def local(e, lo=lo, hi=hi):
            assert lo <= e < hi, f"device {g} asked for expert {e} outside its group"
            return experts[e]
        r = O.moe_forward_ep_rank(xb, Wg, local, w.k, w.budget, w.mode, G, g, **extra, **w.params())
        # The routing is the same on every device.
        assert np.array_equal(r["mask"], ref["mask"]) and np.array_equal(r["ids"], ref["ids"])
        assert np.array_equal(r["w"], ref["w"]) and np.array_equal(r["perm"], ref["perm"])
        nz = np.any(r["out"] != 0, axis=1)
        if total is None:
            total, owners = np.zeros_like(r["out"]), np.zeros(len(nz), dtype=int)
        owners += nz
        total += r["out"]
    assert owners.max() <= 1, "an exchange row computed by two devices"
    y = O.ep_combine(ref, total, ns)
    assert np.array_equal(y, ref["y"]), np.abs(y - ref["y"]).max()


def test_ep_group_range_partition():
    """The G groups are contiguous, of N/G experts, and cover E once."""
    for N, G in [(64, 1), (64, 8), (256, 8), (128, 128)]:
        seen = []
        for g in range(G):
            lo, hi = O.expert_group_range(N, G, g)
            assert hi - lo == N // G
            seen.extend(range(lo, hi))
        assert seen == list(range(N))
    with pytest.raises(ValueError):
        O.expert_group_range(100, 8, 0)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    from oracle import xshare_oracle as Orc
    from paper_2602_07265_gb300 import workloads as Wl
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w = Wl.TINY.with_(k0=1, budget=16)
    x, W_g = Wl.router_inputs(w, 5)
    lo, hi = Orc.expert_group_range(w.N, world, rank)
    Wg, Wu, Wd = Wl.expert_weights(w, 5, device="cpu", experts=list(range(lo, hi)))
    local = {lo + i: (Wl.bf16_bits(Wg[i]), Wl.bf16_bits(Wu[i]), Wl.bf16_bits(Wd[i]))
             for i in range(hi - lo)}
    Sg, Su, Sd = Wl.shared_expert_weights(w, 1, 5, device="cpu")
    shared = [(Wl.bf16_bits(Sg[0]), Wl.bf16_bits(Su[0]), Wl.bf16_bits(Sd[0]))]
    r = Orc.moe_forward_ep_rank(Wl.bf16_bits(x), W_g.numpy(), local.__getitem__, w.k, w.budget,
                                w.mode, world, rank, get_shared=shared.__getitem__, n_shared=1,
                                **w.params())
    buf = torch.from_numpy(r["out"].copy())
    dist.all_reduce(buf, op=dist.ReduceOp.SUM)
    y = Orc.ep_combine(r, buf.numpy(), 1)
    q.put((rank, y, np.any(r["out"] != 0, axis=1)))
    dist.destroy_process_group()


def test_ep_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=300) for _ in range(2)), key=lambda v: v[0])
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    w = W.TINY.with_(k0=1, budget=16)
    xb, Wg, experts, shared = _inputs(w, 5, 1)
    ref = O.moe_forward(xb, Wg, experts.__getitem__, w.k, w.budget, w.mode,
                        get_shared=shared.__getitem__, n_shared=1, **w.params())
    (_, y0, nz0), (_, y1, nz1) = res
    assert not np.any(nz0 & nz1), "a row computed on both ranks"
    assert np.array_equal(y0, ref["y"]) and np.array_equal(y1, ref["y"])
