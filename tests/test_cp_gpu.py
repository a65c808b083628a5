"""GPU parity of the context-parallel forward (App. A.3: the Exchange summary (m, l, z) merges
associatively; App. A.3.3-A.3.5: the epilogue from the summary): a sequence computed shard
by shard -- each shard's own causal summary, merged with its summaries over every earlier
shard's keys, then finished at the shard's positions -- against the fp64 oracle of the
whole sequence on every head, and against the single-call forward."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20172_gb300 import binding, workloads
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    binding.load()


def _sharded_forward(q, k, v, bounds, lam, tau):
    """Y, logZ of the whole sequence from shards [bounds[i], bounds[i + 1])."""
    ys, lzs = [], []
    for s in range(len(bounds) - 1):
        a, b = bounds[s], bounds[s + 1]
        qs, ks, vs = (t[:, a:b].contiguous() for t in (q, k, v))
        state = binding.fwd_state(qs, ks, vs, causal=True)
        for e in range(s):  # every earlier shard's keys
            c0, c1 = bounds[e], bounds[e + 1]
            other = binding.fwd_state(qs, k[:, c0:c1].contiguous(), v[:, c0:c1].contiguous(),
                                      causal=False)
            binding.state_merge(state, other)
        y, lz = binding.state_finish(qs, ks, vs, state, lam, tau, pos0=a)
        ys.append(y)
        lzs.append(lz)
    return torch.cat(ys, dim=1), torch.cat(lzs, dim=2)


@pytest.mark.parametrize("d", [48, 64, 128])
@pytest.mark.parametrize("bounds", [(0, 250, 513, 700), (0, 1, 130, 131, 300), (0, 128, 256)])
def test_sharded_forward_matches_the_whole_sequence(d, bounds):
    T = bounds[-1]
    w = workloads.custom(2, 3, T, d, "bf16")
    q, k, v, _ = workloads.make_inputs(w, seed=40 + d + T)
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    dev = torch.device("cuda:0")
    qd, kd, vd = (t.to(dev) for t in (q, k, v))
    y, lz = _sharded_forward(qd, kd, vd, list(bounds), lam, tau)
    y_one, lz_one = binding.fwd(qd, kd, vd, lam, tau, kernel="tcgen05")
    torch.cuda.synchronize()
    y, lz = y.float().cpu(), lz.cpu()
    y_one, lz_one = y_one.float().cpu(), lz_one.cpu()
    for b in range(w.B):
        for h in range(w.H):
            ry, rlz = oracle.fwd(pu.head(q, b, h), pu.head(k, b, h), pu.head(v, b, h), lam, tau)
            pu.check_recorded("context-parallel", f"Y d={d}", y[b, :, h].numpy(), ry, "bf16",
                              "out")
            pu.check_logz(f"logZ[{b},{h}]", lz[b, h].numpy(), rlz, "bf16")
            pu.check(f"sharded vs one call [{b},{h}]", y[b, :, h].numpy(),
                     y_one[b, :, h].numpy(), "bf16", "out")
            assert np.max(np.abs(lz[b, h].numpy() - lz_one[b, h].numpy())) < 1e-3


def test_merge_order_and_the_empty_summary():
    """Merging is associative and commutative up to fp32 rounding, and the empty summary
    (row 0 of a causal shard: m = -inf, l = 0, z = 0) is its identity."""
    w = workloads.custom(1, 2, 384, 64, "bf16")
    q, k, v, _ = workloads.make_inputs(w, seed=9)
    dev = torch.device("cuda:0")
    qd, kd, vd = (t.to(dev) for t in (q, k, v))
    parts = [binding.fwd_state(qd[:, 256:].contiguous(), kd[:, i:i + 128].contiguous(),
                               vd[:, i:i + 128].contiguous(), causal=False)
             for i in (0, 128)]
    own = binding.fwd_state(qd[:, 256:].contiguous(), kd[:, 256:].contiguous(),
                            vd[:, 256:].contiguous(), causal=True)
    clone = lambda st: tuple(t.clone() for t in st)
    a = binding.state_merge(binding.state_merge(clone(own), parts[0]), parts[1])
    b = binding.state_merge(binding.state_merge(clone(parts[1]), parts[0]), own)
    torch.cuda.synchronize()
    assert torch.isinf(own[0][:, :, 0]).all() and (own[1][:, :, 0] == 0).all()
    assert (own[2][:, :, 0] == 0).all()
    # compare z / l (the normalised Exchange mean), which does not depend on the scale m
    za, zb = a[2] / a[1][..., None], b[2] / b[1][..., None]
    assert torch.allclose(za, zb, rtol=1e-5, atol=1e-6)
    la = a[1].log() + a[0]
    lb = b[1].log() + b[0]
    assert torch.allclose(la, lb, rtol=0, atol=1e-5)
    empty = (torch.full_like(own[0], -float("inf")), torch.zeros_like(own[1]),
             torch.zeros_like(own[2]))
    c = binding.state_merge(clone(parts[0]), empty)
    torch.cuda.synchronize()
    for x, y in zip(c, parts[0]):
        assert torch.equal(x, y)


def test_state_against_the_oracle_rows():
    """A shard of 60 queries at positions 100..159 over an earlier shard of 100 keys (a
    ragged key count: the last key tile masked past them), merged with its own causal
    summary and finished at its positions: the whole sequence's rows 100..159 of the
    oracle."""
    w = workloads.custom(1, 2, 160, 64, "bf16")
    q, k, v, _ = workloads.make_inputs(w, seed=17)
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    dev = torch.device("cuda:0")
    qd, kd, vd = (t.to(dev) for t in (q, k, v))
    # queries at positions 100..159 against keys 0..99 only: the causal own part is kept,
    # so the result is the whole forward's rows 100..159
    own = binding.fwd_state(qd[:, 100:].contiguous(), kd[:, 100:].contiguous(),
                            vd[:, 100:].contiguous(), causal=True)
    other = binding.fwd_state(qd[:, 100:].contiguous(), kd[:, :100].contiguous(),
                              vd[:, :100].contiguous(), causal=False)
    binding.state_merge(own, other)
    y, lz = binding.state_finish(qd[:, 100:].contiguous(), kd[:, 100:].contiguous(),
                                 vd[:, 100:].contiguous(), own, lam, tau, pos0=100)
    torch.cuda.synchronize()
    for h in range(w.H):
        ry, rlz = oracle.fwd(pu.head(q, 0, h), pu.head(k, 0, h), pu.head(v, 0, h), lam, tau)
        pu.check(f"rows 100.. h={h}", y[0, :, h].float().cpu().numpy(), ry[100:], "bf16", "out")
        pu.check_logz(f"logZ h={h}", lz[0, h].cpu().numpy(), rlz[100:], "bf16")


def test_sharded_forward_on_bhtd_storage():
    """Shards of [B, H, T, d] storage (permuted views: every stride differs from the dense
    layout) give the dense layout's results."""
    w = workloads.custom(2, 2, 300, 64, "bf16")
    q, k, v, _ = workloads.make_inputs(w, seed=5)
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    dev = torch.device("cuda:0")

    def bhtd(t):
        return t.permute(0, 2, 1, 3).contiguous().to(dev).permute(0, 2, 1, 3)

    def shards(qq, kk, vv):
        a, b = 0, 130
        st = binding.fwd_state(qq[:, b:], kk[:, b:], vv[:, b:], causal=True)
        binding.state_merge(st, binding.fwd_state(qq[:, b:], kk[:, a:b], vv[:, a:b], causal=False))
        return binding.state_finish(qq[:, b:], kk[:, b:], vv[:, b:], st, lam, tau, pos0=b)

    y0, l0 = shards(*(t.to(dev) for t in (q, k, v)))
    y1, l1 = shards(*(bhtd(t) for t in (q, k, v)))
    torch.cuda.synchronize()
    assert torch.equal(y0.contiguous(), y1.contiguous())
    assert torch.equal(l0, l1)
