"""GPU parity of Linear Relation (Sec. 5.2, App. A.4) against the fp64 oracle, every head
element by element, at sizes that span several staged chunks and a ragged tail."""
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


def _heads(x, b, h):
    return x[b, :, h].double().numpy()


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("d", [32, 64, 128])
@pytest.mark.parametrize("T", [1, 17, 200])
def test_linear_forward(dtype, d, T):
    w = workloads.custom(2, 2, T, d, dtype)
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=T + d)
    dev = torch.device("cuda:0")
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y = binding.linear_fwd(p1.to(dev), p2.to(dev), v.to(dev), alpha.to(dev), dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y = y.float().cpu().numpy()
    for b in range(w.B):
        for h in range(w.H):
            ref, _ = oracle.linear_fwd(_heads(p1, b, h), _heads(p2, b, h), _heads(v, b, h),
                                       _heads(alpha, b, h))
            pu.check(f"linear Y ({b},{h})", y[b, :, h], ref, dtype, "out")


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("d", [32, 64, 128])
@pytest.mark.parametrize("T", [1, 8, 9, 100])
def test_linear_backward(dtype, d, T):
    """Gradients of every input, including the retention, against the oracle's reverse-
    mode backward on every head (T spans whole 8-token chunks and ragged tails)."""
    w = workloads.custom(2, 2, T, d, dtype)
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=100 + T + d)
    dev = torch.device("cuda:0")
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    g = binding.linear_bwd(*(t.to(dev) for t in (p1, p2, v, alpha, dy)), kernel="simt",
                           dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    g = [t.float().cpu().numpy() for t in g]
    for b in range(w.B):
        for h in range(w.H):
            ref = oracle.linear_bwd(_heads(p1, b, h), _heads(p2, b, h), _heads(v, b, h),
                                    _heads(alpha, b, h), _heads(dy, b, h))
            for name, got, r in zip(("dp1", "dp2", "dv", "dalpha"), g, ref):
                pu.check(f"linear {name} ({b},{h}) T={T}", got[b, :, h], r,
                         "fp32" if name == "dalpha" and dtype == "fp32" else dtype, "grad")


def test_linear_bhtd_layout():
    """[B, H, T, d] storage (a permuted view) gives the same output as [B, T, H, d]."""
    w = workloads.custom(2, 3, 70, 64, "bf16")
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=1)
    dev = torch.device("cuda:0")

    def bhtd(t):
        return t.permute(0, 2, 1, 3).contiguous().to(dev).permute(0, 2, 1, 3)

    y0 = binding.linear_fwd(*(t.to(dev) for t in (p1, p2, v, alpha)))
    y1 = binding.linear_fwd(*(bhtd(t) for t in (p1, p2, v, alpha)))
    assert torch.equal(y0.cpu(), y1.cpu())


# --- the chunked tensor-core forward ------------------------------------------

@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("T", [1, 2, 127, 128, 129, 300, 513])
def test_linear_forward_chunked_every_head(d, T):
    """The chunked tcgen05 forward (blocks of 128 tokens: T spans whole blocks, ragged
    tails and a single token) against the fp64 recurrence on every head."""
    w = workloads.custom(2, 3, T, d, "bf16")
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=500 + T + d)
    dev = torch.device("cuda:0")
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y = binding.linear_fwd(p1.to(dev), p2.to(dev), v.to(dev), alpha.to(dev), kernel="tcgen05",
                           dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y = y.float().cpu().numpy()
    for b in range(w.B):
        for h in range(w.H):
            ref, _ = oracle.linear_fwd(_heads(p1, b, h), _heads(p2, b, h), _heads(v, b, h),
                                       _heads(alpha, b, h))
            pu.check(f"chunked linear Y ({b},{h}) T={T}", y[b, :, h], ref, "bf16", "out")


@pytest.mark.parametrize("d", [64, 128])
def test_linear_forward_chunked_long_sequence(d):
    """A long sequence (64 blocks of 128 tokens: the state carried through them) on every
    head, and the chunked and recurrent kernels against each other."""
    w = workloads.custom(1, 2, 8192, d, "bf16")
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=77 + d)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha)]
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y_tc = binding.linear_fwd(*args, kernel="tcgen05", dev_status=status)
    y_rec = binding.linear_fwd(*args, kernel="simt", dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y_tc, y_rec = y_tc.float().cpu().numpy(), y_rec.float().cpu().numpy()
    for h in range(w.H):
        ref, _ = oracle.linear_fwd(_heads(p1, 0, h), _heads(p2, 0, h), _heads(v, 0, h),
                                   _heads(alpha, 0, h))
        e = pu.check_recorded("linear 8192", f"Y d={d}", y_tc[0, :, h], ref, "bf16", "out")
        pu.check(f"recurrent linear Y h={h}", y_rec[0, :, h], ref, "bf16", "out")


def test_linear_chunked_reports_decay_beyond_its_range():
    """Retention so small that a 64-token product falls below 2^-120: the chunked kernel
    clamps its ratio factors and says so through dev_status (the output stays finite); the
    recurrent kernel has no such limit."""
    w = workloads.custom(1, 2, 256, 64, "bf16")
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=3)
    alpha = torch.full_like(alpha, 1e-3)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha)]
    st_tc = torch.zeros(1, dtype=torch.int32, device=dev)
    st_rec = torch.zeros(1, dtype=torch.int32, device=dev)
    y = binding.linear_fwd(*args, kernel="tcgen05", dev_status=st_tc)
    binding.linear_fwd(*args, kernel="simt", dev_status=st_rec)
    torch.cuda.synchronize()
    assert int(st_tc.item()) == binding.ERR_UNSUPPORTED
    assert int(st_rec.item()) == 0
    assert torch.isfinite(y.float()).all()


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("T", [1, 129, 1000, 4097])
def test_linear_forward_chunk_parallel(d, T):
    """The chunk-parallel form (few heads: every block's state contribution, the scan over
    blocks, every block's output in parallel) against the fp64 recurrence on every head, and
    against the sequential chunked kernel."""
    w = workloads.custom(1, 2, T, d, "bf16")
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=900 + T + d)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha)]
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    assert binding.linear_fwd_workspace_size(args[0]) > 0
    y = binding.linear_fwd_ws(*args, dev_status=status)
    y_seq = binding.linear_fwd(*args, kernel="tcgen05", dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y, y_seq = y.float().cpu().numpy(), y_seq.float().cpu().numpy()
    for h in range(w.H):
        ref, _ = oracle.linear_fwd(_heads(p1, 0, h), _heads(p2, 0, h), _heads(v, 0, h),
                                   _heads(alpha, 0, h))
        pu.check_recorded("linear chunk-parallel", f"Y d={d}", y[0, :, h], ref, "bf16", "out")
        pu.check(f"chunk-parallel vs sequential h={h}", y[0, :, h], y_seq[0, :, h], "bf16", "out")


def test_linear_forward_ws_many_heads_uses_the_sequential_walk():
    """With at least half as many (head, column) pairs as SMs the workspace entry point takes
    the sequential chunked kernel: its output equals relation_linear_fwd_ex(TCGEN05) bit for
    bit."""
    w = workloads.custom(4, 40, 300, 64, "bf16")
    p1, p2, v, alpha, _ = workloads.make_linear_inputs(w, seed=4)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha)]
    y = binding.linear_fwd_ws(*args)
    y_seq = binding.linear_fwd(*args, kernel="tcgen05")
    torch.cuda.synchronize()
    assert torch.equal(y, y_seq)


# --- the chunked tensor-core backward -----------------------------------------

def _check_grads(tag, g, p1, p2, v, alpha, dy, heads):
    g = [t.float().cpu().numpy() for t in g]
    for b, h in heads:
        ref = oracle.linear_bwd(_heads(p1, b, h), _heads(p2, b, h), _heads(v, b, h),
                                _heads(alpha, b, h), _heads(dy, b, h))
        for name, got, r in zip(("dp1", "dp2", "dv", "dalpha"), g, ref):
            pu.check_recorded(tag, name, got[b, :, h], r, "bf16", "grad")


@pytest.mark.parametrize("T", [1, 2, 64, 127, 128, 129, 300, 513])
def test_linear_backward_chunked_every_head(T):
    """The chunked tcgen05 backward (the states entering and the adjoints leaving every
    128-token block, then every block's gradients in parallel) against the fp64 reverse
    mode of the recurrence on every head: whole blocks, ragged tails, a single token."""
    w = workloads.custom(2, 3, T, 64, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=700 + T)
    dev = torch.device("cuda:0")
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    g = binding.linear_bwd(*(t.to(dev) for t in (p1, p2, v, alpha, dy)), kernel="tcgen05",
                           dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _check_grads("linear chunked bwd", g, p1, p2, v, alpha, dy,
                 [(b, h) for b in range(w.B) for h in range(w.H)])


def test_linear_backward_chunked_long_sequence():
    """32 blocks of 128 tokens (the states and adjoints carried through all of them) on every
    head, against the oracle and against the recurrent backward."""
    w = workloads.custom(1, 2, 4096, 64, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=91)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha, dy)]
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    g_tc = binding.linear_bwd(*args, kernel="tcgen05", dev_status=status)
    g_rec = binding.linear_bwd(*args, kernel="simt", dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _check_grads("linear chunked bwd 4096", g_tc, p1, p2, v, alpha, dy, [(0, 0), (0, 1)])
    for name, a, r in zip(("dp1", "dp2", "dv", "dalpha"), g_tc, g_rec):
        pu.check(f"chunked vs recurrent {name}", a.float().cpu().numpy(),
                 r.float().cpu().numpy(), "bf16", "grad")


def test_linear_backward_auto_takes_the_chunked_kernel():
    """AUTO serves bf16 at d_h = 64 with the chunked kernel: bit-identical results to
    TCGEN05, in a workspace of the chunked family's size."""
    w = workloads.custom(2, 4, 300, 64, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=5)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha, dy)]
    assert binding.linear_bwd_workspace_size(args[0]) == \
        binding.linear_bwd_workspace_size(args[0], "tcgen05") > 0
    g_auto = binding.linear_bwd(*args)
    g_tc = binding.linear_bwd(*args, kernel="tcgen05")
    torch.cuda.synchronize()
    for a, b in zip(g_auto, g_tc):
        assert torch.equal(a, b)


def test_linear_backward_chunked_reports_decay_beyond_its_range():
    """Retention whose 64-token product falls below 2^-120: the chunked backward clamps like
    the chunked forward, reports RELATION_ERR_UNSUPPORTED and keeps every output finite."""
    w = workloads.custom(1, 2, 256, 64, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=3)
    alpha = torch.full_like(alpha, 1e-3)
    dev = torch.device("cuda:0")
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    g = binding.linear_bwd(*(t.to(dev) for t in (p1, p2, v, alpha, dy)), kernel="tcgen05",
                           dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == binding.ERR_UNSUPPORTED
    for t in g:
        assert torch.isfinite(t.float()).all()


def test_linear_backward_chunked_bhtd_layout_and_stride_fallback():
    """The chunked backward on [B, H, T, d] storage (a permuted view) gives the results of
    the [B, T, H, d] layout bit for bit; a row stride that is a multiple of 4 but not of 8
    elements leaves the chunked kernel's reach, and AUTO then runs the recurrence (still
    against the oracle)."""
    w = workloads.custom(2, 3, 200, 64, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=12)
    dev = torch.device("cuda:0")

    def bhtd(t):
        return t.permute(0, 2, 1, 3).contiguous().to(dev).permute(0, 2, 1, 3)

    g0 = binding.linear_bwd(*(t.to(dev) for t in (p1, p2, v, alpha, dy)), kernel="tcgen05")
    g1 = binding.linear_bwd(*(bhtd(t) for t in (p1, p2, v, alpha, dy)), kernel="tcgen05")
    torch.cuda.synchronize()
    for a, b in zip(g0, g1):
        assert torch.equal(a.contiguous(), b.contiguous())

    def padded(t):  # d padded to 68: element strides (T H 68, H 68, 68), multiples of 4 only
        pad = torch.zeros(t.shape[:-1] + (68,), dtype=t.dtype)
        pad[..., :64] = t
        return pad.to(dev)[..., :64]

    args = [padded(t) for t in (p1, p2, v, alpha, dy)]
    assert binding.linear_bwd_workspace_size(args[0], "tcgen05") == 0
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    g = binding.linear_bwd(*args, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    _check_grads("linear bwd strided", g, p1, p2, v, alpha, dy, [(0, 0), (1, 2)])


def test_linear_chunked_at_the_longest_sweep_point():
    """The long-context sweep's last point as the benchmark runs it (B = 1, H = 12,
    T = 32768, d_h = 64, 256 blocks of 128 tokens): the chunk-parallel forward (workspace
    entry point), the sequential chunked forward and the chunked backward, each against the
    fp64 oracle on three heads over the whole sequence."""
    w = workloads.custom(1, 12, 32768, 64, "bf16")
    p1, p2, v, alpha, dy = workloads.make_linear_inputs(w, seed=1)
    dev = torch.device("cuda:0")
    args = [t.to(dev) for t in (p1, p2, v, alpha)]
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y_ws = binding.linear_fwd_ws(*args, dev_status=status)
    y_seq = binding.linear_fwd(*args, kernel="tcgen05", dev_status=status)
    g = binding.linear_bwd(*args, dy.to(dev), kernel="tcgen05", dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y_ws, y_seq = y_ws.float().cpu().numpy(), y_seq.float().cpu().numpy()
    heads = [(0, 0), (0, 5), (0, 11)]
    for b, h in heads:
        ref, _ = oracle.linear_fwd(_heads(p1, b, h), _heads(p2, b, h), _heads(v, b, h),
                                   _heads(alpha, b, h))
        pu.check_recorded("linear 32768", "Y chunk-parallel", y_ws[b, :, h], ref, "bf16", "out")
        pu.check_recorded("linear 32768", "Y sequential", y_seq[b, :, h], ref, "bf16", "out")
    _check_grads("linear 32768 bwd", g, p1, p2, v, alpha, dy, heads)
