"""relation_bwd_static: the backward for callers that cannot allocate device memory.

It must give the same gradients as relation_bwd with a caller workspace, on two calls in a
row (the library's scratch array keeps the previous call's contents, which must not leak
into the next result).  Runs last so that a failure here does not hide other results.
"""
import pytest
import torch

from paper_2608_20172_gb300 import binding, workloads
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    binding.load()


@pytest.mark.parametrize("shape,dtype", [((2, 3, 300, 64), "bf16"), ((1, 2, 257, 128), "bf16"),
                                         ((1, 2, 128, 32), "fp32")])
def test_no_alloc_backward_matches_workspace_backward(shape, dtype):
    B, H, T, d = shape
    w = workloads.custom(B, H, T, d, dtype, qk_std=1.0 if dtype == "bf16" else d ** -0.5)
    dev = torch.device("cuda:0")
    outs = []
    for seed in (21, 22):  # two calls in a row on different inputs
        q, k, v, do = (t.to(dev) for t in workloads.make_inputs(w, seed=seed))
        y, logz = binding.fwd(q, k, v, workloads.LAMBDA_INIT)
        ref = binding.bwd(q, k, v, y, do, logz, workloads.LAMBDA_INIT)
        dq, dk, dv = torch.empty_like(q), torch.empty_like(q), torch.empty_like(q)
        dl = torch.empty(1, device=dev, dtype=torch.float32)
        status = torch.zeros(1, dtype=torch.int32, device=dev)
        binding.bwd_no_alloc(q, k, v, y, do, logz, workloads.LAMBDA_INIT, dq=dq, dk=dk, dv=dv,
                             dlambda=dl, dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        for name, got, want in (("dQ", dq, ref[0]), ("dK", dk, ref[1]), ("dV", dv, ref[2])):
            pu.check(f"{name} no-alloc vs workspace", got.float().cpu().numpy(),
                     want.float().cpu().numpy(), dtype, "grad")
        pu.check_dlambda(float(dl.item()), float(ref[3].item()), dtype)
        outs.append(dq.float().cpu())
    assert not torch.equal(outs[0], outs[1])  # the second call really recomputed


def test_no_alloc_rejects_oversized_shapes():
    # needs more scratch than the fixed array holds: rejected before any launch
    w = workloads.WORKLOADS["long"]
    x = torch.empty((w.B, w.T, w.H, w.d), dtype=torch.bfloat16, device="cuda:0")
    lz = torch.empty((w.B, w.H, w.T), dtype=torch.float32, device="cuda:0")
    dl = torch.empty(1, dtype=torch.float32, device="cuda:0")
    assert binding.workspace_size(x) > binding.STATIC_SCRATCH_BYTES
    with pytest.raises(binding.RelationError) as e:
        binding.bwd_no_alloc(x, x, x, x, x, lz, 0.5, dq=x, dk=x, dv=x, dlambda=dl)
    assert e.value.code == binding.ERR_WORKSPACE


def test_no_alloc_rejects_operands_off_the_current_device():
    """The array used is the current device's copy, so operands elsewhere (here q in pinned
    host memory, as a stand-in for another GPU's memory on a one-GPU machine) are rejected
    before any launch, and the outputs are left untouched."""
    import ctypes
    w = workloads.custom(1, 2, 200, 64, "bf16")
    dev = torch.device("cuda:0")
    q, k, v, do = workloads.make_inputs(w, seed=31)
    kd, vd, dod = (t.to(dev) for t in (k, v, do))
    y, logz = binding.fwd(q.to(dev), kd, vd, workloads.LAMBDA_INIT)
    q_host = q.pin_memory()
    dq = torch.full_like(kd, 7.0)
    dk, dv = torch.empty_like(kd), torch.empty_like(kd)
    dl = torch.empty(1, device=dev, dtype=torch.float32)
    lib = binding.load()
    ptr = lambda t: ctypes.c_void_p(t.data_ptr())
    rc = lib.relation_bwd_static(ptr(q_host), ptr(kd), ptr(vd), ptr(y), ptr(dod), ptr(logz),
                                 ptr(dq), ptr(dk), ptr(dv), ptr(dl),
                                 float(workloads.LAMBDA_INIT), 2.0, binding.shape_of(kd),
                                 binding.BF16, binding.KERNELS["auto"], None,
                                 ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    torch.cuda.synchronize()
    assert rc == binding.ERR_INVALID_ARG
    assert torch.all(dq == 7.0)
