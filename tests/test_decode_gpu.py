"""GPU parity of relation_decode: one new token per sequence against a key/value cache.

The new token of sequence b is cache row len_b - 1, at one-based position len_b; its
output must equal that row of the full forward over the first len_b rows, which the
oracle computes row by row (fwd_rows).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20172_gb300 import binding, workloads
from tests import parity_util as pu

pytestmark = pytest.mark.gpu

LAM = workloads.LAMBDA_INIT


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    binding.load()


def _run(dtype, d, lengths, T, H=2, lam=LAM, seed=0):
    B = len(lengths)
    w = workloads.custom(B, H, T, d, dtype, qk_std=(1.0 / np.sqrt(d)) if dtype == "fp32" else 1.0)
    q, k, v, _ = workloads.make_inputs(w, seed=seed)
    dev = torch.device("cuda:0")
    lens = torch.tensor(lengths, dtype=torch.int32, device=dev)
    # the new token's query is row len_b - 1 of the query sequence
    qn = torch.stack([q[b, lengths[b] - 1] for b in range(B)]).to(dev)  # [B, H, d]
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y, lz = binding.decode(qn, k.to(dev), v.to(dev), lens, lam, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y, lz = y.float().cpu().numpy(), lz.cpu().numpy()
    for b in range(B):
        n = lengths[b]
        for h in range(H):
            yr, lr = oracle.fwd_rows(q[b, :n, h].double().numpy(), k[b, :n, h].double().numpy(),
                                     v[b, :n, h].double().numpy(), [n - 1], lam)
            pu.check(f"Y decode b{b} h{h} len {n}", y[b, h][None], yr, dtype, "out")
            pu.check_logz(f"logZ decode b{b} h{h} len {n}", lz[b, h][None], lr, dtype)


@pytest.mark.parametrize("dtype,d", [("fp32", 64), ("bf16", 64), ("bf16", 128), ("bf16", 48),
                                     ("fp32", 32)])
def test_decode_ragged_lengths(dtype, d):
    # one row (no history), within one chunk, a chunk boundary, several chunks
    _run(dtype, d, [1, 2, 300, 513, 1025, 1200], T=1200, seed=d)


@pytest.mark.parametrize("lam", [0.0, -1.0, 3.0])
def test_decode_lambda(lam):
    _run("bf16", 64, [7, 640], T=700, lam=lam, seed=3)


def test_decode_bad_length_reported():
    """A length outside [1, T] is reported through dev_status and no cache row is read."""
    dev = torch.device("cuda:0")
    k = torch.randn(2, 16, 1, 64, device=dev).to(torch.bfloat16)
    q = torch.randn(2, 1, 64, device=dev).to(torch.bfloat16)
    lens = torch.tensor([16, 17], dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    binding.decode(q, k, k, lens, LAM, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == binding.ERR_INVALID_ARG


def test_decode_at_the_benchmark_cache_size():
    """The benchmark's decode geometry (B = 32 sequences, H = 16, a T = 8192 cache, d_h = 128,
    2.1 GB of bf16 K and V): full-length sequences as the benchmark runs them and a few
    ragged ones, the new token's Y and logZ on sampled (b, h) against the oracle's row."""
    B, H, T, d = 32, 16, 8192, 128
    g = torch.Generator().manual_seed(11)
    kc = torch.randn((B, T, H, d), generator=g).to(torch.bfloat16)
    vc = torch.randn((B, T, H, d), generator=g).to(torch.bfloat16)
    qn = torch.randn((B, H, d), generator=g).to(torch.bfloat16)
    lengths = [T] * B
    lengths[1], lengths[2], lengths[3] = 1, 4097, T - 1
    dev = torch.device("cuda:0")
    lens = torch.tensor(lengths, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y, lz = binding.decode(qn.to(dev), kc.to(dev), vc.to(dev), lens, LAM, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    y, lz = y.float().cpu().numpy(), lz.cpu().numpy()
    for b in (0, 1, 2, 3, 31):
        n = lengths[b]
        for h in (0, 9, 15):
            qs = np.zeros((n, d))
            qs[n - 1] = qn[b, h].double().numpy()
            yr, lr = oracle.fwd_rows(qs, kc[b, :n, h].double().numpy(),
                                     vc[b, :n, h].double().numpy(), [n - 1], LAM)
            pu.check_recorded("decode 8192", "Y", y[b, h][None], yr, "bf16", "out")
            pu.check_logz(f"logZ decode b{b} h{h}", lz[b, h][None], lr, "bf16")
