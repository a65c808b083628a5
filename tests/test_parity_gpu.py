"""GPU parity: the CUDA path through the C ABI against the fp64 oracle.

Small shapes span several tiles and a ragged tail and are compared element by element
on every head.  The 10M, 30M and 100M workloads run at full size in the benchmark's launch
configuration and are compared on every head, element by element; the long sequence on
sampled rows plus two exact restrictions the causal structure allows.  The achieved errors
of the full-size checks are printed at the end of the run.
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




def _all_heads(w):
    return [(b, h) for b in range(w.B) for h in range(w.H)]


# --- fp32 -------------------------------------------------------------------

def test_tiny_fp32_all_heads():
    w = workloads.WORKLOADS["tiny"]
    q, k, v, do = workloads.make_inputs(w)
    res = pu.gpu_run(q, k, v, do, LAM)
    ref = pu.oracle_heads(q, k, v, do, LAM, _all_heads(w))
    pu.compare_heads(res, ref, "fp32")
    pu.check_dlambda(res["dlambda"], sum(r["dlambda"] for r in ref.values()), "fp32")


@pytest.mark.parametrize("T", [1, 2, 3, 65, 200])
@pytest.mark.parametrize("d", [32, 64, 128])
def test_fp32_shapes(T, d):
    w = workloads.custom(2, 1, T, d, "fp32", qk_std=1.0 / np.sqrt(d))
    q, k, v, do = workloads.make_inputs(w, seed=T + d)
    res = pu.gpu_run(q, k, v, do, LAM)
    ref = pu.oracle_heads(q, k, v, do, LAM, _all_heads(w))
    pu.compare_heads(res, ref, "fp32")
    pu.check_dlambda(res["dlambda"], sum(r["dlambda"] for r in ref.values()), "fp32")


# --- bf16, small shapes, every kernel family ----------------------------------

@pytest.mark.parametrize("T", [1, 2, 3, 127, 128, 129, 255, 300, 513])
@pytest.mark.parametrize("d", [64, 128])
def test_bf16_shapes(T, d):
    w = workloads.custom(1, 2, T, d, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=1000 + T + d)
    ref = pu.oracle_heads(q, k, v, do, LAM, _all_heads(w))
    for kf, kb in pu.kernel_combos("bf16", d):
        res = pu.gpu_run(q, k, v, do, LAM, kernel=kf, kernel_bwd=kb)
        pu.compare_heads(res, ref, "bf16")
        pu.check_dlambda(res["dlambda"], sum(r["dlambda"] for r in ref.values()), "bf16")


@pytest.mark.parametrize("lam", [0.0, -1.0, 3.0])
def test_bf16_lambda_values(lam):
    w = workloads.custom(2, 2, 333, 64, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=7)
    ref = pu.oracle_heads(q, k, v, do, lam, _all_heads(w))
    for kf, kb in pu.kernel_combos("bf16", 64):
        res = pu.gpu_run(q, k, v, do, lam, kernel=kf, kernel_bwd=kb)
        pu.compare_heads(res, ref, "bf16")
        pu.check_dlambda(res["dlambda"], sum(r["dlambda"] for r in ref.values()), "bf16")


def test_bf16_32():
    w = workloads.custom(1, 3, 150, 32, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=3)
    ref = pu.oracle_heads(q, k, v, do, LAM, _all_heads(w))
    for kf, kb in pu.kernel_combos("bf16", 32):
        res = pu.gpu_run(q, k, v, do, LAM, kernel=kf, kernel_bwd=kb)
        pu.compare_heads(res, ref, "bf16")


@pytest.mark.parametrize("T", [1, 129, 300])
@pytest.mark.parametrize("d", [16, 48, 80, 96])
def test_bf16_padded_head_sizes(T, d):
    """Head sizes other than 64 and 128 (the paper's layer geometry uses d_h = 48 and 80)
    run the tensor-core kernels on tiles zero-padded to 64 or 128 columns."""
    assert pu.kernel_available("tcgen05", "bf16", d, "fwd")
    assert pu.kernel_available("tcgen05", "bf16", d, "bwd")
    w = workloads.custom(1, 2, T, d, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=2000 + T + d)
    ref = pu.oracle_heads(q, k, v, do, LAM, _all_heads(w))
    res = pu.gpu_run(q, k, v, do, LAM, kernel="tcgen05")
    pu.compare_heads(res, ref, "bf16")
    pu.check_dlambda(res["dlambda"], sum(r["dlambda"] for r in ref.values()), "bf16")


def test_bhtd_layout():
    """[B, H, T, d] storage (a permuted view) gives the same result as [B, T, H, d]."""
    w = workloads.custom(2, 3, 200, 64, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=11)
    dev = torch.device("cuda:0")

    def bhtd(t):
        return t.permute(0, 2, 1, 3).contiguous().to(dev).permute(0, 2, 1, 3)

    qd, kd, vd, dod = (bhtd(t) for t in (q, k, v, do))
    y, lz = binding.fwd(qd, kd, vd, LAM)
    dq, dk, dv, dl = binding.bwd(qd, kd, vd, y, dod, lz, LAM)
    res = pu.gpu_run(q, k, v, do, LAM)
    for name, t in (("Y", y), ("dQ", dq), ("dK", dk), ("dV", dv)):
        assert torch.equal(t.float().cpu(), res[name]), name
    assert torch.equal(lz.cpu(), res["logZ"])


# --- full-size workloads in the benchmark's launch configuration --------------

@pytest.mark.parametrize("name", ["10M", "30M", "100M"])
def test_workload_full_size_all_heads(name):
    """The full workload in the benchmark's launch configuration, every head element by
    element against the fp64 oracle (OpenMP over heads), dlambda over all heads."""
    w = workloads.WORKLOADS[name]
    q, k, v, do = workloads.make_inputs(w)
    res = pu.gpu_run(q, k, v, do, LAM)
    q64, k64, v64, g64 = (t.double().numpy() for t in (q, k, v, do))
    ry, rlz = oracle.mhr_fwd(q64, k64, v64, LAM)
    rdq, rdk, rdv, dl_all = oracle.mhr_bwd(q64, k64, v64, g64, LAM)
    for n in ("Y", "dQ", "dK", "dV", "logZ"):
        assert torch.isfinite(res[n]).all(), n
    for b in range(w.B):
        for h in range(w.H):
            pu.check_recorded(name, "Y", res["Y"][b, :, h].numpy(), ry[b, :, h], "bf16", "out")
            for n, r in (("dQ", rdq), ("dK", rdk), ("dV", rdv)):
                pu.check_recorded(name, n, res[n][b, :, h].numpy(), r[b, :, h], "bf16", "grad")
    e = pu.check_logz(f"{name} logZ", res["logZ"].numpy(), rlz, "bf16")
    pu.record(name, "logZ(abs)", e, 2e-2, 0.0)
    pu.check_dlambda(res["dlambda"], dl_all, "bf16")
    pu.record(name, "dlambda(rel)", abs(res["dlambda"] - dl_all) / max(abs(dl_all), 1e-3), 5e-2,
              0.0)


def test_long_context_full_size():
    w = workloads.WORKLOADS["long"]
    q, k, v, do = workloads.make_inputs(w)
    T = w.T
    res = pu.gpu_run(q, k, v, do, LAM)
    for n in ("Y", "dQ", "dK", "dV", "logZ"):
        assert torch.isfinite(res[n]).all(), n
    # forward on every row of three heads: the first and the last, and one drawn with
    # seed 0 (numpy's default_rng(0).integers(0, B H) = 27: b = 1, h = 11)
    rows = list(range(T))
    pick = int(np.random.default_rng(0).integers(0, w.B * w.H))
    for (b, h) in [(0, 0), (w.B - 1, w.H - 1), divmod(pick, w.H)]:
        qh, kh, vh = pu.head(q, b, h), pu.head(k, b, h), pu.head(v, b, h)
        y, lz = oracle.fwd_rows(qh, kh, vh, rows, LAM)
        pu.check_recorded("long rows", "Y", res["Y"][b, :, h].numpy(), y, "bf16", "out")
        e = pu.check_logz(f"logZ rows [{b},{h}]", res["logZ"][b, h].numpy(), lz, "bf16")
        pu.record("long rows", "logZ(abs)", e, 2e-2, 0.0)
    # backward of one whole head (every row of dQ, dK, dV; the oracle's row-by-row
    # backward from row 0, about half a minute on the host cores)
    b, h = 1, 7
    dq, dk, dv, _ = oracle.bwd_tail(pu.head(q, b, h), pu.head(k, b, h), pu.head(v, b, h),
                                    pu.head(do, b, h), LAM, 0)
    pu.check_recorded("long head", "dQ", res["dQ"][b, :, h].numpy(), dq, "bf16", "grad")
    pu.check_recorded("long head", "dK", res["dK"][b, :, h].numpy(), dk, "bf16", "grad")
    pu.check_recorded("long head", "dV", res["dV"][b, :, h].numpy(), dv, "bf16", "grad")


@pytest.mark.parametrize("B,H,T,d", [(32, 8, 1024, 48), (4, 8, 4096, 80)])
def test_paper_layer_geometries_full_size(B, H, T, d):
    """The paper's layer geometries the benchmark times with head widths that run on
    zero-padded tiles (d_h = 48 on 64-wide, 80 on 128-wide), at full size: every row of two
    heads (forward) and one whole head's gradients, against the oracle."""
    w = workloads.custom(B, H, T, d, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=d)
    res = pu.gpu_run(q, k, v, do, LAM)
    rows = list(range(T))
    for (b, h) in [(0, 0), (B - 1, H - 1)]:
        y, lz = oracle.fwd_rows(pu.head(q, b, h), pu.head(k, b, h), pu.head(v, b, h), rows, LAM)
        pu.check_recorded(f"paper layer d={d}", "Y", res["Y"][b, :, h].numpy(), y, "bf16", "out")
        pu.check_logz(f"logZ [{b},{h}] d={d}", res["logZ"][b, h].numpy(), lz, "bf16")
    b, h = B // 2, H // 2
    dq, dk, dv, _ = oracle.bwd_tail(pu.head(q, b, h), pu.head(k, b, h), pu.head(v, b, h),
                                    pu.head(do, b, h), LAM, 0)
    pu.check_recorded(f"paper layer d={d}", "dQ", res["dQ"][b, :, h].numpy(), dq, "bf16", "grad")
    pu.check_recorded(f"paper layer d={d}", "dK", res["dK"][b, :, h].numpy(), dk, "bf16", "grad")
    pu.check_recorded(f"paper layer d={d}", "dV", res["dV"][b, :, h].numpy(), dv, "bf16", "grad")


def test_long_context_prefix_gradient():
    """dO = 0 on rows >= T' makes every gradient equal to that of the T'-prefix problem
    (rows i >= T' then carry dR_i. = 0): the full-size launch is checked exactly on the
    prefix, on sampled heads, including dlambda over all heads."""
    w = workloads.WORKLOADS["long"]
    q, k, v, do = workloads.make_inputs(w)
    Tp = 1024
    do = do.clone()
    do[:, Tp:] = 0
    res = pu.gpu_run(q, k, v, do, LAM)
    for (b, h) in [(0, 3), (1, 12)]:
        dq, dk, dv, _ = oracle.bwd(pu.head(q, b, h)[:Tp], pu.head(k, b, h)[:Tp],
                                   pu.head(v, b, h)[:Tp], pu.head(do, b, h)[:Tp], LAM)
        pu.check_recorded("long prefix", "dQ", res["dQ"][b, :Tp, h].numpy(), dq, "bf16", "grad")
        pu.check_recorded("long prefix", "dK", res["dK"][b, :Tp, h].numpy(), dk, "bf16", "grad")
        pu.check_recorded("long prefix", "dV", res["dV"][b, :Tp, h].numpy(), dv, "bf16", "grad")
    for n in ("dQ", "dK", "dV"):
        assert torch.count_nonzero(res[n][:, Tp:]) == 0, n
    _, _, _, dl_all = oracle.mhr_bwd(q[:, :Tp].double().numpy(), k[:, :Tp].double().numpy(),
                                     v[:, :Tp].double().numpy(), do[:, :Tp].double().numpy(), LAM)
    pu.check_dlambda(res["dlambda"], dl_all, "bf16")


# --- determinism, invariants, failure detection --------------------------------

def test_deterministic_repeat():
    w = workloads.custom(2, 2, 700, 64, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=5)
    a = pu.gpu_run(q, k, v, do, LAM)
    b = pu.gpu_run(q, k, v, do, LAM)
    for n in ("Y", "logZ", "dK", "dV"):
        assert torch.equal(a[n], b[n]), n
    pu.check("dQ repeat", a["dQ"].numpy(), b["dQ"].numpy(), "bf16", "grad")


@pytest.mark.parametrize("d,T", [(64, 700), (128, 333), (48, 257)])
def test_staged_backward_and_workspace_reuse(d, T):
    """The backward run stage by stage (row pass, tiles, finalisation) into outputs filled
    with NaN equals the one-call backward (every real element written), and a second call
    on the same workspace repeats dK, dV and dlambda bit for bit."""
    w = workloads.custom(2, 3, T, d, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=71 + d)
    dev = torch.device("cuda:0")
    qd, kd, vd, dod = (t.to(dev) for t in (q, k, v, do))
    y, lz = binding.fwd(qd, kd, vd, LAM, kernel="tcgen05")
    ws = torch.empty(binding.workspace_size(qd), device=dev, dtype=torch.uint8)
    one = [t.clone() for t in binding.bwd(qd, kd, vd, y, dod, lz, LAM, kernel="tcgen05",
                                          workspace=ws)]
    outs = [torch.full_like(qd, float("nan")) for _ in range(3)]
    dl = torch.full((1,), float("nan"), device=dev)
    for st in (binding.BWD_PREPARE, binding.BWD_TILES, binding.BWD_FINALIZE):
        binding.bwd(qd, kd, vd, y, dod, lz, LAM, kernel="tcgen05", workspace=ws, dq=outs[0],
                    dk=outs[1], dv=outs[2], dlambda=dl, stages=st)
    again = binding.bwd(qd, kd, vd, y, dod, lz, LAM, kernel="tcgen05", workspace=ws)
    torch.cuda.synchronize()
    for got in ((*outs, dl), again):
        assert torch.equal(got[1], one[1]) and torch.equal(got[2], one[2])
        assert torch.equal(got[3], one[3])
        assert not torch.isnan(got[0]).any()
        pu.check("dQ staged", got[0].float().cpu().numpy(), one[0].float().cpu().numpy(),
                 "bf16", "grad")


def test_large_lambda_keeps_self():
    """lambda >> 0 suppresses Exchange (-lambda log i): Y = V on rows i >= 2 up to bf16."""
    w = workloads.custom(1, 2, 300, 64, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=9)
    res = pu.gpu_run(q, k, v, do, 60.0, bwd=False)
    pu.check("Y ~ V", res["Y"].numpy(), v.float().numpy(), "bf16", "out")


def test_wait_timeout_reports_status():
    dev = torch.device("cuda:0")
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    assert binding.selftest_wait_timeout(st, 2000) == binding.OK
    torch.cuda.synchronize()
    assert int(st.item()) == binding.ERR_TIMEOUT
    # the context is still usable afterwards
    w = workloads.custom(1, 1, 64, 64, "bf16")
    q, k, v, do = workloads.make_inputs(w)
    res = pu.gpu_run(q, k, v, do, LAM)
    assert torch.isfinite(res["Y"]).all()


def test_device_argument_errors():
    dev = torch.device("cuda:0")
    x = torch.randn(1, 64, 2, 64, device=dev).to(torch.bfloat16)
    y, lz = binding.fwd(x, x, x, LAM)
    with pytest.raises(binding.RelationError) as e:
        binding.bwd(x, x, x, y, x, lz, LAM, workspace=torch.empty(16, dtype=torch.uint8, device=dev))
    assert e.value.code == binding.ERR_WORKSPACE
    buf = torch.empty(1 * 64 * 2 * 64 + 1, dtype=torch.bfloat16, device=dev)
    mis = buf[1:].view(1, 64, 2, 64)
    with pytest.raises(binding.RelationError) as e:
        binding.fwd(mis, mis, mis, LAM)
    assert e.value.code == binding.ERR_ALIGNMENT
    odd = torch.zeros(1, 8, 1, 136, dtype=torch.bfloat16, device=dev)
    with pytest.raises(binding.RelationError) as e:
        binding.fwd(odd, odd, odd, LAM)
    assert e.value.code == binding.ERR_UNSUPPORTED
    with pytest.raises(binding.RelationError) as e:
        binding.fwd(x, x, x, float("nan"))
    assert e.value.code == binding.ERR_INVALID_ARG


def test_autograd_wrapper_matches_binding():
    w = workloads.custom(1, 2, 130, 64, "bf16")
    q, k, v, do = workloads.make_inputs(w, seed=13)
    dev = torch.device("cuda:0")
    qd, kd, vd = (t.to(dev).requires_grad_(True) for t in (q, k, v))
    lam = torch.tensor(LAM, device=dev, requires_grad=True)
    y = binding.RelationFunction.apply(qd, kd, vd, lam)
    y.backward(do.to(dev))
    res = pu.gpu_run(q, k, v, do, LAM)
    assert torch.equal(y.detach().float().cpu(), res["Y"])
    assert torch.equal(kd.grad.float().cpu(), res["dK"])
    assert abs(float(lam.grad) - res["dlambda"]) <= 1e-6 * max(1.0, abs(res["dlambda"]))


# --- Self-flow side output ------------------------------------------------------

@pytest.mark.parametrize("dtype,d,T", [("fp32", 64, 200), ("bf16", 64, 300), ("bf16", 128, 257),
                                       ("bf16", 48, 130)])
def test_self_flow_side_output(dtype, d, T):
    """relation_fwd_flow returns F_ii = 1 - g_i per row (the Self share of the flow) next to
    the same Y and logZ as relation_fwd, for every kernel family that serves the shape."""
    w = workloads.custom(2, 2, T, d, dtype, qk_std=(1.0 / np.sqrt(d)) if dtype == "fp32" else 1.0)
    q, k, v, _ = workloads.make_inputs(w, seed=5000 + T + d)
    dev = torch.device("cuda:0")
    qd, kd, vd = (t.to(dev) for t in (q, k, v))
    tol = 1e-5 if dtype == "fp32" else 2e-3
    fams = [f for f in ("simt", "tcgen05") if pu.kernel_available(f, dtype, d, "fwd")]
    assert fams
    for fam in fams:
        y0, lz0 = binding.fwd(qd, kd, vd, LAM, kernel=fam)
        y, lz, fs = binding.fwd_flow(qd, kd, vd, LAM, kernel=fam)
        torch.cuda.synchronize()
        assert torch.equal(y, y0) and torch.equal(lz, lz0), fam
        fs = fs.cpu().numpy()
        for b in range(w.B):
            for h in range(w.H):
                ref = oracle.fwd_factorized(q[b, :, h].double().numpy(), k[b, :, h].double().numpy(),
                                            v[b, :, h].double().numpy(), LAM)
                err = np.abs(fs[b, h] - ref["Fii"]).max()
                assert err <= tol, f"{fam} head ({b},{h}): max |F_ii - ref| = {err:.3g} > {tol}"
                assert fs[b, h, 0] == 1.0


# --- the persistent backward: many (key tile, head) units per CTA ---------------

@pytest.mark.parametrize("B,H,T,d", [(4, 80, 300, 64), (2, 100, 200, 48), (1, 400, 129, 64)])
def test_persistent_backward_many_units(B, H, T, d):
    """More units than SMs, of mixed sizes (ragged last key tile): every CTA walks several
    units, so the cross-unit K/V double buffer, the staging reuse and the zigzag order
    are all exercised.  Sampled heads against the oracle element by element, every head
    against the CUDA-core backward (an independent GPU implementation), and dlambda
    over all heads against the oracle."""
    w = workloads.custom(B, H, T, d, "bf16")
    q, k, v, do = workloads.make_inputs(w)
    res = pu.gpu_run(q, k, v, do, LAM)
    heads = [(0, 0), (B - 1, H - 1), (B // 2, H // 2), (0, H - 1), (B - 1, 1)]
    ref = pu.oracle_heads(q, k, v, do, LAM, heads)
    pu.compare_heads(res, ref, "bf16")
    if pu.kernel_available("simt", "bf16", d, "bwd"):
        alt = pu.gpu_run(q, k, v, do, LAM, kernel_bwd="simt")
        for n in ("dQ", "dK", "dV"):
            for b in range(B):
                for h in range(H):
                    e = pu.err_metric(res[n][b, :, h].numpy(), alt[n][b, :, h].numpy(), "bf16")
                    assert e <= 2 * pu.TOL[("bf16", "grad")], f"{n}[{b},{h}] vs CUDA-core: {e:.3e}"
    _, _, _, dl_all = oracle.mhr_bwd(q.double().numpy(), k.double().numpy(), v.double().numpy(),
                                     do.double().numpy(), LAM)
    pu.check_dlambda(res["dlambda"], dl_all, "bf16")


@pytest.mark.parametrize("d", [64, 128])
def test_forward_maximum_growing_through_the_sequence(d):
    """Keys scaled up along the sequence (by 1 + 6 j / T), so the rows' maximum grows by
    more than 2^8 many times after their first step: the scale is raised a step late,
    after the z update in flight has landed.  Every row of every head against the oracle
    (a rescale racing the update shows up as a few rows with z off by a large factor)."""
    T = 2048
    w = workloads.custom(1, 2, T, d, "bf16")
    q, k, v, _ = workloads.make_inputs(w, seed=31 + d)
    ramp = (1.0 + 6.0 * torch.arange(T, dtype=torch.float32) / T)[None, :, None, None]
    k = (k.float() * ramp).to(torch.bfloat16)
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    res = pu.gpu_run(q, k, v, None, lam, tau, kernel="tcgen05", bwd=False)
    ref = pu.oracle_heads(q, k, v, None, lam, [(0, 0), (0, 1)], tau, bwd=False)
    for (b, h), r in ref.items():
        pu.check_recorded("growing maximum", f"Y d={d}", res["Y"][b, :, h].numpy(), r["Y"],
                          "bf16", "out")
        pu.check_logz(f"logZ[{b},{h}]", res["logZ"][b, h].numpy(), r["logZ"], "bf16")
        # a wrong z shows up as rows far off even when the normwise error stays small
        assert np.max(np.abs(res["Y"][b, :, h].numpy() - r["Y"])) < 0.25
