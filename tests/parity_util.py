"""Helpers shared by the GPU parity tests: tolerances, runs through the C ABI, and
oracle references for selected heads."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_20172_gb300 import binding, workloads

# Tolerances (max-abs for fp32; max_elem|gpu - ref| / max_elem|ref| per tensor for bf16).
TOL = {
    ("fp32", "out"): 1e-4, ("fp32", "grad"): 1e-3,
    ("bf16", "out"): 2e-2, ("bf16", "grad"): 5e-2,
}


# Denominator floor of the bf16 normwise metric: some references are identically zero
# (e.g. dQ, dK at T = 1, where F_11 = 1 whatever Q and K are), and fp32 rounding then
# leaves residues of ~1e-8 that a pure ratio would blow up.
ZERO_REF_FLOOR = 1e-6


def err_metric(got, ref, dtype: str) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    diff = float(np.max(np.abs(got - ref))) if got.size else 0.0
    if dtype == "fp32":
        return diff
    scale = float(np.max(np.abs(ref))) if ref.size else 0.0
    return diff / max(scale, ZERO_REF_FLOOR)


def check(name: str, got, ref, dtype: str, kind: str):
    e = err_metric(got, ref, dtype)
    bound = TOL[(dtype, kind)]
    assert np.all(np.isfinite(np.asarray(got, dtype=np.float64))), f"{name}: non-finite values"
    assert e <= bound, f"{name}: error {e:.3e} > {bound:.1e} ({dtype}, {kind})"
    return e


def check_logz(name: str, got, ref, dtype: str):
    """logZ is fp32 on both paths; absolute bound 1e-4 (fp32 inputs) or 2e-2 (bf16)."""
    got = np.asarray(got, dtype=np.float64)
    e = float(np.max(np.abs(got - np.asarray(ref, dtype=np.float64)))) if got.size else 0.0
    bound = 1e-4 if dtype == "fp32" else 2e-2
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    assert e <= bound, f"{name}: abs error {e:.3e} > {bound:.1e}"
    return e


def check_dlambda(got: float, ref: float, dtype: str):
    bound = 1e-3 if dtype == "fp32" else 5e-2
    assert np.isfinite(got), "dlambda not finite"
    assert abs(got - ref) <= bound * max(abs(ref), 1.0 if dtype == "fp32" else 1e-3), \
        f"dlambda {got} vs {ref}"


def kernel_available(kernel: str, dtype: str, d: int, which: str = "fwd") -> bool:
    """True when the C ABI serves this kernel family for (dtype, d) (host-side query)."""
    return binding.launches_per_call(kernel, dtype, d, which) > 0


def kernel_combos(dtype: str, d: int):
    """(forward family, backward family) pairs to test: the CUDA-core pair always, and
    each tensor-core kernel the library offers for this (dtype, d)."""
    combos = [("simt", "simt")] if kernel_available("simt", dtype, d, "fwd") else []
    if kernel_available("tcgen05", dtype, d, "fwd") and combos:
        combos.append(("tcgen05", "simt"))
    if kernel_available("tcgen05", dtype, d, "bwd"):
        combos.append(("tcgen05", "tcgen05"))
    return combos


def gpu_run(q, k, v, do, lam, tau=workloads.TAU_S, kernel="auto", bwd=True, kernel_bwd=None):
    """Run forward (+ backward) through the C ABI on cuda:0; returns CPU tensors.
    ``kernel`` selects the forward family, ``kernel_bwd`` (default: same) the backward."""
    dev = torch.device("cuda:0")
    qd, kd, vd = (t.to(dev) for t in (q, k, v))
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    y, logz = binding.fwd(qd, kd, vd, lam, tau, kernel=kernel, dev_status=status)
    out = {"Y": y, "logZ": logz}
    if bwd:
        dod = do.to(dev)
        dq, dk, dv, dl = binding.bwd(qd, kd, vd, y, dod, logz, lam, tau,
                                     kernel=kernel_bwd or kernel, dev_status=status)
        out.update({"dQ": dq, "dK": dk, "dV": dv, "dlambda": dl})
    torch.cuda.synchronize()
    st = int(status.item())
    assert st == 0, f"device status {binding.status_string(st)}"
    res = {n: t.float().cpu() for n, t in out.items()}
    res["dlambda"] = float(res["dlambda"].item()) if bwd else None
    return res


def head(t: torch.Tensor, b: int, h: int) -> np.ndarray:
    """[T, d] fp64 numpy view of head (b, h) of a [B, T, H, d] tensor."""
    return t[b, :, h, :].double().numpy()


def oracle_heads(q, k, v, do, lam, heads, tau=workloads.TAU_S, bwd=True):
    """fp64 oracle forward (+ backward) for the listed (b, h) heads."""
    ref = {}
    for (b, h) in heads:
        qh, kh, vh = head(q, b, h), head(k, b, h), head(v, b, h)
        y, lz = oracle.fwd(qh, kh, vh, lam, tau)
        r = {"Y": y, "logZ": lz}
        if bwd:
            dq, dk, dv, dl = oracle.bwd(qh, kh, vh, head(do, b, h), lam, tau)
            r.update({"dQ": dq, "dK": dk, "dV": dv, "dlambda": dl})
        ref[(b, h)] = r
    return ref


def compare_heads(res, ref, dtype, bwd=True):
    errs = {}
    for (b, h), r in ref.items():
        errs[("Y", b, h)] = check(f"Y[{b},{h}]", res["Y"][b, :, h].numpy(), r["Y"], dtype, "out")
        errs[("logZ", b, h)] = check_logz(f"logZ[{b},{h}]", res["logZ"][b, h].numpy(),
                                          r["logZ"], dtype)
        if bwd:
            for n in ("dQ", "dK", "dV"):
                errs[(n, b, h)] = check(f"{n}[{b},{h}]", res[n][b, :, h].numpy(), r[n], dtype,
                                        "grad")
    return errs


# Achieved errors of the full-size checks, printed at the end of the run by conftest's
# terminal summary: (check, tensor) -> [normwise error, bound, elementwise relative error
# over the entries with |ref| >= 1e-2 max|ref| (information only)].
MARGINS = {}


def elem_rel_err(got, ref) -> float:
    """max |got - ref| / |ref| over the entries with |ref| >= 1e-2 max|ref|."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if not ref.size:
        return 0.0
    big = np.abs(ref) >= 1e-2 * float(np.max(np.abs(ref)))
    if not big.any():
        return 0.0
    return float(np.max(np.abs(got[big] - ref[big]) / np.abs(ref[big])))


def record(check_name: str, tensor: str, err: float, bound: float, elem: float):
    cur = MARGINS.get((check_name, tensor))
    if cur is None or err > cur[0]:
        MARGINS[(check_name, tensor)] = [err, bound, max(elem, cur[2] if cur else 0.0)]
    else:
        cur[2] = max(cur[2], elem)


def check_recorded(check_name: str, tensor: str, got, ref, dtype: str, kind: str):
    """check() plus a record of the achieved error for the end-of-run margin table."""
    e = check(f"{check_name} {tensor}", got, ref, dtype, kind)
    record(check_name, tensor, e, TOL[(dtype, kind)], elem_rel_err(got, ref))
    return e
