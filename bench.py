"""Benchmark: FlashRelation forward + backward on one GB300 (replicas on N GPUs).

One step = relation_fwd + relation_bwd over one batch of the workload (every step of
the operator's hot path), inputs resident in HBM.  Timed with CUDA events on the
launching stream, per step, with the L2 flushed (a 256 MiB write) between steps, after
W warm-up steps.  Prints ONE JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config long|100M|30M|10M|tiny]
                  [--also 100M,...|none] [--impl ours|reference] [--no-cpu-baseline]
                  [--no-side]

The headline line is the long-context workload (B=2, H=16, T=16384, d_h=128); the
~100M-scale layer (B=8, H=12, T=2048, d_h=64) is measured in the same run as a
sub-record (``sub_records``) with its own step time, roofline and tokens/s.  --no-side
skips the side measurements (decode, Linear Relation, layer transforms, SDPA context),
e.g. under a profiler.

--impl reference times the fp64 CPU oracle (the reference arm of this operator: there
is no other implementation) on the host cores over a bounded sample of the workload.
Under torchrun (N > 1) every rank runs an independent replica of the workload on its
own GPU (the heads are independent; nothing is exchanged) and the slowest rank's time
is reported.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2608_20172_gb300 import workloads  # noqa: E402

L2_FLUSH_BYTES = 256 << 20


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu=timestamp,{self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [ln for ln in out.splitlines() if ln.strip()]
        return False

    def summary(self, t_begin=None, t_end=None):
        """Median SM clock and active throttle reasons over the samples taken between the
        host times t_begin and t_end (all samples when no window is given)."""
        import datetime
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in getattr(self, "lines", []):
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 10:
                continue
            if t_begin is not None:
                try:
                    ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                except ValueError:
                    ts = None
                if ts is not None and not (t_begin - 0.06 <= ts <= t_end + 0.06):
                    continue
            f = f[1:]
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def _profiled_traffic(w, kernel):
    """DRAM bytes per launch of `kernel` on workload `w`, from the committed ncu record of
    that kernel instantiation on that workload (profiles/<kernel>_<workload>_traffic.json),
    or None when there is none or the kernel source changed since it was taken."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"{kernel}_{w.name}_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        src = os.path.join(ROOT, rec["source"])
        with open(src, "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != rec["source_sha256"]:
                return None
        if [rec.get(k) for k in ("B", "H", "T", "d_h")] != [w.B, w.H, w.T, w.d]:
            return None
        return float(rec["dram_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
        return dist, ws, rank, local
    return None, 1, 0, local


def _barrier(dist, dev):
    if dist is not None:
        dist.barrier(device_ids=[dev.index] if dev.type == "cuda" else None)


def _max_over_ranks(dist, x: float, dev) -> float:
    if dist is None:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------------------
# CPU oracle (baseline leg and --impl reference)
# ------------------------------------------------------------------------------

ORACLE_BUDGET = 128 * 1024 * 1024 * 64  # heads x T^2 x d of one sample (~1 s on 16 cores)


def _sample_plan(w, budget=ORACLE_BUDGET):
    """A bounded sample of the workload for the fp64 oracle: (heads, T') with the first
    `heads` (b, h) heads over their first T' rows.  The first T' rows of a causal head are
    exactly the T'-row problem, so the sample is a smaller instance of the same
    workload.  Whole sequences (T' = T) while at least one head fits the budget, whole
    batches of heads where possible; long sequences take every head over a prefix."""
    per_head = w.T * w.T * w.d
    if per_head <= budget:
        n = max(1, min(w.B * w.H, budget // per_head))
        return (n if n < w.H else (n // w.H) * w.H), w.T
    heads = w.B * w.H
    t = w.T
    while t > 128 and heads * t * t * w.d > budget:
        t //= 2
    return heads, t


_SAMPLE_CACHE = {}


def _oracle_sample(w, n_heads, t_rows):
    """Inputs of the first n_heads (b, h) heads over rows [0, t_rows), fp64 [B', T', H', d]
    (drawn once per sample shape)."""
    key = (w, n_heads, t_rows)
    if key not in _SAMPLE_CACHE:
        _SAMPLE_CACHE.clear()
        _SAMPLE_CACHE[key] = _draw_sample(w, n_heads, t_rows)
    return _SAMPLE_CACHE[key]


def _draw_sample(w, n_heads, t_rows):
    q, k, v, do = workloads.make_inputs(w)
    heads = [(b, h) for b in range(w.B) for h in range(w.H)][:n_heads]
    bs = sorted({b for b, _ in heads})
    hs = sorted({h for _, h in heads})
    sl = (slice(bs[0], bs[-1] + 1), slice(0, t_rows), slice(hs[0], hs[-1] + 1))
    return [t[sl].double().numpy() for t in (q, k, v, do)], len(bs) * len(hs)


def cpu_oracle_run(w, n_heads=None, t_rows=None, min_seconds=0.0, max_reps=20, nthreads=0):
    """Time the fp64 oracle (forward + backward) on a sample of the workload (the first
    n_heads heads over their first t_rows rows), repeating the sample until min_seconds
    of CPU work have run; nthreads = 0: every OpenMP thread."""
    import oracle
    plan_heads, plan_rows = _sample_plan(w)
    n_heads = n_heads or plan_heads
    t_rows = t_rows or plan_rows
    (q, k, v, do), used = _oracle_sample(w, n_heads, t_rows)
    threads = nthreads or oracle.max_threads()
    reps, dt = 0, 0.0
    while reps < max_reps and (reps == 0 or dt < min_seconds):
        t0 = time.perf_counter()
        oracle.mhr_fwd(q, k, v, workloads.LAMBDA_INIT, nthreads=nthreads)
        oracle.mhr_bwd(q, k, v, do, workloads.LAMBDA_INIT, nthreads=nthreads)
        dt += time.perf_counter() - t0
        reps += 1
    flops = 7.0 * used * t_rows * t_rows * w.d * reps
    return {"seconds": dt, "heads": used, "rows": t_rows, "reps": reps, "flops": flops,
            "tflops": flops / dt / 1e12, "tokens_per_s": reps * (used / w.H) * t_rows / dt,
            "cores": threads}


def _sample_text(w, res):
    rows = "" if res["rows"] == w.T else f" over their first {res['rows']} of {w.T} rows"
    return f"{res['heads']} of {w.B * w.H} heads{rows}"


def run_reference(args, w):
    dist, ws, rank, local = _dist()
    if rank != 0:
        return 0
    n, rows = _sample_plan(w, ORACLE_BUDGET // 4)
    for _ in range(args.warmup):
        cpu_oracle_run(w, n_heads=n, t_rows=rows)
    times, res = [], None
    for _ in range(args.steps):
        res = cpu_oracle_run(w, n_heads=n, t_rows=rows)
        times.append(res["seconds"])
    tot_flops = res["flops"] * args.steps
    val = tot_flops / sum(times) / 1e12
    sample = f"{_sample_text(w, res)} per step (fwd+bwd, fp64, OpenMP over heads)"
    line = {
        "impl": "reference", "metric": "FlashRelation fwd+bwd TFLOP/s (7*B*H*T^2*d causal)",
        "value": val, "unit": "TFLOP/s", "n_gpus": 0, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * statistics.mean(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.description, "B": w.B, "H": w.H, "T": w.T, "d_h": w.d,
                   "lambda": workloads.LAMBDA_INIT, "tau_s": workloads.TAU_S},
        "cpu_baseline": {"value": val, "unit": "TFLOP/s", "cores": res["cores"], "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------
# GPU arm
# ------------------------------------------------------------------------------

DECODE_CFG = {"B": 32, "H": 16, "T": 8192, "d_h": 128}  # bf16 cache of 2.1 GB (K + V)


def decode_measure(binding, dev, peaks, steps=20, warmup=3):
    """relation_decode on a bf16 cache larger than L2 (every sequence at full length):
    algorithmic bytes = the K and V rows read + q, Y, logZ; HBM roofline."""
    c = DECODE_CFG
    B, H, T, d = c["B"], c["H"], c["T"], c["d_h"]
    g = torch.Generator(device="cpu").manual_seed(0)
    kc = torch.randn((B, T, H, d), generator=g).to(torch.bfloat16).to(dev)
    vc = torch.randn((B, T, H, d), generator=g).to(torch.bfloat16).to(dev)
    qn = torch.randn((B, H, d), generator=g).to(torch.bfloat16).to(dev)
    lens = torch.full((B,), T, dtype=torch.int32, device=dev)
    out = torch.empty_like(qn)
    logz = torch.empty((B, H), dtype=torch.float32, device=dev)
    wsb = torch.empty(binding.decode_workspace_size(kc), dtype=torch.uint8, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    call = lambda: binding.decode(qn, kc, vc, lens, workloads.LAMBDA_INIT, out=out, logz=logz,
                                  workspace=wsb, dev_status=status, stream=stream)
    for _ in range(warmup):
        call()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    torch.cuda.synchronize(dev)
    ev[0].record(stream)
    for i in range(steps):
        call()
        ev[i + 1].record(stream)
    torch.cuda.synchronize(dev)
    if int(status.item()) != 0:
        raise SystemExit(f"decode device status {binding.status_string(int(status.item()))}")
    ms = statistics.mean(ev[i].elapsed_time(ev[i + 1]) for i in range(steps))
    nbytes = 2.0 * B * T * H * d * 2 + 2.0 * B * H * d * 2 + B * H * 4
    gbs = nbytes / (ms * 1e-3) / 1e9
    return {"config": {**c, "dtype": "bf16", "lengths": "all T",
                       "l2": "cache 2.1 GB > L2, no flush"},
            "ms_per_call": ms, "tokens_per_s": B / (ms * 1e-3),
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"],
                         "unit": "GB/s", "frac": gbs / peaks["hbm_gbs"],
                         "algorithmic_bytes_per_call": nbytes},
            "gpu_launches_per_call": 2}


LAYER_CFG = {"B": 2, "H": 16, "T": 16384, "d_h": 128}  # the long geometry, bf16 (> L2)


def layer_measure(binding, dev, peaks, steps=10, warmup=3):
    """The layer's transforms around the operator (RoPE of P1, P2 and the Givens mixing of
    I; their gradient) on the long geometry: algorithmic bytes = prep reads P1, P2, I and
    writes Q, K, V; grad reads dQ, dK, dV, I and writes dP1, dP2, dI; HBM roofline."""
    c = LAYER_CFG
    B, H, T, d = c["B"], c["H"], c["T"], c["d_h"]
    g = torch.Generator(device="cpu").manual_seed(0)
    xs = [torch.randn((B, T, H, d), generator=g).to(torch.bfloat16).to(dev) for _ in range(4)]
    theta = (torch.rand(H // 2, generator=g) * 2.0 - 1.0).float().to(dev)
    outs = tuple(torch.empty_like(xs[0]) for _ in range(3))
    ws = torch.empty(max(binding.layer_grad_workspace_size(xs[0]), 16), dtype=torch.uint8,
                     device=dev)
    stream = torch.cuda.current_stream(dev)

    def timed(call):
        for _ in range(warmup):
            call()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
        torch.cuda.synchronize(dev)
        ev[0].record(stream)
        for i in range(steps):
            call()
            ev[i + 1].record(stream)
        torch.cuda.synchronize(dev)
        return statistics.mean(ev[i].elapsed_time(ev[i + 1]) for i in range(steps))

    ms_p = timed(lambda: binding.layer_prep(xs[0], xs[1], xs[2], theta, 1, out=outs,
                                            stream=stream))
    ms_g = timed(lambda: binding.layer_grad(xs[0], xs[1], xs[2], xs[3], theta, 1, workspace=ws,
                                            stream=stream))
    one = B * T * H * d * 2.0
    gb_p, gb_g = 6 * one / (ms_p * 1e-3) / 1e9, 7 * one / (ms_g * 1e-3) / 1e9
    return {"config": {**c, "dtype": "bf16", "pairing": "B", "l2": "arrays 134 MB each > L2"},
            "ms_prep": ms_p, "ms_grad": ms_g,
            "roofline": {"bound": "hbm", "kernel": "layer prep_kernel", "achieved": gb_p,
                         "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": gb_p / peaks["hbm_gbs"],
                         "grad_achieved": gb_g, "grad_frac": gb_g / peaks["hbm_gbs"],
                         "algorithmic_bytes_prep": 6 * one, "algorithmic_bytes_grad": 7 * one},
            "gpu_launches_per_call": {"prep": 1, "grad": 2}}


# The paper's layer geometries (App. B model configurations: heads x width, context and
# per-GPU micro-batch of the Relation runs): 10M 8 x 48 at T = 1024, 30M 8 x 64 at 2048,
# 100M 8 x 80 at 4096.
PAPER_LAYERS = {"10M": (32, 8, 1024, 48), "30M": (16, 8, 2048, 64), "100M": (4, 8, 4096, 80)}


def paper_layers_measure(binding, dev, peaks, steps=10, warmup=3):
    """One Relation layer's token mixing at each paper geometry, fwd + bwd through the
    public API: the layer transforms (RoPE of P1, P2 and the Givens mixing of I), the
    operator forward and backward, and the transforms' gradient, on synthetic bf16 inputs
    (P1, P2, I, dY ~ N(0, 1), Givens angles ~ U(-1, 1), lambda = 0.5).  Operator work as
    7 B H T^2 d_h (the real width; d_h = 48 and 80 run on zero-padded 64- and 128-wide
    tiles)."""
    out = {}
    stream = torch.cuda.current_stream(dev)
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    for name, (B, H, T, d) in PAPER_LAYERS.items():
        g = torch.Generator(device="cpu").manual_seed(0)
        p1, p2, info, dy = (torch.randn((B, T, H, d), generator=g).to(torch.bfloat16).to(dev)
                            for _ in range(4))
        theta = (torch.rand(H // 2, generator=g) * 2.0 - 1.0).float().to(dev)
        qkv = tuple(torch.empty_like(p1) for _ in range(3))
        y = torch.empty_like(p1)
        logz = torch.empty((B, H, T), device=dev, dtype=torch.float32)
        dq, dk, dv = torch.empty_like(p1), torch.empty_like(p1), torch.empty_like(p1)
        dl = torch.empty(1, device=dev, dtype=torch.float32)
        wsb = torch.empty(binding.workspace_size(p1), device=dev, dtype=torch.uint8)
        wsg = torch.empty(max(binding.layer_grad_workspace_size(p1), 16), device=dev,
                          dtype=torch.uint8)
        status = torch.zeros(1, dtype=torch.int32, device=dev)
        q, k, v = qkv
        calls = {
            "prep": lambda: binding.layer_prep(p1, p2, info, theta, 0, out=qkv, stream=stream),
            "fwd": lambda: binding.fwd(q, k, v, lam, tau, out=y, logz=logz, dev_status=status,
                                       stream=stream),
            "bwd": lambda: binding.bwd(q, k, v, y, dy, logz, lam, tau, workspace=wsb, dq=dq,
                                       dk=dk, dv=dv, dlambda=dl, dev_status=status,
                                       stream=stream),
            "grad": lambda: binding.layer_grad(dq, dk, dv, info, theta, 0, workspace=wsg,
                                               stream=stream),
        }
        ms = {k2: _time_calls(c, dev, steps, warmup) for k2, c in calls.items()}
        if int(status.item()) != 0:
            raise SystemExit(f"paper layer {name}: device status "
                             f"{binding.status_string(int(status.item()))}")
        tot = sum(ms.values())
        fl = 7.0 * B * H * T * T * d
        out[name] = {"B": B, "H": H, "T": T, "d_h": d, "ms": ms, "ms_step": tot,
                     "tokens_per_s": B * T / (tot * 1e-3),
                     "operator_tflops": fl / ((ms["fwd"] + ms["bwd"]) * 1e-3) / 1e12,
                     "operator_frac": fl / ((ms["fwd"] + ms["bwd"]) * 1e-3) / 1e12 /
                     peaks["bf16_tflops"]}
        del p1, p2, info, dy, qkv, y, dq, dk, dv, wsb, wsg
    return {"layers": out, "dtype": "bf16", "data": "synthetic",
            "note": "one layer's token mixing; the paper's Table of scale-matched runs reports "
                    "whole-model training tok/s on another GPU (context only)"}


def cp_measure(binding, w, dev, peaks, shards=4, steps=5, warmup=2):
    """The forward of workload w computed as `shards` sequence shards on one GPU (each
    shard's own causal summary, its summaries over every earlier shard's keys merged in,
    then the epilogue at its positions), against the single-call forward: the cost of the
    context-parallel form (the same causal pairs, plus the summaries' fp32 traffic)."""
    q, k, v, _ = workloads.make_inputs(w, seed=0)
    qd, kd, vd = (t.to(dev) for t in (q, k, v))
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    stream = torch.cuda.current_stream(dev)
    T = w.T
    bounds = [T * s // shards for s in range(shards + 1)]
    parts = [tuple(t[:, bounds[s]:bounds[s + 1]].contiguous() for t in (qd, kd, vd))
             for s in range(shards)]
    states = [binding.fwd_state(*parts[s], causal=True, stream=stream) for s in range(shards)]
    other = [tuple(torch.empty_like(x) for x in st) for st in states]
    outs = [(torch.empty_like(parts[s][0]),
             torch.empty((w.B, w.H, bounds[s + 1] - bounds[s]), device=dev, dtype=torch.float32))
            for s in range(shards)]
    y_one = torch.empty_like(qd)
    lz_one = torch.empty((w.B, w.H, T), device=dev, dtype=torch.float32)

    def sharded():
        for s in range(shards):
            binding.fwd_state(*parts[s], causal=True, out=states[s], stream=stream)
            for e in range(s):
                binding.fwd_state(parts[s][0], parts[e][1], parts[e][2], causal=False,
                                  out=other[s], stream=stream)
                binding.state_merge(states[s], other[s], stream=stream)
            binding.state_finish(*parts[s], states[s], lam, tau, pos0=bounds[s],
                                 out=outs[s][0], logz=outs[s][1], stream=stream)

    ms_cp = _time_calls(sharded, dev, steps, warmup)
    ms_one = _time_calls(lambda: binding.fwd(qd, kd, vd, lam, tau, out=y_one, logz=lz_one,
                                             stream=stream), dev, steps, warmup)
    err = max(float((outs[s][0].float() - y_one[:, bounds[s]:bounds[s + 1]].float()).abs().max())
              for s in range(shards))
    fl = w.flops_fwd()
    return {"workload": w.name, "shards": shards, "bounds": bounds, "ms_sharded": ms_cp,
            "ms_one_call": ms_one, "overhead": ms_cp / ms_one,
            "sharded_tflops": fl / (ms_cp * 1e-3) / 1e12,
            "max_abs_diff_vs_one_call": err,
            "gpu_launches": sum(2 + 2 * s for s in range(shards))}


def sdpa_context(w, dev, steps=20, warmup=3):
    """Context only, not this library: PyTorch's causal scaled-dot-product attention
    (softmax attention, the paper's comparison operator) forward + backward on the same
    B, H, T, d_h and dtype, counted with the same 7 B H T^2 d convention.  GPU: CUDA
    events with the L2 flushed between steps; CPU (tests): wall clock."""
    g = torch.Generator(device="cpu").manual_seed(0)
    shape = (w.B, w.H, w.T, w.d)
    dt = w.torch_dtype
    q, k, v, do = (torch.randn(shape, generator=g).to(dt).to(dev) for _ in range(4))
    q.requires_grad_(True)
    k.requires_grad_(True)
    v.requires_grad_(True)
    cuda = dev.type == "cuda"
    flush = torch.empty(L2_FLUSH_BYTES if cuda else 16, dtype=torch.uint8, device=dev)

    def step():
        out = torch.nn.functional.scaled_dot_product_attention(q, k, v, is_causal=True)
        out.backward(do)
        q.grad = k.grad = v.grad = None

    for _ in range(warmup):
        step()
    times = []
    for _ in range(steps):
        flush.zero_()
        if cuda:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            step()
            e1.record()
            torch.cuda.synchronize(dev)
            times.append(e0.elapsed_time(e1))
        else:
            t0 = time.perf_counter()
            step()
            times.append((time.perf_counter() - t0) * 1e3)
    ms = statistics.mean(times)
    return {"operator": "torch scaled_dot_product_attention, causal (softmax attention)",
            "ms_per_step": ms, "tflops": w.flops_fwd_bwd() / (ms * 1e-3) / 1e12,
            "note": "context only: a different operator through PyTorch's kernels"}


LINEAR_CFG = {"B": 8, "H": 12, "T": 2048, "d_h": 64}  # the 100M layer geometry, bf16
LINEAR_SWEEP_TOKENS = 32768  # B * T of each point of the long-context sweep (H = 12, d_h = 64)
FP32_FMA_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12  # 152 SMs x 128 FFMA lanes x 2 flops x 2.07 GHz


def _linear_chunked_flops(B, H, T, d):
    """Tensor-core work of the chunked forward per call: per 128-token block and 64-column
    split, S = Qm Km^T (2 128 128 d), E = Qs C_0 (2 128 64 d), E += tril(S) I~ (2 128 64 128)
    and the state C += KL^T I~ (2 128 64 128; d_h = 64 pads the channels to 128)."""
    nb, splits = -(-T // 128), max(1, d // 64)
    per = 2 * 128 * 128 * d + 2 * 128 * 64 * d + 2 * 128 * 64 * 128 + 2 * 128 * 64 * 128
    return float(B * H * nb * splits * per)


def _linear_chunked_bwd_flops(B, H, T, d):
    """Tensor-core work of the chunked backward per call (d_h = 64), as executed: per
    128-token block, the two state passes' block products (KL^T I~ and Qs^T dY, 2 128 64 128
    each with the channels padded to 128), then S = Qm Km^T and dA = G I~^T (2 128 128 64
    each), X = G C_0^T, Y = I~ dC^T and dI~ = KL dC (2 128 64 64 each), dI~ += A^T G,
    X += dA Km and Y += dA^T Qm (2 128 64 128 each)."""
    nb = -(-T // 128)
    per = 2 * (2 * 128 * 64 * 128) + 2 * (2 * 128 * 128 * d) + 3 * (2 * 128 * 64 * d) + \
        3 * (2 * 128 * 64 * 128)
    return float(B * H * nb * per)


def _time_calls(call, dev, steps, warmup):
    stream = torch.cuda.current_stream(dev)
    for _ in range(warmup):
        call()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    torch.cuda.synchronize(dev)
    ev[0].record(stream)
    for i in range(steps):
        call()
        ev[i + 1].record(stream)
    torch.cuda.synchronize(dev)
    return statistics.mean(ev[i].elapsed_time(ev[i + 1]) for i in range(steps))


def linear_measure(binding, dev, peaks, steps=20, warmup=3):
    """Linear Relation on the 100M geometry (bf16): the chunked tensor-core forward and
    backward, the recurrent CUDA-core forward and backward.  Recurrent arithmetic per token and head:
    forward 5 d^2 (decay, read, write), backward 16 d^2; ALU roofline against the fp32 FMA
    peak of the SMs.  Chunked forward: tensor-core work as counted by _linear_chunked_flops,
    against the measured bf16 peak; chunked backward likewise (_linear_chunked_bwd_flops).
    Then the long-context sweep of the chunked forward,
    T = 1k .. 32k at B T = 32768 tokens."""
    c = LINEAR_CFG
    w = workloads.custom(c["B"], c["H"], c["T"], c["d_h"], "bf16")
    p1, p2, v, alpha, dy = (t.to(dev) for t in workloads.make_linear_inputs(w, seed=0))
    out = torch.empty_like(p1)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    need = max(binding.linear_bwd_workspace_size(p1, "simt"),
               binding.linear_bwd_workspace_size(p1, "tcgen05"))
    wsb = torch.empty(need, dtype=torch.uint8, device=dev)
    fwd = lambda fam: (lambda: binding.linear_fwd(p1, p2, v, alpha, kernel=fam, out=out,
                                                  dev_status=status, stream=stream))
    bwd = lambda fam: (lambda: binding.linear_bwd(p1, p2, v, alpha, dy, kernel=fam, workspace=wsb,
                                                  dev_status=status, stream=stream))
    ms_tc = _time_calls(fwd("tcgen05"), dev, steps, warmup)
    ms_f = _time_calls(fwd("simt"), dev, steps, warmup)
    ms_btc = _time_calls(bwd("tcgen05"), dev, steps, warmup)
    ms_b = _time_calls(bwd("simt"), dev, steps, warmup)
    if int(status.item()) != 0:
        raise SystemExit(f"linear device status {binding.status_string(int(status.item()))}")
    tok_h = w.B * w.T * w.H
    fl_f, fl_b = 5.0 * tok_h * w.d * w.d, 16.0 * tok_h * w.d * w.d
    ach = fl_f / (ms_f * 1e-3) / 1e12
    tc_fl = _linear_chunked_flops(w.B, w.H, w.T, w.d)
    tc_ach = tc_fl / (ms_tc * 1e-3) / 1e12
    tcb_fl = _linear_chunked_bwd_flops(w.B, w.H, w.T, w.d)
    tcb_ach = tcb_fl / (ms_btc * 1e-3) / 1e12
    sweep = []
    for T in (1024, 2048, 4096, 8192, 16384, 32768):
        B = max(1, LINEAR_SWEEP_TOKENS // T)
        ws_ = workloads.custom(B, 12, T, 64, "bf16")
        a = [t.to(dev) for t in workloads.make_linear_inputs(ws_, seed=1)[:4]]
        o = torch.empty_like(a[0])
        wsl = torch.empty(max(binding.linear_fwd_workspace_size(a[0]), 16), dtype=torch.uint8,
                          device=dev)
        ms = _time_calls(lambda: binding.linear_fwd_ws(*a, workspace=wsl, out=o,
                                                       dev_status=status, stream=stream),
                         dev, 5, 2)
        fl = _linear_chunked_flops(B, 12, T, 64)
        sweep.append({"B": B, "T": T, "ms_fwd": ms, "tokens_per_s": B * T / (ms * 1e-3),
                      "tensor_tflops": fl / (ms * 1e-3) / 1e12,
                      "tensor_frac": fl / (ms * 1e-3) / 1e12 / peaks["bf16_tflops"]})
        del a, o, wsl
    if int(status.item()) != 0:
        raise SystemExit(f"linear device status {binding.status_string(int(status.item()))}")
    return {"config": {**c, "dtype": "bf16", "alpha": "KDA-style draw (workloads)"},
            "ms_fwd_chunked": ms_tc, "ms_bwd_chunked": ms_btc, "ms_fwd": ms_f, "ms_bwd": ms_b,
            "tokens_per_s": w.B * w.T / ((ms_tc + ms_btc) * 1e-3),
            "roofline": {"bound": "alu", "kernel": "linear fwd_kernel (recurrent)", "achieved": ach,
                         "peak": FP32_FMA_TFLOPS, "unit": "TFLOP/s (fp32 FMA)",
                         "frac": ach / FP32_FMA_TFLOPS,
                         "bwd_achieved": fl_b / (ms_b * 1e-3) / 1e12},
            "roofline_chunked": {"bound": "tensor", "kernel": "lin_tc_fwd_kernel<64>",
                                 "achieved": tc_ach, "peak": peaks["bf16_tflops"],
                                 "unit": "TFLOP/s", "frac": tc_ach / peaks["bf16_tflops"],
                                 "algorithmic_flops_per_launch": tc_fl},
            "roofline_chunked_bwd": {"bound": "tensor",
                                     "kernel": "chunked backward (five launches)",
                                     "achieved": tcb_ach, "peak": peaks["bf16_tflops"],
                                     "unit": "TFLOP/s", "frac": tcb_ach / peaks["bf16_tflops"],
                                     "flops_per_call": tcb_fl},
            "long_context_sweep": {"kernel": "chunked forward with a workspace (chunk-parallel "
                                             "below one (head, column) pair per SM)",
                                   "H": 12, "d_h": 64,
                                   "tokens_per_point": LINEAR_SWEEP_TOKENS, "points": sweep},
            "gpu_launches_per_step": {"fwd_chunked": 1, "bwd_chunked": 5, "fwd": 1, "bwd": 2}}


def measure_workload(binding, w, dev, steps, warmup, family, peaks, dist=None, ws=1,
                     sample_clocks=False, e2e=True):
    """Time `steps` forward + backward steps of workload `w` (inputs resident in HBM, L2
    flushed between steps) and, with `e2e`, the same steps through the public API from
    pinned host buffers.  Returns the metrics of one JSON record."""
    lam, tau = workloads.LAMBDA_INIT, workloads.TAU_S
    q, k, v, do = workloads.make_inputs(w, seed=0)
    qd, kd, vd, dod = (t.to(dev) for t in (q, k, v, do))
    y = torch.empty_like(qd)
    logz = torch.empty((w.B, w.H, w.T), device=dev, dtype=torch.float32)
    dq, dk, dv = torch.empty_like(qd), torch.empty_like(qd), torch.empty_like(qd)
    dl = torch.empty(1, device=dev, dtype=torch.float32)
    wsb = torch.empty(binding.workspace_size(qd), device=dev, dtype=torch.uint8)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        binding.fwd(qd, kd, vd, lam, tau, kernel=family, out=y, logz=logz, dev_status=status,
                    stream=stream)
        binding.bwd(qd, kd, vd, y, dod, logz, lam, tau, kernel=family, workspace=wsb, dq=dq, dk=dk,
                    dv=dv, dlambda=dl, dev_status=status, stream=stream)

    for _ in range(warmup):
        step()
        flush.zero_()
    torch.cuda.synchronize(dev)
    if int(status.item()) != 0:
        raise SystemExit(f"device status {binding.status_string(int(status.item()))}")

    n = steps
    # per step: forward | backward row pass | backward tiles | backward finalisation
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(n)]
    _barrier(dist, dev)
    torch.cuda.synchronize(dev)
    clk = ClockSampler(dev.index) if sample_clocks else None
    if clk is not None:
        clk.__enter__()
        time.sleep(0.3)  # let the sampler start before the timed region
    t_begin = time.time()
    for i in range(n):
        ev[i][0].record(stream)
        binding.fwd(qd, kd, vd, lam, tau, kernel=family, out=y, logz=logz, dev_status=status,
                    stream=stream)
        ev[i][1].record(stream)
        for j, stage in enumerate((binding.BWD_PREPARE, binding.BWD_TILES,
                                   binding.BWD_FINALIZE)):
            binding.bwd(qd, kd, vd, y, dod, logz, lam, tau, kernel=family, workspace=wsb,
                        dq=dq, dk=dk, dv=dv, dlambda=dl, dev_status=status, stream=stream,
                        stages=stage)
            ev[i][2 + j].record(stream)
        flush.zero_()
    torch.cuda.synchronize(dev)
    t_end = time.time()
    if clk is not None:
        time.sleep(0.1)
        clk.__exit__(None, None, None)
    _barrier(dist, dev)
    t_fwd = [ev[i][0].elapsed_time(ev[i][1]) for i in range(n)]
    t_pre = [ev[i][1].elapsed_time(ev[i][2]) for i in range(n)]
    t_til = [ev[i][2].elapsed_time(ev[i][3]) for i in range(n)]
    t_fin = [ev[i][3].elapsed_time(ev[i][4]) for i in range(n)]
    t_bwd = [a + b + c for a, b, c in zip(t_pre, t_til, t_fin)]
    t_step = [a + b for a, b in zip(t_fwd, t_bwd)]
    ms = _max_over_ranks(dist, statistics.mean(t_step), dev)
    ms_fwd = _max_over_ranks(dist, statistics.mean(t_fwd), dev)
    ms_bwd = _max_over_ranks(dist, statistics.mean(t_bwd), dev)
    ms_tiles = _max_over_ranks(dist, statistics.mean(t_til), dev)
    ms_pre = _max_over_ranks(dist, statistics.mean(t_pre), dev)
    ms_fin = _max_over_ranks(dist, statistics.mean(t_fin), dev)
    st = int(status.item())
    if st != 0:
        raise SystemExit(f"device status {binding.status_string(st)}")

    rec = {}
    if e2e:
        # End to end through the public API: every step copies its inputs from pinned host
        # memory and its results (Y, dQ, dK, dV, dlambda) back.  Two device buffer sets: the
        # inputs of step i + 1 go host->device (stream s_in) and the results of step i - 1
        # device->host (stream s_out) while step i computes, so a step costs the largest of
        # the three, not their sum.  The timed region starts drained and ends when the last
        # results have landed.
        hq, hk, hv, hdo = (t.pin_memory() for t in (q, k, v, do))
        hy, hdq, hdk, hdv = (torch.empty_like(t).pin_memory() for t in (q, q, q, q))
        hdl = torch.empty(1, dtype=torch.float32).pin_memory()
        names = ("q", "k", "v", "do", "y", "dq", "dk", "dv", "dl")
        sets = [dict(zip(names, (qd, kd, vd, dod, y, dq, dk, dv, dl)))]
        sets.append({nm: torch.empty_like(t) for nm, t in sets[0].items()})
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        total = n + warmup
        ev_in, ev_cmp, ev_out = ([torch.cuda.Event() for _ in range(total)] for _ in range(3))
        e2e_t0 = torch.cuda.Event(enable_timing=True)
        e2e_t1 = torch.cuda.Event(enable_timing=True)
        for i in range(total):
            bs = sets[i % 2]
            if i == warmup:
                torch.cuda.synchronize(dev)
                e2e_t0.record(s_in)
            if i >= 2:
                s_in.wait_event(ev_cmp[i - 2])  # set i % 2 no longer read by step i - 2
            with torch.cuda.stream(s_in):
                for src, nm in ((hq, "q"), (hk, "k"), (hv, "v"), (hdo, "do")):
                    bs[nm].copy_(src, non_blocking=True)
            ev_in[i].record(s_in)
            stream.wait_event(ev_in[i])
            if i >= 2:
                stream.wait_event(ev_out[i - 2])  # step i - 2's results have left set i % 2
            binding.fwd(bs["q"], bs["k"], bs["v"], lam, tau, kernel=family, out=bs["y"],
                        logz=logz, dev_status=status, stream=stream)
            binding.bwd(bs["q"], bs["k"], bs["v"], bs["y"], bs["do"], logz, lam, tau,
                        kernel=family, workspace=wsb, dq=bs["dq"], dk=bs["dk"], dv=bs["dv"],
                        dlambda=bs["dl"], dev_status=status, stream=stream)
            flush.zero_()
            ev_cmp[i].record(stream)
            s_out.wait_event(ev_cmp[i])
            with torch.cuda.stream(s_out):
                for nm, dst in (("y", hy), ("dq", hdq), ("dk", hdk), ("dv", hdv), ("dl", hdl)):
                    dst.copy_(bs[nm], non_blocking=True)
            ev_out[i].record(s_out)
        e2e_t1.record(s_out)
        torch.cuda.synchronize(dev)
        ms_e2e = _max_over_ranks(dist, e2e_t0.elapsed_time(e2e_t1) / n, dev)
        h2d = sum(t.numel() * t.element_size() for t in (hq, hk, hv, hdo))
        d2h = sum(t.numel() * t.element_size() for t in (hy, hdq, hdk, hdv, hdl))
        rec["e2e"] = {"value": ws * w.flops_fwd_bwd() / (ms_e2e * 1e-3) / 1e12,
                      "unit": "TFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                      "ms_per_step": ms_e2e,
                      "overlap": "two buffer sets: step i+1's H2D and step i-1's D2H run on "
                                 "their own streams during step i's compute (L2 flushed after "
                                 "each step)"}
        del sets

    flops = w.flops_fwd_bwd()
    tflops = ws * flops / (ms * 1e-3) / 1e12
    esz = 2 if w.dtype == "bf16" else 4
    bwd_flops = 5.0 * w.B * w.H * w.T * w.T * w.d  # causal bwd incl. the U recompute
    tiles_tflops = bwd_flops / (ms_tiles * 1e-3) / 1e12
    fwd_tflops = w.flops_fwd() / (ms_fwd * 1e-3) / 1e12
    tc = family != "simt" and w.dtype == "bf16"
    dpad = 64 if w.d <= 64 else 128
    kname = f"bwd_tc_kernel<{dpad}>" if tc else "bwd_dkdv+dq (simt)"
    traffic = _profiled_traffic(w, "bwd_tc_kernel") if tc else None
    rec.update({
        "value": tflops, "unit": "TFLOP/s", "ms_per_step": ms,
        "tokens_per_s": ws * w.tokens / (ms * 1e-3),
        "pct_bf16_peak": 100.0 * tflops / (ws * peaks["bf16_tflops"]),
        "pct_bf16_peak_sustained": 100.0 * tflops / (ws * peaks["bf16_tflops_sustained"]),
        # the same time under the algorithmic minimum without the U recompute, 6 B H T^2 d
        "tflops_6bht2d": tflops * 6.0 / 7.0,
        "ms_fwd": ms_fwd, "ms_bwd": ms_bwd,
        "ms_bwd_stages": {"prepare": ms_pre, "tiles": ms_tiles, "finalize": ms_fin},
        "fwd_tflops": ws * fwd_tflops,
        "bwd_tflops": ws * bwd_flops / (ms_bwd * 1e-3) / 1e12,
        "roofline": {"kernel": kname, "bound": "tensor", "achieved": tiles_tflops,
                     "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                     "frac": tiles_tflops / peaks["bf16_tflops"],
                     "peak_source": f"{peaks['source']} dense bf16 (burst, cuBLAS)",
                     "algorithmic_flops_per_launch": bwd_flops,
                     "traffic": traffic,
                     "algorithmic_bytes_per_launch": 8.0 * w.B * w.T * w.H * w.d * esz,
                     "fwd_kernel": {"kernel": f"fwd_tc_kernel<{dpad}>" if tc else "fwd (simt)",
                                    "achieved": fwd_tflops,
                                    "frac": fwd_tflops / peaks["bf16_tflops"]},
                     "step": {"achieved": tflops / ws,
                              "frac": tflops / ws / peaks["bf16_tflops"]}},
        "gpu_launches": n * (binding.launches_per_call(family, w.dtype, w.d, "fwd")
                             + binding.launches_per_call(family, w.dtype, w.d, "bwd")),
        "config": {"workload": w.description, "B": w.B, "H": w.H, "T": w.T, "d_h": w.d,
                   "lambda": workloads.LAMBDA_INIT, "tau_s": workloads.TAU_S,
                   "kernel": family, "l2": "flushed between steps (256 MiB write)",
                   "inputs": "Q,K,V,dO iid normal, seed 0 (workload recipe)",
                   "parallelism": f"replicas x{ws}"},
        "steps": n,
    })
    if clk is not None:
        rec["clocks"] = clk.summary(t_begin, t_end)
    return rec


def run_ours(args, w):
    from paper_2608_20172_gb300 import binding
    dist, ws, rank, local = _dist()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    binding.load()
    peaks = _peaks()
    family = args.kernel
    head = measure_workload(binding, w, dev, args.steps, args.warmup, family, peaks, dist, ws,
                            sample_clocks=(rank == 0))
    line = {
        "metric": "FlashRelation fwd+bwd TFLOP/s (7*B*H*T^2*d causal)",
        "value": head["value"], "unit": "TFLOP/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": head["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
    }
    line.update({k: v for k, v in head.items() if k not in line})
    # further workloads of the same run, each with its own timed region (more steps on the
    # short ones so that each region lasts tens of milliseconds)
    subs = {}
    for name in args.also:
        sw = workloads.WORKLOADS[name]
        if sw.name == w.name:
            continue
        steps = max(args.steps, int(math.ceil(0.1 / max(sw.flops_fwd_bwd() / 4e14, 1e-6))))
        rec = measure_workload(binding, sw, dev, steps, args.warmup, family, peaks, dist, ws,
                               sample_clocks=(rank == 0))
        subs[name] = rec
    if subs:
        line["sub_records"] = subs
    if rank == 0 and ws == 1 and not args.no_side:
        line["decode"] = decode_measure(binding, dev, peaks)
        line["linear"] = linear_measure(binding, dev, peaks)
        line["layer"] = layer_measure(binding, dev, peaks)
        line["paper_layers"] = paper_layers_measure(binding, dev, peaks)
        line["context_parallel"] = cp_measure(binding, w, dev, peaks)
        try:
            line["context_sdpa"] = sdpa_context(w, dev)
        except Exception as exc:  # context only: never at the expense of the line
            line["context_sdpa"] = {"not_measured": f"{type(exc).__name__}: {exc}"[:200]}
    if rank == 0 and not args.no_cpu_baseline and ws == 1:
        cb = cpu_oracle_run(w, min_seconds=10.0)
        # the same oracle on one thread, over a sample one head wide per thread of the above
        c1 = cpu_oracle_run(w, n_heads=max(1, cb["heads"] // max(1, cb["cores"])),
                            t_rows=cb["rows"], min_seconds=3.0, nthreads=1)
        line["cpu_baseline"] = {
            "value": cb["tflops"], "unit": "TFLOP/s", "cores": cb["cores"], "kind": "oracle",
            "sample": f"{_sample_text(w, cb)} x {cb['reps']}, fwd+bwd, fp64 C oracle "
                      f"(OpenMP over heads), {cb['seconds']:.1f} s",
            "single_thread": {"value": c1["tflops"], "unit": "TFLOP/s", "cores": 1,
                              "sample": f"{_sample_text(w, c1)} x {c1['reps']}, "
                                        f"{c1['seconds']:.1f} s"}}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="long", choices=sorted(workloads.WORKLOADS))
    ap.add_argument("--also", default="100M",
                    help="comma-separated further workloads measured as sub-records, or none")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--kernel", default="auto", choices=["auto", "simt", "tcgen05"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-side", action="store_true",
                    help="skip the decode, Linear Relation, layer-transform and SDPA legs")
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's batch (a slice for profiler captures)")
    ap.add_argument("--heads", type=int, default=None,
                    help="override the workload's head count (a slice for profiler captures)")
    args = ap.parse_args(argv)
    args.also = [] if args.also in ("", "none") else args.also.split(",")
    for name in args.also:
        if name not in workloads.WORKLOADS:
            ap.error(f"--also: unknown workload {name}")
    args.warmup = max(args.warmup, 3)  # at least 3 untimed warm-up steps
    w = workloads.WORKLOADS[args.config]
    if args.batch or args.heads:
        import dataclasses
        B, H = args.batch or w.B, args.heads or w.H
        w = dataclasses.replace(w, B=B, H=H, description=f"{w.description}, slice B={B} H={H}")
    if args.impl == "reference":
        return run_reference(args, w)
    return run_ours(args, w)


if __name__ == "__main__":
    sys.exit(main())
