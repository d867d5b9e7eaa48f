"""Benchmark of the masked second-order HLA hot path on GB300.

One step = one hla2_forward over the long-context workload (B=2, H=16,
n=16384, d=dv=128, chunk 128, bf16 tokens, masked, ratio-normalised; inputs
resident in HBM).  The decode-step workload (B=64, H=32, d=dv=128, fp32 state,
bf16 tokens, state built from a 4096-token prefix) is measured in the same run
and reported under "decode".  Prints ONE JSON line (rank 0).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Multi-GPU (torchrun): every rank runs its own copy of the workload (heads are
independent; no collective on the data path), the timed region is bracketed by
barriers, and the max time over ranks is used: weak scaling.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import hla_inputs  # noqa: E402

METRIC = "masked HLA-2 forward tokens/s at 1 GB300 and % of roofline; decode-step GB/s"
FWD = hla_inputs.WORKLOADS["long_bf16_norm"]
DEC = hla_inputs.WORKLOADS["decode_bf16"]


# DRAM traffic per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one ncu
# capture of the kernel sources (concatenated) whose SHA-256 starts with "sha256"
# (summaries in profiles/); reported as null for any other source or workload.
TRAFFIC = {
    "hla2_fused_kernel": {"src": ["hla_fused_sm103.cu", "sm103_prims.cuh"], "sha256": "7ca8b7c6b836b2ff", "workload": "long_bf16_norm",
                          "n": 16384, "bytes": 526.6e6,
                          "how": "ncu capture at n=8192 (227.5 MB read + 35.8 MB written during the launch; outputs "
                                 "still dirty in L2 at its end are written later) scaled x2 to n=16384"},
    "step2_kernel": {"src": ["hla_step.cu"], "sha256": "7f4bfb053a9af874", "workload": "decode_bf16", "n": 0,
                     "bytes": 750.3e6, "how": "ncu capture of one step at B64 H32 d128 (bench.py --profile-case "
                                              "tuple_step): 406.4 MB read + 343.9 MB written"},
    "c3_kernels": {"src": ["hla3_chunked.cu"], "sha256": "17ac1acd5c9202d1", "workload": "hla3_f32", "n": 4096,
                   "bytes": 432.5e6, "how": "ncu capture of one forward's five launches (bench.py --only hla3_f32): "
                                            "373.0 MB read + 59.5 MB written, 6.4 x the token I/O (per-chunk records)"},
    "hla3_tc_kernels": {"src": ["hla3_sm103.cu", "sm103_prims.cuh"], "sha256": "dd16e8c0a54902eb", "workload": "hla3_f32",
                        "n": 4096, "bytes": 115.0e6,
                        "how": "ncu capture of one forward's three launches (bench.py --only hla3_f32), caches "
                               "flushed per launch: pre-pass 37.8 MB read, sweep 51.6 MB read + 0.1 MB written "
                               "(outputs still dirty in L2 at its end), fix-up 25.6 MB read"},
    "bwd_tc_kernel": {"src": ["hla_backward_sm103.cu", "sm103_prims.cuh"], "sha256": "e1940b86e729b1d1",
                      "workload": "mid_bf16", "n": 2048, "bytes": 448.4e6,
                      "how": "ncu capture of one backward (bench.py --only backward): 278.0 MB read + 170.4 MB "
                             "written; the per-tile records (X hi, lo; S_p, D_p: 96 MB) are written once and read "
                             "back once"},
    "step2_kernel_sde": {"src": ["hla_step.cu"], "sha256": "7f4bfb053a9af874", "workload": "decode_bf16", "n": 0,
                         "bytes": 480.2e6, "how": "ncu capture of one step at B64 H32 d128 (bench.py --profile-case "
                                                  "sde_step): 271.1 MB read + 209.1 MB written"},
}


def traffic(kernel, workload, n):
    import hashlib
    t = TRAFFIC.get(kernel)
    if t is None or t["workload"] != workload or (t["n"] and t["n"] != n):
        return None, None
    h = hashlib.sha256()
    for name in t["src"]:
        with open(os.path.join(ROOT, "paper_2510_27258_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    if not h.hexdigest().startswith(t["sha256"]):
        return None, None
    return t["bytes"], t["how"]


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def fwd_bytes(w):
    """Algorithmic bytes of one forward: read q, k, v once, write out once."""
    s = 2 if w.dtype == "bf16" else 4
    return w.BH * w.n * ((2 * w.d + w.dv) * s + w.dv * s)


def fwd_flops(w):
    """Algorithmic FLOPs of one forward (masks and the symmetry of S exploited):
    per token-head 2C(d+dv) + C^2/3 + 3d^2 + 6 d dv + 2 d^2 dv / C."""
    C, d, dv = w.chunk, w.d, w.dv
    per = 2 * C * (d + dv) + C * C / 3 + 3 * d * d + 6 * d * dv + 2 * d * d * dv / C
    return w.BH * w.n * per


def roofline_record(w, ms, hbm_peak, tc_peak, peak_kind, traffic_bytes, traffic_how, kernel):
    """Roofline of one forward: its bound is the slower of the algorithmic bytes at the measured HBM
    bandwidth and the algorithmic FLOPs at the measured bf16 tensor peak; frac = that time / the
    measured time; the other resource is reported beside it."""
    t_bytes = fwd_bytes(w) / (hbm_peak * 1e9)
    t_flops = fwd_flops(w) / (tc_peak * 1e12)
    gbs = fwd_bytes(w) / (ms * 1e-3) / 1e9
    tfl = fwd_flops(w) / (ms * 1e-3) / 1e12
    hbm = {"achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak}
    ten = {"achieved": tfl, "peak": tc_peak, "unit": "TFLOP/s", "frac": tfl / tc_peak}
    bound, other = ("hbm", ten) if t_bytes >= t_flops else ("tensor", hbm)
    main = hbm if bound == "hbm" else ten
    rec = {"bound": bound, "achieved": main["achieved"], "peak": main["peak"], "unit": main["unit"],
           "frac": main["frac"], "traffic": traffic_bytes, "traffic_how": traffic_how,
           "algorithmic_bytes": fwd_bytes(w), "algorithmic_flops": fwd_flops(w),
           "roofline_us": max(t_bytes, t_flops) * 1e6, "peak_kind": peak_kind, "kernel": kernel}
    rec["tensor_view" if bound == "hbm" else "hbm_view"] = other
    return rec


def hla3_flops(w):
    """FLOPs of one masked third-order forward in the chunk-parallel form the kernels compute
    (Theorem 4; chunk W, 2 per multiply-add): chunk summaries, brackets and outputs."""
    W, d, dv = min(w.chunk, 64 if max(w.d, w.dv) < 128 else 32), w.d, w.dv
    tri, stri = W * (W + 1) // 2, W * (W - 1) // 2
    local = 2 * d * d * W + 3 * d * dv * W + d * d * W + W * W * d + (tri + stri) * dv
    bracket = W * d * d + 2 * d * d * dv + d * dv * W
    out = W * W * d + 2 * W * d * d + W * W * d + W * W * W // 2 + W * d * dv + tri * dv + W * d * dv + 2 * tri * dv
    chunks = w.B * w.H * ((w.n + W - 1) // W)
    return 2 * chunks * (local + bracket + out)


def hla3_tc_flops(w):
    """FLOPs of one masked third-order forward in the 128-token tile form of the tensor-core path
    (2 per multiply-add, triangles counted once): per tile of T tokens, A = Q K^T (T^2 d, the
    squares above the diagonal enter b), Y (T d dv + T^2 dv / 2), Q S^K_p and K S^Q_p (2 T d^2),
    C' on the lower triangle (T^3 / 6 + T^2 d / 2), LA^T aV, LA Z', (L.C') aV (3 T^2 dv / 2),
    Q F_p (T d dv) and the carries K^T K, Q^T Q, K^T V, K^T G', (Q S^K_p)^T aV (2 T d^2 + 3 T d dv)."""
    T, d, dv = 128, w.d, w.dv
    tiles = w.B * w.H * ((w.n + T - 1) // T)
    per_tile = (T * T * d + T * d * dv + T * T * dv / 2 + 2 * T * d * d + T ** 3 / 6 + T * T * d / 2
                + 3 * T * T * dv / 2 + T * d * dv + 2 * T * d * d + 3 * T * d * dv)
    return 2 * tiles * per_tile


def hla3_tc_issued_flops(w, sms=152):
    """Tensor FLOPs the tensor-core path issues (bf16 hi/lo splits, full 128-row tiles): per
    sweep tile 36 K = 16 steps at N = 128, 104 at N = 64 and 24 at N = 32; per pre-pass tile 24
    at N = 64 (segments as the library plans them: sms // (B H) per head, at most one per tile)."""
    T = 128
    M = (w.n + T - 1) // T
    BH = w.B * w.H
    G = max(1, min(M, sms // BH, 160))
    L = (M + G - 1) // G
    G = (M + L - 1) // L
    pre_tiles = BH * (M - (M - (G - 1) * L)) if G > 1 else 0
    step = lambda N: 2 * 128 * N * 16
    return BH * M * (36 * step(128) + 104 * step(64) + 24 * step(32)) + pre_tiles * 24 * step(64)


def ahla_flops(w):
    """Algorithmic FLOPs of one AHLA forward (masks exploited, chunk C): per token-head
    2 * [C d / 2 (Q K^T) + C dv / 2 (A V) + C dv / 2 (A R) + C / 2 (A 1, A s)
         + 4 d dv (Q P_p, Q E_p, K^T V, K^T R) + 2 d (Q m_p, Q n_p) + d^2 dv / C (R^KQ P_p)]."""
    C, d, dv = min(w.chunk, 64), w.d, w.dv
    per = 2 * (C * d / 2 + C * dv + C / 2 + 4 * d * dv + 2 * d + d * d * dv / C)
    return w.BH * w.n * per


def ahla_dec_bytes(w):
    """Algorithmic bytes of one AHLA decode step: read + write of (P, m, E, n) of every head plus token I/O."""
    st = 2 * w.d * w.dv + 2 * w.d
    s = 2 if w.dtype == "bf16" else 4
    return w.BH * (2 * st * 4 + (2 * w.d + w.dv) * s + w.dv * s)


def alu_peak():
    """fp32 CUDA-core peak: 152 SMs x 128 FP32 lanes x 2 FLOP x 2.07 GHz (maximum SM clock)."""
    return 152 * 128 * 2 * 2.07e9 / 1e12


def dec_bytes(w):
    """Algorithmic bytes of one decode step: read + write of the fp32 state tuple
    (S, C, m, G, h) of every head plus the token I/O."""
    st = w.d * w.d + 2 * w.d * w.dv + 2 * w.d
    s = 2 if w.dtype == "bf16" else 4
    return w.BH * (2 * st * 4 + (2 * w.d + w.dv) * s + w.dv * s)


def dec_sde_bytes(w):
    """Algorithmic bytes of one decode step on (S, D, e) states: read + write of S, D, e of every
    head plus the token I/O."""
    st = w.d * w.d + w.d * w.dv + w.d
    s = 2 if w.dtype == "bf16" else 4
    return w.BH * (2 * st * 4 + (2 * w.d + w.dv) * s + w.dv * s)


class ClockSampler:
    """nvidia-smi clock/throttle samples (every 100 ms) around a timed region."""

    FIELDS = ("index,timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.fh,
                                         stderr=subprocess.DEVNULL)
            # nvidia-smi can take seconds to start; a timed region must not include that
            t_end = time.time() + 20.0
            while time.time() < t_end and os.path.getsize(self.path) == 0 and self.proc.poll() is None:
                time.sleep(0.05)
            time.sleep(0.2)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        self.proc.wait()
        self.fh.close()
        rows = [r.split(",") for r in open(self.path).read().strip().splitlines() if r.count(",") >= 9]
        os.unlink(self.path)
        sm = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        smax = [float(r[3]) for r in rows if r[3].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if "Active" in r[6 + i] and "Not" not in r[6 + i]})
        loaded = [x for x in sm if x > 0.5 * max(sm)] if sm else []
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


def dist_setup(gpus, backend=None):
    """One process per GPU (torchrun sets RANK / LOCAL_RANK / WORLD_SIZE / MASTER_*): NCCL on GPUs,
    gloo without one (the host-side logic of the replica mode, tested on CPU)."""
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = backend or ("nccl" if torch.cuda.is_available() else "gloo")
        if backend == "nccl":
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group(backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """The largest of the ranks' values (the step time of a weak-scaling job is its slowest rank's)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(units_per_rank, world, ms):
    """Whole-job throughput: every rank processes its own copy of the workload (heads are
    independent), so the job processes world x units in the slowest rank's time."""
    return units_per_rank * world / (ms * 1e-3)


def cpu_baseline(budget_s=15.0):
    """The fp64 oracle, as it stands, on a bounded sample of the forward workload:
    the first `heads` heads of the same inputs, all n positions, all host cores."""
    import oracle
    cores = os.cpu_count() or 1
    heads = max(1, min(FWD.BH, cores))
    q, k, v = hla_inputs.make_workload(FWD)
    qf, kf, vf = (x.reshape(FWD.BH, FWD.n, -1)[:heads] for x in (q, k, v))
    # size the sample from a short probe so the run stays near the budget
    t0 = time.time()
    oracle.hla2_serial(qf[:, :512], kf[:, :512], vf[:, :512], masked=True, normalized=True, eps=hla_inputs.EPS,
                       nthreads=cores)
    probe = time.time() - t0
    n = int(min(FWD.n, max(512, 512 * budget_s / max(probe, 1e-6))))
    t0 = time.time()
    oracle.hla2_serial(qf[:, :n], kf[:, :n], vf[:, :n], masked=True, normalized=True, eps=hla_inputs.EPS,
                       nthreads=cores)
    dt = time.time() - t0
    token_heads = heads * n
    return {"value": token_heads / FWD.H / dt, "unit": "tokens/s", "cores": min(cores, heads), "kind": "oracle",
            "sample": "fp64 serial oracle on %d of %d heads x first %d of %d positions of the forward workload "
                      "(tokens/s = token-heads/s / H), %.1f s" % (heads, FWD.BH, n, FWD.n, dt)}


def run_reference(args):
    """--impl reference: the oracle on the host cores, one bounded sample per step."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    cores = os.cpu_count() or 1
    heads = max(1, min(FWD.BH, cores))
    q, k, v = hla_inputs.make_workload(FWD)
    n = 1024
    qf, kf, vf = (np.ascontiguousarray(x.reshape(FWD.BH, FWD.n, -1)[:heads, :n]) for x in (q, k, v))
    for _ in range(args.warmup):
        oracle.hla2_serial(qf, kf, vf, masked=True, normalized=True, eps=hla_inputs.EPS, nthreads=cores)
    t0 = time.time()
    for _ in range(args.steps):
        oracle.hla2_serial(qf, kf, vf, masked=True, normalized=True, eps=hla_inputs.EPS, nthreads=cores)
    dt = (time.time() - t0) / args.steps
    value = heads * n / FWD.H / dt
    sample = "fp64 serial oracle on %d of %d heads x first %d positions per step" % (heads, FWD.BH, n)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": "long_bf16_norm (sampled)", "B": FWD.B, "H": FWD.H, "n": FWD.n, "d": FWD.d,
                   "dv": FWD.dv, "chunk": FWD.chunk},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": min(cores, heads), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0, help="timed forward steps (0 = about 2 s worth)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--decode-steps", type=int, default=DEC.decode_steps)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--workload", default="long_bf16_norm", choices=sorted(hla_inputs.WORKLOADS),
                    help="forward workload (default: the long-context one the metric is quoted on)")
    ap.add_argument("--n", type=int, default=0, help="override the sequence length (profiling runs)")
    ap.add_argument("--profile-case", default="", choices=["", "sde_step", "tuple_step", "ahla_step", "ahla_fwd",
                                                             "backward"],
                    help="run a few launches of one kernel family on a small case (for ncu captures) and exit")
    ap.add_argument("--only", default="", choices=["", "mid_bf16", "hla3_f32", "ahla", "backward"],
                    help="time only this secondary workload (the d = 64 forward or third order) and print its object")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.impl == "reference":
        if args.steps <= 0:
            args.steps = 3
        return run_reference(args)

    import torch

    from paper_2510_27258_gb300 import build
    build.build()
    from paper_2510_27258_gb300 import hla

    rank, world, local = dist_setup(args.gpus)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    hbm_peak, tc_peak, peak_kind = peaks()
    if args.profile_case:
        return profile_case(hla, dev, args.profile_case)
    if args.only in ("ahla", "backward"):
        st = torch.cuda.current_stream()
        res = (bench_ahla(hla, dev, st, hbm_peak, world, tc_peak=tc_peak) if args.only == "ahla"
               else bench_backward(hla, dev, st, world, hbm_peak, tc_peak))
        if rank == 0:
            print(json.dumps(res))
        return
    if args.only:
        stream = torch.cuda.current_stream()
        res = bench_others(hla, dev, stream, hbm_peak, tc_peak, world, names=(args.only,),
                           steps=args.steps if args.steps > 0 else 20, warmup=args.warmup)
        if rank == 0:
            print(json.dumps(res[0]))
        return

    # ---------------- forward workload ----------------
    w = hla_inputs.WORKLOADS[args.workload]
    if args.n > 0:
        import dataclasses
        w = dataclasses.replace(w, n=args.n)
    path, launches_per_step = hla.hla2_forward_path(w.B, w.H, w.n, w.d, w.dv, masked=w.masked,
                                                    normalized=w.normalized, chunk=w.chunk,
                                                    dtype=torch.bfloat16 if w.dtype == "bf16" else torch.float32)
    q, k, v = hla_inputs.make_workload(w)
    tq, tk, tv = (hla_inputs.as_torch(x, w.dtype, dev) for x in (q, k, v))
    out = torch.empty((w.B, w.H, w.n, w.dv), dtype=tq.dtype, device=dev)
    ws = hla.alloc_workspace(hla.hla2_workspace_bytes(w.B, w.H, w.n, w.d, w.dv, w.chunk, tq.dtype), dev)
    stream = torch.cuda.current_stream()

    def step():
        hla.hla2_forward(tq, tk, tv, out, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS,
                         chunk=w.chunk, workspace=ws, stream=stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if hla.hla_poll_error(ws) != 0:
        raise RuntimeError("device-side error flag set during warm-up")
    if args.steps <= 0:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        torch.cuda.synchronize()
        args.steps = int(max(10, min(20000, 2000.0 / max(e0.elapsed_time(e1), 1e-3))))

    sampler = ClockSampler(local)
    sampler.start()
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clocks = sampler.stop()
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    if hla.hla_poll_error(ws) != 0:
        raise RuntimeError("device-side error flag set during the timed region")

    # BASELINE protocol beside the contract's K-step mean: >= 50 single launches, each after a
    # 256 MB write that flushes L2, timed one by one with CUDA events on the launching stream; median
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    per = []
    for _ in range(max(50, args.steps)):
        flush.fill_(1)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        step()
        b.record(stream)
        per.append((a, b))
    torch.cuda.synchronize()
    per_ms = sorted(a.elapsed_time(b) for a, b in per)
    med_ms = max_over_ranks(per_ms[len(per_ms) // 2], world)
    del flush, per

    tokens = w.B * w.n  # sequence positions per forward (every head processed)
    if args.workload != "long_bf16_norm" or args.n > 0:
        args.no_cpu_baseline = True  # the CPU baseline samples the long workload only
    value = weak_scaling_value(tokens, world, ms)
    fwd_traffic, fwd_traffic_how = traffic("hla2_fused_kernel", w.name, w.n) if path == 1 else (None, None)

    # ---------------- end to end: pinned host buffers, copies inside the timed region ----------
    # Every step copies its inputs from pinned host memory and its output back.  Steps are
    # independent, so they are pipelined over two sets of device buffers: the host-to-device
    # copy of step i+1 and the read-back of step i-1 run on their own streams while step i's
    # forward runs; the timed region spans all copies of all steps.
    hq, hk, hv = (t.cpu().pin_memory() for t in (tq, tk, tv))
    hout = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    nb = 2
    dins = [[torch.empty_like(t) for t in (tq, tk, tv)] for _ in range(nb)]
    douts = [torch.empty_like(out) for _ in range(nb)]
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev_in, ev_cmp, ev_out = ([torch.cuda.Event() for _ in range(nb)] for _ in range(3))

    def e2e_step(i):
        b = i % nb
        with torch.cuda.stream(s_in):
            s_in.wait_event(ev_cmp[b])  # the forward that read this buffer set (step i - 2) is done
            for dst, src in zip(dins[b], (hq, hk, hv)):
                dst.copy_(src, non_blocking=True)
            ev_in[b].record(s_in)
        stream.wait_event(ev_in[b])
        stream.wait_event(ev_out[b])  # the read-back of this output buffer (step i - 2) is done
        hla.hla2_forward(*dins[b], douts[b], masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS,
                         chunk=w.chunk, workspace=ws, stream=stream)
        ev_cmp[b].record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev_cmp[b])
            hout.copy_(douts[b], non_blocking=True)
            ev_out[b].record(s_out)

    for i in range(2):
        e2e_step(i)
    torch.cuda.synchronize()
    e2e_steps = max(3, min(args.steps, 50))
    barrier(world)
    e0.record(stream)
    s_in.wait_stream(stream)
    for i in range(e2e_steps):
        e2e_step(i)
    stream.wait_stream(s_out)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, world)
    in_bytes = sum(t.numel() * t.element_size() for t in (hq, hk, hv))
    out_bytes = hout.numel() * hout.element_size()
    # the host link alone: the same pinned buffers copied in (and the output back), 5 times each
    link = {}
    for name, copies, nbytes in (("h2d_gbs", [(d_, h_) for d_, h_ in zip(dins[0], (hq, hk, hv))], in_bytes),
                                 ("d2h_gbs", [(hout, douts[0])], out_bytes)):
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(5):
            for dst, src in copies:
                dst.copy_(src, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        link[name] = nbytes * 5 / (e0.elapsed_time(e1) * 1e-3) / 1e9
    link["how"] = "pinned host buffers of the e2e leg, one stream, 5 x the per-step bytes, CUDA events"
    del hq, hk, hv, hout, dins, douts

    result = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if path == 1 else "f32", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "H": w.H, "n": w.n, "d": w.d, "dv": w.dv,
                   "chunk": w.chunk, "masked": w.masked, "normalized": w.normalized, "tokens": w.dtype,
                   "path": "fused tcgen05 kernel" if path == 1 else "generic CUDA-core kernels",
                   "global_batch": w.B * world, "seq_len": w.n, "parallelism": "replicas (heads independent)",
                   "l2": "inputs larger than L2: %.0f MB read + %.0f MB written per step" % (
                       3 * w.BH * w.n * w.d * 2 / 1e6, w.BH * w.n * w.dv * 2 / 1e6)},
        "clocks": clocks,
        "roofline": roofline_record(w, ms, hbm_peak, tc_peak, peak_kind, fwd_traffic, fwd_traffic_how,
                                    "hla2_fused_kernel (the forward's only kernel)" if path == 1
                                    else "hla2_forward (3 kernels)"),
        "median_flushed": {"ms": med_ms, "runs": len(per_ms), "value": tokens * world / (med_ms * 1e-3),
                           "how": "median of single launches, each after a 256 MB write that flushes L2"},
        "e2e": {"value": tokens * world / (e2e_ms * 1e-3), "unit": "tokens/s", "ms_per_step": e2e_ms,
                "h2d_bytes_per_step": in_bytes, "d2h_bytes_per_step": out_bytes, "host_link": link},
        "gpu_launches": launches_per_step * args.steps,
    }
    del tq, tk, tv, out, ws
    torch.cuda.empty_cache()

    # ---------------- decode step workload ----------------
    if not args.no_decode:
        result["decode"] = bench_decode(hla, dev, stream, args.decode_steps, hbm_peak, world)
        result["gpu_launches"] += result["decode"]["launches"]

    # ---------------- the other configs: d = 64 forward and third order ----------------
    if not args.no_decode:
        result["mid"], result["hla3"] = bench_others(hla, dev, stream, hbm_peak, tc_peak, world)
        result["gpu_launches"] += result["mid"]["launches"] + result["hla3"]["launches"]
        result["ahla"] = bench_ahla(hla, dev, stream, hbm_peak, world, tc_peak=tc_peak)
        result["gpu_launches"] += result["ahla"]["forward"]["launches"] + result["ahla"]["decode"]["launches"]
        result["backward"] = bench_backward(hla, dev, stream, world, hbm_peak, tc_peak)
        result["gpu_launches"] += result["backward"]["launches"]
    if rank == 0 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline()
    if rank == 0:
        print(json.dumps(result))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def bench_others(hla, dev, stream, hbm_peak, tc_peak, world, names=("mid_bf16", "hla3_f32"), steps=20, warmup=3):
    """Forward of mid_bf16 (B8 H16 n2048 d64 bf16) and of hla3_f32 (masked third order, B4 H8 n4096 d32
    fp32): `steps` timed calls each after `warmup` calls, CUDA events on the launching stream."""
    import torch
    res = []
    for name in names:
        w = hla_inputs.WORKLOADS[name]
        q, k, v = hla_inputs.make_workload(w)
        tq, tk, tv = (hla_inputs.as_torch(x, w.dtype, dev) for x in (q, k, v))
        out = torch.empty((w.B, w.H, w.n, w.dv), dtype=tq.dtype, device=dev)
        third = w.order == 3
        nbytes = (hla.hla3_workspace_bytes if third else hla.hla2_workspace_bytes)(w.B, w.H, w.n, w.d, w.dv, w.chunk,
                                                                                  tq.dtype)
        ws = hla.alloc_workspace(nbytes, dev)
        fwd = hla.hla3_forward if third else hla.hla2_forward

        def call():
            fwd(tq, tk, tv, out, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS, chunk=w.chunk,
                workspace=ws, stream=stream)
        for _ in range(warmup):
            call()
        torch.cuda.synchronize()
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            call()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = max_over_ranks(e0.elapsed_time(e1) / steps, world)
        if hla.hla_poll_error(ws) != 0:
            raise RuntimeError("device-side error flag set while timing " + name)
        tok = w.B * w.n * world / (ms * 1e-3)
        cfg = {"workload": name, "B": w.B, "H": w.H, "n": w.n, "d": w.d, "dv": w.dv, "chunk": w.chunk,
               "masked": w.masked, "normalized": w.normalized, "tokens": w.dtype, "order": w.order,
               "ms_per_step": ms, "value": tok, "unit": "tokens/s", "steps": steps}
        path, n_launch = (hla.hla3_forward_path(w.B, w.H, w.n, w.d, w.dv, masked=w.masked, normalized=w.normalized,
                                                chunk=w.chunk, dtype=tq.dtype) if third else (None, 1))
        if third and path == 2:
            gbs = fwd_bytes(w) / (ms * 1e-3) / 1e9
            tc_traffic, tc_how = traffic("hla3_tc_kernels", w.name, w.n)
            issued = hla3_tc_issued_flops(w)
            cfg["roofline"] = {
                "bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak,
                "traffic": tc_traffic, "traffic_how": tc_how, "algorithmic_bytes": fwd_bytes(w),
                "algorithmic_flops": hla3_tc_flops(w),
                "roofline_us": max(fwd_bytes(w) / (hbm_peak * 1e9), hla3_tc_flops(w) / (tc_peak * 1e12)) * 1e6,
                "tensor_view": {"achieved": hla3_tc_flops(w) / (ms * 1e-3) / 1e12, "peak": tc_peak,
                                "unit": "TFLOP/s", "frac": hla3_tc_flops(w) / (ms * 1e-3) / 1e12 / tc_peak},
                "issued_tensor": {"flops": issued, "achieved": issued / (ms * 1e-3) / 1e12, "peak": tc_peak,
                                  "unit": "TFLOP/s", "frac": issued / (ms * 1e-3) / 1e12 / tc_peak,
                                  "note": "bf16 hi.hi + hi.lo + lo.hi products on full 128-row tiles"},
                "peak_kind": "measured",
                "kernel": "hla3_tc_kernel (tcgen05 pre-pass and sweep) + hla3_tc_fixup_kernel"}
            cfg["path"] = "tensor cores"
            cfg["launches"] = steps * n_launch
        elif third:
            tf = hla3_flops(w) / (ms * 1e-3) / 1e12
            h3_traffic, h3_how = traffic("c3_kernels", w.name, w.n)
            cfg["roofline"] = {"bound": "alu", "achieved": tf, "peak": alu_peak(), "unit": "TFLOP/s",
                               "frac": tf / alu_peak(), "traffic": h3_traffic, "traffic_how": h3_how,
                               "algorithmic_bytes": fwd_bytes(w), "flops": hla3_flops(w),
                               "peak_kind": "derived (152 SMs x 128 fp32 lanes x 2 x 2.07 GHz)",
                               "kernel": "c3_local/bracket/out (fp32 CUDA cores)"}
            cfg["path"] = "fp32 CUDA cores"
            cfg["launches"] = steps * n_launch
        else:
            cfg["roofline"] = roofline_record(w, ms, hbm_peak, tc_peak, "measured", None, None, "hla2_fused_kernel")
            cfg["launches"] = steps
        res.append(cfg)
        del tq, tk, tv, out, ws
    return res


def profile_case(hla, dev, case):
    """A few launches of one kernel family on a case small enough for an ncu capture (state or
    inputs of a few hundred MB, larger than L2): the decode steps on B64 H32 d128 states (random
    values), the AHLA forward on ahla_bf16, the backward on mid_bf16."""
    import torch
    torch.manual_seed(0)
    if case in ("sde_step", "tuple_step", "ahla_step"):
        B, H, d, dv = 64, 32, 128, 128
        q = (torch.randn(B, H, d, device=dev) / d ** 0.5).to(torch.bfloat16)
        k = (torch.randn(B, H, d, device=dev) / d ** 0.5).to(torch.bfloat16)
        v = torch.randn(B, H, dv, device=dev).to(torch.bfloat16)
        floats = {"sde_step": hla.hla2_sde_state_floats, "tuple_step": hla.hla2_state_floats,
                  "ahla_step": hla.ahla_state_floats}[case](d, dv)
        st = torch.randn(B, H, floats, device=dev)
        step = {"sde_step": lambda: hla.hla2_step_sde(q, k, v, st), "tuple_step": lambda: hla.hla2_step(q, k, v, st),
                "ahla_step": lambda: hla.ahla_step(q, k, v, st)}[case]
        for _ in range(4):
            step()
    else:
        w = hla_inputs.WORKLOADS["ahla_bf16" if case == "ahla_fwd" else "mid_bf16"]
        q, k, v = (hla_inputs.as_torch(x, w.dtype, dev) for x in hla_inputs.make_workload(w))
        for _ in range(2):
            if case == "ahla_fwd":
                hla.ahla_forward(q, k, v, chunk=w.chunk)
            else:
                hla.hla2_backward(q, k, v, torch.randn_like(v), chunk=w.chunk)
    torch.cuda.synchronize()
    print(json.dumps({"profile_case": case, "ok": True}))


def bwd_flops(w, C=None, W=None):
    """Algorithmic FLOPs of one masked second-order backward (chunk C, value width W: dv + 1
    on the CUDA-core kernels, which always carry the denominator column; dv on the tensor-core
    kernel, plain output, C = 128): the forward recompute (as fwd_flops) plus, per token-head,
    2 [C W / 2 (P) + C d / 2 (P^T Q) + d W (V' Gam) + C d / 2 (Y K^T) + C W / 2 (T^T G')
       + d W (X Gam^T) + C d / 2 (P X) + 2 d W (G' D^T, Gam, M) + d^2 (Y S_p) + C d / 2 (B K)
       + d^2 (K Lam) + C d (W^T Y, B^T Q) + 2 d^2 (Lam) + 2 d^2 W / C (scans)]."""
    d = w.d
    C = min(w.chunk, 32 if max(w.d, w.dv) == 128 else 64) if C is None else C
    W = w.dv + 1 if W is None else W
    per = 2 * (C * W / 2 + C * d / 2 + d * W + C * d / 2 + C * W / 2 + d * W + C * d / 2 + 2 * d * W + d * d
               + C * d / 2 + d * d + C * d + 2 * d * d + 2 * d * d * W / C)
    return fwd_flops(w) + w.BH * w.n * per


def bwd_tc_issued_flops(w):
    """Tensor FLOPs the tensor-core backward issues (bf16 hi/lo pairs, full 128-row tiles): per
    128-token tile 48 K = 16 steps at N = 128 and 204 at N = 64 (forward sweep 4 and 44, reverse
    sweep 44 and 160)."""
    M = (w.n + 127) // 128
    step = lambda N: 2 * 128 * N * 16
    return w.BH * M * (48 * step(128) + 204 * step(64))


def bench_backward(hla, dev, stream, world, hbm_peak, tc_peak, steps=10, warmup=3):
    """hla2_backward on mid_bf16 (B8 H16 n2048 d64 bf16, chunk 64), CUDA events on the launching stream."""
    import torch
    w = hla_inputs.WORKLOADS["mid_bf16"]
    q, k, v = hla_inputs.make_workload(w)
    g = hla_inputs.round_to(np.random.default_rng(w.seed + 1).standard_normal((w.B, w.H, w.n, w.dv)), w.dtype)
    tq, tk, tv, tg = (hla_inputs.as_torch(x, w.dtype, dev) for x in (q, k, v, g))
    ws = hla.alloc_workspace(hla.hla2_backward_workspace_bytes(w.B, w.H, w.n, w.d, w.dv, w.chunk, tq.dtype), dev)

    def call():
        hla.hla2_backward(tq, tk, tv, tg, normalized=w.normalized, eps=hla_inputs.EPS, chunk=w.chunk, workspace=ws,
                          stream=stream)
    for _ in range(warmup):
        call()
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / steps, world)
    rec = {"workload": w.name, "B": w.B, "H": w.H, "n": w.n, "d": w.d, "dv": w.dv, "chunk": w.chunk,
           "tokens": w.dtype, "ms_per_step": ms, "value": w.B * w.n * world / (ms * 1e-3), "unit": "tokens/s",
           "steps": steps}
    if hla.hla2_backward_path(w.B, w.H, w.n, w.d, w.dv, normalized=w.normalized, chunk=w.chunk, dtype=tq.dtype) == 1:
        # q, k, v, dout read once, dq, dk, dv written once (the checkpoints are the kernel's own traffic)
        nbytes = w.BH * w.n * (3 * w.d + 4 * w.dv) * (2 if w.dtype == "bf16" else 4)
        flops = bwd_flops(w, C=128, W=w.dv)
        t_b, t_f = nbytes / (hbm_peak * 1e9), flops / (tc_peak * 1e12)
        gbs, tfl = nbytes / (ms * 1e-3) / 1e9, flops / (ms * 1e-3) / 1e12
        hbm = {"achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak}
        ten = {"achieved": tfl, "peak": tc_peak, "unit": "TFLOP/s", "frac": tfl / tc_peak}
        bound, main, other = ("hbm", hbm, ten) if t_b >= t_f else ("tensor", ten, hbm)
        tr, tr_how = traffic("bwd_tc_kernel", w.name, w.n)
        issued = bwd_tc_issued_flops(w)
        rec["roofline"] = {"bound": bound, "achieved": main["achieved"], "peak": main["peak"], "unit": main["unit"],
                           "frac": main["frac"], "traffic": tr, "traffic_how": tr_how, "algorithmic_bytes": nbytes,
                           "flops": flops, "roofline_us": max(t_b, t_f) * 1e6, "peak_kind": "measured",
                           ("tensor_view" if bound == "hbm" else "hbm_view"): other,
                           "issued_tensor": {"flops": issued, "achieved": issued / (ms * 1e-3) / 1e12, "peak": tc_peak,
                                             "unit": "TFLOP/s", "frac": issued / (ms * 1e-3) / 1e12 / tc_peak},
                           "kernel": "bwd_tc_kernel (tcgen05, one launch)"}
        rec["path"] = "tensor cores"
        rec["launches"] = steps
    else:
        tf = bwd_flops(w) / (ms * 1e-3) / 1e12
        rec["roofline"] = {"bound": "alu", "achieved": tf, "peak": alu_peak(), "unit": "TFLOP/s",
                           "frac": tf / alu_peak(), "traffic": None, "flops": bwd_flops(w),
                           "peak_kind": "derived (152 SMs x 128 fp32 lanes x 2 x 2.07 GHz)",
                           "kernel": "bwd_fwd_local/fwd_scan/local1/scan/local2 (fp32 CUDA cores)"}
        rec["path"] = "fp32 CUDA cores"
        rec["launches"] = 5 * steps
    return rec


def bench_ahla(hla, dev, stream, hbm_peak, world, steps=20, warmup=3, decode_steps=256, tc_peak=None):
    """AHLA: the forward on ahla_bf16 (B8 H16 n2048 d64 bf16, chunk 64) and the decode step on
    ahla_decode_bf16 (B64 H32 d128, state built from a 4096-token prefix), CUDA events on the
    launching stream."""
    import torch
    res = {}
    w = hla_inputs.WORKLOADS["ahla_bf16"]
    q, k, v = hla_inputs.make_workload(w)
    tq, tk, tv = (hla_inputs.as_torch(x, w.dtype, dev) for x in (q, k, v))
    out = torch.empty((w.B, w.H, w.n, w.dv), dtype=tq.dtype, device=dev)
    ws = hla.alloc_workspace(hla.ahla_workspace_bytes(w.B, w.H, w.n, w.d, w.dv, w.chunk, tq.dtype), dev)

    def call():
        hla.ahla_forward(tq, tk, tv, out, normalized=w.normalized, eps=hla_inputs.EPS, chunk=w.chunk, workspace=ws,
                         stream=stream)
    for _ in range(warmup):
        call()
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / steps, world)
    tensor_path = hla.ahla_forward_path(w.B, w.H, w.n, w.d, w.dv, normalized=w.normalized, chunk=w.chunk,
                                        dtype=tq.dtype) == 1
    tf = ahla_flops(w) / (ms * 1e-3) / 1e12
    gbs = fwd_bytes(w) / (ms * 1e-3) / 1e9
    if tensor_path:  # the slower of the bytes at HBM bandwidth and the FLOPs at the bf16 tensor peak
        t_bytes, t_flops = fwd_bytes(w) / (hbm_peak * 1e9), ahla_flops(w) / (tc_peak * 1e12)
        hbm = {"achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak}
        ten = {"achieved": tf, "peak": tc_peak, "unit": "TFLOP/s", "frac": tf / tc_peak}
        main, other, bound = (hbm, ten, "hbm") if t_bytes >= t_flops else (ten, hbm, "tensor")
        roof = dict(main, bound=bound, traffic=None, flops=ahla_flops(w), algorithmic_bytes=fwd_bytes(w),
                    kernel="ahla_tc_kernel (tcgen05, one launch)")
        roof["tensor_view" if bound == "hbm" else "hbm_view"] = other
    else:
        roof = {"bound": "alu", "achieved": tf, "peak": alu_peak(), "unit": "TFLOP/s", "frac": tf / alu_peak(),
                "traffic": None, "flops": ahla_flops(w),
                "peak_kind": "derived (152 SMs x 128 fp32 lanes x 2 x 2.07 GHz)",
                "kernel": "ahla_local/scan/out (fp32 CUDA cores)",
                "hbm_view": {"achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak}}
    res["forward"] = {"workload": w.name, "B": w.B, "H": w.H, "n": w.n, "d": w.d, "dv": w.dv, "chunk": w.chunk,
                      "tokens": w.dtype, "ms_per_step": ms, "value": w.B * w.n * world / (ms * 1e-3),
                      "unit": "tokens/s", "steps": steps, "roofline": roof,
                      "launches": (1 if tensor_path else 3) * steps}
    del tq, tk, tv, out, ws
    # decode step
    w = hla_inputs.WORKLOADS["ahla_decode_bf16"]
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w, steps=decode_steps)
    st = torch.zeros((w.B, w.H, hla.ahla_state_floats(w.d, w.dv)), dtype=torch.float32, device=dev)
    tq, tk, tv = (hla_inputs.as_torch(x, w.dtype, dev) for x in (qp, kp, vp))
    hla.ahla_forward(tq, tk, tv, chunk=w.chunk, state_out=st)
    del tq, tk, tv, qp, kp, vp
    toks = [[hla_inputs.as_torch(x[s], w.dtype, dev) for x in (qs, ks, vs)] for s in range(decode_steps)]
    out = torch.empty((w.B, w.H, w.dv), dtype=toks[0][0].dtype, device=dev)
    st0 = st.clone()
    for s in range(min(3, decode_steps)):
        hla.ahla_step(*toks[s], st, out, normalized=w.normalized, eps=hla_inputs.EPS)
    st.copy_(st0)
    del st0
    torch.cuda.synchronize()
    barrier(world)
    e0.record(stream)
    for s in range(decode_steps):
        hla.ahla_step(*toks[s], st, out, normalized=w.normalized, eps=hla_inputs.EPS, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    us = max_over_ranks(e0.elapsed_time(e1) * 1e3 / decode_steps, world)
    gbs = ahla_dec_bytes(w) / (us * 1e-6) / 1e9
    res["decode"] = {"workload": w.name, "B": w.B, "H": w.H, "d": w.d, "dv": w.dv, "prefix": w.decode_prefix,
                     "steps": decode_steps, "us_per_step": us, "value": gbs * world, "unit": "GB/s",
                     "tokens_per_s": w.B * world / (us * 1e-6),
                     "roofline": {"bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s",
                                  "frac": gbs / hbm_peak, "traffic": None, "algorithmic_bytes": ahla_dec_bytes(w),
                                  "kernel": "ahla_step_staged_kernel"},
                     "launches": decode_steps}
    return res


def bench_decode(hla, dev, stream, steps, hbm_peak, world):
    import torch
    w = DEC
    (qp, kp, vp), (qs, ks, vs) = hla_inputs.make_decode(w, steps=steps)
    st = torch.zeros((w.B, w.H, hla.hla2_state_floats(w.d, w.dv)), dtype=torch.float32, device=dev)
    tq, tk, tv = (hla_inputs.as_torch(x, w.dtype, dev) for x in (qp, kp, vp))
    hla.hla2_forward(tq, tk, tv, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS, chunk=w.chunk,
                     state_out=st)
    del tq, tk, tv
    toks = [[hla_inputs.as_torch(x[s], w.dtype, dev) for x in (qs, ks, vs)] for s in range(steps)]
    out = torch.empty((w.B, w.H, w.dv), dtype=toks[0][0].dtype, device=dev)
    st_init = st.clone()
    for s in range(min(3, steps)):  # warm-up on a copy, then restore
        hla.hla2_step(*toks[s], st, out, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS)
    st.copy_(st_init)
    torch.cuda.synchronize()
    barrier(world)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(steps):
        hla.hla2_step(*toks[s], st, out, masked=w.masked, normalized=w.normalized, eps=hla_inputs.EPS,
                      stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    us = max_over_ranks(e0.elapsed_time(e1) * 1e3 / steps, world)
    gbs = dec_bytes(w) / (us * 1e-6) / 1e9
    dec_traffic, dec_how = traffic("step2_kernel", "decode_bf16", 0)
    res = {"workload": "decode_bf16", "B": w.B, "H": w.H, "d": w.d, "dv": w.dv, "prefix": w.decode_prefix,
           "steps": steps, "us_per_step": us, "value": gbs * world, "unit": "GB/s",
           "tokens_per_s": w.B * world / (us * 1e-6),
           "roofline": {"bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak,
                        "traffic": dec_traffic, "traffic_how": dec_how, "algorithmic_bytes": dec_bytes(w),
                        "kernel": "step2_kernel"},
           "launches": steps}

    # the same steps on the (S, D, e) state (D = S C - G, e = S m - h): same outputs, a third fewer bytes
    st.copy_(st_init)
    sde = hla.hla2_state_to_sde(st, w.d, w.dv)
    del st, st_init
    torch.cuda.synchronize()
    for s in range(min(3, steps)):
        hla.hla2_step_sde(*toks[s], sde, out, normalized=w.normalized, eps=hla_inputs.EPS)
    torch.cuda.synchronize()
    barrier(world)
    e0.record(stream)
    for s in range(steps):
        hla.hla2_step_sde(*toks[s], sde, out, normalized=w.normalized, eps=hla_inputs.EPS, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    us2 = max_over_ranks(e0.elapsed_time(e1) * 1e3 / steps, world)
    gbs2 = dec_sde_bytes(w) / (us2 * 1e-6) / 1e9
    sde_traffic, sde_how = traffic("step2_kernel_sde", "decode_bf16", 0)
    res["sde"] = {"state": "(S, D, e)", "us_per_step": us2, "value": gbs2 * world, "unit": "GB/s",
                  "tokens_per_s": w.B * world / (us2 * 1e-6),
                  "roofline": {"bound": "hbm", "achieved": gbs2, "peak": hbm_peak, "unit": "GB/s",
                               "frac": gbs2 / hbm_peak, "traffic": sde_traffic, "traffic_how": sde_how,
                               "algorithmic_bytes": dec_sde_bytes(w), "kernel": "step2_kernel (S, D, e)"},
                  "launches": steps}
    res["launches"] += steps
    return res


if __name__ == "__main__":
    main()
