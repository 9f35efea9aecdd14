#!/usr/bin/env python3
"""Throughput of the four fused composite sparse expressions on GB300.

One step = one pass of the whole hot path: the four fused expressions of the
SparseLNR benchmark set (Sec. 6.2) at their full synthetic sizes,
  <SDDMM,SpMM>  R-MAT 100k x 100k, 2M nnz, L = K = 64
  <SpMM,GEMM>   R-MAT 2^20 x 2^20, 16.8M nnz, K = L = 128
  MTTKRP        CSF 10k^3, 10M nnz, Zipf(1.2) slices, L = 32
  <SpTTM,SpTTM> CSF 5k^3, 20M nnz, power-law fibers (mean 8), L = M = 64
each through the C ABI with inputs resident in HBM.  L2 is flushed (a write of
2x its size) before every expression, outside the timed events.  Metric:
useful GFLOP/s (the flops the fused schedule must do, Sec. 3.1.3 / 6.2
complexity) over the step; per-expression GFLOP/s, time and achieved HBM
GB/s (minimum bytes / time) are reported beside it.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl slnr|reference]

--suite next times the three further expressions of Sec. 6.2 instead
(<SDDMM,SpMM,GEMM> on the <SDDMM,SpMM> graph with k,l,m = 64; <MTTKRP,GEMM>
on the MTTKRP tensor with rank 32 and m = 64; <SpMMH,GEMM> on the 2^20 R-MAT
graph with j,l = 128), with the same JSON line.

Under torchrun each rank runs an independent replica on its own GPU (the
expressions need no exchange between GPUs); value = all ranks' flops / the
slowest rank's time.  --impl reference times the CPU oracle instead (on rank 0).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as wl  # noqa: E402

BENCH_CONFIGS = (1, 2, 3, 4)   # full-size workloads timed in one step (index 0 is the small parity case)
CSR_OPS = ("spmm_gemm", "sddmm_spmm", "sddmm_spmm_gemm", "spmmh_gemm")


# ---------------------------------------------------------------------------
# algorithmic counts

def _distinct(a) -> int:
    if a.shape[0] == 0:
        return 0
    return int(np.unique(a).shape[0])


def row_sizes(w):
    """Work units of each expression's output rows and their nonzero counts."""
    if w.op in CSR_OPS:
        return np.diff(w.B.pos).astype(np.int64)
    if w.op == "spttm_ttm":
        return np.diff(w.B.pos3).astype(np.int64)
    sizes = np.zeros(w.B.dims[0], np.int64)
    fib = np.diff(w.B.pos3).astype(np.int64)
    if w.B.nfibers:
        sizes[w.B.crd1] = np.add.reduceat(fib, w.B.pos2[:-1]) if w.B.nslices else 0
    return sizes


def row_flops(w) -> np.ndarray:
    """Useful flops per output row under the fused schedule (Sec. 6.2 complexities)."""
    d = w.dims
    if w.op == "spmm_gemm":      # 2 nnz K + 2 K L per non-empty row
        n = np.diff(w.B.pos).astype(np.int64)
        return 2 * n * d["K"] + 2 * (n > 0) * d["K"] * d["L"]
    if w.op == "sddmm_spmm":     # per nonzero: dot (2L), scale (1), axpy (2K)
        n = np.diff(w.B.pos).astype(np.int64)
        return n * (2 * d["L"] + 1 + 2 * d["K"])
    if w.op in ("mttkrp", "mttkrp_gemm"):  # 2 nnz L + 2 nfibers L per slice (+ 2 L M per slice)
        L = d["L"]
        f = np.zeros(w.B.dims[0], np.int64)
        if w.B.nslices:
            pos3 = w.B.pos3.astype(np.int64)
            nnz_s = np.diff(pos3[w.B.pos2])           # nonzeros per slice (0 for a slice without fibers)
            nfib_s = np.diff(w.B.pos2).astype(np.int64)
            f[w.B.crd1] = 2 * nnz_s * L + 2 * nfib_s * L
            if w.op == "mttkrp_gemm":
                f[w.B.crd1] += 2 * L * d["M"]
        return f
    if w.op == "sddmm_spmm_gemm":  # per nonzero: dot (2K), scale (1), axpy (2L); 2 L M per non-empty row
        n = np.diff(w.B.pos).astype(np.int64)
        return n * (2 * d["K"] + 1 + 2 * d["L"]) + 2 * (n > 0) * d["L"] * d["M"]
    if w.op == "spmmh_gemm":     # per nonzero: Hadamard product and axpy (3J); 2 J L per non-empty row
        n = np.diff(w.B.pos).astype(np.int64)
        return 3 * n * d["J"] + 2 * (n > 0) * d["J"] * d["L"]
    if w.op == "spttm_ttm":      # 2 nnz L + 2 L M per fiber
        n = np.diff(w.B.pos3).astype(np.int64)
        return 2 * n * d["L"] + 2 * d["L"] * d["M"]
    raise ValueError(w.op)


def useful_flops(w) -> int:
    return int(row_flops(w).sum())


def min_bytes(w, referenced_only: bool = True) -> int:
    """Bytes an ideal evaluation moves: sparse structure and values once, each
    dense operand row that is actually referenced once (every row of every
    dense input with referenced_only=False, the count that names every dense
    input once), every output once."""
    if not referenced_only:
        return min_bytes_all_rows(w)
    d, B = w.dims, w.B
    if w.op == "spmm_gemm":
        K, L = d["K"], d["L"]
        return 4 * (B.nrows + 1) + 8 * B.nnz + 4 * K * _distinct(B.crd) + 4 * K * L + 4 * B.nrows * L
    if w.op == "sddmm_spmm":
        K, L = d["K"], d["L"]
        nonempty = int(np.count_nonzero(np.diff(B.pos)))
        cols = _distinct(B.crd)
        return 4 * (B.nrows + 1) + 8 * B.nnz + 4 * L * nonempty + 4 * (L + K) * cols + 4 * B.nrows * K
    if w.op == "sddmm_spmm_gemm":
        K, L, M = d["K"], d["L"], d["M"]
        nonempty = int(np.count_nonzero(np.diff(B.pos)))
        cols = _distinct(B.crd)
        return 4 * (B.nrows + 1) + 8 * B.nnz + 4 * K * nonempty + 4 * (K + L) * cols + 4 * L * M + 4 * B.nrows * M
    if w.op == "spmmh_gemm":
        J, L = d["J"], d["L"]
        return 4 * (B.nrows + 1) + 8 * B.nnz + 8 * J * _distinct(B.crd) + 4 * J * L + 4 * B.nrows * L
    structure = 8 + 4 * B.nslices + 4 * (B.nslices + 1) + 4 * B.nfibers + 4 * (B.nfibers + 1) + 8 * B.nnz
    if w.op == "mttkrp_gemm":
        L, M = d["L"], d["M"]
        return structure + 4 * L * (_distinct(B.crd2) + _distinct(B.crd3)) + 4 * L * M + 4 * B.dims[0] * M
    if w.op == "mttkrp":
        L = d["L"]
        return structure + 4 * L * (_distinct(B.crd2) + _distinct(B.crd3)) + 4 * B.dims[0] * L
    if w.op == "spttm_ttm":
        L, M = d["L"], d["M"]
        out_index = 8 + 4 * B.nslices + 4 * (B.nslices + 1) + 4 * B.nfibers
        return structure + 4 * L * _distinct(B.crd3) + 4 * L * M + 4 * B.nfibers * M + out_index
    raise ValueError(w.op)


def min_bytes_all_rows(w) -> int:
    """min_bytes with every row of every dense input read once."""
    B = w.B
    dense = sum(int(v.size) * 4 for v in w.dense.values())
    if w.op in CSR_OPS:
        sparse = 4 * (B.nrows + 1) + 8 * B.nnz
    else:
        sparse = 8 + 4 * B.nslices + 4 * (B.nslices + 1) + 4 * B.nfibers + 4 * (B.nfibers + 1) + 8 * B.nnz
    d = w.dims
    if w.op in CSR_OPS:
        width = {"spmm_gemm": "L", "sddmm_spmm": "K", "sddmm_spmm_gemm": "M", "spmmh_gemm": "L"}[w.op]
        out = 4 * B.nrows * d[width]
    elif w.op == "spttm_ttm":
        out = 4 * B.nfibers * d["M"] + 8 + 4 * B.nslices + 4 * (B.nslices + 1) + 4 * B.nfibers
    else:
        out = 4 * B.dims[0] * (d["M"] if w.op == "mttkrp_gemm" else d["L"])
    return sparse + dense + out


def consumer_flops(w) -> int:
    """Flops of the dense consumer contraction (the tensor-core part where it
    runs on TF32): 2 K L per non-empty row of <SpMM,GEMM>, 2 L M per fiber of
    <SpTTM,SpTTM>, 2 J L per non-empty row of <SpMMH,GEMM>; 0 otherwise."""
    d = w.dims
    if w.op in ("spmm_gemm", "spmmh_gemm"):
        n = np.diff(w.B.pos)
        k = d["K"] if w.op == "spmm_gemm" else d["J"]
        return int(2 * np.count_nonzero(n) * k * d["L"])
    if w.op == "spttm_ttm":
        return int(2 * w.B.nfibers * d["L"] * d["M"])
    return 0


def gather_bytes(w) -> int:
    """Bytes the fused producers read as whole gathered rows, one (or two)
    per nonzero and one per fiber where a fiber scales a row: nnz 4K for
    <SpMM,GEMM>, nnz 4L for <SpTTM,SpTTM>, nnz 8J for <SpMMH,GEMM>, nnz 4(L+K)
    for <SDDMM,SpMM>, nnz 4(K+L) for <SDDMM,SpMM,GEMM>, (nnz + nfibers) 4L for
    MTTKRP.  Almost all of them hit in L2; their rate, not HBM's, is the
    realistic ceiling of the gathering kernels."""
    d, B = w.dims, w.B
    per_nnz = {"spmm_gemm": lambda: 4 * d["K"], "spttm_ttm": lambda: 4 * d["L"], "spmmh_gemm": lambda: 8 * d["J"],
               "sddmm_spmm": lambda: 4 * (d["L"] + d["K"]), "sddmm_spmm_gemm": lambda: 4 * (d["K"] + d["L"]),
               "mttkrp": lambda: 4 * d["L"], "mttkrp_gemm": lambda: 4 * d["L"]}[w.op]()
    extra = 4 * d["L"] * B.nfibers if w.op in ("mttkrp", "mttkrp_gemm") else 0
    return int(per_nnz * B.nnz + extra)


def gather_row_width(w) -> int:
    """Width (fp32 values) of the rows the producers gather, as a power of two
    in [4, 128] for the gather peak kernel."""
    d = w.dims
    width = {"spmm_gemm": "K", "spttm_ttm": "L", "spmmh_gemm": "J", "sddmm_spmm": "K", "sddmm_spmm_gemm": "L",
             "mttkrp": "L", "mttkrp_gemm": "L"}[w.op]
    v = 4
    while v * 2 <= min(d[width], 128):
        v *= 2
    return v


# sources whose code runs outside the measured calls: the peak kernels, the
# entry point without a workspace, the perfect-loop-nest comparator
OUTSIDE_MEASURED = ("peaks.cu", "noalloc.cu", "original.cu")


def kernel_source_hash() -> str:
    """Hash of the kernel sources that run inside the measured calls."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2205_11622_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")) and name not in OUTSIDE_MEASURED:
            h.update(name.encode())
            h.update(open(os.path.join(csrc, name), "rb").read())
    return h.hexdigest()[:16]


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        j = json.load(open(p))
        return float(j["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def ncu_traffic(expr_name: str):
    """DRAM bytes per call of an expression from the committed ncu summary, if it
    was taken on the current kernel sources (else None)."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    j = json.load(open(p))
    if j.get("kernel_source_hash") != kernel_source_hash():
        return None
    e = j.get("expressions", {}).get(expr_name)
    return None if e is None else float(e["dram_bytes_per_call"])


# ---------------------------------------------------------------------------
# clocks during the timed region

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_uuid: str | None):
        self.samples, self.proc, self.thread = [], None, None
        self.uuid = gpu_uuid

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                self.samples.append(parts)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["clocks not sampled"]}
        sm = [float(s[1]) for s in self.samples if s[1].replace(".", "").isdigit()]
        mx = [float(s[2]) for s in self.samples if s[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for s in self.samples for n, v in zip(names, s[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.samples)}


# ---------------------------------------------------------------------------
# CPU oracle on a bounded sample (the cpu_baseline leg and the reference arm)

def oracle_sample(w, flop_budget: float, seed: int):
    """Seeded uniform sample of output rows whose useful flops reach flop_budget."""
    rf = row_flops(w)
    rng = np.random.default_rng(seed)
    order = rng.permutation(rf.shape[0])
    cum = np.cumsum(rf[order])
    n = int(np.searchsorted(cum, flop_budget)) + 1
    rows = np.sort(order[:max(1, min(n, order.shape[0]))]).astype(np.int32)
    return rows, int(rf[rows].sum())


def time_oracle(ws, flop_budget: float, seed: int = 11):
    import oracle
    orc = oracle.get()
    secs, flops, parts = 0.0, 0, []
    for w in ws:
        rows, f = oracle_sample(w, flop_budget, seed)
        t0 = time.perf_counter()
        orc.run(w, rows=rows)
        dt = time.perf_counter() - t0
        secs += dt
        flops += f
        parts.append(f"{w.name}: {rows.shape[0]} rows, {f / 1e9:.2f} GFLOP, {dt:.2f} s")
    return flops, secs, "; ".join(parts)


# ---------------------------------------------------------------------------

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def job_throughput(step_ms, step_flops, world, pg=None, device=None):
    """Whole-job throughput of replicas: every rank runs the same step on its
    own GPU, the job takes as long as the slowest rank (max over ranks of the
    step time), and the job does world x step_flops of useful work in that
    time.  Returns (max step ms, GFLOP/s).  pg is torch.distributed (or None
    for one process); device is where the reduction tensor lives (a CUDA
    device under NCCL, the CPU under gloo)."""
    if pg is not None:
        import torch
        t = torch.tensor([float(step_ms)], dtype=torch.float64, device=device)
        pg.all_reduce(t, op=pg.ReduceOp.MAX)
        step_ms = float(t.item())
        pg.barrier()
    return step_ms, world * step_flops / (step_ms / 1e3) / 1e9


def run_reference(args, rank, world):
    if rank != 0:
        return 0
    ws = select_workloads(args)
    budget = args.ref_gflop_per_expr * 1e9
    times, flops_total, sample = [], 0, ""
    for step in range(args.warmup + args.steps):
        flops, secs, sample = time_oracle(ws, budget, seed=100 + step)
        if step >= args.warmup:
            times.append(secs)
            flops_total += flops
    secs = sum(times)
    value = flops_total / secs / 1e9
    line = {
        "impl": "reference", "metric": metric_name(args), "value": round(value, 4),
        "unit": "GFLOP/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * secs / args.steps, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_block(ws),
        "cpu_baseline": {"value": round(value, 4), "unit": "GFLOP/s", "cores": 1, "kind": "oracle",
                         "sample": "per step, a seeded uniform sample of output rows of each expression worth "
                                   f"{args.ref_gflop_per_expr} GFLOP (oracle computes value and magnitude "
                                   f"companion in fp64, single thread); last step: {sample}"},
        "e2e": {"value": round(value, 4), "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def select_workloads(args):
    if args.suite == "next":
        ws = [wl.next_full(i, args.scale) for i in range(len(wl.NEXT_OPS))]
    else:
        ws = [wl.full(i, args.scale) for i in BENCH_CONFIGS]
    ws = [w for w in ws if args.expr in w.name]
    if not ws:
        raise SystemExit(f"no workload matches --expr {args.expr!r}")
    return ws


def metric_name(args):
    if args.suite == "next":
        return "useful GFLOP/s (3 further fused sparse expressions of Sec. 6.2)"
    return "useful GFLOP/s (4 fused sparse expressions)"


def config_block(ws):
    return {
        "workload": " + ".join(w.name for w in ws),
        "expressions": {w.name: w.recipe for w in ws},
        "l2": "flushed before every expression by writing a buffer of 2x the L2 size (outside the timed events)",
        "variant": "fused", "allow_tf32": True,
        "parallelism": "replicas (one independent full step per GPU)",
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["slnr", "reference"], default="slnr")
    ap.add_argument("--variant", choices=["fused", "unfused"], default="fused")
    ap.add_argument("--no-tf32", action="store_true")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--skip-cpu", action="store_true")
    ap.add_argument("--cpu-gflop-per-expr", type=float, default=4.0)
    ap.add_argument("--ref-gflop-per-expr", type=float, default=1.0)
    ap.add_argument("--expr", default="", help="only the expressions whose name contains this (profiling)")
    ap.add_argument("--scale", type=float, default=1.0, help="shrink the workloads (profiling captures)")
    ap.add_argument("--sweep-k", default="", help="sweep: only these K (comma list; default all)")
    ap.add_argument("--sweep-l", default="", help="sweep: only these L (comma list; default all)")
    ap.add_argument("--original", action="store_true",
                    help="sweep: also time the perfect loop nest (O(nnz K L); use with --scale, Fig. 8b)")
    ap.add_argument("--suite", choices=["main", "next", "sweep"], default="main",
                    help="main: the four benchmark expressions (the step); next: <SDDMM,SpMM,GEMM>, "
                         "<MTTKRP,GEMM>, <SpMMH,GEMM> at full size; sweep: <SpMM,GEMM> fused and unfused "
                         "over the inner dimensions K, L (Sec. 6.3)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank, world, local = dist_env()
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.suite == "sweep":
        return run_sweep(args, rank, world, local)

    import torch

    import paper_2205_11622_gb300 as slnr

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    slnr.build()
    slnr.lib()
    allow_tf32 = not args.no_tf32

    ws = select_workloads(args)
    flops = [useful_flops(w) for w in ws]
    mbytes = [min_bytes(w) for w in ws]

    # device-resident inputs, preallocated outputs and workspaces
    def upload(w):
        if w.op in CSR_OPS:
            B = slnr.DeviceCSR.from_host(w.B, dev)
        else:
            B = slnr.DeviceCSF3.from_host(w.B, dev)
        dense = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dev) for k, v in w.dense.items()}
        return B, dense

    dev_inputs = [upload(w) for w in ws]
    wspaces = [slnr.Workspace(device=dev) for _ in ws]
    outs = [None] * len(ws)

    def call(i, out=None, on_stream=None):
        w = ws[i]
        B, dense = dev_inputs[i]
        return slnr.run(w.op, B, dense, out=out, variant=args.variant, allow_tf32=allow_tf32, workspace=wspaces[i],
                        stream=on_stream)

    for i in range(len(ws)):
        outs[i] = call(i)
    torch.cuda.synchronize()

    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_buf = torch.empty(max(2 * l2, 64 << 20), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def one_step(hook):
        """One call of every expression (L2 flushed before each); with hook, the
        library's per-launch event hook is on and its kernel times are read
        back.  The timed steps run without it: its event records sit between
        the launches."""
        slnr.timing_enable(hook)
        per_expr, per_kernel, launches = [], [], 0
        for i in range(len(ws)):
            flush_buf.fill_(i & 0xFF)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            call(i, out=outs[i])
            b.record(stream)
            b.synchronize()
            per_expr.append(a.elapsed_time(b))
            per_kernel.append(slnr.timing_read() if hook else [])
            launches += slnr.timing_launches()  # this library's kernels in the call
        slnr.timing_enable(False)
        return per_expr, per_kernel, launches

    for _ in range(args.warmup):
        one_step(False)
    torch.cuda.synchronize()
    if pg is not None:
        pg.barrier()
    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        uuid = None
    clocks = ClockSampler(uuid)
    clocks.start()
    time.sleep(0.5)
    torch.cuda.synchronize()
    expr_ms = [[] for _ in ws]
    gpu_launches = 0
    for _ in range(args.steps):
        pe, _, nl = one_step(False)
        gpu_launches += nl
        for i in range(len(ws)):
            expr_ms[i].append(pe[i])
    torch.cuda.synchronize()
    time.sleep(0.3)
    clocks.stop()
    # the per-phase breakdown from as many steps again with the hook on,
    # outside the timed region
    kern_ms = [dict() for _ in ws]
    for _ in range(args.steps):
        _, pk, _ = one_step(True)
        for i in range(len(ws)):
            for name, ms in pk[i]:
                kern_ms[i][name] = kern_ms[i].get(name, 0.0) + ms
    mean_ms = [statistics.mean(x) for x in expr_ms]
    total_flops = sum(flops)
    step_ms, value = job_throughput(sum(mean_ms), total_flops, world, pg, dev)

    peak, peak_kind = measured_peaks()
    per_expression = {}
    for i, w in enumerate(ws):
        kms = {k: round(v / args.steps, 4) for k, v in kern_ms[i].items()}
        all_rows = min_bytes_all_rows(w)
        per_expression[w.name] = {
            "ms": round(mean_ms[i], 4), "gflops": round(flops[i] / (mean_ms[i] / 1e3) / 1e9, 2),
            "min_bytes": mbytes[i], "gbs": round(mbytes[i] / (mean_ms[i] / 1e3) / 1e9, 1),
            "hbm_frac": round(mbytes[i] / (mean_ms[i] / 1e3) / 1e9 / peak, 4),
            "min_bytes_all_rows": all_rows, "hbm_frac_all_rows": round(all_rows / (mean_ms[i] / 1e3) / 1e9 / peak, 4),
            "kernels_ms": kms, "useful_flops": flops[i], "in_headline": True}
    # config 1 (the small <SpMM,GEMM>, launch-bound): timed the same way, reported beside the step
    small = config1_latency(torch, slnr, dev, args, allow_tf32, flush_buf, stream)
    per_expression[small["name"]] = small["entry"]
    # the dominant call and, inside it, its dominant kernel (the timing hook's per-launch events)
    dom = int(np.argmax(mean_ms))
    dw = ws[dom]
    kname = max(kern_ms[dom], key=kern_ms[dom].get)
    k_ms = kern_ms[dom][kname] / args.steps
    achieved = mbytes[dom] / (k_ms / 1e3) / 1e9
    all_rows = min_bytes_all_rows(dw)
    traffic = ncu_traffic(dw.name)
    pk = slnr.peaks(stream, gather_width=gather_row_width(dw)) if rank == 0 else {}
    gb = gather_bytes(dw)
    cflops = consumer_flops(dw)
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": traffic,
                "kernel": f"{kname} of {dw.name} ({k_ms:.4f} ms per launch); achieved = the call's "
                          f"{mbytes[dom]} algorithmic bytes (each referenced dense row once) per launch",
                "peak_kind": f"{peak_kind} HBM copy bandwidth",
                "frac_call": round(mbytes[dom] / (mean_ms[dom] / 1e3) / 1e9 / peak, 4),
                "min_bytes_all_rows": all_rows,
                "frac_all_rows": round(all_rows / (k_ms / 1e3) / 1e9 / peak, 4),
                "compute": {"unit": "TFLOP/s", "tf32_peak_measured": round(pk.get("tf32_tflops", 0.0), 1),
                            "ffma_peak_measured": round(pk.get("ffma_tflops", 0.0), 1),
                            "tf32_achieved": round(cflops / (k_ms / 1e3) / 1e12, 2),
                            "tf32_frac": round(cflops / (k_ms / 1e3) / 1e12 / pk["tf32_tflops"], 4)
                            if pk.get("tf32_tflops") else None,
                            "note": "the dense consumer contraction of the dominant kernel (2 K L per non-empty "
                                    "row) against this library's own tcgen05 kind::tf32 peak kernel"},
                "gather": {"bytes": gb, "unit": "GB/s", "achieved": round(gb / (k_ms / 1e3) / 1e9, 1),
                           "l2_gather_peak_measured": round(pk.get("l2_gather_gbs", 0.0), 1),
                           "hbm_gather_peak_measured": round(pk.get("hbm_gather_gbs", 0.0), 1),
                           "frac_l2": round(gb / (k_ms / 1e3) / 1e9 / pk["l2_gather_gbs"], 4)
                           if pk.get("l2_gather_gbs") else None,
                           "row_width": gather_row_width(dw),
                           "note": "whole rows the producers gather (one per nonzero), against this library's own "
                                   "row-gather kernel on an L2-resident table (a quarter of L2) and on a 2 GB table"}}

    cpu = None
    if rank == 0 and world == 1 and not args.skip_cpu:
        cf, cs, sample = time_oracle(ws, args.cpu_gflop_per_expr * 1e9)
        cpu = {"value": round(cf / cs / 1e9, 4), "unit": "GFLOP/s", "cores": 1, "kind": "oracle",
               "sample": f"seeded uniform sample of output rows per expression (oracle computes value and "
                         f"magnitude companion in fp64, single thread): {sample}"}

    e2e = None
    if not args.skip_e2e:
        e2e = measure_e2e(torch, slnr, ws, dev_inputs, outs, call, stream, args.steps, total_flops, world, pg, dev)

    line = {
        "metric": metric_name(args), "value": round(value, 2), "unit": "GFLOP/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_ms, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32 (tf32 tensor-core contractions allowed)" if allow_tf32 else "f32",
        "data": "synthetic", "config": config_block(ws), "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": gpu_launches, "clocks": clocks.summary(), "per_expression": per_expression,
    }
    line["config"]["variant"] = args.variant
    line["config"]["allow_tf32"] = allow_tf32
    if rank == 0:
        print(json.dumps(line))
    if pg is not None:
        pg.destroy_process_group()
    return 0


SWEEP_DIMS = (16, 32, 64, 128, 256, 512)


def run_sweep(args, rank, world, local):
    """Sec. 6.3's case study on GB300: <SpMM,GEMM> on the 2^20-vertex R-MAT
    graph of the benchmark (16 nonzeros per row) for every inner-dimension
    pair K, L in SWEEP_DIMS, fused and unfused (TF32 allowed), kernel time per
    call (median, L2 flushed before each).  C (n x K) and D (K x L) are N(0,1)
    from a seed derived from K and L; the graph is generated once.  With
    --original, also the perfect loop nest i, j, k, l (Fig. 8b's comparator,
    O(nnz K L); 1 warm-up and up to 3 timed calls per cell)."""
    import torch

    import paper_2205_11622_gb300 as slnr
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    slnr.build()
    slnr.lib()
    n = int((1 << 20) * args.scale)
    seed = wl.SEED_BASE + 2
    base = wl.spmm_gemm_rmat(seed, n, 16, 16, 16)
    B = slnr.DeviceCSR.from_host(base.B, dev)
    flush = torch.empty(2 * torch.cuda.get_device_properties(dev).L2_cache_size, dtype=torch.uint8, device=dev)
    ws = slnr.Workspace(device=dev)
    stream = torch.cuda.current_stream()
    grid, t0 = [], time.time()
    ks = [int(x) for x in args.sweep_k.split(",")] if args.sweep_k else list(SWEEP_DIMS)
    ls = [int(x) for x in args.sweep_l.split(",")] if args.sweep_l else list(SWEEP_DIMS)
    for K in ks:
        rk = wl.Rng(seed ^ (K << 20))
        C = torch.from_numpy(wl.normal(rk, (n, K))).to(dev)
        for L in ls:
            rl = wl.Rng(seed ^ (K << 20) ^ (L << 8) ^ 1)
            D = torch.from_numpy(wl.normal(rl, (K, L))).to(dev)
            w = wl.Workload(f"spmm_gemm_rmat_k{K}_l{L}", "spmm_gemm", base.B, {}, {"K": K, "L": L})
            out = torch.empty((n, L), dtype=torch.float32, device=dev)
            res = {"K": K, "L": L, "useful_flops": useful_flops(w), "min_bytes": min_bytes(w)}
            for variant in ("fused", "unfused"):
                slnr.spmm_gemm(B, C, D, out=out, variant=variant, workspace=ws)
                ts = []
                for it in range(args.warmup + args.steps):
                    flush.fill_(it & 0xFF)
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    slnr.spmm_gemm(B, C, D, out=out, variant=variant, workspace=ws)
                    b.record(stream)
                    b.synchronize()
                    if it >= args.warmup:
                        ts.append(a.elapsed_time(b))
                res[f"{variant}_ms"] = round(statistics.median(ts), 4)
                if slnr.device_flags() != 0:
                    raise SystemExit(f"device flags {slnr.device_flags():#x} at K={K}, L={L}, {variant}")
            if args.original:  # the comparator: 1 warm-up, up to 3 timed calls
                ts = []
                for it in range(1 + min(3, args.steps)):
                    flush.fill_(it & 0xFF)
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    slnr.spmm_gemm_original(B, C, D, out=out)
                    b.record(stream)
                    b.synchronize()
                    if it >= 1:
                        ts.append(a.elapsed_time(b))
                res["original_ms"] = round(statistics.median(ts), 4)
                res["original_over_fused"] = round(res["original_ms"] / res["fused_ms"], 2)
            res["unfused_over_fused"] = round(res["unfused_ms"] / res["fused_ms"], 3)
            res["fused_gflops"] = round(res["useful_flops"] / res["fused_ms"] / 1e6, 1)
            res["fused_hbm_frac"] = round(res["min_bytes"] / res["fused_ms"] / 1e6 / measured_peaks()[0], 4)
            grid.append(res)
            del out, D
        del C
    best = max(grid, key=lambda r: r["unfused_over_fused"])
    line = {
        "metric": "<SpMM,GEMM> unfused/fused time ratio over the inner dimensions (Sec. 6.3)",
        "value": round(statistics.geometric_mean(r["unfused_over_fused"] for r in grid), 3), "unit": "x (geomean)",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "n/a",
        "vs_baseline": None, "dtype": "f32 (tf32 tensor-core contractions allowed)", "data": "synthetic",
        "config": {"workload": f"spmm_gemm R-MAT {n}x{n}, 16 nnz/row (seed {seed:#x}), K in {ks}, L in {ls}",
                   "l2": "flushed before every call", "timing": "median kernel time per call, CUDA events"},
        "best": {"K": best["K"], "L": best["L"], "unfused_over_fused": best["unfused_over_fused"]},
        "original_over_fused_geomean": round(statistics.geometric_mean(r["original_over_fused"] for r in grid), 2)
        if args.original else None,
        "grid": grid, "seconds": round(time.time() - t0, 1),
    }
    if rank == 0:
        print(json.dumps(line))
    return 0


def config1_latency(torch, slnr, dev, args, allow_tf32, flush_buf, stream):
    """Config 1 (<SpMM,GEMM> on a 1024^2 matrix with 10 uniform nonzeros per
    row, K = L = 32): far too small for a bandwidth roofline (it fits in L2),
    so its latency is reported beside the step, not in the headline value.
    Same protocol: warm-up, L2 flushed before each call, CUDA events."""
    w = wl.full(0)
    B = slnr.DeviceCSR.from_host(w.B, dev)
    dense = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dev) for k, v in w.dense.items()}
    ws = slnr.Workspace(device=dev)
    out = slnr.run(w.op, B, dense, variant=args.variant, allow_tf32=allow_tf32, workspace=ws)
    ts = []
    for it in range(args.warmup + args.steps):
        flush_buf.fill_(it & 0xFF)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        slnr.run(w.op, B, dense, out=out, variant=args.variant, allow_tf32=allow_tf32, workspace=ws)
        b.record(stream)
        b.synchronize()
        if it >= args.warmup:
            ts.append(a.elapsed_time(b))
    slnr.timing_enable(True)  # one more call for the kernel breakdown
    flush_buf.fill_(0)
    slnr.run(w.op, B, dense, out=out, variant=args.variant, allow_tf32=allow_tf32, workspace=ws)
    kt = slnr.timing_read()
    slnr.timing_enable(False)
    ms = statistics.mean(ts)
    return {"name": w.name, "entry": {
        "ms": round(ms, 4), "gflops": round(useful_flops(w) / (ms / 1e3) / 1e9, 2), "min_bytes": min_bytes(w),
        "kernels_ms": {k: round(v, 4) for k, v in kt}, "useful_flops": useful_flops(w), "in_headline": False,
        "note": "config 1, latency-bound (fits in L2): timed beside the step, not part of value"}}


def measure_e2e(torch, slnr, ws, dev_inputs, outs, call, stream, steps, total_flops, world, pg, dev):
    """Same step through the public API with host buffers: every step copies all
    inputs from pinned host memory to the device and all outputs back.  The
    copies run on two streams of their own (host-to-device and device-to-host,
    both directions of the link at once) and overlap the calls of the other
    expressions: expression i computes once its inputs have arrived and its
    previous outputs have been read back, and its outputs are copied out as
    soon as it is done; a step's inputs overwrite the device buffers only
    after the previous step's call that reads them has finished."""
    n = len(ws)
    host_in, dev_in, host_out, dev_out = [[] for _ in range(n)], [[] for _ in range(n)], [[] for _ in range(n)], \
        [[] for _ in range(n)]
    for i, w in enumerate(ws):
        B, dense = dev_inputs[i]
        arrays = [getattr(B, f) for f in ("pos", "crd", "vals")] if w.op in CSR_OPS else \
            [getattr(B, f) for f in ("pos1", "crd1", "pos2", "crd2", "pos3", "crd3", "vals")]
        arrays += list(dense.values())
        for a in arrays:
            dev_in[i].append(a)
            host_in[i].append(a.cpu().pin_memory())
        o = outs[i]
        for t in (o if isinstance(o, tuple) else (o,)):
            dev_out[i].append(t)
            host_out[i].append(torch.empty(t.shape, dtype=t.dtype, pin_memory=True))
    # the device-resident path's outputs for the same inputs: the read-back
    # outputs must equal them bit for bit (every kernel sums in a fixed order)
    expect = [[t.cpu() for t in dev_out[i]] for i in range(n)]
    h2d = sum(t.numel() * t.element_size() for hs in host_in for t in hs)
    d2h = sum(t.numel() * t.element_size() for hs in host_out for t in hs)
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    in_ready = [torch.cuda.Event() for _ in range(n)]
    done = [torch.cuda.Event() for _ in range(n)]
    read_back = [torch.cuda.Event() for _ in range(n)]
    for i in range(n):  # nothing pending before the first step
        done[i].record(stream)
        read_back[i].record(stream)

    def step():
        for i in range(n):
            s_in.wait_event(done[i])            # the previous call reading these inputs has finished
            with torch.cuda.stream(s_in):
                for d, h in zip(dev_in[i], host_in[i]):
                    d.copy_(h, non_blocking=True)
            in_ready[i].record(s_in)
        for i in range(n):
            stream.wait_event(in_ready[i])
            stream.wait_event(read_back[i])     # the previous outputs have been read back
            call(i, out=outs[i], on_stream=stream)
            done[i].record(stream)
            s_out.wait_event(done[i])
            with torch.cuda.stream(s_out):
                for h, d in zip(host_out[i], dev_out[i]):
                    h.copy_(d, non_blocking=True)
            read_back[i].record(s_out)

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    if pg is not None:
        pg.barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    s_in.wait_stream(stream)
    s_out.wait_stream(stream)
    for _ in range(steps):
        step()
    stream.wait_stream(s_in)
    stream.wait_stream(s_out)
    b.record(stream)
    b.synchronize()
    ms = a.elapsed_time(b) / steps
    torch.cuda.synchronize()
    differ = sum(int(not torch.equal(h, e)) for i in range(n) for h, e in zip(host_out[i], expect[i]))
    if pg is not None:
        t = torch.tensor([ms], dtype=torch.float64, device=dev)
        pg.all_reduce(t, op=pg.ReduceOp.MAX)
        ms = float(t.item())
    return {"value": round(world * total_flops / (ms / 1e3) / 1e9, 2), "unit": "GFLOP/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": round(ms, 3),
            "link_gbs": round((h2d + d2h) / (ms / 1e3) / 1e9, 1),
            "outputs_read_back": sum(len(x) for x in expect), "outputs_differing_from_device_path": differ}


if __name__ == "__main__":
    sys.exit(main())
