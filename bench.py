#!/usr/bin/env python
"""Benchmark of the UniSVQ linear layer (libunisvq) on GB300.

Workload (the decode sweep of the Llama-2-7B-shaped projection set): 32
layers x {q, k, v, o: 4096x4096; gate, up: 11008x4096; down: 4096x11008},
2-bit codes with d = 2 and one fp16 affine per matrix, bf16 activations with
1% outlier channels, batch M in {1, 2, 4, 8, 16}. One step = one pass of the
whole layer stack at every M of the sweep (5 x 224 layer calls), replayed from
CUDA graphs. The 1.62 GB of packed codes per pass is far larger than L2, so
no flush is needed between steps.

Metric: HBM GB/s = algorithmic bytes (N*K/4 codes + affine + 2*M*K + 2*M*N)
per step / step time. With --prefill (default on) a second object reports the
tcgen05 prefill GEMM on the Llama-3-8B-shaped set at M = 2048 in TFLOP/s.

--impl reference times the CPU oracle (the fp64 NumPy restatement of the
method) on a bounded sample of the same workload, on the host cores.

Multi-GPU (torchrun): the path does not shard, so every rank runs an
independent replica; value = bytes of all ranks / max time over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "UniSVQ linear: GEMV HBM GB/s (% of ~8 TB/s); prefill TFLOPS (% of bf16 peak)"
M_SWEEP = (1, 2, 4, 8, 16)
# Projections of the Llama-2-7B set (synth.LLAMA2_7B order) that share an input.
GROUPS_7B = [[0, 1, 2], [3], [4, 5], [6]]
PREFILL_M = 2048
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


def algo_bytes(N, K, M, d=2):
    return N * K // 4 + (d * d + d) * 2 + 2 * M * K + 2 * M * N


def group_bytes(shapes, grp, M, d=2):
    """Algorithmic bytes of one call over the projections `grp`, which share
    one input: codes, affine and output per projection, the input x once."""
    K = shapes[grp[0]][2]
    return sum(shapes[i][1] * K // 4 + (d * d + d) * 2 + 2 * M * shapes[i][1] for i in grp) + 2 * M * K


KERNEL_NAMES = {1: "decode", 2: "prefill_kernel", 3: "gemv_kernel", 4: "decode_kernel", 5: "gemv_rows_kernel",
                6: "gemv_grouped_kernel"}
GROUPED_LAYERS = 16   # 16 x 69.6 MB of codes + per-group maps: larger than L2


def variant_layers(args):
    """Layers of the secondary sweeps: 16, or --layers when one of them runs
    alone (--only grouped / rht / bits3, a profiling aid)."""
    return args.layers if args.only in ("grouped", "rht", "bits3") else GROUPED_LAYERS
# Sources whose change invalidates a committed ncu traffic figure, per kernel.
KERNEL_SOURCES = {
    "gemv_kernel": ("paper_2606_10520_gb300/csrc/gemv.cu", "paper_2606_10520_gb300/csrc/mma_sync.cuh",
                    "paper_2606_10520_gb300/csrc/common.cuh", "paper_2606_10520_gb300/csrc/layout.h"),
    "decode_kernel": ("paper_2606_10520_gb300/csrc/decode.cu", "paper_2606_10520_gb300/csrc/common.cuh",
                      "paper_2606_10520_gb300/csrc/layout.h"),
}


def traffic_summary_path(kernel):
    return os.path.join(ROOT, "profiles", f"{kernel}_llama2_7b_decode_sweep.txt")


def source_digest(kernel):
    import hashlib
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def measured_traffic(kernel):
    """DRAM bytes per launch of `kernel` from its committed ncu summary, or None
    when the kernel's sources changed since those counters were taken."""
    try:
        fields = {}
        with open(traffic_summary_path(kernel)) as f:
            for ln in f:
                if ":" in ln:
                    k, v = ln.split(":", 1)
                    fields[k.strip()] = v.strip()
        if fields.get("source_sha256") != source_digest(kernel):
            return None
        return float(fields["dram_bytes_per_launch"])
    except Exception:
        return None


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle baseline (bounded sample)
# ---------------------------------------------------------------------------
def cpu_threads():
    """Threads the oracle's BLAS runs with: from threadpoolctl where it is
    installed, else the thread-count environment variables, else every core
    (the BLAS default)."""
    try:
        from threadpoolctl import threadpool_info
        n = [p.get("num_threads") for p in threadpool_info() if p.get("user_api") == "blas"]
        if n and all(isinstance(v, int) for v in n):
            return max(n)
    except Exception:
        pass
    for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(v, "").isdigit():
            return int(os.environ[v])
    return os.cpu_count() or 1


def oracle_sample_one_thread(budget_s: float):
    """oracle_sample in a child process whose BLAS runs one thread."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = ("import json, sys; sys.path.insert(0, %r); import bench; "
            "g, t, n = bench.oracle_sample(%f); print(json.dumps([g, t, len(n), bench.cpu_threads()]))") % (ROOT, budget_s)
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    if r.returncode != 0:
        return None
    g, t, n, th = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": g, "unit": "GB/s", "cores": th, "seconds": t, "calls": n}


def oracle_sample(budget_s: float):
    """Time the oracle on layer-0 projections at M = 1 until `budget_s` passes."""
    import oracle
    t0 = time.perf_counter()
    nbytes = 0
    done = []
    i = 0
    while True:
        name, N, K = synth.LLAMA2_7B[i % len(synth.LLAMA2_7B)]
        codes, A, B = synth.layer_inputs(0, 1, 0, i % 7, N, K, 2)
        xb = synth.activations(0, 1, 1, 1, K)
        t1 = time.perf_counter()
        oracle.linear(xb, codes, A, B)
        dt = time.perf_counter() - t1
        nbytes += algo_bytes(N, K, 1)
        done.append((name, dt))
        i += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    t_oracle = sum(dt for _, dt in done)
    return nbytes / t_oracle / 1e9, t_oracle, [n for n, _ in done]


# ---------------------------------------------------------------------------
# reference arm: the oracle on the host cores
# ---------------------------------------------------------------------------
def max_over_ranks(values, world, device):
    """Element-wise maximum of per-rank floats over the process group (every
    rank receives it); the identity for one rank."""
    if world <= 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist
    tt = torch.tensor([float(v) for v in values], device=device, dtype=torch.float64)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return [float(v) for v in tt.tolist()]


def whole_job_gbs(bytes_per_step_per_rank, steps, world, t_max):
    """Whole-job throughput: every rank's bytes over the slowest rank's time."""
    return bytes_per_step_per_rank * steps * world / t_max / 1e9


def run_reference(args, rank, world):
    """The oracle on a bounded sample of the workload: step i is one call on
    512 output rows of projection i mod 7 of the layer-0 set at M =
    M_SWEEP[(i // 7) mod 5], so K steps cover the projections and batch sizes
    in the workload's proportions (the 32 layers are copies of layer 0)."""
    if rank != 0:
        return
    import oracle
    shapes = synth.LLAMA2_7B
    mats = [synth.layer_inputs(0, 1, 0, pi, N, K, 2) for pi, (_, N, K) in enumerate(shapes)]
    xs = {(M, K): synth.activations(0, 1, 100 + M, M, K) for M in M_SWEEP for K in {K for _, _, K in shapes}}

    rows = 512   # output rows per step, cycling over each matrix

    def step(i):
        pi = i % len(shapes)
        M = M_SWEEP[(i // len(shapes)) % len(M_SWEEP)]
        _, N, K = shapes[pi]
        codes, A, B = mats[pi]
        r0 = (i // (len(shapes) * len(M_SWEEP)) * rows) % N
        part = codes[r0:r0 + rows]
        oracle.linear(xs[(M, K)], part, A, B)
        return algo_bytes(part.shape[0], K, M)
    for i in range(args.warmup):
        step(i)
    nbytes = 0
    t0 = time.perf_counter()
    for i in range(args.steps):
        nbytes += step(i)
    dt = time.perf_counter() - t0
    gbs = nbytes / dt / 1e9
    sample = (f"{args.steps} oracle.linear calls (fp64 NumPy), each on {rows} output rows of one projection, "
              f"cycling over the 7 layer-0 projections, M in {list(M_SWEEP)} and the rows of each matrix")
    line = {
        "impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1000 / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(args),
        "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": cpu_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def workload_config(args):
    return {"workload": f"Llama-2-7B-shaped projection set x {args.layers} layers, decode sweep M in "
                        f"{list(M_SWEEP)}, 2-bit codes d=2, per-matrix fp16 affine",
            "layers": args.layers, "d": 2, "m_sweep": list(M_SWEEP),
            "l2": "inputs larger than L2 (1.62 GB of packed codes per pass at 32 layers)",
            "timing": "CUDA graphs of the full layer stack per M, CUDA events on the capture stream",
            "calls": ("one unisvq_linear per projection (7 per layer)" if getattr(args, "ungrouped", False) else
                      "q/k/v and gate/up as one unisvq_linear_group call each (shared input), o and down "
                      "as unisvq_linear: 4 calls per layer"),
            "parallelism": "replicas"}


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def build_stack(binding, shapes, layers, config_id, d=2):
    """Distinct random matrices for layer 0; the other layers are device copies."""
    base = []
    for pi, (_, N, K) in enumerate(shapes):
        codes, A, B = synth.layer_inputs(0, config_id, 0, pi, N, K, d)
        base.append(binding.UniSVQLinear(codes, A, B))
    stack = [base]
    for _ in range(layers - 1):
        stack.append([b.clone() for b in base])
    return stack


def time_graphs(torch, graphs, steps, warmup, stream):
    """Replay `graphs` `steps` times on `stream`; seconds between CUDA events
    recorded on that same stream (graph replays launch on the current stream)."""
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            for g in graphs:
                g.replay()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            for g in graphs:
                g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
    return e0.elapsed_time(e1) / 1000.0


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    from paper_2606_10520_gb300 import binding

    torch.cuda.set_device(local_rank)
    binding.load()
    peaks, peak_src = load_peaks()
    if args.only == "prefill":
        side = torch.cuda.Stream()
        print(json.dumps({"prefill": run_prefill(torch, binding, peaks, args, side)}), flush=True)
        return
    variants = {"grouped": ("per_group_affine", run_grouped), "rht": ("rht", run_rht), "bits3": ("bits3", run_bits3),
                "rht7": ("rht_llama2_7b", lambda *a: run_rht(*a, which="llama2_7b"))}
    if args.only in variants:
        key, fn = variants[args.only]
        print(json.dumps({key: fn(torch, binding, peaks, args, torch.cuda.Stream())}), flush=True)
        return
    if args.only == "decode":
        args.no_e2e = args.no_cpu = args.no_prefill = args.no_grouped = args.no_rht = args.no_bits3 = True
        args.no_70b = args.no_dense = True
    shapes = synth.LLAMA2_7B
    stack = build_stack(binding, shapes, args.layers, 1)

    # Projections that read the same input are issued as one grouped call
    # (q, k, v and gate, up), as a decode step issues them; --ungrouped makes
    # one unisvq_linear call per projection.
    groups = [[i] for i in range(len(shapes))] if args.ungrouped else GROUPS_7B
    xs, ys, graphs, step_bytes, launches = {}, {}, [], 0, 0
    for M in M_SWEEP:
        for pi, (_, N, K) in enumerate(shapes):
            if (M, K) not in xs:
                xb = synth.activations(0, 1, 100 + M, M, K)
                xs[(M, K)] = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
            ys[(M, pi)] = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")

    # The library's choice per call (the same for every layer of the stack).
    def call_info(grp, M):
        layer0 = stack[0]
        if len(grp) == 1:
            return layer0[grp[0]].query(M)
        return binding.query_group([layer0[i] for i in grp], M)

    def issue(layer, grp, M, sp):
        K = shapes[grp[0]][2]
        if len(grp) == 1:
            st = layer[grp[0]].forward_ptr(xs[(M, K)].data_ptr(), ys[(M, grp[0])].data_ptr(), M, sp,
                                           binding.KERNEL_AUTO)
        else:
            st = binding.linear_group_ptr([layer[i] for i in grp], xs[(M, K)].data_ptr(),
                                          [ys[(M, i)].data_ptr() for i in grp], M, sp)
        if st != 0:
            raise RuntimeError(f"unisvq call failed: {binding.status_string(st)}")

    side = torch.cuda.Stream()
    # calls per kernel class: {kernel id: [(M, group index), ...]}
    kinds = {}
    kind_bytes, kind_main_launches = {}, {}
    for M in M_SWEEP:
        def one_pass(M=M):
            sp = torch.cuda.current_stream().cuda_stream
            for layer in stack:
                for grp in groups:
                    issue(layer, grp, M, sp)
        with torch.cuda.stream(side):
            one_pass()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            one_pass()
        graphs.append(g)
        for gi, grp in enumerate(groups):
            info = call_info(grp, M)
            kid = info["kernel"]
            nbytes = group_bytes(shapes, grp, M) * args.layers
            step_bytes += nbytes
            launches += info["launches"] * args.layers
            kinds.setdefault(kid, []).append((M, gi))
            kind_bytes[kid] = kind_bytes.get(kid, 0) + nbytes
            # the streaming kernel's launches (the skinny path adds one fold launch each)
            main = info["launches"] // 2 if kid == binding.KERNEL_SKINNY else info["launches"]
            kind_main_launches[kid] = kind_main_launches.get(kid, 0) + main * args.layers
    torch.cuda.synchronize()
    st = binding.sync_status()
    if st != 0:
        raise RuntimeError(f"device status {binding.status_string(st)}")

    # ---- timed region: decode sweep ------------------------------------
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clk = ClockSampler(local_rank)
    clk.start()
    time.sleep(0.3)
    t = time_graphs(torch, graphs, args.steps, args.warmup, side)
    clocks = clk.stop()
    t = max_over_ranks([t], world, "cuda")[0]
    st = binding.sync_status(side)
    if st != 0:
        raise RuntimeError(f"device status {binding.status_string(st)}")
    value = whole_job_gbs(step_bytes, args.steps, world, t)
    per_rank = step_bytes * args.steps / t / 1e9

    # per-kernel-class timing: graphs holding only the calls that run that
    # kernel, so each kernel's throughput (and launch interval) is measured
    # on its own stream; the dominant class (most time) gives the roofline.
    kind_time = {}
    for kid, calls in kinds.items():
        kgraphs = []
        for M in M_SWEEP:
            sel = [gi for (m, gi) in calls if m == M]
            if not sel:
                continue
            def kpass(M=M, sel=sel):
                sp = torch.cuda.current_stream().cuda_stream
                for layer in stack:
                    for gi in sel:
                        issue(layer, groups[gi], M, sp)
            with torch.cuda.stream(side):
                kpass()
            torch.cuda.synchronize()
            kg = torch.cuda.CUDAGraph()
            with torch.cuda.graph(kg, stream=side):
                kpass()
            kgraphs.append(kg)
        kind_time[kid] = time_graphs(torch, kgraphs, args.steps, args.warmup, side)
    kids = sorted(kind_time)
    for kid, tk in zip(kids, max_over_ranks([kind_time[k] for k in kids], world, "cuda")):
        kind_time[kid] = tk

    def roofline_for(kid):
        name = KERNEL_NAMES.get(kid, "?")
        t_k = kind_time[kid]
        ach = kind_bytes[kid] * args.steps / t_k / 1e9
        n_main = kind_main_launches[kid]
        extra = " (each call: fold_kernel + decode_kernel)" if kid == binding.KERNEL_SKINNY else ""
        return {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": ach / peaks["hbm_gbs"],
                "traffic": measured_traffic(name) if name in KERNEL_SOURCES else None,
                "algorithmic_bytes_per_launch": kind_bytes[kid] / max(1, n_main),
                "avg_launch_us": t_k / args.steps / max(1, n_main) * 1e6,
                "launches_per_step": n_main,
                "share_of_step_time": t_k / max(1e-12, sum(kind_time.values())),
                "kernel": name + extra,
                "how": ("achieved = algorithmic bytes of the calls that run this kernel / their time, "
                        "timed alone from CUDA graphs of those calls (CUDA events on the launching stream)"),
                "peak_source": f"{peak_src} hbm_gbs (copy, burst)",
                "frac_of_8TBs": ach / 8000.0}

    dominant = max(kind_time, key=lambda k: kind_time[k])

    # per-M breakdown (separate short timing of each graph)
    sweep = []
    for M, g in zip(M_SWEEP, graphs):
        tm = time_graphs(torch, [g], max(3, args.steps // 4), 2, side)
        nb = sum(group_bytes(shapes, grp, M) for grp in groups) * args.layers
        n_calls = len(shapes) * args.layers
        gbs = nb * max(3, args.steps // 4) / tm / 1e9
        sweep.append({"M": M, "GB/s": round(gbs, 1), "frac_of_measured_hbm": round(gbs / peaks["hbm_gbs"], 4),
                      "frac_of_8TBs": round(gbs / 8000.0, 4),
                      "us_per_projection": round(tm / max(3, args.steps // 4) / n_calls * 1e6, 3),
                      "kernels": {"+".join(shapes[i][0] for i in grp): KERNEL_NAMES.get(call_info(grp, M)["kernel"], "?")
                                  for grp in groups}})

    # ---- e2e: pinned host buffers; every step copies its inputs in and its
    # results out inside the timed graphs (activations stay on the device
    # between the layers of a step, as in a model) ---------------------------
    e2e = None
    if not args.no_e2e:
        hx = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True).copy_(v.cpu()) for k, v in xs.items()}
        hy = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in ys.items()}
        egraphs, h2d, d2h = [], 0, 0
        for M in M_SWEEP:
            in_keys = sorted(k for k in xs if k[0] == M)
            out_keys = sorted(k for k in ys if k[0] == M)
            def e2e_pass(M=M, in_keys=in_keys, out_keys=out_keys):
                sp = torch.cuda.current_stream().cuda_stream
                for k in in_keys:
                    xs[k].copy_(hx[k], non_blocking=True)
                for layer in stack:
                    for grp in groups:
                        issue(layer, grp, M, sp)
                for k in out_keys:
                    hy[k].copy_(ys[k], non_blocking=True)
            with torch.cuda.stream(side):
                e2e_pass()
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                e2e_pass()
            egraphs.append(g)
            h2d += sum(xs[k].numel() * xs[k].element_size() for k in in_keys)
            d2h += sum(ys[k].numel() * ys[k].element_size() for k in out_keys)
        te = time_graphs(torch, egraphs, args.steps, args.warmup, side)
        te = max_over_ranks([te], world, "cuda")[0]
        e2e = {"value": whole_job_gbs(step_bytes, args.steps, world, te), "unit": "GB/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "how": "per step (the sweep's M passes): pinned-host -> device copies of the step's activations "
                      "before the layers, the library calls, device -> pinned-host copies of every projection's "
                      "output after them; replayed from CUDA graphs"}

    # ---- per-(row, 128-column group) affine layers ------------------------
    grouped = None
    if not args.no_grouped:
        grouped = run_grouped(torch, binding, peaks, args, side)

    # ---- 3-bit codes --------------------------------------------------------
    bits3 = None
    if not args.no_bits3:
        bits3 = run_bits3(torch, binding, peaks, args, side)

    # ---- inverse RHT around the layers -------------------------------------
    rht = rht7 = None
    if not args.no_rht:
        rht = run_rht(torch, binding, peaks, args, side)
        rht7 = run_rht(torch, binding, peaks, args, side, "llama2_7b")

    # ---- prefill (tcgen05 GEMM), Llama-3-8B-shaped set at M = 2048 -------
    prefill = None
    if not args.no_prefill:
        prefill = run_prefill(torch, binding, peaks, args, side)

    # ---- configs 0, 3 (70B stack), 4 (crossover) and the dense reference ----
    config0 = run_config0(torch, binding, peaks, args, side)
    cfg3 = crossover = None
    if not args.no_70b:
        cfg3, stack70 = run_70b(torch, binding, peaks, args, side)
        crossover = run_crossover(torch, binding, peaks, args, side, stack70)
        for layer in stack70:
            for h in layer:
                h.close()
        del stack70
    dense = None if args.no_dense else run_cublas_decode(torch, peaks, args, side, sweep)

    # ---- CPU oracle baseline (rank 0, N=1 only) --------------------------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        gbs_cpu, t_cpu, names = oracle_sample(args.cpu_budget)
        cpu = {"value": gbs_cpu, "unit": "GB/s", "cores": cpu_threads(), "kind": "oracle",
               "sample": f"oracle.linear (fp64 NumPy) at M=1 on {len(names)} projection calls cycling over "
                         f"the layer-0 set ({', '.join(n for n, _, _ in synth.LLAMA2_7B)}), "
                         f"{t_cpu:.1f} s of CPU work",
               "single_thread": oracle_sample_one_thread(min(8.0, args.cpu_budget))}

    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t * 1000 / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16 I/O; e4m3 tcgen05 MMA (decode_kernel) / f16 mma.sync (gemv_kernel); f32 accumulate",
        "data": "synthetic (seeded codes, affine and activations; layers 1..31 are device copies of layer 0)",
        "config": workload_config(args),
        "roofline": roofline_for(dominant),
        "roofline_other": {KERNEL_NAMES.get(k, "?"): roofline_for(k) for k in kind_time if k != dominant},
        "step_throughput_per_gpu": per_rank,
        "sweep": sweep,
        "e2e": e2e,
        "gpu_launches": launches * args.steps,
        "clocks": clocks,
        "cpu_baseline": cpu,
        "prefill": prefill,
        "config0_4096x4096_m1": config0,
        "llama2_70b": cfg3,
        "crossover_70b": crossover,
        "cublas_dense_decode": dense,
        "per_group_affine": grouped,
        "rht": rht,
        "rht_llama2_7b": rht7,
        "bits3": bits3,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


def sweep_variant(torch, binding, args, stream, base, kernel_id):
    """The Llama-2-7B decode sweep (GROUPED_LAYERS layers: `base` and device
    copies) for one layer variant; returns (GB/s over the sweep, per-M list,
    launches per step). Bytes are the library's algorithmic bytes per call.
    kernel_id: the kernel every call must resolve to, or None for the
    library's own pick (then reported per M and call)."""
    shapes = synth.LLAMA2_7B
    nl = variant_layers(args)
    stack = [base] + [[b.clone() for b in base] for _ in range(nl - 1)]
    xs, ys = {}, {}
    for M in M_SWEEP:
        for pi, (_, N, K) in enumerate(shapes):
            if (M, K) not in xs:
                xb = synth.activations(0, 1, 100 + M, M, K)
                xs[(M, K)] = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
            ys[(M, pi)] = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    graphs, sweep_bytes, launches, kernels = [], [], 0, []
    for M in M_SWEEP:
        def one_pass(M=M):
            sp = torch.cuda.current_stream().cuda_stream
            for layer in stack:
                for grp in GROUPS_7B:
                    K = shapes[grp[0]][2]
                    st = binding.linear_group_ptr([layer[i] for i in grp], xs[(M, K)].data_ptr(),
                                                  [ys[(M, i)].data_ptr() for i in grp], M, sp)
                    if st != 0:
                        raise RuntimeError(f"unisvq call failed: {binding.status_string(st)}")
        with torch.cuda.stream(stream):
            one_pass()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            one_pass()
        graphs.append(g)
        nbytes = 0
        kern_m = {}
        for grp in GROUPS_7B:
            info = binding.query_group([base[i] for i in grp], M)
            assert kernel_id is None or info["kernel"] == kernel_id
            kern_m["+".join(shapes[i][0] for i in grp)] = KERNEL_NAMES.get(info["kernel"], "?")
            nbytes += info["algo_bytes"] * nl
            launches += info["launches"] * nl
        sweep_bytes.append(nbytes)
        kernels.append(kern_m)
    st = binding.sync_status(stream)
    if st != 0:
        raise RuntimeError(f"device status {binding.status_string(st)}")
    steps = max(5, args.steps // 4)
    t = time_graphs(torch, graphs, steps, args.warmup, stream)
    per_m = []
    for M, g, nb, km in zip(M_SWEEP, graphs, sweep_bytes, kernels):
        tm = time_graphs(torch, [g], steps, 2, stream)
        per_m.append({"M": M, "GB/s": round(nb * steps / tm / 1e9, 1),
                      "us_per_layer": round(tm / steps / nl * 1e6, 3), "kernels": km})
    for layer in stack:
        for b in layer:
            b.close()
    return sum(sweep_bytes) * steps / t / 1e9, per_m, launches


def run_grouped(torch, binding, peaks, args, stream):
    """The decode sweep on Llama-2-7B-shaped layers with one fp16 affine map
    per (output row, 128-column group): the per-group GEMV (gemv_grouped_kernel),
    algorithmic bytes counting the maps (N * K/128 * 12 bytes at d = 2)."""
    base = []
    for pi, (_, N, K) in enumerate(synth.LLAMA2_7B):
        codes, A, B = synth.layer_inputs_grouped(0, 1, 0, pi, N, K, 2)
        base.append(binding.UniSVQLinear(codes, A, B, group_cols=128))
    gbs, per_m, launches = sweep_variant(torch, binding, args, stream, base, binding.KERNEL_GROUPED)
    return {"workload": f"Llama-2-7B-shaped projection set x {variant_layers(args)} layers, decode sweep M in "
                        f"{list(M_SWEEP)}, 2-bit codes d=2, one fp16 affine per output row per 128-column group",
            "GB/s": gbs, "frac_of_measured_hbm": gbs / peaks["hbm_gbs"], "sweep": per_m,
            "kernel": "gemv_grouped_kernel", "launches_per_step": launches,
            "bytes": "codes N*K/4 + maps N*ceil(K/128)*12 + x + y per call",
            "timing": "CUDA graphs of the layer stack per M, CUDA events on the capture stream"}


def run_bits3(torch, binding, peaks, args, stream):
    """The decode sweep on Llama-2-7B-shaped layers with 3-bit codes (z in
    0..7, Sec. 5.2) through the library's own pick: the tcgen05 decode path
    (decode_kernel, 3-bit instance) for q/k/v and gate/up, the GEMV with the
    high-bit plane (gemv_kernel, BITS = 3) for o and down."""
    base = []
    for pi, (_, N, K) in enumerate(synth.LLAMA2_7B):
        codes, A, B = synth.layer_inputs_bits(0, 1, 0, pi, N, K, 2, 3)
        base.append(binding.UniSVQLinear(codes, A, B, bits=3))
    gbs, per_m, launches = sweep_variant(torch, binding, args, stream, base, None)
    return {"workload": f"Llama-2-7B-shaped projection set x {variant_layers(args)} layers, decode sweep M in "
                        f"{list(M_SWEEP)}, 3-bit codes d=2, per-matrix fp16 affine",
            "GB/s": gbs, "frac_of_measured_hbm": gbs / peaks["hbm_gbs"], "sweep": per_m,
            "kernel": "decode_kernel / gemv_kernel (3-bit instances), per call as listed in sweep",
            "launches_per_step": launches,
            "bytes": "codes 3*N*K/8 + affine + x + y per call",
            "timing": "CUDA graphs of the layer stack per M, CUDA events on the capture stream"}


RHT_SETS = {"llama3_8b": ("Llama-3-8B", synth.LLAMA3_8B, 2), "llama2_7b": ("Llama-2-7B", synth.LLAMA2_7B, 1)}


def run_rht(torch, binding, peaks, args, stream, which="llama3_8b"):
    """The decode sweep on Llama-3-8B- or Llama-2-7B-shaped layers with and
    without the inverse randomized Hadamard transform around each layer (Eq.
    def:hadamard): q/k/v and gate/up share their input rotation S_V V, every
    layer has its own output rotation U S_U. Widths: 4096 = 2^12, 14336 =
    2^9 * 28, 11008 = 2^5 * 344. GB/s counts the layers' algorithmic bytes
    only (a group call's shared x once)."""
    label, shapes, config_id = RHT_SETS[which]
    g = np.random.default_rng(5)
    base = []
    for pi, (_, N, K) in enumerate(shapes):
        codes, A, B = synth.layer_inputs(0, config_id, 0, pi, N, K, 2)
        base.append(binding.UniSVQLinear(codes, A, B))
    s_in = {K: g.choice([-1.0, 1.0], K) for K in sorted({K for _, _, K in shapes})}
    s_out = [g.choice([-1.0, 1.0], N) for _, N, _ in shapes]
    nl = variant_layers(args)
    stack = [base] + [[b.clone() for b in base] for _ in range(nl - 1)]
    xs, ys = {}, {}
    for M in M_SWEEP:
        for pi, (_, N, K) in enumerate(shapes):
            if (M, K) not in xs:
                xb = synth.activations(0, config_id, 100 + M, M, K)
                xs[(M, K)] = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
            ys[(M, pi)] = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    step_bytes = sum(group_bytes(shapes, grp, M) for M in M_SWEEP for grp in GROUPS_7B) * nl
    steps = max(5, args.steps // 4)
    out = {}
    for rht in (False, True):
        for layer in stack:
            for pi, b in enumerate(layer):
                if rht:
                    b.set_rht(s_in[shapes[pi][2]], s_out[pi], max_tokens=max(M_SWEEP))
                else:
                    b.set_rht(None, None)
        graphs = []
        for M in M_SWEEP:
            def one_pass(M=M):
                sp = torch.cuda.current_stream().cuda_stream
                for layer in stack:
                    for grp in GROUPS_7B:
                        K = shapes[grp[0]][2]
                        st = binding.linear_group_ptr([layer[i] for i in grp], xs[(M, K)].data_ptr(),
                                                      [ys[(M, i)].data_ptr() for i in grp], M, sp)
                        if st != 0:
                            raise RuntimeError(f"unisvq call failed: {binding.status_string(st)}")
            with torch.cuda.stream(stream):
                one_pass()
            torch.cuda.synchronize()
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream):
                one_pass()
            graphs.append(gr)
        st = binding.sync_status(stream)
        if st != 0:
            raise RuntimeError(f"device status {binding.status_string(st)}")
        t = time_graphs(torch, graphs, steps, args.warmup, stream)
        out["with_rht" if rht else "without_rht"] = step_bytes * steps / t / 1e9
    for layer in stack:
        for b in layer:
            b.close()
    return {"workload": f"{label}-shaped projection set x {nl} layers, decode sweep M in "
                        f"{list(M_SWEEP)}, d=2, per-matrix fp16 affine, inverse RHT around every layer",
            "GB/s": out["with_rht"], "GB/s_without_rht": out["without_rht"],
            "frac_of_measured_hbm": out["with_rht"] / peaks["hbm_gbs"],
            "kernels": "rht_kernel (input and output rotations, a cluster of 8 or 16 CTAs per row) + the layers' kernels",
            "bytes": "the layers' algorithmic bytes (codes + affine + x + y); the rotations are overhead",
            "timing": "CUDA graphs of the layer stack per M, CUDA events on the capture stream"}


def run_prefill(torch, binding, peaks, args, stream):
    from paper_2606_10520_gb300 import binding as b
    shapes = synth.LLAMA3_8B
    layers = []
    for pi, (_, N, K) in enumerate(shapes):
        codes, A, B = synth.layer_inputs(0, 2, 0, pi, N, K, 2)
        layers.append(b.UniSVQLinear(codes, A, B))
    q = layers[0].query(PREFILL_M)
    if q["kernel"] != b.KERNEL_PREFILL:
        for l in layers:
            l.close()
        return {"unavailable": "prefill kernel not supported in this build"}
    M = PREFILL_M
    xs = {K: torch.from_numpy(synth.activations(0, 2, K, M, K).view(np.int16)).view(torch.bfloat16).cuda()
          for K in sorted({K for _, _, K in shapes})}
    ys = {N: torch.empty((M, N), dtype=torch.bfloat16, device="cuda") for N in sorted({N for _, N, _ in shapes})}

    def one_pass():
        sp = torch.cuda.current_stream().cuda_stream
        for (_, N, K), h in zip(shapes, layers):
            st = h.forward_ptr(xs[K].data_ptr(), ys[N].data_ptr(), M, sp, b.KERNEL_PREFILL)
            if st != 0:
                raise RuntimeError(b.status_string(st))
    with torch.cuda.stream(stream):
        one_pass()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        one_pass()
    reps = max(5, args.steps // 2)
    t = time_graphs(torch, [g], reps, 3, stream)
    flops = sum(2.0 * M * N * K for _, N, K in shapes)
    tflops_single = flops * reps / t / 1e12
    # the set as a model issues it: q/k/v and gate/up as one call each (one
    # persistent launch over the tiles of the layers that share x)
    yp = [torch.empty((M, N), dtype=torch.bfloat16, device="cuda") for _, N, _ in shapes]

    def group_pass():
        sp = torch.cuda.current_stream().cuda_stream
        for grp in GROUPS_7B:
            K = shapes[grp[0]][2]
            st = b.linear_group_ptr([layers[i] for i in grp], xs[K].data_ptr(), [yp[i].data_ptr() for i in grp],
                                    M, sp, b.KERNEL_PREFILL)
            if st != 0:
                raise RuntimeError(b.status_string(st))
    with torch.cuda.stream(stream):
        group_pass()
    torch.cuda.synchronize()
    gg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gg, stream=stream):
        group_pass()
    tg = time_graphs(torch, [gg], reps, 3, stream)
    tflops = flops * reps / tg / 1e12
    group_launches = sum(b.query_group([layers[i] for i in grp], M)["launches"] for grp in GROUPS_7B)
    del gg, yp
    # per-projection timing
    per = []
    for (nm, N, K), h in zip(shapes, layers):
        def single(h=h, N=N, K=K):
            sp = torch.cuda.current_stream().cuda_stream
            h.forward_ptr(xs[K].data_ptr(), ys[N].data_ptr(), M, sp, b.KERNEL_PREFILL)
        with torch.cuda.stream(stream):
            single()
        torch.cuda.synchronize()
        gs = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gs, stream=stream):
            single()
        ts = time_graphs(torch, [gs], reps, 3, stream)
        per.append({"proj": nm, "N": N, "K": K, "TFLOP/s": round(2.0 * M * N * K * reps / ts / 1e12, 1),
                    "us": round(ts / reps * 1e6, 1)})
    # cuBLAS bf16 dense GEMM on the same shapes (speed reference)
    Wd = {(N, K): torch.randn(N, K, device="cuda").to(torch.bfloat16) for _, N, K in shapes}

    def dense_pass():
        for _, N, K in shapes:
            torch.matmul(xs[K], Wd[(N, K)].t(), out=ys[N])
    with torch.cuda.stream(stream):
        dense_pass()
    torch.cuda.synchronize()
    gd = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gd, stream=stream):
        dense_pass()
    td = time_graphs(torch, [gd], reps, 3, stream)
    for l in layers:
        l.close()
    # the same set with one affine map per (row, 128-column group), d = 1, 2, 4 and 8
    # (d = 8: without down, whose 4096 x 14336 maps do not fit the per-group
    # GEMV's shared memory, so that it does not pack)
    per_group = {}
    shapes_d8 = [sh for sh in shapes if sh[2] <= 4096]
    flops_d8 = sum(2.0 * M * N * K for _, N, K in shapes_d8)
    for dg in (1, 2, 4, 8):
        sset = shapes_d8 if dg == 8 else shapes
        glayers = []
        for pi, (_, N, K) in enumerate(sset):
            codes, A, B = synth.layer_inputs_grouped(0, 2, 0, pi, N, K, dg)
            glayers.append(b.UniSVQLinear(codes, A, B, group_cols=128))
        per_group[dg] = time_prefill_layers(torch, b, sset, glayers, xs, ys, M, reps, stream)
        if dg == 2:
            per_group["calls"] = time_prefill_groups(torch, b, shapes, glayers, xs, M, reps, stream)
        for l in glayers:
            l.close()
    # the same set with 3-bit codes (per-matrix maps)
    l3 = []
    for pi, (_, N, K) in enumerate(shapes):
        codes, A, B = synth.layer_inputs_bits(0, 2, 0, pi, N, K, 2, 3)
        l3.append(b.UniSVQLinear(codes, A, B, bits=3))
    t3 = time_prefill_layers(torch, b, shapes, l3, xs, ys, M, reps, stream)
    for l in l3:
        l.close()
    l34 = []   # 3-bit codes, d = 4 (pair tables)
    for pi, (_, N, K) in enumerate(shapes):
        codes, A, B = synth.layer_inputs_bits(0, 2, 0, pi, N, K, 4, 3)
        l34.append(b.UniSVQLinear(codes, A, B, bits=3))
    t34 = time_prefill_layers(torch, b, shapes, l34, xs, ys, M, reps, stream)
    for l in l34:
        l.close()
    # the same set with vectors of length 8 (per-matrix maps, pair tables)
    l8 = []
    for pi, (_, N, K) in enumerate(shapes):
        codes, A, B = synth.layer_inputs(0, 2, 0, pi, N, K, 8)
        l8.append(b.UniSVQLinear(codes, A, B))
    t8 = time_prefill_layers(torch, b, shapes, l8, xs, ys, M, reps, stream)
    for l in l8:
        l.close()
    return {"workload": f"Llama-3-8B-shaped projection set (7 GEMMs) at M={M}, d=2",
            "TFLOP/s": tflops, "frac_of_measured_bf16": tflops / peaks["bf16_tflops"],
            "calls": (f"q/k/v and gate/up as one unisvq_linear_group call each, o and down alone: "
                      f"{group_launches} prefill launches"),
            "TFLOP/s_one_call_per_projection": tflops_single,
            "per_group_maps_TFLOP/s": flops * reps / per_group[2] / 1e12,
            "per_group_maps_group_calls_TFLOP/s": flops * reps / per_group["calls"] / 1e12,
            "per_group_maps_d4_TFLOP/s": flops * reps / per_group[4] / 1e12,
            "per_group_maps_d1_TFLOP/s": flops * reps / per_group[1] / 1e12,
            "per_group_maps_d8_without_down_TFLOP/s": flops_d8 * reps / per_group[8] / 1e12,
            "bits3_TFLOP/s": flops * reps / t3 / 1e12,
            "bits3_d4_TFLOP/s": flops * reps / t34 / 1e12,
            "d8_TFLOP/s": flops * reps / t8 / 1e12,
            "frac_of_measured_bf16_sustained": tflops / peaks["bf16_tflops_sustained"],
            "us_per_layer_set": tg / reps * 1e6, "per_projection": per,
            "cublas_bf16_dense_TFLOP/s": flops * reps / td / 1e12,
            "kernel": "prefill_kernel (tcgen05)"}


def time_prefill_groups(torch, b, shapes, layers, xs, M, reps, stream):
    """Seconds for `reps` passes of the set as a model issues it (q/k/v and
    gate/up as one group call each, forced to the prefill GEMM)."""
    yp = [torch.empty((M, N), dtype=torch.bfloat16, device="cuda") for _, N, _ in shapes]

    def group_pass():
        sp = torch.cuda.current_stream().cuda_stream
        for grp in GROUPS_7B:
            K = shapes[grp[0]][2]
            st = b.linear_group_ptr([layers[i] for i in grp], xs[K].data_ptr(), [yp[i].data_ptr() for i in grp],
                                    M, sp, b.KERNEL_PREFILL)
            if st != 0:
                raise RuntimeError(b.status_string(st))
    with torch.cuda.stream(stream):
        group_pass()
    torch.cuda.synchronize()
    gg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gg, stream=stream):
        group_pass()
    return time_graphs(torch, [gg], reps, 3, stream)


def time_prefill_layers(torch, b, shapes, glayers, xs, ys, M, reps, stream):
    """Seconds for `reps` passes of the prefill GEMM over the layer set `glayers`."""
    def grouped_pass():
        sp = torch.cuda.current_stream().cuda_stream
        for (_, N, K), h in zip(shapes, glayers):
            st = h.forward_ptr(xs[K].data_ptr(), ys[N].data_ptr(), M, sp, b.KERNEL_PREFILL)
            if st != 0:
                raise RuntimeError(b.status_string(st))
    with torch.cuda.stream(stream):
        grouped_pass()
    torch.cuda.synchronize()
    gg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gg, stream=stream):
        grouped_pass()
    return time_graphs(torch, [gg], reps, 3, stream)


# ---------------------------------------------------------------------------
# configs 0, 3, 4 and the dense decode reference
# ---------------------------------------------------------------------------
def capture(torch, fn, stream):
    """Run `fn` once on `stream`, then capture it in a CUDA graph."""
    with torch.cuda.stream(stream):
        fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    return g


def make_io(torch, shapes, M):
    xs, ys = {}, {}
    for pi, (_, N, K) in enumerate(shapes):
        if K not in xs:
            xb = synth.activations(0, 4, 100 + M, M, K)
            xs[K] = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
        ys[pi] = torch.empty((M, N), dtype=torch.bfloat16, device="cuda")
    return xs, ys


def stack_pass(binding, stack, shapes, groups, xs, ys, M):
    def fn():
        sp = __import__("torch").cuda.current_stream().cuda_stream
        for layer in stack:
            for grp in groups:
                K = shapes[grp[0]][2]
                st = binding.linear_group_ptr([layer[i] for i in grp], xs[K].data_ptr(),
                                              [ys[i].data_ptr() for i in grp], M, sp)
                if st != 0:
                    raise RuntimeError(f"unisvq call failed: {binding.status_string(st)}")
    return fn


def run_config0(torch, binding, peaks, args, stream):
    """One 4096 x 4096 projection at M = 1 (d = 2): 64 distinct device copies
    (268 MB, larger than L2) called one after the other from a CUDA graph."""
    N = K = 4096
    copies = 64
    codes, A, B = synth.layer_inputs(0, 0, 0, 0, N, K, 2)
    base = binding.UniSVQLinear(codes, A, B)
    hs = [base] + [base.clone() for _ in range(copies - 1)]
    x = torch.from_numpy(synth.activations(0, 0, 1, 1, K).view(np.int16)).view(torch.bfloat16).cuda()
    y = torch.empty((1, N), dtype=torch.bfloat16, device="cuda")

    def fn():
        sp = torch.cuda.current_stream().cuda_stream
        for h in hs:
            st = h.forward_ptr(x.data_ptr(), y.data_ptr(), 1, sp, binding.KERNEL_AUTO)
            if st != 0:
                raise RuntimeError(binding.status_string(st))
    g = capture(torch, fn, stream)
    reps = max(5, args.steps // 8)
    t = time_graphs(torch, [g], reps, args.warmup, stream)
    us = t / reps / copies * 1e6
    nb = algo_bytes(N, K, 1)
    gbs = nb / (us * 1e-6) / 1e9
    kern = KERNEL_NAMES.get(base.query(1)["kernel"], "?")
    for h in hs:
        h.close()
    return {"workload": "one 4096x4096 projection, M=1, d=2 (64 device copies cycled: 268 MB, L2-cold)",
            "us_per_call": round(us, 3), "GB/s": round(gbs, 1), "frac_of_measured_hbm": round(gbs / peaks["hbm_gbs"], 4),
            "roofline_us": round(nb / (peaks["hbm_gbs"] * 1e9) * 1e6, 3), "kernel": kern,
            "timing": "CUDA graph of 64 calls, CUDA events on the launching stream"}


def run_70b(torch, binding, peaks, args, stream):
    """The Llama-2-70B-shaped stack: args.layers_70b layers x {q, o: 8192^2;
    k, v: 1024x8192; gate, up: 28672x8192; down: 8192x28672} (17.1 GB of codes
    at 80 layers), decode batches M in {1, 8, 32}. Returns (result, stack)."""
    shapes = synth.LLAMA2_70B
    nl = args.layers_70b
    stack = build_stack(binding, shapes, nl, 3)
    out = []
    for M in (1, 8, 32):
        xs, ys = make_io(torch, shapes, M)
        g = capture(torch, stack_pass(binding, stack, shapes, GROUPS_7B, xs, ys, M), stream)
        reps = max(3, args.steps // 40)
        t = time_graphs(torch, [g], reps, args.warmup, stream)
        nb = sum(group_bytes(shapes, grp, M) for grp in GROUPS_7B) * nl
        gbs = nb * reps / t / 1e9
        kerns = {"+".join(shapes[i][0] for i in grp):
                 KERNEL_NAMES.get(binding.query_group([stack[0][i] for i in grp], M)["kernel"], "?") for grp in GROUPS_7B}
        out.append({"M": M, "GB/s": round(gbs, 1), "frac_of_measured_hbm": round(gbs / peaks["hbm_gbs"], 4),
                    "ms_per_pass": round(t / reps * 1e3, 3), "kernels": kerns})
        del g
    st = binding.sync_status(stream)
    if st != 0:
        raise RuntimeError(f"device status {binding.status_string(st)}")
    code_gb = sum(N * K // 4 for _, N, K in shapes) * nl / 1e9
    return ({"workload": f"Llama-2-70B-shaped projection set x {nl} layers ({code_gb:.1f} GB of 2-bit codes), d=2",
             "per_M": out, "calls": "q/k/v and gate/up as one group call each, o and down alone",
             "l2": "inputs larger than L2"}, stack)


CROSSOVER_M = (1, 2, 4, 8, 16, 32, 64, 128, 512, 2048)


def run_crossover(torch, binding, peaks, args, stream, stack70):
    """GEMV-to-GEMM crossover on the 70B shapes: for d = 2 (the first 16 layers
    of the 70B stack) and d = 4 (16 fresh layers), every M of CROSSOVER_M
    through unisvq_linear_group's own pick; per M the kernel of each call,
    time per layer and the fraction of the roofline max(bytes / HBM, flops /
    bf16 peak)."""
    shapes = synth.LLAMA2_70B
    nl = min(16, len(stack70))
    rows = []
    for d in (2, 4):
        stack = stack70[:nl] if d == 2 else build_stack(binding, shapes, nl, 4, d=4)
        for M in CROSSOVER_M:
            xs, ys = make_io(torch, shapes, M)
            g = capture(torch, stack_pass(binding, stack, shapes, GROUPS_7B, xs, ys, M), stream)
            reps = 3 if M >= 512 else max(3, args.steps // 40)
            t = time_graphs(torch, [g], reps, 2, stream) / reps
            nb = sum(group_bytes(shapes, grp, M, d) for grp in GROUPS_7B) * nl
            fl = sum(2.0 * M * N * K for _, N, K in shapes) * nl
            t_hbm = nb / (peaks["hbm_gbs"] * 1e9)
            t_tc = fl / (peaks["bf16_tflops"] * 1e12)
            kerns = {"+".join(shapes[i][0] for i in grp):
                     KERNEL_NAMES.get(binding.query_group([stack[0][i] for i in grp], M)["kernel"], "?")
                     for grp in GROUPS_7B}
            rows.append({"d": d, "M": M, "kernels": kerns, "us_per_layer": round(t / nl * 1e6, 2),
                         "GB/s": round(nb / t / 1e9, 1), "TFLOP/s": round(fl / t / 1e12, 1),
                         "bound": "hbm" if t_hbm >= t_tc else "tensor",
                         "frac_of_roofline": round(max(t_hbm, t_tc) / t, 4)})
            del g, xs, ys
        if d == 4:
            for layer in stack:
                for h in layer:
                    h.close()
    st = binding.sync_status(stream)
    if st != 0:
        raise RuntimeError(f"device status {binding.status_string(st)}")
    return {"workload": f"Llama-2-70B-shaped projection set x {nl} layers per d, M in {list(CROSSOVER_M)}",
            "roofline": "max(algorithmic bytes / measured HBM, 2MNK / measured bf16 burst)", "rows": rows}


def run_cublas_decode(torch, peaks, args, stream, ours_sweep):
    """cuBLAS bf16 dense GEMM (torch.matmul) on the decode shapes of the
    Llama-2-7B set, 8 layers of dense weights (1.6 GB, larger than L2), per M of
    the sweep: the speed a dense fp16/bf16 layer has on this GPU."""
    shapes = synth.LLAMA2_7B
    nl = 8
    W = [[torch.randn(N, K, device="cuda", dtype=torch.bfloat16) for _, N, K in shapes] for _ in range(nl)]
    out = []
    for M, ours in zip(M_SWEEP, ours_sweep):
        xs, ys = make_io(torch, shapes, M)

        def fn():
            for layer in W:
                for pi, (_, N, K) in enumerate(shapes):
                    torch.matmul(xs[K], layer[pi].t(), out=ys[pi])
        g = capture(torch, fn, stream)
        reps = max(5, args.steps // 20)
        t = time_graphs(torch, [g], reps, args.warmup, stream) / reps
        dense_bytes = sum(2 * N * K + 2 * M * K + 2 * M * N for _, N, K in shapes) * nl
        us_layer = t / nl * 1e6
        ours_us = ours["us_per_projection"] * len(shapes)
        out.append({"M": M, "dense_us_per_layer": round(us_layer, 2), "dense_GB/s": round(dense_bytes / t / 1e9, 1),
                    "unisvq_us_per_layer": round(ours_us, 2), "speedup_vs_dense": round(us_layer / ours_us, 3)})
        del g
    del W
    return {"workload": "Llama-2-7B projection shapes, dense bf16 weights, 8 layers, torch.matmul (cuBLAS)",
            "per_M": out}


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-bits3", action="store_true", help="skip the 3-bit-code sweep")
    ap.add_argument("--no-rht", action="store_true",
                    help="skip the inverse-RHT sweep (Llama-3-8B shapes)")
    ap.add_argument("--no-grouped", action="store_true",
                    help="skip the per-(row, 128-column group) affine sweep")
    ap.add_argument("--ungrouped", action="store_true",
                    help="one unisvq_linear call per projection instead of grouped calls for q/k/v and gate/up")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--layers-70b", type=int, default=80)
    ap.add_argument("--no-70b", action="store_true", help="skip config 3 (70B stack) and the crossover table")
    ap.add_argument("--no-dense", action="store_true", help="skip the cuBLAS dense decode reference")
    ap.add_argument("--only", choices=["decode", "prefill", "grouped", "rht", "rht7", "bits3"], default=None,
                    help="profiling aid: run only the decode sweep (no e2e/cpu/secondary sweeps), only the "
                         "prefill set, or only one secondary sweep (with --layers layers)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    try:
        run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
