"""Benchmark of the CD verification step on GB300.

One step = one pass of the whole hot path over one batch: the per-row kernel
(Eq. 1 target, reductions, greedy/sampled acceptance, terminal draws) and the tree
walk, through the C ABI (dcd_score_rows + dcd_tree_walk, i.e. dcd_verify_sample
without the test-only residual output), on the batched-serving workload:
32 sequences x 60-node trees of depth 7 (1920 rows), V = 128256, bf16 logits,
alpha in {0.05, 0.1, 0.2}, even sequences greedy and odd ones sampled at T = 1.
Inputs are seeded synthetic data resident in HBM (1.97 GB, larger than the 129 MB
L2, so no flush is needed; about 1.05 GB of it is read per step); each step advances
the Philox offset.

`--workload diagnostics` times the per-row diagnostics pass (dcd_row_diagnostics: the signal
at the CD argmax and the drafter-alignment terms over the same logits plus an fp32 q row per
node, 1.97 GB read per step).

`--workload fused` times the fused LM-head variant instead (dcd_verify_fused_lmhead:
64 sequences x 60 nodes = 3840 rows, hidden states of 8192 and 2048, V = 128256,
bf16, greedy): one step is both output projections on the tensor cores with the CD
epilogue, the per-row combine and the tree walk.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload batched|fused|diagnostics|small]

Prints one JSON line (rank 0).  `--impl reference` times the fp64 CPU oracle on a
bounded sample of the same workload instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "batched_B32_tree60_V128256_bf16_mixed"
FUSED_WORKLOAD = "fused_lmhead_B64_tree60_V128256_Hexp8192_Hama2048_bf16_greedy"
METRIC = "verified draft nodes/sec (CD verification step, 1 GPU)"
DIAG_WORKLOAD = "diagnostics_B32_tree60_V128256_bf16_q_f32"
DIAG_METRIC = "diagnosed rows/sec (per-row CD diagnostics, 1 GPU)"
NOMINAL_HBM_GBS = 8000.0
ROW_WARMUP, ROW_LAUNCHES = 10, 60  # the row kernel's own timing loop  # GB300 HBM3e nominal bandwidth (context; the roofline uses the measured copy)


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _bf16_peak():
    """Sustained dense bf16 TFLOP/s (the fused kernel runs back to back for seconds)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops_sustained"]), "measured bf16_tflops_sustained"
    except Exception:
        return 1700.0, "fallback sustained bf16"


ROW_KERNEL_FILES = ("dcd_cluster.cu", "dcd_device.cuh", "dcd_internal.h")


def _kernel_source_hash(files=ROW_KERNEL_FILES) -> str:
    h = hashlib.sha256()
    for name in files:
        with open(os.path.join(ROOT, "paper_2608_12913_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def _profiled_traffic(kernel_hash: str, summary: str = "cluster_rows_kernel_batched_B32_tree60_V128256.md"):
    """DRAM bytes per launch of a kernel from its committed ncu summary, if it was taken on the
    current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", summary)
    try:
        text = open(path).read()
    except OSError:
        return None
    m_hash = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", text)
    m_bytes = re.search(r"dram_bytes_per_launch:\s*([0-9.e+]+)", text)
    if not m_hash or not m_bytes or m_hash.group(1) != kernel_hash:
        return None
    return float(m_bytes.group(1))


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampler (50 ms period) around the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.samples = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)

    def summary(self, t0: float, t1: float):
        win = [s for t, s in self.samples if t0 - 1.0 <= t <= t1 + 0.1]
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]}
        sm = [float(s[0]) for s in win if s[0].replace(".", "").isdigit()]
        mx = [float(s[1]) for s in win if s[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in win for i in range(4) if len(s) > 4 + i and "Active" in s[4 + i]
                          and "Not" not in s[4 + i]})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(win), "window": "from 1 s before the timed region to its end"}


def algorithmic_bytes(w, residual_rows: float) -> float:
    """Bytes the step must move: both logit rows of every node (bf16), the draft distribution q
    of every row whose sampled rule needs a residual (a rejected sibling; the other rows need q
    only at their children's tokens), the tree, parameters and outputs."""
    es = 2 if w.dtype == "bf16" else 4
    logits = 2 * w.R * w.V * es
    qb = residual_rows * w.V * 4
    small = w.R * (4 + 4) + w.B * 12 + w.R * 12 + w.B * (8 + w.N * 4)
    return logits + qb + small


def residual_rows_per_step(w, out, ws, stream, offsets, distinct: bool = False) -> float:
    """Mean number of rows handed to residual passes over the given Philox offsets (the
    workspace header's word 4 counts them; the outcome depends only on inputs and offset)."""
    import torch
    from paper_2608_12913_gb300 import dcd
    if w.q is None:
        return 0.0
    counts = []
    for off in offsets:
        dcd.dcd_score_rows(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, q=w.q,
                           temperature=w.temperature, seed=w.seed, offset=off, out=out, workspace=ws, stream=stream,
                           distinct=distinct)
        counts.append(ws[16:20].view(torch.int32).clone())
    torch.cuda.synchronize()
    return float(torch.stack(counts).double().mean().item())


def max_over_ranks(ms: float, dist, device) -> float:
    """The slowest rank's time: every rank of the job calls it (a MAX all-reduce)."""
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world: int, units_per_rank: int, ms_per_step: float) -> float:
    """Whole-job throughput: every rank processes its own batch (weak scaling), so the job's
    units per step are world x units_per_rank, over the slowest rank's step time."""
    return world * units_per_rank / (ms_per_step / 1e3)


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local



def _parse_cpulist(text: str) -> list:
    cpus = []
    for part in text.split(","):
        if "-" in part:
            a, b = part.split("-")
            cpus.extend(range(int(a), int(b) + 1))
        elif part.strip():
            cpus.append(int(part))
    return cpus


def gpu_numa_cpus(index: int):
    """The NUMA node the GPU is attached to (from its PCI device in sysfs) and that node's CPUs;
    (None, []) where the platform does not say."""
    try:
        bus = subprocess.run(["nvidia-smi", "-i", str(index), "--query-gpu=pci.bus_id", "--format=csv,noheader"],
                             capture_output=True, text=True, timeout=30).stdout.strip()
        dom, rest = bus.split(":", 1)
        sysid = f"{int(dom, 16):04x}:{rest}".lower()
        with open(f"/sys/bus/pci/devices/{sysid}/numa_node") as f:
            node = int(f.read().strip())
        if node < 0:
            return None, []
        with open(f"/sys/devices/system/node/node{node}/cpulist") as f:
            return node, _parse_cpulist(f.read().strip())
    except Exception:
        return None, []


class near_gpu:
    """Runs the enclosed host allocations on the CPUs of the GPU's NUMA node, so that page-locked
    buffers are placed in the memory next to it (the allocating thread's node)."""

    def __init__(self, index: int):
        self.node, self.cpus = gpu_numa_cpus(index)
        self.saved = None

    def __enter__(self):
        if self.cpus and hasattr(os, "sched_setaffinity"):
            self.saved = os.sched_getaffinity(0)
            try:
                os.sched_setaffinity(0, self.cpus)
            except OSError:
                self.saved = None
        return self

    def __exit__(self, *exc):
        if self.saved is not None:
            os.sched_setaffinity(0, self.saved)
        return False


def _parity_summary(gpu: dict, ref: dict, seqs) -> dict:
    """Token, length and path mismatches and the largest |cd_logprob| difference of the given
    sequences (outputs on the host; the oracle's in fp64)."""
    import numpy as np
    seqs = list(seqs)
    al = np.asarray(gpu["accept_len"])[seqs]
    bo = np.asarray(gpu["bonus"])[seqs]
    pa = np.asarray(gpu["accept_path"])[seqs]
    mism = int(((al != ref["accept_len"][seqs]) | (bo != ref["bonus"][seqs]) |
                (pa != ref["accept_path"][seqs]).any(axis=1)).sum())
    lg = np.asarray(gpu["cd_logprob"], dtype=np.float64)[seqs]
    lr = ref["cd_logprob"][seqs]
    fin = np.isfinite(lr)
    dl = float(np.abs(lg[fin] - lr[fin]).max()) if fin.any() else 0.0
    return {"sequences": len(seqs), "mismatched_sequences": mism, "max_abs_dlogprob": dl,
            "nonfinite_pattern_equal": bool(np.array_equal(np.isfinite(lg), fin))}


def small_config(cfg: int, dev, warmup: int = 5, graph_calls: int = 64, reps: int = 4) -> dict:
    """The three small workloads as one call each (a 6-node fp32 chain at V = 32000; a 60-node bf16
    tree at V = 128256, greedy or sampled at T = 1): microseconds per call from CUDA-graph replays of
    `graph_calls` calls (the host's launch cost left out), eagerly launched, and end to end (inputs
    from pinned host memory, results back); the oracle on the same inputs, timed on the host cores,
    and the parity of one call against it."""
    import numpy as np
    import torch

    import oracle
    from paper_2608_12913_gb300 import dcd, workloads

    w_host = workloads.make_config(cfg, margin_fn=oracle.margin_fn)
    w = w_host.to(dev)
    B, N, V = w.B, w.N, w.V
    R = B * N
    sampled = w.q is not None and bool((w.temperature > 0).any())
    out = dcd.alloc_outputs(B, N, dev)
    ws = dcd.alloc_workspace(B, N, V, dev, dtype=dcd.DCD_F32 if w.dtype == "f32" else dcd.DCD_BF16)
    keys = ("z_exp", "z_ama", "q", "tokens", "parents", "alpha", "beta", "temperature")
    resident = {k: getattr(w, k) for k in keys if getattr(w, k) is not None}

    def call(i, stream, d=resident):
        if sampled:
            dcd.dcd_verify_sample(d["z_exp"], d["z_ama"], d["q"], d["tokens"], d["parents"], d["alpha"],
                                  d["temperature"], w.seed, i, d.get("beta"), out=out, workspace=ws, stream=stream)
        else:
            dcd.dcd_verify_greedy(d["z_exp"], d["z_ama"], d["tokens"], d["parents"], d["alpha"], d.get("beta"),
                                  out=out, workspace=ws, stream=stream)

    stream = torch.cuda.Stream(device=dev)
    # parity of one call (offset w.offset) against the oracle, and the oracle's time per call
    with torch.cuda.stream(stream):
        call(w.offset, stream)
    stream.synchronize()
    if dcd.dcd_get_device_error(ws, stream) != 0:
        raise RuntimeError(f"config {cfg}: device error bits set")
    gpu = {k: out[k].cpu().numpy() for k in ("accept_len", "accept_path", "bonus", "cd_logprob")}
    threads = oracle.max_threads()
    t0 = time.perf_counter()
    ref = oracle.verify_workload(w_host, nthreads=threads)
    oracle_s = time.perf_counter() - t0
    parity = _parity_summary(gpu, ref, range(B))
    with torch.cuda.stream(stream):
        for i in range(warmup):
            call(i, stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for i in range(graph_calls):
            call(i, stream)
    graph.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        graph.replay()
    b.record()
    torch.cuda.synchronize()
    graph_us = a.elapsed_time(b) * 1e3 / (reps * graph_calls)
    calls = reps * graph_calls
    with torch.cuda.stream(stream):
        a.record(stream)
        for i in range(calls):
            call(i, stream)
        b.record(stream)
    torch.cuda.synchronize()
    eager_us = a.elapsed_time(b) * 1e3 / calls
    with near_gpu(dev.index if dev.index is not None else 0):
        host = {k: v.cpu().pin_memory() for k, v in resident.items()}
        res_host = {k: torch.empty_like(out[k], device="cpu").pin_memory() for k in ("accept_len", "accept_path",
                                                                                     "bonus")}
    dst = {k: torch.empty_like(v, device=dev) for k, v in host.items()}
    h2d = dcd.upload_inputs(host, dst, N, stream)
    d2h = sum(v.numel() * v.element_size() for v in res_host.values())

    def e2e_call(i):
        dcd.upload_inputs(host, dst, N, stream)
        call(i, stream, dst)
        with torch.cuda.stream(stream):
            for k in res_host:
                res_host[k].copy_(out[k], non_blocking=True)

    e2e_call(0)
    torch.cuda.synchronize()
    n_e2e = graph_calls
    a.record(stream)
    for i in range(n_e2e):
        e2e_call(i + 1)
    b.record(stream)
    torch.cuda.synchronize()
    e2e_us = a.elapsed_time(b) * 1e3 / n_e2e
    if dcd.dcd_get_device_error(ws, stream) != 0:
        raise RuntimeError(f"config {cfg}: device error bits set")
    path = ("one launch (greedy_small_kernel)" if not sampled and R <= 512 and N <= 256
            else "cluster row kernel + tree walk")
    es = 4 if w.dtype == "f32" else 2
    return {"workload": w.name, "B": B, "N": N, "V": V, "logits": w.dtype, "sampled": sampled, "path": path,
            "us_per_call_graph": graph_us, "us_per_call_eager": eager_us, "us_per_call_e2e": e2e_us,
            "nodes_per_s_graph": R / (graph_us / 1e6),
            "algorithmic_bytes_per_call": float(R * V * 2 * es),
            "e2e_h2d_bytes_per_call": h2d, "e2e_d2h_bytes_per_call": d2h,
            "timing": f"{reps} replays of a CUDA graph of {graph_calls} calls; eager and end-to-end: "
                      f"{calls} and {n_e2e} back-to-back calls",
            "oracle": {"ms_per_call": oracle_s * 1e3, "cores": threads, "kind": "oracle",
                       "sample": "the whole call"},
            "parity": parity}


def fused_config(dev, steps: int = 30, warmup: int = 3, soak_s: float = 1.0) -> dict:
    """The fused LM-head workload (64 x 60 rows, hidden 8192 and 2048, V = 128256,
    bf16, greedy): the tensor-core launch's TFLOP/s against the measured sustained bf16 peak, from
    CUDA events around it on every step, with the clocks sampled while it runs; the oracle (fp64
    logits and the row definition) on one sequence, and that sequence's parity."""
    import numpy as np
    import torch

    import oracle
    from paper_2608_12913_gb300 import dcd, workloads

    w = workloads.make_fused_torch(device=dev, seed=4)
    B, N, V = w.B, w.N, w.V
    R = B * N
    H_exp, H_ama = w.h_exp.shape[1], w.h_ama.shape[1]
    flop = 2.0 * R * V * (H_exp + H_ama)
    out = dcd.alloc_outputs(B, N, dev)
    ws = torch.empty(dcd.fused_workspace_bytes(B, N, V), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(evs=None):
        dcd.dcd_verify_fused_lmhead(w.h_exp, w.w_exp, w.h_ama, w.w_ama, w.tokens, w.parents, w.alpha, None, out=out,
                                    workspace=ws, stream=stream, gemm_events=evs)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    if dcd.dcd_get_device_error(ws) != 0:
        raise RuntimeError("fused: device error bits set")
    gpu = {k: out[k].cpu().numpy() for k in ("accept_len", "accept_path", "bonus", "cd_logprob")}
    sampler = ClockSampler(dev.index if dev.index is not None else 0)
    sampler.start()
    t_soak = time.time()
    while time.time() - t_soak < soak_s:
        step()
        torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    t0 = time.time()
    start.record(stream)
    for k in range(steps):
        step(evs[k])
    stop.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    sampler.stop()
    gemm_ms = statistics.median(a.elapsed_time(b) for a, b in evs)
    step_ms = start.elapsed_time(stop) / steps
    peak, peak_src = _bf16_peak()
    achieved = flop / (gemm_ms / 1e3) / 1e12
    threads = oracle.max_threads()
    t2 = time.perf_counter()
    ref = oracle.verify_fused_workload(w, nthreads=threads, seqs=[0])
    oracle_s = time.perf_counter() - t2
    rows = ref["rows"].reshape(-1)[:N]
    amb = int((rows["gap_argmax"] < 2e-4).sum())  # within the GEMM's fp32 rounding of the logits
    parity = _parity_summary(gpu, {k: ref[k] for k in ("accept_len", "accept_path", "bonus", "cd_logprob")}, [0])
    parity["ambiguous_rows"] = amb
    return {"workload": FUSED_WORKLOAD, "B": B, "N": N, "V": V, "H_exp": H_exp, "H_ama": H_ama,
            "ms_per_step": step_ms, "nodes_per_s": R / (step_ms / 1e3),
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                         "frac": achieved / peak, "kernel": "fused_lmhead_kernel", "peak_source": peak_src,
                         "algorithmic_flops_per_launch": flop, "gemm_kernel_ms": gemm_ms,
                         "gemm_kernel_samples": steps},
            "clocks": sampler.summary(t0, t1),
            "oracle": {"s_per_sequence": oracle_s, "cores": threads, "kind": "oracle",
                       "sample": f"sequence 0 of {B} ({N} rows: fp64 logits and the row oracle)"},
            "parity": parity}


def diag_config(w, dev, launches: int = 60, warmup: int = 10) -> dict:
    """The per-row diagnostics pass over a resident batch `w` (its logits and q, x* and cd_lse from a
    greedy verification call): the streaming kernel's GB/s from CUDA events around each of
    `launches` launches; the oracle on two rows, timed on one host thread, and their parity."""
    import numpy as np
    import torch

    import oracle
    from paper_2608_12913_gb300 import dcd

    B, N, V = w.B, w.N, w.V
    R = B * N
    zp, zq, q = w.z_exp.reshape(R, V), w.z_ama.reshape(R, V), w.q.reshape(R, V)
    stream = torch.cuda.current_stream()
    o = dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, stream=stream)
    xstar = o["cd_argmax"].reshape(-1).contiguous()
    cd_lse = o["cd_lse"].reshape(-1).contiguous()
    wsd = torch.empty(dcd.diagnostics_workspace_bytes(B, N, V), dtype=torch.uint8, device=dev)
    diag = torch.empty(R, dcd.DIAG_COLS, dtype=torch.float32, device=dev)

    def step(evs=None):
        dcd.dcd_row_diagnostics(zp, zq, B, N, q=q, xstar=xstar, cd_lse=cd_lse, alpha=w.alpha, beta=w.beta, out=diag,
                                workspace=wsd, stream=stream, pass_events=evs)

    for _ in range(warmup):
        step()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(launches)]
    torch.cuda.synchronize()
    for e in evs:
        step(e)
    torch.cuda.synchronize()
    pass_ms = statistics.median(a.elapsed_time(b) for a, b in evs)
    alg = float(R * V * (2 * 2 + 4))
    peak, peak_kind = _peaks()
    achieved = alg / (pass_ms / 1e3) / 1e9
    rows = [1, R - 1]
    xs = xstar.cpu().numpy()
    got = diag[rows].cpu().numpy().astype(np.float64)
    t0 = time.perf_counter()
    ref = _diag_oracle_rows(w, rows, xs)
    oracle_s = time.perf_counter() - t0
    fin = ~np.isnan(ref)
    err = np.abs(got[fin] - ref[fin]) / np.maximum(1.0, np.abs(ref[fin]))
    return {"workload": DIAG_WORKLOAD, "rows": R, "pass_ms": pass_ms, "rows_per_s": R / (pass_ms / 1e3),
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "frac_nominal": achieved / NOMINAL_HBM_GBS, "kernel": "diag_partial_kernel",
                         "peak_source": f"{peak_kind} hbm_gbs", "algorithmic_bytes_per_launch": alg,
                         "pass_kernel_samples": launches},
            "oracle": {"ms_per_row": oracle_s * 1e3 / len(rows), "cores": 1, "kind": "oracle",
                       "sample": f"rows {rows}, one thread"},
            "parity": {"rows": len(rows), "max_scaled_error": float(err.max()) if err.size else 0.0,
                       "nan_pattern_equal": bool(np.array_equal(np.isnan(got), np.isnan(ref)))}}

def run_reference(args):
    """The fp64 CPU oracle timed as the reference arm (rank 0 only)."""
    ws, rank, _ = _dist_env()
    if rank != 0:
        return 0
    import oracle
    from paper_2608_12913_gb300 import workloads
    if args.workload == "diagnostics":
        return run_reference_diagnostics(args, ws)
    w = workloads.make_config(3, B=2)  # sequences 0 (greedy) and 1 (sampled) of the batched workload
    threads = oracle.max_threads()
    for _ in range(args.warmup):
        oracle.verify_workload(w, nthreads=threads)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.verify_workload(w, nthreads=threads)
    dt = (time.perf_counter() - t0) / max(1, args.steps)
    value = w.R / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "nodes/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "sample": "sequences 0-1 of the batch (120 rows, one greedy, one sampled)",
                   "V": w.V, "N": w.N},
        "cpu_baseline": {"value": value, "unit": "nodes/s", "cores": threads, "kind": "oracle",
                         "sample": "2 of 32 sequences (120 of 1920 rows) per step"},
        "e2e": {"value": value, "unit": "nodes/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def _diag_oracle_rows(w, rows, xstar):
    """The oracle's diagnostics for the given rows of workload `w` (inputs as stored), with the
    decomposition column for sequences with beta = 0 (greedy, as the benchmark's x* call)."""
    import numpy as np

    import oracle
    from paper_2608_12913_gb300 import dcd
    R = w.B * w.N
    zp = w.z_exp.reshape(R, w.V)
    zq = w.z_ama.reshape(R, w.V)
    q = w.q.reshape(R, w.V)
    out = np.full((len(rows), dcd.DIAG_COLS), np.nan)
    for i, g in enumerate(rows):
        b = g // w.N
        beta = 0.0 if w.beta is None else float(w.beta[b])
        d = oracle.row_diagnostics(zp[g].cpu(), zq[g].cpu(), int(xstar[g]), q=q[g].cpu().numpy(), dtype=w.dtype,
                                   alpha=float(w.alpha[b]) if beta == 0.0 else None)
        out[i] = [d[k] for k in dcd.DIAG_FIELDS]
    return out


def run_reference_diagnostics(args, world):
    from paper_2608_12913_gb300 import workloads
    w = workloads.make_config(3, B=2)
    R = w.B * w.N
    xstar = [(g * 7919) % w.V for g in range(R)]
    for _ in range(args.warmup):
        _diag_oracle_rows(w, range(R), xstar)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _diag_oracle_rows(w, range(R), xstar)
    dt = (time.perf_counter() - t0) / max(1, args.steps)
    value = R / dt
    line = {
        "impl": "reference", "metric": DIAG_METRIC, "value": value, "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": DIAG_WORKLOAD, "sample": "sequences 0-1 of the batch (120 rows) per step",
                   "V": w.V, "N": w.N},
        "cpu_baseline": {"value": value, "unit": "rows/s", "cores": 1, "kind": "oracle",
                         "sample": "2 of 32 sequences (120 of 1920 rows) per step, one thread"},
        "e2e": {"value": value, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def cpu_baseline(w_dev, budget_s: float = 8.0):
    """Times the oracle, as it stands, on the first k sequences of the benchmark batch."""
    import oracle
    threads = oracle.max_threads()
    k = 2
    best = None
    while True:
        t0 = time.perf_counter()
        oracle.verify_workload(w_dev, nthreads=threads, seqs=list(range(k)))
        dt = time.perf_counter() - t0
        best = (k, dt)
        if dt * 2.2 > budget_s or k >= w_dev.B:
            break
        k = min(w_dev.B, 2 * k)
    k, dt = best
    # the same oracle on one thread, over the first two sequences (one greedy, one sampled)
    t0 = time.perf_counter()
    oracle.verify_workload(w_dev, nthreads=1, seqs=[0, 1])
    dt1 = time.perf_counter() - t0
    return {"value": k * w_dev.N / dt, "unit": "nodes/s", "cores": threads, "kind": "oracle",
            "sample": f"first {k} of {w_dev.B} sequences ({k * w_dev.N} rows, V={w_dev.V}), {dt:.1f} s wall",
            "single_thread": {"value": 2 * w_dev.N / dt1, "unit": "nodes/s", "cores": 1,
                              "sample": f"sequences 0-1 ({2 * w_dev.N} rows), {dt1:.1f} s wall"}}


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2608_12913_gb300 import dcd, workloads

    world, rank, local = _dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    # weak scaling: every rank verifies its own full batch
    w = workloads.make_config_torch(3, device=dev, seed=3 + rank, B=args.batch or 32,
                                    temperatures=(0.0,) if args.greedy else (0.0, 1.0))
    B, N, V = w.B, w.N, w.V
    R = B * N
    out = dcd.alloc_outputs(B, N, dev)
    ws = dcd.alloc_workspace(B, N, V, dev)
    stream = torch.cuda.current_stream()

    def step(i, evs=None):
        if evs is not None:
            evs[0].record(stream)
        if w.q is None:
            dcd.dcd_score_rows(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, out=out, workspace=ws,
                               stream=stream)
        else:
            dcd.dcd_score_rows(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, q=w.q,
                               temperature=w.temperature, seed=w.seed, offset=i, out=out, workspace=ws, stream=stream,
                               distinct=args.distinct)
        if evs is not None:
            evs[1].record(stream)
        dcd.dcd_tree_walk(B, N, V, out, ws, stream=stream)

    for i in range(args.warmup):
        step(i)
    if dcd.dcd_get_device_error(ws) != 0:
        raise RuntimeError("device error bits set during warm-up")
    sampler = ClockSampler(local)
    sampler.start()
    # keep the GPU busy for a second so the clock samples describe the loaded state
    t_soak = time.time()
    i = args.warmup
    while not args.no_soak and time.time() - t_soak < 1.0:
        step(i)
        i += 1
        if i % 64 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()

    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    start.record(stream)
    for k in range(args.steps):
        step(1_000_000 + k)
    stop.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_wall1 = time.time()
    # The row kernel's own duration: CUDA events around each of ROW_LAUNCHES launches after
    # ROW_WARMUP more, whatever --steps is (an event between the row kernel and the tree walk
    # breaks the walk's programmatic dependent launch, so the step loop above has none)
    for k in range(ROW_WARMUP):
        step(3_000_000 + k)
    row_evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(ROW_LAUNCHES)]
    t_row0 = time.time()
    for k in range(ROW_LAUNCHES):
        step(4_000_000 + k, row_evs[k])
    torch.cuda.synchronize()
    t_row1 = time.time()
    sampler.stop()
    elapsed_ms = start.elapsed_time(stop)
    row_ms = [a.elapsed_time(b) for a, b in row_evs]
    if world > 1:
        elapsed_ms = max_over_ranks(elapsed_ms, dist, dev)
    if dcd.dcd_get_device_error(ws) != 0:
        raise RuntimeError("device error bits set during the timed region")
    ms_per_step = elapsed_ms / args.steps
    value = job_value(world, R, ms_per_step)

    # roofline of the dominant kernel (the row kernel) from its own events; the rows that took
    # residual passes are counted on a replay of every 32nd timed offset
    replay = [4_000_000 + k for k in range(0, ROW_LAUNCHES, 4)]
    res_rows = residual_rows_per_step(w, out, ws, stream, replay, args.distinct)
    alg = algorithmic_bytes(w, res_rows)
    row_avg_s = statistics.median(row_ms) / 1e3
    achieved = alg / row_avg_s / 1e9
    peak, peak_kind = _peaks()
    # the library streams rows with the cluster-per-row kernel (both sibling rules)
    kname = "cluster_rows_kernel"
    khash = _kernel_source_hash(ROW_KERNEL_FILES)
    # the profile covers the default workload (32 sequences, mixed, i.i.d. siblings) only
    traffic = _profiled_traffic(khash) if B == 32 and not args.greedy and not args.distinct else None
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "frac_nominal": achieved / NOMINAL_HBM_GBS, "nominal_peak": NOMINAL_HBM_GBS,
                "traffic": traffic, "kernel": kname, "peak_source": f"{peak_kind} hbm_gbs",
                "algorithmic_bytes_per_launch": alg, "residual_rows_per_step": res_rows,
                "row_kernel_ms": row_avg_s * 1e3, "row_kernel_samples": len(row_ms),
                "row_kernel_timing": f"median of {ROW_LAUNCHES} event-timed launches after {ROW_WARMUP} warm-ups",
                "clocks": sampler.summary(t_row0, t_row1),
                "kernel_source_sha256_16": khash}

    # end to end through the public API: pinned host inputs -> device, verify, results -> host
    e2e = None
    if not args.no_e2e:
        # page-locked buffers in the memory of the GPU's NUMA node (allocated from its CPUs)
        with near_gpu(local) as place:
            host = {k: getattr(w, k).cpu().pin_memory() for k in ("z_exp", "z_ama", "q", "tokens", "parents",
                                                                   "alpha", "beta", "temperature")
                    if getattr(w, k) is not None}
            res_host = {k: torch.empty_like(out[k], device="cpu").pin_memory()
                        for k in ("accept_len", "accept_path", "bonus")}
        dst = {k: torch.empty_like(v, device=dev) for k, v in host.items()}
        # q is copied only for the sampled sequences: the verification reads no other row of it
        h2d = dcd.upload_inputs(host, dst, N, stream)
        d2h = sum(v.numel() * v.element_size() for v in res_host.values())
        n_e2e = max(3, min(args.steps, 10))

        def e2e_step(i):
            dcd.upload_inputs(host, dst, N, stream)
            o = dcd.dcd_verify_sample(dst["z_exp"], dst["z_ama"], dst.get("q"), dst["tokens"], dst["parents"],
                                      dst["alpha"], dst["temperature"], w.seed, 2_000_000 + i, dst["beta"], out=out,
                                      workspace=ws, stream=stream, distinct=args.distinct)
            for k in res_host:
                res_host[k].copy_(o[k], non_blocking=True)

        e2e_step(0)
        torch.cuda.synchronize()
        a, b2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(n_e2e):
            e2e_step(i + 1)
        b2.record(stream)
        torch.cuda.synchronize()
        e_ms = a.elapsed_time(b2) / n_e2e
        # the host link alone: the same upload without the verification, each timed on its own
        # (back-to-back uploads contend with one another), the median
        ups = []
        for i in range(n_e2e):
            a.record(stream)
            dcd.upload_inputs(host, dst, N, stream)
            b2.record(stream)
            torch.cuda.synchronize()
            ups.append(a.elapsed_time(b2))
        up_ms = statistics.median(ups)
        if world > 1:
            e_ms = max_over_ranks(e_ms, dist, dev)
        e2e = {"value": job_value(world, R, e_ms), "unit": "nodes/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e_ms, "steps": n_e2e,
               "h2d_ms_per_step": up_ms, "h2d_gbs": h2d / (up_ms / 1e3) / 1e9,
               "pinned_numa_node": place.node,
               "bound": "host link: the step's inputs cross it every step (its rate is h2d_gbs)"}
        del dst, host

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "nodes/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": (WORKLOAD if B == 32 else f"{WORKLOAD} (profiling case, B={B})") +
                       (" siblings-without-replacement" if args.distinct else ""),
                       "B": B, "N": N, "V": V, "rows": R, "logits": "bf16",
                       "sampled_sequences": int((w.temperature > 0).sum().item()),
                       "bytes_per_step": alg, "l2": "inputs (1.97 GB resident) larger than L2; no flush",
                       "parallelism": f"replicas x{world} (sequence batches, no collective in the path)"},
            "roofline": roofline,
            "clocks": sampler.summary(t_wall0, t_wall1),
            "e2e": e2e,
            "gpu_launches": 2 * args.steps,
        }
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(w)
        if not args.no_configs:
            line["configs"] = all_configs(w, dev, out, ws, stream, line)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def all_configs(w, dev, out, ws, stream, line) -> dict:
    """Every benchmark workload measured in the same run, each with the oracle's time on the
    host cores and a parity summary: the three small calls (0-2), this batch (3, the headline), the
    fused LM-head variant (4), and the per-row diagnostics pass over this batch."""
    import oracle
    from paper_2608_12913_gb300 import dcd
    res = {}
    for cfg, key in ((0, "0_tiny_chain"), (1, "1_tree_greedy"), (2, "2_tree_sampled")):
        res[key] = small_config(cfg, dev)
    # config 3: the headline (above), with the parity of sequences 0-1 of one call
    off = 5_000_000
    dcd.dcd_score_rows(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, q=w.q, temperature=w.temperature,
                       seed=w.seed, offset=off, out=out, workspace=ws, stream=stream)
    dcd.dcd_tree_walk(w.B, w.N, w.V, out, ws, stream=stream)
    gpu = {k: out[k].cpu().numpy() for k in ("accept_len", "accept_path", "bonus", "cd_logprob")}
    import dataclasses
    ref = oracle.verify_workload(dataclasses.replace(w, offset=off), nthreads=oracle.max_threads(), seqs=[0, 1])
    rows = ref["rows"][:2]
    amb = int(((rows["gap_argmax"] < 2e-5) | (rows["gap_accept"] < 1e-5) | (rows["gap_race"] < 1e-4)).sum())
    par = _parity_summary(gpu, ref, [0, 1])
    par["ambiguous_rows"] = amb
    cb = line.get("cpu_baseline", {})
    res["3_batched"] = {"workload": WORKLOAD, "ms_per_step": line["ms_per_step"], "nodes_per_s": line["value"],
                        "roofline": {k: line["roofline"][k] for k in ("achieved", "peak", "frac", "frac_nominal",
                                                                        "row_kernel_ms")},
                        "oracle": {"nodes_per_s": cb.get("value"), "cores": cb.get("cores"),
                                   "sample": cb.get("sample")},
                        "parity": par}
    res["4_fused"] = fused_config(dev)
    res["diagnostics"] = diag_config(w, dev)
    return res


def run_fused(args):
    """The fused LM-head variant: tensor-core bound; roofline in TFLOP/s of the GEMM kernel."""
    import torch
    import torch.distributed as dist

    from paper_2608_12913_gb300 import dcd, workloads

    world, rank, local = _dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = workloads.make_fused_torch(device=dev, seed=4 + rank, beta=args.beta, B=args.batch)
    B, N, V = w.B, w.N, w.V
    R = B * N
    H_exp, H_ama = w.h_exp.shape[1], w.h_ama.shape[1]
    beta = w.beta if args.beta > 0 else None
    # with a plausibility mask the expert's GEMM runs twice (a max sweep, then the masked sweep)
    flop = 2.0 * R * V * (H_exp + H_ama + (H_exp if beta is not None else 0))
    out = dcd.alloc_outputs(B, N, dev)
    ws = torch.empty(dcd.fused_workspace_bytes(B, N, V), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    steps = args.steps

    def step(evs=None):
        dcd.dcd_verify_fused_lmhead(w.h_exp, w.w_exp, w.h_ama, w.w_ama, w.tokens, w.parents, w.alpha, beta,
                                    out=out, workspace=ws, stream=stream, gemm_events=evs)

    for _ in range(args.warmup):
        step()
    if dcd.dcd_get_device_error(ws) != 0:
        raise RuntimeError("device error bits set during warm-up")
    sampler = ClockSampler(local)
    sampler.start()
    t_soak = time.time()
    while not args.no_soak and time.time() - t_soak < 1.0:
        step()
        torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for e in evs:  # create the events outside the timed region
        e[0].record(stream)
        e[1].record(stream)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    start.record(stream)
    for k in range(steps):
        step(evs[k])
    stop.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_wall1 = time.time()
    sampler.stop()
    elapsed_ms = start.elapsed_time(stop)
    gemm_ms = statistics.mean(a.elapsed_time(b) for a, b in evs)
    if world > 1:
        elapsed_ms = max_over_ranks(elapsed_ms, dist, dev)
    if dcd.dcd_get_device_error(ws) != 0:
        raise RuntimeError("device error bits set during the timed region")
    ms_per_step = elapsed_ms / steps
    value = job_value(world, R, ms_per_step)
    peak, peak_src = _bf16_peak()
    achieved = flop / (gemm_ms / 1e3) / 1e12
    khash = _kernel_source_hash(("dcd_fused.cu", "dcd_fused.h", "dcd_tc.cuh", "dcd_device.cuh"))
    # DRAM bytes of one tensor-core launch from the committed launch list (the unmasked call; the
    # masked call runs two sweeps of different traffic, not captured)
    traffic = (_profiled_traffic(khash, "fused_lmhead_kernel_B64_tree60_V128256_H8192_2048.md")
               if beta is None and B == 64 else None)
    roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": traffic, "kernel": "fused_lmhead_kernel", "peak_source": peak_src,
                "kernel_source_sha256_16": khash,
                "algorithmic_flops_per_launch": flop, "gemm_kernel_ms": gemm_ms,
                "flops_counted": "both LM-head GEMMs" + ("; with beta the expert's twice (max sweep, then masked)"
                                                           if beta is not None else "")}

    # end to end: the step's hidden states and tree come from pinned host memory (the weights
    # are the models' resident parameters), the results go back
    e2e = None
    if not args.no_e2e:
        host = {k: getattr(w, k).cpu().pin_memory() for k in ("h_exp", "h_ama", "tokens", "parents", "alpha")}
        dst = {k: torch.empty_like(v, device=dev) for k, v in host.items()}
        res_host = {k: torch.empty_like(out[k], device="cpu").pin_memory() for k in ("accept_len", "accept_path",
                                                                                     "bonus")}
        h2d = sum(v.numel() * v.element_size() for v in host.values())
        d2h = sum(v.numel() * v.element_size() for v in res_host.values())
        n_e2e = max(3, min(steps, 10))

        def e2e_step():
            for k in host:
                dst[k].copy_(host[k], non_blocking=True)
            o = dcd.dcd_verify_fused_lmhead(dst["h_exp"], w.w_exp, dst["h_ama"], w.w_ama, dst["tokens"],
                                            dst["parents"], dst["alpha"], beta, out=out, workspace=ws, stream=stream)
            for k in res_host:
                res_host[k].copy_(o[k], non_blocking=True)

        e2e_step()
        torch.cuda.synchronize()
        a, b2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n_e2e):
            e2e_step()
        b2.record(stream)
        torch.cuda.synchronize()
        e_ms = a.elapsed_time(b2) / n_e2e
        if world > 1:
            e_ms = max_over_ranks(e_ms, dist, dev)
        e2e = {"value": job_value(world, R, e_ms), "unit": "nodes/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e_ms, "steps": n_e2e}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "nodes/s", "n_gpus": world, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": FUSED_WORKLOAD + (f" beta={args.beta:g}" if beta is not None else "") +
                       (f" (profiling case, B={B})" if B != 64 else ""),
                       "B": B, "N": N, "V": V, "rows": R, "H_exp": H_exp,
                       "H_ama": H_ama, "flop_per_step": flop, "beta": args.beta,
                       "l2": "weights (2.6 GB) larger than L2; no flush",
                       "parallelism": f"replicas x{world} (sequence batches, no collective in the path)"},
            "roofline": roofline,
            "clocks": sampler.summary(t_wall0, t_wall1),
            "e2e": e2e,
            # children, GEMM, combine and walk kernels; with a mask also the max sweep and the row max
            "gpu_launches": (6 if beta is not None else 4) * steps,
        }
        if not args.no_cpu_baseline:
            import oracle
            threads = oracle.max_threads()
            t0 = time.perf_counter()
            oracle.verify_fused_workload(w, nthreads=threads, seqs=[0])
            dt = time.perf_counter() - t0
            # the fp64 logits alone (the blocked library GEMM), reported apart from the CD part
            t1 = time.perf_counter()
            oracle.fused_logits(w.h_exp[:N], w.w_exp)
            oracle.fused_logits(w.h_ama[:N], w.w_ama)
            dt_gemm = time.perf_counter() - t1
            line["cpu_baseline"] = {"value": N / dt, "unit": "nodes/s", "cores": threads, "kind": "oracle",
                                    "sample": f"sequence 0 of {B} ({N} rows: fp64 logits and the row oracle), "
                                              f"{dt:.1f} s wall",
                                    "gemm_s": dt_gemm, "cd_s": max(0.0, dt - dt_gemm)}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def run_diagnostics(args):
    """Per-row diagnostics (signal at the CD argmax, alignment terms) over the batched workload's
    logits and q: a streaming pass bound by HBM; roofline in GB/s of the streaming kernel."""
    import torch
    import torch.distributed as dist

    from paper_2608_12913_gb300 import dcd, workloads

    world, rank, local = _dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = workloads.make_config_torch(3, device=dev, seed=3 + rank, B=args.batch or 32)
    B, N, V = w.B, w.N, w.V
    R = B * N
    zp, zq, q = w.z_exp.reshape(R, V), w.z_ama.reshape(R, V), w.q.reshape(R, V)
    stream = torch.cuda.current_stream()
    o = dcd.dcd_verify_greedy(w.z_exp, w.z_ama, w.tokens, w.parents, w.alpha, w.beta, stream=stream)
    xstar = o["cd_argmax"].reshape(-1).contiguous()  # the CD argmax of every node
    cd_lse = o["cd_lse"].reshape(-1).contiguous()  # its CD normaliser (D_KL(pi_p || pi_CD) by App. B's lemma)
    ws = torch.empty(dcd.diagnostics_workspace_bytes(B, N, V), dtype=torch.uint8, device=dev)
    diag = torch.empty(R, dcd.DIAG_COLS, dtype=torch.float32, device=dev)
    steps = args.steps

    def step(evs=None):
        dcd.dcd_row_diagnostics(zp, zq, B, N, q=q, xstar=xstar, cd_lse=cd_lse, alpha=w.alpha, beta=w.beta, out=diag,
                                workspace=ws, stream=stream, pass_events=evs)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.start()
    t_soak = time.time()
    while not args.no_soak and time.time() - t_soak < 1.0:
        for _ in range(32):
            step()
        torch.cuda.synchronize()
    # the pass's own duration is sampled on every 8th step (the median is reported): events between
    # the pass and the combine break the combine's programmatic dependent launch, so the other
    # steps run as a user's back-to-back calls do
    evs = {k: (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for k in range(0, steps, 8)}
    for e in evs.values():  # create the events outside the timed region
        e[0].record(stream)
        e[1].record(stream)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    start.record(stream)
    for k in range(steps):
        step(evs.get(k))
    stop.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_wall1 = time.time()
    sampler.stop()
    elapsed_ms = start.elapsed_time(stop)
    pass_ms = statistics.median(a.elapsed_time(b) for a, b in evs.values())
    if world > 1:
        elapsed_ms = max_over_ranks(elapsed_ms, dist, dev)
    if not torch.isfinite(diag).all():
        raise RuntimeError("non-finite diagnostics on finite inputs")
    ms_per_step = elapsed_ms / steps
    value = job_value(world, R, ms_per_step)
    alg = float(R * V * (2 * 2 + 4))  # both bf16 logit rows and the fp32 q row of every node
    peak, peak_kind = _peaks()
    achieved = alg / (pass_ms / 1e3) / 1e9
    khash = _kernel_source_hash(("dcd_diag.cu", "dcd_diag.h", "dcd_device.cuh"))
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": (_profiled_traffic(khash, "diag_partial_kernel_B32_tree60_V128256.md")
                            if B == 32 else None),
                "kernel": "diag_partial_kernel", "peak_source": f"{peak_kind} hbm_gbs",
                "algorithmic_bytes_per_launch": alg, "pass_kernel_ms": pass_ms,
                "pass_kernel_samples": len(evs), "kernel_source_sha256_16": khash}

    e2e = None
    if not args.no_e2e:
        host = {"zp": zp.cpu().pin_memory(), "zq": zq.cpu().pin_memory(), "q": q.cpu().pin_memory(),
                "xstar": xstar.cpu().pin_memory(), "cd_lse": cd_lse.cpu().pin_memory()}
        dst = {k: torch.empty_like(v, device=dev) for k, v in host.items()}
        res_host = torch.empty((R, dcd.DIAG_COLS), dtype=torch.float32).pin_memory()
        h2d = sum(v.numel() * v.element_size() for v in host.values())
        d2h = res_host.numel() * 4
        n_e2e = max(3, min(steps, 10))

        def e2e_step():
            for k in host:
                dst[k].copy_(host[k], non_blocking=True)
            r = dcd.dcd_row_diagnostics(dst["zp"], dst["zq"], B, N, q=dst["q"], xstar=dst["xstar"],
                                        cd_lse=dst["cd_lse"], alpha=w.alpha, beta=w.beta, out=diag, workspace=ws,
                                        stream=stream)
            res_host.copy_(r, non_blocking=True)

        e2e_step()
        torch.cuda.synchronize()
        a, b2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n_e2e):
            e2e_step()
        b2.record(stream)
        torch.cuda.synchronize()
        e_ms = a.elapsed_time(b2) / n_e2e
        if world > 1:
            e_ms = max_over_ranks(e_ms, dist, dev)
        e2e = {"value": job_value(world, R, e_ms), "unit": "rows/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e_ms, "steps": n_e2e}
        del dst, host

    if rank == 0:
        line = {
            "metric": DIAG_METRIC, "value": value, "unit": "rows/s", "n_gpus": world, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": DIAG_WORKLOAD if B == 32 else f"{DIAG_WORKLOAD} (profiling case, B={B})",
                       "B": B, "N": N, "V": V, "rows": R, "logits": "bf16", "q": "fp32, every row",
                       "bytes_per_step": alg, "l2": "inputs (1.97 GB resident) larger than L2; no flush",
                       "parallelism": f"replicas x{world} (sequence batches, no collective in the path)"},
            "roofline": roofline,
            "clocks": sampler.summary(t_wall0, t_wall1),
            "e2e": e2e,
            "gpu_launches": 2 * steps,
        }
        if not args.no_cpu_baseline:
            rows = range(min(R, 240))
            xs = xstar.cpu().numpy()
            t0 = time.perf_counter()
            _diag_oracle_rows(w, rows, xs)
            dt = time.perf_counter() - t0
            line["cpu_baseline"] = {"value": len(rows) / dt, "unit": "rows/s", "cores": 1, "kind": "oracle",
                                    "sample": f"first {len(rows)} of {R} rows, one thread, {dt:.1f} s wall"}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def run_small(args):
    """Latency of one small verification call (the small workloads: a 6-node chain at V = 32000,
    or a 60-node tree at V = 128256, greedy or sampled), through the public API.  The device time
    per call is taken from CUDA-graph replays of 64 calls (the host's launch cost left out); the
    eager per-call time is reported beside it."""
    import torch
    import torch.distributed as dist

    from paper_2608_12913_gb300 import dcd, workloads

    world, rank, local = _dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    cfg = args.config
    w = workloads.make_config_torch(cfg, device=dev, seed=cfg + rank)
    B, N, V = w.B, w.N, w.V
    R = B * N
    sampled = w.q is not None
    out = dcd.alloc_outputs(B, N, dev)
    ws = dcd.alloc_workspace(B, N, V, dev, dtype=dcd.DCD_F32 if w.dtype == "f32" else dcd.DCD_BF16)

    keys = ("z_exp", "z_ama", "q", "tokens", "parents", "alpha", "beta", "temperature")
    resident = {k: getattr(w, k) for k in keys if getattr(w, k) is not None}

    def call(i, stream, d=resident):
        if sampled:
            dcd.dcd_verify_sample(d["z_exp"], d["z_ama"], d["q"], d["tokens"], d["parents"], d["alpha"],
                                  d["temperature"], w.seed, i, d["beta"], out=out, workspace=ws, stream=stream)
        else:
            dcd.dcd_verify_greedy(d["z_exp"], d["z_ama"], d["tokens"], d["parents"], d["alpha"], d["beta"], out=out,
                                  workspace=ws, stream=stream)

    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        for i in range(max(args.warmup, 3)):
            call(i, stream)
    stream.synchronize()
    if dcd.dcd_get_device_error(ws, stream) != 0:
        raise RuntimeError("device error bits set during warm-up")
    per_graph = 64
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for i in range(per_graph):
            call(i, stream)
    graph.replay()
    torch.cuda.synchronize()
    reps = max(1, args.steps // per_graph)
    sampler = ClockSampler(local)
    sampler.start()
    t_soak = time.time()
    while not args.no_soak and time.time() - t_soak < 1.0:
        graph.replay()
        torch.cuda.synchronize()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    start.record()
    for _ in range(reps):
        graph.replay()
    stop.record()
    torch.cuda.synchronize()
    t_wall1 = time.time()
    sampler.stop()
    steps = reps * per_graph
    ms_per_step = start.elapsed_time(stop) / steps
    if world > 1:
        ms_per_step = max_over_ranks(ms_per_step, dist, dev)
    # eager calls, the host's launch cost included
    with torch.cuda.stream(stream):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(steps):
            call(i, stream)
        b.record(stream)
    torch.cuda.synchronize()
    eager_ms = a.elapsed_time(b) / steps
    # end to end: every call's inputs come from pinned host memory and its results go back
    host = {k: v.cpu().pin_memory() for k, v in resident.items()}
    dst = {k: torch.empty_like(v, device=dev) for k, v in host.items()}
    res_host = {k: torch.empty_like(out[k], device="cpu").pin_memory() for k in ("accept_len", "accept_path",
                                                                                 "bonus")}
    h2d = dcd.upload_inputs(host, dst, N, stream)
    d2h = sum(v.numel() * v.element_size() for v in res_host.values())
    n_e2e = min(steps, 256)

    def e2e_call(i):
        dcd.upload_inputs(host, dst, N, stream)
        call(i, stream, dst)
        with torch.cuda.stream(stream):
            for k in res_host:
                res_host[k].copy_(out[k], non_blocking=True)

    e2e_call(0)
    torch.cuda.synchronize()
    a2, b2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a2.record(stream)
    for i in range(n_e2e):
        e2e_call(i + 1)
    b2.record(stream)
    torch.cuda.synchronize()
    e2e_ms = a2.elapsed_time(b2) / n_e2e
    if world > 1:
        e2e_ms = max_over_ranks(e2e_ms, dist, dev)
    if dcd.dcd_get_device_error(ws, stream) != 0:
        raise RuntimeError("device error bits set during the timed region")
    es = 4 if w.dtype == "f32" else 2
    alg = float(R * V * 2 * es)  # both logit rows of every node (q: only at children unless rejected)
    peak, peak_kind = _peaks()
    achieved = alg / (ms_per_step / 1e3) / 1e9
    path = "one launch (greedy_small_kernel)" if not sampled and R <= 512 else "cluster row kernel + tree walk"
    if rank == 0:
        line = {
            "metric": METRIC + ", small call", "value": job_value(world, R, ms_per_step), "unit": "nodes/s",
            "n_gpus": world, "steps": steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic",
            "config": {"workload": w.name, "B": B, "N": N, "V": V, "rows": R, "logits": w.dtype,
                       "path": path, "timing": f"CUDA-graph replays of {per_graph} calls",
                       "eager_ms_per_call": eager_ms,
                       "l2": "inputs smaller than L2 and re-read every call: latency, not bandwidth",
                       "parallelism": f"replicas x{world}"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": None, "kernel": "whole call (latency-bound)",
                         "peak_source": f"{peak_kind} hbm_gbs", "algorithmic_bytes_per_launch": alg},
            "clocks": sampler.summary(t_wall0, t_wall1),
            "e2e": {"value": job_value(world, R, e2e_ms), "unit": "nodes/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms, "steps": n_e2e},
            "gpu_launches": (1 if path.startswith("one") else 2) * steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle timing (profiling runs)")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end leg (profiling runs)")
    ap.add_argument("--no-soak", action="store_true", help="skip the 1 s clock soak (profiling runs)")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the per-configuration sub-results (small calls, fused, diagnostics)")
    ap.add_argument("--greedy", action="store_true", help="every sequence greedy (profiling case)")
    ap.add_argument("--batch", type=int, default=None,
                    help="sequences per GPU; the benchmark workloads use 32 (batched, diagnostics) and 64 "
                         "(fused); other values are profiling cases")
    ap.add_argument("--distinct", action="store_true",
                    help="sampled rule for siblings drawn without replacement (DCD_SIBLINGS_DISTINCT)")
    ap.add_argument("--beta", type=float, default=0.0,
                    help="fused workload: plausibility threshold of every sequence (0: no mask, one sweep)")
    ap.add_argument("--workload", choices=("batched", "fused", "diagnostics", "small"), default="batched",
                    help="batched: the streaming step on materialised logits (the headline); fused: the "
                         "fused LM-head variant; diagnostics: the per-row diagnostics pass; small: the "
                         "latency of one small call (--config)")
    ap.add_argument("--config", type=int, choices=(0, 1, 2), default=0,
                    help="small workload: 0 = 6-node chain (fp32, V 32000, greedy), 1 = 60-node tree "
                         "(bf16, V 128256, greedy), 2 = the same tree sampled at T = 1")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        return run_reference(args)
    if args.workload == "fused":
        return run_fused(args)
    if args.workload == "diagnostics":
        return run_diagnostics(args)
    if args.workload == "small":
        return run_small(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
