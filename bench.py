#!/usr/bin/env python3
"""Throughput of the ALR slot-loss hot path on GB300.

One step = the whole path over one batch of the 8B-text workload (d=4096, V=151936, B=16,
2048 anchors = 32768 slot rows; seeded synthetic inputs, rollout feature buffer of 16
sequences x 4096 positions):
    IRA gather of the target hidden rows  ->  fused forward (logits, online LSE, soft CE,
    greedy argmaxes, slot weights, Eq. 1; both logit matrices kept in fp16)  ->  accepted
    length  ->  logit gradient G from the kept logits  ->  dH_d = G W^T  ->  dW += H_d^T G.
The step that recomputes the logits in the backward instead of keeping them is timed beside
it (`recompute`).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gpu|reference]

Prints one JSON line (rank 0).  `value` is slot rows per second over all ranks with inputs
resident in HBM; `e2e` repeats the measurement with the step's inputs copied from pinned host
memory (on a second stream, overlapping the previous step) and the loss / acceptance histogram
read back inside the timed region.  Under
torchrun every rank runs its own batch (weak scaling, no collective on the data path).
`--impl reference` times the CPU oracle on a bounded sample of the same workload.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ALR slot-loss fwd+bwd rows/s and % bf16 tensor peak (d=4096,V=151936,B=16)"
UNIT = "rows/s"
WORKLOAD = "text8b"


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gpu", "reference"], default="gpu")
    ap.add_argument("--sigma", type=float, default=0.5)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-anchors", type=int, default=1)
    ap.add_argument("--step", choices=["keep", "recompute"], default="keep",
                    help="the timed step: the forward keeps the logits for the backward (default), "
                         "or the backward recomputes them; the other one is timed beside it")
    ap.add_argument("--no-recompute", action="store_true",
                    help="skip the measurement of the other step variant")
    ap.add_argument("--no-erase", action="store_true",
                    help="skip the erase-mode steps and the accepted-length histograms at other "
                         "noise levels")
    ap.add_argument("--no-topk", action="store_true",
                    help="skip the compact-label (top-8 + tail) step measurement")
    ap.add_argument("--no-other-workloads", action="store_true",
                    help="skip the vl7b step and the small-workload forward measured beside the "
                         "headline workload")
    ap.add_argument("--gather-only", action="store_true",
                    help="profiling only: run just the IRA gather measurement and print its "
                         "result (no step, a little over 2 GB of device memory)")
    ap.add_argument("--anchors", type=int, default=0,
                    help="profiling only: fewer anchors than the workload (config says so)")
    ap.add_argument("--oracle-rates", action="store_true",
                    help="internal: print the CPU oracle's rows/s at each workload and exit")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return dict(bf16=j["bf16_tflops"], bf16_sustained=j["bf16_tflops_sustained"],
                    hbm=j["hbm_gbs"], source="measured")
    return dict(bf16=1900.0, bf16_sustained=1700.0, hbm=6800.0, source="fallback")


# ------------------------------------------------------------------ DRAM traffic ---
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "loss_gemm_traffic.json")
_CSRC = "paper_2609_38795_gb300/csrc/"
_LOSS_KERNEL = [_CSRC + "loss_gemm_kernel.cuh", _CSRC + "tc_common.cuh", _CSRC + "kernels.h"]
_GRAD_KERNELS = [_CSRC + "grad_kernels.cu", _CSRC + "tc_common.cuh", _CSRC + "kernels.h"]
# the sources each recorded kernel is built from: its counters stay valid while their code does
KERNEL_SOURCES = {"fwd": _LOSS_KERNEL, "fwd_recompute": _LOSS_KERNEL,
                  "logit_grad_recompute": _LOSS_KERNEL, "logit_grad": _GRAD_KERNELS}


def _code_only(text):
    """Source text without comments and blank space: a change to a comment is no change to the
    kernel the counters were taken from."""
    import re
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_sources_sha256(files, read=None):
    """Digest of the code of `files` (repository-relative).  `read(rel)` returns a file's text
    (default: the working tree)."""
    import hashlib
    if read is None:
        def read(rel):
            with open(os.path.join(ROOT, rel), encoding="utf-8") as f:
                return f.read()
    h = hashlib.sha256()
    for rel in files:
        h.update(_code_only(read(rel)).encode())
    return h.hexdigest()


def kernel_traffic(phase):
    """DRAM bytes per full-size launch of the kernel of a step phase ("fwd": the fused forward
    keeping the logits; "logit_grad": G from the kept logits; "*_recompute": the step that keeps
    nothing), from the committed ncu summary, or None when that summary is missing or the
    kernel's sources changed since its capture."""
    try:
        with open(TRAFFIC_FILE) as f:
            j = json.load(f)
    except (OSError, ValueError):
        return None
    k = j.get("kernels", {}).get(phase)
    if k is None or phase not in KERNEL_SOURCES:
        return None
    if k.get("sources_sha256") != kernel_sources_sha256(KERNEL_SOURCES[phase]):
        return None
    return k["bytes_per_full_launch"]


# ------------------------------------------------------------------ rank reductions ---
def max_over_ranks(values, device):
    """Element-wise maximum of per-rank timings over the process group (identity when the
    group is absent or has one rank)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(values, device=device, dtype=torch.float64)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_rows_per_s(world, rows_per_rank, steps, slowest_ms):
    """Whole-job throughput: every rank processes rows_per_rank rows per step (weak scaling),
    and the job takes as long as its slowest rank."""
    return world * rows_per_rank * steps / (slowest_ms / 1e3)


# ------------------------------------------------------------------ clocks sampler ---
class Clocks:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return parse_clocks(lines)


def parse_clocks(lines):
    """Summary of nvidia-smi samples in the Clocks.QUERY column order (csv, no header, no
    units): median SM clock over the loaded samples (above half the highest, so idle samples
    at the edges of the timed region do not pull it down), the maximum clock, and every
    throttle reason seen active.  None when no sample parses."""
    sm, smax, reasons = [], [], set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for line in lines:
        parts = [x.strip() for x in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            sm.append(float(parts[1]))
            smax.append(float(parts[2]))
        except ValueError:
            continue
        for n, v in zip(names, parts[5:9]):
            if v.lower() == "active":
                reasons.add(n)
    if not sm:
        return None
    loaded = [s for s in sm if s > 0.5 * max(sm)] or sm
    return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax),
            "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------- CPU oracle ---
def oracle_sample(wl, inputs, n_anchors):
    """Rows of the workload for the CPU oracle: the first n_anchors anchors' rows and W."""
    import numpy as np
    rows = n_anchors * wl.B
    Hd = inputs["Hd"][:rows].float().cpu().numpy()
    Ht = inputs["Ht"][:rows].float().cpu().numpy()
    W = inputs["W"].float().cpu().numpy()
    mask = inputs["row_valid"][:rows].float().cpu().numpy().astype(np.float64)
    return Hd, Ht, W, mask


def oracle_step(wl, Hd, Ht, W, mask):
    """The oracle's fwd + bwd over its sample (as it stands; its own fp64 conversions)."""
    from oracle import alr_oracle as orc
    out = orc.slot_loss_forward(Hd, Ht, W, wl.B, row_mask=mask)
    G = orc.logit_grad(out["z_d"], out["z_t"], out["weight"], 1.0)
    orc.slot_loss_backward(Hd, W, G)
    return out["loss_total"]


def cores_used():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def time_oracle(wl, inputs, n_anchors, reps, budget_s=30.0):
    Hd, Ht, W, mask = oracle_sample(wl, inputs, n_anchors)
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        oracle_step(wl, Hd, Ht, W, mask)
        times.append(time.perf_counter() - t0)
        if sum(times) > budget_s:
            break
    rows = n_anchors * wl.B
    return rows * len(times) / sum(times), times


def time_oracle_single_thread(sigma, n_anchors):
    """The oracle on one host core: this script's reference arm in a child process whose BLAS
    and OpenMP pools are limited to one thread (one step over the same bounded sample)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               RANK="0", WORLD_SIZE="1")
    cmd = [sys.executable, os.path.abspath(__file__), "--impl", "reference", "--steps", "1",
           "--warmup", "0", "--sigma", str(sigma), "--cpu-sample-anchors", str(n_anchors)]
    try:
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=300)
        line = [ln for ln in r.stdout.splitlines() if ln.startswith("{")][-1]
        j = json.loads(line)
        return {"value": j["value"], "unit": j["unit"], "cores": 1,
                "seconds": j["ms_per_step"] / 1e3}
    except (subprocess.SubprocessError, IndexError, ValueError, KeyError) as e:
        return {"unavailable": f"{type(e).__name__}"}


ORACLE_WORKLOADS = ("small", "vl7b", "text8b")


def oracle_rates(n_anchors, reps=2):
    """The oracle's forward-only and forward+backward rows/s at each workload's d and V, on
    n_anchors anchors of seeded CPU inputs (the workload's recipe without a feature buffer);
    the best of `reps` timings each.  Runs in whatever thread budget the process has."""
    import numpy as np
    import torch
    from oracle import alr_oracle as orc
    from paper_2609_38795_gb300 import synthetic
    out = {}
    for name in ORACLE_WORKLOADS:
        wl = synthetic.WORKLOADS[name]
        b = synthetic.slot_batch(wl.d, wl.V, n_anchors, wl.B, wl.sigma, dtype=torch.bfloat16, seed=0)
        Hd, Ht, W = (b[k].float().numpy() for k in ("Hd", "Ht", "W"))
        mask = np.ones(n_anchors * wl.B)
        rows = n_anchors * wl.B
        t_f, t_s = [], []
        for _ in range(reps):
            t0 = time.perf_counter()
            orc.slot_loss_forward(Hd, Ht, W, wl.B, row_mask=mask)
            t_f.append(time.perf_counter() - t0)
            t0 = time.perf_counter()
            oracle_step(wl, Hd, Ht, W, mask)
            t_s.append(time.perf_counter() - t0)
        out[name] = {"fwd": rows / min(t_f), "fwd_bwd": rows / min(t_s)}
    return out


def oracle_rates_child(n_anchors, threads=None):
    """oracle_rates in a fresh interpreter (never a fork of this CUDA process); threads=1 limits
    its BLAS and OpenMP pools to one thread.  Returns flat keys for the cpu_baseline record."""
    env = dict(os.environ, RANK="0", WORLD_SIZE="1")
    if threads is not None:
        env.update(OMP_NUM_THREADS=str(threads), OPENBLAS_NUM_THREADS=str(threads),
                   MKL_NUM_THREADS=str(threads))
    cmd = [sys.executable, os.path.abspath(__file__), "--oracle-rates",
           "--cpu-sample-anchors", str(n_anchors)]
    suffix = "" if threads is None else f"_{threads}core"
    try:
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=600)
        j = json.loads([ln for ln in r.stdout.splitlines() if ln.startswith("{")][-1])
    except (subprocess.SubprocessError, IndexError, ValueError) as e:
        return {f"oracle_rates{suffix}": f"unavailable: {type(e).__name__}"}
    return {f"{kind}_rows_per_s_{wl}{suffix}": v[kind] for wl, v in j.items() for kind in v}


# ------------------------------------------------------------- gather bandwidth ---
def gather_bandwidth(device, reps=24, warmup=4, n_sets=4):
    """IRA gather at the vl7b shape (512 anchors x 16 rows of d=3584 bf16 from a feature
    buffer [32, 2048, d]).  Inputs larger than L2: the launches cycle through n_sets feature
    buffers and output buffers (4 x 58.7 MB read + 4 x 58.7 MB written per cycle, > L2), so no
    launch finds its rows in L2.  The reps launches are captured once in a CUDA graph and the
    graph's replay is timed with CUDA events (mean time per launch); the same launches issued
    one by one from the host are timed beside it (`us_per_launch_stream`)."""
    import torch
    from paper_2609_38795_gb300 import alr, synthetic
    wl = synthetic.WORKLOADS["vl7b"]
    g = torch.Generator(device=device).manual_seed(5)
    sets = []
    for _ in range(n_sets):
        F = torch.randn(wl.S, wl.L, wl.d, generator=g, device=device).to(torch.bfloat16)
        seq, pos = synthetic.anchor_positions(wl.A, wl.S, wl.L, wl.B, device=device, g=g)
        out = torch.empty(wl.N, wl.d, dtype=torch.bfloat16, device=device)
        valid = torch.empty(wl.N, dtype=torch.float32, device=device)
        sets.append((F, seq, pos, out, valid))
    for i in range(warmup):
        F, seq, pos, out, valid = sets[i % n_sets]
        alr.alr_gather_ira_blocks(F, seq, pos, wl.B, out, valid)
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)

    def launches():
        for i in range(reps):
            F, seq, pos, out, valid = sets[i % n_sets]
            alr.alr_gather_ira_blocks(F, seq, pos, wl.B, out, valid)

    a.record()
    launches()
    b.record()
    torch.cuda.synchronize()
    ms_stream = a.elapsed_time(b) / reps
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        launches()
    graph.replay()
    torch.cuda.synchronize()
    a.record()
    graph.replay()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / reps
    check_device_status("gather")
    nbytes = 2 * wl.N * wl.d * 2 + wl.N * 4       # rows read + rows written + row_valid
    gbs = nbytes / (ms / 1e3) / 1e9
    return {"workload": f"vl7b: {wl.A} anchors x {wl.B} rows, d={wl.d}, feature buffer "
                        f"{wl.S}x{wl.L}", "bytes": nbytes, "us_per_launch": ms * 1e3,
            "GB/s": gbs, "us_per_launch_stream": ms_stream * 1e3,
            "GB/s_stream": nbytes / (ms_stream / 1e3) / 1e9,
            "l2": f"inputs larger than L2 ({n_sets} rotating input/output sets)",
            "reps": reps, "timing": "one CUDA graph of reps launches, replayed"}


def ira_context_bandwidth(device, reps=24, warmup=4, n_sets=3):
    """Context rows of the IRA secondary blocks at the paper's shape (App. A: 6 samples per
    GPU, 128 anchors per sample, K = 15, the five target layers' outputs stored for
    y*_1..y*_13, d = 4096 bf16): 64 secondaries per sample, each a [13, 5 d] context buffer
    filled from its primary's store (j - 1 rows copied, the rest zeroed).  The draws come from
    seeded random integers; the algorithmic bytes are the copied rows read and written plus the
    zero rows written, from the actual offsets.  Rotating input/output sets larger than L2; a
    CUDA graph of reps launches replayed, as for the gather."""
    import numpy as np
    import torch
    from paper_2609_38795_gb300 import alr
    S, L, K, max_b, C, F = 6, 4096, 15, 128, 13, 5 * 4096
    H, P = max_b // 2, max_b - max_b // 2
    g = torch.Generator(device=device).manual_seed(11)
    sets = []
    for _ in range(n_sets):
        ok = torch.ones(S, L, dtype=torch.uint8, device=device)
        keys = torch.randint(-(1 << 31), 1 << 31, (S, L), generator=g, device=device,
                             dtype=torch.int64).to(torch.int32)
        off_u = torch.randint(-(1 << 31), 1 << 31, (S, H), generator=g, device=device,
                              dtype=torch.int64).to(torch.int32)
        d = dict(n_valid=torch.empty(S, dtype=torch.int32, device=device),
                 anchor_pos=torch.empty(S, max_b, dtype=torch.int32, device=device),
                 offsets=torch.empty(S, H, dtype=torch.int32, device=device))
        alr.alr_ira_draw(K, max_b, ok, keys, off_u, d)
        store = torch.randn(S * P, C, F, generator=g, device=device).to(torch.bfloat16)
        rlen = torch.full((S * P,), K, dtype=torch.int32, device=device)
        ctx = torch.empty(S, H, C, F, dtype=torch.bfloat16, device=device)
        sets.append((store, d, rlen, ctx))

    def launch(i):
        store, d, rlen, ctx = sets[i % n_sets]
        alr.alr_ira_context(K, max_b, store, d["n_valid"], rlen, d["offsets"], d["anchor_pos"], ctx)

    for i in range(warmup):
        launch(i)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for i in range(reps):
        launch(i)
    b.record()
    torch.cuda.synchronize()
    ms_stream = a.elapsed_time(b) / reps
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for i in range(reps):
            launch(i)
    graph.replay()
    torch.cuda.synchronize()
    a.record()
    graph.replay()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / reps
    check_device_status("IRA context")
    row = F * 2
    nbytes = []
    for _, d, _, _ in sets:                         # mean over the rotating sets' offsets
        copied = int((d["offsets"].cpu().numpy().astype(np.int64) - 1).sum())
        nbytes.append(2 * copied * row + (S * H * C - copied) * row)
    nb = sum(nbytes) / len(nbytes)
    return {"workload": f"{S} samples x {H} secondary blocks, {C} stored rows of 5 x 4096 bf16 "
                        f"features (K={K}, 128 anchors, length {L})",
            "bytes": nb, "us_per_launch": ms * 1e3, "GB/s": nb / (ms / 1e3) / 1e9,
            "us_per_launch_stream": ms_stream * 1e3,
            "GB/s_stream": nb / (ms_stream / 1e3) / 1e9,
            "l2": f"inputs larger than L2 ({n_sets} rotating input/output sets)",
            "reps": reps, "timing": "one CUDA graph of reps launches, replayed"}


# ------------------------------------------------------------------------ GPU arm ---
def make_inputs(wl, sigma, device, seed):
    import torch
    from paper_2609_38795_gb300 import synthetic
    b = synthetic.rollout_batch(wl.d, wl.V, wl.A, wl.B, wl.S, wl.L, sigma, dtype=torch.bfloat16,
                                device=device, seed=seed)
    b["Ht"] = torch.empty(wl.N, wl.d, dtype=torch.bfloat16, device=device)
    b["row_valid"] = torch.empty(wl.N, dtype=torch.float32, device=device)
    return b


class Step:
    """Buffers and the sequence of C-ABI calls of one step.  keep: the forward keeps both
    logit matrices (fp16 relative to 16-column group references) and G is computed from them
    in place of z_d; otherwise G is computed by recomputing both head products."""
    N_PHASES = 6
    PHASES = ["gather", "fwd", "accept_len", "logit_grad", "dH_gemm", "dW_gemm"]
    KERNELS_PER_STEP = 8   # gather, fwd (loss, combine, finalize), accept, logit grad, dH, dW

    def __init__(self, wl, inputs, device, keep=True, mode=0, corpus_tok=None):
        import torch
        from paper_2609_38795_gb300 import alr
        self.alr, self.wl, self.x, self.keep = alr, wl, inputs, keep
        self.corpus_tok = corpus_tok
        self.sl = alr.SlotLoss(wl.N, wl.d, wl.V, wl.B, dtype=torch.bfloat16, device=device,
                               keep_logits=keep, mode=mode)
        self.G = (self.sl.G if keep else
                  torch.empty(wl.N, wl.V, dtype=torch.bfloat16, device=device))
        self.dH = torch.empty(wl.N, wl.d, dtype=torch.float32, device=device)
        self.dW = torch.zeros(wl.d, wl.V, dtype=torch.float32, device=device)

    def run(self, events=None):
        alr, x, sl, wl = self.alr, self.x, self.sl, self.wl
        rec = (lambda i: events[i].record()) if events is not None else (lambda i: None)
        rec(0)
        alr.alr_gather_ira_blocks(x["F"], x["seq"], x["pos"], wl.B, x["Ht"], x["row_valid"])
        rec(1)
        sl.forward(x["Hd"], x["Ht"], x["W"], row_mask=x["row_valid"], corpus_tok=self.corpus_tok)
        rec(2)
        sl.accept(active=x["row_valid"])
        rec(3)
        o = sl.out
        if self.keep:
            alr.alr_logit_grad_from_logits(sl.params, sl.Zd, sl.Zt, sl.Zd_ref, sl.Zt_ref,
                                           o["weight"], o["weight_sum"], o["lse_d"], o["lse_t"],
                                           self.G)
        else:
            alr.alr_logit_grad(sl.params, x["Hd"], x["Ht"], x["W"], o["weight"],
                               o["weight_sum"], o["lse_d"], o["lse_t"], self.G)
        rec(4)
        alr.alr_gemm(self.G, x["W"], self.dH, wl.N, wl.d, wl.V)                    # G W^T
        rec(5)
        alr.alr_gemm(x["Hd"], self.G, self.dW, wl.d, wl.V, wl.N, a_mn=True, b_mn=True,
                     accumulate=True)                                               # H_d^T G
        rec(6)


class TopkStep:
    """The compact-label step (the paper's own loss form): label readout of H_t (top-8 target
    probabilities, tail, greedy token) -> top-8 + tail soft CE forward on H_d keeping z_d ->
    accepted length -> logit gradient from the kept z_d (in place) -> dH = G W^T ->
    dW += H_d^T G.  It reuses the full-vocabulary step's z_d buffer."""
    PHASES = ["readout", "fwd", "accept_len", "logit_grad", "dH_gemm", "dW_gemm"]
    KERNELS_PER_STEP = 8   # readout (+ merge), fwd (+ merge, finalize), accept, grad, dH, dW

    def __init__(self, step):
        import torch
        from paper_2609_38795_gb300 import alr
        self.s, self.alr = step, alr
        wl, dev = step.wl, step.G.device
        N = wl.N
        self.params = alr.make_params(N, wl.d, wl.V, wl.B, torch.bfloat16)
        f = lambda *sh: torch.empty(*sh, dtype=torch.float32, device=dev)  # noqa: E731
        i = lambda *sh: torch.empty(*sh, dtype=torch.int32, device=dev)  # noqa: E731
        self.lab = dict(top_idx=i(N, alr.ALR_TOPK), top_prob=f(N, alr.ALR_TOPK), tail=f(N),
                        lse_t=f(N), argmax_t=i(N), gap_t=f(N))
        self.out = dict(loss_row=f(N), lse_d=f(N), tail_q=f(N), argmax_d=i(N), gap_d=f(N),
                        weight=f(N), loss_total=f(1), weight_sum=f(1))
        self.ws_r = torch.empty(alr.alr_readout_workspace_size(self.params), dtype=torch.uint8,
                                device=dev)
        self.ws_f = torch.empty(alr.alr_topk_fwd_workspace_size(self.params), dtype=torch.uint8,
                                device=dev)

    def run(self, events=None):
        alr, s, x, lab, o = self.alr, self.s, self.s.x, self.lab, self.out
        wl = s.wl
        rec = (lambda i: events[i].record()) if events is not None else (lambda i: None)
        rec(0)
        alr.alr_label_readout(self.params, x["Ht"], x["W"], lab, self.ws_r)
        rec(1)
        alr.alr_topk_loss_fwd_keep_logits(self.params, x["Hd"], x["W"], lab["top_idx"],
                                          lab["top_prob"], lab["tail"], s.sl.Zd, s.sl.Zd_ref, o,
                                          self.ws_f, row_mask=x["row_valid"])
        rec(2)
        alr.alr_accept_len(o["argmax_d"], lab["argmax_t"], wl.B, s.sl.acc_len, s.sl.hist,
                           active=x["row_valid"])
        rec(3)
        alr.alr_topk_logit_grad_from_logits(self.params, s.sl.Zd, s.sl.Zd_ref, lab["top_idx"],
                                            lab["top_prob"], lab["tail"], o["weight"],
                                            o["weight_sum"], o["lse_d"], o["tail_q"], s.G)
        rec(4)
        alr.alr_gemm(s.G, x["W"], s.dH, wl.N, wl.d, wl.V)
        rec(5)
        alr.alr_gemm(x["Hd"], s.G, s.dW, wl.d, wl.V, wl.N, a_mn=True, b_mn=True, accumulate=True)
        rec(6)


def check_device_status(what):
    """Raise if a bounded pipeline wait of the library timed out (its kernels then return
    early and their outputs and timings are void)."""
    from paper_2609_38795_gb300 import alr
    if alr.alr_device_status() != alr.ALR_OK:
        raise RuntimeError(f"{what}: device status: {alr.alr_last_error()}")


def time_variant(wl, x, device, K, warmup, keep):
    """The other step variant, timed beside the headline one: keep=False, the backward
    recomputes both head products (12 NdV tensor flops, no logit storage); keep=True, the
    forward keeps the logits (8 NdV)."""
    import torch
    st = Step(wl, x, device, keep=keep)
    for _ in range(warmup):
        st.run()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(7)] for _ in range(K)]
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for k in range(K):
        st.run(ev[k])
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / K
    check_device_status("recomputing step")
    NdV = wl.N * wl.d * wl.V
    phase = {p: sum(ev[k][i].elapsed_time(ev[k][i + 1]) for k in range(K)) / K
             for i, p in enumerate(Step.PHASES)}
    what = ("same step, logits kept by the forward for the backward" if keep else
            "same step, logits recomputed by the backward (nothing kept)")
    out = {"what": what, "ms_per_step": ms, "rows_per_s": wl.N / (ms / 1e3),
           ("executed_tflops_8NdV" if keep else "executed_tflops_12NdV"):
               (8 if keep else 12) * NdV / (ms / 1e3) / 1e12, "phase_ms": phase,
           "gpu_launches": Step.KERNELS_PER_STEP * K, "loss": st.sl.out["loss_total"].item()}
    del st
    torch.cuda.empty_cache()
    return out


def time_erase(wl, x, device, K, warmup, argmax_t):
    """The kept-logits step in the erase comparator's modes (Eq. 2): corpus tokens are the
    greedy target tokens, each replaced with probability 0.2 by a uniform token.  The label rows
    are the same as in ALR mode, so the difference is the cost of the weighting only."""
    import torch
    from paper_2609_38795_gb300 import alr, synthetic
    mask, rnd = synthetic.corpus_replacement(wl.N, wl.V, 0.2, device=device, seed=3)
    tok = synthetic.corpus_tokens(argmax_t, mask, rnd)
    out = {"workload": "erase: as text8b, sigma 0.5, corpus = greedy target token replaced "
                       "w.p. 0.2"}
    for name, mode in (("soft", alr.ALR_MODE_ERASE_SOFT), ("hard", alr.ALR_MODE_ERASE_HARD)):
        st = Step(wl, x, device, keep=True, mode=mode, corpus_tok=tok)
        for _ in range(warmup):
            st.run()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(K):
            st.run()
        b.record()
        torch.cuda.synchronize()
        check_device_status(f"erase ({name}) steps")
        ms = a.elapsed_time(b) / K
        out[name] = {"ms_per_step": ms, "rows_per_s": wl.N / (ms / 1e3),
                     "loss": st.sl.out["loss_total"].item(),
                     "weight_sum": st.sl.out["weight_sum"].item()}
        del st
        torch.cuda.empty_cache()
    return out


def time_other_workloads(device, K, warmup):
    """Beside the headline workload, two configurations timed for reference (not bench
    lines): the vl7b step (gather from its 32 x 2048 feature buffer, forward keeping the
    logits, accepted length, gradient, dH, dW) and the small workload's forward alone.  The
    small forward's head (131 MB) is about the size of L2, so L2 is flushed (a 256 MB write)
    before every timed repetition; the vl7b inputs are larger than L2."""
    import torch
    from paper_2609_38795_gb300 import alr, synthetic
    out = {}
    wl = synthetic.WORKLOADS["vl7b"]
    x = make_inputs(wl, 0.5, device, seed=7)
    st = Step(wl, x, device, keep=True)
    for _ in range(warmup):
        st.run()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(7)] for _ in range(K)]
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for k in range(K):
        st.run(ev[k])
    b.record()
    torch.cuda.synchronize()
    check_device_status("vl7b step")
    ms = a.elapsed_time(b) / K
    phase = {p: sum(ev[k][i].elapsed_time(ev[k][i + 1]) for k in range(K)) / K
             for i, p in enumerate(Step.PHASES)}
    NdV = wl.N * wl.d * wl.V
    out["vl7b_step"] = {
        "workload": f"vl7b: d={wl.d} V={wl.V} B={wl.B} A={wl.A} rows={wl.N}, feature buffer "
                    f"{wl.S}x{wl.L}", "ms_per_step": ms, "rows_per_s": wl.N / (ms / 1e3),
        "executed_tflops_8NdV": 8 * NdV / (ms / 1e3) / 1e12, "phase_ms": phase,
        "fwd_rows_per_s": wl.N / (phase["fwd"] / 1e3),
        "loss": st.sl.out["loss_total"].item()}
    del st, x
    torch.cuda.empty_cache()

    wl = synthetic.WORKLOADS["small"]
    bt = synthetic.slot_batch(wl.d, wl.V, wl.A, wl.B, wl.sigma, dtype=torch.bfloat16,
                              device=device, seed=8)
    sl = alr.SlotLoss(wl.N, wl.d, wl.V, wl.B)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    for _ in range(warmup):
        sl.forward(bt["Hd"], bt["Ht"], bt["W"])
    times = []
    for _ in range(K):
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        sl.forward(bt["Hd"], bt["Ht"], bt["W"])
        e1.record()
        times.append((e0, e1))
    torch.cuda.synchronize()
    check_device_status("small forward")
    ms = sum(e0.elapsed_time(e1) for e0, e1 in times) / K
    out["small_forward"] = {
        "workload": f"small: d={wl.d} V={wl.V} B={wl.B} A={wl.A} rows={wl.N}",
        "ms": ms, "rows_per_s": wl.N / (ms / 1e3),
        "tflops_4NdV": 4 * wl.N * wl.d * wl.V / (ms / 1e3) / 1e12,
        "l2": "flushed (256 MB write) before every repetition", "gpu_launches": 3 * K}
    del sl, bt, flush
    torch.cuda.empty_cache()
    return out


def mean_accepted_tokens(hist):
    """MAT of Sec. 4: the mean over anchors of (accepted slots + 1), from a histogram whose
    entry n counts the anchors with n accepted slots."""
    total = sum(hist)
    return None if total == 0 else 1.0 + sum(n * c for n, c in enumerate(hist)) / total


def acc_hist_by_sigma(wl, step, device, sigmas):
    """Accepted-length histogram of one step at other drafter noise levels (the same seeded
    target features and head; only the drafter's noise scale changes)."""
    import torch
    hist = {}
    x0 = step.x
    for sg in sigmas:
        step.x = make_inputs(wl, sg, device, seed=0)
        step.run()
        torch.cuda.synchronize()
        hist[str(sg)] = step.sl.hist.cpu().tolist()
    step.x = x0
    torch.cuda.empty_cache()
    return hist


def time_topk(step, K, warmup):
    import torch
    ts = TopkStep(step)
    for _ in range(warmup):
        ts.run()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(7)] for _ in range(K)]
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for k in range(K):
        ts.run(ev[k])
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / K
    check_device_status("compact-label step")
    wl = step.wl
    NdV = wl.N * wl.d * wl.V
    phase = {p: sum(ev[k][i].elapsed_time(ev[k][i + 1]) for k in range(K)) / K
             for i, p in enumerate(TopkStep.PHASES)}
    loss_ms = ms - phase["readout"]
    return {"what": "compact labels (top-8 + tail bin): readout of H_t, then the loss fwd+bwd "
                    "with z_d kept by the forward",
            "ms_per_step": ms, "rows_per_s": wl.N / (ms / 1e3),
            "loss_fwd_bwd_rows_per_s": wl.N / (loss_ms / 1e3),
            "loss_tflops_6NdV": 6 * NdV / (loss_ms / 1e3) / 1e12,
            "readout_tflops_2NdV": 2 * NdV / (phase["readout"] / 1e3) / 1e12,
            "phase_ms": phase, "gpu_launches": TopkStep.KERNELS_PER_STEP * K,
            "loss": ts.out["loss_total"].item()}


def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist
    from paper_2609_38795_gb300 import alr, build_lib, synthetic

    torch.cuda.set_device(local_rank)
    device = f"cuda:{local_rank}"
    build_lib.build()
    alr.lib()
    if alr.alr_device_supported() != alr.ALR_OK:
        raise RuntimeError(alr.alr_last_error())
    wl = synthetic.WORKLOADS[WORKLOAD]
    if args.anchors:
        import dataclasses
        wl = dataclasses.replace(wl, A=args.anchors, S=max(1, args.anchors // 128))
    x = make_inputs(wl, args.sigma, device, seed=rank)
    keep = args.step == "keep"
    step = Step(wl, x, device, keep=keep)
    for _ in range(args.warmup):
        step.run()
    torch.cuda.synchronize()
    check_device_status("warm-up")

    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(7)] for _ in range(K)]
    clocks = Clocks(local_rank)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_stop = torch.cuda.Event(enable_timing=True)
    t_start.record()
    for k in range(K):
        step.run(ev[k])
    t_stop.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_stop)
    phase_ms = {p: sum(ev[k][i].elapsed_time(ev[k][i + 1]) for k in range(K)) / K
                for i, p in enumerate(Step.PHASES)}
    check_device_status("timed steps")
    acc_hist = step.sl.hist.cpu().tolist()
    loss = step.sl.out["loss_total"].item()

    # ---- end to end through host buffers (pinned), copies inside the timed region ----
    # Every step copies its inputs (H_d, the feature buffer, anchor positions) from pinned host
    # memory and reads its loss, sum omega and acceptance histogram back.  The copies run on a
    # second stream into two alternating device buffers, so step k + 1's inputs travel while
    # step k computes; the first copy starts after the timed region opens and the last step's
    # read-back ends before it closes.
    e2e = None
    if not args.no_e2e:
        keys = ("Hd", "F", "seq", "pos")
        host = {k: x[k].cpu().pin_memory() for k in keys}
        sets = [x, dict(x, **{k: torch.empty_like(x[k]) for k in keys})]
        res = {"loss": torch.empty(2, dtype=torch.float32).pin_memory(),
               "hist": torch.empty(wl.B + 1, dtype=torch.int64).pin_memory()}
        h2d = sum(t.numel() * t.element_size() for t in host.values())
        d2h = 2 * 4 + (wl.B + 1) * 8
        comp = torch.cuda.current_stream()
        copy_stream = torch.cuda.Stream()
        ready = [torch.cuda.Event(), torch.cuda.Event()]
        free = [torch.cuda.Event(), torch.cuda.Event()]

        def issue_copy(k, after=None):
            b = k % 2
            with torch.cuda.stream(copy_stream):
                if after is not None:
                    copy_stream.wait_event(after)
                copy_stream.wait_event(free[b])      # the step that last read buffer b is done
                for key in keys:
                    sets[b][key].copy_(host[key], non_blocking=True)
                ready[b].record(copy_stream)

        def e2e_run(n, start_event=None):
            issue_copy(0, start_event)
            for k in range(n):
                if k + 1 < n:
                    issue_copy(k + 1)
                b = k % 2
                comp.wait_event(ready[b])
                step.x = sets[b]
                step.run()
                free[b].record(comp)
                res["loss"][0:1].copy_(step.sl.out["loss_total"], non_blocking=True)
                res["loss"][1:2].copy_(step.sl.out["weight_sum"], non_blocking=True)
                res["hist"].copy_(step.sl.hist, non_blocking=True)

        for e in free:
            e.record(comp)
        e2e_run(max(1, args.warmup))
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(comp)
        e2e_run(K, start_event=a)
        b.record(comp)
        torch.cuda.synchronize()
        step.x = x
        e2e_ms = a.elapsed_time(b)
        check_device_status("end-to-end steps")
        if world > 1:
            dist.barrier()
        e2e = {"ms": e2e_ms, "h2d": h2d, "d2h": d2h}

    # ---- max over ranks ----
    total_ms, e2e_ms = max_over_ranks([total_ms, e2e["ms"] if e2e else 0.0], device)

    gather = gather_bandwidth(device) if rank == 0 else None
    ira_ctx = ira_context_bandwidth(device) if rank == 0 else None
    topk = time_topk(step, K, args.warmup) if (rank == 0 and not args.no_topk) else None
    other = (time_variant(wl, x, device, K, args.warmup, keep=not keep)
             if (rank == 0 and not args.no_recompute) else None)
    erase = (time_erase(wl, x, device, K, args.warmup, step.sl.out["argmax_t"].clone())
             if (rank == 0 and not args.no_erase) else None)
    others = (time_other_workloads(device, K, args.warmup)
              if (rank == 0 and not args.no_other_workloads and not args.anchors) else None)
    hist_sigma = None
    if rank == 0 and not args.no_erase:
        hist_sigma = acc_hist_by_sigma(wl, step, device, [0.25, 1.0])
        hist_sigma[str(args.sigma)] = acc_hist

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rps, ts = time_oracle(wl, x, args.cpu_sample_anchors, reps=10)
        cpu = {"value": rps, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
               "sample": f"{args.cpu_sample_anchors} anchor(s) x {wl.B} rows of the {WORKLOAD} "
                         f"workload, full d={wl.d} and V={wl.V}, fwd+bwd in fp64, "
                         f"{len(ts)} repetition(s), {sum(ts):.1f} s",
               "single_thread": time_oracle_single_thread(args.sigma, args.cpu_sample_anchors)}
        # flat keys: forward-only and forward+backward oracle rates at every workload's d and V,
        # on all host cores and on one
        cpu["rates_sample"] = (f"{args.cpu_sample_anchors} anchor(s) x B rows of seeded CPU "
                               f"inputs per workload, best of 2")
        cpu.update(oracle_rates_child(args.cpu_sample_anchors))
        cpu.update(oracle_rates_child(args.cpu_sample_anchors, threads=1))
        cpu["single_thread_rows_per_s"] = cpu["single_thread"].get("value")
    if rank != 0:
        return None

    pk = peaks()
    NdV = wl.N * wl.d * wl.V
    ms_step = total_ms / K
    rows_per_s = job_rows_per_s(world, wl.N, K, total_ms)
    algo_tf = 8 * NdV / (ms_step / 1e3) / 1e12
    exec_tf = (8 if keep else 12) * NdV / (ms_step / 1e3) / 1e12
    # dominant kernel by measured time (the tensor-core phases); its flops per launch
    flops = {"fwd": 4 * NdV, "dH_gemm": 2 * NdV, "dW_gemm": 2 * NdV}
    if not keep:
        flops["logit_grad"] = 4 * NdV
    # the logit gradient from kept logits streams z_d, z_t (fp16) and their 16-column group
    # references (fp16) in and G (bf16) out
    g_bytes = 6 * wl.N * wl.V + 4 * wl.N * ((wl.V + 15) // 16)
    dom = max(flops, key=lambda p: phase_ms[p])
    achieved = flops[dom] / (phase_ms[dom] / 1e3) / 1e12
    out = {
        "metric": METRIC, "value": rows_per_s, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{WORKLOAD}{' PROFILING SUBSET' if args.anchors else ''}: d={wl.d} V={wl.V} B={wl.B} A={wl.A} rows={wl.N} "
                               f"sigma={args.sigma} feature buffer {wl.S}x{wl.L}",
                   "kernel_forms": dict(zip(("gemm", "loss"), alr.alr_kernel_forms())),
                   "global_batch_rows": world * wl.N, "l2": "inputs larger than L2 "
                   "(W 1.24 GB, H 268 MB each, kept logits 2 x 10 GB)", "parallelism": f"replicas{world}"},
        "tensor_tflops": {"executed": exec_tf, "algorithmic_8NdV": algo_tf,
                          "pct_peak_executed": exec_tf / pk["bf16"],
                          "pct_peak_algorithmic": algo_tf / pk["bf16"],
                          "peak_tflops": pk["bf16"], "peak_source": pk["source"]},
        "phase_ms": phase_ms,
        "fwd": {"rows_per_s": world * wl.N / (phase_ms["fwd"] / 1e3),
                "tflops_4NdV": 4 * NdV / (phase_ms["fwd"] / 1e3) / 1e12},
        # each tensor phase against the sustained peak (the phases run inside a long step)
        "phase_tflops": {ph: {"tflops": fl / (phase_ms[ph] / 1e3) / 1e12,
                              "frac_of_sustained": fl / (phase_ms[ph] / 1e3) / 1e12
                              / pk["bf16_sustained"]}
                         for ph, fl in (("fwd", 4 * NdV), ("dH_gemm", 2 * NdV),
                                        ("dW_gemm", 2 * NdV))},
        "roofline": {"bound": "tensor", "kernel": dom, "achieved": achieved,
                     "peak": pk["bf16_sustained"], "unit": "TFLOP/s",
                     "frac": achieved / pk["bf16_sustained"],
                     "frac_of_burst_peak": achieved / pk["bf16"], "traffic": kernel_traffic(dom if keep else dom + "_recompute"),
                     "peak_note": f"{pk['source']} sustained bf16 (kernel timed inside a long step)",
                     "flops_per_launch": flops[dom]},
        "logit_grad_hbm": ({"bytes": g_bytes, "GB/s": g_bytes / (phase_ms["logit_grad"] / 1e3) / 1e9,
                            "frac_of_hbm": g_bytes / (phase_ms["logit_grad"] / 1e3) / 1e9 / pk["hbm"],
                            "traffic": kernel_traffic("logit_grad")} if keep else None),
        "step": ("forward keeps the logits (fp16 with group references), the backward reads "
                 "them" if keep else "backward recomputes the logits"),
        ("recompute" if keep else "keep"): other,
        "gpu_launches": Step.KERNELS_PER_STEP * K,
        "ira_gather": dict(gather, frac_of_hbm=gather["GB/s"] / pk["hbm"], hbm_peak_gbs=pk["hbm"]),
        "ira_context": dict(ira_ctx, frac_of_hbm=ira_ctx["GB/s"] / pk["hbm"]),
        "compact_labels": topk,
        "loss": loss, "acc_hist": acc_hist, "acc_hist_by_sigma": hist_sigma,
        # mean accepted length per anchor + 1: the tokens a verification round yields (MAT)
        "mat": mean_accepted_tokens(acc_hist),
        "mat_by_sigma": (None if hist_sigma is None else
                         {sg: mean_accepted_tokens(h) for sg, h in hist_sigma.items()}),
        "erase": erase,
        "other_workloads": others,
        "clocks": clk,
        "cpu_baseline": cpu,
    }
    # The step that never stores the logits (the backward recomputes its logit tiles), with
    # its own roofline record: timed as `recompute` beside the default kept-logits step, or as
    # the main step under --step recompute.
    rc = other if keep else {"ms_per_step": ms_step, "rows_per_s": rows_per_s,
                             "phase_ms": phase_ms}
    if rc is not None:
        rc_flops = {"fwd": 4 * NdV, "logit_grad": 4 * NdV, "dH_gemm": 2 * NdV, "dW_gemm": 2 * NdV}
        rc_dom = max(rc_flops, key=lambda ph: rc["phase_ms"][ph])
        rc_ach = rc_flops[rc_dom] / (rc["phase_ms"][rc_dom] / 1e3) / 1e12
        out["recompute_rows_per_s"] = rc["rows_per_s"]
        rec = out.setdefault("recompute", {}) if not keep else out["recompute"]
        rec.update({
            "what": "logits never stored: the forward reduces both logit tiles on chip, the "
                    "backward recomputes them (12 NdV tensor flops per step)",
            "rows_per_s": rc["rows_per_s"], "ms_per_step": rc["ms_per_step"],
            "executed_tflops_12NdV": 12 * NdV / (rc["ms_per_step"] / 1e3) / 1e12,
            "algorithmic_tflops_8NdV": 8 * NdV / (rc["ms_per_step"] / 1e3) / 1e12,
            "roofline": {"bound": "tensor", "kernel": rc_dom, "achieved": rc_ach,
                         "peak": pk["bf16_sustained"], "unit": "TFLOP/s",
                         "frac": rc_ach / pk["bf16_sustained"],
                         "frac_of_burst_peak": rc_ach / pk["bf16"],
                         "traffic": kernel_traffic(rc_dom + "_recompute"),
                         "flops_per_launch": rc_flops[rc_dom],
                         "peak_note": f"{pk['source']} sustained bf16"}})
    if e2e is not None:
        out["e2e"] = {"value": job_rows_per_s(world, wl.N, K, e2e_ms), "unit": UNIT,
                      "h2d_bytes_per_step": e2e["h2d"], "d2h_bytes_per_step": e2e["d2h"],
                      "ms_per_step": e2e_ms / K}
    return out


# ---------------------------------------------------------------- reference arm ---
def run_reference(args):
    import torch
    from paper_2609_38795_gb300 import synthetic
    wl = synthetic.WORKLOADS[WORKLOAD]
    n_a = args.cpu_sample_anchors
    rows = n_a * wl.B
    # the sample's inputs, drawn on the CPU with the same recipe (first n_a anchors)
    g = torch.Generator().manual_seed(0)
    W = (torch.randn(wl.d, wl.V, generator=g) * synthetic.HEAD_STD).to(torch.bfloat16)
    Ht = torch.randn(rows, wl.d, generator=g).to(torch.bfloat16)
    Hd = (Ht.float() + args.sigma * torch.randn(rows, wl.d, generator=g)).to(torch.bfloat16)
    x = {"Hd": Hd, "Ht": Ht, "W": W, "row_valid": torch.ones(rows)}
    Hd_n, Ht_n, W_n, mask = oracle_sample(wl, x, n_a)
    for _ in range(args.warmup):
        oracle_step(wl, Hd_n, Ht_n, W_n, mask)
    ts = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_step(wl, Hd_n, Ht_n, W_n, mask)
        ts.append(time.perf_counter() - t0)
    total = sum(ts)
    v = rows * len(ts) / total
    sample = (f"{n_a} anchor(s) x {wl.B} rows of the {WORKLOAD} workload per step, full d={wl.d} "
              f"and V={wl.V}, fwd+bwd in fp64")
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(ts),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": f"{WORKLOAD}{' PROFILING SUBSET' if args.anchors else ''}: d={wl.d} V={wl.V} B={wl.B} (CPU oracle sample)"},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.oracle_rates:
        print(json.dumps(oracle_rates(args.cpu_sample_anchors)), flush=True)
        return
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return
    if args.gather_only:
        import torch
        from paper_2609_38795_gb300 import alr, build_lib
        torch.cuda.set_device(local_rank)
        build_lib.build()
        alr.lib()
        if rank == 0:
            g = gather_bandwidth(f"cuda:{local_rank}")
            c = ira_context_bandwidth(f"cuda:{local_rank}")
            pk = peaks()
            print(json.dumps({"ira_gather": dict(g, frac_of_hbm=g["GB/s"] / pk["hbm"],
                                                  hbm_peak_gbs=pk["hbm"]),
                              "ira_context": dict(c, frac_of_hbm=c["GB/s"] / pk["hbm"])}),
                  flush=True)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    out = run_gpu(args, rank, world, local_rank)
    if out is not None:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
