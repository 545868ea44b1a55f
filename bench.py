#!/usr/bin/env python3
"""Benchmark of the LAMB optimizer step on the BERT-large parameter layout.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Workload: BERT-large (24 layers, hidden 1024, FFN 4096, vocab 30522): 391
tensors, 335,141,888 parameters; bf16 gradients, fp32 master weights and Adam
moments, a bf16 weight copy written every step; beta1 0.9, beta2 0.999,
eps 1e-6, lambda 0.01 (biases / LayerNorm masked), phi = clip[0, 10],
eta = 2e-3, measured from step t = 1000 on (the step counter lives on the
device and is advanced by the kernels).  Inputs are seeded synthetic arrays
(workloads.bert_large_layout); the W warm-up steps run t = 1..W from m = v = 0
(W >= 3 gives the configured three warm-up steps).  All state (5.4 GB) is far
larger than L2, so no explicit L2 flush is needed between steps.

One JSON line is printed by rank 0:
  value     parameters/s of the whole job, state resident in HBM, timed with
            CUDA events on the launching stream over K steps
  e2e       the same metric through the same C-ABI call, but every step also
            copies that step's bf16 gradients host->device from pinned memory
            and reads the step's result (the per-tensor trust ratios) back;
            upload_gbs is the rate the loop moved gradients at, h2d_copy_gbs
            that of a plain pinned copy of the same bytes, timed alone
  roofline  the dominant kernel's algorithmic bytes / its event-timed
            duration, against the measured HBM copy bandwidth
  cpu_baseline  the fp64 oracle on a bounded sample, on this host's cores
Multi-GPU (torchrun): every rank runs an independent replica (the step has no
data-path exchange on one node here); value = all ranks' parameters / the
slowest rank's time.
"""
from __future__ import annotations

import argparse
import datetime as _dt
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("LAMB step params/sec and achieved HBM GB/s vs GB300 peak "
          "(BERT-large layout)")
UNIT = "params/s"
FALLBACK_HBM_GBS = 6800.0
# nominal HBM3e bandwidth of one GB300 GPU from NVIDIA's GB300 NVL72
# specification (576 TB/s over 72 GPUs); context for the measured peak
NOMINAL_HBM_GBS = 8000.0
CLOCK_WINDOW_S = 0.25     # the clock record spans at least this long
# algorithmic bytes per parameter of each kernel (bf16 g, bf16 copy)
BYTES_PASS1 = 2 + 4 + 4 + 4 + 4 + 4      # read g,m,v,w ; write m,v = 22
BYTES_PASS2 = 4 + 4 + 4 + 4 + 2          # read m,v,w ; write w, copy = 18
BYTES_STEP = BYTES_PASS1 + BYTES_PASS2   # 40
BYTES_SINGLE_TOUCH = 2 + 12 + 12 + 2     # 28
ALGO_CODES = {"auto": 0, "two_pass": 1, "on_chip": 3}
# the committed ncu summaries holding measured DRAM traffic per launch, per
# (algorithm, layout, optimizer), and the kernel sources they were taken on
TWO_PASS_SOURCES = ("lamb_kernels.cu", "lamb_device.cuh", "lamb_internal.h")
ONCHIP_SOURCES = ("lamb_onchip.cu", "lamb_onchip.h", "lamb_device.cuh",
                  "lamb_internal.h")
PROFILES = {
    (1, "bert_large", "lamb"): (
        os.path.join(ROOT, "profiles", "lamb_kernels_bert_large.md"),
        None, TWO_PASS_SOURCES),
    (3, "resnet50", "lamb"): (
        os.path.join(ROOT, "profiles", "onchip_step_kernel.md"),
        "resnet50/lamb", ONCHIP_SOURCES),
    (3, "resnet50", "lars"): (
        os.path.join(ROOT, "profiles", "onchip_step_kernel.md"),
        "resnet50/lars", ONCHIP_SOURCES),
}
# kept for the tests of the committed two-pass summary
KERNELS = {1: (["lamb_pass1_kernel<bf16>", "lamb_pass2_kernel<copy>"],
               [BYTES_PASS1, BYTES_PASS2], PROFILES[(1, "bert_large",
                                                     "lamb")][0])}


def two_pass_bytes(opt, gb, cb):
    """Algorithmic bytes per parameter of a two-pass step (g gb bytes,
    bf16 copy cb bytes)."""
    if opt == "lars":
        return (gb + 8 + 4) + (8 + 4 + cb)
    if opt in ("nlamb", "nnlamb"):
        return (gb + 12 + 8) + (12 + gb + 4 + cb)
    return (gb + 12 + 8) + (12 + 4 + cb)


def single_touch_bytes(opt, gb, cb):
    """Bytes per parameter when every operand is read and written once."""
    if opt == "lars":
        return gb + 8 + 4 + 4 + cb
    return gb + 12 + 8 + 4 + cb


def kernel_model(opt, algo, gb, cb, variant="plain", streamed_frac=0.0):
    """(kernel names, algorithmic bytes per parameter of each kernel).
    The skip-on-non-finite variant moves the m, v (LARS: m) writes from
    pass 1 to pass 2, which then reads g as well."""
    if algo == 3 and variant in ("plain", "decoupled"):
        # tensors too large for a round go through the two-pass kernels
        # first; bytes are per parameter of the whole layout
        f = streamed_frac
        on = ([f"onchip_step_kernel<{opt},g{8 * gb},copy{8 * cb}>"],
              [(1 - f) * single_touch_bytes(opt, gb, cb)])
        if f == 0:
            return on
        names, per = kernel_model(opt, 1, gb, cb, variant)
        return ([n + "(streamed)" for n in names] + on[0],
                [b * f for b in per] + on[1])
    defer = variant == "skip_nonfinite"
    if opt == "lars":
        if defer:
            return (["lars_pass1_kernel", "lars_pass2_kernel"],
                    [gb + 8, gb + 8 + 4 + 4 + cb])
        return (["lars_pass1_kernel", "lars_pass2_kernel"],
                [gb + 8 + 4, 8 + 4 + cb])
    nest = opt in ("nlamb", "nnlamb")
    names = [f"{'n' if nest else ''}lamb_pass1_kernel",
             f"{'n' if nest else ''}lamb_pass2_kernel"]
    if defer:
        return names, [gb + 12, gb + 12 + 8 + 4 + cb]
    return names, [gb + 12 + 8, 12 + (gb if nest else 0) + 4 + cb]


def noalloc_overhead(st, L, hyper, d_step, d_lr, stream, one_step, n=20):
    """Device time and host enqueue time per call of lamb_step_noalloc
    against the plan's lamb_step, on the same state, n calls each after
    three of each untimed.  The no-alloc call rebuilds its tables on the
    device every call; the difference is its per-call overhead."""
    from ctypes import byref, c_int64, c_uint8, c_void_p

    import torch
    from paper_1904_00962_gb300 import binding as B
    from paper_1904_00962_gb300.state import _dtype_code
    lib = B.load()
    k = L.n_tensors
    sizes = (c_int64 * k)(*[int(x) for x in L.sizes])
    mask = (c_uint8 * k)(*[1 if d else 0 for d in L.decay])
    arrs = [B._ptr_array(st.ptrs(x)) for x in ("w", "g", "m", "v", "copy")]
    gcode, ccode = _dtype_code(st.grad_dtype), _dtype_code(st.copy_dtype)
    hp = byref(hyper)
    ds, dl = c_void_p(d_step.data_ptr()), c_void_p(d_lr.data_ptr())
    sp = c_void_p(stream.cuda_stream)

    def na():
        rc = lib.lamb_step_noalloc(sizes, k, mask, gcode, ccode, *arrs, hp,
                                   ds, dl, None, sp)
        if rc:
            raise B.LambError(rc, B.lamb_last_error())

    for _ in range(3):
        na()
        one_step()
    res = {}
    for name, fn in (("plan", one_step), ("noalloc", na)):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        t0 = time.perf_counter()
        for _ in range(n):
            fn()
        t1 = time.perf_counter()
        e1.record(stream)
        e1.synchronize()
        res[name] = (e0.elapsed_time(e1) / n, (t1 - t0) / n * 1e6)
    return {"calls": n, "ms_per_call": res["noalloc"][0],
            "plan_ms_per_call": res["plan"][0],
            "overhead_ms": res["noalloc"][0] - res["plan"][0],
            "host_us_per_call": res["noalloc"][1],
            "plan_host_us_per_call": res["plan"][1]}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-streams", type=int, default=1,
                    help="copy streams the e2e gradient upload is split over")
    ap.add_argument("--e2e-steps", type=int, default=None,
                    help="steps of the end-to-end loop (default: min(K, 50))")
    ap.add_argument("--cpu-seconds", type=float, default=10.0,
                    help="wall time of the bounded oracle sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--algo", choices=list(ALGO_CODES), default="auto",
                    help="step algorithm of the plan (auto = library default)")
    ap.add_argument("--chunk-elems", type=int, default=0,
                    help="two-pass chunk size (0 = library default)")
    ap.add_argument("--layout", default="bert_large",
                    choices=["bert_large", "bert_base", "resnet50", "ragged",
                             "mlp"],
                    help="parameter layout (default: the BERT-large headline)")
    ap.add_argument("--optimizer", default="lamb",
                    choices=["lamb", "lars", "nlamb", "nnlamb"])
    ap.add_argument("--variant", default="plain",
                    choices=["plain", "grad_norm", "skip_nonfinite",
                             "decoupled"],
                    help="optional step flags: the fused gradient check, "
                         "skip-on-non-finite, or decoupled weight decay")
    ap.add_argument("--shard-world", type=int, default=0,
                    help="time the sharded step of this many ranks, run in "
                         "turn on one GPU, instead of the plain step")
    ap.add_argument("--layers", type=int, default=24,
                    help="encoder layers of the layout (24 = BERT-large; "
                         "fewer only for small profiling captures)")
    return ap.parse_args()


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------

def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash(sources=TWO_PASS_SOURCES):
    """sha256 (16 hex digits) of the kernels' code with comments and
    whitespace removed, so that editing a comment does not invalidate the
    committed ncu traffic figures while any change of code does."""
    h = hashlib.sha256()
    for name in sources:
        with open(os.path.join(ROOT, "paper_1904_00962_gb300", "csrc",
                               name)) as f:
            src = f.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(profile_file, kernel_idx, key=None,
                     sources=TWO_PASS_SOURCES):
    """Per-launch DRAM bytes from the committed ncu summary, if it was taken
    on the current kernel source; else None.  A summary covering several
    workloads labels its lines traffic_bytes_per_launch[<key>][<i>]."""
    try:
        text = open(profile_file).read()
    except OSError:
        return None
    m = re.search(r"kernel_source_sha256:\s*([0-9a-f]+)", text)
    if not m or m.group(1) != kernel_source_hash(sources):
        return None
    label = "" if key is None else rf"\[{re.escape(key)}\]"
    m = re.search(rf"traffic_bytes_per_launch{label}\[{kernel_idx}\]:\s*"
                  r"([0-9.e+]+)", text)
    return float(m.group(1)) if m else None


class ClockSampler:
    """nvidia-smi sampled every 100 ms into a temp file; samples whose
    timestamps fall inside [start, end] are summarised."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,"
              "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id=None):
        self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv",
                                               delete=False)
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}",
               "--format=csv,noheader,nounits", "-lms", "100"]
        if gpu_id:
            cmd.insert(1, f"--id={gpu_id}")
        try:
            self.proc = subprocess.Popen(cmd, stdout=self.tmp,
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        self.window = None

    def mark(self, start, end):
        self.window = (start, end)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.tmp.flush()
        rows = []
        with open(self.tmp.name) as f:
            for line in f:
                p = [x.strip() for x in line.split(",")]
                if len(p) < 9:
                    continue
                try:
                    ts = _dt.datetime.strptime(p[0], "%Y/%m/%d %H:%M:%S.%f")
                    rows.append((ts, float(p[1]), float(p[2]), p[3], p[4:]))
                except ValueError:
                    continue
        os.unlink(self.tmp.name)
        if not rows:
            return None
        sel = rows
        if self.window:
            a, b = self.window
            inside = [r for r in rows if a <= r[0] <= b]
            sel = inside if inside else rows
        names = ["active", "hw_slowdown", "hw_thermal_slowdown",
                 "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in sel:
            for name, val in zip(names[1:], r[4][1:]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r[1] for r in sel),
                "sm_max_mhz": max(r[2] for r in sel),
                "samples": len(sel),
                "reasons": sorted(reasons)}


def max_over_ranks(value: float, device=None) -> float:
    """Largest `value` over all ranks (the slowest rank's time); identity
    without an initialised process group."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def select_params(L, target, pool):
    """Whole tensors from `pool` (cycled) until `target` parameters."""
    out, n, i = [], 0, 0
    while n < target:
        k = pool[i % len(pool)]
        out.append(k)
        n += L.sizes[k]
        i += 1
    return out


def oracle_sample(L, h, seconds=None, target=None):
    """Times the fp64 oracle on whole BERT-large encoder-layer tensors.
    Either for `seconds` of wall time (cycling over the tensors) or over a
    fixed selection of `target` parameters.  Returns (params, seconds)."""
    from oracle import lamb_oracle as O
    pool = [k for k, n in enumerate(L.names) if n.startswith("layer0.")]
    inputs = {}

    def inp(k):
        if k not in inputs:
            m, v = L.state_warm(k)
            inputs[k] = (L.weights(k), L.grad(k, 1), m, v)
        return inputs[k]

    kw = dict(t=1000, lr=float(h.lr), beta1=h.beta1, beta2=h.beta2,
              eps=h.eps, weight_decay=h.weight_decay, phi_kind=h.phi,
              gamma_l=h.gamma_l, gamma_u=h.gamma_u, g_dtype=L.grad_dtype)
    done, spent, i = 0, 0.0, 0
    ks = select_params(L, target, pool) if target else None
    while True:
        if ks is not None:
            if i >= len(ks):
                break
            k = ks[i]
        else:
            if spent >= seconds:
                break
            k = pool[i % len(pool)]
        w, g, m, v = inp(k)
        t0 = time.perf_counter()
        O.lamb_tensor(w, g, m, v, decay=bool(L.decay[k]), **kw)
        spent += time.perf_counter() - t0
        done += L.sizes[k]
        i += 1
    return done, spent


def _oracle_pool_worker(ks, barrier, q):
    """One process of the all-core oracle baseline: builds the inputs of its
    tensors (untimed), waits for every worker, then runs the oracle on them."""
    sys.path.insert(0, ROOT)
    from oracle import lamb_oracle as O
    from paper_1904_00962_gb300.workloads import bert_large_layout
    L = bert_large_layout()
    h = L.hyper
    kw = dict(t=1000, lr=float(h.lr), beta1=h.beta1, beta2=h.beta2,
              eps=h.eps, weight_decay=h.weight_decay, phi_kind=h.phi,
              gamma_l=h.gamma_l, gamma_u=h.gamma_u, g_dtype=L.grad_dtype)
    inputs = []
    for k in ks:
        m, v = L.state_warm(k)
        inputs.append((k, L.weights(k), L.grad(k, 1), m, v))
    barrier.wait()
    t0 = time.time()
    n = 0
    for k, w, g, m, v in inputs:
        O.lamb_tensor(w, g, m, v, decay=bool(L.decay[k]), **kw)
        n += L.sizes[k]
    q.put((n, t0, time.time()))


def oracle_pool(L, per_core_params, workers):
    """The oracle over all host cores: a process per core (spawned, so no
    CUDA state is inherited), each given whole BERT-large layer-0 tensors
    totalling ~per_core_params, timed from a common start to the last
    finish.  Returns (params, wall seconds)."""
    import multiprocessing as mp
    pool = [k for k, n in enumerate(L.names) if n.startswith("layer0.")]
    assign = [[] for _ in range(workers)]
    load = [0] * workers
    i = 0
    while min(load) < per_core_params:
        k = pool[i % len(pool)]
        j = load.index(min(load))
        assign[j].append(k)
        load[j] += L.sizes[k]
        i += 1
    ctx = mp.get_context("spawn")
    barrier = ctx.Barrier(workers)
    q = ctx.Queue()
    procs = [ctx.Process(target=_oracle_pool_worker, args=(a, barrier, q))
             for a in assign]
    for pr in procs:
        pr.start()
    import queue as _queue
    res, deadline = [], time.time() + 900
    while len(res) < len(procs):
        try:
            res.append(q.get(timeout=5))
        except _queue.Empty:
            dead = [pr.exitcode for pr in procs if pr.exitcode not in (None, 0)]
            if dead or time.time() > deadline:
                for pr in procs:
                    if pr.is_alive():
                        pr.terminate()
                raise RuntimeError(f"oracle pool failed (exit codes {dead})")
    for pr in procs:
        pr.join(timeout=60)
    params = sum(r[0] for r in res)
    wall = max(r[2] for r in res) - min(r[1] for r in res)
    return params, wall


def host_description():
    """CPU model and core count of this host (for the CPU baseline)."""
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True,
                             timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if model is None:
        try:
            for line in open("/proc/cpuinfo"):
                if line.lower().startswith(("model name", "cpu part")):
                    model = line.split(":", 1)[1].strip()
                    break
        except OSError:
            pass
    import platform
    return {"cpu_count": os.cpu_count(), "cpu_model": model,
            "machine": platform.machine()}


# ---------------------------------------------------------------------------
# reference arm: the fp64 oracle on the host cores
# ---------------------------------------------------------------------------

def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_1904_00962_gb300.workloads import bert_large_layout
    L = bert_large_layout()
    h = L.hyper
    # each step: whole layer-0 tensors totalling ~target parameters, sized so
    # that K + W steps take about 90 s at the ~5e7 params/s one core of the
    # GPU machine's host reaches (at most all of layer 0, 12.6M parameters)
    target = int(min(max(5.0e7 * 90.0 / max(args.steps + args.warmup, 1),
                         4096), 12.6e6))
    for _ in range(args.warmup):
        oracle_sample(L, h, target=target)
    done, spent = 0, 0.0
    for _ in range(args.steps):
        d, s = oracle_sample(L, h, target=target)
        done += d
        spent += s
    value = done / spent
    sample = (f"per step: whole BERT-large layer-0 tensors totalling >= "
              f"{target} params (fp64 NumPy oracle, one tensor at a time, "
              f"1 thread)")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * spent / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic",
        "config": {"workload": "bert_large_layout", "n_params": L.n_params,
                   "n_tensors": L.n_tensors, "grad_dtype": "bf16",
                   "sample_params_per_step": target},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def layout_hyper(L, opt, variant="plain"):
    """The layout's hyper-parameters for optimizer `opt` (LARS takes the
    layout's own LARS settings, else lr 1, kappa 1e-3, no bias correction)
    and the C-ABI struct for one step with them (t incremented per step)."""
    from paper_1904_00962_gb300 import binding as B
    lars = opt == "lars"
    h = L.lars_hyper if (lars and L.lars_hyper) else L.hyper
    if lars and not L.lars_hyper:
        h = type(h)(lr=1.0, beta1=0.9, weight_decay=1e-4, trust_coef=1e-3,
                    bias_correction=False)
    hyper = B.make_hyper(beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                         weight_decay=h.weight_decay, phi=h.phi,
                         gamma_l=h.gamma_l, gamma_u=h.gamma_u,
                         trust_coef=h.trust_coef,
                         bias_correction=not lars, increment_step=True,
                         grad_norm=variant == "grad_norm",
                         skip_nonfinite=variant == "skip_nonfinite",
                         decoupled_decay=variant == "decoupled")
    return h, hyper


def run_ours(args):
    import numpy as np
    import torch

    from paper_1904_00962_gb300 import binding as B
    from paper_1904_00962_gb300 import build as build_mod
    from paper_1904_00962_gb300.state import DeviceState, LambPlan
    from paper_1904_00962_gb300.workloads import bert_large_layout, bert_layout

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if not os.path.exists(B.LIB_PATH):
        build_mod.build()
    B.load()

    from paper_1904_00962_gb300.workloads import get_layout
    if args.layout == "bert_large" and args.layers != 24:
        L = bert_layout(args.layers, 1024, 4096, name="bert_large",
                        grad_dtype="bf16", copy_dtype="bf16",
                        measured_step=1000)
        workload = f"bert_large_layout_{args.layers}_layers"
    else:
        L = get_layout(args.layout)
        workload = f"{args.layout}_layout"
    opt = args.optimizer
    if opt != "lamb":
        workload += f"_{opt}"
    if args.variant != "plain":
        workload += f"_{args.variant}"
    lars = opt == "lars"
    h, hyper = layout_hyper(L, opt, args.variant)
    P = L.n_params
    st = DeviceState(L.sizes, grad_dtype=L.grad_dtype,
                     copy_dtype=L.copy_dtype, device=dev, with_v=not lars)
    for k in range(L.n_tensors):
        st.upload("w", k, L.weights(k))
        st.upload("g", k, L.grad(k, 1))
    plan = LambPlan(st, L.decay, algorithm=ALGO_CODES[args.algo],
                    chunk_elems=args.chunk_elems)
    info = plan.info()
    algo = info["algorithm"]
    if args.algo == "auto" and opt == "lars" and algo == 3 and \
            info["n_rounds"] > 1:
        algo = 1   # AUTO runs LARS over several rounds on the two-pass kernels
    streamed = 0
    if algo == 3:
        cap = info["grid_blocks"] * info["rows_per_cta"] * info["row_elems"]
        streamed = sum(s for s in L.sizes if s > cap)
    kernel_names, kernel_bytes = kernel_model(
        opt, algo, 2 if L.grad_dtype == "bf16" else 4,
        2 if L.copy_dtype == "bf16" else 0, args.variant, streamed / P)
    profile = PROFILES.get((algo, args.layout, opt)) if (
        args.variant == "plain" and args.layers == 24) else None
    d_step = torch.ones(1, dtype=torch.int64, device=dev)
    d_lr = torch.full((1,), float(np.float32(h.lr)), dtype=torch.float32,
                      device=dev)
    d_prod = torch.ones(1, dtype=torch.float64, device=dev)

    stream = torch.cuda.current_stream(dev)
    # one step per call, arguments marshalled once per plan
    calls = {}

    def one_step(pl=plan):
        c = calls.get(pl.handle)
        if c is None:
            c = calls[pl.handle] = pl.step_call(
                opt, hyper, d_step, d_lr, d_prod if opt in ("nlamb", "nnlamb")
                else None, 0.004, stream)
        c()

    def barrier():
        torch.cuda.synchronize(dev)
        if world > 1:
            torch.distributed.barrier()

    # warm-up: t = 1..W from m = v = 0, then jump to the measured step
    for _ in range(args.warmup):
        one_step()
    d_step.fill_(1000)
    barrier()

    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        gpu_id = None
    clocks = ClockSampler(gpu_id) if rank == 0 else None
    time.sleep(0.3)   # let the sampler start

    # ---- device-resident timed region ----------------------------------
    barrier()
    wall0 = _dt.datetime.now()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        one_step()
    e1.record(stream)
    barrier()
    ms_total = e0.elapsed_time(e1)
    # Per-kernel durations: the same K steps again, with the event pair the
    # library records around each kernel on the launching stream.  They are
    # kept out of the region above because on a layout whose step takes a
    # few microseconds the events themselves add to the step.
    B.lamb_plan_set_timing(plan.handle, True)
    e0.record(stream)
    for _ in range(args.steps):
        one_step()
    e1.record(stream)
    barrier()
    ms_instr = e0.elapsed_time(e1)
    n_timed, ms_kernels = B.lamb_plan_read_timing(plan.handle, 3)
    B.lamb_plan_set_timing(plan.handle, False)
    # The first K timed steps are the measurement.  When the two regions take
    # less than CLOCK_WINDOW_S, the same K-step region runs again (each timed
    # the same way) until the clock sampler has watched the GPU for that long,
    # so the clock record never rests on one or two samples.
    repeats_ms = [ms_total, ms_instr]
    while sum(repeats_ms) < CLOCK_WINDOW_S * 1e3 and len(repeats_ms) < 1000:
        e0.record(stream)
        for _ in range(args.steps):
            one_step()
        e1.record(stream)
        e1.synchronize()
        repeats_ms.append(e0.elapsed_time(e1))
    barrier()
    wall1 = _dt.datetime.now()
    if clocks:
        clocks.mark(wall0, wall1)
    ms_total = max_over_ranks(ms_total, dev)
    status = plan.query(clear=True)

    # ---- end to end: pinned host gradients in, trust ratios out ----------
    # Every step uploads its gradients from pinned host memory and the host
    # reads its trust ratios back.  Two gradient buffers, each with a plan
    # over the same w, m, v (and copy), let the upload of step s+1's
    # gradients (copy streams) run while step s computes, as in a training
    # loop whose backward pass fills one buffer while the optimizer consumes
    # the other; an upload into a buffer waits for the step that last read
    # it.  The host takes step s-1's trust ratios while step s runs.
    k_e2e = args.e2e_steps if args.e2e_steps is not None else min(args.steps, 50)
    g_host = torch.empty(st.total, dtype=st.g.dtype).pin_memory()
    g_host.copy_(st.g.cpu())
    ratio_host = torch.empty(2, L.n_tensors, dtype=torch.float64).pin_memory()
    h2d = L.n_params * st.g.element_size()
    d2h = L.n_tensors * 8
    g_dev = [st.g, torch.empty_like(st.g)]
    plan2 = LambPlan(st, L.decay, algorithm=ALGO_CODES[args.algo],
                     chunk_elems=args.chunk_elems)
    es = st.g.element_size()
    B.lamb_plan_bind(plan2.handle, st.ptrs("w"),
                     [g_dev[1].data_ptr() + es * o for o in st.offsets],
                     st.ptrs("m"), st.ptrs("v"), st.ptrs("copy"))
    plans = [plan, plan2]
    n_up = max(1, args.e2e_streams)
    up_streams = [torch.cuda.Stream(dev) for _ in range(n_up)]
    bounds = [st.total * j // n_up for j in range(n_up + 1)]
    copied = [[torch.cuda.Event() for _ in range(n_up)] for _ in range(2)]
    consumed = [torch.cuda.Event(), torch.cuda.Event()]
    done = [torch.cuda.Event(), torch.cuda.Event()]

    def upload(i):
        for j, us in enumerate(up_streams):
            us.wait_event(consumed[i])
            with torch.cuda.stream(us):
                a, b = bounds[j], bounds[j + 1]
                g_dev[i][a:b].copy_(g_host[a:b], non_blocking=True)
            copied[i][j].record(us)

    barrier()
    e2 = torch.cuda.Event(enable_timing=True)
    e3 = torch.cuda.Event(enable_timing=True)
    e2.record(stream)
    for us in up_streams:
        us.wait_event(e2)
    upload(0)
    for s_ in range(k_e2e):
        i = s_ % 2
        if s_ + 1 < k_e2e:
            upload(1 - i)
        for ev in copied[i]:
            stream.wait_event(ev)
        one_step(plans[i])
        consumed[i].record(stream)
        B.lamb_plan_copy_trust_ratios(plans[i].handle,
                                      ratio_host[i].data_ptr(),
                                      stream=stream.cuda_stream)
        done[i].record(stream)
        if s_ >= 1:
            done[1 - i].synchronize()
            assert math.isfinite(float(ratio_host[1 - i][0]))
    e3.record(stream)
    barrier()
    ms_e2e = e2.elapsed_time(e3)
    ms_e2e = max_over_ranks(ms_e2e, dev)
    assert math.isfinite(float(ratio_host[(k_e2e - 1) % 2][0]))
    # The host link's own rate, outside the timed region: plain uploads of
    # the same gradient bytes with nothing else running.
    c0 = torch.cuda.Event(enable_timing=True)
    c1 = torch.cuda.Event(enable_timing=True)
    us = up_streams[0]
    us.wait_stream(stream)
    c0.record(us)
    with torch.cuda.stream(us):
        for _ in range(4):
            g_dev[1].copy_(g_host, non_blocking=True)
    c1.record(us)
    c1.synchronize()
    h2d_copy_gbs = 4 * h2d / (c0.elapsed_time(c1) * 1e6)
    calls.pop(plan2.handle, None)
    plan2.destroy()
    del g_dev[1]
    clk = clocks.stop() if clocks else None
    noalloc = None
    if rank == 0 and opt == "lamb" and args.variant == "plain":
        try:
            noalloc = noalloc_overhead(st, L, hyper, d_step, d_lr, stream,
                                       one_step)
        except B.LambError as e:   # beyond the entry point's limits
            noalloc = {"unavailable": str(e)}

    if rank != 0:
        plan.destroy()
        if world > 1:
            torch.distributed.destroy_process_group()
        return 0

    # ---- roofline of the dominant kernel --------------------------------
    peak, peak_src = load_peaks()
    per_launch_ms = [ms / max(n_timed, 1)
                     for ms in ms_kernels[:len(kernel_names)]]
    dom = int(np.argmax(per_launch_ms))
    alg_bytes = kernel_bytes[dom] * P
    achieved = alg_bytes / (per_launch_ms[dom] * 1e-3) / 1e9
    traffic = profiled_traffic(profile[0], dom, profile[1], profile[2]) \
        if profile else None
    ms_step = ms_total / args.steps
    step_bytes = sum(kernel_bytes)
    single_bytes = single_touch_bytes(opt, 2 if L.grad_dtype == "bf16" else 4,
                                      2 if L.copy_dtype == "bf16" else 0)
    two_bytes = two_pass_bytes(opt, 2 if L.grad_dtype == "bf16" else 4,
                               2 if L.copy_dtype == "bf16" else 0)
    step_gbs = step_bytes * P / (ms_step * 1e-3) / 1e9

    cpu = None
    if not args.no_cpu_baseline and world == 1:
        L_ref = L if args.layout == "bert_large" and args.layers == 24 \
            else bert_large_layout()
        h_ref = L_ref.hyper
        done_p, spent = oracle_sample(L_ref, h_ref, seconds=args.cpu_seconds)
        rate1 = done_p / spent
        cores = os.cpu_count() or 1
        per_core = int(rate1 * min(args.cpu_seconds, 5.0))
        pool_p, pool_s = oracle_pool(L_ref, per_core, cores)
        cpu = {"value": rate1, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": (f"{done_p} params: whole BERT-large layer-0 tensors "
                          f"cycled for ~{args.cpu_seconds:.0f} s, fp64 NumPy "
                          f"oracle, 1 process on 1 core"),
               "all_cores": {
                   "value": pool_p / pool_s, "unit": UNIT, "cores": cores,
                   "kind": "oracle",
                   "sample": (f"{pool_p} params: whole BERT-large layer-0 "
                              f"tensors, ~{per_core} per process, one spawned "
                              f"process per core, wall time from a common "
                              f"start to the last finish ({pool_s:.2f} s)")},
               "host": host_description()}

    line = {
        "metric": METRIC,
        "value": P * world * args.steps / (ms_total * 1e-3),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": workload, "n_params": P,
                   "n_tensors": L.n_tensors, "grad_dtype": L.grad_dtype,
                   "master_dtype": "f32", "copy_dtype": L.copy_dtype,
                   "optimizer": opt, "variant": args.variant,
                   "step_t": 1000, "lr": float(h.lr),
                   "phi": h.phi if h.phi == "identity" else
                   f"clip[{h.gamma_l:g},{h.gamma_u:g}]",
                   "l2": "inputs larger than L2" if P * 16 > 130e6 else
        "state smaller than L2 (no flush; not a bandwidth number)",
                   "parallelism": f"replicas{world}" if world > 1 else "1gpu"},
        # the step's own algorithmic bytes (what the chosen kernels must move)
        "alg_bytes_per_param": step_bytes,
        "hbm_gbs_step": step_gbs,
        "frac_of_peak_alg": step_gbs / peak,
        # the same time against the two fixed byte models
        "two_pass_bytes_per_param": two_bytes,
        "frac_of_peak_two_pass_model": two_bytes * P / (ms_step * 1e-3) /
        1e9 / peak,
        "single_touch_bytes_per_param": single_bytes,
        "frac_of_peak_single_touch_model": single_bytes * P /
        (ms_step * 1e-3) / 1e9 / peak,
        "algorithm": {1: "two_pass", 3: "on_chip"}[algo],
        "kernels": {kernel_names[i]: {"ms_per_launch": per_launch_ms[i],
                                      "alg_bytes_per_param": kernel_bytes[i]}
                    for i in range(len(kernel_names))},
        "frac_of_nominal_alg": step_gbs / NOMINAL_HBM_GBS,
        "nominal_hbm_gbs": NOMINAL_HBM_GBS,
        "ms_per_step_with_kernel_events": ms_instr / args.steps,
        "clock_window": {"regions": len(repeats_ms), "steps_each": args.steps,
                         "ms_per_step_median": statistics.median(
                             repeats_ms) / args.steps,
                         "s": sum(repeats_ms) / 1e3},
        "roofline": {"bound": "hbm", "kernel": kernel_names[dom],
                     "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak,
                     "frac_of_nominal": achieved / NOMINAL_HBM_GBS,
                     "traffic": traffic,
                     "peak_source": f"{peak_src} (MEASURED_PEAKS hbm_gbs)"
                     if peak_src == "measured" else "fallback 6800 GB/s"},
        "e2e": {"value": P * world * k_e2e / (ms_e2e * 1e-3), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "steps": k_e2e, "upload_streams": n_up,
                "upload_gbs": h2d * k_e2e / (ms_e2e * 1e6),
                "h2d_copy_gbs": h2d_copy_gbs,
                "overlap": "upload of step s+1 overlaps step s "
                           "(two gradient buffers)"},
        "noalloc": noalloc,
        "gpu_launches": len(kernel_names) * args.steps,
        "device_status": status,
        "clocks": clk,
        "cpu_baseline": cpu,
    }
    print(json.dumps(line))
    plan.destroy()
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_shard(args):
    """The data-parallel (sharded) step of a W-way split, timed per rank on
    one GPU: each step runs every rank's lamb_shard_pass1, then adds the
    ranks' per-chunk sums arrays and puts the total back into every plan (what
    an all-reduce over NCCL leaves on each rank; here device copies and adds,
    outside the ranks' timings), then every rank's lamb_shard_pass2.  A rank's
    time is its two launches, timed with events on the launching stream.  The
    line gives the slowest rank's time per step beside the unsharded two-pass
    step's time divided by W, which a perfectly split step would reach.
    --chunk-elems sets the sharded plans' chunk size (the unsharded plan
    keeps the library default)."""
    import numpy as np
    import torch

    from paper_1904_00962_gb300 import binding as B
    from paper_1904_00962_gb300 import build as build_mod
    from paper_1904_00962_gb300.state import DeviceState, LambPlan
    from paper_1904_00962_gb300.workloads import get_layout

    rank, world, _ = dist_env()
    if world > 1:   # the emulation is a one-process, one-GPU measurement
        if rank == 0:
            print(json.dumps({"impl": "ours", "unavailable":
                              "--shard-world runs as one process on one GPU"}))
        return 0
    n_ranks = args.shard_world
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    if not os.path.exists(B.LIB_PATH):
        build_mod.build()
    B.load()
    L = get_layout(args.layout)
    opt = args.optimizer
    h, hyper = layout_hyper(L, opt)
    code = {"lamb": B.LAMB_OPT_LAMB, "lars": B.LAMB_OPT_LARS,
            "nlamb": B.LAMB_OPT_NLAMB, "nnlamb": B.LAMB_OPT_NNLAMB}[opt]
    psi = 0.004
    st = DeviceState(L.sizes, grad_dtype=L.grad_dtype,
                     copy_dtype=L.copy_dtype, device=dev,
                     with_v=opt != "lars")
    for k in range(L.n_tensors):
        st.upload("w", k, L.weights(k))
        st.upload("g", k, L.grad(k, 1))
    stream = torch.cuda.current_stream(dev)
    full = LambPlan(st, L.decay, algorithm=B.LAMB_ALGO_TWO_PASS)
    plans = [LambPlan(st, L.decay, algorithm=B.LAMB_ALGO_TWO_PASS,
                      chunk_elems=args.chunk_elems, shard_world=n_ranks,
                      shard_rank=r)
             for r in range(n_ranks)]
    infos = [p.info() for p in plans]
    lr32 = float(np.float32(h.lr))

    def scalars():
        return (torch.ones(1, dtype=torch.int64, device=dev),
                torch.full((1,), lr32, dtype=torch.float32, device=dev),
                torch.ones(1, dtype=torch.float64, device=dev))

    sc = [scalars() for _ in range(n_ranks + 1)]   # the last: unsharded
    nested = opt in ("nlamb", "nnlamb")
    full_step = full.step_call(opt, hyper, sc[-1][0], sc[-1][1],
                               sc[-1][2] if nested else None, psi, stream)
    _, n_sums = B.lamb_plan_partials(plans[0].handle)
    bufs = [torch.empty(n_sums, dtype=torch.float32, device=dev)
            for _ in range(n_ranks)]
    total = torch.empty(n_sums, dtype=torch.float32, device=dev)
    sid = stream.cuda_stream

    def pass_(r, second):
        d_step, d_lr, d_prod = sc[r]
        fn = plans[r].shard_pass2 if second else plans[r].shard_pass1
        fn(hyper, code, d_step, d_lr, d_prod if nested else None,
           momentum_decay=psi, stream=stream)

    def exchange():
        for r, p in enumerate(plans):
            B.lamb_plan_copy_partials(p.handle, bufs[r].data_ptr(), False,
                                      sid)
        torch.sum(torch.stack(bufs), 0, out=total)
        for p in plans:
            B.lamb_plan_copy_partials(p.handle, total.data_ptr(), True, sid)

    def sharded_step(ev=None):
        for r in range(n_ranks):
            if ev:
                ev[r][0].record(stream)
            pass_(r, False)
            if ev:
                ev[r][1].record(stream)
        exchange()
        for r in range(n_ranks):
            if ev:
                ev[r][2].record(stream)
            pass_(r, True)
            if ev:
                ev[r][3].record(stream)

    for _ in range(args.warmup):
        full_step()
        sharded_step()
    for d_step, _, _ in sc:
        d_step.fill_(1000)
    torch.cuda.synchronize(dev)

    gpu_id = None
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        gpu_id = None
    clocks = ClockSampler(gpu_id)
    time.sleep(0.3)
    wall0 = _dt.datetime.now()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        full_step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    ms_full = e0.elapsed_time(e1) / args.steps
    # The host enqueues a sharded step (2W launches, 4W events and the
    # emulated exchange) more slowly than small layouts run it, so a short
    # spin kernel holds the GPU while every timed step is enqueued: the
    # events then time the launches alone, never a wait for the host.  The
    # timed steps are capped so that all of them fit the stream's queue.
    ops = 9 * n_ranks + 3   # stream operations per sharded step
    k_shard = max(1, min(args.steps, 800 // ops))
    t0 = time.perf_counter()
    sharded_step()
    torch.cuda.synchronize(dev)
    host_s = time.perf_counter() - t0
    evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(4)]
            for _ in range(n_ranks)] for _ in range(k_shard)]
    torch.cuda._sleep(int(min(1.0, 3 * k_shard * host_s) * 2.1e9))  # cycles
    for k in range(k_shard):
        sharded_step(evs[k])
    torch.cuda.synchronize(dev)
    wall1 = _dt.datetime.now()
    clocks.mark(wall0, wall1)
    p1 = [sum(evs[k][r][0].elapsed_time(evs[k][r][1])
              for k in range(k_shard)) / k_shard for r in range(n_ranks)]
    p2 = [sum(evs[k][r][2].elapsed_time(evs[k][r][3])
              for k in range(k_shard)) / k_shard for r in range(n_ranks)]
    per_rank = [a + b for a, b in zip(p1, p2)]
    status = [p.query(clear=True) for p in plans + [full]]
    clk = clocks.stop()
    worst = max(per_rank)
    line = {
        "metric": "sharded step: slowest rank's time per step "
                  "(every rank's launches run in turn on one GPU)",
        "value": worst, "unit": "ms", "higher_is_better": False,
        "world": n_ranks, "steps": k_shard, "unsharded_steps": args.steps,
        "warmup": args.warmup, "per_rank_ms": per_rank, "pass1_ms": p1, "pass2_ms": p2,
        "rank_chunks": [i["shard_chunk_end"] - i["shard_chunk_begin"]
                        for i in infos],
        "chunk_elems": infos[0]["chunk_elems"],
        "unsharded_ms": ms_full, "ideal_ms": ms_full / n_ranks,
        "ideal_over_slowest": ms_full / n_ranks / worst,
        "sums_exchanged_bytes": 4 * n_sums,
        "exchange": "per-chunk sums added on the device outside the ranks' "
                    "timings (an all-reduce over NCCL on several GPUs)",
        "dtype": "f32", "data": "synthetic",
        "config": {"workload": f"{args.layout}_layout"
                   + ("" if opt == "lamb" else f"_{opt}"),
                   "n_params": L.n_params, "n_tensors": L.n_tensors,
                   "grad_dtype": L.grad_dtype, "optimizer": opt,
                   "step_t": 1000, "l2": "inputs larger than L2"},
        "device_status": status, "clocks": clk,
    }
    print(json.dumps(line))
    for p in plans + [full]:
        p.destroy()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.shard_world > 1:
        return run_shard(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
