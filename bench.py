"""Throughput of the fused LIF scan, forward + BPTT, on GB300.

One step = the whole hot path over one batch: the Leaky forward scan (Eqs.
3-4) and its BPTT reverse scan with the arctan surrogate, per-neuron beta and
threshold gradients reduced over the batch.  Default workload: I[T=500,
B=64, N=8192] bf16 storage with fp32 state; BPTT from the stored mem/spk
traces (--save recompute: from fp32 checkpoints every 8 steps).

Other scan workloads (`--workload`, the names in workloads.SCAN_WORKLOADS)
time the same step on their shapes.  The network workloads time a whole
training step as one CUDA graph: the dense SNN (Tab. I DSNN) and its
population-coded variant, and the convolutional SNN (Tab. I CSNN) --
forward (by default each GEMM layer fused with its scan), loss (with the
readout's BPTT in the same launch), BPTT (for T > 1 each dense input-gradient
GEMM fused with the lower layer's reverse scan) and AdamW -- in the same
metric, with images/s and per-op times beside it.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle (the
only other implementation of this path) on a bounded sample of the same
workload instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)
# the oracle legs are timed on one host core: keep numpy's BLAS to one thread
for _var in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "OMP_NUM_THREADS"):
    os.environ.setdefault(_var, "1")

METRIC = "neuron-steps/sec (fwd+BPTT) on 1 GB300; achieved HBM GB/s vs roofline"
UNIT = "neuron-steps/s"
DEFAULT_WORKLOAD = "leaky_bf16_T500_B64_N8192"
FALLBACK_HBM_GBS = 6800.0
# scan workloads: the save variant (and checkpoint interval) timed by
# default, the faster one on GB300; the others are timed beside it
DEFAULT_SAVE = {"leaky_bf16_T500_B64_N8192": ("recompute", 8),
                "rleaky_bf16_T500_B64_N8192": ("recompute", 8)}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    # scan workloads: DEFAULT_SAVE names the variant timed by default (the
    # others are timed beside it).  Networks: "fused" (the default) runs
    # each GEMM layer with its scan in the epilogue and stores every trace.
    p.add_argument("--save", default=None, choices=["mem", "recompute", "fused"])
    p.add_argument("--no-graph", action="store_true",
                   help="dense-SNN workload: launch the step eagerly, not as a CUDA graph")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-networks", action="store_true",
                   help="default workload: skip the network training-step records")
    p.add_argument("--no-variants", action="store_true",
                   help="scan workloads: skip timing the other save variants")
    p.add_argument("--ckpt-every", type=int, default=None,
                   help="recompute variant: checkpoint interval K")
    p.add_argument("--batch", type=int, default=None,
                   help="scan workloads: another batch size B (a smaller case for profiling)")
    p.add_argument("--no-torch-eager", action="store_true",
                   help="skip the PyTorch-eager per-timestep context measurement")
    p.add_argument("--cpu-seconds", type=float, default=15.0)
    p.add_argument("--reference-seconds", type=float, default=120.0,
                   help="--impl reference: about how long the whole run takes")
    return p.parse_args()


def workload(args):
    from paper_2211_10725_gb300 import workloads as W
    w = W.SCAN_WORKLOADS[args.workload]
    save = args.save or DEFAULT_SAVE.get(w.name, ("mem", w.ckpt_every))[0]
    k = args.ckpt_every or DEFAULT_SAVE.get(w.name, ("mem", w.ckpt_every))[1]
    if args.batch and args.batch != w.B:
        w = w.scaled(B=args.batch, name=w.name.replace(f"_B{w.B}_", f"_B{args.batch}_"))
    return w.scaled(save=save, ckpt_every=k)


def is_net(args):
    """A whole-network training step (dense or convolutional SNN)."""
    from paper_2211_10725_gb300 import workloads as W
    return args.workload in W.DENSE_WORKLOADS or args.workload in W.CONV_WORKLOADS


def net_workload(name):
    from paper_2211_10725_gb300 import workloads as W
    return W.DENSE_WORKLOADS.get(name) or W.CONV_WORKLOADS[name]


def is_conv(w):
    return hasattr(w, "convs")


def net_inputs(w, seed=None):
    from paper_2211_10725_gb300 import workloads as W
    return W.make_conv_inputs(w, seed) if is_conv(w) else W.make_dense_inputs(w, seed)


def net_neurons(w):
    """Spiking neurons per sample (unpadded): every layer's neurons."""
    if is_conv(w):
        shapes, _ = w.shapes()
        return sum(ho * wo * cout for (_, _, _, cout, _, ho, wo, _, _) in shapes) + w.n_classes
    return sum(w.sizes[1:])


def net_config(w):
    if is_conv(w):
        return {"workload": w.name, "input": [w.H, w.W, w.Cin],
                "convs": [list(c) for c in w.convs], "pool": "2x2 max", "T": w.T, "B": w.B,
                "classes": w.n_classes, "reset": w.reset,
                "beta": "per channel, learnable (conv layers)"}
    return {"workload": w.name, "sizes": list(w.sizes), "T": w.T, "B": w.B,
            "classes": w.n_classes, "neurons_per_class": w.pop}


def net_oracle_pass(w, host, bs):
    """The oracle's forward + loss + BPTT over samples bs of the batch."""
    from oracle import snn_oracle as O
    import numpy as np
    n = len(bs)
    if is_conv(w):
        X = host["X"][:, bs].reshape(w.T * n, w.H, w.W, w.Cin)
        betas = [np.full(c, w.beta) for c, _ in w.convs]
        fwd = O.csnn_forward(X, host["convs"], host["Wfc"], w.T, n, betas, w.beta_fc, w.thr,
                             reset=w.reset)
        O.csnn_backward(fwd, host["convs"], host["Wfc"], host["y"][bs], w.T, n, betas,
                        w.beta_fc, w.thr, w.sg_param, reset=w.reset)
    else:
        xb = host["X"][:, bs].reshape(w.T * n, -1)
        fwd = O.dsnn_forward(xb, host["W"], w.T, n, w.beta, w.thr)
        O.dsnn_backward(fwd, host["W"], host["y"][bs], w.T, n, w.beta, w.thr, w.sg_param,
                        pop=w.pop)


def net_oracle_host(w, inp):
    import numpy as np
    f64 = lambda t: t.float().numpy().astype(np.float64)
    host = {"y": inp["labels"].numpy().astype(np.int64)}
    if is_conv(w):
        host["X"] = f64(inp["X"])                                  # [T, B, H, W, Cin]
        host["convs"] = [f64(c) for c in inp["convs"]]
        host["Wfc"] = f64(inp["Wfc"])
    else:
        host["X"] = f64(inp["X"])                                  # [T, B, K0]
        host["W"] = [f64(x) for x in inp["W"]]
    return host


# ---------------------------------------------------------------------------
# Bytes and peaks
# ---------------------------------------------------------------------------

def esize(dt):
    return 4 if dt == "f32" else 2


def algorithmic_bytes(w):
    """Bytes per neuron-step the contract must touch, per pass (fwd, bwd).

    Forward: read I, write spk (and mem when the layer's mem output is
    requested).  Backward: read grad_spk, read the cheaper saved state (I or
    the mem trace), write grad_I (and read grad_mem when it is given; no
    workload gives it).  Checkpoints, the store variant's trace and spike
    bits, parameters and reductions are overhead, not contract bytes."""
    ei, eo = esize(w.in_dtype), esize(w.io_dtype)
    fwd = ei + eo + (eo if w.want_mem else 0)
    bwd = eo + min(ei, eo) + eo
    return fwd, bwd


def moved_bytes(w):
    """Bytes per neuron-step each pass of the chosen variant moves (fwd,
    bwd): the contract bytes plus the variant's own.  Store: the forward
    writes the mem trace (unless it is an output anyway) and, for half
    storage, one spike bit; the backward reads them back.  Recompute: fp32
    checkpoints every K steps, written once and read once."""
    ei, eo = esize(w.in_dtype), esize(w.io_dtype)
    fwd, bwd = algorithmic_bytes(w)
    if w.save == "recompute":
        ck = 4.0 / w.ckpt_every * (2 if w.neuron == "synaptic" else 1)
        return fwd + ck, bwd + (ei - min(ei, eo)) + ck
    bits = 0.125 if eo != 4 else 0.0
    syn = eo if w.neuron == "synaptic" else 0      # the syn trace for grad_alpha
    return (fwd + (0 if w.want_mem else eo) + bits + syn,
            bwd + (eo - min(ei, eo)) + bits + syn)


def kernel_names(w):
    """Names of the forward and backward scan kernels the variant launches."""
    bwd = "scan_bwd_staged"
    half_in = w.in_dtype != "f32" and w.in_dtype == w.io_dtype
    if w.save == "recompute" and w.neuron != "synaptic" and w.reset != "none" and \
            (w.ckpt_every == 8 or (w.ckpt_every == 16 and half_in)):
        bwd = "scan_bwd_seg"
    return "scan_fwd_staged", bwd


def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            v = float(json.load(f)["hbm_gbs"])
        return v, "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


SCAN_SOURCES = ("scan_kernels.cuh", "scan_dispatch.cuh", "scan_host.cuh", "snn_device.cuh",
                "scan_seg.cuh", "scan_seg_launch.cuh", "scan_bwd_leaky_seg.cu",
                "scan_bwd_leaky_seg8.cu", "scan_bwd_leaky_seg12.cu",
                "scan_fwd.cu", "scan_bwd_leaky.cu", "scan_bwd_leaky_recompute.cu",
                "scan_bwd_synaptic.cu", "scan_bwd_synaptic_recompute.cu", "snn_api.cu")


def kernel_source_hash():
    """Hash of the sources the scan kernels are built from (and launched by)."""
    h = hashlib.sha256()
    for f in sorted(os.path.join(ROOT, "paper_2211_10725_gb300", "csrc", n) for n in SCAN_SOURCES):
        with open(f, "rb") as fh:
            h.update(os.path.basename(f).encode())
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel_key, workload_name):
    """DRAM bytes per launch from a committed ncu summary, valid only if the
    kernel sources are unchanged since it was taken."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            data = json.load(f)
        ent = data[workload_name][kernel_key]
        if ent.get("source_hash") != kernel_source_hash():
            return None
        return float(ent["dram_bytes_per_launch"])
    except Exception:
        return None


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class NvmlClocks:
    """SM clock, power and clock-event reasons read through NVML (the
    driver's management library, called with ctypes) every few
    milliseconds from a thread, so that a timed region of a few tens of
    milliseconds still gets samples.  The GPU is found by its UUID, which
    does not depend on device numbering."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, uuid, period_s=0.002):
        import ctypes
        self.ct = ctypes
        self.lib = ctypes.CDLL("libnvidia-ml.so.1")
        if self.lib.nvmlInit_v2() != 0:
            raise RuntimeError("nvmlInit failed")
        self.h = ctypes.c_void_p()
        if self.lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(self.h)) != 0:
            raise RuntimeError("GPU not found by UUID")
        self.reasons_fn = getattr(self.lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            self.lib.nvmlDeviceGetCurrentClocksThrottleReasons
        mx = ctypes.c_uint()
        self.lib.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx))   # NVML_CLOCK_SM
        self.max_mhz = float(mx.value)
        self.period = period_s
        self.samples = []
        self.stop_flag = False

    def _one(self):
        ct = self.ct
        mhz, mw, rs = ct.c_uint(), ct.c_uint(), ct.c_ulonglong()
        self.lib.nvmlDeviceGetClockInfo(self.h, 1, ct.byref(mhz))
        self.lib.nvmlDeviceGetPowerUsage(self.h, ct.byref(mw))
        self.reasons_fn(self.h, ct.byref(rs))
        return time.time(), float(mhz.value), mw.value / 1000.0, int(rs.value)

    def _run(self):
        while not self.stop_flag:
            self.samples.append(self._one())
            time.sleep(self.period)

    def start(self):
        self.thread = threading.Thread(target=self._run, daemon=True)
        self.thread.start()

    def stop(self):
        self.stop_flag = True
        self.thread.join(timeout=2)

    def summary(self, t0, t1):
        inside = [r for r in self.samples if t0 <= r[0] <= t1]
        note = "NVML, sampled every 2 ms during the timed region"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [],
                    "note": "no samples in the timed region"}
        sm = sorted(r[1] for r in inside)
        reasons = set()
        for r in inside:
            for bit, name in self.REASONS.items():
                if r[3] & bit:
                    reasons.add(name)
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": self.max_mhz, "sm_min_mhz": sm[0],
                "power_w_max": max(r[2] for r in inside), "reasons": sorted(reasons),
                "samples": len(inside), "note": note}


def clock_sampler(dev_index):
    """NVML sampling when the library is there, else nvidia-smi."""
    try:
        import torch
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev_index).uuid)
        return NvmlClocks(uuid)
    except Exception:
        return ClockSampler(dev_index)


class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.samples = []
        self.proc = None
        self.window = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        rows = []
        for ts, line in self.samples:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((ts, float(parts[1]), float(parts[2]), parts))
            except ValueError:
                continue
        inside = [r for r in rows if t0 <= r[0] <= t1]
        note = "sampled during the timed region"
        if not inside and rows:
            mid = 0.5 * (t0 + t1)
            inside = sorted(rows, key=lambda r: abs(r[0] - mid))[:3]
            note = "timed region shorter than the sampling period: nearest samples (warm-up)"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "note": "no samples"}
        sm = sorted(r[1] for r in inside)
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in inside:
            for name, val in zip(names, r[3][5:9]):
                if val.strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[2] for r in inside),
                "reasons": sorted(reasons), "samples": len(inside), "note": note}


# ---------------------------------------------------------------------------
# CPU oracle leg
# ---------------------------------------------------------------------------

def oracle_inputs(w, inp):
    """Host arrays the oracle reads (converted once, outside any timing)."""
    from oracle import snn_oracle as O
    T, B, N = w.T, w.B, w.N
    host = {"I": inp["I"].float().numpy().reshape(T, B * N),
            "gs": inp["grad_spk"].float().numpy().reshape(T, B * N)}
    for name, mode in (("beta", w.beta_mode), ("thr", w.thr_mode), ("alpha", w.alpha_mode),
                       ("v", w.v_mode)):
        if name in inp:
            host[name] = O.lane_param(inp[name].numpy(), B, N, mode, w.C, w.HW)
    return host


def oracle_step(w, host, lanes):
    """One oracle fwd+bwd pass (float64, as it stands) over a lane sample."""
    from oracle import snn_oracle as O
    import numpy as np
    I = host["I"][:, lanes].astype(np.float64)
    gs = host["gs"][:, lanes].astype(np.float64)
    beta, thr = host["beta"][lanes], host["thr"][lanes]
    if w.neuron == "synaptic":
        alpha = host["alpha"][lanes]
        spk, mem, syn = O.synaptic_forward(I, alpha, beta, thr, w.reset)
        O.synaptic_backward(mem, spk, syn, gs, alpha, beta, thr, w.reset, w.detach_reset,
                            w.surrogate, w.sg_param)
    elif w.neuron == "rleaky":
        v = host["v"][lanes]
        spk, mem = O.rleaky_forward(I, v, beta, thr)
        O.rleaky_backward(mem, spk, gs, v, beta, thr, w.detach_reset, w.surrogate, w.sg_param)
    else:
        spk, mem = O.leaky_forward(I, beta, thr, w.reset)
        O.leaky_backward(mem, spk, gs, beta, thr, w.reset, w.detach_reset, w.surrogate,
                         w.sg_param)


def time_oracle(w, inp, seconds, threads=1, host=None):
    """Time the oracle on a bounded sample of the workload: consecutive
    chunks of lanes (all T steps each) until about `seconds` of wall time.

    With threads > 1 the chunks run on a thread pool, one chunk per thread
    at a time: the oracle's per-step work is numpy vector arithmetic over a
    chunk's lanes, which releases the interpreter lock, so the threads run
    on separate cores.  Returns (neuron-steps/s, lanes done, seconds)."""
    import concurrent.futures
    import numpy as np
    L = w.B * w.N
    host = host or oracle_inputs(w, inp)
    chunk = min(L, 16384 if threads > 1 else 65536)
    starts = list(range(0, L, chunk))
    done, t_total, k = 0, 0.0, 0
    with concurrent.futures.ThreadPoolExecutor(max_workers=threads) as ex:
        while t_total < seconds and done < L:
            batch = [starts[(k + j) % len(starts)] for j in range(min(threads, len(starts)))]
            k += len(batch)
            lanes = [np.arange(a, min(L, a + chunk)) for a in batch]
            t0 = time.perf_counter()
            list(ex.map(lambda ln: oracle_step(w, host, ln), lanes))
            t_total += time.perf_counter() - t0
            done += sum(len(x) for x in lanes)
    return w.T * done / t_total, done, t_total


def cpu_baseline(w, inp, seconds):
    """The oracle on one host core and on all of them (a thread per core)."""
    host = oracle_inputs(w, inp)
    cores = os.cpu_count() or 1
    v1, n1, dt1 = time_oracle(w, inp, seconds / 3, 1, host)
    vn, nn, dtn = time_oracle(w, inp, seconds, cores, host)
    return {"value": vn, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{nn} of {w.B * w.N} lanes in chunks of 16384 on {cores} threads, all "
                      f"T={w.T} steps, float64 numpy oracle fwd+BPTT, {dtn:.1f} s",
            "single_core": {"value": v1, "cores": 1,
                            "sample": f"{n1} lanes in chunks of 65536, {dt1:.1f} s"}}


def run_net_reference(args):
    """The oracle's network forward + loss + BPTT on a bounded sample of the
    batch per step (samples are independent until the dW sums)."""
    import concurrent.futures
    import numpy as np
    w = net_workload(args.workload)
    host = net_oracle_host(w, net_inputs(w))
    cores = os.cpu_count() or 1
    pool = concurrent.futures.ThreadPoolExecutor(max_workers=cores)

    def step(bs):
        # samples are independent until the dW sums: one chunk per host core
        chunks = [c for c in np.array_split(bs, min(cores, len(bs))) if len(c)]
        list(pool.map(lambda c: net_oracle_pass(w, host, c), chunks))

    t0 = time.perf_counter()
    probe = min(w.B, 4)
    net_oracle_pass(w, host, np.arange(probe))
    per_sample = (time.perf_counter() - t0) / probe / cores
    total = max(1, args.steps + args.warmup)
    n = int(max(1, min(w.B, args.reference_seconds / total / per_sample)))
    rng = np.random.default_rng(0)
    samples = [np.sort(rng.choice(w.B, n, replace=False)) for _ in range(total)]
    for i in range(args.warmup):
        step(samples[i])
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(samples[args.warmup + i])
    dt = time.perf_counter() - t0
    pool.shutdown()
    value = w.T * n * net_neurons(w) * args.steps / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": dict(net_config(w), sample_batch_per_step=n),
        "images_per_s": n * args.steps / dt,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{n} random samples of {w.B} per step on {cores} threads, "
                                   f"all T={w.T} steps, float64 oracle forward+loss+BPTT "
                                   f"(no optimiser)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    if is_net(args):
        run_net_reference(args)
        return
    import numpy as np
    from paper_2211_10725_gb300 import workloads as W
    import concurrent.futures
    w = workload(args)
    inp = oracle_inputs(w, W.make_scan_inputs(w))
    L = w.B * w.N
    cores = os.cpu_count() or 1
    pool = concurrent.futures.ThreadPoolExecutor(max_workers=cores)

    def step(lanes):
        # the sample in one chunk per host core (numpy releases the
        # interpreter lock inside its vector loops)
        list(pool.map(lambda c: oracle_step(w, inp, c), np.array_split(lanes, cores)))

    # size one step's lane sample so that warm-up + steps take about 2 minutes
    probe = min(L, 2048 * cores)
    t0 = time.perf_counter()
    step(np.arange(probe))
    per_lane = (time.perf_counter() - t0) / probe
    total = max(1, args.steps + args.warmup)
    n = int(max(64 * cores, min(L, args.reference_seconds / total / per_lane)))
    rng = np.random.default_rng(0)
    samples = [np.sort(rng.choice(L, n, replace=False)) for _ in range(total)]
    for i in range(args.warmup):
        step(samples[i])
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(samples[args.warmup + i])
    dt = time.perf_counter() - t0
    pool.shutdown()
    value = w.T * n * args.steps / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "T": w.T, "B": w.B, "N": w.N,
                   "sample_lanes_per_step": n},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{n} random lanes of {L} per step on {cores} threads, all "
                                   f"T={w.T} steps, float64 numpy oracle fwd+BPTT"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------

def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2211_10725_gb300 import snn
    from paper_2211_10725_gb300 import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = workload(args)
    # weak scaling: every rank scans its own batch of the same shape
    inp = W.make_scan_inputs(w, seed=W.SEED_BASE + w.seed_index + 1000 * rank)
    d = {k: v.to(dev) for k, v in inp.items()}
    layer = snn.ScanLayer(w, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        layer.forward(d["I"], d["beta"], d["thr"], d.get("alpha"), v=d.get("v"))
        layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"),
                       want_state_grads=False, v=d.get("v"))

    c0 = snn.snn_kernel_launches()
    warm = max(1, args.warmup)
    for _ in range(warm):
        step()
    torch.cuda.synchronize()
    launches_per_step = (snn.snn_kernel_launches() - c0) // warm
    status = layer.status()
    if status != 0:
        raise RuntimeError(f"kernel status {status} after warm-up")

    sampler = clock_sampler(local)
    if rank == 0:
        sampler.start()
        time.sleep(0.3)
    K = args.steps
    # the K steps back to back, bracketed by two events: an event recorded
    # between two launches would stop the second from starting early under
    # programmatic dependent launch, so the per-pass times come from a
    # second loop of K steps with events between the passes
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    e0.record(stream)
    for k in range(K):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    t_wall1 = time.time()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3 * K + 1)]
    ev[0].record(stream)
    for k in range(K):
        layer.forward(d["I"], d["beta"], d["thr"], d.get("alpha"), v=d.get("v"))
        ev[3 * k + 1].record(stream)
        layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"),
                       want_state_grads=False, v=d.get("v"))
        ev[3 * k + 2].record(stream)
        ev[3 * k + 3].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    if rank == 0:
        time.sleep(0.2)
        sampler.stop()
    total_ms = e0.elapsed_time(e1)
    fwd_ms = sum(ev[3 * k].elapsed_time(ev[3 * k + 1]) for k in range(K)) / K
    bwd_ms = sum(ev[3 * k + 1].elapsed_time(ev[3 * k + 2]) for k in range(K)) / K
    if world > 1:
        t = torch.tensor([total_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    status = layer.status()
    if status != 0:
        raise RuntimeError(f"kernel status {status} in the timed region")

    ns_per_step = w.T * w.B * w.N
    value = world * ns_per_step * K / (total_ms * 1e-3)

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, w, inp, layer, dev, world)

    link = link_bandwidth(dev) if (e2e is not None and rank == 0) else None
    if e2e is not None and link is not None:
        moved = e2e["h2d_bytes_per_step"] + e2e["d2h_bytes_per_step"]
        step_s = ns_per_step * world / e2e["value"]
        e2e["link"] = dict(link, achieved_gbs=moved / step_s / 1e9,
                           frac_of_bidir=moved / step_s / 1e9 / link["bidir_gbs"])

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    peak, peak_kind = hbm_peak()
    fwd_alg, bwd_alg = algorithmic_bytes(w)
    fwd_mov, bwd_mov = moved_bytes(w)
    fwd_name, bwd_name = kernel_names(w)
    step_ms = total_ms / K

    def kern(name, ms, alg, mov):
        gbs = alg * ns_per_step / (ms * 1e-3) / 1e9
        return {"name": name, "ms": ms, "algorithmic_bytes_per_ns": alg,
                "achieved": gbs, "frac": gbs / peak,
                "moved_bytes_per_ns": mov, "moved_gbs": mov * ns_per_step / (ms * 1e-3) / 1e9}

    kf = kern(fwd_name, fwd_ms, fwd_alg, fwd_mov)
    kb = kern(bwd_name + " + parameter reduction", bwd_ms, bwd_alg, bwd_mov)
    dom = kf if fwd_ms >= bwd_ms else kb   # the longer pass
    dom_key = f"{dom['name'].split(' ')[0]}[{w.neuron},{w.save}"
    dom_key += f",K{w.ckpt_every}]" if w.save == "recompute" else "]"
    minimal = fwd_alg + bwd_alg
    path_gbs = minimal * ns_per_step / (step_ms * 1e-3) / 1e9
    clocks = sampler.summary(t_wall0, t_wall1)
    eager = None
    if not args.no_torch_eager and world == 1:
        eager = time_torch_eager(w, inp, dev)
    variants = None
    if not args.no_variants and world == 1:
        variants = time_other_variants(args, w, inp, dev)
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        cpu = cpu_baseline(w, inp, args.cpu_seconds)
    networks = None
    if not args.no_networks and world == 1 and args.workload == DEFAULT_WORKLOAD:
        networks = time_networks()
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.io_dtype, "state_dtype": "f32",
        "data": "synthetic",
        "config": {"workload": w.name, "T": w.T, "B": w.B, "N": w.N, "neuron": w.neuron,
                   "storage": w.io_dtype, "input": w.in_dtype, "save": w.save,
                   "ckpt_every": w.ckpt_every if w.save == "recompute" else None,
                   "surrogate": w.surrogate, "reset": w.reset,
                   "params": f"beta {w.beta_mode}, thr {w.thr_mode}",
                   "l2": "inputs larger than L2 (each [T,B,N] tensor >> 129 MB), no flush",
                   "timing": "K steps back to back between two CUDA events; the per-pass "
                             "times (roofline kernels) from a second loop of K steps with "
                             "events between the passes",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        # dominant kernel = the longer pass, judged on the contract bytes
        # (read I, write spk; read grad_spk and the saved state, write
        # grad_I); the variant's own bytes (trace, spike bits, checkpoints)
        # are in moved_bytes_per_ns, and in `traffic` when ncu measured them
        "roofline": {"bound": "hbm", "kernel": dom["name"], "achieved": dom["achieved"],
                     "peak": peak, "unit": "GB/s", "frac": dom["frac"],
                     "peak_kind": peak_kind + " copy bandwidth",
                     "algorithmic_bytes_per_ns": dom["algorithmic_bytes_per_ns"],
                     "units_per_launch": ns_per_step,
                     "traffic": profiled_traffic(dom_key, w.name),
                     "kernels": {"fwd": kf, "bwd": kb},
                     "path": {"minimal_bytes_per_ns": minimal, "achieved": path_gbs,
                              "frac": path_gbs / peak,
                              "frac_of_8tbs": path_gbs / 8000.0,
                              "target_frac_of_8tbs": 0.70}},
        "clocks": clocks,
        # counted by the library over the warm-up steps: forward scan,
        # backward scan, one reduction per parameter layout
        "gpu_launches": launches_per_step * K,
        "gpu_launches_per_step": launches_per_step,
        "variants": variants,
        # the training steps of the paper's networks (Tab. I DSNN and CSNN,
        # Sec. VII population code), each in a process of its own: context
        # for the same kernels inside whole networks
        "networks": networks,
        "cpu_baseline": cpu,
        "torch_eager_context": eager,
        "e2e": e2e,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def time_networks(steps=30, warmup=3):
    """The default bench line's network records: `bench.py --workload <net>`
    run in a child process per network (graph-replayed training steps), the
    main figures of its JSON line kept."""
    from paper_2211_10725_gb300 import workloads as W
    out = {}
    for name in list(W.DENSE_WORKLOADS) + list(W.CONV_WORKLOADS):
        cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--workload", name, "--steps",
               str(steps), "--warmup", str(warmup), "--no-e2e", "--no-cpu-baseline"]
        try:
            r = subprocess.run(cmd, capture_output=True, text=True, timeout=600)
            line = json.loads(r.stdout.strip().splitlines()[-1])
        except Exception as exc:  # report, do not hide: the record says what failed
            out[name] = {"error": f"{type(exc).__name__}: {exc}"[:300]}
            continue
        rf = line.get("roofline", {})
        out[name] = {k: line.get(k) for k in ("value", "unit", "ms_per_step", "images_per_s",
                                              "gpu_launches_per_step", "clocks")}
        out[name]["config"] = {k: line["config"].get(k) for k in ("save", "launch", "T", "B")}
        out[name]["roofline"] = {k: rf.get(k) for k in ("bound", "kernel", "achieved", "peak",
                                                       "unit", "frac")}
    return out


def time_other_variants(args, w, inp, dev, steps=10):
    """Forward + BPTT of the same workload with the other ways of saving
    state for the reverse pass (store the trace / recompute from
    checkpoints every 8, 12 or 16 steps), timed like the headline: steps
    back to back for the value, then a loop with events between the passes
    for fwd_ms and bwd_ms."""
    import torch
    from paper_2211_10725_gb300 import snn
    out = []
    d = {k: v.to(dev) for k, v in inp.items()}
    cands = [("mem", w.ckpt_every), ("recompute", 8), ("recompute", 12), ("recompute", 16)]
    for save, k in cands:
        if save == w.save and (save == "mem" or k == w.ckpt_every):
            continue
        v = w.scaled(save=save, ckpt_every=k)
        layer = snn.ScanLayer(v, device=dev)

        def fwd():
            layer.forward(d["I"], d["beta"], d["thr"], d.get("alpha"), v=d.get("v"))

        def bwd():
            layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"),
                           want_state_grads=False, v=d.get("v"))

        for _ in range(3):
            fwd()
            bwd()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(steps):
            fwd()
            bwd()
        e1.record()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3 * steps)]
        for i in range(steps):
            ev[3 * i].record()
            fwd()
            ev[3 * i + 1].record()
            bwd()
            ev[3 * i + 2].record()
        torch.cuda.synchronize()
        if layer.status() != 0:
            raise RuntimeError(f"kernel status {layer.status()} ({save})")
        step_ms = e0.elapsed_time(e1) / steps
        f = sum(ev[3 * i].elapsed_time(ev[3 * i + 1]) for i in range(steps)) / steps
        b = sum(ev[3 * i + 1].elapsed_time(ev[3 * i + 2]) for i in range(steps)) / steps
        fm, bm = moved_bytes(v)
        out.append({"save": save, "ckpt_every": k if save == "recompute" else None,
                    "value": w.T * w.B * w.N / (step_ms * 1e-3), "ms_per_step": step_ms,
                    "fwd_ms": f, "bwd_ms": b,
                    "kernels": list(kernel_names(v)), "moved_bytes_per_ns": fm + bm,
                    "steps": steps})
        del layer
        torch.cuda.empty_cache()
    return out


# ---------------------------------------------------------------------------
# Dense SNN training step (784-1000-1000-10, T=25, B=128)
# ---------------------------------------------------------------------------

def tensor_peak(sustained):
    key = "bf16_tflops_sustained" if sustained else "bf16_tflops"
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)[key]), "measured"
    except Exception:
        return (1700.0 if sustained else 1900.0), "fallback"


def net_flops(w):
    """Algorithmic GEMM flops of one training step (unpadded sizes): the
    forward currents of every layer, every dW, and dX of every layer but the
    first (a convolution as its patch-row product)."""
    M = w.T * w.B
    if is_conv(w):
        shapes, n_flat = w.shapes()
        conv = [2 * M * ho * wo * k * k * cin * cout
                for (_, _, cin, cout, k, ho, wo, _, _) in shapes]
        fc = 2 * M * n_flat * w.n_classes
        fwd = sum(conv) + fc
        return fwd, fwd, sum(conv[1:]) + fc
    fwd = sum(2 * M * k * n for k, n in zip(w.sizes[:-1], w.sizes[1:]))
    dx = sum(2 * M * k * n for k, n in zip(w.sizes[1:-1], w.sizes[2:]))
    return fwd, fwd, dx


def conv_op_bytes(net):
    """Bytes each op of the CSNN step must read and write as designed (the
    sizes of its operands and results, each once), for the per-op HBM
    roofline; the scans by the scan byte model (I, spk, grad_spk, grad_I;
    checkpoints excluded)."""
    nb = lambda t: 0 if t is None else t.numel() * t.element_size()
    T, B, M = net.w.T, net.w.B, net.M
    out = {}
    for l, g in enumerate(net.geo):
        x_bytes = M * g[0] * g[1] * g[2] * 2
        layer = net.layers[l]
        ns = T * B * layer.w.N
        f, b = algorithmic_bytes(layer.w)
        if net.cols[l] is None:   # direct convolution: reads the input map itself
            out[f"conv_fwd{l}"] = x_bytes + nb(net.W[l]) + nb(net.I[l])
        else:
            out[f"im2col{l}"] = x_bytes + nb(net.cols[l])
            if net.I[l] is None:  # GEMM with the scan in its epilogue
                out[f"conv_scan_fwd{l}"] = (nb(net.cols[l]) + nb(net.W[l]) + nb(layer.spk)
                                            + nb(layer.mem) + nb(layer.ckpt))
            else:
                out[f"conv_fwd{l}"] = nb(net.cols[l]) + nb(net.W[l]) + nb(net.I[l])
        if net.I[l] is not None:
            out[f"scan_fwd{l}"] = f * ns
        out[f"pool_fwd{l}"] = nb(layer.spk) + nb(net.pool[l]) + nb(net.idx[l])
        out[f"pool_bwd{l}"] = nb(net.grad_pool[l]) + nb(net.idx[l]) + nb(net.grad_spk[l])
        out[f"scan_bwd{l}"] = b * ns
        src = x_bytes if net.cols[l] is None else nb(net.cols[l])
        out[f"conv_bwd{l}"] = (src + nb(layer.grad_I) + nb(net.W[l]) + nb(net.dcols[l])
                               + nb(net.dW[l]))
        if l > 0:
            out[f"col2im{l}"] = nb(net.dcols[l]) + nb(net.grad_pool[l - 1])
    o = net.out_layer
    f, b = algorithmic_bytes(o.w)
    ns = T * B * o.w.N
    flat = nb(net.pool[-1])
    if net.I_fc is None:
        out["fc_scan_fwd"] = flat + nb(net.W[-1]) + nb(o.spk) + nb(o.mem) + nb(o.ckpt)
    else:
        out["fc_fwd"] = flat + nb(net.W[-1]) + nb(net.I_fc)
        out["scan_fwd_out"] = f * ns
    out["ce_loss"] = nb(o.spk) + nb(net.grad_out)
    if net.fused_loss:   # the readout's BPTT in the loss launch: its trace in, dL/dI out
        out["ce_loss"] += nb(o.mem) + nb(o.grad_I)
    else:
        out["scan_bwd_out"] = b * ns
    out["fc_bwd"] = flat + nb(net.W[-1]) + nb(o.grad_I) + nb(net.grad_pool[-1]) + nb(net.dW[-1])
    out["adamw"] = (4 * 2 * nb(net.W32_flat) + nb(net.W_flat)
                    + 4 * 2 * nb(net.beta_flat))
    return out


def _timing_events(external):
    import torch
    if external:
        return torch.cuda.Event(enable_timing=True, external=True)
    return torch.cuda.Event(enable_timing=True)


def run_net(args):
    """The training step of a whole network (the dense SNN of Tab. I, its
    population-coded variant, or the convolutional SNN) as one CUDA graph."""
    import torch
    import torch.distributed as dist

    from paper_2211_10725_gb300 import snn

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = net_workload(args.workload)
    # the fastest parity-tested variant: every GEMM layer's forward fused
    # with its scan, every scan storing its bf16 trace for the BPTT
    save = args.save or "fused"
    from paper_2211_10725_gb300 import workloads as W
    inp = net_inputs(w, seed=W.SEED_BASE + w.seed_index + 1000 * rank)
    if is_conv(w):
        from paper_2211_10725_gb300.csnn import ConvSNN
        net = ConvSNN(w, inp["convs"], inp["Wfc"], device=dev, save=save)
        X = inp["X"].reshape(w.T * w.B, w.H, w.W, w.Cin).to(dev)
        scans = net.layers + [net.out_layer]
    else:
        from paper_2211_10725_gb300.dsnn import DenseSNN
        net = DenseSNN(w, inp["W"], device=dev, save=save)
        X = inp["X"].reshape(w.T * w.B, -1).to(dev)
        scans = net.layers
    labels = inp["labels"].to(dev)
    stream = torch.cuda.Stream(dev)
    if world > 1:
        # data parallel: this rank's samples are its shard of a global batch
        # of world * B; dW (and dbeta) and the loss are summed over the ranks
        # (NCCL) before the AdamW update
        from paper_2211_10725_gb300.data_parallel import allreduce_sum_
        net.batch_total = world * w.B
        from paper_2211_10725_gb300.data_parallel import grad_buffers
        grads = grad_buffers(net)

    # the weight-gradient products off the reverse pass's critical path run
    # on a second stream in the timed graph; the graph with timing events
    # between the ops keeps them in line so that each op's time is its own
    side = snn.SideStream(dev)

    def step_ops(st=None, sd=None):
        ops = net.ops(X, labels, st, sd)
        if world > 1:
            ops.insert(len(ops) - 1, ("allreduce_grads", lambda: allreduce_sum_(grads)))
        return ops

    names = [n for n, _ in step_ops()]

    c0 = snn.snn_kernel_launches()
    warm = max(1, args.warmup)
    with torch.cuda.stream(stream):
        for _ in range(warm):
            for _, call in step_ops(sd=side):
                call()
    stream.synchronize()
    launches = (snn.snn_kernel_launches() - c0) // warm
    for layer in scans:
        if layer.status() != 0:
            raise RuntimeError("kernel status after warm-up")

    # one step as a CUDA graph; a second graph of the same step has a timing
    # event between consecutive ops (event nodes), for the per-op times
    def capture(with_events):
        evs = [_timing_events(True) for _ in range(len(names) + 1)] if with_events else None
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if evs:
                evs[0].record()
            for i, (_, call) in enumerate(step_ops(sd=None if with_events else side)):
                call()
                if evs:
                    evs[i + 1].record()
        return g, evs

    graph = graph_ev = None
    evs = None
    if not args.no_graph and world == 1:
        graph, _ = capture(False)
        try:
            graph_ev, evs = capture(True)
        except TypeError:
            graph_ev, evs = None, None   # no graph-capturable timing events in this torch
    if graph_ev is None:
        evs = [_timing_events(False) for _ in range(len(names) + 1)]

    def launch(with_events):
        if graph is not None and not with_events:
            graph.replay()
        elif graph_ev is not None:
            graph_ev.replay()
        else:
            evs[0].record(stream)
            for i, (_, call) in enumerate(step_ops(stream)):
                call()
                evs[i + 1].record(stream)

    with torch.cuda.stream(stream):
        for _ in range(3):
            launch(False)
            launch(True)
    stream.synchronize()

    sampler = clock_sampler(local)
    if rank == 0:
        sampler.start()
        time.sleep(0.3)
    K = args.steps
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(K):
            launch(graph is None)
        e1.record(stream)
    torch.cuda.synchronize()
    t_wall1 = time.time()
    if world > 1:
        dist.barrier()
    # per-op durations: a timed region of the graph with event nodes (K2
    # steps), each op averaged over the steps
    K2 = max(1, min(K, 100))
    per_op = [0.0] * len(names)
    ev_total = 0.0
    with torch.cuda.stream(stream):
        for _ in range(K2):
            launch(True)
            torch.cuda.synchronize()
            per_op = [acc + evs[i].elapsed_time(evs[i + 1]) for i, acc in enumerate(per_op)]
            ev_total += evs[0].elapsed_time(evs[-1])
    per_op = [x / K2 for x in per_op]
    if rank == 0:
        time.sleep(0.2)
        sampler.stop()
    total_ms = e0.elapsed_time(e1)
    if world > 1:
        t = torch.tensor([total_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    for layer in scans:
        if layer.status() != 0:
            raise RuntimeError("kernel status in the timed region")
    loss = float(net.loss.item())
    if not (loss == loss):
        raise RuntimeError("loss is NaN")

    ns_per_step = w.T * w.B * net_neurons(w)
    ms = total_ms / K
    value = world * ns_per_step / (ms * 1e-3)
    e2e = None if args.no_e2e else run_net_e2e(args, w, inp, net, dev, world)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    fwd_f, dw_f, dx_f = net_flops(w)
    op_ms = dict(zip(names, per_op))
    clocks = sampler.summary(t_wall0, t_wall1)
    cpu = None
    if not args.no_cpu_baseline and world == 1:
        cpu = time_net_oracle(w, inp, args.cpu_seconds)
    if is_conv(w):
        # every op is memory-bound (the GEMMs' K is 32 or 400, N 16 or 64):
        # the HBM roofline of the op that takes longest
        ob = conv_op_bytes(net)
        top = max(ob, key=lambda k: op_ms.get(k, 0.0))
        peak, peak_kind = hbm_peak()
        achieved = ob[top] / (op_ms[top] * 1e-3) / 1e9
        roofline = {"bound": "hbm", "kernel": top, "achieved": achieved, "peak": peak,
                    "unit": "GB/s", "frac": achieved / peak, "peak_kind": peak_kind,
                    "traffic": None, "bytes_per_launch": ob[top],
                    "op_bytes": ob,
                    "op_gbs": {k: ob[k] / (op_ms[k] * 1e-3) / 1e9 for k in ob if op_ms.get(k)},
                    "flops_per_step": {"fwd": fwd_f, "dW": dw_f, "dX": dx_f}}
        step_desc = ("per conv layer im2col, tcgen05 GEMM, Leaky scan, 2x2 max pool; dense "
                     "readout GEMM + scan; rate-coded CE loss; BPTT (max-pool routing, scans "
                     "with per-channel dbeta, GEMM dX/dW, col2im); AdamW on weights and betas")
        l2 = "working set ~1.2 GB, larger than L2; no flush"
    else:
        fused = save == "fused"
        gemm_fwd_ms = sum(v for k, v in op_ms.items()
                          if k.startswith("dense_scan_fwd" if fused else "dense_fwd"))
        peak, peak_kind = tensor_peak(sustained=True)
        achieved = fwd_f / (gemm_fwd_ms * 1e-3) / 1e12
        kname = ("gemm_leaky_tcgen05 (forward GEMMs with the Leaky scan in the epilogue; the "
                 "scan's time counts against the GEMM)") if fused else "gemm_tn_tcgen05 (forward GEMMs)"
        roofline = {"bound": "tensor", "kernel": kname,
                    "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                    "frac": achieved / peak, "peak_kind": f"{peak_kind} sustained bf16",
                    "traffic": None, "flops_per_step": {"fwd": fwd_f, "dW": dw_f, "dX": dx_f}}
        step_desc = ("forward GEMMs + Leaky scans, rate-coded CE loss, BPTT scans, dense "
                     "backward (dX, dW), AdamW")
        if fused:
            step_desc = ("forward GEMMs with the Leaky scan in their epilogue, rate-coded CE "
                         "loss, the readout's BPTT scan, dW GEMMs, dX GEMMs with the lower "
                         "layer's BPTT scan in their epilogue, AdamW")
        l2 = "working set (~70 MB) fits in L2; no flush between steps"
    roofline.update({"op_ms": op_ms, "op_timed_step_ms": ev_total / K2,
                     "timing": "per-op: a second timed region of the same step graph with "
                               "event nodes between the ops (weight gradients in line, not "
                               "on the side stream), averaged over its steps"})
    cfg = net_config(w)
    cfg.update({"step": step_desc, "neuron_steps_per_step": ns_per_step, "save": save,
                "launch": ("CUDA graph replay, weight gradients on a second stream"
                           if graph is not None else "eager"), "l2": l2,
                "parallelism": (f"data parallel x{world} (global batch {world * w.B}, "
                                "gradients all-reduced over NCCL)") if world > 1
                else "single GPU"})
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": cfg,
        "images_per_s": world * w.B / (ms * 1e-3),
        "roofline": roofline,
        "clocks": clocks,
        # counted by the library over the eager warm-up steps
        "gpu_launches": launches * K,
        "gpu_launches_per_step": launches,
        "cpu_baseline": cpu,
        "e2e": e2e,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def time_net_oracle(w, inp, seconds):
    """The oracle's forward + loss + BPTT of the network on consecutive
    sample batches (at most the whole batch), repeated for about `seconds`,
    one chunk of each batch per host core (threads; samples are independent
    until the dW sums)."""
    import concurrent.futures
    import numpy as np
    host = net_oracle_host(w, inp)
    cores = os.cpu_count() or 1
    t0 = time.perf_counter()
    probe = min(w.B, 4)
    net_oracle_pass(w, host, np.arange(probe))
    per_sample = (time.perf_counter() - t0) / probe
    n = int(max(1, min(w.B, cores * seconds / 3 / per_sample)))
    done, t_total, start = 0, 0.0, 0
    with concurrent.futures.ThreadPoolExecutor(max_workers=cores) as pool:
        while t_total < seconds or done == 0:
            bs = np.sort((start + np.arange(n)) % w.B)
            chunks = [c for c in np.array_split(bs, min(cores, n)) if len(c)]
            t0 = time.perf_counter()
            list(pool.map(lambda c: net_oracle_pass(w, host, c), chunks))
            t_total += time.perf_counter() - t0
            done += n
            start = (start + n) % w.B
    ns = w.T * done * net_neurons(w)
    return {"value": ns / t_total, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{done} samples in batches of {n} (of {w.B}) on {cores} threads, all "
                      f"T={w.T} steps, oracle forward+loss+BPTT (no optimiser), {t_total:.1f} s, "
                      f"BLAS on one thread per host thread"}


def run_net_e2e(args, w, inp, net, dev, world):
    """Training steps through the public API with the batch copied from
    pinned host memory each step and the loss read back."""
    import torch
    import torch.distributed as dist
    shape = (w.T * w.B, w.H, w.W, w.Cin) if is_conv(w) else (w.T * w.B, -1)
    hX = inp["X"].reshape(shape).pin_memory()
    hy = inp["labels"].pin_memory()
    dX = torch.empty_like(hX, device=dev)
    dy = torch.empty_like(hy, device=dev)
    out = torch.empty(1, dtype=torch.float32).pin_memory()
    stream = torch.cuda.current_stream(dev)

    if world > 1 and not is_conv(w):
        from paper_2211_10725_gb300.data_parallel import DataParallelDenseSNN
        train = DataParallelDenseSNN(net, world * w.B).train_step
    elif world > 1:
        from paper_2211_10725_gb300.data_parallel import DataParallelConvSNN
        train = DataParallelConvSNN(net, world * w.B).train_step
    else:
        train = net.train_step

    def step():
        dX.copy_(hX, non_blocking=True)
        dy.copy_(hy, non_blocking=True)
        train(dX, dy)
        out.copy_(net.loss, non_blocking=True)

    K = max(3, min(args.steps, 200))
    for _ in range(3):
        step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    if world > 1:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    nb = lambda t: t.numel() * t.element_size()
    return {"value": world * w.T * w.B * net_neurons(w) * K / (ms * 1e-3), "unit": UNIT,
            "h2d_bytes_per_step": nb(hX) + nb(hy), "d2h_bytes_per_step": nb(out), "steps": K,
            "launch": "eager"}


def time_torch_eager(w, inp, dev, steps=2):
    """Context only: the same fwd + BPTT as a PyTorch-eager per-timestep loop
    with autograd on the same GPU (the shape of the paper's GPU path),
    written from Eqs. (3)-(7): fp32 state, the surrogate as a custom
    backward, the reset detached as the workload says.  Returns NS/s."""
    import math
    import torch

    fast = w.surrogate == "fast_sigmoid"
    k, a_half, b_arg = w.sg_param, 0.5 * w.sg_param, math.pi * 0.5 * w.sg_param

    class Spike(torch.autograd.Function):
        @staticmethod
        def forward(ctx, x):
            ctx.save_for_backward(x)
            return (x > 0).float()

        @staticmethod
        def backward(ctx, g):
            (x,) = ctx.saved_tensors
            if fast:
                return g / (1.0 + k * x.abs()) ** 2
            return g * a_half / (1.0 + (b_arg * x) ** 2)

    def lane(p, mode):
        t = p.to(dev).float()
        if mode == "per_channel":
            t = t.repeat_interleave(w.HW).repeat(w.N // (w.C * w.HW))
        return t.reshape(1, -1).expand(w.B, w.N)

    I = inp["I"].to(dev)
    gs = inp["grad_spk"].to(dev).float()

    def one():
        beta = lane(inp["beta"], w.beta_mode).clone().requires_grad_(True)
        thr = lane(inp["thr"], w.thr_mode).clone().requires_grad_(True)
        x = I.float().requires_grad_(True)
        third = None
        if w.neuron == "synaptic":
            third = lane(inp["alpha"], w.alpha_mode).clone().requires_grad_(True)
        elif w.neuron == "rleaky":
            third = lane(inp["v"], w.v_mode).clone().requires_grad_(True)
        u = torch.zeros(w.B, w.N, device=dev)
        i = torch.zeros_like(u)
        z = torch.zeros_like(u)
        loss = 0.0
        for t in range(w.T):
            zr = z.detach() if w.detach_reset else z
            inp_t = x[t]
            if w.neuron == "synaptic":
                i = third * i + x[t]
                inp_t = i
            if w.reset == "zero":
                u = beta * ((1 - zr) * u) + inp_t
            elif w.reset == "none":
                u = beta * u + inp_t
            else:
                u = beta * u + inp_t - zr * thr
            if w.neuron == "rleaky":
                u = u + z * third
            z = Spike.apply(u - thr)
            loss = loss + (z * gs[t]).sum()
        loss.backward()

    one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        one()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    return {"value": w.T * w.B * w.N / (ms * 1e-3), "unit": UNIT, "ms_per_step": ms,
            "steps": steps, "kind": "context",
            "note": "PyTorch eager per-timestep loop with autograd on the same GPU, fp32 "
                    "state; context for the paper's GPU path, not a baseline of this build"}


def link_bandwidth(dev, nbytes=1 << 30):
    """Pinned host <-> device copy rates of this machine (GB/s, best of 3):
    host to device, device to host, and both at once on two streams."""
    import torch
    h = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    h2 = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    d = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    d2 = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def timed(fn):
        best = None
        for _ in range(3):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            dt = time.perf_counter() - t0
            best = dt if best is None else min(best, dt)
        return best

    def both():
        with torch.cuda.stream(s1):
            d.copy_(h, non_blocking=True)
        with torch.cuda.stream(s2):
            h2.copy_(d2, non_blocking=True)

    t_h2d = timed(lambda: d.copy_(h, non_blocking=True))
    t_d2h = timed(lambda: h2.copy_(d2, non_blocking=True))
    t_bi = timed(both)
    del h, h2, d, d2
    return {"h2d_gbs": nbytes / t_h2d / 1e9, "d2h_gbs": nbytes / t_d2h / 1e9,
            "bidir_gbs": 2 * nbytes / t_bi / 1e9,
            "how": "1 GiB pinned copies, best of 3, each direction alone and both at once"}


def run_e2e(args, w, inp, layer, dev, world):
    """Same metric through the public API, with each step's inputs copied
    from pinned host memory and its results read back to pinned host memory.

    A training loop that streams batches from the host overlaps them: two
    sets of device buffers (and two ScanLayers) alternate, so the copy-in of
    step k+1 and the copy-out of step k-1 run on their own streams while
    step k computes.  Every step's copies are inside the timed region."""
    import torch
    import torch.distributed as dist
    from paper_2211_10725_gb300 import snn
    hI = inp["I"].pin_memory()
    hG = inp["grad_spk"].pin_memory()
    beta, thr = inp["beta"].to(dev), inp["thr"].to(dev)
    alpha = inp["alpha"].to(dev) if "alpha" in inp else None
    v = inp["v"].to(dev) if "v" in inp else None
    layers = [layer, snn.ScanLayer(w, device=dev)]
    dI = [torch.empty_like(hI, device=dev) for _ in range(2)]
    dG = [torch.empty_like(hG, device=dev) for _ in range(2)]
    outs = [{k: torch.empty_like(getattr(L, k), device="cpu").pin_memory()
             for k in ("spk", "grad_I", "grad_beta", "grad_thr")} for L in layers]
    s_in, s_comp, s_out = (torch.cuda.Stream(dev) for _ in range(3))
    ev = {name: [torch.cuda.Event() for _ in range(2)] for name in ("in", "comp", "out")}
    used = [False, False]

    def step(k):
        b = k % 2
        L = layers[b]
        with torch.cuda.stream(s_in):
            if used[b]:
                s_in.wait_event(ev["comp"][b])   # the previous use of these inputs is done
            dI[b].copy_(hI, non_blocking=True)
            dG[b].copy_(hG, non_blocking=True)
            ev["in"][b].record(s_in)
        with torch.cuda.stream(s_comp):
            s_comp.wait_event(ev["in"][b])
            if used[b]:
                s_comp.wait_event(ev["out"][b])  # the previous results have been read out
            L.forward(dI[b], beta, thr, alpha, v=v)
            L.backward(dI[b], beta, thr, dG[b], alpha=alpha, want_state_grads=False, v=v)
            ev["comp"][b].record(s_comp)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev["comp"][b])
            for name, host in outs[b].items():
                host.copy_(getattr(L, name), non_blocking=True)
            ev["out"][b].record(s_out)
        used[b] = True

    K = max(3, min(args.steps, 50))
    for k in range(4):
        step(k)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    s_in.wait_event(e0)
    for k in range(K):
        step(k)
    for s in (s_in, s_comp):
        s_out.wait_stream(s)
    e1.record(s_out)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    if world > 1:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    nb = lambda t: t.numel() * t.element_size()
    return {"value": world * w.T * w.B * w.N * K / (ms * 1e-3), "unit": UNIT,
            "h2d_bytes_per_step": nb(hI) + nb(hG),
            "d2h_bytes_per_step": sum(nb(t) for t in outs[0].values()),
            "steps": K, "overlap": "copy-in, compute and copy-out on three streams, two buffer sets"}


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif is_net(args):
        run_net(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
