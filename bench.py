"""Benchmark of the DARB hot path on the FC6/FC7 workload (AlexNet FC layers).

One step = BMWM re-encode of FC6 (4096x9216) and FC7 (4096x4096), bf16
weights, then darb_spmm of both at batch 1, 16, 64 and 256.  The reported value
is effective GB/s: the algorithmic bytes of every call in the step (dense W
read once by the encoder plus the encoded matrix written; for each product the
kept values, stored offsets, per-row metadata, X read once and Y written once)
over the device time of the step.  Inputs rotate over several sets of distinct
buffers whose total is well above the 129 MB L2, so every call reads cold HBM.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Under torchrun every rank runs its own copy of the workload (independent
problems, no data-path collective): weak scaling.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "fc6_fc7"
BATCHES = (1, 16, 64, 256)
METRIC = ("darb_spmm effective GB/s & % of HBM roofline at batch 1/16/64/256; encode GB/s")
NSETS = 4
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=("darb", "reference"), default="darb")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--no-rnn", action="store_true")
    p.add_argument("--no-baselines", action="store_true", help="skip the cuSPARSE comparison section")
    p.add_argument("--step-only", action="store_true",
                   help="time the step and its calls only (no tensor-core, gemv_1024, RNN, assignment or "
                        "baseline sections): the run whose launch list the profiles summarise")
    p.add_argument("--path", choices=("auto", "tensor"), default="auto",
                   help="kernel family of the products: darb_spmm (auto), or the opt-in tensor-core path "
                        "(darb_spmm_ex with DARB_PATH_TENSOR_CORES; for profiling it)")
    p.add_argument("--calls", default="",
                   help="comma list restricting the step to some calls, e.g. fc6_spmm_b256 (profiling)")
    return p.parse_args()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def measured_bf16_tflops():
    """Dense bf16 tensor peak (burst: a kernel timed alone), measured or fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_BF16_TFLOPS, "fallback"


# The CUDA sources each profiled call's kernels are built from (the shared
# headers included): a summary stays valid while these files are unchanged.
_COMMON_SOURCES = ("darb_internal.h", "launch.cuh", "tma.cuh", "spmm.cu")
_CALL_SOURCES = {
    "encode": ("encode.cu",),
    "b1": ("gemv.cuh", "kernels_common.cuh"),
    "b16": ("batch.cuh", "kernels_common.cuh", "rnn_epilogue.cuh", "spmm_batch.cu", "xres.cuh"),
    "xres": ("xres.cuh", "kernels_common.cuh", "spmm_batch.cu", "batch.cuh", "rnn_epilogue.cuh"),
    "tc": ("tc.cuh", "tcgen05.cuh", "spmm_tc.cu"),
}


def call_sources(call: str):
    """The csrc files the kernels of a bench call (e.g. fc6_spmm_b256, or
    fc6_tc_b256 for the opt-in tensor-core path) come from."""
    if call.endswith("_encode"):
        kind = "encode"
    elif "_tc_b" in call:
        kind = "tc"
    else:
        b = int(call.rsplit("_b", 1)[1])
        kind = "b1" if b == 1 else ("b16" if b <= 16 else "xres")
    return tuple(sorted(_COMMON_SOURCES + _CALL_SOURCES[kind]))


def library_source_hash(call: str) -> str:
    """sha1 over the CUDA sources of a call's kernels: identifies the kernels a profile was taken on."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_1911_08020_gb300", "csrc")
    h = hashlib.sha1()
    for name in call_sources(call):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:12]


def profiled_traffic(call: str):
    """DRAM bytes per launch of `call` from the committed ncu summaries under
    profiles/ (lines 'traffic: <call> <bytes> src=<hash>'), or None when no
    summary was taken on the current sources of the call's kernels."""
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir):
        return None
    want = library_source_hash(call)
    for name in sorted(os.listdir(pdir)):
        if not name.endswith((".md", ".txt")):
            continue
        with open(os.path.join(pdir, name)) as f:
            for ln in f:
                parts = ln.strip().strip("`").split()
                if len(parts) == 4 and parts[0] == "traffic:" and parts[1] == call and parts[3] == f"src={want}":
                    return int(parts[2])
    return None


def capture(torch, fn):
    """Record fn's launches (made on the current stream) into a CUDA graph."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side):
            fn()
    torch.cuda.current_stream().wait_stream(side)
    return g


def call_name(kind, mi, b):
    return ("fc6" if mi == 0 else "fc7") + ("_encode" if kind == "encode" else f"_spmm_b{b}")


# ----------------------------------------------------------------------------- clocks
def pci_bus_id(torch, device: int):
    """domain:bus:device.0 of a CUDA device (hex), or None where torch does not report it."""
    p = torch.cuda.get_device_properties(device)
    try:
        return f"{p.pci_domain_id:x}:{p.pci_bus_id:x}:{p.pci_device_id:x}.0"
    except AttributeError:
        return None


class NvmlPoller:
    """SM clock and clock-event reasons read through NVML (the driver's
    libnvidia-ml, read-only queries) every ~0.5 ms from a thread while the
    timed region runs: a region of a few milliseconds is far shorter than
    nvidia-smi's sampling period.  Inert where NVML is missing."""
    CLOCK_SM = 1
    # clock-event reason bits of NVML's public header
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown"}

    def __init__(self, index: int, pci: str | None = None):
        import ctypes
        self.c = ctypes
        self.samples = []
        self.lib = self.dev = None
        self.max_mhz = None
        self.stop = threading.Event()
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            dev = ctypes.c_void_p()
            # the GPU CUDA runs on, by PCI address (CUDA and NVML may number devices differently)
            found = pci is not None and lib.nvmlDeviceGetHandleByPciBusId_v2(pci.encode(), ctypes.byref(dev)) == 0
            if not found and lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(index), ctypes.byref(dev)) != 0:
                lib.nvmlShutdown()
                return
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(dev, ctypes.c_int(self.CLOCK_SM), ctypes.byref(mx)) == 0:
                self.max_mhz = float(mx.value)
            self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons", None)
            self.lib, self.dev = lib, dev
        except (OSError, AttributeError):
            self.lib = None

    def _poll(self):
        c = self.c
        clk, rs = c.c_uint(), c.c_ulonglong()
        while not self.stop.is_set():
            if self.lib.nvmlDeviceGetClockInfo(self.dev, c.c_int(self.CLOCK_SM), c.byref(clk)) == 0:
                mask = rs.value if (self.reasons_fn is not None and self.reasons_fn(self.dev, c.byref(rs)) == 0) else 0
                self.samples.append((float(clk.value), int(mask)))
            time.sleep(0.0005)

    def __enter__(self):
        if self.lib is not None:
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()
        return self

    def __exit__(self, *exc):
        if self.lib is not None:
            self.stop.set()
            self.thread.join(timeout=5)
            self.lib.nvmlShutdown()

    def summary(self):
        if not self.samples:
            return None
        reasons = sorted({name for _, m in self.samples for bit, name in self.REASONS.items() if m & bit})
        return {"sm_mhz": statistics.median(v for v, _ in self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(self.samples), "source": "nvml, during the timed region"}


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons around the timed region
    (used when NVML cannot be read; a short region may see none of its own)."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index   # an nvidia-smi -i argument: index or PCI bus id
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
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
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "source": "nvidia-smi, around the timed region"}


# ----------------------------------------------------------------------------- distributed
def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(value: float, world: int) -> float:
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------- bytes
def spmm_bytes(info, batch):
    return (info["value_bytes"] + info["offset_bytes"] + info["meta_bytes"]
            + info["cols"] * batch * 4 + info["rows"] * batch * 4)


def encode_bytes(info):
    esz = 2 if info["wtype"] == 1 else 4
    return info["rows"] * info["cols"] * esz + info["value_bytes"] + info["offset_bytes"] + info["meta_bytes"]


def tensor_flops(mat, batch):
    """FLOPs of the densified product on the tensor cores: rows x cols x batch
    multiply-adds for each of the two bf16 parts of X."""
    return 2.0 * 2.0 * mat["rows"] * mat["cols"] * batch


def roofline(wl, di, dom, dom_ms, achieved, peak, peak_kind, tpeak, tpeak_kind, traffic, step_ms_sum,
             gather_peak):
    """Roofline of the dominant call against HBM: algorithmic bytes (kept values
    + offsets + row metadata + X + Y, or dense W + encoding) over the mean call
    time.  For a call on the tensor cores the work that binds it -- the
    densified product they execute, zeros and both bf16 parts of X included --
    is reported beside it, not as achieved work."""
    kind, mi, b, nbytes = wl.calls[di]
    share = round(dom_ms / step_ms_sum, 3) if step_ms_sum > 0 else None
    if wl.paths[di][0] == "tensor":
        tfl = tensor_flops(wl.mats[mi], b) / (dom_ms * 1e-3) / 1e12
        nnzb = wl.mats[mi]["info"]["nnzb"]
        return {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1),
                "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / peak, 4),
                "frac_of_nominal_8000": round(achieved / 8000.0, 4), "share_of_step": share,
                "traffic": traffic,
                "binding": "tensor pipe: the densified product of the tensor-core path",
                "tensor_executed": {"tflops": round(tfl, 1), "peak": tpeak, "peak_kind": tpeak_kind,
                                    "frac": round(tfl / tpeak, 4),
                                    "flops_per_call": tensor_flops(wl.mats[mi], b),
                                    "algorithmic_flops_per_call": 2 * nnzb * b},
                "gather_equiv_frac": round(nnzb * b * 4 / (dom_ms * 1e-3) / 1e9 / gather_peak, 4),
                "note": "achieved = algorithmic bytes per call (values + offsets + row metadata + X read once"
                        " + Y written once) / mean call time (the split of X and the product kernel),"
                        " against the measured HBM copy peak. The call runs on the tensor cores, which"
                        " execute 2 x 2 x rows x cols x batch FLOPs of densified tiles (tensor_executed:"
                        " not algorithmic work); that work, not HBM, binds it. gather_equiv_frac = the"
                        " (kept weight, column) operands per second against the CUDA-core gather bound"
                        " of 128 B/clk/SM"}
    out = {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1),
           "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / peak, 4),
           "frac_of_nominal_8000": round(achieved / 8000.0, 4), "share_of_step": share,
           "traffic": traffic,
           "note": "achieved = algorithmic bytes per launch (values + offsets + row metadata + X + Y,"
                   " or dense W + encoding for encode) / median launch time; for batch > 4 the"
                   " on-chip activation gather, not HBM, binds: gather_frac"}
    if kind == "spmm" and b > 4:
        nnzb = wl.mats[mi]["info"]["nnzb"]
        out["gather_frac"] = round(nnzb * b * 4 / (dom_ms * 1e-3) / 1e9 / gather_peak, 4)
        out["gather_peak_gbs"] = round(gather_peak, 1)
        out["binding"] = ("on-chip activation gather: every (kept weight, batch column) product reads a 4-byte "
                          "activation from shared memory, at most 128 B/clk/SM")
    return out


# ----------------------------------------------------------------------------- GPU arm
class Workload:
    """Rotating sets of device buffers for the FC6/FC7 step."""

    def __init__(self, torch, darb, synth, only=(), path="auto"):
        self.torch, self.darb = torch, darb
        self.tensor = path == "tensor"
        wl = synth.WORKLOADS[WORKLOAD]
        dev = torch.device("cuda", torch.cuda.current_device())
        self.dev = dev
        self.mats = []
        for i, (rows, cols) in enumerate(wl.shapes):
            _, bits, m = synth.matrix(wl, i)
            W = torch.from_numpy(bits.view(np.int16)).to(dev).view(torch.bfloat16)
            h = darb.darb_encode(W, m)
            exp = darb.darb_export(h)
            info = darb.darb_info(h)
            self.mats.append(dict(rows=rows, cols=cols, m=m, W=W, h=h, exp=exp, info=info,
                                  bits=bits))
        self.sets = []
        for s in range(NSETS):
            st = {"W": [], "enc": [], "spmm": {}, "X": {}, "Y": {}}
            for mi, mat in enumerate(self.mats):
                st["W"].append(mat["W"].clone())
                val, off, _, m = mat["exp"]
                st["enc"].append(darb.darb_import(val, off, m, darb.BF16, mat["rows"], mat["cols"]))
                for b in BATCHES:
                    st["spmm"][(mi, b)] = darb.darb_import(val, off, m, darb.BF16, mat["rows"], mat["cols"])
                    X = torch.from_numpy(synth.activations(mat["cols"], b, seed=wl.seed, sub=10 * s + b)).to(dev)
                    st["X"][(mi, b)] = X
                    st["Y"][(mi, b)] = torch.empty((mat["rows"], b), device=dev)
            self.sets.append(st)
        torch.cuda.synchronize()
        # the calls of one step, with their algorithmic bytes
        self.calls = []
        for mi, mat in enumerate(self.mats):
            self.calls.append(("encode", mi, None, encode_bytes(mat["info"])))
        for b in BATCHES:
            for mi, mat in enumerate(self.mats):
                self.calls.append(("spmm", mi, b, spmm_bytes(mat["info"], b)))
        if only:
            self.calls = [c for c in self.calls if call_name(*c[:3]) in only]
        self.step_bytes = sum(c[3] for c in self.calls)
        # kernel family and launches of each call, as the library reports them
        self.paths = []
        for kind, mi, b, _ in self.calls:
            if kind == "encode":
                self.paths.append(("encode", 1))
            elif self.tensor:
                self.paths.append(("tensor", 2))   # split_kernel + tc_kernel
            else:
                path, kernels = darb.darb_spmm_path(self.mats[mi]["h"], b)
                self.paths.append(("tensor" if path == darb.PATH_TENSOR_CORES else "cuda", kernels))
        self.step_launches = sum(k for _, k in self.paths)

    def launch(self, call, s, stream):
        kind, mi, b, _ = call
        st = self.sets[s % NSETS]
        if kind == "encode":
            self.darb.darb_reencode(st["enc"][mi], st["W"][mi], stream)
        elif self.tensor:
            self.darb.darb_spmm_ex(st["spmm"][(mi, b)], st["X"][(mi, b)], st["Y"][(mi, b)],
                                   self.darb.PATH_TENSOR_CORES, stream)
        else:
            self.darb.darb_spmm(st["spmm"][(mi, b)], st["X"][(mi, b)], st["Y"][(mi, b)], stream)

    def check_encode(self):
        for st in self.sets:
            for h in st["enc"]:
                self.darb.darb_sync_status(h)
            for h in st["spmm"].values():
                self.darb.darb_sync_status(h)

    def close(self):
        for st in self.sets:
            for h in st["enc"]:
                self.darb.darb_destroy(h)
            for h in st["spmm"].values():
                self.darb.darb_destroy(h)
        for mat in self.mats:
            self.darb.darb_destroy(mat["h"])


def run_gpu(args, world, rank, local):
    import torch

    from paper_1911_08020_gb300 import darb, synth
    torch.cuda.set_device(local)
    only = tuple(c for c in args.calls.split(",") if c)
    wl = Workload(torch, darb, synth, only, args.path)
    stream = torch.cuda.current_stream()
    sid = stream.cuda_stream
    ncalls = len(wl.calls)

    # eager warm-up: first launches set kernel attributes and fill caches
    for s in range(max(1, min(args.warmup, NSETS))):
        for c in wl.calls:
            wl.launch(c, s, sid)
    torch.cuda.synchronize()
    wl.check_encode()

    # One CUDA graph per buffer set holds a whole step (the launches and their
    # PDL edges), so host-side launch cost is out of the measured device time.
    step_graphs = [capture(torch, lambda s=s: [wl.launch(c, s, None) for c in wl.calls]) for s in range(NSETS)]
    for s in range(args.warmup):
        step_graphs[s % NSETS].replay()
    torch.cuda.synchronize()
    wl.check_encode()

    # timed region: K steps back to back, rotating the buffer sets
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    pci = pci_bus_id(torch, local)
    with ClockSampler(pci or local) as clk:
        with NvmlPoller(local, pci) as nv:
            start.record(stream)
            for s in range(args.steps):
                step_graphs[s % NSETS].replay()
            end.record(stream)
            torch.cuda.synchronize()
    barrier(world)
    elapsed_ms = start.elapsed_time(end)
    wl.check_encode()
    elapsed_ms = max_over_ranks(elapsed_ms, world)
    ms_per_step = elapsed_ms / args.steps

    # the same step without programmatic dependent launch: every kernel starts
    # only when the previous one has finished
    darb.darb_set_pdl(False)
    try:
        graphs_off = [capture(torch, lambda s=s: [wl.launch(c, s, None) for c in wl.calls]) for s in range(NSETS)]
        for s in range(args.warmup):
            graphs_off[s % NSETS].replay()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record(stream)
        for s in range(args.steps):
            graphs_off[s % NSETS].replay()
        b.record(stream)
        torch.cuda.synchronize()
        ms_pdl_off = a.elapsed_time(b) / args.steps
    finally:
        darb.darb_set_pdl(True)
    wl.check_encode()

    # per-call breakdown: each call of the step launched back to back over the
    # rotating buffer sets (still cold in L2), from a graph replayed REPEATS
    # times with events around each replay: median (and mean) per call
    per_call = np.zeros(ncalls)
    per_call_mean = np.zeros(ncalls)
    reps = max(1, args.steps // NSETS)
    for i, c in enumerate(wl.calls):
        g = capture(torch, lambda c=c: [wl.launch(c, s, None) for _ in range(reps) for s in range(NSETS)])
        per_call[i], per_call_mean[i] = replay_times(torch, g, stream, reps * NSETS)
    wl.check_encode()
    peak, peak_kind = measured_peaks()
    clocks = nv.summary() or clk.summary()
    sm_mhz = (clocks or {}).get("sm_mhz") or 2070.0
    nsm = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    # on-chip gather bound: every (kept weight, batch column) product reads its
    # 4-byte activation from shared memory, at most 128 bytes/clock/SM
    gather_peak = 128.0 * nsm * sm_mhz * 1e6 / 1e9   # GB/s
    tpeak, tpeak_kind = measured_bf16_tflops()
    parts = []
    for i, (kind, mi, b, nbytes) in enumerate(wl.calls):
        name = call_name(kind, mi, b)
        sec = per_call[i] * 1e-3
        gbs = nbytes / sec / 1e9
        path, kernels = wl.paths[i]
        part = {"call": name, "path": path, "kernels": kernels, "bytes": int(nbytes),
                "us": round(per_call[i] * 1e3, 3), "us_mean": round(per_call_mean[i] * 1e3, 3),
                "gbs": round(gbs, 1), "hbm_frac": round(gbs / peak, 4)}
        if kind == "spmm":
            nnzb = wl.mats[mi]["info"]["nnzb"]
            part["gflops"] = round(2 * nnzb * b / sec / 1e9, 1)
            if path == "tensor":
                # the densified product the tensor cores execute (not algorithmic
                # work): rows x cols x batch, twice (x = hi + lo)
                tfl = tensor_flops(wl.mats[mi], b) / sec / 1e12
                part["executed_tensor_tflops"] = round(tfl, 1)
                part["executed_tensor_frac"] = round(tfl / tpeak, 4)
            if b > 4:
                part["gather_frac"] = round(nnzb * b * 4 / sec / 1e9 / gather_peak, 4)
        parts.append(part)
    # dominant kernel: the single call with the largest share of the step
    di = int(np.argmax(per_call))
    dom = parts[di]["call"]
    dom_ms = float(per_call[di])
    achieved = wl.calls[di][3] / (dom_ms * 1e-3) / 1e9
    traffic = profiled_traffic(dom)
    step_ms_sum = float(per_call.sum())
    value = world * wl.step_bytes / (ms_per_step * 1e-3) / 1e9

    result = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": "fc6_fc7_4096x9216_4096x4096_bf16_weights",
                   "batches": list(BATCHES), "calls_per_step": ncalls,
                   "weights": "bf16 kept values, fp32 accumulate; X and Y fp32",
                   "block_sizes": "per row from {16,32,64} w.p. (.4,.3,.3)",
                   "pruning_ratio": [round(m["rows"] * m["cols"] / m["info"]["nnzb"], 2) for m in wl.mats],
                   "l2": f"inputs rotate over {NSETS} buffer sets (>4x L2), every call reads cold HBM",
                   "parallelism": f"replicas{world}"},
        "roofline": roofline(wl, di, dom, dom_ms, achieved, peak, peak_kind, tpeak, tpeak_kind, traffic,
                             step_ms_sum, gather_peak),
        "gather_peak_gbs": round(gather_peak, 1),
        "parts": parts,
        "parts_note": f"per call: {reps * NSETS} launches of that call alone, back to back on rotating cold"
                      f" buffers, from a CUDA graph replayed {REPEATS} times: us = median over the replays,"
                      " us_mean = their mean",
        "pdl_off": {"ms_per_step": round(ms_pdl_off, 5),
                    "value": round(world * wl.step_bytes / (ms_pdl_off * 1e-3) / 1e9, 2), "unit": "GB/s",
                    "note": "the same step captured with programmatic dependent launch off (darb_set_pdl)"},
        "timing": "CUDA-graph replay of whole steps (one graph per buffer set); CUDA events on the stream",
        "gpu_launches": wl.step_launches * args.steps,
        "clocks": clocks,
    }
    extras = not only and not args.step_only
    if extras:
        result["tensor_cores"] = run_tensor(torch, darb, wl, stream)
        result["gemv_1024"] = run_gemv_1024(torch, darb, synth, peak, stream)
    if not args.no_rnn and extras:
        result["rnn"] = run_rnn(torch, darb, synth, peak)
        result["assign"] = run_assign(torch, darb, wl, peak)
    if not args.no_baselines and extras:
        result["baselines"] = run_baselines(torch, darb, wl)
    if not args.no_e2e:
        result["e2e"] = run_e2e(args, wl, torch, darb)
    wl.close()
    return result


REPEATS = 10   # replays of a per-call graph, for the median


def replay_times(torch, g, stream, calls, repeats=REPEATS):
    """Median and mean time per call (ms) of a graph holding `calls` launches,
    replayed `repeats` times after one warm-up replay, CUDA events around each."""
    g.replay()
    times = []
    for _ in range(repeats):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        times.append(a.elapsed_time(b) / calls)
    return statistics.median(times), statistics.mean(times)


def run_tensor(torch, darb, wl, stream):
    """The opt-in tensor-core path (darb_spmm_ex with DARB_PATH_TENSOR_CORES;
    not darb_spmm, not the paper's per-block selection: densified tiles, X split
    into two bf16 parts) on the step's wide products, timed like `parts`."""
    out = {}
    tpeak, tpeak_kind = measured_bf16_tflops()
    for mi, mat in enumerate(wl.mats):
        for b in (64, 256):
            def launch(b=b, mi=mi):
                for s in range(NSETS):
                    st = wl.sets[s]
                    darb.darb_spmm_ex(st["spmm"][(mi, b)], st["X"][(mi, b)], st["Y"][(mi, b)],
                                      darb.PATH_TENSOR_CORES)
            launch()
            torch.cuda.synchronize()
            g = capture(torch, launch)
            med, mean = replay_times(torch, g, stream, NSETS)
            nbytes = spmm_bytes(mat["info"], b)
            tfl = tensor_flops(mat, b) / (med * 1e-3) / 1e12
            out[f"{'fc6' if mi == 0 else 'fc7'}_tc_b{b}"] = {
                "us": round(med * 1e3, 3), "us_mean": round(mean * 1e3, 3),
                "gbs_algorithmic": round(nbytes / (med * 1e-3) / 1e9, 1),
                "executed_tensor_tflops": round(tfl, 1), "executed_tensor_frac": round(tfl / tpeak, 4),
                "tensor_peak_kind": tpeak_kind}
    wl.check_encode()
    out["note"] = ("opt-in densified-tile product on the tensor cores (darb_spmm_ex, DARB_PATH_TENSOR_CORES): "
                   "executed FLOPs = 2 x 2 x rows x cols x batch (zeros and both bf16 parts of X), not "
                   "algorithmic work; darb_spmm itself never takes this path")
    return out


def run_gemv_1024(torch, darb, synth, peak, stream, nsets=48):
    """Workload gemv_1024 (a 1024 x 1024 fp32 matrix, per-row block sizes from
    {8, 16, 32, 64}): DARB encode, then the product at batch 1.  The dense
    matrices (4 MiB each) rotate over `nsets` sets (> L2), so every call reads
    cold HBM; per call: median over replays, as `parts`."""
    wl1 = synth.WORKLOADS["gemv_1024"]
    rows, cols = wl1.shapes[0]
    dev = torch.device("cuda", torch.cuda.current_device())
    _, stored, m = synth.matrix(wl1, 0)
    W0 = torch.from_numpy(stored).to(dev)
    h0 = darb.darb_encode(W0, m)
    info = darb.darb_info(h0)
    val, off, _, mm = darb.darb_export(h0)
    Ws = [W0.clone() for _ in range(nsets)]
    hs = [darb.darb_import(val, off, mm, darb.F32, rows, cols) for _ in range(nsets)]
    Xs = [torch.from_numpy(synth.activations(cols, 1, seed=wl1.seed, sub=s)).to(dev) for s in range(nsets)]
    Ys = [torch.empty((rows, 1), device=dev) for _ in range(nsets)]
    enc_b, spmm_b = encode_bytes(info), spmm_bytes(info, 1)
    out = {"rows": rows, "cols": cols, "dtype": "f32", "nnzb": info["nnzb"],
           "pruning_ratio": round(rows * cols / info["nnzb"], 2)}
    calls = {"encode": lambda s: darb.darb_reencode(hs[s], Ws[s]),
             "spmm_b1": lambda s: darb.darb_spmm(hs[s], Xs[s], Ys[s]),
             "step": lambda s: (darb.darb_reencode(hs[s], Ws[s]), darb.darb_spmm(hs[s], Xs[s], Ys[s]))}
    for name, fn in calls.items():
        for s in range(nsets):
            fn(s)
        torch.cuda.synchronize()
        g = capture(torch, lambda fn=fn: [fn(s) for s in range(nsets)])
        med, mean = replay_times(torch, g, stream, nsets)
        nbytes = {"encode": enc_b, "spmm_b1": spmm_b, "step": enc_b + spmm_b}[name]
        gbs = nbytes / (med * 1e-3) / 1e9
        out[name] = {"us": round(med * 1e3, 3), "us_mean": round(mean * 1e3, 3), "bytes": int(nbytes),
                     "gbs": round(gbs, 1), "hbm_frac": round(gbs / peak, 4)}
    for h in hs:
        darb.darb_sync_status(h)
        darb.darb_destroy(h)
    darb.darb_destroy(h0)
    return out


def run_assign(torch, darb, wl, peak, reps=3):
    """Block sizes from the weights (the step before encoding): a 4% top-K
    magnitude mask of FC6 and FC7, timed with CUDA events around the call (it
    synchronises).  Bytes: the radix passes and the counting pass each read W."""
    out = {}
    for mi, mat in enumerate(wl.mats):
        W = mat["W"]
        keep = mat["rows"] * mat["cols"] // 25
        darb.darb_assign_from_weights(W, keep)          # warm-up
        best = None
        for _ in range(reps):
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            darb.darb_assign_from_weights(W, keep)
            b.record()
            torch.cuda.synchronize()
            ms = a.elapsed_time(b)
            best = ms if best is None else min(best, ms)
        passes = 3   # bf16: two radix passes and the count
        nbytes = passes * mat["rows"] * mat["cols"] * 2
        out["fc6" if mi == 0 else "fc7"] = {"keep_fraction": 0.04, "us": round(best * 1e3, 1),
                                            "gbs": round(nbytes / (best * 1e-3) / 1e9, 1),
                                            "hbm_frac": round(nbytes / (best * 1e-3) / 1e9 / peak, 4),
                                            "note": "three reads of W (two radix passes and the row count)"
                                                    " plus the host rounding rule and the copies"}
    return out


def run_baselines(torch, darb, wl, reps=20):
    """darb_spmm next to cuSPARSE on the formats the paper compares with
    (Sec. 4.2): the same kept weights as CSR, and 4x4 / 8x8 block pruning of
    the same W at the same density as BSR (fp32 values, fp32 X and Y for the
    vendor library).  Each product is timed alone: `reps` calls captured in a
    CUDA graph and replayed, CUDA events around the replay; the matrices stay
    L2-resident across the calls for every format alike."""
    from paper_1911_08020_gb300 import baselines
    dev = wl.dev

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        try:
            g = capture(torch, lambda: [fn() for _ in range(reps)])
            run = g.replay
        except RuntimeError:   # not capturable: launched eagerly instead
            run = lambda: [fn() for _ in range(reps)]
        run()
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        run()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) * 1e3 / reps   # us per call

    out = {}
    for mi, mat in enumerate(wl.mats):
        name = "fc6" if mi == 0 else "fc7"
        rows, cols, nnzb = mat["rows"], mat["cols"], mat["info"]["nnzb"]
        rp, ci, vv = baselines.csr_from_darb(mat["h"])
        csr = [torch.from_numpy(a).to(dev) for a in (rp, ci, vv)]
        Wf = (mat["bits"].astype(np.uint32) << 16).view(np.float32)
        bsr = {}
        for bs in (4, 8):
            brp, bci, bvals, _ = baselines.block_prune(Wf, bs, round(nnzb / (bs * bs)))
            bsr[bs] = [torch.from_numpy(a).to(dev) for a in (brp, bci, bvals.reshape(-1))]
        entry = {"rows": rows, "cols": cols, "kept_weights": {"darb": nnzb, "csr": int(len(vv)),
                 "bsr4": int(bsr[4][1].numel() * 16), "bsr8": int(bsr[8][1].numel() * 64)}}
        for B in BATCHES:
            X = torch.randn((cols, B), device=dev)
            Y = torch.empty((rows, B), device=dev)
            XT = X.t().contiguous()                       # the same X, each batch column contiguous
            YT = torch.empty((B, rows), device=dev)
            t_darb = timed(lambda: darb.darb_spmm(mat["h"], X, Y))
            row = {"darb_us": round(t_darb, 2)}
            # each vendor product in the dense layout it runs fastest in (the layout change is not timed)
            for fmt, call in [("csr", lambda Xd, Yd, lay: baselines.csr_spmm(*csr, rows, cols, Xd, Yd, lay))] + \
                             [(f"bsr{bs}", (lambda bs_: lambda Xd, Yd, lay: baselines.bsr_spmm(
                                 *bsr[bs_], rows, cols, bs_, Xd, Yd, lay))(bs)) for bs in (4, 8)]:
                t_rows = timed(lambda: call(X, Y, baselines.DENSE_ROWS))
                t_cols = timed(lambda: call(XT, YT, baselines.DENSE_COLS))
                row[f"{fmt}_us"] = round(min(t_rows, t_cols), 2)
                row[f"{fmt}_layout"] = "rows" if t_rows <= t_cols else "cols"
            entry[f"b{B}"] = row
        out[name] = entry
    out["note"] = ("vendor-library figures, not a tuned block-sparse or CSR kernel and not the paper's "
                   "Sec. 4.2 comparison: cuSPARSE SpMM with fp32 values (DARB: bf16 values, so the bytes "
                   "differ), in the faster of the two dense layouts (batch contiguous, or each batch column "
                   "contiguous; the transposition is not timed); CSR = DARB's kept weights; BSR = the "
                   "largest-L1 bs x bs blocks of the same W at the same kept-weight count; every matrix "
                   "L2-resident")
    return out


def run_rnn(torch, darb, synth, peak, reps=3):
    """The fused RNN steps on their workloads: whole sequences, device-timed.

    The gate matrices (at most ~3 MB encoded) stay in L2 from one step to the
    next, so the per-step GB/s here are L2-served, not HBM."""
    dev = torch.device("cuda", torch.cuda.current_device())
    out = {}

    def seq_time(run, graph):
        """Median device time of one whole sequence: replayed from a CUDA graph,
        or launched eagerly from Python (host launch cost included)."""
        run()
        torch.cuda.synchronize()
        g = capture(torch, run) if graph else None
        times = []
        for _ in range(reps):
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            if g is not None:
                g.replay()
            else:
                run()
            b.record()
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b))
        return statistics.median(times)

    def dev_matrix(wl, i):
        _, stored, m = synth.matrix(wl, i)
        if wl.dtype == "bf16":
            W = torch.from_numpy(stored.view(np.int16)).to(dev).view(torch.bfloat16)
        else:
            W = torch.from_numpy(stored).to(dev)
        h = darb.darb_encode(W, m)
        return h, darb.darb_info(h)

    def step_bytes(info, I, H, B, cell):
        io = (I + H) * B * 4 + (2 if cell == "lstm" else 1) * H * B * 4   # inputs + outputs
        io += H * B * 4 if cell == "lstm" else 0                           # c_prev
        bias = info["rows"] * 4 * (1 if cell == "lstm" else 2)
        return info["value_bytes"] + info["offset_bytes"] + info["meta_bytes"] + io + bias

    for name in ("lstm_1024", "lstm_lm_1500", "gru_1024"):
        wl = synth.WORKLOADS[name]
        I, H = wl.input_size, wl.hidden
        hs = [dev_matrix(wl, i) for i in range(wl.layers)]
        for B in wl.batches:
            xs = torch.from_numpy(np.ascontiguousarray(synth.rnn_inputs(wl, B, wl.steps))).to(dev)
            hbuf = [torch.zeros((wl.layers, H, B), device=dev) for _ in range(2)]
            cbuf = [torch.zeros((wl.layers, H, B), device=dev) for _ in range(2)]
            bias = [torch.from_numpy(synth.bias(h[1]["rows"], seed=wl.seed + li)).to(dev) for li, h in enumerate(hs)]
            bias2 = [torch.from_numpy(synth.bias(h[1]["rows"], seed=wl.seed + 7 + li)).to(dev) for li, h in enumerate(hs)]
            for h, _ in hs:
                darb.darb_rnn_reserve(h, B)

            def run():
                for t in range(wl.steps):
                    src, dst = t % 2, (t + 1) % 2
                    inp = xs[t]
                    for li, (h, _) in enumerate(hs):
                        if wl.kind == "lstm":
                            darb.darb_lstm_step(h, I, H, B, inp, hbuf[src][li], cbuf[src][li], bias[li],
                                                hbuf[dst][li], cbuf[dst][li])
                        else:
                            darb.darb_gru_step(h, I, H, B, inp, hbuf[src][li], bias[li], bias2[li],
                                               hbuf[dst][li])
                        inp = hbuf[dst][li]

            ms = seq_time(run, graph=True)
            ms_eager = seq_time(run, graph=False)

            # the same layers, each as one persistent launch over all its steps
            hseq = [torch.empty((wl.steps, H, B), device=dev) for _ in hs]
            clast = [torch.empty((H, B), device=dev) for _ in hs]
            zero = torch.zeros((H, B), device=dev)

            def run_seq():
                inp = xs
                for li, (h, _) in enumerate(hs):
                    if wl.kind == "lstm":
                        darb.darb_lstm_sequence(h, wl.steps, I, H, B, inp, zero, zero, bias[li], hseq[li],
                                                None, clast[li])
                    else:
                        darb.darb_gru_sequence(h, wl.steps, I, H, B, inp, zero, bias[li], bias2[li], hseq[li])
                    inp = hseq[li]

            try:
                ms_seq = seq_time(run_seq, graph=False)
            except darb.DarbError as e:
                ms_seq = None
                seq_note = str(e)
            nsteps = wl.steps * wl.layers
            us = ms * 1e3 / nsteps
            nbytes = sum(step_bytes(info, I, H, B, wl.kind) for _, info in hs) / wl.layers
            out[f"{name}_b{B}"] = {"cell": wl.kind, "layers": wl.layers, "timesteps": wl.steps, "batch": B,
                                   "us_per_cell_step": round(us, 2), "gbs_l2_served": round(nbytes / (us * 1e-6) / 1e9, 1),
                                   "gflops": round(2 * sum(i["nnzb"] for _, i in hs) / wl.layers * B / (us * 1e-6) / 1e9, 1),
                                   "sequence_ms": round(ms, 3),
                                   "us_per_cell_step_eager": round(ms_eager * 1e3 / nsteps, 2),
                                   "us_per_cell_step_persistent": (round(ms_seq * 1e3 / nsteps, 2)
                                                                   if ms_seq is not None else seq_note),
                                   "sequence_ms_persistent": round(ms_seq, 3) if ms_seq is not None else None,
                                   "timing": "CUDA-graph replay of the whole sequence; eager: one Python call per "
                                             "step; persistent: one darb_*_sequence launch per layer"}
        for h, _ in hs:
            darb.darb_destroy(h)
    return out


def run_e2e(args, wl, torch, darb):
    """The same step through the C ABI with HOST buffers: per step, for each
    matrix darb_reencode_host (the dense W, pinned on the host, copied into the
    set's device buffer and re-encoded) and for each product darb_spmm_host (X
    in, product, Y out into pinned host memory).  Each buffer set has its own
    stream, so step s+1's copies overlap step s's kernels and its copies back;
    a set is reused only by the next step on its stream.  Every step moves all
    of its inputs and outputs inside the timed region."""
    main = torch.cuda.current_stream()
    streams = [torch.cuda.Stream() for _ in range(NSETS)]
    host_W = [torch.from_numpy(m["bits"].view(np.int16)).pin_memory().view(torch.bfloat16) for m in wl.mats]
    host_X, host_Y = {}, {}
    st0 = wl.sets[0]
    for key, X in st0["X"].items():
        host_X[key] = X.cpu().pin_memory()
        host_Y[key] = [torch.empty(st0["Y"][key].shape, dtype=torch.float32).pin_memory() for _ in range(NSETS)]
    h2d = sum(w.numel() * 2 for w in host_W) + sum(x.numel() * 4 for x in host_X.values())
    d2h = sum(y[0].numel() * 4 for y in host_Y.values())

    def step(s):
        # the re-encodes (the big weight copies) first: issuing the products
        # first measured slower (223-228 against 237 GB/s), and so did a second
        # stream per set for the products (213 GB/s)
        k = s % NSETS
        st, sid = wl.sets[k], streams[k].cuda_stream
        for mi in range(len(wl.mats)):
            darb.darb_reencode_host(st["enc"][mi], host_W[mi], st["W"][mi], sid)
        for (kind, mi, b, _) in wl.calls:
            if kind == "spmm":
                darb.darb_spmm_host(st["spmm"][(mi, b)], host_X[(mi, b)], host_Y[(mi, b)][k],
                                    st["X"][(mi, b)], st["Y"][(mi, b)], sid)

    def run(n):
        for x in streams:
            x.wait_stream(main)
        for s in range(n):
            step(s)
        for x in streams:
            main.wait_stream(x)

    steps = max(3, args.steps // 2)
    run(args.warmup)
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(main)
    run(steps)
    b.record(main)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / steps
    return {"value": round(wl.step_bytes / (ms * 1e-3) / 1e9, 2), "unit": "GB/s",
            "ms_per_step": round(ms, 4), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "api": "darb_reencode_host + darb_spmm_host (host W, X, Y; the library copies them)",
            "pipeline": f"one stream per buffer set ({NSETS}): step s+1's copies overlap step s's kernels",
            "link_note": "host -> device over the Grace link tops out near 208 GB/s here (copy engines or "
                         "kernels reading pinned host memory alike): the dense W of a step alone is 127 MB"}


# ----------------------------------------------------------------------------- CPU oracle arm
def cpu_model() -> str:
    """The host CPU's name, from /proc/cpuinfo (x86 'model name', or the Arm
    implementer / part numbers) or lscpu."""
    try:
        with open("/proc/cpuinfo") as f:
            info = f.read()
        for key in ("model name", "Model name"):
            for ln in info.splitlines():
                if ln.startswith(key):
                    return ln.split(":", 1)[1].strip()
        impl = [ln.split(":", 1)[1].strip() for ln in info.splitlines() if ln.startswith("CPU implementer")]
        part = [ln.split(":", 1)[1].strip() for ln in info.splitlines() if ln.startswith("CPU part")]
        if impl and part:
            return f"Arm implementer {impl[0]} part {part[0]}"
    except OSError:
        pass
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.startswith("Model name"):
                return ln.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return "unknown"


class OracleStep:
    """The step the GPU arm times -- BMWM encode of FC6 and FC7, then the
    product of each at batch 1, 16, 64 and 256 -- run by the CPU oracle as it
    stands: its encoder, and its fp32-accumulate product loop (OpenMP over
    rows).  Bytes: the same algorithmic bytes as the GPU step."""

    def __init__(self):
        import oracle
        from paper_1911_08020_gb300 import synth
        self.oracle = oracle
        wl = synth.WORKLOADS[WORKLOAD]
        self.mats = []
        self.bytes = 0
        for i, (rows, cols) in enumerate(wl.shapes):
            _, bits, m = synth.matrix(wl, i)
            X = {b: synth.activations(cols, b, seed=wl.seed, sub=90 + b) for b in BATCHES}
            nnzb = int(oracle.block_pointers(m, cols)[-1])
            info = {"rows": rows, "cols": cols, "wtype": 1, "value_bytes": nnzb * 2,
                    "offset_bytes": sum(-(-cols // int(x)) * (4 if x <= 16 else 8) for x in m) // 8,
                    "meta_bytes": rows * 6}
            self.bytes += encode_bytes(info) + sum(spmm_bytes(info, b) for b in BATCHES)
            self.mats.append((bits, m, X))

    def run(self) -> float:
        """One step; returns its wall time in seconds."""
        t0 = time.perf_counter()
        encs = [self.oracle.encode(bits, m, "bf16") for bits, m, _ in self.mats]
        for b in BATCHES:
            for enc, (_, _, X) in zip(encs, self.mats):
                self.oracle.darb_spmm_f32(enc, X[b])
        return time.perf_counter() - t0


def cpu_protocol(runs: int = 5):
    """The oracle on the GPU step's calls at 1 thread and at nproc threads,
    median of `runs` steps each, with the CPU named."""
    import oracle
    oracle.build()
    step = OracleStep()
    nproc = os.cpu_count() or 1
    out = {"cpu_model": cpu_model(), "nproc": nproc, "runs": runs, "bytes_per_step": int(step.bytes)}
    for threads in (1, nproc):
        used = oracle.set_threads(threads)
        step.run()   # warm-up: page in, first-touch
        times = [step.run() for _ in range(runs)]
        med = statistics.median(times)
        out[f"threads_{threads}" if threads == 1 else "threads_nproc"] = {
            "threads": used, "median_s": round(med, 4), "min_s": round(min(times), 4),
            "gbs": round(step.bytes / med / 1e9, 3)}
    oracle.set_threads(nproc)
    out["sample"] = ("the whole FC6 + FC7 step: oracle encode (bf16) + oracle darb_spmm_f32 (fp32 accumulate) "
                     "at batch 1/16/64/256, median of %d steps" % runs)
    return out


def cpu_configs(runs: int = 3):
    """The oracle as it stands on the other four configs, at 1 thread and at
    nproc threads (median of `runs` after one untimed run): config 1's encode
    (fp32) plus its batch-1 product, and one fp64 cell step of each RNN
    workload's first layer (the unit the `rnn` section's per-step times use)."""
    import oracle
    from paper_1911_08020_gb300 import synth
    oracle.build()
    nproc = os.cpu_count() or 1
    cases = {}
    wl = synth.WORKLOADS["gemv_1024"]
    _, stored, m = synth.matrix(wl, 0)
    x1 = synth.activations(wl.shapes[0][1], 1, seed=wl.seed)
    cases["gemv_1024"] = (lambda: oracle.darb_spmm_f32(oracle.encode(stored, m, wl.dtype), x1),
                          "oracle encode (fp32) + darb_spmm_f32 at batch 1")
    for name, batches in (("lstm_1024", (1, 32)), ("lstm_lm_1500", (20,)), ("gru_1024", (64,))):
        wr = synth.WORKLOADS[name]
        _, st_r, m_r = synth.matrix(wr, 0)
        enc = oracle.encode(st_r, m_r, wr.dtype)
        I, H = wr.input_size, wr.hidden
        for B in batches:
            x, h0 = synth.activations(I, B, seed=1), synth.state(H, B, seed=2)
            if wr.kind == "lstm":
                c0 = synth.state(H, B, seed=3, scale=1.0)
                fn = (lambda enc=enc, I=I, H=H, x=x, h0=h0, c0=c0: oracle.lstm_step(enc, I, H, x, h0, c0))
            else:
                fn = (lambda enc=enc, I=I, H=H, x=x, h0=h0: oracle.gru_step(enc, I, H, x, h0))
            cases[f"{name}_b{B}"] = (fn, f"one oracle {wr.kind} cell step (fp64), first layer")
    out = {"cpu_model": cpu_model(), "nproc": nproc, "runs": runs}
    for key, (fn, what) in cases.items():
        entry = {"sample": what}
        for threads in (1, nproc):
            used = oracle.set_threads(threads)
            fn()
            times = []
            for _ in range(runs):
                t0 = time.perf_counter()
                fn()
                times.append(time.perf_counter() - t0)
            entry["threads_1" if threads == 1 else "threads_nproc"] = {
                "threads": used, "us": round(statistics.median(times) * 1e6, 1)}
        out[key] = entry
    oracle.set_threads(nproc)
    return out


def run_reference(args, world, rank):
    """The reference arm: the CPU oracle as it stands (the paper ships no code)
    runs the GPU arm's step at nproc threads; `value` = the step's algorithmic
    bytes over the mean step time."""
    if rank != 0:
        return None
    import oracle
    oracle.build()
    step = OracleStep()
    cores = oracle.set_threads(os.cpu_count() or 1)
    for _ in range(args.warmup):
        step.run()
    times = [step.run() for _ in range(args.steps)]
    ms = 1e3 * statistics.mean(times)
    gbs = step.bytes / (ms * 1e-3) / 1e9
    sample = ("the whole FC6 + FC7 step per timed step: oracle encode (bf16) + oracle darb_spmm_f32 (fp32 "
              "accumulate) at batch 1/16/64/256")
    return {
        "metric": METRIC, "value": round(gbs, 3), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "impl": "reference",
        "config": {"workload": "fc6_fc7_4096x9216_4096x4096_bf16_weights",
                   "batches": list(BATCHES), "sample": sample, "parallelism": "cpu"},
        "cpu_baseline": {"value": round(gbs, 3), "unit": "GB/s", "cores": cores, "kind": "oracle",
                         "sample": sample, "cpu_model": cpu_model()},
        "e2e": {"value": round(gbs, 3), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    args = parse_args()
    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        res = run_reference(args, world, rank)
        if rank == 0 and res is not None:
            print(json.dumps(res), flush=True)
        return
    res = run_gpu(args, world, rank, local)
    if rank == 0:
        if not args.no_cpu and world == 1:
            cp = cpu_protocol()
            res["cpu_baseline"] = {"value": cp["threads_nproc"]["gbs"], "unit": "GB/s",
                                   "cores": cp["threads_nproc"]["threads"], "kind": "oracle",
                                   "sample": cp["sample"], "cpu_model": cp["cpu_model"],
                                   "threads_1": cp["threads_1"], "threads_nproc": cp["threads_nproc"],
                                   "same_step_as_gpu": True}
            if "rnn" in res or "gemv_1024" in res:
                # the GPU numbers of configs 1-4 are in `gemv_1024` and `rnn`
                res["cpu_configs"] = cpu_configs()
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
