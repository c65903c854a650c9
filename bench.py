"""Benchmark of the CCI-sparse forward layer (arXiv 1910.11971) on GB300.

Headline workload: the K/G sweep, a 4096 -> 4096 product over N = 8192 columns
in bf16 (W ~ N(0, 1/4096), X ~ N(0, 1), seeded synthetic data), at its middle
point G = 8, K = 2 (75 % sparse).  One step = the whole hot path on one batch:
cci_pack of the dense weights (per-group top-K, Sec. 3.1 / 5.1) + the product
(Alg. 2) through the library's production path, inputs resident in HBM.  The
metric is nonzero TFLOP/s (2*N*R*Cout*K/G per step).  L2 (129 MB) is flushed
between timed steps by writing a 256 MB buffer outside the timed events.

stdout gets ONE short JSON line, last: the headline with its roofline, CPU
baseline (the fp64 oracle on a bounded sample), end-to-end figure (host buffers,
copies inside the timed region), clocks, and a compact per-(G, K) array of the
sweep.  Every other measurement (fp32 bottleneck, 3x3 convolution, ResNet-50 and
MobileNetV2 stacks, Eq. 1, targeted dropout, CCI against balanced sparsity) is
printed to stderr, one JSON line each.

``--impl reference`` times the fp64 CPU oracle on a bounded sample of the same
workload instead.  Multi-GPU (torchrun): every rank runs its own batch (weak
scaling, no collective on the data path); the step time is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_1910_11971_gb300 import workloads as wl  # noqa: E402

METRIC = "CCI layer nonzero TFLOP/s & fraction of roofline vs K/G; speedup over dense"
UNIT = "TFLOP/s"
MEASURED_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
# CUDA-core fp32 FMA peak from unit counts and clock: 152 SMs x 128 FP32 lanes
# x 2 flop x 2.070 GHz (maximum SM clock); the FFMA path is ALU-bound.
N_SM, FMA_LANES, SM_MAX_GHZ = 152, 128, 2.070
ALU_PEAK_TFLOPS = N_SM * FMA_LANES * 2 * SM_MAX_GHZ / 1e3
L2_FLUSH_BYTES = 256 << 20
HBM_ROOF_GBS = 8000.0  # the workload's stated memory roof (8 TB/s)
HEADLINE = wl.sweep_case(8, 2)  # the middle point of the K/G sweep
# --algo names -> cci_algo values (profiling runs only)
ALGOS = {"auto": 0, "generic": 1, "regtile": 2, "fused": 3, "expand": 4, "ws": 5}


def measured_peaks():
    try:
        with open(MEASURED_PEAKS) as f:
            return json.load(f)
    except (OSError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def tensor_peak(dtype_name: str) -> float:
    """Dense tensor-core peak for the operand type: the measured bf16 burst figure,
    times the nominal tf32/bf16 ratio (1.1 / 2.25 PFLOP/s) for tf32."""
    bf16 = float(measured_peaks()["bf16_tflops"])
    return bf16 if dtype_name == "bf16" else bf16 * 1.1 / 2.25


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--extras", type=int, default=1,
                    help="also measure the other workloads (stderr, one JSON line each)")
    ap.add_argument("--cpu-sample-seconds", type=float, default=12.0)
    ap.add_argument("--profile", type=int, default=0,
                    help="only the warm-up and timed steps of the main path (for ncu)")
    ap.add_argument("--workload", default=HEADLINE.name,
                    help="sweep_4096_G<G>_K<K> (default G8_K2) or bottleneck_1x1: the product timed; with "
                         "--profile 1 also a convolution: conv3x3_28, resnet50_lNN_K<K> (layer NN of "
                         "the ResNet-50 stack) or mobilenetv2_pwNN (pointwise layer NN of MobileNetV2)")
    ap.add_argument("--algo", default="auto", choices=sorted(ALGOS),
                    help="with --profile 1: the kernel family of the timed product")
    return ap.parse_args()


# ---------------------------------------------------------------------------
# distributed plumbing (weak scaling: no collective on the data path)
# ---------------------------------------------------------------------------
def dist_init(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int, device) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    """SM clock and clock-event reasons during the timed region.

    Reads NVML through ctypes (read-only queries: clocks and event reasons),
    polling about every millisecond so that a timed region of a few ms still has
    samples; falls back to `nvidia-smi -lms 200` when NVML cannot be loaded."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device: torch.device):
        self.device = device
        self.samples = []  # (sm_mhz, max_mhz, reasons bitmask)
        self.smi_lines = []
        self.proc = None
        self.nvml = None
        self.stop = threading.Event()
        try:
            import ctypes
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                raise OSError("nvmlInit failed")
            h = ctypes.c_void_p()
            uuid = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
            if lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) != 0:
                raise OSError("device handle")
            self.nvml, self.handle, self.ct = lib, h, ctypes
        except (OSError, AttributeError, RuntimeError):
            self.nvml = None

    def _poll_nvml(self):
        ct, lib = self.ct, self.nvml
        cur, mx, rs = ct.c_uint(), ct.c_uint(), ct.c_ulonglong()
        get_reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self.stop.is_set():
            if (lib.nvmlDeviceGetClockInfo(self.handle, 1, ct.byref(cur)) == 0
                    and lib.nvmlDeviceGetMaxClockInfo(self.handle, 1, ct.byref(mx)) == 0):
                r = rs.value if get_reasons(self.handle, ct.byref(rs)) == 0 else 0
                self.samples.append((float(cur.value), float(mx.value), int(r)))
            time.sleep(0.001)

    def _read_smi(self):
        for line in self.proc.stdout:
            self.smi_lines.append(line.strip())

    def __enter__(self):
        if self.nvml is not None:
            self.thread = threading.Thread(target=self._poll_nvml, daemon=True)
            self.thread.start()
            t0 = time.time()
            while not self.samples and time.time() - t0 < 1.0:
                time.sleep(0.001)
            self.samples.clear()  # keep only the samples taken in the timed region
        else:
            try:
                self.proc = subprocess.Popen(
                    ["nvidia-smi", f"--id={self.device.index or 0}", f"--query-gpu={self.FIELDS}",
                     "--format=csv,noheader,nounits", "-lms", "200"],
                    stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
                self.thread = threading.Thread(target=self._read_smi, daemon=True)
                self.thread.start()
            except (OSError, FileNotFoundError):
                self.proc = None
        return self

    def __exit__(self, *exc):
        self.stop.set()
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        elif self.nvml is not None:
            self.thread.join(timeout=1.0)

    def summary(self):
        if self.nvml is not None:
            if not self.samples:
                return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "source": "nvml"}
            reasons = set()
            for _, _, r in self.samples:
                for bit, name in self.REASONS.items():
                    if r & bit:
                        reasons.add(name)
            return {"sm_mhz": statistics.median(s[0] for s in self.samples),
                    "sm_max_mhz": max(s[1] for s in self.samples), "reasons": sorted(reasons),
                    "samples": len(self.samples)}
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.smi_lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "source": "nvidia-smi"}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "source": "nvidia-smi"}


# ---------------------------------------------------------------------------
# the reported CPU baseline: the fp64 oracle on a bounded sample
# ---------------------------------------------------------------------------
def oracle_rate(case: wl.LinearCase, seconds: float):
    """Nonzero TFLOP/s of the oracle on the first `rows` columns of the workload,
    with `rows` grown until one call takes about `seconds`; when the whole
    workload takes less, whole passes repeat until `seconds` have elapsed.
    Returns (rate, rows, passes, seconds spent, threads)."""
    import numpy as np

    import oracle
    X, W = wl.linear_inputs(case)
    Xf = X.to(torch.float64).numpy()
    v, i = oracle.pack(W.to(torch.float64).numpy(), case.G, case.K)
    Wd, mask = oracle.decompress(v, i, case.Cout, case.G)
    rows = 64
    while True:
        t0 = time.perf_counter()
        oracle.linear(Xf[:rows], Wd, mask)
        dt = time.perf_counter() - t0
        if dt >= seconds or rows >= Xf.shape[0]:
            break
        rows = min(Xf.shape[0], int(rows * max(2.0, 1.2 * seconds / max(dt, 1e-3))))
    passes, total = 1, dt
    while total < seconds:
        t0 = time.perf_counter()
        oracle.linear(Xf[:rows], Wd, mask)
        total += time.perf_counter() - t0
        passes += 1
    flops = 2.0 * rows * case.R * case.Cout * case.K / case.G * passes
    return flops / total / 1e12, rows, passes, total, oracle.threads()


def run_reference(args, rank, world):
    """The reference arm: the fp64 oracle (pack, decompression, dense-mask product)
    on the host cores, on a bounded sample of the headline workload per step."""
    case = workload_case(args.workload)
    if rank != 0:
        return 0
    import oracle
    X, W = wl.linear_inputs(case, N=4096)
    Xf = X.to(torch.float64).numpy()
    Wf = W.to(torch.float64).numpy()
    # size one step's sample so that warmup + steps stay within a few minutes
    v, i = oracle.pack(Wf, case.G, case.K)
    Wd, mask = oracle.decompress(v, i, case.Cout, case.G)
    rows = 16
    t0 = time.perf_counter()
    oracle.linear(Xf[:rows], Wd, mask)
    dt = time.perf_counter() - t0
    budget = 90.0 / max(1, args.steps + args.warmup)
    rows = max(4, min(Xf.shape[0], int(rows * budget / max(dt, 1e-4))))
    for _ in range(args.warmup):
        oracle.pack(Wf, case.G, case.K)
        oracle.linear(Xf[:rows], Wd, mask)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        vv, ii = oracle.pack(Wf, case.G, case.K)
        Wd, mask = oracle.decompress(vv, ii, case.Cout, case.G)
        oracle.linear(Xf[:rows], Wd, mask)
    dt = (time.perf_counter() - t0) / args.steps
    flops = 2.0 * rows * case.R * case.Cout * case.K / case.G
    value = flops / dt / 1e12
    sample = (f"{rows} of {case.N} columns per step (pack + decompress + dense-mask product in "
              f"fp64), {case.Cin}->{case.Cout}, G={case.G}, K={case.K}")
    line = {
        "impl": "reference", "metric": METRIC, "value": sig(value), "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sig(dt * 1e3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(case, extra={"sample_columns": rows}),
        "cpu_baseline": {"value": sig(value), "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": sig(value), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def sig(x, n: int = 4):
    """x rounded to n significant digits (keeps the headline line short)."""
    if x is None or not isinstance(x, (int, float)) or x == 0 or not math.isfinite(x):
        return x
    return float(f"{x:.{n}g}")


def config_of(case, extra=None):
    c = {"workload": case.name, "N": case.N, "Cin": case.Cin, "Cout": case.Cout, "G": case.G,
         "K": case.K, "dtype_in": case.dtype, "l2": "flushed (256 MB write, untimed)",
         "parallelism": "one batch/GPU"}
    if case.name.startswith("sweep_4096"):
        c["workload"] = f"sweep_4096 (K/G sweep, 11 points); value at G={case.G} K={case.K}"
    if extra:
        c.update(extra)
    return c


def extra(name: str, payload) -> None:
    """One measurement beside the headline, as its own JSON line on stderr (the
    headline stays the last, short line on stdout)."""
    print(json.dumps({"extra": name, "data": payload}), file=sys.stderr, flush=True)


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
# the sources of the tensor-core product (decompression and GEMM): a DRAM-traffic
# record in profiles/traffic.txt holds for the sources it was taken on
PRODUCT_SOURCES = ("cci_common.cuh", "cci_kernels.h", "cci_tc_common.cuh", "cci_gemm_ws.cuh",
                   "cci_gemm_ws_bf16.cu", "cci_gemm_ws_tf32.cu", "cci_dense_tc.cu")


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_1910_11971_gb300", "csrc")
    for name in PRODUCT_SOURCES:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def measured_traffic(kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current kernel sources (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    r = rec.get(kernel)
    if not r or r.get("source_hash") != kernel_source_hash():
        return None
    return r.get("dram_bytes_per_launch")


def time_device(fn, reps, flush, stream):
    """Per-rep CUDA-event durations (ms) on `stream`, L2 flushed before each rep."""
    out = []
    for _ in range(reps):
        flush()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record(stream)
        fn()
        e.record(stream)
        e.synchronize()
        out.append(s.elapsed_time(e))
    return out


def workload_case(name: str) -> wl.LinearCase:
    if name == wl.BOTTLENECK_1X1.name:
        return wl.BOTTLENECK_1X1
    for G, K in wl.SWEEP_POINTS:
        if name == wl.sweep_case(G, K).name:
            return wl.sweep_case(G, K)
    raise SystemExit(f"unknown workload {name}")


def conv_case(name: str):
    """A convolution workload by name, or None."""
    if name == wl.CONV3X3_28.name:
        return wl.CONV3X3_28
    if name.startswith("resnet50_l") and "_K" in name:
        li, k = name[len("resnet50_l"):].split("_K")
        return wl.resnet50_layers(K=int(k))[int(li)]
    if name.startswith("mobilenetv2_pw"):
        return wl.mobilenetv2_pointwise_layers()[int(name[len("mobilenetv2_pw"):])]
    return None


def profile_conv(cci, case, args, dev, stream):
    """Warm-up and timed steps (pack + convolution) of one convolution layer, for
    profiler captures; prints the mean step time."""
    X, W = wl.conv_inputs(case, device=str(dev))
    values = torch.empty((case.Cout // case.G, case.R, case.K), dtype=X.dtype, device=dev)
    idx = torch.empty((case.Cout // case.G, case.R, case.K), dtype=torch.uint8, device=dev)
    Y = torch.empty((case.B, case.P, case.Q, case.Cout), dtype=torch.float32, device=dev)
    ws = cci.auto_workspace(X.dtype, case.Cin, case.R, case.Cout, case.G, case.K, dev)
    status = cci.new_status(dev)
    flush_buf = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def step():
        cci.pack(W, case.G, case.K, status=status, check=False, out=(values, idx))
        cci.conv2d(X, values, idx, case.Cout, case.G, case.K, case.KH, case.KW, (case.stride,) * 2,
                   (case.pad,) * 2, out=Y, status=status, workspace=ws)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    ms = time_device(step, args.steps, lambda: flush_buf.fill_(1.0), stream)
    assert cci.read_status(status) == 0
    print(json.dumps({"workload": case.name, "ms_per_step": statistics.mean(ms), "steps": args.steps,
                      "note": "profiling helper: pack + convolution per step"}), flush=True)
    return 0


def launches_per_product(cci, dtype, case) -> int:
    """Kernels one product launches on the production path (AUTO): the workspace
    family runs a decompression and the GEMM, every other family one kernel."""
    name = cci.kernel_name(dtype, case.Cin, case.R, case.Cout, case.G, case.K, cci.ALGO_AUTO)
    return 2 if name.startswith("dense_tc_ws") else 1


def run_ours(args, rank, world, local):
    import paper_1910_11971_gb300 as cci
    from paper_1910_11971_gb300 import build as cci_build

    cci_build.build()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.backends.cudnn.allow_tf32 = False
    cc = conv_case(args.workload)
    if cc is not None:
        if not args.profile:
            raise SystemExit("convolution workloads are profiling helpers: pass --profile 1")
        return profile_conv(cci, cc, args, dev, stream)
    case = workload_case(args.workload)
    X, W = wl.linear_inputs(case, device="cpu")
    X_host = X.pin_memory()
    W_host = W.pin_memory()
    Xd, Wd = X.to(dev), W.to(dev)
    values = torch.empty((case.Cout // case.G, case.R, case.K), dtype=Xd.dtype, device=dev)
    idx = torch.empty((case.Cout // case.G, case.R, case.K), dtype=torch.uint8, device=dev)
    Y = torch.empty((case.N, case.Cout), dtype=torch.float32, device=dev)
    # the library's production path: AUTO (with the workspace it asks for, if any)
    algo = ALGOS[args.algo] if args.profile else cci.ALGO_AUTO
    if algo == cci.ALGO_AUTO:
        ws = cci.auto_workspace(Xd.dtype, case.Cin, case.R, case.Cout, case.G, case.K, dev)
    else:
        ws = cci.new_workspace(algo, Xd.dtype, case.Cout, case.R, dev)
    kname = cci.kernel_name(Xd.dtype, case.Cin, case.R, case.Cout, case.G, case.K, cci.ALGO_AUTO)
    on_tc = kname.startswith("dense_tc")
    status = cci.new_status(dev)
    flush_buf = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def flush():
        flush_buf.fill_(1.0)

    def product():
        cci.linear(Xd, values, idx, case.Cout, case.G, case.K, out=Y, status=status, algo=algo, workspace=ws)

    def step():
        cci.pack(Wd, case.G, case.K, status=status, check=False, out=(values, idx))
        product()

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    assert cci.read_status(status) == 0

    # ---- timed region: K steps, per-step events (pack | product), L2 flushed between ----
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize(dev)
    with ClockSampler(dev) as clk:
        t_wall0 = time.perf_counter()
        for k in range(args.steps):
            flush()
            a, b, c = ev[k]
            a.record(stream)
            cci.pack(Wd, case.G, case.K, status=status, check=False, out=(values, idx))
            b.record(stream)
            product()
            c.record(stream)
        torch.cuda.synchronize(dev)
        t_wall = time.perf_counter() - t_wall0
    barrier(world)
    if args.profile:
        return 0
    step_ms = [a.elapsed_time(c) for a, b, c in ev]
    lin_ms = [b.elapsed_time(c) for a, b, c in ev]
    pack_ms = [a.elapsed_time(b) for a, b, c in ev]
    assert cci.read_status(status) == 0
    ms_step = max_over_ranks(sum(step_ms) / len(step_ms), world, dev)
    nzf = case.nz_flops()
    value = world * nzf / (ms_step * 1e-3) / 1e12
    lin_avg = statistics.mean(lin_ms)
    achieved = nzf / (lin_avg * 1e-3) / 1e12
    es = X.element_size()
    alg_bytes = algorithmic_bytes(case, es)
    tdt = "bf16" if X.dtype == torch.bfloat16 else "tf32"
    if on_tc:
        # tensor time in units of the dtype peak: fp32 runs one tf32 pass (hi*hi) and
        # two bf16 passes (the cross terms) at twice the tf32 rate
        passes = 1 if tdt == "bf16" else 2
        peak = tensor_peak(tdt)
        executed = passes * case.dense_flops()
        roofline = {"bound": "tensor", "achieved": sig(achieved), "peak": sig(peak), "unit": "TFLOP/s",
                    "frac": sig(achieved / peak), "traffic": measured_traffic(kname), "kernel": kname,
                    "peak_source": "measured bf16 burst" + (" x 1.1/2.25" if tdt == "tf32" else ""),
                    "tensor_util": sig(executed / (lin_avg * 1e-3) / 1e12 / peak)}
    else:
        roofline = {"bound": "alu", "achieved": sig(achieved), "peak": sig(ALU_PEAK_TFLOPS), "unit": "TFLOP/s",
                    "frac": sig(achieved / ALU_PEAK_TFLOPS), "traffic": measured_traffic(kname), "kernel": kname,
                    "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 flop x 2.070 GHz"}
    # the workload's own roofline (the metric's): the slower of its nonzero flops at
    # the CUDA-core FMA peak and its compressed bytes at 8 TB/s
    floor_s = max(nzf / (ALU_PEAK_TFLOPS * 1e12), alg_bytes / (HBM_ROOF_GBS * 1e9))
    roofline["metric_frac"] = sig(floor_s / (lin_avg * 1e-3))

    # ---- end to end through the public API: W host -> device and packed, then
    # cci_linear_host: X from pinned host memory, Y back to it, in column chunks
    # whose copies (own streams) overlap the product ----
    Y_host = torch.empty((case.N, case.Cout), dtype=torch.float32).pin_memory()
    chunk = cci.host_chunk(case.N)
    hbuf = cci.host_buffer(X.dtype, case.Cin, case.Cout, chunk, dev)

    def e2e_step():
        Wd.copy_(W_host, non_blocking=True)
        cci.pack(Wd, case.G, case.K, status=status, check=False, out=(values, idx))
        cci.linear_host(X_host, values, idx, case.Cout, case.G, case.K, out=Y_host, status=status, chunk=chunk,
                        buffer=hbuf)

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize(dev)
    e2e_ms = statistics.mean(time_device(e2e_step, max(3, args.steps // 4), flush, stream))
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    e2e = {"value": sig(world * nzf / (e2e_ms * 1e-3) / 1e12), "unit": UNIT,
           "h2d_bytes_per_step": X_host.numel() * X_host.element_size() + W_host.numel() * W_host.element_size(),
           "d2h_bytes_per_step": Y_host.numel() * 4, "ms_per_step": sig(e2e_ms)}
    extra("e2e_path", "H2D copy of W + cci_pack + cci_linear_host (X and Y in pinned host memory, column "
                      f"chunks of {chunk}, copies on their own streams overlapping the product)")

    sweep = []
    if rank == 0 and case.name.startswith("sweep_4096"):
        sweep = run_sweep(cci, dev, stream, flush)
    if args.extras and rank == 0:
        run_extras(cci, dev, stream, flush)

    cpu = None
    if rank == 0 and world == 1:
        rate, rows, passes, dt, cores = oracle_rate(case, args.cpu_sample_seconds)
        cpu = {"value": sig(rate), "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"fp64 dense-mask product, first {rows}/{case.N} columns x {passes}, {dt:.0f} s"}

    if rank == 0:
        extra("timed_region", {"wall_ms_per_step_incl_flush": t_wall * 1e3 / args.steps, "clocks": clk.summary()})
        line = {
            "metric": METRIC, "value": sig(value), "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": sig(ms_step), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if tdt == "bf16" else "f32",
            "data": "synthetic", "config": config_of(case), "roofline": roofline, "cpu_baseline": cpu,
            "e2e": e2e, "gpu_launches": (1 + launches_per_product(cci, X.dtype, case)) * args.steps,
            "clocks": clk.summary(),
            "ms": {"pack": sig(statistics.mean(pack_ms)), "product": sig(lin_avg)},
            "sweep": sweep,
        }
        print(json.dumps(line, separators=(",", ":")), flush=True)
    return 0


def run_sweep(cci, dev, stream, flush, reps=10):
    """The K/G sweep (4096 -> 4096, N = 8192, bf16): per (G, K) the production
    product (pack excluded), cuBLAS bf16 on the masked dense weights, and the same
    tensor-core GEMM on the unpruned dense weights without decompression.  Keys:
    ms (CCI product), nz (nonzero TFLOP/s), frac (the workload roofline: nonzero
    flops at the CUDA-core FMA peak, or bytes at 8 TB/s, over ms),
    cublas (cuBLAS ms / CCI ms), same (the same kernel on dense weights, its ms /
    CCI ms: what the sparsity buys); the tensor utilisation (dense flops executed /
    ms / measured bf16 peak) and kernel names go to stderr."""
    out, tu = [], []
    dense_same_ms = None
    peak = tensor_peak("bf16")
    for G, K in wl.SWEEP_POINTS:
        case = wl.sweep_case(G, K)
        X, W = wl.linear_inputs(case, device=str(dev))
        v, i = cci.pack(W, G, K)
        Y = torch.empty((case.N, case.Cout), dtype=torch.float32, device=dev)
        ws = cci.auto_workspace(X.dtype, case.Cin, case.R, case.Cout, G, K, dev)
        fn = lambda: cci.linear(X, v, i, case.Cout, G, K, out=Y, workspace=ws)  # noqa: E731
        fn()
        ms = statistics.median(time_device(fn, reps, flush, stream))
        Wm = torch.zeros((case.Cout, case.R), dtype=W.dtype, device=dev)
        Wm.view(case.Cout // G, G, case.R).scatter_(1, i.permute(0, 2, 1).long(), v.permute(0, 2, 1))
        dms = statistics.median(time_device(lambda: torch.matmul(X, Wm.t()), reps, flush, stream))
        if dense_same_ms is None:  # one shape for every point: the unpruned W of the first
            Wp = cci.dense_planes(W)
            fd = lambda: cci.dense_linear_tc(X, Wp, case.Cout, out=Y)  # noqa: E731
            fd()
            dense_same_ms = statistics.median(time_device(fd, reps, flush, stream))
            del Wp
        nz = case.nz_flops() / (ms * 1e-3) / 1e12
        floor_s = max(case.nz_flops() / (ALU_PEAK_TFLOPS * 1e12),
                      algorithmic_bytes(case, 2) / (HBM_ROOF_GBS * 1e9))
        out.append({"G": G, "K": K, "ms": sig(ms), "nz": sig(nz, 3), "frac": sig(floor_s / (ms * 1e-3), 3),
                    "cublas": sig(dms / ms, 3), "same": sig(dense_same_ms / ms, 3)})
        tu.append({"G": G, "K": K, "tensor_util": case.dense_flops() / (ms * 1e-3) / 1e12 / peak,
                   "cublas_ms": dms, "kernel": cci.kernel_name(X.dtype, case.Cin, case.R, case.Cout, G, K,
                                                               cci.ALGO_AUTO)})
        del X, W, v, i, Y, Wm, ws
    torch.cuda.empty_cache()
    extra("sweep_4096_details", {"same_kernel_dense_ms": dense_same_ms, "points": tu,
                                 "same_kernel": "the tensor-core GEMM on unpruned bf16 W, no decompression"})
    return out


def algorithmic_bytes(case, elem: int) -> int:
    """Bytes a product or convolution must move at least: its input once (the
    NHWC tensor for a convolution), its fp32 output once and the packed weights
    (values and uint8 indices)."""
    x = case.B * case.H * case.W * case.Cin if isinstance(case, wl.ConvCase) else case.N * case.Cin
    return x * elem + case.N * case.Cout * 4 + (case.Cout // case.G) * case.R * case.K * (elem + 1)


def kernel_families(cci, case, X, v, i, Y, conv, flush, stream, reps=5):
    """The product of one workload on every kernel family that has it: the CUDA-core
    scatter families (jump dispatch and expand), the workspace tensor-core family
    and the fused tensor-core family; ms and nonzero TFLOP/s of each."""
    G, K = case.G, case.K
    res = {}
    for name, algo in (("regtile_jump", cci.ALGO_REGTILE), ("expand", cci.ALGO_EXPAND),
                       ("dense_tc_ws", cci.ALGO_DENSE_TC_WS), ("dense_tc_fused", cci.ALGO_DENSE_TC)):
        kn = cci.kernel_name(X.dtype, case.Cin, case.R, case.Cout, G, K, algo)
        if not kn:
            continue
        ws = cci.new_workspace(algo, X.dtype, case.Cout, case.R, X.device) if algo == cci.ALGO_DENSE_TC_WS else None
        if conv:
            fn = lambda a=algo, w=ws: cci.conv2d(X, v, i, case.Cout, G, K, case.KH, case.KW,  # noqa: E731
                                                 (case.stride,) * 2, (case.pad,) * 2, out=Y, algo=a, workspace=w)
        else:
            fn = lambda a=algo, w=ws: cci.linear(X, v, i, case.Cout, G, K, out=Y, algo=a, workspace=w)  # noqa: E731
        fn()
        ms = statistics.median(time_device(fn, reps, flush, stream))
        res[name] = {"kernel": kn, "ms": sig(ms), "nz": sig(case.nz_flops() / (ms * 1e-3) / 1e12)}
    return res


def run_bottleneck_fp32(cci, dev, stream, flush, reps=10):
    """The ResNet 1x1 bottleneck as an fp32 product (N = 100352, 256 -> 1024, G = 8,
    K = 2): the production path, every kernel family, cuBLAS fp32 (TF32 off) on the
    masked dense weights and the same tensor-core GEMM on the unpruned weights."""
    case = wl.BOTTLENECK_1X1
    X, W = wl.linear_inputs(case, device=str(dev))
    v, i = cci.pack(W, case.G, case.K)
    Y = torch.empty((case.N, case.Cout), dtype=torch.float32, device=dev)
    ws = cci.auto_workspace(X.dtype, case.Cin, case.R, case.Cout, case.G, case.K, dev)
    fn = lambda: cci.linear(X, v, i, case.Cout, case.G, case.K, out=Y, workspace=ws)  # noqa: E731
    fn()
    ms = statistics.median(time_device(fn, reps, flush, stream))
    Wm = torch.zeros_like(W)
    Wm.view(case.Cout // case.G, case.G, case.R).scatter_(1, i.permute(0, 2, 1).long(), v.permute(0, 2, 1))
    dms = statistics.median(time_device(lambda: torch.matmul(X, Wm.t()), reps, flush, stream))
    Wp = cci.dense_planes(W)
    fd = lambda: cci.dense_linear_tc(X, Wp, case.Cout, out=Y)  # noqa: E731
    fd()
    sms = statistics.median(time_device(fd, reps, flush, stream))
    nzf = case.nz_flops()
    floor_s = max(nzf / (ALU_PEAK_TFLOPS * 1e12), algorithmic_bytes(case, 4) / (HBM_ROOF_GBS * 1e9))
    return {"workload": case.name, "ms": ms, "nz_tflops": nzf / (ms * 1e-3) / 1e12,
            "metric_roofline_frac": floor_s / (ms * 1e-3),
            "kernel": cci.kernel_name(X.dtype, case.Cin, case.R, case.Cout, case.G, case.K, cci.ALGO_AUTO),
            "cublas_fp32_simt_ms": dms, "speedup_over_cublas_fp32": dms / ms,
            "same_kernel_dense_ms": sms, "sparsity_gain": sms / ms,
            "tensor_vs_simt": dms / sms,
            "families": kernel_families(cci, case, X, v, i, Y, False, flush, stream)}


def run_conv3x3(cci, dev, stream, flush, reps=10):
    """The 3x3 convolution workload (batch 64, 28x28, 128 -> 128, G = 16, K = 4,
    bf16): the production path, every kernel family, cuDNN bf16 on the masked dense
    weights and the same tensor-core GEMM on the unpruned weights."""
    case = wl.CONV3X3_28
    X, W = wl.conv_inputs(case, device=str(dev))
    v, i = cci.pack(W, case.G, case.K)
    Y = torch.empty((case.B, case.P, case.Q, case.Cout), dtype=torch.float32, device=dev)
    ws = cci.auto_workspace(X.dtype, case.Cin, case.R, case.Cout, case.G, case.K, dev)
    fn = lambda: cci.conv2d(X, v, i, case.Cout, case.G, case.K, 3, 3, (1, 1), (1, 1), out=Y,  # noqa: E731
                            workspace=ws)
    fn()
    ms = statistics.median(time_device(fn, reps, flush, stream))
    Wm = torch.zeros((case.Cout, case.R), dtype=W.dtype, device=dev)
    Wm.view(case.Cout // case.G, case.G, case.R).scatter_(1, i.permute(0, 2, 1).long(), v.permute(0, 2, 1))
    w4 = Wm.view(case.Cout, 3, 3, case.Cin).permute(0, 3, 1, 2).contiguous(memory_format=torch.channels_last)
    x4 = X.permute(0, 3, 1, 2)  # NHWC memory, NCHW view = channels_last
    dms = statistics.median(time_device(lambda: torch.nn.functional.conv2d(x4, w4, padding=1), reps, flush, stream))
    fd = lambda: cci.dense_conv2d_tc(X, W, case.Cout, 3, 3, (1, 1), (1, 1), out=Y)  # noqa: E731
    fd()
    sms = statistics.median(time_device(fd, reps, flush, stream))
    nzf = case.nz_flops()
    return {"workload": case.name, "ms": ms, "nz_tflops": nzf / (ms * 1e-3) / 1e12,
            "metric_roofline_frac": layer_floor_us(case) * 1e-3 / ms,
            "dense_equiv_tflops": case.dense_flops() / (ms * 1e-3) / 1e12,
            "kernel": cci.kernel_name(X.dtype, case.Cin, case.R, case.Cout, case.G, case.K, cci.ALGO_AUTO),
            "cudnn_bf16_ms": dms, "speedup_over_cudnn": dms / ms,
            "same_kernel_dense_ms": sms, "sparsity_gain": sms / ms,
            "families": kernel_families(cci, case, X, v, i, Y, True, flush, stream)}


def run_extras(cci, dev, stream, flush):
    """Every measurement beside the headline, each printed as its own stderr line:
    the fp32 bottleneck product, the 3x3 convolution, the ResNet-50 and MobileNetV2
    stacks, Eq. 1's allocation error, the targeted-dropout step and CCI against
    balanced sparsity."""
    for name, fn in (("bottleneck_1x1_fp32", run_bottleneck_fp32), ("conv3x3_28", run_conv3x3),
                     ("resnet50_stack", run_resnet_stack), ("mobilenetv2_pointwise", run_pointwise_stack),
                     ("allocation_error", run_allocation_error), ("td_mask", run_td_mask),
                     ("cci_vs_bbs", run_cci_vs_bbs)):
        extra(name, fn(cci, dev, stream, flush))
        torch.cuda.empty_cache()


def run_cci_vs_bbs(cci, dev, stream, flush, reps=5):
    """The paper's comparison format (Sec. 3.4) on the same shapes: balanced
    sparsity (groups of G inputs per output channel) against CCI (groups of G
    output channels per input), each on the tensor cores (decompression + the
    same GEMM) and on CUDA cores (BBS: gather kernel; CCI: branch-free expand and
    jump dispatch)."""
    res = []
    shapes = [("sweep_4096_G8_K2", wl.sweep_case(8, 2)), ("sweep_4096_G16_K4", wl.sweep_case(16, 4)),
              ("bottleneck_1x1", wl.BOTTLENECK_1X1)]
    for name, case in shapes:
        X, W = wl.linear_inputs(case, device=str(dev))
        G, K = case.G, case.K
        Y = torch.empty((case.N, case.Cout), dtype=torch.float32, device=dev)
        ws = cci.new_workspace(cci.ALGO_DENSE_TC_WS, X.dtype, case.Cout, case.R, dev)
        cv, ci = cci.pack(W, G, K)
        bv, bi = cci.bbs_pack(W, G, K)
        row = {"shape": name, "G": G, "K": K, "dtype": case.dtype, "nz_gflop": case.nz_flops() / 1e9}
        runs = {
            "cci_tc_ms": lambda: cci.linear(X, cv, ci, case.Cout, G, K, out=Y, algo=cci.ALGO_DENSE_TC_WS,
                                            workspace=ws),
            "bbs_tc_ms": lambda: cci.bbs_linear(X, bv, bi, case.Cout, G, K, out=Y, algo=cci.ALGO_DENSE_TC_WS,
                                                workspace=ws),
            "bbs_cuda_core_gather_ms": lambda: cci.bbs_linear(X, bv, bi, case.Cout, G, K, out=Y,
                                                              algo=cci.ALGO_GENERIC),
            "cci_cuda_core_expand_ms": lambda: cci.linear(X, cv, ci, case.Cout, G, K, out=Y, algo=cci.ALGO_EXPAND),
            "cci_cuda_core_jump_ms": lambda: cci.linear(X, cv, ci, case.Cout, G, K, out=Y, algo=cci.ALGO_REGTILE),
        }
        for key, fn in runs.items():
            try:
                fn()
            except Exception as e:  # a family without this (G, K) or shape
                row[key] = None
                row[key.replace("_ms", "_why")] = str(e)[:80]
                continue
            ms = statistics.median(time_device(fn, reps, flush, stream))
            row[key] = ms
            row[key.replace("_ms", "_nz_tflops")] = case.nz_flops() / (ms * 1e-3) / 1e12
        res.append(row)
        del X, W, Y, ws, cv, ci, bv, bi
    return res


def run_td_mask(cci, dev, stream, flush, reps=10):
    """One targeted-dropout step (Sec. 5.1) on a 4096 x 8192 weight matrix, G = 8,
    K = 2, rate 0.75, per dtype: bytes moved (W, uniforms, W_out, mask) against
    the measured HBM copy bandwidth."""
    res = []
    Cout, R = 4096, 8192
    for dt in (torch.float32, torch.bfloat16):
        g = torch.Generator(device=str(dev)).manual_seed(11)
        W = torch.randn((Cout, R), generator=g, device=dev).to(dt)
        u = torch.rand((Cout, R), generator=g, device=dev)
        Wo = torch.empty_like(W)
        m = torch.empty((Cout, R), dtype=torch.uint8, device=dev)
        fn = lambda: cci.td_mask(W, 8, 2, 0.75, u, out=Wo, mask=m)  # noqa: E731
        fn()
        ms = statistics.median(time_device(fn, reps, flush, stream))
        nbytes = Cout * R * (2 * W.element_size() + 4 + 1)
        gbs = nbytes / (ms * 1e-3) / 1e9
        res.append({"dtype": str(dt).replace("torch.", ""), "ms": ms, "gbs": gbs,
                    "hbm_frac": gbs / float(measured_peaks()["hbm_gbs"]),
                    "dropped_frac_of_candidates": float((m == 0).sum().item()) / (Cout * R * 6 / 8)})
        del W, u, Wo, m
    return res


def run_pointwise_stack(cci, dev, stream, flush, reps=5):
    """The 34 pointwise convolutions of MobileNetV2 (batch 128, bf16, G = 8, K = 2:
    the paper's 75 % case), each on its own synthetic input, captured in CUDA
    graphs: fp32 outputs (the library's product), bf16 outputs with bias through
    the fused epilogue, cuDNN on the masked dense weights (bf16 output) and the
    library's tensor-core GEMM on the unpruned weights (fp32 output)."""
    layers = wl.mobilenetv2_pointwise_layers()
    plain, fused, dense, same, keep = [], [], [], [], []
    for c in layers:
        X, W = wl.conv_inputs(c, device=str(dev))
        v, i = cci.pack(W, c.G, c.K)
        Y = torch.empty((c.B, c.P, c.Q, c.Cout), dtype=torch.float32, device=dev)
        Yb = torch.empty((c.B, c.P, c.Q, c.Cout), dtype=torch.bfloat16, device=dev)
        bias = torch.zeros(c.Cout, dtype=torch.float32, device=dev)
        ws = cci.auto_workspace(X.dtype, c.Cin, c.R, c.Cout, c.G, c.K, dev)
        wsf = cci.new_workspace(cci.ALGO_DENSE_TC_WS, X.dtype, c.Cout, c.R, dev)
        Wm = torch.zeros((c.Cout, c.R), dtype=W.dtype, device=dev)
        Wm.view(c.Cout // c.G, c.G, c.R).scatter_(1, i.permute(0, 2, 1).long(), v.permute(0, 2, 1))
        w4 = Wm.view(c.Cout, 1, 1, c.Cin).permute(0, 3, 1, 2).contiguous(memory_format=torch.channels_last)
        x4 = X.permute(0, 3, 1, 2)
        del Wm
        keep.append((X, v, i, Y, Yb, bias, ws, wsf, w4, x4, W))
        plain.append(lambda c=c, X=X, v=v, i=i, Y=Y, ws=ws: cci.conv2d(
            X, v, i, c.Cout, c.G, c.K, 1, 1, (1, 1), (0, 0), out=Y, workspace=ws))
        fused.append(lambda c=c, X=X, v=v, i=i, Yb=Yb, ws=wsf, bias=bias: cci.conv2d_fused(
            X, v, i, c.Cout, c.G, c.K, 1, 1, (1, 1), (0, 0), bias=bias, out=Yb, workspace=ws))
        dense.append(lambda x4=x4, w4=w4: torch.nn.functional.conv2d(x4, w4))
        same.append(lambda c=c, X=X, W=W, Y=Y: cci.dense_conv2d_tc(X, W, c.Cout, 1, 1, out=Y))
    res = {"layers": len(layers), "batch": layers[0].B, "G": 8, "K": 2}
    for name, calls in (("ms", plain), ("fused_bf16_out_ms", fused), ("dense_cudnn_bf16_ms", dense),
                        ("same_kernel_dense_ms", same)):
        for f in calls:
            f()
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for f in calls:
                f()
        g.replay()
        torch.cuda.synchronize(dev)
        res[name] = statistics.median(time_device(g.replay, reps, flush, stream))
        del g
    nzf = sum(c.nz_flops() for c in layers)
    floor_ms = sum(layer_floor_us(c) for c in layers) * 1e-3
    res.update({"nz_gflop": nzf / 1e9, "nz_tflops": nzf / (res["ms"] * 1e-3) / 1e12,
                "dense_equiv_tflops": sum(c.dense_flops() for c in layers) / (res["ms"] * 1e-3) / 1e12,
                "roofline_floor_ms": floor_ms, "roofline_frac": floor_ms / res["ms"],
                "speedup_over_dense": res["dense_cudnn_bf16_ms"] / res["ms"],
                "fused_speedup_over_dense": res["dense_cudnn_bf16_ms"] / res["fused_bf16_out_ms"],
                "sparsity_gain": res["same_kernel_dense_ms"] / res["ms"]})
    del keep, plain, fused, dense, same
    torch.cuda.empty_cache()
    return res


def run_allocation_error(cci, dev, stream, flush, reps=5):
    """Eq. 1 measured: cci_pack_stats on 4096 x 8192 fp32 weight matrices whose
    zeros are independent with probability Ps (seeded), K = G (1 - Ps), next to the
    closed form (tests/golden/eq1_pd.txt); plus the counting kernel's rate
    (weights read once)."""
    eq1 = {}
    with open(os.path.join(ROOT, "tests", "golden", "eq1_pd.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                ps, g, _, pd = line.split()
                num, den = ps.split("/")
                eq1[(int(num) / int(den), int(g))] = float(pd)
    Cout, R = 4096, 8192
    rows = []
    for Ps in (0.5, 0.75, 0.875, 0.9375):
        g = torch.Generator(device=str(dev)).manual_seed(int(Ps * 10000))
        W = torch.randn((Cout, R), generator=g, device=dev)
        W[torch.rand((Cout, R), generator=g, device=dev) < Ps] = 0
        for G in (2, 4, 8, 16, 32, 64, 128, 256):
            K = G * (1 - Ps)
            if K < 1 or abs(K - round(K)) > 1e-9:
                continue
            K = int(round(K))
            counts = cci.pack_stats(W, G, K)
            nz, dropped = counts.cpu().tolist()
            rows.append({"Ps": Ps, "G": G, "K": K, "measured_Pd": dropped / nz, "eq1_Pd": eq1.get((Ps, G))})
        del W
    W = torch.randn((Cout, R), device=dev)
    counts = torch.zeros(2, dtype=torch.int64, device=dev)
    ms = statistics.median(time_device(lambda: cci.pack_stats(W, 8, 2, counts=counts), reps, flush, stream))
    return {"points": rows, "stats_kernel_ms_4096x8192_f32": ms,
            "stats_kernel_gbs": Cout * R * 4 / (ms * 1e-3) / 1e9,
            "what": "dropped nonzero weights / nonzero weights when packing iid-sparse matrices (Eq. 1)"}


def layer_floor_us(c) -> float:
    """The workload roofline of one layer: the slower of its nonzero flops at the
    CUDA-core FMA peak and its compressed bytes (X, Y, values + idx) at 8 TB/s."""
    es = 2 if c.dtype == "bf16" else 4
    nbytes = c.B * c.H * c.W * c.Cin * es + c.N * c.Cout * 4 + (c.Cout // c.G) * c.R * c.K * (es + 1)
    return max(c.nz_flops() / (ALU_PEAK_TFLOPS * 1e12), nbytes / (HBM_ROOF_GBS * 1e9)) * 1e6


def run_resnet_stack(cci, dev, stream, flush, reps=5):
    """The 52 convolutions of ResNet-50 after the stem, batch 128, bf16 inputs,
    G = 8, K in {1, 2, 4}: every layer once, in network order, each on its own
    synthetic input (the library's layers take bf16 activations and write fp32,
    so layer outputs are not chained).  Both sequences are captured in CUDA
    graphs (launch overhead out of the measurement) and replayed after an L2
    flush; the dense line is cuDNN on the masked dense bf16 weights (bf16 output)."""
    res = []
    for K in (1, 2, 4):
        layers = wl.resnet50_layers(K=K)
        ours_calls, dense_calls, same_calls = [], [], []
        keep = []
        for c in layers:
            X, W = wl.conv_inputs(c, device=str(dev))
            v, i = cci.pack(W, c.G, c.K)
            Y = torch.empty((c.B, c.P, c.Q, c.Cout), dtype=torch.float32, device=dev)
            ws = cci.auto_workspace(X.dtype, c.Cin, c.R, c.Cout, c.G, c.K, dev)
            wsf = cci.new_workspace(cci.ALGO_DENSE_TC_WS, X.dtype, c.Cout, c.R, dev)
            Wm = torch.zeros((c.Cout, c.R), dtype=W.dtype, device=dev)
            Wm.view(c.Cout // c.G, c.G, c.R).scatter_(1, i.permute(0, 2, 1).long(), v.permute(0, 2, 1))
            w4 = Wm.view(c.Cout, c.KH, c.KW, c.Cin).permute(0, 3, 1, 2).contiguous(
                memory_format=torch.channels_last)
            x4 = X.permute(0, 3, 1, 2)
            del Wm
            keep.append((X, v, i, Y, wsf, w4, x4, W, ws))
            ours_calls.append(lambda c=c, X=X, v=v, i=i, Y=Y, ws=ws: cci.conv2d(
                X, v, i, c.Cout, c.G, c.K, c.KH, c.KW, (c.stride, c.stride), (c.pad, c.pad), out=Y,
                workspace=ws))
            dense_calls.append(lambda c=c, x4=x4, w4=w4: torch.nn.functional.conv2d(
                x4, w4, stride=c.stride, padding=c.pad))
            same_calls.append(lambda c=c, X=X, W=W, Y=Y: cci.dense_conv2d_tc(
                X, W, c.Cout, c.KH, c.KW, (c.stride, c.stride), (c.pad, c.pad), out=Y))

        def ours():
            for f in ours_calls:
                f()

        def dense():
            for f in dense_calls:
                f()

        def same():
            for f in same_calls:
                f()

        ours()
        dense()
        same()
        torch.cuda.synchronize(dev)
        g_ours, g_dense, g_same = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_ours):
            ours()
        with torch.cuda.graph(g_dense):
            dense()
        with torch.cuda.graph(g_same):
            same()
        g_ours.replay()
        g_dense.replay()
        g_same.replay()
        torch.cuda.synchronize(dev)
        ms = statistics.median(time_device(g_ours.replay, reps, flush, stream))
        dms = statistics.median(time_device(g_dense.replay, reps, flush, stream))
        sms = statistics.median(time_device(g_same.replay, reps, flush, stream))
        per_layer = []
        if K == 2:  # each layer alone, for the breakdown
            for c, fo, fd, fs, kp in zip(layers, ours_calls, dense_calls, same_calls, keep):
                lm = statistics.median(time_device(fo, reps, flush, stream))
                ld = statistics.median(time_device(fd, reps, flush, stream))
                ls = statistics.median(time_device(fs, reps, flush, stream))
                per_layer.append({"layer": c.name, "ms": round(lm, 5), "floor_ms": round(layer_floor_us(c) * 1e-3, 5),
                                  "cudnn_ms": round(ld, 5), "same_kernel_dense_ms": round(ls, 5),
                                  "kernel": cci.kernel_name(torch.bfloat16, c.Cin, c.R, c.Cout, c.G, c.K,
                                                            cci.ALGO_AUTO)})
        # the same 52 layers chained through the fused epilogue: each layer reads
        # the bf16 output of the layer before it in its block (the first block its
        # synthetic input), adds a bias, applies ReLU (a and b) and writes bf16
        roles = wl.resnet50_roles()
        fused_calls, fkeep = [], []
        x_in = wl.draw_x((layers[0].B, layers[0].H, layers[0].W, layers[0].Cin), "relu_normal", "bf16",
                         1000 + K, str(dev))
        block_in, prev, pending = x_in, None, None
        for c, role, (X, v, i, Y, ws, w4, x4, _, _) in zip(layers, roles, keep):
            if role == "a" and pending is not None:  # a new block reads the last block's output
                block_in, pending = pending, None
            src = block_in if role in ("a", "proj") else prev
            assert tuple(src.shape) == (c.B, c.H, c.W, c.Cin), (c.name, tuple(src.shape))
            out = torch.empty((c.B, c.P, c.Q, c.Cout), dtype=torch.bfloat16, device=dev)
            bias = (torch.randn(c.Cout, generator=torch.Generator(device="cpu").manual_seed(c.seed)) * 0.1
                    ).to(dev)
            fkeep.append((out, bias))
            fused_calls.append(lambda c=c, src=src, v=v, i=i, out=out, ws=ws, bias=bias, relu=role in ("a", "b"):
                               cci.conv2d_fused(src, v, i, c.Cout, c.G, c.K, c.KH, c.KW, (c.stride,) * 2,
                                                (c.pad,) * 2, bias=bias, relu=relu, out=out, workspace=ws))
            if role in ("a", "b"):
                prev = out
            elif role == "c":
                pending = out
        for f in fused_calls:
            f()
        torch.cuda.synchronize(dev)
        assert torch.isfinite(fkeep[-1][0].float()).all()
        g_fused = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_fused):
            for f in fused_calls:
                f()
        g_fused.replay()
        torch.cuda.synchronize(dev)
        fms = statistics.median(time_device(g_fused.replay, reps, flush, stream))
        nzf = sum(c.nz_flops() for c in layers)
        dense_f = sum(c.dense_flops() for c in layers)
        floor_ms = sum(layer_floor_us(c) for c in layers) * 1e-3
        res.append({"G": 8, "K": K, "layers": len(layers), "batch": layers[0].B, "ms": ms,
                    "nz_gflop": nzf / 1e9, "nz_tflops": nzf / (ms * 1e-3) / 1e12,
                    "dense_equiv_tflops": dense_f / (ms * 1e-3) / 1e12,
                    "roofline_floor_ms": floor_ms, "roofline_frac": floor_ms / ms,
                    "dense_cudnn_bf16_ms": dms, "speedup_over_dense": dms / ms,
                    "same_kernel_dense_ms": sms, "sparsity_gain": sms / ms,
                    "fused_chained": {"ms": fms, "nz_tflops": nzf / (fms * 1e-3) / 1e12,
                                      "speedup_over_dense": dms / fms,
                                      "what": "cci_conv2d_fused per layer: bias, ReLU on the 1x1-reduce and 3x3 "
                                              "layers, bf16 output read by the next layer of the block "
                                              "(residual adds left out)"},
                    "captured": "CUDA graph of the 52 calls (ours) / 52 cuDNN convolutions (dense)"})
        if per_layer:
            res[-1]["per_layer"] = per_layer
        del keep, ours_calls, dense_calls, same_calls, g_ours, g_dense, g_same, fused_calls, fkeep, g_fused, block_in, prev, pending, x_in
        torch.cuda.empty_cache()
    return res


def main():
    args = parse()
    if args.impl == "reference":
        # the CPU oracle needs no process group: rank 0 runs it, other ranks exit
        return run_reference(args, int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")))
    rank, world, local = dist_init(args)
    rc = run_ours(args, rank, world, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return rc


if __name__ == "__main__":
    sys.exit(main())
