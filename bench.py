"""Benchmark of the FLARE++ routing chain on GB300: one JSON line on stdout.

A step is one flarepp_route_fwd over the whole workload (encode call 1, combine, encode
call 2, combine, decode call 3; Sec. 3.2). The default workload is the 3D-mesh shape
B=1, H=8, N=1,048,576, M=512, D=32, bf16, with clustered keys; its five B*H*N*D tensors
(2.7 GB) are far larger than the 129 MB L2, so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Under torchrun every rank runs an independent replica on its own GPU (the chain has no
cross-GPU exchange on one box); rank 0 prints the aggregate.
"""
import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_11519_gb300 import inputs  # noqa: E402

METRIC = "routed tokens·heads/sec for the 3-call FLARE++ chain; % of roofline"
UNIT = "token·heads/s"
# the files that fix what a kernel launch reads and writes: the kernels and the plan that
# sets their launch configuration (the C ABI's argument handling is not among them)
KERNEL_SOURCES = tuple("paper_2608_11519_gb300/csrc/" + f for f in (
    "combine.cu", "flarepp_internal.h", "plan.cu", "simt_f32.cu", "simt_kernels.cuh",
    "tc_kernels.cu", "tc_ptx.cuh"))
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                  "source": "fallback"}


# ------------------------------------------------------------------ helpers

def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        d["source"] = "measured"
        return d
    return dict(FALLBACK_PEAKS)


# A timed region at least this long runs the tensor cores into the power cap, as the
# driver's sustained GEMM loop does; a shorter one sees the burst rate.
SUSTAINED_REGION_S = 2.0


def tc_peak_for(peaks, timed_s, bf16=True):
    """The dense bf16 tensor peak that a kernel timed over a region of ``timed_s`` seconds is
    compared with, and its name: the measured burst figure unless the timed region is
    seconds-long (SUSTAINED_REGION_S or more), then the sustained one."""
    if not bf16:
        return None, None
    kind = "bf16_tflops_sustained" if timed_s >= SUSTAINED_REGION_S else "bf16_tflops"
    return peaks[kind], kind + " (" + peaks["source"] + ")"


def kernel_source_hash():
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(os.path.basename(rel).encode() + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload, stage, how=False):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current
    kernel sources (else None); with ``how``, also the record's note on how it was taken."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    e = None
    if os.path.exists(p):
        with open(p) as f:
            e = json.load(f).get(workload, {}).get(stage)
        if e and e.get("source_hash") != kernel_source_hash():
            e = None
    value = e.get("dram_bytes_per_launch") if e else None
    return (value, e.get("how") if e else None) if how else value


def stage_work(w, stage):
    """Algorithmic flops and bytes of one launch of a stage.

    encode (calls 1, 2): S = s Q K^T and O = P V over all tokens: 4*B*H*N*M*D flops; reads
      the call's K and V: 2*B*H*N*D elements.
    decode (call 3): S^T = s K Q^T and Y = P Z: 4*B*H*N*M*D flops; reads K, writes Y:
      2*B*H*N*D elements.
    combine: reads the chunk partials, writes Q or Z (latent-sized; no algorithmic tokens).
    """
    tok = w.B * w.H * w.N
    flops = 4.0 * tok * w.M * w.D
    byts = 2.0 * tok * w.D * w.elt_bytes
    if stage.startswith("combine"):
        return 0.0, 2.0 * w.B * w.H * w.M * w.D * 4
    return flops, byts


class NvmlSampler:
    """SM clock, power and clock-event reasons read through NVML's C API (read-only queries)
    by a thread that polls every 2 ms between start() and stop(), so that even a timed
    region of a few tens of milliseconds gets many samples."""

    # clock-event reason bits of nvml.h
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, cuda_index, lib=None):
        import ctypes
        import threading
        self.ct = ctypes
        self.nvml = lib if lib is not None else ctypes.CDLL("libnvidia-ml.so.1")
        if self.nvml.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        self.dev = ctypes.c_void_p()
        vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").strip()
        ent = vis.split(",")[cuda_index].strip() if vis else str(cuda_index)
        if ent.isdigit():
            rc = self.nvml.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(int(ent)),
                                                         ctypes.byref(self.dev))
        else:
            rc = self.nvml.nvmlDeviceGetHandleByUUID(ent.encode(), ctypes.byref(self.dev))
        if rc != 0:
            raise OSError(f"no NVML handle for CUDA device {cuda_index}")
        self.get_reasons = getattr(self.nvml, "nvmlDeviceGetCurrentClocksEventReasons", None) \
            or self.nvml.nvmlDeviceGetCurrentClocksThrottleReasons
        self.smax = self._clock(self.nvml.nvmlDeviceGetMaxClockInfo)
        self.samples = []
        self.stop_flag = threading.Event()
        self.thread = threading.Thread(target=self._poll, daemon=True)

    def _clock(self, fn):
        v = self.ct.c_uint()
        return float(v.value) if fn(self.dev, 1, self.ct.byref(v)) == 0 else None  # 1: SM

    def _poll(self):
        ct = self.ct
        mw, reasons = ct.c_uint(), ct.c_ulonglong()
        while not self.stop_flag.is_set():
            sm = self._clock(self.nvml.nvmlDeviceGetClockInfo)
            pw = mw.value / 1000.0 if self.nvml.nvmlDeviceGetPowerUsage(
                self.dev, ct.byref(mw)) == 0 else None
            rs = reasons.value if self.get_reasons(self.dev, ct.byref(reasons)) == 0 else 0
            if sm is not None:
                self.samples.append((sm, pw, rs))
            time.sleep(0.002)

    def start(self):
        self.thread.start()

    def stop(self):
        self.stop_flag.set()
        self.thread.join(timeout=5)
        self.nvml.nvmlShutdown()
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.smax, "reasons": ["no samples"]}
        reasons = sorted({name for _, _, r in self.samples
                          for bit, name in self.REASONS.items() if r & bit})
        power = [p for _, p, _ in self.samples if p is not None]
        return {"sm_mhz": statistics.median(s for s, _, _ in self.samples),
                "sm_max_mhz": self.smax, "power_w_max": max(power) if power else None,
                "power_w_median": statistics.median(power) if power else None,
                "samples": len(self.samples), "source": "nvml, 2 ms polling",
                "reasons": reasons}


class ClockSampler:
    """SM clocks and throttle reasons during the timed region: NVML polling where the driver's
    NVML library loads, else nvidia-smi sampling every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self):
        self.proc = None
        self.path = None
        self.nvml = None

    def start(self, cuda_index=0):
        try:
            self.nvml = NvmlSampler(cuda_index)
            self.nvml.start()
            return
        except (OSError, AttributeError, IndexError):
            self.nvml = None
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=self.out, stderr=subprocess.DEVNULL)
            time.sleep(0.3)  # let nvidia-smi start before the timed region
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self, gpu_index):
        if self.nvml is not None:
            return self.nvml.stop()
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        sm, smax, reasons, power = [], [], set(), []
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    if int(parts[0]) != gpu_index:
                        continue
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                    power.append(float(parts[3]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [s for s in sm if s > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax),
                "power_w_max": max(power) if power else None, "samples": len(sm),
                "source": "nvidia-smi, 200 ms sampling", "reasons": sorted(reasons)}


def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """The largest of the ranks' values (every rank gets it): the job's time is its slowest
    rank's. A device tensor under NCCL, a host tensor under gloo."""
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ CPU baseline (oracle)

def oracle_call(f, w, variant):
    """The float64 oracle of the benchmarked variant on numpy inputs."""
    import oracle
    if variant == "flare":
        return oracle.flare(f["seeds"], f["K"], f["V"], w.scale)
    if variant == "shared":
        return oracle.route(f["seeds"], f["K"], f["V"], f["K"], f["V"], w.scale)
    if variant == "train":  # the oracle's backward runs the forward itself
        dY = np.ones_like(f["K"])
        return oracle.route_bwd(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale, dY)
    return oracle.route(f["seeds"], f["Kt"], f["Vt"], f["K"], f["V"], w.scale)


def cpu_oracle_sample(w, target_s, seed=0, variant="flarepp"):
    """Time the float64 oracle on one (b, h) slice with a token prefix of the workload,
    sized from a short probe to take about ``target_s`` seconds. Returns a cpu_baseline dict."""
    import oracle
    x = inputs.make_inputs(w.with_(B=1, H=1, N=min(w.N, 4096)), seed)
    f = inputs.to_f64_numpy(x)
    t0 = time.perf_counter()
    oracle_call(f, w, variant)
    probe = time.perf_counter() - t0
    n = int(min(w.N, max(1024, f["K"].shape[2] * target_s / max(probe, 1e-3))))
    x = inputs.make_inputs(w.with_(B=1, H=1, N=n), seed)
    f = inputs.to_f64_numpy(x)
    t0 = time.perf_counter()
    oracle_call(f, w, variant)
    dt = time.perf_counter() - t0
    return {"value": n / dt, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "sample": f"one head, N={n} tokens of the {w.name} shape (M={w.M}, D={w.D}), "
                      f"float64, {dt:.2f} s"}


# ------------------------------------------------------------------ reference arm

def reference_step(args, w, n):
    """One step of the reference arm on an n-token sample of the workload: returns the call,
    the heads it routes and a description of the sample."""
    import oracle
    if args.variant == "mixer_train":
        # the layer's forward and backward on one batch element
        m = inputs.to_f64_numpy(inputs.make_mixer_inputs(w.with_(B=1, N=n), args.seed, "cpu"))
        dO = np.random.default_rng(args.seed).standard_normal(m["X"].shape)
        return (lambda: oracle.mixer_bwd(m["X"], m["W_in"], m["Wo"], m["seeds"], w.scale, dO),
                w.H, f"one batch element, N={n} tokens, H={w.H} heads of the {w.name} shape "
                     f"(M={w.M}, D={w.D}), float64 oracle (forward and backward), per step")
    if args.variant.startswith("mixer"):
        # the whole layer on one batch element: all H heads of n tokens
        m = inputs.to_f64_numpy(inputs.make_mixer_inputs(
            w.with_(B=1, N=n), args.seed, "cpu", 2 if args.variant == "mixer_shared" else 4))
        return (lambda: oracle.mixer(m["X"], m["W_in"], m["Wo"], m["seeds"], w.scale),
                w.H, f"one batch element, N={n} tokens, H={w.H} heads of the {w.name} shape "
                     f"(M={w.M}, D={w.D}), float64 oracle on the host cores, per step")
    f = inputs.to_f64_numpy(inputs.make_inputs(w.with_(B=1, H=1, N=n), args.seed))
    return (lambda: oracle_call(f, w, args.variant), 1,
            f"one head, N={n} tokens of the {w.name} shape (M={w.M}, D={w.D}), float64 "
            f"oracle on the host cores, per step")


def run_reference(args, w):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    # the sample: at most --ref-tokens tokens, fewer when the warm-up and timed steps would
    # take more than about --ref-seconds (a probe on 1024 tokens gives the time per token),
    # but no fewer than 1024 tokens, so that the tokens still outnumber the routes
    cap = int(min(w.N, args.ref_tokens))
    n0 = min(cap, 1024)
    probe_step = reference_step(args, w, n0)[0]
    t0 = time.perf_counter()
    probe_step()
    per_token = (time.perf_counter() - t0) / n0
    del probe_step
    calls = max(1, args.steps + args.warmup)
    n = int(min(cap, max(n0, args.ref_seconds / (calls * per_token))))
    step, heads, sample = reference_step(args, w, n)
    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = (time.perf_counter() - t0) / args.steps
    value = heads * n / dt
    metric = {"flare": FLARE_METRIC, "train": TRAIN_METRIC, "mixer": MIXER_METRIC,
              "mixer_shared": MIXER_METRIC,
              "mixer_train": MIXER_TRAIN_METRIC}.get(args.variant, METRIC)
    line = {"impl": "reference", "metric": metric, "value": value, "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": arm_config(w, args.variant, world, args.l2),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.max_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ our arm

FLARE_METRIC = "routed tokens·heads/sec for the 2-call FLARE layer (fixed queries); % of roofline"


L2_BYTES = 129e6
FLUSH_BYTES = 256 << 20  # twice the L2


def chain_inputs_fit_l2(w, variant):
    """Whether the chain's streamed tensors (K~, V~, K, V and Y; K, V and Y when shared) stay
    within twice the L2, so that a warm L2 could hold a large share of them across steps."""
    n = 3 if variant == "shared" else 5
    return n * w.B * w.H * w.N * w.D * w.elt_bytes <= 2 * L2_BYTES


def l2_mode(mode, w, variant):
    """'flush' or 'warm' for the chain variants: `auto` flushes exactly when the streamed
    tensors are near the L2's size, where leftover lines would flatter a step."""
    if mode == "auto":
        return "flush" if chain_inputs_fit_l2(w, variant) else "warm"
    return mode


def l2_flush_buffer(mode, w, variant, dev):
    """A buffer larger than the L2 that each timed step overwrites first, or None."""
    if l2_mode(mode, w, variant) != "flush":
        return None
    return torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=dev)


def arm_config(w, variant, world, l2="auto"):
    """The `config` of a bench line; both arms of one variant print the same one."""
    cfg = {"workload": w.name, "variant": variant, "B": w.B, "H": w.H, "N": w.N, "M": w.M,
           "D": w.D}
    tok = w.B * w.H * w.N
    big = "inputs larger than L2 (no flush)"
    if variant in ("flarepp", "shared"):
        cfg["keys"] = f"clustered, {w.n_centres} centres" if w.n_centres else "iid"
        if l2_mode(l2, w, variant) == "flush":
            cfg["l2"] = "flushed before each step (256 MiB written between the step's events)"
        elif chain_inputs_fit_l2(w, variant):
            cfg["l2"] = "warm: no flush, inputs near L2 size"
        else:
            cfg["l2"] = big
    elif variant == "flare":
        cfg["queries"] = "the workload's seeds, as learned queries"
        cfg["l2"] = big if 3 * tok * w.D * w.elt_bytes > 2 * 129e6 else "inputs near L2 size"
    elif variant == "train":
        cfg["l2"] = big
    else:  # the mixer variants
        cfg["C"] = w.H * w.D
        cfg["projections"] = 2 if variant == "mixer_shared" else 4
        cfg["l2"] = big
    cfg["parallelism"] = f"replicas x{world}"
    return cfg


def chain_bwd_launches(w):
    """Kernels of one chain backward: on the tensor-core path c3, two operand copies, R3 and
    its reduce, T23 (with, for D <= 32, the range and flag kernels, the w dZ operand and the
    merged pass before it), R2 and its reduce, T1, R1 and the seeds' reduce; on the
    CUDA-core path c3 and three route passes, two token passes and three reduces."""
    if w.dtype != "bf16":
        return 9
    return 11 + (4 if w.D <= 32 else 0)


def chain_fwd_launches(w):
    """Kernels of one chain forward: on the tensor-core path each encode and the decode is a
    fast kernel followed by its safe kernel (which returns at once unless the fast one
    overflowed), plus two merges and, for a negative scale, the negation of the seeds: 8
    (9); on the CUDA-core path encode, merge, encode, merge, decode: 5."""
    if w.dtype != "bf16":
        return 5
    return 8 + (1 if w.scale < 0 else 0)


def flare_launches(w):
    """Kernels of one FLARE call: encode, merge and decode (the encode and decode as a fast
    and a safe kernel on the tensor-core path), plus the negation of the bf16 queries when
    the scale is negative."""
    if w.dtype != "bf16":
        return 3
    return 5 + (1 if w.scale < 0 else 0)


def run_flare(args, w, flarepp, world, rank, dev, peaks, x, Y, ws, stream):
    """FLARE (Sec. 3, eq. prelim_flare_sdpa) with the seeds as the learned queries: whole
    calls timed with CUDA events (a call is one encode, one merge and one decode)."""
    Q, K, V = x["seeds"], x["K"], x["V"]
    for _ in range(args.warmup):
        flarepp.flare_fwd(Q, K, V, w.scale, Y=Y, workspace=ws, stream=stream)
    torch.cuda.synchronize(dev)
    clocks = ClockSampler()
    if rank == 0:
        clocks.start(dev.index)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    t0.record(stream)
    for _ in range(args.steps):
        flarepp.flare_fwd(Q, K, V, w.scale, Y=Y, workspace=ws, stream=stream)
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop(dev.index) if rank == 0 else None
    ms = max_over_ranks(t0.elapsed_time(t1), world) / args.steps
    tok = w.B * w.H * w.N
    value = tok * world / (ms * 1e-3)
    # algorithmic work of a call: 8 BNMHD flops (two token-latent SDPA calls); K, V read
    # and Y written, 3 BHND elements
    flops = 8.0 * tok * w.M * w.D
    byts = 3.0 * tok * w.D * w.elt_bytes
    tc_peak, tc_kind = tc_peak_for(peaks, ms * args.steps * 1e-3, w.dtype == "bf16")
    bw = peaks["hbm_gbs"]
    t_tc = flops / (tc_peak * 1e12) if tc_peak else 0.0
    t_mem = byts / (bw * 1e9)
    if t_tc >= t_mem and tc_peak:
        roof = {"bound": "tensor", "achieved": flops / (ms * 1e-3) / 1e12, "peak": tc_peak,
                "unit": "TFLOP/s", "peak_kind": tc_kind}
    else:
        roof = {"bound": "hbm", "achieved": byts / (ms * 1e-3) / 1e9, "peak": bw, "unit": "GB/s",
                "peak_kind": "hbm_gbs (" + peaks["source"] + ")"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["kernel"] = "whole call (encode, merge, decode)"
    roof["ms_per_launch"] = ms
    roof["algorithmic_flops_per_launch"] = flops
    roof["algorithmic_bytes_per_launch"] = byts
    roof["traffic"] = None
    e2e = None
    if not args.no_e2e:
        # through the library's host entry: copies overlapped with the compute by head groups
        xh = {k: x[k].to("cpu").pin_memory() for k in ("seeds", "K", "V")}
        Yh = torch.empty(Y.shape, dtype=Y.dtype, pin_memory=True)
        hws = flarepp.Workspace()

        def e2e_call():
            flarepp.flare_fwd_host(xh["seeds"], xh["K"], xh["V"], w.scale, Y_host=Yh,
                                   device=dev, workspace=hws, stream=stream)

        for _ in range(2):
            e2e_call()
        n_e2e = max(1, min(args.steps, args.e2e_steps))
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        barrier(world)
        torch.cuda.synchronize(dev)
        e0.record(stream)
        for _ in range(n_e2e):
            e2e_call()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / n_e2e, world)
        e2e = {"value": tok * world / (e2e_ms * 1e-3), "unit": UNIT, "ms_per_step": e2e_ms,
               "steps": n_e2e, "copies": "overlapped with the compute by head groups",
               "h2d_bytes_per_step": sum(t.numel() * t.element_size() for t in xh.values()),
               "d2h_bytes_per_step": Yh.numel() * Yh.element_size()}
        del xh, Yh, hws
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_oracle_sample(w, args.cpu_seconds, args.seed, "flare")
    if rank == 0:
        line = {
            "metric": FLARE_METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
            "config": arm_config(w, "flare", world),
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": flare_launches(w) * args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


TRAIN_METRIC = ("routed tokens·heads/sec for a training step of the 3-call FLARE++ chain "
                "(forward with saved state + backward); % of roofline")


def run_train(args, w, flarepp, world, rank, dev, peaks, x, Y, ws, stream):
    """A training step of the chain: flarepp_route_fwd_train then flarepp_route_bwd (App. A.5)
    on device-resident inputs and output gradient, each part bracketed by CUDA events."""
    args_ = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    dY = inputs.make_output_grad(w, args.seed + rank, device=dev)
    saved = None
    ws_b = flarepp.Workspace()
    grads = tuple(torch.empty_like(t) for t in args_)

    def step(ev=None):
        nonlocal saved
        if ev:
            ev[0].record(stream)
        _, saved = flarepp.route_fwd_train(*args_, w.scale, Y=Y, saved=saved, workspace=ws,
                                           stream=stream)
        if ev:
            ev[1].record(stream)
        flarepp.route_bwd(*args_, Y, dY, saved, w.scale, grads=grads, workspace=ws_b,
                          stream=stream)
        if ev:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    clocks = ClockSampler()
    if rank == 0:
        clocks.start(dev.index)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    t0.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop(dev.index) if rank == 0 else None
    ms = max_over_ranks(t0.elapsed_time(t1), world) / args.steps
    fwd_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps
    bwd_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / args.steps
    tok = w.B * w.H * w.N
    value = tok * world / (ms * 1e-3)
    # backward algorithmic work: per SDPA, S (recomputed), dP, dV, dK and dQ, 2 NMD flops
    # each: 30 BNMHD over the three calls; reads Kt, Vt, K, V, Y, dY and writes four
    # gradients: 10 BHND elements
    flops = 30.0 * tok * w.M * w.D
    byts = 10.0 * tok * w.D * w.elt_bytes
    tc_peak, tc_kind = tc_peak_for(peaks, ms * args.steps * 1e-3, w.dtype == "bf16")
    bw = peaks["hbm_gbs"]
    t_tc = flops / (tc_peak * 1e12) if tc_peak else 0.0
    t_mem = byts / (bw * 1e9)
    if t_tc >= t_mem and tc_peak:
        roof = {"bound": "tensor", "achieved": flops / (bwd_ms * 1e-3) / 1e12, "peak": tc_peak,
                "unit": "TFLOP/s", "peak_kind": tc_kind}
    else:
        roof = {"bound": "hbm", "achieved": byts / (bwd_ms * 1e-3) / 1e9, "peak": bw,
                "unit": "GB/s", "peak_kind": "hbm_gbs (" + peaks["source"] + ")"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["kernel"] = "backward (all passes)"
    roof["ms_per_launch"] = bwd_ms
    roof["algorithmic_flops_per_launch"] = flops
    roof["algorithmic_bytes_per_launch"] = byts
    roof["traffic"] = None
    t_step = max((12.0 + 30.0) * tok * w.M * w.D / ((tc_peak or peaks["bf16_tflops"]) * 1e12),
                 15.0 * tok * w.D * w.elt_bytes / (bw * 1e9))
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_oracle_sample(w, args.cpu_seconds, args.seed, "train")
    if rank == 0:
        line = {
            "metric": TRAIN_METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
            "config": arm_config(w, "train", world),
            "stage_ms": {"forward_train": fwd_ms, "backward": bwd_ms},
            "roofline": roof,
            "step_roofline": {"roofline_us": t_step * 1e6, "frac": t_step / (ms * 1e-3),
                              "flops": "42 BNMHD", "tensors": 15},
            "cpu_baseline": cpu, "e2e": None, "clocks": clk,
            "gpu_launches": (chain_fwd_launches(w) + chain_bwd_launches(w)) * args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


MIXER_METRIC = ("routed tokens·heads/sec for the FLARE++ mixer layer (projections, 3-call chain, "
                "output projection); % of roofline")


def mixer_cpu_sample(w, target_s, seed, n_proj):
    """The oracle's mixer on one batch element with a token prefix sized from a short probe."""
    import oracle
    probe_n = min(w.N, 2048)
    x = inputs.to_f64_numpy(inputs.make_mixer_inputs(w.with_(B=1, N=probe_n), seed, "cpu", n_proj))
    t0 = time.perf_counter()
    oracle.mixer(x["X"], x["W_in"], x["Wo"], x["seeds"], w.scale)
    probe = time.perf_counter() - t0
    n = int(min(w.N, max(512, probe_n * target_s / max(probe, 1e-3))))
    x = inputs.to_f64_numpy(inputs.make_mixer_inputs(w.with_(B=1, N=n), seed, "cpu", n_proj))
    t0 = time.perf_counter()
    oracle.mixer(x["X"], x["W_in"], x["Wo"], x["seeds"], w.scale)
    dt = time.perf_counter() - t0
    return {"value": w.H * n / dt, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "sample": f"one batch element, N={n} tokens of the {w.name} shape (H={w.H}, M={w.M}, "
                      f"D={w.D}), float64, {dt:.2f} s"}


MIXER_TRAIN_METRIC = ("routed tokens·heads/sec for a training step of the FLARE++ mixer layer "
                      "(forward with saved state + backward); % of roofline")


def run_mixer_train(args, w, flarepp, world, rank, dev, peaks, stream):
    """A training step of the mixer layer: flarepp_mixer_fwd_train then flarepp_mixer_bwd, each
    bracketed by CUDA events, on device-resident inputs and output gradient."""
    x = inputs.make_mixer_inputs(w, args.seed + rank, device=dev, n_proj=4)
    dO = inputs.make_output_grad(w.with_(H=1, D=w.H * w.D), args.seed + rank,
                                 device=dev).reshape(x["X"].shape)
    O = torch.empty_like(x["X"])
    ws_f, ws_b = flarepp.Workspace(), flarepp.Workspace()
    grads = (torch.empty_like(x["X"]), torch.empty_like(x["W_in"]), torch.empty_like(x["Wo"]),
             torch.empty_like(x["seeds"]))
    saved = None

    def step(ev=None):
        nonlocal saved
        if ev:
            ev[0].record(stream)
        _, saved = flarepp.mixer_fwd_train(x["X"], x["W_in"], x["Wo"], x["seeds"], w.scale, O=O,
                                           saved=saved, workspace=ws_f, stream=stream)
        if ev:
            ev[1].record(stream)
        flarepp.mixer_bwd(x["X"], x["W_in"], x["Wo"], x["seeds"], saved, dO, w.scale,
                          grads=grads, workspace=ws_b, stream=stream)
        if ev:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    clocks = ClockSampler()
    if rank == 0:
        clocks.start(dev.index)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    t0.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop(dev.index) if rank == 0 else None
    ms = max_over_ranks(t0.elapsed_time(t1), world) / args.steps
    fwd_ms = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps
    bwd_ms = sum(e[1].elapsed_time(e[2]) for e in evs) / args.steps
    tok = w.B * w.H * w.N
    BN, C = w.B * w.N, w.H * w.D
    # backward algorithmic flops: the chain's 30 BNMHD, and per token 2 C^2 (dY) + 2 C^2 (dWo)
    # + 2 C (4C) each for dW_in and dX (the projections' recompute is not counted)
    flops = 30.0 * tok * w.M * w.D + BN * (4.0 * C * C + 16.0 * C * C)
    tc_peak, tc_kind = tc_peak_for(peaks, ms * args.steps * 1e-3)
    roof = {"bound": "tensor", "achieved": flops / (bwd_ms * 1e-3) / 1e12, "peak": tc_peak,
            "unit": "TFLOP/s", "peak_kind": tc_kind}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["kernel"] = "mixer backward (all launches)"
    roof["ms_per_launch"] = bwd_ms
    roof["algorithmic_flops_per_launch"] = flops
    roof["traffic"] = None
    if rank == 0:
        line = {
            "metric": MIXER_TRAIN_METRIC, "value": tok * world / (ms * 1e-3), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": arm_config(w, "mixer_train", world),
            "stage_ms": {"forward_train": fwd_ms, "backward": bwd_ms}, "roofline": roof,
            "cpu_baseline": None, "e2e": None, "clocks": clk,
            # forward: projection, the chain's kernels, output projection; backward: two
            # weight transposes, dY, dWo and its reduce, the chain's backward, dW_in and its
            # reduce, dX
            "gpu_launches": (2 + chain_fwd_launches(w) + 8 + chain_bwd_launches(w))
                            * args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def run_mixer(args, w, flarepp, world, rank, dev, peaks, stream):
    """The FLARE++ mixer layer (Fig. 1) on device-resident inputs, each stage bracketed by the
    library's own events."""
    n_proj = 2 if args.variant == "mixer_shared" else 4
    x = inputs.make_mixer_inputs(w, args.seed + rank, device=dev, n_proj=n_proj)
    O = torch.empty_like(x["X"])
    ws = flarepp.Workspace()
    call = lambda ev=None: flarepp.mixer_fwd(x["X"], x["W_in"], x["Wo"], x["seeds"], w.scale,
                                             O=O, workspace=ws, stream=stream, events=ev)
    for _ in range(args.warmup):
        call()
    torch.cuda.synchronize(dev)
    evs = [flarepp.MixerEvents(stream) for _ in range(args.steps)]
    clocks = ClockSampler()
    if rank == 0:
        clocks.start(dev.index)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize(dev)
    t0.record(stream)
    for i in range(args.steps):
        call(evs[i])
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clk = clocks.stop(dev.index) if rank == 0 else None
    ms = max_over_ranks(t0.elapsed_time(t1), world) / args.steps
    stage_ms = {s: 0.0 for s in flarepp.MIXER_STAGES}
    for e in evs:
        for s, v in e.stage_ms().items():
            stage_ms[s] += v / args.steps
    tok = w.B * w.H * w.N
    BN, C = w.B * w.N, w.H * w.D
    e = w.elt_bytes
    # algorithmic work of each stage (the stages as built, each reading and writing HBM)
    work = {
        "projection": (2.0 * BN * C * n_proj * C, (1 + n_proj) * BN * C * e),
        "chain": (12.0 * tok * w.M * w.D, (3 if n_proj == 2 else 5) * tok * w.D * e),
        "output": (2.0 * BN * C * C, 2 * BN * C * e),
    }
    tc_peak, tc_kind = tc_peak_for(peaks, ms * args.steps * 1e-3)
    bw = peaks["hbm_gbs"]
    roof_t = {s: max(f / (tc_peak * 1e12), b / (bw * 1e9)) for s, (f, b) in work.items()}
    dominant = max(stage_ms, key=stage_ms.get)
    f, b = work[dominant]
    t_dom = stage_ms[dominant] * 1e-3
    if f / (tc_peak * 1e12) >= b / (bw * 1e9):
        roof = {"bound": "tensor", "achieved": f / t_dom / 1e12, "peak": tc_peak,
                "unit": "TFLOP/s", "peak_kind": tc_kind}
    else:
        roof = {"bound": "hbm", "achieved": b / t_dom / 1e9, "peak": bw, "unit": "GB/s",
                "peak_kind": "hbm_gbs (" + peaks["source"] + ")"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["kernel"] = dominant
    roof["ms_per_launch"] = stage_ms[dominant]
    roof["algorithmic_flops_per_launch"] = f
    roof["algorithmic_bytes_per_launch"] = b
    roof["traffic"] = None
    stage_frac = {s: roof_t[s] / (stage_ms[s] * 1e-3) for s in stage_ms}
    layer = {"roofline_us": sum(roof_t.values()) * 1e6,
             "frac": sum(roof_t.values()) / (ms * 1e-3),
             "stage_frac": stage_frac,
             "note": "sum of the stages' own rooflines (each stage streams its tensors through HBM)"}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = mixer_cpu_sample(w, args.cpu_seconds, args.seed, n_proj)
    if rank == 0:
        line = {
            "metric": MIXER_METRIC, "value": tok * world / (ms * 1e-3), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": arm_config(w, args.variant, world),
            "stage_ms": stage_ms, "roofline": roof, "layer_roofline": layer,
            "cpu_baseline": cpu, "e2e": None, "clocks": clk,
            "gpu_launches": (2 + chain_fwd_launches(w)) * args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def run_ours(args, w):
    from paper_2608_11519_gb300 import flarepp

    world, rank, local = dist_setup(args.gpus)
    dev = torch.device("cuda", local if world > 1 else 0)
    flarepp.load()
    peaks = load_peaks()

    x = inputs.make_inputs(w, args.seed + rank, device=dev)
    Y = torch.empty_like(x["K"])
    ws = flarepp.Workspace()
    stream = torch.cuda.current_stream(dev)
    args_ = (x["seeds"], x["Kt"], x["Vt"], x["K"], x["V"])
    if args.variant == "shared":  # Kt, Vt tied to K, V (App. cost_model)
        args_ = (x["seeds"], x["K"], x["V"], x["K"], x["V"])
    if args.variant == "flare":
        return run_flare(args, w, flarepp, world, rank, dev, peaks, x, Y, ws, stream)
    if args.variant == "train":
        return run_train(args, w, flarepp, world, rank, dev, peaks, x, Y, ws, stream)
    if args.variant in ("mixer", "mixer_shared"):
        del x, Y
        return run_mixer(args, w, flarepp, world, rank, dev, peaks, stream)
    if args.variant == "mixer_train":
        del x, Y
        return run_mixer_train(args, w, flarepp, world, rank, dev, peaks, stream)

    for _ in range(args.warmup):
        flarepp.route_fwd(*args_, scale=w.scale, Y=Y, workspace=ws, stream=stream)
    torch.cuda.synchronize(dev)

    # the timed region: whole calls of the public entry, no events inside a step; with the L2
    # flushed, each step is bracketed by its own events and the flush runs between them
    flush = l2_flush_buffer(args.l2, w, args.variant, dev)
    clocks = ClockSampler()
    if rank == 0:
        clocks.start(dev.index)
    barrier(world)
    torch.cuda.synchronize(dev)
    if flush is None:
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for i in range(args.steps):
            flarepp.route_fwd(*args_, scale=w.scale, Y=Y, workspace=ws, stream=stream)
        t_end.record(stream)
        torch.cuda.synchronize(dev)
        total_ms = t_start.elapsed_time(t_end)
    else:
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        for i in range(args.steps):
            flush.fill_(i & 0x7F)
            evs[i][0].record(stream)
            flarepp.route_fwd(*args_, scale=w.scale, Y=Y, workspace=ws, stream=stream)
            evs[i][1].record(stream)
        torch.cuda.synchronize(dev)
        total_ms = sum(a.elapsed_time(b) for a, b in evs)
    barrier(world)
    clk = clocks.stop(dev.index) if rank == 0 else None
    total_ms = max_over_ranks(total_ms, world)
    ms_per_step = total_ms / args.steps

    # per-stage durations: separate calls that record events between the stages (the events
    # keep each stage's kernels from overlapping the next stage's start)
    n_prof = max(1, min(args.steps, 20))
    ev_sets = [flarepp.StageEvents(stream) for _ in range(n_prof)]
    for i in range(n_prof):
        if flush is not None:
            flush.fill_(i & 0x7F)
        flarepp.route_fwd_profiled(*args_, ev_sets[i], scale=w.scale, Y=Y, workspace=ws)
    torch.cuda.synchronize(dev)
    stage_ms = {s: 0.0 for s in flarepp.STAGES}
    for e in ev_sets:
        for s, v in e.stage_ms().items():
            stage_ms[s] += v / n_prof
    dominant = max(stage_ms, key=stage_ms.get)
    flops, byts = stage_work(w, dominant)
    t_dom = stage_ms[dominant] * 1e-3
    tc_peak, tc_kind = tc_peak_for(peaks, total_ms * 1e-3, w.dtype == "bf16")
    bw_peak = peaks["hbm_gbs"]
    t_tc = flops / (tc_peak * 1e12) if tc_peak else 0.0
    t_mem = byts / (bw_peak * 1e9)
    if t_tc >= t_mem and tc_peak:
        roof = {"bound": "tensor", "achieved": flops / t_dom / 1e12, "peak": tc_peak,
                "unit": "TFLOP/s", "peak_kind": tc_kind}
    else:
        roof = {"bound": "hbm", "achieved": byts / t_dom / 1e9, "peak": bw_peak, "unit": "GB/s",
                "peak_kind": "hbm_gbs (" + peaks["source"] + ")"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    if roof["bound"] == "tensor" and peaks.get("bf16_tflops_sustained"):
        roof["frac_vs_sustained_peak"] = roof["achieved"] / peaks["bf16_tflops_sustained"]
    roof["timed_region_s"] = total_ms * 1e-3
    roof["kernel"] = dominant
    roof["ms_per_launch"] = stage_ms[dominant]
    roof["algorithmic_flops_per_launch"] = flops
    roof["algorithmic_bytes_per_launch"] = byts
    roof["traffic"], how = recorded_traffic(w.name, dominant, how=True)
    if how:
        roof["traffic_source"] = how

    # whole-chain roofline: max(12 BNMHD / tensor peak, 5 BHND elt / HBM); the shared
    # projection streams 3 token tensors (K, V, Y) instead of 5
    tok = w.B * w.H * w.N
    n_tensors = 3.0 if args.variant == "shared" else 5.0
    t_chain_tc = 12.0 * tok * w.M * w.D / ((tc_peak or peaks["bf16_tflops"]) * 1e12)
    t_chain_mem = n_tensors * tok * w.D * w.elt_bytes / (bw_peak * 1e9)
    t_chain = max(t_chain_tc, t_chain_mem)
    t_chain_burst = max(12.0 * tok * w.M * w.D / (peaks["bf16_tflops"] * 1e12), t_chain_mem)
    t_chain_sus = max(12.0 * tok * w.M * w.D / (peaks["bf16_tflops_sustained"] * 1e12),
                      t_chain_mem)
    chain = {"roofline_us": t_chain * 1e6, "bound": "tensor" if t_chain_tc >= t_chain_mem else "hbm",
             "frac": t_chain / (ms_per_step * 1e-3), "peak_kind": tc_kind,
             "frac_vs_burst_peak": t_chain_burst / (ms_per_step * 1e-3),
             "frac_vs_sustained_peak": t_chain_sus / (ms_per_step * 1e-3),
             "peaks": {"bf16_tflops_sustained": peaks.get("bf16_tflops_sustained"),
                       "bf16_tflops": peaks.get("bf16_tflops"), "hbm_gbs": bw_peak,
                       "source": peaks["source"]}}

    value = tok * world / (ms_per_step * 1e-3)

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        xh = {k: v.to("cpu").pin_memory() for k, v in x.items()}
        Yh = torch.empty(Y.shape, dtype=Y.dtype, pin_memory=True)
        bufs = {}
        ha = (xh["seeds"], xh["Kt"], xh["Vt"], xh["K"], xh["V"])
        if args.variant == "shared":
            ha = (xh["seeds"], xh["K"], xh["V"], xh["K"], xh["V"])
        for _ in range(2):
            flarepp.route_fwd_host(*ha, w.scale, Y_host=Yh, device=dev, workspace=ws, dev_bufs=bufs)
        n_e2e = max(1, min(args.steps, args.e2e_steps))
        barrier(world)
        torch.cuda.synchronize(dev)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(n_e2e):
            flarepp.route_fwd_host(*ha, w.scale, Y_host=Yh, device=dev, workspace=ws, dev_bufs=bufs)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / n_e2e, world)
        h2d = sum(t.numel() * t.element_size() for t in {id(t): t for t in ha}.values())
        d2h = Yh.numel() * Yh.element_size()
        e2e = {"value": tok * world / (e2e_ms * 1e-3), "unit": UNIT, "ms_per_step": e2e_ms,
               "steps": n_e2e, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
        del xh, Yh, bufs

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_oracle_sample(w, args.cpu_seconds, args.seed, args.variant)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
            "config": arm_config(w, args.variant, world, args.l2),
            "roofline": roof, "chain_roofline": chain, "stage_ms": stage_ms,
            "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": chain_fwd_launches(w) * args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default="mesh3d", choices=sorted(inputs.WORKLOADS))
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--variant", choices=("flarepp", "shared", "flare", "train", "mixer",
                                          "mixer_shared", "mixer_train"),
                    default="flarepp",
                    help="flarepp: the routing chain (default); shared: the chain with Kt, Vt "
                         "tied to K, V; flare: FLARE with fixed learned queries; train: the "
                         "chain's training forward and backward; mixer(_shared): the whole "
                         "FLARE++ mixer layer with four (two) projections")
    ap.add_argument("--l2", choices=("auto", "flush", "warm"), default="auto",
                    help="chain variants: flush the L2 before each timed step, or not; auto "
                         "flushes when the streamed tensors are near the L2's size")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-tokens", type=int, default=16384,
                    help="largest token sample per reference step")
    ap.add_argument("--ref-seconds", type=float, default=60.0,
                    help="about how long the reference arm's warm-up and timed steps take; "
                         "the token sample shrinks to fit")
    args = ap.parse_args()
    w = inputs.get(args.workload)
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        return run_reference(args, w)
    return run_ours(args, w)


if __name__ == "__main__":
    sys.exit(main())
