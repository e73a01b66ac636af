"""WHTMix forward benchmark: tokens/s and achieved HBM GB/s against the measured GB300 peak.

One step = one whtmix_forward call (the whole hot path: load, forward 2D WHT, gain, inverse 2D
WHT, store) over one batch of synthetic input already resident in HBM.  Default workload: the
full-image global-mixing shape, X [1, 65536, 128] bf16 (two 135x240 maps flattened, zero-padded
to 65536 tokens), G [65536, 128] fp32.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]

Prints one JSON line (rank 0).  Under torchrun (N > 1) every rank runs its own copy of the
workload (independent planes, no collective on the data path: weak scaling); the timed region is
bracketed by a barrier and a device synchronisation on both sides and the MAX over ranks is used.

Timing: CUDA events on the stream the kernels run on.  The inputs rotate over enough buffer sets
that their total exceeds 3x the L2 size, so every step streams X and G from HBM.  Clocks and
throttle reasons are sampled with nvidia-smi during the run.  ``--impl reference`` times the CPU
oracle (float64, single-threaded) on the host as the reference arm.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_25234_gb300 import inputs  # noqa: E402

DEFAULT_WORKLOAD = "fullimage_1x65536x128_bf16"
NOMINAL_HBM_GBS = 7900.0
FALLBACK_HBM_GBS = 6800.0
REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap", 0x8: "hw_slowdown",
           0x10: "sync_boost", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
           0x80: "hw_power_brake_slowdown", 0x100: "display_clock_setting"}
# The device-code files each kernel family is compiled from: a committed DRAM-traffic figure is
# used only while the hash of its family's files is unchanged (and only for the kernel it names).
KERNEL_FAMILY_SOURCES = {
    "k_forward_fast": ("whtmix_kernels.cuh", "whtmix_fast.cuh", "whtmix_fast_launch.cuh"),
    "k_backward_fast": ("whtmix_kernels.cuh", "whtmix_fast.cuh", "whtmix_fast_launch.cuh", "whtmix_fast_bwd.cuh"),
    "k_block_fast": ("whtmix_kernels.cuh", "whtmix_fast.cuh", "whtmix_block.cuh", "whtmix_block.cu"),
    "k_forward_plane": ("whtmix_kernels.cuh", "whtmix_fast.cuh", "whtmix_plane.cuh", "whtmix_plane.cu"),
}


def block_fused(w) -> bool:
    """True where whtmix_block_forward runs the whole block as one fused launch (mirrors the C ABI)."""
    m = (w.N * w.C).bit_length() - 1
    return w.block and w.dtype == "bf16" and w.C == 128 and 21 <= m <= 23


def kernel_name(w) -> str:
    """The kernel one whtmix_forward call launches for this workload (mirrors the C ABI's dispatch)."""
    m = (w.N * w.C).bit_length() - 1
    if block_fused(w):
        return f"k_block_fast<bf16, R=14, Q={m - 14}>"
    padded_ok = w.n_valid is None or (w.n_valid * w.C * (2 if w.dtype == "bf16" else 4)) % 16 == 0
    if (w.dtype in ("f32", "bf16") and 14 <= m <= 16 and (m < 16 or w.B >= 80) and w.gains == "full"
            and not w.block and (not w.padded_io or padded_ok)):
        return f"k_forward_plane<{w.dtype}, column bits {m - 14}> (one plane per CTA, in tensor memory)"
    if w.dtype in ("f32", "bf16") and 14 <= m <= 23:
        r = 14 if m == 21 else 13
        sep = ", separable gains" if w.gains == "separable" else ""
        pad = ", in-kernel token padding" if w.padded_io else ""
        x16 = ", bf16 exchange" if w.exchange == "bf16" else ""
        name = f"k_forward_fast<{w.dtype}, R={r}, Q={m - r}{sep}{pad}{x16}>"
        return f"k_proj<C={w.C}> + {name} + k_proj<C={w.C}>" if w.block else name
    return "k_forward_s" if m <= 13 else "k_forward_m"


def backward_kernel_name(w) -> str:
    """The kernel one whtmix_backward call launches for this workload (mirrors the C ABI's dispatch);
    for the block, the mixer backward inside whtmix_block_backward."""
    m = (w.N * w.C).bit_length() - 1
    if w.dtype in ("f32", "bf16") and 14 <= m <= 23:
        r = 14 if m >= 21 else 13
        return f"k_backward_fast<{w.dtype}, R={r}, Q={m - r}>"
    return "k_backward_s" if m <= 13 else "k_backward_m" if m <= 26 else "k_pass_* (five launches per group)"


def kernel_source_hash(kernel: str) -> str:
    """Hash of the source files of the kernel family `kernel` belongs to ("" if unknown)."""
    family = next((f for f in KERNEL_FAMILY_SOURCES if kernel.startswith(f)), None)
    if family is None:
        return ""
    h = hashlib.sha256()
    for f in sorted(KERNEL_FAMILY_SOURCES[family]):
        path = os.path.join(ROOT, "paper_2607_25234_gb300", "csrc", f)
        if os.path.exists(path):
            h.update(open(path, "rb").read())
    return h.hexdigest()[:16]


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def input_rotation(w, l2: int):
    """Buffer sets the timed loop rotates over so that their inputs and outputs exceed 3x the L2
    size (every step then streams from HBM): (sets, bytes per set)."""
    es = 2 if w.dtype == "bf16" else 4
    nv = w.n_valid if w.padded_io else w.N
    plane_b = w.B * nv * w.C * es
    g_b = (w.N + w.C) * 4 if w.gains == "separable" else w.N * w.C * 4
    set_bytes = 2 * plane_b + g_b + ((2 * plane_b + g_b) if w.backward else 0)
    return max(2, -(-3 * l2 // set_bytes)), set_bytes


def workload_config(w, world: int, l2: int) -> dict:
    """The JSON line's config, the same for both arms: the workload and how its steps defeat L2."""
    nsets, set_bytes = input_rotation(w, l2)
    return {"workload": w.name, "B": w.B, "N": w.N, "C": w.C, "io_dtype": w.dtype,
            "gain_dtype": "f32" if w.dtype != "i32" else "i32", "gains": w.gains,
            "stored_tokens": w.n_valid if w.padded_io else w.N, "exchange": w.exchange,
            "parallelism": f"replicas{world}",
            "l2": f"inputs rotate over {nsets} buffer sets ({nsets * set_bytes / 2**20:.0f} MiB, "
                  f"{nsets * set_bytes / l2:.1f}x L2)"}


def device_l2_bytes() -> int:
    """L2 size of GPU 0 (the fallback where none is visible)."""
    try:
        import torch
        if torch.cuda.is_available():
            return int(getattr(torch.cuda.get_device_properties(0), "L2_cache_size", 0) or 132 * 2**20)
    except Exception:
        pass
    return 132 * 2**20


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return ws, int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0"))


def max_over_ranks(value: float, world: int, device) -> float:
    """The job's time is its slowest rank's: a MAX all-reduce over the ranks (each timed the same
    K steps between two barriers)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.item()


def whole_job_tokens_per_s(world: int, tokens_per_step: int, steps: int, elapsed_ms: float) -> float:
    """Weak scaling, replicas: every rank runs the whole workload, so the job processes world times
    the tokens of one step per step."""
    return world * tokens_per_step * steps / (elapsed_ms / 1e3)


class ClockSampler:
    """nvidia-smi samples (timestamped on the host) for one GPU while the bench runs."""

    def __init__(self, gpu_index: str):
        self.samples = []  # (host_time, sm_mhz, max_mhz, reasons_mask)
        self.proc = None
        self.gpu = gpu_index
        self._t = None

    def start(self):
        cmd = ["nvidia-smi", "-i", self.gpu, "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active",
               "--format=csv,noheader,nounits", "-lms", "50"]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self._t = threading.Thread(target=self._read, daemon=True)
        self._t.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 3:
                continue
            try:
                self.samples.append((time.time(), float(parts[0]), float(parts[1]), int(parts[2], 16)))
            except ValueError:
                pass

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
        if self._t is not None:
            self._t.join(timeout=5)

    def summary(self, t0: float, t1: float):
        inside = [s for s in self.samples if t0 <= s[0] <= t1]
        window = "timed_region"
        if not inside:
            inside, window = self.samples, "whole_run"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "window": "none"}
        mask = 0
        for s in inside:
            mask |= s[3]
        return {"sm_mhz": statistics.median(s[1] for s in inside), "sm_max_mhz": max(s[2] for s in inside),
                "reasons": [n for b, n in REASONS.items() if mask & b and n != "gpu_idle"],
                "samples": len(inside), "window": window}


def host_cpu():
    """(usable cores, CPU model) of the host the bench runs on."""
    try:
        cores = len(os.sched_getaffinity(0))
    except Exception:
        cores = os.cpu_count() or 1
    model = ""
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                model = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    if not model:
        try:
            out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
            for line in out.splitlines():
                if line.strip().lower().startswith("model name"):
                    model = line.split(":", 1)[1].strip()
                    break
        except Exception:
            pass
    return cores, model or "unknown"


def oracle_time_plane(w: inputs.Workload, n_tokens: int, reps: int, threads: int = 1):
    """Median wall time of the CPU oracle on one [n_tokens, C] plane of the workload: the forward,
    plus the backward for a training-step workload, with `threads` OpenMP threads (the results
    are bit-identical to one thread's)."""
    import numpy as np
    import oracle
    oracle.set_threads(threads)
    d = inputs.make_inputs(1, n_tokens, w.C, w.dtype, seed=0,
                           n_valid=None if w.n_valid is None else min(w.n_valid, n_tokens), with_dy=w.backward)
    x = inputs.as_float64(d["x"], w.dtype)
    g = d["g"].astype(np.float64)
    dy = inputs.as_float64(d["dy"], w.dtype) if w.backward else None
    g_t, g_c = (a.astype(np.float64) for a in inputs.make_log_gains(n_tokens, w.C, 0))
    w_in, w_out = (inputs.as_float64(a, "bf16") for a in inputs.make_projections(w.C, 0))
    oracle.forward(x[:, :8, :], g[:8, :])  # load / compile outside the timing
    times = []
    for _ in range(reps):
        t = time.perf_counter()
        if w.block:
            oracle.block_forward(x, w_in, g, w_out)
        elif w.gains == "separable":
            oracle.forward_separable(x, g_t, g_c)
        else:
            oracle.forward(x, g)
        if dy is not None:
            if w.block:
                oracle.block_backward(x, w_in, g, w_out, dy)
            else:
                oracle.backward(x, g, dy)
        times.append(time.perf_counter() - t)
    oracle.set_threads(1)
    return statistics.median(times), times


def reference_arm(args, w):
    """The CPU oracle as the reference arm: each step runs the oracle forward on a bounded sample
    (one plane; the full [N, C] plane when K+W steps of it fit in about three minutes, else a
    plane with fewer tokens) and the metric is tokens/s of that sample."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    import numpy as np
    import oracle
    cores, model = host_cpu()
    t_full, _ = oracle_time_plane(w, w.N, 1, cores)
    budget = 180.0
    n = w.N
    while n > 64 and (args.steps + args.warmup) * t_full * n / w.N > budget:
        n //= 2
    d = inputs.make_inputs(1, n, w.C, w.dtype, seed=0, n_valid=None if w.n_valid is None else min(w.n_valid, n),
                           with_dy=w.backward)
    x = inputs.as_float64(d["x"], w.dtype)
    g = d["g"].astype(np.float64)
    dy = inputs.as_float64(d["dy"], w.dtype) if w.backward else None
    if w.block:
        w_in, w_out = (inputs.as_float64(a, "bf16") for a in inputs.make_projections(w.C, 0))
        fwd_run = lambda: oracle.block_forward(x, w_in, g, w_out)
        bwd_run = lambda: oracle.block_backward(x, w_in, g, w_out, dy)
    elif w.gains == "separable":
        g_t, g_c = (a.astype(np.float64) for a in inputs.make_log_gains(n, w.C, 0))
        fwd_run = lambda: oracle.forward_separable(x, g_t, g_c)
        bwd_run = lambda: oracle.backward_separable(x, g_t, g_c, dy)
    else:
        fwd_run = lambda: oracle.forward(x, g)
        bwd_run = lambda: oracle.backward(x, g, dy)

    def run():
        fwd_run()
        if w.backward:
            bwd_run()

    threads = oracle.set_threads(cores)
    for _ in range(args.warmup):
        run()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        run()
    el = time.perf_counter() - t0
    oracle.set_threads(1)
    value = args.steps * n / el
    sample = (f"per step one [{n},{w.C}] plane of the workload (full plane [{w.N},{w.C}] is {t_full:.2f} s), "
              f"float64 oracle{' forward + backward' if w.backward else ''} on {threads} OpenMP threads, CPU {model}")
    metric = ("WHTMix block fwd+bwd tokens/s" if w.backward and w.block else "WHTMix fwd+bwd tokens/s" if w.backward
              else "WHTMix block fwd tokens/s" if w.block else "WHTMix fwd tokens/s")
    line = {"impl": "reference", "metric": metric, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * el / max(args.steps, 1), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, world, device_l2_bytes()),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle", "sample": sample,
                             "cpu_model": model},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def alu_floor(w, sms: int, sm_mhz):
    """The adds of the transform against the SMs' fp32 lanes: 2 L log2(L) adds (forward, two
    transforms) and L multiplies per plane; the backward adds 3 L log2(L) + 2 L.  Floor = adds /
    (SMs x 128 lanes x SM clock): the packed add.f32x2 halves the instructions but, measured on
    this part, not the add rate."""
    L = w.N * w.C
    lg = L.bit_length() - 1
    adds = 2 * L * lg
    muls = L
    if w.backward:
        adds += 3 * L * lg
        muls += 2 * L
    adds *= w.B
    muls *= w.B
    if not sm_mhz:
        return {"adds": adds, "muls": muls, "floor_us": None}
    floor_s = adds / (sms * 128 * sm_mhz * 1e6)
    return {"adds": adds, "muls": muls, "sms": sms, "sm_mhz": sm_mhz, "lanes_per_sm": 128, "floor_us": 1e6 * floor_s}


def traffic_from_profile(workload: str):
    """DRAM bytes per launch from a committed ncu summary, only for the kernel the workload launches and
    only while that kernel's source files are unchanged."""
    p = os.path.join(ROOT, "profiles", "roofline_traffic.json")
    try:
        d = json.load(open(p))
    except Exception:
        return None
    e = d.get(workload)
    if not e:
        return None
    w = inputs.WORKLOADS.get(workload)
    launched = kernel_name(w) + (" " + backward_kernel_name(w) if w is not None and w.backward else "") if w else ""
    if e.get("kernel") not in launched or e.get("kernel_source_hash") != kernel_source_hash(e.get("kernel", "")):
        return None
    return e.get("dram_bytes_per_launch")


def ours(args, w):
    import ctypes
    import numpy as np
    import torch
    from paper_2607_25234_gb300 import whtmix

    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())
    lib = whtmix.library()
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 0) or 132 * 2**20

    d = inputs.workload_inputs(w, seed=rank)
    nv = w.n_valid if w.padded_io else w.N  # tokens stored per plane in X and Y
    if w.padded_io:
        d["x"] = np.ascontiguousarray(d["x"][:, :nv])
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16, "i32": torch.int32}[w.dtype]
    x_host = torch.from_numpy(d["x"].view(np.int16) if w.dtype == "bf16" else d["x"])
    if w.dtype == "bf16":
        x_host = x_host.view(torch.bfloat16)
    # the gains: G [N, C], or for the separable workload g_t [N] and g_c [C] in one buffer
    sep = w.gains == "separable"
    g_host = torch.from_numpy(np.concatenate([d["g_t"], d["g_c"]]) if sep else d["g"])
    x0 = x_host.to(dev)
    g0 = g_host.to(dev)
    # a training step (forward + backward) also reads dY and writes dX and dG
    dy_host = None
    if w.backward:
        dy_host = torch.from_numpy(d["dy"].view(np.int16) if w.dtype == "bf16" else d["dy"])
        if w.dtype == "bf16":
            dy_host = dy_host.view(torch.bfloat16)
    nsets, set_bytes = input_rotation(w, l2)
    xs = [x0] + [x0.clone() for _ in range(nsets - 1)]
    gs = [g0] + [g0.clone() for _ in range(nsets - 1)]
    ys = [torch.empty_like(x0) for _ in range(nsets)]
    if w.backward:
        dys = [dy_host.to(dev) for _ in range(nsets)]
        dxs = [torch.empty_like(x0) for _ in range(nsets)]
        dgs = [torch.empty_like(g0) for _ in range(nsets)]
    code = whtmix.DTYPE_CODE[tdt]
    stream = torch.cuda.current_stream(dev)
    sp = int(stream.cuda_stream)
    args_c = [(xs[i].data_ptr(), gs[i].data_ptr(), ys[i].data_ptr()) for i in range(nsets)]
    bargs_c = [(dys[i].data_ptr(), dxs[i].data_ptr(), dgs[i].data_ptr()) for i in range(nsets)] if w.backward else None
    fwd = lib.whtmix_forward
    bwd = lib.whtmix_backward
    fwd_sep = lib.whtmix_forward_separable
    fwd_pad = lib.whtmix_forward_padded
    fwd_block = lib.whtmix_block_forward
    fwd_x16 = lib.whtmix_forward_x16
    bwd_block = lib.whtmix_block_backward
    # launches of our kernels per step; the block backward: projection, mixer forward, weight
    # transpose, projection, weight gradient and its reduction, mixer backward, weight gradient
    # and reduction, weight transpose, projection
    block_bwd_launches = 11
    launches_per_step = ((1 if block_fused(w) else 3) + block_bwd_launches if w.block and w.backward else
                         2 if w.backward else 3 if w.block and not block_fused(w) else 1)
    if w.block:
        wi = torch.from_numpy(d["w_in"].view(np.int16)).to(dev).view(torch.bfloat16)
        wo = torch.from_numpy(d["w_out"].view(np.int16)).to(dev).view(torch.bfloat16)
        dwis = [torch.empty(w.C, w.C, dtype=torch.float32, device=dev) for _ in range(nsets)]
        dwos = [torch.empty(w.C, w.C, dtype=torch.float32, device=dev) for _ in range(nsets)]

    def step(i):
        a = args_c[i % nsets]
        if w.block:
            rc = fwd_block(a[0], wi.data_ptr(), a[1], wo.data_ptr(), a[2], w.B, w.N, w.C, code, sp)
        elif sep:
            rc = fwd_sep(a[0], a[1], a[1] + 4 * w.N, a[2], w.B, nv, w.N, w.C, code, sp)
        elif w.padded_io:
            rc = fwd_pad(a[0], a[1], a[2], w.B, nv, w.N, w.C, code, sp)
        elif w.exchange == "bf16":
            rc = fwd_x16(a[0], a[1], a[2], w.B, w.N, w.C, code, sp)
        else:
            rc = fwd(a[0], a[1], a[2], w.B, w.N, w.C, code, sp)
        if rc != 0:
            raise whtmix.WhtmixError(rc, "whtmix_forward")
        if w.backward:
            bb = bargs_c[i % nsets]
            if w.block:
                k = i % nsets
                rc = bwd_block(a[0], wi.data_ptr(), a[1], wo.data_ptr(), bb[0], bb[1], dwis[k].data_ptr(), bb[2],
                               dwos[k].data_ptr(), w.B, w.N, w.C, code, sp)
            else:
                rc = bwd(a[0], a[1], bb[0], bb[1], bb[2], w.B, w.N, w.C, code, sp)
            if rc != 0:
                raise whtmix.WhtmixError(rc, "whtmix_block_backward" if w.block else "whtmix_backward")

    # warm-up (also allocates the cached workspace on this stream)
    for i in range(max(args.warmup, 3)):
        step(i)
    whtmix.sync(stream)
    exchange = None
    if w.exchange == "bf16" and rank == 0:
        # the 16-bit exchange changes the arithmetic: how far its output is from the fp32-exchange
        # forward's on the first buffer set (the parity tests bound both against the float64
        # oracle), beside the bf16 acceptance tolerance (relative L2 <= 1e-2)
        y_f32x = whtmix.forward(xs[0], gs[0])
        whtmix.sync(stream)
        a, b = ys[0].double().reshape(w.B, -1), y_f32x.double().reshape(w.B, -1)
        rel = ((a - b).norm(dim=1) / b.norm(dim=1)).max().item()
        exchange = {"dtype": "bf16", "rel_l2_vs_fp32_exchange": rel, "tolerance": 1e-2}

    gpu_index = os.environ.get("CUDA_VISIBLE_DEVICES", str(local)).split(",")[local if world > 1 and
                                                                          "CUDA_VISIBLE_DEVICES" in os.environ else 0]
    sampler = ClockSampler(gpu_index if "CUDA_VISIBLE_DEVICES" in os.environ else str(local))
    sampler.start()
    time.sleep(0.3)
    for i in range(max(args.warmup, 3)):
        step(i)

    # The timed region: K steps back to back between two events on the launch stream (no event
    # between steps, so nothing but the launches themselves separates them).
    K = args.steps
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_host0 = time.time()
    start.record(stream)
    for i in range(K):
        step(i)
    end.record(stream)
    torch.cuda.synchronize(dev)
    t_host1 = time.time()
    if world > 1:
        dist.barrier()
    rc = lib.whtmix_sync(ctypes.c_void_p(sp))
    if rc != 0:
        raise whtmix.WhtmixError(rc, "device-side check after the timed loop")
    elapsed_ms = start.elapsed_time(end)
    # The spread of single steps: a shorter pass with events around each step (informational; the
    # events add their own gap to each step).
    KD = min(K, 200)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(KD)]
    for i in range(KD):
        ev[i][0].record(stream)
        step(i)
        ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    kern_ms = [a.elapsed_time(b) for a, b in ev]
    time.sleep(0.2)
    sampler.stop()
    clocks = sampler.summary(t_host0, t_host1)

    elapsed_ms = max_over_ranks(elapsed_ms, world, dev)
    tokens_per_step = w.B * w.N
    value = whole_job_tokens_per_s(world, tokens_per_step, K, elapsed_ms)
    step_ms = elapsed_ms / K  # average launch (or launch pair) duration over the timed region
    ideal = w.ideal_bytes()
    peak, peak_kind = measured_peaks()
    achieved = ideal / (step_ms / 1e3) / 1e9

    # End to end through the public Python API: every step copies its inputs in from pinned host
    # memory and its result back out.  Two device buffer sets and three streams (copies in,
    # compute, copies out) let step i + 1's copies in and step i - 1's copy out run beside step i's
    # launch, as a serving loop would; events order each buffer set's reuse.
    e2e = None
    if rank == 0 or world > 1:
        xh = x_host.pin_memory()
        gh = g_host.pin_memory()
        yh = torch.empty_like(xh).pin_memory()
        dyh = dy_host.pin_memory() if w.backward else None
        dxh = torch.empty_like(dyh).pin_memory() if w.backward else None
        dgh = torch.empty_like(gh).pin_memory() if w.backward else None
        dwih = torch.empty(w.C, w.C).pin_memory() if w.backward and w.block else None
        dwoh = torch.empty(w.C, w.C).pin_memory() if w.backward and w.block else None
        NB = 2
        s_in, s_comp, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        ev_in = [torch.cuda.Event() for _ in range(NB)]
        ev_comp = [torch.cuda.Event() for _ in range(NB)]
        ev_out = [torch.cuda.Event() for _ in range(NB)]

        def copies_in(k):
            pairs = [(xs[k], xh), (gs[k], gh)]
            if w.backward:
                pairs.append((dys[k], dyh))
            return pairs

        def copies_out(k):
            pairs = [(yh, ys[k])]
            if w.backward:
                pairs += [(dxh, dxs[k]), (dgh, dgs[k])]
            if w.backward and w.block:
                pairs += [(dwih, dwis[k]), (dwoh, dwos[k])]
            return pairs

        def e2e_step(i):
            k = i % NB
            with torch.cuda.stream(s_in):
                if i >= NB:
                    s_in.wait_event(ev_comp[k])  # the set's previous inputs are consumed
                for dst, src in copies_in(k):
                    dst.copy_(src, non_blocking=True)
                ev_in[k].record(s_in)
            with torch.cuda.stream(s_comp):
                s_comp.wait_event(ev_in[k])
                if i >= NB:
                    s_comp.wait_event(ev_out[k])  # the set's previous outputs are copied out
                xd, gd, yd = xs[k], gs[k], ys[k]
                if w.block:
                    whtmix.block_forward(xd, wi, gd, wo, out=yd)
                elif sep:
                    whtmix.forward_separable(xd, gd[:w.N], gd[w.N:], out=yd)
                elif w.padded_io:
                    whtmix.forward_padded(xd, gd, out=yd)
                elif w.exchange == "bf16":
                    whtmix.forward_x16(xd, gd, out=yd)
                else:
                    whtmix.forward(xd, gd, out=yd)
                if w.backward and w.block:
                    whtmix.block_backward(xd, wi, gd, wo, dys[k], dx=dxs[k], dw_in=dwis[k], dg=dgs[k], dw_out=dwos[k])
                elif w.backward:
                    whtmix.backward(xd, gd, dys[k], dx=dxs[k], dg=dgs[k])
                ev_comp[k].record(s_comp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_comp[k])
                for dst, src in copies_out(k):
                    dst.copy_(src, non_blocking=True)
                ev_out[k].record(s_out)

        ke = max(3, min(K, 50))
        for i in range(4):
            e2e_step(i)
        torch.cuda.synchronize(dev)
        s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record(s_in)
        for i in range(ke):
            e2e_step(i)
        e2.record(s_out)
        torch.cuda.synchronize(dev)
        e2e_ms = s2.elapsed_time(e2) / ke
        e2e = {"value": tokens_per_step / (e2e_ms / 1e3), "unit": "tokens/s",
               "h2d_bytes_per_step": sum(src.numel() * src.element_size() for _, src in copies_in(0)),
               "d2h_bytes_per_step": sum(dst.numel() * dst.element_size() for dst, _ in copies_out(0)),
               "steps": ke, "ms_per_step": e2e_ms,
               "pipeline": "copies in, compute, copies out on three streams, two buffer sets"}
        rc = lib.whtmix_sync(ctypes.c_void_p(int(s_comp.cuda_stream)))
        if rc != 0:
            raise whtmix.WhtmixError(rc, "device-side check after the end-to-end loop")

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    cpu = None
    if not args.no_cpu_baseline:
        # the oracle as it stands on the host: all usable cores (OpenMP over rows, column blocks and
        # elements, bit-identical to one thread) and, beside it, one thread
        cores, model = host_cpu()
        reps = 1 if w.backward else 3
        t_all, times_all = oracle_time_plane(w, w.N, reps, cores)
        t_one, times_one = oracle_time_plane(w, w.N, reps, 1)
        what = f"float64 oracle{' forward + backward' if w.backward else ''}"
        cpu = {"value": w.N / t_all, "unit": "tokens/s", "cores": cores, "kind": "oracle", "cpu_model": model,
               "sample": f"one full [{w.N},{w.C}] plane of the workload (B={w.B} planes would take "
                         f"{w.B * t_all:.2f} s), {what} on {cores} OpenMP threads, median of {len(times_all)} "
                         f"run(s): " + ", ".join(f"{t:.3f}" for t in times_all) + " s",
               "single_thread": {"value": w.N / t_one, "unit": "tokens/s", "cores": 1,
                                 "sample": f"the same plane on one thread, median of {len(times_one)} run(s): "
                                           + ", ".join(f"{t:.3f}" for t in times_one) + " s"}}

    metric = ("WHTMix block fwd+bwd tokens/s" if w.backward and w.block else "WHTMix fwd+bwd tokens/s" if w.backward
              else "WHTMix block fwd tokens/s" if w.block else "WHTMix fwd tokens/s")
    line = {"metric": metric, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": elapsed_ms / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "i32" if w.dtype == "i32" else "f32",
            "data": "synthetic",
            "config": workload_config(w, world, l2),
            "hbm_gbs": achieved, "pct_of_measured_peak": 100.0 * achieved / peak,
            "pct_of_nominal_peak": 100.0 * achieved / NOMINAL_HBM_GBS,
            "kernel_us": {"per_step": 1e3 * step_ms,
                          "single_step_events": {"steps": KD, "mean": 1e3 * statistics.mean(kern_ms),
                                                 "median": 1e3 * statistics.median(kern_ms),
                                                 "p10": 1e3 * sorted(kern_ms)[len(kern_ms) // 10],
                                                 "p90": 1e3 * sorted(kern_ms)[(9 * len(kern_ms)) // 10]}},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic_from_profile(w.name),
                         "peak_kind": peak_kind, "algorithmic_bytes_per_launch": ideal,
                         "kernel": kernel_name(w) + (
                             f" + the block backward ({block_bwd_launches} launches, the largest "
                             f"{backward_kernel_name(w)})" if w.backward and w.block else
                             f" + {backward_kernel_name(w)} (two launches per step)" if w.backward
                             else " (one launch per step)")},
            "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": K * launches_per_step, "clocks": clocks}
    if exchange is not None:
        line["exchange"] = exchange
    alu = alu_floor(w, torch.cuda.get_device_properties(dev).multi_processor_count, clocks.get("sm_mhz"))
    if alu["floor_us"] is not None:
        alu["frac_of_step"] = alu["floor_us"] / (elapsed_ms * 1e3 / K)
    line["alu_floor"] = alu
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def sweep(args):
    """Isolated-mixer latency against the token count N at batch 1, C = 64 (the paper's Section
    IV-C measurement of the mixer alone, power-of-two N, no padding).  Each point: one
    whtmix_forward call on resident bf16 inputs, CUDA events around each of 200 calls after 20
    warm-up calls on the same buffers (a latency, so the caches are warm as in a repeated call).
    Prints one JSON line with the per-N medians and the log-log slope."""
    import math
    import numpy as np
    import torch
    from paper_2607_25234_gb300 import whtmix
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    C = 64
    points = []
    for N in [1 << k for k in range(10, 17)]:
        d = inputs.make_inputs(1, N, C, "bf16", seed=0)
        x = torch.from_numpy(d["x"].view(np.int16)).to(dev).view(torch.bfloat16)
        g = torch.from_numpy(d["g"]).to(dev)
        y = torch.empty_like(x)
        for _ in range(20):
            whtmix.forward(x, g, out=y)
        whtmix.sync()
        ts = []
        for _ in range(200):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            whtmix.forward(x, g, out=y)
            b.record()
            ts.append((a, b))
        torch.cuda.synchronize(dev)
        us = statistics.median(a.elapsed_time(b) * 1e3 for a, b in ts)
        points.append({"N": N, "C": C, "us": us, "kernel": kernel_name(inputs.Workload("s", 1, N, C, "bf16"))})
    xs = [math.log(p["N"]) for p in points]
    ys = [math.log(p["us"]) for p in points]
    mx, my = sum(xs) / len(xs), sum(ys) / len(ys)
    slope = sum((a - mx) * (b - my) for a, b in zip(xs, ys)) / sum((a - mx) ** 2 for a in xs)
    print(json.dumps({"metric": "WHTMix isolated mixer latency vs N (batch 1, C=64, bf16)", "unit": "us",
                      "points": points, "loglog_slope": slope,
                      "paper_context": "paper (RTX 4090): isolated WHTMix slope 0.25, attention 1.70"}), flush=True)


def floor(args):
    """The memory-only floor of the three-phase forward on the full-image plane (2^23 elements,
    bf16 X and Y, fp32 G and workspace): bench_floor.cu moves the mixer's data phase by phase (X ->
    workspace rows, workspace and G columns, workspace rows -> Y) with coalesced 16-byte accesses,
    the same per-CTA ownership and the same barriers, and computes no butterflies.  Timed like the
    mixer (K launches back to back, inputs rotating over > 3x L2), with the mixer itself timed
    beside it on the same buffers; per-phase times come from global-timer stamps of every CTA
    (phase k ends when its last CTA leaves it).  Prints one JSON line."""
    import ctypes
    import numpy as np
    import torch
    from paper_2607_25234_gb300 import build, whtmix
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    lib = whtmix.library()
    flib = ctypes.CDLL(build.FLOOR_LIB)
    p, i = ctypes.c_void_p, ctypes.c_int
    flib.whtmix_floor_three_phase.argtypes = [p, p, p, p, p, i, i, p]
    flib.whtmix_floor_three_phase.restype = ctypes.c_int
    w = inputs.WORKLOADS[DEFAULT_WORKLOAD]
    m = (w.N * w.C).bit_length() - 1
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    l2 = getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0) or 132 * 2**20
    d = inputs.workload_inputs(w, seed=0)
    x0 = torch.from_numpy(d["x"].view(np.int16)).to(dev).view(torch.bfloat16)
    g0 = torch.from_numpy(d["g"]).to(dev)
    set_bytes = 2 * x0.numel() * 2 + g0.numel() * 4
    nsets = max(2, -(-3 * l2 // set_bytes))
    xs = [x0] + [x0.clone() for _ in range(nsets - 1)]
    gs = [g0] + [g0.clone() for _ in range(nsets - 1)]
    ys = [torch.empty_like(x0) for _ in range(nsets)]
    ws = torch.zeros(256 + 4 * (1 << m), dtype=torch.uint8, device=dev)
    KS = 50
    stamps = torch.zeros(KS, sms, 4, dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    sp = int(stream.cuda_stream)

    def fl(k, st=None):
        rc = flib.whtmix_floor_three_phase(xs[k % nsets].data_ptr(), gs[k % nsets].data_ptr(), ys[k % nsets].data_ptr(),
                                           ws.data_ptr(), (st if st is not None else stamps[0]).data_ptr(), m, sms, sp)
        if rc != 0:
            raise RuntimeError(f"floor kernel launch failed: cudaError {rc}")

    def mx(k):
        whtmix.forward(xs[k % nsets], gs[k % nsets], out=ys[k % nsets])

    def timed(f, K):
        for k in range(max(args.warmup, 3)):
            f(k)
        torch.cuda.synchronize(dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for k in range(K):
            f(k)
        b.record(stream)
        torch.cuda.synchronize(dev)
        return 1e3 * a.elapsed_time(b) / K

    K = args.steps
    floor_us = timed(fl, K)
    mixer_us = timed(mx, K)
    floor_us2 = timed(fl, K)
    for k in range(KS):
        fl(k, stamps[k])
    torch.cuda.synchronize(dev)
    whtmix.sync()
    hdr = ws[:256].view(torch.int32)
    if hdr[2].item() != 0:
        raise RuntimeError("floor kernel: a bounded barrier wait gave up")
    st = stamps.cpu().numpy().astype(np.float64)
    t0 = st[:, :, 0].min(axis=1)
    ends = [st[:, :, k].max(axis=1) for k in (1, 2, 3)]
    ph = [np.median(ends[0] - t0) / 1e3, np.median(ends[1] - ends[0]) / 1e3, np.median(ends[2] - ends[1]) / 1e3]
    ideal = w.ideal_bytes()
    peak, peak_kind = measured_peaks()
    fus = min(floor_us, floor_us2)
    print(json.dumps({
        "metric": "three-phase memory-only floor (no butterflies) vs the mixer, full-image plane",
        "workload": w.name, "steps": K, "floor_us": fus, "floor_us_runs": [floor_us, floor_us2],
        "mixer_us": mixer_us, "mixer_over_floor": mixer_us / fus,
        "floor_phases_us": {"phase1_rows_in": ph[0], "phase2_columns_incl_barrier": ph[1],
                            "phase3_rows_out_incl_barrier": ph[2], "stamped_launches": KS},
        "bytes": {"hbm_algorithmic": ideal, "l2_workspace": 4 * 4 * (1 << m)},
        "floor_frac_of_hbm_peak": ideal / (fus * 1e-6) / 1e9 / peak, "peak_gbs": peak, "peak_kind": peak_kind,
        "l2": f"inputs rotate over {nsets} buffer sets ({nsets * set_bytes / l2:.1f}x L2)"}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=inputs.WORKLOAD_ORDER)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true", help="isolated-mixer latency vs N (batch 1, C=64) instead")
    ap.add_argument("--floor", action="store_true",
                    help="memory-only floor of the three-phase forward on the full-image plane instead")
    args = ap.parse_args()
    if args.sweep:
        sweep(args)
        return
    if args.floor:
        floor(args)
        return
    w = inputs.WORKLOADS[args.workload]
    if args.impl == "reference":
        reference_arm(args, w)
    else:
        ours(args, w)


if __name__ == "__main__":
    main()
