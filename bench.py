"""Throughput of the ES step on one GB300: param*seed/s of a full generation
(N perturb + N restore + reward normalisation + one fused N-seed update) on a
synthetic parameter set shaped like the paper's workloads.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload qwen27b]
                    [--impl ours|reference] [--no-e2e] [--no-cpu-baseline] [--unfused]
    python bench.py --sweep [--populations 1,2,4,...] [--workload qwen4b]
    python bench.py --replay [--population N] [--generations K]
    python bench.py --antithetic
    python bench.py --generator [--gen-log2 31]
    python bench.py --pipe-peaks [--probes name,name,...]

Prints one JSON line (rank 0). `value` is measured with the inputs resident in
HBM; `e2e` is the same metric with the parameters in pinned host memory and
copied to the device and back inside every timed step. The reference arm
(`--impl reference`) times the CPU oracle, on every host core, on a bounded
sample of the same workload. The other modes time one part of the path each:
es_update per population size, seed-log replay, antithetic generations, the
noise generator alone and the register-only pipe probes. The roofline is the
nominal integer-multiply rate (the FMA-heavy pipe's rate for Philox's
products); each kernel is also reported against the kernels' own generator
run in registers in the same process (`generator_frac`). With --gpus N > 1 (under torchrun) every rank runs an independent
replica of the step (replicas only: the ES step has no exchange between GPUs
besides N scalar rewards) and the slowest rank's time is reported.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_17310_gb300 import inputs as I  # noqa: E402

METRIC = "ES step param*seed/s (perturb+restore+update) and % of HBM/ALU roofline"
UNIT = "param*seed/s"
SIGMA_FINAL = {"qwen27b": 2.5e-4, "qwen4b": 5e-4, "qwen4b_f32": 5e-4, "qwen4b_4layer": 5e-4,
               "toy": 1e-3}
SCHEDULE_T = 100


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--workload", default="qwen27b",
                   choices=["qwen27b", "qwen4b", "qwen4b_f32", "qwen4b_fp8", "qwen4b_4layer", "toy"])
    p.add_argument("--population", type=int, default=None, help="override N")
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--e2e-steps", type=int, default=None,
                   help="generations timed by the e2e leg (default: --steps, at least 5)")
    p.add_argument("--unfused", action="store_true",
                   help="separate es_restore / es_perturb launches instead of es_restore_perturb")
    p.add_argument("--sweep", action="store_true",
                   help="instead of the step: time es_update alone for each N of --populations "
                        "(default workload qwen4b) and print one JSON line with every point")
    p.add_argument("--populations", default="1,2,4,8,16,32,64,128",
                   help="comma-separated N values of --sweep")
    p.add_argument("--replay", action="store_true",
                   help="instead of the step: K logged generations applied by one es_replay "
                        "against K es_update calls (default workload qwen4b)")
    p.add_argument("--generations", type=int, default=16, help="K of --replay")
    p.add_argument("--generator", action="store_true",
                   help="instead of the step: the noise generator alone through es_noise_fill "
                        "(2^31 Gaussians per launch) and es_noise_bits")
    p.add_argument("--gen-log2", type=int, default=31,
                   help="--generator: 2^k Gaussians per es_noise_fill launch")
    p.add_argument("--pipe-peaks", action="store_true",
                   help="instead of the step: the register-only pipe probes (integer "
                        "multiply, MUFU, FMA, LOP3, their mixes, a warp-split overlap test, "
                        "the generator) in ops per clock per SM")
    p.add_argument("--probes", default=None,
                   help="--pipe-peaks: only these probes (comma-separated names), at 4 CTAs "
                        "per SM")
    p.add_argument("--antithetic", action="store_true",
                   help="instead of the step: a generation of N/2 antithetic pairs (the +/- "
                        "flip as one es_restore_perturb on one seed)")
    args = p.parse_args()
    if args.e2e_steps is None:
        args.e2e_steps = max(5, args.steps)
    if (args.sweep or args.replay) and "--workload" not in " ".join(sys.argv):
        args.workload = "qwen4b"
    return args


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d.get("sm_max_mhz", 2070.0)), "measured"
    return 6800.0, 2070.0, "fallback"


# --- distributed plumbing -------------------------------------------------------------

def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if world == 1:
        return 0, 1, None
    import torch
    import torch.distributed as dist
    local = int(os.environ.get("LOCAL_RANK", "0"))
    backend = "nccl" if torch.cuda.is_available() else "gloo"
    if backend == "nccl":
        torch.cuda.set_device(local)
    dist.init_process_group(backend)
    return dist.get_rank(), dist.get_world_size(), dist


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(x: float, dist) -> float:
    if dist is None:
        return x
    import torch
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --- clocks -------------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        # nvidia-smi numbers GPUs by itself; address the torch device by UUID
        self.device_id = str(device_index)
        try:
            import torch
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            if uuid:
                self.device_id = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            pass
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.device_id}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for name, val in zip(names, f[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# --- the step -------------------------------------------------------------------------------

L2_BYTES = 129 * 1024 * 1024     # GB300 L2


ELEM_BYTES = {"bf16": 2, "f32": 4, "e4m3": 1}


def param_set(es, workload: str):
    """(flat buffer, views, plan, bytes per element) of a workload's parameter
    set on the current CUDA device; FP8 sets get a scaled plan."""
    import torch
    wl = I.WORKLOADS[workload]
    specs = I.shapes_for(workload)
    if wl.dtype == "e4m3":
        flat, params, scales = I.init_params_flat_e4m3(specs, "cuda", seed=0)
        return flat, params, es.plan_from_tensors(params, scales=scales), 1
    dtype = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    flat, params = I.init_params_flat(specs, dtype, "cuda", seed=0)
    return flat, params, es.plan_from_tensors(params), ELEM_BYTES[wl.dtype]


def workload_config(workload: str, n: int, world: int) -> dict:
    """The `config` object of the JSON line (shared by both arms)."""
    wl = I.WORKLOADS[workload]
    specs = I.shapes_for(workload)
    P = sum(s.numel for s in specs)
    esize = ELEM_BYTES[wl.dtype]
    return {"workload": workload, "params": P, "population": n, "storage": wl.dtype,
            "segments": len(specs), "description": wl.description, "alpha": wl.alpha,
            "l2": ("inputs larger than L2 (%.1f GB of parameters)" % (P * esize / 1e9)
                   if P * esize > L2_BYTES else
                   "inputs smaller than L2 (%.1f MB of parameters): not an HBM measurement"
                   % (P * esize / 1e6)),
            "parallelism": "replicas" if world > 1 else "single GPU"}


def generation_inputs(wl, step: int, n: int):
    """Seeds and rewards of one generation (rewards stand in for rollouts)."""
    seeds = I.population_seeds(n, generation=step)
    rewards = I.rewards(wl.rewards if wl.rewards != "quadratic" else "uniform", n, seed=step)
    return seeds, rewards


def run_step(es, plan, wl, step, n, sigma, sigma_next, stream, timers=None, fused=True):
    """One ES generation through the C ABI. Returns the number of kernels launched.

    Fused (the library's steady-state loop): on entry theta carries the
    perturbation of this generation's first member, applied by the previous
    step's es_update_perturb; each step does N - 1 es_restore_perturb, one
    es_restore and one es_update_perturb (update fused with the next
    generation's first perturb): N perturbs, N restores and one update per
    generation. Unfused: N x (es_perturb, es_restore), then es_update.
    """
    seeds, rewards = generation_inputs(wl, step, n)
    launches = [0]

    def call(name, fn, *args):
        if timers is not None:
            timers.start(name)
        fn(*args)
        if timers is not None:
            timers.stop(name, 1)
        launches[0] += 1

    # (the rollout of each perturbed model happens after its perturb; its
    # reward is an input here)
    if fused:
        for i in range(1, n):
            call("restore_perturb", es.es_restore_perturb, plan, int(seeds[i - 1]), sigma,
                 int(seeds[i]), sigma, stream)
        call("restore", es.es_restore, plan, int(seeds[n - 1]), sigma, stream)
    else:
        for i in range(n):
            call("perturb", es.es_perturb, plan, int(seeds[i]), sigma, stream)
            call("restore", es.es_restore, plan, int(seeds[i]), sigma, stream)
    rhat = es.es_normalize_rewards(rewards, 1e-8)
    coeffs = es.es_update_coeffs(rhat, wl.alpha, sigma, es.ES_SCALE_PAPER)
    if fused:
        first_next = int(generation_inputs(wl, step + 1, n)[0][0])
        call("update_perturb", es.es_update_perturb, plan, seeds, coeffs, first_next,
             sigma_next, stream)
    elif np.any(coeffs != 0):
        call("update", es.es_update, plan, seeds, coeffs, stream)
    else:
        es.es_update(plan, seeds, coeffs, stream)   # no launch: the no-update rule
    return launches[0]


def start_loop(es, plan, wl, step, n, sigma, stream, fused):
    """Before the first fused step: perturb with that generation's first member."""
    if fused:
        es.es_perturb(plan, int(generation_inputs(wl, step, n)[0][0]), sigma, stream)


class KernelTimers:
    """CUDA-event pairs around kernel launches on the launching stream."""

    def __init__(self, torch, stream):
        self.torch = torch
        self.stream = stream
        self.pairs = {}
        self._open = {}

    def start(self, name):
        e = self.torch.cuda.Event(enable_timing=True)
        e.record(self.stream)
        self._open[name] = e

    def stop(self, name, count):
        e = self.torch.cuda.Event(enable_timing=True)
        e.record(self.stream)
        self.pairs.setdefault(name, []).append((self._open.pop(name), e, count))

    def names(self):
        return list(self.pairs)

    def count(self, name):
        return sum(c for _, _, c in self.pairs.get(name, []))

    def mean_ms(self, name):
        cnt = self.count(name)
        return self.total_ms(name) / cnt if cnt else None

    def total_ms(self, name):
        return sum(a.elapsed_time(b) for a, b, _ in self.pairs.get(name, []))


# Gaussians each launch kind draws per parameter (the update draws N).
GAUSS_PER_ELEM = {"perturb": 1, "restore": 1, "restore_perturb": 2}
KERNEL_NAME = {"perturb": "axpy_noise_kernel<1 step> (es_perturb)",
               "restore": "axpy_noise_kernel<1 step> (es_restore)",
               "restore_perturb": "axpy_noise_kernel<2 steps> (es_restore_perturb)",
               "update": "update_kernel<single generation> (es_update)",
               "update_perturb": "update_kernel<generations + perturb> (es_update_perturb)"}


def gauss_per_elem(kind, n):
    if kind in GAUSS_PER_ELEM:
        return GAUSS_PER_ELEM[kind]
    return n + 1 if kind == "update_perturb" else n
# Philox4x32-10 on counter (j_lo, j_hi, 0, 0): 10 rounds x 2 products of
# 32x32->64 bits per 4 outputs, less the first round's product by 0 and the
# second round's product of (key, j_hi) alone (shared by a tile): 18 products
# (mad.wide.u32), each two 32-bit multiplies (high and low word), i.e. 9 per
# Gaussian. The nominal rate is 64 32-bit multiplies per clock per SM.
IMUL_PER_GAUSS = 9
WIDE_PER_GAUSS = IMUL_PER_GAUSS / 2
IMUL_PER_CLK_SM = 64
# Box-Muller: log2, sqrt, sin and cos per pair on the MUFU pipe (nominal 16
# per clock per SM): 2 per Gaussian.
MUFU_PER_GAUSS = 2
MUFU_PER_CLK_SM = 16
# Three-input XORs of those rounds (lop3): 19 per block of 4 Gaussians.
LOP3_PER_GAUSS = 19 / 4


# The device code of the kernels whose DRAM traffic is recorded.
KERNEL_SOURCES = ("es_internal.h", "es_kernels.cu", "es_noise.cuh")


def strip_comments(src):
    """C/C++ source without comments, trailing blanks or blank lines, so that
    an edit to comments or layout leaves the code digest unchanged. String and
    character literals are kept as written."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        elif c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        else:
            out.append(c)
            i += 1
    lines = (" ".join(line.split()) for line in "".join(out).split("\n"))
    return "\n".join(line for line in lines if line)


def kernel_code_digest(csrc=None):
    """First 16 hex digits of the sha256 over the kernels' device sources
    (KERNEL_SOURCES in order), comments and layout stripped."""
    import hashlib
    csrc = csrc or os.path.join(ROOT, "paper_2608_17310_gb300", "csrc")
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(csrc, f), encoding="utf-8") as fh:
            h.update(strip_comments(fh.read()).encode())
            h.update(b"\0")
    return h.hexdigest()[:16]


def traffic_per_element(kind):
    """DRAM bytes per parameter of one launch from the committed ncu summary,
    or None if the kernels' code changed since that capture."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    if not os.path.exists(path):
        return None
    digest = kernel_code_digest()
    for line in open(path):
        f = line.split()
        if len(f) == 3 and not line.startswith("#") and f[0] == kind:
            return float(f[1]) if f[2] == digest else None
    return None


def pipe_occupancy(kind):
    """FMA-heavy and XU cycles active (% of elapsed) of a launch kind from the
    committed ncu summary, or None if the kernels' code changed since."""
    path = os.path.join(ROOT, "profiles", "pipe_occupancy.txt")
    if not os.path.exists(path):
        return None
    digest = kernel_code_digest()
    for line in open(path):
        f = line.split()
        if len(f) == 4 and not line.startswith("#") and f[0] == kind and f[3] == digest:
            heavy, xu = float(f[1]), float(f[2])
            return {"fmaheavy_pct": heavy, "xu_pct": xu, "sum_pct": round(heavy + xu, 1),
                    "source": "ncu sm__pipe_fmaheavy_cycles_active + sm__pipe_xu_cycles_active, "
                              "profiles/pipe_occupancy.txt"}
    return None


def run_ours(args, rank, world, dist):
    import torch
    from paper_2608_17310_gb300 import build, esopt as es

    build.build_library()
    dev_index = torch.cuda.current_device()
    torch.cuda.init()
    wl = I.WORKLOADS[args.workload]
    n = args.population or wl.population
    flat, params, plan, esize = param_set(es, args.workload)
    P = plan.numel
    stream = torch.cuda.current_stream()
    s_handle = stream.cuda_stream
    sigma0, sigmaT = wl.sigma, SIGMA_FINAL.get(args.workload, wl.sigma)

    def sigma_at(t):
        return float(np.float32(es.es_sigma_cosine(sigma0, sigmaT, t, SCHEDULE_T)))

    fused = not args.unfused
    start_loop(es, plan, wl, 0, n, sigma_at(0), s_handle, fused)
    for w in range(args.warmup):
        run_step(es, plan, wl, w, n, sigma_at(w), sigma_at(w + 1), s_handle, None, fused)
    torch.cuda.synchronize()
    barrier(dist)
    torch.cuda.synchronize()

    timers = KernelTimers(torch, stream)
    launches = 0
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev_index) as clk:
        ev0.record(stream)
        for k in range(args.steps):
            t = args.warmup + k
            launches += run_step(es, plan, wl, t, n, sigma_at(t), sigma_at(t + 1), s_handle,
                                 timers, fused)
        ev1.record(stream)
        torch.cuda.synchronize()
    barrier(dist)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    ms_max = max_over_ranks(ms, dist)
    per_step_ms = ms_max / args.steps
    value = world * P * n * args.steps / (ms_max / 1e3)

    imul_peak, gauss_peak, gen_peak, sms, sm_max_mhz, hbm_gbs, peak_src, ceilings = \
        alu_peaks(torch, dev_index)
    bytes_per_launch = 2 * esize * P
    gen_pipe = ceilings["generator_pipelined"]["gauss_per_s"]
    kernels = {}
    for name in timers.names():
        mean = timers.mean_ms(name)
        g = gauss_per_elem(name, n) * P
        gbs = bytes_per_launch / (mean / 1e3) / 1e9
        gps = g / (mean / 1e3)
        hbm_frac, alu_frac = gbs / hbm_gbs, gps / gauss_peak
        kernels[name] = {"kernel": KERNEL_NAME[name], "launches": timers.count(name),
                         "mean_ms": mean, "share": timers.total_ms(name) / ms,
                         "gbs": gbs, "gauss_per_s": gps, "hbm_frac": hbm_frac,
                         "alu_frac": alu_frac, "generator_frac": gps / gen_peak,
                         "generator_pipelined_frac": gps / gen_pipe,
                         "bound": "alu" if alu_frac > hbm_frac else "hbm"}
    dom = max(kernels, key=lambda k: kernels[k]["share"])
    d = kernels[dom]
    tpe = traffic_per_element(dom)
    traffic = tpe * P if tpe is not None else None
    if d["bound"] == "hbm":
        roof = {"bound": "hbm", "achieved": d["gbs"], "peak": hbm_gbs, "unit": "GB/s",
                "frac": d["hbm_frac"], "traffic": traffic,
                "peak_source": f"{peak_src} MEASURED_PEAKS.json hbm_gbs"}
    else:
        roof = {"bound": "alu", "achieved": d["gauss_per_s"] * IMUL_PER_GAUSS / 1e12,
                "peak": imul_peak / 1e12, "unit": "T imul32/s", "frac": d["alu_frac"],
                "traffic": traffic,
                "peak_source": f"{sms} SMs x {IMUL_PER_CLK_SM} 32-bit integer multiplies/clk x "
                               f"{sm_max_mhz:.0f} MHz; {IMUL_PER_GAUSS} multiplies per Gaussian"}
    roof["generator_bound"] = {
        "gauss_per_s": gen_peak, "frac": d["gauss_per_s"] / gen_peak,
        "source": "measured in this run: the kernels' own generator (Philox, Box-Muller) in a "
                  "register-only loop with no memory traffic, 4 CTAs per SM, scaled to the "
                  "maximum SM clock: what this instruction stream reaches on its own "
                  "(bench.py --pipe-peaks has every probe)",
        "pipelined": {"gauss_per_s": gen_pipe, "frac": d["gauss_per_s"] / gen_pipe,
                      "source": "the same generator with two seeds' blocks alternating, the "
                                "next seed's Philox words beside the current seed's transform, "
                                "as in the update's seed loop"}}
    roof["measured_ceilings"] = ceilings
    roof["pipe_occupancy"] = pipe_occupancy(dom)
    roof.update({"kernel": d["kernel"], "hbm_frac": d["hbm_frac"], "alu_frac": d["alu_frac"],
                 "algorithmic_bytes_per_launch": bytes_per_launch,
                 "gaussians_per_launch": gauss_per_elem(dom, n) * P})

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, torch, es, plan, flat, params, wl, n, esize, sigma_at, s_handle, dist,
                      world, fused)

    cpu = None
    if not args.no_cpu_baseline and rank == 0 and world == 1:
        cpu = cpu_baseline(args.workload, n, sigma_at(args.warmup))

    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic",
        "config": dict(workload_config(args.workload, n, world), sigma=sigma_at(args.warmup),
                       generation_loop=("es_restore_perturb x (N-1), es_restore, es_update_perturb"
                                        if fused else "separate calls")),
        "roofline": roof,
        "kernels": kernels,
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    plan.close()
    if rank == 0:
        print(json.dumps(out), flush=True)


def probe_lib():
    """The register-only pipe probes (csrc/es_probes.cu, _build/libesprobe.so)."""
    import ctypes
    from paper_2608_17310_gb300 import build
    build.build_library()
    L = ctypes.CDLL(build.PROBE_LIB)
    L.esprobe_count.restype = ctypes.c_int
    L.esprobe_name.argtypes = [ctypes.c_int]
    L.esprobe_name.restype = ctypes.c_char_p
    L.esprobe_unit.argtypes = [ctypes.c_int]
    L.esprobe_unit.restype = ctypes.c_char_p
    L.esprobe_run.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int,
                              ctypes.POINTER(ctypes.c_double)]
    L.esprobe_run.restype = ctypes.c_int
    return L


def run_probe(L, name, ctas_per_sm=4, target_ms=20.0):
    """One probe, its iteration count scaled so the timed launch takes about
    target_ms. Rates are per SM per clock (the probe times itself in SM cycles)."""
    import ctypes
    ids = {L.esprobe_name(i).decode(): i for i in range(L.esprobe_count())}
    pid = ids[name]
    out = (ctypes.c_double * 7)()
    iters = 256
    for _ in range(2):
        rc = L.esprobe_run(pid, ctas_per_sm, iters, out)
        if rc != 0:
            raise RuntimeError(f"probe {name}: esprobe_run returned {rc}")
        if out[0] >= 0.5 * target_ms:
            break
        iters = max(256, int(iters * target_ms / max(out[0], 1e-3)) // 4 * 4)
    return {"probe": name, "unit": L.esprobe_unit(pid).decode(), "ctas_per_sm": int(out[6]),
            "iters": iters, "ms": out[0], "cycles": out[1], "sm_mhz": out[2],
            "ops_per_clk_sm": out[3], "ops": out[4], "threads_per_sm": out[5]}


def measured_ceilings(res, sms, sm_max_mhz):
    """ALU ceilings of the generator from probe results (`res`: name -> run_probe
    dict), in Gaussians/s at the maximum SM clock:
      imad_wide      a chain of mad.wide.u32 with a 64-bit addend, per 4.5 per
                     Gaussian. ncu counts 1.5 FMA-heavy instructions and 5 pipe
                     cycles per operation of this chain, against 4 cycles for
                     the kernels' mul.wide, so it understates the pipe: the
                     nominal 64 multiplies per clock per SM (32 mul.wide at 4
                     cycles each) is the pipe's rate;
      lop3           the three-input XOR alone: lop3 rate / 4.75;
      mufu           the MUFU pipe alone: its rate / 2;
      imad_mufu_mix  mad.wide and MUFU in the generator's ratio (9 : 4) in one
                     thread;
      generator      the streaming kernels' generator (Philox with scheduled
                     round keys, the packed transform, the near-one series on a
                     rare branch) in registers, no memory traffic: the rate this
                     instruction stream reaches on its own;
      generator_pipelined  the same generator with two seeds' blocks
                     alternating, the next seed's Philox words computed beside
                     the current seed's transform (the update's seed loop)."""
    hz = sms * sm_max_mhz * 1e6
    out = {}
    for name, per_g in (("imad_wide", WIDE_PER_GAUSS), ("lop3", LOP3_PER_GAUSS),
                        ("mufu", MUFU_PER_GAUSS)):
        if name in res:
            r = res[name]["ops_per_clk_sm"]
            out[name] = {"ops_per_clk_sm": r, "per_gaussian": per_g, "gauss_per_s": r / per_g * hz}
    if "imad_wide" in out:
        out["imad_wide"]["imul32_per_clk_sm"] = 2 * out["imad_wide"]["ops_per_clk_sm"]
    if "mix_imad_wide_mufu_9_4" in res:
        r = res["mix_imad_wide_mufu_9_4"]["ops_per_clk_sm"]
        out["imad_mufu_mix"] = {"wide_per_clk_sm": r, "gauss_per_s": r / WIDE_PER_GAUSS * hz}
    if "mix_imad_hi_lo_1_1" in res:
        r = res["mix_imad_hi_lo_1_1"]["ops_per_clk_sm"]
        out["imad_hi_lo"] = {"pairs_per_clk_sm": r, "imul32_per_clk_sm": 2 * r,
                             "gauss_per_s": r / WIDE_PER_GAUSS * hz}
    if "mix_imad_hi_lo_mufu_9_4" in res:
        r = res["mix_imad_hi_lo_mufu_9_4"]["ops_per_clk_sm"]
        out["imad_hi_lo_mufu_mix"] = {"pairs_per_clk_sm": r, "gauss_per_s": r / WIDE_PER_GAUSS * hz}
    if "generator" in res:
        r = res["generator"]["ops_per_clk_sm"]
        out["generator"] = {"gauss_per_clk_sm": r, "gauss_per_s": r * hz}
    if "generator_pipelined" in res:
        r = res["generator_pipelined"]["ops_per_clk_sm"]
        out["generator_pipelined"] = {"gauss_per_clk_sm": r, "gauss_per_s": r * hz}
    if all(k in res for k in ("split_imad_wide_only", "split_mufu_only", "split_both")):
        ti = res["split_imad_wide_only"]["cycles"]
        tm = res["split_mufu_only"]["cycles"]
        tb = res["split_both"]["cycles"]
        out["warp_split"] = {"cycles_imad_only": ti, "cycles_mufu_only": tm, "cycles_both": tb,
                             "overlap": (ti + tm - tb) / min(ti, tm)}
    return out


CEILING_PROBES = ("imad_wide", "lop3", "mufu", "mix_imad_wide_mufu_9_4", "mix_imad_hi_lo_1_1",
                  "mix_imad_hi_lo_mufu_9_4", "generator", "generator_pipelined")


def alu_peaks(torch, dev_index, probes=True):
    """(imul32/s at the nominal integer-multiply rate, Gaussians/s at that
    roofline, Gaussians/s of the register-only generator, SM count, max SM MHz,
    HBM GB/s, peak source, measured ceilings).

    The roofline is the nominal one: 64 32-bit multiplies per clock per SM x
    SMs x the maximum SM clock, 9 multiplies per Gaussian. It is the FMA-heavy
    pipe's rate for mul.wide.u32 (4 pipe cycles per warp instruction, ncu). The
    generator rate is measured live by the register-only probe of the kernels'
    own generator (no memory traffic); without probes it is None."""
    hbm_gbs, sm_max_mhz, peak_src = peaks()
    sms = torch.cuda.get_device_properties(dev_index).multi_processor_count
    imul_peak = sms * IMUL_PER_CLK_SM * sm_max_mhz * 1e6
    ceilings = {}
    gen_peak = None
    if probes:
        L = probe_lib()
        res = {name: run_probe(L, name, 4, 10.0) for name in CEILING_PROBES}
        ceilings = measured_ceilings(res, sms, sm_max_mhz)
        ceilings["source"] = ("bench.py probes (csrc/es_probes.cu): register-only loops, 4 CTAs "
                              "of 256 threads per SM, each SM timed on its own clock from its "
                              "first CTA's start to its last CTA's end, scaled to the maximum "
                              "SM clock")
        gen_peak = ceilings["generator"]["gauss_per_s"]
    return (imul_peak, imul_peak / IMUL_PER_GAUSS, gen_peak, sms, sm_max_mhz, hbm_gbs,
            peak_src, ceilings)


def run_pipe_peaks(args, rank, world, dist):
    """Every register-only probe of csrc/es_probes.cu: single pipes, two-pipe
    mixes, the warp-split overlap test and the library's generator, at 4 CTAs of
    256 threads per SM, and at 1, 2 and 8 (where the registers allow) for the
    main ones. Rates are per SM per clock;
    ceilings are scaled to the maximum SM clock."""
    import torch
    torch.cuda.init()
    dev_index = torch.cuda.current_device()
    hbm_gbs, sm_max_mhz, peak_src = peaks()
    sms = torch.cuda.get_device_properties(dev_index).multi_processor_count
    L = probe_lib()
    names = [L.esprobe_name(i).decode() for i in range(L.esprobe_count())]
    if args.probes:
        wanted = [x.strip() for x in args.probes.split(",") if x.strip()]
        unknown = [x for x in wanted if x not in names]
        if unknown:
            raise SystemExit(f"--probes: unknown probe(s) {unknown}; known: {names}")
        names = wanted
    res, occupancy = {}, []
    with ClockSampler(dev_index) as clk:
        for name in names:
            res[name] = run_probe(L, name, 4, 25.0)
        for name in ("imad_wide", "mufu", "mix_imad_wide_mufu_9_4", "mix_imad_hi_lo_1_1",
                     "mix_imad_hi_lo_mufu_9_4", "philox", "generator", "generator_pipelined"):
            if args.probes:
                break
            for ctas in (1, 2, 8):
                occupancy.append(run_probe(L, name, ctas, 25.0))
    out = {"mode": "pipe_peaks", "metric": "ops per clock per SM of register-only pipe probes",
           "unit": "ops/clk/SM", "n_gpus": 1, "data": "synthetic (register-only loops)",
           "config": {"threads_per_cta": 256, "ctas_per_sm": 4, "sms": sms,
                      "sm_max_mhz": sm_max_mhz,
                      "nominal": {"imul32_per_clk_sm": IMUL_PER_CLK_SM,
                                  "mufu_per_clk_sm": MUFU_PER_CLK_SM}},
           "probes": [res[n] for n in names], "occupancy": occupancy,
           "ceilings": measured_ceilings(res, sms, sm_max_mhz),
           "gpu_launches": 2 * (len(res) + len(occupancy)) * 2, "clocks": clk.summary()}
    if rank == 0:
        print(json.dumps(out), flush=True)


def run_sweep(args, rank, world, dist):
    """es_update alone on one parameter set for each population size N: where
    the fused update turns from HBM-bound (small N: 2 * sizeof bytes per
    parameter, N Gaussians) to generator-bound (large N). Each launch is timed
    with CUDA events on the launching stream; the set is larger than L2."""
    import torch
    from paper_2608_17310_gb300 import build, esopt as es

    build.build_library()
    dev_index = torch.cuda.current_device()
    torch.cuda.init()
    wl = I.WORKLOADS[args.workload]
    flat, params, plan, esize = param_set(es, args.workload)
    P = plan.numel
    stream = torch.cuda.current_stream()
    s_handle = stream.cuda_stream
    imul_peak, gauss_peak, gen_peak, sms, sm_max_mhz, hbm_gbs, peak_src, ceilings = \
        alu_peaks(torch, dev_index)
    gen_pipe = ceilings["generator_pipelined"]["gauss_per_s"]
    bytes_per_launch = 2 * esize * P
    pops = [int(x) for x in args.populations.split(",") if x.strip()]
    points = []
    launches = 0
    with ClockSampler(dev_index) as clk:
        for n in pops:
            seeds = I.population_seeds(n, generation=n, first=7)
            # N(0, 1) rewards used as the normalised rewards directly (a z-score
            # of a single reward would be 0: no update to time at N = 1)
            rhat = I.rewards("normal", n, seed=n)
            coeffs = es.es_update_coeffs(rhat, wl.alpha, float(np.float32(wl.sigma)),
                                         es.ES_SCALE_PAPER)
            for _ in range(args.warmup):
                es.es_update(plan, seeds, coeffs, s_handle)
            torch.cuda.synchronize()
            evs = []
            for _ in range(args.steps):
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                es.es_update(plan, seeds, coeffs, s_handle)
                e1.record(stream)
                evs.append((e0, e1))
                launches += 1
            torch.cuda.synchronize()
            ms = sum(a.elapsed_time(b) for a, b in evs) / len(evs) if evs else float("nan")
            gbs = bytes_per_launch / (ms / 1e3) / 1e9
            gps = n * P / (ms / 1e3)
            t_hbm = bytes_per_launch / (hbm_gbs * 1e9) * 1e3
            t_imul = n * P / gauss_peak * 1e3
            t_gen = n * P / gen_peak * 1e3
            points.append({
                "population": n, "mean_ms": ms, "gbs": gbs, "gauss_per_s": gps,
                "hbm_frac": gbs / hbm_gbs, "alu_frac": gps / gauss_peak,
                "generator_frac": gps / gen_peak, "generator_pipelined_frac": gps / gen_pipe,
                "bound": "alu" if t_imul > t_hbm else "hbm",
                "roofline_frac": max(t_hbm, t_imul) / ms,
                "t_hbm_ms": t_hbm, "t_imul_ms": t_imul, "t_generator_ms": t_gen})
    plan.close()
    out = {"mode": "sweep", "metric": "es_update param*seed/s per population size",
           "unit": UNIT, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
           "dtype": "f32", "data": "synthetic",
           "config": dict(workload_config(args.workload, pops[-1] if pops else 0, 1),
                          populations=pops, call="es_update",
                          rewards="N(0,1) used as the normalised rewards; paper-scale coefficients"),
           "peaks": {"hbm_gbs": hbm_gbs, "hbm_source": peak_src,
                     "imul32_per_s": imul_peak, "gauss_per_s_imul": gauss_peak,
                     "gauss_per_s_generator": gen_peak,
                     "gauss_per_s_generator_pipelined": gen_pipe, "sms": sms,
                     "sm_max_mhz": sm_max_mhz},
           "bytes_per_launch": bytes_per_launch, "points": points,
           "gpu_launches": launches, "clocks": clk.summary()}
    if rank == 0:
        print(json.dumps(out), flush=True)


def _timed(torch, stream, fn, reps):
    """Mean milliseconds of fn() over reps runs, CUDA events on `stream`."""
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def _rates(P, gaussians_per_param, bytes_total, ms, peaks_):
    imul_peak, gauss_peak, gen_peak, _, _, hbm_gbs, _, _ = peaks_
    gps = gaussians_per_param * P / (ms / 1e3)
    gbs = bytes_total / (ms / 1e3) / 1e9
    return {"ms": ms, "gauss_per_s": gps, "gbs": gbs, "hbm_frac": gbs / hbm_gbs,
            "alu_frac": gps / gauss_peak, "generator_frac": gps / gen_peak}


def run_replay(args, rank, world, dist):
    """es_replay of K logged generations (N seeds each) in one pass over the
    parameters, against the same K generations as K es_update calls."""
    import torch
    from paper_2608_17310_gb300 import build, esopt as es

    build.build_library()
    dev_index = torch.cuda.current_device()
    torch.cuda.init()
    wl = I.WORKLOADS[args.workload]
    n = args.population or wl.population
    K = args.generations
    flat, params, plan, esize = param_set(es, args.workload)
    P = plan.numel
    stream = torch.cuda.current_stream()
    sh = stream.cuda_stream
    sigma = float(np.float32(wl.sigma))
    seeds, coeffs = [], []
    for g in range(K):
        # N(0, 1) rewards used as the normalised rewards (as in the sweep): no
        # generation of the log degenerates to an all-zero update
        seeds.append(I.population_seeds(n, generation=g))
        coeffs.append(es.es_update_coeffs(I.rewards("normal", n, seed=g), wl.alpha, sigma,
                                          es.ES_SCALE_PAPER))
    all_seeds, all_coeffs = np.concatenate(seeds), np.concatenate(coeffs)
    counts = np.full(K, n, dtype=np.int32)
    # launches es_replay makes: generations of fewer than 4 non-zero seeds
    # share a pass (<= ES_MAX_SEEDS seeds, <= 256 generations); a larger one
    # has a pass of its own; passes break only between generations
    passes, in_pass, gens = 0, 0, 0
    for g in range(K):
        nz = int(np.count_nonzero(coeffs[g]))
        own = nz >= 4
        if nz and gens and (own or in_pass + nz > es.ES_MAX_SEEDS or gens == 256):
            passes, in_pass, gens = passes + 1, 0, 0
        if nz:
            in_pass, gens = in_pass + nz, gens + 1
        if own:
            passes, in_pass, gens = passes + 1, 0, 0
    passes += 1 if gens else 0

    def replay():
        es.es_replay(plan, all_seeds, all_coeffs, counts, sh)

    def separate():
        for g in range(K):
            es.es_update(plan, seeds[g], coeffs[g], sh)

    pk = alu_peaks(torch, dev_index)
    with ClockSampler(dev_index) as clk:
        for _ in range(args.warmup):
            replay()
            separate()
        ms_r = _timed(torch, stream, replay, args.steps)
        ms_s = _timed(torch, stream, separate, args.steps)
    plan.close()
    live = int(sum(np.count_nonzero(c) for c in coeffs))      # seeds that are applied
    live_gens = int(sum(1 for c in coeffs if np.any(c != 0)))  # es_update calls that launch
    r = _rates(P, live, passes * 2 * esize * P, ms_r, pk)
    sep = _rates(P, live, live_gens * 2 * esize * P, ms_s, pk)
    out = {"mode": "replay", "metric": "seed-log replay param*seed/s", "unit": UNIT,
           "value": P * live / (ms_r / 1e3), "n_gpus": 1, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": ms_r, "higher_is_better": True,
           "dtype": "f32", "data": "synthetic",
           "config": dict(workload_config(args.workload, n, 1), generations=K,
                          seeds_per_replay=live, replay_passes=passes,
                          rewards="N(0,1) used as the normalised rewards"),
           "replay": r, "separate_updates": sep, "speedup": ms_s / ms_r,
           "gpu_launches": args.steps * (passes + live_gens), "clocks": clk.summary()}
    if rank == 0:
        print(json.dumps(out), flush=True)


def run_generator(args, rank, world, dist):
    """The generator alone: es_noise_fill materialises 2^k Gaussians of one
    seed (4 bytes written per Gaussian, below what HBM sustains at the
    generator's rate, so the launch is generator-bound), and es_noise_bits
    writes the raw Philox words of as many elements (HBM-bound)."""
    import torch
    from paper_2608_17310_gb300 import build, esopt as es

    build.build_library()
    dev_index = torch.cuda.current_device()
    torch.cuda.init()
    stream = torch.cuda.current_stream()
    sh = stream.cuda_stream
    n = 1 << args.gen_log2
    eps = torch.empty(n, dtype=torch.float32, device="cuda")
    nblocks = n >> 2
    words = torch.empty(4 * nblocks, dtype=torch.int32, device="cuda")
    pk = alu_peaks(torch, dev_index)
    seed = [1000]

    def fill():
        es.es_noise_fill(seed[0], 0, n, eps, sh)
        seed[0] += 1

    def bits():
        es.es_noise_bits(seed[0], 0, nblocks, words, sh)
        seed[0] += 1

    with ClockSampler(dev_index) as clk:
        for _ in range(args.warmup):
            fill()
            bits()
        ms_fill = _timed(torch, stream, fill, args.steps)
        ms_bits = _timed(torch, stream, bits, args.steps)
    fill_rates = _rates(n, 1, 4 * n, ms_fill, pk)
    bits_gbs = 16 * nblocks / (ms_bits / 1e3) / 1e9
    out = {"mode": "generator", "metric": "Gaussians/s of the noise generator (es_noise_fill)",
           "unit": "Gaussians/s", "value": fill_rates["gauss_per_s"], "n_gpus": 1,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_fill,
           "higher_is_better": True, "dtype": "f32", "data": "synthetic",
           "config": {"gaussians_per_launch": n,
                      "output": "fp32, %.2f GB (%s than L2)" % (4 * n / 1e9,
                                                                "larger" if 4 * n > L2_BYTES else "smaller"),
                      "philox_blocks_per_bits_launch": nblocks},
           "noise_fill": fill_rates,
           "noise_bits": {"ms": ms_bits, "words_per_s": 4 * nblocks / (ms_bits / 1e3),
                          "gbs": bits_gbs, "hbm_frac": bits_gbs / pk[5]},
           "gpu_launches": 2 * args.steps, "clocks": clk.summary()}
    if rank == 0:
        print(json.dumps(out), flush=True)


def run_antithetic(args, rank, world, dist):
    """A generation of N/2 antithetic pairs, steady state: each pair's flip from
    +sigma eps_i to -sigma eps_i is one es_restore_perturb on one seed (noise
    generated once); between pairs es_restore_perturb moves to the next seed;
    the generation ends with es_restore and es_update_perturb over the folded
    per-pair coefficients."""
    import torch
    from paper_2608_17310_gb300 import build, esopt as es

    build.build_library()
    dev_index = torch.cuda.current_device()
    torch.cuda.init()
    wl = I.WORKLOADS[args.workload]
    pairs = (args.population or wl.population) // 2
    flat, params, plan, esize = param_set(es, args.workload)
    P = plan.numel
    stream = torch.cuda.current_stream()
    sh = stream.cuda_stream
    sigma0, sigmaT = wl.sigma, SIGMA_FINAL.get(args.workload, wl.sigma)

    def sigma_at(t):
        return float(np.float32(es.es_sigma_cosine(sigma0, sigmaT, t, SCHEDULE_T)))

    def inputs(t):
        seeds = I.population_seeds(pairs, generation=t)
        rewards = I.rewards("uniform", 2 * pairs, seed=t)
        return seeds, rewards

    launches = [0]

    def step(t):
        sigma, sigma_next = sigma_at(t), sigma_at(t + 1)
        seeds, rewards = inputs(t)
        for i, sd in enumerate(seeds):
            es.es_restore_perturb(plan, int(sd), sigma, int(sd), -sigma, sh)      # + -> -
            if i + 1 < pairs:
                es.es_restore_perturb(plan, int(sd), -sigma, int(seeds[i + 1]), sigma, sh)
            else:
                es.es_restore(plan, int(sd), -sigma, sh)
        rhat = es.es_normalize_rewards(rewards, 1e-8)
        coeffs = es.es_fold_antithetic(rhat[:pairs], rhat[pairs:], wl.alpha, sigma,
                                       es.ES_SCALE_PAPER)
        es.es_update_perturb(plan, seeds, coeffs, int(inputs(t + 1)[0][0]), sigma_next, sh)
        launches[0] += 2 * pairs + 1

    es.es_perturb(plan, int(inputs(0)[0][0]), sigma_at(0), sh)
    pk = alu_peaks(torch, dev_index)
    for w in range(args.warmup):
        step(w)
    launches[0] = 0
    t_box = [args.warmup]

    def timed_step():
        step(t_box[0])
        t_box[0] += 1

    with ClockSampler(dev_index) as clk:
        ms = _timed(torch, stream, timed_step, args.steps)
    plan.close()
    members = 2 * pairs
    gauss = pairs * 1 + (pairs - 1) * 2 + 1 + (pairs + 1)
    passes = 2 * pairs + 1
    out = {"mode": "antithetic", "metric": "ES step param*member/s, antithetic pairs",
           "unit": "param*member/s", "value": P * members / (ms / 1e3), "n_gpus": 1,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
           "higher_is_better": True, "dtype": "f32", "data": "synthetic",
           "config": dict(workload_config(args.workload, members, 1), pairs=pairs,
                          gaussians_per_param=gauss, passes=passes),
           "rates": _rates(P, gauss, passes * 2 * esize * P, ms, pk),
           "gpu_launches": launches[0], "clocks": clk.summary()}
    if rank == 0:
        print(json.dumps(out), flush=True)


class PinnedHostBuffer:
    """Page-locked host memory for the e2e copies: anonymous mmap with
    transparent huge pages requested (madvise), registered with
    cudaHostRegister. On the GB300 machines huge-page-backed buffers copy at a
    steady 211 GB/s (H2D) / 193 GB/s (D2H); cudaHostAlloc'd memory varied
    between 100 and 204 GB/s from run to run, and a buffer with 11 % of its
    pages split to base size made the e2e step 2.2x slower. Falls back to
    torch's pinned allocator if registration fails."""

    def __init__(self, torch, like):
        import ctypes
        import mmap
        self.torch = torch
        self.addr = None
        self.hugepages_at_registration = None
        nbytes = like.numel() * like.element_size()
        self.nbytes = nbytes
        try:
            self.map = mmap.mmap(-1, nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
            addr = ctypes.addressof(ctypes.c_char.from_buffer(self.map))
            libc = ctypes.CDLL(None)
            libc.madvise(ctypes.c_void_p(addr), ctypes.c_size_t(nbytes), 14)  # MADV_HUGEPAGE
            arr = np.frombuffer(self.map, dtype=np.uint8)
            # The registration faults the pages in itself. Pages the CPU had
            # faulted in first were, in some runs, split out of their huge
            # pages once the GPU wrote to them, and copies through a partly
            # split buffer ran 5-9x slower; pages faulted in by the
            # registration were never split (measured).
            if int(torch.cuda.cudart().cudaHostRegister(addr, nbytes, 0)) != 0:
                raise OSError("cudaHostRegister failed")
            self.addr = addr
            self.hugepages_at_registration = self.hugepage_fraction()
            self.tensor = torch.from_numpy(arr).view(like.dtype)
            self.kind = "mmap + MADV_HUGEPAGE + cudaHostRegister"
        except Exception:
            self.map = None
            self.tensor = torch.empty(like.shape, dtype=like.dtype, pin_memory=True)
            self.kind = "torch pin_memory"

    def hugepage_fraction(self):
        """Share of the buffer backed by transparent huge pages (None if the
        buffer is torch's, or /proc/self/smaps cannot be read)."""
        if self.addr is None:
            return None
        lo, hi = self.addr, self.addr + self.nbytes
        huge, cur = 0, False
        try:
            with open("/proc/self/smaps") as f:
                for line in f:
                    head = line.split()[0]
                    if "-" in head and not head.endswith(":"):
                        a, b = (int(x, 16) for x in head.split("-"))
                        cur = a < hi and b > lo
                    elif cur and head == "AnonHugePages:":
                        huge += int(line.split()[1]) * 1024
        except (OSError, ValueError):
            return None
        return min(1.0, huge / self.nbytes)

    def close(self):
        if self.addr is not None:
            self.torch.cuda.synchronize()
            self.torch.cuda.cudart().cudaHostUnregister(self.addr)
            self.addr = None
        self.tensor = None
        self.map = None     # the mapping is released with its last reference


def host_memory_available() -> int:
    """MemAvailable of this node in bytes (0 if unknown)."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def e2e_fits(torch, nbytes: int, dist) -> bool:
    """Whether every rank on this node can page-lock its own copy of the
    parameter set with room to spare; all ranks take the same decision."""
    local = int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
    ok = host_memory_available() >= 1.5 * local * nbytes
    if dist is None:
        return ok
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([1 if ok else 0], dtype=torch.int32, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MIN)
    return bool(t.item())


def copy_groups(sizes, groups=8):
    """Ends (exclusive tensor indices) of the contiguous copy groups of the e2e
    leg. A group's copy back (and its copy in for the next step) starts when
    its last pass is done, so whatever copying is left when the last pass of
    the step ends is exposed. The groups therefore shrink towards the end: the
    last holds the trailing tensors up to 1/32 of the elements (at least one
    tensor), and each group before it up to twice as much as the one after it,
    while that stays below 1/groups of the elements; the tensors before them
    are split into groups of about 1/groups of the elements each. A tail group's
    round trip then overlaps the last passes of the groups after it."""
    total = sum(sizes)
    share = total / groups
    tail_ends, end, cap = [], len(sizes), total / 32
    while end > 1 and cap < share:
        start, acc = end, 0
        while start > 1 and (acc == 0 or acc + sizes[start - 1] <= cap):
            start -= 1
            acc += sizes[start]
        tail_ends.append(end)
        end = start
        cap = max(2 * cap, 2 * acc)
    head = sum(sizes[:end])
    nhead = max(1, round(head / share))
    ends, acc = [], 0
    for k in range(end):
        acc += sizes[k]
        if acc >= head * (len(ends) + 1) / nhead or k == end - 1:
            ends.append(k + 1)
    return ends + tail_ends[::-1]


class E2ELoop:
    """The generation with the parameter set in pinned host memory: every step
    copies it to the device, runs the generation through the C ABI and copies
    it back. The tensors are split into `groups` contiguous groups with a plan
    each, so that each group's first pass starts when its copy has landed and
    its copy back starts when its last pass is done (the middle passes use the
    whole plan). With copy_next, a group's copy to the device for the next step
    follows its copy back at once, on the same stream, so it runs while the
    other groups' last passes still compute; the next step's first pass of
    that group waits for it. The results are those of the unsplit calls: every
    call is elementwise (tested)."""

    def __init__(self, torch, es, plan, flat, params, wl, n, esize, sigma_at, s_handle, fused,
                 groups=8, nstreams=4, lead=2):
        self.torch, self.es, self.plan, self.flat = torch, es, plan, flat
        self.wl, self.n, self.sigma_at, self.s_handle, self.fused = wl, n, sigma_at, s_handle, fused
        self.nstreams, self.lead = nstreams, lead
        self.pending = None  # per group: the event of its copy in issued by the previous step
        # The first use of a fresh page-locked buffer sometimes splits some of
        # its huge pages, and copies through it then run 5-9x slower (the
        # kernel's thp_split_page count rises; a buffer allocated after a
        # release does not show it). So the buffer makes one round trip and,
        # if its huge-page share fell, is released and allocated again.
        self.attempts = 0
        for self.attempts in range(1, 6):
            self.pinned = PinnedHostBuffer(torch, flat)
            self.host = self.pinned.tensor
            self.host.copy_(flat)
            flat.copy_(self.host)
            torch.cuda.synchronize()
            before, after = self.pinned.hugepages_at_registration, self.pinned.hugepage_fraction()
            if before is None or after is None or after >= before - 0.005 or self.attempts == 5:
                break
            self.host = None
            self.pinned.close()
            self.pinned = None
        self.stream = torch.cuda.current_stream()
        self.copy_streams = [torch.cuda.Stream() for _ in range(nstreams)]
        self.bytes_per_copy = flat.numel() * esize
        ends = copy_groups([p.numel() for p in params], groups)
        self.spans, start = [], 0
        segs_all = es.segments_from_tensors(params)
        for e in ends:
            lo = params[start].data_ptr() - flat.data_ptr()
            hi = params[e - 1].data_ptr() - flat.data_ptr() + params[e - 1].numel() * esize
            if plan.scales is not None:
                group = es.es_plan_create_scaled(segs_all[start:e], plan.scales[start:e],
                                                 plan.dtype, params[start:e])
            else:
                group = es.es_plan_create(segs_all[start:e], plan.dtype, params[start:e])
            self.spans.append((lo // esize, hi // esize, group))
            start = e

    def _copy_in(self, g):
        """Copy of group g to the device on its copy stream; returns its event."""
        torch = self.torch
        a, b, _ = self.spans[g]
        cs = self.copy_streams[g % self.nstreams]
        with torch.cuda.stream(cs):
            self.flat[a:b].copy_(self.host[a:b], non_blocking=True)
            done = torch.cuda.Event()
            done.record(cs)
        return done

    def passes(self, seeds, sigma):
        """The generation's passes before its last one, in order, as
        (call, arguments after the plan) pairs."""
        es, n, sh = self.es, self.n, self.s_handle
        out = []
        if self.fused:
            # the previous step's last pass perturbed with seeds[0]
            for i in range(1, n):
                out.append((es.es_restore_perturb,
                            (int(seeds[i - 1]), sigma, int(seeds[i]), sigma, sh)))
            out.append((es.es_restore, (int(seeds[n - 1]), sigma, sh)))
        else:
            for i in range(n):
                out.append((es.es_perturb, (int(seeds[i]), sigma, sh)))
                out.append((es.es_restore, (int(seeds[i]), sigma, sh)))
        return out

    def step(self, t, record=None, copy_next=False):
        torch, es, plan = self.torch, self.es, self.plan
        wl, n, sh, stream = self.wl, self.n, self.s_handle, self.stream
        seeds, rewards = generation_inputs(wl, t, n)
        sigma, sigma_next = self.sigma_at(t), self.sigma_at(t + 1)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        ev[0].record(stream)
        # in: unless the previous step already issued them, every copy waits
        # only for the previous step; each group's first passes wait only for
        # its own copy
        if self.pending is None:
            for cs in self.copy_streams:
                cs.wait_stream(stream)
            landed = [self._copy_in(g) for g in range(len(self.spans))]
        else:
            landed, self.pending = self.pending, None
        # the first `lead` passes group by group, so that the groups copied
        # last (the smallest) get the earlier groups' passes to land in; the
        # rest on the whole plan
        todo = self.passes(seeds, sigma)
        lead = min(self.lead, len(todo))
        for (a, b, gplan), done in zip(self.spans, landed):
            stream.wait_event(done)
            for call, rest in todo[:lead]:
                call(gplan, *rest)
        ev[1].record(stream)
        for call, rest in todo[lead:]:
            call(plan, *rest)
        coeffs = es.es_update_coeffs(es.es_normalize_rewards(rewards, 1e-8), wl.alpha, sigma,
                                     es.ES_SCALE_PAPER)
        first_next = int(generation_inputs(wl, t + 1, n)[0][0])
        ev[2].record(stream)
        # out: last pass per group, then copy it back (and with copy_next, at
        # once to the device again for the next step)
        pending = []
        for g, (a, b, gplan) in enumerate(self.spans):
            if self.fused:
                es.es_update_perturb(gplan, seeds, coeffs, first_next, sigma_next, sh)
            else:
                es.es_update(gplan, seeds, coeffs, sh)
            cs = self.copy_streams[g % self.nstreams]
            cs.wait_stream(stream)
            with torch.cuda.stream(cs):
                self.host[a:b].copy_(self.flat[a:b], non_blocking=True)
            if copy_next:
                pending.append(self._copy_in(g))
        if copy_next:
            self.pending = pending
        else:
            for cs in self.copy_streams:
                stream.wait_stream(cs)
        ev[3].record(stream)
        if record is not None:
            record.append(ev)

    def close(self):
        for _, _, gplan in self.spans:
            gplan.close()
        self.spans = []
        self.host = None
        self.pinned.close()


def run_e2e(args, torch, es, plan, flat, params, wl, n, esize, sigma_at, s_handle, dist, world,
            fused, groups=8, nstreams=4):
    """e2e leg of the JSON line: E2ELoop timed over args.e2e_steps generations."""
    nbytes = flat.numel() * esize
    if not e2e_fits(torch, nbytes, dist):
        local = int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
        return {"value": None, "unit": UNIT, "unavailable":
                f"host memory: {local} ranks x {nbytes / 1e9:.1f} GB page-locked would exceed "
                f"2/3 of the {host_memory_available() / 1e9:.0f} GB available"}
    loop = E2ELoop(torch, es, plan, flat, params, wl, n, esize, sigma_at, s_handle, fused,
                   groups, nstreams)
    stream = loop.stream
    loop.step(0)
    torch.cuda.synchronize()
    barrier(dist)
    evs = []
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for k in range(args.e2e_steps):
        # each step's copy to the device is issued by the step before it,
        # except the first one's, which the first step issues itself: every
        # copy of the timed steps lies inside the timed region
        loop.step(args.warmup + k, evs, copy_next=k + 1 < args.e2e_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1), dist)
    phases = {"copy_in_and_first_passes": 0.0, "middle_passes": 0.0,
              "last_pass_and_copy_out": 0.0}
    for ev in evs:
        for name, a, b in (("copy_in_and_first_passes", 0, 1), ("middle_passes", 1, 2),
                           ("last_pass_and_copy_out", 2, 3)):
            phases[name] += ev[a].elapsed_time(ev[b]) / len(evs)
    kind, ngroups, bytes_per_copy = loop.pinned.kind, len(loop.spans), loop.bytes_per_copy
    lead = loop.lead
    huge = loop.pinned.hugepage_fraction()
    hp_fault = loop.pinned.hugepages_at_registration
    attempts = loop.attempts
    loop.close()
    P = sum(p.numel() for p in params)
    return {"value": world * P * n * args.e2e_steps / (ms / 1e3), "unit": UNIT,
            "steps": args.e2e_steps, "ms_per_step": ms / args.e2e_steps,
            "h2d_bytes_per_step": bytes_per_copy, "d2h_bytes_per_step": bytes_per_copy,
            "phase_ms": phases, "host_hugepage_fraction": huge,
            "host_hugepage_fraction_at_registration": hp_fault,
            "host_buffer_attempts": attempts,
            "layout": f"one page-locked host buffer ({kind}) and one device buffer "
                      f"holding every tensor; {ngroups} groups with a plan each, copies over "
                      f"{nstreams} streams, the groups shrinking towards the end; a group's "
                      f"copy back and its copy in for the next step run while the other "
                      f"groups' last passes compute, and its first {lead} passes (group by "
                      f"group) wait only for its own copy"}


# --- CPU oracle (cpu_baseline leg and the reference arm) ---------------------------------

def oracle_generation(workload: str, n: int, sigma: float, lo: int, count: int, step: int):
    """One ES generation (N perturb + restore pairs, the update) of the oracle on
    parameters [lo, lo + count) of the workload's first weight tensor. Returns
    (seconds of oracle work, parameters)."""
    from oracle import oracle as O
    wl = I.WORKLOADS[workload]
    g = np.arange(lo, lo + count, dtype=np.uint64)
    theta32 = I.normal_f32(g.size, lo, 0.02)
    dt = wl.dtype
    scale = 1.0
    if dt == "bf16":
        import torch
        theta = torch.from_numpy(theta32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    elif dt == "e4m3":
        import torch
        scale = float(np.float32(np.abs(theta32).max() / 448.0))
        theta = torch.from_numpy(theta32 / np.float32(scale)).to(torch.float8_e4m3fn) \
            .view(torch.uint8).numpy().copy()
    else:
        theta = theta32
    seeds, rewards = generation_inputs(wl, step, n)
    t0 = time.perf_counter()
    for i in range(n):
        theta = O.perturb(theta, g, int(seeds[i]), sigma, dt, scale)
        theta = O.restore(theta, g, int(seeds[i]), sigma, dt, scale)
    coeffs = O.update_coeffs(O.zscore(rewards), wl.alpha, sigma, 0)
    theta = O.update(theta, g, seeds, coeffs, dt, scale)
    return time.perf_counter() - t0, g.size


def _oracle_worker_init():
    import torch  # noqa: F401  (bf16 conversion of the inputs, loaded before timing)
    from oracle import oracle as O
    O.lib()


def _oracle_task(a):
    return oracle_generation(*a)


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return "unknown"


class OraclePool:
    """The unchanged oracle on every host core: one spawned worker per core,
    each running whole generations on its own slice of the parameters (the
    step is elementwise, so slices are independent). Spawned, never forked, so
    it is safe after CUDA has been initialised."""

    def __init__(self, workers: int):
        import multiprocessing as mp
        self.workers = workers
        self.pool = mp.get_context("spawn").Pool(workers, initializer=_oracle_worker_init)

    def generation(self, workload, n, sigma, per_worker, step):
        """Wall seconds of one generation over workers x per_worker parameters
        (fewer where the tensor is smaller), and the parameters covered."""
        numel = I.shapes_for(workload)[0].numel
        tasks = [(workload, n, sigma, lo, min(per_worker, numel - lo), step)
                 for lo in range(0, min(numel, self.workers * per_worker), per_worker)]
        t0 = time.perf_counter()
        res = self.pool.map(_oracle_task, tasks, chunksize=1)
        return time.perf_counter() - t0, sum(m for _, m in res)

    def close(self):
        self.pool.close()
        self.pool.join()


def cpu_baseline(workload, n, sigma):
    """The oracle on all host cores over about 2^22 parameters (10-30 s of CPU
    work), plus its single-thread rate on 2^20 parameters."""
    cores = host_cores()
    per_worker = max(1 << 16, (1 << 22) // cores)
    pool = OraclePool(cores)
    try:
        pool.generation(workload, n, sigma, 1 << 12, 0)            # workers up and warm
        wall, m = pool.generation(workload, n, sigma, per_worker, 0)
    finally:
        pool.close()
    secs1, m1 = oracle_generation(workload, n, sigma, 0, 1 << 20, 0)
    return {"value": m * n / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"one generation (N={n} perturb+restore, update) on {m} parameters of "
                      f"the {workload} set's first weight tensor, split over {cores} spawned "
                      f"workers of the unchanged plain-C oracle; {wall:.1f} s wall",
            "single_thread": {"value": m1 * n / secs1, "cores": 1, "params": m1,
                              "seconds": secs1},
            "cpu_model": cpu_model()}


def run_reference(args, rank, world):
    if rank != 0:
        return
    wl = I.WORKLOADS[args.workload]
    n = args.population or wl.population
    # the sigma the GPU line reports: the cosine schedule at the first timed step
    # (the oracle's schedule, equal to the library's to 1e-15)
    from oracle import oracle as O
    sigma = float(np.float32(O.sigma_cosine(wl.sigma, SIGMA_FINAL.get(args.workload, wl.sigma),
                                            args.warmup, SCHEDULE_T)))
    cores = host_cores()
    per_worker = 1 << 17
    pool = OraclePool(cores)
    try:
        for w in range(args.warmup):
            pool.generation(args.workload, n, sigma, per_worker, w)
        tot, m = 0.0, 0
        for k in range(args.steps):
            secs, m = pool.generation(args.workload, n, sigma, per_worker, args.warmup + k)
            tot += secs
    finally:
        pool.close()
    value = m * n * args.steps / tot if tot > 0 else 0.0
    desc = (f"each step: one generation (N={n}) of the unchanged plain-C oracle on {m} "
            f"parameters of the {args.workload} set, split over {cores} spawned workers")
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": 1e3 * tot / args.steps if args.steps else 0.0,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "f64", "data": "synthetic", "impl": "reference",
           "config": dict(workload_config(args.workload, n, 1), sigma=sigma, sample_params=m),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                            "sample": desc, "cpu_model": cpu_model()},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0},
           "gpu_launches": 0}
    print(json.dumps(out), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        # CPU work on rank 0 alone: no process group and no GPU for any rank.
        run_reference(args, int(os.environ.get("RANK", "0")),
                      int(os.environ.get("WORLD_SIZE", "1")))
        return
    rank, world, dist = dist_setup(args)
    try:
        if args.sweep:
            run_sweep(args, rank, world, dist)
        elif args.replay:
            run_replay(args, rank, world, dist)
        elif args.antithetic:
            run_antithetic(args, rank, world, dist)
        elif args.generator:
            run_generator(args, rank, world, dist)
        elif args.pipe_peaks:
            run_pipe_peaks(args, rank, world, dist)
        else:
            run_ours(args, rank, world, dist)
    finally:
        if dist is not None:
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
