#!/usr/bin/env python
"""Benchmark of the TGV-KV eviction step (score + budget + select + compact).

Prints ONE JSON line on stdout (rank 0).  Metric: eviction microseconds per
decoder layer for the fused tgvkv_evict over all layers of one request, plus
the achieved HBM bandwidth of the step and the roofline of its dominant kernel.

  python bench.py [--gpus N --steps K --warmup W] [--config next --ratio 0.05]
  python bench.py --impl reference ...   (the fp64 CPU oracle, same metric)

The headline line is the LLaVA-NeXT-shaped workload (32 layers, 32/32 heads,
N = 3008, 788 MB of K: the largest by bytes, where the HBM roof binds) at 5%
vision retention; the same line carries a `per_config` block with every
workload and budget (bounded steps each).

Multi-GPU (torchrun, one rank per GPU): every rank runs its own replica of the
workload (the step has no data-path exchange); the timed region is bracketed by
a barrier and synchronisation and the max over ranks is reported.
"""
import os
import sys

if "reference" in sys.argv[1:]:
    # the reference arm is the single-threaded oracle: BLAS gets one thread
    # before numpy is first imported
    for _k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS",
               "BLIS_NUM_THREADS", "VECLIB_MAXIMUM_THREADS"):
        os.environ[_k] = "1"

import argparse
import ctypes
import hashlib
import json
import math
import statistics
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2606_03075_gb300 import synth  # noqa: E402

METRIC = "eviction µs/layer and achieved HBM GB/s vs peak (score+budget+select+compact)"
UNIT = "µs/layer"
L2_BYTES = 129 * 2 ** 20


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="tgvkv", choices=["tgvkv", "reference"])
    ap.add_argument("--config", default="next", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--ratio", type=float, default=None)
    ap.add_argument("--layers", type=int, default=0,
                    help="profiling: cut the workload to this many layers (0 = all)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="wall-clock target of the oracle CPU-baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-next-rows", action="store_true",
                    help="skip timing the Eq. 7 / all-token basis / sink variants of the step")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip the per_config block (every workload and budget)")
    ap.add_argument("--per-config-steps", type=int, default=100)
    ap.add_argument("--record-traffic", metavar="CSV",
                    help="record the DRAM bytes of one kernel launch from `ncu -i REP --page raw "
                         "--csv` output into profiles/traffic.json (for --stage and --config)")
    ap.add_argument("--stage", default="score", choices=["score", "budget", "select", "compact"])
    return ap.parse_args()


# --------------------------------------------------------------------------
# workload description and algorithmic byte counts
# --------------------------------------------------------------------------
def workload_of(args):
    """The named workload, cut to --layers layers when given (small profiling
    cases of the same launch configuration)."""
    wl = synth.WORKLOADS[args.config]
    if args.layers:
        import dataclasses
        wl = dataclasses.replace(wl, L=args.layers)
    return wl


def rotation_sets(wl):
    """Input sets the GPU arm rotates through so that every step's inputs
    miss L2 (their total is above twice the L2 size)."""
    in_bytes = sum(wl.input_bytes().values())
    return max(2, math.ceil(2 * L2_BYTES / in_bytes) + 1), in_bytes


def full_config(wl, ratio, world):
    """The `config` of a bench line (both arms)."""
    n_sets, in_bytes = rotation_sets(wl)
    return dict(workload_config(wl, ratio),
                l2="inputs larger than L2: %d rotating input sets of %.0f MB "
                   "(L2 %d MB)" % (n_sets, in_bytes / 1e6, L2_BYTES >> 20),
                parallelism=f"replicas x{world}")


def workload_config(wl, ratio):
    return {"workload": f"{wl.name}: L={wl.L} H_q/H_kv={wl.H_q}/{wl.H_kv} d={wl.d} "
                        f"N={wl.N} (N_v={wl.N_v}, N_t={wl.N_t}) query rows={wl.n_win} "
                        f"budget r={ratio} of vision KV",
            "L": wl.L, "H_q": wl.H_q, "H_kv": wl.H_kv, "head_dim": wl.d, "N": wl.N,
            "N_v": wl.N_v, "n_win": wl.n_win, "ratio": ratio, "weights": wl.weights,
            "keys": wl.keys}


def budget_total(wl, ratio):
    return int(math.floor(ratio * float(wl.N_v * wl.L) + 0.5))


def step_bytes(wl, ratio):
    """Roofline bytes of one step: K read once + compacted K/V written."""
    rows = wl.H_kv * (wl.L * wl.N_t + budget_total(wl, ratio))
    k_read = wl.L * wl.H_kv * wl.N * wl.d * 2
    kv_written = 2 * rows * wl.d * 2
    return k_read + kv_written, rows


def full_step_bytes(wl, ratio):
    """All algorithmic bytes of one fused step: K read once, Q read, scores
    written and read back, the kept K/V rows read and written, idx and offsets."""
    _, rows = step_bytes(wl, ratio)
    k = wl.L * wl.H_kv * wl.N * wl.d * 2
    q = wl.L * wl.H_q * wl.n_win * wl.d * 2
    scores = wl.L * wl.H_kv * wl.N_v * 4
    return k + q + 2 * scores + 4 * rows * wl.d * 2 + 4 * rows + 8 * (wl.L * wl.H_kv + 1)


def stage_bytes(wl, ratio):
    """Algorithmic bytes of each kernel launch (all layers)."""
    _, rows = step_bytes(wl, ratio)
    k = wl.L * wl.H_kv * wl.N * wl.d * 2
    q = wl.L * wl.H_q * wl.n_win * wl.d * 2
    scores = wl.L * wl.H_kv * wl.N_v * 4
    return {
        "score": k + q + scores,
        "budget": 8 * wl.L,
        "select": scores + 4 * rows + 8 * (wl.L * wl.H_kv + 1),
        "compact": 4 * rows * wl.d * 2 + 4 * rows,
        # the fused select + gather of tgvkv_evict (tgvkv_select_compact)
        "tail": scores + 4 * rows * wl.d * 2 + 4 * rows + 8 * (wl.L * wl.H_kv + 1),
    }


NOMINAL_HBM_GBS = 7900.0      # GB300 HBM3e, nominal
NOMINAL_BF16_TFLOPS = 2250.0  # dense, nominal
MUFU_EX2_PER_CLK_SM = 32      # ex2.approx.f32 results per clock per SM, measured on GB300
GB300_SMS = 152


def score_exps(wl):
    """Exponentials of the score kernel's two passes: every (query row, visible
    key) pair in pass A, every (query row, visible vision key) pair in pass B."""
    pos = wl.text_pos.astype(np.int64)
    vis_le = np.cumsum(wl.modality.astype(np.int64))[pos]
    return int(wl.L * wl.H_q * ((pos + 1).sum() + vis_le.sum()))


def score_flops(wl):
    """Algorithmic FLOPs of the score kernel: the logits q.k of every text-query
    row of every query head against each key it attends to (causal), once."""
    visible = int((wl.text_pos.astype(np.int64) + 1).sum())
    return 2 * wl.d * wl.L * wl.H_q * visible


# each kernel's source with the headers it includes (a change to any of them
# invalidates a recorded ncu traffic figure)
KERNEL_SOURCES = {"score": ("score_tc.cu", "budget.cuh", "rowstat.cuh", "tc05.cuh", "common.cuh"),
                  "budget": ("budget.cu", "budget.cuh", "common.cuh"),
                  "select": ("select.cu", "common.cuh"),
                  "compact": ("compact.cu", "common.cuh"),
                  "tail": ("select.cu", "compact.cu", "common.cuh")}


def source_hash(stage):
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[stage]:
        with open(os.path.join(ROOT, "paper_2606_03075_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(stage, workload):
    """DRAM bytes per launch from a committed ncu capture, if the kernel source
    is unchanged since the capture."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        rec = json.load(open(path))[stage][workload]
    except (OSError, KeyError, ValueError):
        return None
    return rec["dram_bytes_per_launch"] if rec.get("source_sha") == source_hash(stage) else None


_BYTE_UNITS = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}


def record_traffic(csv_path, stage, workload):
    """Write dram__bytes_read.sum + dram__bytes_write.sum of the first kernel in
    an ncu raw-page CSV export to profiles/traffic.json."""
    import csv
    rows = list(csv.reader(open(csv_path)))
    head, units, vals = rows[0], rows[1], rows[2]
    total = 0.0
    for name in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
        i = head.index(name)
        total += float(vals[i].replace(",", "")) * _BYTE_UNITS[units[i]]
    kernel = vals[head.index("Kernel Name")] if "Kernel Name" in head else "?"
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        rec = json.load(open(path))
    except (OSError, ValueError):
        rec = {}
    rec.setdefault(stage, {})[workload] = {
        "dram_bytes_per_launch": int(round(total)), "source_sha": source_hash(stage),
        "kernel": kernel.split("(")[0]}
    with open(path, "w") as f:
        json.dump(rec, f, indent=1, sort_keys=True)
        f.write("\n")
    print(json.dumps(rec[stage][workload]))


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


def kernel_roof(wl, ratio, stage, launch_ms, peaks, peak_src="measured"):
    """Binding roof of one kernel launch: HBM unless the kernel's algorithmic
    FLOPs take longer than its bytes at the measured peaks (grouped-query
    shapes of the score kernel)."""
    hbm_peak = float(peaks["hbm_gbs"])
    tensor_peak = float(peaks["bf16_tflops"])
    nbytes = stage_bytes(wl, ratio)[stage]
    flops = score_flops(wl) if stage == "score" else 0
    if flops / (tensor_peak * 1e12) > nbytes / (hbm_peak * 1e9):
        roof = {"bound": "tensor", "achieved": flops / (launch_ms * 1e-3) / 1e12,
                "peak": tensor_peak, "unit": "TFLOP/s",
                "peak_source": f"{peak_src} bf16_tflops (MEASURED_PEAKS.json, burst)"}
    else:
        roof = {"bound": "hbm", "achieved": nbytes / (launch_ms * 1e-3) / 1e9,
                "peak": hbm_peak, "unit": "GB/s",
                "peak_source": f"{peak_src} hbm_gbs (MEASURED_PEAKS.json)"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["frac_nominal"] = roof["achieved"] / (NOMINAL_HBM_GBS if roof["bound"] == "hbm"
                                               else NOMINAL_BF16_TFLOPS)
    roof["bytes_per_launch"] = nbytes
    roof["flops_per_launch"] = flops
    return roof


def _roof_brief(roof, launch_ms):
    return {"launch_ms": launch_ms, "bound": roof["bound"], "achieved": roof["achieved"],
            "unit": roof["unit"], "peak": roof["peak"], "frac": roof["frac"],
            "bytes_per_launch": roof["bytes_per_launch"]}


def mufu_of(wl, score_ms, clk_mhz):
    """The score kernel's exponentials against the MUFU rate at the clock seen."""
    exps = score_exps(wl)
    m = {"exps_per_launch": exps,
         "achieved_G_per_s": exps / (score_ms * 1e-3) / 1e9,
         "peak_G_per_s": MUFU_EX2_PER_CLK_SM * GB300_SMS * clk_mhz * 1e6 / 1e9,
         "peak_source": f"{MUFU_EX2_PER_CLK_SM} ex2/clk/SM measured x {GB300_SMS} SMs x "
                        f"{clk_mhz:.0f} MHz median under load"}
    m["frac"] = m["achieved_G_per_s"] / m["peak_G_per_s"]
    return m


# --------------------------------------------------------------------------
# clocks during the timed region (NVML through ctypes; nvidia-smi fallback)
# --------------------------------------------------------------------------
_REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
            0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}


_REJECTING = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


def clocks_rejected(summary) -> bool:
    """A timed region whose clocks saw a hardware or thermal slowdown, or whose
    median SM clock sat below 80% of the maximum with no reason recorded (a
    clock lock left behind by someone else), does not count; sw_power_cap is
    normal under load and is only noted."""
    reasons = set(summary.get("reasons") or ())
    if reasons & set(_REJECTING):
        return True
    mhz, top = summary.get("sm_mhz"), summary.get("sm_max_mhz")
    return bool(mhz and top and mhz < 0.8 * top and not reasons)


class ClockSampler:
    def __init__(self, torch_dev):
        self.samples, self.reasons, self.max_mhz, self.ok = [], set(), None, False
        self._stop = threading.Event()
        try:
            self.nvml = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nvml.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            got = False
            try:
                import torch
                pr = torch.cuda.get_device_properties(torch_dev)
                bus = f"{pr.pci_domain_id:08x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0"
                got = self.nvml.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(self.h)) == 0
            except Exception:
                got = False
            if not got:
                vis = os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0]
                idx = int(vis) if vis.isdigit() else 0
                if self.nvml.nvmlDeviceGetHandleByIndex_v2(idx, ctypes.byref(self.h)) != 0:
                    return
            m = ctypes.c_uint()
            if self.nvml.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(m)) == 0:
                self.max_mhz = m.value
            self.ok = True
        except OSError:
            self.ok = False

    def _run(self):
        c, r = ctypes.c_uint(), ctypes.c_ulonglong()
        get_r = getattr(self.nvml, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            self.nvml.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if self.nvml.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(c)) == 0:
                self.samples.append(c.value)
            if get_r(self.h, ctypes.byref(r)) == 0:
                for bit, name in _REASONS.items():
                    if r.value & bit:
                        self.reasons.add(name)
            time.sleep(0.002)

    def __enter__(self):
        if self.ok:
            self.t = threading.Thread(target=self._run, daemon=True)
            self.t.start()
        return self

    def __exit__(self, *a):
        if self.ok:
            self._stop.set()
            self.t.join()

    def summary(self):
        if not self.ok or not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                    "samples": len(self.samples), "source": "nvml unavailable"}
        return {"sm_mhz": statistics.median(self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": sorted(self.reasons), "samples": len(self.samples), "source": "nvml"}


# --------------------------------------------------------------------------
# CPU baseline: the oracle on a bounded sample of the workload
# --------------------------------------------------------------------------
def oracle_unit(wl, layer_inputs, l, g, ratio):
    """The oracle's work for one (layer, KV head): Eq. 2/6/8 scores of its G
    query heads, a TVB split, TPR selection and the compaction gather."""
    import numpy as np
    import oracle
    q, k, v, w = layer_inputs
    G = wl.G
    scale = 1.0 / math.sqrt(wl.d)
    qq = oracle.widen_bf16(q[g * G:(g + 1) * G])[None]
    kk = oracle.widen_bf16(k[g:g + 1])[None]
    s, st = oracle.twr_scores_tvb_stat(qq, kk, wl.modality, wl.text_pos, w[None].astype(np.float64),
                                       scale, 1)
    total = budget_total(wl, ratio)
    budgets = oracle.tvb_budgets(np.full(wl.L, st[0]), total, wl.N_v)
    off, idx = oracle.tpr_select(s, budgets[l:l + 1], wl.modality)
    oracle.compact(k[None, g:g + 1], v[None, g:g + 1], off, idx)


_ONE_THREAD = {"OMP_NUM_THREADS": "1", "OPENBLAS_NUM_THREADS": "1", "MKL_NUM_THREADS": "1",
               "BLIS_NUM_THREADS": "1", "VECLIB_MAXIMUM_THREADS": "1"}


def _oracle_units_worker(job):
    """Run the oracle on the given (layer, KV head) units and return the seconds
    the oracle took (a process of its own, BLAS limited to one thread by the
    environment; the inputs are drawn before the clock starts)."""
    name, ratio, seed, units = job
    wl = synth.WORKLOADS[name]
    layers = {l: synth.draw_layer(wl, seed, l) for l in sorted({l for l, _ in units})}
    t = time.perf_counter()
    for l, g in units:
        oracle_unit(wl, layers[l], l, g, ratio)
    return time.perf_counter() - t


_ARM_PARTS = {"0xd4f": "Arm Neoverse-V2", "0xd40": "Arm Neoverse-V1", "0xd0c": "Arm Neoverse-N1",
              "0xd49": "Arm Neoverse-N2"}


def cpu_model():
    try:
        for line in open("/proc/cpuinfo"):
            key = line.split(":")[0].strip().lower()
            if key in ("model name", "cpu part", "hardware"):
                val = line.split(":", 1)[1].strip()
                return _ARM_PARTS.get(val.lower(), val)
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def run_cpu_baseline(wl, ratio, seed, seconds):
    """The fp64 oracle on this host: single-threaded, and on all cores (one
    single-threaded process per core over (layer, KV head) units)."""
    import multiprocessing as mp
    cores = os.cpu_count() or 1
    all_units = [(l, g) for l in range(wl.L) for g in range(wl.H_kv)]
    # the sample cycles over the workload's units when the whole workload takes
    # less than the time asked for
    units = [all_units[i % len(all_units)] for i in range(64 * len(all_units))]
    saved = {k: os.environ.get(k) for k in _ONE_THREAD}
    os.environ.update(_ONE_THREAD)
    try:
        ctx = mp.get_context("spawn")      # never fork after the GPU has been used
        with ctx.Pool(1) as pool:          # single-threaded: grow the sample to ~seconds/2
            n, spent1 = 1, 0.0
            while True:
                spent1 = pool.map(_oracle_units_worker, [(wl.name, ratio, seed, units[:n])])[0]
                if spent1 > seconds / 2 or n >= len(units):
                    break
                n = min(len(units), max(n + 1, int(n * (seconds / 2) / max(spent1, 1e-3))))
        single = spent1 / n * wl.H_kv * 1e6
        # all cores: about seconds/4 of oracle work per process, all processes at once;
        # the slowest process's time stands for the parallel wall time
        per_core = max(1, int(n * 0.5))
        jobs = [(wl.name, ratio, seed, [units[(c * per_core + i) % len(units)] for i in range(per_core)])
                for c in range(cores)]
        with ctx.Pool(cores) as pool:
            pool.map(_oracle_units_worker, [(wl.name, ratio, seed, units[:1])] * cores, chunksize=1)
            wall = max(pool.map(_oracle_units_worker, jobs, chunksize=1))
        multi = wall / (cores * per_core) * wl.H_kv * 1e6
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return {"value": multi, "unit": UNIT, "cores": cores, "kind": "oracle",
            "single_thread_value": single, "cpu_model": cpu_model(),
            "sample": f"fp64 numpy oracle, BLAS one thread per process: {n} (layer, KV head) "
                      f"units of {wl.name} (cycling over its {len(all_units)}) single-threaded "
                      f"({spent1:.1f} s), then {per_core} "
                      f"units on each of {cores} cores in parallel processes ({wall:.1f} s wall); "
                      f"us/layer = time per unit x H_kv={wl.H_kv} (value: all cores)"}


# --------------------------------------------------------------------------
# reference arm: the oracle, timed per step on a bounded sample
# --------------------------------------------------------------------------
def run_reference(args, rank, world):
    if rank != 0:
        return 0
    wl = workload_of(args)
    ratio = args.ratio if args.ratio is not None else wl.ratios[0]
    units = [(l, g) for l in range(wl.L) for g in range(wl.H_kv)]
    cache = {}

    def step(s):
        l, g = units[s % len(units)]
        if l not in cache:
            cache.clear()
            cache[l] = synth.draw_layer(wl, args.seed, l)
        t = time.perf_counter()
        oracle_unit(wl, cache[l], l, g, ratio)
        return time.perf_counter() - t

    for s in range(args.warmup):
        step(s)
    times = [step(args.warmup + s) for s in range(args.steps)]
    mean = sum(times) / len(times)
    value = mean * wl.H_kv * 1e6
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": mean * 1e3, "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": full_config(wl, ratio, world),
            "cpu_baseline": {"kind": "oracle", "cores": 1, "value": value,
                             "unit": UNIT,
                             "sample": f"each step = one (layer, KV head) unit of {wl.name} "
                                       f"(scores of its {wl.G} query heads, TVB split, TPR "
                                       f"select, gather), fp64 numpy on one thread (BLAS "
                                       f"limited to one thread); µs/layer = step "
                                       f"time x H_kv={wl.H_kv}"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------------------
# every workload and budget, bounded steps each
# --------------------------------------------------------------------------
PER_CONFIG = [("tiny", 0.25), ("llava15", 0.05), ("llava15", 0.20), ("next", 0.05),
              ("next", 0.10), ("next", 0.20), ("qwen25", 0.05), ("video", 0.05)]


def run_per_config(api, torch, dev, stream, barrier, seed, n_steps, inputs=None):
    """The fused step (tgvkv_evict), its score kernel alone (tgvkv_score), its
    select + gather alone (tgvkv_select_compact) and one decode step over the
    compacted cache it made (tgvkv_decode) on every workload and budget:
    n_steps timed calls each after 3 warm-up calls, inputs rotated past L2.
    Returns {"<name> r=<ratio>": {...}} and the clocks seen over the whole
    block."""
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks["hbm_gbs"])
    res = {}
    with ClockSampler(dev) as clocks:
        for name in dict.fromkeys(n for n, _ in PER_CONFIG):
            wl = synth.WORKLOADS[name]
            inp = (inputs or {}).get(name) or synth.generate(wl, seed=seed)
            in_bytes = sum(wl.input_bytes().values())
            n_sets = max(2, math.ceil(2 * L2_BYTES / in_bytes) + 1)

            def up(a, dtype=None):
                t = torch.from_numpy(np.ascontiguousarray(a)).to(dev)
                return t.view(dtype) if dtype is not None else t

            sets = [dict(q=up(inp["q"], torch.bfloat16), k=up(inp["k"], torch.bfloat16),
                         v=up(inp["v"], torch.bfloat16), modality=up(inp["modality"]),
                         text_pos=up(inp["text_pos"]), w=up(inp["w"])) for _ in range(n_sets)]
            del inp
            desc = api.desc_for_workload(wl)
            ws = api.new_workspace(desc, dev)
            for cname, ratio in PER_CONFIG:
                if cname != name:
                    continue
                out = api.alloc_outputs(desc, ratio, dev)

                def evict(i):
                    x = sets[i % n_sets]
                    api.tgvkv_evict(desc, x["q"], x["k"], x["v"], x["modality"], x["text_pos"],
                                    x["w"], ratio, out, ws, stream)

                def score(i):
                    x = sets[i % n_sets]
                    api.tgvkv_score(desc, x["q"], x["k"], x["modality"], x["text_pos"], x["w"],
                                    out.scores, out.tvb_stat, ws, stream)

                def timed(call):
                    for i in range(3):
                        call(i)
                    barrier()
                    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    for i in range(n_steps):
                        call(3 + i)
                    b.record(stream)
                    barrier()
                    return a.elapsed_time(b) / n_steps      # ms per call

                def tail(i):
                    # the evict's select + gather alone, on the last evict's
                    # scores and budgets, K/V rotated as above
                    x = sets[i % n_sets]
                    api.tgvkv_select_compact(desc, out.scores, None, out.budgets, x["modality"],
                                             x["k"], x["v"], out.offsets, out.idx, out.k_out,
                                             out.v_out, ws, stream)

                step_ms = timed(evict)
                score_ms = timed(score)
                evict(0)
                tail_ms = timed(tail)

                # one decode step over the compacted cache this step made (the
                # consumer), copies of the cache rotated past L2
                n_rows = int(out.offsets[-1].item())
                comp_bytes = 2 * n_rows * wl.d * 2
                n_cp = max(2, math.ceil(2 * L2_BYTES / max(comp_bytes, 1)) + 1)
                comp = [(out.k_out[:n_rows].clone(), out.v_out[:n_rows].clone())
                        for _ in range(n_cp)]
                offs = out.offsets.clone()
                qdec = torch.from_numpy(synth.to_bf16_bits(
                    np.random.default_rng(seed + 11).standard_normal((wl.L, wl.H_q, wl.d))
                    .astype(np.float32))).to(dev).view(torch.bfloat16)
                odec = torch.empty((wl.L, wl.H_q, wl.d), dtype=torch.float32, device=dev)

                def decode(i):
                    kk, vv = comp[i % n_cp]
                    api.tgvkv_decode(desc, qdec, kk, vv, offs, odec, ws, stream)

                dec_ms = timed(decode)
                del comp
                bits = api.tgvkv_status(ws, stream)
                if bits != 0:
                    raise RuntimeError(f"device status bits 0x{bits:x} in {name} r={ratio}")
                sbytes, rows = step_bytes(wl, ratio)
                step_gbs = sbytes / (step_ms * 1e-3) / 1e9
                roof = kernel_roof(wl, ratio, "score", score_ms, peaks, peak_src)
                clk = clocks.summary().get("sm_mhz") or float(peaks.get("sm_max_mhz", 2070.0))
                res[f"{name} r={ratio}"] = {
                    "us_per_layer": step_ms * 1e3 / wl.L, "step_ms": step_ms,
                    "step_bytes": sbytes, "step_gbs": step_gbs, "step_frac": step_gbs / hbm_peak,
                    "score_kernel": {"launch_ms": score_ms, "bound": roof["bound"],
                                     "achieved": roof["achieved"], "unit": roof["unit"],
                                     "peak": roof["peak"], "frac": roof["frac"],
                                     "share_of_step": score_ms / step_ms,
                                     "traffic": recorded_traffic("score", name)},
                    "score_mufu_frac": mufu_of(wl, score_ms, clk)["frac"],
                    "tail_kernel": _roof_brief(kernel_roof(wl, ratio, "tail", tail_ms, peaks,
                                                           peak_src), tail_ms),
                    "tail_ms": step_ms - score_ms, "rows_kept": rows, "steps": n_steps,
                    "decode": {"us_per_token": dec_ms * 1e3,
                               "gbs": comp_bytes / (dec_ms * 1e-3) / 1e9,
                               "frac": comp_bytes / (dec_ms * 1e-3) / 1e9 / hbm_peak,
                               "rows": n_rows}}
                del out
            del sets, ws
            torch.cuda.empty_cache()
    return res, clocks.summary()


# --------------------------------------------------------------------------
# GPU arm
# --------------------------------------------------------------------------
def main():
    args = parse()
    if args.record_traffic:
        return record_traffic(args.record_traffic, args.stage, args.config)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if args.impl == "reference":
        return run_reference(args, rank, world)

    import torch
    import torch.distributed as dist

    from paper_2606_03075_gb300 import build
    build.build()
    from paper_2606_03075_gb300 import api

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    wl = workload_of(args)
    ratio = args.ratio if args.ratio is not None else wl.ratios[0]
    desc = api.desc_for_workload(wl)
    inp = synth.generate(wl, seed=args.seed + rank)
    n_sets, in_bytes = rotation_sets(wl)

    def upload(a, dtype=None):
        t = torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        return t.view(dtype) if dtype is not None else t

    sets = []
    for i in range(n_sets):
        sets.append(dict(q=upload(inp["q"], torch.bfloat16), k=upload(inp["k"], torch.bfloat16),
                         v=upload(inp["v"], torch.bfloat16), modality=upload(inp["modality"]),
                         text_pos=upload(inp["text_pos"]), w=upload(inp["w"])))
    ws = api.new_workspace(desc, dev)
    out = api.alloc_outputs(desc, ratio, dev)
    launches_per_step = api.tgvkv_evict_launches(desc)
    stream = torch.cuda.current_stream(dev)

    def evict(s):
        x = sets[s % n_sets]
        api.tgvkv_evict(desc, x["q"], x["k"], x["v"], x["modality"], x["text_pos"], x["w"],
                        ratio, out, ws, stream)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    # ---- warm-up, then the timed region (fused path)
    for s in range(args.warmup):
        evict(s)
    bits = api.tgvkv_status(ws, stream)
    if bits != 0:
        raise RuntimeError(f"device status bits 0x{bits:x} set during warm-up")
    # Events only at the two ends: an event recorded between two evictions
    # would end the programmatic dependency between the previous eviction's
    # select + gather and the next score kernel, and time a different program
    # from the one a caller runs back to back.
    def timed_region():
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier()
        with ClockSampler(dev) as clocks:
            t_wall = time.perf_counter()
            t0.record(stream)
            for s in range(args.steps):
                evict(args.warmup + s)
            t1.record(stream)
            barrier()
            t_wall = time.perf_counter() - t_wall
        return t0.elapsed_time(t1), t_wall, clocks.summary()

    region_ms, t_wall, clocks = timed_region()
    # a region the clocks disqualify is measured once more (every rank agrees)
    bad = torch.tensor([1.0 if clocks_rejected(clocks) else 0.0], device=dev)
    if world > 1:
        dist.all_reduce(bad, op=dist.ReduceOp.MAX)
    rejected_clocks = None
    if bad.item() > 0:
        rejected_clocks = clocks
        region_ms, t_wall, clocks = timed_region()
    bits = api.tgvkv_status(ws, stream)
    if bits != 0:
        raise RuntimeError(f"device status bits 0x{bits:x} set in the timed region")
    region = torch.tensor([region_ms], device=dev, dtype=torch.float64)
    if world > 1:
        dist.all_reduce(region, op=dist.ReduceOp.MAX)
    region_ms = float(region.item())
    us_per_layer = region_ms * 1e3 / (args.steps * wl.L * world)

    # ---- per-step spread (event pair around each eviction)
    n_iso = min(args.steps, 64)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(n_iso)]
    barrier()
    for s in range(n_iso):
        ev[s][0].record(stream)
        evict(s)
        ev[s][1].record(stream)
    barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev]

    # ---- per-stage breakdown (the entry points with events between them; the
    # fused select + gather follows the budget, as in the step)
    stages = ["score", "budget", "tail", "select", "compact"]
    sev = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(args.steps)]
    barrier()
    for s in range(args.steps):
        x = sets[s % n_sets]
        e = sev[s]
        e[0].record(stream)
        api.tgvkv_score(desc, x["q"], x["k"], x["modality"], x["text_pos"], x["w"], out.scores,
                        out.tvb_stat, ws, stream)
        e[1].record(stream)
        api.tgvkv_budget(desc, out.tvb_stat, ratio, out.budgets, ws, stream)
        e[2].record(stream)
        api.tgvkv_select_compact(desc, out.scores, None, out.budgets, x["modality"], x["k"], x["v"],
                                 out.offsets, out.idx, out.k_out, out.v_out, ws, stream)
        e[3].record(stream)
        api.tgvkv_select(desc, out.scores, out.budgets, x["modality"], out.offsets, out.idx, ws,
                         stream)
        e[4].record(stream)
        api.tgvkv_compact(desc, x["k"], x["v"], out.offsets, out.idx, out.k_out, out.v_out, ws,
                          stream)
        e[5].record(stream)
    barrier()
    stage_ms = {st: statistics.mean(sev[s][i].elapsed_time(sev[s][i + 1]) for s in range(args.steps))
                for i, st in enumerate(stages)}

    # ---- the widened path (Eq. 7 weights, all-token basis, sinks): the same
    # evict call with the descriptor's options, inputs rotated as above
    next_rows = {}
    if not args.no_next_rows:
        variants = {"eq7_weights": dict(weights="eq7"),
                    "all_token_basis": dict(basis="all"),
                    "sinks_4_1": dict(keep_first=4, keep_last=1),
                    "eq7_all_sinks": dict(weights="eq7", basis="all", keep_first=4, keep_last=1)}
        n_var = max(3, min(args.steps, 100))
        for vname, opts in variants.items():
            dv = api.desc_for_workload(wl, **opts)
            wsv = api.new_workspace(dv, dev)
            outv = api.alloc_outputs(dv, ratio, dev)

            def evict_v(s):
                x = sets[s % n_sets]
                api.tgvkv_evict(dv, x["q"], x["k"], x["v"], x["modality"], x["text_pos"],
                                None if opts.get("weights") == "eq7" else x["w"], ratio, outv,
                                wsv, stream)

            for s in range(3):
                evict_v(s)
            barrier()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for s in range(n_var):
                evict_v(3 + s)
            b.record(stream)
            barrier()
            bits = api.tgvkv_status(wsv, stream)
            if bits != 0:
                raise RuntimeError(f"device status bits 0x{bits:x} set in the {vname} run")
            bud = outv.budgets.cpu().numpy()
            next_rows[vname] = {
                "us_per_layer": a.elapsed_time(b) * 1e3 / (n_var * wl.L), "steps": n_var,
                "launches_per_step": api.tgvkv_evict_launches(dv),
                "rows_kept": int(outv.offsets[-1].item()),
                "layers_text_only": int((bud <= wl.N_t).sum()) if opts.get("basis") == "all" else 0,
                "options": opts}
            del outv, wsv

    # ---- decode over the compacted cache vs over the full cache: the consumer
    # of the step (one new token per layer), copies rotated past L2
    decode = None
    if not args.no_next_rows:
        evict(0)
        barrier()
        n_rows = int(out.offsets[-1].item())
        comp_bytes = 2 * n_rows * wl.d * 2
        n_cp = max(2, math.ceil(2 * L2_BYTES / max(comp_bytes, 1)) + 1)
        comp = [(out.k_out[:n_rows].clone(), out.v_out[:n_rows].clone()) for _ in range(n_cp)]
        offs = out.offsets.clone()
        full_off = torch.arange(wl.L * wl.H_kv + 1, dtype=torch.int64, device=dev) * wl.N
        qdec = torch.from_numpy(synth.to_bf16_bits(
            np.random.default_rng(args.seed + 11).standard_normal((wl.L, wl.H_q, wl.d))
            .astype(np.float32))).to(dev).view(torch.bfloat16)
        odec = torch.empty((wl.L, wl.H_q, wl.d), dtype=torch.float32, device=dev)
        n_dec = max(3, min(args.steps, 200))

        def time_decode(pick):
            for s in range(3):
                kk, vv, oo = pick(s)
                api.tgvkv_decode(desc, qdec, kk, vv, oo, odec, ws, stream)
            barrier()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for s in range(n_dec):
                kk, vv, oo = pick(3 + s)
                api.tgvkv_decode(desc, qdec, kk, vv, oo, odec, ws, stream)
            b.record(stream)
            barrier()
            return a.elapsed_time(b) * 1e3 / n_dec

        t_comp = time_decode(lambda s: (comp[s % n_cp][0], comp[s % n_cp][1], offs))
        t_full = time_decode(lambda s: (sets[s % n_sets]["k"], sets[s % n_sets]["v"], full_off))
        bits = api.tgvkv_status(ws, stream)
        if bits != 0:
            raise RuntimeError(f"device status bits 0x{bits:x} set in the decode runs")
        full_bytes = 2 * wl.L * wl.H_kv * wl.N * wl.d * 2
        decode = {"what": "one decode step of every layer (one new token), attention over the "
                          "cached K/V of each KV head's query heads",
                  "compacted_us_per_token": t_comp, "full_us_per_token": t_full,
                  "speedup": t_full / t_comp, "rows_compacted": n_rows,
                  "rows_full": wl.L * wl.H_kv * wl.N,
                  "compacted_gbs": comp_bytes / (t_comp * 1e-6) / 1e9,
                  "full_gbs": full_bytes / (t_full * 1e-6) / 1e9,
                  "launches": api.tgvkv_decode_launches(desc), "steps": n_dec}
        pk = float(measured_peaks()[0]["hbm_gbs"])
        decode["compacted_frac"] = decode["compacted_gbs"] / pk
        decode["full_frac"] = decode["full_gbs"] / pk
        del comp

    # ---- the prefill side: causal attention over every token that also keeps
    # the query rows' (m, Z, vision mass), then the eviction that reads them
    # instead of running its own pass over the row statistics
    prefill = None
    if not args.no_next_rows:
        pinp = synth.generate_prefill(wl, seed=args.seed + rank, inp=inp)
        kv_bytes = 2 * inp["k"].nbytes
        n_q = max(2, math.ceil(2 * L2_BYTES / (pinp["q_all"].nbytes + kv_bytes)) + 1)
        q_alls = [upload(pinp["q_all"], torch.bfloat16) for _ in range(n_q)]
        del pinp
        o_pf = torch.empty_like(q_alls[0])
        qt_pf = torch.empty((wl.L, wl.H_q, wl.n_win, wl.d), dtype=torch.bfloat16, device=dev)
        rs_pf = torch.empty((wl.L, wl.H_q, wl.n_win, 3), dtype=torch.float32, device=dev)
        # the same attention without query rows: no statistics to keep
        desc_plain = api.make_desc(wl.L, wl.H_q, wl.H_kv, wl.d, wl.N, wl.N_v, 0)
        ws_plain = api.new_workspace(desc_plain, dev)
        n_pf = max(3, min(args.steps, 50))

        def time_calls(call, n):
            for s in range(3):
                call(s)
            barrier()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for s in range(n):
                call(3 + s)
            b.record(stream)
            barrier()
            return a.elapsed_time(b) / n      # ms per call

        def prefill_call(dsc, wsp):
            def call(s):
                x = sets[s % n_sets]
                api.tgvkv_prefill(dsc, q_alls[s % n_q], x["k"], x["v"], x["modality"],
                                  x["text_pos"], o_pf, qt_pf, rs_pf, wsp, stream)
            return call

        t_pf = time_calls(prefill_call(desc, ws), n_pf)
        t_pf_plain = time_calls(prefill_call(desc_plain, ws_plain), n_pf)

        def evict_stats(s):
            x = sets[s % n_sets]
            api.tgvkv_evict_with_stats(desc, qt_pf, x["k"], x["v"], x["modality"], x["text_pos"],
                                       x["w"], ratio, rs_pf, out, ws, stream)

        n_ev = max(3, min(args.steps, 200))
        t_ev_stats = time_calls(evict_stats, n_ev)
        bits = api.tgvkv_status(ws, stream) | api.tgvkv_status(ws_plain, stream)
        if bits != 0:
            raise RuntimeError(f"device status bits 0x{bits:x} set in the prefill runs")
        # causal attention FLOPs: QK^T and PV over every visible (row, key) pair
        pairs = wl.N * (wl.N + 1) // 2
        flops = 4.0 * wl.d * wl.H_q * wl.L * pairs
        peaks = measured_peaks()[0]
        peak_tf = float(peaks.get("bf16_tflops", 0.0)) or None
        tf = flops / (t_pf * 1e-3) / 1e12
        prefill = {
            "what": "causal prefill attention of every token (all layers) that also keeps the "
                    "eviction rows' statistics; then tgvkv_evict_with_stats",
            "prefill_ms": t_pf, "prefill_plain_ms": t_pf_plain,
            "stats_overhead_frac": t_pf / t_pf_plain - 1.0,
            "flops_per_launch": flops, "tflops": tf,
            "frac_of_measured_bf16": tf / peak_tf if peak_tf else None,
            "evict_with_stats_us_per_layer": t_ev_stats * 1e3 / wl.L,
            "evict_us_per_layer": us_per_layer,
            "evict_saving_frac": 1.0 - (t_ev_stats * 1e3 / wl.L) / us_per_layer,
            "steps": n_pf}
        # context only: the library attention (PyTorch SDPA) on the same tensors
        try:
            import torch.nn.functional as F
            kq = sets[0]["k"].view(wl.L, wl.H_kv, wl.N, wl.d)
            vq = sets[0]["v"].view(wl.L, wl.H_kv, wl.N, wl.d)

            def sdpa(s):
                F.scaled_dot_product_attention(q_alls[s % n_q], kq, vq, is_causal=True,
                                               enable_gqa=wl.H_q != wl.H_kv)

            t_sdpa = time_calls(sdpa, n_pf)
            prefill["sdpa_ms"] = t_sdpa
            prefill["sdpa_tflops"] = flops / (t_sdpa * 1e-3) / 1e12
        except Exception as exc:   # noqa: BLE001 - context figure only
            prefill["sdpa_ms"] = None
            prefill["sdpa_error"] = str(exc)[:200]
        del q_alls, o_pf

    # ---- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        pin = {k: torch.from_numpy(np.ascontiguousarray(inp[k])).pin_memory()
               for k in ("q", "k", "v", "modality", "text_pos", "w")}
        rows = api.tgvkv_retained_rows(desc, ratio)
        host_out = dict(k_out=torch.empty((rows, wl.d), dtype=torch.bfloat16).pin_memory(),
                        v_out=torch.empty((rows, wl.d), dtype=torch.bfloat16).pin_memory(),
                        idx=torch.empty(rows, dtype=torch.int32).pin_memory(),
                        offsets=torch.empty(wl.L * wl.H_kv + 1, dtype=torch.int64).pin_memory(),
                        budgets=torch.empty(wl.L, dtype=torch.int32).pin_memory())
        x = sets[0]
        dst = dict(q=x["q"].view(torch.int16), k=x["k"].view(torch.int16),
                   v=x["v"].view(torch.int16), modality=x["modality"], text_pos=x["text_pos"],
                   w=x["w"])
        h2d = sum(pin[k].numel() * pin[k].element_size() for k in pin)
        d2h = sum(t.numel() * t.element_size() for t in host_out.values())
        n_e2e = max(3, min(args.steps, 200))

        def e2e_step():
            for key in pin:
                dst[key].copy_(pin[key], non_blocking=True)
            api.tgvkv_evict(desc, x["q"], x["k"], x["v"], x["modality"], x["text_pos"], x["w"],
                            ratio, out, ws, stream)
            host_out["k_out"].copy_(out.k_out[:rows], non_blocking=True)
            host_out["v_out"].copy_(out.v_out[:rows], non_blocking=True)
            host_out["idx"].copy_(out.idx[:rows], non_blocking=True)
            host_out["offsets"].copy_(out.offsets, non_blocking=True)
            host_out["budgets"].copy_(out.budgets, non_blocking=True)

        for _ in range(3):
            e2e_step()
        barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n_e2e):
            e2e_step()
        b.record(stream)
        barrier()
        e2e_ms = torch.tensor([a.elapsed_time(b)], device=dev, dtype=torch.float64)
        if world > 1:
            dist.all_reduce(e2e_ms, op=dist.ReduceOp.MAX)
        e2e = {"value": float(e2e_ms.item()) * 1e3 / (n_e2e * wl.L * world), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n_e2e,
               "path": "pinned host -> tgvkv_evict (C ABI) -> pinned host, one stream"}

    # ---- roofline of the dominant kernel and of the whole step
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks["hbm_gbs"])
    dom = max(stages, key=lambda s: stage_ms[s])
    traffic = recorded_traffic(dom, wl.name)
    roof = kernel_roof(wl, ratio, dom, stage_ms[dom], peaks, peak_src)
    clk_mhz = clocks.get("sm_mhz") or float(peaks.get("sm_max_mhz", 2070.0))
    mufu = mufu_of(wl, stage_ms["score"], clk_mhz)
    sbytes, rows = step_bytes(wl, ratio)
    step_gbs = sbytes * args.steps * world / (region_ms * 1e-3) / 1e9
    fbytes = full_step_bytes(wl, ratio)
    full_gbs = fbytes * args.steps * world / (region_ms * 1e-3) / 1e9

    # ---- every workload and budget (the main workload's inputs reused)
    per_config, per_config_clocks = None, None
    if not args.no_per_config and not args.layers:
        del sets
        torch.cuda.empty_cache()
        per_config, per_config_clocks = run_per_config(
            api, torch, dev, stream, barrier, args.seed + rank, args.per_config_steps,
            inputs={wl.name: inp})

    line = None
    if rank == 0:
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            cpu = run_cpu_baseline(wl, ratio, args.seed, args.cpu_seconds)
        line = {
            "metric": METRIC, "value": us_per_layer, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": region_ms / args.steps, "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16->f32",
            "data": "synthetic",
            "config": full_config(wl, ratio, world),
            "hbm_step": {"bytes_per_step": sbytes, "bytes_per_layer": sbytes / wl.L,
                         "gbs": step_gbs, "peak": hbm_peak, "frac": step_gbs / hbm_peak,
                         "frac_nominal": step_gbs / NOMINAL_HBM_GBS,
                         "definition": "K read once + compacted K/V written, per step",
                         "full_bytes_per_step": fbytes, "full_gbs": full_gbs,
                         "full_frac": full_gbs / hbm_peak,
                         "full_definition": "plus Q read, scores written and read, kept K/V "
                                            "rows read, idx and offsets"},
            "roofline": {"bound": roof["bound"], "kernel": dom, "achieved": roof["achieved"],
                         "peak": roof["peak"], "unit": roof["unit"], "frac": roof["frac"],
                         "traffic": traffic, "source_sha": source_hash(dom),
                         "bytes_per_launch": roof["bytes_per_launch"],
                         "flops_per_launch": roof["flops_per_launch"],
                         "launch_ms": stage_ms[dom],
                         "peak_source": roof["peak_source"], "frac_nominal": roof["frac_nominal"]},
            "score_mufu": mufu,
            # the evict's fused select + gather timed alone after the budget
            # (tgvkv_select_compact, the same kernel), against its own roof
            "tail_kernel": _roof_brief(kernel_roof(wl, ratio, "tail", stage_ms["tail"], peaks,
                                                   peak_src), stage_ms["tail"]),
            "stage_ms": stage_ms,
            "next_rows": next_rows,
            "decode": decode,
            "prefill": prefill,
            "fused_tail_ms": region_ms / args.steps - stage_ms["score"],
            # per-step spread from a separate pass with an event pair around
            # each eviction (no overlap between evictions there)
            "step_ms_median_isolated": statistics.median(step_ms),
            "wall_s_timed_region": t_wall,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches_per_step * args.steps,
            "clocks": clocks,
            # the clocks of a first timed region they disqualified (then re-measured)
            "clocks_rejected_first_run": rejected_clocks,
            "per_config": per_config,
            "per_config_clocks": per_config_clocks,
        }
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    if line is not None:
        print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
