"""Benchmark of the hybrid packed-CKKS linear layer on GB300.

One step = one evaluation of the whole layer (every signed sum, shared signed
sum, scale PMult, raw PMult-MAC and the final reduction) through the C ABI
(fiona_linear_eval), on synthetic residues already resident in HBM.

  value        nonzero ciphertext terms per second (raw + signed terms with
               t != 0) of the whole job, all ranks
  roofline     minimal HBM bytes per launch (each used input, plaintext and
               output limb moved once) / average kernel time, against the
               measured copy bandwidth
  e2e          the same metric through fiona_linear_eval_host: host inputs
               (pinned) -> device -> kernel -> host outputs every step; the
               plaintexts (the model's weights) stay resident on the device
  cpu_baseline the CPU oracle on a bounded sample of the same layer, on every
               host core (one spawn process per core)

--op rescale times the rescale that follows the layer instead (fiona_rescale
on the layer's 2 n_out output polys, N and L of the workload): value is
polys rescaled per second and the roofline is the integer-multiply pipe
(the NTT butterflies), not HBM.

--op encode times the plaintext encoding (fiona_encode: slot vectors ->
integer coefficients -> RNS NTT form) of up to 256 of the layer's plaintexts.

--impl reference times the CPU oracle as the reference arm.
Multi-GPU (torchrun): every rank evaluates its own replica of the layer
(independent queries, weak scaling, no data-path collective).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2609_35352_gb300 import workloads as W  # noqa: E402

METRIC = "hybrid linear layer ciphertext-terms/s and HBM GB/s (% of GB300 peak), N=2^16"
UNIT = "ciphertext-terms/s"
DEFAULT_WORKLOAD = "bert"
WORKLOAD_TEXT = {
    "wsum-pmult": "64-ciphertext weighted sum -> 1 output, all PMult",
    "wsum-ternary": "64-ciphertext weighted sum -> 1 output, all ternary (one scale PMult)",
    "wsum-hybrid": "64-ciphertext weighted sum -> 1 output, 50/50 hybrid (32 raw, 32 signed)",
    "vgg": "VGG11-style conv layer, 144 rotated inputs -> 16 outputs, 79% ternary",
    "vit": "ViT-B-style BSGS projection, 32 -> 24, 65% ternary, 25% shared sums",
    "bert": "BERT-base-style FFN column packing, 96 -> 96, 53% ternary, 30% shared sums",
    "bert-const": "the bert layer with every raw weight broadcast to all slots (constant raw plaintexts)",
}
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e, the ~8 TB/s the target is stated against


# ----------------------------------------------------------------------------
# CPU oracle on a sample (spawned workers; never forked after CUDA init)
# ----------------------------------------------------------------------------
_WORKER_BYTES = 32 << 20  # bound on the sampled residues one worker holds


def _oracle_time(state) -> float:
    import oracle
    p, q, X, P = state
    t0 = time.perf_counter()
    oracle.linear_eval(p, q, X, P)
    return time.perf_counter() - t0


def _oracle_state(name: str, limb: int, coefs: list):
    """The residues of one limb and some coefficients of a workload: every
    input (both polys) and every plaintext."""
    wl = W.make_workload(name)
    p = wl.plan
    k = np.asarray(coefs, dtype=np.uint64)
    X = wl.input_values(np.arange(p.n_in).reshape(-1, 1, 1), np.arange(2).reshape(1, -1, 1),
                        limb, k.reshape(1, 1, -1)).reshape(p.n_in, 2, 1, -1)
    P = wl.plaintext_values(np.arange(p.n_pt).reshape(-1, 1), limb, k.reshape(1, -1))
    return p, [wl.moduli[limb]], X, P.reshape(p.n_pt, 1, -1)


def _oracle_worker(conn, name, limb, coefs):
    """One spawned process with a fixed task: it generates its positions'
    residues once (untimed), then times the oracle on them each time it is
    asked, until it receives None."""
    import oracle
    oracle.build()
    state = _oracle_state(name, limb, coefs)
    conn.send(("ready", len(coefs)))
    while conn.recv() is not None:
        conn.send((_oracle_time(state), len(coefs)))
    conn.close()


class OracleSampler:
    """Runs the oracle over sampled (limb, coefficient) positions of a layer
    on `cores` spawned processes, each with its own fixed positions (the same
    every step; their residues generated once, untimed).  The sample is sized
    to about `budget_s` seconds of oracle time per process and step, and to at
    most _WORKER_BYTES of residues per process."""

    def __init__(self, name: str, cores: int, budget_s: float):
        import oracle
        oracle.build()
        self.name = name
        self.wl = W.make_workload(name)
        self.cores = cores
        # calibrate here (not timed in the line): a few positions, one process
        state = _oracle_state(name, 0, list(range(8)))
        _oracle_time(state)
        per_pos = max(_oracle_time(state) / 8, 1e-7)
        p = self.wl.plan
        values_per_pos = 2 * p.n_in + p.n_pt
        per_core = min(int(budget_s / per_pos), _WORKER_BYTES // (8 * values_per_pos), self.wl.N)
        self.per_core = max(1, per_core)
        self.positions = self.per_core * cores
        ctx = mp.get_context("spawn")
        self.procs, self.conns = [], []
        wl = self.wl
        for c in range(cores):
            limb = c % wl.L
            start = ((c // wl.L) * self.per_core) % max(1, wl.N - self.per_core + 1)
            a, b = ctx.Pipe()
            pr = ctx.Process(target=_oracle_worker,
                             args=(b, name, limb, list(range(start, start + self.per_core))), daemon=True)
            pr.start()
            self.procs.append(pr)
            self.conns.append(a)
        for a in self.conns:
            a.recv()  # ready

    def step(self):
        for a in self.conns:
            a.send(1)
        res = [a.recv() for a in self.conns]
        wall = max(r[0] for r in res)
        pos = sum(r[1] for r in res)
        return wall, pos

    def throughput(self, wall: float, pos: int) -> float:
        frac = pos / (self.wl.L * self.wl.N)
        return frac * self.wl.plan.counts()["nonzero"] / wall

    def sample_text(self, pos: int) -> str:
        return ("oracle on %d sampled (limb, coefficient) positions of %d per step "
                "(all outputs, both polys), %d spawned processes, the slowest one's time; "
                "terms/s scaled by the sampled fraction" % (pos, self.wl.L * self.wl.N, self.cores))

    def close(self):
        for a in self.conns:
            try:
                a.send(None)
            except OSError:
                pass
        for pr in self.procs:
            pr.join(timeout=5)
            if pr.is_alive():
                pr.terminate()


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------
# NVML clock-event reason bits (nvml.h)
_NVML_REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
                 0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}


class _Nvml:
    """Read-only NVML queries through ctypes (the driver's libnvidia-ml):
    SM clock, its maximum, power draw and the active clock-event reasons of
    one device.  Raises OSError when NVML cannot be used."""

    def __init__(self, device: int):
        import ctypes
        self.ct = ctypes
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        self.lib = lib
        self.h = ctypes.c_void_p()
        ok = False
        try:  # the CUDA device's own identity (CUDA and NVML orders may differ)
            import torch
            props = torch.cuda.get_device_properties(device)
            uuid = getattr(props, "uuid", None)
            if uuid is not None:
                u = str(uuid)
                u = u if u.startswith("GPU-") else "GPU-" + u
                ok = lib.nvmlDeviceGetHandleByUUID(u.encode(), ctypes.byref(self.h)) == 0
            if not ok and hasattr(props, "pci_bus_id"):
                bus = "%08x:%02x:%02x.0" % (props.pci_domain_id, props.pci_bus_id, props.pci_device_id)
                ok = lib.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(self.h)) == 0
        except Exception:  # noqa: BLE001 - fall back to the index
            ok = False
        if not ok and lib.nvmlDeviceGetHandleByIndex_v2(device, ctypes.byref(self.h)) != 0:
            raise OSError("no NVML handle for device %d" % device)
        self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons

    def sample(self):
        ct = self.ct
        sm, smax, mw = ct.c_uint(), ct.c_uint(), ct.c_uint()
        bits = ct.c_ulonglong()
        if self.lib.nvmlDeviceGetClockInfo(self.h, 1, ct.byref(sm)) != 0:  # NVML_CLOCK_SM
            return None
        self.lib.nvmlDeviceGetMaxClockInfo(self.h, 1, ct.byref(smax))
        if self.lib.nvmlDeviceGetPowerUsage(self.h, ct.byref(mw)) != 0:
            mw.value = 0
        if self.reasons_fn(self.h, ct.byref(bits)) != 0:
            bits.value = 0
        return float(sm.value), float(smax.value), mw.value / 1000.0, int(bits.value)


class ClockSampler:
    """SM clock, power and throttle reasons of one GPU while the timed region
    runs.  NVML is polled every millisecond from a thread started before the
    region (an NVML query can take a millisecond: none runs on the launching
    thread before the last launch is queued, so the GPU never waits for one);
    mark_begin() after the first launch is queued opens the window, a
    synchronous sample at mark_end() (the GPU still busy with queued work)
    closes it, and stop(t_done) keeps the samples taken from the first launch
    to the final synchronize.  Without NVML, nvidia-smi samples every 20 ms
    instead."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device: int):
        self.device = device
        self.samples = []  # (sm_mhz, max_mhz, watts, reason names)
        self.nvml = None
        self.thread = None
        self.stop_flag = False
        self.proc = None
        self.file = None
        self.skip = 0
        self.t_begin = None
        self.source = "nvml"
        try:
            self.nvml = _Nvml(device)
        except (OSError, AttributeError):
            self.nvml = None
            self.source = "nvidia-smi"

    def _take(self):
        t0 = time.monotonic()
        s = self.nvml.sample()
        if s is not None:
            names = [n for b, n in _NVML_REASONS.items() if s[3] & b]
            self.samples.append((s[0], s[1], s[2], names, t0))

    def _loop(self):
        while not self.stop_flag:
            self._take()
            time.sleep(0.001)

    def start(self):
        """Call before the timed region."""
        if self.nvml is not None:
            import threading
            self.thread = threading.Thread(target=self._loop, daemon=True)
            self.thread.start()
            return
        try:
            self.file = tempfile.TemporaryFile(mode="w+")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.device), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None

    def mark_begin(self):
        """Call right after the timed region's first launch is queued."""
        self.t_begin = time.monotonic()

    def mark_end(self):
        """Call after the last launch is queued, before the final synchronize."""
        if self.nvml is not None:
            self._take()

    def stop(self, t_done=None) -> dict:
        """`t_done`: time.monotonic() right after the region's final synchronize."""
        if self.nvml is not None:
            self.stop_flag = True
            if self.thread is not None:
                self.thread.join(timeout=2)
            lo = self.t_begin if self.t_begin is not None else float("-inf")
            hi = t_done if t_done is not None else float("inf")
            self.samples = [x for x in self.samples if lo <= x[4] <= hi]
        elif self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.file.seek(0)
            names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
            for line in self.file.read().splitlines():
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    vals = float(parts[1]), float(parts[2]), float(parts[3])
                except ValueError:
                    continue
                self.samples.append(vals + ([n for n, v in zip(names, parts[5:9]) if v.lower() == "active"],))
        else:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no clock source (NVML, nvidia-smi)"],
                    "samples": 0, "source": None}
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "source": self.source}
        sm = [x[0] for x in self.samples]
        reasons = sorted(set(r for x in self.samples for r in x[3]))
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(x[1] for x in self.samples),
                "sm_mhz_min": min(sm), "reasons": reasons, "samples": len(sm),
                "power_w_max": max(x[2] for x in self.samples), "source": self.source}


# ----------------------------------------------------------------------------
def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


KERNEL_FILES = {"direct": ["kernel_direct.cu", "rns.cuh"],
                "tiled": ["kernel_tiled.cu", "kernel_tiled_off.cu", "kernel_tiled_w12.cu", "tiled_kernel.cuh", "tiled.h", "lower_tiled.cpp",
                          "rns.cuh", "tile_math.cuh", "async.cuh", "tc_signed.cuh", "tc_geometry.h", "../build.py"]}


def kernel_source_hash(kernel: str) -> str:
    """Hash of the device code of one kernel variant."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_35352_gb300", "csrc")
    for f in KERNEL_FILES[kernel]:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(f.encode() + b"\0" + fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current sources of this kernel; None otherwise."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except (OSError, ValueError):
        return None
    ent = d.get("%s/%s" % (kernel, workload))
    if not ent or ent.get("kernel_src_sha") != kernel_source_hash(kernel):
        return None
    return ent.get("dram_bytes_per_launch")


def workload_config(wl: W.Workload, name: str) -> dict:
    """The workload, from the plan description alone: both arms print the
    same dict for the same layer."""
    c = wl.plan.counts()
    bytes_min = W.min_bytes(wl.plan, wl.L, wl.N)
    return {
        "workload": "%s (%s): N=2^%d, L=%d RNS limbs of %d-bit primes, %d inputs -> %d outputs"
                    % (name, WORKLOAD_TEXT.get(name, name), wl.N.bit_length() - 1, wl.L,
                       max(wl.moduli).bit_length(), wl.plan.n_in, wl.plan.n_out),
        "N": wl.N, "L": wl.L, "n_in": wl.plan.n_in, "n_out": wl.plan.n_out,
        "nonzero_terms": c["nonzero"], "raw_terms": c["raw"], "signed_terms": c["plus"] + c["minus"],
        "shared_sums": wl.plan.n_nodes, "bytes_min_per_step": bytes_min,
        "l2": "inputs larger than L2 (%.2f GB read per step, L2 129 MB)" % (bytes_min / 1e9),
    }


def max_over_ranks(x: float, device: str = "cuda") -> float:
    """The largest x over the ranks of the default process group (x itself
    without one): a step takes as long as its slowest rank."""
    import torch
    dist = torch.distributed
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier() -> None:
    """Barrier of the default process group, if there is one."""
    import torch
    dist = torch.distributed
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()


def whole_job_rate(units_per_rank_step: float, steps: int, world: int, elapsed_s: float) -> float:
    """Units all ranks processed per second: every rank processes the same
    units each step (weak scaling), and elapsed_s is the slowest rank's."""
    return world * units_per_rank_step * steps / elapsed_s


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def run_reference(args, rank: int, world: int) -> None:
    if rank != 0:
        return
    cores = host_cores()
    wl = W.make_workload(args.workload)
    # sized so that warmup + steps stay within about two minutes (the
    # worker-side time of each step is what is measured; at least one
    # position per core)
    budget = max(0.02, min(5.0, 120.0 / max(1, args.steps + args.warmup)))
    smp = OracleSampler(args.workload, cores, budget)
    for _ in range(args.warmup):
        smp.step()
    walls, poss = [], []
    for _ in range(args.steps):
        w, p = smp.step()
        walls.append(w)
        poss.append(p)
    smp.close()
    wall = sum(walls)
    frac = sum(poss) / (wl.L * wl.N)
    value = frac * wl.plan.counts()["nonzero"] / wall
    cfg = workload_config(wl, args.workload)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * wall / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u64", "data": "synthetic", "config": cfg,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": smp.sample_text(poss[0] if poss else 0)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args, rank: int, world: int, local_rank: int) -> None:
    import torch

    from paper_2609_35352_gb300 import build as B
    from paper_2609_35352_gb300 import fiona as F

    if rank == 0:
        B.build()
    barrier()
    torch.cuda.set_device(local_rank)
    dev = local_rank
    name = args.workload
    wl = W.make_workload(name, L=args.limbs)
    p = wl.plan

    # CPU baseline first (rank 0, N = 1): spawned workers, before heavy GPU use
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu and args.limbs is None:
        cores = host_cores()
        smp = OracleSampler(name, cores, args.cpu_budget)
        walls, poss = [], []
        while not walls or sum(walls) < args.cpu_budget:  # about cpu_budget s on every core
            w, pos = smp.step()
            walls.append(w)
            poss.append(pos)
        cpu = {"value": smp.throughput(sum(walls), sum(poss)), "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": smp.sample_text(poss[0]) + ", %d steps" % len(walls)}
        smp.close()

    ctx = F.Context(wl.N, wl.moduli, device=dev)
    plan = F.Plan(ctx, p)
    stats = plan.stats()
    n_in = 2 * p.n_in * wl.L * wl.N
    n_pt = p.n_pt * wl.L * wl.N
    n_out = 2 * p.n_out * wl.L * wl.N
    d_in = torch.empty(max(n_in, 2), dtype=torch.int64, device="cuda")
    d_pt = torch.empty(max(n_pt, 2), dtype=torch.int64, device="cuda")
    d_out = torch.empty(max(n_out, 2), dtype=torch.int64, device="cuda")
    stream = torch.cuda.Stream()
    F.device_fill(d_in, 2 * p.n_in, wl.L, wl.N, wl.moduli, wl.key(W.STREAM_INPUTS), 0, stream)
    F.device_fill(d_pt, p.n_pt, wl.L, wl.N, wl.moduli, wl.key(W.STREAM_PLAINTEXTS), 0, stream)
    if wl.const_pts:  # constant raw plaintexts (one residue per limb) come first
        F.device_fill(d_pt, wl.const_pts, wl.L, wl.N, wl.moduli, wl.key(W.STREAM_PLAINTEXTS), 2, stream)
    stream.synchronize()

    for _ in range(args.warmup):
        plan.eval(d_in, d_pt, d_out, stream=stream)
    stream.synchronize()

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    stops = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(dev)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    t_begin = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_begin.record(stream)
    for s in range(args.steps):
        starts[s].record(stream)
        plan.eval(d_in, d_pt, d_out, stream=stream)
        stops[s].record(stream)
        if s == 0:
            clocks.mark_begin()
    t_end.record(stream)
    clocks.mark_end()
    torch.cuda.synchronize()
    t_done = time.monotonic()
    barrier()
    clk = clocks.stop(t_done)
    elapsed_ms = t_begin.elapsed_time(t_end)
    kernel_ms = [a.elapsed_time(b) for a, b in zip(starts, stops)]
    elapsed_ms = max_over_ranks(elapsed_ms)
    ms_per_step = elapsed_ms / args.steps
    terms = stats["n_nonzero_terms"]
    value = whole_job_rate(terms, args.steps, world, elapsed_ms / 1e3)

    avg_kernel_s = statistics.mean(kernel_ms) / 1e3
    peak, peak_kind = measured_peak()
    achieved = stats["bytes_min"] / avg_kernel_s / 1e9
    kernel = "tiled" if stats["kernel"] == 2 else "direct"
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak,
                "peak_nominal": NOMINAL_HBM_GBS, "frac_nominal": achieved / NOMINAL_HBM_GBS,
                "traffic": profiled_traffic(name, kernel) if args.limbs is None else None,
                "kernel": kernel,
                "peak_kind": peak_kind,
                "algorithmic_bytes_per_launch": stats["bytes_min"],
                "kernel_ms_median": statistics.median(kernel_ms)}
    # the secondary roof: 50-bit x 50-bit products against the measured rate
    # of the same product-accumulate (fiona_mul_roof), outside the timed region
    narrow = max(wl.moduli) < (1 << 52)
    mul_achieved = stats["wide_products"] / avg_kernel_s
    try:
        mul_peak = F.mul_roof()["narrow" if narrow else "wide"]
    except RuntimeError as e:  # the line keeps its HBM figures without it
        mul_peak, why = None, str(e)
    alu = {"bound": "alu", "unit": "products/s", "achieved": mul_achieved, "peak": mul_peak,
           "frac": mul_achieved / mul_peak if mul_peak else None,
           "peak_kind": ("measured (fiona_mul_roof: the %s product-accumulate on every SM)"
                         % ("radix-2^26 Karatsuba" if narrow else "64x64->128")) if mul_peak else
                        "unavailable: " + why,
           "products_per_launch": stats["wide_products"]}

    # end to end: host inputs -> result on the host, plaintexts resident
    e2e = None
    if not args.no_e2e:
        h_in = torch.empty(max(n_in, 2), dtype=torch.int64, pin_memory=True)
        h_out = torch.empty(max(n_out, 2), dtype=torch.int64, pin_memory=True)
        h_in.copy_(d_in.cpu())
        e2e_steps = max(3, min(args.steps, args.e2e_steps))
        for _ in range(2):
            plan.eval_host(h_in, d_pt, h_out, d_in, d_out, stream=stream)
        barrier()
        # a stream of queries (fiona_linear_eval_host_async): every step
        # copies its inputs in and its result out; consecutive steps overlap
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            plan.eval_host_async(h_in, d_pt, h_out, d_in, d_out, stream=stream)
        plan.eval_host_join(stream=stream)
        stream.synchronize()
        dt = time.perf_counter() - t0
        dt = max_over_ranks(dt)
        # one synchronous call a step (fiona_linear_eval_host), beside it
        t1 = time.perf_counter()
        for _ in range(3):
            plan.eval_host(h_in, d_pt, h_out, d_in, d_out, stream=stream)
        dt_sync = max_over_ranks(time.perf_counter() - t1) / 3
        e2e = {"value": whole_job_rate(terms, e2e_steps, world, dt), "unit": UNIT,
               "h2d_bytes_per_step": n_in * 8, "d2h_bytes_per_step": n_out * 8,
               "ms_per_step": 1e3 * dt / e2e_steps, "steps": e2e_steps,
               "call": "fiona_linear_eval_host_async, queued back to back, then fiona_linear_eval_host_join",
               "sync_ms_per_step": 1e3 * dt_sync}

    if rank == 0:
        cfg = workload_config(wl, name)
        if cfg["bytes_min_per_step"] != stats["bytes_min"]:
            raise RuntimeError("minimal bytes: the library counts %d, the plan description %d"
                               % (stats["bytes_min"], cfg["bytes_min_per_step"]))
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64",
            "data": "synthetic (seeded SplitMix64 residues, filled on the device)",
            "config": cfg,
            "hbm_gbs": achieved, "hbm_frac": achieved / peak,
            "roofline": roofline, "alu": alu, "cpu_baseline": cpu, "e2e": e2e,
            "clocks": clk, "gpu_launches": args.steps,
            "parallelism": "replicas x%d (independent layer per GPU)" % world,
            "kernel": {"name": kernel, "tile_coeffs": stats["tile_coeffs"],
                       "warps_per_cta": stats["warps_per_cta"], "ctas_per_sm": stats["ctas_per_sm"],
                       "shared_sums_formed": stats["nodes_materialized"],
                       "addsub_executed": stats.get("addsub_executed"),
                       "tensor_core_sums": stats.get("tensor_core_sums"),
                       "source_offsets": stats.get("source_offsets"),
                       "const_raw_all": stats.get("const_raw_all")},
        }
        print(json.dumps(line), flush=True)
    plan.close()
    ctx.close()


# ----------------------------------------------------------------------------
# --op rescale
# ----------------------------------------------------------------------------
# Integer multiplies (IMAD on the FMA-heavy pipe, 64 per clock per SM) that
# one forward butterfly needs at least: the quotient estimate (a wide
# product and two high halves) and the two 64-bit low products (a wide
# product and two plain multiplies each); a wide product takes two issue
# slots.  The derived peak: 152 SMs x 64 multiplies per clock x 2070 MHz /
# 12 slots = 1678 G butterflies/s.
IMAD_SLOTS_PER_BUTTERFLY = 12
IMAD_PER_CLK_PER_SM = 64
SM_COUNT = 152
SM_MAX_MHZ = 2070.0


def rescale_butterflies(N: int, L: int) -> int:
    """Radix-2 butterflies of one poly's rescale: one inverse transform of
    the last limb and L - 1 forward transforms."""
    return L * (N // 2) * (N.bit_length() - 1)


def run_rescale(args, rank: int, world: int, local_rank: int) -> None:
    import torch

    from paper_2609_35352_gb300 import build as B
    from paper_2609_35352_gb300 import fiona as F

    if rank == 0:
        B.build()
    barrier()
    torch.cuda.set_device(local_rank)
    dev = local_rank
    name = args.workload
    wl = W.make_workload(name, L=args.limbs)
    N, L = wl.N, wl.L
    count = 2 * wl.plan.n_out
    unit = "polys/s"

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        import oracle
        oracle.build()
        flat = np.arange(L * N, dtype=np.uint64).reshape(1, L, N)
        y0 = W.residues_np(wl.key(W.STREAM_INPUTS), flat, wl.moduli_np.reshape(1, L, 1))
        dt, done = 0.0, 0
        while done < count and (done == 0 or dt < args.cpu_budget):
            t0 = time.perf_counter()
            oracle.rescale(wl.moduli, y0)
            dt += time.perf_counter() - t0
            done += 1
        cpu = {"value": done / dt, "unit": unit, "cores": 1, "kind": "oracle",
               "sample": "%d rescales of the first of the %d polys (radix-2 NTT oracle, one thread)"
                         % (done, count)}

    ctx = F.Context(N, wl.moduli, device=dev)
    n_y, n_o = count * L * N, count * (L - 1) * N
    d_y = torch.empty(n_y, dtype=torch.int64, device="cuda")
    d_o = torch.empty(n_o, dtype=torch.int64, device="cuda")
    stream = torch.cuda.Stream()
    F.device_fill(d_y, count, L, N, wl.moduli, wl.key(W.STREAM_INPUTS), 0, stream)
    stream.synchronize()
    for _ in range(args.warmup):
        ctx.rescale(L, count, d_y, d_o, stream=stream)
    stream.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    stops = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clocks = ClockSampler(dev)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    for s in range(args.steps):
        starts[s].record(stream)
        ctx.rescale(L, count, d_y, d_o, stream=stream)
        stops[s].record(stream)
        if s == 0:
            clocks.mark_begin()
    clocks.mark_end()
    torch.cuda.synchronize()
    t_done = time.monotonic()
    barrier()
    clk = clocks.stop(t_done)
    step_ms = [a.elapsed_time(b) for a, b in zip(starts, stops)]
    elapsed_ms = sum(step_ms)
    elapsed_ms = max_over_ranks(elapsed_ms)
    value = whole_job_rate(count, args.steps, world, elapsed_ms / 1e3)
    avg_s = statistics.mean(step_ms) / 1e3
    bfly = count * rescale_butterflies(N, L)
    derived_bfly = SM_COUNT * IMAD_PER_CLK_PER_SM * SM_MAX_MHZ * 1e6 / IMAD_SLOTS_PER_BUTTERFLY
    # the measured roof: the rescale's own forward butterfly (fiona_bfly_roof),
    # outside the timed region; the fast form when every modulus is below 2^56
    try:
        roof = F.bfly_roof()
        peak_bfly = roof["fast" if max(wl.moduli) < (1 << 56) else "general"]
        peak_kind = ("measured (fiona_bfly_roof: the rescale's %s forward butterfly on every SM)"
                     % ("fast" if max(wl.moduli) < (1 << 56) else "general"))
    except RuntimeError as e:
        peak_bfly, peak_kind = derived_bfly, "derived (the measurement failed: %s)" % e
    achieved = bfly / avg_s
    hbm_bytes = count * (2 * L - 1) * N * 8
    hbm_peak, hbm_kind = measured_peak()
    roofline = {"bound": "alu", "achieved": achieved / 1e9, "peak": peak_bfly / 1e9, "unit": "Gbutterfly/s",
                "frac": achieved / peak_bfly, "traffic": None,
                "kernel": "rescale (k_inv_low, k_inv_high, k_fwd_high, k_fwd_low)",
                "peak_kind": peak_kind,
                "derived_peak": derived_bfly / 1e9,
                "derived_peak_kind": "%d SMs x %d IMAD/clk x %.0f MHz / %d IMAD slots per butterfly"
                                     % (SM_COUNT, IMAD_PER_CLK_PER_SM, SM_MAX_MHZ, IMAD_SLOTS_PER_BUTTERFLY),
                "butterflies_per_launch": bfly,
                "hbm_gbs_algorithmic": hbm_bytes / avg_s / 1e9,
                "hbm_frac": hbm_bytes / avg_s / 1e9 / hbm_peak, "hbm_peak_kind": hbm_kind,
                "step_ms_median": statistics.median(step_ms)}

    e2e = None
    if not args.no_e2e:
        h_y = torch.empty(n_y, dtype=torch.int64, pin_memory=True)
        h_o = torch.empty(n_o, dtype=torch.int64, pin_memory=True)
        h_y.copy_(d_y.cpu())
        e2e_steps = max(3, min(args.steps, args.e2e_steps))

        def one():
            with torch.cuda.stream(stream):
                d_y.copy_(h_y, non_blocking=True)
                ctx.rescale(L, count, d_y, d_o, stream=stream)
                h_o.copy_(d_o, non_blocking=True)
            stream.synchronize()

        one()
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            one()
        dt = max_over_ranks(time.perf_counter() - t0)
        e2e = {"value": whole_job_rate(count, e2e_steps, world, dt), "unit": unit, "h2d_bytes_per_step": n_y * 8,
               "d2h_bytes_per_step": n_o * 8, "ms_per_step": 1e3 * dt / e2e_steps, "steps": e2e_steps}

    if rank == 0:
        line = {
            "metric": "rescale of the layer's outputs: polys/s, NTT butterflies/s (%% of the integer-multiply "
                      "pipe), N=2^%d" % (N.bit_length() - 1),
            "value": value, "unit": unit, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "u64",
            "data": "synthetic (seeded SplitMix64 residues, filled on the device)",
            "config": {"workload": "rescale of the %s layer's outputs: %d polys, N=2^%d, L=%d -> %d limbs of "
                                   "%d-bit primes" % (name, count, N.bit_length() - 1, L, L - 1,
                                                      max(wl.moduli).bit_length()),
                       "polys": count, "N": N, "L": L,
                       "l2": "inputs larger than L2 (%.2f GB per step, L2 129 MB)" % (hbm_bytes / 1e9)},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": 4 * args.steps,
        }
        print(json.dumps(line), flush=True)
    ctx.close()


# ----------------------------------------------------------------------------
# --op encode
# ----------------------------------------------------------------------------
FP64_NOMINAL_TFLOPS = 1.25   # GB300 dense fp64 (nominal)
FLOPS_PER_COMPLEX_BUTTERFLY = 10  # one complex product (6) and a complex sum and difference (4)


def run_encode(args, rank: int, world: int, local_rank: int) -> None:
    import torch

    from paper_2609_35352_gb300 import build as B
    from paper_2609_35352_gb300 import fiona as F

    if rank == 0:
        B.build()
    barrier()
    torch.cuda.set_device(local_rank)
    dev = local_rank
    name = args.workload
    wl = W.make_workload(name, L=args.limbs)
    N, L = wl.N, wl.L
    count = min(wl.plan.n_pt, 256)
    unit = "plaintexts/s"
    scale = 2.0 ** 40
    rng = np.random.default_rng(wl.seed)
    h_slots = rng.uniform(-1.0, 1.0, size=(count, N // 2, 2))
    h_slots[:, :, 1] = 0.0  # weights are real

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        import oracle
        oracle.build()
        # the definition sum costs N/2 terms per coefficient: time it on a
        # sample of coefficients and scale to N; the NTT form on a whole poly
        z = h_slots[0, :, 0] + 0j
        n_idx = 256
        idx = np.arange(0, N, N // n_idx, dtype=np.uint32)
        t0 = time.perf_counter()
        oracle.ckks_embed(z, scale, idx)
        t_emb = (time.perf_counter() - t0) * N / n_idx
        c = np.zeros(N, np.int64)
        t0 = time.perf_counter()
        oracle.encode_coeffs(wl.moduli, c)
        t_ntt = time.perf_counter() - t0
        cpu = {"value": 1.0 / (t_emb + t_ntt), "unit": unit, "cores": 1, "kind": "oracle",
               "sample": "one plaintext, one thread: the embedding sum timed on %d of its %d coefficients and "
                         "scaled by %d (%.1f s), the RNS NTT form of %d limbs timed whole (%.2f s)"
                         % (n_idx, N, N // n_idx, t_emb, L, t_ntt)}

    ctx = F.Context(N, wl.moduli, device=dev)
    d_slots = torch.from_numpy(h_slots).to("cuda")
    d_c = torch.empty(count * N, dtype=torch.int64, device="cuda")
    d_w = torch.empty(count * N, dtype=torch.float64, device="cuda")
    d_o = torch.empty(count * L * N, dtype=torch.int64, device="cuda")
    stream = torch.cuda.Stream()
    for _ in range(args.warmup):
        ctx.encode(L, count, d_slots, scale, d_c, d_w, d_o, stream=stream)
    stream.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(dev)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    for i, (a, b, c) in enumerate(ev):
        a.record(stream)
        ctx.ckks_embed(count, d_slots, scale, d_c, d_w, stream=stream)
        b.record(stream)
        ctx.encode_coeffs(L, count, d_c, d_o, stream=stream)
        c.record(stream)
        if i == 0:
            clocks.mark_begin()
    clocks.mark_end()
    torch.cuda.synchronize()
    t_done = time.monotonic()
    barrier()
    clk = clocks.stop(t_done)
    if ctx.device_check(stream) != F.FIONA_OK:
        raise RuntimeError("encoding reported a coefficient out of range")
    step_ms = [a.elapsed_time(c) for a, b, c in ev]
    emb_ms = [a.elapsed_time(b) for a, b, c in ev]
    ntt_ms = [b.elapsed_time(c) for a, b, c in ev]
    elapsed_ms = max_over_ranks(sum(step_ms))
    value = whole_job_rate(count, args.steps, world, elapsed_ms / 1e3)
    logn = N.bit_length() - 1
    # the embedding is a complex transform of size N/2
    emb_flops = count * (N // 4) * (logn - 1) * FLOPS_PER_COMPLEX_BUTTERFLY
    achieved = emb_flops / (statistics.mean(emb_ms) / 1e3) / 1e12
    ntt_bfly = count * L * (N // 2) * logn
    peak_bfly = SM_COUNT * IMAD_PER_CLK_PER_SM * SM_MAX_MHZ * 1e6 / IMAD_SLOTS_PER_BUTTERFLY
    roofline = {"bound": "fp64", "achieved": achieved, "peak": FP64_NOMINAL_TFLOPS, "unit": "TFLOP/s",
                "frac": achieved / FP64_NOMINAL_TFLOPS, "traffic": None,
                "kernel": "embedding (k_embed_low, k_embed_high): complex fp64 transform",
                "peak_kind": "nominal GB300 dense fp64", "flops_per_launch": emb_flops,
                "embed_ms_median": statistics.median(emb_ms),
                "rns_ntt": {"bound": "alu", "ms_median": statistics.median(ntt_ms),
                            "achieved_gbfly_s": ntt_bfly / (statistics.mean(ntt_ms) / 1e3) / 1e9,
                            "peak_gbfly_s": peak_bfly / 1e9,
                            "frac": ntt_bfly / (statistics.mean(ntt_ms) / 1e3) / peak_bfly}}

    e2e = None
    if not args.no_e2e:
        h_in = torch.from_numpy(h_slots).pin_memory()
        h_out = torch.empty(count * L * N, dtype=torch.int64, pin_memory=True)
        e2e_steps = max(3, min(args.steps, args.e2e_steps))

        def one():
            with torch.cuda.stream(stream):
                d_slots.copy_(h_in, non_blocking=True)
                ctx.encode(L, count, d_slots, scale, d_c, d_w, d_o, stream=stream)
                h_out.copy_(d_o, non_blocking=True)
            stream.synchronize()

        one()
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            one()
        dt = max_over_ranks(time.perf_counter() - t0)
        e2e = {"value": whole_job_rate(count, e2e_steps, world, dt), "unit": unit, "h2d_bytes_per_step": h_slots.nbytes,
               "d2h_bytes_per_step": count * L * N * 8, "ms_per_step": 1e3 * dt / e2e_steps, "steps": e2e_steps}

    if rank == 0:
        line = {
            "metric": "plaintext encoding: plaintexts/s (slots -> RNS NTT form), N=2^%d" % logn,
            "value": value, "unit": unit, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64+u64", "data": "synthetic (seeded uniform real weights in [-1, 1])",
            "config": {"workload": "encoding of %d of the %s layer's plaintexts: N=2^%d, %d limbs of %d-bit primes, "
                                   "scale 2^40" % (count, name, logn, L, max(wl.moduli).bit_length()),
                       "plaintexts": count, "N": N, "L": L},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": 4 * args.steps,
        }
        print(json.dumps(line), flush=True)
    ctx.close()


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(WORKLOAD_TEXT))
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-budget", type=float, default=2.0,
                    help="seconds of oracle work per host core for cpu_baseline")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--op", choices=["layer", "rescale", "encode"], default="layer")
    ap.add_argument("--limbs", type=int, default=None,
                    help="profiling aid: the same layer with this many RNS limbs (no cpu_baseline)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
    try:
        run = {"layer": run_ours, "rescale": run_rescale, "encode": run_encode}[args.op]
        run(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
