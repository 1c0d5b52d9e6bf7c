#!/usr/bin/env python3
"""Benchmark of the PSS hashed shared-array embedding step on GB300.

One step = the whole hot path over one batch: fused hash + gather + sum-pool
forward, then the backward scatter fused with the optimizer update of the
shared array.  Default workload: the Criteo-TB-shaped 10000x-compressed case
(26 tables, ~195M ids capped at 40M per table, d = 128, M = 2.5M fp32,
Z = 32, batch 65536, Zipf(1.05) ids, Adagrad).

Prints ONE JSON line (rank 0).  ``--impl reference`` times the CPU oracle
instead (the reference arm: a deliberately plain program).

Usage:  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload tb]
        torchrun --nproc-per-node N bench.py --gpus N ...   (independent replicas)
"""
from __future__ import annotations

import argparse
import datetime as _dt
import hashlib
import json
import os
import re
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2207_10731_gb300 import workloads as wl  # noqa: E402

METRIC = "pooled lookups/sec and fused fwd+bwd+update GB/s vs HBM/L2 roofline, 1 GB300"
UNIT = "lookups/s"
WORKLOAD_DESC = {
    "tb": "criteo-tb-shaped 10000x: 26 tables (log-uniform cards in [3,40M], ~195M ids), d=128, "
          "M=2.5M fp32 (10 MB), Z=32, G=4, batch 65536, one Zipf(1.05) id per bag, Adagrad",
    "kaggle": "criteo-kaggle-shaped: 26 tables (log-uniform cards in [3,10M]), d=16, M=1Mi fp32, "
              "Z=32, G=4, batch 2048, one Zipf(1.05) id per bag, Adagrad",
    "multihot": "multi-hot contention: 26 tables as criteo-tb, d=64, M=2.5M fp32, Z=32, G=4, "
                "batch 16384, Poisson(20) bags, Zipf(1.2) ids, SGD",
    "sweep": "criteo-tb shape with shared array M chosen by --M, Z=32, G=4, batch 65536, Adagrad",
    "microbench": "paper micro-benchmark shape: 26 tables, d=128, M=2.5M, Z=32, batch 10240, "
                  "all-ones upstream gradient, SGD",
    "tiny": "tiny: 8 tables x 1000 ids, d=16, M=16384, Z=16, batch 256, SGD",
}


def _host():
    """Host cores and CPU model (for the CPU-oracle baseline)."""
    model = None
    try:
        with open("/proc/cpuinfo") as f:
            info = f.read()
        for key in ("model name", "Hardware", "cpu model"):
            m = re.search(rf"^{key}\s*:\s*(.+)$", info, flags=re.M)
            if m:
                model = m.group(1).strip()
                break
        if model is None:
            try:
                out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
                m = re.search(r"^Model name:\s*(.+)$", out, flags=re.M)
                if m:
                    model = m.group(1).strip()
            except (OSError, subprocess.SubprocessError):
                pass
        if model is None:
            impl = re.search(r"^CPU implementer\s*:\s*(\S+)", info, flags=re.M)
            part = re.search(r"^CPU part\s*:\s*(\S+)", info, flags=re.M)
            if impl and part:
                model = f"arm implementer {impl.group(1)} part {part.group(1)}"
    except OSError:
        pass
    if model is None:
        import platform
        model = platform.processor() or platform.machine()
    return {"nproc": os.cpu_count(), "cpu_model": model}


def _l2_peaks(torch, dev, sm_count):
    """L2 rates measured live with the library's probe kernels over a 32 MB
    device buffer (L2-resident): uniformly random 128-byte block gathers (the
    L2 peak of the roofline: the forward's block reads have this shape),
    streaming 128-byte line reads, and fp64 / 16-byte fp32 reductions into
    random 32-lane blocks (consecutive elements per instruction, as the
    kernels issue them).  Best of 5 timed calls after 2 warm-up calls, CUDA
    events on the launch stream."""
    from paper_2207_10731_gb300 import binding
    nbytes = 32 << 20
    buf = torch.zeros(nbytes // 4, dtype=torch.float32, device=dev)
    ctas = sm_count * 16
    stream = torch.cuda.current_stream()
    out = {"buffer_mb": nbytes >> 20, "ctas": ctas}
    for kind, iters, key in ((0, 1024, "gather_gbs"), (3, 1024, "read_gbs"),
                             (1, 256, "red_f64_adds_per_s"), (2, 256, "red_v4_f32_adds_per_s")):
        best = None
        for rep_ in range(7):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            binding.probe_l2(kind, buf, iters, ctas, stream)
            b.record(stream)
            torch.cuda.synchronize()
            if rep_ >= 2:
                ms = a.elapsed_time(b)
                best = ms if best is None else min(best, ms)
        if kind in (0, 3):
            it = -(-iters // 8) * 8
            out[key] = ctas * 8 * it * 128 / (best / 1e3) / 1e9
        else:
            out[key] = ctas * 256 * iters * (4 if kind == 2 else 1) / (best / 1e3)
    del buf
    return out


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# the C ABI's host code: no device code, so no bearing on a kernel's DRAM traffic
_HOST_ONLY = {"pss_api.cu"}


def _code_only(src: str) -> str:
    """Source text without comments and blank lines (the sources keep no comment
    markers inside string literals)."""
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    lines = (ln.split("//", 1)[0].rstrip() for ln in src.splitlines())
    return "\n".join(ln for ln in lines if ln)


def _kernel_sha():
    """Hash of the code of the library's device-code sources: the kernels,
    their launchers and the headers they share, comments left out (traffic
    figures go stale with it)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2207_10731_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        if f.endswith((".cu", ".cuh", ".h")) and f not in _HOST_ONLY:
            with open(os.path.join(csrc, f), encoding="utf-8") as fh:
                h.update(f.encode() + b"\0" + _code_only(fh.read()).encode())
    return h.hexdigest()[:16]


def _traffic(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if the kernel
    source has not changed since it was captured."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            t = json.load(f)
        e = t.get(f"{kernel}@{workload}")
        if e and e.get("kernel_sha") == _kernel_sha():
            return float(e["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi clock/throttle samples with their own timestamps."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.rows = []
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", gpu_id], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                text=True)
        except Exception:
            self.proc = None
            return
        self.th = threading.Thread(target=self._read, daemon=True)
        self.th.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                ts = _dt.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                self.rows.append((ts, float(parts[1]), float(parts[2]), parts[4:8]))
            except ValueError:
                continue

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0: float, t1: float):
        if not self.rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "nvidia-smi unavailable"}
        inside = [r for r in self.rows if t0 <= r[0] <= t1]
        note = "samples inside the timed region"
        if not inside:
            mid = 0.5 * (t0 + t1)
            inside = sorted(self.rows, key=lambda r: abs(r[0] - mid))[:3]
            note = "timed region shorter than the sampling period: nearest samples"
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i, v in enumerate(r[3]) if v == "Active"})
        return {"sm_mhz": float(np.median([r[1] for r in inside])),
                "sm_max_mhz": float(max(r[2] for r in inside)), "reasons": reasons,
                "samples": len(inside), "note": note}


def _gpu_id(torch, dev):
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
        return vis.split(",")[dev] if vis else str(dev)


def _algorithmic_bytes(w: wl.Workload):
    """Bytes each kernel must move per launch to do the method's work (not
    what an implementation adds on top), and the L2 bytes of the array."""
    nnz, nb, row = w.nnz, w.T * w.B, w.B * w.T * w.d * 4
    stream = 8 * nnz + 8 * (nb + 1)
    per_elem = 16 if w.opt == "adagrad" else 8
    return {
        "forward": stream + row,             # indices + offsets read, pooled rows written
        "scatter": stream + row,             # indices + offsets read, grad_out read (atomic path)
        "reduce": row,                       # grad_out read once (sorted path)
        "update": per_elem * w.M,            # w (and the Adagrad accumulator) read + written
        "step": 2 * stream + 2 * row,        # the whole fused step's HBM streams
        "l2_gather": 4 * nnz * w.d,          # hashed blocks read from the shared array
        "l2_scatter": 4 * nnz * w.d,         # contributions added into the shared array
    }


def _touched_elements(h, dbatches, L, torch):
    """Mean number of distinct elements of M that a batch's blocks cover (the
    touched update reads and writes only these): the union of the intervals
    [loc, loc + L) over the batch's locations, from the library's own hash."""
    tot = 0
    for i, o, _ in dbatches:
        nb = (o.numel() - 1) // h.T
        loc = h.compute_locations(i, o, nb)
        u = torch.unique(loc[loc >= 0])
        if u.numel():
            tot += int(torch.clamp(torch.diff(u), max=L).sum().item()) + L
    torch.cuda.synchronize()
    return tot / max(1, len(dbatches))


def _step_roofline(ab, step_s, hbm_peak, l2, forward_only, array_in_l2):
    """The step's bound: HBM time of its streamed bytes against L2 time of its
    shared-array gathers and adds (when the array is L2-resident), the larger
    of the two; frac = that bound over the measured step time."""
    hbm_bytes = ab["forward"] if forward_only else ab["step"]
    l2_bytes = ab["l2_gather"] + (0 if forward_only else ab["l2_scatter"])
    t_hbm = hbm_bytes / (hbm_peak * 1e9)
    t_l2 = l2_bytes / (l2["gather_gbs"] * 1e9) if (l2 and array_in_l2) else 0.0
    bound = "l2" if t_l2 > t_hbm else "hbm"
    return {"bound": bound, "t_hbm_ms": t_hbm * 1e3, "t_l2_ms": t_l2 * 1e3,
            "hbm_bytes": hbm_bytes, "l2_bytes": l2_bytes if array_in_l2 else None,
            "frac": max(t_hbm, t_l2) / step_s, "target_frac": 0.60,
            "note": "fused forward + backward + update against max(HBM time, L2 time); "
                    "L2 time uses the measured random 128-byte L2 gather rate"}


def _oracle_sample(w: wl.Workload, rows: int):
    """First ``rows`` batch rows of every table as a smaller batch."""
    idx_parts, lens = [], []
    for t in range(w.T):
        for b in range(rows):
            s = t * w.B + b
            idx_parts.append(w.indices[w.offsets[s]:w.offsets[s + 1]])
            lens.append(idx_parts[-1].shape[0])
    off = np.zeros(len(lens) + 1, dtype=np.int64)
    np.cumsum(lens, out=off[1:])
    go = w.grad_out.reshape(w.B, w.T, w.d)[:rows].reshape(-1).copy()
    return np.concatenate(idx_parts).astype(np.int64), off, go


def _oracle_rate(w: wl.Workload, budget_s: float, forward_only: bool = False,
                 max_rows: int = None, signed: bool = False):
    """Time the CPU oracle (as it stands) on bounded samples of the workload."""
    import oracle
    o = oracle.OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, signed=signed)
    wcur = w.w0.copy() if w.w0 is not None else None
    Gcur = np.zeros(w.M, np.float32)
    rows = min(w.B, max_rows or 256)
    # grow the sample until one step takes about budget/5
    while True:
        idx, off, go = _oracle_sample(w, rows)
        t0 = time.perf_counter()
        out, _ = o.forward(wcur, idx, off, rows)
        if not forward_only:
            wcur, Gcur, _ = o.step(wcur, Gcur, idx, off, rows, go, w.opt, w.lr, w.eps)
        dt = time.perf_counter() - t0
        if dt > budget_s / 5 or rows >= w.B or (max_rows and rows >= max_rows):
            break
        rows = min(w.B, rows * 2)
    reps, tot, lookups = 0, 0.0, 0
    while tot < budget_s and reps < 20:
        t0 = time.perf_counter()
        out, _ = o.forward(wcur, idx, off, rows)
        if not forward_only:
            wcur, Gcur, _ = o.step(wcur, Gcur, idx, off, rows, go, w.opt, w.lr, w.eps)
        tot += time.perf_counter() - t0
        reps += 1
        lookups += idx.shape[0]
    return lookups / tot, rows, reps, idx.shape[0], tot


def reduce_over_ranks(dist, device, elapsed_ms: float, work: float):
    """Replicas: the job's time is the slowest rank's timed region, its work
    the sum over ranks (one all-reduce each; the process group may be NCCL on
    GPUs or gloo on the host)."""
    import torch
    t = torch.tensor([elapsed_ms, float(work)], dtype=torch.float64, device=device)
    tmax = t.clone()
    dist.all_reduce(tmax[:1], op=dist.ReduceOp.MAX)
    dist.all_reduce(t[1:], op=dist.ReduceOp.SUM)
    return float(tmax[0]), float(t[1])


def _shape_overrides(args):
    """Chunk size Z, offset alignment G and id distribution given on the command line."""
    over = {k: v for k, v in (("Z", args.Z), ("G", args.G)) if v is not None}
    if args.ids == "uniform":
        over["ids"] = ("uniform",)
    return over


def _workload_desc(args, w):
    """The named workload's description with the batch and M actually run."""
    desc = re.sub(r"batch \d+", f"batch {w.B}", WORKLOAD_DESC[args.workload])
    if args.M is not None:
        desc = re.sub(r"M=[0-9.]+M[i]? fp32( \(\d+ MB\))?|M chosen by --M", f"M={w.M} fp32", desc)
    return desc


def _sort_desc(h, binding, args):
    """How the sorted path grouped the pairs in the timed steps."""
    info = h.info()
    if info["last_path"] != binding.PATH_SORTED:
        return {}
    if args.deterministic:
        return {"sort": "stable radix sort of all pairs"}
    if info["last_collision_rate"] < 0:
        return {"sort": "segment-local: pairs grouped by location within 8192-pair segments"}
    return {"sort": ("counting sort of all pairs" if info["R"] <= (1 << 22) else
                     "radix sort of all pairs"),
            "collision_rate": info["last_collision_rate"]}


def _config_extra(args, w):
    """Config keys that differ from the named workload's defaults."""
    extra = {}
    if args.Z is not None or args.G is not None:
        extra.update({"Z": w.Z, "G": w.G})
    if args.forward_only:
        extra["mode"] = "forward only (inference): hash + gather + sum-pool, no backward"
    if args.signed:
        extra["signed_hash"] = True
    if args.deterministic:
        extra["deterministic"] = ("stable radix sort and window reduce: run-to-run identical bits "
                                  "(PSS_OPT_DETERMINISTIC)")
    if args.ids == "uniform":
        extra["ids"] = "uniform over each table"
    return extra


def run_reference(args):
    """Reference arm: the CPU oracle timed on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w = wl.make_workload(args.workload, M=args.M, B=args.B, **_shape_overrides(args))
    import oracle
    o = oracle.OraclePSS(w.cards, d=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, signed=args.signed)
    total_budget = 90.0
    per_step = total_budget / max(1, args.steps + args.warmup)
    # size the per-step sample so K+W steps fit the budget
    rows = 64
    idx, off, go = _oracle_sample(w, rows)
    t0 = time.perf_counter()
    wcur, Gcur = w.w0.copy(), np.zeros(w.M, np.float32)
    o.forward(wcur, idx, off, rows)
    if not args.forward_only:
        o.step(wcur, Gcur, idx, off, rows, go, w.opt, w.lr, w.eps)
    dt = time.perf_counter() - t0
    rows = int(max(1, min(w.B, rows * per_step / max(dt, 1e-6) * 0.8)))
    idx, off, go = _oracle_sample(w, rows)
    for _ in range(args.warmup):
        o.forward(wcur, idx, off, rows)
        if not args.forward_only:
            wcur, Gcur, _ = o.step(wcur, Gcur, idx, off, rows, go, w.opt, w.lr, w.eps)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        o.forward(wcur, idx, off, rows)
        if not args.forward_only:
            wcur, Gcur, _ = o.step(wcur, Gcur, idx, off, rows, go, w.opt, w.lr, w.eps)
    el = time.perf_counter() - t0
    value = idx.shape[0] * args.steps / el
    sample = (f"first {rows} of {w.B} batch rows x {w.T} tables ({idx.shape[0]} lookups) per step; "
              + ("forward only" if args.forward_only else "forward + gradient + update")
              + ", single thread")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64+f32",
        "data": "synthetic",
        "config": dict({"workload": _workload_desc(args, w), "global_batch": w.B, "seq_len": 1,
                        "parallelism": "single host thread"}, **_config_extra(args, w)),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "host": _host(), "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_gpu(args):
    import torch
    import torch.distributed as dist

    from paper_2207_10731_gb300 import binding

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE={world}")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    # one replica per rank, each with its own batch (no data-path exchange)
    w = wl.make_workload(args.workload, seed=0, M=args.M, B=args.B, **_shape_overrides(args))
    batches = [(w.indices, w.offsets, w.grad_out)]
    for k in range(1, args.rotate):
        batches.append(wl.make_batch(w.cards, w.B, w.d, wl.CONFIGS[args.workload]["bag"],
                                     _shape_overrides(args).get("ids",
                                                                wl.CONFIGS[args.workload]["ids"]),
                                     seed=rank, batch=k,
                                     grad=wl.CONFIGS[args.workload].get("grad", "normal")))
    dbatches = [(torch.from_numpy(i).to(dev), torch.from_numpy(o).to(dev),
                 torch.from_numpy(g).to(dev)) for i, o, g in batches]
    h = binding.PSS(w.cards, dim=w.d, M=w.M, Z=w.Z, G=w.G, seed=w.seed, optimizer=w.opt,
                    eps=w.eps)
    if w.w0 is not None:
        h.set_weights(torch.from_numpy(w.w0).to(dev))
    else:
        base = torch.from_numpy(w.w0_base).to(dev)
        h.set_weights(base.repeat(-(-w.M // base.numel()))[: w.M].contiguous())
        del base
    h.set_option(binding.OPT_ACCUM, binding.ACCUM_F32 if args.accum == "f32" else binding.ACCUM_F64)
    if args.signed:
        h.set_option(binding.OPT_SIGNED, 1)
    if args.deterministic:
        h.set_option(binding.OPT_DETERMINISTIC, 1)
    h.set_option(binding.OPT_SORT_SCOPE, {"auto": binding.SORT_AUTO, "global": binding.SORT_GLOBAL,
                                          "local": binding.SORT_LOCAL}[args.sort])
    h.set_option(binding.OPT_UPDATE_MODE, {"auto": binding.UPDATE_AUTO, "dense": binding.UPDATE_DENSE,
                                           "touched": binding.UPDATE_TOUCHED}[args.update])
    # forward-only: no backward follows, so the forward emits nothing for one
    h.set_option(binding.OPT_BACKWARD_PATH,
                 binding.PATH_ATOMIC if args.forward_only else
                 {"auto": binding.PATH_AUTO, "atomic": binding.PATH_ATOMIC,
                  "sorted": binding.PATH_SORTED}[args.path])
    out = torch.empty((w.B, w.T, w.d), dtype=torch.float32, device=dev)
    nnz_per_step = [int(b[0].shape[0]) for b in batches]
    stream = torch.cuda.current_stream()

    def step(k):
        i, o, g = dbatches[k % len(dbatches)]
        h.forward(i, o, w.B, out=out)
        if not args.forward_only:
            h.backward_update(g, w.lr)

    for k in range(args.warmup):
        step(k)
    torch.cuda.synchronize()

    def timed(nsteps, profile):
        """Time nsteps steps with CUDA events on the launch stream (barrier +
        synchronize on both sides); with `profile`, the library also records
        CUDA events around each kernel group (they cost ~2 us each of stream
        time, so the headline region runs without them)."""
        h.set_option(binding.OPT_PROFILE, 1 if profile else 0)
        h.reset_profile()
        l0 = h.info()["kernel_launches"]
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.time()
        a.record(stream)
        for k in range(nsteps):
            step(k)
        b.record(stream)
        torch.cuda.synchronize()
        t1 = time.time()
        if world > 1:
            dist.barrier()
        pr = {}
        if profile:
            for kid, name in enumerate(binding.KERNEL_NAMES):
                n, ms = h.profile(kid)
                if n:
                    pr[name] = (n, ms)
        h.set_option(binding.OPT_PROFILE, 0)
        return a.elapsed_time(b), h.info()["kernel_launches"] - l0, pr, t0, t1

    sampler = ClockSampler(_gpu_id(torch, local)) if rank == 0 else None
    time.sleep(0.3 if sampler else 0)
    # headline region: the K steps, no per-kernel events
    elapsed_ms, launches, _, wall0, wall1 = timed(args.steps, False)
    # per-kernel split (and the roofline's launch durations): a second timed
    # region with the library's CUDA events around each kernel group
    split_steps = max(1, min(args.steps, 200))
    split_ms, _, prof, _, wall2 = timed(split_steps, True)
    if sampler:
        time.sleep(0.3)
        sampler.stop()
    lookups = sum(nnz_per_step[k % len(nnz_per_step)] for k in range(args.steps))
    if world > 1:
        elapsed_ms, lookups = reduce_over_ranks(dist, dev, elapsed_ms, lookups)

    # end to end through the same C-ABI calls with pinned HOST buffers:
    # every step copies indices, offsets and grad_out in and the pooled output out.
    e2e_steps = max(3, min(args.steps, args.e2e_steps))
    hb = [(torch.from_numpy(i).pin_memory(), torch.from_numpy(o).pin_memory(),
           torch.from_numpy(g).pin_memory()) for i, o, g in batches]
    hout = torch.empty((w.B, w.T, w.d), dtype=torch.float32, pin_memory=True)

    def step_host(k):
        i, o, g = hb[k % len(hb)]
        h.forward(i, o, w.B, out=hout)
        if not args.forward_only:
            h.backward_update(g, w.lr)

    step_host(0)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for k in range(e2e_steps):
        step_host(k)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    e2e_lookups = sum(nnz_per_step[k % len(nnz_per_step)] for k in range(e2e_steps))
    if world > 1:
        e2e_ms, e2e_lookups = reduce_over_ranks(dist, dev, e2e_ms, e2e_lookups)
    h2d = int(np.mean([i.nbytes + o.nbytes + (0 if args.forward_only else g.nbytes)
                       for i, o, g in batches]))
    d2h = int(hout.numel() * 4)
    props = torch.cuda.get_device_properties(dev)
    l2 = _l2_peaks(torch, dev, props.multi_processor_count) if rank == 0 else None
    # the shared array's working set (w, the Adagrad accumulator and the fp64
    # gradient: 16 bytes per element) fits in L2
    l2_size = getattr(props, "L2_cache_size", 0) or (126 << 20)
    array_in_l2 = 16 * w.M <= l2_size // 2
    # the optimizer pass visits only the touched blocks when the library chose
    # its touched update
    L = min(w.Z, w.d)
    touched_elems = None
    if (not args.forward_only and rank == 0
            and h.info()["last_update"] == binding.UPDATE_TOUCHED):
        touched_elems = _touched_elements(h, dbatches, L, torch)

    if rank == 0:
        clocks = sampler.summary(wall0, wall2) if sampler else None
        value = lookups / (elapsed_ms / 1e3)
        peak, peak_kind = _peaks()
        ab = _algorithmic_bytes(w)
        if touched_elems is not None:
            ab["update"] = (16 if w.opt == "adagrad" else 8) * touched_elems
        # dominant kernel with an algorithmic byte count (sort passes are pure
        # implementation overhead and have none)
        cands = {k: v for k, v in prof.items() if k in ab} or {"forward": (1, float("nan"))}
        dom = max(cands.items(), key=lambda kv: kv[1][1])[0]
        n_dom, ms_dom = cands[dom]
        avg_s = ms_dom / max(1, n_dom) / 1e3
        bytes_dom = ab[dom]
        achieved = bytes_dom / avg_s / 1e9
        kroof = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak,
                 "unit": "GB/s", "frac": achieved / peak, "traffic": _traffic(dom, args.workload),
                 "peak_kind": peak_kind, "algorithmic_bytes_per_launch": bytes_dom,
                 "avg_launch_ms": avg_s * 1e3}
        if dom == "update" and touched_elems is not None:
            kroof["note"] = (f"touched update: {touched_elems:.0f} distinct elements of M per batch "
                             "(union of the batch's blocks), each read and written once")
        if dom == "forward" and array_in_l2 and l2:
            # the forward's block gathers from the L2-resident array take
            # longer at the measured L2 gather rate than its HBM streams
            t_l2 = ab["l2_gather"] / (l2["gather_gbs"] * 1e9)
            if t_l2 > bytes_dom / (peak * 1e9):
                a_l2 = ab["l2_gather"] / avg_s / 1e9
                kroof.update({"bound": "l2", "achieved": a_l2, "peak": l2["gather_gbs"],
                              "frac": a_l2 / l2["gather_gbs"],
                              "peak_kind": "measured (L2 random 128-byte gather probe)",
                              "algorithmic_bytes_per_launch": ab["l2_gather"], "traffic": None})
        step_bytes = ab["forward"] if args.forward_only else ab["step"]
        step_gbs = step_bytes / (elapsed_ms / args.steps / 1e3) / 1e9 * world
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            rate, rows, reps, nnz_s, tot = _oracle_rate(w, args.cpu_budget, args.forward_only,
                                                        signed=args.signed)
            cpu = {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle", "host": _host(),
                   "sample": (f"first {rows} of {w.B} batch rows x {w.T} tables "
                              f"({nnz_s} lookups) per step, {reps} steps, {tot:.1f} s: "
                              + ("forward only" if args.forward_only else
                                 "forward + gradient + update") + ", single host thread")}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": _workload_desc(args, w), "global_batch": w.B * world,
                       "seq_len": 1,
                       "parallelism": "independent replicas" if world > 1 else "single GPU",
                       "grad_accumulator": args.accum,
                       "backward_path": ["auto", "atomic", "sorted"][h.info()["last_path"]],
                       **_sort_desc(h, binding, args),
                       **({} if args.forward_only else
                          {"update": {binding.UPDATE_DENSE: "dense", binding.UPDATE_TOUCHED: "touched blocks"}
                           .get(h.info()["last_update"], "SGD scattered into M")}),
                       "l2": (f"inputs larger than L2: {args.rotate}-batch rotation, "
                              f"{w.B * w.T * w.d * 4 / 1e6:.0f} MB output and "
                              f"{w.B * w.T * w.d * 4 / 1e6:.0f} MB upstream gradient per step"),
                       **_config_extra(args, w)},
            "step_gbs": step_gbs,
            "bags_per_s": w.B * w.T * args.steps * world / (elapsed_ms / 1e3),
            "roofline": dict(kroof, step_frac=step_gbs / world / peak),
            "step_roofline": _step_roofline(ab, elapsed_ms / args.steps / 1e3, peak, l2,
                                            args.forward_only, array_in_l2),
            "l2_peaks": l2,
            "kernels_ms": {k: v[1] / v[0] for k, v in prof.items()},
            "kernel_split": {"steps": split_steps, "ms_per_step_with_events": split_ms / split_steps,
                             "note": "kernels_ms and roofline.avg_launch_ms come from a second "
                                     "timed region of these steps with CUDA events around each "
                                     "kernel group; the headline region has none"},
            "gpu_launches": launches * world,
            "e2e": {"value": e2e_lookups / (e2e_ms / 1e3), "unit": UNIT,
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "steps": e2e_steps},
            "cpu_baseline": cpu,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    h.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(wl.CONFIGS), default="tb")
    ap.add_argument("--M", type=int, default=None, help="shared-array length (sweep workload)")
    ap.add_argument("--rotate", type=int, default=2, help="distinct batches cycled through")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-budget", type=float, default=15.0, help="seconds of oracle timing")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--accum", choices=["f64", "f32"], default="f64",
                    help="gradient accumulator precision of the atomic path")
    ap.add_argument("--B", type=int, default=None, help="override the batch size (profiling)")
    ap.add_argument("--path", choices=["auto", "atomic", "sorted"], default="auto",
                    help="backward path")
    ap.add_argument("--Z", type=int, default=None, help="override the chunk size Z")
    ap.add_argument("--G", type=int, default=None, help="override the offset alignment G")
    ap.add_argument("--forward-only", action="store_true",
                    help="time the forward (inference) alone")
    ap.add_argument("--signed", action="store_true", help="signed hashing (PSS_OPT_SIGNED)")
    ap.add_argument("--update", choices=["auto", "dense", "touched"], default="auto",
                    help="how the optimizer pass visits M (PSS_OPT_UPDATE_MODE)")
    ap.add_argument("--sort", choices=["auto", "global", "local"], default="auto",
                    help="sorted path: one sort over all pairs, the segment-local sort, or the "
                         "library's choice (PSS_OPT_SORT_SCOPE)")
    ap.add_argument("--deterministic", action="store_true",
                    help="run-to-run identical bits on the sorted path (PSS_OPT_DETERMINISTIC)")
    ap.add_argument("--ids", choices=["workload", "uniform"], default="workload",
                    help="id distribution: the workload's own (Zipf for the Criteo shapes) or "
                         "uniform over each table")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        raise SystemExit("--warmup must be at least 3")
    if args.workload == "sweep" and args.M is None:
        args.M = 1 << 24
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
