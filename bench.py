"""Throughput of one global round of distributed sign momentum with local steps.

A step is one global round of Algorithm 1 on the synthetic workload: tau
times (synthetic gradient fill for all n workers + one local base-optimizer
step on all n replicas), then the fused global step and its statistics.
By default the round is fused (the last local step runs inside the global
step and the replica reset is deferred to the next round's first local
step); --no-fused runs every step separately.  Both give identical results.
All inputs are resident in HBM when the timed region starts.

Metric: params/s per global round = d x rounds / device time (whole job).
Also reported: the dominant kernel's roofline (algorithmic bytes per launch
over its CUDA-event duration, against the measured HBM copy bandwidth), an
end-to-end figure through the C ABI with host gradient buffers, the SM
clocks seen during the timed region, and the C++ CPU oracle timed on a
bounded sample of the same workload.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload gpt2s] [--impl reference]

Under torchrun rank r of G runs shard r of one model made of G copies of
the workload's tensor list (d parameters per rank, starting at element r*d);
the path is elementwise, so the shards need no communication, and rank 0
prints one JSON line.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "params/s per global round (τ local + sign-momentum step); % HBM roofline"
UNIT = "params/s"
# the CPU oracle's samples: all host cores, and one thread (about 10-30 s of CPU work on the GPT-2 workloads)
CPU_SAMPLE_ELEMS = 1 << 27
CPU_ONE_CORE_ELEMS = 1 << 24
# the sources of the local-step kernels (their arithmetic lives in the shared device header)
KERNELS_SRC = [os.path.join(ROOT, "paper_2411_17866_gb300", "csrc", f) for f in ("dsm_device.cuh", "dsm_local.cu")]


def kernels_source_hash() -> str:
    h = hashlib.sha256()
    for f in KERNELS_SRC:
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default=W.BENCH_WORKLOAD, choices=sorted(W.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    # the five workloads' short CUDA-event runs (the line's "workloads" record)
    ap.add_argument("--no-workloads", action="store_true")
    # smaller cases of a workload (profiling captures): fewer workers, fewer local steps, or a
    # prefix of the tensor list holding at most this many parameters
    ap.add_argument("--n-workers", type=int, default=None)
    ap.add_argument("--tau", type=int, default=None)
    ap.add_argument("--max-params", type=int, default=None)
    # or one flat weight tensor of this many parameters (the workload's n, tau, hyper-parameters and the
    # first tensor's gradient scale)
    ap.add_argument("--flat-params", type=int, default=None)
    # the global step: Algorithm 1 (default) or a variant of the ablations
    ap.add_argument("--global-mode", default=None, choices=sorted(GLOBAL_MODES))
    # fused round (default): the last local step inside the global step, lazy replica reset
    ap.add_argument("--no-fused", dest="fused", action="store_false")
    # the variant in which every round restarts each worker's base optimizer from zero state
    ap.add_argument("--reset-local-state", action="store_true")
    return ap.parse_args()


GLOBAL_MODES = {"sign_momentum": W.GLOBAL_SIGN_MOMENTUM, "slowmo": W.GLOBAL_SLOWMO,
                "signed_slowmo": W.GLOBAL_SIGNED_SLOWMO, "lookahead": W.GLOBAL_LOOKAHEAD,
                "adamw": W.GLOBAL_ADAMW}


def select_workload(args):
    wl = W.WORKLOADS[args.workload]
    changes = {}
    notes = []
    if args.n_workers:
        changes["n"] = args.n_workers
        notes.append(f"n={args.n_workers}")
    if args.tau:
        changes["tau"] = args.tau
        notes.append(f"tau={args.tau}")
    if args.global_mode and GLOBAL_MODES[args.global_mode] != wl.hp.global_mode:
        mode = GLOBAL_MODES[args.global_mode]
        changes["hp"] = dataclasses.replace(wl.hp, global_mode=mode,
                                            sign_mode=wl.hp.sign_mode if mode == W.GLOBAL_SIGN_MOMENTUM else W.SIGN)
        notes.append(f"global step {args.global_mode}")
    if args.fused:   # an execution option: the results are bit-identical to the unfused round
        hp = changes.get("hp", wl.hp)
        changes["hp"] = dataclasses.replace(hp, flags=hp.flags | W.FLAG_FUSED_ROUND)
    else:
        notes.append("unfused round")
    if args.reset_local_state:   # a variant of the method: every round restarts the base optimizer
        hp = changes.get("hp", wl.hp)
        changes["hp"] = dataclasses.replace(hp, flags=hp.flags | W.FLAG_RESET_LOCAL_STATE)
        notes.append("base optimizer restarted every round")
    if args.max_params:
        keep, total = [], 0
        for t in wl.tensors:
            if keep and total + t.numel > args.max_params:
                break
            keep.append(t)
            total += t.numel
        changes["tensors"] = tuple(keep)
        notes.append(f"reduced to the first {len(keep)} tensors ({total} params)")
    if args.flat_params:
        changes["tensors"] = W.flat_layout(args.flat_params, wl.tensors[0].grad_scale)
        notes.append(f"one flat tensor of {args.flat_params} params")
    if changes:
        if notes:
            changes["name"] = wl.name + " [" + ", ".join(notes) + "]"
        wl = dataclasses.replace(wl, **changes)
    return wl


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(seconds: float, world: int) -> float:
    """The slowest rank's time (host-side gloo reduction; nothing on the data path)."""
    if world <= 1:
        return seconds
    import torch
    import torch.distributed as dist
    t = torch.tensor([seconds], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# A timed region whose clocks show one of these reasons, or SM clocks well below their maximum with no
# reason given (a clock lock left by someone else), is measured again once.
REJECTED_CLOCK_REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


def clocks_rejected(clocks) -> bool:
    if not clocks:
        return False
    if set(REJECTED_CLOCK_REASONS) & set(clocks["reasons"]):
        return True
    return not clocks["reasons"] and clocks["sm_mhz"] < 0.9 * clocks["sm_max_mhz"]


def any_rank(flag: bool, world: int) -> bool:
    """True on every rank if any rank's flag is true (host-side gloo reduction)."""
    return max_over_ranks(1.0 if flag else 0.0, world) > 0.5


def rank_shard(wl, world: int, rank: int):
    """Rank r's part of the weak-scaling model: `world` copies of the workload's tensor list, cut into
    `world` contiguous shards of d parameters (shard r is copy r and starts at element r*d of that model).
    Every step is elementwise, so the shards need no communication; together they compute exactly the
    one-process run of the whole model."""
    from paper_2411_17866_gb300.shard import repeated_model, shard_layout
    return shard_layout(repeated_model(wl.tensors, world), world, rank)


def whole_job_value(d_per_rank: int, world: int, rounds: int, seconds: float) -> float:
    """params/s over all ranks: every rank processes its own shard of d parameters per round."""
    return world * d_per_rank * rounds / seconds


def bytes_per_elem_local(wl, zero_state=False) -> int:
    """Algorithmic bytes of one local step per worker-element: every state read and written once
    (zero_state: the base optimizer restarts, its state is written but not read)."""
    g = 2 if wl.hp.grad_dtype == W.BF16 else 4
    states = 2 if wl.hp.base == W.BASE_ADAMW else 1
    # read x, the states and g; write x and the states
    return 4 + 4 * states * (1 if zero_state else 2) + g + 4


def local_step_bytes(wl, from_x=False, zero_state=False) -> int:
    """Algorithmic bytes of one local-step launch (from_x: every worker starts from the global x,
    read once per tile)."""
    b = bytes_per_elem_local(wl, zero_state)
    return wl.n * wl.d * (b - 4) + wl.d * 4 if from_x else wl.n * wl.d * b


def bytes_per_param_global(wl, lazy_reset=False) -> int:
    # read x, m (and the global AdamW second moment) and n replicas; write them all (the replicas
    # only when the reset is not deferred)
    return 8 * (wl.n + 2 + (1 if wl.hp.global_mode == W.GLOBAL_ADAMW else 0)) - (4 * wl.n if lazy_reset else 0)


def fused_round_active(wl) -> bool:
    """The library runs the last local step inside the global step with n <= 8 workers."""
    return bool(wl.hp.flags & W.FLAG_FUSED_ROUND) and wl.n <= 8


def lazy_reset_active(wl) -> bool:
    """With the fused-round flag the replicas' reset is deferred for any n: the next round's first
    local step starts every worker from x."""
    return bool(wl.hp.flags & W.FLAG_FUSED_ROUND)


def bytes_per_param_fused_last(wl, from_x=False, zero_state=False) -> int:
    """Fused last local step + global step: per worker read x_i (unless every worker starts from x),
    the optimizer state (unless it restarts from zero) and g, and write the state back (not when the
    round restarts the base optimizer; x_i is never written); read and write x and m (and the global
    AdamW second moment); no replica reset."""
    g = 2 if wl.hp.grad_dtype == W.BF16 else 4
    states = 2 if wl.hp.base == W.BASE_ADAMW else 1
    reset = bool(wl.hp.flags & W.FLAG_RESET_LOCAL_STATE)
    per_worker = (0 if from_x else 4) + g + (0 if zero_state else 4 * states) + (0 if reset else 4 * states)
    return wl.n * per_worker + 16 + (8 if wl.hp.global_mode == W.GLOBAL_ADAMW else 0)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def committed_traffic(kernel_key):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current kernels."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        j = json.load(f)
    ent = j.get(kernel_key)
    if not ent or ent.get("kernels_sha256_16") != kernels_source_hash():
        return None
    return ent.get("bytes_per_launch")


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.proc = None
        self.gpu = self.smi_id(gpu_index)

    @staticmethod
    def smi_id(local_index: int) -> str:
        """nvidia-smi's -i for CUDA device `local_index`: nvidia-smi ignores CUDA_VISIBLE_DEVICES, so use the
        device's UUID (or the listed id) rather than the CUDA index."""
        try:
            import torch
            uuid = str(torch.cuda.get_device_properties(local_index).uuid)
            if uuid:
                return uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            pass
        visible = os.environ.get("CUDA_VISIBLE_DEVICES", "").strip()
        if visible:
            ids = [v.strip() for v in visible.split(",") if v.strip()]
            if local_index < len(ids):
                return ids[local_index]
        return str(local_index)

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(self.gpu)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.3)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.strip().splitlines():
            f = [c.strip() for c in line.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append(dict(sm=float(f[1]), max=float(f[2]), power=float(f[3]), hw=f[5], hwt=f[6],
                                 swt=f[7], pcap=f[8]))
            except ValueError:
                continue
        if not rows:
            return None
        pmax = max(r["power"] for r in rows)
        loaded = [r for r in rows if r["power"] >= 0.5 * pmax] or rows
        reasons = set()
        for r in rows:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in loaded), "sm_max_mhz": rows[0]["max"],
                "reasons": sorted(reasons), "samples": len(rows), "power_w_max": pmax, "gpu": self.gpu}


def cxx_oracle_round(wl, count, threads, steps=1, warmup=0):
    """The C++ oracle, as it stands, over elements [0, count) of the workload with `threads` OpenMP threads
    (0: every host core): `warmup` untimed rounds, then the wall time of each of `steps` rounds."""
    import numpy as np

    from oracle.cxx_oracle import CxxOracleRun
    ora = CxxOracleRun(wl.tensors, wl.n, wl.tau, wl.hp, elems=np.arange(count, dtype=np.int64), threads=threads)
    for _ in range(warmup):
        ora.run_round()
    walls = []
    for _ in range(steps):
        t0 = time.perf_counter()
        ora.run_round()
        walls.append(time.perf_counter() - t0)
    return walls


def oracle_threads() -> int:
    from oracle.cxx_oracle import load
    return int(load().dsmo_max_threads())


def cpu_baseline(wl, elems_count=CPU_SAMPLE_ELEMS, one_core_count=CPU_ONE_CORE_ELEMS):
    """The C++ oracle, as it stands: one round over a contiguous sample of the workload on every host core
    (OpenMP over elements), and one round over a smaller sample on one thread."""
    count = min(elems_count, wl.d)
    one = min(one_core_count, wl.d)
    cores = oracle_threads()
    wall = cxx_oracle_round(wl, count, 0)[0]
    wall1 = cxx_oracle_round(wl, one, 1)[0]
    return {"value": count / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"1 round (tau={wl.tau} local steps x n={wl.n} workers + global step) over elements "
                      f"[0, {count}) of the {wl.d}-parameter layout: the C++ oracle (g++ -O2 -ffp-contract=off), "
                      f"OpenMP over elements on {cores} threads; {wall:.2f} s",
            "one_core": {"value": one / wall1, "cores": 1,
                         "sample": f"1 round over elements [0, {one}), one thread; {wall1:.2f} s"}}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    wl = select_workload(args)
    # each step one round over a contiguous sample, sized so that the whole run stays near a minute of
    # wall time whatever --steps and --warmup are (about 2^23 elements per step at the defaults)
    per_step = (1 << 23) * (20 + 3) // max(1, args.steps + args.warmup)
    per_step = per_step * 48 // (wl.n * wl.tau)          # the defaults' n*tau is 48
    count = int(min(max(per_step, 1 << 14), 1 << 25, wl.d))
    cores = oracle_threads()
    walls = cxx_oracle_round(wl, count, 0, steps=args.steps, warmup=args.warmup)
    dt = sum(walls)
    value = count * args.steps / dt
    sample = (f"each step: one round (tau={wl.tau} x n={wl.n} local steps + global step) over elements "
              f"[0, {count}) of the {wl.d}-parameter layout; the C++ oracle (g++ -O2 -ffp-contract=off), "
              f"OpenMP over elements on {cores} threads")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": compute_dtype(wl),
            "data": "synthetic", "config": workload_config(wl, args.gpus),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def workload_config(wl, gpus):
    return {"workload": wl.name, "d": wl.d, "n_workers": wl.n, "tau": wl.tau, "tensors": len(wl.tensors),
            "base": "adamw" if wl.hp.base == W.BASE_ADAMW else "sgd-momentum",
            "grad_dtype": "bf16" if wl.hp.grad_dtype == W.BF16 else "f32",
            "sign": ["sign", "rand-sign-2", "rand-sign-1"][wl.hp.sign_mode],
            "global_step": {v: k for k, v in GLOBAL_MODES.items()}[wl.hp.global_mode],
            "fused_round": bool(wl.hp.flags & W.FLAG_FUSED_ROUND),
            "parallelism": (f"parameter shards x{gpus}: rank r holds elements [r*d, (r+1)*d) of {gpus} copies "
                            "of the tensor list, no collective on the data path") if gpus > 1 else "single GPU",
            "l2": l2_note(wl)}


L2_BYTES = 129e6


def l2_note(wl) -> str:
    """How the timed rounds stand to the 129 MB L2 (no flush between rounds: the launches stream more than L2,
    except on workloads whose whole state fits in it)."""
    launch = wl.n * wl.d * bytes_per_elem_local(wl)
    if launch > L2_BYTES:
        return f"inputs larger than L2 (129 MB): each local-step launch streams {launch / 1e9:.1f} GB"
    return (f"not flushed: each local-step launch streams {launch / 1e9:.3f} GB, less than L2 (129 MB), "
            "so these rounds run partly from L2")


SPEC_HBM_GBS = 8000.0   # GB300's HBM3e figure (~8 TB/s) that the 80 % per-kernel target is stated against


def round_events(run, wl, stream, t, tau, fused, lazy, reset, rec):
    """Enqueue one global round; with `rec` (a dict of lists) bracket each launch with CUDA events on the
    launching stream and record the algorithmic bytes of every local-step and global-step launch."""
    import torch

    def ev():
        return torch.cuda.Event(enable_timing=True)

    for k in range(tau):
        if rec is not None:
            a, b = ev(), ev()
            a.record(stream)
            run.fill_synthetic_grads(t * tau + k, stream)
            b.record(stream)
            rec["fill"].append((a, b, 0))
        else:
            run.fill_synthetic_grads(t * tau + k, stream)
        if rec is not None and not (fused and k == tau - 1):
            a, b = ev(), ev()
            a.record(stream)
            run.local_step(stream)
            b.record(stream)
            # deferred reset: the first local step starts every worker from x (read once per tile);
            # restarted base optimizer: the first local step reads no state
            nbytes = local_step_bytes(wl, from_x=lazy and k == 0 and t > 0, zero_state=reset and k == 0 and t > 0)
            rec["local"].append((a, b, nbytes))
        else:
            run.local_step(stream)
    if rec is not None:
        a, b = ev(), ev()
        a.record(stream)
        run.global_step(stream)
        b.record(stream)
        if fused:   # with tau = 1 the fused launch is also the round's first local step
            first = tau == 1 and t > 0
            gbytes = wl.d * bytes_per_param_fused_last(wl, from_x=first, zero_state=reset and first)
        else:
            gbytes = wl.d * bytes_per_param_global(wl, lazy)
        rec["global"].append((a, b, gbytes))
    else:
        run.global_step(stream)


def time_rounds(run, wl, stream, t, warmup, steps, world=1, sampler=None):
    """W untimed rounds, then K rounds between CUDA events on the launching stream (barrier and
    synchronize on both sides).  Returns the next round index and the per-kernel timings."""
    import torch
    import torch.distributed as dist
    fused, lazy = fused_round_active(wl), lazy_reset_active(wl)
    reset = bool(wl.hp.flags & W.FLAG_RESET_LOCAL_STATE)
    for _ in range(warmup):
        round_events(run, wl, stream, t, wl.tau, fused, lazy, reset, None)
        t += 1
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
    rec = {"fill": [], "local": [], "global": []}
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(steps):
        round_events(run, wl, stream, t, wl.tau, fused, lazy, reset, rec)
        t += 1
    end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop() if sampler else None
    res = {"elapsed": max_over_ranks(start.elapsed_time(end) / 1e3, world), "clocks": clocks, "fused": fused,
           "lazy": lazy}
    for key, evs in rec.items():
        res[key + "_ms"] = [a.elapsed_time(b) for a, b, _ in evs]
        res[key + "_bytes"] = [nb for _, _, nb in evs]
    return t, res


def kernel_figures(wl, res, peak):
    """Per-kernel achieved bandwidth (algorithmic bytes over CUDA-event time) against both peaks."""
    local_ms, global_ms = res["local_ms"], res["global_ms"]
    global_gbs = sum(res["global_bytes"]) / (sum(global_ms) / 1e3) / 1e9
    out = {"global_gbs": global_gbs, "global_frac": global_gbs / peak, "global_spec_frac": global_gbs / SPEC_HBM_GBS,
           "global_avg_ms": statistics.mean(global_ms), "global_bytes": statistics.mean(res["global_bytes"])}
    if local_ms:
        local_gbs = sum(res["local_bytes"]) / (sum(local_ms) / 1e3) / 1e9
        out.update(local_gbs=local_gbs, local_frac=local_gbs / peak, local_spec_frac=local_gbs / SPEC_HBM_GBS,
                   local_avg_ms=statistics.mean(local_ms), local_bytes=local_step_bytes(wl))
    out["optimizer_only_value"] = wl.d * len(global_ms) / ((sum(local_ms) + sum(global_ms)) / 1e3)
    return out


def copy_gbs(nbytes, dev, stream, reps=8):
    """Bandwidth of a plain device-to-device copy that moves `nbytes` (half read, half written; capped at
    2 GiB), over its CUDA-event time (median of `reps`), with L2 flushed before each copy: the copy roofline
    at a launch of that size, which small launches (ramp and tail of a short kernel) keep below the large
    copy's peak."""
    import torch
    nbytes = min(int(nbytes), 2 << 30)
    src = torch.empty(max(nbytes // 8, 1), dtype=torch.float32, device=dev)
    dst = torch.empty_like(src)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)   # larger than the 129 MB L2
    times = []
    for r in range(reps + 2):
        flush.zero_()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        dst.copy_(src)
        b.record(stream)
        torch.cuda.synchronize()
        if r >= 2:
            times.append(a.elapsed_time(b) / 1e3)
    moved = 2 * src.numel() * 4
    del src, dst, flush
    return moved / statistics.median(times) / 1e9


def workload_sweep(dev, stream, peak, skip, steps=3, warmup=2):
    """Every measured workload (fused round, as configured) timed briefly in this process with CUDA events:
    params/s of the round and each kernel's fraction of both peaks.  `skip` maps a workload already timed
    in this job to its figures."""
    import torch

    from paper_2411_17866_gb300 import dsm
    out = {}
    for key in ("flat1m", "gpt2s", "gpt2m", "gpt2l", "gpt2xl"):
        if key in skip:
            out[key] = skip[key]
            continue
        wl = W.WORKLOADS[key]
        wl = dataclasses.replace(wl, hp=dataclasses.replace(wl.hp, flags=wl.hp.flags | W.FLAG_FUSED_ROUND))
        run = dsm.DistributedSignMomentum(wl.tensors, wl.n, wl.tau, wl.hp, device=dev)
        _, res = time_rounds(run, wl, stream, 0, warmup, steps)
        run.close()
        del run
        torch.cuda.empty_cache()
        out[key] = sweep_entry(wl, res, peak, steps)
    for key, e in out.items():   # the plain copy's bandwidth at each workload's local-step launch size
        wl = W.WORKLOADS[key]
        c = copy_gbs(local_step_bytes(wl), dev, stream)
        e["copy_gbs_at_launch_size"] = c
        if "local_step_gbs" in e:
            e["local_step_frac_of_copy_at_launch_size"] = e["local_step_gbs"] / c
        torch.cuda.empty_cache()
    return out


def sweep_entry(wl, res, peak, steps):
    f = kernel_figures(wl, res, peak)
    e = {"params_per_s": wl.d * steps / res["elapsed"], "ms_per_round": res["elapsed"] / steps * 1e3,
         "rounds_timed": steps, "optimizer_only_params_per_s": f["optimizer_only_value"],
         "fused_last_plus_global_gbs": f["global_gbs"], "fused_last_plus_global_frac": f["global_frac"],
         "fused_last_plus_global_frac_of_8tbs": f["global_spec_frac"],
         "grad_fill_ms": statistics.mean(res["fill_ms"])}
    if "local_gbs" in f:
        e.update(local_step_gbs=f["local_gbs"], local_step_frac=f["local_frac"],
                 local_step_frac_of_8tbs=f["local_spec_frac"])
    return e


def compute_dtype(wl) -> str:
    """The arithmetic type of the path, with the gradients' storage type where it differs."""
    return "f32 (bf16 grads)" if wl.hp.grad_dtype == W.BF16 else "f32"


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    rank, world, local = dist_env()

    import torch
    import torch.distributed as dist

    from paper_2411_17866_gb300 import dsm
    if world > 1:
        dist.init_process_group("gloo", rank=rank, world_size=world)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    wl = select_workload(args)
    shard = rank_shard(wl, world, rank)
    run = dsm.DistributedSignMomentum(shard.tensors, wl.n, wl.tau, wl.hp, device=dev,
                                      first_element=shard.first_element)
    stream = torch.cuda.current_stream(dev)
    tau = wl.tau

    sampler = ClockSampler(local) if (rank == 0 and not args.no_clocks) else None
    t, res = time_rounds(run, wl, stream, 0, args.warmup, args.steps, world, sampler)
    if any_rank(clocks_rejected(res["clocks"]), world):   # throttled or clock-locked: measure once more
        first = res["clocks"]
        sampler = ClockSampler(local) if (rank == 0 and not args.no_clocks) else None
        t, res = time_rounds(run, wl, stream, t, 1, args.steps, world, sampler)
        if res["clocks"] is not None and first is not None:
            res["clocks"]["remeasured_after"] = {k: first[k] for k in ("sm_mhz", "reasons")}
    elapsed, clocks, fused, lazy = res["elapsed"], res["clocks"], res["fused"], res["lazy"]

    # end to end through the C ABI with host buffers: per round, tau x (pinned host -> device
    # gradient copy + local step), the global step, and the new x read back to pinned host memory
    e2e = None
    if not args.no_e2e:
        esz = 2 if wl.hp.grad_dtype == W.BF16 else 4
        gdt = torch.bfloat16 if esz == 2 else torch.float32
        host_g = torch.empty((wl.n, wl.d), dtype=gdt).pin_memory()
        run.fill_synthetic_grads(t * tau, stream)   # the gradients of one synthetic step, staged once
        for i in range(wl.n):
            run.read(dsm.BUF_GRAD, i, out=host_g[i], stream=stream)
        host_x = torch.empty(wl.d, dtype=torch.float32).pin_memory()
        copy_stream = torch.cuda.Stream(dev)

        def e2e_round():
            for k in range(tau):
                # the copy of each chunk of gradients overlaps the update of the previous chunk
                run.local_step_host_grads(host_g, stream, copy_stream)
            run.global_step(stream)
            run.read(dsm.BUF_X, out=host_x, stream=stream)   # synchronises the stream

        e2e_round()   # one untimed round: first use of the pinned buffers and of the chunk events
        t += 1
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_round()
            t += 1
        e2e_dt = max_over_ranks(time.perf_counter() - t0, world)
        e2e = {"value": whole_job_value(wl.d, world, args.e2e_steps, e2e_dt), "unit": UNIT,
               "h2d_bytes_per_step": tau * wl.n * wl.d * esz, "d2h_bytes_per_step": wl.d * 4,
               "steps": args.e2e_steps, "path": "dsm_local_step_host_grads (pinned host gradients, chunked "
                                                 "copies on a second stream) x tau, dsm_global_step, "
                                                 "dsm_read_params(x -> pinned host)"}
        del host_g, host_x
    run.close()
    del run
    torch.cuda.empty_cache()

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return 0

    peak, peak_kind = measured_peaks()
    f = kernel_figures(wl, res, peak)
    grad_bytes = wl.n * wl.d * (2 if wl.hp.grad_dtype == W.BF16 else 4)
    if "local_gbs" in f:   # the dominant kernel: the local step
        achieved, avg_local_ms, local_bytes = f["local_gbs"], f["local_avg_ms"], f["local_bytes"]
        kname = "local_adamw" if wl.hp.base == W.BASE_ADAMW else "local_sgdm"
        # the traffic record holds for the workload as configured by default (a full local-step launch)
        default = wl.name == W.WORKLOADS[args.workload].name
        traffic = committed_traffic(f"{kname}:{args.workload}") if default else None
    else:          # tau = 1 in the fused round: the only launch is the fused last step + global step
        achieved, avg_local_ms, local_bytes = f["global_gbs"], f["global_avg_ms"], f["global_bytes"]
        kname, traffic = "fused_last_global", None
    value = whole_job_value(wl.d, world, args.steps, elapsed)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": elapsed / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": compute_dtype(wl), "data": "synthetic",
        "config": workload_config(wl, world),
        "roofline": {"bound": "hbm", "kernel": kname, "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "spec_peak": SPEC_HBM_GBS, "spec_frac": achieved / SPEC_HBM_GBS,
                     "traffic": traffic, "algorithmic_bytes_per_launch": local_bytes,
                     "avg_launch_ms": avg_local_ms},
        "global_step": {"bytes_per_launch": f["global_bytes"], "avg_ms": f["global_avg_ms"],
                        "achieved_gbs": f["global_gbs"], "frac": f["global_frac"], "spec_frac": f["global_spec_frac"],
                        "note": ("last local step fused with the global step, + statistics reduction"
                                 if fused else "fused global step + statistics reduction" +
                                 (" (replica reset deferred)" if lazy else "")) +
                                ", CUDA events around both"},
        "grad_fill": {"avg_ms": statistics.mean(res["fill_ms"]), "bytes_written_per_launch": grad_bytes,
                      "write_gbs": grad_bytes / (statistics.mean(res["fill_ms"]) / 1e3) / 1e9,
                      "note": "synthetic gradients (stand-in for the backward pass); bound by instruction "
                              "issue of the SplitMix64 hash"},
        "optimizer_only_value": f["optimizer_only_value"],
        # per round: tau gradient fills, tau local steps (tau - 1 in the fused round), the global step and
        # the statistics reduction
        "gpu_launches": args.steps * (2 * tau + (1 if fused else 2)),
        "e2e": e2e,
        "clocks": clocks,
    }
    if not args.no_workloads and world == 1:
        sampler = ClockSampler(local) if not args.no_clocks else None
        if sampler:
            sampler.start()
        done = {}
        if wl.name == W.WORKLOADS[args.workload].name and fused:
            done[args.workload] = sweep_entry(wl, res, peak, args.steps)
        sweep = workload_sweep(dev, stream, peak, done)
        line["workloads"] = {"note": "each workload's fused round as configured, timed in this job with CUDA "
                                     "events (2 untimed + 3 timed rounds; the bench workload's entry is the "
                                     "timed region above); fractions of the measured copy peak and of 8 TB/s, "
                                     "and of a plain copy moving one local-step launch's bytes (at most 2 GiB, "
                                     "L2 flushed before each copy)",
                             "clocks": sampler.stop() if sampler else None, **sweep}
    if not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = cpu_baseline(wl)
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
