#!/usr/bin/env python
"""Benchmark of the GB300 BD-LRU scan (RecBLR, arXiv 2406.12580, Sec. 3.2-3.3).

One step = one forward scan plus one backward scan (the whole training hot
path: gates, decay and input normalisation, forward scan, reverse scan,
dLambda) over one batch of synthetic input. The headline workload is the
long-sequence one, B=8, L=32768, D=512, bfloat16 I/O with float32 state
(XLong-like histories scaled up): its inputs (2.9 GB a step) are larger than
L2, so K steps run back to back between two CUDA events, each C-ABI call also
bracketed by its own events for the per-kernel roofline. Inputs are resident
in HBM when the timed region starts.

The other workloads are reported beside it, each with its own roofline
(`configs`): they fit L2, so L2 is flushed (a 2x L2 write) before every timed
call, the backward's included.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--config 0-4] [--extras]

Prints one JSON line on rank 0 (--extras: a second line with further
workloads on stderr). Under torchrun each rank runs its own replica of the
workload (the scan shards over batch rows and channels with no exchange), so
the value is the sum over ranks ("weak" scaling).

--impl reference times the float64 CPU oracle, as it stands, on the host
cores (there is no other implementation of this method to compare against).
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "BD-LRU scan fwd+bwd elements/s and achieved HBM GB/s vs GB300 peak (1 GPU)"
UNIT = "elements/s"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e nominal, reported beside the measured-peak fractions

# Compulsory HBM bytes per element (inputs read once, outputs written once;
# the per-tile carries and O(B*D) state are overhead, not counted):
#   forward : x, rho, iota read, h written             = 4 values
#   backward: dh, x, rho, iota read, dx, drho, diota   = 7 values
#   step    : h_prev (f32), x, rho, iota read, h_t (f32) written
FWD_VALUES, BWD_VALUES = 4, 7


def io_bytes(io: str) -> int:
    return 2 if io == "bf16" else 4


def step_bytes_per_elem(io: str) -> int:
    return 4 + 3 * io_bytes(io) + 4


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=4, help="workload (0-4); 4 is the headline")
    ap.add_argument("--quick", action="store_true", help="skip the other workloads and e2e")
    ap.add_argument("--extras", action="store_true",
                    help="also time the gated, varlen, K-step and layer workloads (stderr)")
    ap.add_argument("--seq-len", type=int, default=0,
                    help="replace the workload's L (smaller cases for profiler captures)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--io", choices=["f32", "bf16"], default="",
                    help="override the workload's I/O dtype (profiling other kernel families)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_workload(cfg, rank: int):
    """The workload rank `rank` scans in a multi-GPU run: the same shape with
    its own seed (batch rows are independent problems, so ranks share no data
    and need no collective on the data path). Rank 0 scans the workload itself."""
    if rank == 0:
        return cfg
    return dataclasses.replace(cfg, seed=cfg.seed + 7919 * rank)


def max_over_ranks(local: float, world: int, device=None) -> float:
    """The largest of the ranks' values (the step time of the slowest rank);
    `device` is where the reduction tensor lives (CUDA for NCCL, CPU for gloo)."""
    if world == 1:
        return local
    import torch
    import torch.distributed as dist
    t = torch.tensor([local], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def code_text(src: str) -> str:
    """A CUDA/C++ source without its comments and blank lines, each line
    stripped: what the compiler sees, so that a comment edit leaves it alone."""
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    lines = (re.sub(r"//.*", "", ln).strip() for ln in src.splitlines())
    return "\n".join(ln for ln in lines if ln)


def kernel_sources_sha() -> str:
    """Hash of the library's code (comments excluded), which the committed ncu
    traffic figures are tied to."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2406_12580_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name), encoding="utf-8") as f:
            h.update(name.encode() + b"\0" + code_text(f.read()).encode())
    return h.hexdigest()[:16]


def scan_kernels(cfg):
    """(forward kernels, backward kernels, our kernels per forward call, per
    backward call) of the family the library runs on this shape
    (blr_scan_family). The chained kernels also clear their records with one
    cudaMemsetAsync a call, which is not counted as a kernel of ours."""
    from paper_2406_12580_gb300 import (FAMILY_SEGMENTED, FAMILY_SERIAL, Desc,
                                        blr_scan_family)
    fam = blr_scan_family(Desc(cfg.B, cfg.L, cfg.D, 0 if cfg.io == "f32" else 1, cfg.c))
    if fam == FAMILY_SERIAL:
        return "seq_fwd_kernel", "seq_bwd_kernel", 1, 1
    if fam == FAMILY_SEGMENTED:
        return "chain_fwd_kernel", "chain_bwd_kernel", 1, 1
    return "prep_kernel+scan_fwd_kernel", "prep_kernel+scan_bwd_kernel", 2, 2


def config_dict(cfg, world: int, l2: str) -> dict:
    """The `config` object of the JSON line (the same for both arms)."""
    return {"workload": cfg.name, "B": cfg.B, "L": cfg.L, "D": cfg.D, "io": cfg.io,
            "state": "f32", "parallelism": f"replicas{world}" if world > 1 else "single",
            "l2": l2, "inputs": "seeded synthetic (paper_2406_12580_gb300.inputs), resident in HBM"}


def l2_policy(cfg, l2_bytes: int):
    """(flush between timed calls?, description): workloads whose per-step
    traffic exceeds twice the L2 run back to back, the others flush L2."""
    step_bytes = cfg.elements * (FWD_VALUES + BWD_VALUES) * io_bytes(cfg.io)
    if step_bytes > 2 * l2_bytes:
        return False, f"inputs larger than L2 ({step_bytes / 1e9:.2f} GB a step): no flush"
    return True, f"flushed before every timed call ({2 * l2_bytes >> 20} MiB write)"


def ncu_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources (else None)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except Exception:
        return None
    if d.get("sources_sha") != kernel_sources_sha():
        return None
    return d.get("kernels", {}).get(kernel, {}).get(workload)


# ------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 100 ms."""

    QUERY = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.t0 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t0 = time.time()
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return []
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=10)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            if self.uuid and self.uuid not in f[0]:
                continue
            try:
                rows.append(dict(sm=float(f[1]), sm_max=float(f[2]), power=float(f[3]),
                                 hw_slowdown=f[5] == "Active", hw_thermal=f[6] == "Active",
                                 sw_thermal=f[7] == "Active", sw_power_cap=f[8] == "Active"))
            except ValueError:
                continue
        return rows

    @staticmethod
    def summary(rows):
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        loaded = [r for r in rows if r["power"] > 200.0] or rows
        reasons = sorted({k for r in loaded for k in ("hw_slowdown", "hw_thermal", "sw_thermal",
                                                      "sw_power_cap") if r[k]})
        return {"sm_mhz": statistics.median(r["sm"] for r in loaded),
                "sm_max_mhz": max(r["sm_max"] for r in rows), "reasons": reasons,
                "samples": len(loaded), "power_w_max": max(r["power"] for r in rows)}


# ------------------------------------------------------------ CPU baseline

def cpu_oracle_rate(inp, target_s: float = 10.0, max_reps: int = 1000, threads: int = 0):
    """The float64 oracle, as it stands, on the host cores (all of them, or
    `threads`): fwd + bwd over the whole workload, repeated for about
    `target_s` seconds. Returns (elements/s, threads, reps, seconds)."""
    import oracle
    orc = oracle.load()
    threads = threads or os.cpu_count() or 1
    n = inp.cfg.elements
    t = time.perf_counter()
    reps = 0
    while True:
        orc.fwd(inp.x, inp.gl, inp.lam, inp.h0, c=inp.cfg.c, threads=threads)
        if inp.dh is not None:
            orc.bwd(inp.dh, inp.x, inp.gl, inp.lam, inp.h0, inp.dh_last, c=inp.cfg.c,
                    threads=threads)
        reps += 1
        el = time.perf_counter() - t
        if el >= target_s or reps >= max_reps:
            break
    threads_used = threads if orc.has_openmp else 1
    return n * reps / el, threads_used, reps, el


# --------------------------------------------------------------- reference

def nominal_l2_bytes() -> int:
    """L2 size of the device if torch can see one, else GB300's 129 MiB."""
    try:
        import torch
        if torch.cuda.is_available():
            v = int(getattr(torch.cuda.get_device_properties(0), "L2_cache_size", 0) or 0)
            if v > 0:
                return v
    except Exception:
        pass
    return 129 << 20


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2406_12580_gb300 import inputs as I
    import oracle
    orc = oracle.load()
    cfg = I.CONFIGS[args.config]
    threads = os.cpu_count() or 1
    # One reference step = fwd + bwd of the oracle over a bounded sample of the
    # workload (whole batch rows), sized so that warm-up and timed steps take
    # about two minutes in all.
    per_step_s = min(1.0, 120.0 / max(1, args.steps + args.warmup))
    probe_rows = 1 if cfg.L * cfg.D > (1 << 20) else max(1, min(cfg.B, 8))
    probe = I.make_scan_inputs(I.scaled(cfg, B=probe_rows))
    t = time.perf_counter()
    orc.fwd(probe.x, probe.gl, probe.lam, probe.h0, c=cfg.c, threads=threads)
    if probe.dh is not None:
        orc.bwd(probe.dh, probe.x, probe.gl, probe.lam, probe.h0, probe.dh_last, c=cfg.c,
                threads=threads)
    per_row = (time.perf_counter() - t) / probe.cfg.B
    Bs = int(max(1, min(cfg.B, per_step_s / max(per_row, 1e-9))))
    inp = probe if Bs == probe_rows else I.make_scan_inputs(I.scaled(cfg, B=Bs))

    def step():
        orc.fwd(inp.x, inp.gl, inp.lam, inp.h0, c=cfg.c, threads=threads)
        if inp.dh is not None:
            orc.bwd(inp.dh, inp.x, inp.gl, inp.lam, inp.h0, inp.dh_last, c=cfg.c, threads=threads)

    for _ in range(args.warmup):
        step()
    t = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t
    value = inp.cfg.elements * args.steps / el
    sample = f"{Bs} of {cfg.B} batch rows of {cfg.name} per step (fwd+bwd, float64 oracle)"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": config_dict(cfg, args.gpus, l2_policy(cfg, nominal_l2_bytes())[1]),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads if orc.has_openmp else 1,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# -------------------------------------------------------------------- ours

def time_calls(buf, reps, flush=None, with_bwd=True):
    """Times `reps` steps (forward, then backward) with CUDA events on the
    launching stream: per call, and, when nothing runs between the steps
    (flush is None), the whole region. With `flush`, L2 is flushed before
    every call. Returns (fwd ms list, bwd ms list, region ms or None)."""
    import torch
    E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    ev = [(E(), E(), E(), E()) for _ in range(reps)]
    r0, r1 = E(), E()
    r0.record()
    for e0, e1, e2, e3 in ev:
        if flush is not None:
            flush()
        e0.record()
        buf.fwd()
        e1.record()
        if with_bwd:
            if flush is not None:
                flush()
            e2.record()
            buf.bwd()
            e3.record()
    r1.record()
    torch.cuda.synchronize()
    fwd_ms = [a.elapsed_time(b) for a, b, _, _ in ev]
    bwd_ms = [c.elapsed_time(d) for _, _, c, d in ev] if with_bwd else []
    return fwd_ms, bwd_ms, (r0.elapsed_time(r1) if flush is None else None)


def time_step_kernel(sbuf, reps, flush):
    import torch
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(reps)]
    for k in range(reps):
        flush()
        ev[k][0].record()
        sbuf.step()
        ev[k][1].record()
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in ev]


def call_roofline(kernel: str, alg_bytes: float, ms: float, peak: float, peak_kind: str, traffic):
    """Roofline block of one C-ABI call: algorithmic bytes over its mean
    event-timed duration, against the measured copy bandwidth."""
    gbs = alg_bytes / (ms * 1e-3) / 1e9
    return {"bound": "hbm", "kernel": kernel, "achieved": gbs, "peak": peak, "peak_kind": peak_kind,
            "unit": "GB/s", "frac": gbs / peak, "traffic": traffic, "algorithmic_bytes": alg_bytes,
            "us": ms * 1e3}


def workload_rooflines(cfg, fwd_ms, bwd_ms, peak, peak_kind, tag):
    """Per-call rooflines (mean times) and the fwd+bwd fraction of a workload."""
    n, ib = cfg.elements, io_bytes(cfg.io)
    fk, bk, _, _ = scan_kernels(cfg)
    f = sum(fwd_ms) / len(fwd_ms)
    out = {"workload": cfg.name,
           "fwd": call_roofline(fk, n * FWD_VALUES * ib, f, peak, peak_kind, ncu_traffic(fk, tag))}
    if bwd_ms:
        b = sum(bwd_ms) / len(bwd_ms)
        out["bwd"] = call_roofline(bk, n * BWD_VALUES * ib, b, peak, peak_kind, ncu_traffic(bk, tag))
        gbs = n * (FWD_VALUES + BWD_VALUES) * ib / ((f + b) * 1e-3) / 1e9
        out.update(elements_per_s=n / ((f + b) * 1e-3), fwd_bwd_gbs=gbs, fwd_bwd_frac=gbs / peak)
    else:
        out["elements_per_s"] = n / (f * 1e-3)
    return out


def run_ours(args):
    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import ScanBuffers

    peak, peak_kind = measured_peaks()
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 0) or 0) or nominal_l2_bytes()
    flush_buf = torch.empty(2 * l2 // 4 + 1024, dtype=torch.float32, device=dev)
    flush = lambda: flush_buf.fill_(1.0)  # noqa: E731

    cfg = I.CONFIGS[args.config]
    if args.seq_len > 0:
        cfg = dataclasses.replace(cfg, name=f"{cfg.name} at L={args.seq_len}", L=args.seq_len)
    if args.io and args.io != cfg.io:
        cfg = dataclasses.replace(cfg, name=f"{cfg.name} as {args.io}", io=args.io)
    cfg = rank_workload(cfg, rank)
    inp = I.make_scan_inputs(cfg)
    buf = ScanBuffers.from_inputs(inp, device=dev)
    n = cfg.elements
    do_flush, l2_note = l2_policy(cfg, l2)
    tflush = flush if do_flush else None

    def step():
        if tflush is not None:
            tflush()
        buf.fwd()
        if not cfg.fwd_only:
            if tflush is not None:
                tflush()
            buf.bwd()

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    uuid = None
    try:
        uuid = str(props.uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    sampler.start()
    # Untimed pre-roll of the same steps (about 0.5 s) so that the clock
    # samples see the GPU under this load before and during the timed region.
    t_pre = time.time()
    preroll = 0
    while time.time() - t_pre < 0.5:
        for _ in range(20):
            step()
        preroll += 20
        torch.cuda.synchronize()

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    fwd_ms, bwd_ms, region_ms = time_calls(buf, args.steps, tflush, with_bwd=not cfg.fwd_only)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    wall = time.perf_counter() - wall0
    clock_rows = sampler.stop()

    total_ms = region_ms if region_ms is not None else sum(fwd_ms) + sum(bwd_ms)
    t_max_ms = max_over_ranks(total_ms, world, device=dev)
    value = world * n * args.steps / (t_max_ms * 1e-3)
    tag = f"config{args.config}" if args.seq_len == 0 and not args.io else None
    rl = workload_rooflines(cfg, fwd_ms, bwd_ms, peak, peak_kind, tag)
    dominant = rl["bwd"] if "bwd" in rl and rl["bwd"]["us"] > rl["fwd"]["us"] else rl["fwd"]
    _, _, kf, kb = scan_kernels(cfg)
    ib = io_bytes(cfg.io)
    step_gbs = n * ((FWD_VALUES + (0 if cfg.fwd_only else BWD_VALUES)) * ib) * args.steps / (
        total_ms * 1e-3) / 1e9

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": max(3, args.warmup), "preroll_steps": preroll,
        "ms_per_step": t_max_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32" if cfg.io == "f32" else "bf16", "data": "synthetic",
        "config": config_dict(cfg, world, l2_note),
        "hbm_gbs": step_gbs, "hbm_frac": step_gbs / peak, "hbm_frac_nominal": step_gbs / NOMINAL_HBM_GBS,
        "roofline": dominant,
        "calls": {k: rl[k] for k in ("fwd", "bwd") if k in rl},
        "gpu_launches": (kf + (0 if cfg.fwd_only else kb)) * args.steps,
        "wall_s_timed_region": wall,
        "timing": ("CUDA events on the launching stream: the K steps back to back between two "
                   "events (value), and each C-ABI call between its own (per-call rooflines)"
                   if region_ms is not None else
                   "CUDA events around each C-ABI call, L2 flushed before each (value and rooflines)"),
    }

    rows_summary = ClockSampler.summary(clock_rows)
    line["clocks"] = {k: rows_summary[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")}
    line["clocks"]["samples"] = rows_summary["samples"]
    line["clocks"]["window"] = "0.5 s pre-roll of the same steps plus the timed region"

    if rank == 0 and not args.quick:
        # end to end through the public API: pinned host inputs -> HBM, fwd,
        # bwd, results -> pinned host, every step
        del buf
        torch.cuda.empty_cache()
        line["e2e"] = e2e_pipelined(inp, min(args.steps, 20), world, dev)
        configs = other_workloads(flush, peak, peak_kind, dev, args.config)
    else:
        configs = None

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg)
    if configs is not None:
        line["configs"] = configs  # last, so that a kept tail of the line holds it
    if rank == 0:
        print(json.dumps(line), flush=True)
        if args.extras:
            print(json.dumps({"extras": extra_workloads(flush, peak, dev)}), file=sys.stderr,
                  flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def cpu_baseline(cfg, target_s: float = 10.0):
    """The float64 oracle, as it stands, on the host cores, over a bounded
    sample of the workload (whole batch rows, about a second a repetition),
    repeated for about `target_s` seconds; and on one thread."""
    from paper_2406_12580_gb300 import inputs as I
    rows = 1 if cfg.L * cfg.D > (1 << 20) else cfg.B
    sample = I.make_scan_inputs(I.scaled(cfg, B=rows))
    rate, threads, reps, secs = cpu_oracle_rate(sample, target_s=target_s)
    if rows < cfg.B:  # grow the sample towards about a second a repetition
        per = secs / reps
        rows2 = int(max(1, min(cfg.B, rows / max(per, 1e-9))))
        if rows2 > rows:
            sample = I.make_scan_inputs(I.scaled(cfg, B=rows2))
            rate, threads, reps, secs = cpu_oracle_rate(sample, target_s=target_s)
    rate1, _, reps1, secs1 = cpu_oracle_rate(sample, target_s=3.0, threads=1)
    return {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{reps} x fwd+bwd of {sample.cfg.B} of {cfg.B} batch rows "
                      f"({sample.cfg.elements} elements) in {secs:.1f} s, float64",
            "single_thread": {"value": rate1, "unit": UNIT, "cores": 1,
                              "sample": f"{reps1} x fwd+bwd in {secs1:.1f} s"}}


def e2e_pipelined(inp, reps, world, dev, nsets=3):
    """Same metric through the C ABI with host buffers, steps streamed: every
    step copies its inputs from pinned host memory and reads every output back.
    Three streams — host-to-device copies, the scan, device-to-host copies —
    and `nsets` device buffer sets in rotation, so that step k's outputs go
    back while step k+1 computes and step k+2's inputs arrive."""
    import torch
    from paper_2406_12580_gb300.device import ScanBuffers, to_device
    cfg = inp.cfg
    pin = lambda name: to_device(inp.io_array(name), cfg.io, "cpu", pin=False).pin_memory()  # noqa: E731
    hx, hgl, hdh = pin("x"), pin("gl"), pin("dh") if not cfg.fwd_only else None
    bufs = [ScanBuffers.from_inputs(inp, device=dev) for _ in range(nsets)]
    outs = [[b.h, b.h_last] + ([] if cfg.fwd_only else [b.dx, b.dgl, b.dlam]) for b in bufs]
    host_outs = [[torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs[0]]
                 for _ in range(nsets)]
    h2d = sum(t.numel() * t.element_size() for t in (hx, hgl, hdh) if t is not None)
    d2h = sum(t.numel() * t.element_size() for t in host_outs[0])
    s_in, s_run, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    freed = [None] * nsets  # set j's outputs copied back: its buffers are free again

    def step(k):
        j = k % nsets
        b = bufs[j]
        with torch.cuda.stream(s_in):
            if freed[j] is not None:
                s_in.wait_event(freed[j])
            b.x.copy_(hx, non_blocking=True)
            b.gl.copy_(hgl, non_blocking=True)
            if hdh is not None:
                b.dh.copy_(hdh, non_blocking=True)
            ready = torch.cuda.Event()
            ready.record(s_in)
        with torch.cuda.stream(s_run):
            s_run.wait_event(ready)
            b.fwd()
            if not cfg.fwd_only:
                b.bwd()
            computed = torch.cuda.Event()
            computed.record(s_run)
        with torch.cuda.stream(s_out):
            s_out.wait_event(computed)
            for d, o in zip(host_outs[j], outs[j]):
                d.copy_(o, non_blocking=True)
            freed[j] = torch.cuda.Event()
            freed[j].record(s_out)

    for k in range(nsets + 1):
        step(k)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    s_run.wait_event(e0)
    s_out.wait_event(e0)
    for k in range(reps):
        step(k)
    e1.record(s_out)  # after the last step's copies back, which follow all of its work
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    return {"value": world * cfg.elements / (ms * 1e-3), "unit": UNIT, "ms_per_step": ms,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "pipelining": (f"three streams (copies in, scan, copies out) and {nsets} device buffer "
                           "sets: step k's copies back overlap step k+1's scan and step k+2's "
                           "copies in")}


def other_workloads(flush, peak, peak_kind, dev, headline):
    """The other workloads (parity-test shapes beside the headline), each with
    per-call rooflines; L2 flushed before every call; the recurrent step; and
    one training step of the gated recurrent layer (tokens/s)."""
    import torch
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import ScanBuffers, StepBuffers
    out = {}
    for k in (0, 1, 2, 3, 4):
        if k == headline:
            continue
        cfg = I.CONFIGS[k]
        inp = I.make_scan_inputs(cfg)
        buf = ScanBuffers.from_inputs(inp, device=dev)
        time_calls(buf, 3, flush, with_bwd=not cfg.fwd_only)
        f, b, _ = time_calls(buf, 30, flush, with_bwd=not cfg.fwd_only)
        out[f"config{k}"] = compact(workload_rooflines(cfg, f, b, peak, peak_kind, f"config{k}"))
        del buf, inp
        torch.cuda.empty_cache()
    for io in ("f32", "bf16"):
        scfg = I.StepConfig(f"recurrent step B=65536 D=64 {io}", 65536, 64, io, seed=4)
        sbuf = StepBuffers.from_inputs(I.make_step_inputs(scfg), device=dev)
        time_step_kernel(sbuf, 3, flush)
        ms = sum(time_step_kernel(sbuf, 30, flush)) / 30
        r = call_roofline("step_kernel", scfg.elements * step_bytes_per_elem(io), ms, peak,
                          peak_kind, None)
        out[f"step_{io}"] = {"us": round(r["us"], 2), "frac": round(r["frac"], 3)}
        del sbuf
    g = step_graph(flush, peak, dev)
    out["step_f32_graph8"] = {"us": round(g["ms_per_step"] * 1e3, 2), "frac": round(g["frac"], 3)}
    t = layer_workload(flush, dev, serial=False)
    out["layer_train_step"] = {"ms": round(t["ms_fused_kernels"], 3),
                               "tokens_per_s": round(t["tokens_per_s"])}
    return out


def compact(rl):
    """A workload's rooflines, short enough for the end of the JSON line: per
    call the mean event-timed microseconds, fraction of the measured copy
    bandwidth and ncu DRAM bytes per launch (null if not captured on these
    kernel sources); and the fwd+bwd fraction."""
    out = {}
    for k in ("fwd", "bwd"):
        if k in rl:
            out[k] = {"kernel": rl[k]["kernel"], "us": round(rl[k]["us"], 2),
                      "frac": round(rl[k]["frac"], 3), "traffic": rl[k]["traffic"]}
    if "fwd_bwd_frac" in rl:
        out["frac"] = round(rl["fwd_bwd_frac"], 3)
    return out


def extra_workloads(flush, peak, dev):
    """Workloads beyond the scope table's configurations (--extras)."""
    out = {}
    for io in ("f32", "bf16"):
        out[f"steps_k8_{io}"] = steps_workload(io, flush, peak, dev)
    for k in (1, 2):
        out[f"gated_config{k}"] = gated_workload(k, flush, peak, dev)
    out["gated_layer_train_step"] = layer_workload(flush, dev)
    out["varlen_config2"] = varlen_workload(flush, peak, dev)
    out["padding_table"] = padding_table(flush, dev)
    return out


def steps_workload(io, flush, peak, dev, B=65536, K=8, D=64, reps=20):
    """K = 8 recurrent steps per row in one call (blr_steps), state and I/O in
    the same dtype, per-step states not written: compulsory bytes per (row,
    channel) are the state in and out plus K x (x, rho, iota)."""
    import torch
    from paper_2406_12580_gb300 import blr_steps
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import io_code, to_device, torch_io_dtype
    cfg = I.ScanConfig(f"{K} recurrent steps B={B} D={D} {io}", B, K, D, io, seed=6,
                       fwd_only=True, random_h0=True)
    inp = I.make_scan_inputs(cfg)
    x, gl = to_device(inp.io_array("x"), io, dev), to_device(inp.io_array("gl"), io, dev)
    lam = to_device(inp.lam, "f32", dev)
    h = torch.from_numpy(inp.h0).to(dev).to(torch_io_dtype(io))
    code = io_code(io)
    for _ in range(3):
        blr_steps(B, K, D, code, code, 1.0, h, x, gl, lam, h)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(reps)]
    for e0, e1 in ev:
        flush()
        e0.record()
        blr_steps(B, K, D, code, code, 1.0, h, x, gl, lam, h)
        e1.record()
    torch.cuda.synchronize()
    ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    ib = io_bytes(io)
    gbs = B * D * (2 + 3 * K) * ib / (ms * 1e-3) / 1e9
    return {"workload": cfg.name + " in one call", "ms": ms,
            "steps_per_s": B * D * K / (ms * 1e-3), "gbs": gbs, "frac": gbs / peak}


def _time_fwd_bwd(fwd, bwd, flush, reps):
    import torch
    for _ in range(3):
        fwd(); bwd()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(reps)]
    for e in ev:
        flush()
        e[0].record(); fwd(); e[1].record(); bwd(); e[2].record()
    torch.cuda.synchronize()
    return (statistics.median(a.elapsed_time(b) for a, b, c in ev),
            statistics.median(b.elapsed_time(c) for a, b, c in ev))


def varlen_workload(flush, peak, dev, reps=20):
    """The train-shaped workload (20 % of every row left padding) given as rows
    of their own length, 40 of 50 steps (blr_scan_*_varlen: the padding is not
    read), against the padded scan over all 50."""
    import torch
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = I.CONFIGS[2]
    buf = ScanBuffers.from_inputs(I.make_scan_inputs(cfg), device=dev)
    lengths = torch.full((cfg.B,), cfg.L - cfg.pad_rows, dtype=torch.int32, device=dev)
    fp, bp = _time_fwd_bwd(buf.fwd, buf.bwd, flush, reps)
    fv, bv = _time_fwd_bwd(lambda: buf.fwd_varlen(lengths), lambda: buf.bwd_varlen(lengths),
                           flush, reps)
    n_real = cfg.B * (cfg.L - cfg.pad_rows) * cfg.D
    gbs = n_real * 22 * io_bytes(cfg.io) / 2 / ((fv + bv) * 1e-3) / 1e9
    return {"workload": cfg.name + f", as rows of {cfg.L - cfg.pad_rows} steps",
            "padded": {"fwd_ms": fp, "bwd_ms": bp}, "varlen": {"fwd_ms": fv, "bwd_ms": bv},
            "speedup": (fp + bp) / (fv + bv), "varlen_gbs": gbs, "varlen_frac": gbs / peak}


def padding_table(flush, dev, B=256, D=64, reps=20):
    """The shape of the paper's padding comparison (Sec. 4, lengths 200, 100,
    257): fwd + bwd of the sequence length itself (this scan needs no padding)
    against the same scan over the next power of two, the length a two-tree
    scan needs."""
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import ScanBuffers
    rows = {}
    for L in (200, 100, 257):
        L2 = 1 << (L - 1).bit_length()
        t = {}
        for n in (L, L2):
            cfg = I.ScanConfig(f"fwd+bwd B={B} L={n} D={D} fp32", B, n, D, "f32", seed=5)
            buf = ScanBuffers.from_inputs(I.make_scan_inputs(cfg), device=dev)
            f, b = _time_fwd_bwd(buf.fwd, buf.bwd, flush, reps)
            t[n] = f + b
            del buf
        rows[f"L={L}"] = {"ms": t[L], f"ms_at_L={L2}": t[L2], "padded_over_exact": t[L2] / t[L]}
    return {"workload": f"fwd+bwd B={B} D={D} fp32 at L and at the next power of two",
            "rows": rows}


def layer_workload(flush, dev, B=256, L=200, D=64, E=2, reps=10, serial=True):
    """One training step (forward, backward and an Adam update, lr 1e-3) of the
    gated recurrent layer of Alg. 1 (layer.GatedRecurrentLayer: torch GEMMs and
    convolution, the scan and merge on the library's kernels), and (serial)
    the same step with the scan as a step-by-step torch loop on the GPU."""
    import torch
    from paper_2406_12580_gb300.layer import GatedRecurrentLayer
    torch.manual_seed(0)
    layer = GatedRecurrentLayer(D, expand=E, device=dev)
    opt = torch.optim.Adam(layer.parameters(), lr=1e-3)
    h = torch.randn(B, L, D, device=dev, requires_grad=True)
    g = torch.randn(B, L, D, device=dev)

    def train_step(fwd):
        opt.zero_grad(set_to_none=False)
        (fwd(h) * g).sum().backward()
        opt.step()

    def serial_forward(x_in):
        hx, hz = layer.in_proj(x_in).split(layer.ed, dim=-1)
        xc = layer.conv(hx.transpose(1, 2))[..., :L].transpose(1, 2)
        x = torch.nn.functional.silu(xc)
        rho, iota = layer.gate_proj(x).split(layer.ed, dim=-1)
        alpha = torch.exp(-torch.nn.functional.softplus(layer.lam) * torch.sigmoid(rho))
        beta = torch.sqrt(1.0 - alpha * alpha) * torch.sigmoid(iota)
        state = torch.zeros(B, layer.ed, device=dev)
        hs = []
        for t in range(L):
            state = alpha[:, t] * state + beta[:, t] * x[:, t]
            hs.append(state)
        return layer.out_proj(torch.stack(hs, dim=1) * torch.nn.functional.silu(hz))

    res = {}
    variants = (("fused_kernels", layer), ("serial_torch_scan", serial_forward))
    for name, fwd in variants if serial else variants[:1]:
        n = reps if name == "fused_kernels" else max(2, reps // 5)
        for _ in range(2):
            train_step(fwd)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(n)]
        for e0, e1 in ev:
            flush()
            e0.record()
            train_step(fwd)
            e1.record()
        torch.cuda.synchronize()
        res[name] = statistics.median(a.elapsed_time(b) for a, b in ev)
    out = {"workload": f"gated recurrent layer (Alg. 1) d_model={D} E={E} B={B} L={L} f32, "
                       "forward + backward + Adam", "ms_fused_kernels": res["fused_kernels"],
           "tokens_per_s": B * L / (res["fused_kernels"] * 1e-3)}
    if serial:
        out.update(ms_serial_torch_scan=res["serial_torch_scan"],
                   serial_over_fused=res["serial_torch_scan"] / res["fused_kernels"])
    return out


def gated_workload(k, flush, peak, dev, reps=20):
    """Workload k with the gated layer's merge y = h SiLU(z) (Alg. 1): the fused
    entry points against the plain scan followed by the merge as separate torch
    elementwise operations (what a caller without the fused call would run)."""
    import torch
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import ScanBuffers
    cfg = I.scaled(I.CONFIGS[k], gated=True)
    buf = ScanBuffers.from_inputs(I.make_scan_inputs(cfg), device=dev)
    z, dy = buf.z, buf.dh
    dh = torch.empty_like(dy)

    def fused():
        buf.fwd_gated()
        e = torch.cuda.Event(enable_timing=True)
        e.record()
        buf.bwd_gated()
        return e

    def unfused():
        buf.fwd()
        y = buf.h * torch.nn.functional.silu(z)
        e = torch.cuda.Event(enable_timing=True)
        e.record()
        sg = torch.sigmoid(z)
        torch.mul(dy, z * sg, out=dh)
        dz = dy * buf.h * (sg * (1 + z * (1 - sg)))
        blr_scan_bwd_buf(buf, dh)
        return e, y, dz

    def blr_scan_bwd_buf(b, dh_):
        from paper_2406_12580_gb300 import blr_scan_bwd
        blr_scan_bwd(b.desc, dh_, b.dh_last, b.x, b.gl, b.lam, b.h0, b.dx, b.dgl, b.dlam, b.dh0,
                     b.ws)

    res = {}
    for name, fn in (("fused", fused), ("unfused", unfused)):
        for _ in range(3):
            fn()
        ev = []
        for _ in range(reps):
            flush()
            e0, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            r = fn()
            e2.record()
            ev.append((e0, r[0] if isinstance(r, tuple) else r, e2))
        torch.cuda.synchronize()
        f = statistics.median(a.elapsed_time(b) for a, b, c in ev)
        b = statistics.median(b.elapsed_time(c) for a, b, c in ev)
        res[name] = {"fwd_ms": f, "bwd_ms": b}
    n, ib = cfg.elements, io_bytes(cfg.io)
    fu = res["fused"]
    # compulsory bytes of the fused calls: fwd x, rho, iota, z in, y out (5 values);
    # bwd dy, x, rho, iota, z in, dx, drho, diota, dz out (9 values)
    gbs = n * 14 * ib / ((fu["fwd_ms"] + fu["bwd_ms"]) * 1e-3) / 1e9
    return {"workload": cfg.name + ", gated (y = h SiLU(z))", "fused": res["fused"],
            "unfused_scan_then_torch_merge": res["unfused"],
            "fused_elements_per_s": n / ((fu["fwd_ms"] + fu["bwd_ms"]) * 1e-3),
            "fused_speedup": (res["unfused"]["fwd_ms"] + res["unfused"]["bwd_ms"]) /
                             (fu["fwd_ms"] + fu["bwd_ms"]),
            "fused_gbs": gbs, "fused_frac": gbs / peak}


def step_graph(flush, peak, dev, n_tok=8, reps=20):
    """Recurrent serving: n_tok consecutive steps h <- step(h, x_k, gate_logits_k)
    with distinct inputs per step (n_tok x 84 MB, more than L2), launched back to
    back from one CUDA graph; L2 flushed before each replay."""
    import torch
    from paper_2406_12580_gb300 import inputs as I
    from paper_2406_12580_gb300.device import StepBuffers
    bufs = [StepBuffers.from_inputs(I.make_step_inputs(
        I.StepConfig(f"recurrent step B=65536 D=64 f32 token {k}", 65536, 64, "f32", seed=100 + k)),
        device=dev) for k in range(n_tok)]
    h = [bufs[0].h_prev, torch.empty_like(bufs[0].h_prev)]

    def run():
        for k, b in enumerate(bufs):
            b.h_prev, b.h_t = h[k % 2], h[(k + 1) % 2]
            b.step()

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run()  # warm-up outside capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        run()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(reps)]
    for e0, e1 in ev:
        flush()
        e0.record()
        g.replay()
        e1.record()
    torch.cuda.synchronize()
    ms = statistics.median(a.elapsed_time(b) for a, b in ev[3:]) / n_tok
    el = bufs[0].B * bufs[0].D
    gbs = el * step_bytes_per_elem("f32") / (ms * 1e-3) / 1e9
    return {"workload": f"{n_tok} recurrent steps B=65536 D=64 f32 in one CUDA graph",
            "ms_per_step": ms, "elements_per_s": el / (ms * 1e-3), "gbs": gbs, "frac": gbs / peak}


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
