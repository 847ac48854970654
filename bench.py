#!/usr/bin/env python
"""Benchmark of the OSD hot path: speculative-sampling verification and the
distillation loss/gradient, at vocabulary 32000 (bf16 logits).

One step is one pass of the whole hot path over synthetic inputs:
  verify   B=32 sequences, k=5 draft tokens, V=32000, T=1.0, then the greedy
           (T=0) pass over the same logits            -> 2 x 160 verified positions
  distill  reverse KL on the rows the T=1 pass rejected, picked on the device
           from its accepted counts                   -> one row per rejecting sequence
  distill  a buffer flush of N=65536 positions x V=32000, reverse KL then TVD,
           loss and d loss / d draft logits           -> 2 x 65536 distilled positions
The value is positions (verified + distilled) per second for the whole job.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload serving-32k|large-vocab]

With --gpus N > 1 and no torchrun environment, the script starts N ranks
itself (torch.distributed.run on 127.0.0.1), one per GPU; each rank draws its
own shard of the workload (weak scaling, no collective on the data path) and
the job time is the slowest rank's.

`--workload large-vocab` times verify at B=256, k=8, V=128256, T=0.7 followed
by forward-KL distill of its rejected rows (the 128k-vocabulary serving step).
`--impl reference` times the CPU oracle (the correctness reference) on a
bounded sample of the same workload, on the host cores.
Prints one JSON line (rank 0).
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "verified positions/s and distilled positions/s at V=32000; % of HBM peak"
SLEEP_CYCLES = 2_000_000  # ~1 ms of device time ahead of each timed step: covers the host-side
                          # enqueue of the whole step, so no host gap lands inside the events
FALLBACK_HBM_GBS = 6800.0


def _peak_hbm():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def _source_hash(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


DISTILL_SOURCES = ["paper_2310_07177_gb300/csrc/osd_distill.cu", "paper_2310_07177_gb300/csrc/osd_device.cuh",
                   "paper_2310_07177_gb300/csrc/osd_rowspan.cuh"]
VERIFY_SOURCES = ["paper_2310_07177_gb300/csrc/osd_verify.cu", "paper_2310_07177_gb300/csrc/osd_device.cuh",
                  "paper_2310_07177_gb300/csrc/osd_rowstats.cuh"]


def _traffic(kernel: str, files):
    """DRAM bytes per launch from the committed ncu summary, if it still matches the source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)[kernel]
    except Exception:
        return None
    if rec.get("source_sha") != _source_hash(files):
        return None
    return rec.get("dram_bytes_per_launch")


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.lines = []
        self.first = 0

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def wait_lines(self, n: int, timeout_s: float) -> None:
        """Wait (bounded) until at least n sample lines have arrived."""
        t_end = time.perf_counter() + timeout_s
        while self.proc is not None and len(self.lines) < n and time.perf_counter() < t_end:
            time.sleep(0.002)

    def start_region(self) -> None:
        """Mark the start of the timed region once the sampler is running: keep
        the sample just before it, so that a region shorter than the sampling
        period still has the clocks on both sides of it."""
        self.wait_lines(1, 3.0)
        self.first = max(0, len(self.lines) - 1)

    def end_region(self) -> None:
        self.wait_lines(len(self.lines) + 1, 1.0)  # and the sample just after it

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines[self.first:]:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for name, val in zip(names, parts[3:7]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- ranks
def job_time_ms(local_ms: float, device=None) -> float:
    """Whole-job time: the slowest rank's timed total (max over ranks; the
    identity when torch.distributed is not initialised)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(local_ms)
    t = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(positions_per_rank: int, world: int, ms_per_step: float) -> float:
    """Positions per second over all ranks: every rank processes its own shard
    of the same size in the time of the slowest one (weak scaling)."""
    return world * positions_per_rank / (ms_per_step / 1e3)


# ----------------------------------------------------------------------------- workloads
def shard_seed(base_seed: int, rank: int) -> int:
    """Each rank draws its own shard of sequences / rows (weak scaling, no overlap)."""
    return base_seed + 7919 * rank


def _setup_serving_32k(dev, distill_rows=None, rank=0):
    import dataclasses

    from paper_2310_07177_gb300 import workloads as W
    spec_v, spec_d = W.VERIFY[2], W.DISTILL[4]
    if distill_rows:
        spec_d = dataclasses.replace(spec_d, N=distill_rows)
    v = W.verify_inputs(spec_v, seed=shard_seed(W.seed_for(2), rank), device=dev)
    d = W.distill_inputs(spec_d, seed=shard_seed(W.seed_for(4), rank), device=dev)
    return {"v": v, "d": d, "spec_v": spec_v, "spec_d": spec_d,
            "desc": "serving-32k: verify B=32 k=5 V=32000 bf16 T=1.0 -> reverse-KL distill of its "
                    "rejected rows (selected on the device) + greedy T=0 pass; "
                    f"distill flush N={spec_d.N} V=32000 bf16 reverse-KL + TVD"}


def _setup_large_vocab(dev, rank=0):
    from paper_2310_07177_gb300 import workloads as W
    v = W.verify_inputs(W.VERIFY[5], seed=shard_seed(W.seed_for(5), rank), device=dev)
    return {"v": v, "spec_v": W.VERIFY[5],
            "desc": "large-vocab: verify B=256 k=8 V=128256 bf16 T=0.7 -> forward-KL distill of "
                    "its rejected rows (selected and compacted on the device)"}


def _bytes_verify(B, k, V, s_in, greedy):
    return (B * (k + 1) * V * s_in) if greedy else ((B * k + B * (k + 1)) * V * s_in)


# ----------------------------------------------------------------------------- our arm
def run_ours(args):
    import torch
    import paper_2310_07177_gb300 as osd

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    osd.build_library()
    osd.load_library()

    wl = args.workload
    setup = (_setup_serving_32k(dev, args.distill_rows, rank) if wl == "serving-32k"
             else _setup_large_vocab(dev, rank))
    stream = torch.cuda.current_stream(dev)
    v = setup["v"]
    sv = setup["spec_v"]
    s_in = 2 if sv.dtype == torch.bfloat16 else 4
    ws = torch.empty(osd.osd_verify_workspace_size(sv.B, sv.k, sv.V), dtype=torch.uint8, device=dev)
    vout = osd.osd_verify(v["draft"], v["target"], v["tokens"], v["uniforms"], sv.temperature, workspace=ws)
    vout0 = osd.osd_verify(v["draft"], v["target"], v["greedy_tokens"], v["uniforms"], 0.0, workspace=ws)
    l2_flush = torch.empty(2 * 128 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    if wl == "serving-32k":
        d = setup["d"]
        sd = setup["spec_d"]
        dl = torch.empty(sd.N, sd.V, dtype=torch.float32, device=dev)
        loss = torch.empty(sd.N, dtype=torch.float32, device=dev)
        kinds = args.distill_kinds.split(",")
        if kinds != ["rkl", "tvd"]:
            setup["desc"] = setup["desc"].replace("reverse-KL + TVD", " + ".join(k.upper() for k in kinds))
        dist_pos = len(kinds) * sd.N
        dist_bytes = sd.N * sd.V * (2 * 2 + 4)  # per launch
    else:
        kinds = []

    rej_kind = "rkl" if wl == "serving-32k" else "fkl"
    rej = osd.osd_distill_accepted(v["draft"], v["target"], vout.accepted, rej_kind)
    torch.cuda.synchronize()
    n_rej = int(rej.count.item())  # the inputs are the same every step, so is the count
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    n_ver = 2 if wl == "serving-32k" else 1

    def step(record):
        e = [ev() for _ in range(2 + n_ver + (len(kinds) if wl == "serving-32k" else 0))]
        l2_flush.zero_()
        # keep the device busy while the host enqueues the step, so that host-side
        # launch overhead never shows up inside the timed events
        torch.cuda._sleep(SLEEP_CYCLES)
        e[0].record(stream)
        osd.osd_verify(v["draft"], v["target"], v["tokens"], v["uniforms"], sv.temperature,
                       workspace=ws, out=vout)
        e[1].record(stream)
        # the rows this pass rejected, straight from its accepted counts
        osd.osd_distill_accepted(v["draft"], v["target"], vout.accepted, rej_kind, 0.5, out=rej)
        e[2].record(stream)
        if wl == "serving-32k":
            osd.osd_verify(None, v["target"], v["greedy_tokens"], None, 0.0, workspace=ws, out=vout0)
            e[3].record(stream)
            for i, kind in enumerate(kinds):
                osd.osd_distill(d["draft"], d["target"], d["mask"], kind, 0.5, loss=loss, dlogits=dl)
                e[4 + i].record(stream)
        record.append(e)

    warm = []
    for _ in range(args.warmup):
        step(warm)
    torch.cuda.synchronize()

    props = torch.cuda.get_device_properties(dev)
    gpu_id = str(getattr(props, "uuid", local))
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) == 36:
        gpu_id = "GPU-" + gpu_id
    recs = []
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(gpu_id) as clk:
        clk.start_region()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            step(recs)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        clk.end_region()
    if world > 1:
        torch.distributed.barrier()

    step_ms = [r[0].elapsed_time(r[-1]) for r in recs]
    verify_ms = [r[0].elapsed_time(r[1]) for r in recs]
    rej_ms = [r[1].elapsed_time(r[2]) for r in recs]
    if wl == "serving-32k":
        greedy_ms = [r[2].elapsed_time(r[3]) for r in recs]
        dist_ms = [r[3 + i].elapsed_time(r[4 + i]) for r in recs for i in range(len(kinds))]
    total_ms = job_time_ms(sum(step_ms), dev if world > 1 else None)
    ms_step = total_ms / args.steps

    bytes_rej = n_rej * sv.V * (2 * s_in + 4) + sv.B * 4  # the rejected rows, plus the counts
    if wl == "serving-32k":
        ver_pos = 2 * sv.B * sv.k
        positions = ver_pos + dist_pos + n_rej
        launches = 2 * 2 + 1 + len(kinds)
        bytes_v = _bytes_verify(sv.B, sv.k, sv.V, s_in, False)
        bytes_g = _bytes_verify(sv.B, sv.k, sv.V, s_in, True)
    else:
        ver_pos = sv.B * sv.k
        positions = ver_pos + n_rej
        launches = 2 + 1
        bytes_v = _bytes_verify(sv.B, sv.k, sv.V, s_in, False)
    value = job_throughput(positions, world, ms_step)
    peak, peak_src = _peak_hbm()
    avg_ver = statistics.mean(verify_ms)
    avg_rej = statistics.mean(rej_ms)
    kernels = {
        "verify": {"us_per_call": avg_ver * 1e3, "alg_bytes": bytes_v,
                   "gbs": bytes_v / (avg_ver / 1e3) / 1e9,
                   "positions_per_s": sv.B * sv.k / (avg_ver / 1e3)},
        "distill_rejected": {"us_per_call": avg_rej * 1e3, "alg_bytes": bytes_rej, "rows": n_rej,
                             "gbs": bytes_rej / (avg_rej / 1e3) / 1e9,
                             "positions_per_s": n_rej / (avg_rej / 1e3)},
    }
    if wl == "serving-32k":
        avg_dist = statistics.mean(dist_ms)
        kernels["distill"] = {"us_per_call": avg_dist * 1e3, "alg_bytes": dist_bytes,
                              "gbs": dist_bytes / (avg_dist / 1e3) / 1e9,
                              "positions_per_s": sd.N / (avg_dist / 1e3)}
        avg_g = statistics.mean(greedy_ms)
        kernels["verify_greedy"] = {"us_per_call": avg_g * 1e3, "alg_bytes": bytes_g,
                                    "gbs": bytes_g / (avg_g / 1e3) / 1e9,
                                    "positions_per_s": sv.B * sv.k / (avg_g / 1e3)}
    if wl == "serving-32k" and not args.no_extras and rank == 0:
        reps = max(3, args.steps // 2)
        kernels["mixed_sample"] = _time_mixed_sample(osd, d, sd, l2_flush, stream, reps=reps)
        kernels["tree_verify"] = _time_tree_verify(osd, dev, l2_flush, stream, reps=reps)
        kernels.update(_time_large_vocab(osd, dev, l2_flush, stream, reps=max(5, args.steps)))
        kernels["distill_jsd_masked"] = _time_jsd_flush(osd, dev, l2_flush, stream, reps=max(5, args.steps))
    for kv in kernels.values():
        kv["frac_of_peak"] = kv["gbs"] / peak
    # the dominant kernel: distill on the default step, verify's row statistics at 128k
    top = "distill" if wl == "serving-32k" else "verify"
    achieved = kernels[top]["gbs"]
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4),
                # the distill counters were taken on the RKL and TVD launches of the default step
                "traffic": ((_traffic("distill", DISTILL_SOURCES) if kinds == ["rkl", "tvd"] else None)
                            if top == "distill" else _traffic("verify", VERIFY_SOURCES)),
                "kernel": (" + ".join(("distill_tm_kernel " if k in ("rkl", "tvd", "jsd") else "distill_kernel ")
                                      + k.upper() for k in kinds) if top == "distill"
                           else "row_stats_kernel + verify_finalize_kernel"),
                "peak_source": peak_src}

    e2e = None
    if not args.no_e2e:  # every rank runs it (h2d and d2h are per rank), timed over the job
        e2e = run_e2e(args, osd, setup, dev, stream, positions, wl)
    cpu = cpu_baseline(args, setup) if (rank == 0 and world == 1 and not args.no_cpu_baseline) else None

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "positions/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded random logits shaped like 32k/128k-vocabulary LLM outputs; no model weights)",
            "config": {"workload": setup["desc"], "l2": "flushed (256 MiB write) before every step",
                       "parallelism": f"replicas x{world} (rows sharded, no collective)"},
            "roofline": roofline,
            "kernels": {k2: {kk: (round(vv, 3) if isinstance(vv, float) else vv) for kk, vv in kv.items()}
                        for k2, kv in kernels.items()},
            "clocks": clk.summary(),
            "gpu_launches": launches * args.steps,
            "wall_s_timed": round(wall, 3),
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def _time_mixed_sample(osd, d, sd, l2_flush, stream, reps):
    """Mixed sampling (y ~ beta p + (1 - beta) q) over the distill workload's rows,
    timed on its own after the step loop (it is not part of the serving step)."""
    import torch
    g = torch.Generator(device=d["draft"].device)
    g.manual_seed(2310071779)
    u = torch.rand(sd.N, generator=g, device=d["draft"].device)
    tok = torch.empty(sd.N, dtype=torch.int32, device=d["draft"].device)
    for _ in range(2):
        osd.osd_mixed_sample(d["draft"], d["target"], u, 0.5, tokens=tok)
    ms = []
    for _ in range(reps):
        l2_flush.zero_()
        torch.cuda._sleep(SLEEP_CYCLES)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        osd.osd_mixed_sample(d["draft"], d["target"], u, 0.5, tokens=tok)
        b.record(stream)
        b.synchronize()
        ms.append(a.elapsed_time(b))
    avg = statistics.mean(ms)
    alg = sd.N * sd.V * 2 * 2 + sd.N * 8  # both bf16 rows, the uniform and the token
    return {"us_per_call": avg * 1e3, "alg_bytes": alg, "gbs": alg / (avg / 1e3) / 1e9,
            "positions_per_s": sd.N / (avg / 1e3), "in_step": False, "beta": 0.5}


def _timed(fn, l2_flush, stream, reps, warm=2):
    """Mean CUDA-event time (ms) of fn() on `stream`, L2 flushed and the device
    kept busy (so that host enqueue time stays outside the events) before each."""
    import torch
    ms = []
    for i in range(reps + warm):
        l2_flush.zero_()
        torch.cuda._sleep(SLEEP_CYCLES)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        b.synchronize()
        if i >= warm:
            ms.append(a.elapsed_time(b))
    return statistics.mean(ms)


def _time_large_vocab(osd, dev, l2_flush, stream, reps):
    """The 128k-vocabulary serving step's two calls, each timed on its own with L2
    flushed before it: verify at B=256, k=8, V=128256 bf16, T=0.7 (the largest
    verify workload), then the forward-KL distillation of the rows it rejected,
    selected and compacted on the device (osd_distill_accepted)."""
    import torch
    from paper_2310_07177_gb300 import workloads as W
    sv = W.VERIFY[5]
    v = W.verify_inputs(sv, seed=W.seed_for(5), device=dev)
    ws = torch.empty(osd.osd_verify_workspace_size(sv.B, sv.k, sv.V), dtype=torch.uint8, device=dev)
    out = osd.osd_verify(v["draft"], v["target"], v["tokens"], v["uniforms"], sv.temperature, workspace=ws)
    rej = osd.osd_distill_accepted(v["draft"], v["target"], out.accepted, "fkl", 0.5)
    torch.cuda.synchronize()
    n_rej = int(rej.count.item())
    t_v = _timed(lambda: osd.osd_verify(v["draft"], v["target"], v["tokens"], v["uniforms"], sv.temperature,
                                        workspace=ws, out=out), l2_flush, stream, reps)
    t_d = _timed(lambda: osd.osd_distill_accepted(v["draft"], v["target"], out.accepted, "fkl", 0.5, out=rej),
                 l2_flush, stream, reps)
    bv = _bytes_verify(sv.B, sv.k, sv.V, 2, False)
    bd = n_rej * sv.V * (2 * 2 + 4) + sv.B * 4
    res = {
        "verify_large_vocab": {"us_per_call": t_v * 1e3, "alg_bytes": bv, "gbs": bv / (t_v / 1e3) / 1e9,
                               "positions_per_s": sv.B * sv.k / (t_v / 1e3), "in_step": False,
                               "workload": "B=256 k=8 V=128256 bf16 T=0.7"},
        "distill_rejected_large_vocab": {"us_per_call": t_d * 1e3, "alg_bytes": bd, "rows": n_rej,
                                         "gbs": bd / (t_d / 1e3) / 1e9, "positions_per_s": n_rej / (t_d / 1e3),
                                         "in_step": False, "kind": "fkl",
                                         "workload": "the rows the verify above rejected, V=128256 bf16"},
    }
    del v, ws, out, rej
    return res


def _time_jsd_flush(osd, dev, l2_flush, stream, reps):
    """The 16384 x 32128 buffer flush: generalised JSD (beta = 1/2) loss and
    gradient under its 40 % mask, timed on its own with L2 flushed before it."""
    import torch
    from paper_2310_07177_gb300 import workloads as W
    spec = W.DISTILL[3]
    inp = W.distill_inputs(spec, seed=W.seed_for(3), device=dev)
    loss = torch.empty(spec.N, dtype=torch.float32, device=dev)
    dl = torch.empty(spec.N, spec.V, dtype=torch.float32, device=dev)
    n_on = int(inp["mask"].sum().item())
    t = _timed(lambda: osd.osd_distill(inp["draft"], inp["target"], inp["mask"], "jsd", 0.5, loss=loss,
                                       dlogits=dl), l2_flush, stream, reps)
    alg = n_on * spec.V * (2 * 2 + 4)
    del inp, loss, dl
    return {"us_per_call": t * 1e3, "alg_bytes": alg, "rows": n_on, "gbs": alg / (t / 1e3) / 1e9,
            "positions_per_s": n_on / (t / 1e3), "in_step": False,
            "workload": f"N={spec.N} V={spec.V} bf16, {n_on} rows active (40 % mask), JSD beta=0.5"}


def _time_tree_verify(osd, dev, l2_flush, stream, reps):
    """Token-tree verification of B=32 sequences over the 27-node Medusa-style
    tree at V=32000 bf16, T=1, timed on its own after the step loop."""
    import torch
    from paper_2310_07177_gb300 import workloads as W
    par = W.MEDUSA_TREE
    B, V = 32, 32000
    inp = W.tree_inputs(B, par, V, torch.bfloat16, 1.0, seed=2310071778, device=dev, target_noise=0.8)
    n = len(par)
    ws = torch.empty(osd.osd_verify_tree_workspace_size(B, n, V), dtype=torch.uint8, device=dev)
    res = osd.osd_verify_tree(inp["draft"], inp["target"], par, inp["tokens"], inp["uniforms"], 1.0, workspace=ws)
    ms = []
    for i in range(reps + 2):
        l2_flush.zero_()
        torch.cuda._sleep(SLEEP_CYCLES)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        osd.osd_verify_tree(inp["draft"], inp["target"], par, inp["tokens"], inp["uniforms"], 1.0,
                            workspace=ws, out=res)
        b.record(stream)
        b.synchronize()
        if i >= 2:
            ms.append(a.elapsed_time(b))
    avg = statistics.mean(ms)
    alg = 2 * B * n * V * 2  # every node's draft and target row, read once by the statistics pass
    acc = res.accepted.float().mean().item()
    return {"us_per_call": avg * 1e3, "alg_bytes": alg, "gbs": alg / (avg / 1e3) / 1e9,
            "positions_per_s": B * (acc + 1) / (avg / 1e3), "mean_accepted": round(acc, 3),
            "nodes": n, "in_step": False}


def run_e2e(args, osd, setup, dev, stream, positions, wl):
    """Same step through the public API from pinned host buffers: every step's
    inputs are copied host->device and its results read device->host inside
    the timed region.  As a server would, the step pipelines: the upload of
    step i+1's inputs (into the second of two device buffer sets, on a copy
    stream) runs while step i's kernels run."""
    import torch
    v = setup["v"]
    sv = setup["spec_v"]
    nbuf = 2
    host = {k: v[k].cpu().pin_memory() for k in ("draft", "target", "tokens", "greedy_tokens", "uniforms")}
    dv = [{k: torch.empty_like(v[k]) for k in host} for _ in range(nbuf)]
    h_out = {"acc": torch.empty(sv.B, dtype=torch.int32).pin_memory(),
             "tok": torch.empty(sv.B, sv.k + 1, dtype=torch.int32).pin_memory(),
             "mask": torch.empty(sv.B, sv.k, dtype=torch.uint8).pin_memory()}
    ws = torch.empty(osd.osd_verify_workspace_size(sv.B, sv.k, sv.V), dtype=torch.uint8, device=dev)
    h2d = sum(t.numel() * t.element_size() for k, t in host.items()
              if wl == "serving-32k" or k != "greedy_tokens")
    rej_kind = "rkl" if wl == "serving-32k" else "fkl"
    rej = osd.DistillAcceptedResult(torch.empty(sv.B, dtype=torch.float32, device=dev),
                                    torch.empty(sv.B, sv.V, dtype=torch.float32, device=dev),
                                    torch.empty(sv.B, dtype=torch.int32, device=dev),
                                    torch.empty(1, dtype=torch.int32, device=dev))
    h_rej = {"loss": torch.empty(sv.B, dtype=torch.float32).pin_memory(),
             "seq": torch.empty(sv.B, dtype=torch.int32).pin_memory(),
             "count": torch.empty(1, dtype=torch.int32).pin_memory()}
    d2h = (h_out["acc"].numel() * 4 + h_out["tok"].numel() * 4 + h_out["mask"].numel()
           + sum(t.numel() * 4 for t in h_rej.values()))
    hd, dd = {}, [{} for _ in range(nbuf)]
    if wl == "serving-32k":
        d = setup["d"]
        sd = setup["spec_d"]
        hd = {"draft": d["draft"].cpu().pin_memory(), "target": d["target"].cpu().pin_memory()}
        dd = [{k: torch.empty_like(d[k]) for k in hd} for _ in range(nbuf)]
        loss = torch.empty(sd.N, dtype=torch.float32, device=dev)
        dl = torch.empty(sd.N, sd.V, dtype=torch.float32, device=dev)
        h_loss = torch.empty(2, sd.N, dtype=torch.float32).pin_memory()
        # the greedy pass's results land in pinned buffers of their own, next to the T=1 pass's
        h_out0 = {key: torch.empty_like(val).pin_memory() for key, val in h_out.items()}
        h2d += sum(t.numel() * t.element_size() for t in hd.values())
        d2h += sum(t.numel() * t.element_size() for t in h_out0.values()) + h_loss.numel() * 4

    copy_stream = torch.cuda.Stream(dev)
    copied = [torch.cuda.Event() for _ in range(nbuf)]
    free = [torch.cuda.Event() for _ in range(nbuf)]
    for ev in free:
        ev.record(stream)

    def upload(i):
        """Step i's inputs into buffer set i % 2, once step i-2's kernels are done with it."""
        bi = i % nbuf
        copy_stream.wait_event(free[bi])
        with torch.cuda.stream(copy_stream):
            for k in host:
                dv[bi][k].copy_(host[k], non_blocking=True)
            for k in hd:
                dd[bi][k].copy_(hd[k], non_blocking=True)
        copied[bi].record(copy_stream)

    def compute(i):
        bi = i % nbuf
        stream.wait_event(copied[bi])
        x, xd = dv[bi], dd[bi]
        r = osd.osd_verify(x["draft"], x["target"], x["tokens"], x["uniforms"], sv.temperature, workspace=ws)
        h_out["acc"].copy_(r.accepted, non_blocking=True)
        h_out["tok"].copy_(r.out_tokens, non_blocking=True)
        h_out["mask"].copy_(r.mismatch_mask, non_blocking=True)
        osd.osd_distill_accepted(x["draft"], x["target"], r.accepted, rej_kind, 0.5, out=rej)
        h_rej["loss"].copy_(rej.loss, non_blocking=True)
        h_rej["seq"].copy_(rej.seq_of_row, non_blocking=True)
        h_rej["count"].copy_(rej.count, non_blocking=True)
        if wl == "serving-32k":
            r0 = osd.osd_verify(None, x["target"], x["greedy_tokens"], None, 0.0, workspace=ws)
            h_out0["acc"].copy_(r0.accepted, non_blocking=True)
            h_out0["tok"].copy_(r0.out_tokens, non_blocking=True)
            h_out0["mask"].copy_(r0.mismatch_mask, non_blocking=True)
            for i2, kind in enumerate(("rkl", "tvd")):
                osd.osd_distill(xd["draft"], xd["target"], None, kind, 0.5, loss=loss, dlogits=dl)
                h_loss[i2].copy_(loss, non_blocking=True)
        free[bi].record(stream)

    def steps(count):
        upload(0)
        for i in range(count):
            if i + 1 < count:
                upload(i + 1)
            compute(i)

    steps(max(2, args.warmup))
    torch.cuda.synchronize()
    n = max(3, args.steps // 2)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if world > 1:
        torch.distributed.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(copy_stream)  # before the first upload
    steps(n)
    e1.record(stream)       # after the last step's kernels and read-backs
    e1.synchronize()
    # whole job: every rank ran its own shard; the slowest rank's time counts
    ms = job_time_ms(e0.elapsed_time(e1), dev if world > 1 else None) / n
    return {"value": round(job_throughput(positions, world, ms), 1), "unit": "positions/s",
            "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": round(ms, 3), "steps": n,
            "pipelined": "step i+1's upload overlaps step i's kernels (two device buffer sets, a copy stream)",
            "note": "dlogits stays on the device, where the draft model's backward pass consumes it"}


# ----------------------------------------------------------------------------- CPU oracle
def _oracle_step_time(setup, n_rows, threads):
    """Time the oracle on the verify batch (whole, with the distillation of the
    rows it rejects) and on n_rows distill rows per loss kind; returns
    (seconds, positions) of that bounded sample."""
    import concurrent.futures as cf

    import numpy as np
    import oracle

    v = setup["v"]
    sv = setup["spec_v"]
    z = v["draft"].cpu()
    t = v["target"].cpu()
    y = v["tokens"].cpu()
    yg = v["greedy_tokens"].cpu()
    u = v["uniforms"].cpu()
    T = float(np.float32(sv.temperature))

    def chunks(n, parts):
        step = max(1, (n + parts - 1) // parts)
        return [(i, min(n, i + step)) for i in range(0, n, step)]

    rej_kind = "rkl" if "d" in setup else "fkl"

    def verify_and_distill(a, b):
        r = oracle.verify(z[a:b], t[a:b], y[a:b], u[a:b], T)
        n_rej = oracle.distill_rejected(z[a:b], t[a:b], r["accepted"], rej_kind, 0.5)[3]
        return (b - a) * sv.k + n_rej

    jobs = []
    for (a, b) in chunks(sv.B, threads):
        jobs.append(lambda a=a, b=b: verify_and_distill(a, b))
        if "d" in setup:
            jobs.append(lambda a=a, b=b: (oracle.verify(z[a:b], t[a:b], yg[a:b], u[a:b], 0.0), (b - a) * sv.k)[1])
    if "d" in setup:
        d = setup["d"]
        zd = d["draft"][:n_rows].cpu()
        td = d["target"][:n_rows].cpu()
        for kind in ("rkl", "tvd"):
            # blocks of at most 256 rows: the oracle holds each block in double precision
            for (a, b) in chunks(n_rows, max(threads, (n_rows + 255) // 256)):
                jobs.append(lambda a=a, b=b, kind=kind: (oracle.distill(zd[a:b], td[a:b], None, kind, 0.5),
                                                         b - a)[1])
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        positions = sum(ex.map(lambda f: f(), jobs))
    return time.perf_counter() - t0, positions


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the platform)."""
    import platform
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() == "Model name":
                return f"{line.split(':', 1)[1].strip()} ({platform.machine()})"
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return f"{line.split(':', 1)[1].strip()} ({platform.machine()})"
    except Exception:
        pass
    return platform.processor() or platform.machine()


def cpu_baseline(args, setup):
    threads = os.cpu_count() or 1
    n_rows = args.cpu_rows
    secs, pos = _oracle_step_time(setup, n_rows, threads)
    # one thread on a smaller sample of the same mix (a few seconds)
    n1 = max(64, n_rows // 32)
    secs1, pos1 = _oracle_step_time(setup, n1, 1)
    return {"value": round(pos / secs, 2), "unit": "positions/s", "cores": threads, "kind": "oracle",
            "sample": f"whole verify batch (both passes, with its rejected rows distilled) + {n_rows} "
                      f"distill rows per loss kind, "
                      f"{secs:.1f} s on {threads} host threads (double-precision C oracle)",
            "single_thread": {"value": round(pos1 / secs1, 2), "unit": "positions/s", "cores": 1,
                              "sample": f"whole verify batch + {n1} distill rows per loss kind, "
                                        f"{secs1:.1f} s on one thread"},
            "cpu_model": cpu_model()}


def run_reference(args):
    """The oracle (plain double-precision C) as the reference arm, on host cores."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch
    dev = "cpu"
    setup = (_setup_serving_32k(dev, args.distill_rows) if args.workload == "serving-32k"
             else _setup_large_vocab(dev))
    threads = os.cpu_count() or 1
    for _ in range(args.warmup):
        _oracle_step_time(setup, max(16, args.ref_rows // 8), threads)
    times, pos = [], 0
    for _ in range(args.steps):
        s, pos = _oracle_step_time(setup, args.ref_rows, threads)
        times.append(s)
    ms = 1e3 * sum(times) / len(times)
    value = pos / (ms / 1e3)
    sample = (f"per step: whole verify batch (both passes, with its rejected rows distilled) + "
              f"{args.ref_rows} distill rows per loss kind "
              f"of the same workload, {threads} host threads")
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": "positions/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded random logits)", "config": {"workload": setup["desc"]},
            "cpu_baseline": {"value": round(value, 2), "unit": "positions/s", "cores": threads,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 2), "unit": "positions/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "torch": torch.__version__}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- launcher
def _free_port() -> int:
    import socket
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as sock:
        sock.bind(("127.0.0.1", 0))
        return sock.getsockname()[1]


def launch_ranks(n: int, argv) -> int:
    """Start this script as n ranks on this node (torch.distributed.run, one
    process per GPU, rendezvous on 127.0.0.1) and return their exit status."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr", "127.0.0.1", f"--master-port={_free_port()}", os.path.abspath(__file__), *argv]
    return subprocess.call(cmd)


def run_launcher_check(args):
    """CPU-only check of the multi-rank plumbing (gloo, no GPU): every rank
    times its own stand-in step (rank r sleeps (r + 1) ms), the job time is the
    slowest rank's, and rank 0 prints the line with the number of ranks."""
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1:
        dist.init_process_group("gloo")
    local = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        time.sleep(1e-3 * (rank + 1))
        local.append((time.perf_counter() - t0) * 1e3)
    ms = job_time_ms(sum(local)) / args.steps
    if rank == 0:
        print(json.dumps({"check": "launcher", "n_gpus": world, "steps": args.steps, "ms_per_step": round(ms, 4),
                          "value": job_throughput(1, world, ms), "scaling": "weak"}), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["serving-32k", "large-vocab"], default="serving-32k")
    ap.add_argument("--cpu-rows", type=int, default=65536,
                    help="distill rows per loss kind in the cpu_baseline oracle sample (65536: the whole step, "
                         "about 7 s on 16 Neoverse-V2 cores)")
    ap.add_argument("--ref-rows", type=int, default=16384,
                    help="distill rows per loss kind in each step of --impl reference (about 2 s a step on "
                         "16 Neoverse-V2 cores)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the kernels timed outside the step (mixed sampling, tree verification)")
    ap.add_argument("--distill-rows", type=int, default=None,
                    help="override the distill buffer size N (small cases for profiling)")
    ap.add_argument("--distill-kinds", default="rkl,tvd",
                    help="loss kinds of the timed step's buffer flush, comma-separated (profiling one kind; "
                         "the e2e and CPU legs keep RKL and TVD)")
    ap.add_argument("--launcher-check", action="store_true",
                    help="CPU-only check of the multi-rank launcher (gloo ranks, no GPU work)")
    args = ap.parse_args()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # not started under torchrun: start the N ranks here, one process per GPU
        sys.exit(launch_ranks(args.gpus, sys.argv[1:]))
    if "WORLD_SIZE" in os.environ and int(os.environ["WORLD_SIZE"]) != args.gpus:
        print(f"warning: --gpus {args.gpus} but WORLD_SIZE={os.environ['WORLD_SIZE']}; the ranks decide",
              file=sys.stderr)
    if args.launcher_check:
        run_launcher_check(args)
        return
    if any(k not in ("fkl", "rkl", "jsd", "tvd", "ce") for k in args.distill_kinds.split(",")):
        ap.error("--distill-kinds takes fkl, rkl, jsd, tvd, ce")
    if args.warmup < 3:
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
