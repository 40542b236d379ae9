"""Benchmark of the quantised-state recurrence on GB300.

A step is one pass of the whole hot path over one batch of the KDA decode workload
(B = 256, H = 32, dk = dv = 128, T = 1024 tokens, per-token write-back, 4-bit mean payload,
widths 0..8, log-quantised decay rates with 2 bits): the log-uniform decay quantiser over the
batch's rates, then T write-backs, each the fused write-back kernel followed by the bit
allocation for the next one.  Inputs (17 GB) are resident in HBM when the timed region starts
and exceed L2, so no flush is needed.  Prints one JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--fit-every F]
                    [--workload gdn_decode|mamba2_decode|kda_prefill|...]

``--workload`` runs another of the paper's layer shapes (a labelled secondary measurement);
the default is KDA decode.

Under torchrun each rank runs the same per-GPU batch (batch elements are independent: weak
scaling, no collective); the reported value is the sum over ranks divided by the slowest rank.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

WORKLOAD = "kda_decode"
METRIC = "quantised-state recurrence tokens/s and achieved HBM GB/s (% of ~8 TB/s), 1\u00d7GB300"
PEAK_FALLBACK_GBS = 6800.0


def algorithmic_bytes(w, fit_every=1):
    """Bytes the method must move per write-back launch (the fused kernel, C tokens) and per
    allocation launch.  Per head, with u units and g scale groups per head (row unit: u = g =
    dk; head unit: u = 1, g = dk dv / 32):
      payload read + write        2 dk dv bbar / 8
      FP16 scales read + write    2 * 2 g
      widths read (in + out)      2 u
      fitted-factor index r + w   2 g
      head offsets (in + out)     8
      EMA statistics r + w        2 * 2 * 4 u
      range write                 4 u
    and per token
      q, k, v                     4 (2 dk + dv)
      decay rates                 dk (row, log-coded), 4 dk (row, FP32), 4 (head)
      beta                        4 (delta rule)
      readout o                   4 dv
    Allocation per batch element: EMA + range read 12 per unit, widths 1 per unit, offsets 4 H."""
    dk, dv = w.dk, w.dv
    row = w.unit == "row"
    u = dk if row else 1
    g = dk if row else dk * dv // 32
    rates = (dk if w.gate_bits else 4 * dk) if w.per_row_decay else 4
    per_token = 4 * (2 * dk + dv) + rates + (4 if w.erase else 0) + 4 * dv
    per_head = (2 * dk * dv * w.bbar // 8 + 4 * g + 2 * u + 2 * g + 8 + 16 * u + 4 * u +
                w.C * per_token)
    writeback = per_head * w.B * w.H
    alloc = w.B * (w.H * u * 13 + 4 * w.H)
    return writeback, alloc, per_head


# Committed ncu summaries that carry a DRAM traffic figure, per (workload, interval form):
# the summary and the kernel sources its figure was taken on.
_CORE = ("qs_wb_row.cuh", "qs_common.cuh", "qs_internal.h")
TRAFFIC_PROFILES = {
    ("kda_decode", "token"): ("writeback_kda_decode.md", _CORE),
    ("kda_prefill", "chunk"): ("writeback_kda_prefill_chunk.md", _CORE + ("qs_chunk.cuh", "qs_tc.cuh")),
    ("gdn_decode", "token"): ("head_kernel_gdn_decode.md", ("qs_head.cuh", "qs_common.cuh", "qs_internal.h")),
    ("mamba2_decode", "token"): ("writeback_mamba2_decode.md", _CORE),
}


def kernel_sha(files=_CORE):
    """Hash of the write-back kernel's sources (ties an ncu traffic figure to the kernel it was
    taken on)."""
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2609_30950_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload, form):
    """(kernel sha, DRAM bytes per write-back + allocation launch pair) from the committed ncu
    summary of this workload and interval form, the bytes None unless the summary was taken on
    the current kernel sources (or there is no summary)."""
    entry = TRAFFIC_PROFILES.get((workload, form))
    if entry is None:
        return kernel_sha(), None
    name, files = entry
    sha = kernel_sha(files)
    path = os.path.join(ROOT, "profiles", name)
    if not os.path.exists(path):
        return sha, None
    vals = {}
    for line in open(path):
        if ":" in line and line.strip().startswith("- "):
            k, v = line.strip()[2:].split(":", 1)
            vals[k.strip()] = v.strip()
    if vals.get("kernel_sha") != sha:
        return sha, None
    try:
        return sha, float(vals["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return sha, None


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return PEAK_FALLBACK_GBS, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    def __init__(self, gpu_index=0):
        # raw samples go to a scratch file; the JSON line carries their summary
        out = os.environ.get("QSTATE_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out, f"qstate_clocks_rank{gpu_index}_{os.getpid()}.csv")
        os.makedirs(out, exist_ok=True)
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        try:
            rows = [r.split(",") for r in open(self.path).read().strip().splitlines() if r.strip()]
        except Exception:
            return None
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            for n, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(rows)}


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(w, budget_s=12.0, parallel=False):
    """The oracle as it stands on a bounded sample of the workload: the log-decay quantiser over
    the sample's rates (when rates are coded), then per write-back one pass over every head of
    the sampled batch elements and the allocation.  Single-threaded (the plain build), or with
    ``parallel`` the OpenMP timing build, whose threads share out the heads of each write-back
    over every host core this process may use (same arithmetic).  Returns tokens/s and the
    sample."""
    import numpy as np
    from oracle import oracle as orc
    cores = host_cores() if parallel else 1
    if parallel:
        os.environ["OMP_NUM_THREADS"] = str(cores)
    nb, nt = 4, max(64, w.C)
    sub = synth.scaled(w, B=nb)
    cfg = orc.Cfg.from_workload(sub)
    t_start = time.perf_counter()
    inp = synth.host_inputs(sub, t_range=(0, nt))
    gen_s = time.perf_counter() - t_start
    t0 = time.perf_counter()
    codes = lut = None
    if w.gate_bits:
        codes, lut, _ = orc.quant_decay(inp["s"], w.H * w.dk, w.gate_bits)
    src, dst = orc.init_state(cfg)
    o = np.zeros((nb, nt, w.H, w.dv), np.float32)
    ms, mr, R = (np.zeros(cfg.units * nb, np.float32) for _ in range(3))
    tokens = 0
    for wi, t in enumerate(range(0, nt, w.C)):
        orc.step(cfg, src, dst, inp, t, t + w.C, wi, o, ms, mr, R, codes, lut, parallel=parallel)
        src.widths[:], src.head_off[:] = orc.alloc(cfg, ms, mr, R)
        src, dst = dst, src
        tokens += nb * w.C
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    how = f"OpenMP over the heads, {cores} threads" if parallel else "single thread"
    return tokens / el, dict(cores=cores, sample=f"{nb} batch elements x {tokens // nb} tokens x "
                                                 f"{w.H} heads, {how} (input synthesis "
                                                 f"{gen_s:.1f}s excluded)",
                             seconds=el)


def cpu_baselines(w, budget_s):
    """The oracle on all host cores (the reported baseline) and single-threaded beside it."""
    one, info1 = cpu_baseline(w, budget_s)
    try:
        par, info = cpu_baseline(w, budget_s, parallel=True)
    except Exception as e:   # no OpenMP compiler: the single-thread figure only
        return one, info1, {"value": one, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                            "sample": info1["sample"], "all_cores": f"unavailable: {e}"}
    return par, info, {"value": par, "unit": "tokens/s", "cores": info["cores"], "kind": "oracle",
                       "sample": info["sample"],
                       "single_thread": {"value": one, "unit": "tokens/s", "cores": 1,
                                         "sample": info1["sample"]}}


def run_reference(args, w):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    vals = []
    for i in range(args.warmup + args.steps):
        v, info = cpu_baseline(w, budget_s=max(3.0, 40.0 / max(1, args.steps + args.warmup)),
                               parallel=True)
        if i >= args.warmup:
            vals.append(v)
    value = statistics.median(vals)
    line = {"metric": METRIC, "value": value,
            "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * w.B * w.T / value, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "impl": "reference",
            "config": config_of(w, args),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": info["cores"],
                             "kind": "oracle", "sample": info["sample"]},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def slowest_ms(ms, world, device):
    """Max over ranks of a per-rank time (ms); the job is as fast as its slowest rank."""
    if world <= 1:
        return float(ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank, world, ms):
    """Whole-job tokens/s: every rank runs its own batch of independent sequences (weak scaling,
    no exchange on the data path), so the job processes world x tokens_per_rank per step."""
    return tokens_per_rank * world / (ms / 1000.0)


def rank_seed_offset(rank):
    """Each rank draws its own batch of sequences (a shard of the job's batch)."""
    return rank


def config_of(w, args):
    return {"workload": w.name, "B": w.B, "H": w.H, "dk": w.dk, "dv": w.dv, "T": w.T, "C": w.C,
            "bbar": w.bbar, "widths": [w.bmin, w.bmax], "gate_bits": w.gate_bits,
            "fit_every": args.fit_every, "alloc_mode": getattr(args, "alloc_mode", 0),
            "interval_form": getattr(args, "form", "token"),
            "global_batch": w.B * args.gpus, "seq_len": w.T,
            "parallelism": f"dp{args.gpus}",
            "l2": (f"inputs {input_gb(w) * 1e3:.0f} MB > 129 MB L2: no flush" if input_gb(w) > 0.129
                   else f"inputs {input_gb(w) * 1e3:.1f} MB fit in L2 (small case)")}


def input_gb(w):
    """Token inputs of one step (q, k, v, FP32 rates, beta), which each step streams through."""
    rates = w.dk if w.per_row_decay else 1
    return w.B * w.T * w.H * (2 * w.dk + w.dv + rates + 1) * 4 / 1e9


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--fit-every", type=int, default=1)
    ap.add_argument("--alloc-mode", type=int, default=0,
                    help="0: widths from the previous write-back's statistics; 1: from this one's")
    ap.add_argument("--form", default="auto", choices=["auto", "token", "chunk"],
                    help="write-back intervals token by token, or in 16-token blocks on the tensor "
                         "cores (row unit, 128 x 128, C > 1); auto: the chunked form where it applies")
    ap.add_argument("--T", type=int, default=None, help="tokens per step (default: workload T)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-chunk", type=int, default=0,
                    help="tokens per host-staging chunk of the end-to-end run (default: 64 when the "
                         "state is written back every token, else max(256, C))")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--scan-partitions", type=int, default=0,
                    help="batch partitions of each scan, one stream each (0: the library's choice)")
    ap.add_argument("--workload", default=WORKLOAD, choices=sorted(synth.WORKLOADS),
                    help="the paper's layer shape to run (default: KDA decode)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    w = synth.WORKLOADS[args.workload]
    if args.T:
        w = synth.scaled(w, T=args.T)
    if args.form == "auto":
        args.form = ("chunk" if w.C > 1 and w.unit == "row" and w.dk == 128 and w.dv == 128
                     and not w.general else "token")
    if args.impl == "reference":
        return run_reference(args, w)

    import torch
    import torch.distributed as dist
    import paper_2609_30950_gb300 as q

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    q.load(build_if_missing=True)

    cfg = q.Config.from_workload(w, fit_every=args.fit_every, alloc_mode=args.alloc_mode,
                                 interval_form=q.FORM_CHUNK if args.form == "chunk" else q.FORM_TOKEN)
    x = synth.device_inputs(w, device=dev, seed_offset=rank_seed_offset(rank))
    nchan = w.H * w.dk
    coded = w.gate_bits > 0
    codes = lut = thr = None
    if coded:
        L = 1 << w.gate_bits
        codes = torch.empty(x["s"].shape, dtype=torch.uint8, device=dev)
        lut = torch.empty(nchan * L, dtype=torch.float32, device=dev)
        thr = torch.empty(nchan * (L - 1), dtype=torch.float32, device=dev)
    beta = x["beta"] if w.erase else None
    o = torch.empty((w.B, w.T, w.H, w.dv), dtype=torch.float32, device=dev)
    A, Bst = q.new_state(cfg, dev), q.new_state(cfg, dev)
    st = q.new_stats(cfg, dev)
    X = q.Inputs(x["q"], x["k"], x["v"], None if coded else x["s"], codes, lut, beta, w.T)
    stream = torch.cuda.current_stream(dev)
    q.qstate_set_scan_partitions(args.scan_partitions)
    parts = q.qstate_scan_partition_count(cfg, X, st)

    def quant_decay(s):
        if coded:
            q.qstate_quant_decay(cfg, x["s"], codes, lut, thr, s)

    def step():
        quant_decay(stream)
        q.qstate_init(cfg, A, Bst, stream)
        q.qstate_scan(cfg, A, Bst, X, 0, w.T, 0, o, st, stream)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for _ in range(args.warmup):
        step()
    q.qstate_check(stream)
    barrier()

    # timed region: K steps; events split each step into the decay quantiser and the scan
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        barrier()
        t0 = time.perf_counter()
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for e0, e1, e2 in ev:
            e0.record(stream)
            quant_decay(stream)
            q.qstate_init(cfg, A, Bst, stream)
            e1.record(stream)
            q.qstate_scan(cfg, A, Bst, X, 0, w.T, 0, o, st, stream)
            e2.record(stream)
        end.record(stream)
        barrier()
        wall = time.perf_counter() - t0
    q.qstate_check(stream)
    ms_total = slowest_ms(start.elapsed_time(end), world, dev)
    ms_step = ms_total / args.steps
    tokens_step = w.B * w.T
    value = job_throughput(tokens_step, world, ms_step)
    scan_ms = statistics.median(e1.elapsed_time(e2) for _, e1, e2 in ev)
    decay_ms = statistics.median(e0.elapsed_time(e1) for e0, e1, _ in ev)
    n_wb = -(-w.T // w.C)
    per_wb_ms = scan_ms / n_wb       # write-back kernel + allocation kernel per write-back

    wb_bytes, alloc_bytes, per_head = algorithmic_bytes(w, args.fit_every)
    peak, peak_kind = peaks()
    achieved = (wb_bytes + alloc_bytes) / (per_wb_ms / 1000.0) / 1e9
    sha, traffic = recorded_traffic(w.name, args.form)

    # end to end through the public API: pinned host inputs -> device, the step, o -> host.
    # The rates go first (the log-decay levels are taken over all tokens of the step); q, k,
    # v and beta then stream in chunk by chunk on a copy stream while the compute stream scans
    # the previous chunk, and readouts stream back (qstate_scan_host).
    e2e = None
    if not args.no_e2e:
        names = ["q", "k", "v", "s"] + (["beta"] if w.erase else [])
        host_in = {n: torch.empty(x[n].shape, dtype=x[n].dtype, pin_memory=True) for n in names}
        for n in names:
            host_in[n].copy_(x[n])
        host_o = torch.empty(o.shape, dtype=o.dtype, pin_memory=True)
        h2d = sum(t.numel() * t.element_size() for t in host_in.values())
        d2h = host_o.numel() * host_o.element_size()
        comp, copy_stream = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        comp.wait_stream(stream)
        xh = q.Inputs(host_in["q"], host_in["k"], host_in["v"], None if coded else host_in["s"],
                      None, None, host_in.get("beta"), w.T)
        # per-token write-back: 64-token chunks (larger ones measured no faster); write-back
        # intervals of C > 1 tokens: at least 1024 tokens (several intervals per chunk, fewer
        # staging launches and stream handoffs per write-back; the prefill measured 2.34M
        # tokens/s at 256, 2.48M at 512, 2.55M at 1024 and 2048)
        chunk = args.e2e_chunk if args.e2e_chunk > 0 else (64 if w.C == 1 else max(1024, w.C))
        chunk = -(-chunk // w.C) * w.C   # a multiple of C

        def e2e_step():
            if coded:   # the levels are taken over all tokens: the rates go first
                with torch.cuda.stream(comp):
                    x["s"].copy_(host_in["s"], non_blocking=True)
                quant_decay(comp)
            q.qstate_init(cfg, A, Bst, comp)
            q.qstate_scan_host(cfg, A, Bst, xh, X, 0, w.T, 0, host_o, o, st, chunk, comp,
                               copy_stream)

        e2e_step()
        barrier()
        k2 = max(1, min(args.steps, 3))
        s0 = torch.cuda.Event(enable_timing=True)
        s1 = torch.cuda.Event(enable_timing=True)
        s0.record(comp)
        for _ in range(k2):
            e2e_step()
        s1.record(comp)
        barrier()
        e_ms = slowest_ms(s0.elapsed_time(s1) / k2, world, dev)
        e2e = {"value": job_throughput(tokens_step, world, e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e_ms,
               "staging": f"qstate_scan_host, {chunk}-token chunks on a copy stream"}
        q.qstate_check(comp)

    # decay quantiser (4), init (alloc + pack), then per write-back: write-back + alloc, or with
    # current-statistics allocation a statistics pass + alloc + write-back
    launches_per_step = (4 if coded else 0) + 2 + (3 if args.alloc_mode == 1 else 2) * n_wb * parts
    clocks = clk.summary()
    if rank != 0:
        if world > 1:
            dist.barrier()
            dist.destroy_process_group()
        return
    cpu = None
    if not args.no_cpu:
        _, _, cpu = cpu_baselines(w, 10.0)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": config_of(w, args),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_source": peak_kind,
                     "kernel": "write-back + allocation per token",
                     "algorithmic_bytes_per_launch": wb_bytes + alloc_bytes,
                     "kernel_sha": sha},
        "breakdown": {"decay_quantiser_ms": decay_ms, "scan_ms": scan_ms,
                      "per_writeback_us": per_wb_ms * 1000.0, "wall_s": wall,
                      "bits_per_element": q.bits_per_element(cfg),
                      "pct_of_8TBps": 100.0 * achieved / 8000.0},
        "e2e": e2e, "gpu_launches": launches_per_step * args.steps, "clocks": clocks,
        "cpu_baseline": cpu,
    }
    line["config"]["scan_partitions"] = parts
    print(json.dumps(line))
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
