#!/usr/bin/env python3
"""Benchmark of the MPCache decode path on one GB300 (or N replicas).

One step = the whole method over one batch of synthetic input: look-once
static eviction of the leader layers, gathering + clustering of every
layer, then all E decode steps (selection for the leaders, append + sparse
attention for every layer).  The metric is selected-KV tokens per second:
the rows every decode step attends (selected clusters plus tail, summed over
layers, sequences and kv heads) divided by the whole step's time.

Prints one JSON line on rank 0.  ``--impl reference`` times the fp64 CPU
oracle on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2501_06807_gb300 import synth  # noqa: E402

# The headline metric names three figures; `value` is the last (selected KV
# tokens attended per second over the whole job), and the line also carries
# the decode-step latency (decode_step_us) and its HBM GB/s (decode).
METRIC = "decode-step latency (\u00b5s) and achieved HBM GB/s vs ~8 TB/s; selected-KV tokens/s"
UNIT = "selected-KV tokens/s"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# fp32 FFMA peak of a GB300 at its maximum SM clock: 152 SMs x 128 lanes x 2 flops
FFMA_PEAK_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=synth.C5.name, choices=sorted(synth.WORKLOADS))
    p.add_argument("--decode-steps", type=int, default=None)
    p.add_argument("--no-e2e", action="store_true")
    # the paper's ablation axes, applied to --workload (the line's config
    # reports them): alpha of Eq. 3, the window ratios of static eviction,
    # the static budget, the cluster size, the hierarchy (fanouts and kept
    # ratio per level, finest first), the sharing group size, and the
    # cross-layer correlation of the synthetic inputs
    p.add_argument("--alpha", type=float)
    p.add_argument("--window-ppm", type=int)
    p.add_argument("--long-window-ppm", type=int)
    p.add_argument("--keep-ppm", type=int)
    p.add_argument("--cluster-size", type=int)
    p.add_argument("--fanouts", help="comma-separated children per coarser cluster ('' for one level)")
    p.add_argument("--level-keep-ppm", help="comma-separated kept ppm per level, finest first")
    p.add_argument("--share-every", type=int)
    p.add_argument("--layer-rho-ppm", type=int)
    # the decode step's form: speculative first selection round (-1 auto),
    # and one fused kernel (1) or the selection + attention launches (-1 / 0)
    p.add_argument("--speculate", type=int, choices=[-1, 0, 1], default=-1)
    p.add_argument("--fuse", type=int, choices=[-1, 0, 1], default=-1)
    # measured side reports instead of the bench line (one JSON line each):
    # adaptive-sharing: commonality of unshared selections, the group size the
    # adaptive rule picks, and the decode step with it; tokenwise: selection
    # and decode step of the clustered path and of the token-wise comparator
    # read-floor: the time to read one decode step's attention tiles and
    # nothing else (bench_floor.cu), at the step's size and multiples of it
    p.add_argument("--report", choices=["adaptive-sharing", "tokenwise", "read-floor"])
    p.add_argument("--share-threshold", type=float, default=0.25)
    # internal: print the oracle sample of --workload as JSON (the bench runs
    # it in a child process with one BLAS thread for the single-core figure)
    p.add_argument("--oracle-sample", action="store_true", help=argparse.SUPPRESS)
    return p.parse_args()


def peaks():
    try:
        with open(PEAKS_FILE) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return FALLBACK, "fallback"


# ------------------------------------------------------------ workload ----

def _ints(text):
    return tuple(int(v) for v in text.split(",") if v.strip())


# (flag, Workload field, parser)
OVERRIDES = (("--alpha", "alpha", float), ("--window-ppm", "window_ppm", int),
             ("--long-window-ppm", "long_window_ppm", int), ("--keep-ppm", "keep_ppm", int),
             ("--cluster-size", "cluster_size", int), ("--fanouts", "fanouts", _ints),
             ("--level-keep-ppm", "level_keep_ppm", _ints), ("--share-every", "share_every", int),
             ("--layer-rho-ppm", "layer_rho_ppm", int))


def _attr(flag):
    return flag[2:].replace("-", "_")


def overrides_of(args):
    """{field: value} of the ablation flags given on the command line."""
    return {field: parse(getattr(args, _attr(flag))) if parse is _ints else getattr(args, _attr(flag))
            for flag, field, parse in OVERRIDES if getattr(args, _attr(flag)) is not None}


def override_argv(args):
    """The ablation flags as given, to pass on to a child process."""
    return [a for flag, _, _ in OVERRIDES if getattr(args, _attr(flag)) is not None
            for a in (flag, str(getattr(args, _attr(flag))))]


def workload_of(args):
    """--workload with the ablation flags applied."""
    w = synth.WORKLOADS[args.workload]
    ov = overrides_of(args)
    if not ov:
        return w
    w = w.replace(**ov)
    if len(w.level_keep_ppm) != w.n_levels:
        raise SystemExit(f"--level-keep-ppm needs {w.n_levels} ratios (one per level, finest first)")
    if w.cluster_size < 1 or w.share_every < 1 or not 0 <= w.alpha <= 1:
        raise SystemExit("cluster size and share_every must be >= 1 and alpha in [0, 1]")
    return w

def rules(w):
    from paper_2501_06807_gb300 import mpcache
    R = mpcache.window_rows_bound(w.prompt_len, w.window_ppm, w.long_window_ppm, w.long_prompt_threshold)
    leaders = sorted({mpcache.sharing_leader(l, w.share_every) for l in range(w.n_layers)})
    return R, leaders


# ---------------------------------------------------------- replicas ----
#
# The path has no exchange step: --gpus N runs N independent replicas (one
# process per GPU, each with its own seeded workload) and reports the units
# all ranks processed over the slowest rank's time.

def replica_workload(w, rank):
    """The workload of one replica: rank r draws its inputs from seed + 7919 r."""
    return w.replace(seed=w.seed + 7919 * rank) if rank else w


def max_over_ranks(x, dist, device=None):
    """max over the ranks of a float (a time), through one all-reduce."""
    if dist is None:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(units_per_rank, world, ms):
    """Whole-job throughput: the units every rank processed over the slowest time."""
    return units_per_rank * world / (ms / 1e3)


def select_rows(w, n_tok):
    """Representative rows the hierarchical selection of one (leader, b, kv
    head) scores for a cache of n_tok rows: every cluster of the coarsest
    level, then the children of each level's kept clusters."""
    from paper_2501_06807_gb300 import mpcache
    C = [n_tok // w.cluster_size]
    for f in w.fanouts:
        C.append(-(-C[-1] // f))
    rows, cand = 0, C[-1]
    for l in range(len(C) - 1, -1, -1):
        rows += cand
        k = min(mpcache.ppm_count(C[l], w.level_keep_ppm[l]), cand)
        if l > 0:
            cand = min(C[l - 1], k * w.fanouts[l - 1])
    return rows


def static_flops(w, lens, n_leaders):
    """Algorithmic FLOPs of the two score passes: every (window row, causal
    key) pair of every leader layer and query head, 2 d flops per pass."""
    from paper_2501_06807_gb300 import mpcache
    total = 0
    for T in lens:
        wl = mpcache.ppm_count(T, w.long_window_ppm if T > w.long_prompt_threshold else w.window_ppm)
        pairs = wl * (T - wl) + wl * (wl + 1) // 2
        total += pairs
    return 2 * 2 * w.head_dim * total * w.n_q_heads * n_leaders


# ------------------------------------------------------------- clocks ----

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        """Starts sampling every 50 ms and returns once the first sample is
        out (nvidia-smi takes a while to start), so that the samples read at
        stop() fall inside the region between the two calls."""
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.proc.stdout.readline()
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out = ""
        rows = [r.split(",") for r in out.strip().splitlines() if r.strip()]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, r[4:8]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------ our arm ----

def make_engine(w, E):
    from paper_2501_06807_gb300 import mpcache
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    return mpcache.Engine(n_layers=w.n_layers, batch=w.batch, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                          head_dim=w.head_dim, dtype=dt, t_max=w.prompt_len, keep_ppm=w.keep_ppm,
                          cluster_size=w.cluster_size, fanouts=w.fanouts, level_keep_ppm=w.level_keep_ppm,
                          share_every=w.share_every, max_decode_steps=E, alpha=w.alpha,
                          window_ppm=w.window_ppm, long_window_ppm=w.long_window_ppm,
                          long_prompt_threshold=w.long_prompt_threshold)


def run_ours(args, rank, world, dist):
    from paper_2501_06807_gb300 import build, mpcache
    build.build()
    mpcache.load()
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    w = replica_workload(workload_of(args), rank)
    E = args.decode_steps or w.decode_steps
    R, leaders = rules(w)
    x = synth.generate(w, R, device="cuda", decode_steps=E)
    lens = x.prompt_lens.cuda()
    pt = x.page_table.cuda() if x.page_table is not None else None
    eng = make_engine(w, E)
    out_all = torch.empty((E, w.n_layers, w.batch, w.n_q_heads, w.head_dim), dtype=torch.float32, device=dev)

    def prefill():
        eng.prefill(x.k, x.v, x.q_win, lens, pt, w.page_size)

    step_kw = dict(speculate=args.speculate, fuse=args.fuse)
    # kernel launches of one decode step (the library's choice of form)
    step_launches = eng.decode_step_launches(x.q[0], x.k_new[0], x.v_new[0], out=out_all[0], fuse=args.fuse)

    def decode_all():
        for e in range(E):
            eng.decode_step(x.q[e], x.k_new[e], x.v_new[e], out=out_all[e], **step_kw)

    # eager pass: counts the attended rows of every step, checks the status
    prefill()
    attended = 0
    n_keep = eng.n_keep.cpu().tolist()
    s = w.cluster_size
    rep_rows = 0
    for e in range(E):
        eng.decode_step(x.q[e], x.k_new[e], x.v_new[e], out=out_all[e], **step_kw)
        n_sel = eng.n_sel.cpu().tolist()
        for b in range(w.batch):
            n_tok = n_keep[b] + e
            attended += (n_sel[b] * s + n_tok % s + 1) * w.n_layers * w.n_kv_heads
            rep_rows += select_rows(w, n_tok) * len(leaders) * w.n_kv_heads
    status = mpcache.device_status()
    if status != 0:
        raise RuntimeError(f"device status {status} after the eager pass")

    graph = torch.cuda.CUDAGraph()
    prefill()
    torch.cuda.synchronize()
    with torch.cuda.graph(graph):
        decode_all()
    torch.cuda.synchronize()

    for _ in range(args.warmup):
        prefill()
        graph.replay()
    torch.cuda.synchronize()

    stream = torch.cuda.current_stream()
    ev = lambda: torch.cuda.Event(enable_timing=True)
    marks = [(ev(), ev(), ev(), ev()) for _ in range(args.steps)]
    clocks = ClockSampler(dev.index)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_start, t_end = ev(), ev()
    t_start.record(stream)
    for m in marks:
        m[0].record(stream)
        eng.static_evict(x.k, x.q_win, lens, pt, w.page_size)
        m[1].record(stream)
        eng.build_clusters(x.k, x.v, pt, w.page_size)
        m[2].record(stream)
        graph.replay()
        m[3].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if dist is not None:
        dist.barrier()
    total_ms = max_over_ranks(t_start.elapsed_time(t_end), dist, dev)
    static_ms = sum(m[0].elapsed_time(m[1]) for m in marks) / args.steps
    build_ms = sum(m[1].elapsed_time(m[2]) for m in marks) / args.steps
    decode_ms = sum(m[2].elapsed_time(m[3]) for m in marks) / args.steps
    ms_per_step = total_ms / args.steps
    value = job_value(attended, world, ms_per_step)

    # the same decode steps as one fused kernel per step (bf16), timed beside
    # the two-launch form the job runs
    fused_us = None
    if w.dtype == "bf16":
        gf = torch.cuda.CUDAGraph()
        prefill()
        for e in range(E):  # eager once: the fused call's workspace
            eng.decode_step(x.q[e], x.k_new[e], x.v_new[e], out=out_all[e], speculate=args.speculate, fuse=1)
        prefill()
        torch.cuda.synchronize()
        with torch.cuda.graph(gf):
            for e in range(E):
                eng.decode_step(x.q[e], x.k_new[e], x.v_new[e], out=out_all[e], speculate=args.speculate, fuse=1)
        per = []
        for i in range(5):
            prefill()
            a, b = ev(), ev()
            a.record(stream)
            gf.replay()
            b.record(stream)
            torch.cuda.synchronize()
            if i >= 2:
                per.append(a.elapsed_time(b) / E * 1e3)
        fused_us = statistics.median(per)
        if mpcache.device_status() != 0:
            raise RuntimeError("device status set by the fused decode steps")

    # e2e through the public API with host buffers.  A copy stream moves the
    # leaders' keys and window queries to the device (static eviction reads
    # only those), leader by leader, then the decode inputs, then the whole
    # keys and values of the last group; each leader's static eviction starts
    # once its copies have landed.  A gather stream then builds the group's
    # caches from its kept rows (the leader's keys from the device, every
    # other key and value row straight from pinned host memory, so evicted
    # rows never cross the host link) while the next leaders are scored.
    # When the link has time to spare during scoring, the last group, whose
    # gather would end the prefill, is copied whole and gathers from the
    # device.  Non-leader window queries are never read, so they are not
    # copied.
    e2e = None
    if not args.no_e2e:
        host = {n: getattr(x, n).cpu().pin_memory() for n in ("k", "v", "q_win", "q", "k_new", "v_new")}
        host_lens = x.prompt_lens.pin_memory()
        out_host = torch.empty(out_all.shape, dtype=out_all.dtype).pin_memory()
        members = {lead: [l for l in range(w.n_layers) if eng.group_of[l] == eng.group_of[lead] and l != lead]
                   for lead in leaders}
        copies = [(x.k[l], host["k"][l]) for l in leaders] + [(x.q_win[l], host["q_win"][l]) for l in leaders]
        decode_in = [(getattr(x, n), host[n]) for n in ("q", "k_new", "v_new")]
        esz_kv = host["k"].element_size()
        kept_rows = sum(int(t) for t in eng.n_keep.tolist()) * w.n_kv_heads  # per layer
        n_last = sum(1 for l in range(w.n_layers) if eng.group_of[l] == eng.group_of[leaders[-1]])
        row_bytes = kept_rows * w.head_dim * esz_kv  # one layer's kept K (or V) rows
        gathered = row_bytes * (len(leaders) + 2 * (w.n_layers - len(leaders)))
        copied = sum(src.numel() * src.element_size() for _, src in copies + decode_in) + host_lens.numel() * 4
        # the last group whole: its other layers' K and every V, instead of
        # their kept rows; worth it if the link (about 200 GB/s) still idles
        # while the leaders are scored
        whole_last = (2 * n_last - 1) * host["k"][0].numel() * esz_kv
        last_kept = row_bytes * (1 + 2 * (n_last - 1))
        last_whole = (copied + gathered - last_kept + whole_last) / 200e6 < static_ms
        h2d = copied + gathered + (whole_last - last_kept if last_whole else 0)
        d2h = out_host.numel() * out_host.element_size()
        side = torch.cuda.Stream(device=dev)
        gat = torch.cuda.Stream(device=dev)
        # the first and the last leader are scored alone (the first starts as
        # soon as its copies land, the last ends the chain), the others two at
        # a time (larger grids, fewer launches)
        mid = leaders[1:-1]
        batches = [leaders[:1]] + [mid[i:i + 2] for i in range(0, len(mid), 2)] + [leaders[-1:]]
        batches = [bt for bt in batches if bt]
        last = [l for l in range(w.n_layers) if eng.group_of[l] == eng.group_of[leaders[-1]]]
        landed = [torch.cuda.Event() for _ in batches]
        last_landed = torch.cuda.Event()

        def e2e_step():
            lens.copy_(host_lens, non_blocking=True)
            side.wait_stream(stream)  # the previous step is done with the inputs
            gat.wait_stream(stream)   # ... and with the caches
            with torch.cuda.stream(side):
                for i, batch in enumerate(batches):
                    for lead in batch:
                        x.k[lead].copy_(host["k"][lead], non_blocking=True)
                        x.q_win[lead].copy_(host["q_win"][lead], non_blocking=True)
                    landed[i].record(side)
                for dst, src in decode_in:
                    dst.copy_(src, non_blocking=True)
                if last_whole:
                    for l in last:
                        if l != leaders[-1]:  # the leader's keys are already there
                            x.k[l].copy_(host["k"][l], non_blocking=True)
                        x.v[l].copy_(host["v"][l], non_blocking=True)
                last_landed.record(side)
            for i, batch in enumerate(batches):
                stream.wait_event(landed[i])
                eng.static_evict(x.k, x.q_win, lens, pt, w.page_size, layers=batch)
                gat.wait_stream(stream)
                with torch.cuda.stream(gat):
                    if i == len(batches) - 1 and last_whole:
                        gat.wait_event(last_landed)
                        eng.build_clusters(x.k, x.v, pt, w.page_size, layers=last)
                        continue
                    eng.build_clusters(x.k, host["v"], pt, w.page_size, layers=batch)
                    rest = [l for lead in batch for l in members[lead]]
                    if rest:
                        eng.build_clusters(host["k"], host["v"], pt, w.page_size, layers=rest)
            stream.wait_stream(gat)
            stream.wait_stream(side)
            graph.replay()
            out_host.copy_(out_all, non_blocking=True)

        for _ in range(max(3, args.warmup)):  # first passes over new pinned pages run slow
            e2e_step()
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        # per-step events: the host link is shared with other tenants of the
        # machine and some passes copy several times slower, so the median step
        # is the figure and the mean is reported beside it
        em = [(ev(), ev()) for _ in range(args.steps)]
        for m in em:
            m[0].record(stream)
            e2e_step()
            m[1].record(stream)
        torch.cuda.synchronize()
        per = [m[0].elapsed_time(m[1]) for m in em]
        e2e_ms = max_over_ranks(statistics.median(per), dist, dev)
        e2e = {"value": job_value(attended, world, e2e_ms), "unit": UNIT, "ms_per_step": e2e_ms,
               "ms_per_step_mean": max_over_ranks(sum(per) / len(per), dist, dev),
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "last_group_copied_whole": bool(last_whole)}

    pk, pk_kind = peaks()
    n_lead = len(leaders)
    flops = static_flops(w, [int(t) for t in x.prompt_lens], n_lead)
    static_tflops = flops / (static_ms / 1e3) / 1e12
    esz = 2 if w.dtype == "bf16" else 4
    # decode bytes: attended K and V rows, the fp32 representatives the
    # selection scores (each level's candidates), q, k_new, v_new, o
    kv_bytes = attended * w.head_dim * 2 * esz
    rep_bytes = rep_rows * w.head_dim * 4
    io_bytes = E * w.n_layers * w.batch * (w.n_q_heads * w.head_dim * (esz + 4) + 2 * w.n_kv_heads * w.head_dim * esz)
    dec_bytes = kv_bytes + rep_bytes + io_bytes
    decode_gbs = dec_bytes / (decode_ms / 1e3) / 1e9
    dominant_static = static_ms >= decode_ms
    # bf16 keys score on tcgen05 (paged keys through their gathered dense copy)
    tensor_path = w.dtype == "bf16"
    # DRAM bytes of one static-eviction call (both score passes), from an ncu
    # capture of the 8k workload (dram__bytes_read.sum + dram__bytes_write.sum
    # of the two score_tc_kernel launches: 302.2 + 10.0 + 310.6 + 5.7 MB):
    # each pass reads its inputs once, so the 32k figure is that capture
    # scaled by the input bytes (939.5 / 302.2 MB).  Valid for the kernel as
    # captured.
    static_traffic = {"c3_llama3_8b_gqa_t8192": 628.4e6,
                      "c5_llama3_8b_gqa_t32768_needles": 628.4e6 * 939.5 / 302.2}.get(w.name)
    if dominant_static and tensor_path:
        # tcgen05 score passes: two launches of a few ms each, so the burst
        # bf16 figure (a GEMM timed alone) is the denominator
        peak_t = pk["bf16_tflops"]
        roof = {"kernel": "mpc_static_evict (score_tc_kernel pass 0 + pass 1 + budget)", "bound": "tensor",
                "achieved": round(static_tflops, 3), "peak": peak_t, "unit": "TFLOP/s",
                "frac": round(static_tflops / peak_t, 4), "traffic": static_traffic,
                "peak_source": pk_kind + " bf16_tflops (burst)"}
    elif dominant_static:
        roof = {"kernel": "mpc_static_evict (rowstats + colsum + budget)", "bound": "alu",
                "achieved": round(static_tflops, 3), "peak": round(FFMA_PEAK_TFLOPS, 1), "unit": "TFLOP/s",
                "frac": round(static_tflops / FFMA_PEAK_TFLOPS, 4), "traffic": None,
                "peak_source": "fp32 FFMA: 152 SMs x 128 lanes x 2 flops x 2.07 GHz"}
    # the decode step (one mpc_decode_step call per step, all layers): bytes
    # it must touch over its CUDA-event time, against the measured copy rate
    roof_dec = {"kernel": "decode step (mpc_decode_step: " + ("decode_step_kernel" if step_launches == 1 else
                                                              "select_kernel + attention kernel") + ")", "bound": "hbm", "achieved": round(decode_gbs, 1),
                "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": round(decode_gbs / pk["hbm_gbs"], 4),
                "traffic": None, "peak_source": pk_kind + " hbm_gbs"}
    if not dominant_static:
        roof = roof_dec
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": w.dtype, "data": "synthetic (seeded generator shaped like the paper's models; no datasets or weights)",
        "config": dict(workload_config(w, E, f"replicas{world}"), speculate=args.speculate, fuse=args.fuse),
        # per step: static eviction (two score passes + budget, plus the gather
        # of paged bf16 keys), gathering (+ coarse levels), and per decode step
        # a selection and an attention kernel, or the fused kernel
        "gpu_launches": args.steps * (3 + (1 if w.paged and w.dtype == "bf16" else 0) + 1 +
                                      (1 if len(w.fanouts) else 0) + step_launches * E),
        "static_scoring_path": "tcgen05" if tensor_path else "simt",
        "phases_ms": {"static_evict": static_ms, "build_clusters": build_ms, "decode_all_steps": decode_ms},
        "decode_step_us": decode_ms / E * 1e3,
        "decode_step_us_fused_kernel": fused_us,
        # one launch pair covers every layer, so a layer's share is the mean
        "decode_step_us_per_layer": decode_ms / E * 1e3 / w.n_layers,
        "decode": {"bytes_per_step": dec_bytes / E, "achieved_gbs": round(decode_gbs, 1),
                   "frac_of_measured_hbm": round(decode_gbs / pk["hbm_gbs"], 4),
                   "frac_of_8tbs": round(decode_gbs / 8000.0, 4)},
        "static_scoring_tflops": round(static_tflops, 3),
        "roofline": roof,
        "roofline_decode": roof_dec,
        "clocks": clk,
        "e2e": e2e,
    }
    return line


# ------------------------------------------------------------ reports ----

def decode_timing(w, E, reps=5, calibrate=None):
    """Graph-timed decode of ``w`` after its prefill: the median over ``reps``
    replays of E whole decode steps (mpc_decode_step, every layer) and of E
    standalone selections of the leaders (mpc_select at the prefill's cache).
    ``calibrate(eng, x)`` runs on the prefilled engine before the timing."""
    from paper_2501_06807_gb300 import mpcache
    R, leaders = rules(w)
    x = synth.generate(w, R, device="cuda", decode_steps=E)
    lens = x.prompt_lens.cuda()
    pt = x.page_table.cuda() if x.page_table is not None else None
    eng = make_engine(w, E)

    def prefill():
        eng.prefill(x.k, x.v, x.q_win, lens, pt, w.page_size)

    extra = {}
    if calibrate is not None:
        prefill()
        extra = calibrate(eng, x)
    # attended rows per step (selected clusters + tail), eager pass
    prefill()
    n_keep = eng.n_keep.cpu().tolist()
    attended = 0
    for e in range(E):
        eng.decode_step(x.q[e], x.k_new[e], x.v_new[e])
        n_sel = eng.n_sel.cpu().tolist()
        attended += sum((n_sel[b] * w.cluster_size + (n_keep[b] + e) % w.cluster_size + 1)
                        for b in range(w.batch)) * w.n_layers * w.n_kv_heads
    if mpcache.device_status() != 0:
        raise RuntimeError("device status set by the eager pass")
    ev = lambda: torch.cuda.Event(enable_timing=True)
    stream = torch.cuda.current_stream()

    def timed(body):
        prefill()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            body()
        out = []
        for i in range(reps + 2):
            prefill()
            a, b = ev(), ev()
            a.record(stream)
            g.replay()
            b.record(stream)
            torch.cuda.synchronize()
            if i >= 2:
                out.append(a.elapsed_time(b) * 1e3 / E)
        return statistics.median(out)

    step_us = timed(lambda: [eng.decode_step(x.q[e], x.k_new[e], x.v_new[e]) for e in range(E)])
    sel_us = timed(lambda: [eng.select(x.q[e]) for e in range(E)])
    res = {"decode_step_us": round(step_us, 2), "select_us": round(sel_us, 2), "leaders": len(leaders),
           "attended_rows_per_step": attended / E,
           "scored_rep_rows_per_step": sum(select_rows(w, n_keep[b]) for b in range(w.batch)) * len(leaders) *
           w.n_kv_heads, **extra}
    del eng, x
    torch.cuda.empty_cache()
    return res


def run_report(args):
    from paper_2501_06807_gb300 import build, mpcache
    build.build()
    mpcache.load()
    torch.cuda.set_device(0)
    if args.report == "read-floor":
        import tempfile
        exe = os.path.join(tempfile.mkdtemp(prefix="mpc_floor_"), "bench_floor")
        subprocess.run(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17", "-o", exe,
                        os.path.join(ROOT, "bench_floor.cu")], check=True)
        for w in (synth.C3, synth.C5):
            E = args.decode_steps or w.decode_steps
            keep = mpcache.ppm_count(w.prompt_len, w.keep_ppm)
            s = w.cluster_size
            cap_rows = ((keep + E + s - 1) // s) * s + s  # the engine's cache rows per (layer, kv head)
            clusters = keep // s
            k1 = mpcache.ppm_count(clusters, w.level_keep_ppm[0])
            units = w.n_layers * w.batch * w.n_kv_heads
            r = subprocess.run([exe, str(units), str(clusters), str(k1), str(cap_rows), "6", "4", str(w.seed)],
                               check=True, capture_output=True, text=True)
            print(json.dumps({"report": "read-floor", "workload": w.name, **json.loads(r.stdout)}), flush=True)
        return
    if args.report == "tokenwise":
        # the clustered method and the token-wise comparator (every prompt
        # token kept, one token per cluster) on the same shapes and inputs
        for clustered, tokenwise in ((synth.C3, synth.C3_TOKENWISE), (synth.C5, synth.C5_TOKENWISE)):
            for w in (clustered, tokenwise):
                E = args.decode_steps or w.decode_steps
                r = decode_timing(w, E)
                print(json.dumps({"report": "tokenwise", "workload": w.name, "decode_steps": E,
                                  "cluster_size": w.cluster_size, "keep_ppm": w.keep_ppm,
                                  "fanouts": list(w.fanouts), "level_keep_ppm": list(w.level_keep_ppm), **r}),
                      flush=True)
        return
    # adaptive-sharing: each layer its own leader for a few calibration steps,
    # the commonality of their selected tokens (windows of 2 .. 4 layers), the
    # group size the adaptive rule picks at --share-threshold, then the
    # decode step with no sharing, the picked group size and the workload's
    ms = (1, 2, 3)
    for base in (synth.C2, synth.C3, synth.C5):
        for rho in (0, 950_000):
            w1 = base.replace(share_every=1, layer_rho_ppm=rho)
            E = args.decode_steps or base.decode_steps
            n_cal = min(4, E)

            def calibrate(eng, x):
                acc = {m: [] for m in ms}
                for e in range(n_cal):
                    eng.decode_step(x.q[e], x.k_new[e], x.v_new[e])
                    for m in ms:
                        acc[m].append(float(eng.commonality(m)[1].mean()))
                return {"commonality": {m + 1: round(statistics.mean(v), 4) for m, v in acc.items()}}

            r1 = decode_timing(w1, E, calibrate=calibrate)
            com = {m: r1["commonality"][m + 1] for m in ms}
            chosen = mpcache.choose_share_every(com, args.share_threshold)
            timings = {1: r1}
            for se in sorted({chosen, base.share_every} - {1}):
                timings[se] = decode_timing(base.replace(share_every=se, layer_rho_ppm=rho), E)
            print(json.dumps({"report": "adaptive-sharing", "workload": base.name, "layer_rho_ppm": rho,
                              "calibration_steps": n_cal, "commonality_by_layers": r1["commonality"],
                              "threshold": args.share_threshold, "chosen_share_every": chosen,
                              "fixed_share_every": base.share_every, "decode_steps": E,
                              "decode_step_us": {se: r["decode_step_us"] for se, r in timings.items()},
                              "select_us": {se: r["select_us"] for se, r in timings.items()},
                              "leaders": {se: r["leaders"] for se, r in timings.items()}}), flush=True)


# ------------------------------------------------------ oracle sample ----

def oracle_sample(w, E_sample=4):
    """Times the fp64 oracle on one (leader layer, sequence 0, kv head 0) unit
    of the workload: static scoring, eviction, clustering and E_sample decode
    steps (selection + attention), and extrapolates to the whole job."""
    from oracle import mpcache_oracle as O
    from paper_2501_06807_gb300 import mpcache
    R, leaders = rules(w)
    ws = w.replace(n_layers=1, batch=1)
    x = synth.generate(ws, R, decode_steps=E_sample)
    T = int(x.prompt_lens[0])
    G, d, s = w.group, w.head_dim, w.cluster_size
    kd, vd = x.dense_kv(0, 0)  # dense view (paged workloads keep a page pool)
    K = kd[0, :T].double().numpy()
    V = vd[0, :T].double().numpy()
    wl = O.window_length(T, w.window_ppm, w.long_window_ppm, w.long_prompt_threshold)
    qw = x.q_win[0, 0, :G, R - wl:].double().numpy()
    t0 = time.perf_counter()
    score = O.accumulated_attention(qw, K, 1 / math.sqrt(d))
    kept = O.static_evict(score, O.kept_count(T, w.keep_ppm))
    t1 = time.perf_counter()
    ck, cv = K[kept], V[kept]
    t_dec = 0.0
    t_build = 0.0
    for e in range(E_sample):
        n_tok = len(ck)
        tb = time.perf_counter()
        levels = O.cluster_pyramid(ck, s, w.fanouts, w.alpha)
        t_build += time.perf_counter() - tb
        td = time.perf_counter()
        qg = x.q[e, 0, 0, :G].double().numpy()
        sel = O.hierarchical_select(qg, levels, w.fanouts, w.level_keep_ppm)
        ck = np.vstack([ck, x.k_new[e, 0, 0, 0].double().numpy()[None]])
        cv = np.vstack([cv, x.v_new[e, 0, 0, 0].double().numpy()[None]])
        toks = O.attended_tokens(n_tok, s, sel)
        for g in range(G):
            O.sparse_attention(qg[g], ck[toks], cv[toks], 1 / math.sqrt(d))
        t_dec += time.perf_counter() - td
    t_static = t1 - t0
    E = w.decode_steps
    units = w.batch * w.n_kv_heads
    whole = (t_static * len(leaders) * units + (t_build / E_sample) * len(leaders) * units
             + (t_dec / E_sample) * E * w.n_layers * units)
    n_keep = len(kept)
    k1_of = {}

    def k1(n_tok):
        c1 = n_tok // s
        if c1 not in k1_of:
            zero = O.cluster_pyramid(np.zeros((c1 * s, 1)), s, w.fanouts, w.alpha)
            k1_of[c1] = len(O.hierarchical_select(np.zeros((1, 1)), zero, w.fanouts, w.level_keep_ppm))
        return k1_of[c1]

    tokens = sum(k1(n_keep + e) * s + (n_keep + e) % s + 1 for e in range(E)) * w.n_layers * units
    sample = (f"1 of {len(leaders) * units} leader units static-scored at full T={T} "
              f"({t_static:.1f} s), {E_sample} decode steps of 1 unit; extrapolated to "
              f"{len(leaders)} leaders x {units} (b, kv head) units and {E} steps x {w.n_layers} layers")
    return {"value": tokens / whole, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": sample, "seconds": t1 - t0 + t_build + t_dec, "whole_job_s_estimate": whole}


def cpu_baseline(args):
    """The oracle sample on all host cores (numpy's BLAS threads), and again
    in a child process limited to one thread, each with its core count."""
    allc = oracle_sample(workload_of(args))
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               BLIS_NUM_THREADS="1", VECLIB_MAXIMUM_THREADS="1", NUMEXPR_NUM_THREADS="1")
    try:
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-sample", "--workload", args.workload,
                            *override_argv(args)],
                           env=env, capture_output=True, text=True, timeout=600)
        one = json.loads(r.stdout.strip().splitlines()[-1])
        allc["single_thread"] = {"value": one["value"], "unit": one["unit"], "cores": 1,
                                 "seconds": one["seconds"], "whole_job_s_estimate": one["whole_job_s_estimate"]}
    except Exception as e:  # the all-core figure stands on its own
        allc["single_thread"] = {"unavailable": f"{type(e).__name__}: {e}"[:200]}
    return allc


def workload_config(w, E, parallelism):
    """The bench line's ``config``: the workload by its sizes (both arms)."""
    kv_gb = 2 * w.n_layers * w.batch * w.n_kv_heads * w.prompt_len * w.head_dim * (2 if w.dtype == "bf16" else 4) / 1e9
    return {"workload": w.name, "layers": w.n_layers, "batch": w.batch, "q_heads": w.n_q_heads,
            "kv_heads": w.n_kv_heads, "head_dim": w.head_dim, "prompt_len": w.prompt_len,
            "decode_steps": E, "cluster_size": w.cluster_size, "fanouts": list(w.fanouts),
            "level_keep_ppm": list(w.level_keep_ppm), "keep_ppm": w.keep_ppm,
            "share_every": w.share_every, "alpha": w.alpha, "window_ppm": w.window_ppm,
            "long_window_ppm": w.long_window_ppm, "layer_rho_ppm": w.layer_rho_ppm,
            "paged": w.paged, "parallelism": parallelism,
            "l2": "inputs larger than L2 (prompt KV up to %.1f GB per step)" % kv_gb}


def run_reference(args, rank, world):
    if rank != 0:
        return None
    w = workload_of(args)
    for _ in range(args.warmup):
        oracle_sample(w, E_sample=1)
    vals, secs, whole = [], [], []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        r = oracle_sample(w, E_sample=2)
        secs.append(time.perf_counter() - t0)
        vals.append(r["value"])
        whole.append(r["whole_job_s_estimate"])
    v = statistics.median(vals)
    # a step is one bounded sample of the job (ms_per_step is its measured
    # time); the whole job's estimated time is reported beside it
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": statistics.median(secs) * 1e3,
            "whole_job_ms_estimate": statistics.median(whole) * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(w, args.decode_steps or w.decode_steps, "cpu"),
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                             "sample": r["sample"]},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    dist = None
    if world > 1:
        import torch.distributed as tdist
        backend = "nccl" if torch.cuda.is_available() and args.impl == "ours" else "gloo"
        if args.impl == "ours":
            torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        tdist.init_process_group(backend)
        dist = tdist
    if args.oracle_sample:
        print(json.dumps(oracle_sample(workload_of(args))), flush=True)
        return
    if args.report:
        if rank == 0 and world == 1:
            run_report(args)
        return
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        line = run_ours(args, rank, world, dist)
        if rank == 0 and world == 1:
            line["cpu_baseline"] = cpu_baseline(args)
    if rank == 0 and line is not None:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
