#!/usr/bin/env python3
"""Benchmark of the CompressKV prefill KV-compression step on GB300.

One step = ckv_compress_layer (score + pool + top-k + gather) for every layer of the
needle-style long-prefix workload (Llama-3.1-8B-shaped: 32 layers, 32 query / 8 KV heads,
d = 128, one sequence of 131072 prefix tokens with a planted 64-token span, w = 32, 2 selected
heads per group, max-pool 7, 128 tokens kept per KV head), on synthetic seeded inputs already
resident in HBM.  Each layer has its own K/V/Q buffers, so one step streams far more than the
129 MB L2; the step is replayed from a CUDA graph.  `--workload` picks another workload.

Prints one JSON line (rank 0).  `--impl reference` times the fp64 CPU oracle instead (the
reference arm of this build) on whole layers of the same workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
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

METRIC = "KV-compress prefix tokens/s per layer (score+topk+gather); % of HBM peak"
UNIT = "prefix tokens/s per layer"
WORKLOAD = "needle_l131072"
HBM_FALLBACK_GBS = 6800.0

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) of the scoring kernel per layer, per
# workload, from an ncu capture of a two-layer launch of the same kernel (bench.py --layers 2 on
# the workload), halved; keyed by the sha256 of the scoring kernels' sources (SCORE_SOURCES), so
# a changed kernel reports null until it is captured again.  Rounded to 10 kB.
SCORE_SOURCES = ('score_layers.cu', 'score_layers.cuh', 'score_resident.cu', 'score_lse.cu', 'score_common.cuh',
                 'ckv_device.cuh')
SCORE_TRAFFIC = {
    "2420f73d42000877d15e1e55b8936cf6b89b5eaa3076715573ec3b7a0d634c9a": {
        "needle_l131072": 362_430_000,
        "llama8b_l32768": 73_830_000,
        "ragged_qwen7b": 223_730_000,
        "needle_l131072+lse": 272_310_000,
        "llama8b_l32768+lse": 69_040_000,
        "ragged_qwen7b+lse": 174_490_000,
    },
}
# Sequences up to this many tokens are selected by one block per (sequence, KV head)
# (one launch); longer ones by the chunked kernels (two launches).
SELECT_UNIT_LEN = 16384


def _window_lse(q, k, cu_seqlens, w, Hq, Hkv):
    """The window rows' lse, [Hq, S*w] fp32 natural log, as a prefill attention kernel returns
    it: log sum_{j <= P+r} exp(q_r.k_j / sqrt(d)) (NaN for rows before the sequence start).
    Plain PyTorch, for preparing the input of the given-lse path."""
    import torch
    S = len(cu_seqlens) - 1
    G = Hq // Hkv
    d = q.shape[-1]
    out = torch.full((Hq, S * w), float("nan"), dtype=torch.float32, device=q.device)
    for s in range(S):
        t0, t1 = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        L, P = t1 - t0, t1 - t0 - w
        if L <= 0:
            continue
        for h in range(Hq):
            qs = q[s, :, h].float()                       # [w, d]
            ks = k[t0:t1, h // G].float()                 # [L, d]
            logits = (qs @ ks.T) / (d ** 0.5)            # [w, L]
            j = torch.arange(L, device=q.device)[None, :]
            r = torch.arange(w, device=q.device)[:, None]
            logits = logits.masked_fill(j > P + r, float("-inf"))
            lse = torch.logsumexp(logits, dim=1)
            lse[P + torch.arange(w, device=q.device) < 0] = float("nan")
            out[h, s * w:(s + 1) * w] = lse
    return out


def _args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--min-seconds", type=float, default=1.0,
                    help="the K-step timed region is repeated until this much GPU time has been "
                         "timed (at least 3 times); the median repetition is reported")
    ap.add_argument("--layers", type=int, default=0, help="use only the first N layers (0 = all)")
    ap.add_argument("--breakdown", action="store_true", help="per-stage times on stderr")
    ap.add_argument("--score-path", choices=("auto", "resident", "reload"), default="auto",
                    help="scoring kernel: logits kept in TMEM, K re-read in pass 2, or the "
                         "library's choice")
    ap.add_argument("--srs", action="store_true",
                    help="time the Semantic Retrieval Score accumulation (Eq. 5) instead: every "
                         "head scored, the window rows as decode steps, all of them in the answer")
    ap.add_argument("--calls", choices=("layers", "layer"), default="layers",
                    help="layers: one ckv_compress_layers call over every layer of the step (one "
                         "persistent scoring launch, then the selections); layer: one "
                         "ckv_compress_layer call per layer, layers round-robin on streams")
    ap.add_argument("--split-select", action="store_true",
                    help="with --calls layer: each layer as ckv_score_window then "
                         "ckv_select_compact, the selection on a stream of its own, so that the "
                         "next layer's scoring need not wait")
    ap.add_argument("--lse", action="store_true",
                    help="the window rows' lse given (as a prefill attention kernel returns it): "
                         "ckv_compress_layers_lse (with --calls layer: ckv_compress_layer_lse), "
                         "one pass over K")
    ap.add_argument("--max-ctas", type=int, default=0,
                    help="CTAs one call's scoring kernel may occupy (0: all SMs with --calls "
                         "layers; SMs / streams with --calls layer, so that one scoring kernel "
                         "per stream is resident at once)")
    ap.add_argument("--streams", type=int, default=0,
                    help="layers are issued round-robin on this many streams (one workspace each); "
                         "0 = min(layers, 16)")
    return ap.parse_args()


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return HBM_FALLBACK_GBS, "fallback"


def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


# Replicas only: the ranks share nothing in the data path; they meet for the barriers around
# the timed region and for the maximum of their times.
def _rank_barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def _max_over_ranks(ms, world, device):
    """The largest of the ranks' times (every rank gets it)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _job_throughput(world, units_per_rank, ms_per_step):
    """Whole-job units per second: every rank processes its own units in the slowest rank's time."""
    return world * units_per_rank / (ms_per_step / 1e3)


def _workload_config(wl, world):
    """The workload both arms run, as the `config` of their JSON lines."""
    d = wl.head_dim
    per_layer = (wl.num_seqs * wl.window * wl.num_q_heads * d + 2 * wl.total_tokens * wl.num_kv_heads * d) * 2
    step_gb = per_layer * wl.num_layers / 1e9
    return {"workload": wl.name, "layers": wl.num_layers, "seq_len": wl.total_tokens,
            "seqs": wl.num_seqs, "q_heads": wl.num_q_heads, "kv_heads": wl.num_kv_heads,
            "head_dim": d, "window": wl.window, "heads_per_group": wl.heads_per_group,
            "heads_per_layer": wl.heads_per_layer, "scope": wl.scope,
            "pool": f"{wl.pool_type}{wl.pool_kernel}", "head_order": wl.head_order,
            "budget_total": int(wl.budgets().sum()), "parallelism": f"replicas{world}",
            "l2": f"inputs larger than L2 (distinct per-layer buffers, {step_gb:.2f} GB per step)"}


# ----------------------------------------------------------------------------- clocks
_REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
            0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
            0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
            0x100: "display_clock_setting"}


class ClockSampler:
    def __init__(self, device_index: int):
        self.path = tempfile.mktemp(prefix="ckv_clocks_", suffix=".csv")
        self.dev = device_index
        self.proc = None

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev),
                 "--query-gpu=clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 4:
                    continue
                try:
                    rows.append((float(parts[0]), float(parts[1]), float(parts[2]), int(parts[3], 16)))
                except ValueError:
                    continue
        finally:
            try:
                os.unlink(self.path)
            except OSError:
                pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        busy = [r for r in rows if not (r[3] & 0x1)] or rows
        reasons = sorted({name for r in busy for bit, name in _REASONS.items()
                          if r[3] & bit and bit != 0x1})
        return {"sm_mhz": statistics.median(r[0] for r in busy), "sm_max_mhz": max(r[1] for r in rows),
                "power_w_max": max(r[2] for r in rows), "reasons": reasons, "samples": len(busy)}


# ----------------------------------------------------------------------------- our arm
def run_ours(args):
    import numpy as np
    import torch

    import ckv_synth as cs
    import __graft_entry__ as entry

    rank, world, local = _dist()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    entry.build()
    import paper_2508_02401_gb300 as ckv

    wl = cs.workload(args.workload)
    if args.layers:
        wl = wl.with_(num_layers=args.layers)
    path = {"auto": ckv.SCORE_AUTO, "resident": ckv.SCORE_RESIDENT, "reload": ckv.SCORE_RELOAD}[args.score_path]
    cfg = ckv.Config.from_workload(wl, score_path=path)
    batch = ckv.Batch(wl.cu_seqlens(), device=f"cuda:{local}")
    T, Hkv, nl = wl.total_tokens, wl.num_kv_heads, wl.num_layers

    def dev(bits):
        return torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)

    layers = []
    host_layers = []
    for l in range(nl):
        li = wl.layer(l)
        host_layers.append(li)
        idx, cu_keep_dev, k_out, v_out, cu_keep = ckv.new_outputs(cfg, l, batch)
        layers.append(dict(q=dev(li.q_win), k=dev(li.k), v=dev(li.v), idx=idx, cu_keep_dev=cu_keep_dev,
                           k_out=k_out, v_out=v_out, t_keep=int(cu_keep[-1])))
        if args.lse:  # input preparation, outside every timed region
            layers[-1]["lse"] = _window_lse(layers[-1]["q"], layers[-1]["k"], wl.cu_seqlens(), wl.window,
                                            wl.num_q_heads, Hkv)
    ws_bytes = max(ckv.ckv_workspace_size(cfg, l, batch) for l in range(nl))
    # Layers are independent: by default they go round-robin on min(layers, 16) streams, and
    # each call's scoring kernel is capped at SMs / streams CTAs, so that one per stream is
    # resident at once (in even waves: a stream's next layer starts when its previous one is
    # done) and the SMs they leave free run the selections in between.
    nstreams = args.streams if args.streams > 0 else min(nl, 16)
    sms = torch.cuda.get_device_properties(local).multi_processor_count
    cap = args.max_ctas if args.max_ctas > 0 else max(1, sms // nstreams)
    cfg = ckv.Config.from_workload(wl, max_ctas=cap, score_path=path)
    wss = [torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda") for _ in range(nstreams)]
    ws = wss[0]
    stream = torch.cuda.Stream()
    side = [torch.cuda.Stream() for _ in range(nstreams)]
    if args.split_select:  # per layer a score buffer; per stream a selection stream + workspace
        sel_side = [torch.cuda.Stream() for _ in range(nstreams)]
        sel_wss = [torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda") for _ in range(nstreams)]
        n_sel_max = max(ckv.ckv_keep_lengths(cfg, l, batch)[1] for l in range(nl))
        for d in layers:
            d["scores"] = torch.empty((n_sel_max, T), dtype=torch.float32, device="cuda")

    # One call for every layer of the step: ckv_compress_layers (the layers' scoring in one
    # persistent launch over all SMs, then the selections), with the window rows' lse computed.
    multi = args.calls == "layers" and not args.split_select
    if multi:
        cap = args.max_ctas if args.max_ctas > 0 else 0
        cfg = ckv.Config.from_workload(wl, max_ctas=cap, score_path=path)
        nstreams = 1
        ios = [ckv.LayerIO(layer=l, q_win=d["q"], k=d["k"], v=d["v"], idx=d["idx"],
                           cu_keep_dev=d["cu_keep_dev"], k_out=d["k_out"], v_out=d["v_out"],
                           lse=d.get("lse"))
               for l, d in enumerate(layers)]
        compress_layers = ckv.ckv_compress_layers_lse if args.lse else ckv.ckv_compress_layers
        wss = [ckv.new_layers_workspace(cfg, ios, batch)]
        ws = wss[0]

    def over_layers(fn, selections=False):
        # Layers are independent: layer l runs on side stream l % nstreams with its own
        # workspace, so the calls of consecutive layers overlap on the GPU (and, with
        # `selections`, its selection on the matching selection stream).
        for sd in side:
            sd.wait_stream(stream)
        for l, d in enumerate(layers):
            fn(l, d, wss[l % nstreams], side[l % nstreams])
        for sd in side + (sel_side if selections else []):
            stream.wait_stream(sd)

    def compress(l, d, w, st):
        if args.split_select:
            i = l % nstreams
            if args.lse:
                ckv.ckv_score_window_lse(cfg, l, batch, d["q"], d["k"], d["lse"], d["scores"], w,
                                         stream=st)
            else:
                ckv.ckv_score_window(cfg, l, batch, d["q"], d["k"], d["scores"], w, stream=st)
            ev = torch.cuda.Event()
            ev.record(st)
            sel_side[i].wait_event(ev)
            ckv.ckv_select_compact(cfg, l, batch, d["scores"], d["k"], d["v"], d["idx"],
                                   d["cu_keep_dev"], d["k_out"], d["v_out"], sel_wss[i],
                                   stream=sel_side[i])
            return sel_side[i]  # the stream on which the layer's outputs are complete
        if args.lse:
            ckv.ckv_compress_layer_lse(cfg, l, batch, d["q"], d["k"], d["v"], d["lse"], d["idx"],
                                       d["cu_keep_dev"], d["k_out"], d["v_out"], w, stream=st)
        else:
            ckv.ckv_compress_layer(cfg, l, batch, d["q"], d["k"], d["v"], d["idx"], d["cu_keep_dev"],
                                   d["k_out"], d["v_out"], w, stream=st)
        return st

    def step():
        if multi:
            compress_layers(cfg, ios, batch, ws, stream=stream)
        else:
            over_layers(compress, selections=args.split_select)

    with torch.cuda.stream(stream):
        for _ in range(max(1, args.warmup)):
            step()
    torch.cuda.synchronize()
    for w in wss + (sel_wss if args.split_select else []):
        code, detail = ckv.ckv_read_device_status(w, stream=stream)
        if code != 0:
            raise RuntimeError(f"device status {code} ({detail}) after warm-up")

    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step()
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            graph.replay()
    torch.cuda.synchronize()

    def barrier():
        _rank_barrier(world)

    # The timed region: exactly `steps` graph replays between a barrier and a synchronize on
    # both sides, repeated until at least `min_seconds` of GPU time (and 3 repetitions) so
    # that the clock sampler sees the GPU under load; the median repetition is reported.
    reps_ms = []
    with ClockSampler(local) as clk:
        while len(reps_ms) < 3 or sum(reps_ms) < 1e3 * args.min_seconds:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            barrier()
            torch.cuda.synchronize()
            with torch.cuda.stream(stream):
                e0.record(stream)
                for _ in range(args.steps):
                    graph.replay()
                e1.record(stream)
            torch.cuda.synchronize()
            barrier()
            reps_ms.append(_max_over_ranks(e0.elapsed_time(e1), world, "cuda"))
            if len(reps_ms) >= 1000:
                break
    ms = statistics.median(reps_ms)
    clocks = clk.summary()
    for w in wss + (sel_wss if args.split_select else []):
        code, detail = ckv.ckv_read_device_status(w, stream=stream)
        if code != 0:
            raise RuntimeError(f"device status {code} ({detail}) after the timed region")
    ms_per_step = ms / args.steps
    value = _job_throughput(world, nl * T, ms_per_step)

    # --- the same step issued eagerly (no graph): the host's wall time per call (argument
    # checks, planning, tensor-map encoding and the launches, through the Python binding) and
    # the GPU time of a step issued that way.
    eager_reps = 3
    host_s = []
    ea, eb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        ea.record(stream)
        for _ in range(eager_reps):
            t_issue = time.perf_counter()
            step()
            host_s.append(time.perf_counter() - t_issue)
        eb.record(stream)
    torch.cuda.synchronize()
    eager = {"host_us_per_call": round(statistics.median(host_s) / nl * 1e6, 2),
             "gpu_ms_per_step": round(ea.elapsed_time(eb) / eager_reps, 5)}

    # per layer: the scoring kernel, then the selection (pool, top-k, compaction and gather)
    lens = list(wl.seqlens)
    sel_per_layer = (1 if min(lens) <= SELECT_UNIT_LEN else 0) + (2 if max(lens) > SELECT_UNIT_LEN else 0)
    if multi:  # per 32 layers one scoring launch (two-pass, or single-pass with the lse given)
        # and one selection launch (the workloads here fit one launch's unit table; the
        # counter resets are memsets, not kernels)
        launches_per_step = 2 * -(-nl // 32)
    else:
        launches_per_step = (1 + sel_per_layer) * nl

    # --- scoring stage (the dominant kernels): a graph of every layer's ckv_score_window,
    # timed with events on its stream; the average per layer is one pass-1 + pass-2 pair.
    hbm_peak, peak_kind = _peaks()
    n_sel = int(cfg.head_mask[0].sum())
    score_rows = [torch.empty((int(cfg.head_mask[l].sum()), T), dtype=torch.float32, device="cuda")
                  for l in range(nl)]
    pooled_rows = [torch.empty((Hkv, T), dtype=torch.float32, device="cuda") for _ in range(nl)]

    def stage(fn):
        with torch.cuda.stream(stream):
            fn()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        reps = 20
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            g.replay()
            a.record(stream)
            for _ in range(reps):
                g.replay()
            b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps / nl  # ms per layer

    def score_one(l, d, w, st):
        if args.lse:
            ckv.ckv_score_window_lse(cfg, l, batch, d["q"], d["k"], d["lse"], score_rows[l], w, stream=st)
        else:
            ckv.ckv_score_window(cfg, l, batch, d["q"], d["k"], score_rows[l], w, stream=st)

    def score_all():
        if multi and args.lse:
            ckv.ckv_score_windows_lse(cfg, score_ios, batch, ws, stream=stream)
        elif multi:
            ckv.ckv_score_windows(cfg, score_ios, batch, ws, stream=stream)
        else:
            over_layers(score_one)

    if multi:
        score_ios = [ckv.LayerIO(layer=l, q_win=d["q"], k=d["k"], scores=score_rows[l],
                                 lse=d["lse"] if args.lse else None)
                     for l, d in enumerate(layers)]

    score_ms = stage(score_all)
    if args.breakdown:
        def pool_all():
            over_layers(lambda l, d, w, st: ckv.ckv_pool(cfg, l, batch, score_rows[l],
                                                         pooled_rows[l], stream=st))

        def select_all():
            over_layers(lambda l, d, w, st: ckv.ckv_select_topk(
                cfg, l, batch, pooled_rows[l], d["idx"], d["cu_keep_dev"], w, stream=st))

        def gather_all():
            over_layers(lambda l, d, w, st: ckv.ckv_gather_compact(
                cfg, batch, d["t_keep"], d["k"], d["v"], d["idx"], d["cu_keep_dev"], d["k_out"],
                d["v_out"], w, stream=st))
        parts = {"score": score_ms, "pool": stage(pool_all), "select": stage(select_all),
                 "gather": stage(gather_all), "step": ms_per_step / nl}
        print("per-layer stage times (us): " + ", ".join(f"{k}={v * 1e3:.2f}" for k, v in parts.items()),
              file=sys.stderr, flush=True)
    # K is read once per (token, KV head) whose group has a selected head in the layer
    G = wl.num_q_heads // Hkv
    scored = [int((cfg.head_mask[l].reshape(Hkv, G) != 0).any(axis=1).sum()) for l in range(nl)]
    k_bytes = T * 256 * sum(scored) / nl
    score_gbs = k_bytes / (score_ms / 1e3) / 1e9
    digest = hashlib.sha256()
    for f in SCORE_SOURCES:
        digest.update(open(os.path.join(ROOT, "paper_2508_02401_gb300", "csrc", f), "rb").read())
    traffic = SCORE_TRAFFIC.get(digest.hexdigest(), {}).get(args.workload + ("+lse" if args.lse else ""))
    kernel_desc = ("single-pass scoring kernel (ckv_score_windows_lse): every layer of the step "
                   f"in one persistent launch on {cap or sms} CTAs; per layer" if multi and args.lse else
                   "two-pass scoring kernel (ckv_score_windows): every layer of the step in one "
                   f"persistent launch on {cap or sms} CTAs; per layer" if multi else
                   "scoring kernel (ckv_score_window), per layer, layers overlapped on "
                   f"{nstreams} streams, {cap} CTAs per call")
    roofline = {"bound": "hbm", "kernel": kernel_desc,
                "achieved": round(score_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                "frac": round(score_gbs / hbm_peak, 4), "peak_kind": peak_kind,
                "frac_of_8TBs": round(score_gbs / 8000.0, 4),
                "traffic": traffic, "algorithmic_bytes_per_launch": int(k_bytes),
                "avg_launch_us": round(score_ms * 1e3, 2)}
    keep_bytes = sum(4 * 256 * Hkv * d["t_keep"] for d in layers) / nl
    layer_bytes = k_bytes + keep_bytes
    layer_gbs = layer_bytes / (ms_per_step / nl / 1e3) / 1e9

    # --- end to end through the public API from pinned host memory
    e2e = None
    if args.e2e_steps > 0:
        hq = [torch.from_numpy(h.q_win.view(np.int16)).view(torch.bfloat16).pin_memory() for h in host_layers]
        hk = [torch.from_numpy(h.k.view(np.int16)).view(torch.bfloat16).pin_memory() for h in host_layers]
        hv = [torch.from_numpy(h.v.view(np.int16)).view(torch.bfloat16).pin_memory() for h in host_layers]
        hl = [d["lse"].cpu().pin_memory() for d in layers] if args.lse else []
        oi = [torch.empty(d["idx"].shape, dtype=torch.int32, pin_memory=True) for d in layers]
        ok = [torch.empty(d["k_out"].shape, dtype=torch.bfloat16, pin_memory=True) for d in layers]
        ov = [torch.empty(d["v_out"].shape, dtype=torch.bfloat16, pin_memory=True) for d in layers]
        h2d = sum(x.numel() * 2 for x in hq + hk + hv) + sum(x.numel() * 4 for x in hl)
        d2h = sum(x.numel() * x.element_size() for x in oi + ok + ov)

        # Per layer: its inputs on one of two copy streams, its compression on its own stream once
        # they have landed, its outputs back on a read-back stream once it is done; the copies of
        # one layer overlap the other layers' compressions.
        copy_streams = [torch.cuda.Stream() for _ in range(2)]
        back = torch.cuda.Stream()
        every = copy_streams + side + [back] + (sel_side if args.split_select else [])

        E = 4  # layers per ckv_compress_layers call in the end-to-end step

        def e2e_step_multi():
            # Per chunk of E layers: its inputs on one of two copy streams, one
            # ckv_compress_layers call on the compute stream once they have landed, its outputs
            # back on the read-back stream; the copies overlap the other chunks' compressions.
            for st in copy_streams + [back]:
                st.wait_stream(stream)
            for c0 in range(0, nl, E):
                cp = copy_streams[(c0 // E) % len(copy_streams)]
                with torch.cuda.stream(cp):
                    for l in range(c0, min(nl, c0 + E)):
                        d = layers[l]
                        d["q"].copy_(hq[l], non_blocking=True)
                        d["k"].copy_(hk[l], non_blocking=True)
                        d["v"].copy_(hv[l], non_blocking=True)
                        if args.lse:
                            d["lse"].copy_(hl[l], non_blocking=True)
                landed = torch.cuda.Event()
                landed.record(cp)
                stream.wait_event(landed)
                compress_layers(cfg, ios[c0:c0 + E], batch, ws, stream=stream)
                done = torch.cuda.Event()
                done.record(stream)
                back.wait_event(done)
                with torch.cuda.stream(back):
                    for l in range(c0, min(nl, c0 + E)):
                        oi[l].copy_(layers[l]["idx"], non_blocking=True)
                        ok[l].copy_(layers[l]["k_out"], non_blocking=True)
                        ov[l].copy_(layers[l]["v_out"], non_blocking=True)
            for st in copy_streams + [back]:
                stream.wait_stream(st)

        def e2e_step():
            if multi:
                e2e_step_multi()
                return
            for st in every:
                st.wait_stream(stream)
            for l, d in enumerate(layers):
                cp = copy_streams[l % len(copy_streams)]
                with torch.cuda.stream(cp):
                    d["q"].copy_(hq[l], non_blocking=True)
                    d["k"].copy_(hk[l], non_blocking=True)
                    d["v"].copy_(hv[l], non_blocking=True)
                    if args.lse:
                        d["lse"].copy_(hl[l], non_blocking=True)
                landed = torch.cuda.Event()
                landed.record(cp)
                st = side[l % nstreams]
                st.wait_event(landed)
                out_st = compress(l, d, wss[l % nstreams], st)
                done = torch.cuda.Event()
                done.record(out_st)
                back.wait_event(done)
                with torch.cuda.stream(back):
                    oi[l].copy_(d["idx"], non_blocking=True)
                    ok[l].copy_(d["k_out"], non_blocking=True)
                    ov[l].copy_(d["v_out"], non_blocking=True)
            for st in every:
                stream.wait_stream(st)

        with torch.cuda.stream(stream):
            for _ in range(2):
                e2e_step()
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(args.e2e_steps):
                e2e_step()
            b.record(stream)
        torch.cuda.synchronize()
        e2e_ms = a.elapsed_time(b) / args.e2e_steps
        h2d_peak = _h2d_peak(torch, stream)
        h2d_gbs = h2d / (e2e_ms / 1e3) / 1e9
        e2e = {"value": world * nl * T / (e2e_ms / 1e3), "unit": UNIT, "ms_per_step": round(e2e_ms, 4),
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "h2d_gbs": round(h2d_gbs, 1), "h2d_peak_gbs": round(h2d_peak, 1),
               "frac_of_h2d_peak": round(h2d_gbs / h2d_peak, 4)}

    cpu = None
    if rank == 0 and world == 1 and args.cpu_seconds > 0:
        cpu = _cpu_baseline(wl, host_layers, args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": _workload_config(wl, world),
            "run": {"graph": "one CUDA graph per step",
                    "streams": ("one stream" if multi else
                                f"layers round-robin on {nstreams} streams, scoring capped at {cap} CTAs per call"),
                    "lse": ("window-row lse given (PyTorch logsumexp outside the timed region; "
                            "one pass over K)") if args.lse else "computed (two passes)",
                    "calls": (("ckv_compress_layers_lse" if args.lse else "ckv_compress_layers") +
                              " over every layer of the step" if multi else
                              "ckv_score_window + ckv_select_compact, the selection on a stream "
                              "of its own" if args.split_select else "ckv_compress_layer per layer"),
                    "repetitions": len(reps_ms),
                    "ms_per_step_spread": {"min": round(min(reps_ms) / args.steps, 5),
                                           "median": round(ms_per_step, 5),
                                           "max": round(max(reps_ms) / args.steps, 5)},
                    "timed_gpu_s": round(sum(reps_ms) / 1e3, 3),
                    "eager": eager},
            "roofline": roofline,
            "layer_roofline": {"bound": "hbm", "achieved": round(layer_gbs, 1), "peak": hbm_peak,
                               "unit": "GB/s", "frac": round(layer_gbs / hbm_peak, 4),
                               "frac_of_8TBs": round(layer_gbs / 8000.0, 4),
                               "algorithmic_bytes_per_layer": int(layer_bytes)},
            "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks,
            "gpu_launches": launches_per_step * args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def _h2d_peak(torch, stream, nbytes=1 << 30, reps=5):
    """A plain host-to-device copy of one pinned 1 GiB buffer: the best of `reps`, in GB/s."""
    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    d = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    best = float("inf")
    with torch.cuda.stream(stream):
        for _ in range(reps):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            d.copy_(h, non_blocking=True)
            b.record(stream)
            torch.cuda.synchronize()
            best = min(best, a.elapsed_time(b))
    del h, d
    return nbytes / (best / 1e3) / 1e9


# ----------------------------------------------------------------------------- the oracle
def _oracle_cores(wl, threads):
    """Threads that the oracle keeps busy: it runs OpenMP over (sequence, selection) units."""
    units = wl.num_seqs * (1 if wl.scope == "layer" else wl.num_kv_heads)
    return min(threads, units)


def _cpu_baseline(wl, host_layers, seconds):
    """The fp64 oracle as it stands, whole layers in order until `seconds` have passed."""
    import oracle
    oracle.build()
    cores = _oracle_cores(wl, oracle.threads(0))
    t0 = time.perf_counter()
    done = 0
    while True:  # sweeps of the layers, in order, until `seconds` have passed
        l = done % len(host_layers)
        li = host_layers[l]
        oracle.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), wl.head_mask()[l],
                              int(wl.budgets()[l]), wl.window, wl.pool_kernel,
                              0 if wl.pool_type == "max" else 1,
                              0 if wl.head_order == "pool_then_sum" else 1,
                              scope=1 if wl.scope == "layer" else 0)
        done += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    return {"value": round(done * wl.total_tokens / dt, 2), "unit": UNIT, "cores": cores,
            "kind": "oracle", "sample": f"{done} whole-layer calls (layers in order), {dt:.1f} s, "
                                        f"OpenMP over (sequence, selection) units: {cores} of "
                                        f"{oracle.threads(0)} host threads busy"}


def run_reference(args):
    """The reference arm: the fp64 oracle as it stands, on all host cores, one whole layer of the
    workload per step (cycling over its first four layers), as the GPU line's cpu_baseline."""
    rank, world, local = _dist()
    if rank != 0:
        return
    import ckv_synth as cs
    import oracle
    oracle.build()
    wl = cs.workload(args.workload)
    if args.layers:
        wl = wl.with_(num_layers=args.layers)
    cores = _oracle_cores(wl, oracle.threads(0))
    masks, budgets, cu = wl.head_mask(), wl.budgets(), wl.cu_seqlens()
    cache = {}
    n_distinct = min(wl.num_layers, 4)

    def sample(i):
        l = i % n_distinct
        if l not in cache:
            cache[l] = wl.layer(l)
        li = cache[l]
        t = time.perf_counter()
        oracle.compress_layer(li.q_win, li.k, li.v, cu, masks[l], int(budgets[l]), wl.window,
                              wl.pool_kernel, 0 if wl.pool_type == "max" else 1,
                              0 if wl.head_order == "pool_then_sum" else 1,
                              scope=1 if wl.scope == "layer" else 0)
        return time.perf_counter() - t

    for i in range(args.warmup):
        sample(i)
    times = [sample(args.warmup + i) for i in range(args.steps)]
    per_layer = statistics.mean(times)
    value = wl.total_tokens / per_layer
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(per_layer * 1e3, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": _workload_config(wl, world),
            "cpu_baseline": {"value": round(value, 2), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"one whole layer per step (layers 0..{n_distinct - 1} in turn), "
                                       f"OpenMP over (sequence, selection) units: {cores} of "
                                       f"{oracle.threads(0)} host threads busy"},
            "e2e": {"value": round(value, 2), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_srs(args):
    """ckv_semantic_retrieval_scores over every layer of the workload: the window queries act as
    the decode steps (all flagged as answer tokens), the answer span is 64 positions from a third
    of each sequence, every query head is scored.  One JSON line; 1 GPU."""
    import numpy as np
    import torch

    import __graft_entry__ as entry
    import ckv_synth as cs
    entry.build()
    import paper_2508_02401_gb300 as ckv

    wl = cs.workload(args.workload)
    if args.layers:
        wl = wl.with_(num_layers=args.layers)
    nl, T, Hkv, Hq = wl.num_layers, wl.total_tokens, wl.num_kv_heads, wl.num_q_heads
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    nstreams = args.streams if args.streams > 0 else min(nl, 16)
    cap = args.max_ctas if args.max_ctas > 0 else max(1, sms // nstreams)
    cfg = ckv.Config.from_workload(wl, head_mask=np.ones((nl, Hq), np.uint8), max_ctas=cap)
    batch = ckv.Batch(wl.cu_seqlens())
    cu = wl.cu_seqlens()
    lens = np.diff(cu)
    span = torch.from_numpy(np.array([[L // 3, min(L, L // 3 + 64)] for L in lens], np.int32)).cuda()
    flags = torch.ones(wl.num_seqs * wl.window, dtype=torch.uint8, device="cuda")
    layers = []
    for l in range(nl):
        li = wl.layer(l)
        q = torch.from_numpy(li.q_win.view(np.int16)).cuda().view(torch.bfloat16)
        k = torch.from_numpy(li.k.view(np.int16)).cuda().view(torch.bfloat16)
        layers.append(dict(q=q, k=k, lse=_window_lse(q, k, cu, wl.window, Hq, Hkv)))
    srs = torch.zeros(Hq, dtype=torch.float32, device="cuda")
    ws_bytes = max(ckv.ckv_workspace_size(cfg, l, batch) for l in range(nl))
    wss = [torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda") for _ in range(nstreams)]
    stream = torch.cuda.Stream()
    side = [torch.cuda.Stream() for _ in range(nstreams)]

    def step():
        for sd in side:
            sd.wait_stream(stream)
        for l, d in enumerate(layers):
            ckv.ckv_semantic_retrieval_scores(cfg, l, batch, d["q"], d["k"], d["lse"], flags, span, srs,
                                              wss[l % nstreams], stream=side[l % nstreams])
        for sd in side:
            stream.wait_stream(sd)

    with torch.cuda.stream(stream):
        for _ in range(max(1, args.warmup)):
            step()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step()
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clk:
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                graph.replay()
            e1.record(stream)
        torch.cuda.synchronize()
    for w in wss:
        code, detail = ckv.ckv_read_device_status(w, stream=stream)
        if code != 0:
            raise RuntimeError(f"device status {code} ({detail}) after the timed region")
    ms_per_step = e0.elapsed_time(e1) / args.steps
    hbm_peak, peak_kind = _peaks()
    k_bytes = T * Hkv * 256  # K read once per (token, KV head): the floor; each head batch reads it
    gbs = k_bytes * nl / (ms_per_step / 1e3) / 1e9
    line = {
        "metric": "SRS accumulation (Eq. 5) prefix tokens/s per layer", "value": round(nl * T / (ms_per_step / 1e3), 1),
        "unit": UNIT, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": wl.name, "layers": nl, "seq_len": T, "q_heads": Hq, "kv_heads": Hkv,
                   "decode_steps": wl.window, "heads_scored": Hq,
                   "streams": f"layers round-robin on {nstreams} streams, scoring capped at {cap} CTAs per call"},
        "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                     "frac": round(gbs / hbm_peak, 4), "peak_kind": peak_kind, "traffic": None,
                     "algorithmic_bytes_per_layer": k_bytes},
        "clocks": clk.summary(), "gpu_launches": 3 * nl * args.steps,
    }
    print(json.dumps(line), flush=True)


def main():
    args = _args()
    if args.impl == "reference":
        run_reference(args)
    elif args.srs:
        run_srs(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
