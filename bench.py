#!/usr/bin/env python3
"""Benchmark: decode attention over a block-wise low-rank KV prefix (MILO).

A step is one decode-attention call per decoder layer (all layers of the
workload), i.e. the whole hot path once over one batch of synthetic queries.
The per-layer calls go through the libmilo C ABI and are captured in one CUDA
graph; inputs are resident in HBM before timing starts.

Metric: tokens-attended/s = sum over layers and queries of (prefix tokens +
the query's tail tokens) per second (all heads of a layer count once), plus
achieved algorithmic HBM GB/s as a fraction of the measured copy bandwidth
and, where the contraction binds, algorithmic FLOP/s against the measured
sustained bf16 tensor throughput.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config C] [--only]
                  [--impl milo|reference]

Prints one JSON line (rank 0).  The line's headline is workload --config
(default 1, the 28-layer Qwen2.5-7B-shaped prefix at batch 1); unless --only
is given, "workloads" adds a record for each of the other four workloads,
measured in the same process with the same warm-up and step count.  Under
torchrun (N > 1) every rank runs an independent replica of the workload (the
path has no cross-GPU exchange): value = all ranks' tokens / the slowest
rank's time, scaling "weak".
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode tokens-attended/s over low-rank KV prefix; HBM GB/s as % of GB300 peak"
UNIT = "tokens/s"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
L2_BYTES = 129 * 2 ** 20
PARITY_ATOL, PARITY_RTOL_L2 = 1e-2, 2e-3
# workloads on which the reconstruct-then-attend path and its pre-RoPE
# variant are timed beside the rank-space path; the rotary base of the
# Qwen2.5 models
RECON_WORKLOADS = ("qwen7b-28L-32k-b1", "qwen7b-28L-32k-b64")
ROPE_THETA = 1e6


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", type=int, default=1, help="headline workload index 0..4 (1 = batch-1 7B)")
    ap.add_argument("--only", action="store_true", help="measure the headline workload only")
    ap.add_argument("--impl", default="milo", choices=["milo", "reference"])
    ap.add_argument("--no-check", action="store_true", help="skip the parity checks")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU baseline sample time")
    ap.add_argument("--no-recon", action="store_true",
                    help="skip timing the reconstruct-then-attend path beside the rank-space path")
    ap.add_argument("--no-encode", action="store_true", help="skip timing the compression stage")
    ap.add_argument("--no-paths", action="store_true",
                    help="skip timing each workload on the other decode path (chunk grid / tensor-core grid)")
    ap.add_argument("--no-offload", action="store_true", help="skip timing the offloaded prefix")
    ap.add_argument("--no-int8", action="store_true", help="skip timing the INT8-stored factors")
    return ap.parse_args(argv)


def peaks():
    """Measured HBM copy GB/s and sustained bf16 TFLOP/s (or the fallbacks)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return (float(d["hbm_gbs"]), float(d.get("bf16_tflops_sustained", FALLBACK_BF16_TFLOPS_SUSTAINED)),
                "measured")
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


# ------------------------------------------------------------ accounting
def layer_totals(num_q_heads, num_kv_heads, head_dim, block_len, rank_k, rank_v, tail_lengths, batch):
    """(tokens attended, algorithmic bytes, algorithmic flops) of one call.

    Bytes: the factors at their true ranks (C^K, P^K, C^V, P^V), the dense
    tails, the q reads and the fp32 output writes.  Flops (multiply-add = 2):
    per KV head and query row, 2 (n_b + d)(r^k + r^v) per prefix entry (scores
    and rank-space values over its n_b tokens, projection and
    back-projection over d), and 4 d per tail token."""
    d = int(head_dim)
    hk = int(num_kv_heads)
    G = int(num_q_heads) // hk
    n = np.asarray(block_len, np.int64)[np.arange(len(rank_k)) // hk]
    r = np.asarray(rank_k, np.int64) + np.asarray(rank_v, np.int64)
    per_row = int((2 * (n + d) * r).sum())
    tails = int(np.asarray(tail_lengths, np.int64).sum())
    bytes_ = per_row + tails * hk * d * 2 * 2 + batch * num_q_heads * d * (2 + 4)
    flops = batch * G * per_row + tails * G * hk * 4 * d
    tokens = batch * int(np.asarray(block_len).sum()) + tails
    return tokens, bytes_, flops


def workload_totals(cfg, W):
    """Per-step totals of a workload from its tables alone (no factor data)."""
    tok = byt = flo = 0
    for l in range(cfg.layers):
        ranks = W.draw_ranks(cfg, l).reshape(-1)
        tl = W.draw_tail_lengths(cfg, l)
        a, b, c = layer_totals(cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                               np.full(cfg.num_blocks, cfg.block_len), ranks, ranks, tl, cfg.batch)
        tok, byt, flo = tok + a, byt + b, flo + c
    return tok, byt, flo


def shared_config(cfg, totals, world):
    """The workload's `config` object, the same on both arms."""
    tokens, bytes_, flops = totals
    l2 = ("inputs larger than L2 (a step reads %.2f GB > 129 MB); no flush" % (bytes_ / 1e9)
          if bytes_ > 2 * L2_BYTES else
          "inputs smaller than L2 (%.2f MB): L2 flushed (a %d MB write) before each timed step" %
          (bytes_ / 1e6, 4 * L2_BYTES >> 20))
    return {"workload": cfg.name, "layers": cfg.layers, "batch": cfg.batch,
            "prefix_tokens": cfg.prefix_tokens, "num_q_heads": cfg.num_q_heads,
            "num_kv_heads": cfg.num_kv_heads, "head_dim": cfg.head_dim,
            "tokens_per_step": tokens, "algorithmic_bytes_per_step": bytes_,
            "algorithmic_flops_per_step": flops, "l2": l2,
            "parallelism": "replicas" if world > 1 else "single GPU"}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.dev), "-lms", "100"], stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.3)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or not self.path:
            return None
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(dict(sm=float(parts[1]), smax=float(parts[2]), power=float(parts[3]),
                                 hw=parts[5], hwt=parts[6], swt=parts[7], swp=parts[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        loaded = [r for r in rows if r["power"] > 200.0] or rows
        reasons = set()
        for r in rows:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("swp", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in loaded),
                "sm_max_mhz": max(r["smax"] for r in rows), "reasons": sorted(reasons),
                "samples": len(rows)}


def cpu_baseline(layers_host, target_s: float):
    """The oracle, as it stands, on the host cores over a bounded sample of
    the workload's layers: returns tokens-attended/s and a description."""
    from oracle import milo_oracle
    milo_oracle.build()
    cores = milo_oracle.max_threads()
    done_tokens, t_used, used = 0, 0.0, 0
    while t_used < target_s and used < 200:
        bits, toks = layers_host[used % len(layers_host)]
        t0 = time.perf_counter()
        milo_oracle.attention(**bits)
        t_used += time.perf_counter() - t0
        done_tokens += toks
        used += 1
    return {"value": done_tokens / t_used, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{used} single-layer oracle calls cycling over the first "
                      f"{len(layers_host)} layers of the workload (all queries, all heads), "
                      f"{t_used:.1f} s of fp64 CPU work"}


def reference_arm(args, cfg, W):
    """The oracle timed as the reference implementation (rank 0 only).  A
    step is one layer of the workload (a bounded sample: the whole step of
    the GPU arm would take minutes); ms_per_step is that step's mean time and
    value the tokens it attends per second."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    from oracle import milo_oracle
    milo_oracle.build()
    layers = [W.make_config_layer(cfg, l, device="cpu") for l in range(min(cfg.layers, 2))]
    host = [(L.to_numpy_bits(), layer_totals(L.num_q_heads, L.num_kv_heads, L.head_dim, L.block_len,
                                             L.rank_k, L.rank_v, np.diff(L.tail_offsets), L.batch)[0])
            for L in layers]
    times, toks = [], []
    per = max(1, int(args.steps))
    for s in range(args.warmup + per):
        bits, tk = host[s % len(host)]
        t0 = time.perf_counter()
        milo_oracle.attention(**bits)
        dt = time.perf_counter() - t0
        if s >= args.warmup:
            times.append(dt)
            toks.append(tk)
    value = sum(toks) / sum(times)
    sample = (f"each step is one layer of {cfg.name} (layers 0 and 1 in turn), all queries and heads; "
              f"{per} timed steps after {args.warmup} warm-up")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * sum(times) / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": shared_config(cfg, workload_totals(cfg, W), world),
            "step": "one layer of the workload per step (a bounded sample of the GPU arm's step)",
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": milo_oracle.max_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def max_over_ranks(x, dist, device):
    """The largest of every rank's x (a time in ms); x itself without a
    process group.  Replicas report the slowest rank's time."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(world, tokens_per_rank, ms_step):
    """Whole-job tokens/s: every replica attends tokens_per_rank per step, and
    the step takes the slowest rank's ms_step."""
    return world * tokens_per_rank / (ms_step * 1e-3)


def pack_tensors(tensors, dev):
    """Copy device tensors (None allowed) into one byte buffer, each at a
    256-byte boundary; returns the buffer and a view of it per tensor."""
    import torch
    offs, n = [], 0
    for t in tensors:
        offs.append(n)
        if t is not None:
            n += (t.numel() * t.element_size() + 255) // 256 * 256
    buf = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)
    views = []
    for t, o in zip(tensors, offs):
        if t is None:
            views.append(None)
            continue
        v = buf[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape)
        v.copy_(t)
        views.append(v)
    return buf, views


def parity_layer0(layer, out0, ref=None):
    """Layer 0's whole output [batch, Hq, d] against the oracle (ref: the
    oracle's output, when already computed)."""
    if ref is None:
        from oracle import milo_oracle
        milo_oracle.build()
        ref = milo_oracle.attention(**layer.to_numpy_bits())
    got = out0.double().cpu().numpy()
    d = got.shape[-1]
    g2, r2 = got.reshape(-1, d), ref.reshape(-1, d)
    rows = np.linalg.norm(g2 - r2, axis=1) / np.maximum(np.linalg.norm(r2, axis=1), 1e-30)
    err = float(np.abs(got - ref).max())
    rel = float(np.linalg.norm(got - ref) / np.linalg.norm(ref))
    return {"max_abs": err, "rel_l2": rel, "worst_row_rel_l2": float(rows.max()),
            "pass": bool(err <= PARITY_ATOL and rel <= PARITY_RTOL_L2),
            "rows": f"layer 0, every query and head ({got.shape[0]} x {got.shape[1]} rows of {d})"}


def kernel_names(path: int, has_tail: bool) -> list:
    """The kernels one layer call launches, for the JSON line's description."""
    if path == 1:
        return (["chunk_kernel (dense-tail items)"] if has_tail else []) + ["batch_tc_kernel", "finish_kernel"]
    return ["chunk_kernel", "finish_kernel"]


def time_graph(step, stream, steps, warmup, flush):
    """Capture step(stream) in a CUDA graph, replay it `warmup` times, then
    time `steps` replays with CUDA events on `stream` (replay by replay after
    writing `flush`, when given).  Returns the total ms."""
    import torch
    with torch.cuda.stream(stream):
        step(stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step(stream)
    for _ in range(max(warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    if flush is None:
        start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        with torch.cuda.stream(stream):
            for _ in range(steps):
                graph.replay()
        stop.record(stream)
        torch.cuda.synchronize()
        return start.elapsed_time(stop), graph
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    with torch.cuda.stream(stream):
        for a, b in evs:
            flush.fill_(1.0)
            a.record(stream)
            graph.replay()
            b.record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs), graph


def measure(cfg, W, milo, dev, steps, warmup, dist=None, rank=0, world=1, *, check=True,
            e2e=False, cpu_seconds=0.0, recon=False, offload=False, int8=False, paths=False):
    """Time one workload (all its layers per step) and return its record."""
    import torch
    plans, qs, tks, tvs, toffs = [], [], [], [], []
    host_layers = []
    check_layer = None
    max_tail = 0
    t_gen = time.perf_counter()
    for l in range(cfg.layers):
        layer = W.make_config_layer(cfg, l, device=dev)
        max_tail = max(max_tail, int(np.diff(layer.tail_offsets).max()))
        pre = milo.Prefix.from_layer(layer)
        plans.append(pre)
        qs.append(layer.q)
        tks.append(layer.tail_k)
        tvs.append(layer.tail_v)
        toffs.append(torch.as_tensor(layer.tail_offsets, device=dev))
        if l == 0 and check and rank == 0:
            check_layer = layer
        if rank == 0 and cpu_seconds > 0 and len(host_layers) < 3:
            host_layers.append((layer.to_numpy_bits(), layer_totals(
                layer.num_q_heads, layer.num_kv_heads, layer.head_dim, layer.block_len, layer.rank_k,
                layer.rank_v, np.diff(layer.tail_offsets), layer.batch)[0]))
        if l > 0 or check_layer is None:
            layer.arena = None  # the packed copy in the plan is all the decode reads
    torch.cuda.synchronize()
    t_gen = time.perf_counter() - t_gen
    totals = workload_totals(cfg, W)
    tokens, alg_bytes, alg_flops = totals
    batch = cfg.batch
    call = milo.milo_call_info(plans[0].plan, batch, max_tail)
    ws_bytes = max(p.workspace_size(batch, max_tail) for p in plans)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    # A step's inputs (every layer's q and dense tails, layer by layer) sit in
    # one device buffer and its outputs in another, so that the end-to-end
    # step moves them in a few large copies.
    L = cfg.layers
    in_buf, views = pack_tensors([x for l in range(L) for x in (qs[l], tks[l], tvs[l])], dev)
    qs, tks, tvs = views[0::3], views[1::3], views[2::3]
    out_buf = torch.empty((L, batch, cfg.num_q_heads, cfg.head_dim), dtype=torch.float32, device=dev)
    outs = [out_buf[l] for l in range(L)]
    stream = torch.cuda.Stream(device=dev)

    def run_step(s):
        for l in range(L):
            plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws, stream=s)

    with torch.cuda.stream(stream):
        run_step(stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        run_step(stream)
    for _ in range(max(warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    for p in plans:
        assert p.status() == 0, "device status word set during warm-up"

    ref0 = None
    if check_layer is not None:
        from oracle import milo_oracle
        milo_oracle.build()
        ref0 = milo_oracle.attention(**check_layer.to_numpy_bits())
    check = parity_layer0(check_layer, outs[0], ref0) if check_layer is not None else None

    # ---- timed region: K graph replays.  Inputs larger than L2 need no
    # flush; a workload that fits in L2 is timed replay by replay with a
    # buffer larger than L2 written before each (outside the events).
    flush = torch.empty(4 * L2_BYTES // 4, dtype=torch.float32, device=dev) if alg_bytes <= 2 * L2_BYTES else None
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev.index if dev.index is not None else 0) as clocks:
        if flush is None:
            start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            start.record(stream)
            with torch.cuda.stream(stream):
                for _ in range(steps):
                    graph.replay()
            stop.record(stream)
            torch.cuda.synchronize()
            ms_total = start.elapsed_time(stop)
        else:
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(steps)]
            with torch.cuda.stream(stream):
                for a, b in evs:
                    flush.fill_(1.0)
                    a.record(stream)
                    graph.replay()
                    b.record(stream)
            torch.cuda.synchronize()
            ms_total = sum(a.elapsed_time(b) for a, b in evs)
    if dist:
        dist.barrier()
    ms_step = max_over_ranks(ms_total / steps, dist, dev)
    for p in plans:
        assert p.status() == 0, "device status word set during the timed region"

    hbm, tf_sus, peak_kind = peaks()
    achieved = alg_bytes / (ms_step * 1e-3) / 1e9
    flops_s = alg_flops / (ms_step * 1e-3) / 1e12
    roof_ms = max(alg_bytes / (hbm * 1e9), alg_flops / (tf_sus * 1e12)) * 1e3
    rec = {
        "workload": cfg.name, "ms_per_step": ms_step, "value": replica_throughput(world, tokens, ms_step),
        "unit": UNIT, "steps": steps, "warmup": warmup,
        "config": shared_config(cfg, totals, world),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "traffic": None,
                     "peak_source": f"{peak_kind} copy bandwidth (hbm_gbs)"},
        "tensor": {"achieved_tflops": flops_s, "peak_tflops": tf_sus, "frac": flops_s / tf_sus,
                   "peak_source": f"{peak_kind} sustained cuBLAS bf16 (bf16_tflops_sustained)"},
        "roofline_time": {"ms": roof_ms, "frac": roof_ms / ms_step,
                          "how": "max(algorithmic bytes / hbm_gbs, algorithmic flops / bf16_tflops_sustained)"},
        "path": {0: "chunk grid (mma.sync)", 1: "tensor-core batched grid (tcgen05)"}[call["path"]],
        "kernels_per_layer": call["kernels"],
        "kernels": kernel_names(call["path"], max_tail > 0),
        "gpu_launches": call["kernels"] * L * steps,
        "clocks": clocks.summary(), "parity_check": check, "setup_s": t_gen,
    }
    if paths:
        rec["other_path"] = measure_other_path(milo, plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps,
                                               warmup, flush, dist, dev, world, tokens, ms_step, call["path"], ref0)
    if recon:
        rec["reconstruct_then_attend"] = measure_recon(cfg, plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream,
                                                      steps, warmup, flush, dist, dev, world, tokens, ms_step,
                                                      check_layer, ref0)
    offload_check = check_layer
    if check_layer is not None:
        check_layer.arena = None
    check_layer = None
    rec["roofline"]["traffic"] = traffic_record(cfg.name)
    rec["roofline"]["traffic_of"] = (
        "DRAM bytes per launch of the tensor-core prefix grid (the prefix only), from profiles/traffic.json"
        if call["path"] == 1 else "DRAM bytes per launch of chunk_kernel, from profiles/traffic.json")
    if e2e:
        rec["e2e"] = measure_e2e(plans, stream, in_buf, out_buf, qs, tks, tvs, toffs, outs, ws, max_tail,
                                 steps, dist, dev, world, tokens)
    if offload:  # (last: it moves the plans' arenas to host memory)
        rec["offload"] = measure_offload(plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup,
                                         dist, dev, world, tokens, ms_step, offload_check, ref0, milo)
    if int8:
        for p in plans:
            p.close()
        plans = []
        torch.cuda.empty_cache()
        rec["int8"] = measure_int8(cfg, W, milo, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup,
                                   dist, dev, world, tokens, ms_step, rec.get("offload"), offload_check is not None,
                                   ref0, alg_bytes)
    if cpu_seconds > 0 and rank == 0 and world == 1 and host_layers:
        rec["cpu_baseline"] = cpu_baseline(host_layers, cpu_seconds)
    for p in plans:
        p.close()
    del plans, graph, ws, in_buf, out_buf
    torch.cuda.empty_cache()
    return rec


def measure_recon(cfg, plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup, flush, dist, dev,
                  world, tokens, ms_rank_space, check_layer, ref0):
    """The same step by reconstruct-then-attend (the paper's own path: dense
    keys and values rebuilt from the factors, then attended), on the same
    plans and inputs; then the pre-RoPE variant (every reconstructed prefix
    key rotated to its position, rotary base ROPE_THETA).  Each is timed like
    the rank-space step and checked on layer 0 against the oracle."""
    L = len(plans)
    kernels = (1 if max_tail > 0 else 0) + 2

    def step(s):
        for l in range(L):
            plans[l].decode_reconstruct(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws,
                                        stream=s)

    def one(label):
        ms_total, _ = time_graph(step, stream, steps, warmup, flush)
        for p in plans:
            assert p.status() == 0, f"device status word set during the {label} timing"
        ms = max_over_ranks(ms_total / steps, dist, dev)
        return {"ms_per_step": ms, "value": replica_throughput(world, tokens, ms), "unit": UNIT,
                "gpu_launches": kernels * L * steps,
                "kernels": (["chunk_kernel (dense-tail items)"] if max_tail > 0 else []) +
                           ["recon_kernel", "finish_kernel"]}

    out = one("reconstruct")
    out["rank_space_ms_per_step"] = ms_rank_space
    out["rank_space_speedup"] = out["ms_per_step"] / ms_rank_space
    out["how"] = ("the same graph of per-layer calls through milo_attn_decode_reconstruct: per tile of 64 "
                  "tokens, K^ = C^K P^K and V^ = C^V P^V rebuilt in fp16 in shared memory, then flash "
                  "decoding; rank_space_speedup = this ms / the rank-space ms on the same inputs")
    if check_layer is not None:
        out["parity_check"] = parity_layer0(check_layer, outs[0], ref0)
    for p in plans:
        p.set_rope(ROPE_THETA)
    try:
        rope = one("pre-RoPE")
        rope["rope_theta"] = ROPE_THETA
        rope["how"] = ("reconstruct-then-attend over pre-RoPE factors: every reconstructed prefix key turns "
                       "to its position (the blocks' starts in the concatenated prefix) before scoring")
        if check_layer is not None:
            from oracle import milo_oracle
            ref_rope = milo_oracle.attention(**check_layer.to_numpy_bits(), rope_theta=ROPE_THETA)
            rope["parity_check"] = parity_layer0(check_layer, outs[0], ref_rope)
        out["pre_rope"] = rope
    finally:
        for p in plans:
            p.set_rope(0.0)
    return out


def measure_offload(plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup, dist, dev, world, tokens,
                    ms_resident, check_layer, ref0, milo=None):
    """The same step with every layer's packed factors in pinned host memory
    (milo_prefix_offload): layer l is copied into device buffer l % 2 on a
    copy stream (milo_prefix_stage) while the decode stream runs layer l - 1;
    the copy into a buffer waits for the decode two layers back.  One CUDA
    graph per step.  The interconnect's copy rate is measured in the same run
    (one pinned host-to-device copy of the step's bytes)."""
    import torch
    L = len(plans)
    for p in plans:
        p.offload()
    nbytes = max(int(p.info["packed_bytes"]) for p in plans)
    total_bytes = sum(int(p.info["packed_bytes"]) for p in plans)
    bufs = [torch.empty(nbytes + 128, dtype=torch.uint8, device=dev) for _ in range(2)]
    copy = torch.cuda.Stream(device=dev)
    staged = [torch.cuda.Event() for _ in range(L)]
    done = [torch.cuda.Event() for _ in range(L)]
    fork = torch.cuda.Event()

    def step(s):
        fork.record(s)
        copy.wait_event(fork)
        for l in range(L):
            if l >= 2:
                copy.wait_event(done[l - 2])
            plans[l].stage(bufs[l % 2], stream=copy)
            staged[l].record(copy)
            s.wait_event(staged[l])
            plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws, stream=s)
            done[l].record(s)
        s.wait_stream(copy)

    ms_total, _ = time_graph(step, stream, steps, warmup, None)
    for p in plans:
        assert p.status() == 0, "device status word set during the offloaded timing"
    ms = max_over_ranks(ms_total / steps, dist, dev)
    # the host-to-device copy rate of the same bytes, one copy
    host = torch.empty(total_bytes, dtype=torch.uint8).pin_memory()
    dst = torch.empty(total_bytes, dtype=torch.uint8, device=dev)
    dst.copy_(host, non_blocking=True)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(3):
        dst.copy_(host, non_blocking=True)
    b.record()
    torch.cuda.synchronize()
    h2d = 3 * total_bytes / (a.elapsed_time(b) * 1e-3) / 1e9
    achieved = total_bytes / (ms * 1e-3) / 1e9
    rec = {"ms_per_step": ms, "value": replica_throughput(world, tokens, ms), "unit": UNIT,
           "resident_ms_per_step": ms_resident,
           "interconnect": {"achieved": achieved, "peak": h2d, "unit": "GB/s", "frac": achieved / h2d,
                            "peak_source": "pinned host-to-device copy of the step's bytes, measured in this run"},
           "gpu_launches": sum(1 for _ in plans) * steps * milo.milo_call_info(plans[0].plan, qs[0].shape[0], max_tail)["kernels"],
           "how": "packed arenas in pinned host memory; per layer one cudaMemcpyAsync into one of two device "
                  "buffers on a copy stream, overlapped with the previous layer's decode; one CUDA graph a step"}
    if check_layer is not None:
        rec["parity_check"] = parity_layer0(check_layer, outs[0], ref0)
    return rec


def measure_int8(cfg, W, milo, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup, dist, dev, world,
                 tokens, ms_resident, offload_rec, check, ref0, alg_bytes):
    """The same step with every layer's factors held as INT8 (Sec. 5.3,
    Table 2; milo_prefix_quantize_int8), in two placements, each on plans
    built afresh from the same layers:
      offloaded: codes in mapped pinned host memory; per layer one staging
        kernel reads them over the chip-to-chip link and writes the bf16
        read-back into device buffer l % 2 on a copy stream, overlapped with
        the previous layer's decode (the structure of the bf16 offloaded step);
      resident: codes in device memory, staged the same way from HBM;
      resident_direct: the same plans unstaged, the chunk grid reading the
        codes itself (one decode per layer, half the factor bytes).
    One CUDA graph per step.  Parity: layer 0 against the oracle's attention
    over the oracle's INT8 read-back of the same factors; the distance to the
    bf16 result is the quantisation's effect."""
    import torch
    from oracle import milo_int8, milo_oracle
    L = cfg.layers
    rec = {"what": "MILO + INT8 (asymmetric, one bf16 minimum and step per 8x8 tile of a factor)"}
    layer0_bits = None
    ref_q = None
    for mode, to_host in (("offloaded", True), ("resident", False)):
        plans = []
        for l in range(L):
            layer = W.make_config_layer(cfg, l, device=dev)
            if l == 0 and check and layer0_bits is None:
                layer0_bits = layer.to_numpy_bits()
            pre = milo.Prefix.from_layer(layer)
            pre.quantize_int8(to_host=to_host)
            plans.append(pre)
            layer.arena = None
        torch.cuda.synchronize()
        nbytes = max(int(p.info["packed_bytes"]) for p in plans)
        stored = sum(p.storage()["bytes"] for p in plans)
        bf16_bytes = sum(int(p.info["packed_bytes"]) for p in plans)
        bufs = [torch.empty(nbytes + 128, dtype=torch.uint8, device=dev) for _ in range(2)]
        copy = torch.cuda.Stream(device=dev)
        staged = [torch.cuda.Event() for _ in range(L)]
        done = [torch.cuda.Event() for _ in range(L)]
        fork = torch.cuda.Event()

        def step(s):
            fork.record(s)
            copy.wait_event(fork)
            for l in range(L):
                if l >= 2:
                    copy.wait_event(done[l - 2])
                plans[l].stage(bufs[l % 2], stream=copy)
                staged[l].record(copy)
                s.wait_event(staged[l])
                plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws, stream=s)
                done[l].record(s)
            s.wait_stream(copy)

        ms_total, graph = time_graph(step, stream, steps, warmup, None)
        for p in plans:
            assert p.status() == 0, "device status word set during the INT8 timing"
        ms = max_over_ranks(ms_total / steps, dist, dev)
        r = {"ms_per_step": ms, "value": replica_throughput(world, tokens, ms), "unit": UNIT,
             "stored_bytes_per_step": stored, "bf16_bytes_per_step": bf16_bytes,
             "gpu_launches": L * steps * (1 + milo.milo_call_info(plans[0].plan, qs[0].shape[0], max_tail)["kernels"])}
        # the staging kernel alone: every layer staged into one buffer, on one stream
        def stage_only(s):
            for l in range(L):
                plans[l].stage(bufs[0], stream=s)
        ms_stage, _ = time_graph(stage_only, stream, max(steps // 4, 5), warmup, None)
        ms_stage /= max(steps // 4, 5)
        if to_host:
            ach = stored / (ms * 1e-3) / 1e9
            r["interconnect"] = {"achieved": ach, "peak": offload_rec["interconnect"]["peak"] if offload_rec else None,
                                 "unit": "GB/s", "bytes": "INT8 codes and group parameters of every layer"}
            if offload_rec:
                r["interconnect"]["frac"] = ach / offload_rec["interconnect"]["peak"]
                r["speedup_vs_bf16_offloaded"] = offload_rec["ms_per_step"] / ms
            r["stage_kernel"] = {"us_per_layer": 1e3 * ms_stage / L,
                                 "link_gbs": stored / (ms_stage * 1e-3) / 1e9,
                                 "how": "dequant_plan_kernel reading mapped host memory, all layers back to back"}
        else:
            hbm = (stored + bf16_bytes) / (ms_stage * 1e-3) / 1e9
            peak_gbs, _, peak_kind = peaks()
            r["stage_kernel"] = {"us_per_layer": 1e3 * ms_stage / L, "achieved_gbs": hbm,
                                 "peak_gbs": peak_gbs, "frac": hbm / peak_gbs, "peak_source": peak_kind,
                                 "how": "dequant_plan_kernel from device memory: reads codes and parameters "
                                        "(68 B per 128 B core), writes the bf16 core; all layers back to back"}
            r["vs_bf16_resident"] = ms_resident / ms
            rec["resident_direct"] = measure_int8_direct(milo, plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream,
                                                         steps, warmup, dist, dev, world, tokens, ms_resident,
                                                         alg_bytes, stored, ref_q, ref0)
        if mode == "offloaded" and layer0_bits is not None:
            milo_oracle.build()
            deq, _ = milo_int8.quantize_arena(arena=layer0_bits["arena"], **{
                k: layer0_bits[k] for k in ("num_kv_heads", "head_dim", "block_len", "rank_k", "rank_v",
                                            "off_ck", "off_pk", "off_cv", "off_pv")})
            bits = dict(layer0_bits, arena=deq)
            ref_q = milo_oracle.attention(**bits)
            pc = parity_layer0(None, outs[0], ref_q)
            if ref0 is not None:
                got = outs[0].double().cpu().numpy()
                pc["rel_l2_vs_bf16_factors"] = float(np.linalg.norm(got - ref0) / np.linalg.norm(ref0))
            pc["what"] = "against the oracle's attention over its own INT8 read-back of layer 0's factors"
            r["parity_check"] = pc
        rec[mode] = r
        for p in plans:
            p.close()
        del plans, graph, bufs
        torch.cuda.empty_cache()
    rec["reduction_vs_bf16_factors"] = rec["offloaded"]["bf16_bytes_per_step"] / rec["offloaded"]["stored_bytes_per_step"]
    return rec


def measure_other_path(milo, plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup, flush, dist,
                       dev, world, tokens, ms_default, path_default, ref0):
    """The same step on the other decode path, chosen per plan with
    milo_prefix_set_tensor_min_rows (the chunk grid for a workload that takes
    the tensor-core grid, and the reverse), timed the same way; the plans go
    back to the default threshold afterwards."""
    import torch
    other = 1 - path_default
    for p in plans:
        p.set_tensor_min_rows(1 if other == 1 else 1 << 30)
    try:
        batch = qs[0].shape[0]
        need = max(p.workspace_size(batch, max_tail) for p in plans)
        wsx = ws if ws.numel() >= need else torch.empty(need, dtype=torch.uint8, device=dev)
        L = len(plans)

        def step(s):
            for l in range(L):
                plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=wsx, stream=s)

        ms_total, _ = time_graph(step, stream, steps, warmup, flush)
        for p in plans:
            assert p.status() == 0, "device status word set on the other path"
        ms = max_over_ranks(ms_total / steps, dist, dev)
        call = milo.milo_call_info(plans[0].plan, batch, max_tail)
        assert call["path"] == other
        r = {"path": {0: "chunk grid (mma.sync)", 1: "tensor-core batched grid (tcgen05)"}[other],
             "ms_per_step": ms, "value": replica_throughput(world, tokens, ms), "unit": UNIT,
             "default_speedup": ms / ms_default, "gpu_launches": call["kernels"] * L * steps,
             "how": "milo_prefix_set_tensor_min_rows on every plan, one CUDA graph a step as for the default path"}
        if ref0 is not None:
            r["parity_check"] = parity_layer0(None, outs[0], ref0)
        return r
    finally:
        for p in plans:
            p.set_tensor_min_rows(milo.milo_tensor_min_rows())


def measure_int8_direct(milo, plans, qs, tks, tvs, toffs, outs, ws, max_tail, stream, steps, warmup, dist, dev,
                        world, tokens, ms_resident, alg_bytes, stored, ref_q, ref0):
    """The resident INT8 plans unstaged (milo_prefix_stage with no buffer):
    each layer's decode is one chunk grid that reads the codes and group
    parameters (68 B per 128-byte core) and reads them back in shared memory.
    Algorithmic bytes: the bf16 step's, with the factors' true-rank bf16
    bytes replaced by the INT8 bytes stored."""
    import torch
    L = len(plans)
    for p in plans:
        p.stage(None)
    need = max(p.workspace_size(qs[0].shape[0], max_tail) for p in plans)
    if ws.numel() < need:
        ws = torch.empty(need, dtype=torch.uint8, device=dev)

    def step(s):
        for l in range(L):
            plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws, stream=s)

    ms_total, _ = time_graph(step, stream, steps, warmup, None)
    for p in plans:
        assert p.status() == 0, "device status word set during the INT8 direct timing"
    ms = max_over_ranks(ms_total / steps, dist, dev)
    logical = sum(int(p.info["logical_factor_bytes"]) for p in plans)
    nbytes = alg_bytes - logical + stored
    ach = nbytes / (ms * 1e-3) / 1e9
    peak_gbs, _, peak_kind = peaks()
    call = milo.milo_call_info(plans[0].plan, qs[0].shape[0], max_tail)
    r = {"ms_per_step": ms, "value": replica_throughput(world, tokens, ms), "unit": UNIT,
         "vs_bf16_resident": ms_resident / ms,
         "path": "chunk grid reading INT8 codes (%s)" % milo.PATH_NAMES[call["path"]],
         "gpu_launches": call["kernels"] * L * steps,
         "roofline": {"bound": "hbm", "achieved": ach, "peak": peak_gbs, "unit": "GB/s", "frac": ach / peak_gbs,
                      "peak_source": f"{peak_kind} copy bandwidth (hbm_gbs)", "bytes_per_step": nbytes,
                      "how": "the bf16 step's algorithmic bytes with the factors' true-rank bf16 bytes "
                             "replaced by the INT8 codes and parameters stored"}}
    if ref_q is not None:
        pc = parity_layer0(None, outs[0], ref_q)
        if ref0 is not None:
            got = outs[0].double().cpu().numpy()
            pc["rel_l2_vs_bf16_factors"] = float(np.linalg.norm(got - ref0) / np.linalg.norm(ref0))
        pc["what"] = "against the oracle's attention over its own INT8 read-back of layer 0's factors"
        r["parity_check"] = pc
    return r


def measure_encode(cfg, W, milo, dev, reps=5, cpu_seconds=0.0):
    """The compression stage (milo_encode, Alg. 1 Stage 1) on one layer of
    the workload's shape: dense keys and values drawn with a decaying
    spectrum, budgets of a mean rank of d/2 (the paper's 50% rank budget),
    r_min 16, r_max d.  Timed end to end per call (host staging included) on
    the device; checked against the oracle's greedy on the GPU's singular
    values and the oracle's SVD of one block; the oracle's own compression
    timed on a bounded sample of blocks on the host."""
    import torch
    bl = [cfg.block_len] * cfg.num_blocks
    hkv, d = cfg.num_kv_heads, cfg.head_dim
    k, v = W.make_dense_kv(bl, hkv, d, seed=cfg.seed, device=dev)
    budget = (d // 2) * cfg.num_blocks
    kw = dict(r_min=16, r_max=d, budget_k=budget, budget_v=budget)
    enc = milo.encode(k, v, bl, **kw)  # warm-up
    torch.cuda.synchronize()
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        enc = milo.encode(k, v, bl, **kw)
        torch.cuda.synchronize()
        times.append(time.perf_counter() - t0)
    ms = 1e3 * statistics.median(times)
    tokens = int(sum(bl))
    rec = {"ms_per_layer": ms, "value": tokens / (ms * 1e-3), "unit": "prefix tokens encoded/s (all KV heads)",
           "matrices_per_layer": 2 * cfg.num_blocks * hkv, "mean_rank_k": float(enc["rank_k"].mean()),
           "mean_rank_v": float(enc["rank_v"].mean()),
           "how": "median of %d milo_encode calls on one %d x %d-token layer, %d KV heads, d %d (three grids: "
                  "Gram + Jacobi eigen-decomposition, allocation, factors)" % (reps, cfg.num_blocks,
                                                                                 cfg.block_len, hkv, d)}
    from oracle import milo_oracle
    milo_oracle.build()
    sig = enc["sigma"].cpu().numpy().astype(np.float64)
    gsig = [sig[2 * (b * hkv)][:min(cfg.block_len, d)] for b in range(cfg.num_blocks)]
    want = milo_oracle.allocate_ranks(gsig, kw["r_min"], kw["r_max"], budget, 1e-6)
    got = np.array([enc["rank_k"][b * hkv] for b in range(cfg.num_blocks)])
    X = (k[:cfg.block_len, 0, :].float().cpu().numpy()).astype(np.float64)
    t0 = time.perf_counter()
    s_ref = milo_oracle.svd(X)[0]
    t_svd = time.perf_counter() - t0
    rec["parity_check"] = {
        "ranks_equal_oracle_greedy_on_gpu_sigma": bool(np.array_equal(got, want)),
        "sigma2_max_err_over_sigma1_2_block0": float(np.abs(sig[0][:len(s_ref)] ** 2 - s_ref ** 2).max() / s_ref[0] ** 2),
        "what": "KV head 0 keys: the oracle's greedy (Eq. 7) fed the GPU's singular values gives the GPU's ranks; "
                "block 0's singular values against the oracle's fp64 Jacobi SVD"}
    if cpu_seconds > 0:
        # the oracle's compression (SVD of K and V of each block, then the
        # greedy) of as many blocks of KV head 0 as fit the time
        Kh = k[:, 0, :].float().cpu().numpy().astype(np.float64)
        Vh = v[:, 0, :].float().cpu().numpy().astype(np.float64)
        nb = max(1, min(cfg.num_blocks, int(cpu_seconds / max(2 * t_svd, 1e-3))))
        n = cfg.block_len
        t0 = time.perf_counter()
        milo_oracle.compress_blocks([Kh[i * n:(i + 1) * n] for i in range(nb)], [Vh[i * n:(i + 1) * n] for i in range(nb)],
                                    R_tot_k=(d // 2) * nb, R_tot_v=(d // 2) * nb, r_min=16, r_max=d)
        dt = time.perf_counter() - t0
        rec["cpu_baseline"] = {"value": nb * n / dt, "unit": "prefix tokens encoded/s (one KV head)",
                               "cores": milo_oracle.max_threads(), "kind": "oracle",
                               "sample": f"{nb} blocks of {n} tokens of one KV head (keys and values), {dt:.1f} s"}
    return rec


def measure_e2e(plans, stream, in_buf, out_buf, qs, tks, tvs, toffs, outs, ws, max_tail, steps, dist, dev,
                world, tokens):
    """The same step through the public API with host buffers: each step
    copies every layer's q and tails from pinned host memory, runs the
    per-layer calls and reads every layer's output back.  The layers are cut
    into segments, each a captured graph whose inputs arrive by one copy on
    a second stream and whose outputs leave by one copy on a third, so that
    later segments' input copies and earlier segments' output copies overlap
    the calls in between."""
    import torch
    L = len(plans)
    in_host = in_buf.cpu().pin_memory()
    out_host = torch.empty_like(out_buf, device="cpu").pin_memory()
    h2d = sum(x.numel() * x.element_size() for x in qs + tks + tvs if x is not None)
    d2h = out_host.numel() * out_host.element_size()
    # four segments: more (or segments of 1, 2, 4, ... layers) measured no
    # better, each cross-stream edge costing the calls their chaining
    nseg = min(4, L)
    cuts = [round(k * L / nseg) for k in range(nseg + 1)]
    base = in_buf.data_ptr()
    seg_bytes = [qs[a].data_ptr() - base for a in cuts[:-1]] + [in_buf.numel()]
    copy_stream = torch.cuda.Stream(device=dev)
    out_stream = torch.cuda.Stream(device=dev)
    seg_done = [torch.cuda.Event() for _ in range(nseg)]
    seg_out = [torch.cuda.Event() for _ in range(nseg)]

    def body(s):
        copy_stream.wait_stream(s)  # the previous step's calls have read their inputs
        out_stream.wait_stream(s)
        with torch.cuda.stream(copy_stream):
            for k in range(nseg):
                lo, hi = seg_bytes[k], seg_bytes[k + 1]
                in_buf[lo:hi].copy_(in_host[lo:hi], non_blocking=True)
                seg_done[k].record(copy_stream)
        for k in range(nseg):
            s.wait_event(seg_done[k])
            for l in range(cuts[k], cuts[k + 1]):
                plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws, stream=s)
            seg_out[k].record(s)
            out_stream.wait_event(seg_out[k])
            with torch.cuda.stream(out_stream):
                out_host[cuts[k]:cuts[k + 1]].copy_(out_buf[cuts[k]:cuts[k + 1]], non_blocking=True)
        s.wait_stream(out_stream)  # the step ends when its last output is on the host

    # the whole step (copies, calls, event edges) is one CUDA graph, so the
    # host issues one launch a step
    with torch.cuda.stream(stream):
        body(stream)
    stream.synchronize()
    step_graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(step_graph, stream=stream):
        body(stream)

    def e2e_step(s):
        step_graph.replay()

    with torch.cuda.stream(stream):
        for _ in range(2):
            e2e_step(stream)
    stream.synchronize()
    e_steps = max(3, min(steps, 10))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(e_steps):
            e2e_step(stream)
    e1.record(stream)
    torch.cuda.synchronize()
    e_ms = max_over_ranks(e0.elapsed_time(e1) / e_steps, dist, dev)
    return {"value": replica_throughput(world, tokens, e_ms), "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e_ms,
            "segments": nseg,
            "how": "one CUDA graph a step: every layer's q and tails copied from pinned host memory in %d "
                   "copies on a second stream, each releasing its layers' calls, whose outputs are copied to "
                   "pinned host memory on a third stream; the step ends when the last output copy is done"
                   % nseg}


def traffic_record(cfg_name):
    """DRAM bytes per launch of the dominant kernel from profiles/traffic.json,
    while the kernel's source still hashes to the profiled one."""
    try:
        import hashlib
        from paper_2609_29913_gb300 import build as b
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            tr = json.load(f)
        entry = tr.get(cfg_name)
        if not entry:
            return None
        h = hashlib.sha256(open(os.path.join(b.CSRC, entry["kernel_source"]), "rb").read()).hexdigest()[:16]
        return entry["dram_bytes_per_launch"] if entry.get("kernel_sha") == h else None
    except Exception:
        return None


def main():
    args = parse()
    from paper_2609_29913_gb300 import workloads as W
    cfg = W.CONFIGS[args.config]
    if args.impl == "reference":
        reference_arm(args, cfg, W)
        return

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2609_29913_gb300 import build as milo_build
    milo_build.build()
    from paper_2609_29913_gb300 import milo

    dev = torch.device("cuda", local)
    head = measure(cfg, W, milo, dev, args.steps, args.warmup, dist, rank, world, check=not args.no_check,
                   e2e=True, cpu_seconds=0.0 if args.no_cpu else args.cpu_seconds,
                   recon=not args.no_recon and cfg.name in RECON_WORKLOADS, offload=not args.no_offload,
                   int8=not args.no_int8, paths=not args.no_paths)
    others = []
    if not args.only:
        for k, other in enumerate(W.CONFIGS):
            if k == args.config:
                continue
            others.append(measure(other, W, milo, dev, args.steps, args.warmup, dist, rank, world,
                                  check=not args.no_check,
                                  recon=not args.no_recon and other.name in RECON_WORKLOADS,
                                  paths=not args.no_paths))
    if not args.no_encode and rank == 0:
        head["encode"] = measure_encode(cfg, W, milo, dev, cpu_seconds=0.0 if args.no_cpu else 4.0)
    roof = dict(head["roofline"])
    roof["kernel"] = ", ".join(head["kernels"])
    roof["per_launch_bytes"] = head["config"]["algorithmic_bytes_per_step"] // cfg.layers
    roof["per_launch_us"] = head["ms_per_step"] * 1e3 / cfg.layers
    roof["how"] = ("algorithmic bytes of a layer call / the mean time of a layer call inside the timed "
                   "CUDA graph (consecutive calls overlap through programmatic dependent launch)")
    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": head["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": head["config"],
        "launch": "one CUDA graph of %d per-layer calls (%s per call)" % (cfg.layers, ", ".join(head["kernels"])),
        "roofline": roof, "tensor": head["tensor"], "roofline_time": head["roofline_time"],
        "cpu_baseline": head.get("cpu_baseline"),
        "e2e": head["e2e"], "gpu_launches": head["gpu_launches"], "clocks": head["clocks"],
        "parity_check": head["parity_check"], "path": head["path"], "setup_s": head["setup_s"],
        "other_path": head.get("other_path"),
        "reconstruct_then_attend": head.get("reconstruct_then_attend"),
        "encode": head.get("encode"),
        "offload": head.get("offload"),
        "int8": head.get("int8"),
        "workloads": [{k: v for k, v in o.items() if k not in ("unit",)} for o in others],
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
