#!/usr/bin/env python3
"""Benchmark: decode attention over a block-wise low-rank KV prefix (MILO).

A step is one decode-attention call per decoder layer (all layers of the
workload), i.e. the whole hot path once over one batch of synthetic queries.
The per-layer calls go through the libmilo C ABI and are captured in one CUDA
graph; inputs are resident in HBM before timing starts.

Metric: tokens-attended/s = sum over layers and queries of (prefix tokens +
the query's tail tokens) per second (all heads of a layer count once), plus
achieved algorithmic HBM GB/s as a fraction of the measured copy bandwidth.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config C] [--impl milo|reference]

Prints one JSON line (rank 0).  Under torchrun (N > 1) every rank runs an
independent replica of the workload (the path has no cross-GPU exchange):
value = all ranks' tokens / the slowest rank's time, scaling "weak".
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


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", type=int, default=1, help="workload index 0..4 (1 = headline)")
    ap.add_argument("--impl", default="milo", choices=["milo", "reference"])
    ap.add_argument("--no-check", action="store_true", help="skip the parity spot check")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU baseline sample time")
    return ap.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def algorithmic_bytes(layer) -> int:
    """Bytes the method must move for one call: factors at their true ranks
    (C^K, P^K, C^V, P^V), the dense tails, q reads and fp32 output writes."""
    d = layer.head_dim
    n = layer.block_len[np.arange(len(layer.rank_k)) // layer.num_kv_heads].astype(np.int64)
    r = (layer.rank_k + layer.rank_v).astype(np.int64)
    factors = int(((n + d) * r).sum()) * 2
    tails = int(layer.tail_offsets[-1]) * layer.num_kv_heads * d * 2 * 2
    qo = layer.batch * layer.num_q_heads * d * (2 + 4)
    return factors + tails + qo


def tokens_attended(layer) -> int:
    return int(layer.batch * int(layer.block_len.sum()) + int(layer.tail_offsets[-1]))


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
    """The oracle timed as the reference implementation (rank 0 only)."""
    import torch  # noqa: F401
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from oracle import milo_oracle
    milo_oracle.build()
    layers = [W.make_config_layer(cfg, l, device="cpu") for l in range(min(cfg.layers, 2))]
    host = [(L.to_numpy_bits(), tokens_attended(L)) for L in layers]
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
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * sum(times) / len(times) * cfg.layers,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": cfg.name, "layers": cfg.layers,
                                            "sample": "each step is one layer of the workload"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": milo_oracle.max_threads(),
                             "kind": "oracle",
                             "sample": f"{per} single-layer calls of {cfg.name} after {args.warmup} warm-up"},
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
    # ---- inputs resident in HBM, one plan per layer (logical arenas freed)
    plans, qs, tks, tvs, toffs, metas = [], [], [], [], [], []
    check_layer = None
    host_layers = []
    alg_bytes = 0
    tokens = 0
    max_tail = 0
    t_gen = time.perf_counter()
    for l in range(cfg.layers):
        layer = W.make_config_layer(cfg, l, device=dev)
        alg_bytes += algorithmic_bytes(layer)
        tokens += tokens_attended(layer)
        max_tail = max(max_tail, int(np.diff(layer.tail_offsets).max()))
        pre = milo.Prefix.from_layer(layer)
        plans.append(pre)
        qs.append(layer.q)
        tks.append(layer.tail_k)
        tvs.append(layer.tail_v)
        toffs.append(torch.as_tensor(layer.tail_offsets, device=dev))
        if l == 0 and not args.no_check:
            check_layer = (layer, layer.to_numpy_bits())
        if rank == 0 and not args.no_cpu and len(host_layers) < 3:
            host_layers.append((layer.to_numpy_bits(), tokens_attended(layer)))
        layer.arena = None  # the packed copy in the plan is all the decode reads
    torch.cuda.synchronize()
    t_gen = time.perf_counter() - t_gen
    batch = cfg.batch
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
        for l in range(cfg.layers):
            plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws,
                            stream=s)

    # warm once eagerly, then capture the step in a graph
    with torch.cuda.stream(stream):
        run_step(stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        run_step(stream)
    for _ in range(max(args.warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    for p in plans:
        assert p.status() == 0, "device status word set during warm-up"

    # ---- parity spot check (outside the timed region): one KV head of layer 0
    check = None
    if check_layer is not None:
        from oracle import milo_oracle
        milo_oracle.build()
        check_layer, bits = check_layer
        hkv, G = cfg.num_kv_heads, cfg.num_q_heads // cfg.num_kv_heads
        ent = np.arange(cfg.num_blocks) * hkv
        qsel = list(range(min(batch, 2)))
        sub = dict(num_kv_heads=1, head_dim=cfg.head_dim, block_len=check_layer.block_len,
                   rank_k=check_layer.rank_k[ent], rank_v=check_layer.rank_v[ent],
                   off_ck=check_layer.off_ck[ent], off_pk=check_layer.off_pk[ent],
                   off_cv=check_layer.off_cv[ent], off_pv=check_layer.off_pv[ent],
                   arena=bits["arena"], q=np.ascontiguousarray(bits["q"][qsel][:, :G]))
        if "tail_k" in bits:
            tk, tv, to = [], [], [0]
            for i in qsel:
                a, b = check_layer.tail_offsets[i], check_layer.tail_offsets[i + 1]
                tk.append(bits["tail_k"][a:b, 0:1])
                tv.append(bits["tail_v"][a:b, 0:1])
                to.append(to[-1] + b - a)
            sub.update(tail_k=np.ascontiguousarray(np.concatenate(tk)),
                       tail_v=np.ascontiguousarray(np.concatenate(tv)), tail_offsets=np.array(to))
        ref = milo_oracle.attention(**sub)
        got = outs[0][qsel][:, :G].double().cpu().numpy()
        check = {"max_abs": float(np.abs(got - ref).max()),
                 "rel_l2": float(np.linalg.norm(got - ref) / np.linalg.norm(ref)),
                 "rows": f"layer 0, KV head 0, queries {qsel}"}
        check_layer = None

    # ---- timed region: K graph replays (inputs > L2: no flush needed)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clocks:
        torch.cuda.nvtx.range_push("milo_timed")
        start.record(stream)
        with torch.cuda.stream(stream):
            for _ in range(args.steps):
                graph.replay()
        stop.record(stream)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    if dist:
        dist.barrier()
    ms_total = start.elapsed_time(stop)
    ms_step = max_over_ranks(ms_total / args.steps, dist, dev)
    for p in plans:
        assert p.status() == 0, "device status word set during the timed region"

    # ---- end to end through the public API with host buffers: each step
    # copies every layer's q and tails from pinned host memory, runs the
    # per-layer calls and reads every layer's output back.  The layers are
    # cut into a few segments, each a captured graph whose inputs arrive by
    # one copy on a second stream, so that later segments' copies overlap
    # earlier segments' calls.
    in_host = in_buf.cpu().pin_memory()
    out_host = torch.empty_like(out_buf, device="cpu").pin_memory()
    h2d = sum(x.numel() * x.element_size() for x in qs + tks + tvs if x is not None)
    d2h = out_host.numel() * out_host.element_size()
    nseg = min(4, L)
    cuts = [round(k * L / nseg) for k in range(nseg + 1)]
    base = in_buf.data_ptr()
    seg_bytes = [qs[a].data_ptr() - base for a in cuts[:-1]] + [in_buf.numel()]
    seg_graphs = []
    for a, b in zip(cuts, cuts[1:]):
        gs = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gs, stream=stream):
            for l in range(a, b):
                plans[l].decode(qs[l], tks[l], tvs[l], toffs[l], max_tail, out=outs[l], workspace=ws,
                                stream=stream)
        seg_graphs.append(gs)
    copy_stream = torch.cuda.Stream(device=dev)
    seg_done = [torch.cuda.Event() for _ in range(nseg)]

    def e2e_step(s):
        copy_stream.wait_stream(s)  # the previous step's calls have read their inputs
        with torch.cuda.stream(copy_stream):
            for k in range(nseg):
                lo, hi = seg_bytes[k], seg_bytes[k + 1]
                in_buf[lo:hi].copy_(in_host[lo:hi], non_blocking=True)
                seg_done[k].record(copy_stream)
        for k in range(nseg):
            s.wait_event(seg_done[k])
            seg_graphs[k].replay()
        out_host.copy_(out_buf, non_blocking=True)

    with torch.cuda.stream(stream):
        for _ in range(2):
            e2e_step(stream)
    stream.synchronize()
    e_steps = max(3, min(args.steps, 10))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(e_steps):
            e2e_step(stream)
    e1.record(stream)
    torch.cuda.synchronize()
    e_ms = max_over_ranks(e0.elapsed_time(e1) / e_steps, dist, dev)

    # ---- CPU oracle baseline (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu and host_layers:
        cpu = cpu_baseline(host_layers, args.cpu_seconds)

    peak, peak_kind = peaks()
    achieved = alg_bytes / (ms_step * 1e-3) / 1e9
    traffic = None
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            tr = json.load(f)
        from paper_2609_29913_gb300 import build as b
        import hashlib
        entry = tr.get(cfg.name)
        src = entry.get("kernel_source", "milo_decode.cu") if entry else "milo_decode.cu"
        h = hashlib.sha256(open(os.path.join(b.CSRC, src), "rb").read()).hexdigest()[:16]
        if entry and entry.get("kernel_sha") == h:
            traffic = entry["dram_bytes_per_launch"]
    except Exception:
        traffic = None
    value = replica_throughput(world, tokens, ms_step)
    # up to 8 query heads per KV head: the chunk grid (a block per prefix
    # chunk and row group of 8 query rows, and per tail item, adding into
    # per-row accumulators) and its finish grid; more: the persistent kernel
    # and the merge kernel
    short = cfg.num_q_heads // cfg.num_kv_heads <= 8
    kernels_per_layer = 2
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": cfg.name, "layers": cfg.layers, "batch": cfg.batch,
                   "prefix_tokens": cfg.prefix_tokens, "num_q_heads": cfg.num_q_heads,
                   "num_kv_heads": cfg.num_kv_heads, "head_dim": cfg.head_dim,
                   "tokens_per_step": tokens, "algorithmic_bytes_per_step": alg_bytes,
                   "l2": "inputs larger than L2 (step reads %.2f GB > 129 MB); no flush" % (alg_bytes / 1e9),
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "launch": ("one CUDA graph of %d per-layer calls, each a grid of two-warp blocks (prefix "
                              "chunks per row group of 8 query rows, and dense-tail items, adding into per-row "
                              "accumulators) and a finish grid of one warp per KV head and row group "
                              "(programmatic dependent launch)"
                              if short else
                              "one CUDA graph of %d per-layer calls, each a persistent decode and a merge "
                              "kernel (programmatic dependent launch)") % cfg.layers},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "peak_source": f"{peak_kind} copy bandwidth",
                     "kernel": ("chunk_kernel (two warps per prefix chunk and row group, accumulator merge; "
                                "finish_kernel chained)" if short
                                else "decode_kernel (persistent rank-space split-K decode)"),
                     "per_launch_bytes": alg_bytes // cfg.layers,
                     "per_launch_us": ms_step * 1e3 / cfg.layers},
        "cpu_baseline": cpu,
        "e2e": {"value": replica_throughput(world, tokens, e_ms), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e_ms,
                "how": "per step: every layer's q and tails copied from pinned host memory in %d copies on a "
                       "second stream, each releasing a captured graph of its layers' calls, then one copy "
                       "of every layer's output to pinned host memory" % nseg},
        "gpu_launches": kernels_per_layer * cfg.layers * args.steps,
        "clocks": clocks.summary(),
        "parity_check": check,
        "setup_s": t_gen,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    for p in plans:
        p.close()
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
