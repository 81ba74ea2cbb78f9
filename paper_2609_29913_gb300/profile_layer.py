"""Run decode calls on the first layers of a named workload, for profilers.

  python -m paper_2609_29913_gb300.profile_layer --workload qwen7b-1L-1M-b8 \
      [--layers 1] [--calls 3] [--reconstruct [--rope-theta 1e6]] [--int8 device|host|direct]

Builds the plans of layers 0 .. layers-1 of the workload (seeded synthetic
inputs, as the benchmark draws them), then makes `calls` rounds of one
decode call per layer on the current stream, synchronises and checks every
plan's device status word.  Each call launches the kernels milo_call_info
names, so a profiler can select them by name and count (e.g. ncu -k
regex:batch_tc -s 1 -c 1 skips the first round's launch).  With
--reconstruct the calls go through milo_attn_decode_reconstruct (kernel
recon_kernel), with --rope-theta over pre-RoPE factors.  With --int8 the
plans hold their factors as INT8 codes (device memory or mapped host
memory) and every call is preceded by its staging kernel
(dequant_plan_kernel) into one device buffer; with --int8 direct the codes
stay in device memory and the chunk grid reads them itself (chunk_kernel's
INT8 variant, no staging).  It keeps the device
footprint to the chosen layers, well under the full workload's.
"""
from __future__ import annotations

import argparse
import sys

import numpy as np


def main(argv=None) -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", required=True)
    ap.add_argument("--layers", type=int, default=1)
    ap.add_argument("--calls", type=int, default=3)
    ap.add_argument("--reconstruct", action="store_true")
    ap.add_argument("--rope-theta", type=float, default=0.0)
    ap.add_argument("--int8", choices=("device", "host", "direct"), default=None)
    args = ap.parse_args(argv)

    import torch
    from . import build, milo, workloads

    build.build()
    cfg = workloads.by_name(args.workload)
    plans, layers = [], []
    for l in range(min(args.layers, cfg.layers)):
        layer = workloads.make_config_layer(cfg, l, device="cuda")
        plans.append(milo.Prefix.from_layer(layer))
        layers.append(layer)
    toffs = [torch.as_tensor(L.tail_offsets, device="cuda") for L in layers]
    if args.rope_theta > 0:
        for pre in plans:
            pre.set_rope(args.rope_theta)
    buf = None
    if args.int8:
        for pre in plans:
            pre.quantize_int8(to_host=args.int8 == "host")
        if args.int8 != "direct":
            buf = torch.empty(max(int(p.info["packed_bytes"]) for p in plans) + 128, dtype=torch.uint8,
                              device="cuda")
    max_tail = max(int(np.diff(L.tail_offsets).max()) for L in layers)
    for _ in range(args.calls):
        for L, pre, toff in zip(layers, plans, toffs):
            if buf is not None:
                pre.stage(buf)
            (pre.decode_reconstruct if args.reconstruct else pre.decode)(L.q, L.tail_k, L.tail_v, toff, max_tail)
    torch.cuda.synchronize()
    for pre in plans:
        if pre.status() != 0:
            print("device status word set", file=sys.stderr)
            return 1
    info = milo.milo_call_info(plans[0].plan, cfg.batch, max_tail)
    path = "reconstruct" if args.reconstruct else milo.PATH_NAMES[info['path']]
    print(f"{cfg.name}: {len(plans)} layer(s) x {args.calls} call(s), path {path}, "
          f"{info['kernels']} kernels per call, {info['blocks']} blocks in the prefix grid")
    for pre in plans:
        pre.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
