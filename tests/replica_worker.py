"""One rank of the replica timing check, launched by torchrun over gloo (CPU
only): each rank reports a different local step time, and every rank must
end with the slowest one and the whole job's throughput."""
import importlib.util
import json
import os
import sys

import torch.distributed as dist

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def main():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    dist.init_process_group("gloo")
    rank, world = dist.get_rank(), dist.get_world_size()
    local_ms = 1.0 + 2.5 * rank  # rank r's own step time
    dist.barrier()
    ms = bench.max_over_ranks(local_ms, dist, "cpu")
    value = bench.replica_throughput(world, int(sys.argv[1]), ms)
    dist.barrier()
    # one file per rank: the ranks' standard outputs interleave
    with open(os.path.join(sys.argv[2], f"rank{rank}.json"), "w") as f:
        json.dump({"rank": rank, "world": world, "local_ms": local_ms, "ms": ms, "value": value}, f)
    dist.destroy_process_group()


if __name__ == "__main__":
    main()
