"""A rank of a CPU stand-in for bench.py's multi-GPU run, started by bench.launch_ranks.

Each rank joins the process group through bench.init_dist (gloo on CPU, where the GPU run
uses NCCL), gathers one timing per rank and rank 0 prints the aggregate as one JSON line."""
import json
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402


def main():
    rank = int(os.environ["RANK"])
    world = int(os.environ["WORLD_SIZE"])
    dist = bench.init_dist(world, "cpu")
    times = bench.gather_times(dist, 0.5 + 0.25 * rank, "cpu")
    agg = bench.aggregate(64, 100, times)
    if rank == 0:
        print(json.dumps({"world": dist.get_world_size(), "backend": dist.get_backend(),
                          "times": times, "value": agg["value"]}), flush=True)
    dist.barrier()
    dist.destroy_process_group()


if __name__ == "__main__":
    main()
