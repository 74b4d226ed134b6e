"""One rank of bench.py's replica harness on the CPU (`gloo`), for
tests/test_bench_spawn.py.

The step is a host sleep whose length depends on the rank (rank r sleeps
20 (r + 1) ms), standing in for one replica's work; nothing of the
attention is computed.  Each rank writes its own timing, rank 0 also the
job's fields, as JSON into the directory given on the command line.
"""
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import torch.distributed as dist  # noqa: E402

import bench  # noqa: E402


def main():
    out_dir, steps, ops = sys.argv[1], int(sys.argv[2]), float(sys.argv[3])
    world, rank, _ = bench.dist_env()
    dist.init_process_group("gloo")
    try:
        step = lambda: time.sleep(0.02 * (rank + 1))
        own_ms, job_ms = bench.time_replicas(step, steps, dist, bench.HostTimer())
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"rank": rank, "world": world, "ms": own_ms, "job_ms": job_ms}, f)
        if rank == 0:
            with open(os.path.join(out_dir, "job.json"), "w") as f:
                json.dump(bench.replica_fields(world, ops, steps, job_ms), f)
    finally:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
