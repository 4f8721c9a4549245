"""One rank of the multi-process CPU test (launched by torch.distributed.run with the gloo
backend): bench.py's barrier, max over ranks and whole-job rate, as the N-GPU bench uses them."""

import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

import bench  # noqa: E402


def main():
    world, rank, _ = bench.dist_env()
    bench.init_dist(world, "gloo")
    bench.barrier(world)
    ms = 100.0 + 10.0 * rank  # rank r "took" 100 + 10 r ms
    slowest = bench.max_over_ranks(ms, world, "cpu")
    rate = bench.whole_job_rate(1000, 5, world, slowest)
    bench.barrier(world)
    # one file per rank: the ranks' standard outputs interleave under torch.distributed.run
    with open(os.path.join(os.environ["OPD_TEST_OUT"], f"rank{rank}.json"), "w") as f:
        json.dump({"rank": rank, "world": world, "max_ms": slowest, "rate": rate}, f)
    torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
