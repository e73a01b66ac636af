"""One rank of the world-size-2 CPU test of bench.py's multi-rank logic (launched by
test_multirank_cpu.py the way torchrun launches the bench: RANK, WORLD_SIZE, MASTER_ADDR and
MASTER_PORT in the environment; gloo instead of NCCL)."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import torch  # noqa: E402
import torch.distributed as dist  # noqa: E402

import bench  # noqa: E402


def main():
    world, rank, local = bench.dist_env()
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # every rank reports a different elapsed time; the job's time is the slowest
    elapsed = bench.max_over_ranks(10.0 + 5.0 * rank, world, torch.device("cpu"))
    value = bench.whole_job_tokens_per_s(world, tokens_per_step=65536, steps=100, elapsed_ms=elapsed)
    dist.barrier()
    dist.destroy_process_group()
    print(json.dumps({"rank": rank, "world": world, "local": local, "elapsed": elapsed, "value": value}), flush=True)


if __name__ == "__main__":
    main()
