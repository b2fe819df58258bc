"""One rank of the world-size-2 replica check (CPU, gloo backend).

Run by tests/test_multirank.py under ``torch.distributed.run``. Each rank draws
its replica's inputs with ``bench.rank_seed`` and reduces a rank-dependent
step time with ``bench.max_over_ranks``, the two pieces of host logic the
multi-GPU bench adds to a single-GPU run; it writes what it saw to
``<out_dir>/rank<r>.json``.
"""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import torch  # noqa: E402
import torch.distributed as dist  # noqa: E402

import bench  # noqa: E402
import workloads as W  # noqa: E402


def main() -> None:
    out_dir = sys.argv[1]
    dist.init_process_group("gloo")
    rank, world = dist.get_rank(), dist.get_world_size()
    step_ms = bench.max_over_ranks(1.5 + rank, torch.device("cpu"))
    w = W.make("tiny", seed=bench.rank_seed("tiny", rank))
    qsum = float(w.q.float().sum())
    qsums = [None] * world
    dist.all_gather_object(qsums, qsum)
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"rank": rank, "world": world, "max": step_ms, "qsums": qsums, "shape": list(w.q.shape)}, f)
    dist.destroy_process_group()


if __name__ == "__main__":
    main()
