"""One rank of a CPU process group (gloo), launched by torchrun from
tests/test_bench_ranks.py: each replica reports a different step time and
takes the benchmark's aggregation of it over the group."""
import json
import os
import sys

import torch.distributed as dist

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402

rank, world = int(os.environ["RANK"]), int(os.environ["WORLD_SIZE"])
dist.init_process_group("gloo")
ms = 10.0 + 5.0 * rank                       # the higher ranks are the slower replicas
slowest = bench.max_over_ranks(ms, world, "cpu")
value = bench.job_tops(2.0e12, slowest, world)
results = [None] * world
dist.all_gather_object(results, {"rank": rank, "slowest_ms": slowest, "tops": value})
if rank == 0:    # one line: the ranks share stdout
    print(json.dumps({"world": world, "ranks": results}), flush=True)
dist.destroy_process_group()
