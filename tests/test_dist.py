"""The N>1 host logic of bench.py (replicas, barrier, max-over-ranks timing, whole-job
aggregation) on two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update({"RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    import bench
    r, w, local = bench.dist_env()
    dist = bench.init_dist(w, "gloo")
    bench.barrier(dist)
    # each rank "timed" its replica; the whole job takes as long as the slowest rank
    t = bench.max_over_ranks(10.0 + rank, dist)
    s = bench.sum_over_ranks(1.0, dist)
    q.put((r, w, local, t, s))
    dist.destroy_process_group()


def test_two_rank_timing_reduction():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[0] for o in out] == [0, 1]
    assert all(o[1] == 2 for o in out)
    assert all(o[3] == 11.0 for o in out)      # max over ranks
    assert all(o[4] == 2.0 for o in out)       # whole-job count


def test_single_process_has_no_collective():
    import bench
    assert bench.init_dist(1, "gloo") is None
    assert bench.max_over_ranks(3.5, None) == 3.5


def test_clock_summary_flags_throttling():
    import bench
    rows = [["0", "1965", "2070", "900.5", "0x0", "Not Active", "Not Active", "Not Active", "Not Active"],
            ["0", "1950", "2070", "1100.0", "0x4", "Not Active", "Not Active", "Not Active", "Active"],
            ["0", "345", "2070", "150.0", "0x0", "Not Active", "Not Active", "Not Active", "Not Active"]]
    c = bench.summarize_clocks(rows)
    assert c["sm_mhz"] == pytest.approx(1957.5)
    assert c["sm_max_mhz"] == 2070
    assert c["reasons"] == ["sw_power_cap"]


def test_launch_count_matches_grouping():
    import bench

    class T:
        def __init__(self, p):
            self.p = p

        def data_ptr(self):
            return self.p
    x1, x2 = T(1), T(2)
    specs = [(0, None, 2048, 2048, x1, None), (0, None, 256, 2048, x1, None),
             (0, None, 256, 2048, x1, None), (0, None, 2048, 2048, x2, None),
             (0, None, 16384, 2048, x1, None)]
    assert bench.count_launches(specs) == 3
