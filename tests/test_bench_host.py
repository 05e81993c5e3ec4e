"""Host-side logic of bench.py, on CPU: multi-rank aggregation over gloo
(world size 2, as torchrun would launch the replicas), the clock-sample
parser and the workload arithmetic."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each replica's timed region and launch count
        ms = [120.0, 180.0][rank]
        launches = [96, 100][rank]
        bench.barrier()
        q.put((rank, bench.max_over_ranks(ms), bench.sum_over_ranks(launches), bench.dist_env()))
    finally:
        dist.destroy_process_group()


def test_two_rank_aggregation_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, mx, sm, env in res:
        assert mx == 180.0          # the slowest replica sets the job time
        assert sm == 196.0          # launches summed over replicas
        assert env == (rank, rank, 2)


def test_single_process_aggregation_is_identity():
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.sum_over_ranks(7) == 7


def test_clock_parser():
    lines = [
        "1980, 2070, 650.5, Not Active, Not Active, Not Active, Not Active",
        "2010, 2070, 700.0, Not Active, Not Active, Not Active, Active",
        "345, 2070, 120.0, Not Active, Not Active, Not Active, Not Active",   # idle sample
        "garbage",
    ]
    c = bench.parse_clock_lines(lines)
    assert c["sm_mhz"] == pytest.approx(1995.0)
    assert c["sm_max_mhz"] == 2070.0
    assert c["reasons"] == ["sw_power_cap"]
    assert c["samples"] == 3
    assert bench.parse_clock_lines([])["sm_mhz"] is None


def test_attended_rows_follow_the_growth_law():
    cfg = bench.CONFIGS["long"]
    N = 1374
    assert bench.attended_rows(cfg, 1) == N                     # frame 1: no memory
    assert bench.attended_rows(cfg, 2) == 2 * N                 # anchor stored whole
    assert bench.attended_rows(cfg, 2000) - N == N + 1998 * 14  # |M_1999| = N + 1998 k


def test_default_window_is_centred_on_the_mean_attended_length():
    cfg = bench.CONFIGS["long"]
    S0 = bench.default_start_frame(cfg["frames"], 20)
    assert S0 == 991
    frames = bench.window_frames(S0, 20)
    assert frames[0] == 991 and frames[-1] == 1010
    # the memory grows linearly (Eq. 6), so the mean over the stream is the
    # middle frame's length; the window's mean is within one frame's k of it
    whole = bench.mean_attended(cfg, range(1, cfg["frames"] + 1))
    assert abs(bench.mean_attended(cfg, frames) - whole) <= cfg["k"]
    assert bench.default_start_frame(100, 20) == 41
    assert bench.default_start_frame(8, 6) == 2
    assert bench.default_start_frame(2000, 0) == 1 and bench.default_start_frame(50, 50) == 1


def test_reference_arm_line_uses_the_same_frames_and_config():
    """The oracle arm runs on CPU: its config equals the GPU arm's config for
    the same command line, and its steps sample the timed window."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "tiny",
                          "--steps", "3", "--warmup", "1"], cwd=root, capture_output=True,
                         text=True, timeout=300)
    assert out.returncode == 0, out.stderr[-2000:]
    d = json.loads(out.stdout.strip().splitlines()[-1])
    cfg = bench.CONFIGS["tiny"]
    S0 = bench.default_start_frame(cfg["frames"], 3)
    assert d["impl"] == "reference" and d["steps"] == 3 and d["warmup"] == 1
    assert d["config"] == json.loads(json.dumps(bench.bench_config(cfg, "tiny", S0, 3, 1)))
    assert d["config"]["first_frame"] == S0 == 4  # frames 4-6 of 8, centred on frame 5
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
    assert d["value"] > 0 and d["unit"] == bench.UNIT and d["metric"] == bench.METRIC


def test_cpulist_parser():
    assert bench.parse_cpulist("0-3,8,10-11\n") == {0, 1, 2, 3, 8, 10, 11}
    assert bench.parse_cpulist("72-143") == set(range(72, 144))
    assert bench.parse_cpulist("") == set()
