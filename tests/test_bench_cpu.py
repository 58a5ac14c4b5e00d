"""Host logic of bench.py that needs no GPU: the clock-record rule that
rejects a timing (a slowdown, or a clock stuck low with no reason), the
replica launch of `--gpus N` (torchrun on 127.0.0.1, rank 0 prints one line
with n_gpus = N), the whole-job throughput from the slowest rank's time over
gloo, and the tensor rate at a sampled clock."""

import bench


def rec(mhz, reasons, mx=2070.0):
    return {"sm_mhz": mhz, "sm_max_mhz": mx, "reasons": reasons, "samples": 10}


def test_power_cap_is_kept():
    assert not bench.clocks_rejected(rec(1672.0, ["sw_power_cap"]))
    assert not bench.clocks_rejected(rec(1200.0, ["sw_power_cap"]))


def test_slowdowns_are_rejected():
    for r in bench.SLOWDOWNS:
        assert bench.clocks_rejected(rec(2000.0, [r]))
        assert bench.clocks_rejected(rec(1600.0, ["sw_power_cap", r]))


def test_stuck_clock_without_reason_is_rejected():
    assert bench.clocks_rejected(rec(1000.0, []))
    assert not bench.clocks_rejected(rec(1900.0, []))


def test_no_record_is_not_rejected():
    assert not bench.clocks_rejected(None)


# ---------------------------------------------------------------- replicas
import json
import os
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_replica_command_runs_one_process_per_gpu_on_loopback():
    cmd = bench.replica_command(4, ["--steps", "3", "--gpus", "4"], 29555)
    assert cmd[:3] == [sys.executable, "-m", "torch.distributed.run"]
    assert "--nproc-per-node=4" in cmd and "--nnodes=1" in cmd
    assert cmd[cmd.index("--master-addr") + 1] == "127.0.0.1"
    assert cmd[cmd.index("--master-port") + 1] == "29555"
    assert cmd[-5] == os.path.join(ROOT, "bench.py") and cmd[-4:] == ["--steps", "3", "--gpus", "4"]


def test_tensor_peak_at_clock():
    # 152 SMs x 8192 FLOP/clk at 1800 MHz
    assert abs(bench.tensor_peak_at_clock(1800.0) - 152 * 8192 * 1.8e9 / 1e12) < 1e-9


def _line_worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench as b
        ms = b.max_over_ranks(20.0 + 5.0 * rank, world, device="cpu")
        q.put(b.result_line(world, 4, 4096, ms))
    finally:
        dist.destroy_process_group()


def test_two_replicas_report_the_whole_job():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    procs = [ctx.Process(target=_line_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    lines = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for ln in lines:
        assert ln["n_gpus"] == 2 and ln["ms_per_step"] == 25.0  # the slowest rank's time
        assert abs(ln["value"] - 2 * 4 * 4096 / 0.025) < 1e-6 and ln["scaling"] == "weak"


def test_gpus_flag_launches_the_replicas_itself():
    # --gpus 2 with no WORLD_SIZE set: bench.py starts two ranks through
    # torchrun; on the reference arm (CPU oracle) rank 0 alone measures and
    # prints, the other rank exits 0
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "tiny",
                        "--gpus", "2", "--steps", "2", "--warmup", "1"], capture_output=True, text=True, env=env,
                       timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [json.loads(x) for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    ln = lines[0]
    assert ln["impl"] == "reference" and ln["n_gpus"] == 2 and ln["steps"] == 2
    assert ln["config"]["workload"] == "tiny" and ln["value"] > 0
