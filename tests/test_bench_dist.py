"""The multi-process paths of bench.py on CPU: world size 2 over gloo.

The (batch, head) pairs are independent, so N GPUs run N replicas: the only
cross-rank operations are the barrier and the max over ranks of the step time,
and the reference arm (the fp64 oracle) runs on rank 0 alone.
"""
import json
import os
import socket

import torch
import torch.multiprocessing as mp

import bench

WS = 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _env(rank, port):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      LOCAL_RANK=str(rank), WORLD_SIZE=str(WS))


def _max_worker(rank, port, out):
    _env(rank, port)
    ws, r, _ = bench.dist_env()
    bench.init_dist(ws, "gloo")
    bench.barrier(ws)
    m = bench.max_over_ranks(float(10 * (r + 1)), ws, torch.device("cpu"))
    bench.barrier(ws)
    torch.distributed.destroy_process_group()
    with open(os.path.join(out, f"max{rank}"), "w") as f:
        f.write(repr(m))


def _reference_worker(rank, port, out):
    _env(rank, port)
    import contextlib
    import io
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.main(["--impl", "reference", "--gpus", str(WS), "--workload",
                    "tiny_fp32_b1_h2_n256_d32", "--steps", "2", "--warmup", "3"])
    with open(os.path.join(out, f"ref{rank}"), "w") as f:
        f.write(buf.getvalue())


def test_max_over_ranks_gloo(tmp_path):
    mp.start_processes(_max_worker, args=(_free_port(), str(tmp_path)), nprocs=WS,
                       start_method="spawn")
    vals = [float((tmp_path / f"max{r}").read_text()) for r in range(WS)]
    assert vals == [10.0 * WS] * WS


def test_reference_arm_prints_on_rank0_only(tmp_path):
    import oracle
    oracle.load()  # build the C oracle once, before the ranks start
    mp.start_processes(_reference_worker, args=(_free_port(), str(tmp_path)), nprocs=WS,
                       start_method="spawn")
    out0 = (tmp_path / "ref0").read_text().strip().splitlines()
    out1 = (tmp_path / "ref1").read_text().strip()
    assert out1 == ""
    assert len(out0) == 1
    line = json.loads(out0[0])
    assert line["impl"] == "reference" and line["n_gpus"] == WS and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0
