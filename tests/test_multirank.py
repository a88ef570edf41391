"""The bench's multi-rank host logic on CPU: world size 2 over gloo.

Ranks rendezvous on 127.0.0.1, meet at barriers, agree on the slowest rank's
time, count the steps of all ranks (weak scaling), share identical datastores
but draw their own sequences, and only rank 0 runs the reference arm.  No GPU
is touched: this is the path `torchrun --nproc-per-node N bench.py` takes
before and after its timed region.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank), CUDA_VISIBLE_DEVICES="")
    import sys
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    r, w, local = bench.dist_setup(ws)
    assert (r, w, local) == (rank, ws, rank) and dist.get_backend() == "gloo"
    bench.barrier(w)
    t_max = bench.max_over_ranks(10.0 + 5.0 * r, w)  # rank-dependent "timed region" in ms
    inp = bench.make_inputs(1e-4, 4, r, 3)
    ref = bench.run_reference(bench.parse_args(["--impl", "reference", "--steps", "1", "--warmup", "0"]), r, w) \
        if r != 0 else "skipped"
    bench.barrier(w)
    out[rank] = dict(t_max=t_max, value=bench.weak_value(8, w, t_max), ref=ref, seed=inp["seed"],
                     corpora=[np.asarray(T).copy() for T in inp["corpora"]], ctx=np.asarray(inp["ctx"]).copy())
    dist.destroy_process_group()


@pytest.mark.timeout(300)
def test_two_ranks_gloo():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(240)
        assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
        r0, r1 = out[0], out[1]
    # both ranks report the slowest rank's time, and the job counts both ranks' steps
    assert r0["t_max"] == r1["t_max"] == 15.0
    assert r0["value"] == pytest.approx(2 * 8 / 15e-3)
    # identical datastores, distinct per-rank sequences
    for a, b in zip(r0["corpora"], r1["corpora"]):
        assert np.array_equal(a, b)
    assert r0["seed"] != r1["seed"] and not np.array_equal(r0["ctx"], r1["ctx"])
    # the reference arm runs on rank 0 alone; the others return without work
    assert r1["ref"] is None


def test_weak_value_single_rank():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.weak_value(256, 1, 200.0) == pytest.approx(1280.0)
    assert bench.max_over_ranks(3.5, 1) == 3.5
