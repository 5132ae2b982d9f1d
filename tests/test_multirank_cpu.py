"""The N > 1 path of bench.py on CPU: each rank is an independent replica;
a gloo process group carries only the barrier and the timing reduction
(queries of all ranks over the slowest rank's time)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    os.environ.update({"RANK": str(rank), "LOCAL_RANK": str(rank), "WORLD_SIZE": str(world),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    import bench
    d = bench.Dist()
    d.barrier()
    # rank r processed (r + 1) * 1000 queries in (r + 1) seconds
    value, tmax = bench.aggregate(d, (rank + 1) * 1000.0, rank + 1.0)
    out[rank] = (value, tmax)
    d.close()


def test_replica_aggregation_two_ranks():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(world):
        value, tmax = out[r]
        assert tmax == 2.0                  # max over ranks
        assert value == pytest.approx(1500.0)  # (1000 + 2000) queries / 2 s


def test_single_rank_aggregation_is_identity():
    import bench
    d = bench.Dist()
    assert d.world == int(os.environ.get("WORLD_SIZE", "1"))
    if d.world == 1:
        assert bench.aggregate(d, 500.0, 2.0) == (250.0, 2.0)


def test_insert_roofline_arithmetic():
    """The insert's rooflines: 2 C d flops per row over the kernel time
    against SMs x 128 lanes x 2 flops x clock for the FP32 certify kernels;
    for the tensor kernel, 8 d + 16 bytes per row against the HBM peak (the
    bound: the flops at the TF32 peak take less time), with the TF32 and ALU
    figures beside it."""
    import bench
    import synth
    w = synth.WORKLOADS["scale"]
    flops = 2 * w.N * w.C * w.d
    alu = 152 * 128 * 2 * 2070e6 / 1e12
    r = bench.insert_summary(w, w.N, 20.0, 152, {"sm_max_mhz": 2070}, kernel=("k_certify_wt", 8.0, 62, 0, 0, 0))
    assert r["rows_per_s"] == w.N / 0.02
    assert abs(r["e2e"]["achieved"] - flops / 0.02 / 1e12) < 1e-9
    assert abs(r["roofline"]["achieved"] - flops / 0.008 / 1e12) < 1e-9
    assert abs(r["roofline"]["peak"] - alu) < 1e-9
    assert r["roofline"]["bound"] == "alu" and 0 < r["e2e"]["frac_alu"] < r["roofline"]["frac"] < 1
    assert r["kernel"] == "k_certify_wt" and abs(r["kernel_ms"] - 8.0 / 62) < 1e-12
    r = bench.insert_summary(w, w.N, 20.0, 152, {"sm_max_mhz": 2070},
                             kernel=("k_certify_tc", 5.0, 62, 2.6 * w.N, 0, 1234), tf32_peak=937.7, hbm_peak=6686.8)
    # bytes at the HBM peak take longer than the flops at the TF32 peak: HBM-bound
    nbytes = w.N * (8 * w.d + 16)
    assert nbytes / 6686.8e9 > flops / 937.7e12
    assert r["roofline"]["bound"] == "hbm" and r["roofline"]["peak"] == 6686.8
    assert abs(r["roofline"]["frac"] - nbytes / 0.005 / 1e9 / 6686.8) < 1e-12
    assert abs(r["roofline"]["tensor_equiv"]["frac"] - flops / 0.005 / 1e12 / 937.7) < 1e-12
    assert abs(r["roofline"]["alu_equiv"]["frac"] - flops / 0.005 / 1e12 / alu) < 1e-12
    assert r["rows_fp64_pass"] == 1234
    assert abs(r["roofline"]["refined_pairs_per_row"] - 2.6) < 1e-12
    r = bench.insert_summary(w, w.N, 20.0, 152, {"sm_max_mhz": 2070})
    assert r["roofline"]["achieved"] == r["e2e"]["achieved"]
