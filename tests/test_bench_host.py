"""Host-side logic of bench.py for N > 1 (replicas): the max-over-ranks reduction and the
whole-job time-per-token figure, run as two gloo ranks on the CPU."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update({"RANK": str(rank), "LOCAL_RANK": str(rank), "WORLD_SIZE": str(world),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    d = bench.Dist("gloo")
    d.barrier()
    out[rank] = d.max(10.0 + 5.0 * rank)
    d.close()


def test_two_gloo_ranks_reduce_the_slowest_time():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        ps = [ctx.Process(target=_rank, args=(r, 2, port, out)) for r in range(2)]
        for p in ps:
            p.start()
        for p in ps:
            p.join(120)
            assert p.exitcode == 0
        assert dict(out) == {0: 15.0, 1: 15.0}


def test_whole_job_ms_per_token():
    # two replicas decoding 128 tokens each in at most 64 ms: 0.25 ms per token of the job
    assert bench.whole_job_ms_per_token(64.0, 128, 2) == 0.25
    assert bench.whole_job_ms_per_token(64.0, 128, 1) == 0.5


def test_single_process_dist_is_a_no_op(monkeypatch):
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    d = bench.Dist("gloo")
    assert d.world == 1 and d.max(3.5) == 3.5
    d.barrier()
    d.close()


def test_decode_weight_bytes_of_the_masks():
    """Weight bytes per decode token: 2.000 GB all bf16, 1.459 GB under FFN 5+5 + lm_head
    (the FFN blocks of 10 layers and the 262144 x 1152 table at one byte per weight)."""
    five = sum(1 << l for l in list(range(5)) + list(range(21, 26)))
    assert bench.decode_weight_bytes(0, 0, 0) == 26 * (1536 * 1152 + 1152 * 1024 + 3 * 6912 * 1152) * 2 + 262144 * 1152 * 2
    saved = 10 * 3 * 6912 * 1152 + 262144 * 1152
    assert bench.decode_weight_bytes(five, 0, 1) == bench.decode_weight_bytes(0, 0, 0) - saved
    assert bench.decode_weight_bytes(five, 0, 1) == pytest.approx(1.4586e9, rel=1e-4)
