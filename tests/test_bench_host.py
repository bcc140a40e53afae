"""Host-side pieces of bench.py: the visible-pair FLOP model against the oracle's
mask, and the multi-rank aggregation (max time over ranks, whole-job units) on a
world-size-2 gloo group."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import oracle
from paper_2607_08186_gb300.inputs import AttnShape, CROSS, LOCAL, WITHIN


@pytest.mark.parametrize("n,L", [(1, 9), (2, 7), (4, 5), (8, 3)])
def test_visible_pair_model_matches_oracle_mask(n, L):
    s = AttnShape(1, L, n, 1, 1, 64)
    for mode, w in ((WITHIN, 0), (CROSS, 0), (LOCAL, 3), (LOCAL, 100)):
        cnt = sum(oracle.visible(t, tk, n, mode, w) for t in range(1, s.nL + 1) for tk in range(1, s.nL + 1))
        assert bench.visible_pairs(s, mode, w) == cnt


@pytest.mark.parametrize("n,L", [(1, 9), (2, 7), (4, 5), (3, 6)])
def test_final_stream_pair_model_matches_oracle_mask(n, L):
    # the final-stream queries (1-indexed positions t = i*n) against every key position
    for mode, w in ((WITHIN, 0), (CROSS, 0), (LOCAL, 3), (LOCAL, 100)):
        count = sum(oracle.visible(i * n, tk, n, mode, w) for i in range(1, L + 1) for tk in range(1, n * L + 1))
        assert bench.final_pairs(L, n, mode, w) == count, (mode, w)


def test_flop_model_headline_workload():
    s = bench.SHAPES[bench.WORKLOAD]
    assert bench.visible_pairs(s, WITHIN) == 33_562_624
    assert bench.attn_flops(s, WITHIN, 14) == pytest.approx(1.924615110656e12)


def _free_port():
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        return sk.getsockname()[1]


def _worker(rank, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE="2")
    dist.init_process_group("gloo", rank=rank, world_size=2)
    try:
        secs = [0.5, 2.0][rank]
        val, tmax = bench.job_throughput(10.0, secs, 2)
        q.put((rank, val, tmax, bench.reduce_max(float(rank + 3), 2)))
    finally:
        dist.destroy_process_group()


def test_job_throughput_two_ranks_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = [q.get(timeout=120) for _ in range(2)]
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, val, tmax, m in res:
        assert tmax == 2.0                 # slowest rank's time
        assert val == pytest.approx(10.0)  # 2 ranks x 10 units / 2 s
        assert m == 4.0
