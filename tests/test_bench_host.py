"""Host-side logic of the bench, on CPU: the multi-replica aggregation (one
process per GPU, launched by torch.distributed.run: job time = the slowest
rank's timed region, tokens = the sum over ranks), exercised with two gloo
ranks, and the algorithmic byte model its roofline divides by."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, ws, port, out_dir):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    ms, toks = bench.aggregate_over_ranks(10.0 + 5.0 * rank, 100 + rank, ws, device="cpu")
    with open(os.path.join(out_dir, f"r{rank}.txt"), "w") as f:
        f.write(f"{ms} {toks}")
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_take_max_time_and_sum_tokens(tmp_path):
    mp = pytest.importorskip("torch.multiprocessing")
    port = _free_port()
    mp.spawn(_rank, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    for r in range(2):
        ms, toks = open(tmp_path / f"r{r}.txt").read().split()
        assert float(ms) == 15.0 and int(toks) == 201


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_over_ranks(3.5, 7, 1) == (3.5, 7)


def test_roofline_byte_model_from_the_model_shapes():
    """The algorithmic bytes the bench divides by: the 8B target streams
    32 x 218.1 M layer parameters + the 525.3 M LM head + norms in bf16 (15.01 GB
    per forward), and each token of context costs 2 (K, V) x 32 layers x 8 kv
    heads x 128 x 2 B = 131072 B of KV read per verify; the K+1 verified rows
    write as much per row."""
    import synthetic as S
    sys.path.insert(0, ROOT)
    import bench as b
    wl = S.WORKLOADS["8b_greedy"]
    t = wl.target
    per_layer = 4096 * (32 * 128 + 2 * 8 * 128) + 32 * 128 * 4096 + 3 * 4096 * 14336 + 2 * 4096
    weights = 2 * (32 * per_layer + 128256 * 4096 + 4096)
    assert t.streamed_weight_bytes() == weights and abs(weights / 1e9 - 15.01) < 0.01
    assert t.kv_bytes_per_token() == 2 * 32 * 8 * 128 * 2 == 131072
    ctx = 600.0
    assert b.verify_bytes(wl, ctx) == weights + ctx * 131072 + (wl.K + 1) * 131072
    d = wl.draft
    assert b.draft_bytes(wl, ctx) == d.streamed_weight_bytes() + ctx * d.kv_bytes_per_token()
