"""One prefill split over ranks by (batch, KV head) pairs, on the CPU.

Alg. 1 treats every query head on its own, and a query head reads only its KV
head, so the B * Hkv pairs (each with its G query heads) are independent
problems.  Checked here: the partition covers every pair exactly once with
the query heads following their KV head, and two gloo ranks that each run the
fp64 oracle on their shard and all-gather the outputs reproduce the
whole-problem oracle bit for bit."""
import os
import socket
import sys

import numpy as np
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from paper_2505_11254_gb300.replicas import head_shard, shard_views  # noqa: E402

PROBLEM = dict(B=2, Hq=8, Hkv=2, N=96, d=16, n_sink=2, window=20, gamma=8)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _problem():
    p = PROBLEM
    g = torch.Generator().manual_seed(5)
    Q = torch.randn((p["B"], p["Hq"], p["N"], p["d"]), generator=g).to(torch.bfloat16)
    K = (1.5 * torch.randn((p["B"], p["Hkv"], p["N"], p["d"]), generator=g)).to(torch.bfloat16)
    V = torch.randn((p["B"], p["Hkv"], p["N"], p["d"]), generator=g).to(torch.bfloat16)
    return Q, K, V


def _bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def test_partition_covers_every_pair_once():
    for B in (1, 2, 3):
        for Hkv in (1, 2, 8):
            for world in (1, 2, 3, 4, 8, 16):
                ranges = [head_shard(B, Hkv, r, world) for r in range(world)]
                assert ranges[0][0] == 0 and ranges[-1][1] == B * Hkv
                assert all(a[1] == b[0] for a, b in zip(ranges, ranges[1:])), "contiguous, no overlap"
                sizes = [p1 - p0 for p0, p1 in ranges]
                assert max(sizes) - min(sizes) <= 1, "balanced"


def test_query_heads_follow_their_kv_head():
    Q, K, V = _problem()
    B, Hq, Hkv = PROBLEM["B"], PROBLEM["Hq"], PROBLEM["Hkv"]
    G = Hq // Hkv
    for world in (1, 2, 3):
        for r in range(world):
            p0, p1 = head_shard(B, Hkv, r, world)
            q, k, v = shard_views(Q, K, V, Hkv, p0, p1)
            for i, pair in enumerate(range(p0, p1)):
                b, g = divmod(pair, Hkv)
                assert torch.equal(q[i], Q[b, g * G:(g + 1) * G])
                assert torch.equal(k[i, 0], K[b, g]) and torch.equal(v[i, 0], V[b, g])


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import oracle
    from paper_2505_11254_gb300.replicas import Replicas, gather_shards, head_shard, shard_views
    rep = Replicas().init(backend="gloo")
    p = PROBLEM
    Q, K, V = _problem()
    p0, p1 = head_shard(p["B"], p["Hkv"], rank, world)
    q, k, v = shard_views(Q, K, V, p["Hkv"], p0, p1)
    part = oracle.delta_attn(_bits(q), _bits(k), _bits(v), p["n_sink"], p["window"], p["gamma"])["A"]
    whole = gather_shards(torch.from_numpy(part), p["B"], p["Hq"], p["Hkv"], world)
    out.put((rank, p1 - p0, whole.numpy()))
    rep.barrier()
    rep.close()


def test_two_gloo_ranks_reproduce_the_whole_problem():
    import oracle
    p = PROBLEM
    Q, K, V = _problem()
    ref = oracle.delta_attn(_bits(Q), _bits(K), _bits(V), p["n_sink"], p["window"], p["gamma"])["A"]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for pr in procs:
        pr.start()
    res = sorted((q.get(timeout=180) for _ in procs), key=lambda x: x[0])
    for pr in procs:
        pr.join(timeout=60)
        assert pr.exitcode == 0
    assert [r[1] for r in res] == [2, 2], "each rank holds two of the four pairs"
    for _, _, whole in res:
        assert whole.shape == ref.shape and np.array_equal(whole, ref), "bit-identical to the whole problem"
