"""One prefill split by rows over ranks (context parallelism), on the CPU.

The partition cuts the sequence at multiples of lcm(128, gamma) into
contiguous, balanced ranges.  Two gloo ranks each hold only their rows of Q,
K and V, exchange the K and V row shards (the one collective), evaluate the
fp64 oracle on their own rows, seeing zeros for every other rank's Q, and
all-gather the outputs: the result equals the whole-problem oracle bit for
bit, because Eq. 6 evaluates a row from its own query, its sample's query (in
the same range) and the keys up to it."""
import math
import os
import socket
import sys

import numpy as np
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from paper_2505_11254_gb300.replicas import context_shard  # noqa: E402

PROBLEM = dict(B=1, Hq=4, Hkv=2, N=700, d=16, n_sink=3, window=150, gamma=16)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _problem():
    p = PROBLEM
    g = torch.Generator().manual_seed(11)
    Q = torch.randn((p["B"], p["Hq"], p["N"], p["d"]), generator=g).to(torch.bfloat16)
    K = (1.5 * torch.randn((p["B"], p["Hkv"], p["N"], p["d"]), generator=g)).to(torch.bfloat16)
    V = torch.randn((p["B"], p["Hkv"], p["N"], p["d"]), generator=g).to(torch.bfloat16)
    return Q, K, V


def _bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def test_partition_is_contiguous_and_aligned():
    for N in (1, 127, 128, 700, 4096, 100000):
        for gamma in (1, 3, 16, 48, 64, 200):
            for world in (1, 2, 3, 4, 8):
                unit = math.lcm(128, gamma)
                ranges = [context_shard(N, gamma, r, world) for r in range(world)]
                assert ranges[0][0] == 0 and ranges[-1][1] == N
                assert all(a[1] == b[0] for a, b in zip(ranges, ranges[1:]))
                assert all(r0 % unit == 0 for r0, _ in ranges), "a range starts on a tile and a sample group"
                counts = [-(-(r1 - r0) // unit) for r0, r1 in ranges]
                assert max(counts) - min(counts) <= 1, "balanced in units"


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import oracle
    from paper_2505_11254_gb300.replicas import Replicas, context_shard, gather_context, gather_kv
    rep = Replicas().init(backend="gloo")
    p = PROBLEM
    Q, K, V = _problem()
    r0, r1 = context_shard(p["N"], p["gamma"], rank, world)
    # what this rank holds: its rows of Q, K and V
    Q_own, K_own, V_own = Q[:, :, r0:r1].clone(), K[:, :, r0:r1].clone(), V[:, :, r0:r1].clone()
    K_all, V_all = gather_kv(K_own, V_own, p["N"], p["gamma"], world)
    Q_seen = torch.zeros_like(Q)
    Q_seen[:, :, r0:r1] = Q_own
    part = oracle.delta_attn(_bits(Q_seen), _bits(K_all), _bits(V_all), p["n_sink"], p["window"], p["gamma"],
                             rows=(r0, r1))["A"]
    whole = gather_context(torch.from_numpy(part), p["N"], p["gamma"], world)
    out.put((rank, r1 - r0, whole.numpy()))
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
    assert [r[1] for r in res] == [384, 316], "rows per rank"
    for _, _, whole in res:
        assert whole.shape == ref.shape and np.array_equal(whole, ref), "bit-identical to the whole problem"
