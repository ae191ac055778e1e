"""The multi-rank plumbing of bench.py on CPU: two gloo ranks, the job time is the slowest
rank's (max over ranks) and every rank sees the same value; the barrier releases both."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

from conftest import ROOT


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench

    r, w, dist = bench.dist_init()
    assert (r, w) == (rank, world) and dist is not None
    bench.barrier(dist)
    got = bench.max_over_ranks(10.0 + 5.0 * rank, dist)
    q.put((rank, got))
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_max_over_ranks_gloo_two_ranks(monkeypatch):
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(90)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(2))
    assert res == [(0, 15.0), (1, 15.0)]


def test_single_process_needs_no_process_group(monkeypatch):
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    sys.path.insert(0, ROOT)
    import bench

    assert bench.dist_init() == (0, 1, None)
    assert bench.max_over_ranks(3.5, None) == 3.5


# ----------------------------------------------------------------------------- row sharding
def _oracle_row_ptr(N, d, S):
    import numpy as np

    import oracle

    counts = oracle.mask_counts(oracle.MaskSpec(N=N, mode=0, density=d, seeds=list(range(S))))
    return np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)


def test_row_split_balances_pairs():
    """Balanced cuts of a causal mask's rows: contiguous, non-empty, each part's pair count
    within one row's count of total / parts (rows near the end cost more)."""
    import numpy as np

    from paper_2607_21927_gb300 import ris

    rp = _oracle_row_ptr(3000, 0.05, 3)
    total = int(rp[-1])
    for parts in (1, 2, 3, 7, 64):
        b = ris.ris_row_split(rp, parts)
        assert b[0] == 0 and b[-1] == 3000 and all(b[k] < b[k + 1] for k in range(parts))
        sizes = [int(rp[b[k + 1]] - rp[b[k]]) for k in range(parts)]
        biggest_row = int(np.diff(rp).max())
        assert max(abs(sz - total / parts) for sz in sizes) <= biggest_row + 1
    b = ris.ris_row_split(np.arange(11, dtype=np.int64), 10)  # ten one-pair rows, ten parts
    assert b == list(range(11))
    with pytest.raises(ris.RisError):
        ris.ris_row_split(rp, 0)
    with pytest.raises(ris.RisError):
        ris.ris_row_split(rp, 3001)


def _shard_rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch
    import torch.distributed as dist

    from paper_2607_21927_gb300 import ris

    dist.init_process_group("gloo")
    # every rank derives the same counts (the mask is a pure function of its seeds) and takes
    # its own part: no exchange of mask data between ranks
    rp = _oracle_row_ptr(2000, 0.03, 2)
    b = ris.ris_row_split(rp, world)
    mine = torch.tensor([b[rank], b[rank + 1], int(rp[b[rank + 1]] - rp[b[rank]])], dtype=torch.int64)
    got = [torch.zeros(3, dtype=torch.int64) for _ in range(world)]
    dist.all_gather(got, mine)
    q.put((rank, [g.tolist() for g in got], int(rp[-1])))
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_row_shards_partition_rows_gloo(monkeypatch):
    """Two gloo ranks take balanced row ranges of the same mask: together they cover every row
    once and every sampled pair once."""
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_shard_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(90)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(2))
    parts, total = res[0][1], res[0][2]
    assert res[1][1] == parts
    assert parts[0][0] == 0 and parts[0][1] == parts[1][0] and parts[1][1] == 2000
    assert parts[0][2] + parts[1][2] == total and abs(parts[0][2] - parts[1][2]) <= 0.01 * total


def _kv_gather_rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch
    import torch.distributed as dist

    from paper_2607_21927_gb300 import inputs, ris, shard

    dist.init_process_group("gloo")
    N, Hkv, D = 2000, 2, 128
    # the same pure function on every rank: the mask's row counts and the balanced cuts
    rp = _oracle_row_ptr(N, 0.03, 2)
    b = ris.ris_row_split(rp, world)
    _, k, v = inputs.make_qkv(N, 6, Hkv, D, dtype=torch.bfloat16, seed=9, outliers=True)
    # this rank holds only its own rows of K and V
    k_full, v_full = shard.kv_allgather(k[b[rank]:b[rank + 1]].clone(), v[b[rank]:b[rank + 1]].clone(), b)
    q.put((rank, b, bool(torch.equal(k_full, k)), bool(torch.equal(v_full, v)), tuple(k_full.shape)))
    dist.destroy_process_group()


@pytest.mark.timeout(120)
@pytest.mark.parametrize("world", [2, 3])
def test_kv_allgather_of_row_shards_gloo(monkeypatch, world):
    """Ranks that hold only their own balanced row range of K and V rebuild the layer's whole K
    and V bit for bit with one all-gather each (ragged parts padded to the longest)."""
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_kv_gather_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(90)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(world))
    bounds = res[0][1]
    assert len(bounds) == world + 1 and len({tuple(r[1]) for r in res}) == 1
    assert len({bounds[k + 1] - bounds[k] for k in range(world)}) > 1  # ragged parts
    for rank, _, k_ok, v_ok, shape in res:
        assert k_ok and v_ok and shape == (2000, 2, 128), rank
