"""Multi-GPU partition of the path, run as two gloo ranks on the CPU: the head
partition keeps GQA groups whole and its gathered per-head values equal the
single-process ones; the key-range split of a decode cache, with each rank's
local top k (the oracle on its range) exchanged and merged, equals the top k
over the whole range.  The merge here is the oracle's ranking of the union;
the library's saki_merge_topk is checked against the same on the GPU
(test_gpu_merge.py)."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import dist as D


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_blocks_cover_everything_once():
    for n in (0, 1, 5, 8, 13, 256):
        for world in (1, 2, 3, 8):
            got = [D.block(n, world, r) for r in range(world)]
            assert got[0][0] == 0 and got[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(got, got[1:]))
            sizes = [h - l for l, h in got]
            assert max(sizes) - min(sizes) <= 1


def test_head_range_keeps_gqa_groups_whole():
    Hq, Hk = 32, 8
    for world in (1, 2, 3, 8):
        seen = []
        for r in range(world):
            q0, q1, g0, g1 = D.head_range(Hq, Hk, world, r)
            assert (q0, q1) == (g0 * 4, g1 * 4)
            seen += [h // 4 for h in range(q0, q1)]
            assert all(g0 <= h // 4 < g1 for h in range(q0, q1))
        assert seen == [h // 4 for h in range(Hq)]
    with pytest.raises(ValueError):
        D.head_range(30, 8, 2, 0)


def _case():
    rng = np.random.default_rng(3)
    Hq, d, r, N, T, k = 3, 16, 8, 301, 4, 16
    Q = rng.standard_normal((Hq, T, d))
    L = rng.standard_normal((Hq, d, r))
    sketch = np.round(rng.standard_normal((Hq, N, r)) * 4) / 4     # quarter steps: many exact ties
    return Hq, N, T, k, Q, L, sketch


def _worker(rank, world, port, out):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        Hq, N, T, k, Q, L, sketch = _case()
        # key-range split: this rank's top k of its own range, part-local indices
        lo, hi = D.key_range(N, world, rank)
        off = np.array([0, hi - lo], np.int64)
        idx, sc = O.score_topk(Q, L, sketch[:, lo:hi], off, np.zeros(T, np.int32), np.full(T, hi - lo), k)
        ip, sp, offs = D.exchange_candidates(torch.from_numpy(idx.astype(np.int32)),
                                             torch.from_numpy(sc.astype(np.float32)), lo)
        # the union with global indices, ranked by the oracle (score desc, lower index)
        merged = np.full((Hq, T, k), -1, np.int64)
        for h in range(Hq):
            for t in range(T):
                cand = {}
                for p in range(world):
                    for j, s in zip(ip[p, h, t].tolist(), sp[p, h, t].tolist()):
                        if j >= 0:
                            cand[j + offs[p]] = s
                keys = np.array(sorted(cand))
                vals = np.array([cand[j] for j in keys])
                order = np.lexsort((keys, -vals))[:k]
                merged[h, t, :len(order)] = keys[order]
        # head partition: per-head values of this rank's heads, gathered in head order
        q0, q1, _, _ = D.head_range(8, 2, world, rank)
        local = torch.arange(q0, q1, dtype=torch.float32) * 0.5
        gathered = D.gather_head_values(local, 8, 2)
        out[rank] = (merged, offs, gathered.numpy())
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_key_range_split_reproduces_the_full_range_top_k(world):
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    Hq, N, T, k, Q, L, sketch = _case()
    ref, _ = O.score_topk(Q, L, sketch, np.array([0, N]), np.zeros(T, np.int32), np.full(T, N), k)
    for r in range(world):
        merged, offs, gathered = out[r]
        assert offs == [D.key_range(N, world, p)[0] for p in range(world)]
        np.testing.assert_array_equal(merged, ref)
        np.testing.assert_array_equal(gathered, np.arange(8) * 0.5)
