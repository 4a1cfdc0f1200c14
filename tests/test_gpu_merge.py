"""saki_merge_topk, the exchange step of a key-range split: the k best of
per-part lists must equal the oracle's ranking of their union (exact, ties by
the lower global index), and splitting a decode cache into ranges, selecting
each with saki_score_topk and merging must give the whole-range selection."""
import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import f32, to_dev

pytestmark = pytest.mark.gpu
D = 128


@pytest.mark.parametrize("k,parts", [(64, 2), (16, 5), (100, 3), (1, 4)])
def test_merge_equals_the_ranking_of_the_union(lib, k, parts):
    import torch
    rng = np.random.default_rng(k + parts)
    rows = 37
    offs = [0] + sorted(rng.choice(np.arange(1, 5000), parts - 1, replace=False).tolist())
    idx = np.full((parts, rows, k), -1, np.int32)
    sc = np.full((parts, rows, k), -np.inf, np.float32)
    for p in range(parts):
        span = (offs[p + 1] if p + 1 < parts else 6000) - offs[p]
        for r in range(rows):
            n = int(rng.integers(0, min(k, span) + 1))
            idx[p, r, :n] = rng.choice(span, n, replace=False)
            sc[p, r, :n] = rng.integers(-3, 4, n) * 0.5          # many equal scores
    cfg = lib.make_config(4, 1, 32, k, "bf16")
    out_i = torch.empty((rows, k), dtype=torch.int32, device="cuda")
    out_s = torch.empty((rows, k), dtype=torch.float32, device="cuda")
    lib.saki_merge_topk(cfg, torch.from_numpy(idx).cuda(), torch.from_numpy(sc).cuda(), offs, out_i, out_s)
    got_i, got_s = out_i.cpu().numpy(), out_s.cpu().numpy()
    for r in range(rows):
        keys = np.concatenate([idx[p, r][idx[p, r] >= 0] + offs[p] for p in range(parts)])
        vals = np.concatenate([sc[p, r][idx[p, r] >= 0] for p in range(parts)])
        order = np.lexsort((keys, -vals))[:k]
        ref = np.full(k, -1)
        ref[:len(order)] = keys[order]
        np.testing.assert_array_equal(got_i[r], ref, err_msg=f"row {r}")
        np.testing.assert_array_equal(got_s[r][:len(order)], vals[order])


def test_range_split_selection_merges_to_the_whole_range(lib):
    """A 20,000-key decode cache split in three ranges (as three GPUs would hold
    it): per-range saki_score_topk, then saki_merge_topk, equals one
    saki_score_topk over the whole cache, index for index."""
    import torch
    Hq, Hk, r, k, N, T = 4, 1, 32, 64, 20000, 8
    rng = np.random.default_rng(5)
    Q = synth.round_to_bf16_grid(rng.standard_normal((Hq, T, D)).astype(np.float32))
    L = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    sk = O.round_bf16(rng.standard_normal((Hq, N, r))).astype(np.float32)
    cfg = lib.make_config(Hq, Hk, r, k, "bf16", flags=lib.SAKI_FLAG_SORTED)
    Qd, Ld = to_dev(Q, "bf16"), f32(L)

    def select(lo, hi):
        lay = lib.HostLayout(np.array([0, hi - lo]), np.zeros(T, np.int32), np.full(T, hi - lo))
        i = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
        s = torch.empty((Hq, T, k), dtype=torch.float32, device="cuda")
        lib.saki_score_topk(cfg, lay, Qd, Ld, to_dev(np.ascontiguousarray(sk[:, lo:hi]), "bf16"), i, score=s)
        return i, s

    full_i, full_s = select(0, N)
    bounds = [0, 7001, 13500, N]
    parts = [select(a, b) for a, b in zip(bounds, bounds[1:])]
    out_i = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
    out_s = torch.empty((Hq, T, k), dtype=torch.float32, device="cuda")
    lib.saki_merge_topk(cfg, torch.stack([p[0] for p in parts]), torch.stack([p[1] for p in parts]), bounds[:-1],
                        out_i, out_s)
    np.testing.assert_array_equal(out_i.cpu().numpy(), full_i.cpu().numpy())
    np.testing.assert_array_equal(out_s.cpu().numpy(), full_s.cpu().numpy())
