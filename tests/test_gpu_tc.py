"""GPU parity of the tensor-core selection path (bf16 prefill-like layouts):
approximate top-k (K = r) and exact top-k (K = d) against the fp64 oracle."""
import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import RECALL_ABS, check_topk_rows, f32, to_dev

pytestmark = pytest.mark.gpu
D = 128


def _causal_layout(lens, starts=None):
    off = np.zeros(len(lens) + 1, np.int64)
    off[1:] = np.cumsum(lens)
    q_seq, q_vis = [], []
    for s, L in enumerate(lens):
        first = 0 if starts is None else starts[s]
        for t in range(first, L):
            q_seq.append(s)
            q_vis.append(t + 1)
    return off, np.array(q_seq, np.int32), np.array(q_vis, np.int64)


def _run_score(lib, Hq, Hk, r, k, off, q_seq, q_vis, Q, L, sk, flags=0, nu=None):
    import torch
    T = len(q_seq)
    cfg = lib.make_config(Hq, Hk, r, k, "bf16", flags=flags, center=1 if nu is not None else 0)
    lay = lib.HostLayout(off, q_seq, q_vis)
    idx = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
    sc = torch.empty((Hq, T, k), dtype=torch.float32, device="cuda")
    ws = torch.empty(lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay), dtype=torch.uint8, device="cuda")
    lib.saki_score_topk(cfg, lay, to_dev(Q, "bf16"), f32(L), to_dev(sk, "bf16"), idx, score=sc,
                        nu=None if nu is None else f32(nu), workspace=ws)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), sc.cpu().numpy()


def _random_case(Hq, r, lens, seed, starts=None):
    rng = np.random.default_rng(seed)
    off, q_seq, q_vis = _causal_layout(lens, starts)
    T, N = len(q_seq), int(off[-1])
    Q = synth.round_to_bf16_grid(rng.standard_normal((Hq, T, D)).astype(np.float32))
    L = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    sk = O.round_bf16(rng.standard_normal((Hq, N, r))).astype(np.float32)
    return off, q_seq, q_vis, Q, L, sk


@pytest.mark.parametrize("r", [16, 32, 64, 128])
def test_tc_score_topk_causal(lib, r):
    Hq, Hk, k = 4, 2, 64
    off, q_seq, q_vis, Q, L, sk = _random_case(Hq, r, (700,), seed=r)
    idx, sc = _run_score(lib, Hq, Hk, r, k, off, q_seq, q_vis, Q, L, sk)
    waived = 0
    for h in range(Hq):
        rows = [O.approx_scores(Q[h, t], L[h], sk[h, :q_vis[t]]) for t in range(len(q_seq))]
        waived += check_topk_rows(idx[h], rows, k, gpu_scores=sc[h], label=f"r{r} h{h}")[1]
    assert waived <= 0.05 * Hq * len(q_seq)


@pytest.mark.parametrize("k,flags", [(16, 1), (33, 0), (64, 1), (1, 0)])
def test_tc_score_topk_multi_sequence(lib, k, flags):
    """Two prefill sequences, the second starting mid-way; sorted and unsorted lists."""
    Hq, Hk, r = 2, 1, 32
    off, q_seq, q_vis, Q, L, sk = _random_case(Hq, r, (300, 900), seed=k, starts=(0, 500))
    idx, sc = _run_score(lib, Hq, Hk, r, k, off, q_seq, q_vis, Q, L, sk, flags=flags)
    for h in range(Hq):
        rows = [O.approx_scores(Q[h, t], L[h], sk[h, off[q_seq[t]]:off[q_seq[t]] + q_vis[t]])
                for t in range(len(q_seq))]
        check_topk_rows(idx[h], rows, k, gpu_scores=sc[h], label=f"k{k} h{h}")
        if flags & 1:
            for t in range(len(q_seq)):
                v = sc[h, t][idx[h, t] >= 0]
                assert np.all(np.diff(v) <= 0)


def test_tc_score_topk_exact_ties(lib):
    """Integer-valued u and codes make many exactly equal scores: the selection must
    be the oracle's, including the lower-index rule for ties (no tolerance)."""
    Hq, Hk, r, k = 2, 1, 32, 64
    rng = np.random.default_rng(9)
    off, q_seq, q_vis = _causal_layout((600,))
    T, N = len(q_seq), int(off[-1])
    Q = np.zeros((Hq, T, D), np.float32)
    Q[:, np.arange(T), np.arange(T) % D] = 1.0                  # one-hot queries: u = row of L
    L = rng.integers(-1, 2, (Hq, D, r)).astype(np.float32)
    sk = rng.integers(-2, 3, (Hq, N, r)).astype(np.float32)    # integer scores in [-64, 64]
    for flags in (0, 1):
        idx, sc = _run_score(lib, Hq, Hk, r, k, off, q_seq, q_vis, Q, L, sk, flags=flags)
        for h in range(Hq):
            for t in range(T):
                s = O.approx_scores(Q[h, t], L[h], sk[h, :q_vis[t]])
                ref, val = O.topk(s, k)
                got = idx[h, t]
                assert set(got[got >= 0].tolist()) == set(ref[ref >= 0].tolist()), (flags, h, t)
                if flags:
                    np.testing.assert_array_equal(got, ref)


def test_tc_score_topk_mean_term(lib):
    Hq, r, k = 2, 32, 64
    off, q_seq, q_vis, Q, L, sk = _random_case(Hq, r, (400,), seed=5)
    nu = np.random.default_rng(6).standard_normal((Hq, D)).astype(np.float32)
    idx, sc = _run_score(lib, Hq, 1, r, k, off, q_seq, q_vis, Q, L, sk, nu=nu)
    for h in range(Hq):
        rows = [O.approx_scores(Q[h, t], L[h], sk[h, :q_vis[t]]) + float(Q[h, t].astype(np.float64) @ nu[h])
                for t in range(len(q_seq))]
        check_topk_rows(idx[h], rows, k, gpu_scores=sc[h], label=f"nu h{h}")


def test_tc_exact_topk_and_recall(lib):
    """saki_recall on a bf16 prefill layout takes the tensor-core exact path (K = d)."""
    import torch
    w = synth.Workload("tcx", 8, 2, rank=32, dtype="bf16", n_calib=512, seq_lens=(640,), spikes=(6, 6), seed=21)
    data = synth.make_numpy(w)
    ref = O.fit(data["q_calib"], data["k_calib"], data["A"], w.rank, center=False)
    sketch = O.build_index(data["K"], ref["R"], None, "bf16", w.group)
    ia, _ = O.score_topk(data["Q"], ref["L"], sketch, data["seq_offsets"], data["q_seq"], data["q_visible"], w.topk)
    ie, _ = O.exact_topk(data["Q"], data["A"], data["K"], data["seq_offsets"], data["q_seq"], data["q_visible"],
                         w.topk, w.group)
    cfg = lib.make_config(w.num_q_heads, w.num_kv_heads, w.rank, w.topk, "bf16")
    lay = lib.HostLayout(data["seq_offsets"], data["q_seq"], data["q_visible"])
    T = len(data["q_seq"])
    idx_e = torch.empty((w.num_q_heads, T, w.topk), dtype=torch.int32, device="cuda")
    rec = torch.empty((w.num_q_heads,), device="cuda")
    lib.saki_recall(cfg, lay, w.topk + 1, to_dev(data["Q"], "bf16"), f32(data["A"]), to_dev(data["K"], "bf16"),
                    torch.from_numpy(ia.astype(np.int32)).cuda(), rec, idx_exact=idx_e)
    idx_e = idx_e.cpu().numpy()
    waived = 0
    for h in range(w.num_q_heads):
        rows = [O.exact_scores(data["Q"][h, t], data["A"][h], data["K"][h // w.group, :data["q_visible"][t]])
                for t in range(T)]
        waived += check_topk_rows(idx_e[h], rows, w.topk, label=f"exact h{h}")[1]
    ref_rec = O.head_recall(ia, ie, data["q_visible"], w.topk + 1, w.topk)
    np.testing.assert_allclose(rec.cpu().numpy(), ref_rec, atol=RECALL_ABS + waived / (w.topk * (T - w.topk)))


def test_tc_end_to_end_bf16(lib):
    """fit -> index -> tensor-core select -> tensor-core exact + recall on a bf16
    prefill workload, against the oracle chain (recall within 1e-3 per head)."""
    import torch
    w = synth.Workload("tce2e", 8, 2, rank=32, dtype="bf16", n_calib=1024, seq_lens=(1024,), spikes=(2, 16), seed=22)
    data = synth.make_numpy(w)
    Hq, Hk, r, k = w.num_q_heads, w.num_kv_heads, w.rank, w.topk
    T, N = len(data["q_seq"]), data["K"].shape[1]
    cfg = lib.make_config(Hq, Hk, r, k, "bf16")
    L = torch.empty((Hq, D, r), device="cuda")
    R = torch.empty((Hq, D, r), device="cuda")
    Qd, Kd, Ad = to_dev(data["Q"], "bf16"), to_dev(data["K"], "bf16"), f32(data["A"])
    lib.saki_fit(cfg, to_dev(data["q_calib"], "bf16"), to_dev(data["k_calib"], "bf16"), Ad, L, R)
    sk = torch.empty((Hq, N, r), dtype=torch.bfloat16, device="cuda")
    lib.saki_build_index(cfg, Kd, R, sk)
    lay = lib.HostLayout(data["seq_offsets"], data["q_seq"], data["q_visible"])
    idx = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
    lib.saki_score_topk(cfg, lay, Qd, L, sk, idx)
    rec = torch.empty((Hq,), device="cuda")
    lib.saki_recall(cfg, lay, k + 1, Qd, Ad, Kd, idx, rec)
    ref = O.fit(data["q_calib"], data["k_calib"], data["A"], r, center=False)
    sketch = O.build_index(data["K"], ref["R"], None, "bf16", w.group)
    ia, _ = O.score_topk(data["Q"], ref["L"], sketch, data["seq_offsets"], data["q_seq"], data["q_visible"], k)
    ie, _ = O.exact_topk(data["Q"], data["A"], data["K"], data["seq_offsets"], data["q_seq"], data["q_visible"], k,
                         w.group)
    ref_rec = O.head_recall(ia, ie, data["q_visible"], k + 1, k)
    got = rec.cpu().numpy()
    # bf16 codes built from the GPU's fp32 fit differ from the oracle's in rare
    # round-to-nearest decisions, which can swap near-tie keys: allow 1e-3 per head
    np.testing.assert_allclose(got, ref_rec, atol=RECALL_ABS)
