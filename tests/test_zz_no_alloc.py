"""saki_score_topk_noalloc -- the selection call for callers that cannot
allocate device memory (a plugin whose host framework owns the device pool, a
decode loop that must not risk cudaMalloc's device synchronisation).  It uses
the library's static device scratch instead of a workspace; its results must
match saki_score_topk's, call after call, since every call reuses that scratch.
This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import SCORE_REL, f32, to_dev

pytestmark = pytest.mark.gpu
D = 128


def _inputs(Hq, r, dtype, lens, q_vis, seed):
    rng = np.random.default_rng(seed)
    off = np.zeros(len(lens) + 1, np.int64)
    off[1:] = np.cumsum(lens)
    q_seq = np.concatenate([np.full(len(v), s, np.int32) for s, v in enumerate(q_vis)])
    vis = np.concatenate([np.asarray(v, np.int64) for v in q_vis])
    T, N = len(q_seq), int(off[-1])
    Q = synth.round_to_bf16_grid(rng.standard_normal((Hq, T, D)).astype(np.float32))
    L = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    sk = O.round_to(dtype, rng.standard_normal((Hq, N, r))).astype(np.float32)
    return off, q_seq, vis, Q, L, sk


def _compare(lib, cfg, lay, Q, L, sk, nu=None):
    """One saki_score_topk call with a workspace, then the no-alloc call on the
    same inputs; sets and scores must agree."""
    import torch
    Hq, T, k = Q.shape[0], Q.shape[1], cfg.topk
    Qd, Ld, skd = to_dev(Q, "bf16"), f32(L), to_dev(sk, "bf16")
    nud = None if nu is None else f32(nu)
    ref_i = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
    ref_s = torch.empty((Hq, T, k), dtype=torch.float32, device="cuda")
    lib.saki_score_topk(cfg, lay, Qd, Ld, skd, ref_i, score=ref_s, nu=nud)
    got_i = torch.full((Hq, T, k), -7, dtype=torch.int32, device="cuda")
    got_s = torch.zeros((Hq, T, k), dtype=torch.float32, device="cuda")
    lib.saki_score_topk_noalloc(cfg, lay, Qd, Ld, skd, got_i, score=got_s, nu=nud)
    lib.saki_noalloc_status()   # synchronises; raises if a bounded wait gave up
    ri, rs = ref_i.cpu().numpy(), ref_s.cpu().numpy()
    gi, gs = got_i.cpu().numpy(), got_s.cpu().numpy()
    for h in range(Hq):
        for t in range(T):
            assert set(gi[h, t].tolist()) == set(ri[h, t].tolist()), (h, t)
            finite = np.isfinite(rs[h, t])
            np.testing.assert_array_equal(np.isfinite(gs[h, t]), finite)
            scale = np.max(np.abs(rs[h, t][finite])) if finite.any() else 1.0
            np.testing.assert_allclose(gs[h, t][finite], rs[h, t][finite], rtol=0, atol=SCORE_REL * scale)


def test_noalloc_matches_workspace_path_on_consecutive_calls(lib):
    Hq, Hk, r, k = 4, 1, 32, 64
    cases = [
        # long decode sequence: the plan splits it, so candidate lists live in the scratch
        ((20000,), [[20000] * 8]),
        # a different, ragged layout right after, reusing the same scratch
        ((700, 50, 3000), [[700, 350], [50, 10], [3000, 2999, 1500, 64]]),
        # 192 tail queries of one 4096-key sequence: the tensor-core tile path
        # (projection split, mean terms and error word in the scratch)
        ((4096,), [list(range(3905, 4097))]),
    ]
    for n, (lens, q_vis) in enumerate(cases):
        off, q_seq, vis, Q, L, sk = _inputs(Hq, r, "bf16", lens, q_vis, seed=40 + n)
        tc_case = n == 2
        cfg = lib.make_config(Hq, Hk, r, k, "bf16", flags=lib.SAKI_FLAG_SORTED, center=1 if tc_case else 0)
        lay = lib.HostLayout(off, q_seq, vis)
        assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay) <= lib.SAKI_NOALLOC_SCRATCH_BYTES
        nu = np.random.default_rng(50 + n).standard_normal((Hq, D)).astype(np.float32) if tc_case else None
        _compare(lib, cfg, lay, Q, L, sk, nu)


def test_noalloc_runs_the_unseeded_plan_when_the_seeded_one_does_not_fit(lib):
    """32 decode groups of eight queries over 20,000 keys each, k = 100: the
    seeded plan (sample lists and seeds) needs more than the scratch holds, the
    plan without the sample pass fits, and the results are the same."""
    Hq, Hk, r, k = 4, 1, 32, 100
    lens = (20000,) * 32
    off, q_seq, vis, Q, L, sk = _inputs(Hq, r, "bf16", lens, [[20000] * 8] * 32, seed=60)
    cfg = lib.make_config(Hq, Hk, r, k, "bf16")
    lay = lib.HostLayout(off, q_seq, vis)
    seeded = lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay)
    unseeded = lib.saki_workspace_size(lib.make_config(Hq, Hk, r, k, "f32"), lib.SAKI_OP_SCORE_TOPK, lay)
    assert unseeded <= lib.SAKI_NOALLOC_SCRATCH_BYTES < seeded
    _compare(lib, cfg, lay, Q, L, sk)


def test_noalloc_rejects_layouts_beyond_its_scratch(lib):
    """Five million queries: even the work list alone exceeds the scratch.  The
    buffers are real and sized for the layout, so a regression that let the call
    run would still touch only valid memory; the call must refuse before any
    launch and leave the outputs untouched."""
    import torch
    Hq, r, k, N = 1, 32, 64, 16
    T = 5_000_000
    lay = lib.HostLayout(np.array([0, N], np.int64), np.zeros(T, np.int32), np.full(T, N, np.int64))
    cfg = lib.make_config(Hq, 1, r, k, "bf16")
    assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay) > lib.SAKI_NOALLOC_SCRATCH_BYTES
    Q = torch.zeros((Hq, T, D), dtype=torch.bfloat16, device="cuda")
    L = torch.zeros((Hq, D, r), dtype=torch.float32, device="cuda")
    sk = torch.zeros((Hq, N, r), dtype=torch.bfloat16, device="cuda")
    idx = torch.full((Hq, T, k), -7, dtype=torch.int32, device="cuda")
    st = lib._lib.saki_score_topk_noalloc(ctypes.byref(cfg), ctypes.byref(lay.c), Q.data_ptr(), L.data_ptr(),
                                          sk.data_ptr(), None, idx.data_ptr(), None, None)
    assert st == 6   # SAKI_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert bool((idx == -7).all())
    del Q, idx
    torch.cuda.empty_cache()
