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


def test_noalloc_matches_workspace_path_on_consecutive_calls(lib):
    import torch
    Hq, Hk, r, k = 4, 1, 32, 64
    cases = [
        # long decode sequence: the plan splits it, so candidate lists live in the scratch
        ((20000,), [[20000] * 8]),
        # a different, ragged layout right after, reusing the same scratch
        ((700, 50, 3000), [[700, 350], [50, 10], [3000, 2999, 1500, 64]]),
    ]
    for n, (lens, q_vis) in enumerate(cases):
        off, q_seq, vis, Q, L, sk = _inputs(Hq, r, "bf16", lens, q_vis, seed=40 + n)
        cfg = lib.make_config(Hq, Hk, r, k, "bf16", flags=lib.SAKI_FLAG_SORTED)
        lay = lib.HostLayout(off, q_seq, vis)
        assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay) <= lib.SAKI_NOALLOC_SCRATCH_BYTES
        Qd, Ld, skd = to_dev(Q, "bf16"), f32(L), to_dev(sk, "bf16")
        T = len(q_seq)
        ref_i = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
        ref_s = torch.empty((Hq, T, k), dtype=torch.float32, device="cuda")
        lib.saki_score_topk(cfg, lay, Qd, Ld, skd, ref_i, score=ref_s)
        got_i = torch.full((Hq, T, k), -7, dtype=torch.int32, device="cuda")
        got_s = torch.zeros((Hq, T, k), dtype=torch.float32, device="cuda")
        lib.saki_score_topk_noalloc(cfg, lay, Qd, Ld, skd, got_i, score=got_s)
        torch.cuda.synchronize()
        ri, rs = ref_i.cpu().numpy(), ref_s.cpu().numpy()
        gi, gs = got_i.cpu().numpy(), got_s.cpu().numpy()
        for h in range(Hq):
            for t in range(T):
                assert set(gi[h, t].tolist()) == set(ri[h, t].tolist()), (n, h, t)
                finite = np.isfinite(rs[h, t])
                np.testing.assert_array_equal(np.isfinite(gs[h, t]), finite)
                scale = np.max(np.abs(rs[h, t][finite])) if finite.any() else 1.0
                np.testing.assert_allclose(gs[h, t][finite], rs[h, t][finite], rtol=0, atol=SCORE_REL * scale)


def test_noalloc_rejects_layouts_beyond_its_scratch(lib):
    Hq = 1
    T = 5_000_000   # the work list alone needs more than the static scratch holds
    lay = lib.HostLayout(np.array([0, 16], np.int64), np.zeros(T, np.int32), np.full(T, 16, np.int64))
    cfg = lib.make_config(Hq, 1, 32, 64, "bf16")
    assert lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay) > lib.SAKI_NOALLOC_SCRATCH_BYTES
    fake = 1 << 20   # aligned and never dereferenced: the call must stop before any launch
    st = lib._lib.saki_score_topk_noalloc(ctypes.byref(cfg), ctypes.byref(lay.c), fake, fake, fake, None, fake, None,
                                          None)
    assert st == 6   # SAKI_ERR_WORKSPACE
