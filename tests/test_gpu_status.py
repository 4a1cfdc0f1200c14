"""Failure reporting on the GPU without a fault: every wait inside the library's
tensor-core kernels is bounded, and a kernel whose wait runs out stops, sets
the error word in its workspace header and returns, leaving the context usable.
The test hook saki_debug_inject_stall makes the next launch's TMA producer issue
no loads, so the other roles' waits run out (about two seconds); the call must
then report SAKI_ERR_TIMEOUT (through SAKI_FLAG_CHECK or saki_workspace_status)
and the next call on the same workspace must succeed with correct results.
Stream capture is refused before anything is enqueued."""
import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import check_topk_rows, f32, to_dev

pytestmark = pytest.mark.gpu
D = 128
TIMEOUT = 7
UNSUPPORTED = 2


def _causal_case(Hq, r, n, seed):
    rng = np.random.default_rng(seed)
    off = np.array([0, n], np.int64)
    q_seq = np.zeros(n, np.int32)
    q_vis = np.arange(1, n + 1, dtype=np.int64)
    Q = synth.round_to_bf16_grid(rng.standard_normal((Hq, n, D)).astype(np.float32))
    L = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    sk = O.round_bf16(rng.standard_normal((Hq, n, r))).astype(np.float32)
    return off, q_seq, q_vis, Q, L, sk


def _check_selection(idx, Q, L, sk, q_vis, k):
    for h in range(idx.shape[0]):
        rows = [O.approx_scores(Q[h, t], L[h], sk[h, :q_vis[t]]) for t in range(len(q_vis))]
        check_topk_rows(idx[h], rows, k, label=f"h{h}")


def test_stalled_selection_reports_timeout_and_the_next_call_recovers(lib):
    import torch
    Hq, Hk, r, k, n = 2, 1, 32, 64, 384
    off, q_seq, q_vis, Q, L, sk = _causal_case(Hq, r, n, seed=71)
    lay = lib.HostLayout(off, q_seq, q_vis)
    Qd, Ld, skd = to_dev(Q, "bf16"), f32(L), to_dev(sk, "bf16")
    check = lib.make_config(Hq, Hk, r, k, "bf16", flags=lib.SAKI_FLAG_CHECK)
    plain = lib.make_config(Hq, Hk, r, k, "bf16")
    ws = torch.empty(lib.saki_workspace_size(plain, lib.SAKI_OP_SCORE_TOPK, lay), dtype=torch.uint8, device="cuda")
    idx = torch.empty((Hq, n, k), dtype=torch.int32, device="cuda")
    # a healthy call under SAKI_FLAG_CHECK reports ok
    lib.saki_score_topk(check, lay, Qd, Ld, skd, idx, workspace=ws)
    # the stalled launch: the call itself reports the timeout ...
    lib.saki_debug_inject_stall(lib.SAKI_KERNEL_SELECT)
    with pytest.raises(lib.SakiError) as e:
        lib.saki_score_topk(check, lay, Qd, Ld, skd, idx, workspace=ws)
    assert e.value.status == TIMEOUT
    # ... and without the flag the call returns at once and the workspace keeps the word
    lib.saki_debug_inject_stall(lib.SAKI_KERNEL_SELECT)
    lib.saki_score_topk(plain, lay, Qd, Ld, skd, idx, workspace=ws)
    with pytest.raises(lib.SakiError) as e:
        lib.saki_workspace_status(ws)
    assert e.value.status == TIMEOUT
    # the context is still usable: the next call clears the word and is correct
    idx.fill_(-7)
    lib.saki_score_topk(plain, lay, Qd, Ld, skd, idx, workspace=ws)
    lib.saki_workspace_status(ws)
    _check_selection(idx.cpu().numpy(), Q, L, sk, q_vis, k)


def test_stalled_exact_selection_reports_timeout(lib):
    import torch
    Hq, Hk, r, k, n = 2, 1, 32, 64, 256
    off, q_seq, q_vis, Q, _, _ = _causal_case(Hq, r, n, seed=72)
    rng = np.random.default_rng(73)
    K = synth.round_to_bf16_grid(rng.standard_normal((Hk, n, D)).astype(np.float32))
    A = (rng.standard_normal((Hq, D, D)) / np.sqrt(D)).astype(np.float32)
    lay = lib.HostLayout(off, q_seq, q_vis)
    cfg = lib.make_config(Hq, Hk, r, k, "bf16", flags=lib.SAKI_FLAG_CHECK)
    ia = torch.zeros((Hq, n, k), dtype=torch.int32, device="cuda")
    ie = torch.empty((Hq, n, k), dtype=torch.int32, device="cuda")
    rec = torch.empty((Hq,), device="cuda")
    args = (cfg, lay, k + 1, to_dev(Q, "bf16"), f32(A), to_dev(K, "bf16"), ia, rec)
    lib.saki_debug_inject_stall(lib.SAKI_KERNEL_EXACT)
    with pytest.raises(lib.SakiError) as e:
        lib.saki_recall(*args, idx_exact=ie)
    assert e.value.status == TIMEOUT
    lib.saki_recall(*args, idx_exact=ie)
    got = ie.cpu().numpy()
    for h in range(Hq):
        rows = [O.exact_scores(Q[h, t], A[h], K[0, :q_vis[t]]) for t in range(n)]
        check_topk_rows(got[h], rows, k, label=f"exact h{h}")


def test_stalled_decode_selection_reports_timeout(lib):
    """The tensor-core decode kernel (groups of at least four bf16 queries)."""
    import torch
    Hq, Hk, r, k, n = 2, 1, 32, 64, 3000
    rng = np.random.default_rng(74)
    off = np.array([0, n], np.int64)
    q_seq = np.zeros(8, np.int32)
    q_vis = np.full(8, n, np.int64)
    Q = synth.round_to_bf16_grid(rng.standard_normal((Hq, 8, D)).astype(np.float32))
    L = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    sk = O.round_bf16(rng.standard_normal((Hq, n, r))).astype(np.float32)
    lay = lib.HostLayout(off, q_seq, q_vis)
    cfg = lib.make_config(Hq, Hk, r, k, "bf16", flags=lib.SAKI_FLAG_CHECK)
    idx = torch.empty((Hq, 8, k), dtype=torch.int32, device="cuda")
    args = (cfg, lay, to_dev(Q, "bf16"), f32(L), to_dev(sk, "bf16"), idx)
    lib.saki_debug_inject_stall(lib.SAKI_KERNEL_SELECT)
    with pytest.raises(lib.SakiError) as e:
        lib.saki_score_topk(*args)
    assert e.value.status == TIMEOUT
    lib.saki_score_topk(*args)
    _check_selection(idx.cpu().numpy(), Q, L, sk, q_vis, k)


def test_stalled_index_build_reports_timeout(lib):
    import torch
    Hq, Hk, r, n = 8, 2, 32, 1000
    rng = np.random.default_rng(75)
    K = synth.round_to_bf16_grid(rng.standard_normal((Hk, n, D)).astype(np.float32))
    R = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    cfg = lib.make_config(Hq, Hk, r, 64, "bf16", flags=lib.SAKI_FLAG_CHECK)
    sk = torch.empty((Hq, n, r), dtype=torch.bfloat16, device="cuda")
    Kd, Rd = to_dev(K, "bf16"), f32(R)
    lib.saki_debug_inject_stall(lib.SAKI_KERNEL_BUILD)
    with pytest.raises(lib.SakiError) as e:
        lib.saki_build_index(cfg, Kd, Rd, sk)
    assert e.value.status == TIMEOUT
    lib.saki_build_index(cfg, Kd, Rd, sk)
    exact = np.stack([K[h // (Hq // Hk)].astype(np.float64) @ R[h].astype(np.float64) for h in range(Hq)])
    got = sk.float().cpu().numpy()
    assert np.mean(got == O.round_bf16(exact)) >= 0.999


def test_stream_capture_is_refused_before_anything_is_enqueued(lib):
    import torch
    Hq, Hk, r, k, n = 2, 1, 32, 64, 256
    off, q_seq, q_vis, Q, L, sk = _causal_case(Hq, r, n, seed=76)
    lay = lib.HostLayout(off, q_seq, q_vis)
    cfg = lib.make_config(Hq, Hk, r, k, "bf16")
    Qd, Ld, skd = to_dev(Q, "bf16"), f32(L), to_dev(sk, "bf16")
    idx = torch.empty((Hq, n, k), dtype=torch.int32, device="cuda")
    ws = torch.empty(lib.saki_workspace_size(cfg, lib.SAKI_OP_SCORE_TOPK, lay), dtype=torch.uint8, device="cuda")
    lib.saki_score_topk_noalloc(cfg, lay, Qd, Ld, skd, idx)   # the scratch address is looked up before capture
    torch.cuda.synchronize()
    codes = []
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for call in (lambda: lib.saki_score_topk(cfg, lay, Qd, Ld, skd, idx, workspace=ws),
                     lambda: lib.saki_score_topk_noalloc(cfg, lay, Qd, Ld, skd, idx)):
            try:
                call()
                codes.append(0)
            except lib.SakiError as e:
                codes.append(e.status)
    assert codes == [UNSUPPORTED, UNSUPPORTED]
    # nothing was enqueued, so an ordinary call afterwards runs normally
    lib.saki_score_topk(cfg, lay, Qd, Ld, skd, idx, workspace=ws)
    _check_selection(idx.cpu().numpy(), Q, L, sk, q_vis, k)
