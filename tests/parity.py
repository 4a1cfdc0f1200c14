"""Helpers of the GPU parity tests: run the oracle and the CUDA library on the
same seeded inputs and compare them element by element.

Tolerances: top-k sets must be identical wherever the oracle's k-th/(k+1)-th
score gap exceeds GAP_REL x the row's largest |score|; reported scores agree
within SCORE_REL x that maximum (fp32 accumulation of bf16 inputs); recall
within RECALL_ABS; the rank-r map M_r within MAP_REL relative Frobenius."""
from __future__ import annotations

import numpy as np

from oracle import saki_oracle as O

GAP_REL = 1e-4     # top-k sets must match where the k-th/(k+1)-th gap exceeds this x row max |score|
SCORE_REL = 2e-3   # reported scores within this x row max |score|
MAP_REL = 1e-4     # M_r relative Frobenius error (heads with relative gap >= 1e-3)
RECALL_ABS = 1e-3


def to_dev(x, dtype: str, device="cuda"):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x))
    t = t.to(torch.bfloat16) if dtype == "bf16" else t.to(torch.float32)
    return t.to(device)


def f32(x, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(device)


def check_topk_rows(gpu_idx, rows_scores, k, gpu_scores=None, label=""):
    """gpu_idx [rows][k]; rows_scores: list of full oracle score vectors (visible
    prefix).  Returns the number of rows compared exactly and the number waived
    as near-ties (whose selections are still checked for validity)."""
    exact = waived = 0
    for r, s in enumerate(rows_scores):
        s = np.asarray(s, np.float64)
        got = np.asarray(gpu_idx[r])
        n = len(s)
        valid = got[got >= 0]
        assert len(valid) == min(n, k), (label, r, got)
        assert np.all(got[len(valid):] == -1) and np.all(got[:len(valid)] >= 0), (label, r, got)
        assert len(set(valid.tolist())) == len(valid), (label, r, "duplicate indices")
        assert np.all(valid < n), (label, r)
        if n == 0:
            continue
        mx = np.max(np.abs(s))
        ref_idx, ref_val = O.topk(s, k)
        if n <= k:
            assert set(valid.tolist()) == set(range(n)), (label, r)
            exact += 1
        else:
            srt = np.sort(s)[::-1]
            gap = srt[k - 1] - srt[k]
            if gap > GAP_REL * mx:
                assert set(valid.tolist()) == set(ref_idx.tolist()), (label, r, gap / mx)
                exact += 1
            else:
                # near-tie: the set is not unique at this margin, but every selected
                # key must score within the same margin of the oracle's k-th
                assert np.all(s[valid] >= srt[k - 1] - GAP_REL * mx), (label, r)
                waived += 1
        if gpu_scores is not None:
            gs = np.asarray(gpu_scores[r])[:len(valid)]
            np.testing.assert_allclose(gs, s[valid], atol=SCORE_REL * mx, rtol=0, err_msg=f"{label} row {r}")
    return exact, waived


def map_rel_err(L_gpu, R_gpu, M_ref):
    M = np.asarray(L_gpu, np.float64) @ np.asarray(R_gpu, np.float64).T
    return np.linalg.norm(M - M_ref) / np.linalg.norm(M_ref)


def recall_allowance(ref_rows, alt_rows, k, min_visible):
    """How far a head's recall may move when the approximate scores change from
    ``ref_rows`` (the oracle chain's) to ``alt_rows`` (the same formula evaluated
    on the library's fitted factors), counted row by row (Prop. 2).

    In a row where every score moved by at most e, a key can enter or leave the
    top k only if it scores within 2 e of the oracle's k-th score; each such key
    changes that row's recall by at most 1/k.  Returns the sum over qualifying
    rows of min(k, #such keys) / k, divided by the number of qualifying rows."""
    total, rows = 0.0, 0
    for s, t in zip(ref_rows, alt_rows):
        s = np.asarray(s, np.float64)
        if len(s) < min_visible:
            continue
        rows += 1
        e = float(np.max(np.abs(np.asarray(t, np.float64) - s)))
        kth = np.sort(s)[::-1][k - 1]
        m = int(np.sum(np.abs(s - kth) <= 2 * e)) if e > 0 else 0
        total += min(k, m) / k
    return total / max(1, rows)
