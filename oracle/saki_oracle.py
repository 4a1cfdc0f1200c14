"""SAKI oracle: a plain, slow, fp64 CPU restatement of the paper's definitions.

TEST INFRASTRUCTURE.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this module.  It shares
no code with the CUDA library and imports nothing from it; its inputs are the
seeded arrays of the synthetic generator (or values the paper prints).

What it follows (sections and equations of arXiv 2608.03228, "SAKI"):

* Sec. 3 (Setup): scores ``s_ij = q_i^T A_h k_j``; GQA query head ``h`` reads
  KV group ``g(h) = floor(h / (Hq/Hk))`` (the paper names GQA without a
  mapping; this is the usual repeat-kv convention).
* Eq. (1): score distortion ``L(P) = tr[A(I-P) Sk (I-P)^T A^T Sq]``; with the
  rank-r score map ``M = A P`` this is ``|| Sq^{1/2} (A - M) Sk^{1/2} ||_F^2``.
* Prop. 1, Eq. (3) and App. A: ``C = Sq^{1/2} A Sk^{1/2}``, truncated SVD
  ``C_r = U_r Lambda_r V_r^T``, optimum ``M_r = Sq^{-1/2} C_r Sk^{-1/2}`` with
  ``L(M_r) = sum_{i>r} lambda_i(C)^2``; singular covariances use pseudoinverse
  roots, eigenvalues below ``1e-6 * lambda_max`` are treated as zero.
* Sec. 6 (SAKI): ``Sq`` uncentered second moment of queries, ``Sk`` and ``mu``
  from centered keys (uncentered keys are the ``mu = 0`` case, App. A
  "Centering"); factors ``B_q = Sq^{-1/2} U_r Lambda_r^{1/2}`` (called ``L``
  here) and ``B_k = Sk^{-1/2} V_r Lambda_r^{1/2}`` (called ``R``); key code
  ``c_j = R^T (k_j - mu)``; score ``s_hat = (L^T q)^T c_j + q^T A mu``.
* Sec. 3 protocol: recall of the true top-k attended positions, i.e. the
  fraction of the exact top-k set (by ``q^T A k``) found by the index.
* Tab. 1 (Sec. 3 baselines) comparison indexes: key PCA (the rank-r principal
  projector of the keys, M = A P) and weight SVD (the operator's truncated
  SVD, M = A_r).  Sec. 6's projector variants SAP-svd (the raw span of C's
  right singular vectors) and SAP-map (the optimum's key-side span,
  orthonormalised): the paper names them without formulas; the readings are
  the docstrings of ``sap_svd_head`` and ``sap_map_head``.

Readings where the paper is silent:

* lambda_i(C) in Eq. (3) are the singular values of the (non-symmetric) C.
* Moments are normalised by 1/n.
* The eigenvalue floor is a pseudo-inverse: floored eigenvalues are zero in
  both the root and the inverse root.
* Signs of singular vectors are arbitrary; ``canonical_signs`` flips each
  column pair (L[:, c], R[:, c]) so that the largest-magnitude entry of
  R[:, c] is positive.
* Ranking: descending score, equal scores broken by the lower key index.
* Sketch storage: codes are rounded to the sketch dtype (round-to-nearest-even)
  because that is what an index stores; query projections ``u = L^T q`` are
  kept exact.
* The mean term ``q^T A mu`` is a per-query constant: it is added to reported
  scores but cannot change a ranking, so ranking uses ``u . c`` alone.
"""
from __future__ import annotations

import numpy as np

F64 = np.float64


# --------------------------------------------------------------------------
# Sec. 6: calibration moments
# --------------------------------------------------------------------------
def moments(X, center: bool):
    """Second moment of the rows of X [n][d]: ``(1/n) sum_t x_t x_t^T``.

    ``center=True`` returns the covariance of the centered rows and their mean
    (keys, Sec. 6 / App. A "Centering"); ``center=False`` the uncentered second
    moment and a zero mean (queries, and the ``mu = 0`` special case)."""
    X = np.asarray(X, F64)
    n = X.shape[0]
    mu = X.mean(axis=0) if center else np.zeros(X.shape[1])
    Xc = X - mu
    return (Xc.T @ Xc) / n, mu


# --------------------------------------------------------------------------
# Prop. 1 / App. A: roots of the covariances with the eigenvalue floor
# --------------------------------------------------------------------------
def psd_roots(S, floor_rel: float = 1e-6):
    """Symmetric root ``S^{1/2}`` and pseudo-inverse root ``S^{+1/2}``.

    Eigenvalues below ``floor_rel * lambda_max`` count as zero in both (App. A,
    "Singular covariances")."""
    S = np.asarray(S, F64)
    lam, U = np.linalg.eigh(0.5 * (S + S.T))
    lmax = lam.max() if lam.size else 0.0
    keep = (lam > 0) & (lam >= floor_rel * lmax)
    Uk, lk = U[:, keep], lam[keep]
    root = (Uk * np.sqrt(lk)) @ Uk.T
    iroot = (Uk / np.sqrt(lk)) @ Uk.T
    return root, iroot


def canonical_signs(L, R):
    """Flip column pairs so that each R column's largest-|.| entry is positive."""
    L = L.copy()
    R = R.copy()
    for c in range(R.shape[1]):
        i = int(np.argmax(np.abs(R[:, c])))
        if R[i, c] < 0:
            R[:, c] = -R[:, c]
            L[:, c] = -L[:, c]
    return L, R


def fit_head(Sq, Sk, A, r: int, floor_rel: float = 1e-6) -> dict:
    """Prop. 1 (Eq. 3, Sec. 5) and the Sec. 6 factors for one head.

    Returns L = B_q [d][r], R = B_k [d][r], the score map M_r = L R^T, the
    singular values of C (all d, descending) and the optimum
    ``loss = sum_{i>r} sigma_i^2``."""
    A = np.asarray(A, F64)
    rq, iq = psd_roots(Sq, floor_rel)
    rk, ik = psd_roots(Sk, floor_rel)
    C = rq @ A @ rk
    U, sig, Vt = np.linalg.svd(C)
    V = Vt.T
    sh = np.sqrt(sig[:r])
    L = iq @ (U[:, :r] * sh)
    R = ik @ (V[:, :r] * sh)
    L, R = canonical_signs(L, R)
    M = iq @ (U[:, :r] * sig[:r]) @ V[:, :r].T @ ik
    return dict(L=L, R=R, M=M, sigma=sig, loss=float(np.sum(sig[r:] ** 2)), C=C)


def score_loss(M, A, Sq, Sk) -> float:
    """Eq. (1) written directly: ``tr[(A - M) Sk (A - M)^T Sq]``."""
    E = np.asarray(A, F64) - np.asarray(M, F64)
    return float(np.trace(E @ np.asarray(Sk, F64) @ E.T @ np.asarray(Sq, F64)))


def ledoit_wolf(X, center: bool):
    """Ledoit-Wolf shrinkage of the second moment of the rows of X [n][d] (Sec. 7
    applies it to both moments; Ledoit & Wolf 2004): S* = (1 - rho) S + rho m I
    with m = tr(S) / d, rho = min(b2, d2) / d2, d2 = ||S - m I||_F^2 and
    b2 = (1/n^2) sum_t ||x_t x_t^T - S||_F^2 (x_t centered when ``center``).
    Returns (S*, rho, mu)."""
    S, mu = moments(X, center)
    Xc = np.asarray(X, F64) - mu
    n, d = Xc.shape
    m = np.trace(S) / d
    d2 = float(np.sum((S - m * np.eye(d)) ** 2))
    b2 = sum(float(np.sum((np.outer(x, x) - S) ** 2)) for x in Xc) / n ** 2
    rho = min(b2, d2) / d2 if d2 > 0 else 0.0
    return (1 - rho) * S + rho * m * np.eye(d), rho, mu


def fit(q_calib, k_calib, A, rank: int, center: bool, floor_rel: float = 1e-6, shrink: bool = False) -> dict:
    """All heads: q_calib [Hq][n][d], k_calib [Hk][n][d], A [Hq][d][d].
    ``shrink`` replaces both moments by their Ledoit-Wolf shrinkage.

    Returns L, R [Hq][d][r]; M [Hq][d][d]; mu [Hk][d]; nu = A_h mu_g [Hq][d];
    sigma [Hq][d]; loss [Hq]; Sq [Hq][d][d]; Sk [Hk][d][d]."""
    Hq, Hk = len(q_calib), len(k_calib)
    G = Hq // Hk
    if shrink:
        Sk, _, mu = zip(*[ledoit_wolf(k_calib[g], center) for g in range(Hk)])
        Sq = [ledoit_wolf(q_calib[h], False)[0] for h in range(Hq)]
    else:
        Sk, mu = zip(*[moments(k_calib[g], center) for g in range(Hk)])
        Sq = [moments(q_calib[h], False)[0] for h in range(Hq)]
    out = {k: [] for k in ("L", "R", "M", "sigma", "loss", "nu")}
    for h in range(Hq):
        g = h // G
        res = fit_head(Sq[h], Sk[g], A[h], rank, floor_rel)
        for k in ("L", "R", "M", "sigma", "loss"):
            out[k].append(res[k])
        out["nu"].append(np.asarray(A[h], F64) @ mu[g])
    res = {k: np.array(v) for k, v in out.items()}
    res.update(mu=np.array(mu), Sq=np.array(Sq), Sk=np.array(Sk))
    return res


# --------------------------------------------------------------------------
# Tab. 1 comparison indexes: key PCA and weight SVD
# --------------------------------------------------------------------------
def key_pca_head(Sk, A, r: int, floor_rel: float = 1e-6) -> dict:
    """Key PCA for one head (Tab. 1; Sec. 5 states that PCA minimises
    ``||(I - P) Sk^{1/2}||_F^2``): P = V_r V_r^T projects onto the r leading
    eigenvectors of the key moment Sk, the score map is M = A P, and the
    factors are L = A V_r, R = V_r, so a key's code is its principal
    coordinates.  sigma are the square roots of Sk's eigenvalues (descending,
    the App. A floor applied) and loss is the discarded key energy
    ``sum_{i>r} lambda_i(Sk)``.  Directions whose eigenvalue is floored are
    left out (zero columns)."""
    lam, V = np.linalg.eigh(0.5 * (np.asarray(Sk, F64) + np.asarray(Sk, F64).T))
    order = np.argsort(-lam, kind="stable")
    lam, V = lam[order], V[:, order]
    lmax = lam[0] if lam.size else 0.0
    lam = np.where((lam > 0) & (lam >= floor_rel * lmax), lam, 0.0)
    R = V[:, :r] * (lam[:r] > 0)
    L = np.asarray(A, F64) @ R
    L, R = canonical_signs(L, R)
    return dict(L=L, R=R, M=L @ R.T, sigma=np.sqrt(lam), loss=float(np.sum(lam[r:])))


def weight_svd_head(A, r: int) -> dict:
    """Weight SVD for one head (Tab. 1; Sec. 4 (b)): the operator's own
    truncated SVD, blind to the data.  A = U Sigma V^T, L = U_r Sigma_r^{1/2},
    R = V_r Sigma_r^{1/2}, M = A_r; loss = ``sum_{i>r} sigma_i(A)^2``."""
    U, sig, Vt = np.linalg.svd(np.asarray(A, F64))
    sh = np.sqrt(sig[:r])
    L, R = canonical_signs(U[:, :r] * sh, Vt[:r].T * sh)
    return dict(L=L, R=R, M=(U[:, :r] * sig[:r]) @ Vt[:r], sigma=sig, loss=float(np.sum(sig[r:] ** 2)))


def _orth(X):
    """Orthonormal basis of the column span of X (d x r, full column rank) by
    modified Gram-Schmidt."""
    Q = np.array(X, F64)
    for c in range(Q.shape[1]):
        for p in range(c):
            Q[:, c] -= (Q[:, p] @ Q[:, c]) * Q[:, p]
        Q[:, c] /= np.linalg.norm(Q[:, c])
    return Q


def _projector_head(Q, A) -> dict:
    L, R = canonical_signs(np.asarray(A, F64) @ Q, Q)
    return dict(L=L, R=R, M=L @ R.T)


def sap_svd_head(Sq, Sk, A, r: int, floor_rel: float = 1e-6) -> dict:
    """SAP-svd (Sec. 6, Tab. 1): the projector onto the raw span of the r
    leading right singular vectors V_r of C = Sq^{1/2} A Sk^{1/2}, used directly
    as key-space directions (the whitening is not undone); M = A V_r V_r^T,
    L = A V_r, R = V_r."""
    rq, _ = psd_roots(Sq, floor_rel)
    rk, _ = psd_roots(Sk, floor_rel)
    _, _, Vt = np.linalg.svd(rq @ np.asarray(A, F64) @ rk)
    return _projector_head(Vt[:r].T, A)


def sap_map_head(Sq, Sk, A, r: int, floor_rel: float = 1e-6) -> dict:
    """SAP-map (Sec. 6, Tab. 1): the orthogonal projector onto the key-side span
    of the optimum M_r, i.e. span((Sk^{1/2})^+ V_r), with (Sk^{1/2})^+ the
    pseudo-inverse of the symmetric root (eigenvalues below the App. A floor
    count as zero), which is the column span of the factor R of ``fit_head``,
    orthonormalised; M = A Q Q^T, L = A Q, R = Q."""
    _, ik = psd_roots(Sk, floor_rel)
    rq, _ = psd_roots(Sq, floor_rel)
    rk, _ = psd_roots(Sk, floor_rel)
    _, _, Vt = np.linalg.svd(rq @ np.asarray(A, F64) @ rk)
    return _projector_head(_orth(ik @ Vt[:r].T), A)


def fit_baseline(method: str, k_calib, A, rank: int, center: bool, num_q_heads: int,
                 floor_rel: float = 1e-6) -> dict:
    """All heads of a comparison index, ``method`` "key_pca" or "weight_svd";
    the keys' moments and means follow the same centering reading as ``fit``
    (the mean term nu = A_h mu_g is unchanged).  Returns L, R, M, sigma, loss,
    mu, nu like ``fit``."""
    Hq, Hk = num_q_heads, len(k_calib)
    G = Hq // Hk
    Sk, mu = zip(*[moments(k_calib[g], center) for g in range(Hk)])
    out = {k: [] for k in ("L", "R", "M", "sigma", "loss", "nu")}
    for h in range(Hq):
        g = h // G
        res = key_pca_head(Sk[g], A[h], rank, floor_rel) if method == "key_pca" else weight_svd_head(A[h], rank)
        for k in ("L", "R", "M", "sigma", "loss"):
            out[k].append(res[k])
        out["nu"].append(np.asarray(A[h], F64) @ mu[g])
    res = {k: np.array(v) for k, v in out.items()}
    res.update(mu=np.array(mu), Sk=np.array(Sk))
    return res


# --------------------------------------------------------------------------
# Sec. 6: key codes (the index)
# --------------------------------------------------------------------------
def round_bf16(x):
    """Round fp64 values to the bf16 grid, nearest with ties to even.

    bf16 keeps 8 significant bits and the fp32 exponent range; below 2^-126
    its spacing is the fixed subnormal step 2^-133.  Magnitudes beyond the
    largest finite bf16 are not produced by this workload and raise."""
    x = np.asarray(x, F64)
    m, e = np.frexp(x)                         # x = m 2^e, 0.5 <= |m| < 1
    out = np.ldexp(np.rint(m * 256.0), e - 8)
    small = np.abs(x) < 2.0 ** -126
    out[small] = np.rint(x[small] * 2.0 ** 133) * 2.0 ** -133
    if np.any(np.abs(out) > 3.3895313892515355e38):
        raise OverflowError("value outside the bf16 range")
    return out


def round_to(dtype: str, x):
    """Storage rounding of an index entry: 'f32' (IEEE round-to-nearest-even)
    or 'bf16' (:func:`round_bf16`)."""
    if dtype == "f32":
        return np.asarray(x, F64).astype(np.float32).astype(F64)
    if dtype == "bf16":
        return round_bf16(x)
    raise ValueError(dtype)


def build_index(K, R, mu, dtype: str, group: int):
    """Key codes ``c_j = R_h^T (k_j - mu_g)`` for every query head h (Sec. 6).

    K [Hk][N][d]; R [Hq][d][r]; mu [Hk][d] or None.  Returns [Hq][N][r] rounded
    to the index dtype."""
    K = np.asarray(K, F64)
    Hq = R.shape[0]
    out = []
    for h in range(Hq):
        g = h // group
        kc = K[g] - (0.0 if mu is None else np.asarray(mu[g], F64))
        out.append(round_to(dtype, kc @ np.asarray(R[h], F64)))
    return np.array(out)


# --------------------------------------------------------------------------
# Selection: approximate and exact scores, top-k, recall
# --------------------------------------------------------------------------
def approx_scores(q, L, sketch):
    """``s_hat_j = (L^T q)^T c_j`` for every code row of ``sketch`` (Sec. 6)."""
    u = np.asarray(L, F64).T @ np.asarray(q, F64)
    return np.asarray(sketch, F64) @ u


def exact_scores(q, A, K):
    """``s_j = q^T A k_j`` for every key row of ``K`` (Sec. 3)."""
    return np.asarray(K, F64) @ (np.asarray(A, F64).T @ np.asarray(q, F64))


def topk(scores, k: int):
    """Indices of the k largest scores, descending, equal scores by lower index.

    Returns (idx [k] int64 padded with -1, values [k] padded with -inf)."""
    s = np.asarray(scores, F64)
    n = s.shape[0]
    order = np.lexsort((np.arange(n), -s))[:k]
    idx = np.full(k, -1, np.int64)
    val = np.full(k, -np.inf)
    idx[:len(order)] = order
    val[:len(order)] = s[order]
    return idx, val


def score_topk(Q, L, sketch, seq_offsets, q_seq, q_visible, k: int, nu=None,
               heads=None, rows=None):
    """Per (head, query): top-k of ``u . c_j`` over the query's visible prefix of
    its own sequence.  Q [Hq][T][d]; L [Hq][d][r]; sketch [Hq][Ntot][r].

    ``heads``/``rows`` restrict the work to a sample.  Returns (idx, scores)
    with idx seq-local int64 [len(heads)][len(rows)][k] (-1 pad) and scores
    including the ``q^T nu`` term when ``nu`` is given."""
    Hq, T = Q.shape[0], Q.shape[1]
    heads = range(Hq) if heads is None else heads
    rows = range(T) if rows is None else rows
    I = np.full((len(heads), len(rows), k), -1, np.int64)
    S = np.full((len(heads), len(rows), k), -np.inf)
    for a, h in enumerate(heads):
        for b, t in enumerate(rows):
            base = int(seq_offsets[q_seq[t]])
            vis = int(q_visible[t])
            s = approx_scores(Q[h, t], L[h], sketch[h, base:base + vis])
            idx, val = topk(s, k)
            I[a, b] = idx
            if nu is not None:
                val = val + float(np.asarray(Q[h, t], F64) @ np.asarray(nu[h], F64))
            S[a, b] = val
    return I, S


def exact_topk(Q, A, K, seq_offsets, q_seq, q_visible, k: int, group: int,
               heads=None, rows=None):
    """Exact top-k by ``q^T A k`` (the recall reference of Sec. 3)."""
    Hq, T = Q.shape[0], Q.shape[1]
    heads = range(Hq) if heads is None else heads
    rows = range(T) if rows is None else rows
    I = np.full((len(heads), len(rows), k), -1, np.int64)
    S = np.full((len(heads), len(rows), k), -np.inf)
    for a, h in enumerate(heads):
        g = h // group
        for b, t in enumerate(rows):
            base = int(seq_offsets[q_seq[t]])
            vis = int(q_visible[t])
            s = exact_scores(Q[h, t], A[h], K[g, base:base + vis])
            I[a, b], S[a, b] = topk(s, k)
    return I, S


def recall_rows(idx_approx, idx_exact, q_visible, min_visible: int, k: int):
    """Per-row recall ``|S_hat & S| / k`` (Sec. 3 protocol); NaN for rows with
    fewer than ``min_visible`` visible keys.  Inputs [rows][k]."""
    out = np.full(len(idx_approx), np.nan)
    for t in range(len(idx_approx)):
        if q_visible[t] < min_visible:
            continue
        a = set(int(i) for i in idx_approx[t] if i >= 0)
        e = set(int(i) for i in idx_exact[t] if i >= 0)
        out[t] = len(a & e) / k
    return out


def head_recall(idx_approx, idx_exact, q_visible, min_visible: int, k: int):
    """Mean recall per head over qualifying rows; inputs [H][rows][k]."""
    res = []
    for h in range(len(idx_approx)):
        r = recall_rows(idx_approx[h], idx_exact[h], q_visible, min_visible, k)
        res.append(np.nanmean(r) if np.any(~np.isnan(r)) else np.nan)
    return np.array(res)


def median_over_heads(recall):
    """Median across heads (Tab. 1 reports medians over all heads)."""
    return float(np.median(np.asarray(recall, F64)))


# --------------------------------------------------------------------------
# Sec. 7: a random-matrix view of the key moments, and App. C's measured
# score-MSE reduction
# --------------------------------------------------------------------------
def correlation_spectrum(S):
    """Eigenvalues (descending) of the correlation matrix D^{-1/2} S D^{-1/2},
    D = diag(S) (a zero diagonal entry leaves its row and column zero)."""
    S = np.asarray(S, F64)
    dg = np.diag(S)
    inv = np.where(dg > 0, 1.0 / np.sqrt(np.where(dg > 0, dg, 1.0)), 0.0)
    Rm = S * inv[:, None] * inv[None, :]
    return np.sort(np.linalg.eigvalsh(0.5 * (Rm + Rm.T)))[::-1]


def mp_upper_edge(d: int, n: int, tau_int: float = 1.0) -> float:
    """Marchenko-Pastur upper edge (1 + sqrt(q_eff))^2 with q_eff = d / T_eff and
    T_eff = n / tau_int (Sec. 7)."""
    return (1.0 + np.sqrt(d * tau_int / n)) ** 2


def mp_spike_count(S, n: int, tau_int: float = 1.0) -> int:
    """Eigenvalues of the correlation matrix of S above the MP upper edge."""
    lam = correlation_spectrum(S)
    return int(np.sum(lam > mp_upper_edge(len(lam), n, tau_int)))


def score_mse(Q, A, K, L, codes, nu, seq_offsets, q_seq, q_visible, group: int, key_stride: int = 1):
    """App. C measurement: per query head, over the causal (query, key) pairs
    (every key_stride-th visible key of each query), the sums of s^2 and
    (s - s_hat)^2 with s = q^T A k and s_hat = (L^T q)^T c + q^T nu.
    Returns [Hq][3]: sum s^2, sum (s - s_hat)^2, pairs.  The measured
    reduction is 1 - column 1 / column 0."""
    Hq, T = Q.shape[0], Q.shape[1]
    out = np.zeros((Hq, 3))
    for h in range(Hq):
        g = h // group
        for t in range(T):
            base, vis = int(seq_offsets[q_seq[t]]), int(q_visible[t])
            keys = np.arange(0, vis, key_stride)
            if len(keys) == 0:
                continue
            q = np.asarray(Q[h, t], F64)
            s = exact_scores(q, A[h], K[g, base + keys])
            sh = approx_scores(q, L[h], codes[h, base + keys]) + (0.0 if nu is None else q @ np.asarray(nu[h], F64))
            out[h] += (np.sum(s ** 2), np.sum((s - sh) ** 2), len(keys))
    return out


# --------------------------------------------------------------------------
# Online moment tracking (Sec. 2: online updates of Sq, Sk) and composition with
# RoPE (Sec. 6: reconstruct k_hat = mu + M_r (k - mu) and rotate)
# --------------------------------------------------------------------------
def merge_moments(S1, mu1, n1: int, S2, mu2, n2: int, center: bool):
    """Moments (1/n normalisation) of the union of two batches from each batch's
    moments: S = (n1 S1 + n2 S2) / n, plus (n1 n2 / n^2) (mu1 - mu2)(mu1 - mu2)^T
    for centered moments (the pooled-variance identity); mu = (n1 mu1 + n2 mu2) / n."""
    n = n1 + n2
    S1, S2 = np.asarray(S1, F64), np.asarray(S2, F64)
    if n1 == 0:
        return S2.copy(), np.asarray(mu2, F64).copy()
    S = (n1 * S1 + n2 * S2) / n
    if not center:
        return S, np.zeros(S.shape[0])
    m1, m2 = np.asarray(mu1, F64), np.asarray(mu2, F64)
    dm = m1 - m2
    return S + (n1 * n2 / n ** 2) * np.outer(dm, dm), (n1 * m1 + n2 * m2) / n


def rope(x, pos, theta: float):
    """Rotary position embedding, rotate-half convention: dimension i < d/2 pairs
    with i + d/2 and turns by pos * theta^(-2i/d)."""
    x = np.asarray(x, F64)
    d = x.shape[-1]
    half = d // 2
    ang = np.asarray(pos, F64)[..., None] * theta ** (-2.0 * np.arange(half) / d)
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def reconstruct_keys(codes, L, nu, rows, positions=None, theta: float = 10000.0):
    """k_hat_j = nu_h + L_h c_j for the given code rows of every query head (in the
    head coordinates of the paper, where A is absorbed, this is
    mu + M_r (k - mu)); q^T k_hat_j is the index's score with the mean term.
    With positions, each k_hat_j is then rotated by RoPE at positions[j].
    codes [Hq][N][r], L [Hq][d][r], nu [Hq][d] or None; returns [Hq][len(rows)][d]."""
    codes = np.asarray(codes, F64)
    rows = np.asarray(rows)
    out = np.einsum("hdr,hnr->hnd", np.asarray(L, F64), codes[:, rows])
    if nu is not None:
        out = out + np.asarray(nu, F64)[:, None, :]
    if positions is not None:
        out = rope(out, np.asarray(positions)[None, :], theta)
    return out
