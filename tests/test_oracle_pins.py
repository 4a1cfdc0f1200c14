"""Pins for the CPU oracle: each test checks it against something other than
itself -- a hand-derived closed form, a textbook special case, an inequality
the paper proves, an independent construction, or brute force."""
import json
import math
import os

import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _case(d=16, s=3, seed=0, n=None):
    """Small seeded (Sq, Sk, A) from the generator recipe (population moments
    when n is None, sample moments of n draws otherwise)."""
    w = synth.Workload("pin", 1, 1, head_dim=d, spikes=(s, s), seed=seed)
    f = synth.head_factors(w)
    if n is None:
        Sq = f.Fq[0] @ f.Fq[0].T
        Sk = f.Fk[0] @ f.Fk[0].T
    else:
        rng = np.random.default_rng(seed + 100)
        Xq = rng.standard_normal((n, d)) @ f.Fq[0].T
        Xk = rng.standard_normal((n, d)) @ f.Fk[0].T
        Sq, Sk = Xq.T @ Xq / n, Xk.T @ Xk / n
    return Sq, Sk, f.A[0].astype(np.float64)


# ---------------------------------------------------------------- closed forms
@pytest.mark.parametrize("name", ["eckart_young_golden_ratio", "query_weighting_beats_key_pca",
                                  "weight_svd_is_blind_to_data"])
def test_hand_examples(name):
    g = _gold("hand_examples.json")[name]
    res = O.fit_head(np.array(g["Sq"]), np.array(g["Sk"]), np.array(g["A"]), g["r"])
    np.testing.assert_allclose(res["sigma"], g["sigma"], rtol=1e-12, atol=1e-12)
    assert abs(res["loss"] - g["loss"]) < 1e-12
    np.testing.assert_allclose(res["M"], g["M"], rtol=1e-12, atol=1e-12)
    if "L" in g:
        np.testing.assert_allclose(res["L"], g["L"], atol=1e-12)
        np.testing.assert_allclose(res["R"], g["R"], atol=1e-12)
    if "M_squared_over_M" in g:
        M = res["M"]
        np.testing.assert_allclose(M @ M, g["M_squared_over_M"] * M, atol=1e-12)
    if "pca_loss" in g:
        pca = O.key_pca_head(np.array(g["Sk"]), np.array(g["A"]), g["r"])
        assert abs(O.score_loss(pca["M"], g["A"], g["Sq"], g["Sk"]) - g["pca_loss"]) < 1e-12
    if "weight_svd_loss" in g:
        wsvd = O.weight_svd_head(np.array(g["A"]), g["r"])
        assert abs(O.score_loss(wsvd["M"], g["A"], g["Sq"], g["Sk"]) - g["weight_svd_loss"]) < 1e-12
    if np.allclose(g["Sq"], np.eye(len(g["A"]))) and np.allclose(g["Sk"], np.eye(len(g["A"]))):
        # identity moments: the weight SVD is the optimum itself (Eckart-Young)
        np.testing.assert_allclose(O.weight_svd_head(np.array(g["A"]), g["r"])["M"], g["M"], atol=1e-12)


# ------------------------------------------------------- Prop. 1 identities
@pytest.mark.parametrize("r", [1, 4, 8, 15])
@pytest.mark.parametrize("seed", [0, 1])
def test_optimum_equals_discarded_singular_energy(r, seed):
    """Prop. 1: L(M_r) computed from Eq. (1) directly = sum_{i>r} sigma_i^2."""
    Sq, Sk, A = _case(seed=seed)
    res = O.fit_head(Sq, Sk, A, r)
    direct = O.score_loss(res["M"], A, Sq, Sk)
    assert abs(direct - res["loss"]) <= 1e-10 * max(1.0, res["loss"])
    # the total energy is ||C||_F^2 = L(0)
    assert abs(O.score_loss(0 * A, A, Sq, Sk) - np.sum(res["sigma"] ** 2)) <= 1e-9 * np.sum(res["sigma"] ** 2)


def test_full_rank_reproduces_A():
    Sq, Sk, A = _case(d=24, seed=3)
    res = O.fit_head(Sq, Sk, A, 24)
    np.testing.assert_allclose(res["M"], A, atol=1e-10 * np.abs(A).max())
    assert res["loss"] < 1e-20


@pytest.mark.parametrize("r", [1, 5, 11])
def test_map_has_rank_r(r):
    Sq, Sk, A = _case(seed=4)
    s = np.linalg.svd(O.fit_head(Sq, Sk, A, r)["M"], compute_uv=False)
    assert s[r - 1] / s[0] > 1e-8
    assert s[r] / s[0] < 1e-12


@pytest.mark.parametrize("r", [1, 2, 4, 8, 12])
def test_saki_never_loses_to_key_pca_or_weight_svd(r):
    """Remark 1: projector-based maps (key PCA) and operator-only truncation
    are rank-r maps too, so the exact optimum can only be better."""
    for seed in range(3):
        Sq, Sk, A = _case(seed=seed)
        res = O.fit_head(Sq, Sk, A, r)
        pca = O.score_loss(O.key_pca_head(Sk, A, r)["M"], A, Sq, Sk)
        wsvd = O.score_loss(O.weight_svd_head(A, r)["M"], A, Sq, Sk)
        assert res["loss"] <= pca * (1 + 1e-12)
        assert res["loss"] <= wsvd * (1 + 1e-12)


def test_identity_covariances_reduce_to_eckart_young():
    _, _, A = _case(seed=5)
    I = np.eye(A.shape[0])
    res = O.fit_head(I, I, A, 6)
    U, s, Vt = np.linalg.svd(A)
    np.testing.assert_allclose(res["M"], (U[:, :6] * s[:6]) @ Vt[:6], atol=1e-12)


def test_identity_operator_with_equal_moments_is_pca_projector():
    Sq, _, _ = _case(seed=6)
    d = Sq.shape[0]
    res = O.fit_head(Sq, Sq, np.eye(d), 5)
    lam, V = np.linalg.eigh(Sq)
    Vr = V[:, ::-1][:, :5]
    np.testing.assert_allclose(res["M"], Vr @ Vr.T, atol=1e-10)


def test_cholesky_roots_give_the_same_map():
    """Any F with F F^T = S gives ||F_q^T X F_k||_F^2 = tr(X^T Sq X Sk), so the
    optimum built from Cholesky factors must equal the symmetric-root one."""
    Sq, Sk, A = _case(seed=7, n=400)
    r = 6
    Lq, Lk = np.linalg.cholesky(Sq), np.linalg.cholesky(Sk)
    U, s, Vt = np.linalg.svd(Lq.T @ A @ Lk)
    Mc = np.linalg.solve(Lq.T, (U[:, :r] * s[:r]) @ Vt[:r]) @ np.linalg.inv(Lk)
    res = O.fit_head(Sq, Sk, A, r)
    np.testing.assert_allclose(res["M"], Mc, atol=1e-9 * np.abs(Mc).max())
    np.testing.assert_allclose(res["sigma"], s, rtol=1e-10)


def test_scaling_moments_leaves_the_map_unchanged():
    Sq, Sk, A = _case(seed=8)
    a = O.fit_head(Sq, Sk, A, 4)["M"]
    b = O.fit_head(3.7 * Sq, 0.21 * Sk, A, 4)["M"]
    np.testing.assert_allclose(a, b, atol=1e-10 * np.abs(a).max())


def test_local_optimality_under_rank_r_perturbations():
    Sq, Sk, A = _case(seed=9)
    r = 5
    res = O.fit_head(Sq, Sk, A, r)
    rng = np.random.default_rng(0)
    for _ in range(40):
        X = rng.standard_normal(res["L"].shape)
        Y = rng.standard_normal(res["R"].shape)
        for eps in (1e-3, 1e-1):
            M = (res["L"] + eps * X) @ (res["R"] + eps * Y).T
            assert O.score_loss(M, A, Sq, Sk) >= res["loss"] * (1 - 1e-12)
    # random rank-r maps are much worse
    for _ in range(10):
        M = rng.standard_normal((16, r)) @ rng.standard_normal((r, 16))
        assert O.score_loss(M, A, Sq, Sk) > res["loss"]


def test_factorisation_identity_and_non_idempotence():
    """App. A: (L^T q).(R^T k) = q^T M_r k with M_r = Sq^-1/2 C_r Sk^-1/2; Remark 1."""
    Sq, Sk, A = _case(seed=10)
    r = 4
    res = O.fit_head(Sq, Sk, A, r)
    rng = np.random.default_rng(1)
    for _ in range(5):
        q, k = rng.standard_normal(16), rng.standard_normal(16)
        assert abs((res["L"].T @ q) @ (res["R"].T @ k) - q @ res["M"] @ k) < 1e-10
    M = res["M"]
    assert np.linalg.norm(M @ M - M) > 0.1 * np.linalg.norm(M)


def test_singular_covariances_match_the_restricted_problem():
    """App. A 'Singular covariances': with n < d the covariances are rank n; the
    optimum is the full-rank solution on range(Sq) x range(Sk), zero outside."""
    d, n, r = 16, 9, 4
    rng = np.random.default_rng(2)
    Xq = rng.standard_normal((n, d))
    Xk = rng.standard_normal((n, d)) * np.linspace(3, 0.5, d)
    _, _, A = _case(seed=11)
    Sq, Sk = Xq.T @ Xq / n, Xk.T @ Xk / n
    res = O.fit_head(Sq, Sk, A, r)
    Bq, _ = np.linalg.qr(Xq.T)          # orthonormal bases of the ranges
    Bk, _ = np.linalg.qr(Xk.T)
    Sqr, Skr = Bq.T @ Sq @ Bq, Bk.T @ Sk @ Bk
    Lq, Lk = np.linalg.cholesky(Sqr), np.linalg.cholesky(Skr)
    U, s, Vt = np.linalg.svd(Lq.T @ (Bq.T @ A @ Bk) @ Lk)
    X = np.linalg.solve(Lq.T, (U[:, :r] * s[:r]) @ Vt[:r]) @ np.linalg.inv(Lk)
    M_ref = Bq @ X @ Bk.T
    np.testing.assert_allclose(res["M"], M_ref, atol=1e-8 * np.abs(M_ref).max())
    assert abs(O.score_loss(res["M"], A, Sq, Sk) - res["loss"]) < 1e-9 * max(res["loss"], 1)


# ------------------------------------------------------------ moments, rounding
def test_moments_match_numpy_cov():
    rng = np.random.default_rng(3)
    X = rng.standard_normal((300, 7)) + np.arange(7)
    S, mu = O.moments(X, center=True)
    np.testing.assert_allclose(S, np.cov(X.T, bias=True), atol=1e-12)
    np.testing.assert_allclose(mu, np.average(X, axis=0), atol=1e-12)
    S0, mu0 = O.moments(X, center=False)
    ref = sum(np.outer(x, x) for x in X) / len(X)
    np.testing.assert_allclose(S0, ref, atol=1e-12)
    assert not np.any(mu0)


def test_bf16_rounding_golden_cases():
    for c in _gold("bf16_rounding.json")["cases"]:
        got = float(O.round_bf16(np.array([c["x"]]))[0])
        assert got == c["bf16"], c


def test_bf16_rounding_matches_torch_on_fp32_values():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(4)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                        (1 + (2 * rng.integers(0, 128, 2000) + 1) * 2.0 ** -8)]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.round_bf16(x.astype(np.float64)), ref)


def test_round_to_float32_is_round_to_nearest_even():
    """Hand cases of IEEE binary32 rounding (24-bit significand): halfway
    values go to the even neighbour, anything above halfway rounds up."""
    u = 2.0 ** -23   # float32 spacing at 1
    cases = [(1 + u / 2, 1.0),                    # halfway, 1 is even
             (1 + 3 * u / 2, 1 + 2 * u),          # halfway, 1 + 2u is even
             (1 + u / 2 + 2.0 ** -40, 1 + u),     # just above halfway
             (-(1 + u / 2), -1.0),
             (3.0, 3.0)]
    for x, want in cases:
        assert float(O.round_to("f32", np.array([x]))[0]) == want, x
    x = np.random.default_rng(9).standard_normal(64)
    np.testing.assert_array_equal(O.round_to("bf16", x), O.round_bf16(x))
    with pytest.raises(ValueError):
        O.round_to("f16", x)


# ------------------------------------------------------------ oracle helpers
def test_psd_roots_match_scipy_sqrtm_on_a_definite_matrix():
    scipy_linalg = pytest.importorskip("scipy.linalg")
    rng = np.random.default_rng(10)
    B = rng.standard_normal((12, 12))
    S = B @ B.T + 0.5 * np.eye(12)
    root, iroot = O.psd_roots(S)
    ref = np.real(scipy_linalg.sqrtm(S))
    np.testing.assert_allclose(root, ref, atol=1e-10)
    np.testing.assert_allclose(iroot, np.linalg.inv(ref), atol=1e-10)


def test_psd_roots_drop_eigenvalues_below_the_floor():
    """App. A: eigenvalues below floor * lambda_max count as zero in both roots.
    Built from a seeded orthogonal basis with eigenvalues 40 x (1, 0.5, 2e-6,
    5e-7, 0): at the 1e-6 relative floor the third is kept and the last two are
    dropped (an absolute floor of 1e-6 would keep the fourth, 2e-5)."""
    U, _ = np.linalg.qr(np.random.default_rng(11).standard_normal((5, 5)))
    lam = 40.0 * np.array([1.0, 0.5, 2e-6, 5e-7, 0.0])
    S = (U * lam) @ U.T
    root, iroot = O.psd_roots(S, floor_rel=1e-6)
    kept = U[:, :3]
    P = kept @ kept.T
    np.testing.assert_allclose(root @ root, S - lam[3] * np.outer(U[:, 3], U[:, 3]), atol=1e-11)
    np.testing.assert_allclose(iroot @ root, P, atol=1e-8)
    np.testing.assert_allclose(root @ iroot, P, atol=1e-8)
    np.testing.assert_allclose(iroot @ S @ iroot, P, atol=1e-8)
    np.testing.assert_allclose(iroot @ U[:, 3], 0.0, atol=1e-8)   # dropped directions vanish
    np.testing.assert_allclose(root, root.T, atol=1e-14)
    np.testing.assert_allclose(iroot, iroot.T, atol=1e-8)


def test_canonical_signs_hand_example_and_ties():
    """Each column pair is flipped so that R's largest-magnitude entry is
    positive (ties: the first such row); L R^T is unchanged."""
    L = np.array([[1.0, 2.0, 5.0], [3.0, 4.0, 6.0]])
    R = np.array([[1.0, -3.0, -2.0], [2.0, 1.0, 2.0]])
    L2, R2 = O.canonical_signs(L, R)
    np.testing.assert_array_equal(R2, [[1.0, 3.0, 2.0], [2.0, -1.0, -2.0]])
    np.testing.assert_array_equal(L2, [[1.0, -2.0, -5.0], [3.0, -4.0, -6.0]])
    np.testing.assert_array_equal(L2 @ R2.T, L @ R.T)
    np.testing.assert_array_equal(R, [[1.0, -3.0, -2.0], [2.0, 1.0, 2.0]])   # inputs untouched


def test_orthonormal_basis_spans_the_columns_and_matches_householder_qr():
    X = np.random.default_rng(12).standard_normal((16, 5))
    Q = O._orth(X)
    np.testing.assert_allclose(Q.T @ Q, np.eye(5), atol=1e-12)
    np.testing.assert_allclose(Q @ Q.T, X @ np.linalg.solve(X.T @ X, X.T), atol=1e-12)
    Qh, Rh = np.linalg.qr(X)   # Householder; Gram-Schmidt gives R a positive diagonal
    np.testing.assert_allclose(Q, Qh * np.sign(np.diag(Rh)), atol=1e-12)


def test_projector_map_factors():
    rng = np.random.default_rng(13)
    Q = O._orth(rng.standard_normal((8, 3)))
    A = rng.standard_normal((8, 8))
    out = O._projector_head(Q, A)
    np.testing.assert_allclose(out["M"], A @ Q @ Q.T, atol=1e-12)
    np.testing.assert_allclose(out["R"].T @ out["R"], np.eye(3), atol=1e-12)
    np.testing.assert_allclose(np.abs(out["R"]), np.abs(Q), atol=0)
    np.testing.assert_allclose(out["L"], A @ out["R"], atol=1e-12)


# ------------------------------------------------------------ selection, recall
def test_topk_against_brute_force_with_ties():
    rng = np.random.default_rng(5)
    for n in (1, 5, 63, 64, 65, 200):
        s = rng.integers(-5, 5, n).astype(float)     # many exact ties
        for k in (1, 8, 64):
            idx, val = O.topk(s, k)
            ref = sorted(range(n), key=lambda j: (-s[j], j))[:k]
            assert list(idx[:len(ref)]) == ref
            assert np.all(idx[len(ref):] == -1) and np.all(np.isneginf(val[len(ref):]))
            np.testing.assert_array_equal(val[:len(ref)], s[ref])


def test_recall_golden_example():
    g = _gold("hand_examples.json")["recall_example"]
    rows = O.recall_rows(np.array(g["idx_approx"]), np.array(g["idx_exact"]),
                         np.array(g["q_visible"]), g["min_visible"], g["k"])
    for got, want in zip(rows, g["row_recall"]):
        assert (np.isnan(got) and want is None) or got == want
    h = O.head_recall(np.array([g["idx_approx"]]), np.array([g["idx_exact"]]),
                      np.array(g["q_visible"]), g["min_visible"], g["k"])
    assert h[0] == g["head_recall"]
    assert O.median_over_heads([0.2, 0.9, 0.5, 0.7]) == 0.6


def test_recall_boundary_divisor_and_head_mean():
    """Sec. 3 protocol: a row with exactly min_visible visible keys counts; the
    divisor is k even when fewer than k keys are visible (a row of 3 visible
    keys with min_visible 3 and k 4 scores 3/4 with every key found); a head's
    recall is the mean of its rows (1, 1 and 1/4: 0.75, where the median is 1)."""
    k = 4
    ia = np.array([[0, 1, 2, 3], [0, 1, 2, -1], [9, 8, 7, 3]])
    ie = np.array([[3, 2, 1, 0], [2, 1, 0, -1], [0, 1, 2, 3]])
    rows = O.recall_rows(ia, ie, np.array([10, 3, 10]), 3, k)
    np.testing.assert_array_equal(rows, [1.0, 0.75, 0.25])
    rows = O.recall_rows(ia, ie, np.array([10, 3, 10]), 4, k)
    assert np.isnan(rows[1]) and rows[0] == 1.0
    ia2 = np.array([[[0, 1, 2, 3], [4, 5, 6, 7], [9, 8, 7, 3]]])
    ie2 = np.array([[[0, 1, 2, 3], [7, 6, 5, 4], [0, 1, 2, 3]]])
    assert O.head_recall(ia2, ie2, np.array([10, 10, 10]), 5, k)[0] == 0.75


def test_bf16_rounding_matches_torch_in_the_subnormal_range():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(14)
    x = (rng.uniform(-1, 1, 20000) * 2.0 ** rng.integers(-149, -120, 20000)).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.round_bf16(x.astype(np.float64)), ref)


def test_margin_condition_guarantees_exact_top_k():
    """Prop. 2: |s - s_hat| <= eps for all j and 2 eps < gamma_k => same top-k set;
    at 2 eps > gamma_k a perturbation exists that swaps the boundary pair."""
    rng = np.random.default_rng(6)
    k = 8
    for _ in range(200):
        s = rng.standard_normal(60)
        srt = np.sort(s)[::-1]
        gamma = srt[k - 1] - srt[k]
        eps = 0.49 * gamma
        s_hat = s + rng.uniform(-eps, eps, s.shape)
        assert set(O.topk(s, k)[0]) == set(O.topk(s_hat, k)[0])
    s = np.array([5.0, 4.0, 3.0, 2.9, 1.0])
    gamma, eps = 0.1, 0.06
    s_hat = s.copy()
    s_hat[2] -= eps
    s_hat[3] += eps
    assert set(O.topk(s, 3)[0]) != set(O.topk(s_hat, 3)[0])


# ------------------------------------------------------- index and scores
def test_full_rank_index_reproduces_exact_scores_with_centering():
    """r = d: codes c_j = R^T (k_j - mu) and s_hat = u.c + q^T A mu equal q^T A k."""
    d = 16
    Sq, Sk, A = _case(d=d, seed=12)
    rng = np.random.default_rng(7)
    kc = rng.standard_normal((300, d)) + 2.0
    qc = rng.standard_normal((300, d))
    res = O.fit(qc[None], kc[None], A[None], d, center=True)
    K = rng.standard_normal((1, 40, d)) + 2.0
    q = rng.standard_normal(d)
    codes = O.build_index(K, res["R"], res["mu"], "f32", 1)
    s_hat = O.approx_scores(q, res["L"][0], codes[0]) + q @ res["nu"][0]
    np.testing.assert_allclose(s_hat, O.exact_scores(q, A, K[0]), rtol=2e-5, atol=2e-5)
    # the selection's returned scores carry the same q^T nu term
    Q = q[None, None, :]
    off, seq, vis = np.array([0]), np.array([0]), np.array([40])
    _, S_hat = O.score_topk(Q, res["L"], codes, off, seq, vis, 8, nu=res["nu"])
    _, S = O.exact_topk(Q, A[None], K, off, seq, vis, 8, 1)
    np.testing.assert_allclose(S_hat[0, 0], S[0, 0], rtol=2e-5, atol=2e-5)


def test_build_index_maps_query_heads_to_their_kv_head():
    """GQA (Sec. 6): with 2 KV heads and groups of 2, query head h codes the
    keys of KV head h // 2.  KV head g holds keys (g + 1) e_0 with mean
    (g + 1) / 2 e_0 (head 0) or e_0 (head 1); R_h has (h + 1) at (0, 0), so code
    entry 0 is (g + 1 - mu_g) (h + 1): 0.5, 1, 3, 4 for h = 0..3."""
    d, N, r = 4, 3, 2
    K = np.zeros((2, N, d))
    K[0, :, 0], K[1, :, 0] = 1.0, 2.0
    R = np.zeros((4, d, r))
    for h in range(4):
        R[h, 0, 0] = h + 1
    mu = np.array([[0.5, 0, 0, 0], [1.0, 0, 0, 0]])
    codes = O.build_index(K, R, mu, "f32", group=2)
    np.testing.assert_array_equal(codes[:, :, 0], np.array([[0.5] * N, [1.0] * N, [3.0] * N, [4.0] * N]))
    np.testing.assert_array_equal(codes[:, :, 1], 0.0)


def test_exact_scores_by_double_loop():
    rng = np.random.default_rng(8)
    d = 5
    A = rng.standard_normal((d, d))
    K = rng.standard_normal((7, d))
    q = rng.standard_normal(d)
    ref = [sum(q[a] * A[a, b] * K[j, b] for a in range(d) for b in range(d)) for j in range(7)]
    np.testing.assert_allclose(O.exact_scores(q, A, K), ref, rtol=1e-12)


def test_predicted_mse_reduction_matches_independent_draws():
    """Remark 2 / App. C: with independent q ~ N(0,Sq), k ~ N(0,Sk) the measured
    score-MSE reduction equals 1 - sum_{i>r} sigma^2 / sum sigma^2 up to
    sampling noise (E s^2 = ||C||_F^2 and E (s - s_hat)^2 = L(M_r))."""
    w = synth.Workload("pin", 1, 1, head_dim=16, spikes=(3, 3), seed=13)
    f = synth.head_factors(w)
    Sq, Sk, A = f.Fq[0] @ f.Fq[0].T, f.Fk[0] @ f.Fk[0].T, f.A[0].astype(float)
    r = 4
    res = O.fit_head(Sq, Sk, A, r)
    pred = 1 - res["loss"] / np.sum(res["sigma"] ** 2)
    rng = np.random.default_rng(9)
    n = 400000
    q = rng.standard_normal((n, 16)) @ f.Fq[0].T
    k = rng.standard_normal((n, 16)) @ f.Fk[0].T
    s = np.einsum("ni,ij,nj->n", q, A, k)
    e = s - np.einsum("ni,ij,nj->n", q, res["M"], k)
    meas = 1 - np.mean(e ** 2) / np.mean(s ** 2)
    # relative std of a mean of squared Gaussian bilinear forms is ~3/sqrt(n)
    tol = 5 * 3 / math.sqrt(n) * (1 - pred + 0.05)
    assert abs(meas - pred) < tol, (meas, pred, tol)


# ------------------------------------------------- comparison indexes (Tab. 1)
def _rotation(d, seed):
    """An orthogonal matrix built from Givens rotations by fixed angles (no
    factorisation routine involved)."""
    Q = np.eye(d)
    rng = np.random.default_rng(seed)
    for i in range(d - 1):
        for j in range(i + 1, d):
            t = rng.uniform(0, 2 * np.pi)
            G = np.eye(d)
            G[i, i] = G[j, j] = np.cos(t)
            G[i, j], G[j, i] = -np.sin(t), np.sin(t)
            Q = Q @ G
    return Q


def test_weight_svd_closed_form():
    """A = Q1 diag(4, 3, 2, 1) Q2^T: the rank-2 weight SVD keeps Q1 diag(4, 3, 0, 0)
    Q2^T, sigma = (4, 3, 2, 1), loss = 2^2 + 1^2 = 5, and L R^T = M."""
    Q1, Q2 = _rotation(4, 1), _rotation(4, 2)
    A = Q1 @ np.diag([4.0, 3.0, 2.0, 1.0]) @ Q2.T
    res = O.weight_svd_head(A, 2)
    np.testing.assert_allclose(res["M"], Q1 @ np.diag([4.0, 3.0, 0.0, 0.0]) @ Q2.T, atol=1e-12)
    np.testing.assert_allclose(res["sigma"], [4.0, 3.0, 2.0, 1.0], atol=1e-12)
    assert abs(res["loss"] - 5.0) < 1e-12
    np.testing.assert_allclose(res["L"] @ res["R"].T, res["M"], atol=1e-12)
    # each R column is sqrt(sigma) times a unit right singular vector
    np.testing.assert_allclose(np.sum(res["R"] ** 2, axis=0), [4.0, 3.0], atol=1e-12)


def test_key_pca_closed_form():
    """Sk = Q diag(9, 4, 1, 1/4) Q^T: rank-2 key PCA keeps the first two columns
    of Q (R R^T = Q_2 Q_2^T, R orthonormal), L = A R, sigma = (3, 2, 1, 1/2),
    loss = 1 + 1/4."""
    Q = _rotation(4, 3)
    Sk = Q @ np.diag([9.0, 4.0, 1.0, 0.25]) @ Q.T
    A = _rotation(4, 4) @ np.diag([2.0, 1.0, 0.5, 0.1])
    res = O.key_pca_head(Sk, A, 2)
    np.testing.assert_allclose(res["R"] @ res["R"].T, Q[:, :2] @ Q[:, :2].T, atol=1e-12)
    np.testing.assert_allclose(res["R"].T @ res["R"], np.eye(2), atol=1e-12)
    np.testing.assert_allclose(res["L"], A @ res["R"], atol=1e-12)
    np.testing.assert_allclose(res["M"], A @ Q[:, :2] @ Q[:, :2].T, atol=1e-12)
    np.testing.assert_allclose(res["sigma"], [3.0, 2.0, 1.0, 0.5], atol=1e-12)
    assert abs(res["loss"] - 1.25) < 1e-12


def test_key_pca_drops_floored_directions():
    """App. A floor: an eigenvalue below 1e-6 lambda_max counts as zero, so a
    rank-3 key PCA of a rank-2 moment keeps two directions."""
    Sk = np.diag([1.0, 0.5, 1e-9, 0.0])
    res = O.key_pca_head(Sk, np.eye(4), 3)
    np.testing.assert_allclose(res["M"], np.diag([1.0, 1.0, 0.0, 0.0]), atol=1e-15)
    np.testing.assert_allclose(res["sigma"], [1.0, np.sqrt(0.5), 0.0, 0.0], atol=1e-15)


def test_baselines_from_calibration_keys():
    """fit_baseline on keys whose centered moment is diagonal by construction
    (rows mu +- sqrt(n lambda_i / 2) e_i): key PCA picks the largest-variance
    axes, nu = A mu; weight SVD ignores the data entirely."""
    d, n = 6, 12
    lam = np.array([0.5, 3.0, 0.25, 2.0, 1.0, 0.1])
    mu = np.arange(1.0, d + 1.0)
    K = np.tile(mu, (n, 1))
    for i in range(d):
        K[2 * i] += np.sqrt(n * lam[i] / 2) * np.eye(d)[i]
        K[2 * i + 1] -= np.sqrt(n * lam[i] / 2) * np.eye(d)[i]
    A = np.stack([_rotation(d, 5), _rotation(d, 6)])
    res = O.fit_baseline("key_pca", K[None], A, 2, True, 2)
    P = np.zeros((d, d))
    P[1, 1] = P[3, 3] = 1.0
    for h in range(2):
        np.testing.assert_allclose(res["M"][h], A[h] @ P, atol=1e-12)
        np.testing.assert_allclose(res["nu"][h], A[h] @ mu, atol=1e-12)
    np.testing.assert_allclose(res["mu"][0], mu, atol=1e-12)
    a = O.fit_baseline("weight_svd", K[None], A, 2, True, 2)
    b = O.fit_baseline("weight_svd", 2.0 * K[None] + 1.0, A, 2, True, 2)
    np.testing.assert_allclose(a["M"], b["M"], atol=1e-15)


# --------------------------------------------------- SAP projector variants (Sec. 6)
def test_sap_variants_hand_example():
    """A = [[1, 1], [0, 1]], Sq = I, Sk = diag(4, 1), r = 1.  C = A Sk^{1/2} =
    [[2, 1], [0, 1]]; C^T C = [[4, 2], [2, 2]] has top eigenvalue 3 + sqrt5 with
    eigenvector v = (2, sqrt5 - 1), |v|^2 = 10 - 2 sqrt5.  SAP-svd projects on v;
    SAP-map on Sk^{-1/2} v = (1, sqrt5 - 1), |.|^2 = 7 - 2 sqrt5."""
    A = np.array([[1.0, 1.0], [0.0, 1.0]])
    Sq, Sk = np.eye(2), np.diag([4.0, 1.0])
    s5 = math.sqrt(5.0)
    v = np.array([2.0, s5 - 1.0])
    w = np.array([1.0, s5 - 1.0])
    P_svd = np.outer(v, v) / (10.0 - 2.0 * s5)
    P_map = np.outer(w, w) / (7.0 - 2.0 * s5)
    np.testing.assert_allclose(O.sap_svd_head(Sq, Sk, A, 1)["M"], A @ P_svd, atol=1e-12)
    np.testing.assert_allclose(O.sap_map_head(Sq, Sk, A, 1)["M"], A @ P_map, atol=1e-12)


def test_sap_variants_reduce_to_weight_svd_with_identity_moments():
    """Sq = Sk = I: C = A, both spans are A's leading right singular vectors, and
    A V_r V_r^T = A_r (rotated diagonal spectrum, kept part diag(4, 3))."""
    Q1, Q2 = _rotation(4, 7), _rotation(4, 8)
    A = Q1 @ np.diag([4.0, 3.0, 2.0, 1.0]) @ Q2.T
    want = Q1 @ np.diag([4.0, 3.0, 0.0, 0.0]) @ Q2.T
    for f in (O.sap_svd_head, O.sap_map_head):
        np.testing.assert_allclose(f(np.eye(4), np.eye(4), A, 2)["M"], want, atol=1e-12)


@pytest.mark.parametrize("r", [1, 3, 6])
def test_sap_variants_are_projector_maps_that_never_beat_saki(r):
    """Remark 1: an orthogonal projector P gives the rank-r map A P, so the exact
    optimum's loss is no larger; R has orthonormal columns and P = R R^T."""
    for seed in range(3):
        Sq, Sk, A = _case(seed=seed + 20)
        best = O.fit_head(Sq, Sk, A, r)["loss"]
        for f in (O.sap_svd_head, O.sap_map_head):
            res = f(Sq, Sk, A, r)
            R = res["R"]
            np.testing.assert_allclose(R.T @ R, np.eye(r), atol=1e-10)
            np.testing.assert_allclose(res["M"], A @ R @ R.T, atol=1e-10)
            assert best <= O.score_loss(res["M"], A, Sq, Sk) * (1 + 1e-12)


# ------------------------------------------------------------ layouts and GQA
def _two_sequence_layout():
    """Two sequences in one key tensor: sequence 0 holds rows 0..4, sequence 1
    rows 5..10.  Each query names its sequence and how many of that sequence's
    keys it sees (the causal or decode prefix)."""
    seq_offsets = np.array([0, 5, 11], np.int64)
    #            t:  0  1  2  3  4  5
    q_seq = np.array([0, 1, 1, 0, 1, 0], np.int32)
    q_visible = np.array([3, 4, 6, 1, 0, 5], np.int64)
    # one-dimensional codes (r = 1) chosen so that a visible prefix one key too
    # long or too short, or a sequence read from the wrong base row, changes the
    # top two
    codes0 = [5.0, 1.0, 4.0, 9.0, 3.0]
    codes1 = [0.0, 9.0, 7.0, 8.0, 6.0, 10.0]
    u = np.array([1.0, 1.0, 1.0, 1.0, 1.0, -1.0])      # the last query ranks keys by -code
    # the expected sequence-local top-2 of every query, worked out by hand:
    #   t0: seq 0, keys 0..2, codes 5 1 4        -> 0, 2
    #   t1: seq 1, keys 0..3, codes 0 9 7 8      -> 1, 3
    #   t2: seq 1, keys 0..5, codes 0 9 7 8 6 10 -> 5, 1
    #   t3: seq 0, key 0 only                    -> 0, -1
    #   t4: seq 1, no key                        -> -1, -1
    #   t5: seq 0, keys 0..4, scores -5 -1 -4 -9 -3 -> 1, 4
    expected = np.array([[0, 2], [1, 3], [5, 1], [0, -1], [-1, -1], [1, 4]])
    return seq_offsets, q_seq, q_visible, np.array(codes0 + codes1), u, expected


def test_score_topk_slices_each_query_by_its_sequence_and_prefix():
    off, q_seq, q_vis, codes, u, expected = _two_sequence_layout()
    d = 4
    Q = np.zeros((1, len(q_seq), d))
    Q[0, :, 2] = u                                   # u = L^T q = q[2] with L = e_2
    L = np.zeros((1, d, 1))
    L[0, 2, 0] = 1.0
    sketch = codes.reshape(1, -1, 1)
    idx, val = O.score_topk(Q, L, sketch, off, q_seq, q_vis, 2)
    np.testing.assert_array_equal(idx[0], expected)
    assert list(val[0, 0]) == [5.0, 4.0] and list(val[0, 5]) == [-1.0, -3.0]
    assert np.isneginf(val[0, 3, 1]) and np.all(np.isneginf(val[0, 4]))


def test_exact_topk_slices_the_same_layout_and_maps_query_heads_to_kv_heads():
    """Four query heads over two KV heads (G = 2): heads 0 and 1 must read KV head
    0, heads 2 and 3 KV head 1.  KV head 1 holds the negated keys, so a wrong
    head mapping reverses the ranking."""
    off, q_seq, q_vis, codes, u, expected = _two_sequence_layout()
    d = 3
    K = np.zeros((2, len(codes), d))
    K[0, :, 1] = codes
    K[1, :, 1] = -codes
    A = np.zeros((4, d, d))
    A[:, 0, 1] = 1.0                                 # s = q[0] * k[1]
    Q = np.zeros((4, len(q_seq), d))
    Q[:, :, 0] = u
    idx, _ = O.exact_topk(Q, A, K, off, q_seq, q_vis, 2, group=2)
    for h in (0, 1):
        np.testing.assert_array_equal(idx[h], expected)
    # KV head 1: every query ranks by -code (the last one by +code), worked by hand
    neg = np.array([[1, 2], [0, 2], [0, 4], [0, -1], [-1, -1], [3, 0]])
    for h in (2, 3):
        np.testing.assert_array_equal(idx[h], neg)


def _diag_calibration(lams, d):
    """n = d calibration rows whose uncentered second moment is exactly
    diag(lams): row i = sqrt(d * lams[i]) e_i."""
    X = np.zeros((d, d))
    X[np.arange(d), np.arange(d)] = np.sqrt(d * np.asarray(lams, float))
    return X


def test_fit_maps_query_heads_to_their_own_kv_head():
    """Hq = 4, Hk = 2.  With A = I and Sq = I exactly, the optimum is the
    projector onto the r leading eigenvectors of the head's own Sk (Prop. 1:
    C = Sk^{1/2}, M_r = Sk^{-1/2} C_r Sk^{-1/2}).  KV head 0 has its energy on
    axes 0, 1 and KV head 1 on axes 2, 3, so heads 0, 1 must get diag(1, 1, 0,
    ...) and heads 2, 3 diag(0, 0, 1, 1, 0, ...)."""
    d, r = 8, 2
    lam0 = [9.0, 4.0, 1.0, 0.5, 0.25, 0.2, 0.1, 0.05]
    lam1 = [1.0, 0.5, 9.0, 4.0, 0.25, 0.2, 0.1, 0.05]
    k_cal = np.stack([_diag_calibration(lam0, d), _diag_calibration(lam1, d)])
    q_cal = np.stack([_diag_calibration(np.ones(d), d)] * 4)
    A = np.stack([np.eye(d)] * 4)
    res = O.fit(q_cal, k_cal, A, r, center=False)
    P0 = np.diag([1.0, 1, 0, 0, 0, 0, 0, 0])
    P1 = np.diag([0.0, 0, 1, 1, 0, 0, 0, 0])
    for h, P in zip(range(4), (P0, P0, P1, P1)):
        np.testing.assert_allclose(res["M"][h], P, atol=1e-12)
    # loss = the discarded key energy of the head's own KV head
    np.testing.assert_allclose(res["loss"], [1.0 + 0.5 + 0.25 + 0.2 + 0.1 + 0.05] * 2 +
                               [1.0 + 0.5 + 0.25 + 0.2 + 0.1 + 0.05] * 2, rtol=1e-12)
    for method in ("key_pca", "weight_svd"):
        base = O.fit_baseline(method, k_cal, A, r, False, 4)
        if method == "key_pca":      # R spans the two leading axes of the head's KV head
            for h, P in zip(range(4), (P0, P0, P1, P1)):
                np.testing.assert_allclose(base["R"][h] @ base["R"][h].T, P, atol=1e-12)
            np.testing.assert_allclose(base["loss"], [2.1] * 4, rtol=1e-12)
        else:                        # data-blind: every head keeps two unit directions of I
            np.testing.assert_allclose(base["loss"], [d - r] * 4, rtol=1e-12)


# ------------------------------------------------------- Sec. 7 diagnostics
@pytest.mark.parametrize("center", [False, True])
def test_ledoit_wolf_matches_sklearn(center):
    cov = pytest.importorskip("sklearn.covariance")
    rng = np.random.default_rng(21)
    X = rng.standard_normal((60, 12)) @ rng.standard_normal((12, 12)) + (1.5 if center else 0.0)
    S, rho, _ = O.ledoit_wolf(X, center)
    ref, ref_rho = cov.ledoit_wolf(X, assume_centered=not center)
    np.testing.assert_allclose(S, ref, rtol=1e-10, atol=1e-12)
    assert abs(rho - ref_rho) <= 1e-12


def test_ledoit_wolf_limits():
    rng = np.random.default_rng(22)
    # many samples of a strongly anisotropic distribution: almost no shrinkage
    X = rng.standard_normal((20000, 8)) * np.array([10, 5, 3, 2, 1, 1, 0.5, 0.2])
    _, rho, _ = O.ledoit_wolf(X, False)
    assert 0 <= rho < 1e-3
    # fewer samples than dimensions of an isotropic distribution: heavy shrinkage
    X = rng.standard_normal((8, 64))
    S, rho, _ = O.ledoit_wolf(X, False)
    assert rho > 0.5
    np.testing.assert_allclose(np.trace(S), np.trace(X.T @ X / 8), rtol=1e-12)   # the trace is kept


def test_ledoit_wolf_clips_the_intensity_at_one():
    """rho = min(b2, d2) / d2: four draws in six dimensions (seed 0) give an
    estimated error b2 above the dispersion d2, so S* is the scaled identity."""
    X = np.random.default_rng(0).standard_normal((4, 6))
    S, _ = O.moments(X, False)
    m = np.trace(S) / 6
    d2 = np.sum((S - m * np.eye(6)) ** 2)
    b2 = sum(np.sum((np.outer(x, x) - S) ** 2) for x in X) / 16
    assert b2 > d2
    S_star, rho, _ = O.ledoit_wolf(X, False)
    assert rho == 1.0
    np.testing.assert_allclose(S_star, m * np.eye(6), atol=1e-14)
    sk = pytest.importorskip("sklearn.covariance")
    np.testing.assert_allclose(sk.ledoit_wolf(X, assume_centered=True)[1], 1.0)


def test_correlation_spectrum_and_mp_edge():
    rng = np.random.default_rng(23)
    d, n = 64, 4096
    # white data: the largest sample eigenvalue sits at the MP edge, no spike
    X = rng.standard_normal((n, d)) * rng.uniform(0.5, 3.0, d)     # scales drop out of the correlation
    S = X.T @ X / n
    lam = O.correlation_spectrum(S)
    assert abs(lam.sum() - d) < 1e-9                                # unit diagonal
    edge = O.mp_upper_edge(d, n)
    assert edge == pytest.approx((1 + np.sqrt(d / n)) ** 2)
    assert abs(lam[0] - edge) < 0.08 and O.mp_spike_count(S, n) == 0
    # five planted spikes far above the edge are all counted
    U = np.linalg.qr(rng.standard_normal((d, 5)))[0]
    Xs = rng.standard_normal((n, d)) + (rng.standard_normal((n, 5)) * np.sqrt([40, 30, 20, 15, 10])) @ U.T
    assert O.mp_spike_count(Xs.T @ Xs / n, n) == 5
    # autocorrelation shrinks the effective sample: the edge moves out
    assert O.mp_upper_edge(d, n, tau_int=3.2) > edge


def test_score_mse_reduction_by_double_loop_and_full_rank():
    rng = np.random.default_rng(24)
    d, Hq, N = 6, 2, 9
    Q = rng.standard_normal((Hq, N, d))
    K = rng.standard_normal((1, N, d)) + 0.5
    A = rng.standard_normal((Hq, d, d))
    L = rng.standard_normal((Hq, d, 3))
    codes = rng.standard_normal((Hq, N, 3))
    nu = rng.standard_normal((Hq, d))
    off, q_seq, q_vis = np.array([0, N]), np.zeros(N, np.int32), np.arange(1, N + 1)
    out = O.score_mse(Q, A, K, L, codes, nu, off, q_seq, q_vis, group=2, key_stride=2)
    for h in range(Hq):
        ss = se = cnt = 0.0
        for t in range(N):
            for j in range(0, t + 1, 2):
                s = sum(Q[h, t, a] * A[h, a, b] * K[0, j, b] for a in range(d) for b in range(d))
                sh = sum(sum(L[h, a, c] * Q[h, t, a] for a in range(d)) * codes[h, j, c] for c in range(3))
                sh += sum(Q[h, t, a] * nu[h, a] for a in range(d))
                ss, se, cnt = ss + s * s, se + (s - sh) ** 2, cnt + 1
        np.testing.assert_allclose(out[h], [ss, se, cnt], rtol=1e-12)
    # r = d with centered codes and the mean term: the index reproduces q^T A k
    kc = rng.standard_normal((300, d)) + 1.0
    qc = rng.standard_normal((300, d))
    res = O.fit(qc[None], kc[None], A[:1], d, center=True)
    codes = O.build_index(K, res["R"], res["mu"], "f32", 1)
    out = O.score_mse(Q[:1], A[:1], K, res["L"], codes, res["nu"], off, q_seq, q_vis, group=1)
    assert out[0, 1] <= 1e-12 * out[0, 0]


# ------------------------------------------- online moments, RoPE composition
@pytest.mark.parametrize("center", [False, True])
def test_merged_moments_equal_the_moments_of_the_union(center):
    rng = np.random.default_rng(41)
    X1 = rng.standard_normal((37, 10)) + 1.0
    X2 = rng.standard_normal((91, 10)) * 2.0 - 0.5
    S1, m1 = O.moments(X1, center)
    S2, m2 = O.moments(X2, center)
    S, mu = O.merge_moments(S1, m1, 37, S2, m2, 91, center)
    Su, mu_u = O.moments(np.concatenate([X1, X2]), center)
    np.testing.assert_allclose(S, Su, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(mu, mu_u, rtol=1e-12, atol=1e-12)
    S0, mu0 = O.merge_moments(np.zeros((10, 10)), np.zeros(10), 0, S2, m2, 91, center)
    np.testing.assert_allclose(S0, S2)


def test_rope_hand_example_and_relative_positions():
    # d = 4: pairs (0, 2) and (1, 3) turn by pos and pos / 100 (theta = 10^4)
    x = np.array([1.0, 2.0, 3.0, 4.0])
    got = O.rope(x, 1.0, 10000.0)
    c0, s0, c1, s1 = np.cos(1.0), np.sin(1.0), np.cos(0.01), np.sin(0.01)
    np.testing.assert_allclose(got, [1 * c0 - 3 * s0, 2 * c1 - 4 * s1, 3 * c0 + 1 * s0, 4 * c1 + 2 * s1], rtol=1e-15)
    rng = np.random.default_rng(42)
    q, k = rng.standard_normal(16), rng.standard_normal(16)
    assert np.linalg.norm(O.rope(k, 37.0, 500.0)) == pytest.approx(np.linalg.norm(k))
    base = O.rope(q, 3.0, 500.0) @ O.rope(k, 11.0, 500.0)
    assert O.rope(q, 103.0, 500.0) @ O.rope(k, 111.0, 500.0) == pytest.approx(base, rel=1e-12)


def test_reconstructed_keys_reproduce_the_index_scores_and_the_keys_at_full_rank():
    rng = np.random.default_rng(43)
    d = 12
    A = rng.standard_normal((1, d, d))
    kc = rng.standard_normal((400, d)) + 1.0
    qc = rng.standard_normal((400, d))
    K = rng.standard_normal((1, 20, d)) + 1.0
    q = rng.standard_normal(d)
    for r in (4, d):
        res = O.fit(qc[None], kc[None], A, r, center=True)
        codes = O.build_index(K, res["R"], res["mu"], "f32", 1)
        rows = np.array([3, 0, 19, 7])
        kh = O.reconstruct_keys(codes, res["L"], res["nu"], rows)
        s_hat = O.approx_scores(q, res["L"][0], codes[0, rows]) + q @ res["nu"][0]
        np.testing.assert_allclose(kh[0] @ q, s_hat, rtol=1e-10, atol=1e-10)
        if r == d:   # M_d = A: the reconstruction is A k itself
            np.testing.assert_allclose(kh[0], K[0, rows] @ A[0].T, rtol=2e-5, atol=2e-5)
    rot = O.reconstruct_keys(codes, res["L"], res["nu"], rows, positions=[5, 6, 7, 8], theta=10000.0)
    np.testing.assert_allclose(rot[0], O.rope(kh[0], np.array([5, 6, 7, 8]), 10000.0), rtol=1e-14)
