"""GPU parity of online moment tracking (saki_moments merged batch by batch,
then saki_fit_moments) against saki_fit on all rows at once and the oracle,
and of the key reconstruction with RoPE (saki_reconstruct_keys) against the
oracle, with q^T k_hat checked against the selection's own reported scores."""
import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import MAP_REL, SCORE_REL, f32, map_rel_err, to_dev

pytestmark = pytest.mark.gpu
D = 128


@pytest.mark.parametrize("center", [0, 1])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_running_moments_and_fit_from_moments(lib, center, dtype):
    import torch
    w = synth.Workload("onl", 4, 2, rank=16, dtype=dtype, n_calib=700, seq_lens=(64,), spikes=(6, 6), seed=51)
    data = synth.make_numpy(w)
    Hq, Hk, r = w.num_q_heads, w.num_kv_heads, w.rank
    cfg = lib.make_config(Hq, Hk, r, 16, dtype, center=center)
    qc, kc = data["q_calib"], data["k_calib"]
    Sq = torch.empty((Hq, D, D), device="cuda")
    Sk = torch.empty((Hk, D, D), device="cuda")
    mu = torch.empty((Hk, D), device="cuda")
    n_prev = 0
    for a, b in ((0, 250), (250, 251), (251, 700)):     # batches of 250, 1 and 449 rows
        lib.saki_moments(cfg, to_dev(np.ascontiguousarray(qc[:, a:b]), dtype), to_dev(np.ascontiguousarray(kc[:, a:b]), dtype),
                         n_prev, Sq, Sk, mu=mu)
        n_prev += b - a
    torch.cuda.synchronize()
    ref = O.fit(qc, kc, data["A"], r, center=bool(center))
    for h in range(Hq):
        assert np.linalg.norm(Sq[h].cpu().numpy() - ref["Sq"][h]) <= 1e-5 * np.linalg.norm(ref["Sq"][h])
    for g in range(Hk):
        assert np.linalg.norm(Sk[g].cpu().numpy() - ref["Sk"][g]) <= 1e-5 * np.linalg.norm(ref["Sk"][g])
        np.testing.assert_allclose(mu[g].cpu().numpy(), ref["mu"][g], atol=1e-5)
    L = torch.empty((Hq, D, r), device="cuda")
    R = torch.empty_like(L)
    sig = torch.empty((Hq, D), device="cuda")
    lib.saki_fit_moments(cfg, Sq, Sk, f32(data["A"]), L, R, mu=mu, sigma=sig)
    Lg, Rg, sg = L.cpu().numpy(), R.cpu().numpy(), sig.cpu().numpy()
    for h in range(Hq):
        s = ref["sigma"][h]
        np.testing.assert_allclose(sg[h], s, atol=1e-4 * s[0], rtol=0)
        if (s[r - 1] - s[r]) / s[0] >= 1e-3:
            assert map_rel_err(Lg[h], Rg[h], ref["M"][h]) <= MAP_REL, h
    with pytest.raises(lib.SakiError) as e:   # shrinkage needs the rows themselves
        lib.saki_fit_moments(lib.make_config(Hq, Hk, r, 16, dtype, center=center, flags=lib.SAKI_FLAG_SHRINK),
                             Sq, Sk, f32(data["A"]), L, R, mu=mu)
    assert e.value.status == 2


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_reconstructed_keys_with_rope(lib, dtype):
    import torch
    rng = np.random.default_rng(52)
    Hq, Hk, r, k, N = 4, 1, 32, 16, 900
    L = (rng.standard_normal((Hq, D, r)) / np.sqrt(D)).astype(np.float32)
    nu = rng.standard_normal((Hq, D)).astype(np.float32)
    codes = O.round_to(dtype, rng.standard_normal((Hq, N, r))).astype(np.float32)
    rows = np.array([0, 5, 899, 17, 431, 431, 2], np.int64)
    pos = np.array([0, 1, 65535, 1 << 20, 7, 8, 123456], np.int64)
    cfg = lib.make_config(Hq, Hk, r, k, dtype)
    out = torch.empty((Hq, len(rows), D), dtype=torch.bfloat16 if dtype == "bf16" else torch.float32, device="cuda")
    skd = to_dev(codes, dtype)
    for theta in (10000.0, 500000.0):
        for p in (None, pos):
            lib.saki_reconstruct_keys(cfg, torch.from_numpy(rows).cuda(), skd, f32(L), out, nu=f32(nu),
                                      positions=None if p is None else torch.from_numpy(p).cuda(), rope_theta=theta)
            got = out.float().cpu().numpy()
            ref = O.reconstruct_keys(codes, L, nu, rows, positions=p, theta=theta)
            scale = np.abs(ref).max()
            tol = (2.0 ** -8 if dtype == "bf16" else 0.0) * np.abs(ref) + 1e-5 * scale
            assert np.all(np.abs(got - ref) <= tol), (theta, p is None, np.abs(got - ref).max())
    # without rotation q^T k_hat is the index's score: the selection reports the same
    if dtype != "f32":
        return
    T = 3
    Q = rng.standard_normal((Hq, T, D)).astype(np.float32)
    lay = lib.HostLayout(np.array([0, N]), np.zeros(T, np.int32), np.full(T, N))
    idx = torch.empty((Hq, T, k), dtype=torch.int32, device="cuda")
    sc = torch.empty((Hq, T, k), dtype=torch.float32, device="cuda")
    lib.saki_score_topk(lib.make_config(Hq, Hk, r, k, "f32", center=1), lay, to_dev(Q, "f32"), f32(L), skd, idx,
                        score=sc, nu=f32(nu))
    kh = torch.empty((Hq, k, D), dtype=torch.float32, device="cuda")
    for t in range(T):
        sel = idx[:, t].cpu().numpy()
        for h in range(Hq):
            lib.saki_reconstruct_keys(cfg, torch.from_numpy(sel[h].astype(np.int64)).cuda(), skd, f32(L), kh,
                                      nu=f32(nu))
            s = kh[h].cpu().numpy().astype(np.float64) @ Q[h, t].astype(np.float64)
            ref = sc[h, t].cpu().numpy()
            np.testing.assert_allclose(s, ref, atol=SCORE_REL * np.abs(ref).max(), rtol=0)
