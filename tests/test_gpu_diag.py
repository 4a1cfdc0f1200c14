"""GPU parity of the Sec. 7 diagnostics and App. C's measurement against the
oracle: Ledoit-Wolf shrinkage of both moments inside saki_fit, the key
correlation spectrum with its Marchenko-Pastur spike count, and the measured
score-MSE reduction."""
import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import MAP_REL, f32, map_rel_err, to_dev

pytestmark = pytest.mark.gpu
D = 128


@pytest.mark.parametrize("center", [0, 1])
@pytest.mark.parametrize("dtype,n", [("f32", 512), ("bf16", 96)])
def test_fit_with_ledoit_wolf_shrinkage(lib, center, dtype, n):
    import torch
    w = synth.Workload("lw", 4, 2, rank=16, dtype=dtype, n_calib=n, seq_lens=(64,), spikes=(6, 6), seed=31)
    data = synth.make_numpy(w)
    Hq, Hk, r = w.num_q_heads, w.num_kv_heads, w.rank
    cfg = lib.make_config(Hq, Hk, r, 16, dtype, center=center, flags=lib.SAKI_FLAG_SHRINK)
    L = torch.empty((Hq, D, r), device="cuda")
    R = torch.empty_like(L)
    mu = torch.empty((Hk, D), device="cuda")
    ws = torch.empty(lib.saki_workspace_size(cfg, lib.SAKI_OP_FIT, n_calib=n), dtype=torch.uint8, device="cuda")
    lib.saki_fit(cfg, to_dev(data["q_calib"], dtype), to_dev(data["k_calib"], dtype), f32(data["A"]), L, R, mu=mu,
                 workspace=ws)
    torch.cuda.synchronize()
    nm = Hq + Hk
    S = ws[: nm * D * D * 4].view(torch.float32).reshape(nm, D, D).cpu().numpy()
    ref = O.fit(data["q_calib"], data["k_calib"], data["A"], r, center=bool(center), shrink=True)
    for h in range(Hq):   # shrunk moments: fp32 accumulation, then the same convex combination
        assert np.linalg.norm(S[h] - ref["Sq"][h]) <= 2e-5 * np.linalg.norm(ref["Sq"][h]), h
    for g in range(Hk):
        assert np.linalg.norm(S[Hq + g] - ref["Sk"][g]) <= 2e-5 * np.linalg.norm(ref["Sk"][g]), g
    Lg, Rg = L.cpu().numpy(), R.cpu().numpy()
    for h in range(Hq):
        s = ref["sigma"][h]
        if (s[r - 1] - s[r]) / s[0] >= 1e-3:
            assert map_rel_err(Lg[h], Rg[h], ref["M"][h]) <= MAP_REL, h


@pytest.mark.parametrize("center", [0, 1])
def test_key_spectrum_and_spike_count(lib, center):
    import torch
    w = synth.Workload("spec", 8, 4, rank=16, dtype="f32", n_calib=1024, seq_lens=(64,), spikes=(2, 14), seed=32)
    data = synth.make_numpy(w)
    Hk = w.num_kv_heads
    cfg = lib.make_config(w.num_q_heads, Hk, w.rank, 16, "f32", center=center)
    eig = torch.empty((Hk, D), device="cuda")
    spikes = torch.empty((Hk,), dtype=torch.int32, device="cuda")
    for tau in (1.0, 3.2):
        lib.saki_key_spectrum(cfg, to_dev(data["k_calib"], "f32"), eig, spikes, tau_int=tau)
        ev, sp = eig.cpu().numpy(), spikes.cpu().numpy()
        edge = O.mp_upper_edge(D, w.n_calib, tau)
        for g in range(Hk):
            Sk = O.moments(data["k_calib"][g], bool(center))[0]
            ref = O.correlation_spectrum(Sk)
            np.testing.assert_allclose(ev[g], ref, atol=2e-5 * ref[0], rtol=0)
            # the count is unique unless an eigenvalue sits within rounding of the edge
            if np.all(np.abs(ref - edge) > 1e-4 * ref[0]):
                assert sp[g] == O.mp_spike_count(Sk, w.n_calib, tau), (g, tau)
        assert abs(ev.sum(axis=1) - D).max() < 1e-2   # unit diagonal: the trace is d


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_score_mse_matches_the_oracle(lib, dtype):
    import torch
    w = synth.Workload("mse", 4, 2, rank=16, dtype=dtype, n_calib=512, seq_lens=(300, 200), spikes=(6, 6), seed=33)
    data = synth.make_numpy(w)
    Hq, Hk, r = w.num_q_heads, w.num_kv_heads, w.rank
    ref = O.fit(data["q_calib"], data["k_calib"], data["A"], r, center=True)
    L = ref["L"].astype(np.float32)
    codes = O.build_index(data["K"], ref["R"].astype(np.float32), ref["mu"].astype(np.float32), dtype, w.group)
    codes = codes.astype(np.float32)
    nu = ref["nu"].astype(np.float32)
    cfg = lib.make_config(Hq, Hk, r, 16, dtype, center=1)
    lay = lib.HostLayout(data["seq_offsets"], data["q_seq"], data["q_visible"])
    out = torch.empty((Hq, 3), dtype=torch.float64, device="cuda")
    for stride in (1, 7):
        lib.saki_score_mse(cfg, lay, to_dev(data["Q"], dtype), f32(data["A"]), to_dev(data["K"], dtype), f32(L),
                           to_dev(codes, dtype), out, nu=f32(nu), key_stride=stride)
        got = out.cpu().numpy()
        exp = O.score_mse(data["Q"], data["A"], data["K"], L, codes, nu, data["seq_offsets"], data["q_seq"],
                          data["q_visible"], w.group, key_stride=stride)
        np.testing.assert_array_equal(got[:, 2], exp[:, 2])
        np.testing.assert_allclose(got[:, 0], exp[:, 0], rtol=1e-5)
        np.testing.assert_allclose(got[:, 1], exp[:, 1], rtol=1e-4)
        # measured reduction near the predicted one (App. C; finite-sample noise)
        pred = 1 - ref["loss"] / np.sum(ref["sigma"] ** 2, axis=1)
        meas = 1 - got[:, 1] / got[:, 0]
        assert np.all(np.abs(meas - pred) < 0.1), (meas, pred)
