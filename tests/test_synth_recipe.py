"""The synthetic input recipe, checked on CPU: planted spectra, per-head
determinism (sampled full-size tests draw single heads and must see the same
data as the whole workload), bf16 data on the bf16 grid, and the query layouts
of the causal, tail and decode workloads."""
import numpy as np
import pytest

from paper_2608_03228_gb300 import synth


def test_population_spectra_carry_the_planted_spikes():
    """Sigma = Q diag(spec) Q^T: the s spikes linspace(50, 5, s) sit above a
    Marchenko-Pastur bulk of aspect 0.5, whose edge (1 + sqrt(0.5))^2 < 3 < 5."""
    w = synth.Workload("recipe", 4, 2, spikes=(2, 16), seed=7)
    f = synth.head_factors(w)
    for F, s in [(F, s) for F, s in zip(f.Fq, f.spikes_q)] + [(F, s) for F, s in zip(f.Fk, f.spikes_k)]:
        assert 2 <= s <= 16
        lam = np.sort(np.linalg.eigvalsh(F @ F.T))[::-1]
        np.testing.assert_allclose(lam[:s], np.linspace(50.0, 5.0, s), rtol=1e-10)
        assert lam[s] < 3.0 and lam[-1] > 0.0


def test_operator_has_the_power_law_profile():
    """A_h = G diag(i^-0.8) O with G ~ N(0, 1/d): A_h^T A_h = O^T D G^T G D O, so
    its eigenvalues are those of D G^T G D, whose trace is sum_i i^-1.6 |g_i|^2
    (about sum_i i^-1.6 on average over the d Gaussian columns)."""
    w = synth.Workload("recipe", 64, 8, seed=3)
    A = synth.head_factors(w).A.astype(np.float64)
    d = w.head_dim
    ref = np.sum(np.arange(1, d + 1) ** -1.6)
    fro2 = np.mean(np.sum(A * A, axis=(1, 2)))
    assert fro2 == pytest.approx(ref, rel=0.05)
    # strongly non-normal, as Sec. 4 reports for real heads
    dep = np.linalg.norm(A @ np.transpose(A, (0, 2, 1)) - np.transpose(A, (0, 2, 1)) @ A, axis=(1, 2))
    assert np.all(dep > 0.1 * np.linalg.norm(A, axis=(1, 2)) ** 2)


def test_draws_depend_only_on_seed_and_head():
    w = synth.Workload("recipe", 8, 2, rank=16, n_calib=64, seq_lens=(96,), seed=5)
    full = synth.make_numpy(w)
    part = synth.make_numpy(w, heads=[5])
    np.testing.assert_array_equal(part["A"][0], full["A"][5])
    np.testing.assert_array_equal(part["q_calib"][0], full["q_calib"][5])
    np.testing.assert_array_equal(part["Q"][0], full["Q"][5])
    np.testing.assert_array_equal(part["k_calib"][0], full["k_calib"][5 // w.group])
    np.testing.assert_array_equal(part["K"][0], full["K"][5 // w.group])


def test_bf16_data_sits_on_the_bf16_grid():
    torch = pytest.importorskip("torch")
    w = synth.Workload("recipe", 2, 1, rank=16, n_calib=64, seq_lens=(64,), seed=1)
    data = synth.make_numpy(w)
    for key in ("q_calib", "k_calib", "Q", "K"):
        x = torch.from_numpy(data[key])
        assert torch.equal(x.to(torch.bfloat16).to(torch.float32), x), key
    x = np.random.default_rng(2).standard_normal(5000).astype(np.float32)
    np.testing.assert_array_equal(synth.round_to_bf16_grid(x),
                                  torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy())


def test_query_layouts():
    off, q_seq, vis, pos = synth.seq_layout(synth.Workload("c", 1, 1, seq_lens=(5, 3)))
    np.testing.assert_array_equal(off, [0, 5, 8])
    np.testing.assert_array_equal(q_seq, [0] * 5 + [1] * 3)
    np.testing.assert_array_equal(vis, [1, 2, 3, 4, 5, 1, 2, 3])          # causal: query t sees keys 0..t
    w = synth.WORKLOADS["ragged64_mistral7b_r64"]
    off, q_seq, vis, pos = synth.seq_layout(w)
    lens = np.diff(off)
    assert len(lens) == 64 and lens.min() >= 4096 and lens.max() <= 65536
    for s in (0, 31, 63):                                                # tail: the last 4 positions
        np.testing.assert_array_equal(vis[q_seq == s], lens[s] - np.arange(3, -1, -1))
    off, q_seq, vis, pos = synth.seq_layout(synth.WORKLOADS["decode_n1m_b8_r32"])
    assert len(vis) == 8 and np.all(vis == 1 << 20) and np.all(pos == (1 << 20) - 1)
