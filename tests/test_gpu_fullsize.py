"""Parity at the benchmark workloads' full sizes, in the launch configuration the
benchmark times (every head and every query in one call per entry point),
checked on sampled heads, rows and keys that the oracle computes one by one from
host copies of the same generator inputs.

Each stage runs on generator inputs: the calibration and evaluation tensors of
``synth.make_torch``, and for the stages after the fit, seeded random
projections and random bf16 codes, so no oracle input ever comes from the
library's own outputs."""
import numpy as np
import pytest

from oracle import saki_oracle as O
from paper_2608_03228_gb300 import synth
from tests.parity import MAP_REL, check_topk_rows, map_rel_err

pytestmark = pytest.mark.gpu
D = 128


def _torch():
    import torch
    return torch


def _randn(shape, seed, scale=1.0, dtype=None):
    torch = _torch()
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    x = torch.randn(shape, generator=g, device="cuda") * scale
    return x.to(dtype) if dtype is not None else x


def _host(t):
    return t.float().cpu().numpy().astype(np.float64)


def _causal_rows(T, k, seed, extra=10):
    fixed = [0, 1, k - 2, k - 1, k, k + 1, 127, 128, 129, T // 2 - 1, T // 2, T - 2, T - 1]
    rng = np.random.default_rng(seed)
    rows = set(t for t in fixed if 0 <= t < T) | set(rng.integers(0, T, extra).tolist())
    return sorted(rows)


def _sample_rows(w, lay_arrays, seed):
    off, q_seq, q_vis, _ = lay_arrays
    T = len(q_seq)
    if w.queries == "causal" and len(off) == 2:
        return _causal_rows(T, w.topk, seed)
    if w.queries == "decode":
        return list(range(T))
    # ragged tail queries: every query of the first, a middle and the last sequence
    S = len(off) - 1
    seqs = sorted({0, S // 2, S - 1})
    return [t for t in range(T) if q_seq[t] in seqs]


def _select(lib, w, data, L, codes, exact=False, A=None):
    """One saki_score_topk (or saki_recall) call over the whole workload."""
    torch = _torch()
    Hq, T = w.num_q_heads, len(data["q_seq"])
    cfg = lib.make_config(Hq, w.num_kv_heads, w.rank, w.topk, w.dtype)
    lay = lib.HostLayout(data["seq_offsets"], data["q_seq"], data["q_visible"])
    idx = torch.empty((Hq, T, w.topk), dtype=torch.int32, device="cuda")
    if not exact:
        sc = torch.empty((Hq, T, w.topk), dtype=torch.float32, device="cuda")
        lib.saki_score_topk(cfg, lay, data["Q"], L, codes, idx, score=sc)
        torch.cuda.synchronize()
        return idx, sc
    dummy = torch.zeros((Hq, T, w.topk), dtype=torch.int32, device="cuda")
    rec = torch.empty((Hq,), device="cuda")
    lib.saki_recall(cfg, lay, w.topk + 1, data["Q"], A, data["K"], dummy, rec, idx_exact=idx)
    torch.cuda.synchronize()
    r = rec.cpu().numpy()
    assert np.all((r >= 0) & (r <= 1))
    return idx, None


def _check_rows(w, data, idx, sc, heads, rows, src, score_fn, label):
    """src(h, g) -> the device tensor the row scores read ([N][.]); score_fn(h, q,
    X) -> oracle scores of query q against host rows X.  Each (head, sequence)
    prefix is copied to the host once, at its longest visible length."""
    off, q_seq, q_vis = data["seq_offsets"], data["q_seq"], data["q_visible"]
    waived = total = 0
    for h in heads:
        g = h // w.group
        gi = idx[h, rows].cpu().numpy()
        gs = sc[h, rows].cpu().numpy() if sc is not None else None
        Qh = _host(data["Q"][h, rows])
        cache = {}
        for t in rows:
            s = int(q_seq[t])
            cache[s] = max(cache.get(s, 0), int(q_vis[t]))
        X = src(h, g)
        cache = {s: _host(X[int(off[s]):int(off[s]) + v]) for s, v in cache.items()}
        vectors = [score_fn(h, Qh[i], cache[int(q_seq[t])][:int(q_vis[t])]) for i, t in enumerate(rows)]
        e, wv = check_topk_rows(gi, vectors, w.topk, gpu_scores=gs, label=f"{label} h{h}")
        waived += wv
        total += len(rows)
    # A row is waived when the oracle's own k-th/(k+1)-th gap is below 1e-4 of the
    # row maximum; its selection is still checked key by key against that margin.
    # The count depends on the data alone (a simulation of Gaussian scores: about
    # 8 % of rows over 4096 keys, 12 % over 1M); the bound, 30 % of the rows or
    # four, only keeps the exact comparison from becoming vacuous.
    assert waived <= max(4, (3 * total + 9) // 10), (label, waived, total)


# ------------------------------------------------------------------ Llama-3.1-8B shapes
@pytest.fixture(scope="module")
def llama():
    torch = _torch()
    w = synth.WORKLOADS["llama31_8b_t4096_r32"]
    data = synth.make_torch(w, "cuda")
    yield w, data
    del data
    torch.cuda.empty_cache()


def test_fullsize_fit_llama31(lib, llama):
    """saki_fit over all 1024 query heads; M_r, sigma and loss of sampled heads."""
    torch = _torch()
    w, data = llama
    Hq, Hk, r = w.num_q_heads, w.num_kv_heads, w.rank
    cfg = lib.make_config(Hq, Hk, r, w.topk, w.dtype)
    L = torch.empty((Hq, D, r), device="cuda")
    R = torch.empty((Hq, D, r), device="cuda")
    sig = torch.empty((Hq, D), device="cuda")
    loss = torch.empty((Hq,), device="cuda")
    lib.saki_fit(cfg, data["q_calib"], data["k_calib"], data["A"], L, R, sigma=sig, loss=loss)
    torch.cuda.synchronize()
    for h in (0, 517, Hq - 1):
        g = h // w.group
        ref = O.fit(_host(data["q_calib"][h:h + 1]), _host(data["k_calib"][g:g + 1]),
                    _host(data["A"][h:h + 1]), r, center=False)
        s_ref = ref["sigma"][0]
        if (s_ref[r - 1] - s_ref[r]) / s_ref[0] >= 1e-3:
            assert map_rel_err(L[h].cpu().numpy(), R[h].cpu().numpy(), ref["M"][0]) <= MAP_REL, h
        np.testing.assert_allclose(sig[h].cpu().numpy(), s_ref, atol=1e-4 * s_ref[0], rtol=0)
        np.testing.assert_allclose(loss[h].item(), ref["loss"][0], rtol=1e-4, atol=1e-4 * np.sum(s_ref ** 2))


def test_fullsize_build_llama31(lib, llama):
    """saki_build_index over 1024 heads x 4096 keys; sampled codes against the oracle."""
    torch = _torch()
    w, data = llama
    Hq, r = w.num_q_heads, w.rank
    N = data["K"].shape[1]
    R = _randn((Hq, D, r), seed=11, scale=D ** -0.5)
    cfg = lib.make_config(Hq, w.num_kv_heads, r, w.topk, w.dtype)
    sk = torch.empty((Hq, N, r), dtype=torch.bfloat16, device="cuda")
    lib.saki_build_index(cfg, data["K"], R, sk)
    torch.cuda.synchronize()
    keys = np.unique(np.concatenate([[0, 1, 127, 128, N - 1], np.random.default_rng(12).integers(0, N, 200)]))
    for h in (0, 333, Hq - 1):
        g = h // w.group
        Kh = _host(data["K"][g, keys])
        Rh = R[h].cpu().numpy()
        got = sk[h, keys].float().cpu().numpy()
        exact = O.build_index(Kh[None], Rh[None].astype(np.float32), None, "bf16", 1)[0]
        raw = Kh @ Rh.astype(np.float64)
        acc = D * 2.0 ** -24 * (np.abs(Kh) @ np.abs(Rh.astype(np.float64)))
        assert np.all(np.abs(got - raw) <= 2.0 ** -7 * np.abs(raw) + acc + 1e-38), h
        assert np.mean(got == exact) >= 0.999, h


def test_fullsize_select_llama31(lib, llama):
    """saki_score_topk over 1024 heads x 4096 causal queries (the benchmark call)."""
    torch = _torch()
    w, data = llama
    Hq, r = w.num_q_heads, w.rank
    N = data["K"].shape[1]
    L = _randn((Hq, D, r), seed=21, scale=D ** -0.5)
    codes = _randn((Hq, N, r), seed=22, dtype=torch.bfloat16)
    idx, sc = _select(lib, w, data, L, codes)
    rows = _causal_rows(len(data["q_seq"]), w.topk, seed=23)
    Lh = {h: L[h].cpu().numpy() for h in (0, 600, Hq - 1)}

    _check_rows(w, data, idx, sc, sorted(Lh), rows, lambda h, g: codes[h],
                lambda h, q, X: O.approx_scores(q, Lh[h], X), "llama select")


def test_fullsize_exact_llama31(lib, llama):
    """saki_recall's exact top-64 over 1024 heads x 4096 causal queries."""
    w, data = llama
    idx, _ = _select(lib, w, data, None, None, exact=True, A=data["A"])
    rows = _causal_rows(len(data["q_seq"]), w.topk, seed=31)
    heads = (5, 700, w.num_q_heads - 1)
    Ah = {h: _host(data["A"][h]) for h in heads}

    _check_rows(w, data, idx, None, heads, rows, lambda h, g: data["K"][g],
                lambda h, q, X: O.exact_scores(q, Ah[h], X), "llama exact")


# ------------------------------------------------------------------ the other workloads
@pytest.mark.parametrize("name", ["qwen25_7b_t4096_r32_n512", "qwen25_7b_t4096_r32_n32768"])
def test_fullsize_fit_calibration_sweep(lib, name):
    """saki_fit over all 784 Qwen2.5-7B-shaped heads at the ends of the
    calibration-length sweep (512 and 32,768 tokens, Fig. 2A); M_r, sigma and
    loss of sampled heads against the oracle."""
    torch = _torch()
    w = synth.WORKLOADS[name]
    data = synth.make_torch(w, "cuda")
    Hq, Hk, r = w.num_q_heads, w.num_kv_heads, w.rank
    cfg = lib.make_config(Hq, Hk, r, w.topk, w.dtype)
    L = torch.empty((Hq, D, r), device="cuda")
    R = torch.empty((Hq, D, r), device="cuda")
    sig = torch.empty((Hq, D), device="cuda")
    loss = torch.empty((Hq,), device="cuda")
    lib.saki_fit(cfg, data["q_calib"], data["k_calib"], data["A"], L, R, sigma=sig, loss=loss)
    torch.cuda.synchronize()
    for h in (0, 391, Hq - 1):
        g = h // w.group
        ref = O.fit(_host(data["q_calib"][h:h + 1]), _host(data["k_calib"][g:g + 1]),
                    _host(data["A"][h:h + 1]), r, center=False)
        s_ref = ref["sigma"][0]
        if (s_ref[r - 1] - s_ref[r]) / s_ref[0] >= 1e-3:
            assert map_rel_err(L[h].cpu().numpy(), R[h].cpu().numpy(), ref["M"][0]) <= MAP_REL, h
        np.testing.assert_allclose(sig[h].cpu().numpy(), s_ref, atol=1e-4 * s_ref[0], rtol=0)
        np.testing.assert_allclose(loss[h].item(), ref["loss"][0], rtol=1e-4, atol=1e-4 * np.sum(s_ref ** 2))
    del data
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["qwen25_7b_t4096_r32", "qwen25_7b_t4096_r16", "qwen25_7b_t4096_r64",
                                  "llama32_3b_t4096_r32", "decode_n1m_b1_r32", "decode_n1m_b8_r32",
                                  "ragged64_mistral7b_r64"])
def test_fullsize_select_workloads(lib, name):
    """Approximate and exact selection at each workload's full size."""
    torch = _torch()
    w = synth.WORKLOADS[name]
    data = synth.make_torch(w, "cuda")
    lay_arrays = (data["seq_offsets"], data["q_seq"], data["q_visible"], None)
    Hq, r = w.num_q_heads, w.rank
    N = data["K"].shape[1]
    L = _randn((Hq, D, r), seed=41, scale=D ** -0.5)
    codes = _randn((Hq, N, r), seed=42, dtype=torch.bfloat16)
    rows = _sample_rows(w, lay_arrays, seed=43)
    heads = (0, Hq - 1)
    idx, sc = _select(lib, w, data, L, codes)
    Lh = {h: L[h].cpu().numpy() for h in heads}

    _check_rows(w, data, idx, sc, heads, rows, lambda h, g: codes[h],
                lambda h, q, X: O.approx_scores(q, Lh[h], X), f"{name} select")
    del idx, sc, codes
    idx, _ = _select(lib, w, data, None, None, exact=True, A=data["A"])
    Ah = {h: _host(data["A"][h]) for h in heads[:1]}

    _check_rows(w, data, idx, None, heads[:1], rows, lambda h, g: data["K"][g],
                lambda h, q, X: O.exact_scores(q, Ah[h], X), f"{name} exact")
    del idx, data
    torch.cuda.empty_cache()
