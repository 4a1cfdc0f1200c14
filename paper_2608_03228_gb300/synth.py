"""Seeded synthetic inputs shaped like the SAKI paper's retrieval workloads.

This module only draws random data.  It holds none of the method's
arithmetic (no moments, no fit, no sketch, no scoring, no selection): both the
CUDA path and the CPU oracle consume the arrays it returns, and neither side's
results ever flow back into it.

Recipe (the paper's protocol, Sec. 3, uses activations of real models on
natural text; these synthetic stand-ins keep its shapes and spectra):

* Score operator per query head: ``A_h = G diag(i^-0.8) O`` with ``G_ij ~
  N(0, 1/d)`` and ``O`` Haar-orthogonal (QR of a Gaussian matrix with the sign
  of ``diag(R)`` folded in).  Such an operator is strongly non-normal, as the
  paper's Sec. 4 reports for real heads.
* Key covariance per KV head and query covariance per query head:
  ``Sigma = Q diag(spec) Q^T`` with ``Q`` Haar and ``spec`` = ``s`` spikes
  ``linspace(50, 5, s)`` followed by a Marchenko-Pastur bulk (the sorted
  eigenvalues of one Wishart sample ``X^T X / m`` with aspect ratio
  ``(d - s) / m = 0.5``).  Queries use an independent basis and bulk draw.
* Vectors: ``x = Q diag(sqrt(spec)) z`` with ``z ~ N(0, I)``; calibration and
  evaluation draws are independent.  bf16 workloads round the fp32 draws to
  the bf16 grid (round-to-nearest-even); those rounded values *are* the data.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np

__all__ = ["Workload", "WORKLOADS", "HeadFactors", "head_factors", "make_numpy",
           "make_torch", "seq_layout", "round_to_bf16_grid"]


@dataclass(frozen=True)
class Workload:
    """Shapes of one retrieval workload.  Layers are folded into the head axis."""

    name: str
    num_q_heads: int
    num_kv_heads: int
    head_dim: int = 128
    rank: int = 32
    topk: int = 64
    dtype: str = "bf16"            # "f32" or "bf16": q, k, calibration data, sketch
    n_calib: int = 4096
    seq_lens: tuple = (4096,)      # keys per sequence
    queries: str = "causal"        # "causal" | "tail" | "decode"
    q_per_seq: int = 0             # queries per sequence for "tail" / "decode"
    spikes: tuple = (8, 8)         # inclusive range of spike counts per head
    center: int = 0
    seed: int = 0
    layers: int = 1                # informational: heads = layers x heads/layer
    ragged: tuple = ()             # (num_seqs, min_len, max_len) drawn from seed

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    def lens(self) -> tuple:
        if self.ragged:
            ns, lo, hi = self.ragged
            rng = np.random.default_rng(np.random.SeedSequence([self.seed, 0x5E9]))
            return tuple(int(v) for v in rng.integers(lo, hi + 1, size=ns))
        return tuple(self.seq_lens)


# The five workloads (Sec. 3 protocol shapes; decode and ragged batches follow the
# 1M-token motivation of Sec. 1).  Names say what they are, with their sizes.
WORKLOADS = {
    # 4 query heads on 1 KV head, fp32, T = N = 512 causal, r = 16
    "tiny_f32_t512": Workload("tiny_f32_t512", 4, 1, rank=16, dtype="f32",
                              n_calib=512, seq_lens=(512,), spikes=(8, 8), seed=0),
    # LLaMA-3.1-8B shape: 32 layers x 32 query heads / 8 KV heads, T = N = 4096 causal
    "llama31_8b_t4096_r32": Workload("llama31_8b_t4096_r32", 32 * 32, 32 * 8, rank=32,
                                     n_calib=4096, seq_lens=(4096,), spikes=(2, 16),
                                     seed=1, layers=32),
    # Qwen2.5-7B shape: 28 layers x 28 query heads / 4 KV heads (GQA 7)
    "qwen25_7b_t4096_r32": Workload("qwen25_7b_t4096_r32", 28 * 28, 28 * 4, rank=32,
                                    n_calib=4096, seq_lens=(4096,), spikes=(2, 16),
                                    seed=2, layers=28),
    # the rank sweep at that shape (Tab. 2 reports r = 16, 32, 64)
    "qwen25_7b_t4096_r16": Workload("qwen25_7b_t4096_r16", 28 * 28, 28 * 4, rank=16,
                                    n_calib=4096, seq_lens=(4096,), spikes=(2, 16),
                                    seed=2, layers=28),
    "qwen25_7b_t4096_r64": Workload("qwen25_7b_t4096_r64", 28 * 28, 28 * 4, rank=64,
                                    n_calib=4096, seq_lens=(4096,), spikes=(2, 16),
                                    seed=2, layers=28),
    # the calibration-length sweep at r = 32 (Fig. 2A: 512 to 32,768 tokens)
    "qwen25_7b_t4096_r32_n512": Workload("qwen25_7b_t4096_r32_n512", 28 * 28, 28 * 4, rank=32,
                                         n_calib=512, seq_lens=(4096,), spikes=(2, 16),
                                         seed=2, layers=28),
    "qwen25_7b_t4096_r32_n32768": Workload("qwen25_7b_t4096_r32_n32768", 28 * 28, 28 * 4, rank=32,
                                           n_calib=32768, seq_lens=(4096,), spikes=(2, 16),
                                           seed=2, layers=28),
    # Llama-3.2-3B shape: 28 layers x 24 query heads / 8 KV heads
    "llama32_3b_t4096_r32": Workload("llama32_3b_t4096_r32", 28 * 24, 28 * 8, rank=32,
                                     n_calib=4096, seq_lens=(4096,), spikes=(2, 16),
                                     seed=3, layers=28),
    # one layer, 32 query / 8 KV heads, 1,048,576 cached keys, decode batch of 8
    "decode_n1m_b8_r32": Workload("decode_n1m_b8_r32", 32, 8, rank=32, n_calib=4096,
                                  seq_lens=(1 << 20,), queries="decode", q_per_seq=8,
                                  spikes=(8, 8), seed=4),
    "decode_n1m_b1_r32": Workload("decode_n1m_b1_r32", 32, 8, rank=32, n_calib=4096,
                                  seq_lens=(1 << 20,), queries="decode", q_per_seq=1,
                                  spikes=(8, 8), seed=4),
    # Mistral-7B shape, 64 sequences of 4096..65536 keys, 4 queries each, r = 64
    "ragged64_mistral7b_r64": Workload("ragged64_mistral7b_r64", 32, 8, rank=64,
                                       n_calib=4096, queries="tail", q_per_seq=4,
                                       spikes=(8, 8), seed=5, ragged=(64, 4096, 65536)),
}


def _haar(rng: np.random.Generator, d: int) -> np.ndarray:
    z = rng.standard_normal((d, d))
    q, r = np.linalg.qr(z)
    return q * np.sign(np.diag(r))


def _spectrum(rng: np.random.Generator, d: int, s: int) -> np.ndarray:
    spikes = np.linspace(50.0, 5.0, s) if s > 0 else np.zeros(0)
    p = d - s
    m = int(round(p / 0.5))
    x = rng.standard_normal((m, p))
    bulk = np.sort(np.linalg.eigvalsh(x.T @ x / m))[::-1]
    return np.concatenate([spikes, bulk])


@dataclass
class HeadFactors:
    """Per-head generator factors: x = F z gives covariance F F^T."""

    A: np.ndarray        # [Hq][d][d] float32 score operator, s = q^T A k
    Fq: np.ndarray       # [Hq][d][d] float64 query factor
    Fk: np.ndarray       # [Hk][d][d] float64 key factor
    spikes_q: np.ndarray
    spikes_k: np.ndarray


def head_factors(w: Workload, heads: tuple | None = None) -> HeadFactors:
    """Draw A_h and the covariance factors.  ``heads`` restricts to a subset of
    query heads (their KV heads follow); draws depend only on (seed, head)."""
    d = w.head_dim
    hq = list(range(w.num_q_heads)) if heads is None else list(heads)
    hk = sorted({h // w.group for h in hq})
    lo, hi = w.spikes
    A = np.empty((len(hq), d, d), np.float32)
    Fq = np.empty((len(hq), d, d))
    Fk = np.empty((len(hk), d, d))
    sq = np.empty(len(hq), np.int64)
    sk = np.empty(len(hk), np.int64)
    for i, h in enumerate(hq):
        rng = np.random.default_rng(np.random.SeedSequence([w.seed, 1, h]))
        g = rng.standard_normal((d, d)) / math.sqrt(d)
        o = _haar(rng, d)
        A[i] = (g * (np.arange(1, d + 1, dtype=np.float64) ** -0.8)) @ o
        s = int(rng.integers(lo, hi + 1))
        spec = _spectrum(rng, d, s)
        Fq[i] = _haar(rng, d) * np.sqrt(spec)
        sq[i] = s
    for i, g_ in enumerate(hk):
        rng = np.random.default_rng(np.random.SeedSequence([w.seed, 2, g_]))
        s = int(rng.integers(lo, hi + 1))
        spec = _spectrum(rng, d, s)
        Fk[i] = _haar(rng, d) * np.sqrt(spec)
        sk[i] = s
    return HeadFactors(A, Fq, Fk, sq, sk)


def round_to_bf16_grid(x: np.ndarray) -> np.ndarray:
    """Round float32 data to the nearest bf16 value (ties to even); returns
    float32 holding exactly representable values.  Data preparation only."""
    x = np.ascontiguousarray(x, np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) & 0xFFFF0000
    return b.astype(np.uint32).view(np.float32)


def seq_layout(w: Workload):
    """Host layout: seq_offsets [S+1] int64, q_seq [T] int32, q_visible [T] int64,
    q_pos [T] int64 (position of each query inside its sequence)."""
    lens = w.lens()
    off = np.zeros(len(lens) + 1, np.int64)
    off[1:] = np.cumsum(lens)
    qs, qv, qp = [], [], []
    for s, L in enumerate(lens):
        if w.queries == "causal":
            pos = np.arange(L)
            vis = pos + 1
        elif w.queries == "tail":
            pos = np.arange(L - w.q_per_seq, L)
            vis = pos + 1
        elif w.queries == "decode":
            pos = np.full(w.q_per_seq, L - 1)
            vis = np.full(w.q_per_seq, L)
        else:
            raise ValueError(w.queries)
        qs.append(np.full(len(pos), s, np.int32))
        qv.append(vis.astype(np.int64))
        qp.append(pos.astype(np.int64))
    return off, np.concatenate(qs), np.concatenate(qv), np.concatenate(qp)


def _draw(rng: np.random.Generator, F: np.ndarray, n: int) -> np.ndarray:
    z = rng.standard_normal((n, F.shape[0]))
    return (z @ F.T).astype(np.float32)


def make_numpy(w: Workload, heads: tuple | None = None) -> dict:
    """All inputs on the host as float32 arrays (bf16 workloads: values on the bf16
    grid).  Keys: A, q_calib, k_calib, Q, K, seq_offsets, q_seq, q_visible, q_pos."""
    f = head_factors(w, heads)
    off, q_seq, q_vis, q_pos = seq_layout(w)
    T, N = len(q_seq), int(off[-1])
    n = w.n_calib
    hq = list(range(w.num_q_heads)) if heads is None else list(heads)
    hk = sorted({h // w.group for h in hq})
    rnd = round_to_bf16_grid if w.dtype == "bf16" else (lambda a: a)
    q_cal = np.empty((len(hq), n, w.head_dim), np.float32)
    Q = np.empty((len(hq), T, w.head_dim), np.float32)
    for i, h in enumerate(hq):
        q_cal[i] = rnd(_draw(np.random.default_rng(np.random.SeedSequence([w.seed, 3, h])), f.Fq[i], n))
        Q[i] = rnd(_draw(np.random.default_rng(np.random.SeedSequence([w.seed, 4, h])), f.Fq[i], T))
    k_cal = np.empty((len(hk), n, w.head_dim), np.float32)
    K = np.empty((len(hk), N, w.head_dim), np.float32)
    for i, g in enumerate(hk):
        k_cal[i] = rnd(_draw(np.random.default_rng(np.random.SeedSequence([w.seed, 5, g])), f.Fk[i], n))
        K[i] = rnd(_draw(np.random.default_rng(np.random.SeedSequence([w.seed, 6, g])), f.Fk[i], N))
    return dict(A=f.A, q_calib=q_cal, k_calib=k_cal, Q=Q, K=K, seq_offsets=off,
                q_seq=q_seq, q_visible=q_vis, q_pos=q_pos, factors=f)


def make_torch(w: Workload, device, seed_offset: int = 0) -> dict:
    """Same recipe with the Gaussian draws made on ``device`` by torch (for the
    full-size workloads).  Factors come from :func:`head_factors`; vectors are
    drawn in chunks so peak temporary memory stays small.  Returns torch
    tensors in the workload dtype plus the host layout arrays."""
    import torch

    f = head_factors(w)
    off, q_seq, q_vis, q_pos = seq_layout(w)
    T, N = len(q_seq), int(off[-1])
    n, d = w.n_calib, w.head_dim
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    gen = torch.Generator(device=device)
    gen.manual_seed(w.seed * 1000003 + seed_offset)

    def draw(F: np.ndarray, rows: int) -> "torch.Tensor":
        H = F.shape[0]
        out = torch.empty((H, rows, d), dtype=dt, device=device)
        Ft = torch.from_numpy(np.ascontiguousarray(np.transpose(F, (0, 2, 1)))).to(device, torch.float32)
        step = max(1, (1 << 26) // (rows * d))
        for h0 in range(0, H, step):
            h1 = min(H, h0 + step)
            z = torch.randn((h1 - h0, rows, d), generator=gen, device=device, dtype=torch.float32)
            out[h0:h1] = torch.bmm(z, Ft[h0:h1]).to(dt)
        return out

    return dict(A=torch.from_numpy(f.A).to(device), q_calib=draw(f.Fq, n), k_calib=draw(f.Fk, n),
                Q=draw(f.Fq, T), K=draw(f.Fk, N), seq_offsets=off, q_seq=q_seq,
                q_visible=q_vis, q_pos=q_pos, factors=f)
