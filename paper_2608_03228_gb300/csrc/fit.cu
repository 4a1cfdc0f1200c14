// The closed-form fit of Prop. 1 (Eq. 3, Sec. 5), Sec. 6 and App. A, one CTA per matrix.
//
// factor_kernel: for each moment matrix S (query heads, then KV heads) a factor F
//   with F F^T = S and G = F^{+T}.  Fast path: Cholesky S = F F^T, G = F^{-T},
//   taken only when lambda_min(S) >= 1/||F^{-1}||_F^2 >= floor * trace(S) >=
//   floor * lambda_max(S) proves that the eigenvalue floor of App. A drops
//   nothing.  Otherwise the floor is applied exactly: eigenpairs of S from a
//   one-sided Jacobi run on S (S V = V Lambda for a PSD matrix), F = V_+
//   Lambda_+^{1/2}, G = V_+ Lambda_+^{-1/2} over the kept eigenvalues.  F is
//   stored row-major, G column-major (the fit kernel reads G's columns with
//   consecutive rows in consecutive lanes).
//   Any factor with F F^T = S yields the same optimum, because
//   ||F_q^T X F_k||_F^2 = tr(X^T Sq X Sk) for every X.
//
// fit_kernel: per query head h with KV head g,
//   C' = Fq^T A_h Fk (singular values equal those of Sq^{1/2} A_h Sk^{1/2}),
//   C' = Q1 R1 (Householder QR, as preconditioning), one-sided (Hestenes)
//   Jacobi on R1^T: its columns converge to V Sigma with V the right singular
//   vectors of C' (C'^T = R1^T Q1^T); then
//   R = Gk V_r Sigma_r^{1/2}  and  L = Gq (C' V_r) Sigma_r^{-1/2} = Gq U_r Sigma_r^{1/2},
//   so L R^T = M_r, loss = sum_{i>r} sigma_i^2 and nu = A_h mu_g.
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {

constexpr int kFitThreads = 512;

__device__ __forceinline__ void rr_pair(int round, int k, int& pa, int& pb) {
  // round-robin (circle) schedule of kD players: position 0 fixed, others rotate
  auto player = [&](int p) { return p == 0 ? 0 : ((p - 1 + round) % (kD - 1)) + 1; };
  pa = player(k);
  pb = player(kD - 1 - k);
}

// One-sided Jacobi on the columns of X (column-major, leading dimension kLdS) until
// every pair satisfies |x_a . x_b| <= tol ||x_a|| ||x_b||.  Columns of norm below
// 1e-7 ||X||_F count as zero (their pairs are not rotated): they carry no
// singular value that matters, and rounding noise left in exactly rank-deficient
// inputs would otherwise keep rotating.  Needs kFitThreads threads; returns true
// on convergence within max_sweeps.
__device__ bool jacobi_columns(float* X, int max_sweeps, float tol, int* s_counter) {
  __shared__ float s_red[kFitThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float fro = 0.f;
  for (int o = tid; o < kD * kD; o += kFitThreads) {
    const float v = X[(o / kD) * kLdS + (o % kD)];
    fro = fmaf(v, v, fro);
  }
  fro = warp_sum(fro);
  if (lane == 0) s_red[warp] = fro;
  __syncthreads();
  fro = 0.f;
  for (int w = 0; w < kFitThreads / 32; ++w) fro += s_red[w];
  const float tiny = fro * 1e-14f;   // squared column norm treated as zero
  for (int sweep = 0; sweep < max_sweeps; ++sweep) {
    if (tid == 0) *s_counter = 0;
    __syncthreads();
    int rot = 0;
    for (int round = 0; round < kD - 1; ++round) {
      // eight lanes per pair: lane group q = lane / 8 of the warp holds rows
      // sub + 8u (u < 16) of the pair's two columns, so a dot product needs only
      // three butterfly steps inside the group, and the four pairs run side by side
      // pair index (warp % 8) + 8 q + 32 (warp / 8): the four groups' columns sit 8
      // apart, so their 8-bank windows of shared memory do not overlap
      const int q = lane >> 3, sub = lane & 7;
      int pa, pb;
      rr_pair(round, (warp & 7) + 8 * q + 32 * (warp >> 3), pa, pb);
      float* xa = X + pa * kLdS + sub;
      float* xb = X + pb * kLdS + sub;
      float a[16], b[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        a[u] = xa[8 * u];
        b[u] = xb[8 * u];
      }
      float al0 = 0.f, al1 = 0.f, be0 = 0.f, be1 = 0.f, ga0 = 0.f, ga1 = 0.f;
#pragma unroll
      for (int u = 0; u < 16; u += 2) {
        al0 = fmaf(a[u], a[u], al0);
        al1 = fmaf(a[u + 1], a[u + 1], al1);
        be0 = fmaf(b[u], b[u], be0);
        be1 = fmaf(b[u + 1], b[u + 1], be1);
        ga0 = fmaf(a[u], b[u], ga0);
        ga1 = fmaf(a[u + 1], b[u + 1], ga1);
      }
      float al = al0 + al1, be = be0 + be1, ga = ga0 + ga1;
#pragma unroll
      for (int m = 4; m > 0; m >>= 1) {  // butterflies leave the group's sums in all eight lanes
        al += __shfl_xor_sync(0xffffffffu, al, m);
        be += __shfl_xor_sync(0xffffffffu, be, m);
        ga += __shfl_xor_sync(0xffffffffu, ga, m);
      }
      if (ga != 0.f && al > tiny && be > tiny && fabsf(ga) > tol * sqrtf(al) * sqrtf(be)) {
        const float zeta = (be - al) / (2.f * ga);
        const float t = fabsf(zeta) > 1e18f ? 0.5f / zeta
                                            : copysignf(1.f, zeta) / (fabsf(zeta) + sqrtf(fmaf(zeta, zeta, 1.f)));
        const float c = 1.f / sqrtf(fmaf(t, t, 1.f));
        const float sn = c * t;
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          xa[8 * u] = c * a[u] - sn * b[u];
          xb[8 * u] = sn * a[u] + c * b[u];
        }
        if (sub == 0) ++rot;
      }
      __syncthreads();
    }
    if ((lane & 7) == 0 && rot) atomicAdd(s_counter, rot);   // one counter per pair group
    __syncthreads();
    const int total = *s_counter;
    __syncthreads();
    if (total == 0) return true;
  }
  return false;
}

// x . y over the 128 rows that a lane group of eight holds (16 per lane as
// float2 pairs), in all eight lanes.
__device__ __forceinline__ float group_dot(const float2 (&x)[8], const float2 (&y)[8]) {
  float2 p = make_float2(0.f, 0.f);
#pragma unroll
  for (int e = 0; e < 8; ++e) p = __ffma2_rn(x[e], y[e], p);
  float v = p.x + p.y;
#pragma unroll
  for (int m = 4; m > 0; m >>= 1) v += __shfl_xor_sync(0xffffffffu, v, m);
  return v;
}

// Leading dimension of the fit kernel's Jacobi matrix: 16-byte aligned columns
// whose starts step through the banks by four.
constexpr int kLdJ = kD + 4;

// jacobi_columns for a matrix with leading dimension kLdJ, with 16-byte shared
// accesses, packed fp32 pairs and a pair order that keeps one column of every
// pair in registers (the same rotation rule and threshold; it also stops after
// a sweep whose rotations were all within sqrt(tol) of orthogonal, see below):
// lane group q = lane / 8 of a warp holds rows 32 w + 4 sub + j (w, j < 4,
// sub = lane % 8) of its pair's two columns, so a column moves in four 16-byte
// accesses per lane and the group's eight lanes cover all 32 banks; the dot
// products and the rotation run on float2 pairs (two fp32 FMAs per instruction,
// each rounded as the scalar one).  With both columns of every pair loaded and
// stored each round, the sweeps were bound by shared-memory bandwidth (128 KB
// per round); the nested order halves that, with as many sweeps (fp32 emulation
// on the bench's operators: 7 or 8 either way, the same singular values and
// rank-r maps).
__device__ bool jacobi_columns_v4(float* X, int max_sweeps, float tol) {
  __shared__ float s_red[kFitThreads / 32];
  __shared__ unsigned int s_off;   // bits of the sweep's largest rotated off-diagonality (>= 0)
  __shared__ float s_nrm[kD];      // squared norms of the rotating columns, carried through a level
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float fro = 0.f;
  for (int o = tid; o < kD * kD; o += kFitThreads) {
    const float v = X[(o / kD) * kLdJ + (o % kD)];
    fro = fmaf(v, v, fro);
  }
  fro = warp_sum(fro);
  if (lane == 0) s_red[warp] = fro;
  __syncthreads();
  fro = 0.f;
  for (int w = 0; w < kFitThreads / 32; ++w) fro += s_red[w];
  const float tiny = fro * 1e-14f;   // squared column norm treated as zero
  const int q = lane >> 3, sub = lane & 7;
  const float stop_off = sqrtf(tol);
  for (int sweep = 0; sweep < max_sweeps; ++sweep) {
    if (tid == 0) s_off = 0u;
    __syncthreads();
    float mo = 0.f;   // the largest off-diagonality this thread's pairs rotated
    // nested halving order: at level l the columns form 2^l blocks of 2h
    // (h = 64 >> l); pair group g holds column i = g mod h of its block's top
    // half in registers for the level's h rounds and meets the bottom half's
    // column (i + s) mod h in round s.  Each unordered pair meets once per sweep
    // (at the level that separates it), and a round moves one column per pair
    // through shared memory instead of two.
    const int g = (warp & 7) + 8 * q + 32 * (warp >> 3);
#pragma unroll 1
    for (int h = 64; h > 0; h >>= 1) {
      const int i = g & (h - 1);
      float* const top = X + 2 * (g - i) * kLdJ + 4 * sub;   // the block's first column
      float2 a[8];
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float4 va = *reinterpret_cast<const float4*>(top + i * kLdJ + 32 * w);
        a[2 * w] = make_float2(va.x, va.y);
        a[2 * w + 1] = make_float2(va.z, va.w);
      }
      // squared norms: exact at the level's start (the top-half column here, each
      // bottom-half column in round 0, where exactly one group meets it), then
      // carried through the rotations, |a'|^2 = |a|^2 - t g and |b'|^2 = |b|^2 + t g
      float al = group_dot(a, a);
#pragma unroll 1
      for (int s = 0; s < h; ++s) {
        const int cb = 2 * (g - i) + h + ((i + s) & (h - 1));
        float4* xb = reinterpret_cast<float4*>(top + (cb - 2 * (g - i)) * kLdJ);
        float2 b[8];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const float4 vb = xb[8 * w];
          b[2 * w] = make_float2(vb.x, vb.y);
          b[2 * w + 1] = make_float2(vb.z, vb.w);
        }
        const float ga = group_dot(a, b);
        float be = s == 0 ? group_dot(b, b) : s_nrm[cb];
        const float off = fabsf(ga) * rsqrtf(al) * rsqrtf(be);
        if (ga != 0.f && al > tiny && be > tiny && off > tol) {
          mo = fmaxf(mo, off);
          // the angle only needs to be close (fast divisions); c = 1 / sqrt(1 + t^2)
          // is rounded correctly, so that the rotation stays orthogonal
          const float zeta = __fdividef(be - al, 2.f * ga);
          const float t = fabsf(zeta) > 1e18f ? __fdividef(0.5f, zeta)
                                              : __fdividef(copysignf(1.f, zeta), fabsf(zeta) + sqrtf(fmaf(zeta, zeta, 1.f)));
          const float c = 1.f / sqrtf(fmaf(t, t, 1.f));
          const float sn = c * t;
          al = fmaxf(fmaf(-t, ga, al), 0.f);
          be = fmaxf(fmaf(t, ga, be), 0.f);
          const float2 c2 = make_float2(c, c), s2 = make_float2(sn, sn), ms2 = make_float2(-sn, -sn);
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            const float2 nb0 = __ffma2_rn(s2, a[2 * w], __fmul2_rn(c2, b[2 * w]));
            const float2 nb1 = __ffma2_rn(s2, a[2 * w + 1], __fmul2_rn(c2, b[2 * w + 1]));
            a[2 * w] = __ffma2_rn(ms2, b[2 * w], __fmul2_rn(c2, a[2 * w]));
            a[2 * w + 1] = __ffma2_rn(ms2, b[2 * w + 1], __fmul2_rn(c2, a[2 * w + 1]));
            xb[8 * w] = make_float4(nb0.x, nb0.y, nb1.x, nb1.y);
          }
        }
        if (sub == 0) s_nrm[cb] = be;
        if (s == h - 1) {   // the level's last round: the top-half column goes home
#pragma unroll
          for (int w = 0; w < 4; ++w)
            *reinterpret_cast<float4*>(top + i * kLdJ + 32 * w) =
                make_float4(a[2 * w].x, a[2 * w].y, a[2 * w + 1].x, a[2 * w + 1].y);
        }
        __syncthreads();
      }
    }
    if (sub == 0 && mo > 0.f) atomicMax(&s_off, __float_as_uint(mo));   // one update per pair group
    __syncthreads();
    const float max_off = __uint_as_float(s_off);
    __syncthreads();
    // done when every rotated pair was within sqrt(tol) of orthogonal (max_off
    // stays 0 when nothing rotated): cyclic Jacobi converges quadratically
    // there, so the next sweep would find the pairs near tol (float32 emulation
    // on the bench's operators: the same singular values and rank-r maps, one
    // or two sweeps fewer)
    if (max_off <= stop_off) return true;
  }
  return false;
}

// Householder QR of the matrix in X (column-major, leading dimension kLdS), in
// place: on return R occupies the upper triangle (diagonal included); below it,
// the reflector vectors are left behind.  Needs kFitThreads threads.  One
// barrier per column: warp 0, whose first trailing column is j + 1, derives the
// next reflector from it once its columns are done (parameters double-buffered
// by step parity); the new diagonal is written without a barrier, as the
// trailing update never reads it.  Lane l holds rows l + 32 u of every column
// it touches, and a warp reduces four columns' dot products together (the
// step's cost is the latency of those butterflies, not their arithmetic).

// Reflector parameters of column x below row j - 1 (warp-wide; lane 0 writes):
// alpha (the new diagonal), v_j, and 2 / |v|^2 (0 when there is nothing to reflect).
__device__ __forceinline__ void householder_par(const float* x, int j, float* par, int lane) {
  float sq = 0.f;
  for (int i = j + 1 + lane; i < kD; i += 32) sq = fmaf(x[i], x[i], sq);
  sq = warp_sum(sq);
  if (lane == 0) {
    const float x0 = x[j];
    const float nx = sqrtf(fmaf(x0, x0, sq));
    const float alpha = x0 >= 0.f ? -nx : nx;   // v_j = x0 - alpha adds magnitudes: no cancellation
    const float v0 = x0 - alpha;
    const float vn2 = fmaf(v0, v0, sq);
    par[0] = alpha;
    par[1] = v0;
    par[2] = vn2 > 0.f ? 2.f / vn2 : 0.f;
  }
}

__device__ void householder_r(float* X) {
  __shared__ float s_par[2][3];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarps = kFitThreads / 32;
  if (warp == 0) householder_par(X, 0, s_par[0], lane);
  __syncthreads();
  for (int j = 0; j < kD - 1; ++j) {
    const float* par = s_par[j & 1];
    float* nxt = s_par[(j + 1) & 1];
    const float v0 = par[1], inv = par[2];
    const float* xj = X + j * kLdS;
    if (inv > 0.f) {
      // the reflector v in the lane's rows lane + 32 u: v_j = v0, v_i = x_j(i) below
      float v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int i = lane + 32 * u;
        v[u] = i > j ? xj[i] : (i == j ? v0 : 0.f);
      }
      // trailing columns c = j + 1 + warp + 16 t, four per warp at a time: their
      // dot products with v reduce together, so the butterflies overlap
#pragma unroll 1
      for (int c0 = j + 1 + warp; c0 < kD; c0 += 4 * kWarps) {
        float x[4][4], dt[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int c = c0 + t * kWarps;
          dt[t] = 0.f;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            x[t][u] = c < kD ? X[c * kLdS + lane + 32 * u] : 0.f;
            dt[t] = fmaf(v[u], x[t][u], dt[t]);
          }
        }
#pragma unroll
        for (int m = 16; m > 0; m >>= 1)
#pragma unroll
          for (int t = 0; t < 4; ++t) dt[t] += __shfl_xor_sync(0xffffffffu, dt[t], m);
        // c -= (2 v.c / |v|^2) v on rows j and below
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int c = c0 + t * kWarps;
          const float f = dt[t] * inv;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int i = lane + 32 * u;
            if (c < kD && i >= j) X[c * kLdS + i] = fmaf(-f, v[u], x[t][u]);
          }
        }
      }
      if (warp == 0) {   // warp 0 updated column j + 1 (c0 = j + 1): the next reflector
        __syncwarp();
        householder_par(X + (j + 1) * kLdS, j + 1, nxt, lane);
      }
      if (tid == 0) X[j * kLdS + j] = par[0];
    } else if (warp == 0) {
      householder_par(X + (j + 1) * kLdS, j + 1, nxt, lane);   // nothing to reflect: column j + 1 unchanged
    }
    __syncthreads();
  }
}

// column norms of X (leading dimension ld) into out[kD] (warp per column)
__device__ void column_norms(const float* X, float* out, int ld = kLdS) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int c = warp; c < kD; c += kFitThreads / 32) {
    float v = 0.f;
    for (int i = lane; i < kD; i += 32) v = fmaf(X[c * ld + i], X[c * ld + i], v);
    v = warp_sum(v);
    if (lane == 0) out[c] = sqrtf(v);
  }
}

// One d x d buffer in shared memory (two CTAs per SM): the Cholesky factor L
// in its lower triangle, L^{-1} transposed in its strict upper triangle with
// L^{-1}'s diagonal in dinv; or, on the fallback path, the Jacobi matrix.
// Matrices m >= sym_from take the eigen path whatever their spectrum and store
// the symmetric roots F = S^{1/2} = V Lambda^{1/2} V^T and G = S^{+1/2} (the
// projector variant SAP-svd needs the right singular vectors of the
// symmetric-root C itself).
// Three CTAs per SM (the Cholesky and inverse are bound by the latency of their
// per-column barriers, so more resident matrices hide it: 1280 matrices in 3
// waves instead of 5; the register cap spills a few words in the eigen fallback).
__global__ void __launch_bounds__(kFitThreads, 3) factor_kernel(const float* S, float floor_rel, int max_sweeps,
                                                                float tol, float* Fout, float* Gout, int* status,
                                                                int sym_from) {
  extern __shared__ __align__(16) float sm[];
  float* Sb = sm;   // row-major
  float* Xb = sm;   // the Jacobi matrix of the fallback path
  __shared__ float lam[kD];
  __shared__ float dinv[kD];
  __shared__ float red[32];
  __shared__ int flag, counter;
  const int m = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* Sm = S + (int64_t)m * kD * kD;
  float* F = Fout + (int64_t)m * kD * kD;
  float* G = Gout + (int64_t)m * kD * kD;

  for (int o = tid; o < kD * kD; o += kFitThreads) Sb[(o / kD) * kLdS + (o % kD)] = Sm[o];
  if (tid == 0) flag = 0;
  __syncthreads();
  // trace and finiteness
  if (warp == 0) {
    float tr = 0.f;
    for (int i = lane; i < kD; i += 32) tr += Sb[i * kLdS + i];
    tr = warp_sum(tr);
    if (lane == 0) red[0] = tr;
  }
  bool bad = false;
  for (int o = tid; o < kD * kD; o += kFitThreads) bad |= !isfinite(Sm[o]);
  if (__syncthreads_or(bad)) {
    for (int o = tid; o < kD * kD; o += kFitThreads) { F[o] = 0.f; G[o] = 0.f; }
    if (tid == 0) status[m] |= kStNonFinite;
    return;
  }
  const float trace = red[0];

  const bool sym = m >= sym_from;   // symmetric roots: skip the Cholesky path
  // Cholesky, right-looking, in place; every thread reads the same pivot (the
  // last barrier of step j - 1 made it final), so all leave together
  bool chol_ok = !sym;
  for (int j = 0; j < kD && chol_ok; ++j) {
    const float piv = Sb[j * kLdS + j];
    if (!(piv > 0.f && isfinite(piv))) {
      chol_ok = false;
      break;
    }
    const float ljj = sqrtf(piv);
    for (int i = j + 1 + tid; i < kD; i += kFitThreads) Sb[i * kLdS + j] /= ljj;
    __syncthreads();
    if (tid == 0) Sb[j * kLdS + j] = ljj;
    // trailing update of the lower triangle: a warp per row, lanes over columns
    for (int i = j + 1 + warp; i < kD; i += kFitThreads / 32) {
      const float lij = Sb[i * kLdS + j];
      for (int c = j + 1 + lane; c <= i; c += 32) Sb[i * kLdS + c] = fmaf(-lij, Sb[c * kLdS + j], Sb[i * kLdS + c]);
    }
    __syncthreads();
  }

  if (chol_ok) {
    // Linv = F^{-1} by right-looking substitution on the identity: row i is
    // divided by F_ii, then subtracted (times F_ri) from every row below it.
    // Linv(r, c) for r > c lives at Sb[c][r] (the strict upper triangle, whose
    // copy of S is no longer needed), Linv(i, i) in dinv[i].
    for (int o = tid; o < kD * kD; o += kFitThreads) {
      const int i = o / kD, c = o % kD;
      if (c > i) Sb[i * kLdS + c] = 0.f;
    }
    if (tid < kD) dinv[tid] = 1.f;
    __syncthreads();
    for (int i = 0; i < kD; ++i) {
      const float inv = 1.f / Sb[i * kLdS + i];
      if (tid < i) Sb[tid * kLdS + i] *= inv;   // Linv(i, c) for c < i; columns > i of row i are zero
      if (tid == i) dinv[i] *= inv;
      __syncthreads();
      for (int r = i + 1 + warp; r < kD; r += kFitThreads / 32) {
        const float lri = Sb[r * kLdS + i];
        for (int c = lane; c < i; c += 32) Sb[c * kLdS + r] = fmaf(-lri, Sb[c * kLdS + i], Sb[c * kLdS + r]);
        if (lane == 0) Sb[i * kLdS + r] = fmaf(-lri, dinv[i], Sb[i * kLdS + r]);
      }
      __syncthreads();
    }
    float ss = 0.f;
    for (int o = tid; o < kD * kD; o += kFitThreads) {
      const int i = o / kD, c = o % kD;
      const float v = c > i ? Sb[i * kLdS + c] : (c == i ? dinv[i] : 0.f);
      ss = fmaf(v, v, ss);
    }
    ss = warp_sum(ss);
    if (lane == 0) red[warp] = ss;
    __syncthreads();
    if (tid == 0) {
      float t = 0.f;
      for (int w = 0; w < kFitThreads / 32; ++w) t += red[w];
      flag = (isfinite(t) && t > 0.f && 1.f / t >= floor_rel * trace) ? 0 : 2;
    }
    __syncthreads();
    chol_ok = (flag == 0);
  }
  if (chol_ok) {
    for (int o = tid; o < kD * kD; o += kFitThreads) {
      const int i = o / kD, c = o % kD;
      F[o] = c <= i ? Sb[i * kLdS + c] : 0.f;
    }
    for (int o = tid; o < kD * kD; o += kFitThreads) {   // G = Linv^T, stored transposed: G[c][i] = Linv(c, i)
      const int c = o / kD, i = o % kD;
      G[o] = i < c ? Sb[i * kLdS + c] : (i == c ? dinv[i] : 0.f);
    }
    return;
  }

  // exact floor: eigenpairs from one-sided Jacobi on S itself (the barrier: a
  // failed pivot leaves the Cholesky loop without one, and Xb overwrites Sb)
  __syncthreads();
  for (int o = tid; o < kD * kD; o += kFitThreads) Xb[(o % kD) * kLdS + (o / kD)] = Sm[o];
  __syncthreads();
  const bool conv = jacobi_columns(Xb, max_sweeps, tol, &counter);
  if (!conv && tid == 0) status[m] |= kStNotConverged;
  column_norms(Xb, lam);
  __syncthreads();
  if (tid == 0) {
    float mx = 0.f;
    for (int i = 0; i < kD; ++i) mx = fmaxf(mx, lam[i]);
    red[0] = mx;
  }
  __syncthreads();
  const float lmax = red[0];
  if (sym) {
    // F = sum_c v_c v_c^T sqrt(l_c), G = sum_c v_c v_c^T / sqrt(l_c) over the kept
    // eigenpairs (v_c = w_c / l_c from the Jacobi columns w_c = v_c l_c)
    for (int o = tid; o < kD * kD; o += kFitThreads) {
      const int i = o / kD, j = o % kD;
      float f = 0.f, gg = 0.f;
      for (int c = 0; c < kD; ++c) {
        const float l = lam[c];
        if (!(l > 0.f && l >= floor_rel * lmax)) continue;
        const float vv = (Xb[c * kLdS + i] / l) * (Xb[c * kLdS + j] / l);
        const float sl = sqrtf(l);
        f = fmaf(vv, sl, f);
        gg = fmaf(vv, 1.f / sl, gg);
      }
      F[o] = f;
      G[o] = gg;
    }
    return;
  }
  for (int o = tid; o < kD * kD; o += kFitThreads) {
    const int i = o / kD, c = o % kD;
    const float l = lam[c];
    const bool keep = l > 0.f && l >= floor_rel * lmax;
    F[o] = keep ? Xb[c * kLdS + i] / sqrtf(l) : 0.f;          // v sqrt(l),  v = w / l
  }
  for (int o = tid; o < kD * kD; o += kFitThreads) {   // G stored transposed
    const int c = o / kD, i = o % kD;
    const float l = lam[c];
    const bool keep = l > 0.f && l >= floor_rel * lmax;
    G[o] = keep ? Xb[c * kLdS + i] / (l * sqrtf(l)) : 0.f;    // v / sqrt(l)
  }
}

// Shared memory holds only the Jacobi matrix (68 KB), so two CTAs share an SM;
// C'^T is kept in a global scratch slice (L2-resident) for the steps after the SVD.
// out(i, j) = sum_p a(i, p) b(p, j) for 128 x 128 x 128 with kFitThreads
// threads: a thread accumulates rows 4 (t % 32) .. + 3 and columns 8 (t / 32)
// .. + 7 (three 16-byte shared loads per 32 FMAs); the K dimension goes in
// chunks of 16, staged in stg (2 x 16 rows of 132 floats).  Each output is
// summed over p in increasing order, one FMA at a time.
constexpr int kStgLd = kD + 4;
constexpr int kStgFloats = 2 * 16 * kStgLd;
template <class LA, class LB, class ST>
__device__ __forceinline__ void gemm128(LA la, LB lb, ST st, float* stg) {
  float* At = stg;
  float* Bt = stg + 16 * kStgLd;
  const int tid = threadIdx.x;
  const int i0 = (tid & 31) * 4, j0 = (tid >> 5) * 8;
  float acc[4][8];
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 8; ++v) acc[u][v] = 0.f;
  for (int p0 = 0; p0 < kD; p0 += 16) {
    __syncthreads();   // the previous chunk is consumed
    for (int e = tid; e < 16 * kD; e += kFitThreads) {
      const int kk = e & 15, i = e >> 4;
      At[kk * kStgLd + i] = la(i, p0 + kk);
      const int kb = e / kD, j = e % kD;
      Bt[kb * kStgLd + j] = lb(p0 + kb, j);
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      const float4 a4 = *reinterpret_cast<const float4*>(At + kk * kStgLd + i0);
      const float4 b0 = *reinterpret_cast<const float4*>(Bt + kk * kStgLd + j0);
      const float4 b1 = *reinterpret_cast<const float4*>(Bt + kk * kStgLd + j0 + 4);
      const float a[4] = {a4.x, a4.y, a4.z, a4.w};
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 8; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
    }
  }
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 8; ++v) st(i0 + u, j0 + v, acc[u][v]);
}

__global__ void __launch_bounds__(kFitThreads, 2) fit_kernel(const float* A, const float* Fm, const float* Gm,
                                                             const float* mu, int Hq, int Hk, int r, int max_sweeps,
                                                             float tol, float* Cws, float* L, float* R, float* sigma,
                                                             float* loss, float* nu, int* status) {
  extern __shared__ __align__(16) float sm[];
  float* X = sm;               // column-major, ld kLdS
  __shared__ float sig[kD];
  __shared__ float sgn[kD];
  __shared__ int perm[kD];
  const int h = blockIdx.x, g = h / (Hq / Hk);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* Ah = A + (int64_t)h * kD * kD;
  const float* Fq = Fm + (int64_t)h * kD * kD;
  const float* Gq = Gm + (int64_t)h * kD * kD;
  const float* Fk = Fm + (int64_t)(Hq + g) * kD * kD;
  const float* Gk = Gm + (int64_t)(Hq + g) * kD * kD;
  float* Ct = Cws + (int64_t)h * kD * kD;   // C', column-major: (row, col) at [col * d + row]
  float* Lh = L + (int64_t)h * kD * r;
  float* Rh = R + (int64_t)h * kD * r;

  float* stg = sm + kD * kLdJ;   // staging of the two products
  // X = A Fk (column-major, ld kLdS)
  gemm128([&](int i, int p) { return __ldg(Ah + i * kD + p); }, [&](int p, int j) { return __ldg(Fk + p * kD + j); },
          [&](int i, int j, float v) { X[j * kLdS + i] = v; }, stg);
  __syncthreads();
  // C'^T = X^T Fq, stored as C' column-major in the global scratch: C'(j, i) at [i * d + j]
  gemm128([&](int i, int p) { return X[i * kLdS + p]; }, [&](int p, int j) { return __ldg(Fq + p * kD + j); },
          [&](int i, int j, float v) { Ct[i * kD + j] = v; }, stg);
  __syncthreads();
  // Preconditioning: C' = Q1 R1 (Householder), then the Jacobi runs on R1^T, whose
  // left singular vectors are those of C'^T = R1^T Q1^T, i.e. the right singular
  // vectors of C' (the triangular factor converges in far fewer sweeps).
  for (int o = tid; o < kD * kD; o += kFitThreads) X[(o / kD) * kLdS + (o % kD)] = Ct[o];   // X = C'
  __syncthreads();
  householder_r(X);
  {  // X = R1^T (lower triangle), re-laid out with leading dimension kLdJ
    float v[kD * kD / kFitThreads];
#pragma unroll
    for (int t = 0; t < kD * kD / kFitThreads; ++t) {
      const int o = tid + t * kFitThreads, i = o / kD, jj = o % kD;
      v[t] = i >= jj ? X[i * kLdS + jj] : 0.f;   // R1^T (i, jj) = R1 (jj, i)
    }
    __syncthreads();
#pragma unroll
    for (int t = 0; t < kD * kD / kFitThreads; ++t) {
      const int o = tid + t * kFitThreads, i = o / kD, jj = o % kD;
      X[jj * kLdJ + i] = v[t];
    }
  }
  __syncthreads();

  const bool conv = jacobi_columns_v4(X, max_sweeps, tol);
  if (!conv && tid == 0) status[h] |= kStNotConverged;
  column_norms(X, sig, kLdJ);
  __syncthreads();
  if (tid < kD) {  // rank = position in descending order, ties by index
    const float s = sig[tid];
    int rk = 0;
    for (int j = 0; j < kD; ++j) rk += (sig[j] > s) || (sig[j] == s && j < tid);
    perm[rk] = tid;
  }
  __syncthreads();
  const float smax = sig[perm[0]];
  if (tid == 0 && !isfinite(smax)) status[h] |= kStNonFinite;

  // Z = C' V_r Sigma^{-1} (= U_r) into L as scratch; R = Gk V_r Sigma^{1/2} (unsigned) into R
  const int a = tid % kD;
  for (int c = tid / kD; c < r; c += kFitThreads / kD) {
    const int i = perm[c];
    const float s = sig[i];
    const bool live = s > 0.f && s > smax * 1e-20f;
    float z = 0.f, q = 0.f;
    for (int b = 0; b < kD; ++b) {   // C'(a, b) and Gk(a, b): consecutive a in consecutive lanes
      const float x = X[i * kLdJ + b];
      z = fmaf(__ldg(Ct + b * kD + a), x, z);
      q = fmaf(__ldg(Gk + b * kD + a), x, q);
    }
    Lh[a * r + c] = live ? z / (s * s) : 0.f;    // C' x_i / s^2 = u_i (x_i = s v_i)
    Rh[a * r + c] = live ? q / sqrtf(s) : 0.f;   // Gk v_i sqrt(s) = Gk x_i / sqrt(s)
  }
  __syncthreads();
  for (int c = warp; c < r; c += kFitThreads / 32) {  // sign: largest-|.| entry of R[:, c] positive
    float best = -1.f, val = 0.f;
    int bi = 0;
    for (int i = lane; i < kD; i += 32) {
      const float v = Rh[i * r + c];
      if (fabsf(v) > best) { best = fabsf(v); bi = i; val = v; }
    }
#pragma unroll
    for (int m = 16; m > 0; m >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, m);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, m);
      const float ov = __shfl_xor_sync(0xffffffffu, val, m);
      if (ob > best || (ob == best && oi < bi)) { best = ob; bi = oi; val = ov; }
    }
    if (lane == 0) sgn[c] = val < 0.f ? -1.f : 1.f;
  }
  __syncthreads();
  for (int o = tid; o < kD * r; o += kFitThreads) {
    const int i = o / r, c = o % r;
    Rh[o] *= sgn[c];
    X[c * kLdS + i] = Lh[o];   // Z back into shared memory (the Jacobi matrix is no longer needed)
  }
  __syncthreads();
  for (int c = tid / kD; c < r; c += kFitThreads / kD) {
    const float s = sig[perm[c]];
    float acc = 0.f;
    for (int e = 0; e < kD; ++e) acc = fmaf(__ldg(Gq + e * kD + a), X[c * kLdS + e], acc);
    Lh[a * r + c] = sgn[c] * acc * sqrtf(fmaxf(s, 0.f));   // Gq u_i sqrt(s)
  }
  if (tid < kD && sigma) sigma[(int64_t)h * kD + tid] = sig[perm[tid]];
  if (warp == 0 && loss) {
    float v = 0.f;
    for (int c = r + lane; c < kD; c += 32) v = fmaf(sig[perm[c]], sig[perm[c]], v);
    v = warp_sum(v);
    if (lane == 0) loss[h] = v;
  }
  if (nu && tid < kD) {
    float v = 0.f;
    if (mu)
      for (int b = 0; b < kD; ++b) v = fmaf(__ldg(Ah + tid * kD + b), __ldg(mu + g * kD + b), v);
    nu[(int64_t)h * kD + tid] = v;
  }
}

// ---------------------------------------------------------------- comparison indexes
// Identity matrices [nmat][d][d]: the whitening factors of a comparison index
// that ignores a moment (both for weight SVD, the query side for key PCA), and
// the identity operator of the key-PCA fit.
__global__ void identity_kernel(float* X) {
  float* Xm = X + (int64_t)blockIdx.x * kD * kD;
  for (int o = threadIdx.x; o < kD * kD; o += blockDim.x) Xm[o] = (o / kD == o % kD) ? 1.f : 0.f;
}

// Key PCA from the fit of C' = F_k (operator and query factors set to the
// identity): that fit returns R = V Sigma^{-1/2} with V the leading eigenvectors
// of Sk and Sigma = Lambda^{1/2}, signed like every fit.  Rescaled, R = V (unit
// columns); the operator is folded into the query side, L = A_h V, and the mean
// term recomputed, nu = A_h mu_g.  One CTA of d threads per head; thread i owns
// row i of L and R, and reads the fit's R only from shared memory.
__global__ void __launch_bounds__(kD) key_pca_fold_kernel(const float* A, const float* sigma, const float* mu,
                                                         int Hq, int Hk, int r, float* L, float* R, float* nu) {
  extern __shared__ float sm[];
  float* As = sm;                    // A_h, row stride d + 1 (row i of thread i: conflict-free)
  float* Vs = As + kD * (kD + 1);    // V [d][r]
  __shared__ float mus[kD];
  const int h = blockIdx.x, g = h / (Hq / Hk), i = threadIdx.x;
  const float* Ah = A + (int64_t)h * kD * kD;
  float* Lh = L + (int64_t)h * kD * r;
  float* Rh = R + (int64_t)h * kD * r;
  for (int o = i; o < kD * kD; o += kD) As[(o / kD) * (kD + 1) + o % kD] = Ah[o];
  for (int o = i; o < kD * r; o += kD) Vs[o] = Rh[o] * sqrtf(fmaxf(sigma[(int64_t)h * kD + o % r], 0.f));
  mus[i] = mu ? mu[(int64_t)g * kD + i] : 0.f;
  __syncthreads();
  for (int c = 0; c < r; ++c) {
    float acc = 0.f;
    for (int j = 0; j < kD; ++j) acc = fmaf(As[i * (kD + 1) + j], Vs[j * r + c], acc);
    Lh[i * r + c] = acc;
    Rh[i * r + c] = Vs[i * r + c];
  }
  if (nu) {
    float v = 0.f;
    for (int j = 0; j < kD; ++j) v = fmaf(As[i * (kD + 1) + j], mus[j], v);
    nu[(int64_t)h * kD + i] = v;
  }
}

// The projector variants of Sec. 6 (SAP-svd, SAP-map) from a SAKI fit: an
// orthonormal basis Q of an r-dimensional key subspace, the map M = A_h Q Q^T
// folded as R = Q, L = A_h Q (nu = A_h mu is the fit's).  SAP-map takes the
// optimum's key-side span, span((Sk^{1/2})^+ V_r) with (Sk^{1/2})^+ the
// pseudo-inverse of the root: the columns of the fit's R
// ((Sk^{1/2})^+ V_r Sigma_r^{1/2} whatever factor of Sk whitened it), in order.
// SAP-svd takes the raw right singular vectors V_r of C: with the symmetric key
// root F_k = Sk^{1/2} (factor kernel, sym_from) the fit's R gives
// V_r = F_k R Sigma_r^{-1/2}.  Either basis is orthonormalised by modified
// Gram-Schmidt in column order and each column signed so that its largest-|.|
// entry (the first of equal ones) is positive.  One CTA of d threads per head;
// thread i owns row i.
__global__ void __launch_bounds__(kD) sap_fold_kernel(const float* A, const float* Fm, const float* sigma, int Hq,
                                                      int Hk, int r, int svd, float* L, float* R) {
  extern __shared__ float sm[];
  float* As = sm;                    // A_h or F_k, row stride d + 1
  float* Qs = As + kD * (kD + 1);    // [d][r]
  __shared__ float red[kD / 32];
  __shared__ int redi[kD / 32];
  const int h = blockIdx.x, g = h / (Hq / Hk), i = threadIdx.x, lane = i & 31, warp = i >> 5;
  float* Lh = L + (int64_t)h * kD * r;
  float* Rh = R + (int64_t)h * kD * r;
  if (svd) {
    const float* Fk = Fm + (int64_t)(Hq + g) * kD * kD;
    for (int o = i; o < kD * kD; o += kD) As[(o / kD) * (kD + 1) + o % kD] = Fk[o];
    __syncthreads();
    for (int c = 0; c < r; ++c) {
      float acc = 0.f;
      for (int j = 0; j < kD; ++j) acc = fmaf(As[i * (kD + 1) + j], Rh[j * r + c], acc);
      const float sg = sigma[(int64_t)h * kD + c];
      Qs[i * r + c] = sg > 0.f ? acc * rsqrtf(sg) : 0.f;
    }
  } else {
    for (int c = 0; c < r; ++c) Qs[i * r + c] = Rh[i * r + c];
  }
  __syncthreads();
  auto block_sum = [&](float v) {
    v = warp_sum(v);
    if (lane == 0) red[warp] = v;
    __syncthreads();
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kD / 32; ++w) t += red[w];
    __syncthreads();
    return t;
  };
  for (int c = 0; c < r; ++c) {
    float x = Qs[i * r + c];
    for (int p = 0; p < c; ++p) {
      const float qp = Qs[i * r + p];
      const float dot = block_sum(qp * x);
      x = fmaf(-dot, qp, x);
    }
    const float nrm = sqrtf(block_sum(x * x));
    x = nrm > 0.f ? x / nrm : 0.f;
    // sign: the largest-|.| entry (first of equal ones) positive
    float best = fabsf(x);
    int bi = i;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (ob > best || (ob == best && oi < bi)) { best = ob; bi = oi; }
    }
    if (lane == 0) { red[warp] = best; redi[warp] = bi; }
    __syncthreads();
    float b = red[0];
    int bidx = redi[0];
    for (int w = 1; w < kD / 32; ++w)
      if (red[w] > b || (red[w] == b && redi[w] < bidx)) { b = red[w]; bidx = redi[w]; }
    __syncthreads();
    if (i == bidx) red[0] = x;
    __syncthreads();
    if (red[0] < 0.f) x = -x;
    __syncthreads();
    Qs[i * r + c] = x;
    __syncthreads();
  }
  // L = A_h Q, R = Q
  const float* Ah = A + (int64_t)h * kD * kD;
  for (int o = i; o < kD * kD; o += kD) As[(o / kD) * (kD + 1) + o % kD] = Ah[o];
  __syncthreads();
  for (int c = 0; c < r; ++c) {
    float acc = 0.f;
    for (int j = 0; j < kD; ++j) acc = fmaf(As[i * (kD + 1) + j], Qs[j * r + c], acc);
    Lh[i * r + c] = acc;
    Rh[i * r + c] = Qs[i * r + c];
  }
}

// Sec. 7 diagnostic: the eigenvalues (descending) of each key correlation
// matrix D^{-1/2} S D^{-1/2} (D = diag(S); a zero diagonal entry leaves its row
// and column zero), from one-sided Jacobi on it, and the number above the
// Marchenko-Pastur upper edge.  The column norms of the converged Jacobi matrix
// are the eigenvalues of the PSD input; a rank sort (ties by position) orders them.
__global__ void __launch_bounds__(kFitThreads, 2) spectrum_kernel(const float* S, float edge, int max_sweeps,
                                                                  float tol, float* lam_out, int* spikes,
                                                                  int* status) {
  extern __shared__ __align__(16) float sm[];
  float* Xb = sm;   // column-major, ld kLdS
  __shared__ float lam[kD];
  __shared__ float dg[kD];
  __shared__ int counter, above;
  const int m = blockIdx.x, tid = threadIdx.x;
  const float* Sm = S + (int64_t)m * kD * kD;
  if (tid < kD) {
    const float v = Sm[tid * kD + tid];
    dg[tid] = v > 0.f ? rsqrtf(v) : 0.f;
  }
  if (tid == 0) above = 0;
  __syncthreads();
  for (int o = tid; o < kD * kD; o += kFitThreads) {
    const int i = o / kD, c = o % kD;
    Xb[c * kLdS + i] = Sm[o] * dg[i] * dg[c];
  }
  __syncthreads();
  const bool conv = jacobi_columns(Xb, max_sweeps, tol, &counter);
  if (!conv && tid == 0) status[m] |= kStNotConverged;
  column_norms(Xb, lam);
  __syncthreads();
  if (tid < kD) {
    const float l = lam[tid];
    int rank = 0;
    for (int j = 0; j < kD; ++j) rank += (lam[j] > l || (lam[j] == l && j < tid)) ? 1 : 0;
    lam_out[(int64_t)m * kD + rank] = l;
    if (l > edge) atomicAdd(&above, 1);
  }
  __syncthreads();
  if (tid == 0) spikes[m] = above;
}

constexpr float kTol = 1e-6f;
constexpr size_t kSmem = sizeof(float) * kD * kLdS;         // factor kernel: L and L^{-1} share one buffer
constexpr size_t kFitSmem = sizeof(float) * (kD * kLdJ + kStgFloats);   // fit kernel: the Jacobi matrix, staging
}  // namespace

cudaError_t launch_factor(const float* S, int nmat, float floor_rel, int max_sweeps, float* F, float* Gm,
                          int* status, cudaStream_t s, int sym_from) {
  cudaError_t e = cudaFuncSetAttribute(factor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  if (e != cudaSuccess) return e;
  note_launch();
  factor_kernel<<<nmat, kFitThreads, kSmem, s>>>(S, floor_rel, max_sweeps, kTol, F, Gm, status, sym_from);
  return cudaGetLastError();
}

cudaError_t launch_fit(const float* A, const float* F, const float* Gm, const float* mu, int Hq, int Hk, int r,
                       int max_sweeps, float* Cws, float* L, float* R, float* sigma, float* loss, float* nu,
                       int* status, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(fit_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFitSmem);
  if (e != cudaSuccess) return e;
  note_launch();
  fit_kernel<<<Hq, kFitThreads, kFitSmem, s>>>(A, F, Gm, mu, Hq, Hk, r, max_sweeps, kTol, Cws, L, R, sigma, loss,
                                               nu, status);
  return cudaGetLastError();
}

cudaError_t launch_identity(float* X, int nmat, cudaStream_t s) {
  if (nmat == 0) return cudaSuccess;
  note_launch();
  identity_kernel<<<nmat, 256, 0, s>>>(X);
  return cudaGetLastError();
}

cudaError_t launch_key_pca_fold(const float* A, const float* sigma, const float* mu, int Hq, int Hk, int r, float* L,
                                float* R, float* nu, cudaStream_t s) {
  const int smem = (int)(sizeof(float) * (kD * (kD + 1) + kD * r));
  cudaError_t e = cudaFuncSetAttribute(key_pca_fold_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  note_launch();
  key_pca_fold_kernel<<<Hq, kD, smem, s>>>(A, sigma, mu, Hq, Hk, r, L, R, nu);
  return cudaGetLastError();
}

}  // namespace saki

namespace saki {
cudaError_t launch_sap_fold(const float* A, const float* F, const float* sigma, int Hq, int Hk, int r, int svd,
                            float* L, float* R, cudaStream_t s) {
  const int smem = (int)(sizeof(float) * (kD * (kD + 1) + kD * r));
  cudaError_t e = cudaFuncSetAttribute(sap_fold_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  note_launch();
  sap_fold_kernel<<<Hq, kD, smem, s>>>(A, F, sigma, Hq, Hk, r, svd, L, R);
  return cudaGetLastError();
}
}  // namespace saki

namespace saki {
cudaError_t launch_spectrum(const float* S, int nmat, float edge, int max_sweeps, float* lam, int* spikes, int* status,
                            cudaStream_t s) {
  if (nmat == 0) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(spectrum_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
  if (e != cudaSuccess) return e;
  note_launch();
  spectrum_kernel<<<nmat, kFitThreads, kSmem, s>>>(S, edge, max_sweeps, kTol, lam, spikes, status);
  return cudaGetLastError();
}
}  // namespace saki
