// Sec. 7 estimation diagnostics and App. C's measured score-MSE reduction:
//   fourth_moment_kernel + shrink_kernel: Ledoit-Wolf shrinkage of the
//     calibration moments (Ledoit & Wolf 2004), S* = (1 - rho) S + rho m I with
//     m = tr(S) / d, rho = min(b2, d2) / d2, d2 = ||S - m I||_F^2 and
//     b2 = (1/n^2) sum_t ||x_t x_t^T - S||_F^2 = (sum_t ||x_t||^4 / n - ||S||_F^2) / n
//     (the cross term sums to 2 n ||S||_F^2 because S = (1/n) sum_t x_t x_t^T);
//   score_mse_kernel: per query head, over every key_stride-th visible key of
//     each query, the sums of s^2 and (s - s_hat)^2 with s = q^T A k and
//     s_hat = (L^T q)^T c + q^T nu, accumulated in fp64.
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {

// sum_t ||x_t - mu||^4 of each calibration matrix (queries first, never
// centered; keys centered on mu when it is given) added into acc[m] (fp64,
// zeroed by the caller).  One warp per row, four dimensions per lane.
template <typename Tin>
__global__ void __launch_bounds__(256) fourth_moment_kernel(const Tin* Xq, const Tin* Xk, int64_t n, int Hq,
                                                            const float* mu, double* acc) {
  const int m = blockIdx.y;
  const Tin* X = m < Hq ? Xq + (int64_t)m * n * kD : Xk + (int64_t)(m - Hq) * n * kD;
  const float* mum = (m >= Hq && mu) ? mu + (int64_t)(m - Hq) * kD : nullptr;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float mloc[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) mloc[c] = mum ? mum[lane * 4 + c] : 0.f;
  double local = 0.0;
  for (int64_t t = (int64_t)blockIdx.x * 8 + warp; t < n; t += (int64_t)gridDim.x * 8) {
    float s2 = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const float x = Vec<Tin>::load1(X + t * kD + lane * 4 + c) - mloc[c];
      s2 = fmaf(x, x, s2);
    }
    s2 = warp_sum(s2);
    local += (double)s2 * (double)s2;
  }
  if (lane == 0 && local != 0.0) atomicAdd(acc + m, local);
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Ledoit-Wolf shrinkage of each d x d moment matrix, in place; rho[m] if given.
__global__ void __launch_bounds__(256) shrink_kernel(float* S, const double* acc4, int64_t n, float* rho_out) {
  __shared__ double red[2][8];
  const int m = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float* Sm = S + (int64_t)m * kD * kD;
  double tr = 0.0, fro = 0.0;
  for (int o = tid; o < kD * kD; o += 256) {
    const double v = Sm[o];
    fro += v * v;
    if (o / kD == o % kD) tr += v;
  }
  tr = warp_sum_d(tr);
  fro = warp_sum_d(fro);
  if (lane == 0) { red[0][warp] = tr; red[1][warp] = fro; }
  __syncthreads();
  tr = fro = 0.0;
#pragma unroll
  for (int w = 0; w < 8; ++w) { tr += red[0][w]; fro += red[1][w]; }
  const double mid = tr / kD;
  const double d2 = fro - kD * mid * mid;                       // ||S - m I||_F^2
  const double b2bar = fmax((acc4[m] / (double)n - fro) / (double)n, 0.0);
  const double rho = d2 > 0.0 ? fmin(b2bar, d2) / d2 : 0.0;
  __syncthreads();
  for (int o = tid; o < kD * kD; o += 256) {
    const double v = (1.0 - rho) * Sm[o] + (o / kD == o % kD ? rho * mid : 0.0);
    Sm[o] = (float)v;
  }
  if (tid == 0 && rho_out) rho_out[m] = (float)rho;
}

// App. C: one CTA of d threads per (query, head).  qinfo[t] = (key base, visible keys).
template <typename Tin>
__global__ void __launch_bounds__(kD) score_mse_kernel(const Tin* Q, const float* A, const Tin* K, const float* L,
                                                       const Tin* codes, const float* nu, const int64_t* qinfo,
                                                       int64_t T, int64_t N, int Hq, int G, int r, int64_t stride,
                                                       double* out) {
  __shared__ float qs[kD], as[kD], us[kD];
  __shared__ float red[4];
  __shared__ double dred[4][3];
  const int64_t t = blockIdx.x;
  const int h = blockIdx.y, i = threadIdx.x, lane = i & 31, warp = i >> 5;
  qs[i] = Vec<Tin>::load1(Q + ((int64_t)h * T + t) * kD + i);
  __syncthreads();
  const float* Ah = A + (int64_t)h * kD * kD;
  float a = 0.f;
  for (int j = 0; j < kD; ++j) a = fmaf(qs[j], Ah[j * kD + i], a);   // (A^T q)_i
  as[i] = a;
  if (i < r) {
    const float* Lh = L + (int64_t)h * kD * r;
    float u = 0.f;
    for (int j = 0; j < kD; ++j) u = fmaf(qs[j], Lh[j * r + i], u);    // (L^T q)_i
    us[i] = u;
  }
  float qn = nu ? qs[i] * nu[(int64_t)h * kD + i] : 0.f;
  qn = warp_sum(qn);
  if (lane == 0) red[warp] = qn;
  __syncthreads();
  const float qnu = red[0] + red[1] + red[2] + red[3];
  const int64_t base = qinfo[2 * t], vis = qinfo[2 * t + 1];
  const Tin* Kg = K + (int64_t)(h / G) * N * kD;
  const Tin* Ch = codes + (int64_t)h * N * r;
  double ss = 0.0, se = 0.0, cnt = 0.0;
  for (int64_t idx = warp; idx * stride < vis; idx += 4) {
    const int64_t row = base + idx * stride;
    float s = 0.f, sh = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) s = fmaf(as[lane * 4 + c], Vec<Tin>::load1(Kg + row * kD + lane * 4 + c), s);
    for (int c = lane; c < r; c += 32) sh = fmaf(us[c], Vec<Tin>::load1(Ch + row * r + c), sh);
    s = warp_sum(s);
    sh = warp_sum(sh) + qnu;
    ss += (double)s * s;
    se += ((double)s - sh) * ((double)s - sh);
    cnt += 1.0;
  }
  if (lane == 0) { dred[warp][0] = ss; dred[warp][1] = se; dred[warp][2] = cnt; }
  __syncthreads();
  if (i < 3) {
    const double v = dred[0][i] + dred[1][i] + dred[2][i] + dred[3][i];
    if (v != 0.0) atomicAdd(out + (int64_t)h * 3 + i, v);
  }
}

}  // namespace

cudaError_t launch_fourth_moment(const void* q, const void* k, int64_t n, int Hq, int Hk, const float* mu, int dtype,
                                 double* acc, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const int64_t bx = (n + 63) / 64;
  const dim3 grid((unsigned)(bx < 64 ? bx : 64), Hq + Hk);
  note_launch();
  if (dtype == SAKI_BF16)
    fourth_moment_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(q),
                                                             static_cast<const __nv_bfloat16*>(k), n, Hq, mu, acc);
  else
    fourth_moment_kernel<float><<<grid, 256, 0, s>>>(static_cast<const float*>(q), static_cast<const float*>(k), n,
                                                      Hq, mu, acc);
  return cudaGetLastError();
}

cudaError_t launch_shrink(float* S, const double* acc4, int64_t n, int nmat, float* rho, cudaStream_t s) {
  if (nmat == 0) return cudaSuccess;
  note_launch();
  shrink_kernel<<<nmat, 256, 0, s>>>(S, acc4, n, rho);
  return cudaGetLastError();
}

cudaError_t launch_score_mse(const void* Q, const float* A, const void* K, const float* L, const void* codes,
                             const float* nu, const int64_t* qinfo, int64_t T, int64_t N, int Hq, int G, int r,
                             int64_t stride, int dtype, double* out, cudaStream_t s) {
  if (T == 0) return cudaSuccess;
  const dim3 grid((unsigned)T, Hq);
  note_launch();
  if (dtype == SAKI_BF16)
    score_mse_kernel<__nv_bfloat16><<<grid, kD, 0, s>>>(
        static_cast<const __nv_bfloat16*>(Q), A, static_cast<const __nv_bfloat16*>(K), L,
        static_cast<const __nv_bfloat16*>(codes), nu, qinfo, T, N, Hq, G, r, stride, out);
  else
    score_mse_kernel<float><<<grid, kD, 0, s>>>(static_cast<const float*>(Q), A, static_cast<const float*>(K), L,
                                               static_cast<const float*>(codes), nu, qinfo, T, N, Hq, G, r, stride,
                                               out);
  return cudaGetLastError();
}

}  // namespace saki

// ---------------------------------------------------------------- online moments, RoPE composition
namespace saki {
namespace {

// Running moments (in place, n1 rows so far) merged with a batch's moments (n2
// rows): S = (n1 S + n2 B) / n, plus (n1 n2 / n^2) (mu1 - mu2)(mu1 - mu2)^T for
// centered key moments, and mu = (n1 mu1 + n2 mu2) / n (the pooled-variance
// identity).  One CTA per matrix, queries first.
__global__ void __launch_bounds__(256) merge_moments_kernel(float* Sq, float* Sk, float* mu, const float* Sb,
                                                            const float* mub, int Hq, int64_t n1, int64_t n2,
                                                            int center) {
  __shared__ float dm[kD];
  const int m = blockIdx.x, tid = threadIdx.x;
  const bool key = m >= Hq;
  const int g = m - Hq;
  float* S = key ? Sk + (int64_t)g * kD * kD : Sq + (int64_t)m * kD * kD;
  const float* B = Sb + (int64_t)m * kD * kD;
  const double n = (double)(n1 + n2);
  const double w1 = (double)n1 / n, w2 = (double)n2 / n, c = (double)n1 * (double)n2 / (n * n);
  const bool cen = key && center;
  if (tid < kD) dm[tid] = cen && n1 > 0 ? mu[(int64_t)g * kD + tid] - mub[(int64_t)g * kD + tid] : 0.f;
  __syncthreads();
  for (int o = tid; o < kD * kD; o += 256) {
    const int i = o / kD, j = o % kD;
    const double v = w1 * (n1 > 0 ? (double)S[o] : 0.0) + w2 * B[o] + (cen ? c * (double)dm[i] * dm[j] : 0.0);
    S[o] = (float)v;
  }
  if (key && tid < kD && mu) {
    const double m1 = n1 > 0 ? (double)mu[(int64_t)g * kD + tid] : 0.0;
    mu[(int64_t)g * kD + tid] = center ? (float)(w1 * m1 + w2 * mub[(int64_t)g * kD + tid]) : 0.f;
  }
}

// cos and sin of pos * theta^(-2j/d) for j < d/2: the angle in fp64, reduced
// modulo 2 pi before the fp32 evaluation (positions up to 2^31 keep ~1e-7 rad).
__global__ void rope_table_kernel(const int64_t* positions, int64_t n_rows, float theta, float2* table) {
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= n_rows * (kD / 2)) return;
  const int j = (int)(idx % (kD / 2));
  const double inv = pow((double)theta, -2.0 * j / kD);
  double ang = fmod((double)positions[idx / (kD / 2)] * inv, 6.283185307179586476925);
  float sn, cs;
  sincosf((float)ang, &sn, &cs);
  table[idx] = make_float2(cs, sn);
}

// k_hat = nu_h + L_h c for the requested code rows of every query head, then
// (with a table) the rotate-half RoPE rotation: dimension i < d/2 pairs with
// i + d/2.  One warp per (row, head); L_h transposed in shared memory ([c][i],
// conflict-free); lane l holds dimensions l, l+32, l+64, l+96, so both members
// of each rotated pair sit in the same lane.
template <typename Tout, typename Tin>
__global__ void __launch_bounds__(256) reconstruct_kernel(const int64_t* rows, int64_t n_rows, const Tin* codes,
                                                          int64_t N, const float* L, const float* nu, int r,
                                                          const float2* table, Tout* out) {
  extern __shared__ float sm[];
  float* Lt = sm;                 // [r][d]
  float* cs = Lt + r * kD;        // [8][r] code rows of the block's warps
  const int h = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* Lh = L + (int64_t)h * kD * r;
  for (int o = tid; o < kD * r; o += 256) Lt[(o % r) * kD + o / r] = Lh[o];
  __syncthreads();
  const int64_t row = blockIdx.x * 8ll + warp;
  if (row >= n_rows) return;
  const int64_t key = rows[row];
  const bool valid = key >= 0 && key < N;   // a row outside the sketch reads nothing and comes out NaN
  float* c = cs + warp * r;
  for (int i = lane; i < r; i += 32)
    c[i] = valid ? Vec<Tin>::load1(codes + ((int64_t)h * N + key) * r + i) : __int_as_float(0x7fc00000);
  __syncwarp();
  float x[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) x[e] = nu ? nu[(int64_t)h * kD + lane + 32 * e] : 0.f;
  for (int k = 0; k < r; ++k) {
    const float ck = c[k];
#pragma unroll
    for (int e = 0; e < 4; ++e) x[e] = fmaf(Lt[k * kD + lane + 32 * e], ck, x[e]);
  }
  if (table) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const float2 t = table[row * (kD / 2) + lane + 32 * e];
      const float a = x[e], b = x[e + 2];
      x[e] = a * t.x - b * t.y;
      x[e + 2] = b * t.x + a * t.y;
    }
  }
  Tout* o = out + ((int64_t)h * n_rows + row) * kD;
#pragma unroll
  for (int e = 0; e < 4; ++e) o[lane + 32 * e] = from_float<Tout>(x[e]);
}

}  // namespace

cudaError_t launch_merge_moments(float* Sq, float* Sk, float* mu, const float* Sb, const float* mub, int Hq, int Hk,
                                 int64_t n1, int64_t n2, int center, cudaStream_t s) {
  note_launch();
  merge_moments_kernel<<<Hq + Hk, 256, 0, s>>>(Sq, Sk, mu, Sb, mub, Hq, n1, n2, center);
  return cudaGetLastError();
}

cudaError_t launch_reconstruct(const int64_t* rows, int64_t n_rows, const void* codes, int64_t N, const float* L,
                               const float* nu, int Hq, int r, const int64_t* positions, float theta, float2* table,
                               int dtype, void* out, cudaStream_t s) {
  if (n_rows == 0) return cudaSuccess;
  if (positions) {
    const int64_t n = n_rows * (kD / 2);
    note_launch();
    rope_table_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(positions, n_rows, theta, table);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  const float2* tab = positions ? table : nullptr;
  const dim3 grid((unsigned)((n_rows + 7) / 8), Hq);
  const int smem = (int)(sizeof(float) * (r * kD + 8 * r));
  note_launch();
  if (dtype == SAKI_BF16) {
    auto kern = reconstruct_kernel<__nv_bfloat16, __nv_bfloat16>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, 256, smem, s>>>(rows, n_rows, static_cast<const __nv_bfloat16*>(codes), N, L, nu, r, tab,
                                 static_cast<__nv_bfloat16*>(out));
  } else {
    auto kern = reconstruct_kernel<float, float>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, 256, smem, s>>>(rows, n_rows, static_cast<const float*>(codes), N, L, nu, r, tab,
                                 static_cast<float*>(out));
  }
  return cudaGetLastError();
}

}  // namespace saki
