// Calibration moments of Sec. 5: Sq_h = (1/n) sum_t q_t q_t^T for every query
// head (uncentered) and Sk_g = (1/n) sum_t (k_t - mu_g)(k_t - mu_g)^T with
// mu_g = (1/n) sum_t k_t for every KV head (centered keys, App. A "Centering";
// mu = 0 when center = 0).  CUDA-core path: 64 x 64 output tiles per CTA,
// fp32 accumulation, keys centered on load (two passes, no cancellation).
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {

template <typename Tin>
__global__ void __launch_bounds__(128) key_mean_kernel(const Tin* K, int64_t n, float* mu) {
  const int g = blockIdx.x, i = threadIdx.x;
  const Tin* x = K + (int64_t)g * n * kD + i;
  double acc = 0.0;
  for (int64_t t = 0; t < n; ++t) acc += (double)Vec<Tin>::load1(x + t * kD);
  mu[g * kD + i] = (float)(acc / (double)n);
}

constexpr int kTile = 64, kChunk = 32;

template <typename Tin>
__global__ void __launch_bounds__(256) gram_kernel(const Tin* Xq, const Tin* Xk, int64_t n, int Hq,
                                                   int center, const float* mu, float* S) {
  __shared__ float xa[kChunk][kTile + 4];
  __shared__ float xb[kChunk][kTile + 4];
  const int m = blockIdx.y;
  const bool key = m >= Hq;
  const Tin* X = key ? Xk + (int64_t)(m - Hq) * n * kD : Xq + (int64_t)m * n * kD;
  const float* mv = (key && center) ? mu + (m - Hq) * kD : nullptr;
  const int a0 = (blockIdx.x >> 1) * kTile, b0 = (blockIdx.x & 1) * kTile;
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  float acc[4][4] = {};
  for (int64_t t0 = 0; t0 < n; t0 += kChunk) {
    for (int o = tid; o < kChunk * kTile; o += 256) {
      const int tt = o / kTile, c = o % kTile;
      float va = 0.f, vb = 0.f;
      if (t0 + tt < n) {
        va = Vec<Tin>::load1(X + (t0 + tt) * kD + a0 + c);
        vb = Vec<Tin>::load1(X + (t0 + tt) * kD + b0 + c);
        if (mv) { va -= mv[a0 + c]; vb -= mv[b0 + c]; }
      }
      xa[tt][c] = va;
      xb[tt][c] = vb;
    }
    __syncthreads();
#pragma unroll 8
    for (int tt = 0; tt < kChunk; ++tt) {
      float av[4], bv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) { av[u] = xa[tt][ty * 4 + u]; bv[u] = xb[tt][tx * 4 + u]; }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
    }
    __syncthreads();
  }
  const float inv = 1.0f / (float)n;
  float* Sm = S + (int64_t)m * kD * kD;
#pragma unroll
  for (int u = 0; u < 4; ++u)
#pragma unroll
    for (int v = 0; v < 4; ++v) Sm[(a0 + ty * 4 + u) * kD + b0 + tx * 4 + v] = acc[u][v] * inv;
}

template <typename Tin>
cudaError_t gram_t(const void* q, const void* k, int64_t n, int Hq, int Hk, int center, float* S,
                   float* mu, cudaStream_t s) {
  if (center) key_mean_kernel<Tin><<<Hk, 128, 0, s>>>(static_cast<const Tin*>(k), n, mu);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  gram_kernel<Tin><<<dim3(4, Hq + Hk), 256, 0, s>>>(static_cast<const Tin*>(q), static_cast<const Tin*>(k),
                                                    n, Hq, center, mu, S);
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_gram(const void* q_calib, const void* k_calib, int64_t n, int Hq, int Hk, int center,
                        int dtype, float* S, float* mu, cudaStream_t s) {
  return dtype == SAKI_BF16 ? gram_t<__nv_bfloat16>(q_calib, k_calib, n, Hq, Hk, center, S, mu, s)
                            : gram_t<float>(q_calib, k_calib, n, Hq, Hk, center, S, mu, s);
}

}  // namespace saki
