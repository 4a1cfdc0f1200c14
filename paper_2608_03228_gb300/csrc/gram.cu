// Calibration moments of Sec. 6: Sq_h = (1/n) sum_t q_t q_t^T for every query
// head (uncentered) and Sk_g = (1/n) sum_t (k_t - mu_g)(k_t - mu_g)^T with
// mu_g = (1/n) sum_t k_t for every KV head (centered keys, App. A "Centering";
// mu = 0 when center = 0).
//   Tensor-core path (bf16 inputs, uncentered matrices): S = (1/n) X^T X with
//   X (n x d) streamed in chunks of 64 rows; bf16 x bf16 products are exact in
//   the fp32 accumulator.
//   CUDA-core path (fp32 inputs, centered keys): 64 x 64 output tiles per CTA,
//   fp32 accumulation, keys centered on load (two passes, no cancellation).
#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

#include <type_traits>

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
                                                   int center, const float* mu, float* S, int m0) {
  __shared__ float xa[kChunk][kTile + 4];
  __shared__ float xb[kChunk][kTile + 4];
  const int m = m0 + blockIdx.y;
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

// ---------------------------------------------------------------- tensor-core moments
// One CTA (128 threads) per matrix.  A chunk of 64 rows of X is transposed in
// registers (8 x 8 blocks of bf16 by byte permutes) into a K-major tile with
// 128-byte swizzle: row m (a dimension) holds that dimension's 64 values.  The
// same tile is both MMA operands (D[m][n] = sum_k X[k][m] X[k][n]), the fp32
// 128 x 128 accumulator lives in TMEM, and two tiles alternate so that the
// transpose of chunk c+1 overlaps the multiplications of chunk c.
constexpr int kGramChunk = 64;
constexpr int kGramSmem = 2 * 16384 + 1024 + 64 + 16 * 1024;  // tiles, alignment, barriers; caps at 4 CTAs per SM

__device__ __forceinline__ void gram_load(const __nv_bfloat16* X, int64_t n, int64_t r0, int kb, int mb, uint4 (&w)[8]) {
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    const int64_t row = r0 + kb * 8 + r;
    w[r] = row < n ? __ldg(reinterpret_cast<const uint4*>(X + row * kD + mb * 8)) : make_uint4(0u, 0u, 0u, 0u);
  }
}

// Rows [r0, r0 + nrows) of each matrix's n rows; the 1/n-scaled Gram is
// written (add = 0) or added to S (add = 1).  The tensor core's fp32
// accumulation is exact per product but its long sums drift (32,768 rows left
// the moments about 2e-4 low), so the host cuts n into launches of at most
// kGramRows rows and the partial moments are summed in S.
__global__ void __launch_bounds__(128) gram_tc_kernel(const __nv_bfloat16* Xq, const __nv_bfloat16* Xk, int64_t n,
                                                      int Hq, int64_t r0, int64_t nrows, int add, float* S,
                                                      int* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* done = reinterpret_cast<uint64_t*>(smem + 2 * 16384);   // [2] MMA completion per tile
  uint64_t* drain = done + 2;                                        // every multiplication of the CTA
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_f = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int m = blockIdx.x;
  const __nv_bfloat16* X = (m < Hq ? Xq + (int64_t)m * n * kD : Xk + (int64_t)(m - Hq) * n * kD) + r0 * kD;
  const int64_t nl = nrows;
  if (tid == 0) {
    tc::mbar_init(done, 1);
    tc::mbar_init(done + 1, 1);
    tc::mbar_init(drain, 1);
    *abort_f = 0;
    tc::fence_barrier_init();
  }
  if (warp == 0) {
    tc::tmem_alloc(tmem_slot, 128);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;
  const int kb = tid & 7, mb = tid >> 3;   // this thread's 8 x 8 block: rows 8kb.., dimensions 8mb..
  const int nch = (int)((nl + kGramChunk - 1) / kGramChunk);
  constexpr uint32_t idesc = tc::idesc_bf16(128, 128);
  // two chunks of rows in flight per thread beyond the one being transposed
  uint4 w[8], wn[8];
  gram_load(X, nl, 0, kb, mb, w);
  gram_load(X, nl, kGramChunk, kb, mb, wn);   // rows past nl load as zeros
  bool ok = true;
  for (int c = 0; c < nch; ++c) {
    const int b = c & 1;
    uint4 wn2[8];
    if (c + 2 < nch) gram_load(X, nl, (int64_t)(c + 2) * kGramChunk, kb, mb, wn2);
    else
#pragma unroll
      for (int r = 0; r < 8; ++r) wn2[r] = make_uint4(0u, 0u, 0u, 0u);
    if (c >= 2) ok = tc::mbar_wait(done + b, ((c >> 1) & 1) ^ 1, abort_f);
    if (!__syncthreads_and(ok)) break;
    uint8_t* tile = smem + b * 16384;
#pragma unroll
    for (int mm = 0; mm < 8; ++mm) {
      const uint32_t sel = (mm & 1) ? 0x7632u : 0x5410u;
      uint32_t o[4];
#pragma unroll
      for (int f = 0; f < 4; ++f) {
        const uint32_t* lo = reinterpret_cast<const uint32_t*>(&w[2 * f]);
        const uint32_t* hi = reinterpret_cast<const uint32_t*>(&w[2 * f + 1]);
        o[f] = __byte_perm(lo[mm >> 1], hi[mm >> 1], sel);
      }
      const int row = mb * 8 + mm;
      *reinterpret_cast<uint4*>(tile + row * 128 + ((kb ^ (row & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
    }
    tc::fence_proxy_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      const uint32_t base = tc::smem_u32(tile);
#pragma unroll
      for (int kk = 0; kk < kGramChunk / 16; ++kk) {
        const uint64_t d = tc::sdesc(base + kk * 32, 1024, 2);
        tc::mma_bf16(tmem, d, d, idesc, (c > 0 || kk > 0) ? 1u : 0u);
      }
      tc::mma_commit(done + b);
    }
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      w[r] = wn[r];
      wn[r] = wn2[r];
    }
  }
  // one more commit covers every multiplication issued (also after an early exit)
  if (tid == 0) tc::mma_commit(drain);
  const bool drained = tc::mbar_wait_bounded(drain, 0);
  ok = __syncthreads_and(ok && drained);
  tc::fence_after_sync();
  if (ok) {
    const float inv = 1.0f / (float)n;
    float* Sm = S + (int64_t)m * kD * kD + (int64_t)tid * kD;
#pragma unroll
    for (int c0 = 0; c0 < kD; c0 += 32) {
      uint32_t r[32];
      tc::tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + c0, r);
      tc::tmem_ld_wait();
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v = make_float4(__uint_as_float(r[4 * q]) * inv, __uint_as_float(r[4 * q + 1]) * inv,
                               __uint_as_float(r[4 * q + 2]) * inv, __uint_as_float(r[4 * q + 3]) * inv);
        float4* dst = reinterpret_cast<float4*>(Sm + c0 + 4 * q);
        if (add) {
          const float4 o = *dst;
          v.x += o.x; v.y += o.y; v.z += o.z; v.w += o.w;
        }
        *dst = v;
      }
    }
  } else if (tid == 0) {
    atomicOr(err, kStTimeout);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 128);
}

constexpr int64_t kGramRows = 4096;   // rows per tensor-core moment launch

template <typename Tin>
cudaError_t gram_t(const void* q, const void* k, int64_t n, int Hq, int Hk, int center, float* S,
                   float* mu, int* err, cudaStream_t s) {
  if (center) {
    note_launch();
    key_mean_kernel<Tin><<<Hk, 128, 0, s>>>(static_cast<const Tin*>(k), n, mu);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int first_cuda = 0;   // first matrix left to the CUDA-core kernel
  if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
    const int ntc = center ? Hq : Hq + Hk;
    if (ntc > 0 && n > 0) {
      e = cudaFuncSetAttribute(gram_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGramSmem);
      if (e != cudaSuccess) return e;
      for (int64_t r0 = 0; r0 < n; r0 += kGramRows) {
        note_launch();
        gram_tc_kernel<<<ntc, 128, kGramSmem, s>>>(static_cast<const __nv_bfloat16*>(q),
                                                   static_cast<const __nv_bfloat16*>(k), n, Hq, r0,
                                                   n - r0 < kGramRows ? n - r0 : kGramRows, r0 > 0 ? 1 : 0, S, err);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
      }
    }
    first_cuda = ntc;
  }
  const int rest = Hq + Hk - first_cuda;
  if (rest > 0) {
    note_launch();
    gram_kernel<Tin><<<dim3(4, rest), 256, 0, s>>>(static_cast<const Tin*>(q), static_cast<const Tin*>(k), n, Hq,
                                                   center, mu, S, first_cuda);
  }
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_gram(const void* q_calib, const void* k_calib, int64_t n, int Hq, int Hk, int center,
                        int dtype, float* S, float* mu, int* err, cudaStream_t s) {
  return dtype == SAKI_BF16 ? gram_t<__nv_bfloat16>(q_calib, k_calib, n, Hq, Hk, center, S, mu, err, s)
                            : gram_t<float>(q_calib, k_calib, n, Hq, Hk, center, S, mu, err, s);
}

}  // namespace saki
