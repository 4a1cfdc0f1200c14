// Key codes of Sec. 6 on CUDA cores: sketch[h][j] = R_h^T (k_j - mu_g), fp32
// accumulation, rounded to nearest-even into the index dtype.  Any rank; one
// CTA per (128 keys, query head), R_h staged in shared memory.
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {

template <typename Tin>
__global__ void __launch_bounds__(256) build_generic_kernel(const Tin* K, const float* R, const float* mu,
                                                            Tin* sketch, int64_t N, int G, int r, int center) {
  extern __shared__ __align__(16) float smr[];   // R_h [d][r], then mu [d]
  float* mus = smr + kD * r;
  const int h = blockIdx.y, g = h / G;
  const int tid = threadIdx.x;
  for (int o = tid; o < kD * r; o += 256) smr[o] = __ldg(R + (int64_t)h * kD * r + o);
  if (tid < kD) mus[tid] = (center && mu) ? __ldg(mu + g * kD + tid) : 0.f;
  __syncthreads();
  const int64_t j = (int64_t)blockIdx.x * 128 + (tid >> 1);
  if (j >= N) return;
  const int half = tid & 1;
  const Tin* krow = K + ((int64_t)g * N + j) * kD;
  Tin* out = sketch + ((int64_t)h * N + j) * r;
  for (int c0 = half * 16; c0 < r; c0 += 32) {
    float acc[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) acc[u] = 0.f;
    for (int i = 0; i < kD; ++i) {
      const float x = Vec<Tin>::load1(krow + i) - mus[i];
#pragma unroll
      for (int u = 0; u < 16; ++u)
        if (c0 + u < r) acc[u] = fmaf(x, smr[i * r + c0 + u], acc[u]);
    }
#pragma unroll
    for (int u = 0; u < 16; ++u)
      if (c0 + u < r) out[c0 + u] = from_float<Tin>(acc[u]);
  }
}
}  // namespace

cudaError_t launch_build_generic(const void* K, const float* R, const float* mu, void* sketch, int64_t N, int Hq,
                                 int G, int r, int center, int dtype, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  const size_t sm = sizeof(float) * ((size_t)kD * r + kD);
  dim3 grid((unsigned)((N + 127) / 128), Hq);
  if (dtype == SAKI_BF16) {
    auto k = build_generic_kernel<__nv_bfloat16>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    note_launch();
    k<<<grid, 256, sm, s>>>(static_cast<const __nv_bfloat16*>(K), R, mu, static_cast<__nv_bfloat16*>(sketch), N,
                            G, r, center);
  } else {
    auto k = build_generic_kernel<float>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    note_launch();
    k<<<grid, 256, sm, s>>>(static_cast<const float*>(K), R, mu, static_cast<float*>(sketch), N, G, r, center);
  }
  return cudaGetLastError();
}

}  // namespace saki
