// Recall of the Sec. 3 protocol: per (head, query) with at least min_visible
// visible keys, |approx set & exact set| / k, averaged per head.  A warp per
// row inserts the approximate indices into a small open-addressing table in
// shared memory and probes it with the exact ones; integer counts per head are
// accumulated with atomics, so the per-head value is exact and order-free.
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {
constexpr int kSlots = 256;   // >= 2 k for k <= 128

__device__ __forceinline__ uint32_t slot_of(int32_t v) { return ((uint32_t)v * 2654435761u) >> 24; }

__global__ void __launch_bounds__(256) recall_kernel(const int32_t* ia, const int32_t* ie, const int32_t* vis,
                                                     int64_t T, int k, int64_t min_visible,
                                                     unsigned long long* counters) {
  __shared__ int32_t tab[8][kSlots];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int h = blockIdx.y;
  int32_t* tb = tab[warp];
  unsigned long long matches = 0, rows = 0;
  for (int o = lane; o < kSlots; o += 32) tb[o] = -1;
  __syncwarp();
  for (int64_t t = (int64_t)blockIdx.x * 8 + warp; t < T; t += (int64_t)gridDim.x * 8) {
    if (vis[t] < min_visible) continue;   // warp-uniform
    const int32_t* a = ia + ((int64_t)h * T + t) * k;
    const int32_t* e = ie + ((int64_t)h * T + t) * k;
    for (int i = lane; i < k; i += 32) {
      const int32_t v = a[i];
      if (v < 0) continue;
      uint32_t s = slot_of(v);
      while (true) {
        const int32_t prev = atomicCAS(&tb[s], -1, v);
        if (prev == -1 || prev == v) break;
        s = (s + 1) & (kSlots - 1);
      }
    }
    __syncwarp();
    int m = 0;
    for (int i = lane; i < k; i += 32) {
      const int32_t v = e[i];
      if (v < 0) continue;
      uint32_t s = slot_of(v);
      while (true) {
        const int32_t cur = tb[s];
        if (cur == v) { ++m; break; }
        if (cur == -1) break;
        s = (s + 1) & (kSlots - 1);
      }
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) m += __shfl_xor_sync(0xffffffffu, m, d);
    matches += m;
    rows += 1;
    __syncwarp();
    for (int o = lane; o < kSlots; o += 32) tb[o] = -1;
    __syncwarp();
  }
  if (lane == 0 && rows) {
    atomicAdd(counters + 2 * h, matches);
    atomicAdd(counters + 2 * h + 1, rows);
  }
}

__global__ void recall_finish_kernel(const unsigned long long* counters, int Hq, int k, float* recall) {
  const int h = blockIdx.x * blockDim.x + threadIdx.x;
  if (h >= Hq) return;
  const unsigned long long m = counters[2 * h], n = counters[2 * h + 1];
  recall[h] = n ? (float)((double)m / ((double)k * (double)n)) : __int_as_float(0x7fc00000);
}
}  // namespace

cudaError_t launch_recall(const int32_t* idx_a, const int32_t* idx_e, const int32_t* vis, int64_t T, int Hq, int k,
                          int64_t min_visible, unsigned long long* counters, float* recall, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(counters, 0, sizeof(unsigned long long) * 2 * Hq, s);
  if (e != cudaSuccess) return e;
  if (T > 0) {
    const int64_t blocks = (T + 7) / 8;
    dim3 grid((unsigned)(blocks < 1024 ? blocks : 1024), Hq);
    note_launch();
    recall_kernel<<<grid, 256, 0, s>>>(idx_a, idx_e, vis, T, k, min_visible, counters);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  note_launch();
  recall_finish_kernel<<<(Hq + 127) / 128, 128, 0, s>>>(counters, Hq, k, recall);
  return cudaGetLastError();
}

}  // namespace saki
