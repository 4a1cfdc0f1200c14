// Recall of the Sec. 3 protocol: per (head, query) with at least min_visible
// visible keys, |approx set & exact set| / k, averaged per head.  A warp walks a
// contiguous range of (head, query) rows, loading the next row's two index
// lists while it matches the current one.  Where every row sees at most
// kBitmapKeys keys, the warp marks the approximate indices in a bitmap of the
// row's key range in shared memory (one atomic OR per index), tests the exact
// ones against it and clears the words it set; otherwise it inserts them into
// a small open-addressing table.  Integer counts per head are flushed with
// atomics when the head changes, so the per-head value is exact and
// order-free.
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {
constexpr int kSlots = 256;       // >= 2 k for k <= 128
constexpr int kPerLane = 4;       // k <= 128 indices per list: at most 4 per lane
constexpr int64_t kBitmapKeys = 24576;   // bitmap path: 8 warps x 3 KB of shared memory per block

__device__ __forceinline__ uint32_t slot_of(int32_t v) { return ((uint32_t)v * 2654435761u) >> 24; }

// Bitmap matching: words = bitmap words per warp (dynamic shared memory, 8 warps).
// A warp's rows go in groups of four, two groups in registers: the index lists
// of the next group load while the current group is matched (a row alone left
// too few bytes in flight).  KPL = index slots per lane (k <= 32 KPL).
template <int KPL>
__global__ void __launch_bounds__(256) recall_bitmap_kernel(const int32_t* ia, const int32_t* ie, const int32_t* vis,
                                                            int64_t T, int Hq, int k, int64_t min_visible, int words,
                                                            unsigned long long* counters) {
  constexpr int R = 4;
  extern __shared__ uint32_t bm_all[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t* bm = bm_all + warp * words;
  for (int o = lane; o < words; o += 32) bm[o] = 0u;
  __syncwarp();
  const int64_t total = (int64_t)Hq * T;
  const int64_t nwarps = (int64_t)gridDim.x * 8;
  const int64_t per = (total + nwarps - 1) / nwarps;
  const int64_t r0 = ((int64_t)blockIdx.x * 8 + warp) * per;
  const int64_t r1 = r0 + per < total ? r0 + per : total;
  const int64_t nbits = (int64_t)words * 32;
  int cur_h = -1;
  unsigned long long matches = 0, rows = 0;
  int64_t lt = r0 % T;            // query of the next row to load
  int64_t pt = r0 % T;            // query and head of the next row to match
  int ph = (int)(r0 / T);
  auto load_group = [&](int64_t rg, int32_t (&va)[R][KPL], int32_t (&ve)[R][KPL], int32_t (&vv)[R]) {
#pragma unroll
    for (int j = 0; j < R; ++j) {
      const int64_t r = rg + j;
      const bool row_in = r < r1;
#pragma unroll
      for (int u = 0; u < KPL; ++u) {
        const int i = lane + 32 * u;
        const bool in = row_in && i < k;
        va[j][u] = in ? __ldg(ia + r * k + i) : -1;
        ve[j][u] = in ? __ldg(ie + r * k + i) : -1;
      }
      vv[j] = row_in ? __ldg(vis + lt) : 0;
      if (row_in && ++lt == T) lt = 0;
    }
  };
  auto match_group = [&](int64_t rg, const int32_t (&va)[R][KPL], const int32_t (&ve)[R][KPL],
                         const int32_t (&vv)[R]) {
#pragma unroll
    for (int j = 0; j < R; ++j) {
      if (rg + j >= r1) break;   // warp-uniform
      const int h = ph;
      if (++pt == T) {
        pt = 0;
        ++ph;
      }
      if (h != cur_h) {
        if (lane == 0 && rows) {
          atomicAdd(counters + 2 * cur_h, matches);
          atomicAdd(counters + 2 * cur_h + 1, rows);
        }
        cur_h = h;
        matches = rows = 0;
      }
      if (vv[j] < min_visible) continue;   // warp-uniform
      // indices outside the bitmap (none from the selection calls) match nothing
#pragma unroll
      for (int u = 0; u < KPL; ++u)
        if (va[j][u] >= 0 && va[j][u] < nbits) atomicOr(bm + (va[j][u] >> 5), 1u << (va[j][u] & 31));
      __syncwarp();
      int m = 0;
#pragma unroll
      for (int u = 0; u < KPL; ++u)
        if (ve[j][u] >= 0 && ve[j][u] < nbits) m += (bm[ve[j][u] >> 5] >> (ve[j][u] & 31)) & 1u;
      m = __reduce_add_sync(0xffffffffu, m);
      matches += (unsigned long long)m;
      rows += 1;
      __syncwarp();
#pragma unroll
      for (int u = 0; u < KPL; ++u)
        if (va[j][u] >= 0 && va[j][u] < nbits) bm[va[j][u] >> 5] = 0u;
      __syncwarp();
    }
  };
  int32_t aA[R][KPL], eA[R][KPL], vA[R], aB[R][KPL], eB[R][KPL], vB[R];
  load_group(r0, aA, eA, vA);
  load_group(r0 + R, aB, eB, vB);
  for (int64_t rg = r0; rg < r1; rg += 2 * R) {
    match_group(rg, aA, eA, vA);
    load_group(rg + 2 * R, aA, eA, vA);
    match_group(rg + R, aB, eB, vB);
    load_group(rg + 3 * R, aB, eB, vB);
  }
  if (lane == 0 && rows) {
    atomicAdd(counters + 2 * cur_h, matches);
    atomicAdd(counters + 2 * cur_h + 1, rows);
  }
}

__global__ void __launch_bounds__(256) recall_kernel(const int32_t* ia, const int32_t* ie, const int32_t* vis,
                                                     int64_t T, int Hq, int k, int64_t min_visible,
                                                     unsigned long long* counters) {
  __shared__ int32_t tab[8][kSlots];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int32_t* tb = tab[warp];
  for (int o = lane; o < kSlots; o += 32) tb[o] = -1;
  __syncwarp();
  const int64_t total = (int64_t)Hq * T;
  const int64_t nwarps = (int64_t)gridDim.x * 8;
  const int64_t per = (total + nwarps - 1) / nwarps;
  const int64_t r0 = ((int64_t)blockIdx.x * 8 + warp) * per;
  const int64_t r1 = r0 + per < total ? r0 + per : total;
  int cur_h = -1;
  unsigned long long matches = 0, rows = 0;
  // the next row's two index lists are loaded while this row is matched
  int32_t na[kPerLane], ne[kPerLane];
  int64_t nt = r0 % T;   // query of the next row; its head follows from the row index
  int nh = (int)(r0 / T);
  int32_t nvis = r0 < r1 ? __ldg(vis + nt) : 0;
  auto load_row = [&](int64_t r, int32_t (&va)[kPerLane], int32_t (&ve)[kPerLane]) {
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      const int i = lane + 32 * u;
      const bool in = r < r1 && i < k;
      va[u] = in ? __ldg(ia + r * k + i) : -1;
      ve[u] = in ? __ldg(ie + r * k + i) : -1;
    }
  };
  load_row(r0, na, ne);
  for (int64_t r = r0; r < r1; ++r) {
    int32_t av[kPerLane], ev[kPerLane];
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      av[u] = na[u];
      ev[u] = ne[u];
    }
    const int h = nh;
    const int32_t row_vis = nvis;
    if (++nt == T) {
      nt = 0;
      ++nh;
    }
    nvis = r + 1 < r1 ? __ldg(vis + nt) : 0;
    load_row(r + 1, na, ne);
    if (h != cur_h) {
      if (lane == 0 && rows) {
        atomicAdd(counters + 2 * cur_h, matches);
        atomicAdd(counters + 2 * cur_h + 1, rows);
      }
      cur_h = h;
      matches = rows = 0;
    }
    if (row_vis < min_visible) continue;   // warp-uniform
    uint32_t used[kPerLane];
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) used[u] = kSlots;
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      if (av[u] < 0) continue;
      uint32_t sl = slot_of(av[u]);
      while (true) {
        const int32_t prev = atomicCAS(&tb[sl], -1, av[u]);
        if (prev == -1) { used[u] = sl; break; }
        if (prev == av[u]) break;
        sl = (sl + 1) & (kSlots - 1);
      }
    }
    __syncwarp();
    int m = 0;
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      if (ev[u] < 0) continue;
      uint32_t sl = slot_of(ev[u]);
      while (true) {
        const int32_t cur = tb[sl];
        if (cur == ev[u]) { ++m; break; }
        if (cur == -1) break;
        sl = (sl + 1) & (kSlots - 1);
      }
    }
    m = (int)warp_sum((float)m);
    matches += (unsigned long long)m;
    rows += 1;
    __syncwarp();
#pragma unroll
    for (int u = 0; u < kPerLane; ++u)
      if (used[u] < kSlots) tb[used[u]] = -1;
    __syncwarp();
  }
  if (lane == 0 && rows) {
    atomicAdd(counters + 2 * cur_h, matches);
    atomicAdd(counters + 2 * cur_h + 1, rows);
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
                          int64_t min_visible, int64_t max_visible, unsigned long long* counters, float* recall,
                          cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(counters, 0, sizeof(unsigned long long) * 2 * Hq, s);
  if (e != cudaSuccess) return e;
  if (T > 0) {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t rows = (int64_t)Hq * T;
    const int64_t want = (rows + 7) / 8;   // at least one row per warp
    const int64_t blocks = want < (int64_t)sms * 4 ? want : (int64_t)sms * 4;
    note_launch();
    if (max_visible <= kBitmapKeys) {
      const int words = (int)((max_visible + 31) / 32) < 1 ? 1 : (int)((max_visible + 31) / 32);
      const size_t sm = (size_t)8 * words * sizeof(uint32_t);
      // one wave: as many CTAs as are resident (the two row groups in registers
      // leave room for fewer CTAs per SM than the table version)
      auto kern = k <= 64 ? recall_bitmap_kernel<2> : recall_bitmap_kernel<4>;
      int per_sm = 0;
      if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, sm) != cudaSuccess || per_sm < 1)
        per_sm = 1;
      const int64_t bb = want < (int64_t)sms * per_sm ? want : (int64_t)sms * per_sm;
      kern<<<(unsigned)bb, 256, sm, s>>>(idx_a, idx_e, vis, T, Hq, k, min_visible, words, counters);
    } else {
      recall_kernel<<<(unsigned)blocks, 256, 0, s>>>(idx_a, idx_e, vis, T, Hq, k, min_visible, counters);
    }
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  note_launch();
  recall_finish_kernel<<<(Hq + 127) / 128, 128, 0, s>>>(counters, Hq, k, recall);
  return cudaGetLastError();
}

}  // namespace saki
