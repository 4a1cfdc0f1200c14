// Merge of per-part top-k lists (the exchange step of a selection split across
// GPUs by key ranges): every part holds, per row, its k best keys of its own
// contiguous key range with part-local indices; the row's k best over the whole
// range are the k best of the union, indices shifted by each part's offset.
// One warp per row keeps the running k best as 64-bit (score, index) keys
// striped over its lanes: each part's list is sorted by a warp bitonic sort and
// merged in (the best half of two sorted lists).  Ranking: descending score,
// equal scores by the lower global index.
#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {

template <int KP>
__global__ void __launch_bounds__(128) merge_parts_kernel(const int32_t* idx_in, const float* score_in, PartOffsets po,
                                                          int parts, int64_t rows, int k, int32_t* idx, float* score) {
  constexpr int E = KP / 32;
  const int lane = threadIdx.x & 31;
  const int64_t row = blockIdx.x * 4ll + (threadIdx.x >> 5);
  if (row >= rows) return;
  uint64_t best[E], cur[E];
#pragma unroll
  for (int e = 0; e < E; ++e) best[e] = 0ull;
  for (int p = 0; p < parts; ++p) {
    const int64_t base = ((int64_t)p * rows + row) * k;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int i = e * 32 + lane;
      const int32_t j = i < k ? idx_in[base + i] : -1;
      cur[e] = j >= 0 ? make_key(score_in[base + i], (uint32_t)(j + po.off[p])) : 0ull;
    }
    warp_sort_desc<E>(cur);
    warp_merge_top<E>(best, cur);
  }
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = e * 32 + lane;
    if (i < k) {
      idx[row * k + i] = key_index(best[e]);
      if (score) score[row * k + i] = key_score(best[e]);
    }
  }
}

}  // namespace

cudaError_t launch_merge_parts(const int32_t* idx_in, const float* score_in, const PartOffsets& po, int parts,
                               int64_t rows, int k, int32_t* idx, float* score, cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  const unsigned grid = (unsigned)((rows + 3) / 4);
  note_launch();
  if (k <= 64)
    merge_parts_kernel<64><<<grid, 128, 0, s>>>(idx_in, score_in, po, parts, rows, k, idx, score);
  else
    merge_parts_kernel<128><<<grid, 128, 0, s>>>(idx_in, score_in, po, parts, rows, k, idx, score);
  return cudaGetLastError();
}

}  // namespace saki
