// Key codes of Sec. 6 on the tensor cores: sketch[h][j] = R_h^T k_j for all query
// heads h of a GQA group at once (uncentered keys, mu = 0).
//
// One persistent CTA per SM walks items (KV head g, block of <= 128 output
// columns = consecutive heads of the group, range of 128-key tiles).  The
// block's R^T, split exactly into three bf16 parts (R = R0 + R1 + R2), stays in
// shared memory while TMA streams key tiles through a ring of stages; one
// thread issues tcgen05.mma (M = 128 keys, N = block columns, K = d = 128, three
// parts) into one of two TMEM accumulators; four epilogue warps (TMEM lane = key)
// read the fp32 codes, round them to bf16 (nearest even) and store each head's
// r values of the key as one contiguous row segment.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace saki {
namespace {

constexpr int kBStages = 3;
constexpr int kKeyTile = 128;
constexpr int kATile = kKeyTile * kD * 2;                // 32 KB: a key tile, two 64-wide K halves
constexpr int kBPartMax = 128 * kD * 2;                  // 32 KB: one part of a 128-column block
constexpr int kOffB = kBStages * kATile;                 // B after the stages
constexpr int kOffBar = kOffB + 3 * kBPartMax;
constexpr int kBuildSmem = kOffBar + 256 + 1024;

__device__ __forceinline__ bool wait_noabort(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity))
    if (clock64() - t0 > tc::kWaitCycles) return false;
  return true;
}

__global__ void __launch_bounds__(192, 1)
    build_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmB,
                    const BuildItem* items, int n_items, int64_t N, int ncol_total, int r, int G,
                    __nv_bfloat16* sketch, int* err, int stall) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* sA = smem;
  uint8_t* sB = smem + kOffB;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* empty = full + kBStages;
  uint64_t* accf = empty + kBStages;
  uint64_t* acce = accf + 2;
  uint64_t* bfull = acce + 2;
  uint64_t* bfree = bfull + 1;
  uint64_t* drain = bfree + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_f = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kBStages; ++s) {
      tc::mbar_init(full + s, 1);
      tc::mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(accf + b, 1);
      tc::mbar_init(acce + b, 128);
    }
    tc::mbar_init(bfull, 1);
    tc::mbar_init(bfree, 1);
    tc::mbar_init(drain, 1);
    *abort_f = 0;
    tc::fence_barrier_init();
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_slot, 256);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;
  // each CTA takes a contiguous run of items, so consecutive items share a B block
  const int per = (n_items + gridDim.x - 1) / gridDim.x;
  const int i_begin = blockIdx.x * per, i_end = min(n_items, i_begin + per);

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tc::prefetch_tmap(&tmK);
      tc::prefetch_tmap(&tmB);
      uint32_t sc = 0;
      int nb = 0;          // B loads issued
      int prev_g = -1, prev_cb = -1;
      bool ok = true;
      for (int item = stall ? i_end : i_begin; item < i_end && ok; ++item) {
        const BuildItem it = items[item];
        if (it.g != prev_g || it.cb != prev_cb) {
          if (nb > 0 && !(ok = tc::mbar_wait(bfree, (nb - 1) & 1, abort_f))) break;
          // full 128-row boxes (rows past the block are never read by the MMA)
          tc::mbar_arrive_expect_tx(bfull, 3 * kBPartMax);
          for (int part = 0; part < 3; ++part)
            for (int kh = 0; kh < 2; ++kh)
              tc::tma_load_2d(sB + part * kBPartMax + kh * (128 * 128), &tmB, bfull, kh * 64,
                              (it.g * 3 + part) * ncol_total + it.cb * 128);
          ++nb;
          prev_g = it.g;
          prev_cb = it.cb;
        }
        for (int t = it.t0; t < it.t1; ++t) {
          const int st = sc % kBStages;
          if (!(ok = tc::mbar_wait(empty + st, ((sc / kBStages) & 1) ^ 1, abort_f))) break;
          tc::mbar_arrive_expect_tx(full + st, kATile);
          const int y = (int)((int64_t)it.g * N + (int64_t)t * kKeyTile);
          tc::tma_load_2d(sA + st * kATile, &tmK, full + st, 0, y);
          tc::tma_load_2d(sA + st * kATile + kKeyTile * 128, &tmK, full + st, 64, y);
          ++sc;
        }
      }
      for (int s = 0; s < kBStages; ++s) {
        if ((uint32_t)s >= sc) break;
        const uint32_t last = s + kBStages * ((sc - 1 - s) / kBStages);
        if (!wait_noabort(full + s, (last / kBStages) & 1)) *abort_f = 1;
      }
      if (nb > 0 && !wait_noabort(bfull, (nb - 1) & 1)) *abort_f = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t sc = 0, ac = 0;
      int nb = 0;
      int prev_g = -1, prev_cb = -1;
      bool ok = true;
      const uint32_t aBase = tc::smem_u32(sA), bBase = tc::smem_u32(sB);
      for (int item = i_begin; item < i_end && ok; ++item) {
        const BuildItem it = items[item];
        const int ncol = min(128, ncol_total - it.cb * 128);
        const uint32_t idesc = tc::idesc_bf16(128, ncol);
        if (it.g != prev_g || it.cb != prev_cb) {
          if (nb > 0) tc::mma_commit(bfree);   // the previous block's MMAs release B
          if (!(ok = tc::mbar_wait(bfull, nb & 1, abort_f))) break;
          ++nb;
          prev_g = it.g;
          prev_cb = it.cb;
        }
        for (int t = it.t0; t < it.t1; ++t) {
          const uint32_t buf = ac & 1;
          if (!(ok = tc::mbar_wait(acce + buf, ((ac >> 1) & 1) ^ 1, abort_f))) break;
          const int st = sc % kBStages;
          if (!(ok = tc::mbar_wait(full + st, (sc / kBStages) & 1, abort_f))) break;
          tc::fence_after_sync();
          uint32_t acc = 0;
          for (int part = 0; part < 3; ++part)
#pragma unroll
            for (int kh = 0; kh < 2; ++kh)
#pragma unroll
              for (int kk = 0; kk < 4; ++kk) {
                const uint32_t ad = aBase + st * kATile + kh * (kKeyTile * 128) + kk * 32;
                const uint32_t bd = bBase + part * kBPartMax + kh * (128 * 128) + kk * 32;
                tc::mma_bf16(tmem + buf * 128, tc::sdesc(ad, 1024, 2), tc::sdesc(bd, 1024, 2), idesc, acc);
                acc = 1;
              }
          tc::mma_commit(empty + st);
          tc::mma_commit(accf + buf);
          ++sc;
          ++ac;
        }
      }
      tc::mma_commit(drain);
      if (!wait_noabort(drain, 0)) *abort_f = 1;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;
    const int m = quarter * 32 + lane;   // key within the tile
    const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
    uint32_t ac = 0;
    bool ok = true;
    for (int item = i_begin; item < i_end && ok; ++item) {
      const BuildItem it = items[item];
      const int ncol = min(128, ncol_total - it.cb * 128);
      for (int t = it.t0; t < it.t1; ++t) {
        const uint32_t buf = ac & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(accf + buf, (ac >> 1) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
        const int64_t j = (int64_t)t * kKeyTile + m;
        for (int c0 = 0; c0 < ncol; c0 += 32) {
          uint32_t v[32];
          __syncwarp();
          tc::tmem_ld32(tl + buf * 128 + c0, v);
          tc::tmem_ld_wait();
          if (c0 + 32 >= ncol) {
            tc::fence_before_sync();
            tc::mbar_arrive(acce + buf);
          }
          if (j < N) {
            // columns c0.. of the block are (head, code) pairs: col = hl * r + c
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              if (c0 + q * 8 >= ncol) break;
              const int col = it.cb * 128 + c0 + q * 8;
              const int hl = col / r, c = col % r;
              const int h = it.g * G + hl;
              uint4 pk;
              pk.x = pack_bf16_pair(__uint_as_float(v[q * 8 + 0]), __uint_as_float(v[q * 8 + 1]));
              pk.y = pack_bf16_pair(__uint_as_float(v[q * 8 + 2]), __uint_as_float(v[q * 8 + 3]));
              pk.z = pack_bf16_pair(__uint_as_float(v[q * 8 + 4]), __uint_as_float(v[q * 8 + 5]));
              pk.w = pack_bf16_pair(__uint_as_float(v[q * 8 + 6]), __uint_as_float(v[q * 8 + 7]));
              *reinterpret_cast<uint4*>(sketch + ((int64_t)h * N + j) * r + c) = pk;
            }
          }
        }
        ++ac;
      }
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (*abort_f && threadIdx.x == 0) atomicOr(err, 1);
  if (warp == 1) tc::tmem_dealloc(tmem, 256);
}

// R [Hq][d][r] fp32 -> per KV head g: [3][G*r][d] bf16 (row n = hl * r + c holds
// R_{gG+hl}[:, c] transposed), with R = part0 + part1 + part2 exactly.
__global__ void pack_rt_kernel(const float* R, int Hq, int G, int r, __nv_bfloat16* out) {
  const int Hk = Hq / G, ncol = G * r;
  const int64_t n = (int64_t)Hq * r * kD;
  for (int64_t o = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; o < n; o += (int64_t)gridDim.x * blockDim.x) {
    const int i = (int)(o % kD);
    const int c = (int)((o / kD) % r);
    const int h = (int)(o / ((int64_t)kD * r));
    const int g = h / G, hl = h % G;
    const float w = R[((int64_t)h * kD + i) * r + c];
    const __nv_bfloat16 w0 = __float2bfloat16_rn(w);
    const float r1 = w - __bfloat162float(w0);
    const __nv_bfloat16 w1 = __float2bfloat16_rn(r1);
    const __nv_bfloat16 w2 = __float2bfloat16_rn(r1 - __bfloat162float(w1));
    const int64_t row = hl * r + c;
    const int64_t base = ((int64_t)g * 3 * ncol + row) * kD + i;
    out[base] = w0;
    out[base + (int64_t)ncol * kD] = w1;
    out[base + 2 * (int64_t)ncol * kD] = w2;
  }
  (void)Hk;
}

bool make_map2(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint32_t box_inner, uint32_t box_rows) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return false;
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

bool build_tc_supported(int r, int G) {
  return r % 16 == 0 && r >= 16 && r <= 128 && 128 % r == 0 && (G * r) % 16 == 0;
}

size_t build_tc_workspace(int Hq, int r) { return (size_t)Hq * 3 * r * kD * 2; }

cudaError_t launch_build_tc(const void* K, const float* R, void* sketch, int64_t N, int Hq, int G, int r,
                            const BuildItem* items, int n_items, void* wsplit, int* err, int stall,
                            int num_sms, cudaStream_t s) {
  if (n_items == 0) return cudaSuccess;
  const int64_t n = (int64_t)Hq * r * kD;
  const int blocks = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  note_launch();
  pack_rt_kernel<<<blocks, 256, 0, s>>>(R, Hq, G, r, static_cast<__nv_bfloat16*>(wsplit));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int Hk = Hq / G, ncol_total = G * r;
  CUtensorMap mK, mB;
  if (!make_map2(&mK, K, kD, (uint64_t)Hk * N, 64, kKeyTile) ||
      !make_map2(&mB, wsplit, kD, (uint64_t)Hk * 3 * ncol_total, 64, 128))
    return cudaErrorInvalidValue;
  e = cudaFuncSetAttribute(build_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kBuildSmem);
  if (e != cudaSuccess) return e;
  const int grid = n_items < num_sms ? n_items : num_sms;
  note_launch();
  build_tc_kernel<<<grid, 192, kBuildSmem, s>>>(mK, mB, items, n_items, N, ncol_total, r, G,
                                                static_cast<__nv_bfloat16*>(sketch), err, stall);
  return cudaGetLastError();
}

}  // namespace saki
