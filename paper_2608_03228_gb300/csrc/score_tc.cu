// Batched fused score + top-k on the 5th-generation tensor cores (sm_103a).
//
// One persistent CTA per SM walks work items (a tile of up to 128 consecutive
// queries of one sequence, one query head), heaviest tiles first.  Per item:
//   1. projection on the tensor core: u = W^T q for the 128 queries, with the
//      fp32 projection W (L for Sec. 5's selection, A for the exact scores of the
//      Sec. 3 protocol) split exactly into three bf16 parts; the fp32 result in
//      TMEM is split into u_hi + u_lo (bf16 each) and written, swizzled, as the
//      A operand of the main loop (keeping u to ~16 bits, far below the score
//      tolerance);
//   2. main loop over key tiles of the visible range: TMA brings NT key rows
//      (codes, or raw keys for the exact scores) into a ring of shared-memory
//      stages; one thread issues tcgen05.mma (M = 128 queries, N = NT keys,
//      K = P, twice: u_hi and u_lo) into one of two TMEM accumulators;
//   3. four epilogue warps own one query row per thread (TMEM lane = row): they
//      pull 32 scores at a time with tcgen05.ld, mask the causal edge, skip any
//      16-score half whose maximum does not beat the row's threshold, and append
//      the others to the row's candidate column in shared memory; when a column
//      fills, a sampled pivot shrinks it to a set that still holds the row's top
//      k and raises the threshold.  The T x N score matrix is never stored.
//   4. exact top-k of the remaining candidates per row, written coalesced.
// Roles: warp 0 = TMA producer, warp 1 = TMEM owner + MMA issuer, warps 2-5 =
// epilogue.  Every mbarrier wait is bounded (tc.cuh); a timed-out CTA drains its
// copies and MMAs, frees TMEM, flags the error word and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace saki {
namespace {

constexpr int kLdc = 129;   // candidate column stride (words): conflict-free per-row scans and row reads

template <int P>
struct TcCfg {
  static constexpr int NT = P == 128 ? 128 : 256;            // keys per tile (MMA N)
  static constexpr int STAGES = P <= 32 ? 4 : 2;
  static constexpr int CAP = P == 128 ? 128 : (P == 16 ? 208 : 168);   // candidate slots per row
  static constexpr int KB = P == 128 ? 2 : 1;                 // 64-wide K blocks
  static constexpr int KW = P == 128 ? 64 : P;                // K width of one block
  static constexpr int KK = KW / 16;                          // MMA K steps per block
  static constexpr uint32_t SW = KW == 64 ? 2u : (KW == 32 ? 4u : 6u);
  static constexpr uint32_t SBO = 8 * KW * 2;
  static constexpr int A_PART = 128 * P * 2;                  // u_hi (or u_lo) bytes
  static constexpr int A_BYTES = 2 * A_PART > 32768 ? 2 * A_PART : 32768;  // also holds the 128x128 query tile
  static constexpr int STAGE_BYTES = NT * P * 2;
  static constexpr int CAND_BYTES = CAP * kLdc * 4 + ((CAP * kLdc * 2 + 15) & ~15);
  static constexpr int TMEM_COLS = 2 * NT;
  static constexpr int OFF_STAGE = A_BYTES;
  static constexpr int OFF_CAND = OFF_STAGE + STAGES * STAGE_BYTES;
  static constexpr int OFF_BAR = OFF_CAND + CAND_BYTES;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static_assert(STAGE_BYTES >= P * 128, "a projection chunk must fit a stage");
  static_assert(SMEM <= 232448, "shared memory budget");
};

__device__ __forceinline__ float fmax3(float a, float b, float c) { return fmaxf(a, fmaxf(b, c)); }

// ---------------------------------------------------------------- selection
// A row's candidate column: scores (fp32) and key indices (16-bit; the host only
// sends sequences of at most 65535 keys here).
struct Col {
  float* bs;
  uint16_t* bi;
  int row;
  __device__ __forceinline__ float s(int i) const { return bs[i * kLdc + row]; }
  __device__ __forceinline__ int j(int i) const { return bi[i * kLdc + row]; }
  __device__ __forceinline__ void put(int i, float v, int k) const {
    bs[i * kLdc + row] = v;
    bi[i * kLdc + row] = (uint16_t)k;
  }
};

// The passes below keep eight independent shared-memory loads in flight per
// thread: a row's column is scanned with no other parallelism, so latency, not
// bandwidth, bounds them.

// Number of entries scoring >= p.
__device__ __forceinline__ int count_ge(const Col& c, int cnt, float p) {
  int n0 = 0, n1 = 0, i = 0;
  for (; i + 8 <= cnt; i += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = c.s(i + u);
#pragma unroll
    for (int u = 0; u < 8; u += 2) {
      n0 += v[u] >= p;
      n1 += v[u + 1] >= p;
    }
  }
  for (; i < cnt; ++i) n0 += c.s(i) >= p;
  return n0 + n1;
}

// Keep the entries scoring >= p (in place, order preserved); returns their count.
__device__ __forceinline__ int compact_ge(const Col& c, int cnt, float p) {
  int w = 0, i = 0;
  for (; i + 8 <= cnt; i += 8) {
    float v[8];
    int j[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      v[u] = c.s(i + u);
      j[u] = c.j(i + u);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (v[u] >= p) {
        c.put(w, v[u], j[u]);
        ++w;
      }
  }
  for (; i < cnt; ++i) {
    const float v = c.s(i);
    if (v >= p) {
      c.put(w, v, c.j(i));
      ++w;
    }
  }
  return w;
}

// (score, index) worse-than: lower score, or equal score and higher index.
__device__ __forceinline__ bool worse(float a, int ja, float b, int jb) { return a < b || (a == b && ja > jb); }

// Remove the worst entry (lowest score, then highest index); raise thr to its score.
__device__ __forceinline__ void remove_worst(const Col& c, int& cnt, float& thr) {
  float ws[4];
  int wj[4], wp[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) { ws[u] = INFINITY; wj[u] = -1; wp[u] = 0; }
  int i = 0;
  for (; i + 4 <= cnt; i += 4) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float v = c.s(i + u);
      const int jj = c.j(i + u);
      if (worse(v, jj, ws[u], wj[u])) { ws[u] = v; wj[u] = jj; wp[u] = i + u; }
    }
  }
  for (; i < cnt; ++i) {
    const float v = c.s(i);
    const int jj = c.j(i);
    if (worse(v, jj, ws[0], wj[0])) { ws[0] = v; wj[0] = jj; wp[0] = i; }
  }
#pragma unroll
  for (int u = 1; u < 4; ++u)
    if (worse(ws[u], wj[u], ws[0], wj[0])) { ws[0] = ws[u]; wj[0] = wj[u]; wp[0] = wp[u]; }
  --cnt;
  c.put(wp[0], c.s(cnt), c.j(cnt));
  thr = fmaxf(thr, ws[0]);
}

// Keep every entry scoring >= a sampled pivot p, provided at least k and at most
// tmax remain; the threshold becomes p (all later keys have higher indices, so a
// key scoring exactly p loses to all kept entries).  Returns false if no tried
// pivot qualifies.
__device__ __forceinline__ bool pivot_round(const Col& c, int& cnt, float& thr, int k, int aim, int tmax) {
  float s[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) s[u] = c.s(((2 * u + 1) * cnt) >> 4);
  // Batcher odd-even merge sort of 8, descending
  auto cx = [&](int a, int b) {
    const float x = fmaxf(s[a], s[b]), y = fminf(s[a], s[b]);
    s[a] = x;
    s[b] = y;
  };
  cx(0, 1); cx(2, 3); cx(4, 5); cx(6, 7);
  cx(0, 2); cx(1, 3); cx(4, 6); cx(5, 7);
  cx(1, 2); cx(5, 6);
  cx(0, 4); cx(1, 5); cx(2, 6); cx(3, 7);
  cx(2, 4); cx(3, 5);
  cx(1, 2); cx(3, 4); cx(5, 6);
  // sample q (0-based, descending) sits near entry rank (q + 0.5) cnt / 8
  int q = (16 * aim / cnt - 1) >> 1;
  q = q < 0 ? 0 : (q > 7 ? 7 : q);
  for (int attempt = 0; attempt < 3; ++attempt) {
    float p = s[0];
#pragma unroll
    for (int u = 1; u < 8; ++u)
      if (u == q) p = s[u];
    const int n = count_ge(c, cnt, p);
    if (n >= k && n <= tmax) {
      cnt = compact_ge(c, cnt, p);
      thr = fmaxf(thr, p);
      return true;
    }
    if (n < k) {
      if (q == 7) return false;
      ++q;
    } else {
      if (q == 0) return false;
      --q;
    }
  }
  return false;
}

// Warp-wide room making, run at a convergent point whenever any lane of the warp
// has more than tmax candidates: every lane holding more than lo = (k + tmax)/2
// shrinks at the same time (one pivot round for the whole warp instead of one per
// lane, and the lanes' fill levels stay in step).  Lanes above tmax are brought
// to at most tmax in every case; the row's top k is never dropped.
__device__ __forceinline__ void shrink_warp(const Col& c, int& cnt, float& thr, int k, int tmax) {
  const int lo = (k + tmax) >> 1;
  if (cnt > lo) {
    if (!pivot_round(c, cnt, thr, k, k + ((tmax - k) >> 3), lo) && cnt > tmax)
      while (cnt > tmax) remove_worst(c, cnt, thr);
  }
}

// Exactly the k best (or all, if fewer).
__device__ __forceinline__ void finalize(const Col& c, int& cnt, float& thr, int k) {
  for (int guard = 0; cnt - k > 12 && guard < 4; ++guard)
    if (!pivot_round(c, cnt, thr, k, k + 4, cnt - 1)) break;
  while (cnt > k) remove_worst(c, cnt, thr);
}

// 16 scores of one row (register offset OFF of a 32-score load): mask the keys
// the row cannot see and append the ones above thr (lanes diverge here).
template <int OFF>
__device__ __forceinline__ void append16(const uint32_t (&r)[32], int j0, int vis, const Col& c, int& cnt,
                                         float thr) {
  float v[16];
#pragma unroll
  for (int u = 0; u < 16; ++u) v[u] = __uint_as_float(r[OFF + u]);
  if (j0 + 16 > vis) {
#pragma unroll
    for (int u = 0; u < 16; ++u)
      if (j0 + u >= vis) v[u] = -INFINITY;
  }
  const float m = fmaxf(fmax3(fmax3(v[0], v[1], v[2]), fmax3(v[3], v[4], v[5]), fmax3(v[6], v[7], v[8])),
                        fmax3(fmax3(v[9], v[10], v[11]), fmax3(v[12], v[13], v[14]), v[15]));
  if (m > thr) {
    // branch-free: write every key at the next free slot, advance only past
    // the ones above thr (the slot stays in bounds: cnt <= CAP - 16 on entry)
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      c.put(cnt, v[u], j0 + u);
      cnt += v[u] > thr ? 1 : 0;
    }
  }
}

// 32 scores of one row; the capacity check runs with the whole warp converged.
template <int CAP>
__device__ __forceinline__ void take32(const uint32_t (&r)[32], int j0, int vis, const Col& c, int& cnt, float& thr,
                                       int k) {
  append16<0>(r, j0, vis, c, cnt, thr);
  if (__any_sync(0xffffffffu, cnt > CAP - 16)) shrink_warp(c, cnt, thr, k, CAP - 16);
  append16<16>(r, j0 + 16, vis, c, cnt, thr);
  if (__any_sync(0xffffffffu, cnt > CAP - 16)) shrink_warp(c, cnt, thr, k, CAP - 16);
}

template <int P>
__device__ __forceinline__ void store_a_chunk(uint8_t* sA, int part, int m, int c8, uint4 val) {
  using C = TcCfg<P>;
  uint32_t off;
  if constexpr (P == 128) {
    const int kb = c8 >> 3, ch = c8 & 7;
    off = part * C::A_PART + kb * 16384 + m * 128 + ((ch ^ (m & 7)) << 4);
  } else {
    constexpr int RB = 2 * P;
    const int sw = P == 64 ? (m & 7) : (P == 32 ? ((m >> 1) & 3) : ((m >> 2) & 1));
    off = part * C::A_PART + m * RB + ((c8 ^ sw) << 4);
  }
  *reinterpret_cast<uint4*>(sA + off) = val;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo_elem, float hi_elem) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo_elem, hi_elem);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Epilogue: read the projection (P fp32 columns of this row), split u = hi + lo
// into the two bf16 A-operand matrices.
template <int P>
__device__ __forceinline__ void convert_projection(uint32_t taddr, uint8_t* sA, int m) {
#pragma unroll
  for (int c0 = 0; c0 < P; c0 += 16) {
    uint32_t r[16];
    __syncwarp();
    tc::tmem_ld16(taddr + c0, r);
    tc::tmem_ld_wait();
#pragma unroll
    for (int h8 = 0; h8 < 2; ++h8) {
      uint32_t hw[4], lw[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float u0 = __uint_as_float(r[h8 * 8 + 2 * e]), u1 = __uint_as_float(r[h8 * 8 + 2 * e + 1]);
        const float h0 = __bfloat162float(__float2bfloat16_rn(u0)), h1 = __bfloat162float(__float2bfloat16_rn(u1));
        hw[e] = pack_bf16(h0, h1);
        lw[e] = pack_bf16(u0 - h0, u1 - h1);
      }
      const int c8 = (c0 >> 3) + h8;
      store_a_chunk<P>(sA, 0, m, c8, make_uint4(hw[0], hw[1], hw[2], hw[3]));
      store_a_chunk<P>(sA, 1, m, c8, make_uint4(lw[0], lw[1], lw[2], lw[3]));
    }
  }
}

__device__ __forceinline__ bool wait_noabort(uint64_t* bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity))
    if (clock64() - t0 > tc::kWaitCycles) return false;
  return true;
}

template <int P>
__global__ void __launch_bounds__(192, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmW,
                    const __grid_constant__ CUtensorMap tmX, const TcArgs a) {
  using C = TcCfg<P>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // align by pointer arithmetic on the shared array, so the compiler keeps
  // treating every derived pointer as shared memory
  uint8_t* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* sA = smem;
  uint8_t* sStage = smem + C::OFF_STAGE;
  float* bs = reinterpret_cast<float*>(smem + C::OFF_CAND);
  uint16_t* bi = reinterpret_cast<uint16_t*>(smem + C::OFF_CAND + C::CAP * kLdc * 4);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + C::STAGES;
  uint64_t* accf = empty + C::STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* qfull = acce + 2;
  uint64_t* afree = qfull + 1;
  uint64_t* aready = afree + 1;
  uint64_t* drain = aready + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_f = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      tc::mbar_init(full + s, 1);
      tc::mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(accf + b, 1);
      tc::mbar_init(acce + b, 128);
    }
    tc::mbar_init(qfull, 1);
    tc::mbar_init(afree, 1);
    tc::mbar_init(aready, 128);
    tc::mbar_init(drain, 1);
    *abort_f = 0;
    tc::fence_barrier_init();
  }
  if (warp == 1) {
    tc::tmem_alloc(tmem_slot, C::TMEM_COLS);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *tmem_slot;
  const int Hq = a.Hq;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tc::prefetch_tmap(&tmQ);
      tc::prefetch_tmap(&tmW);
      tc::prefetch_tmap(&tmX);
      uint32_t sc = 0;
      int it = 0, q_issued = 0;
      for (int item = blockIdx.x; item < a.n_items; item += gridDim.x, ++it) {
        const TcTile t = a.tiles[item / Hq];
        const int h = item % Hq;
        if (it > 0 && !tc::mbar_wait(afree, (it - 1) & 1, abort_f)) break;
        tc::mbar_arrive_expect_tx(qfull, 32768);
        ++q_issued;
        const int qrow = (int)((int64_t)h * a.T + t.q0);
        tc::tma_load_2d(sA, &tmQ, qfull, 0, qrow);
        tc::tma_load_2d(sA + 16384, &tmQ, qfull, 64, qrow);
        bool ok = true;
        for (int s3 = 0; s3 < 3 && ok; ++s3)
          for (int kh = 0; kh < 2 && ok; ++kh) {
            const int st = sc % C::STAGES;
            if (!(ok = tc::mbar_wait(empty + st, ((sc / C::STAGES) & 1) ^ 1, abort_f))) break;
            tc::mbar_arrive_expect_tx(full + st, P * 128);
            tc::tma_load_2d(sStage + st * C::STAGE_BYTES, &tmW, full + st, kh * 64, (h * 3 + s3) * P);
            ++sc;
          }
        if (!ok) break;
        const int ntiles = (t.vis_max + C::NT - 1) / C::NT;
        const int64_t xrow = (int64_t)(a.exact ? h / a.G : h) * a.N + t.key_base;
        for (int i = 0; i < ntiles; ++i) {
          const int st = sc % C::STAGES;
          if (!(ok = tc::mbar_wait(empty + st, ((sc / C::STAGES) & 1) ^ 1, abort_f))) break;
          tc::mbar_arrive_expect_tx(full + st, C::STAGE_BYTES);
#pragma unroll
          for (int kb = 0; kb < C::KB; ++kb)
            tc::tma_load_2d(sStage + st * C::STAGE_BYTES + kb * (C::NT * 128), &tmX, full + st, kb * 64,
                            (int)(xrow + (int64_t)i * C::NT));
          ++sc;
        }
        if (!ok) break;
      }
      // every issued load has landed before the CTA may exit
      for (int s = 0; s < C::STAGES; ++s) {
        if ((uint32_t)s >= sc) break;
        const uint32_t last = s + C::STAGES * ((sc - 1 - s) / C::STAGES);
        if (!wait_noabort(full + s, (last / C::STAGES) & 1)) *abort_f = 1;
      }
      if (q_issued > 0 && !wait_noabort(qfull, (q_issued - 1) & 1)) *abort_f = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t sc = 0, ac = 0;
      int it = 0;
      constexpr uint32_t idP = tc::idesc_bf16(128, P);
      constexpr uint32_t idN = tc::idesc_bf16(128, C::NT);
      const uint32_t aBase = tc::smem_u32(sA), sBase = tc::smem_u32(sStage);
      for (int item = blockIdx.x; item < a.n_items; item += gridDim.x, ++it) {
        const TcTile t = a.tiles[item / Hq];
        if (!tc::mbar_wait(qfull, it & 1, abort_f)) break;
        uint32_t buf = ac & 1;
        if (!tc::mbar_wait(acce + buf, ((ac >> 1) & 1) ^ 1, abort_f)) break;
        tc::fence_after_sync();
        bool ok = true;
        uint32_t acc = 0;
        for (int s3 = 0; s3 < 3 && ok; ++s3)
          for (int kh = 0; kh < 2; ++kh) {
            const int st = sc % C::STAGES;
            if (!(ok = tc::mbar_wait(full + st, (sc / C::STAGES) & 1, abort_f))) break;
            tc::fence_after_sync();
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              tc::mma_bf16(tmem + buf * C::NT, tc::sdesc(aBase + kh * 16384 + kk * 32, 1024, 2),
                           tc::sdesc(sBase + st * C::STAGE_BYTES + kk * 32, 1024, 2), idP, acc);
              acc = 1;
            }
            tc::mma_commit(empty + st);
            ++sc;
          }
        if (!ok) break;
        tc::mma_commit(accf + buf);
        ++ac;
        if (!tc::mbar_wait(aready, it & 1, abort_f)) break;
        tc::fence_after_sync();
        const int ntiles = (t.vis_max + C::NT - 1) / C::NT;
        for (int i = 0; i < ntiles; ++i) {
          buf = ac & 1;
          if (!(ok = tc::mbar_wait(acce + buf, ((ac >> 1) & 1) ^ 1, abort_f))) break;
          const int st = sc % C::STAGES;
          if (!(ok = tc::mbar_wait(full + st, (sc / C::STAGES) & 1, abort_f))) break;
          tc::fence_after_sync();
          uint32_t accum = 0;
#pragma unroll
          for (int part = 0; part < 2; ++part)
#pragma unroll
            for (int kb = 0; kb < C::KB; ++kb)
#pragma unroll
              for (int kk = 0; kk < C::KK; ++kk) {
                const uint32_t ad = aBase + part * C::A_PART + kb * 16384 + kk * 32;
                const uint32_t bd = sBase + st * C::STAGE_BYTES + kb * (C::NT * 128) + kk * 32;
                tc::mma_bf16(tmem + buf * C::NT, tc::sdesc(ad, C::SBO, C::SW), tc::sdesc(bd, C::SBO, C::SW), idN,
                             accum);
                accum = 1;
              }
          tc::mma_commit(empty + st);
          tc::mma_commit(accf + buf);
          ++sc;
          ++ac;
        }
        if (!ok) break;
        tc::mma_commit(afree);
      }
      tc::mma_commit(drain);
      if (!wait_noabort(drain, 0)) *abort_f = 1;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;
    const int m = quarter * 32 + lane;
    const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
    const Col col{bs, bi, m};
    uint32_t ac = 0;
    int it = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < a.n_items && ok; item += gridDim.x, ++it) {
      const TcTile t = a.tiles[item / Hq];
      const int h = item % Hq;
      if (it == 0) {  // this item's projection (later items convert theirs ahead of time)
        const uint32_t buf = ac & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(accf + buf, (ac >> 1) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
        convert_projection<P>(tl + buf * C::NT, sA, m);
        tc::fence_before_sync();
        tc::mbar_arrive(acce + buf);
        ++ac;
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(aready);
      }
      const int vis = m < t.nrows ? a.vis[t.q0 + m] : 0;
      int cnt = 0;
      float thr = -INFINITY;
      const int ntiles = (t.vis_max + C::NT - 1) / C::NT;
      for (int i = 0; i < ntiles; ++i) {
        const uint32_t buf = ac & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(accf + buf, (ac >> 1) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
#pragma unroll 1
        for (int c = 0; c < C::NT / 32; ++c) {
          uint32_t r[32];
          __syncwarp();
          tc::tmem_ld32(tl + buf * C::NT + c * 32, r);
          tc::tmem_ld_wait();
          if (c == C::NT / 32 - 1) {
            tc::fence_before_sync();
            tc::mbar_arrive(acce + buf);
          }
          const int j0 = i * C::NT + c * 32;
          take32<C::CAP>(r, j0, vis, col, cnt, thr, a.k);
        }
        ++ac;
      }
      if (!ok) break;
      // convert the next item's projection now, so the tensor core can move on
      const int nxt = item + gridDim.x;
      if (nxt < a.n_items) {
        const uint32_t buf = ac & 1;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(accf + buf, (ac >> 1) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
        convert_projection<P>(tl + buf * C::NT, sA, m);
        tc::fence_before_sync();
        tc::mbar_arrive(acce + buf);
        ++ac;
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(aready);
      }
      finalize(col, cnt, thr, a.k);
      // coalesced output: the warp writes its 32 rows one after another
      __syncwarp();
      for (int rr = 0; rr < 32; ++rr) {
        const int row = quarter * 32 + rr;
        const int n = __shfl_sync(0xffffffffu, cnt, rr);
        if (row >= t.nrows) continue;
        const int64_t o = ((int64_t)h * a.T + t.q0 + row) * a.k;
        const float qn = a.qnu ? a.qnu[(int64_t)h * a.T + t.q0 + row] : 0.f;
        if (a.sorted) {
          uint64_t v[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int i = e * 32 + lane;
            v[e] = i < n ? make_key(bs[i * kLdc + row], (uint32_t)bi[i * kLdc + row]) : 0ull;
          }
          warp_sort_desc<2>(v);
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int i = e * 32 + lane;
            if (i < a.k) {
              a.idx[o + i] = key_index(v[e]);
              if (a.score) a.score[o + i] = v[e] ? key_score(v[e]) + qn : -INFINITY;
            }
          }
        } else {
          for (int i = lane; i < a.k; i += 32) {
            a.idx[o + i] = i < n ? bi[i * kLdc + row] : -1;
            if (a.score) a.score[o + i] = i < n ? bs[i * kLdc + row] + qn : -INFINITY;
          }
        }
      }
      __syncwarp();
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (*abort_f && threadIdx.x == 0) atomicOr(a.err, 1);
  if (warp == 1) tc::tmem_dealloc(tmem, C::TMEM_COLS);
}

// W [Hq][d][P] fp32 -> [Hq][3][P][d] bf16 with W = w0 + w1 + w2 exactly
__global__ void pack_w_kernel(const float* W, int Hq, int P, __nv_bfloat16* out) {
  const int64_t n = (int64_t)Hq * P * kD;
  for (int64_t o = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; o < n; o += (int64_t)gridDim.x * blockDim.x) {
    const int i = (int)(o % kD);
    const int p = (int)((o / kD) % P);
    const int h = (int)(o / ((int64_t)kD * P));
    const float w = W[((int64_t)h * kD + i) * P + p];
    const __nv_bfloat16 w0 = __float2bfloat16_rn(w);
    const float r1 = w - __bfloat162float(w0);
    const __nv_bfloat16 w1 = __float2bfloat16_rn(r1);
    const __nv_bfloat16 w2 = __float2bfloat16_rn(r1 - __bfloat162float(w1));
    const int64_t base = (((int64_t)h * 3) * P + p) * kD + i;
    out[base] = w0;
    out[base + (int64_t)P * kD] = w1;
    out[base + 2 * (int64_t)P * kD] = w2;
  }
}

// q^T nu per (head, query)
__global__ void qnu_kernel(const __nv_bfloat16* Q, const float* nu, int64_t T, int Hq, float* out) {
  const int lane = threadIdx.x & 31;
  const int64_t rowi = blockIdx.x * (int64_t)(blockDim.x / 32) + (threadIdx.x >> 5);
  if (rowi >= (int64_t)Hq * T) return;
  const int h = (int)(rowi / T);
  float v = 0.f;
  for (int i = lane; i < kD; i += 32) v = fmaf(__bfloat162float(Q[rowi * kD + i]), nu[(int64_t)h * kD + i], v);
  v = warp_sum(v);
  if (lane == 0) out[rowi] = v;
}

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

bool make_map(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t rows, uint32_t box_inner, uint32_t box_rows,
              CUtensorMapSwizzle sw) {
  auto enc = encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

CUtensorMapSwizzle swz_of(int kw) {
  return kw == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : (kw == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B);
}

template <int P>
cudaError_t launch_tc_t(const TcLaunch& L, cudaStream_t s) {
  using C = TcCfg<P>;
  CUtensorMap mQ, mW, mX;
  const int xrows_heads = L.args.exact ? L.Hk : L.args.Hq;
  const int xcols = L.args.exact ? kD : P;
  if (!make_map(&mQ, L.Q, kD, (uint64_t)L.args.Hq * L.args.T, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&mW, L.Wsplit, kD, (uint64_t)L.args.Hq * 3 * P, 64, P, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map(&mX, L.X, xcols, (uint64_t)xrows_heads * L.args.N, C::KW, C::NT, swz_of(C::KW)))
    return cudaErrorInvalidValue;
  auto kern = score_tc_kernel<P>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int grid = L.args.n_items < L.num_sms ? L.args.n_items : L.num_sms;
  kern<<<grid, 192, C::SMEM, s>>>(mQ, mW, mX, L.args);
  return cudaGetLastError();
}
}  // namespace

bool tc_supported(int P) { return P == 16 || P == 32 || P == 64 || P == 128; }

cudaError_t launch_pack_w(const float* W, int Hq, int P, void* out, cudaStream_t s) {
  const int64_t n = (int64_t)Hq * P * kD;
  const int blocks = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  pack_w_kernel<<<blocks, 256, 0, s>>>(W, Hq, P, static_cast<__nv_bfloat16*>(out));
  return cudaGetLastError();
}

cudaError_t launch_qnu(const void* Q, const float* nu, int64_t T, int Hq, float* out, cudaStream_t s) {
  const int64_t rows = (int64_t)Hq * T;
  qnu_kernel<<<(unsigned)((rows + 7) / 8), 256, 0, s>>>(static_cast<const __nv_bfloat16*>(Q), nu, T, Hq, out);
  return cudaGetLastError();
}

cudaError_t launch_score_tc(const TcLaunch& L, cudaStream_t s) {
  if (L.args.n_items == 0) return cudaSuccess;
  switch (L.P) {
    case 16: return launch_tc_t<16>(L, s);
    case 32: return launch_tc_t<32>(L, s);
    case 64: return launch_tc_t<64>(L, s);
    case 128: return launch_tc_t<128>(L, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace saki
