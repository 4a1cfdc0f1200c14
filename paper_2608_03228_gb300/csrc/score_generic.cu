// Generic fused score + top-k on CUDA cores (any rank, f32 or bf16 inputs).
//
// Serves the decode-shaped work of the selection step (Sec. 6: s_hat = (L^T q)^T c_j
// over the visible keys, keep the k largest) and, with W = A and X = K, the
// exact top-k of the Sec. 3 recall protocol.  A work item is up to kGroupQ
// queries of one sequence against one split of its keys; each lane scores one
// key for all queries of the group from 128-bit loads, so every key row is read
// once per item.  Selection never forms the score matrix: each warp keeps, per
// query, a shared-memory buffer of candidates above its running k-th best key
// and re-selects (warp bitonic sort) when the buffer fills; warps are merged at
// the end, and splits of a long sequence by a second small kernel.
//
// score_decode_tc_kernel runs the same work items with the scores from the
// tensor core (bf16 keys or codes): see its comment.
#include <atomic>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"
#include "tmap.cuh"

namespace saki {

namespace {
constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;

template <typename T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

// Keep the KP best of the warp's buffer of CAP slots (sorted, descending) and
// return the k-th best key (0 while fewer than k are held).
template <int KP, int CAP = 2 * KP>
__device__ __forceinline__ uint64_t reselect(uint64_t* qb, int& cnt, int k) {
  constexpr int E = CAP / 32;
  const int lane = threadIdx.x & 31;
  __syncwarp();
  uint64_t v[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = e * 32 + lane;
    v[e] = i < cnt ? qb[i] : 0ull;
  }
  warp_sort_desc<E>(v);
  __syncwarp();
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int i = e * 32 + lane;
    if (i < KP) qb[i] = v[e];
  }
  cnt = cnt < KP ? cnt : KP;
  uint64_t t = 0;
  const int ke = (k - 1) >> 5;
#pragma unroll
  for (int e = 0; e < E; ++e)
    if (e == ke) t = v[e];
  t = shfl_u64(t, (k - 1) & 31);
  __syncwarp();
  return cnt >= k ? t : 0ull;
}

// Rare path, kept out of line: append the passing keys of this 32-key batch to
// the warp's buffer of one query, re-select when it is nearly full, publish the
// warp's k-th best as a CTA-wide lower bound, and return the new threshold.
template <int KP, int CAP = 2 * KP>
__device__ __noinline__ uint64_t append_keys(uint64_t* qb, int* cnt_s, unsigned long long* cta_thr, uint64_t key,
                                             bool pass, unsigned mask, uint64_t thr, int k) {
  const int lane = threadIdx.x & 31;
  int cnt = *cnt_s;
  if (pass) qb[cnt + __popc(mask & ((1u << lane) - 1u))] = key;
  cnt += __popc(mask);
  if (cnt > CAP - 32) {
    const uint64_t t = reselect<KP, CAP>(qb, cnt, k);
    if (t > thr) thr = t;
    if (lane == 0 && t) atomicMax(cta_thr, (unsigned long long)t);
  }
  __syncwarp();
  if (lane == 0) *cnt_s = cnt;
  __syncwarp();
  const uint64_t c = *cta_thr;
  return c > thr ? c : thr;
}

// Packed fp32x2 fused multiply-add: (acc.x, acc.y) += (a.x, a.y) * (b.x, b.y).
__device__ __forceinline__ void ffma2(unsigned long long& acc, unsigned long long x, unsigned long long y) {
  asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(acc) : "l"(x), "l"(y));
}
__device__ __forceinline__ unsigned long long pk2(float lo, float hi) {
  return ((unsigned long long)__float_as_uint(hi) << 32) | __float_as_uint(lo);
}
__device__ __forceinline__ float sum2(unsigned long long v) {
  return __uint_as_float((uint32_t)v) + __uint_as_float((uint32_t)(v >> 32));
}

// NQ: compile-time width of the query group (1, 2, 4 or 8); the host launches the
// smallest width that holds every group of the call.
template <typename Tin, int KP, int NQ>
__global__ void __launch_bounds__(kThreads) score_generic_kernel(const ScoreArgs a) {
  constexpr int CAP = 2 * KP;
  constexpr int EK = KP / 32;
  constexpr int NV = Vec<Tin>::NV;
  constexpr int kGroupQ = NQ;
  extern __shared__ __align__(16) unsigned char smem[];
  uint64_t* buf = reinterpret_cast<uint64_t*>(smem);                       // [warps][GQ][CAP]
  float* qs = reinterpret_cast<float*>(buf + kWarps * kGroupQ * CAP);      // [GQ][d]
  float* us = qs + kGroupQ * kD;                                           // [GQ][P]
  float* qnu = us + kGroupQ * a.P;                                         // [GQ]
  int* visq = reinterpret_cast<int*>(qnu + kGroupQ);                       // [GQ]
  int* cnt_s = visq + kGroupQ;                                             // [warps][GQ]
  __shared__ unsigned long long cta_thr[kGroupQ];

  // one CTA per (item, query head), the heads of an item adjacent: the G
  // heads of a KV group then stream the same key tiles together (the exact
  // scores read a KV head's keys once from DRAM, the others hit L2)
  const ScoreItem it = a.items[blockIdx.x / a.Hq];
  const int h = (int)(blockIdx.x % a.Hq);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int P = a.P;
  const int nq = it.q_count;

  const Tin* Q = static_cast<const Tin*>(a.Q);
  for (int o = tid; o < kGroupQ * kD; o += kThreads) {
    const int b = o / kD;
    qs[o] = b < nq ? to_f<Tin>(Q[((int64_t)h * a.T + it.q_begin + b) * kD + (o % kD)]) : 0.f;
  }
  if (tid < kGroupQ) {
    visq[tid] = tid < nq ? a.vis[it.q_begin + tid] : 0;
    cta_thr[tid] = 0ull;
  }
  if (tid < kWarps * kGroupQ) cnt_s[tid] = 0;
  for (int o = tid; o < kWarps * kGroupQ * CAP; o += kThreads) buf[o] = 0ull;
  __syncthreads();

  // u_b = W_h^T q_b (fp32), and the mean term q_b^T nu_h
  const float* W = a.W + (int64_t)h * kD * P;
  for (int o = tid; o < kGroupQ * P; o += kThreads) {
    const int b = o / P, p = o % P;
    float acc = 0.f;
    for (int i = 0; i < kD; ++i) acc = fmaf(__ldg(W + i * P + p), qs[b * kD + i], acc);
    us[o] = acc;
  }
  if (warp < kGroupQ) {
    float v = 0.f;
    if (a.nu)
      for (int i = lane; i < kD; i += 32) v = fmaf(qs[warp * kD + i], __ldg(a.nu + (int64_t)h * kD + i), v);
    v = warp_sum(v);
    if (lane == 0) qnu[warp] = v;
  }
  __syncthreads();

  const Tin* X = static_cast<const Tin*>(a.X) +
                 ((int64_t)(a.exact ? h / a.G : h) * a.N + it.key_base) * P;
  uint64_t thr[kGroupQ];
  float thr_f[kGroupQ];   // score part of thr: a key can only pass if its score is >= thr_f
#pragma unroll
  for (int b = 0; b < kGroupQ; ++b) { thr[b] = 0ull; thr_f[b] = -INFINITY; }
  uint64_t* wbuf = buf + warp * kGroupQ * CAP;
  int* wcnt = cnt_s + warp * kGroupQ;
  const int nkeys = it.key_hi - it.key_lo;
  const bool vec = ((P * (int)sizeof(Tin)) % 16) == 0;

  for (int base = warp * 32; base < nkeys; base += kThreads) {
    const int jl = base + lane;
    const int j = it.key_lo + jl;
    float acc[kGroupQ];
#pragma unroll
    for (int b = 0; b < kGroupQ; ++b) acc[b] = 0.f;
    if (jl < nkeys) {
      const Tin* row = X + (int64_t)j * P;
      if (vec) {
        unsigned long long a2[kGroupQ];
#pragma unroll
        for (int b = 0; b < kGroupQ; ++b) a2[b] = 0ull;
        const uint4* r4 = reinterpret_cast<const uint4*>(row);
        const int nv = P / NV;
        for (int v = 0; v < nv; ++v) {
          const uint4 raw = __ldg(r4 + v);
          float x[NV];
          Vec<Tin>::unpack(raw, x);
#pragma unroll
          for (int b = 0; b < kGroupQ; ++b) {
            const ulonglong2* u2 = reinterpret_cast<const ulonglong2*>(us + b * P + v * NV);
#pragma unroll
            for (int e4 = 0; e4 < NV / 4; ++e4) {
              const ulonglong2 uu = u2[e4];
              ffma2(a2[b], uu.x, pk2(x[4 * e4 + 0], x[4 * e4 + 1]));
              ffma2(a2[b], uu.y, pk2(x[4 * e4 + 2], x[4 * e4 + 3]));
            }
          }
        }
#pragma unroll
        for (int b = 0; b < kGroupQ; ++b) acc[b] = sum2(a2[b]);
      } else {
        for (int p = 0; p < P; ++p) {
          const float x = to_f<Tin>(row[p]);
#pragma unroll
          for (int b = 0; b < kGroupQ; ++b) acc[b] = fmaf(us[b * P + p], x, acc[b]);
        }
      }
    }
#pragma unroll
    for (int b = 0; b < kGroupQ; ++b) {
      if (b < nq) {
        const bool ok = (jl < nkeys) && (j < visq[b]) && acc[b] >= thr_f[b];
        if (__ballot_sync(0xffffffffu, ok)) {
          const uint64_t key = make_key(acc[b], (uint32_t)j);
          const bool pass = ok && key > thr[b];
          const unsigned mask = __ballot_sync(0xffffffffu, pass);
          if (mask) {
            thr[b] = append_keys<KP>(wbuf + b * CAP, wcnt + b, cta_thr + b, key, pass, mask, thr[b], a.k);
            thr_f[b] = key_score(thr[b]);
          }
        }
      }
    }
  }
  for (int b = 0; b < nq; ++b) {
    int c = wcnt[b];
    reselect<KP>(wbuf + b * CAP, c, a.k);
  }
  __syncthreads();

  // merge the warps' lists of query `warp`
  if (warp < nq) {
    const int b = warp;
    uint64_t best[EK], other[EK];
#pragma unroll
    for (int e = 0; e < EK; ++e) best[e] = buf[(0 * kGroupQ + b) * CAP + e * 32 + lane];
    for (int w2 = 1; w2 < kWarps; ++w2) {
#pragma unroll
      for (int e = 0; e < EK; ++e) other[e] = buf[(w2 * kGroupQ + b) * CAP + e * 32 + lane];
      warp_merge_top<EK>(best, other);
    }
    if (it.cand < 0) {
      const int64_t row = ((int64_t)h * a.T + it.q_begin + b) * a.k;
#pragma unroll
      for (int e = 0; e < EK; ++e) {
        const int i = e * 32 + lane;
        if (i < a.k) {
          a.idx[row + i] = key_index(best[e]);
          if (a.score) a.score[row + i] = best[e] ? key_score(best[e]) + qnu[b] : -INFINITY;
        }
      }
    } else {
      uint64_t* c = a.cand + ((int64_t)h * a.cand_per_head + it.cand + (int64_t)b * it.cand_stride) * KP;
#pragma unroll
      for (int e = 0; e < EK; ++e) c[e * 32 + lane] = best[e];
    }
  }
}

// The merge of a row's per-split lists (each sorted, striped over a warp): the
// block's four warps each merge every fourth split, the next split's keys
// loaded while the current one is merged (a global load per split would
// otherwise sit on the critical path, split after split), and warp 0 merges
// the other three warps' lists in through shared memory.
template <typename Tin, int KP>
__global__ void __launch_bounds__(128) merge_kernel(const ScoreArgs a) {
  constexpr int EK = KP / 32;
  __shared__ uint64_t part[3][KP];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int m = blockIdx.x;
  const int h = blockIdx.y;
  const MergeItem mi = a.merges[m];
  const uint64_t* c = a.cand + ((int64_t)h * a.cand_per_head + mi.cand) * KP;
  uint64_t best[EK], nxt[EK], cur[EK];
  int sp = warp;
#pragma unroll
  for (int e = 0; e < EK; ++e) best[e] = sp < mi.nsplit ? c[(int64_t)sp * KP + e * 32 + lane] : 0ull;
  sp += 4;
#pragma unroll
  for (int e = 0; e < EK; ++e) nxt[e] = sp < mi.nsplit ? c[(int64_t)sp * KP + e * 32 + lane] : 0ull;
  while (sp < mi.nsplit) {
    const int sn = sp + 4;
#pragma unroll
    for (int e = 0; e < EK; ++e) {
      cur[e] = nxt[e];
      nxt[e] = sn < mi.nsplit ? c[(int64_t)sn * KP + e * 32 + lane] : 0ull;
    }
    warp_merge_top<EK>(best, cur);
    sp = sn;
  }
  if (warp > 0) {
#pragma unroll
    for (int e = 0; e < EK; ++e) part[warp - 1][e * 32 + lane] = best[e];
  }
  __syncthreads();
  if (warp > 0) return;
  for (int j = 0; j < 3; ++j) {
#pragma unroll
    for (int e = 0; e < EK; ++e) cur[e] = part[j][e * 32 + lane];
    warp_merge_top<EK>(best, cur);
  }
  if (a.seed_out) {
    // the row's k-th best key over the merged lists (0 while fewer than k)
    uint64_t t = 0;
#pragma unroll
    for (int e = 0; e < EK; ++e)
      if (e == (a.k - 1) >> 5) t = best[e];
    t = shfl_u64(t, (a.k - 1) & 31);
    if (lane == 0) a.seed_out[(int64_t)h * a.T + mi.t] = t;
    return;
  }
  float qnu = 0.f;
  if (a.nu) {
    const Tin* q = static_cast<const Tin*>(a.Q) + ((int64_t)h * a.T + mi.t) * kD;
    for (int i = lane; i < kD; i += 32) qnu = fmaf(to_f<Tin>(q[i]), __ldg(a.nu + (int64_t)h * kD + i), qnu);
    qnu = warp_sum(qnu);
  }
  const int64_t row = ((int64_t)h * a.T + mi.t) * a.k;
#pragma unroll
  for (int e = 0; e < EK; ++e) {
    const int i = e * 32 + lane;
    if (i < a.k) {
      a.idx[row + i] = key_index(best[e]);
      if (a.score) a.score[row + i] = best[e] ? key_score(best[e]) + qnu : -INFINITY;
    }
  }
}

// ---------------------------------------------------------------- tensor-core variant
// The work items of score_generic_kernel (up to kGroupQ queries of one sequence
// against one split of its keys) with the scores on the tensor core: tiles of
// 128 keys (codes, or keys for the exact scores) are the A operand (M = 128,
// TMA), u = W^T q of the group's queries split into bf16 hi + lo the B operand
// (N = 16, rows past the group zero), D[key][query] in a ring of TMEM
// accumulators.  Each epilogue thread reads one key's scores for all queries (its
// TMEM lane) into registers and compares them with its warp's running k-th best
// of each query (score_generic_kernel's candidate buffer and re-selection, one
// buffer per warp and query), one warp vote per tile for all queries; the four
// warps' lists of a query are merged at the end.  A seeded item starts every
// threshold at the row's seed, so after the first few keys almost no key is
// appended.  With ScoreArgs::sample set, the kernel keeps per query the best
// score each thread sees (a group maximum over the split) and writes the kp
// largest of the CTA's 128 group maxima, from which the seeds are merged.
// Roles: warp 0 TMA producer, warp 1 TMEM owner and MMA issuer, warps 2-5
// projection and selection.  Every mbarrier wait is bounded; a CTA that gives
// up sets kStTimeout in the error word.
template <int P>
struct DcCfg {
  static constexpr int KW = P == 128 ? 64 : P;   // K width of one swizzled block
  static constexpr int KB = P / KW;
  static constexpr int KK = KW / 16;
  static constexpr uint32_t SW = KW == 64 ? 2u : (KW == 32 ? 4u : 6u);
  static constexpr uint32_t SBO = 8 * KW * 2;
  static constexpr int NT = 128;                 // keys per tile (MMA M)
  static constexpr int NQ = 16;                  // queries per MMA (N), the group zero-padded
  static constexpr int NB = 8;                   // TMEM ring of NQ-column accumulators
  static constexpr int STAGES = P == 128 ? 3 : 4;
  static constexpr int STAGE_BYTES = NT * P * 2;
  static constexpr int U_PART = (NQ * P * 2 + 1023) & ~1023;   // u_hi or u_lo
  static constexpr int OFF_U = STAGES * STAGE_BYTES;
  static constexpr int OFF_BUF = OFF_U + 2 * U_PART;
  static constexpr int cap(int kp) { return 2 * kp; }          // candidate slots per warp and query
  static constexpr int LANES = 4 * 32;                          // group maxima per query in a sample pass
  static int smem(int kp) { return OFF_BUF + 4 * kGroupQ * cap(kp) * 8 + 1024; }   // [4 warps][query][cap]
  static_assert(4 * cap(64) >= LANES, "a sample pass's group maxima fit the candidate buffers");
  static_assert(kGroupQ <= NQ && NQ % 16 == 0, "the group fits the MMA's N");
  static_assert(STAGE_BYTES % 1024 == 0 && OFF_U % 1024 == 0, "swizzled blocks on 1024-byte boundaries");
};

// 16 bytes (8 bf16 of K columns 8 c8 .. 8 c8 + 7) of row n of u's part `part`,
// in the swizzled K-major layout the MMA's B descriptor reads.
template <int P>
__device__ __forceinline__ void store_u_chunk(uint8_t* sU, int part, int n, int c8, uint4 v) {
  using C = DcCfg<P>;
  uint32_t off;
  if constexpr (P == 128) {
    const int kb = c8 >> 3, ch = c8 & 7;
    off = part * C::U_PART + kb * (C::NQ * 128) + n * 128 + ((ch ^ (n & 7)) << 4);
  } else {
    const int sw = P == 64 ? (n & 7) : (P == 32 ? ((n >> 1) & 3) : ((n >> 2) & 1));
    off = part * C::U_PART + n * (2 * P) + ((c8 ^ sw) << 4);
  }
  *reinterpret_cast<uint4*>(sU + off) = v;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo_elem, float hi_elem) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo_elem, hi_elem);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ void epilogue_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

template <int P, int KP>
__global__ void __launch_bounds__(192) score_decode_tc_kernel(const __grid_constant__ CUtensorMap tmX,
                                                              const ScoreArgs a) {
  using C = DcCfg<P>;
  constexpr int CAP = C::cap(KP);
  constexpr int EK = KP / 32;
  constexpr int GQ = kGroupQ;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (tc::smem_u32(smem_raw) & 1023u)) & 1023u);
  uint8_t* sStage = smem;
  uint8_t* sU = smem + C::OFF_U;
  uint64_t* buf = reinterpret_cast<uint64_t*>(smem + C::OFF_BUF);   // [4 warps][GQ][CAP]
  __shared__ float qs[GQ][kD];
  __shared__ float us[GQ][P];
  __shared__ float qnu[GQ];
  __shared__ int visq[GQ];
  __shared__ int cnt_s[4 * GQ];
  __shared__ unsigned long long cta_thr[GQ];
  __shared__ __align__(8) uint64_t bars[2 * C::STAGES + 2 * C::NB + 2];
  __shared__ uint32_t tmem_slot;
  __shared__ int abort_s;
  uint64_t* full = bars;
  uint64_t* empty = full + C::STAGES;
  uint64_t* accf = empty + C::STAGES;
  uint64_t* acce = accf + C::NB;
  uint64_t* uready = acce + C::NB;
  uint64_t* drain = uready + 1;
  volatile int* abort_f = &abort_s;

  // one CTA per (item, query head), the heads of an item adjacent: the G
  // heads of a KV group then stream the same key tiles together (the exact
  // scores read a KV head's keys once from DRAM, the others hit L2)
  const ScoreItem it = a.items[blockIdx.x / a.Hq];
  const int h = (int)(blockIdx.x % a.Hq);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nq = it.q_count;
  const int nkeys = it.key_hi - it.key_lo;
  const int ntiles = (nkeys + C::NT - 1) / C::NT;

  if (threadIdx.x == 0) {
    for (int s2 = 0; s2 < C::STAGES; ++s2) {
      tc::mbar_init(full + s2, 1);
      tc::mbar_init(empty + s2, 1);
    }
    for (int b = 0; b < C::NB; ++b) {
      tc::mbar_init(accf + b, 1);
      tc::mbar_init(acce + b, 128);
    }
    tc::mbar_init(uready, 128);
    tc::mbar_init(drain, 1);
    *abort_f = 0;
    tc::fence_barrier_init();
  }
  if (warp == 1) {
    tc::tmem_alloc(&tmem_slot, C::NB * C::NQ);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tc::prefetch_tmap(&tmX);
      const int64_t xrow = (int64_t)(a.exact ? h / a.G : h) * a.N + it.key_base + it.key_lo;
      int issued = 0;
      for (int i = 0; i < (a.stall ? 0 : ntiles); ++i) {
        const int st = i % C::STAGES;
        if (!tc::mbar_wait(empty + st, ((i / C::STAGES) & 1) ^ 1, abort_f)) break;
        tc::mbar_arrive_expect_tx(full + st, C::STAGE_BYTES);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          tc::tma_load_2d(sStage + st * C::STAGE_BYTES + kb * (C::NT * C::KW * 2), &tmX, full + st, kb * C::KW,
                          (int)(xrow + (int64_t)i * C::NT));
        ++issued;
      }
      // every issued load has landed before the CTA may exit
      for (int s2 = 0; s2 < C::STAGES && s2 < issued; ++s2) {
        const int last = s2 + C::STAGES * ((issued - 1 - s2) / C::STAGES);
        if (!tc::mbar_wait_bounded(full + s2, (last / C::STAGES) & 1)) *abort_f = 1;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = tc::idesc_bf16(C::NT, C::NQ);
      const uint32_t sBase = tc::smem_u32(sStage), uBase = tc::smem_u32(sU);
      bool ok = tc::mbar_wait(uready, 0, abort_f);
      if (ok) tc::fence_after_sync();
      for (int i = 0; ok && i < ntiles; ++i) {
        const int st = i % C::STAGES, b = i % C::NB;
        if (!(ok = tc::mbar_wait(acce + b, ((i / C::NB) & 1) ^ 1, abort_f))) break;
        if (!(ok = tc::mbar_wait(full + st, (i / C::STAGES) & 1, abort_f))) break;
        tc::fence_after_sync();
        uint32_t accum = 0;
#pragma unroll
        for (int part = 0; part < 2; ++part)
#pragma unroll
          for (int kb = 0; kb < C::KB; ++kb)
#pragma unroll
            for (int kk = 0; kk < C::KK; ++kk) {
              const uint32_t ad = sBase + st * C::STAGE_BYTES + kb * (C::NT * C::KW * 2) + kk * 32;
              const uint32_t bd = uBase + part * C::U_PART + kb * (C::NQ * C::KW * 2) + kk * 32;
              tc::mma_bf16(tmem + b * C::NQ, tc::sdesc(ad, C::SBO, C::SW), tc::sdesc(bd, C::SBO, C::SW), idesc,
                           accum);
              accum = 1;
            }
        tc::mma_commit(empty + st);
        tc::mma_commit(accf + b);
      }
      tc::mma_commit(drain);
      if (!tc::mbar_wait_bounded(drain, 0)) *abort_f = 1;
    }
  } else {
    // ------------------------------------------------------------ projection and selection
    const int e = warp - 2;                 // candidate buffers of this warp
    const int quarter = warp & 3;           // the TMEM lanes (keys of a tile) this warp may read
    const int et = threadIdx.x - 64;
    const __nv_bfloat16* Q = static_cast<const __nv_bfloat16*>(a.Q);
    for (int o = et; o < GQ * kD; o += 128) {
      const int b = o / kD;
      qs[b][o % kD] = b < nq ? __bfloat162float(Q[((int64_t)h * a.T + it.q_begin + b) * kD + (o % kD)]) : 0.f;
    }
    if (et < GQ) {
      visq[et] = et < nq ? a.vis[it.q_begin + et] : 0;
      cta_thr[et] = 0ull;
    }
    if (et < 4 * GQ) cnt_s[et] = 0;
    for (int o = et; o < 4 * GQ * CAP; o += 128) buf[o] = 0ull;
    epilogue_sync();
    // u_b = W_h^T q_b (fp32) and the mean term q_b^T nu_h
    const float* W = a.W + (int64_t)h * kD * P;
    for (int o = et; o < GQ * P; o += 128) {
      const int b = o / P, p = o % P;
      float acc = 0.f;
      for (int i = 0; i < kD; ++i) acc = fmaf(__ldg(W + i * P + p), qs[b][i], acc);
      us[b][p] = acc;
    }
    for (int b = e; b < GQ; b += 4) {
      float v = 0.f;
      if (a.nu)
        for (int i = lane; i < kD; i += 32) v = fmaf(qs[b][i], __ldg(a.nu + (int64_t)h * kD + i), v);
      v = warp_sum(v);
      if (lane == 0) qnu[b] = v;
    }
    epilogue_sync();
    // u = u_hi + u_lo in bf16, the MMA's B operand; rows past the group are zero
    for (int o = et; o < C::NQ * (P / 8); o += 128) {
      const int n = o / (P / 8), c8 = o % (P / 8);
      uint32_t hw[4], lw[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float u0 = n < nq ? us[n][8 * c8 + 2 * q] : 0.f, u1 = n < nq ? us[n][8 * c8 + 2 * q + 1] : 0.f;
        const float h0 = __bfloat162float(__float2bfloat16_rn(u0)), h1 = __bfloat162float(__float2bfloat16_rn(u1));
        hw[q] = pack_bf16x2(h0, h1);
        lw[q] = pack_bf16x2(u0 - h0, u1 - h1);
      }
      store_u_chunk<P>(sU, 0, n, c8, make_uint4(hw[0], hw[1], hw[2], hw[3]));
      store_u_chunk<P>(sU, 1, n, c8, make_uint4(lw[0], lw[1], lw[2], lw[3]));
    }
    tc::fence_proxy_async_smem();
    tc::mbar_arrive(uready);

    // Each thread owns one key of every tile (its TMEM lane) and holds that
    // key's scores for all queries of the group in registers: one compare per
    // query against the warp's running threshold and one warp vote per tile.
    const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
    int lim[GQ];   // keys of the split visible to query q (0 past the group)
    int lim_min = nkeys;
#pragma unroll
    for (int q = 0; q < GQ; ++q) {
      lim[q] = q < nq ? max(0, min(nkeys, visq[q] - it.key_lo)) : 0;
      if (q < nq) lim_min = min(lim_min, lim[q]);
    }
    if (a.sample) {
      // Sample pass: per query, the best score each thread sees over the split
      // (a group of up to ntiles keys, one per tile).  The k-th largest group
      // maximum over all splits is reached by k distinct visible keys, so it
      // bounds the row's k-th best score from below.
      float mx[GQ];
#pragma unroll
      for (int q = 0; q < GQ; ++q) mx[q] = -INFINITY;
      for (int i = 0; i < ntiles; ++i) {
        const int b = i % C::NB;
        if (!__all_sync(0xffffffffu, tc::mbar_wait(accf + b, (i / C::NB) & 1, abort_f))) break;
        tc::fence_after_sync();
        uint32_t r[8];
        __syncwarp();
        tc::tmem_ld8(tl + b * C::NQ, r);
        tc::tmem_ld_wait(r);
        tc::fence_before_sync();
        tc::mbar_arrive(acce + b);
        const int jl = i * C::NT + quarter * 32 + lane;
#pragma unroll
        for (int q = 0; q < GQ; ++q)
          if (jl < lim[q]) mx[q] = fmaxf(mx[q], __uint_as_float(r[q]));
      }
      uint64_t* gm = buf;   // [GQ][LANES] group maxima as keys (0: the thread saw no visible key)
#pragma unroll
      for (int q = 0; q < GQ; ++q)
        gm[q * C::LANES + quarter * 32 + lane] =
            mx[q] > -INFINITY ? make_key(mx[q], (uint32_t)(it.key_lo + quarter * 32 + lane)) : 0ull;
      epilogue_sync();
      for (int q = e; q < nq; q += 4) {
        int c = C::LANES;
        reselect<KP, C::LANES>(gm + q * C::LANES, c, a.k);
        uint64_t* c2 = a.cand + ((int64_t)h * a.cand_per_head + it.cand + (int64_t)q * it.cand_stride) * KP;
#pragma unroll
        for (int y = 0; y < EK; ++y) c2[y * 32 + lane] = gm[q * C::LANES + y * 32 + lane];
      }
    } else {
      // a seeded item starts each query at its row's seed score: at least k
      // visible keys of the row score that much, so every key of the row's
      // top k still passes
      uint64_t thr[GQ];
      float thr_f[GQ];   // score part of thr: a key can only pass if its score is >= thr_f
#pragma unroll
      for (int q = 0; q < GQ; ++q) {
        thr[q] = 0ull;
        thr_f[q] = q < nq ? -INFINITY : INFINITY;
        const uint64_t sd = it.seeded && a.seed && q < nq ? a.seed[(int64_t)h * a.T + it.q_begin + q] : 0ull;
        if (sd >> 32) {
          thr[q] = (sd & 0xffffffff00000000ull) - 1ull;
          thr_f[q] = key_score(sd);
        }
      }
      uint64_t* wbuf = buf + e * GQ * CAP;
      int* wcnt = cnt_s + e * GQ;
      for (int i = 0; i < ntiles; ++i) {
        const int b = i % C::NB;
        if (!__all_sync(0xffffffffu, tc::mbar_wait(accf + b, (i / C::NB) & 1, abort_f))) break;
        tc::fence_after_sync();
        uint32_t r[8];
        __syncwarp();
        tc::tmem_ld8(tl + b * C::NQ, r);
        tc::tmem_ld_wait(r);
        tc::fence_before_sync();
        tc::mbar_arrive(acce + b);
        const int jl = i * C::NT + quarter * 32 + lane;
        // one bit per query whose score clears its threshold; one vote for all
        const bool inner = (i + 1) * C::NT <= lim_min;   // every key of the tile visible to every query
        unsigned m = 0u;
#pragma unroll
        for (int q = 0; q < GQ; ++q) {
          const bool ok = __uint_as_float(r[q]) >= thr_f[q] && (inner || jl < lim[q]);
          m |= ok ? 1u << q : 0u;
        }
        const unsigned any = __reduce_or_sync(0xffffffffu, m);
        if (any) {
          const uint32_t j = (uint32_t)(it.key_lo + jl);
#pragma unroll
          for (int q = 0; q < GQ; ++q) {
            if (any & (1u << q)) {
              const uint64_t key = make_key(__uint_as_float(r[q]), j);
              const bool pass = ((m >> q) & 1u) && key > thr[q];
              const unsigned mask = __ballot_sync(0xffffffffu, pass);
              if (mask) {
                thr[q] = append_keys<KP, CAP>(wbuf + q * CAP, wcnt + q, cta_thr + q, key, pass, mask, thr[q], a.k);
                thr_f[q] = key_score(thr[q]);
              }
            }
          }
        }
      }
      for (int q = 0; q < nq; ++q) {
        int c = wcnt[q];
        reselect<KP, CAP>(wbuf + q * CAP, c, a.k);
      }
      epilogue_sync();
      // each query's k best: the four warps' sorted lists merged by one warp
      for (int q = e; q < nq; q += 4) {
        uint64_t best[EK], other[EK];
#pragma unroll
        for (int y = 0; y < EK; ++y) best[y] = buf[q * CAP + y * 32 + lane];
        for (int w2 = 1; w2 < 4; ++w2) {
#pragma unroll
          for (int y = 0; y < EK; ++y) other[y] = buf[(w2 * GQ + q) * CAP + y * 32 + lane];
          warp_merge_top<EK>(best, other);
        }
        if (it.cand < 0) {
          const int64_t row = ((int64_t)h * a.T + it.q_begin + q) * a.k;
#pragma unroll
          for (int y = 0; y < EK; ++y) {
            const int ii = y * 32 + lane;
            if (ii < a.k) {
              a.idx[row + ii] = key_index(best[y]);
              if (a.score) a.score[row + ii] = best[y] ? key_score(best[y]) + qnu[q] : -INFINITY;
            }
          }
        } else {
          uint64_t* c2 = a.cand + ((int64_t)h * a.cand_per_head + it.cand + (int64_t)q * it.cand_stride) * KP;
#pragma unroll
          for (int y = 0; y < EK; ++y) c2[y * 32 + lane] = best[y];
        }
      }
    }
  }

  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  if (*abort_f && threadIdx.x == 0) atomicOr(a.err, kStTimeout);
  if (warp == 1) tc::tmem_dealloc(tmem, C::NB * C::NQ);
}

template <int P, int KP>
cudaError_t launch_decode_tc_t(const ScoreArgs& a, cudaStream_t s) {
  using C = DcCfg<P>;
  const int xheads = a.exact ? a.Hq / a.G : a.Hq;
  CUtensorMap mX;
  if (!make_tmap(&mX, a.X, (uint64_t)P, (uint64_t)xheads * a.N, C::KW, C::NT, swizzle_for(C::KW)))
    return cudaErrorInvalidValue;
  const int sm = C::smem(KP);
  auto kern = score_decode_tc_kernel<P, KP>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
  if (e != cudaSuccess) return e;
  note_launch();
  if ((int64_t)a.n_items * a.Hq > 0x7fffffff) return cudaErrorInvalidConfiguration;
  kern<<<(unsigned)(a.n_items * a.Hq), 192, sm, s>>>(mX, a);
  return cudaGetLastError();
}

template <int P, int KP>
int decode_tc_occupancy() {
  using C = DcCfg<P>;
  const int sm = C::smem(KP);
  auto kern = score_decode_tc_kernel<P, KP>;
  int n = 0;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, sm) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, 192, sm) != cudaSuccess)
    n = 0;
  return n;
}

template <int KP>
cudaError_t launch_decode_tc(const ScoreArgs& a, cudaStream_t s) {
  switch (a.P) {
    case 16: return launch_decode_tc_t<16, KP>(a, s);
    case 32: return launch_decode_tc_t<32, KP>(a, s);
    case 64: return launch_decode_tc_t<64, KP>(a, s);
    default: return launch_decode_tc_t<128, KP>(a, s);
  }
}

template <typename Tin, int KP, int NQ>
int score_occupancy(int P) {
  const size_t sm = score_generic_smem(P, KP, NQ);
  auto kern = score_generic_kernel<Tin, KP, NQ>;
  int n = 0;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, kThreads, sm) != cudaSuccess)
    n = 0;
  return n;
}

template <typename Tin, int KP, int NQ>
cudaError_t launch_score_t(const ScoreArgs& a, cudaStream_t s) {
  const size_t sm = score_generic_smem(a.P, KP, NQ);
  auto kern = score_generic_kernel<Tin, KP, NQ>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  note_launch();
  if ((int64_t)a.n_items * a.Hq > 0x7fffffff) return cudaErrorInvalidConfiguration;
  kern<<<(unsigned)(a.n_items * a.Hq), kThreads, sm, s>>>(a);
  return cudaGetLastError();
}
}  // namespace

size_t score_generic_smem(int P, int kp, int nq) {
  return sizeof(uint64_t) * (size_t)kWarps * nq * 2 * kp +
         sizeof(float) * (size_t)(nq * kD + nq * P + nq) + sizeof(int) * (nq + kWarps * nq);
}

namespace {
template <typename Tin, int KP>
cudaError_t launch_nq(const ScoreArgs& a, int nq, cudaStream_t s) {
  switch (nq) {
    case 1: return launch_score_t<Tin, KP, 1>(a, s);
    case 2: return launch_score_t<Tin, KP, 2>(a, s);
    case 4: return launch_score_t<Tin, KP, 4>(a, s);
    default: return launch_score_t<Tin, KP, 8>(a, s);
  }
}
}  // namespace

// bf16 keys or codes of a tensor-core width, in groups of at least four
// queries, take the tensor-core variant (with one query per group the CUDA-core
// kernel streams a decode step faster: 0.50 against 0.53 ms over 32 heads x 1M keys)
bool decode_tc_eligible(int dtype, int P, int nq) {
  return dtype == SAKI_BF16 && nq >= 4 && (P == 16 || P == 32 || P == 64 || P == 128);
}

namespace {
template <typename Tin, int KP>
int occupancy_nq(int P, int nq) {
  switch (nq) {
    case 1: return score_occupancy<Tin, KP, 1>(P);
    case 2: return score_occupancy<Tin, KP, 2>(P);
    case 4: return score_occupancy<Tin, KP, 4>(P);
    default: return score_occupancy<Tin, KP, 8>(P);
  }
}
template <int KP>
int occupancy_tc(int P) {
  switch (P) {
    case 16: return decode_tc_occupancy<16, KP>();
    case 32: return decode_tc_occupancy<32, KP>();
    case 64: return decode_tc_occupancy<64, KP>();
    default: return decode_tc_occupancy<128, KP>();
  }
}
}  // namespace

int score_ctas_per_sm(int dtype, int P, int kp, int nq) {
  // cached per (kernel kind, dtype, P, kp, group width): the query sets the
  // kernel's shared-memory attribute, as its launch does
  static std::atomic<int> cache[2][2][8][2][4];
  const int tc = decode_tc_eligible(dtype, P, nq) ? 1 : 0;
  const int pi = P == 16 ? 0 : P == 32 ? 1 : P == 64 ? 2 : P == 128 ? 3 : (P <= 8 ? 4 : P <= 24 ? 5 : P <= 48 ? 6 : 7);
  const int qi = nq <= 1 ? 0 : nq <= 2 ? 1 : nq <= 4 ? 2 : 3;
  std::atomic<int>& slot = cache[tc][dtype == SAKI_BF16 ? 1 : 0][pi][kp == 64 ? 0 : 1][qi];
  int n = slot.load(std::memory_order_relaxed);
  if (n > 0) return n;
  if (tc) n = kp == 64 ? occupancy_tc<64>(P) : occupancy_tc<128>(P);
  else if (dtype == SAKI_BF16) n = kp == 64 ? occupancy_nq<__nv_bfloat16, 64>(P, nq) : occupancy_nq<__nv_bfloat16, 128>(P, nq);
  else n = kp == 64 ? occupancy_nq<float, 64>(P, nq) : occupancy_nq<float, 128>(P, nq);
  if (n > 0 && (pi < 4)) slot.store(n, std::memory_order_relaxed);   // other ranks' smem varies with P: not cached
  return n;
}

cudaError_t launch_score_generic(const ScoreArgs& a, int dtype, int kp, int nq, cudaStream_t s) {
  if (a.n_items == 0) return cudaSuccess;
  if (a.err && decode_tc_eligible(dtype, a.P, nq))
    return kp == 64 ? launch_decode_tc<64>(a, s) : launch_decode_tc<128>(a, s);
  if (dtype == SAKI_BF16)
    return kp == 64 ? launch_nq<__nv_bfloat16, 64>(a, nq, s) : launch_nq<__nv_bfloat16, 128>(a, nq, s);
  return kp == 64 ? launch_nq<float, 64>(a, nq, s) : launch_nq<float, 128>(a, nq, s);
}

cudaError_t launch_merge(const ScoreArgs& a, int dtype, int kp, cudaStream_t s) {
  if (a.n_merges == 0) return cudaSuccess;
  dim3 grid(a.n_merges, a.Hq);
  if (dtype == SAKI_BF16) {
    if (kp == 64) {
      note_launch();
      merge_kernel<__nv_bfloat16, 64><<<grid, 128, 0, s>>>(a);
    }
    else {
      note_launch();
      merge_kernel<__nv_bfloat16, 128><<<grid, 128, 0, s>>>(a);
    }
  } else {
    if (kp == 64) {
      note_launch();
      merge_kernel<float, 64><<<grid, 128, 0, s>>>(a);
    }
    else {
      note_launch();
      merge_kernel<float, 128><<<grid, 128, 0, s>>>(a);
    }
  }
  return cudaGetLastError();
}

}  // namespace saki
