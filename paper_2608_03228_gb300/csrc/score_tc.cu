// Batched fused score + top-k on the 5th-generation tensor cores (sm_103a).
//
// One persistent CTA per SM walks work items (a tile of up to 128 consecutive
// queries of one sequence, one query head), heaviest tiles first.  Per item:
//   1. projection on the tensor core: u = W^T q for the 128 queries, with the
//      fp32 projection W (L for Sec. 6's selection, A for the exact scores of the
//      Sec. 3 protocol) split exactly into three bf16 parts; the fp32 result in
//      TMEM is split into u_hi + u_lo (bf16 each) and written, swizzled, as the
//      A operand of the main loop (keeping u to ~16 bits, far below the score
//      tolerance);
//   2. main loop over 64-key tiles of the visible range: TMA brings the key
//      rows (codes, or raw keys for the exact scores) into a ring of
//      shared-memory stages; one thread issues tcgen05.mma (M = 128 queries,
//      N = 64 keys, K = P, twice: u_hi and u_lo) into a ring of eight TMEM
//      accumulators of 64 columns (a rank-128 projection spans two);
//   3. four epilogue warps own one query row per thread (TMEM lane = row) and
//      select in two passes over the same scores (the key tiles are multiplied
//      twice; the tensor core has ample headroom): pass 1 folds every score
//      into the row's 128 key-group maxima (one three-input maximum per two
//      scores) and takes their k-th largest, a certified lower bound tau on
//      the row's k-th best score; pass 2 appends the visible keys scoring
//      >= tau to the row's candidate column in shared memory.  The T x N score
//      matrix is never stored.
//   4. exact top-k of the remaining candidates per row, written coalesced.
// Roles: warp 0 = TMA producer, warp 1 = TMEM owner + MMA issuer, warps 2-5 =
// epilogue.  Every mbarrier wait is bounded (tc.cuh); a timed-out CTA drains its
// copies and MMAs, frees TMEM, flags the error word and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <type_traits>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"
#include "tmap.cuh"

namespace saki {
namespace {

constexpr int kLdc = 129;   // candidate column stride (words): conflict-free per-row scans and row reads
constexpr int kGroups = 128;  // pass-1 key groups per row, one maximum each
constexpr int kScr = 36;      // per-row scratch stride (words): 32 scores + pad, conflict-free 16-byte stores

template <int P>
struct TcCfg {
  // keys per tile (MMA N): 64-key tiles keep two chunks per tile in the
  // unrolled selection loops (fewer inlined overflow-cut copies) and halve the
  // stage buffers, so that rank-128 columns get 144 slots
  static constexpr int NT = 64;
  // TMEM accumulator ring of eight 64-column buffers: the four epilogue warps
  // release a buffer together, so its depth is how far they may drift apart
  // (their cut and bound phases take data-dependent time).  A tile takes one
  // buffer, a projection of P columns PB consecutive ones (two at rank 128).
  static constexpr int NB = 8;
  static constexpr int BUFC = 64;                             // TMEM columns per ring buffer
  static constexpr int PB = (P + BUFC - 1) / BUFC;
  // ranks up to 64 store (score, 32-bit key index) pairs of 8 bytes (one
  // 64-bit store per append); rank 128 needs the room for its operands and
  // keeps 16-bit indices in their own array
  static constexpr bool WIDE = P <= 64;
  static constexpr int STAGES = P == 128 ? 2 : 4;
  // candidate slots per row: as many as the shared-memory budget leaves (a
  // multiple of 8); bytes per slot and row: a 4-byte score plus a 4-byte (ranks
  // up to 64) or 2-byte (rank 128) key index
  static constexpr int FIXED_BYTES = (2 * 128 * P * 2 > 32768 ? 2 * 128 * P * 2 : 32768) + STAGES * 64 * P * 2 +
                                     128 * kScr * 4 + 256 + 1024;
  static constexpr int CAP = P == 128 ? 144 : ((232448 - FIXED_BYTES) / (kLdc * 8)) / 8 * 8;
  static constexpr int KB = P == 128 ? 2 : 1;                 // 64-wide K blocks
  static constexpr int KW = P == 128 ? 64 : P;                // K width of one block
  static constexpr int KK = KW / 16;                          // MMA K steps per block
  static constexpr uint32_t SW = KW == 64 ? 2u : (KW == 32 ? 4u : 6u);
  static constexpr uint32_t SBO = 8 * KW * 2;
  static constexpr int A_PART = 128 * P * 2;                  // u_hi (or u_lo) bytes
  static constexpr int A_BYTES = 2 * A_PART > 32768 ? 2 * A_PART : 32768;  // also holds the 128x128 query tile
  static constexpr int STAGE_BYTES = NT * P * 2;
  static constexpr int IDX_BYTES = WIDE ? CAP * kLdc * 4 : ((CAP * kLdc * 2 + 15) & ~15);
  static constexpr int CAND_BYTES = CAP * kLdc * 4 + IDX_BYTES;
  static constexpr int SCR_BYTES = 128 * kScr * 4;
  static constexpr int TMEM_COLS = NB * BUFC;
  static constexpr int OFF_STAGE = A_BYTES;
  static constexpr int OFF_CAND = OFF_STAGE + STAGES * STAGE_BYTES;
  static constexpr int OFF_SCR = OFF_CAND + CAND_BYTES;
  static constexpr int OFF_BAR = OFF_SCR + SCR_BYTES;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static_assert(STAGE_BYTES >= P * 128, "a projection chunk must fit a stage");
  static_assert(CAP % 8 == 0 && CAP >= 64 + 32, "candidate capacity: k + one chunk of appends");
  static_assert(NT == 64, "pass 1 folds a tile's two 32-key halves into one block of 32 groups");
  static_assert(NT <= BUFC && P <= PB * BUFC && P % PB == 0 && TMEM_COLS <= 512,
                "a ring buffer holds a tile's columns, PB of them a projection's");
  static_assert(SMEM <= 232448, "shared memory budget");
  static_assert(OFF_STAGE % 1024 == 0 && STAGE_BYTES % 1024 == 0, "swizzled TMA tiles sit on 1024-byte boundaries");
  static_assert(OFF_SCR % 16 == 0 && OFF_BAR % 16 == 0, "16-byte scratch stores and 8-byte mbarriers stay aligned");
};

// ---------------------------------------------------------------- selection
// Selection of a row's top k runs in two passes over the same tensor-core scores.
//   Pass 1 keeps, per row, the maximum of each of 128 key groups.  These are
//   scores of distinct keys, so their k-th largest, tau, is a certified lower
//   bound on the row's k-th best score: no key of the top k scores below tau.
//   Pass 2 appends only the keys scoring >= tau to the row's candidate column
//   (about 87 per row for independent scores with k = 64, against ~5 k ln(n/k)
//   for a streaming threshold), and a final exact cut leaves the top k.
// Every helper runs with the warp converged: loops over candidate slots run to
// the warp's largest count with per-lane predicates, so the 32 rows of a warp
// never split into separately executed paths.

// A row's candidate column: slot i holds a score (fp32) and its key index.
// ColSplit keeps 16-bit indices in their own array (the host only sends
// sequences of at most 65535 keys here); ColPair keeps (score, 32-bit index)
// pairs of 8 bytes, so an append is a single 64-bit store (shared-memory store
// instructions, predicated or not, are what the append loop is bound by: two
// 32-bit stores per key took twice as long in a stand-alone loop).  kSStride
// is the distance, in floats, between a row's consecutive scores.
struct ColSplit {
  static constexpr bool kWide = false;
  static constexpr int kSStride = kLdc;
  float* bs;
  uint16_t* bi;
  int row;
  __device__ __forceinline__ float* sbase() const { return bs + row; }
  __device__ __forceinline__ float s(int i) const { return bs[i * kLdc + row]; }
  __device__ __forceinline__ int j(int i) const { return bi[i * kLdc + row]; }
  __device__ __forceinline__ void put(int i, float v, int k) const {
    bs[i * kLdc + row] = v;
    bi[i * kLdc + row] = (uint16_t)k;
  }
  __device__ __forceinline__ ColSplit at(int r) const { return ColSplit{bs, bi, r}; }
};
struct ColPair {
  static constexpr bool kWide = true;
  static constexpr int kSStride = 2 * kLdc;
  float2* b;
  int row;
  __device__ __forceinline__ float* sbase() const { return reinterpret_cast<float*>(b + row); }
  __device__ __forceinline__ float s(int i) const { return b[i * kLdc + row].x; }
  __device__ __forceinline__ int j(int i) const { return __float_as_int(b[i * kLdc + row].y); }
  __device__ __forceinline__ void put(int i, float v, int k) const {
    b[i * kLdc + row] = make_float2(v, __int_as_float(k));
  }
  __device__ __forceinline__ ColPair at(int r) const { return ColPair{b, r}; }
};
template <class Col>
__device__ __forceinline__ Col make_col(float* bs, uint16_t* bi, int row) {
  if constexpr (Col::kWide) return Col{reinterpret_cast<float2*>(bs), row};
  else return Col{bs, bi, row};
}

__device__ __forceinline__ int warp_max(int v) { return __reduce_max_sync(0xffffffffu, v); }

// Largest float below t (appending "score > below(tau)" keeps every score >= tau).
__device__ __forceinline__ float below(float t) {
  if (t == -INFINITY) return t;
  const uint32_t b = __float_as_uint(t);
  if ((b & 0x7fffffffu) == 0) return __uint_as_float(0x80000001u);
  return __uint_as_float((b & 0x80000000u) ? b + 1 : b - 1);
}

// Bitonic sort of a register array into descending order (compile-time indices).
template <int N>
__device__ __forceinline__ void sort_desc(float (&s)[N]) {
#pragma unroll
  for (int size = 2; size <= N; size <<= 1)
#pragma unroll
    for (int j = size >> 1; j > 0; j >>= 1)
#pragma unroll
      for (int i = 0; i < N; ++i) {
        const int l = i ^ j;
        if (l > i) {
          const float a = s[i], b = s[l];
          const bool desc = (i & size) == 0;
          s[i] = desc ? fmaxf(a, b) : fminf(a, b);
          s[l] = desc ? fminf(a, b) : fmaxf(a, b);
        }
      }
}

template <int N>
__device__ __forceinline__ float pick(const float (&s)[N], int q) {
  float p = s[0];
#pragma unroll
  for (int u = 1; u < N; ++u) p = (u == q) ? s[u] : p;
  return p;
}

// Lanes with `on` keep their entries scoring >= p (in place, order preserved).
template <class Col>
__device__ __forceinline__ int compact_ge(const Col& c, int cnt, int cmax, float p, bool on) {
  int w = 0;
  for (int i = 0; i < cmax; i += 8) {
    float v[8];
    int j[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      v[u] = c.s(i + u);
      j[u] = c.j(i + u);
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const bool keep = on && i + u < cnt && v[u] >= p;
      if (keep) c.put(w, v[u], j[u]);
      w += keep ? 1 : 0;
    }
  }
  return on ? w : cnt;
}

// (score, index) worse-than: lower score, or equal score and higher index.
__device__ __forceinline__ bool worse(float a, int ja, float b, int jb) { return a < b || (a == b && ja > jb); }

// Lanes with `on` drop their worst entry (lowest score, then highest index) and
// raise thr to its score.
template <class Col>
__device__ __forceinline__ void remove_worst(const Col& c, int& cnt, int cmax, float& thr, bool on) {
  float ws[4];
  int wj[4], wp[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) { ws[u] = INFINITY; wj[u] = -1; wp[u] = 0; }
  for (int i = 0; i < cmax; i += 4) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float v = c.s(i + u);
      const int jj = c.j(i + u);
      if (i + u < cnt && worse(v, jj, ws[u], wj[u])) { ws[u] = v; wj[u] = jj; wp[u] = i + u; }
    }
  }
#pragma unroll
  for (int u = 1; u < 4; ++u)
    if (worse(ws[u], wj[u], ws[0], wj[0])) { ws[0] = ws[u]; wj[0] = wj[u]; wp[0] = wp[u]; }
  if (on && cnt > 0) {
    --cnt;
    const float ls = c.s(cnt);
    const int lj = c.j(cnt);
    c.put(wp[0], ls, lj);
    thr = fmaxf(thr, ws[0]);
  }
}

// Lanes with `on` cut their column to the entries scoring >= a sampled pivot p,
// for a pivot leaving between k and tmax entries; thr becomes p (every later key
// has a higher index, so a later key scoring exactly p loses to all kept ones).
// One counting pass tries four adjacent pivots of 16 sorted samples around
// rank aim and takes the one leaving the fewest entries that still number at
// least k.  Lanes for which no tried pivot qualifies keep their column unchanged.
template <class Col>
__device__ __forceinline__ void pivot_cut(const Col& c, int& cnt, float& thr, int k, int aim, int tmax, bool on) {
  const bool pending = on && cnt > k;
  if (!__any_sync(0xffffffffu, pending)) return;
  const int cmax = warp_max(cnt);
  float s[16];
#pragma unroll
  for (int u = 0; u < 16; ++u) s[u] = c.s(((2 * u + 1) * cnt) >> 5);
  sort_desc<16>(s);
  // sample q (0-based, descending) sits near entry rank (q + 0.5) cnt / 16
  int q = cnt > 0 ? (32 * aim / cnt - 1) >> 1 : 0;
  q = q < 1 ? 1 : (q > 13 ? 13 : q);
  float p[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) p[j] = pick<16>(s, q - 1 + j);
  const float kNaN = __int_as_float(0x7fffffff);   // compares false: slots past the lane's count
  int n[4] = {0, 0, 0, 0};
  for (int i = 0; i < cmax; i += 8) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) v[u] = i + u < cnt ? c.s(i + u) : kNaN;
#pragma unroll
    for (int u = 0; u < 8; ++u)
#pragma unroll
      for (int j = 0; j < 4; ++j) n[j] += v[u] >= p[j] ? 1 : 0;
  }
  // descending pivots give ascending counts: the first count reaching k
  float pc = p[3];
  int nc = n[3];
#pragma unroll
  for (int j = 2; j >= 0; --j)
    if (n[j] >= k) { pc = p[j]; nc = n[j]; }
  const bool ok = pending && nc >= k && nc <= tmax;
  if (__any_sync(0xffffffffu, ok)) cnt = compact_ge(c, cnt, cmax, pc, ok);
  if (ok) thr = fmaxf(thr, pc);
}

// Bitonic sort of 16 (score, index) keys into descending order.
__device__ __forceinline__ void sort16_desc(uint64_t (&key)[16]) {
#pragma unroll
  for (int size = 2; size <= 16; size <<= 1)
#pragma unroll
    for (int jj = size >> 1; jj > 0; jj >>= 1)
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int l = i ^ jj;
        if (l > i) {
          const uint64_t x = key[i], y = key[l];
          const bool desc = (i & size) == 0;
          const bool sw = desc ? (x < y) : (x > y);
          key[i] = sw ? y : x;
          key[l] = sw ? x : y;
        }
      }
}

// Exact cut of the lanes with `on` to their k best entries (slots [0, k)); thr
// rises to a lower bound of the k-th best score (a later key, with a higher
// index, must score above it to matter).  Quickselect by counting over a
// half-open bracket [lo, hi): na entries score >= hi (na <= k, all of them
// kept) and nb score >= lo (nb >= k, so the k best all score >= lo).  A round
// counts the entries at or above five pivots taken from 16 sorted samples of
// the bracket around the k-th entry's expected rank and keeps the tightest
// bracket; once at most 16 entries lie in [lo, hi), they are ranked as 64-bit
// (score, index) keys in registers and fill the remaining places.  Lanes whose
// bracket cannot narrow (many equal scores) fall back to pivot cuts and single
// removals.
template <class Col>
__device__ __forceinline__ void cut_to_k(const Col& c, int& cnt, float& thr, int k, float* scr, bool on) {
  bool pending = on && cnt > k;
  if (!__any_sync(0xffffffffu, pending)) return;
  const int cmax = warp_max(cnt);
  float s[16];
#pragma unroll
  for (int u = 0; u < 16; ++u) s[u] = c.s(((2 * u + 1) * cnt) >> 5);
  sort_desc<16>(s);
  float hi = INFINITY, lo = -INFINITY;
  int na = 0, nb = cnt;
  bool ready = false;
  const float kNaN = __int_as_float(0x7fffffff);   // compares false: slots past the lane's count
  for (int round = 0; round < 4; ++round) {
    const bool act = pending && !ready;
    if (!__any_sync(0xffffffffu, act)) break;
    // sample q sits near rank (q + 0.5) pop / 16 of the bracket's population
    const int pop = nb - na > 0 ? nb - na : 1;
    int qc = (32 * (k - na) / pop - 1) >> 1;
    qc = qc < 2 ? 2 : (qc > 13 ? 13 : qc);
    float p[5];
#pragma unroll
    for (int j = 0; j < 5; ++j) p[j] = pick<16>(s, qc - 2 + j);
    int n[5] = {0, 0, 0, 0, 0};
    for (int i = 0; i < cmax; i += 8) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = i + u < cnt ? c.s(i + u) : kNaN;
#pragma unroll
      for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int j = 0; j < 5; ++j) n[j] += v[u] >= p[j] ? 1 : 0;
    }
    if (act) {
#pragma unroll
      for (int j = 0; j < 5; ++j) {
        if (n[j] <= k && p[j] < hi) { hi = p[j]; na = n[j]; }
        if (n[j] >= k && p[j] > lo) { lo = p[j]; nb = n[j]; }
      }
      ready = nb - na <= 16;
    }
    const bool resample = act && !ready;
    if (__any_sync(0xffffffffu, resample)) {
      // new samples: every stride-th score inside the bracket (pop > 16 there)
      const int stride = (nb - na) >> 4;
      int ns = 0, seen = 0;
      for (int i = 0; i < cmax; i += 8) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = c.s(i + u);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const bool in = resample && i + u < cnt && v[u] >= lo && v[u] < hi;
          const bool take = in && seen == 0 && ns < 16;
          if (take) scr[ns] = v[u];
          ns += take ? 1 : 0;
          seen = in ? (seen + 1 == stride ? 0 : seen + 1) : seen;
        }
      }
      if (resample) {
#pragma unroll
        for (int u = 0; u < 16; ++u) s[u] = u < ns ? scr[u] : -INFINITY;
      }
      sort_desc<16>(s);
    }
  }
  const bool fin = pending && ready;
  if (__any_sync(0xffffffffu, fin)) {
    // entries at or above hi compacted in place, boundary entries to the scratch
    int w = 0, nbd = 0;
    for (int i = 0; i < cmax; i += 8) {
      float v[8];
      int j[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        v[u] = c.s(i + u);
        j[u] = c.j(i + u);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const bool in = fin && i + u < cnt;
        const bool sure = in && v[u] >= hi;
        const bool bnd = in && !sure && v[u] >= lo;
        if (sure) c.put(w, v[u], j[u]);
        if (bnd) {
          scr[2 * nbd] = v[u];
          scr[2 * nbd + 1] = __int_as_float(j[u]);
        }
        w += sure ? 1 : 0;
        nbd += bnd ? 1 : 0;
      }
    }
    uint64_t key[16];
#pragma unroll
    for (int u = 0; u < 16; ++u)
      key[u] = (fin && u < nbd) ? make_key(scr[2 * u], (uint32_t)__float_as_int(scr[2 * u + 1])) : 0ull;
    sort16_desc(key);
    float kth = hi;
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const bool use = fin && w + u < k && u < nbd;
      if (use) c.put(w + u, key_score(key[u]), key_index(key[u]));
      if (use) kth = key_score(key[u]);
    }
    if (fin) {
      cnt = k;
      thr = fmaxf(thr, kth);
      pending = false;
    }
  }
  if (__any_sync(0xffffffffu, pending)) {
    for (int g = 0; g < 3 && __any_sync(0xffffffffu, pending && cnt - k > 8); ++g)
      pivot_cut(c, cnt, thr, k, k + 3, cnt - 1, pending && cnt - k > 8);
    while (__any_sync(0xffffffffu, pending && cnt > k)) remove_worst(c, cnt, warp_max(cnt), thr, pending && cnt > k);
  }
}

// Bin of score v among 64 equal bins over [lo, lo + 64 / scale]: the integer
// nearest (v - lo) * scale, read from the bits of a float near 2^23 (one FMA;
// bias = 2^23 - lo * scale), clamped to [0, 63].  Non-decreasing in v.
__device__ __forceinline__ int bin64(float v, float scale, float bias) {
  const int b = __float_as_int(fmaf(v, scale, bias)) - 0x4B000000;
  return b < 0 ? 0 : (b > 63 ? 63 : b);
}

// Final exact cut of the lanes with `on` to their k best entries (slots
// [0, k)), by histogram: 64 bins over the column's score range, counted with
// shared-memory atomics into 16-bit halves of the row's scratch, locate the bin
// holding the k-th best entry; entries in higher bins are kept, and those of
// that bin (at most 16) are ranked as 64-bit (score, index) keys.  Lanes this
// cannot settle (a degenerate range, or more than 16 entries in the boundary
// bin, e.g. many equal scores) go through cut_to_k.
template <class Col>
__device__ __forceinline__ void cut_hist(const Col& c, int& cnt, float& thr, int k, float* scr, bool on) {
  bool pending = on && cnt > k;
  if (!__any_sync(0xffffffffu, pending)) return;
  const int cmax = warp_max(cnt);
  const float kNaN = __int_as_float(0x7fffffff);   // ignored by fminf / fmaxf
  float lo = INFINITY, hi = -INFINITY;
  for (int i = 0; i < cmax; i += 8) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float v = i + u < cnt ? c.s(i + u) : kNaN;
      lo = fminf(lo, v);
      hi = fmaxf(hi, v);
    }
  }
  const float scale = 64.f / (hi - lo);
  const float bias = 8388608.f - lo * scale;
  const bool ok = pending && hi > lo && scale <= 1e30f && fabsf(bias) <= 1e30f;
  int* h = reinterpret_cast<int*>(scr);
#pragma unroll
  for (int w = 0; w < 32; ++w) h[w] = 0;
  for (int i = 0; i < cmax; i += 8) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const float v = c.s(i + u);
      const int b = bin64(v, scale, bias);
      if (ok && i + u < cnt) atomicAdd(h + (b >> 1), 1 << ((b & 1) << 4));
    }
  }
  // the boundary bin: counting down from the top bin, the first that reaches k
  int bstar = -1, na = 0, nb = 0, acc = 0;
#pragma unroll
  for (int w = 31; w >= 0; --w) {
    const int hw = h[w];
#pragma unroll
    for (int half = 1; half >= 0; --half) {
      const int n = half ? (hw >> 16) : (hw & 0xffff);
      const bool hit = bstar < 0 && acc + n >= k;
      bstar = hit ? 2 * w + half : bstar;
      na = hit ? acc : na;
      nb = hit ? n : nb;
      acc += n;
    }
  }
  const bool fin = ok && bstar >= 0 && nb <= 16;
  if (__any_sync(0xffffffffu, fin)) {
    // entries above the boundary bin compacted in place, its entries to the scratch
    int w = 0, nbd = 0;
    for (int i = 0; i < cmax; i += 8) {
      float v[8];
      int j[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        v[u] = c.s(i + u);
        j[u] = c.j(i + u);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int b = bin64(v[u], scale, bias);
        const bool in = fin && i + u < cnt;
        const bool sure = in && b > bstar;
        const bool bnd = in && b == bstar;
        if (sure) c.put(w, v[u], j[u]);
        if (bnd) {
          scr[2 * nbd] = v[u];
          scr[2 * nbd + 1] = __int_as_float(j[u]);
        }
        w += sure ? 1 : 0;
        nbd += bnd ? 1 : 0;
      }
    }
    uint64_t key[16];
#pragma unroll
    for (int u = 0; u < 16; ++u)
      key[u] = (fin && u < nbd) ? make_key(scr[2 * u], (uint32_t)__float_as_int(scr[2 * u + 1])) : 0ull;
    sort16_desc(key);
    float kth = thr;
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const bool use = fin && w + u < k && u < nbd;
      if (use) c.put(w + u, key_score(key[u]), key_index(key[u]));
      if (use) kth = key_score(key[u]);
    }
    if (fin) {
      cnt = k;
      thr = fmaxf(thr, kth);
      pending = false;
    }
  }
  if (__any_sync(0xffffffffu, pending)) cut_to_k(c, cnt, thr, k, scr, pending);
}

// Three-input maximum (one instruction on sm_100 and later).
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Scores of a key tile (keys j0 .. j0+63 of the row: ra holds the first 32, rb
// the last 32) at or past the row's visible count become -inf.  Only tiles that
// cross some row's visibility boundary take this path.
__device__ __forceinline__ void mask_tile(uint32_t (&ra)[32], uint32_t (&rb)[32], int j0, int vis) {
  const uint32_t ninf = __float_as_uint(-INFINITY);
#pragma unroll
  for (int u = 0; u < 32; ++u) {
    ra[u] = j0 + u < vis ? ra[u] : ninf;
    rb[u] = j0 + 32 + u < vis ? rb[u] : ninf;
  }
}

// Pass 1: fold a tile into 32 of the row's 128 group maxima.  Key j belongs to
// group 32 ((j / 64) mod 4) + (j mod 32), so a tile's keys j and j + 32 share a
// group and one three-input maximum folds both (half an instruction per
// score).  Called from a loop unrolled over the tile index mod 4, so gb is a
// constant and the maxima stay in registers.
__device__ __forceinline__ void fold64(const uint32_t (&ra)[32], const uint32_t (&rb)[32], float (&g)[kGroups],
                                       int gb) {
#pragma unroll
  for (int u = 0; u < 32; ++u) g[gb + u] = max3f(g[gb + u], __uint_as_float(ra[u]), __uint_as_float(rb[u]));
}

// The certified bound of pass 1.  The 128 group maxima are scores of distinct
// visible keys, so the k-th largest of them bounds the row's k-th best score
// from below.  32 of them, sorted, give pivots: a counting pass tests three,
// two samples apart, around the expected rank of the k-th and moves up or down
// until one pivot leaves at least k maxima (lo) and a higher one fewer (hi).
// The maxima between the two (at most 32) are gathered in the row's scratch
// and ranked, which gives the k-th largest exactly; a wider bracket keeps lo,
// and no qualifying pivot at all leaves -inf (every visible key is then a
// candidate).  The maxima are first copied into the row's candidate column,
// still empty, so that the counting and gathering loops run over shared memory
// without unrolling: this code runs once per item and stays small.
template <int S>
__device__ __forceinline__ float select_tau(const float (&g)[kGroups], int k, float* col, float* scr) {
  float s[32];
#pragma unroll
  for (int u = 0; u < 32; ++u) s[u] = g[4 * u + 1];
  sort_desc<32>(s);
#pragma unroll
  for (int i = 0; i < kGroups; ++i) col[i * S] = g[i];
  // sample q (0-based, descending) has about (q + 1) * 128 / 33 maxima at or above it
  int q = (33 * k + 127) / kGroups - 1;
  q = q < 2 ? 2 : (q > 29 ? 29 : q);
  float lo = -INFINITY, hi = INFINITY;
  int nlo = kGroups, nhi = 0;
  bool pending = true;
  for (int attempt = 0; attempt < 4; ++attempt) {
    const float p0 = pick<32>(s, q - 2), p1 = pick<32>(s, q), p2 = pick<32>(s, q + 2);
    int n0 = 0, n1 = 0, n2 = 0;
#pragma unroll 4
    for (int i = 0; i < kGroups; ++i) {
      const float v = col[i * S];
      n0 += v >= p0 ? 1 : 0;
      n1 += v >= p1 ? 1 : 0;
      n2 += v >= p2 ? 1 : 0;
    }
    if (pending) {
      // descending pivots, ascending counts: the highest qualifying one and
      // the lowest failing one narrow the bracket
      if (n2 >= k && p2 > lo) { lo = p2; nlo = n2; }
      if (n1 >= k && p1 > lo) { lo = p1; nlo = n1; }
      if (n0 >= k && p0 > lo) { lo = p0; nlo = n0; }
      if (n0 < k && p0 < hi) { hi = p0; nhi = n0; }
      if (n1 < k && p1 < hi) { hi = p1; nhi = n1; }
      if (n2 < k && p2 < hi) { hi = p2; nhi = n2; }
      const bool up = hi == INFINITY && q > 2;      // every pivot qualified
      const bool down = lo == -INFINITY && q < 29;  // none did
      pending = up || down;
      q = up ? (q < 8 ? 2 : q - 6) : (down ? (q > 23 ? 29 : q + 6) : q);
    }
    if (!__any_sync(0xffffffffu, pending)) break;
  }
  // the (k - nhi)-th largest of the nlo - nhi maxima in [lo, hi)
  const bool ex = nlo - nhi <= 32;
  if (__any_sync(0xffffffffu, ex)) {
    int c = 0;
#pragma unroll 4
    for (int i = 0; i < kGroups; ++i) {
      const float v = col[i * S];
      const bool in = ex && v >= lo && v < hi;
      if (in) scr[c] = v;
      c += in ? 1 : 0;
    }
    float b[32];
#pragma unroll
    for (int u = 0; u < 32; ++u) b[u] = u < c ? scr[u] : -INFINITY;
    sort_desc<32>(b);
    const float t = pick<32>(b, k - nhi - 1);
    if (ex) lo = t;
  }
  return lo;
}

// Rare path of pass 2: lanes whose column is within one chunk of the capacity
// and would overflow with this chunk's appends are cut to between k and CAP - 32
// entries at a sampled pivot (raising thr to it), together with every lane of
// the warp close to the capacity; the exact cut only where no pivot qualifies.
template <int CAP, class Col>
__device__ __forceinline__ void make_room(const uint32_t (&r)[32], float& thr, float* scr, const Col& c, int& cnt,
                                          int k) {
  int n = 0;
#pragma unroll
  for (int u = 0; u < 32; ++u) n += __uint_as_float(r[u]) > thr ? 1 : 0;
  const bool over = cnt + n > CAP;
  const int near = (k + 8 > CAP - 40) ? k + 8 : CAP - 40;
  if (__any_sync(0xffffffffu, over)) {
    pivot_cut(c, cnt, thr, k, k + 8, CAP - 32, over || cnt > near);
    const bool still = over && cnt > CAP - 32;
    if (__any_sync(0xffffffffu, still)) cut_to_k(c, cnt, thr, k, scr, still);
  }
  __syncwarp();
}

// Pass 2: append the keys of 32 scores of a row (keys j0 .. j0+31; keys the row
// cannot see are -inf already) that score above thr.  The appends are
// predicated stores at a running slot pointer: no mask, no scratch, no
// data-dependent loop; the capacity check is one warp vote.
template <int CAP, class Col>
__device__ __forceinline__ void append32(const uint32_t (&r)[32], int j0, float& thr, float* scr, const Col& c,
                                         int& cnt, int k) {
  if (__any_sync(0xffffffffu, cnt > CAP - 32)) make_room<CAP>(r, thr, scr, c, cnt, k);
  if constexpr (Col::kWide) {
    // one 64-bit store per append; the count is the slot pointer's advance
    float2* ps = c.b + cnt * kLdc + c.row;
    float2* const p0 = ps;
#pragma unroll
    for (int u = 0; u < 32; ++u) {
      const float v = __uint_as_float(r[u]);
      const bool t = v > thr;
      if (t) *ps = make_float2(v, __int_as_float(j0 + u));
      ps += t ? kLdc : 0;
    }
    cnt += (int)(ps - p0) / kLdc;
  } else {
    float* ps = c.bs + cnt * kLdc + c.row;
    uint16_t* pi = c.bi + cnt * kLdc + c.row;
    int added = 0;
#pragma unroll
    for (int u = 0; u < 32; ++u) {
      const float v = __uint_as_float(r[u]);
      const bool t = v > thr;
      if (t) {
        *ps = v;
        *pi = (uint16_t)(j0 + u);
      }
      ps += t ? kLdc : 0;
      pi += t ? kLdc : 0;
      added += t ? 1 : 0;
    }
    cnt += added;
  }
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
__device__ __forceinline__ void convert_projection(const uint32_t (&taddr)[2], uint8_t* sA, int m) {
#pragma unroll
  for (int c0 = 0; c0 < P; c0 += 16) {
    uint32_t r[16];
    __syncwarp();
    tc::tmem_ld16(c0 < 64 ? taddr[0] + c0 : taddr[1] + (c0 - 64), r);
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
  float* scr_all = reinterpret_cast<float*>(smem + C::OFF_SCR);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + C::STAGES;
  uint64_t* accf = empty + C::STAGES;
  uint64_t* acce = accf + C::NB;
  uint64_t* qfull = acce + C::NB;
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
    for (int b = 0; b < C::NB; ++b) {
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
      for (int item = a.stall ? a.n_items : blockIdx.x; item < a.n_items; item += gridDim.x, ++it) {
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
        for (int i2 = 0; i2 < 2 * ntiles; ++i2) {   // the two selection passes
          const int i = i2 < ntiles ? i2 : i2 - ntiles;
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
      constexpr uint32_t idP = tc::idesc_bf16(128, P / C::PB);
      constexpr uint32_t idN = tc::idesc_bf16(128, C::NT);
      const uint32_t aBase = tc::smem_u32(sA), sBase = tc::smem_u32(sStage);
      for (int item = blockIdx.x; item < a.n_items; item += gridDim.x, ++it) {
        const TcTile t = a.tiles[item / Hq];
        if (!tc::mbar_wait(qfull, it & 1, abort_f)) break;
        bool ok = true;
#pragma unroll
        for (int q = 0; q < C::PB; ++q)
          ok = ok && tc::mbar_wait(acce + (ac + q) % C::NB, (((ac + q) / C::NB) & 1) ^ 1, abort_f);
        if (!ok) break;
        tc::fence_after_sync();
        uint32_t buf;
        uint32_t acc = 0;
        for (int s3 = 0; s3 < 3 && ok; ++s3)
          for (int kh = 0; kh < 2; ++kh) {
            const int st = sc % C::STAGES;
            if (!(ok = tc::mbar_wait(full + st, (sc / C::STAGES) & 1, abort_f))) break;
            tc::fence_after_sync();
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              // the projection's columns p * P / PB .. of W in rows of the stage
#pragma unroll
              for (int q = 0; q < C::PB; ++q)
                tc::mma_bf16(tmem + ((ac + q) % C::NB) * C::BUFC, tc::sdesc(aBase + kh * 16384 + kk * 32, 1024, 2),
                             tc::sdesc(sBase + st * C::STAGE_BYTES + q * (P / C::PB) * 128 + kk * 32, 1024, 2), idP,
                             acc);
              acc = 1;
            }
            tc::mma_commit(empty + st);
            ++sc;
          }
        if (!ok) break;
#pragma unroll
        for (int q = 0; q < C::PB; ++q) tc::mma_commit(accf + (ac + q) % C::NB);
        ac += C::PB;
        if (!tc::mbar_wait(aready, it & 1, abort_f)) break;
        tc::fence_after_sync();
        const int ntiles = (t.vis_max + C::NT - 1) / C::NT;
        for (int i = 0; i < 2 * ntiles; ++i) {
          buf = ac % C::NB;
          if (!(ok = tc::mbar_wait(acce + buf, ((ac / C::NB) & 1) ^ 1, abort_f))) break;
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
                tc::mma_bf16(tmem + buf * C::BUFC, tc::sdesc(ad, C::SBO, C::SW), tc::sdesc(bd, C::SBO, C::SW), idN,
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
    using Col = typename std::conditional<C::WIDE, ColPair, ColSplit>::type;
    const Col col = make_col<Col>(bs, bi, m);
    float* scr = scr_all + m * kScr;
    uint32_t ac = 0;
    int it = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < a.n_items && ok; item += gridDim.x, ++it) {
      const TcTile t = a.tiles[item / Hq];
      const int h = item % Hq;
      if (it == 0) {  // this item's projection (later items convert theirs ahead of time)
        uint32_t pa[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) pa[q] = tl + ((ac + (q < C::PB ? q : 0)) % C::NB) * C::BUFC;
#pragma unroll
        for (int q = 0; q < C::PB; ++q)
          ok = ok && __all_sync(0xffffffffu, tc::mbar_wait(accf + (ac + q) % C::NB, ((ac + q) / C::NB) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
        convert_projection<P>(pa, sA, m);
        tc::fence_before_sync();
#pragma unroll
        for (int q = 0; q < C::PB; ++q) tc::mbar_arrive(acce + (ac + q) % C::NB);
        ac += C::PB;
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(aready);
      }
      const int vis = m < t.nrows ? a.vis[t.q0 + m] : 0;
      const int wmin = __reduce_min_sync(0xffffffffu, vis);   // tiles past it need masking
      const int ntiles = (t.vis_max + C::NT - 1) / C::NT;
      // pass 1: the maxima of the 128 key groups, then the certified bound
      float g[kGroups];
#pragma unroll
      for (int u = 0; u < kGroups; ++u) g[u] = -INFINITY;
      for (int i0 = 0; i0 < ntiles && ok; i0 += 4) {
#pragma unroll
        for (int sub = 0; sub < 4; ++sub) {
          const int i = i0 + sub;
          if (i >= ntiles) break;
          const uint32_t buf = ac % C::NB;
          ok = __all_sync(0xffffffffu, tc::mbar_wait(accf + buf, (ac / C::NB) & 1, abort_f));
          if (!ok) break;
          tc::fence_after_sync();
          uint32_t ra[32], rb[32];
          __syncwarp();
          tc::tmem_ld32(tl + buf * C::BUFC, ra);
          tc::tmem_ld32(tl + buf * C::BUFC + 32, rb);
          tc::tmem_ld_wait(ra);
          tc::reg_fence(rb);
          tc::fence_before_sync();
          tc::mbar_arrive(acce + buf);   // the scores are in registers: the MMA may reuse the buffer
          ++ac;
          if (i * C::NT + C::NT > wmin) mask_tile(ra, rb, i * C::NT, vis);
          fold64(ra, rb, g, sub * 32);
        }
      }
      if (!ok) break;
      int cnt = 0;
      float thr = below(select_tau<Col::kSStride>(g, a.k, col.sbase(), scr));
      // pass 2: candidates scoring >= tau
      for (int i = 0; i < ntiles; ++i) {
        const uint32_t buf = ac % C::NB;
        ok = __all_sync(0xffffffffu, tc::mbar_wait(accf + buf, (ac / C::NB) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
        uint32_t ra[32], rb[32];
        __syncwarp();
        tc::tmem_ld32(tl + buf * C::BUFC, ra);
        tc::tmem_ld32(tl + buf * C::BUFC + 32, rb);
        tc::tmem_ld_wait(ra);
        tc::reg_fence(rb);
        tc::fence_before_sync();
        tc::mbar_arrive(acce + buf);
        ++ac;
        if (i * C::NT + C::NT > wmin) mask_tile(ra, rb, i * C::NT, vis);
        append32<C::CAP>(ra, i * C::NT, thr, scr, col, cnt, a.k);
        append32<C::CAP>(rb, i * C::NT + 32, thr, scr, col, cnt, a.k);
      }
      if (!ok) break;
      // convert the next item's projection now, so the tensor core can move on
      const int nxt = item + gridDim.x;
      if (nxt < a.n_items) {
        uint32_t pa[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) pa[q] = tl + ((ac + (q < C::PB ? q : 0)) % C::NB) * C::BUFC;
#pragma unroll
        for (int q = 0; q < C::PB; ++q)
          ok = ok && __all_sync(0xffffffffu, tc::mbar_wait(accf + (ac + q) % C::NB, ((ac + q) / C::NB) & 1, abort_f));
        if (!ok) break;
        tc::fence_after_sync();
        convert_projection<P>(pa, sA, m);
        tc::fence_before_sync();
#pragma unroll
        for (int q = 0; q < C::PB; ++q) tc::mbar_arrive(acce + (ac + q) % C::NB);
        ac += C::PB;
        tc::fence_proxy_async_smem();
        tc::mbar_arrive(aready);
      }
      cut_hist(col, cnt, thr, a.k, scr, true);
      if (!a.sorted && (a.k & 3) == 0) {
        // unsorted lists: each thread writes its own row, four entries per store
        if (m < t.nrows) {
          const int64_t o = ((int64_t)h * a.T + t.q0 + m) * a.k;
          const float qn = a.qnu ? a.qnu[(int64_t)h * a.T + t.q0 + m] : 0.f;
#pragma unroll 4
          for (int i = 0; i < a.k; i += 4) {
            int4 v;
            v.x = i < cnt ? col.j(i) : -1;
            v.y = i + 1 < cnt ? col.j(i + 1) : -1;
            v.z = i + 2 < cnt ? col.j(i + 2) : -1;
            v.w = i + 3 < cnt ? col.j(i + 3) : -1;
            *reinterpret_cast<int4*>(a.idx + o + i) = v;
            if (a.score) {
              float4 f;
              f.x = i < cnt ? col.s(i) + qn : -INFINITY;
              f.y = i + 1 < cnt ? col.s(i + 1) + qn : -INFINITY;
              f.z = i + 2 < cnt ? col.s(i + 2) + qn : -INFINITY;
              f.w = i + 3 < cnt ? col.s(i + 3) + qn : -INFINITY;
              *reinterpret_cast<float4*>(a.score + o + i) = f;
            }
          }
        }
        continue;
      }
      // sorted lists: the warp sorts and writes its 32 rows one after another
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
            v[e] = i < n ? make_key(col.at(row).s(i), (uint32_t)col.at(row).j(i)) : 0ull;
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
            a.idx[o + i] = i < n ? col.at(row).j(i) : -1;
            if (a.score) a.score[o + i] = i < n ? col.at(row).s(i) + qn : -INFINITY;
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

template <int P>
cudaError_t launch_tc_t(const TcLaunch& L, cudaStream_t s) {
  using C = TcCfg<P>;
  CUtensorMap mQ, mW, mX;
  const int xrows_heads = L.args.exact ? L.Hk : L.args.Hq;
  const int xcols = L.args.exact ? kD : P;
  if (!make_tmap(&mQ, L.Q, kD, (uint64_t)L.args.Hq * L.args.T, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap(&mW, L.Wsplit, kD, (uint64_t)L.args.Hq * 3 * P, 64, P, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap(&mX, L.X, xcols, (uint64_t)xrows_heads * L.args.N, C::KW, C::NT, swizzle_for(C::KW)))
    return cudaErrorInvalidValue;
  auto kern = score_tc_kernel<P>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int grid = L.args.n_items < L.num_sms ? L.args.n_items : L.num_sms;
  note_launch();
  kern<<<grid, 192, C::SMEM, s>>>(mQ, mW, mX, L.args);
  return cudaGetLastError();
}
}  // namespace

bool tc_supported(int P) { return P == 16 || P == 32 || P == 64 || P == 128; }

cudaError_t launch_pack_w(const float* W, int Hq, int P, void* out, cudaStream_t s) {
  const int64_t n = (int64_t)Hq * P * kD;
  const int blocks = (int)((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  note_launch();
  pack_w_kernel<<<blocks, 256, 0, s>>>(W, Hq, P, static_cast<__nv_bfloat16*>(out));
  return cudaGetLastError();
}

cudaError_t launch_qnu(const void* Q, const float* nu, int64_t T, int Hq, float* out, cudaStream_t s) {
  const int64_t rows = (int64_t)Hq * T;
  note_launch();
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
