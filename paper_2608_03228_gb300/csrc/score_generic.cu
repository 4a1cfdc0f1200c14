// Generic fused score + top-k on CUDA cores (any rank, f32 or bf16 inputs).
//
// Serves the decode-shaped work of the selection step (Sec. 5: s_hat = (L^T q)^T c_j
// over the visible keys, keep the k largest) and, with W = A and X = K, the
// exact top-k of the Sec. 3 recall protocol.  A work item is up to kGroupQ
// queries of one sequence against one split of its keys; each lane scores one
// key for all queries of the group from 128-bit loads, so every key row is read
// once per item.  Selection never forms the score matrix: each warp keeps, per
// query, a shared-memory buffer of candidates above its running k-th best key
// and re-selects (warp bitonic sort) when the buffer fills; warps are merged at
// the end, and splits of a long sequence by a second small kernel.
#include "common.cuh"
#include "kernels.h"

namespace saki {

namespace {
constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;

template <typename T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

// Keep the KP best of the warp's buffer (sorted, descending) and return the
// k-th best key (0 while fewer than k are held).
template <int KP>
__device__ __forceinline__ uint64_t reselect(uint64_t* qb, int& cnt, int k) {
  constexpr int E = 2 * KP / 32;
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
template <int KP>
__device__ __noinline__ uint64_t append_keys(uint64_t* qb, int* cnt_s, unsigned long long* cta_thr, uint64_t key,
                                             bool pass, unsigned mask, uint64_t thr, int k) {
  constexpr int CAP = 2 * KP;
  const int lane = threadIdx.x & 31;
  int cnt = *cnt_s;
  if (pass) qb[cnt + __popc(mask & ((1u << lane) - 1u))] = key;
  cnt += __popc(mask);
  if (cnt > CAP - 32) {
    const uint64_t t = reselect<KP>(qb, cnt, k);
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

  const ScoreItem it = a.items[blockIdx.x];
  const int h = blockIdx.y;
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

template <typename Tin, int KP>
__global__ void __launch_bounds__(128) merge_kernel(const ScoreArgs a) {
  constexpr int EK = KP / 32;
  const int lane = threadIdx.x & 31;
  const int m = blockIdx.x * 4 + (threadIdx.x >> 5);
  if (m >= a.n_merges) return;
  const int h = blockIdx.y;
  const MergeItem mi = a.merges[m];
  const uint64_t* c = a.cand + ((int64_t)h * a.cand_per_head + mi.cand) * KP;
  uint64_t best[EK], other[EK];
#pragma unroll
  for (int e = 0; e < EK; ++e) best[e] = c[e * 32 + lane];
  for (int s = 1; s < mi.nsplit; ++s) {
#pragma unroll
    for (int e = 0; e < EK; ++e) other[e] = c[(int64_t)s * KP + e * 32 + lane];
    warp_merge_top<EK>(best, other);
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

template <typename Tin, int KP, int NQ>
cudaError_t launch_score_t(const ScoreArgs& a, cudaStream_t s) {
  const size_t sm = score_generic_smem(a.P, KP, NQ);
  auto kern = score_generic_kernel<Tin, KP, NQ>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  note_launch();
  kern<<<dim3(a.n_items, a.Hq), kThreads, sm, s>>>(a);
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

cudaError_t launch_score_generic(const ScoreArgs& a, int dtype, int kp, int nq, cudaStream_t s) {
  if (a.n_items == 0) return cudaSuccess;
  if (dtype == SAKI_BF16)
    return kp == 64 ? launch_nq<__nv_bfloat16, 64>(a, nq, s) : launch_nq<__nv_bfloat16, 128>(a, nq, s);
  return kp == 64 ? launch_nq<float, 64>(a, nq, s) : launch_nq<float, 128>(a, nq, s);
}

cudaError_t launch_merge(const ScoreArgs& a, int dtype, int kp, cudaStream_t s) {
  if (a.n_merges == 0) return cudaSuccess;
  dim3 grid((a.n_merges + 3) / 4, a.Hq);
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
