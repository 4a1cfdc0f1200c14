// C-ABI entry points (include/saki.h): argument checks, workspace carving, the
// host-side work plan of the selection kernels, and launches.  No device
// memory is allocated here; every buffer belongs to the caller.
#include <algorithm>
#include <atomic>
#include <climits>
#include <cmath>
#include <cstring>
#include <map>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "kernels.h"

using namespace saki;

namespace {

thread_local bool t_pageable_only = false;

// Pinned host staging for the library's own small transfers (per-call plans up,
// the fit's status words down).  A pageable copy is staged by the driver through
// its bounce buffers, which can stall behind large copies the caller runs on
// other streams; these go through a ring of pinned slots per device instead.  A
// slot is reused only after the event recorded behind its last copy completed.
// Byte copy on the SMs (16-byte words when both ends allow), for the staging
// ring: one side is mapped pinned host memory read or written through its
// device alias, so no copy engine is involved.
__global__ void staged_copy_kernel(uint8_t* dst, const uint8_t* src, size_t n) {
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  size_t i0 = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (((reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(src)) & 15u) == 0) {
    const size_t nv = n / 16;
    for (size_t i = i0; i < nv; i += stride)
      reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
    for (size_t i = nv * 16 + i0; i < n; i += stride) dst[i] = src[i];
  } else {
    for (size_t i = i0; i < n; i += stride) dst[i] = src[i];
  }
}

cudaError_t staged_copy(void* dst, const void* src, size_t n, cudaStream_t s) {
  const size_t words = (n + 15) / 16;
  const int blocks = (int)std::min<size_t>((words + 255) / 256, 64);
  note_launch();
  staged_copy_kernel<<<blocks, 256, 0, s>>>(static_cast<uint8_t*>(dst), static_cast<const uint8_t*>(src), n);
  return cudaGetLastError();
}

// The library's own small transfers (plans up, status words down) go through a
// ring of mapped pinned slots and are carried by staged_copy_kernel: a copy
// engine would queue them behind the caller's large transfers on other
// streams (an input copy of the next batch), stalling this stream for as long.
class Staging {
 public:
  // host -> device: n bytes of src to dst, ordered on s
  cudaError_t upload(void* dst, const void* src, size_t n, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if (t_pageable_only) return cudaMemcpyAsync(dst, src, n, cudaMemcpyHostToDevice, s);
    std::lock_guard<std::mutex> lock(mu_);
    Slot* sl = nullptr;
    cudaError_t e = take(n, &sl);
    if (e != cudaSuccess) return e;
    std::memcpy(sl->p, src, n);
    if ((e = staged_copy(dst, sl->d, n, s)) != cudaSuccess) return e;
    return cudaEventRecord(sl->ev, s);
  }
  // device -> host: n bytes of src to dst; waits for the stream
  cudaError_t download_sync(void* dst, const void* src, size_t n, cudaStream_t s) {
    if (t_pageable_only) {
      const cudaError_t e = cudaMemcpyAsync(dst, src, n, cudaMemcpyDeviceToHost, s);
      return e != cudaSuccess ? e : cudaStreamSynchronize(s);
    }
    std::lock_guard<std::mutex> lock(mu_);
    Slot* sl = nullptr;
    cudaError_t e = take(n, &sl);
    if (e != cudaSuccess) return e;
    if ((e = staged_copy(sl->d, src, n, s)) != cudaSuccess) return e;
    if ((e = cudaEventRecord(sl->ev, s)) != cudaSuccess) return e;
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return e;
    std::memcpy(dst, sl->p, n);
    return cudaSuccess;
  }

 private:
  struct Slot {
    void* p = nullptr;   // host address
    void* d = nullptr;   // its device alias
    size_t cap = 0;
    cudaEvent_t ev = nullptr;
  };
  // A slot is free once the event recorded behind its last copy has completed
  // (queried, never waited on).  When no slot of the device's ring is free the
  // ring grows by one, so the host never blocks on the GPU here: the ring ends
  // as deep as the most uploads the caller ever kept in flight.
  struct Ring {
    std::vector<Slot*> slot;
    size_t cap = size_t(4) << 20;   // capacity of every slot made from now on
  };
  static bool idle(const Slot& sl) { return !sl.ev || cudaEventQuery(sl.ev) == cudaSuccess; }
  static cudaError_t pin(Slot& sl, size_t cap) {
    if (sl.p) cudaFreeHost(sl.p);
    sl.p = sl.d = nullptr;
    sl.cap = 0;
    cudaError_t e = cudaHostAlloc(&sl.p, cap, cudaHostAllocMapped | cudaHostAllocPortable);
    if (e != cudaSuccess) return e;
    if ((e = cudaHostGetDevicePointer(&sl.d, sl.p, 0)) != cudaSuccess) {
      cudaFreeHost(sl.p);
      sl.p = nullptr;
      return e;
    }
    sl.cap = cap;
    return cudaSuccess;
  }
  cudaError_t take(size_t n, Slot** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    Ring& ring = rings_[dev];
    if (ring.cap < n) {
      // Pinning host memory stalls transfers in flight on the GPU's host link
      // (a caller's input copy of 2.75 GB took 174 ms instead of 13 ms when it
      // overlapped one), so every idle slot grows at once, to a power of two of
      // at least 4 MB: after the first calls nothing is pinned again.
      while (ring.cap < n) ring.cap <<= 1;
      for (Slot* o : ring.slot)
        if (o->cap < ring.cap && idle(*o) && (e = pin(*o, ring.cap)) != cudaSuccess) return e;
    }
    Slot* sl = nullptr;
    for (Slot* o : ring.slot)
      if (o->cap >= n && idle(*o)) { sl = o; break; }
    if (!sl) {
      for (Slot* o : ring.slot)   // an idle slot left small by an earlier growth
        if (idle(*o)) { sl = o; break; }
      if (sl && (e = pin(*sl, ring.cap)) != cudaSuccess) return e;
    }
    if (!sl) {
      ring.slot.push_back(new Slot());
      sl = ring.slot.back();
      if ((e = pin(*sl, ring.cap)) != cudaSuccess) return e;
    }
    if (!sl->ev && (e = cudaEventCreateWithFlags(&sl->ev, cudaEventDisableTiming)) != cudaSuccess) return e;
    *out = sl;
    return cudaSuccess;
  }
  std::mutex mu_;
  std::map<int, Ring> rings_;
};

}  // namespace

PageableUploads::PageableUploads() : prev_(t_pageable_only) { t_pageable_only = true; }
PageableUploads::~PageableUploads() { t_pageable_only = prev_; }

namespace {

Staging& staging() {
  static Staging* st = new Staging();   // process lifetime: the pinned slots outlive every call
  return *st;
}

constexpr size_t kAlign = 256;
// Every workspace of the selection, recall and index calls starts with this
// header; its first word is the call's device error word (zeroed by the call's
// plan upload, set by a kernel whose bounded wait gave up), which
// saki_workspace_status reads.
constexpr size_t kHeader = 256;
constexpr int kNumSMs = 152;

// One-shot stall for the failure-reporting test (saki_debug_inject_stall): the
// next launch of the armed kernel kind gets a producer that issues no loads.
std::atomic<int> g_stall_kind{0};
int take_stall(int kind) {
  int expect = kind;
  return g_stall_kind.compare_exchange_strong(expect, 0) ? 1 : 0;
}

// Work lists are uploaded from host memory that lives only for the call, so a
// captured call would replay a copy from freed memory: refuse stream capture.
bool capturing(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  return cudaStreamIsCapturing(s, &st) == cudaSuccess && st != cudaStreamCaptureStatusNone;
}
inline size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }
inline saki_status cuda_status(cudaError_t e) { return e == cudaSuccess ? SAKI_OK : SAKI_ERR_CUDA; }
inline bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline int kp_of(int k) { return k <= 64 ? 64 : 128; }

saki_status check_cfg(const saki_config* c) {
  if (!c) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->num_q_heads < 1 || c->num_kv_heads < 1 || c->num_q_heads % c->num_kv_heads) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->num_q_heads > 65535) return SAKI_ERR_UNSUPPORTED;
  if (c->head_dim < 1) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->head_dim != kD) return SAKI_ERR_UNSUPPORTED;
  if (c->rank < 1 || c->rank > c->head_dim) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->topk < 1) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->topk > 128) return SAKI_ERR_UNSUPPORTED;
  if (c->dtype != SAKI_F32 && c->dtype != SAKI_BF16) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->center != 0 && c->center != 1) return SAKI_ERR_INVALID_ARGUMENT;
  if (!(c->eig_floor_rel >= 0.f && c->eig_floor_rel < 1.f)) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->max_sweeps < 0) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->flags & ~(SAKI_FLAG_SORTED | SAKI_FLAG_CHECK | SAKI_FLAG_SHRINK)) return SAKI_ERR_INVALID_ARGUMENT;
  if (c->method < SAKI_METHOD_SAKI || c->method > SAKI_METHOD_SAP_MAP) return SAKI_ERR_INVALID_ARGUMENT;
  return SAKI_OK;
}

saki_status check_layout(const saki_layout* L, int64_t* total_keys) {
  if (!L || L->num_seqs < 1 || !L->seq_offsets || L->num_queries < 0) return SAKI_ERR_INVALID_ARGUMENT;
  if (L->num_queries > INT32_MAX) return SAKI_ERR_UNSUPPORTED;
  if (L->num_queries > 0 && (!L->q_seq || !L->q_visible)) return SAKI_ERR_INVALID_ARGUMENT;
  if (L->seq_offsets[0] != 0) return SAKI_ERR_INVALID_ARGUMENT;
  for (int s = 0; s < L->num_seqs; ++s) {
    const int64_t len = L->seq_offsets[s + 1] - L->seq_offsets[s];
    if (len < 0) return SAKI_ERR_INVALID_ARGUMENT;
    if (len > INT32_MAX - 1) return SAKI_ERR_UNSUPPORTED;
  }
  for (int64_t t = 0; t < L->num_queries; ++t) {
    const int32_t s = L->q_seq[t];
    if (s < 0 || s >= L->num_seqs) return SAKI_ERR_INVALID_ARGUMENT;
    const int64_t v = L->q_visible[t];
    if (v < 0 || v > L->seq_offsets[s + 1] - L->seq_offsets[s]) return SAKI_ERR_INVALID_ARGUMENT;
  }
  *total_keys = L->seq_offsets[L->num_seqs];
  return SAKI_OK;
}

// ------------------------------------------------------------------ work plan
struct Plan {
  int nq = 1;   // launch width: smallest power of two >= the largest group
  std::vector<ScoreItem> items;
  std::vector<MergeItem> merges;
  std::vector<ScoreItem> sitems;    // sample pass of the seeded groups
  std::vector<MergeItem> smerges;   // its merges, which write the seeds
  std::vector<int32_t> vis;
  int64_t cand_slots = 0, scand_slots = 0;
  // workspace offsets (bytes)
  size_t off_items = 0, off_merges = 0, off_sitems = 0, off_smerges = 0, off_vis = 0, off_err = 0, off_cand = 0,
         off_scand = 0, off_seed = 0, bytes = 0, staged = 0;
};

constexpr int kSeedMinSplits = 8;    // groups cut into at least this many splits are seeded
constexpr int64_t kSeedKeys = 1024;  // sample keys per split (at most an eighth of a split)

// Groups of up to kGroupQ consecutive queries of one sequence; a group's visible
// range is cut into splits so that the grid has several CTAs per SM.
//
// Seeding (groups of the tensor-core decode kernel with many splits): a split
// that starts from an empty candidate buffer admits every key until its
// threshold has risen, and for a 27,648-key split and k = 64 that is about 800
// appends and five re-sorts per query.  A sample pass first reads the first
// kSeedKeys keys of every split and keeps, per query, the best score of each of
// the split's 128 key groups (one key per tile and thread); the seed merge takes
// the k-th largest of these group maxima over all splits of the row.  k distinct
// visible keys reach it, so it bounds the row's k-th best score from below and
// the main pass may start each query's threshold there (about 50 appends per
// split and query in place of 800, no re-sort).  The result is unchanged: every
// key of the row's top k scores at least the seed.
Plan make_plan(const saki_layout* L, int Hq, int kp, int dtype, int P, bool seed = true) {
  Plan p;
  const int64_t T = L->num_queries;
  struct G { int32_t b, n; int64_t vmax; int32_t seq; };
  std::vector<G> groups;
  int64_t work = 0;
  for (int64_t t = 0; t < T;) {
    G g{(int32_t)t, 0, 0, L->q_seq[t]};
    while (t < T && L->q_seq[t] == g.seq && g.n < kGroupQ) {
      g.vmax = std::max(g.vmax, L->q_visible[t]);
      ++g.n;
      ++t;
    }
    work += g.vmax;
    while (p.nq < g.n) p.nq *= 2;
    groups.push_back(g);
  }
  const int64_t target_per_head = std::max<int64_t>(1, (int64_t)8 * kNumSMs / Hq);
  int64_t chunk = std::max<int64_t>(2048, (work + target_per_head - 1) / target_per_head);
  chunk = (chunk + 255) / 256 * 256;
  // split length between 70 % and 100 % of that (never longer: a group keeps at
  // least the splits that make it seeded), chosen so the (item, head) CTAs
  // fill their last wave best (CTAs resident per SM from the scoring kernel's
  // occupancy; 1216 CTAs of three per SM left a last wave two-thirds full)
  const int per_sm = score_ctas_per_sm(dtype, P, kp, p.nq);
  int64_t base_items = 0;
  for (const G& g : groups) base_items += g.vmax > 0 ? (g.vmax + chunk - 1) / chunk : 1;
  // only where the waves are few: past four, a part-filled last wave costs
  // little and the extra splits (more items, longer merges) cost more
  if (per_sm > 0 && !groups.empty() && base_items * Hq <= (int64_t)4 * kNumSMs * per_sm) {
    const int64_t slots = (int64_t)kNumSMs * per_sm;
    double best_fill = -1.0;
    int64_t best_c = chunk;
    for (int i = -6; i <= 0; ++i) {
      const int64_t c = std::min(chunk, (chunk * (20 + i) / 20 + 255) / 256 * 256);
      if (c < 2048) continue;
      int64_t items = 0;
      for (const G& g : groups) items += g.vmax > 0 ? (g.vmax + c - 1) / c : 1;
      const int64_t ctas = items * Hq;
      const double fill = (double)ctas / (double)(((ctas + slots - 1) / slots) * slots);
      if (fill > best_fill + 1e-9 || (fill > best_fill - 1e-9 && c > best_c)) {
        best_fill = fill;
        best_c = c;
      }
    }
    chunk = best_c;
  }
  // the tensor-core kernel takes groups of at least four queries
  const bool seedable = seed && decode_tc_eligible(dtype, P, p.nq);
  const int64_t samp = std::min<int64_t>(kSeedKeys, chunk / 8 / 128 * 128);
  for (const G& g : groups) {
    const int64_t base = L->seq_offsets[g.seq];
    const int32_t S = g.vmax > 0 ? (int32_t)((g.vmax + chunk - 1) / chunk) : 1;
    if (S == 1) {
      p.items.push_back(ScoreItem{g.b, g.n, 0, (int32_t)g.vmax, base, -1, 0, 0});
      continue;
    }
    const bool seeded = seedable && S >= kSeedMinSplits;
    const int64_t slot0 = p.cand_slots;
    p.cand_slots += (int64_t)g.n * S;
    const int64_t sslot0 = p.scand_slots;
    if (seeded) p.scand_slots += (int64_t)g.n * S;
    for (int32_t s = 0; s < S; ++s) {
      const int64_t lo = s * chunk, hi = std::min<int64_t>(g.vmax, lo + chunk);
      p.items.push_back(ScoreItem{g.b, g.n, (int32_t)lo, (int32_t)hi, base, slot0 + s, S, seeded ? 1 : 0});
      if (seeded)
        p.sitems.push_back(ScoreItem{g.b, g.n, (int32_t)lo, (int32_t)std::min(hi, lo + samp), base, sslot0 + s, S, 0});
    }
    for (int32_t b = 0; b < g.n; ++b) {
      p.merges.push_back(MergeItem{g.b + b, S, slot0 + (int64_t)b * S});
      if (seeded) p.smerges.push_back(MergeItem{g.b + b, S, sslot0 + (int64_t)b * S});
    }
  }
  p.vis.resize(T);
  for (int64_t t = 0; t < T; ++t) p.vis[t] = (int32_t)L->q_visible[t];
  p.off_err = 0;   // the header's error word, zeroed by the upload
  p.off_items = kHeader;
  p.off_merges = p.off_items + align_up(p.items.size() * sizeof(ScoreItem));
  p.off_sitems = p.off_merges + align_up(p.merges.size() * sizeof(MergeItem));
  p.off_smerges = p.off_sitems + align_up(p.sitems.size() * sizeof(ScoreItem));
  p.off_vis = p.off_smerges + align_up(p.smerges.size() * sizeof(MergeItem));
  p.staged = p.off_vis + p.vis.size() * sizeof(int32_t);
  p.off_cand = align_up(p.staged);
  p.off_scand = p.off_cand + align_up((size_t)p.cand_slots * Hq * kp * sizeof(uint64_t));
  p.off_seed = p.off_scand + align_up((size_t)p.scand_slots * Hq * kp * sizeof(uint64_t));
  p.bytes = p.off_seed + (p.sitems.empty() ? 0 : align_up((size_t)Hq * T * sizeof(uint64_t)));
  return p;
}

// Score and merge the plan's items: the sample pass and its seed merge first when
// the plan has seeded groups, then every split and the merge into idx / score.
cudaError_t run_plan(ScoreArgs a, const Plan& p, char* ws, int dtype, int kp, cudaStream_t s) {
  cudaError_t e;
  a.seed = nullptr;
  a.seed_out = nullptr;
  a.sample = 0;
  if (!p.sitems.empty()) {
    ScoreArgs b = a;
    b.items = reinterpret_cast<const ScoreItem*>(ws + p.off_sitems);
    b.merges = reinterpret_cast<const MergeItem*>(ws + p.off_smerges);
    b.n_items = (int32_t)p.sitems.size();
    b.n_merges = (int32_t)p.smerges.size();
    b.cand = reinterpret_cast<uint64_t*>(ws + p.off_scand);
    b.cand_per_head = p.scand_slots;
    b.idx = nullptr;
    b.score = nullptr;
    b.seed_out = reinterpret_cast<uint64_t*>(ws + p.off_seed);
    b.sample = 1;
    if ((e = launch_score_generic(b, dtype, kp, p.nq, s)) != cudaSuccess) return e;
    if ((e = launch_merge(b, dtype, kp, s)) != cudaSuccess) return e;
    a.seed = b.seed_out;
  }
  if ((e = launch_score_generic(a, dtype, kp, p.nq, s)) != cudaSuccess) return e;
  return launch_merge(a, dtype, kp, s);
}

// The plan for a call: the seeded one, or the same splits without the sample
// pass when the workspace holds only that (same results, slower; a caller with a
// fixed scratch, such as saki_score_topk_noalloc, keeps working at sizes the
// sample lists would push past it).
Plan plan_for(const saki_layout* L, int Hq, int kp, int dtype, int P, size_t workspace_bytes, size_t extra) {
  Plan p = make_plan(L, Hq, kp, dtype, P);
  if (!p.sitems.empty() && workspace_bytes < p.bytes + extra) {
    Plan q = make_plan(L, Hq, kp, dtype, P, false);
    if (workspace_bytes >= q.bytes + extra) return q;
  }
  return p;
}

saki_status upload_plan(const Plan& p, char* ws, cudaStream_t s) {
  if (p.staged == 0) return SAKI_OK;
  std::vector<char> host(p.staged, 0);
  if (!p.items.empty()) std::memcpy(host.data() + p.off_items, p.items.data(), p.items.size() * sizeof(ScoreItem));
  if (!p.merges.empty())
    std::memcpy(host.data() + p.off_merges, p.merges.data(), p.merges.size() * sizeof(MergeItem));
  if (!p.sitems.empty())
    std::memcpy(host.data() + p.off_sitems, p.sitems.data(), p.sitems.size() * sizeof(ScoreItem));
  if (!p.smerges.empty())
    std::memcpy(host.data() + p.off_smerges, p.smerges.data(), p.smerges.size() * sizeof(MergeItem));
  if (!p.vis.empty()) std::memcpy(host.data() + p.off_vis, p.vis.data(), p.vis.size() * sizeof(int32_t));
  return staging().upload(ws, host.data(), p.staged, s) == cudaSuccess ? SAKI_OK : SAKI_ERR_CUDA;
}

// Tensor-core plan: tiles of up to 128 consecutive queries of one sequence,
// heaviest first; the workspace holds the tiles, the visible counts, the error
// word, the exact three-way bf16 split of the projection and the mean terms.
struct TcPlan {
  std::vector<TcTile> tiles;
  std::vector<int32_t> vis;
  size_t off_vis = 0, off_err = 0, staged = 0, off_w = 0, off_qnu = 0, bytes = 0;
};

TcPlan make_tc_plan(const saki_layout* L, int Hq, int P, bool with_qnu) {
  TcPlan p;
  const int64_t T = L->num_queries;
  for (int64_t t = 0; t < T;) {
    TcTile tl{(int32_t)t, 0, L->seq_offsets[L->q_seq[t]], 0, 0};
    const int32_t seq = L->q_seq[t];
    while (t < T && L->q_seq[t] == seq && tl.nrows < 128) {
      tl.vis_max = std::max<int32_t>(tl.vis_max, (int32_t)L->q_visible[t]);
      ++tl.nrows;
      ++t;
    }
    p.tiles.push_back(tl);
  }
  std::stable_sort(p.tiles.begin(), p.tiles.end(),
                   [](const TcTile& a, const TcTile& b) { return a.vis_max > b.vis_max; });
  p.vis.resize(T);
  for (int64_t t = 0; t < T; ++t) p.vis[t] = (int32_t)L->q_visible[t];
  p.off_err = 0;   // the header's error word, zeroed by the upload
  p.off_vis = kHeader + align_up(p.tiles.size() * sizeof(TcTile));
  p.staged = p.off_vis + p.vis.size() * sizeof(int32_t);
  p.off_w = align_up(p.staged);
  p.off_qnu = p.off_w + align_up((size_t)Hq * 3 * P * kD * 2);
  p.bytes = p.off_qnu + (with_qnu ? align_up((size_t)Hq * T * sizeof(float)) : 0);
  return p;
}

// The tensor-core kernel serves bf16 data, K widths 16/32/64/128, k <= 64, queries
// that see at most 65535 keys, and layouts whose query tiles average at least 32
// rows (prefill-like); everything else goes to the CUDA-core kernel.
bool use_tc(const saki_config* c, const saki_layout* L, int P) {
  if (c->dtype != SAKI_BF16 || !tc_supported(P) || c->topk > 64 || L->num_queries == 0) return false;
  for (int64_t t = 0; t < L->num_queries; ++t)
    if (L->q_visible[t] > 65535) return false;   // candidate lists hold 16-bit key offsets
  int64_t tiles = 0;
  for (int64_t t = 0; t < L->num_queries;) {
    const int32_t seq = L->q_seq[t];
    int n = 0;
    while (t < L->num_queries && L->q_seq[t] == seq && n < 128) { ++n; ++t; }
    ++tiles;
  }
  return L->num_queries >= 32 * tiles;
}

saki_status upload_tc_plan(const TcPlan& p, char* ws, cudaStream_t s) {
  std::vector<char> host(p.staged, 0);
  if (!p.tiles.empty()) std::memcpy(host.data() + kHeader, p.tiles.data(), p.tiles.size() * sizeof(TcTile));
  if (!p.vis.empty()) std::memcpy(host.data() + p.off_vis, p.vis.data(), p.vis.size() * sizeof(int32_t));
  return staging().upload(ws, host.data(), p.staged, s) == cudaSuccess ? SAKI_OK : SAKI_ERR_CUDA;
}

int num_sms() {
  int dev = 0, n = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : kNumSMs;
}

// Run the tensor-core selection: W is L (approximate, X = codes) or A (exact, X = keys).
saki_status run_tc(const saki_config* cfg, const saki_layout* layout, const TcPlan& p, int P, bool exact,
                   const void* Q, const float* W, const void* X, const float* nu, int32_t* idx, float* score,
                   char* ws, cudaStream_t s) {
  saki_status st = upload_tc_plan(p, ws, s);
  if (st != SAKI_OK) return st;
  void* wsplit = ws + p.off_w;
  if (launch_pack_w(W, cfg->num_q_heads, P, wsplit, s) != cudaSuccess) return SAKI_ERR_CUDA;
  float* qnu = nullptr;
  if (nu && score) {
    qnu = reinterpret_cast<float*>(ws + p.off_qnu);
    if (launch_qnu(Q, nu, layout->num_queries, cfg->num_q_heads, qnu, s) != cudaSuccess) return SAKI_ERR_CUDA;
  }
  TcLaunch L{};
  L.Q = Q;
  L.X = X;
  L.Wsplit = wsplit;
  L.P = P;
  L.Hk = cfg->num_kv_heads;
  L.num_sms = num_sms();
  TcArgs& a = L.args;
  a.tiles = reinterpret_cast<const TcTile*>(ws + kHeader);
  a.vis = reinterpret_cast<const int32_t*>(ws + p.off_vis);
  a.qnu = qnu;
  a.idx = idx;
  a.score = score;
  a.err = reinterpret_cast<int*>(ws + p.off_err);
  a.T = layout->num_queries;
  a.N = layout->seq_offsets[layout->num_seqs];
  a.n_items = (int32_t)(p.tiles.size() * cfg->num_q_heads);
  a.Hq = cfg->num_q_heads;
  a.G = cfg->num_q_heads / cfg->num_kv_heads;
  a.k = cfg->topk;
  a.exact = exact ? 1 : 0;
  a.sorted = (cfg->flags & SAKI_FLAG_SORTED) ? 1 : 0;
  a.stall = take_stall(exact ? SAKI_KERNEL_EXACT : SAKI_KERNEL_SELECT);
  KernelTimer kt(exact ? SAKI_KERNEL_EXACT : SAKI_KERNEL_SELECT, s);
  return cuda_status(launch_score_tc(L, s));
}

// Index build on the tensor cores: bf16 data, uncentered keys (codes of centered
// keys keep the CUDA-core path, which subtracts mu before the products), r a
// multiple of 16 dividing 128.  Items: (KV head, 128-column block, 32 key tiles).
struct BuildWs { std::vector<BuildItem> items; size_t off_err, off_w, bytes; bool tc; };
BuildWs build_ws(const saki_config* c, int64_t N) {
  BuildWs w{};
  const int G = c->num_q_heads / c->num_kv_heads;
  w.tc = c->dtype == SAKI_BF16 && !c->center && build_tc_supported(c->rank, G) && N > 0;
  w.off_err = 0;
  if (!w.tc) { w.bytes = kHeader; return w; }
  const int ncb = (G * c->rank + 127) / 128;
  const int64_t tiles = (N + 127) / 128;
  for (int g = 0; g < c->num_kv_heads; ++g)
    for (int cb = 0; cb < ncb; ++cb)
      for (int64_t t = 0; t < tiles; t += 32)
        w.items.push_back(BuildItem{g, cb, (int32_t)t, (int32_t)std::min<int64_t>(tiles, t + 32)});
  w.off_w = kHeader + align_up(w.items.size() * sizeof(BuildItem));
  w.bytes = w.off_w + align_up(build_tc_workspace(c->num_q_heads, c->rank));
  return w;
}

// fit workspace: S, F, G [(Hq+Hk)][d][d], mu [Hk][d], status [Hq+Hk], C'^T scratch [Hq][d][d]
struct FitWs { size_t S, F, G, mu, st, C, I, sig, acc4, bytes; };
// Key PCA also needs an identity operator per query head and its own sigma.
FitWs fit_ws(const saki_config* c) {
  const size_t nm = (size_t)c->num_q_heads + c->num_kv_heads;
  const size_t mat = nm * kD * kD * sizeof(float);
  FitWs w;
  w.S = 0;
  w.F = align_up(mat);
  w.G = w.F + align_up(mat);
  w.mu = w.G + align_up(mat);
  w.st = w.mu + align_up((size_t)c->num_kv_heads * kD * sizeof(float));
  w.C = w.st + align_up(nm * sizeof(int));
  w.I = w.C + align_up((size_t)c->num_q_heads * kD * kD * sizeof(float));
  w.sig = w.I;
  w.bytes = w.I;
  if (c->method == SAKI_METHOD_KEY_PCA) {
    w.sig = w.I + align_up((size_t)c->num_q_heads * kD * kD * sizeof(float));
    w.bytes = w.sig + align_up((size_t)c->num_q_heads * kD * sizeof(float));
  }
  if (c->method == SAKI_METHOD_SAP_SVD) {   // the fold reads sigma_r even when the caller asks for none
    w.sig = w.I;
    w.bytes = w.sig + align_up((size_t)c->num_q_heads * kD * sizeof(float));
  }
  w.acc4 = w.bytes;   // Ledoit-Wolf: sum_t ||x_t||^4 per moment matrix
  if (c->flags & SAKI_FLAG_SHRINK) w.bytes = w.acc4 + align_up(nm * sizeof(double));
  return w;
}

size_t recall_extra(const saki_config* c, int64_t T, bool with_idx) {
  return align_up((size_t)c->num_q_heads * 2 * sizeof(unsigned long long)) +
         (with_idx ? align_up((size_t)c->num_q_heads * T * c->topk * sizeof(int32_t)) : 0);
}

// Read the header's error word once the stream has run up to here.
saki_status read_status(const void* workspace, cudaStream_t s) {
  int word = 0;
  if (staging().download_sync(&word, workspace, sizeof(int), s) != cudaSuccess) return SAKI_ERR_CUDA;
  return word ? SAKI_ERR_TIMEOUT : SAKI_OK;
}

// A call's return: its launch status, then, with SAKI_FLAG_CHECK, the device
// status of what it launched.
saki_status finish(const saki_config* cfg, saki_status st, const void* workspace, cudaStream_t s) {
  if (st != SAKI_OK || !(cfg->flags & SAKI_FLAG_CHECK)) return st;
  return read_status(workspace, s);
}

// The fit after the moments (Prop. 1 / Sec. 6 and the comparison indexes):
// factors of the moments in the workspace's S, the SVD fit, the method's fold,
// and the status words.  Shared by saki_fit and saki_fit_moments.
saki_status fit_from_moments(const saki_config* cfg, const FitWs& w, char* ws, float* muw, const float* A, float* L,
                             float* R, float* nu, float* sigma, float* loss, cudaStream_t s) {
  saki_status st;
  const int Hq = cfg->num_q_heads, Hk = cfg->num_kv_heads, nm = Hq + Hk;
  float* S = reinterpret_cast<float*>(ws + w.S);
  float* F = reinterpret_cast<float*>(ws + w.F);
  float* Gm = reinterpret_cast<float*>(ws + w.G);
  int* status = reinterpret_cast<int*>(ws + w.st);
  const int sweeps = cfg->max_sweeps > 0 ? cfg->max_sweeps : 40;
  // The comparison indexes reuse the fit with other inputs: weight SVD whitens
  // with identity factors (C' = A); key PCA keeps the key factors and sets the
  // query factors and the operator to the identity (C' = F_k, whose left singular
  // vectors are Sk's eigenvectors), then folds A into L.
  const int method = cfg->method;
  float* Iw = reinterpret_cast<float*>(ws + w.I);
  float* sig = (method == SAKI_METHOD_KEY_PCA || method == SAKI_METHOD_SAP_SVD) && !sigma
                   ? reinterpret_cast<float*>(ws + w.sig) : sigma;
  {
    KernelTimer kt(SAKI_KERNEL_FACTOR, s);
    if (method == SAKI_METHOD_WEIGHT_SVD) {
      if ((st = cuda_status(launch_identity(F, nm, s))) != SAKI_OK) return st;
      if ((st = cuda_status(launch_identity(Gm, nm, s))) != SAKI_OK) return st;
    } else {
      // SAP-svd needs the symmetric key roots (the right singular vectors of C itself)
      const int sym_from = method == SAKI_METHOD_SAP_SVD ? Hq : (1 << 30);
      if ((st = cuda_status(launch_factor(S, nm, cfg->eig_floor_rel, sweeps, F, Gm, status, s, sym_from))) !=
          SAKI_OK)
        return st;
    }
    if (method == SAKI_METHOD_KEY_PCA) {
      if ((st = cuda_status(launch_identity(F, Hq, s))) != SAKI_OK) return st;
      if ((st = cuda_status(launch_identity(Gm, Hq, s))) != SAKI_OK) return st;
      if ((st = cuda_status(launch_identity(Iw, Hq, s))) != SAKI_OK) return st;
    }
  }
  {
    KernelTimer kt(SAKI_KERNEL_FIT, s);
    const float* Afit = method == SAKI_METHOD_KEY_PCA ? Iw : A;
    if ((st = cuda_status(launch_fit(Afit, F, Gm, cfg->center ? muw : nullptr, Hq, Hk, cfg->rank, sweeps,
                                     reinterpret_cast<float*>(ws + w.C), L, R, sig, loss, nu, status, s))) !=
        SAKI_OK)
      return st;
    if (method == SAKI_METHOD_KEY_PCA &&
        (st = cuda_status(launch_key_pca_fold(A, sig, cfg->center ? muw : nullptr, Hq, Hk, cfg->rank, L, R, nu,
                                              s))) != SAKI_OK)
      return st;
    if ((method == SAKI_METHOD_SAP_SVD || method == SAKI_METHOD_SAP_MAP) &&
        (st = cuda_status(launch_sap_fold(A, F, sig, Hq, Hk, cfg->rank, method == SAKI_METHOD_SAP_SVD, L, R, s))) !=
            SAKI_OK)
      return st;
  }
  std::vector<int> hst(nm);
  if ((st = cuda_status(staging().download_sync(hst.data(), status, nm * sizeof(int), s))) != SAKI_OK) return st;
  int acc = 0;
  for (int v : hst) acc |= v;
  if (acc & kStTimeout) return SAKI_ERR_TIMEOUT;
  if (acc & kStNonFinite) return SAKI_ERR_NUMERIC;
  if (acc & kStNotConverged) return SAKI_ERR_NOT_CONVERGED;
  return SAKI_OK;
}

}  // namespace

extern "C" {

saki_status saki_workspace_status(const void* workspace, saki_stream stream) {
  if (!workspace || !al16(workspace)) return SAKI_ERR_INVALID_ARGUMENT;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  return read_status(workspace, s);
}

saki_status saki_key_spectrum(const saki_config* cfg, int64_t n_calib, const void* k_calib, float tau_int,
                              float* eig, int32_t* spikes, void* workspace, size_t workspace_bytes,
                              saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (n_calib < 1 || !k_calib || !eig || !spikes || !workspace || !(tau_int >= 1.f)) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {k_calib, (const void*)eig, (const void*)spikes, (const void*)workspace})
    if (!al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  const int Hk = cfg->num_kv_heads;
  const size_t off_mu = align_up((size_t)Hk * kD * kD * sizeof(float));
  const size_t off_st = off_mu + align_up((size_t)Hk * kD * sizeof(float));
  if (workspace_bytes < off_st + align_up((size_t)Hk * sizeof(int))) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  char* ws = static_cast<char*>(workspace);
  float* S = reinterpret_cast<float*>(ws);
  int* status = reinterpret_cast<int*>(ws + off_st);
  if ((st = cuda_status(cudaMemsetAsync(status, 0, Hk * sizeof(int), s))) != SAKI_OK) return st;
  // key moments only (Hq = 0), centered as cfg->center says
  if ((st = cuda_status(launch_gram(nullptr, k_calib, n_calib, 0, Hk, cfg->center, cfg->dtype, S,
                                    reinterpret_cast<float*>(ws + off_mu), status, s))) != SAKI_OK)
    return st;
  const double q_eff = (double)kD * tau_int / (double)n_calib;
  const float edge = (float)((1.0 + std::sqrt(q_eff)) * (1.0 + std::sqrt(q_eff)));
  const int sweeps = cfg->max_sweeps > 0 ? cfg->max_sweeps : 40;
  if ((st = cuda_status(launch_spectrum(S, Hk, edge, sweeps, eig, spikes, status, s))) != SAKI_OK) return st;
  std::vector<int> hst(Hk);
  if ((st = cuda_status(staging().download_sync(hst.data(), status, Hk * sizeof(int), s))) != SAKI_OK) return st;
  int acc = 0;
  for (int v : hst) acc |= v;
  if (acc & kStTimeout) return SAKI_ERR_TIMEOUT;
  if (acc & kStNotConverged) return SAKI_ERR_NOT_CONVERGED;
  return SAKI_OK;
}

saki_status saki_score_mse(const saki_config* cfg, const saki_layout* layout, int64_t key_stride, const void* Q,
                           const float* A, const void* K, const float* L, const void* sketch, const float* nu,
                           double* out, void* workspace, size_t workspace_bytes, saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  int64_t N = 0;
  if ((st = check_layout(layout, &N)) != SAKI_OK) return st;
  const int64_t T = layout->num_queries;
  if (key_stride < 1 || !out || !workspace || (T > 0 && (!Q || !A || !L || (N > 0 && (!K || !sketch)))))
    return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {Q, (const void*)A, K, (const void*)L, sketch, (const void*)nu, (const void*)out,
                        (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  const size_t need = kHeader + align_up((size_t)T * 2 * sizeof(int64_t));
  if (workspace_bytes < need) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  char* ws = static_cast<char*>(workspace);
  std::vector<char> host(kHeader + (size_t)T * 2 * sizeof(int64_t), 0);
  int64_t* qi = reinterpret_cast<int64_t*>(host.data() + kHeader);
  for (int64_t t = 0; t < T; ++t) {
    qi[2 * t] = layout->seq_offsets[layout->q_seq[t]];
    qi[2 * t + 1] = layout->q_visible[t];
  }
  if ((st = cuda_status(staging().upload(ws, host.data(), host.size(), s))) != SAKI_OK) return st;
  const int Hq = cfg->num_q_heads;
  if ((st = cuda_status(cudaMemsetAsync(out, 0, (size_t)Hq * 3 * sizeof(double), s))) != SAKI_OK) return st;
  return finish(cfg,
                cuda_status(launch_score_mse(Q, A, K, L, sketch, nu, reinterpret_cast<const int64_t*>(ws + kHeader), T,
                                             N, Hq, Hq / cfg->num_kv_heads, cfg->rank, key_stride, cfg->dtype, out,
                                             s)),
                ws, s);
}

saki_status saki_merge_topk(const saki_config* cfg, int32_t num_parts, int64_t num_rows, const int32_t* idx_parts,
                            const float* score_parts, const int64_t* part_offsets, int32_t* idx, float* score,
                            saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (num_parts < 1 || num_rows < 0 || !part_offsets) return SAKI_ERR_INVALID_ARGUMENT;
  if (num_parts > kMaxParts) return SAKI_ERR_UNSUPPORTED;
  if (num_rows > 0 && (!idx_parts || !score_parts || !idx)) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {(const void*)idx_parts, (const void*)score_parts, (const void*)idx, (const void*)score})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  PartOffsets po{};
  for (int p = 0; p < num_parts; ++p) {
    if (part_offsets[p] < 0 || part_offsets[p] > INT32_MAX) return SAKI_ERR_INVALID_ARGUMENT;
    po.off[p] = part_offsets[p];
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return cuda_status(launch_merge_parts(idx_parts, score_parts, po, num_parts, num_rows, cfg->topk, idx, score, s));
}

saki_status saki_debug_inject_stall(int32_t kind) {
  if (kind != 0 && kind != SAKI_KERNEL_SELECT && kind != SAKI_KERNEL_EXACT && kind != SAKI_KERNEL_BUILD)
    return SAKI_ERR_INVALID_ARGUMENT;
  g_stall_kind.store(kind);
  return SAKI_OK;
}

const char* saki_status_string(saki_status s) {
  switch (s) {
    case SAKI_OK: return "ok";
    case SAKI_ERR_INVALID_ARGUMENT: return "invalid argument";
    case SAKI_ERR_UNSUPPORTED: return "unsupported by this build";
    case SAKI_ERR_CUDA: return "CUDA launch or copy failed";
    case SAKI_ERR_NUMERIC: return "non-finite calibration data or moments";
    case SAKI_ERR_NOT_CONVERGED: return "Jacobi SVD did not converge within max_sweeps";
    case SAKI_ERR_WORKSPACE: return "workspace too small";
    case SAKI_ERR_TIMEOUT: return "bounded device wait gave up";
  }
  return "unknown status";
}

const char* saki_version(void) { return "0.1.0"; }

size_t saki_workspace_size(const saki_config* cfg, int32_t op, const saki_layout* layout, int64_t n_calib,
                           int64_t total_keys) {
  if (check_cfg(cfg) != SAKI_OK) return 0;
  switch (op) {
    case SAKI_OP_FIT:
      return n_calib >= 1 ? fit_ws(cfg).bytes : 0;
    case SAKI_OP_BUILD_INDEX:
      return total_keys >= 0 ? build_ws(cfg, total_keys).bytes : 0;
    case SAKI_OP_MOMENTS:
      return kHeader + align_up((size_t)(cfg->num_q_heads + cfg->num_kv_heads) * kD * kD * sizeof(float)) +
             align_up((size_t)cfg->num_kv_heads * kD * sizeof(float));
    case SAKI_OP_RECONSTRUCT:   // total_keys: the number of rows to reconstruct
      return total_keys >= 0 ? std::max<size_t>(kAlign, align_up((size_t)total_keys * (kD / 2) * sizeof(float2))) : 0;
    case SAKI_OP_KEY_SPECTRUM:
      return align_up((size_t)cfg->num_kv_heads * kD * kD * sizeof(float)) +
             align_up((size_t)cfg->num_kv_heads * kD * sizeof(float)) +
             align_up((size_t)cfg->num_kv_heads * sizeof(int));
    case SAKI_OP_SCORE_MSE: {
      int64_t n = 0;
      if (check_layout(layout, &n) != SAKI_OK) return 0;
      return kHeader + align_up((size_t)layout->num_queries * 2 * sizeof(int64_t));
    }
    case SAKI_OP_SCORE_TOPK:
    case SAKI_OP_RECALL: {
      int64_t n = 0;
      if (check_layout(layout, &n) != SAKI_OK) return 0;
      const int P = op == SAKI_OP_RECALL ? kD : cfg->rank;
      size_t b;
      if (use_tc(cfg, layout, P))
        b = make_tc_plan(layout, cfg->num_q_heads, P, op == SAKI_OP_SCORE_TOPK).bytes;
      else
        b = make_plan(layout, cfg->num_q_heads, kp_of(cfg->topk), cfg->dtype, P).bytes;
      if (op == SAKI_OP_RECALL) b += recall_extra(cfg, layout->num_queries, true);
      return b;
    }
  }
  return 0;
}

saki_status saki_fit(const saki_config* cfg, int64_t n_calib, const void* q_calib, const void* k_calib,
                     const float* A, float* L, float* R, float* mu, float* nu, float* sigma, float* loss,
                     void* workspace, size_t workspace_bytes, saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (n_calib < 1 || !q_calib || !k_calib || !A || !L || !R || !workspace) return SAKI_ERR_INVALID_ARGUMENT;
  if (cfg->center && !mu) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {q_calib, k_calib, (const void*)A, (const void*)L, (const void*)R, (const void*)mu,
                        (const void*)nu, (const void*)sigma, (const void*)loss, (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  const FitWs w = fit_ws(cfg);
  if (workspace_bytes < w.bytes) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  char* ws = static_cast<char*>(workspace);
  const int Hq = cfg->num_q_heads, Hk = cfg->num_kv_heads, nm = Hq + Hk;
  float* S = reinterpret_cast<float*>(ws + w.S);
  float* muw = mu ? mu : reinterpret_cast<float*>(ws + w.mu);
  int* status = reinterpret_cast<int*>(ws + w.st);
  if ((st = cuda_status(cudaMemsetAsync(status, 0, nm * sizeof(int), s))) != SAKI_OK) return st;
  if (!cfg->center && mu && (st = cuda_status(cudaMemsetAsync(mu, 0, (size_t)Hk * kD * sizeof(float), s))) != SAKI_OK)
    return st;
  {
    KernelTimer kt(SAKI_KERNEL_MOMENTS, s);
    if ((st = cuda_status(launch_gram(q_calib, k_calib, n_calib, Hq, Hk, cfg->center, cfg->dtype, S, muw, status,
                                      s))) != SAKI_OK)
      return st;
  }
  if (cfg->flags & SAKI_FLAG_SHRINK) {   // Sec. 7: Ledoit-Wolf shrinkage of both moments
    double* acc4 = reinterpret_cast<double*>(ws + w.acc4);
    if ((st = cuda_status(cudaMemsetAsync(acc4, 0, nm * sizeof(double), s))) != SAKI_OK) return st;
    if ((st = cuda_status(launch_fourth_moment(q_calib, k_calib, n_calib, Hq, Hk, cfg->center ? muw : nullptr,
                                               cfg->dtype, acc4, s))) != SAKI_OK)
      return st;
    if ((st = cuda_status(launch_shrink(S, acc4, n_calib, nm, nullptr, s))) != SAKI_OK) return st;
  }
  return fit_from_moments(cfg, w, ws, muw, A, L, R, nu, sigma, loss, s);
}

saki_status saki_moments(const saki_config* cfg, int64_t n_new, const void* q_new, const void* k_new, int64_t n_prev,
                         float* Sq, float* Sk, float* mu, void* workspace, size_t workspace_bytes,
                         saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (n_new < 1 || n_prev < 0 || !q_new || !k_new || !Sq || !Sk || !workspace) return SAKI_ERR_INVALID_ARGUMENT;
  if (cfg->center && !mu) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {q_new, k_new, (const void*)Sq, (const void*)Sk, (const void*)mu, (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  const int Hq = cfg->num_q_heads, Hk = cfg->num_kv_heads;
  const size_t off_S = kHeader, off_mu = off_S + align_up((size_t)(Hq + Hk) * kD * kD * sizeof(float));
  if (workspace_bytes < off_mu + align_up((size_t)Hk * kD * sizeof(float))) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  char* ws = static_cast<char*>(workspace);
  float* Sb = reinterpret_cast<float*>(ws + off_S);
  float* mub = reinterpret_cast<float*>(ws + off_mu);
  if ((st = cuda_status(cudaMemsetAsync(ws, 0, sizeof(int), s))) != SAKI_OK) return st;   // the header's error word
  {
    KernelTimer kt(SAKI_KERNEL_MOMENTS, s);
    if ((st = cuda_status(launch_gram(q_new, k_new, n_new, Hq, Hk, cfg->center, cfg->dtype, Sb, mub,
                                      reinterpret_cast<int*>(ws), s))) != SAKI_OK)
      return st;
  }
  return finish(cfg, cuda_status(launch_merge_moments(Sq, Sk, mu, Sb, mub, Hq, Hk, n_prev, n_new, cfg->center, s)),
                ws, s);
}

saki_status saki_fit_moments(const saki_config* cfg, const float* Sq, const float* Sk, const float* mu,
                             const float* A, float* L, float* R, float* nu, float* sigma, float* loss,
                             void* workspace, size_t workspace_bytes, saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (cfg->flags & SAKI_FLAG_SHRINK) return SAKI_ERR_UNSUPPORTED;   // needs the calibration rows
  if (!Sq || !Sk || !A || !L || !R || !workspace) return SAKI_ERR_INVALID_ARGUMENT;
  if (cfg->center && !mu) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {(const void*)Sq, (const void*)Sk, (const void*)mu, (const void*)A, (const void*)L,
                        (const void*)R, (const void*)nu, (const void*)sigma, (const void*)loss, (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  const FitWs w = fit_ws(cfg);
  if (workspace_bytes < w.bytes) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  char* ws = static_cast<char*>(workspace);
  const int Hq = cfg->num_q_heads, Hk = cfg->num_kv_heads, nm = Hq + Hk;
  float* S = reinterpret_cast<float*>(ws + w.S);
  float* muw = reinterpret_cast<float*>(ws + w.mu);
  const size_t mat = (size_t)kD * kD * sizeof(float);
  if ((st = cuda_status(cudaMemsetAsync(ws + w.st, 0, nm * sizeof(int), s))) != SAKI_OK) return st;
  if ((st = cuda_status(cudaMemcpyAsync(S, Sq, Hq * mat, cudaMemcpyDeviceToDevice, s))) != SAKI_OK) return st;
  if ((st = cuda_status(cudaMemcpyAsync(S + (size_t)Hq * kD * kD, Sk, Hk * mat, cudaMemcpyDeviceToDevice, s))) !=
      SAKI_OK)
    return st;
  if (cfg->center &&
      (st = cuda_status(cudaMemcpyAsync(muw, mu, (size_t)Hk * kD * sizeof(float), cudaMemcpyDeviceToDevice, s))) !=
          SAKI_OK)
    return st;
  return fit_from_moments(cfg, w, ws, muw, A, L, R, nu, sigma, loss, s);
}

saki_status saki_reconstruct_keys(const saki_config* cfg, int64_t n_rows, const int64_t* rows, int64_t total_keys,
                                  const void* sketch, const float* L, const float* nu, const int64_t* positions,
                                  float rope_theta, void* keys, void* workspace, size_t workspace_bytes,
                                  saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (n_rows < 0 || total_keys < 0 || (n_rows > 0 && (!rows || !sketch || !L || !keys)))
    return SAKI_ERR_INVALID_ARGUMENT;
  if (positions && (!(rope_theta > 1.f) || !workspace)) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {(const void*)rows, sketch, (const void*)L, (const void*)nu, (const void*)positions,
                        (const void*)keys, (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  if (positions && workspace_bytes < (size_t)n_rows * (kD / 2) * sizeof(float2)) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return cuda_status(launch_reconstruct(rows, n_rows, sketch, total_keys, L, nu, cfg->num_q_heads, cfg->rank,
                                        positions, rope_theta, static_cast<float2*>(workspace), cfg->dtype, keys, s));
}

saki_status saki_build_index(const saki_config* cfg, int64_t total_keys, const void* K, const float* R,
                             const float* mu, void* sketch, void* workspace, size_t workspace_bytes,
                             saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  if (total_keys < 0 || (total_keys > 0 && (!K || !R || !sketch))) return SAKI_ERR_INVALID_ARGUMENT;
  if (cfg->center && !mu) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {K, (const void*)R, (const void*)mu, (const void*)sketch})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const BuildWs w = build_ws(cfg, total_keys);
  if (w.tc) {
    if (!workspace) return SAKI_ERR_INVALID_ARGUMENT;
    if (workspace_bytes < w.bytes) return SAKI_ERR_WORKSPACE;
    if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
    char* ws = static_cast<char*>(workspace);
    std::vector<char> host(kHeader + w.items.size() * sizeof(BuildItem), 0);
    std::memcpy(host.data() + kHeader, w.items.data(), w.items.size() * sizeof(BuildItem));
    if ((st = cuda_status(staging().upload(ws, host.data(), host.size(), s))) != SAKI_OK) return st;
    {
      KernelTimer kt(SAKI_KERNEL_BUILD, s);
      st = cuda_status(launch_build_tc(K, R, sketch, total_keys, cfg->num_q_heads,
                                       cfg->num_q_heads / cfg->num_kv_heads, cfg->rank,
                                       reinterpret_cast<const BuildItem*>(ws + kHeader), (int)w.items.size(),
                                       ws + w.off_w, reinterpret_cast<int*>(ws + w.off_err),
                                       take_stall(SAKI_KERNEL_BUILD), num_sms(), s));
    }
    return finish(cfg, st, workspace, s);
  }
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  // the CUDA-core build has no bounded wait: its status is always ok, and a
  // workspace passed along gets a zeroed header so that it reads so
  if (workspace && workspace_bytes >= kHeader &&
      (st = cuda_status(cudaMemsetAsync(workspace, 0, sizeof(int), s))) != SAKI_OK)
    return st;
  {
    KernelTimer kt(SAKI_KERNEL_BUILD, s);
    st = cuda_status(launch_build_generic(K, R, cfg->center ? mu : nullptr, sketch, total_keys, cfg->num_q_heads,
                                          cfg->num_q_heads / cfg->num_kv_heads, cfg->rank, cfg->center,
                                          cfg->dtype, s));
  }
  return workspace ? finish(cfg, st, workspace, s) : st;
}

saki_status saki_score_topk(const saki_config* cfg, const saki_layout* layout, const void* Q, const float* L,
                            const void* sketch, const float* nu, int32_t* idx, float* score, void* workspace,
                            size_t workspace_bytes, saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  int64_t N = 0;
  if ((st = check_layout(layout, &N)) != SAKI_OK) return st;
  const int64_t T = layout->num_queries;
  if (T > 0 && (!Q || !L || !idx || !workspace || (N > 0 && !sketch))) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {Q, (const void*)L, sketch, (const void*)nu, (const void*)idx, (const void*)score,
                        (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  if (T == 0) return SAKI_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(workspace);
  if (use_tc(cfg, layout, cfg->rank)) {
    const TcPlan tp = make_tc_plan(layout, cfg->num_q_heads, cfg->rank, true);
    if (workspace_bytes < tp.bytes) return SAKI_ERR_WORKSPACE;
    if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
    return finish(cfg, run_tc(cfg, layout, tp, cfg->rank, false, Q, L, sketch, nu, idx, score, ws, s), ws, s);
  }
  const int kp = kp_of(cfg->topk);
  const Plan p = plan_for(layout, cfg->num_q_heads, kp, cfg->dtype, cfg->rank, workspace_bytes, 0);
  if (workspace_bytes < p.bytes) return SAKI_ERR_WORKSPACE;
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;
  if ((st = upload_plan(p, ws, s)) != SAKI_OK) return st;
  ScoreArgs a{};
  a.Q = Q; a.X = sketch; a.W = L; a.nu = nu;
  a.items = reinterpret_cast<const ScoreItem*>(ws + p.off_items);
  a.merges = reinterpret_cast<const MergeItem*>(ws + p.off_merges);
  a.vis = reinterpret_cast<const int32_t*>(ws + p.off_vis);
  a.idx = idx; a.score = score;
  a.cand = reinterpret_cast<uint64_t*>(ws + p.off_cand);
  a.cand_per_head = p.cand_slots;
  a.err = reinterpret_cast<int*>(ws + p.off_err);
  a.T = T; a.N = N;
  a.Hq = cfg->num_q_heads; a.G = cfg->num_q_heads / cfg->num_kv_heads; a.P = cfg->rank; a.k = cfg->topk;
  a.exact = 0;
  a.n_items = (int32_t)p.items.size();
  a.n_merges = (int32_t)p.merges.size();
  a.stall = take_stall(SAKI_KERNEL_SELECT);
  {
    KernelTimer kt(SAKI_KERNEL_SELECT, s);
    st = cuda_status(run_plan(a, p, ws, cfg->dtype, kp, s));
  }
  return finish(cfg, st, ws, s);
}

saki_status saki_recall(const saki_config* cfg, const saki_layout* layout, int64_t min_visible, const void* Q,
                        const float* A, const void* K, const int32_t* idx_approx, int32_t* idx_exact, float* recall,
                        void* workspace, size_t workspace_bytes, saki_stream stream) {
  saki_status st = check_cfg(cfg);
  if (st != SAKI_OK) return st;
  int64_t N = 0;
  if ((st = check_layout(layout, &N)) != SAKI_OK) return st;
  const int64_t T = layout->num_queries;
  if (!recall || !workspace || (T > 0 && (!Q || !A || !idx_approx || (N > 0 && !K)))) return SAKI_ERR_INVALID_ARGUMENT;
  for (const void* p : {Q, (const void*)A, K, (const void*)idx_approx, (const void*)idx_exact, (const void*)recall,
                        (const void*)workspace})
    if (p && !al16(p)) return SAKI_ERR_INVALID_ARGUMENT;
  const int kp = kp_of(cfg->topk);
  const bool tc = use_tc(cfg, layout, kD);
  const size_t extra = recall_extra(cfg, T, idx_exact == nullptr);
  const Plan p = tc ? Plan{} : plan_for(layout, cfg->num_q_heads, kp, cfg->dtype, kD, workspace_bytes, extra);
  const TcPlan tp = tc ? make_tc_plan(layout, cfg->num_q_heads, kD, false) : TcPlan{};
  const size_t base = tc ? tp.bytes : p.bytes;
  const size_t need = base + extra;
  if (workspace_bytes < need) return SAKI_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (capturing(s)) return SAKI_ERR_UNSUPPORTED;   // after every host-side check above
  char* ws = static_cast<char*>(workspace);
  unsigned long long* counters = reinterpret_cast<unsigned long long*>(ws + base);
  int32_t* ie = idx_exact ? idx_exact
                          : reinterpret_cast<int32_t*>(ws + base + align_up((size_t)cfg->num_q_heads * 2 *
                                                                            sizeof(unsigned long long)));
  int64_t vmax = 0;   // the longest visible prefix: sizes the recall kernel's bitmap
  for (int64_t t = 0; t < T; ++t) vmax = layout->q_visible[t] > vmax ? layout->q_visible[t] : vmax;
  if (tc) {
    if ((st = run_tc(cfg, layout, tp, kD, true, Q, A, K, nullptr, ie, nullptr, ws, s)) != SAKI_OK) return st;
    return finish(cfg,
                  cuda_status(launch_recall(idx_approx, ie, reinterpret_cast<const int32_t*>(ws + tp.off_vis), T,
                                            cfg->num_q_heads, cfg->topk, min_visible, vmax, counters, recall, s)),
                  ws, s);
  }
  if (T == 0 && (st = cuda_status(cudaMemsetAsync(ws, 0, sizeof(int), s))) != SAKI_OK) return st;
  if (T > 0) {
    if ((st = upload_plan(p, ws, s)) != SAKI_OK) return st;
    ScoreArgs a{};
    a.Q = Q; a.X = K; a.W = A; a.nu = nullptr;
    a.items = reinterpret_cast<const ScoreItem*>(ws + p.off_items);
    a.merges = reinterpret_cast<const MergeItem*>(ws + p.off_merges);
    a.vis = reinterpret_cast<const int32_t*>(ws + p.off_vis);
    a.idx = ie; a.score = nullptr;
    a.cand = reinterpret_cast<uint64_t*>(ws + p.off_cand);
    a.cand_per_head = p.cand_slots;
    a.err = reinterpret_cast<int*>(ws + p.off_err);
    a.T = T; a.N = N;
    a.Hq = cfg->num_q_heads; a.G = cfg->num_q_heads / cfg->num_kv_heads; a.P = kD; a.k = cfg->topk;
    a.exact = 1;
    a.n_items = (int32_t)p.items.size();
    a.n_merges = (int32_t)p.merges.size();
    a.stall = take_stall(SAKI_KERNEL_EXACT);
    KernelTimer kt(SAKI_KERNEL_EXACT, s);
    if ((st = cuda_status(run_plan(a, p, ws, cfg->dtype, kp, s))) != SAKI_OK) return st;
  }
  const int32_t* vis = reinterpret_cast<const int32_t*>(ws + p.off_vis);
  return finish(cfg,
                cuda_status(launch_recall(idx_approx, ie, vis, T, cfg->num_q_heads, cfg->topk, min_visible, vmax,
                                          counters, recall, s)),
                ws, s);
}

}  // extern "C"
