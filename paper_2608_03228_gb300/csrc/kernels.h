// Internal interface between the C-ABI layer (api.cu) and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace saki {

// ---------------------------------------------------------------- profiling aids
void note_launch();   // called at every kernel launch of the library

// While alive on this thread, the library's plan uploads use plain pageable
// copies instead of its pinned staging ring (whose first use allocates pinned
// host memory): for the entry points that promise to allocate nothing.
class PageableUploads {
 public:
  PageableUploads();
  ~PageableUploads();
  PageableUploads(const PageableUploads&) = delete;
  PageableUploads& operator=(const PageableUploads&) = delete;

 private:
  bool prev_;
};

// Kernel kinds timed by saki_kernel_timer_* (values match the SAKI_KERNEL_* macros).
constexpr int kTimedKinds = 7;
// While the kind is armed, records one CUDA event on construction and one on
// destruction, on stream s (bracket the launch of that kind).
class KernelTimer {
 public:
  KernelTimer(int kind, cudaStream_t s);
  ~KernelTimer();
  KernelTimer(const KernelTimer&) = delete;
  KernelTimer& operator=(const KernelTimer&) = delete;

 private:
  int kind_;
  cudaStream_t s_;
  cudaEvent_t stop_;
};

// One unit of scoring work: up to kGroupQ consecutive queries of one sequence
// against keys [key_lo, key_hi) of that sequence (a split of its visible range).
struct ScoreItem {
  int32_t q_begin;      // first query row in Q
  int32_t q_count;      // queries in the group
  int32_t key_lo;       // sequence-local first key of this split
  int32_t key_hi;       // sequence-local end of this split
  int64_t key_base;     // global row of the sequence's key 0
  int64_t cand;         // -1: write final lists; else candidate slot of (row 0, this split)
  int32_t cand_stride;  // slots between consecutive rows (= number of splits)
  int32_t seeded;       // 1: start each query's threshold at ScoreArgs::seed of its row
};

// Merge of the per-split candidate lists of one query.
struct MergeItem {
  int32_t t;        // query row
  int32_t nsplit;   // number of candidate lists
  int64_t cand;     // slot of split 0 (lists are consecutive slots)
};

constexpr int kGroupQ = 8;  // queries per generic work item

struct ScoreArgs {
  const void* Q;        // [Hq][T][d]
  const void* X;        // codes [Hq][N][P] (approximate) or keys [Hk][N][d] (exact)
  const float* W;       // projection [Hq][d][P]: L (approximate) or A (exact)
  const float* nu;      // [Hq][d] or null
  const ScoreItem* items;
  const MergeItem* merges;
  const int32_t* vis;   // [T] visible keys per query
  int32_t* idx;         // [Hq][T][k]
  float* score;         // [Hq][T][k] or null
  uint64_t* cand;       // candidate lists, kp keys per slot, per head: cand_per_head slots
  int64_t cand_per_head;
  int* err;             // zeroed workspace word; the tensor-core variant sets kStTimeout if a bounded wait gave up
  const uint64_t* seed; // [Hq][T] per-row lower bound on the row's k-th best key (read by seeded items), or null
  uint64_t* seed_out;   // merge only: write each merged row's k-th best key here instead of idx / score
  int64_t T, N;
  int32_t Hq, G, P, k, exact, n_items, n_merges;
  int32_t sample;       // tensor-core variant only: write each query's kp best group maxima (a sample pass)
  int32_t stall;        // test hook: the tensor-core variant's producer issues no loads (its waits run out)
};

// generic CUDA-core scoring (any rank, f32 or bf16)
// nq: query-group width of the launch (1, 2, 4 or 8), at least every item's q_count
cudaError_t launch_score_generic(const ScoreArgs& a, int dtype, int kp, int nq, cudaStream_t s);
// true when launch_score_generic runs the tensor-core variant for these arguments
bool decode_tc_eligible(int dtype, int P, int nq);
cudaError_t launch_merge(const ScoreArgs& a, int dtype, int kp, cudaStream_t s);
size_t score_generic_smem(int P, int kp, int nq);
// CTAs of the decode-shaped scoring kernel that serves (dtype, P, kp, group
// width nq) resident per SM (0 if the query fails)
int score_ctas_per_sm(int dtype, int P, int kp, int nq);

// calibration moments: S [(Hq+Hk)][d][d] (queries first), mu [Hk][d]; err: set to 1
// if a bounded wait of the tensor-core path gave up
cudaError_t launch_gram(const void* q_calib, const void* k_calib, int64_t n, int Hq, int Hk,
                        int center, int dtype, float* S, float* mu, int* err, cudaStream_t s);

// factor F (F F^T = S, floor applied, row-major) and G = pseudo-inverse transpose of F
// (stored transposed, i.e. column-major), per matrix
// matrices m >= sym_from store the symmetric roots (eigen path) instead
cudaError_t launch_factor(const float* S, int nmat, float floor_rel, int max_sweeps,
                          float* F, float* Gm, int* status, cudaStream_t s, int sym_from = 1 << 30);
// projector variants (SAP-svd: svd = 1, SAP-map: svd = 0) folded from a SAKI fit
cudaError_t launch_sap_fold(const float* A, const float* F, const float* sigma, int Hq, int Hk, int r, int svd,
                            float* L, float* R, cudaStream_t s);

// per query head: C' = Fq^T A Fk, Jacobi SVD, factors L, R, sigma, loss, nu
// Cws: scratch [Hq][d][d] (C'^T per head)
cudaError_t launch_fit(const float* A, const float* F, const float* Gm, const float* mu, int Hq,
                       int Hk, int r, int max_sweeps, float* Cws, float* L, float* R, float* sigma,
                       float* loss, float* nu, int* status, cudaStream_t s);
// comparison indexes: identity matrices [nmat][d][d]; the key-PCA rescale and
// operator fold after a fit of C' = F_k (sigma of that fit, mu may be null)
cudaError_t launch_identity(float* X, int nmat, cudaStream_t s);
cudaError_t launch_key_pca_fold(const float* A, const float* sigma, const float* mu, int Hq, int Hk, int r, float* L,
                                float* R, float* nu, cudaStream_t s);

// key codes
cudaError_t launch_build_generic(const void* K, const float* R, const float* mu, void* sketch,
                                 int64_t N, int Hq, int G, int r, int center, int dtype,
                                 cudaStream_t s);

// recall counters [Hq][2] (matches, rows) and final per-head recall
// max_visible: the largest visible count of any query (sizes the bitmap path)
cudaError_t launch_recall(const int32_t* idx_a, const int32_t* idx_e, const int32_t* vis,
                          int64_t T, int Hq, int k, int64_t min_visible, int64_t max_visible,
                          unsigned long long* counters, float* recall, cudaStream_t s);

// ---------------------------------------------------------------- tensor-core path
// A tile: up to 128 consecutive queries of one sequence, ranked against that
// sequence's first vis_max keys (each row against its own visible prefix).
struct TcTile {
  int32_t q0;
  int32_t nrows;
  int64_t key_base;
  int32_t vis_max;
  int32_t pad;
};

struct TcArgs {
  const TcTile* tiles;
  const int32_t* vis;   // [T]
  const float* qnu;     // [Hq][T] mean term added to reported scores, or null
  int32_t* idx;         // [Hq][T][k]
  float* score;         // [Hq][T][k] or null
  int* err;             // set to 1 if a bounded wait gave up
  int64_t T, N;
  int32_t n_items, Hq, G, k, exact, sorted;
  int32_t stall;        // test hook: the producer issues no loads, so the consumers' bounded waits run out
};

struct TcLaunch {
  const void* Q;        // [Hq][T][d] bf16
  const void* X;        // codes [Hq][N][P] (approximate) or keys [Hk][N][d] (exact), bf16
  const void* Wsplit;   // [Hq][3][P][d] bf16 from launch_pack_w
  int P, Hk, num_sms;
  TcArgs args;
};

bool tc_supported(int P);
cudaError_t launch_pack_w(const float* W, int Hq, int P, void* out, cudaStream_t s);
cudaError_t launch_qnu(const void* Q, const float* nu, int64_t T, int Hq, float* out, cudaStream_t s);
cudaError_t launch_score_tc(const TcLaunch& L, cudaStream_t s);

// ---------------------------------------------------------------- tensor-core index build
// A build item: KV head g, block cb of <= 128 output columns (heads hl*r+c of the
// group), key tiles [t0, t1) of 128 keys.
struct BuildItem {
  int32_t g, cb, t0, t1;
};
bool build_tc_supported(int r, int G);
size_t build_tc_workspace(int Hq, int r);
cudaError_t launch_build_tc(const void* K, const float* R, void* sketch, int64_t N, int Hq, int G, int r,
                            const BuildItem* items, int n_items, void* wsplit, int* err, int stall,
                            int num_sms, cudaStream_t s);

// ---------------------------------------------------------------- merge of per-part lists
constexpr int kMaxParts = 64;
struct PartOffsets {
  int64_t off[kMaxParts];   // key offset of each part's range (added to its local indices)
};
// idx_in, score_in [parts][rows][k] (part-local indices, -1 padding); idx, score
// [rows][k]: the k best of the union, descending, global indices
cudaError_t launch_merge_parts(const int32_t* idx_in, const float* score_in, const PartOffsets& po, int parts,
                               int64_t rows, int k, int32_t* idx, float* score, cudaStream_t s);

// ---------------------------------------------------------------- Sec. 7 / App. C diagnostics
// sum_t ||x_t - mu||^4 per calibration matrix (keys centered on mu when given) into acc (zeroed)
cudaError_t launch_fourth_moment(const void* q, const void* k, int64_t n, int Hq, int Hk, const float* mu, int dtype,
                                 double* acc, cudaStream_t s);
// Ledoit-Wolf shrinkage of nmat moment matrices in place (rho per matrix if given)
cudaError_t launch_shrink(float* S, const double* acc4, int64_t n, int nmat, float* rho, cudaStream_t s);
// eigenvalues (descending) of each correlation matrix of S, and the count above edge
cudaError_t launch_spectrum(const float* S, int nmat, float edge, int max_sweeps, float* lam, int* spikes, int* status,
                            cudaStream_t s);
// per head: sum s^2, sum (s - s_hat)^2, pairs over every stride-th visible key (out [Hq][3], zeroed)
cudaError_t launch_score_mse(const void* Q, const float* A, const void* K, const float* L, const void* codes,
                             const float* nu, const int64_t* qinfo, int64_t T, int64_t N, int Hq, int G, int r,
                             int64_t stride, int dtype, double* out, cudaStream_t s);

// ---------------------------------------------------------------- online moments, RoPE composition
// running moments (Sq [Hq], Sk [Hk], mu [Hk], n1 rows) merged in place with a batch's (Sb [(Hq+Hk)], mub, n2 rows)
cudaError_t launch_merge_moments(float* Sq, float* Sk, float* mu, const float* Sb, const float* mub, int Hq, int Hk,
                                 int64_t n1, int64_t n2, int center, cudaStream_t s);
// k_hat = nu + L c of the given code rows per query head, RoPE-rotated when positions are given
// (table: workspace of n_rows * d/2 float2)
cudaError_t launch_reconstruct(const int64_t* rows, int64_t n_rows, const void* codes, int64_t N, const float* L,
                               const float* nu, int Hq, int r, const int64_t* positions, float theta, float2* table,
                               int dtype, void* out, cudaStream_t s);

}  // namespace saki
