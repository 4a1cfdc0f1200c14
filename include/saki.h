/*
 * saki.h -- C ABI of the GB300 (sm_103a) SAKI score-map retrieval library.
 *
 * SAKI (arXiv 2608.03228) indexes a KV cache with a per-head rank-r score map.
 * For query head h reading KV head g(h) = h / (Hq / Hk):
 *   - fit (Prop. 1, Eq. 3, Sec. 5; Sec. 6; App. A): from calibration moments Sq (queries,
 *     uncentered) and Sk, mu (keys), form C = Sq^{1/2} A_h Sk^{1/2}, take its
 *     truncated SVD C_r = U_r Lambda_r V_r^T and fold M_r = Sq^{-1/2} C_r Sk^{-1/2}
 *     into L_h = Sq^{-1/2} U_r Lambda_r^{1/2} and R_h = Sk^{-1/2} V_r Lambda_r^{1/2};
 *   - index (Sec. 6): key codes c_j = R_h^T (k_j - mu_g);
 *   - select (Sec. 1, Sec. 6): s_hat_j = (L_h^T q)^T c_j over the keys a query
 *     can see, keep the k largest;
 *   - evaluate (Sec. 3 protocol): exact s_j = q^T A_h k_j, its top-k, recall@k.
 *
 * Conventions shared by every entry point
 *   Pointers.  Tensor arguments are DEVICE pointers on the current CUDA device,
 *     16-byte aligned, row-major with the last listed dimension fastest.  The
 *     layout description (saki_layout) is HOST memory.  The caller owns every
 *     buffer, including the workspace; the library allocates no device memory.
 *   Host staging.  The library's own small transfers (the work list a call
 *     builds on the host, status words read back) go through a ring of mapped
 *     pinned host slots per device that the library allocates on first use
 *     (cudaHostAlloc, at least 4 MB a slot) and keeps for the life of the
 *     process; a copy kernel on `stream` moves them, so they never queue behind
 *     the caller's large copies on other streams.  A slot is reused once the
 *     copy that last read it has run; when none is free the ring grows by one
 *     slot instead of blocking the host.  saki_score_topk_noalloc stages
 *     through pageable memory instead and pins nothing.
 *   Streams.  Work is enqueued on `stream` (NULL = legacy default stream) and
 *     the calls return without waiting for it, except saki_fit, which
 *     synchronises the stream once to report numeric status, and calls made
 *     with SAKI_FLAG_CHECK.  A stream in capture mode is refused
 *     (SAKI_ERR_UNSUPPORTED, nothing enqueued): each call uploads a work list
 *     from host memory that lives only for the call.
 *   Errors.  Arguments are checked before any launch; on SAKI_ERR_INVALID_ARGUMENT,
 *     SAKI_ERR_UNSUPPORTED or SAKI_ERR_WORKSPACE nothing is launched and no
 *     output is touched.  SAKI_ERR_CUDA reports a failed launch or copy (the
 *     CUDA error is left for cudaGetLastError()).  Every wait inside a kernel
 *     is bounded (about two seconds); a kernel whose wait runs out stops,
 *     leaves its outputs partly written and sets the error word in the first
 *     bytes of the call's workspace.  saki_score_topk, saki_recall and
 *     saki_build_index return before their kernels run, so that word is read
 *     by saki_workspace_status (or by the call itself under SAKI_FLAG_CHECK),
 *     which returns SAKI_ERR_TIMEOUT when it is set.
 *   dtype.  SAKI_F32 or SAKI_BF16 applies to queries, keys, calibration data and
 *     key codes; A, L, R, mu, nu, sigma, loss and scores are always float32.
 *   GQA.  Query head h uses KV head h / (num_q_heads / num_kv_heads).
 */
#ifndef SAKI_H_
#define SAKI_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SAKI_API __attribute__((visibility("default")))
#else
#define SAKI_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* saki_stream; /* same handle as cudaStream_t */

typedef enum saki_status {
  SAKI_OK = 0,
  SAKI_ERR_INVALID_ARGUMENT = 1, /* bad pointer, size, shape or flag */
  SAKI_ERR_UNSUPPORTED = 2,      /* valid request outside what this build implements */
  SAKI_ERR_CUDA = 3,             /* a CUDA launch or copy failed */
  SAKI_ERR_NUMERIC = 4,          /* non-finite calibration data or moments */
  SAKI_ERR_NOT_CONVERGED = 5,    /* Jacobi sweep limit reached for some head */
  SAKI_ERR_WORKSPACE = 6,        /* workspace smaller than saki_workspace_size() */
  SAKI_ERR_TIMEOUT = 7           /* a bounded device-side wait gave up */
} saki_status;

typedef enum saki_dtype { SAKI_F32 = 0, SAKI_BF16 = 1 } saki_dtype;

/* saki_config.flags */
#define SAKI_FLAG_SORTED 1 /* top-k lists in descending score (ties: lower index) */
#define SAKI_FLAG_CHECK 2  /* saki_score_topk, saki_recall, saki_build_index (and the
                              no-alloc selection) synchronise `stream` before returning
                              and report the device status of their kernels, as
                              saki_workspace_status does */
#define SAKI_FLAG_SHRINK 4 /* saki_fit: Ledoit-Wolf shrinkage of both moments (Sec. 7):
                              S <- (1 - rho) S + rho (tr S / d) I, rho = min(b2, d2) / d2,
                              d2 = ||S - (tr S / d) I||_F^2,
                              b2 = (1/n^2) sum_t ||x_t x_t^T - S||_F^2 (keys centered
                              when center = 1) */

/* saki_config.method: which rank-r map saki_fit folds into L and R */
#define SAKI_METHOD_SAKI 0       /* the exact optimum M_r of Prop. 1 (default) */
#define SAKI_METHOD_KEY_PCA 1    /* Tab. 1 comparison: M = A_h V_r V_r^T, V_r the r leading
                                    eigenvectors of Sk; L = A_h V_r, R = V_r */
#define SAKI_METHOD_WEIGHT_SVD 2 /* Tab. 1 comparison: the truncated SVD of A_h itself,
                                    L = U_r Sigma_r^{1/2}, R = V_r Sigma_r^{1/2} */
#define SAKI_METHOD_SAP_SVD 3    /* Sec. 6 projector variant: M = A_h Q Q^T with Q the r
                                    leading right singular vectors of C = Sq^{1/2} A_h Sk^{1/2}
                                    (symmetric roots), used directly as key directions;
                                    L = A_h Q, R = Q */
#define SAKI_METHOD_SAP_MAP 4    /* Sec. 6 projector variant: M = A_h Q Q^T with Q an
                                    orthonormal basis (Gram-Schmidt, in column order) of the
                                    optimum's key-side span, span((Sk^{1/2})^+ V_r),
                                    (Sk^{1/2})^+ the pseudo-inverse of the symmetric root
                                    under the eigenvalue floor;
                                    L = A_h Q, R = Q */

typedef struct saki_config {
  int32_t num_q_heads;   /* Hq >= 1 */
  int32_t num_kv_heads;  /* Hk >= 1, Hq % Hk == 0 */
  int32_t head_dim;      /* d; this build supports d = 128 */
  int32_t rank;          /* r, 1 <= r <= d */
  int32_t topk;          /* k, 1 <= k <= 128 */
  int32_t dtype;         /* saki_dtype */
  int32_t center;        /* 1: centered keys (Sk centered, codes of k - mu); 0: mu = 0 */
  float eig_floor_rel;   /* eigenvalues below eig_floor_rel * lambda_max count as zero
                            (App. A, "Singular covariances"); the paper uses 1e-6 */
  int32_t max_sweeps;    /* Jacobi sweep limit of the fit; 0 selects 40 */
  int32_t flags;         /* SAKI_FLAG_* */
  int32_t method;        /* SAKI_METHOD_*; 0 = SAKI */
} saki_config;

/* Which keys each query may rank (HOST memory).  Keys of sequence s are rows
 * seq_offsets[s] .. seq_offsets[s+1]-1 of the key / code tensors; query t belongs
 * to sequence q_seq[t] and sees its first q_visible[t] keys (causal prefill: t+1;
 * decode: the whole sequence).  Returned key indices are sequence-local. */
typedef struct saki_layout {
  int32_t num_seqs;            /* S >= 1 */
  const int64_t* seq_offsets;  /* [S+1], non-decreasing, seq_offsets[0] == 0 */
  int64_t num_queries;         /* T >= 0 */
  const int32_t* q_seq;        /* [T], values in [0, S) */
  const int64_t* q_visible;    /* [T], 0 <= q_visible[t] <= length of its sequence */
} saki_layout;

/* Operation codes for saki_workspace_size */
#define SAKI_OP_FIT 0
#define SAKI_OP_BUILD_INDEX 1
#define SAKI_OP_SCORE_TOPK 2
#define SAKI_OP_RECALL 3
#define SAKI_OP_KEY_SPECTRUM 4
#define SAKI_OP_SCORE_MSE 5
#define SAKI_OP_MOMENTS 6
#define SAKI_OP_RECONSTRUCT 7   /* total_keys: the number of rows to reconstruct */

/* Bytes of device workspace `op` needs.  FIT uses n_calib; BUILD_INDEX uses
 * total_keys; SCORE_TOPK and RECALL use the layout.  Returns 0 if the arguments
 * are invalid.  For SCORE_TOPK and RECALL this is the size of the fastest plan;
 * when a decode-shaped layout would run a sample pass (see saki_score_topk) and
 * the workspace passed is too small for its lists but holds the plan without
 * it, the call runs that plan instead (same results, slower). */
SAKI_API size_t saki_workspace_size(const saki_config* cfg, int32_t op, const saki_layout* layout,
                           int64_t n_calib, int64_t total_keys);

/* saki_fit -- Prop. 1 (Eq. 3, Sec. 5), Sec. 6 and App. A: calibration moments, the exact
 * rank-r minimiser of the score distortion of Eq. (1), folded into factors.
 *   q_calib [Hq][n][d] dtype   calibration queries of each query head
 *   k_calib [Hk][n][d] dtype   calibration keys of each KV head
 *   A       [Hq][d][d] f32     score operator, s = q^T A k
 * Outputs (float32):
 *   L [Hq][d][r], R [Hq][d][r]  factors with L R^T = M_r; each column pair is
 *                               signed so that the largest-|.| entry of R[:, c]
 *                               is positive; columns follow descending sigma
 *   mu [Hk][d]      key means (required when center = 1, may be NULL otherwise)
 *   nu [Hq][d]      A_h mu_g, the exact mean term q^T nu (NULL = skip)
 *   sigma [Hq][d]   singular values of C, descending (NULL = skip)
 *   loss [Hq]       optimum sum_{i>r} sigma_i^2 (NULL = skip)
 * Moments are normalised by 1/n.  Synchronises `stream`; returns SAKI_ERR_NUMERIC
 * if a moment is not finite and SAKI_ERR_NOT_CONVERGED if a head's Jacobi SVD
 * reached max_sweeps (outputs are then still written from the last sweep).
 * The comparison methods fold other rank-r maps into the same L, R, which the
 * index and selection calls take unchanged:
 *   SAKI_METHOD_KEY_PCA     R = V_r (unit columns), L = A_h V_r; sigma holds the
 *                           square roots of Sk's eigenvalues and loss the
 *                           discarded key energy sum_{i>r} lambda_i(Sk); the
 *                           query calibration data is read but not used;
 *   SAKI_METHOD_WEIGHT_SVD  sigma are A_h's singular values and loss
 *                           sum_{i>r} sigma_i^2; the calibration data is only
 *                           checked and, when center = 1, gives mu;
 *   SAKI_METHOD_SAP_SVD,
 *   SAKI_METHOD_SAP_MAP     the projector variants; sigma and loss are those of
 *                           the SAKI optimum they are derived from (the
 *                           variant's own distortion is larger, Prop. 1).
 *                           Each column of R (= Q) is signed so that its
 *                           largest-|.| entry is positive. */
SAKI_API saki_status saki_fit(const saki_config* cfg, int64_t n_calib, const void* q_calib,
                     const void* k_calib, const float* A, float* L, float* R, float* mu,
                     float* nu, float* sigma, float* loss, void* workspace,
                     size_t workspace_bytes, saki_stream stream);

/* saki_moments -- online tracking of the calibration moments (Sec. 2: online
 * updates of Sq and Sk compose with the method).  Adds a batch of n_new
 * calibration rows to running moments that so far cover n_prev rows:
 *   q_new [Hq][n_new][d], k_new [Hk][n_new][d] (dtype)
 *   Sq [Hq][d][d], Sk [Hk][d][d] f32, in/out; mu [Hk][d] f32 in/out (keys'
 *   running mean, required when center = 1; zeroed when center = 0)
 * Moments are normalised by 1/n; with center = 1 the key moments are merged by
 * the pooled-variance identity, so after any sequence of calls they equal
 * saki_fit's moments of all the rows at once (up to rounding).  n_prev = 0
 * starts afresh (the inputs' previous contents are ignored).  Stream-ordered;
 * workspace of saki_workspace_size(SAKI_OP_MOMENTS) with the error-word header
 * (saki_workspace_status). */
SAKI_API saki_status saki_moments(const saki_config* cfg, int64_t n_new, const void* q_new,
                                  const void* k_new, int64_t n_prev, float* Sq, float* Sk, float* mu,
                                  void* workspace, size_t workspace_bytes, saki_stream stream);

/* saki_fit_moments -- saki_fit from given moments (Sq [Hq][d][d], Sk [Hk][d][d],
 * mu [Hk][d] when center = 1), e.g. the running moments of saki_moments: the
 * same factors, outputs, methods, status codes and workspace (SAKI_OP_FIT) as
 * saki_fit.  SAKI_FLAG_SHRINK needs the calibration rows and is refused
 * (SAKI_ERR_UNSUPPORTED). */
SAKI_API saki_status saki_fit_moments(const saki_config* cfg, const float* Sq, const float* Sk,
                                      const float* mu, const float* A, float* L, float* R, float* nu,
                                      float* sigma, float* loss, void* workspace, size_t workspace_bytes,
                                      saki_stream stream);

/* saki_reconstruct_keys -- composition with RoPE (Sec. 6: reconstruct
 * k_hat = mu + M_r (k - mu) and rotate).  For every query head h and each of
 * the n_rows code rows rows[i] (device int64, rows of the sketch; a row
 * outside [0, total_keys) reads nothing and its key comes out NaN):
 *   k_hat = nu_h + L_h c,  so that q^T k_hat is the index's score with the mean
 *   term (in the paper's head coordinates, where A is absorbed, nu = mu and
 *   L_h c = M_r (k - mu));
 * then, when positions (device int64 [n_rows]) is given, rotated by rotary
 * position embedding at positions[i], rotate-half convention: dimension
 * j < d/2 pairs with j + d/2 and turns by positions[i] * rope_theta^(-2j/d)
 * (rope_theta > 1; the angle is formed in fp64).
 *   sketch [Hq][total_keys][r] dtype, L [Hq][d][r] f32, nu [Hq][d] f32 or NULL,
 *   keys [Hq][n_rows][d] dtype (written).
 * Workspace (only with positions): saki_workspace_size(SAKI_OP_RECONSTRUCT,
 * total_keys = n_rows).  SAKI_ERR_INVALID_ARGUMENT for negative counts, NULL
 * tensors when n_rows > 0, positions without a workspace or with rope_theta
 * <= 1, or a misaligned pointer; SAKI_ERR_WORKSPACE if the workspace is too
 * small.  Stream-ordered; uploads nothing (so it may be captured). */
SAKI_API saki_status saki_reconstruct_keys(const saki_config* cfg, int64_t n_rows, const int64_t* rows,
                                           int64_t total_keys, const void* sketch, const float* L,
                                           const float* nu, const int64_t* positions, float rope_theta,
                                           void* keys, void* workspace, size_t workspace_bytes,
                                           saki_stream stream);

/* saki_build_index -- Sec. 6 key codes c_j = R_h^T (k_j - mu_g) for every query
 * head h and every key row j (all sequences at once).
 *   K      [Hk][total_keys][d] dtype
 *   R      [Hq][d][r] f32
 *   mu     [Hk][d] f32, read only when center = 1 (then required)
 *   sketch [Hq][total_keys][r] dtype, written; rounded to nearest-even.
 * Workspace: saki_workspace_size(SAKI_OP_BUILD_INDEX) bytes, required for bf16
 * uncentered keys (the tensor-core path, which reports a device timeout through
 * the header's error word); other builds take none (NULL allowed; a workspace
 * passed along gets its error word cleared).  SAKI_ERR_INVALID_ARGUMENT for
 * NULL tensors when total_keys > 0, a missing mu when center = 1, a missing
 * workspace on the tensor-core path or a misaligned pointer; SAKI_ERR_WORKSPACE
 * if the workspace is too small.  Stream-ordered. */
SAKI_API saki_status saki_build_index(const saki_config* cfg, int64_t total_keys, const void* K,
                             const float* R, const float* mu, void* sketch, void* workspace,
                             size_t workspace_bytes, saki_stream stream);

/* saki_score_topk -- Sec. 6 selection: per (head h, query t) the k keys of the
 * visible prefix with the largest s_hat = (L_h^T q_t)^T c_j, never forming the
 * T x N score matrix.
 *   Q      [Hq][T][d] dtype      queries
 *   L      [Hq][d][r] f32
 *   sketch [Hq][total_keys][r] dtype, total_keys = seq_offsets[S]
 *   nu     [Hq][d] f32 or NULL   adds q^T nu to reported scores (not to ranking)
 *   idx    [Hq][T][k] int32      sequence-local key indices, -1 where fewer than
 *                                k keys are visible
 *   score  [Hq][T][k] f32 or NULL   s_hat (+ q^T nu) of each idx entry, -inf pad
 * Ranking is by descending s_hat with equal scores ordered by the lower index.
 * Without SAKI_FLAG_SORTED the k entries of a row come in unspecified order.
 * Decode-shaped groups (at least four bf16 queries of one sequence whose keys
 * are cut into eight or more splits) first run a sample pass over the head of
 * every split, whose per-query bound starts each split's selection; the result
 * is the same as without it.
 * Workspace: saki_workspace_size(SAKI_OP_SCORE_TOPK) bytes, required when T > 0
 * (T = 0 returns SAKI_OK and launches nothing).  SAKI_ERR_INVALID_ARGUMENT for
 * a malformed layout (seq_offsets[0] != 0, a decreasing offset, q_seq out of
 * range, q_visible beyond its sequence) or NULL / misaligned tensors;
 * SAKI_ERR_UNSUPPORTED for d != 128, k > 128, more than 65535 query heads,
 * more than 2^31 - 1 queries or a sequence of more than 2^31 - 2 keys;
 * SAKI_ERR_WORKSPACE if the workspace holds neither plan.  Stream-ordered; a
 * device timeout is read by saki_workspace_status. */
SAKI_API saki_status saki_score_topk(const saki_config* cfg, const saki_layout* layout, const void* Q,
                            const float* L, const void* sketch, const float* nu, int32_t* idx,
                            float* score, void* workspace, size_t workspace_bytes,
                            saki_stream stream);

/* saki_recall -- Sec. 3 protocol: exact top-k by s = q^T A_h k over the visible
 * keys, and recall@k = |approx set & exact set| / k averaged over the queries of
 * each head with at least min_visible visible keys (the paper uses k + 1).
 *   Q [Hq][T][d] dtype, A [Hq][d][d] f32, K [Hk][total_keys][d] dtype
 *   idx_approx [Hq][T][k] int32   e.g. the output of saki_score_topk
 *   idx_exact  [Hq][T][k] int32 or NULL (then kept in the workspace)
 *   recall     [Hq] f32, NaN for a head with no qualifying query
 * Medians across heads (Tab. 1) are left to the caller.
 * Workspace: saki_workspace_size(SAKI_OP_RECALL) bytes, always required (it
 * holds the per-head counts, and the exact lists when idx_exact is NULL).
 * Errors as saki_score_topk (recall and workspace must not be NULL).
 * Stream-ordered; a device timeout is read by saki_workspace_status. */
SAKI_API saki_status saki_recall(const saki_config* cfg, const saki_layout* layout, int64_t min_visible,
                        const void* Q, const float* A, const void* K, const int32_t* idx_approx,
                        int32_t* idx_exact, float* recall, void* workspace,
                        size_t workspace_bytes, saki_stream stream);

/* saki_key_spectrum -- Sec. 7's random-matrix diagnostic: per KV head, the
 * eigenvalues of the key correlation matrix D^{-1/2} Sk D^{-1/2} (D = diag(Sk);
 * Sk centered when cfg->center = 1, from the n_calib rows of k_calib
 * [Hk][n][d]) in descending order, and how many lie above the Marchenko-Pastur
 * upper edge (1 + sqrt(q_eff))^2, q_eff = d tau_int / n_calib (tau_int >= 1,
 * the token autocorrelation time; 1 for independent draws).
 *   eig [Hk][d] f32, spikes [Hk] int32 (device); workspace of
 *   saki_workspace_size(SAKI_OP_KEY_SPECTRUM).
 * Synchronises `stream`; SAKI_ERR_NOT_CONVERGED if a Jacobi eigensolve reached
 * max_sweeps (outputs written from the last sweep). */
SAKI_API saki_status saki_key_spectrum(const saki_config* cfg, int64_t n_calib, const void* k_calib,
                                       float tau_int, float* eig, int32_t* spikes, void* workspace,
                                       size_t workspace_bytes, saki_stream stream);

/* saki_score_mse -- App. C's measured score-MSE reduction: per query head, over
 * every key_stride-th visible key of every query of the layout (key_stride >= 1;
 * 1 = all causal pairs), out[h] = { sum s^2, sum (s - s_hat)^2, pairs } in fp64
 * with s = q^T A_h k and s_hat = (L_h^T q)^T c + q^T nu_h (the index's score,
 * mean term included when nu is given).  The measured reduction is
 * 1 - out[h][1] / out[h][0], to compare with the predicted
 * 1 - sum_{i>r} sigma_i^2 / sum_i sigma_i^2 of saki_fit.
 *   Q [Hq][T][d], K [Hk][total_keys][d], sketch [Hq][total_keys][r] (dtype),
 *   A [Hq][d][d], L [Hq][d][r], nu [Hq][d] f32 or NULL, out [Hq][3] double.
 * Workspace: saki_workspace_size(SAKI_OP_SCORE_MSE) bytes, with the error-word
 * header of the selection calls.  SAKI_ERR_INVALID_ARGUMENT for key_stride < 1,
 * NULL out or workspace, NULL inputs when T > 0, a malformed layout or a
 * misaligned pointer; SAKI_ERR_WORKSPACE if too small.  Stream-ordered. */
SAKI_API saki_status saki_score_mse(const saki_config* cfg, const saki_layout* layout, int64_t key_stride,
                                    const void* Q, const float* A, const void* K, const float* L,
                                    const void* sketch, const float* nu, double* out, void* workspace,
                                    size_t workspace_bytes, saki_stream stream);

/* saki_merge_topk -- the exchange step of a selection split by key ranges
 * (several GPUs each holding a contiguous range of a long cache, Sec. 1's
 * 1M-token setting): the k best of the union of per-part top-k lists.
 *   idx_parts   [P][rows][k] int32  part-local key indices, -1 padding
 *   score_parts [P][rows][k] f32    their scores (the ranking key)
 *   part_offsets [P] HOST int64     first key of each part's range, in [0, 2^31)
 *   idx   [rows][k] int32           global indices (local + offset), -1 padding
 *   score [rows][k] f32 or NULL
 * Output lists are in descending score, equal scores by the lower global index,
 * which is the ranking saki_score_topk applies over the whole range, so merging
 * the parts' lists reproduces its result.  k = cfg->topk; P <= 64
 * (SAKI_ERR_UNSUPPORTED above).  Stream-ordered, no workspace. */
SAKI_API saki_status saki_merge_topk(const saki_config* cfg, int32_t num_parts, int64_t num_rows,
                                     const int32_t* idx_parts, const float* score_parts,
                                     const int64_t* part_offsets, int32_t* idx, float* score,
                                     saki_stream stream);

/* saki_workspace_status -- the device status of the last saki_score_topk,
 * saki_recall or saki_build_index call that used `workspace` (the first 256 bytes
 * of every workspace of these calls are a header holding the error word, which
 * each call clears as it starts).  Synchronises `stream`, the stream that call
 * ran on, then returns SAKI_OK, or SAKI_ERR_TIMEOUT if one of the call's kernels
 * gave up a bounded wait (its outputs are then incomplete).  A call that
 * launched nothing (no queries) leaves the header as it was.  saki_fit reports
 * its status itself and keeps no header. */
SAKI_API saki_status saki_workspace_status(const void* workspace, saki_stream stream);

/* Bytes of the static device scratch array behind saki_score_topk_noalloc. */
#define SAKI_NOALLOC_SCRATCH_BYTES (16u << 20)

/* saki_score_topk_noalloc -- the paper has no counterpart; this is a library
 * convenience.  Same arguments, semantics and results as saki_score_topk, minus
 * the workspace, for callers that cannot call cudaMalloc: for example a plugin
 * running inside a serving framework whose allocator owns all device memory, or
 * a decode loop that must not allocate because cudaMalloc can synchronise the
 * device.  Its scratch is a static device array of SAKI_NOALLOC_SCRATCH_BYTES
 * inside the library, held by every GPU that loads the library until the
 * process exits; nothing is allocated per call.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make that first call
 *     before any stream capture.
 *   - The call runs the fastest plan that fits the scratch: saki_workspace_size
 *     (SAKI_OP_SCORE_TOPK) reports the fastest plan, and a decode-shaped layout
 *     whose seeded plan (see saki_score_topk) exceeds SAKI_NOALLOC_SCRATCH_BYTES
 *     runs without the sample pass when that fits (same results).  Only a layout
 *     that even the plan without it does not fit is rejected, with
 *     SAKI_ERR_WORKSPACE, before any launch.
 *   - Its device status is read by saki_noalloc_status (or SAKI_FLAG_CHECK).
 *   - Every call shares the one array and it keeps the last call's contents;
 *     each call rewrites everything it later reads, so nothing needs clearing,
 *     but calls that overlap on the GPU (other streams, other host threads)
 *     race on it: serialise them. */
SAKI_API saki_status saki_score_topk_noalloc(const saki_config* cfg, const saki_layout* layout,
                                             const void* Q, const float* L, const void* sketch,
                                             const float* nu, int32_t* idx, float* score,
                                             saki_stream stream);

/* saki_noalloc_status -- saki_workspace_status for the static scratch of
 * saki_score_topk_noalloc on the current device (SAKI_OK before its first call);
 * no counterpart in the paper. */
SAKI_API saki_status saki_noalloc_status(saki_stream stream);

/* ---------------------------------------------------------------- profiling aids
 * Not part of the method (the paper has no counterpart): a launch count and
 * per-kernel device timing, for benchmarks that report kernel-level rooflines.
 *
 * saki_launch_count: number of kernels this library has launched in the process
 *   (every device and stream).
 * saki_kernel_timer_start(kind): arms one kernel kind.  While armed, every launch
 *   of that kind is bracketed by two CUDA timing events recorded on the stream of
 *   the library call that launches it (events of the device current at the first
 *   timed launch; launches on other devices are not timed).  Several kinds may be
 *   armed at once.  SAKI_ERR_INVALID_ARGUMENT for an unknown kind.
 * saki_kernel_timer_stop(kind, total_ms, launches): waits for the last recorded
 *   event, writes the summed device time (ms) and the number of timed launches,
 *   and disarms the kind.  SAKI_ERR_CUDA if an event query fails.
 * The timer state is process-wide and not synchronised with library calls made
 * concurrently from other threads; each timed launch costs two event records. */
#define SAKI_KERNEL_SELECT 1  /* selection kernel(s) of saki_score_topk */
#define SAKI_KERNEL_EXACT 2   /* exact top-k kernel(s) of saki_recall */
#define SAKI_KERNEL_FIT 3     /* SVD kernel of saki_fit (C', Jacobi, factors L and R) */
#define SAKI_KERNEL_MOMENTS 4 /* calibration-moment kernel(s) of saki_fit */
#define SAKI_KERNEL_BUILD 5   /* key-code kernel(s) of saki_build_index */
#define SAKI_KERNEL_FACTOR 6  /* moment-factor kernel of saki_fit */
SAKI_API int64_t saki_launch_count(void);
/* saki_debug_inject_stall(kind): a test hook for the failure reporting.  Arms a
 * one-shot stall for the next launch of a tensor-core kernel of that kind
 * (SAKI_KERNEL_SELECT, SAKI_KERNEL_EXACT or SAKI_KERNEL_BUILD; 0 disarms): its
 * TMA producer issues no loads, so the other roles' bounded waits run out
 * (about two seconds), the kernel stops without faulting and the call's error
 * word reports SAKI_ERR_TIMEOUT.  A launch of another path (CUDA-core kernels,
 * which do not wait) leaves the stall armed.  SAKI_ERR_INVALID_ARGUMENT for
 * other kinds. */
SAKI_API saki_status saki_debug_inject_stall(int32_t kind);
SAKI_API saki_status saki_kernel_timer_start(int32_t kind);
SAKI_API saki_status saki_kernel_timer_stop(int32_t kind, double* total_ms, int64_t* launches);

/* Static description of a status code (never NULL; "unknown status" for
 * values outside saki_status). */
SAKI_API const char* saki_status_string(saki_status status);

/* Library version as "major.minor.patch". */
SAKI_API const char* saki_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SAKI_H_ */
