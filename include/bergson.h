/*
 * bergson.h -- C ABI of the GB300 projected-gradient attribution library.
 *
 * The library implements the TrackStar-style gradient path of Bergson
 * (Sec. 3.1 "Attribution Pipelines", Fig. 1, App. B, "Gradients"):
 *   per-example gradients of every nn.Linear weight, optional Adafactor-style
 *   factored second-moment normalisation, the double-sided per-module random
 *   projection, unit normalisation into an fp16 gradient store, and exact
 *   cosine top-k queries against that store.
 *
 * Conventions shared by every entry point
 *   - All tensor pointers are DEVICE pointers owned by the caller; the library
 *     never allocates.  Scratch memory comes in through `workspace`, sized by
 *     the matching *_workspace query.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Every call only enqueues work on it; nothing synchronises.
 *   - Arguments are validated on the host before anything is enqueued.  A
 *     failing call returns a negative bergson_status, enqueues nothing and
 *     leaves a message in bergson_last_error().  No call aborts the process.
 *   - Device-side waits are bounded.  A wait that gives up records
 *     BERGSON_EDEVICE_TIMEOUT in a device status word that
 *     bergson_sync_status() reports.
 *   - The device that executes the work is the one that owns `workspace` (or
 *     the output buffer for calls without workspace).
 */
#ifndef BERGSON_H
#define BERGSON_H

#include <stddef.h>
#include <stdint.h>

#if defined(BERGSON_BUILD) && defined(__GNUC__)
#define BERGSON_API __attribute__((visibility("default")))
#else
#define BERGSON_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  BERGSON_OK = 0,
  BERGSON_EINVAL = -1,            /* bad size, null pointer or inconsistent arguments */
  BERGSON_EALIGN = -2,            /* a pointer or leading dimension breaks an alignment rule */
  BERGSON_EUNSUPPORTED = -3,      /* valid request outside what this build implements */
  BERGSON_EWORKSPACE = -4,        /* workspace smaller than the *_workspace query */
  BERGSON_ECUDA = -5,             /* a CUDA runtime/driver call failed */
  BERGSON_EDEVICE_TIMEOUT = -6,   /* a bounded device wait gave up (see bergson_sync_status) */
  BERGSON_EMOMENT = -7            /* a second-moment entry r_i or c_j was not > 0 (recorded by
                                     the device; see bergson_sync_status) */
} bergson_status;

typedef enum {
  BERGSON_AGG_SUM = 0,
  BERGSON_AGG_MEAN = 1
} bergson_aggregation;

typedef enum {
  BERGSON_FISHER_INV_SQRT = 0,    /* M = R^-1/2 (whitening, TrackStar) */
  BERGSON_FISHER_INV = 1          /* M = R^-1 */
} bergson_fisher_power;

typedef enum {
  BERGSON_LAYER_BIAS = 1          /* also write the layer's projected bias gradient */
} bergson_layer_flags;

/*
 * Distribution of the projection entries.  Every kind has mean 0 and variance
 * 1/k per entry (Johnson-Lindenstrauss scaling); entry (i, j) of P [d, k]
 * takes counter e = i*k + j of its seed's stream.  App. B ("Gradients") names
 * Rademacher and uniform projection matrices; Gaussian is the default here.
 */
typedef enum {
  BERGSON_PROJ_GAUSSIAN = 0,      /* z_e / sqrt(k), z_e the Box-Muller normal draw */
  BERGSON_PROJ_IDENTITY = 1,      /* P = I, requires k == d (testing aid) */
  BERGSON_PROJ_RADEMACHER = 2,    /* +-1 / sqrt(k): sign = top bit of h_e = mix(seed ^ mix(e)) */
  BERGSON_PROJ_UNIFORM = 3        /* sqrt(3) x_e / sqrt(k), x_e = (2v + 1 - 2^24) 2^-24 uniform
                                     on (-1, 1), v = top 24 bits of h_e */
} bergson_proj_kind;

/*
 * One nn.Linear module's captured tensors (Bergson App. B, "Gradients": gradient
 * collection from linear layers; Fig. 1: Adafactor normalisation and the
 * double-sided per-module projection).
 *
 *   A      bf16 [B, T, d_in] layer inputs, contiguous, 16-byte aligned.
 *   G      bf16 [B, T, d_out] gradients w.r.t. the layer output, contiguous,
 *          16-byte aligned.
 *   d_in, d_out   multiples of 8, >= 8.
 *   k_in, k_out   projection sizes, each one of 16, 32, 64.
 *   seed_in, seed_out   seeds of P_in [d_in, k_in] and P_out [d_out, k_out].
 *          Entry (i, j) of P is z(seed, i*k + j) / sqrt(k), z the counter-based
 *          SplitMix64 + Box-Muller normal draw, rounded to fp32 (Gaussian kind;
 *          see bergson_proj_kind for the others).
 *   proj_kind    bergson_proj_kind, shared by both sides of the layer.
 *   r, c   fp32 [d_out] and [d_in] factored second moments (> 0), or both
 *          NULL for no normalisation.  The gradient is divided elementwise by
 *          sqrt(r_i c_j).  The values live on the device, so the host cannot
 *          check them: an entry that is not > 0 (zero, negative, NaN) is
 *          recorded as BERGSON_EMOMENT in the device status word (reported by
 *          bergson_sync_status) and the outputs that depend on it are inf/NaN.
 *   out_col_offset   first column of this module's k_out*k_in block in `out`.
 *   flags  0 or BERGSON_LAYER_BIAS.  With BERGSON_LAYER_BIAS the projected
 *          bias gradient P_out^T (sum over valid tokens of g_t / sqrt(r)) --
 *          App. B, gradients of linear "weight and bias" -- is written as
 *          k_out values at bias_col_offset (bergson_project_grads only; the
 *          per-token scores cover the weight blocks).
 */
typedef struct bergson_layer {
  const void* A;
  const void* G;
  int64_t d_in;
  int64_t d_out;
  int64_t k_in;
  int64_t k_out;
  uint64_t seed_in;
  uint64_t seed_out;
  int32_t proj_kind;
  int32_t flags;                  /* bergson_layer_flags */
  const float* r;
  const float* c;
  int64_t out_col_offset;
  int64_t bias_col_offset;        /* used with BERGSON_LAYER_BIAS */
} bergson_layer;

/* Bytes of workspace bergson_project_grads needs for these arguments. */
BERGSON_API int bergson_project_grads_workspace(const bergson_layer* layers, int n_layers,
                                    int64_t B, int64_t T, size_t* ws_bytes);

/*
 * Projected per-example gradients (Bergson Sec. 3.1 "processing ... down-
 * projection"; Fig. 1 double-sided per-module random projection):
 *
 *   out[b, off + i*k_in + j] = ( P_out^T (W_b / sqrt(r c^T)) P_in )[i, j],
 *   W_b = sum over valid tokens t of g_{b,t} a_{b,t}^T,
 *
 * computed without forming W_b, through the token-level projections
 * (A diag(c^-1/2) P_in, G diag(r^-1/2) P_out) and a masked per-example
 * contraction over tokens.  The result is NOT unit-normalised.
 *
 *   mask    u8 [B, T] (nonzero = valid token) or NULL (all valid).  A masked
 *           token contributes nothing, whatever A and G hold there.
 *   out     fp32 [B, ld_out]; only the layers' column blocks are written.
 *           Blocks must lie inside [0, ld_out) and must not overlap.
 *   B, T    >= 0.  T == 0 writes zero blocks.
 *   workspace/ws_bytes   device scratch of at least the queried size,
 *           256-byte aligned; contents on entry are ignored.
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_project_grads(const bergson_layer* layers, int n_layers, int64_t B, int64_t T,
                          const uint8_t* mask, float* out, int64_t ld_out,
                          void* workspace, size_t ws_bytes, void* stream);

/*
 * Gradient-store rows (Bergson Sec. 3.1 on-disk gradient store with unit
 * normalisation; Fig. 1 "unit normalization"):
 *
 *   store[row_offset + b, 0:K] = fp16( proj[b, 0:K] / ||proj[b, 0:K]||_2 )
 *
 * (or fp16(proj) when unit_normalize == 0).  A zero row is stored as zeros.
 *   proj      fp32 [B, ld_proj], 16-byte aligned, ld_proj % 4 == 0, ld_proj >= K.
 *   K         > 0, K % 8 == 0.
 *   store     fp16 [N_cap, ld_store], 16-byte aligned, ld_store % 8 == 0,
 *             ld_store >= K.  Rows outside [row_offset, row_offset + B) are
 *             untouched (stores are built by appending batches).
 *   norms_out optional fp32 [B]: the l2 norms before normalisation.
 * Errors: EINVAL, EALIGN, ECUDA.
 */
BERGSON_API int bergson_build_store(const float* proj, int64_t B, int64_t K, int64_t ld_proj,
                        int unit_normalize, void* store, int64_t ld_store,
                        int64_t row_offset, int64_t N_cap, float* norms_out, void* stream);

/*
 * Gradient-store rows with per-module unit normalisation (Sec. 3.1: the
 * store is indexed by module; Fig. 1 "unit normalization"), the option beside
 * the whole-row normalisation of bergson_build_store:
 *
 *   store[row_offset + b, o_j:o_{j+1}] = fp16( proj[b, o_j:o_{j+1}] / ||proj[b, o_j:o_{j+1}]||_2 )
 *
 * for every block j (typically one module's k_out*k_in block); a zero block
 * is stored as zeros.  Each stored block then has unit norm, so a row has
 * norm sqrt(n_blocks) and bergson_score_topk's score of a unit query q is
 * sum_j q[o_j:o_{j+1}] . s_j, every module weighted alike.
 *   block_offsets  HOST int64 [n_blocks + 1]: 0 = o_0 < o_1 < ... < o_n = K,
 *                  each a multiple of 8.   n_blocks in 1 .. 2048.
 *   norms_out      optional fp32 [B, n_blocks]: the blocks' l2 norms before
 *                  normalisation.
 * Other arguments and rules as for bergson_build_store; with n_blocks = 1 the
 * result equals bergson_build_store with unit_normalize = 1.
 * Errors: EINVAL, EALIGN, ECUDA.
 */
BERGSON_API int bergson_build_store_blocks(const float* proj, int64_t B, int64_t K,
                                           int64_t ld_proj, const int64_t* block_offsets,
                                           int n_blocks, void* store, int64_t ld_store,
                                           int64_t row_offset, int64_t N_cap, float* norms_out,
                                           void* stream);

/* Bytes of workspace bergson_score_topk (and bergson_score_bottomk) needs;
 * N, K, Q and topk follow the calls' size rules (EINVAL, EALIGN, EUNSUPPORTED). */
BERGSON_API int bergson_score_topk_workspace(int64_t N, int64_t K, int64_t Q, int64_t topk, size_t* ws_bytes);

/*
 * Exact cosine top-k of queries against the store (Bergson Sec. 3.1: exact
 * top-k nearest-neighbour lookup over the gradient store; grad-cosine):
 *
 *   S[q, n] = (query_q / ||query_q||) . store_n
 *   out_scores[q, :], out_idx[q, :] = the topk largest S[q, n], ordered by
 *   score descending, then index ascending.
 *
 * Store rows are taken as stored (unit norm when built by bergson_build_store).
 * The N x Q score matrix is never materialised.
 *   store     fp16 [N, ld_store], 16-byte aligned, ld_store % 8 == 0, ld_store >= K.
 *   N         1 .. 2^31-1.   K > 0, K % 8 == 0.
 *   queries   fp32 [Q, ld_q], ld_q >= K, 4-byte aligned; normalised inside
 *             (a zero query scores 0 against every row).
 *   Q         >= 0.   topk in 1 .. min(N, 1024).
 *   out_scores fp32 [Q, topk]; out_idx int64 [Q, topk].
 * NaN scores never enter the result; if fewer than topk scores are usable
 * the tail holds score -inf and index -1.
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_score_topk(const void* store, int64_t N, int64_t K, int64_t ld_store,
                       const float* queries, int64_t Q, int64_t ld_q, int64_t topk,
                       float* out_scores, int64_t* out_idx,
                       void* workspace, size_t ws_bytes, void* stream);

/*
 * The k least influential store rows of each query (Bergson Sec. 3.1: the
 * query tool returns the k most and least influential training items):
 *
 *   out_scores[q, :], out_idx[q, :] = the bottomk smallest S[q, n], ordered by
 *   score ascending, then index ascending.
 *
 * S, the arguments, the limits (bottomk in 1 .. min(N, 1024)) and the errors
 * are those of bergson_score_topk, and so is the workspace
 * (bergson_score_topk_workspace with topk = bottomk).  The search runs on the
 * negated unit query; the scores it returns are exactly the negations of the
 * scores against -q, i.e. the cosines against q.  If fewer than bottomk scores
 * are usable the tail holds score +inf and index -1.
 */
BERGSON_API int bergson_score_bottomk(const void* store, int64_t N, int64_t K, int64_t ld_store,
                          const float* queries, int64_t Q, int64_t ld_q, int64_t bottomk,
                          float* out_scores, int64_t* out_idx,
                          void* workspace, size_t ws_bytes, void* stream);

/*
 * Exact top-k (bottom-k) over a store scored piece by piece (Bergson Sec. 3.1:
 * gradient stores persisted to disk and queried with exact top-k; a store can
 * be far larger than device memory).  One call scores the rows of one chunk,
 *   store[0, N) = rows [row_base, row_base + N) of the whole store,
 * and merges them into a running result held by the caller:
 *   init != 0:  scores/idx <- the top-k of this chunk (contents on entry ignored);
 *   init == 0:  scores/idx <- the top-k of (scores/idx on entry  U  this chunk).
 * Indices are global (row_base + row).  After calls over chunks that cover
 * rows [0, N_total) once each, in any order, scores/idx equal
 * bergson_score_topk over the whole store: the same rows, the same scores
 * bit for bit (every score is computed the same way whatever chunk holds
 * its row), the same order (score descending, index ascending; bottom-k:
 * ascending, index ascending).  With init == 0 the chunk's pass starts from
 * the running k-th score, so chunks after the first cost little beyond
 * streaming them.
 *   N          1 .. 2^31-1 rows in this chunk (may be fewer than topk).
 *   row_base   >= 0, row_base + N < 2^31.  Chunks must not overlap.
 *   scores, idx  fp32 / int64 [Q, topk], in and out; tail entries of a
 *              result with fewer than topk rows are (-inf, -1) for top-k and
 *              (+inf, -1) for bottom-k.
 * Other arguments and rules as for bergson_score_topk / _bottomk; workspace
 * from bergson_score_topk_update_workspace (it does not depend on N).
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_score_topk_update_workspace(int64_t K, int64_t Q, int64_t topk,
                                                    size_t* ws_bytes);
BERGSON_API int bergson_score_topk_update(const void* store, int64_t N, int64_t K,
                                          int64_t ld_store, int64_t row_base,
                                          const float* queries, int64_t Q, int64_t ld_q,
                                          int64_t topk, int init, float* scores, int64_t* idx,
                                          void* workspace, size_t ws_bytes, void* stream);
BERGSON_API int bergson_score_bottomk_update(const void* store, int64_t N, int64_t K,
                                             int64_t ld_store, int64_t row_base,
                                             const float* queries, int64_t Q, int64_t ld_q,
                                             int64_t bottomk, int init, float* scores,
                                             int64_t* idx, void* workspace, size_t ws_bytes,
                                             void* stream);

/*
 * Exact top-k (least == 0) or bottom-k (least != 0) of a store that lives in
 * HOST memory (Sec. 3.1: on-disk, memory-mapped gradient stores), streamed
 * to the device in chunks of chunk_rows rows: chunk c + 1 is copied on
 * `copy_stream` while chunk c is scored on `stream` (two device chunk
 * buffers in the workspace), each chunk merged into the running result as
 * bergson_score_topk_update does.  The result equals bergson_score_topk over
 * the same rows resident on the device.
 *   host_store  fp16 [N, ld_store] host memory, 16-byte aligned rows.  Pinned
 *               (page-locked) memory lets the copies overlap the scoring and
 *               run at the host link's rate; other host memory (e.g. a
 *               numpy.memmap of a store file) works, with copies staged by
 *               the driver.
 *   copy_stream a second stream for the copies, or NULL to copy on `stream`
 *               (no overlap).  The call orders the two streams with events it
 *               creates and destroys itself; on return all its work is
 *               enqueued on `stream` (and copy_stream), nothing is synchronised.
 *   workspace   bergson_score_topk_host_workspace(chunk_rows, K, Q, topk) bytes.
 * N, K, Q, topk, queries and outputs as for bergson_score_topk.
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_score_topk_host_workspace(int64_t chunk_rows, int64_t K, int64_t Q,
                                                  int64_t topk, size_t* ws_bytes);
BERGSON_API int bergson_score_topk_host(const void* host_store, int64_t N, int64_t K,
                                        int64_t ld_store, const float* queries, int64_t Q,
                                        int64_t ld_q, int64_t topk, int least,
                                        int64_t chunk_rows, float* out_scores, int64_t* out_idx,
                                        void* workspace, size_t ws_bytes, void* stream,
                                        void* copy_stream);

/* Bytes of workspace bergson_token_scores needs (n_queries in 1 .. 256). */
BERGSON_API int bergson_token_scores_workspace(const bergson_layer* layers, int n_layers,
                                               int64_t B, int64_t T, int64_t n_queries,
                                               size_t* ws_bytes);

/*
 * Per-token attribution scores (Bergson Fig. 1: attribution scores per token
 * or per sequence; Sec. 3.1 per-token gradient collection):
 *
 *   out[q, b, t] = sum over layers m of  g~_{b,t,m}^T  Q~_{q,m}  a~_{b,t,m}
 *
 * i.e. the Frobenius inner product of token t's own projected (and
 * normalised) gradient P_out'^T g_t a_t^T P_in' with query q's k_out x k_in
 * block Q~_{q,m} = queries[q, off_m : off_m + k_out*k_in] (row-major, the
 * layout bergson_project_grads writes).  Summed over t, the scores give the
 * per-sequence inner product <out_b, queries_q>.  Masked tokens score 0.
 *   queries  fp32 [n_queries, ld_q], 4-byte aligned; the layers' column
 *            blocks must fit in ld_q and must not overlap.
 *   n_queries  1 .. 256.  One pass over A and G serves them all: a module's
 *            query blocks go through shared memory in groups (up to 16
 *            queries; fewer for larger k_in x k_out) for every token tile, and
 *            the inner products a~^T Q~_q^T run on the tensor cores
 *            (3xTF32, fp32 accuracy) except for (k_in, k_out) = (64, 32) and
 *            (64, 64), which stay on the CUDA cores.
 *   out      fp32 [n_queries, B, T] contiguous.
 * The workspace holds per-module partial scores (n_layers x n_queries x B x
 * T floats) that a final pass sums in module order.
 * Other arguments as for bergson_project_grads.  Deterministic.
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_token_scores(const bergson_layer* layers, int n_layers, int64_t B,
                                     int64_t T, const uint8_t* mask, const float* queries,
                                     int64_t n_queries, int64_t ld_q, float* out,
                                     void* workspace, size_t ws_bytes, void* stream);

/* Bytes of workspace bergson_aggregate_rows needs for n rows. */
BERGSON_API int bergson_aggregate_rows_workspace(int64_t n, size_t* ws_bytes);

/*
 * Query aggregation (Bergson Sec. 3.2: queries formed as the mean or sum of
 * the gradients of several generations or dataset items, as LESS builds its
 * evaluation queries; Fig. 2 "unit_normalize: true, aggregation: mean"):
 *
 *   out[g, 0:K] = agg over r in [offsets[g], offsets[g+1]) of  w_r * rows[r, 0:K]
 *
 * with w_r = 1/||rows[r, 0:K]|| when normalize_each (0 for a zero row) else 1,
 * and agg = sum (BERGSON_AGG_SUM) or mean (BERGSON_AGG_MEAN).  An empty group
 * gives a zero row.  Rows are added in order (deterministic).
 *   rows     fp32 [n, ld], out fp32 [G, ld_out]: 16-byte aligned, ld % 4 == 0.
 *   K        multiple of 4.
 *   offsets  DEVICE int64 [G + 1], non-decreasing within [0, n] (entries
 *            outside are clamped; a decreasing pair is an empty group).
 *   workspace  needed only when normalize_each (size from the query above).
 * Errors: EINVAL, EALIGN, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_aggregate_rows(const float* rows, int64_t n, int64_t K, int64_t ld,
                                       const int64_t* offsets, int64_t G, int mode,
                                       int normalize_each, float* out, int64_t ld_out,
                                       void* workspace, size_t ws_bytes, void* stream);

/*
 * TrackStar's empirical-Fisher preconditioner (Bergson Sec. 3.1: the
 * empirical Fisher information matrix of TrackStar, stacked with optimizer
 * normalisation and down-projection; Fig. 2: Fisher fitting and mixing).
 * Three steps, all on the device, fp32:
 *
 *   bergson_fisher_fit:             R = (1/n) sum_i x_i x_i^T  over n rows x_i = rows[i, 0:K]
 *   bergson_fisher_preconditioner:  R = lam R1 + (1 - lam) R2 (R2 = NULL: R = R1),
 *                                   R += damping * (tr(R) / K) * I,
 *                                   M = R^-1/2 (BERGSON_FISHER_INV_SQRT) or R^-1,
 *                                   by `iterations` coupled Newton-Schulz steps
 *                                   (20-30 reach fp32 accuracy for condition
 *                                   numbers up to ~1e4-1e6; damping bounds it)
 *   bergson_precondition_rows:      out[b] = M rows[b]   (M symmetric)
 *
 * Preconditioned rows then go through bergson_build_store / bergson_score_topk
 * (or bergson_score_grads) as usual.  All matrices are fp32 row-major with
 * 16-byte aligned rows (leading dimensions multiples of 4); K % 4 == 0,
 * K <= 65536.  Workspaces: bergson_fisher_fit_workspace(n, K),
 * bergson_fisher_preconditioner_workspace(K) (4 K^2 floats) and, for
 * precondition_rows, bergson_score_grads_workspace(B, K, K).
 * Errors: EINVAL, EALIGN, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_fisher_fit_workspace(int64_t n, int64_t K, size_t* ws_bytes);
BERGSON_API int bergson_fisher_fit(const float* rows, int64_t n, int64_t K, int64_t ld, float* R,
                                   int64_t ldr, void* workspace, size_t ws_bytes, void* stream);
BERGSON_API int bergson_fisher_preconditioner_workspace(int64_t K, size_t* ws_bytes);
BERGSON_API int bergson_fisher_preconditioner(const float* R1, const float* R2, int64_t K,
                                              int64_t ldr, float lam, float damping, int power,
                                              int iterations, float* M, int64_t ldm,
                                              void* workspace, size_t ws_bytes, void* stream);
/*
 * bergson_fisher_preconditioner with a stopping rule (same reading of Sec. 3.1
 * and Fig. 2).  Before each Newton-Schulz update the residual of the current
 * iterate,
 *
 *   res_i = ||I - Z_i Y_i||_F / sqrt(K)     (= ||M_i R M_i - I||_F / sqrt(K)
 *                                            while the iteration keeps Y = R Z / c),
 *
 * is read back to the host; the iteration stops at the first i with
 * res_i <= tol, or after max_iterations updates.  M is formed from that iterate.
 *   residuals   host fp32 [max_iterations + 1] or NULL: res_0, res_1, ... up to
 *               the last iterate computed.
 *   iterations  host int or NULL: the number of updates applied.
 * Unlike the other calls this one synchronises `stream` once per iterate
 * (one 4-byte read each; the call is a one-time setup cost).  tol = 0 runs
 * all max_iterations updates and still records every residual.
 * Errors: those of bergson_fisher_preconditioner, and EINVAL for tol < 0.
 */
BERGSON_API int bergson_fisher_preconditioner_tol(const float* R1, const float* R2, int64_t K,
                                                  int64_t ldr, float lam, float damping,
                                                  int power, int max_iterations, float tol,
                                                  float* M, int64_t ldm, void* workspace,
                                                  size_t ws_bytes, float* residuals,
                                                  int* iterations, void* stream);
BERGSON_API int bergson_precondition_rows(const float* rows, int64_t B, int64_t K, int64_t ld,
                                          const float* M, int64_t ldm, float* out,
                                          int64_t ld_out, void* workspace, size_t ws_bytes,
                                          void* stream);

/* Bytes of workspace bergson_score_grads needs. */
BERGSON_API int bergson_score_grads_workspace(int64_t B, int64_t K, int64_t Q, size_t* ws_bytes);

/*
 * On-the-fly attribution scores (Bergson Sec. 3.1, "bergson score": training
 * gradients are streamed and only their influence on fixed queries is kept,
 * with no gradient store; Table 3 grad-cosine / grad-dot):
 *
 *   scores[b, q] = <x_b, y_q> / (||x_b|| ||y_q||)   (unit_normalize != 0)
 *   scores[b, q] = <x_b, y_q>                        (unit_normalize == 0)
 *
 * with x_b = proj[b, 0:K] (e.g. bergson_project_grads output) and
 * y_q = queries[q, 0:K] (projected query gradients).  fp32 throughout; a zero
 * row or query scores 0 under normalisation.  Deterministic.
 *   proj      fp32 [B, ld_proj], queries fp32 [Q, ld_q]: 16-byte aligned,
 *             ld % 4 == 0, ld >= K.   K > 0, K % 4 == 0.
 *   scores    fp32 [B, ld_scores], ld_scores >= Q.
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, EWORKSPACE, ECUDA.
 */
BERGSON_API int bergson_score_grads(const float* proj, int64_t B, int64_t K, int64_t ld_proj,
                                    const float* queries, int64_t Q, int64_t ld_q,
                                    int unit_normalize, float* scores, int64_t ld_scores,
                                    void* workspace, size_t ws_bytes, void* stream);

/*
 * The projection actually used by bergson_project_grads (Fig. 1 random
 * projection), materialised for inspection:
 *   out[i, j] = scale_i * P[i, j]   (fp32 [d, k], row-major)
 * with P as described for bergson_layer and scale_i = 1/sqrt(moment_i), or 1
 * when `moment` is NULL.  k in 16, 32, 64; identity needs k == d.
 * Errors: EINVAL, EALIGN, EUNSUPPORTED, ECUDA.
 */
BERGSON_API int bergson_projection_matrix(uint64_t seed, int64_t d, int64_t k, int proj_kind,
                              const float* moment, float* out, void* stream);

/*
 * Synchronises `stream`, then reports and clears the device status word:
 * BERGSON_OK, BERGSON_EDEVICE_TIMEOUT (a bounded device wait gave up),
 * BERGSON_EMOMENT (a factored second-moment entry was not > 0) or
 * BERGSON_ECUDA (the stream carried a CUDA error).  The word keeps the first
 * status recorded since it was last cleared.
 */
BERGSON_API int bergson_sync_status(void* stream);

/* Message of the last failing call on this thread ("" if none). */
BERGSON_API const char* bergson_last_error(void);

/*
 * Per-module projection seeds derived from one base seed, so that a model's
 * modules get independent projections (reading of Fig. 1: every module has
 * its own pair of random matrices):
 *   seed_in = mix(base ^ 2m),  seed_out = mix(base ^ (2m + 1)),
 * mix = the SplitMix64 finaliser, m = module index.  Pure host function.
 */
BERGSON_API void bergson_module_seeds(uint64_t base_seed, int64_t module_index, uint64_t* seed_in,
                          uint64_t* seed_out);

/* Library version, major*10000 + minor*100 + patch. */
BERGSON_API int bergson_version(void);

/*
 * Test aid for the bounded-wait machinery: enqueues one kernel that waits on a
 * barrier nothing will ever complete, for at most `timeout_ns`, then records
 * BERGSON_EDEVICE_TIMEOUT in the device status word and returns.  The context
 * stays usable.  timeout_ns in 1 .. 10^10.
 */
BERGSON_API int bergson_debug_wait_probe(uint64_t timeout_ns, void* stream);

/*
 * Test aid for host error paths: the next `count` calls of any entry point
 * that would enqueue work return `status` (e.g. BERGSON_ECUDA) after argument
 * validation, without enqueueing anything.  count = 0 clears it.
 */
BERGSON_API void bergson_debug_inject_status(int status, int count);

/*
 * Test aid for the per-device record behind every kernel-attribute setting
 * (one process may drive several GPUs; CUDA keeps a kernel's shared-memory
 * limit per function and per device).  Runs n_threads host threads that each
 * ask, three times over, for the setting on each of n_devices simulated
 * devices, with a slow fake setting in place of the CUDA call; the first
 * fake setting for fail_device (-1: none) fails.  set_calls[d] receives how
 * often the setting ran for device d (1 expected, 2 for fail_device: a
 * failure is retried) and *failures how many requests saw a failure.
 * Host only: no GPU is touched.  n_threads, n_devices in 1 .. 64.
 */
BERGSON_API int bergson_debug_attr_once(int n_threads, int n_devices, int fail_device,
                                        int64_t* set_calls, int* failures);

/*
 * Test aid for the projection work planner: for the same arguments as
 * bergson_project_grads_workspace, reports the (module, example, tile range)
 * partial slots of all launches (*n_slots), the work items the launches hand
 * out (*n_items), how many of those items are pieces (*n_pieces; a piece
 * projects one side of a slot over a range of 64-column chunks, and the
 * slot's last piece contracts them) and how many layers share their input
 * tensor A with another layer of the same (k_in, k_out) (*n_shared; their
 * items are scheduled side by side).
 * Host only: enqueues nothing.  Returns the validation status; NULL outputs
 * are skipped.
 */
BERGSON_API int bergson_debug_project_plan(const bergson_layer* layers, int n_layers, int64_t B,
                                           int64_t T, int64_t* n_slots, int64_t* n_items,
                                           int64_t* n_pieces, int64_t* n_shared);

/*
 * Test aid for the scorer's launch planner (bergson_score_topk and
 * bergson_score_bottomk): the launches it would make for a store of N rows,
 * Q queries and topk, on a device with `ctas` resident CTAs of the score
 * kernel (the SM count, or for more than 128 queries twice the number of
 * co-resident two-CTA clusters).  *n_launches receives the number of score
 * launches (each followed by a merge); the first min(max_launches,
 * *n_launches) are written to out as rows of 12 int64:
 *   pass, stage (0 = prefix threshold pass, 1 = full pass), store rows,
 *   query groups, first query group, CTAs per group, grid, store tiles,
 *   first query, end query (of the merge), pair (1 = clusters of two CTAs),
 *   128-query tiles per CTA.
 * Host only: enqueues nothing.  Errors: EINVAL.
 */
BERGSON_API int bergson_debug_score_plan(int64_t N, int64_t K, int64_t Q, int64_t topk, int ctas,
                                         int64_t* out, int max_launches, int* n_launches);

/*
 * Test aid for the planner of the skinny tcgen05 product behind
 * bergson_score_grads, bergson_precondition_rows and the Fisher products
 * (C[b, q] = <x_b, y_q> for B rows x, Q rows y of length K).  Writes 19 int64
 * to out (n_out >= 19): batch rows per tile, batch tiles, y tiles, 32-column
 * steps, K slices, pipeline stages, column chunks of the row split, CTA pairs
 * (1/0: batches of up to 64 rows), accumulator buffers, rows of y per tile
 * (256 on pairs, else 128), TMEM columns allocated, the workspace offsets of
 * the x norms, y norms, partial products, x_hi, x_lo and the total, then the
 * TMEM column of the pairs' y operand ring and its 64-column slots (0
 * otherwise).
 * Host only: enqueues nothing.  Errors: EINVAL (B in [1, 2^20], Q in
 * [1, 2^24], K in [4, 2^26] and a multiple of 4).
 */
BERGSON_API int bergson_debug_xgemm_plan(int64_t B, int64_t Q, int64_t K, int64_t* out, int n_out);

/*
 * On-disk gradient store (Bergson Sec. 3.1: gradient stores persisted to disk,
 * read back as memory maps).  The file is N rows of K fp16 values, row-major,
 * with no header (numpy.memmap(path, dtype=float16, shape=(N, K)) opens it).
 *   bergson_store_save: rows [0, rows) of the device store -> file rows
 *     [file_row_offset, file_row_offset + rows); creates or extends the file.
 *   bergson_store_load: file rows [file_row_offset, +rows) -> device store rows [0, rows).
 * Both synchronise `stream` first and return when the data has moved (host
 * I/O through a bounce buffer; not a hot-path call).
 * Errors: EINVAL (bad arguments, I/O failure, file too short), ECUDA.
 */
BERGSON_API int bergson_store_save(const void* store, int64_t rows, int64_t K, int64_t ld_store,
                                   const char* path, int64_t file_row_offset, void* stream);
BERGSON_API int bergson_store_load(const char* path, int64_t file_row_offset, int64_t rows,
                                   int64_t K, void* store, int64_t ld_store, void* stream);

/*
 * Allocation-free variant of bergson_project_grads.  The paper has no
 * counterpart: this exists for callers that cannot supply a workspace, such as
 * plugin or callback interfaces that hand over only input and output buffers,
 * runtimes that own all device memory through their own pool, or loops that
 * must not call cudaMalloc (it can synchronise the device and can fail when
 * memory is short).
 *
 * Same arguments and result as bergson_project_grads, minus the workspace.
 * The scratch is a fixed static device array of BERGSON_NOALLOC_SCRATCH_BYTES
 * that every GPU loading the library keeps until the process exits; requests
 * needing more (see bergson_project_grads_workspace) fail with
 * BERGSON_EWORKSPACE and enqueue nothing.  The call itself allocates nothing
 * (no cudaMalloc, no workspace, no allocating library routine).
 * All calls share the one array: calls that overlap on the GPU (e.g. on two
 * streams) race and must be ordered by the caller.
 *
 * First call on a device: it looks up the array's device address on the
 * device that owns `out` (the current device when out is NULL).  Under CUDA's
 * lazy module loading (the default) that lookup is also the moment the driver
 * loads this part of the library on the device and reserves the array's
 * 32 MiB there, so the first call can fail with BERGSON_ECUDA when the device
 * has no 32 MiB left (e.g. a runtime's pool already holds it all).  To take
 * that step at a time of the caller's choosing, make a warm-up call early:
 * any valid layer array with B = 0 and out = NULL does the lookup (and the
 * reservation) on the current device and enqueues nothing.  Make the first
 * call on each device before any stream capture begins.
 */
#define BERGSON_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

BERGSON_API int bergson_project_grads_noalloc(const bergson_layer* layers, int n_layers,
                                              int64_t B, int64_t T, const uint8_t* mask,
                                              float* out, int64_t ld_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* BERGSON_H */
