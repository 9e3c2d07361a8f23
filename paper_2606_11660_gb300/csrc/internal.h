// Structures shared between the host API (api.cu) and the kernel translation
// units, and the launchers each kernel unit exports to the host API.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

namespace bergson {

// A per-device "done once" record for settings that CUDA keeps per function
// and per device (the dynamic shared-memory limit of a kernel): ensure(dev,
// set) runs set() the first time it is asked for device `dev` and remembers
// success, so that one process can drive several GPUs and two host threads
// making their first calls at the same time neither skip nor repeat it.  A
// failed set() is not remembered (the next call tries again).  Devices past
// the first 64 are not cached: set() runs on every call.
class PerDeviceOnce {
 public:
  template <typename Set>
  cudaError_t ensure(int dev, Set&& set) {
    const bool cached = dev >= 0 && dev < 64;
    const uint64_t bit = cached ? (uint64_t{1} << dev) : 0;
    if (cached && (done_.load(std::memory_order_acquire) & bit) != 0) return cudaSuccess;
    std::lock_guard<std::mutex> lk(mu_);
    if (cached && (done_.load(std::memory_order_relaxed) & bit) != 0) return cudaSuccess;
    const cudaError_t e = set();
    if (e == cudaSuccess && cached) done_.fetch_or(bit, std::memory_order_release);
    return e;
  }

 private:
  std::atomic<uint64_t> done_{0};
  std::mutex mu_;
};

// Sets `kernel`'s dynamic shared-memory limit to `bytes` on the current
// device, once per device (see PerDeviceOnce).
template <typename Kernel>
cudaError_t smem_attr_once(PerDeviceOnce& once, Kernel kernel, int bytes) {
  int dev = -1;
  const cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  return once.ensure(dev, [&] {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  });
}

// Launches `kernel` with programmatic stream serialization: it may be
// scheduled before its predecessor in the stream has finished, and must call
// griddep_wait() before it touches anything that predecessor writes.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block,
                                    size_t smem, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

constexpr int kTileTokens = 128;     // tokens per MMA tile (tcgen05 M)
constexpr int kChunk = 64;           // bf16 elements per 128-byte swizzled row
constexpr int kScoreBN = 256;        // store rows per score tile (tcgen05 N)
constexpr int kScoreQT = 128;        // queries per query tile (tcgen05 M)
constexpr int kMaxTopk = 1024;
constexpr uint64_t kWaitTimeoutNs = 4000000000ull;   // bounded device waits: 4 s
constexpr int kPlanCTAs = 152;   // persistent CTAs work planners assume (one per SM of this part)

// Per-module launch record kept in workspace (global memory).  The tensor maps
// are read by TMA straight from there, so the record is 64-byte aligned.
struct ModDesc {
  CUtensorMap tmA;      // bf16 {d_in, T, B}, box {64, 32, 1}, 128B swizzle
  CUtensorMap tmG;      // bf16 {d_out, T, B}, box {64, 32, 1}, 128B swizzle
  CUtensorMap tmPin;    // bf16 {d_in, 2 k_in} (hi rows then lo rows), box {64, 2 k_in}
  CUtensorMap tmPout;   // bf16 {d_out, 2 k_out}, box {64, 2 k_out}
  int32_t d_in;
  int32_t d_out;
  int64_t col_offset;
  int64_t bias_col_offset;   // -1: no bias block
  int64_t reserved[5];
};
static_assert(alignof(ModDesc) >= 64 && sizeof(ModDesc) % 64 == 0, "TMA needs 64-byte aligned maps");

// One projection matrix to materialise: P'^T as bf16 hi rows [0, k) and lo rows
// [k, 2k), each of length d, with P'[i, j] = scale_i * P[i, j].
struct PrepSeg {
  uint64_t seed;
  const float* moment;      // r (output side) or c (input side), or nullptr
  __nv_bfloat16* dst;       // [2k, d]
  int64_t begin;            // unused (kept zero)
  int32_t d;
  int32_t k;
  int32_t kind;
  int32_t reserved;
};

// One entry of a projection launch's work table.  A fused item projects both
// sides of every tile of its slot and contracts them; a piece projects one
// side over a range of 64-column chunks and stores the fp32 token
// projections, and the last piece of a slot to finish sums them and contracts.
struct WorkItem {
  int32_t slot;              // partial index (m * B + b) * n_chunks + chunk
  int32_t side;              // 0: fused; 1: A-side piece; 2: G-side piece
  int32_t ch_begin, ch_end;  // chunk range of a piece
  int32_t split;             // piece counter index of the slot
  int32_t n_a, n_g;          // pieces of the slot on the A and G side
  int32_t piece;             // index of this piece on its side
  int64_t base;              // float offset of the slot's pieces in piece_buf
};
static_assert(sizeof(WorkItem) == 40, "WorkItem layout");

struct ProjParams {
  const ModDesc* mods;
  int n_mods;
  int B;
  int T;
  int n_tiles;          // ceil(T / 128)
  int tpc;              // tiles per work item
  int n_chunks;         // work items per (module, example)
  int n_items;          // work items (n_mods * B * n_chunks without a work table)
  const uint8_t* mask;        // [B, T] or nullptr
  const uint8_t* tile_valid;  // [B, n_tiles] 4-bit masks of valid 32-token slices, or nullptr
  float* partials;            // [n_items, k_out * k_in]   (projection mode)
  float* bias_partials;       // [n_items, 128] column sums of g~, or nullptr (no bias)
  const float* queries;       // [n_queries, ld_q] query rows          (token mode)
  int64_t ld_q;
  int n_queries;
  float* token_partials;      // [n_mods, n_queries, B, T]             (token mode)
  const WorkItem* items;      // [n_items] work table, or nullptr: item i is fused slot i
  float* piece_buf;           // token projections of pieces (see WorkItem)
  int* split_cnt;             // per split slot: pieces finished, zero on entry
  int* counter;               // dynamic scheduler, zero on entry
  int* status;                // device status word
  uint64_t timeout_ns;
};

struct ScoreParams {
  int N;
  int K;
  int Q;
  int topk;
  int n_qg;             // query groups in this pass
  int qg_base;          // first query group of this pass
  int n_ntiles;         // ceil(N / 256)
  unsigned long long* heaps;  // [grid, topk, QT*128]
  const float* tau0;    // per query starting threshold at tau0[q * topk + topk - 1], or nullptr
  int tau0_negate;      // 1: the threshold is -tau0[...] (tau0 holds scores against q while
                        //    the search runs on -q: a bottom-k state)
  unsigned long long* pace;   // pair kernel, two or more pair groups: [grid] progress words
                              //   (launch tag << 32 | chunks issued), or nullptr
  unsigned int pace_tag;      // this launch's tag (never 0; differs between launches)
  int* status;
  uint64_t timeout_ns;
};

// Sets this thread's bergson_last_error() message (printf format) and returns `code`.
int record_error(int code, const char* fmt, ...);

// ---- launchers (return the launch error, if any) ----

// Both record BERGSON_EMOMENT in *status when a second-moment entry is not > 0.
cudaError_t launch_prep(const PrepSeg* segs, int n_segs, int64_t max_pairs, int* status,
                        cudaStream_t s);
cudaError_t launch_projection_matrix(uint64_t seed, int d, int k, int kind, const float* moment,
                                     int* status, float* out, cudaStream_t s);
cudaError_t launch_tile_valid(const uint8_t* mask, int B, int T, int n_tiles, uint8_t* tile_valid,
                              cudaStream_t s);
cudaError_t launch_wait_probe(int* status, uint64_t timeout_ns, cudaStream_t s);

// token = false: per-example projected gradients (partials); token = true:
// per-token scores against p.queries (token_partials).
cudaError_t launch_project(int k_in, int k_out, bool token, const ProjParams& p, int grid,
                          cudaStream_t s);
// Queries whose blocks token mode holds in shared memory at once (more are
// streamed through in blocks of this many).
int token_query_capacity(int k_in, int k_out);
cudaError_t launch_token_reduce(const float* token_partials, int n_mods, int Q, int B, int T,
                                const uint8_t* mask, float* out, cudaStream_t s);
cudaError_t launch_reduce(const ModDesc* mods, int n_mods, int k_in, int k_out, int B,
                          int n_chunks, const float* partials, const float* bias_partials,
                          float* out, int64_t ld_out, cudaStream_t s);

cudaError_t launch_build_store(const float* proj, int B, int K, int64_t ld_proj, int unit,
                               __half* store, int64_t ld_store, float* norms, cudaStream_t s);
// Column blocks of a store row normalised separately (one module each).
constexpr int kMaxStoreBlocks = 2048;
struct StoreBlocks {
  int32_t offset[kMaxStoreBlocks + 1];   // 0 = offset[0] < ... < offset[n] = K, multiples of 8
  int32_t n;
};
cudaError_t launch_build_store_blocks(const float* proj, int B, int64_t ld_proj,
                                      const StoreBlocks& blocks, __half* store, int64_t ld_store,
                                      float* norms, cudaStream_t s);
cudaError_t launch_normalize_queries(const float* q, int Q, int K, int64_t ld_q, bool negate,
                                     __half* qh, cudaStream_t s);
cudaError_t launch_score(int qt, const CUtensorMap& tm_store, const CUtensorMap& tm_q,
                         const ScoreParams& p, int grid, cudaStream_t s);
// Two-SM variant (clusters of two CTAs, qt x 128 queries per CTA, 128 store
// rows per CTA per tile): the store tensor map has 128-row boxes, grid and
// n_qg are even.
cudaError_t launch_score_pair(int qt, const CUtensorMap& tm_store, const CUtensorMap& tm_q,
                              const ScoreParams& p, int grid, cudaStream_t s);
cudaError_t score_pair_max_ctas(int qt, int sms, int* ctas);
constexpr int kPairMinQueries = 129;   // the pair kernel serves Q >= this
// Final top-k of queries [q_begin, q_end) from the CTAs' heaps.  Heap rows
// are local to the scored rows; the results report row_base + row.  With
// prior_scores / prior_idx (a previous [Q, topk] result over other rows, global
// indices, ordered as this call's output) the prior entries take part in the
// selection too; they may alias out_scores / out_idx.
cudaError_t launch_merge(const unsigned long long* heaps, int grid, int n_qg, int qt, int topk,
                         int q_begin, int q_end, int qg_base, bool negate, int64_t row_base,
                         const float* prior_scores, const int64_t* prior_idx, float* out_scores,
                         int64_t* out_idx, cudaStream_t s);

cudaError_t launch_row_scales(const float* x, int n, int K, int64_t ld, int unit, float* scale,
                              cudaStream_t s);
cudaError_t launch_aggregate(const float* rows, int64_t n, int K, int64_t ld,
                             const int64_t* offsets, int G, int mode, const float* scale,
                             float* out, int64_t ld_out, cudaStream_t s);
size_t fisher_fit_workspace(int64_t n, int64_t K);
cudaError_t launch_fisher_fit(const float* x, int n, int K, int64_t ldx, float* r, int64_t ldr,
                              float* ws, int* status, int sms, cudaStream_t s);
size_t fisher_power_workspace(int64_t K);
// At most `iterations` Newton-Schulz updates.  With residuals != nullptr or
// tol > 0 the residual ||I - Z Y||_F / sqrt(K) of every iterate is read back
// (one stream synchronisation per iterate) into residuals[0 ..] and the
// iteration stops at the first iterate whose residual is <= tol;
// *iterations_done receives the number of updates applied.
cudaError_t launch_fisher_power(const float* r1, const float* r2, int K, int64_t ldr, float lam,
                                float damping, int inverse, int iterations, float tol,
                                float* residuals, int* iterations_done, float* m, int64_t ldm,
                                float* ws, int* status, int sms, cudaStream_t s);

// Skinny fp32 product C[b, q] = <x_b, y_q> on the tensor cores (on-the-fly
// scores, preconditioner application): plan and workspace layout.
struct XGemmPlan {
  int n_pad = 16;          // batch rows per tile (multiple of 16; <= 64 on pairs, <= 128 else)
  int n_ntiles = 1;        // ceil(B / n_pad)
  int n_mtiles = 1;        // ceil(Q / y_rows)
  int steps = 1;           // ceil(K / 32)
  int S = 1;               // K slices (pairs: the most segments of any y tile)
  int n_clusters = 0;      // pairs: clusters the (y tile, step) space is split over
  int stages = 2;          // shared-memory pipeline depth
  int n_chunks = 1;        // column chunks of x for the row split (norm partials per row)
  bool pair = false;       // CTA pairs with y in TMEM (B <= 64)
  int n_buf = 2;           // accumulator sets in TMEM
  int y_rows = 128;        // rows of y per work item (256 on pairs: 128 per CTA)
  int a_base = 0;          // pairs: TMEM column of the y operand ring (a slot per stage)
  int a_slots = 0;         // pairs: slots of that ring (64 columns each; as many as stages)
  bool two_issuers = false;  // pairs: y_hi and y_lo products issued by two threads (n_pad <= 32)
  int sub = 8;             // 32-column steps per accumulation chain (at most)
  int tmem_cols = 32;      // TMEM columns allocated per CTA
  size_t xnorm_off = 0, ynorm_off = 0, partial_off = 0, xh_off = 0, xl_off = 0, total = 0;
};
XGemmPlan xgemm_plan(int64_t B, int64_t Q, int64_t K);

struct XGemmArgs {
  const float* x;          // [B, ldx] fp32, 16-byte aligned rows
  int64_t ldx;
  const float* y;          // [Q, ldy] fp32, 16-byte aligned rows
  int64_t ldy;
  int B, Q, K;
  int unit;                // 1: cosine (scale by both norms), 0: affine (below)
  float alpha = 1.0f;      // unit == 0: out = alpha' <x_b, y_q> + beta out + gamma [b == q],
  const float* alpha_s = nullptr;   //   alpha' = alpha * (*alpha_s) when alpha_s is given
  float beta = 0.0f;
  float gamma = 0.0f;
  float* scores;           // out [B, ld_scores]
  int64_t ld_scores;
  uint8_t* ws;             // workspace laid out by xgemm_plan(B, Q, K)
  int* status;
  uint64_t timeout_ns;
};
// Encodes the tensor maps and launches the split, product and finishing
// kernels.  Returns cudaErrorInvalidValue if a tensor map cannot be encoded.
cudaError_t xgemm_run(const XGemmArgs& a, int sms, cudaStream_t s);

// 2-D tiled tensor map with the 128-byte swizzle (host; defined with the C ABI).
CUresult encode_tmap_2d(CUtensorMap* tm, CUtensorMapDataType dt, const void* ptr, int64_t inner,
                        int64_t outer, int64_t row_bytes, int box_inner, int box_outer);

}  // namespace bergson
