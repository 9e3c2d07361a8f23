// On-the-fly scores (Bergson Sec. 3.1, "bergson score"): projected training
// gradients scored directly against fixed query gradients, with no gradient
// store in between.  Table 3's grad-cosine (unit-normalised rows and queries)
// and grad-dot (raw inner products) are both served:
//   scores[b, q] = <x_b, y_q> * s_b * t_q,  s = 1/||x||, t = 1/||y|| (cosine) or 1.
// The same skinny product applies the preconditioner (Sec. 3.2): there y is
// the K x K matrix M and the outputs are the preconditioned rows M x_b.
//
// The product C[b, q] = <x_b, y_q> runs on the tensor cores (tcgen05,
// kind::tf32) at fp32 accuracy.  tf32 keeps 10 of fp32's 23 mantissa bits, so
// every operand is split into two tf32 values:
//   y ~= y_hi + y_lo,  y_lo = tf32(y - y_hi)   (error <= 2^-22 |y|),
//   <x, y> ~= <x_hi, y_hi> + <x_lo, y_hi> + <x_hi, y_lo>
// (the 3xTF32 scheme of Ootomo and Yokota, 2022); the fourth product
// <x_lo, y_lo> (relative size <= 2^-22) is kept where it comes for free.
//
// y (queries, or M) is the large operand and is streamed from HBM once: TMA
// loads 128-row x 32-column fp32 tiles of y (128-byte swizzle) into a
// shared-memory ring; the tile itself is y_hi (the tensor cores truncate it)
// and converter warps compute its y_lo = tf32(y - trunc(y)) and, for cosine
// scores, the rows' squared norms from the same tile.  x is split by a
// pre-pass into x_hi and x_lo (and its norms) in workspace, and its tiles
// come from L2.  Two kernels:
//
//  * batch tiles of up to 64 rows (the common case: a training batch, a
//    handful of query rows): CTA pairs, y_hi and y_lo in TMEM as the A
//    operands of M = 256 MMAs over both CTAs' y rows (xgemm_pair_kernel);
//  * larger batch tiles (up to 128 rows): single CTAs, y_lo written next to
//    y in shared memory (xgemm_kernel).
//
// Work items are (tile of y, batch tile, K slice), handed out round-robin to
// persistent CTAs or pairs (all items have the same cost); every item writes
// an fp32 partial that a finishing kernel sums over the K slices in order and
// scales (deterministic result).  Every wait is bounded.

#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

namespace bergson {

namespace {

constexpr int kRowThreads = 256;
constexpr int kSplitChunk = 2048;          // fp32 columns of x per splitting CTA
constexpr int kXM = 128;                   // rows of y per tile, M side (MMA M)
constexpr int kXK = 32;                    // fp32 columns per stage: one 128-byte row
constexpr int kYBytes = kXM * 128;         // one y tile, M side
constexpr int kXThreads = 320;             // producer, MMA, 4 converter, 4 epilogue warps
constexpr int kPThreads = 352;             // pairs: the same and a second MMA issuer warp
constexpr int kXSmemBudget = 232448;       // 227 KB opt-in per CTA
constexpr int kXBarBytes = 512;
constexpr int kXMaxStages = 8;
constexpr int kMaxSlices = 64;
constexpr uint64_t kXDrainTimeoutNs = 2000000000ull;
// The tensor cores' fp32 accumulation rounds toward zero: every MMA into a
// running TMEM sum loses up to one ulp of it, so a long chain drifts (about
// -5e-8 of the sum per MMA, measured: -2.7e-5 over 4,096 columns of positive
// terms).  Each accumulation chain therefore covers at most kSubSteps
// 32-column steps of 8 MMAs each (4 MMAs of K = 8 into each of y_hi and y_lo
// terms, which both kernels add into one accumulator): the MMA warp restarts
// the accumulator after that many steps and the epilogue adds the pieces with
// IEEE fp32 adds, in order.
constexpr int kSubSteps = 8;
constexpr int kMaxPad = 128;                 // largest batch tile (n_pad)
constexpr int kMaxPadN = 64;                 // largest batch tile on CTA pairs

struct KahanSum {
  float s = 0.0f, c = 0.0f;
  __device__ __forceinline__ void add(float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
  }
};

// v rounded to the nearest tf32 value (10 explicit mantissa bits; ties away
// from zero), as an fp32 bit pattern whose low 13 bits are zero.
__device__ __forceinline__ float tf32_round(float v) {
  return __uint_as_float((__float_as_uint(v) + 0x1000u) & 0xFFFFE000u);
}

// v = hi + lo + e with hi, lo exact tf32 values and |e| <= 2^-22 |v|: the
// tensor cores read both parts exactly.
__device__ __forceinline__ void tf32_split(float4 v, float4& hi, float4& lo) {
  hi = make_float4(tf32_round(v.x), tf32_round(v.y), tf32_round(v.z), tf32_round(v.w));
  lo = make_float4(tf32_round(v.x - hi.x), tf32_round(v.y - hi.y), tf32_round(v.z - hi.z),
                   tf32_round(v.w - hi.w));
}

__device__ __forceinline__ float tf32_trunc(float v) {
  return __uint_as_float(__float_as_uint(v) & 0xFFFFE000u);
}

// The tensor cores read an fp32 operand of kind::tf32 as tf32 by dropping its
// low 13 mantissa bits (truncation; the fp64 checks of the tests would show
// errors near 2^-12 otherwise).  So y itself serves as y_hi = trunc(y), and
// y_lo = tf32(y - trunc(y)) is what truncation leaves out, rounded to nearest.
__device__ __forceinline__ float4 tf32_remainder(float4 v) {
  return make_float4(tf32_round(v.x - tf32_trunc(v.x)), tf32_round(v.y - tf32_trunc(v.y)),
                     tf32_round(v.z - tf32_trunc(v.z)), tf32_round(v.w - tf32_trunc(v.w)));
}

// scale[i] = 1/||row_i|| (unit, 0 for a zero row) or 1.  One CTA per row,
// 16-byte loads, compensated fp32 sums per thread (fp64 is slow on this part).
__global__ void __launch_bounds__(kRowThreads) row_scales_kernel(
    const float* __restrict__ x, int K, int64_t ld, int unit, float* __restrict__ scale) {
  __shared__ float red[kRowThreads / 32];
  const float4* xr = reinterpret_cast<const float4*>(x + blockIdx.x * ld);
  KahanSum ks;
  for (int i = threadIdx.x; i < K / 4; i += kRowThreads) {
    const float4 v = xr[i];
    ks.add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
  }
  float s = ks.s;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float tot = 0.0f;
    for (int w = 0; w < kRowThreads / 32; ++w) tot += red[w];
    scale[blockIdx.x] = unit ? (tot > 0.0f ? 1.0f / sqrtf(tot) : 0.0f) : 1.0f;
  }
}

// Row b of x -> rows of x_hi and x_lo ([B, K], contiguous) and scale[b] as above.
__global__ void __launch_bounds__(kRowThreads) split_rows_kernel(
    const float* __restrict__ x, int K, int64_t ld, int unit, int n_chunks,
    float* __restrict__ xh, float* __restrict__ xl, float* __restrict__ xnorm) {
  // grid: (rows, chunks of kSplitChunk columns); each CTA splits one chunk of
  // one row and, for cosine scores, writes that chunk's compensated sum of
  // squares (the finishing kernel adds the chunks of a row in order).
  __shared__ float red[kRowThreads / 32];
  griddep_launch_dependents();   // the product kernel may start streaming y meanwhile
  const int64_t b = blockIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + b * ld);
  float4* hr = reinterpret_cast<float4*>(xh + b * K);
  float4* lr = reinterpret_cast<float4*>(xl + b * K);
  for (int c = blockIdx.y; c < n_chunks; c += gridDim.y) {
    const int i0 = c * (kSplitChunk / 4);
    const int i1 = min(K / 4, i0 + kSplitChunk / 4);
    KahanSum ks;
    for (int i = i0 + threadIdx.x; i < i1; i += kRowThreads) {
      const float4 v = xr[i];
      float4 h, l;
      tf32_split(v, h, l);
      hr[i] = h;
      lr[i] = l;
      ks.add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
    }
    if (!unit) continue;
    float s = ks.s;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.0f;
      for (int w = 0; w < kRowThreads / 32; ++w) tot += red[w];
      xnorm[b * n_chunks + c] = tot;
    }
    __syncthreads();
  }
}
struct XGemmParams {
  int B, Q;
  int n_pad, n_mtiles, S, steps, stages;
  int n_items;
  int tmem_cols;
  int sub;            // 32-column steps per accumulation chain
  int a_base;         // pairs: TMEM column of the y_hi / y_lo ring (a slot per stage)
  int n_clusters;     // pairs: clusters sharing the (y tile, step) space evenly
  int unit;
  float* partial;     // [S, B, Q]
  float* ynorm;       // [S, Q] squared norms of y rows over each slice (unit only)
  int* status;
  uint64_t timeout_ns;
};

struct XItem {
  int mt, nt, z, s0, s1;
};

__device__ __forceinline__ XItem decode_xitem(const XGemmParams& p, int item) {
  XItem it;
  it.z = item % p.S;
  const int t = item / p.S;
  it.mt = t % p.n_mtiles;
  it.nt = t / p.n_mtiles;
  it.s0 = static_cast<int>(static_cast<int64_t>(it.z) * p.steps / p.S);
  it.s1 = static_cast<int>(static_cast<int64_t>(it.z + 1) * p.steps / p.S);
  return it;
}

// Pairs split the n_mtiles x steps (y tile, 32-column step) space evenly
// over the clusters in order: cluster c takes positions [c W / n, (c + 1) W
// / n), W = n_mtiles steps, cut at tile boundaries into segments.  The
// segments of a tile are its K slices; a segment's partial plane is its
// cluster's rank among the clusters that meet the tile.  The cluster that
// holds position g: ceil((g + 1) n / W) - 1.
__host__ __device__ __forceinline__ int seg_cluster_of(int64_t g, int64_t W, int n) {
  return static_cast<int>(((g + 1) * n + W - 1) / W) - 1;
}
__host__ __device__ __forceinline__ int seg_planes(int mt, int steps, int64_t W, int n) {
  const int64_t p0 = static_cast<int64_t>(mt) * steps;
  return seg_cluster_of(p0 + steps - 1, W, n) - seg_cluster_of(p0, W, n) + 1;
}

struct SegIter {
  int64_t g, g1, W;
  int steps, n, cid;
  XItem it;
  __device__ __forceinline__ SegIter(const XGemmParams& p, int c) {
    steps = p.steps;
    n = p.n_clusters;
    cid = c;
    W = static_cast<int64_t>(p.n_mtiles) * steps;
    g = c * W / n;
    g1 = (c + 1) * W / n;
    load();
  }
  __device__ __forceinline__ bool valid() const { return g < g1; }
  __device__ __forceinline__ void load() {
    if (g >= g1) return;
    it.mt = static_cast<int>(g / steps);
    it.nt = 0;
    it.s0 = static_cast<int>(g % steps);
    const int64_t end = it.s0 + (g1 - g);
    it.s1 = end < steps ? static_cast<int>(end) : steps;
    it.z = cid - seg_cluster_of(static_cast<int64_t>(it.mt) * steps, W, n);
  }
  __device__ __forceinline__ void next() {
    g += it.s1 - it.s0;
    load();
  }
};

// Lane 0 waits, the warp takes its answer (keeps the warp's control flow
// uniform).  Inline: the converter and epilogue warps keep running sums in
// registers across these waits.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, uint64_t tmo,
                                          const volatile int* abort_flag) {
  bool ok = true;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_inline(bar, parity, tmo, abort_flag);
  return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}

// The producer warp's loop, shared by both kernels: y tiles of y_rows rows at
// once, x tiles (the row split's output) only after griddep_wait(), so the
// first round of stages streams y while the split grid finishes.
__device__ __forceinline__ void xgemm_produce(const CUtensorMap* tm_y, const CUtensorMap* tm_xh,
                                              const CUtensorMap* tm_xl, const XGemmParams& p,
                                              uint32_t sbase, int stage_bytes, int xoff,
                                              int y_rows, uint64_t* full, uint64_t* empty,
                                              volatile int* s_abort) {
  prefetch_tmap(tm_y);
  prefetch_tmap(tm_xh);
  prefetch_tmap(tm_xl);
  const int xbytes = p.n_pad * 128;
  const uint64_t pol_y = policy_evict_first();    // streamed once
  const uint64_t pol_x = policy_evict_last();     // re-read by every tile
  int stage = 0;
  uint32_t ph = 0;
  uint32_t issued = 0, issued_par = 0;
  bool ok = true;
  bool dep = false;
  int n_def = 0;
  int def_st[kXMaxStages], def_nt[kXMaxStages];
  auto load_x = [&](int sg, int st, int nt) {
    const uint32_t fb = smem_u32(&full[sg]);
    const uint32_t dst = sbase + sg * stage_bytes + xoff;
    tma_load_2d_hint(dst, tm_xh, fb, st * kXK, nt * p.n_pad, pol_x);
    tma_load_2d_hint(dst + xbytes, tm_xl, fb, st * kXK, nt * p.n_pad, pol_x);
  };
  auto release = [&]() {
    griddep_wait();
    dep = true;
    for (int d = 0; d < n_def; ++d) load_x(d, def_st[d], def_nt[d]);
    n_def = 0;
  };
  for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x) {
    const XItem it = decode_xitem(p, item);
    for (int st = it.s0; st < it.s1; ++st) {
      if (!mbar_wait(smem_u32(&empty[stage]), ph ^ 1, p.timeout_ns, s_abort)) { ok = false; break; }
      const uint32_t fb = smem_u32(&full[stage]);
      mbar_arrive_expect_tx(fb, y_rows * 128 + 2 * xbytes);
      tma_load_2d_hint(sbase + stage * stage_bytes, tm_y, fb, st * kXK, it.mt * y_rows, pol_y);
      if (dep) {
        load_x(stage, st, it.nt);
      } else {
        def_st[n_def] = st;                     // first round: stage == n_def
        def_nt[n_def] = it.nt;
        if (++n_def == p.stages) release();
      }
      issued |= 1u << stage;
      issued_par = (issued_par & ~(1u << stage)) | (ph << stage);
      if (++stage == p.stages) { stage = 0; ph ^= 1; }
    }
  }
  if (!dep) release();
  griddep_launch_dependents();   // every load issued: the finishing grid may launch
  if (!ok) {
    raise_device_error(p.status, s_abort, kStatusTimeout);
    for (int s = 0; s < p.stages; ++s)
      if (issued >> s & 1)
        mbar_wait(smem_u32(&full[s]), (issued_par >> s) & 1, kXDrainTimeoutNs, nullptr);
  }
}

// y on the M side, batch tiles of up to 128 rows: y_lo is written next to y
// in shared memory, and y_lo x_hi adds into the y_hi x_hi columns so that two
// accumulator sets of 2 n_pad columns fit in TMEM.
__global__ void __launch_bounds__(kXThreads, 1)
    xgemm_kernel(const __grid_constant__ CUtensorMap tm_y, const __grid_constant__ CUtensorMap tm_xh,
                 const __grid_constant__ CUtensorMap tm_xl, const XGemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const int xbytes = p.n_pad * 128;
  const int xoff = 2 * kYBytes;                 // x_hi, x_lo after y and y_lo
  const int stage_bytes = xoff + 2 * xbytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + p.stages * stage_bytes);
  uint64_t* empty = full + p.stages;
  uint64_t* conv = empty + p.stages;
  uint64_t* tfull = conv + p.stages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
      mbar_init(smem_u32(&conv[s]), 128);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), 4);
    }
    mbar_init(smem_u32(drain), 1);
    *s_abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(s_tmem), p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const uint64_t tmo = p.timeout_ns;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0)
      xgemm_produce(&tm_y, &tm_xh, &tm_xl, p, sbase, stage_bytes, xoff, kXM, full, empty, s_abort);
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = make_idesc_tf32(kXM, 2 * p.n_pad);   // y_hi [x_hi; x_lo]^T
      const uint32_t idesc_lo = make_idesc_tf32(kXM, p.n_pad);    // y_lo x_hi^T
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x) {
        const XItem it = decode_xitem(p, item);
        for (int c0 = it.s0; c0 < it.s1 && ok; c0 += p.sub) {
          const int c1 = min(it.s1, c0 + p.sub);
          if (!mbar_wait(smem_u32(&tempty[ab]), aph ^ 1, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          // Set ab, 2 n_pad columns: y_hi [x_hi; x_lo]^T (x_hi and x_lo land
          // next to each other, so one B operand of 2 n_pad rows serves both),
          // with y_lo x_hi^T added into its first n_pad columns.
          const uint32_t d = tmem + ab * 2 * p.n_pad;
          for (int st = c0; st < c1; ++st) {
            if (!mbar_wait(smem_u32(&full[stage]), ph, tmo, s_abort) ||
                !mbar_wait(smem_u32(&conv[stage]), ph, tmo, s_abort)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t yh = sbase + stage * stage_bytes;
            const uint64_t dx = sw128_desc(yh + xoff);
            const uint64_t dyh = sw128_desc(yh);
            const uint64_t dyl = sw128_desc(yh + kYBytes);
#pragma unroll
            for (int kk = 0; kk < kXK / 8; ++kk) {     // 8 tf32 = 32 bytes: +2 in the address field
              const uint64_t o = 2 * kk;
              umma_tf32(d, dyh + o, dx + o, idesc, st != c0 || kk != 0);
              umma_tf32(d, dyl + o, dx + o, idesc_lo, 1u);
            }
            umma_commit(smem_u32(&empty[stage]));
            if (++stage == p.stages) { stage = 0; ph ^= 1; }
          }
          if (!ok) break;
          umma_commit(smem_u32(&tfull[ab]));
          if (++ab == 2) { ab = 0; aph ^= 1; }
        }
      }
      if (!ok) raise_device_error(p.status, s_abort, kStatusTimeout);
      umma_commit(smem_u32(drain));
      mbar_wait(smem_u32(drain), 0, kXDrainTimeoutNs, nullptr);
    }
    __syncwarp();
  } else if (warp < 6) {
    // ------------------------------------------------------------ converter
    // Thread ct owns 16-byte chunks ct + 128 i (i < 8) of each tile: rows
    // ct / 8 + 16 i, whatever the swizzle did to their columns.
    const int ct = threadIdx.x - 64;
    int stage = 0;
    uint32_t ph = 0;
    for (int item = blockIdx.x; item < p.n_items; item += gridDim.x) {
      const XItem it = decode_xitem(p, item);
      KahanSum nrm[8];
      bool aborted = false;
      for (int st = it.s0; st < it.s1; ++st) {
        if (!warp_wait(smem_u32(&full[stage]), ph, tmo, s_abort)) {
          raise_device_error(p.status, s_abort, kStatusTimeout);
          aborted = true;
          break;
        }
        float4* yb = reinterpret_cast<float4*>(smem + stage * stage_bytes);
        float4* lb = yb + kYBytes / 16;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int idx = ct + 128 * i;
          const float4 v = yb[idx];
          lb[idx] = tf32_remainder(v);
          if (p.unit) nrm[i].add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
        }
        fence_proxy_async_smem();
        mbar_arrive(smem_u32(&conv[stage]));
        if (++stage == p.stages) { stage = 0; ph ^= 1; }
      }
      if (aborted) break;
      if (p.unit && it.nt == 0) {
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float s = nrm[i].s;                        // the 8 lanes of a row, in a fixed order
          s += __shfl_xor_sync(0xffffffffu, s, 1);
          s += __shfl_xor_sync(0xffffffffu, s, 2);
          s += __shfl_xor_sync(0xffffffffu, s, 4);
          const int q = it.mt * kXM + ct / 8 + 16 * i;
          if ((ct & 7) == 0 && q < p.Q) p.ynorm[static_cast<int64_t>(it.z) * p.Q + q] = s;
        }
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;                    // TMEM lanes 32*quarter ..
    const int row = 32 * quarter + lane;
    int ab = 0;
    uint32_t aph = 0;
    bool aborted = false;
    for (int item = blockIdx.x; item < p.n_items && !aborted; item += gridDim.x) {
      const XItem it = decode_xitem(p, item);
      const int q = it.mt * kXM + row;
      // The item's chains, added in order in registers (compile-time indices:
      // the column loop is unrolled over the largest batch tile and guarded;
      // 0 + v = v, so the first chain lands unchanged).
      float acc[kMaxPad];
#pragma unroll
      for (int j = 0; j < kMaxPad; ++j) acc[j] = 0.0f;
      for (int c0 = it.s0; c0 < it.s1; c0 += p.sub) {
        if (!warp_wait(smem_u32(&tfull[ab]), aph, tmo, s_abort)) {
          raise_device_error(p.status, s_abort, kStatusTimeout);
          aborted = true;
          break;
        }
        tc_fence_after();
        const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * quarter) << 16) + ab * 2 * p.n_pad;
#pragma unroll
        for (int cb = 0; cb < kMaxPad / 16; ++cb) {
          const int c = 16 * cb;
          if (c < p.n_pad) {
            // <x_b, y_q> ~= (y_hi + y_lo) x_hi + y_hi x_lo
            float v[16], w[16];
            tmem_ld16(tbase + c, v);
            tmem_ld16(tbase + p.n_pad + c, w);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) acc[c + jj] += v[jj] + w[jj];
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&tempty[ab]));
        if (++ab == 2) { ab = 0; aph ^= 1; }
      }
      if (aborted) break;
      if (q < p.Q) {
        float* dst = p.partial + static_cast<int64_t>(it.z) * p.B * p.Q + q;
#pragma unroll
        for (int cb = 0; cb < kMaxPad / 16; ++cb) {
          const int c = 16 * cb;
          if (c < p.n_pad) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int b = it.nt * p.n_pad + c + j;
              if (b < p.B) dst[static_cast<int64_t>(b) * p.Q] = acc[c + j];
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

// Accumulation chains: an item of L steps is cut into ceil(L / sub) chains of
// near-equal length (floor or ceil of L / chains).
__host__ __device__ constexpr int chain_count(int L, int sub) { return (L + sub - 1) / sub; }
__host__ __device__ constexpr int chain_start(int L, int n_ch, int k) { return k * L / n_ch; }

// Batches of up to 64 rows: CTA pairs (clusters of two CTAs on two SMs).
// Each CTA of a pair streams its own 128-row half of a 256-row y tile and
// converts it into its own TMEM (y_hi and y_lo, the tf32 A operands); one
// tcgen05.mma of M = 256 then covers both halves: B = [x_hi; x_lo] (N = 2
// n_pad), x_hi from the even CTA's shared memory and x_lo from the odd CTA's.
// A small-N tcgen05 MMA costs about the same issue time whatever its size,
// and one pair MMA does the work of two single-CTA MMAs, so a pair issues
// half the instructions per byte of y that a lone CTA would (measured: 8
// MMAs per 16 KB stage cap a lone CTA near half the HBM rate).
//
// kTwo (batch tiles of up to 32 rows): one issuing thread still stalls about
// 115 cycles per MMA, so two threads issue.  Warp 1: y_hi [x_hi; x_lo]^T
// into the set's columns [0, 2 n_pad); warp 10: y_lo x_hi^T into [2 n_pad,
// 3 n_pad), its B = x_hi split over the pair (each CTA loads its n_pad / 2
// rows at the same offset).  Each issuer keeps a fixed order into its own
// columns, so the sums stay deterministic.  Without kTwo, one thread issues
// y_hi B^T and y_lo B^T into one 2 n_pad-column set (the fourth product
// y_lo x_lo comes for free).  The epilogue adds the parts.
//
// Work: the (y tile, step) space split evenly over the clusters in
// segments (SegIter); each segment is cut into accumulation chains.
//
// Synchronisation: each CTA's loads complete on its own `full` barrier; its
// converter warps then store the tile's y_hi / y_lo into the TMEM slot of
// that stage and arrive on the even CTA's `conv` barrier (eight arrivals:
// four warps of each CTA; CTA-scope release, as these signals only order
// tcgen05 operations: a cluster-scope release costs a memory barrier per
// arrival, which halved the stream rate).  The even CTA's MMA threads issue
// the stage's MMAs, and their commits free the stage in both CTAs (`empty`,
// multicast, one arrival per issuer) and hand finished accumulator sets to
// both CTAs' epilogues (`tfull`, likewise); every epilogue warp of both CTAs
// releases a set on the even CTA's `tempty`.  A stage's TMEM slot is written
// again only after its `full` barrier completes anew, i.e. after the `empty`
// commits of the MMAs that read it.
template <bool kUnit, bool kTwo>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPThreads, 1)
    xgemm_pair_kernel(const __grid_constant__ CUtensorMap tm_y, const __grid_constant__ CUtensorMap tm_xh,
                      const __grid_constant__ CUtensorMap tm_xl,
                      const __grid_constant__ CUtensorMap tm_xh2, const XGemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const int xbytes = p.n_pad * 128;
  // this CTA's y half, its half of B = [x_hi; x_lo], and with two issuers its
  // half of B' = x_hi for the y_lo products (N = n_pad: rows r n_pad / 2 ..)
  const int stage_bytes = kYBytes + xbytes + (kTwo ? xbytes / 2 : 0);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + p.stages * stage_bytes);
  uint64_t* empty = full + p.stages;
  uint64_t* conv = empty + p.stages;
  uint64_t* tfull = conv + p.stages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;                  // one per issuer
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(drain + 2);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const uint32_t rank = cluster_ctarank();       // 0: issues the MMAs
  const int cid = blockIdx.x >> 1;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), kTwo ? 2 : 1);   // a commit from each MMA issuer
      mbar_init(smem_u32(&conv[s]), 8);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&tfull[i]), kTwo ? 2 : 1);
      mbar_init(smem_u32(&tempty[i]), 8);
    }
    mbar_init(smem_u32(&drain[0]), 1);
    mbar_init(smem_u32(&drain[1]), 1);
    *s_abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(s_tmem), p.tmem_cols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();              // both CTAs' barriers initialised and TMEM allocated
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  const uint64_t tmo = p.timeout_ns;
  // one accumulator set: y_hi [x_hi; x_lo]^T (2 n_pad columns), then with two
  // issuers y_lo x_hi^T (n_pad columns)
  const int set_cols = (kTwo ? 3 : 2) * p.n_pad;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // y at once; x (the row split's output) after griddep_wait(), so the
    // first round of stages streams y while the split grid finishes.
    if (lane == 0) {
      prefetch_tmap(&tm_y);
      const CUtensorMap* tm_x = rank == 0 ? &tm_xh : &tm_xl;
      prefetch_tmap(tm_x);
      if constexpr (kTwo) prefetch_tmap(&tm_xh2);
      const uint64_t pol_y = policy_evict_first();    // streamed once
      const uint64_t pol_x = policy_evict_last();     // re-read by every tile
      int stage = 0;
      uint32_t ph = 0;
      uint32_t issued = 0, issued_par = 0;
      bool ok = true, dep = false;
      int n_def = 0;
      int def_st[kXMaxStages], def_nt[kXMaxStages];
      auto load_x = [&](int sg, int st, int nt) {
        tma_load_2d_hint(sbase + sg * stage_bytes + kYBytes, tm_x, smem_u32(&full[sg]), st * kXK,
                         nt * p.n_pad, pol_x);
        if constexpr (kTwo)
          tma_load_2d_hint(sbase + sg * stage_bytes + kYBytes + xbytes, &tm_xh2,
                           smem_u32(&full[sg]), st * kXK,
                           nt * p.n_pad + static_cast<int>(rank) * (p.n_pad / 2), pol_x);
      };
      auto release = [&]() {
        griddep_wait();
        dep = true;
        for (int d = 0; d < n_def; ++d) load_x(d, def_st[d], def_nt[d]);
        n_def = 0;
      };
      for (SegIter sg(p, cid); sg.valid() && ok; sg.next()) {
        const XItem& it = sg.it;
        for (int st = it.s0; st < it.s1; ++st) {
          if (!mbar_wait(smem_u32(&empty[stage]), ph ^ 1, tmo, s_abort)) { ok = false; break; }
          const uint32_t fb = smem_u32(&full[stage]);
          mbar_arrive_expect_tx(fb, stage_bytes);
          tma_load_2d_hint(sbase + stage * stage_bytes, &tm_y, fb, st * kXK,
                           it.mt * 2 * kXM + static_cast<int>(rank) * kXM, pol_y);
          if (dep) {
            load_x(stage, st, it.nt);
          } else {
            def_st[n_def] = st;                     // first round: stage == n_def
            def_nt[n_def] = it.nt;
            if (++n_def == p.stages) release();
          }
          issued |= 1u << stage;
          issued_par = (issued_par & ~(1u << stage)) | (ph << stage);
          if (++stage == p.stages) { stage = 0; ph ^= 1; }
        }
      }
      if (!dep) release();
      griddep_launch_dependents();   // every load issued: the finishing grid may launch
      if (!ok) {
        raise_device_error(p.status, s_abort, kStatusTimeout);
        for (int s = 0; s < p.stages; ++s)
          if (issued >> s & 1)
            mbar_wait(smem_u32(&full[s]), (issued_par >> s) & 1, kXDrainTimeoutNs, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1 || warp == 10) {
    // ------------------------------------------------------------ MMA issuer(s) (even CTA)
    // kTwo: warp 1 issues the y_hi products into the set's first 2 n_pad
    // columns and warp 10 the y_lo products into the next 2 n_pad, each in a
    // fixed order (two issuing threads keep the tensor pipe fed: one stalls
    // about 115 cycles per MMA instruction at these shapes).
    if (rank == 0 && lane == 0 && (warp == 1 || kTwo)) {
      const int who = warp == 10 ? 1 : 0;           // 1: the y_lo issuer
      // y [x_hi; x_lo]^T, or for the y_lo issuer y_lo x_hi^T; M = 256
      const uint32_t idesc = make_idesc_tf32(2 * kXM, (who ? 1 : 2) * p.n_pad);
      int stage = 0;
      uint32_t ph = 0;
      int ab = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (SegIter sg(p, cid); sg.valid() && ok; sg.next()) {
        const XItem& it = sg.it;
        const int L = it.s1 - it.s0;
        const int n_ch = chain_count(L, p.sub);
        for (int k = 0; k < n_ch && ok; ++k) {
          const int c0 = it.s0 + chain_start(L, n_ch, k), c1 = it.s0 + chain_start(L, n_ch, k + 1);
          if (!mbar_wait(smem_u32(&tempty[ab]), aph ^ 1, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d = tmem + ab * set_cols + who * 2 * p.n_pad;   // y_lo part after y_hi
          for (int st = c0; st < c1; ++st) {
            if (!mbar_wait(smem_u32(&conv[stage]), ph, tmo, s_abort)) { ok = false; break; }
            tc_fence_after();
            const uint32_t ta = tmem + p.a_base + stage * 2 * kXK;    // y_hi, then y_lo
            const uint64_t dx =
                sw128_desc(sbase + stage * stage_bytes + kYBytes + who * xbytes);   // B or B'
#pragma unroll
            for (int kk = 0; kk < kXK / 8; ++kk) {   // 8 tf32 = 32 bytes: +2 in the address field
              const uint32_t acc = st != c0 || kk != 0;
              if constexpr (kTwo) {
                umma_tf32_pair_ta(d, ta + who * kXK + 8 * kk, dx + 2 * kk, idesc, acc);
              } else {
                umma_tf32_pair_ta(d, ta + 8 * kk, dx + 2 * kk, idesc, acc);
                umma_tf32_pair_ta(d, ta + kXK + 8 * kk, dx + 2 * kk, idesc, 1u);
              }
            }
            umma_commit_pair(smem_u32(&empty[stage]), 0x3);
            if (++stage == p.stages) { stage = 0; ph ^= 1; }
          }
          if (!ok) break;
          umma_commit_pair(smem_u32(&tfull[ab]), 0x3);
          if (++ab == 2) { ab = 0; aph ^= 1; }
        }
      }
      if (!ok) raise_device_error(p.status, s_abort, kStatusTimeout);
      umma_commit_pair(smem_u32(&drain[who]), 0x1);
      mbar_wait(smem_u32(&drain[who]), 0, kXDrainTimeoutNs, nullptr);
    }
    __syncwarp();
  } else if (warp < 6) {
    // ------------------------------------------------------------ converter
    // Thread = row r of this CTA's y half = TMEM lane r (warp w reaches lanes
    // 32 (w % 4) ..).  Chunk c (columns 4c .. 4c + 3) of row r sits at chunk
    // c ^ (r % 8) of the 128-byte swizzled row.
    const int quarter = warp & 3;
    const int r = 32 * quarter + lane;
    const uint32_t trow = tmem + (static_cast<uint32_t>(32 * quarter) << 16) + p.a_base;
    int stage = 0;
    uint32_t ph = 0;
    bool aborted = false;
    for (SegIter sg(p, cid); sg.valid() && !aborted; sg.next()) {
      const XItem& it = sg.it;
      KahanSum nrm;
      for (int st = it.s0; st < it.s1; ++st) {
        if (!warp_wait(smem_u32(&full[stage]), ph, tmo, s_abort)) {
          aborted = true;
          break;
        }
        tc_fence_after();          // the MMAs that last read this TMEM slot are done
        const uint8_t* row = smem + stage * stage_bytes + r * 128;
        float hv[kXK], lv[kXK];
#pragma unroll
        for (int c = 0; c < kXK / 4; ++c) {
          const float4 v = *reinterpret_cast<const float4*>(row + ((c ^ (r & 7)) << 4));
          const float4 l = tf32_remainder(v);
          hv[4 * c] = v.x; hv[4 * c + 1] = v.y; hv[4 * c + 2] = v.z; hv[4 * c + 3] = v.w;
          lv[4 * c] = l.x; lv[4 * c + 1] = l.y; lv[4 * c + 2] = l.z; lv[4 * c + 3] = l.w;
          if constexpr (kUnit) nrm.add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
        }
        tmem_st32(trow + stage * 2 * kXK, hv);
        tmem_st32(trow + stage * 2 * kXK + kXK, lv);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(mapa_shared(smem_u32(&conv[stage]), 0));
        if (++stage == p.stages) { stage = 0; ph ^= 1; }
      }
      if (aborted) break;
      if constexpr (kUnit) {
        const int q = it.mt * 2 * kXM + static_cast<int>(rank) * kXM + r;
        if (it.nt == 0 && q < p.Q) p.ynorm[static_cast<int64_t>(it.z) * p.Q + q] = nrm.s;
      }
    }
    if (aborted) raise_device_error(p.status, s_abort, kStatusTimeout);
  } else {
    // ------------------------------------------------------------ epilogue
    // Thread = row of this CTA's y half (TMEM lane); the item's chains are
    // added in order in registers and written once.
    const int quarter = warp & 3;
    const int row = 32 * quarter + lane;
    int ab = 0;
    uint32_t aph = 0;
    bool aborted = false;
    for (SegIter sg(p, cid); sg.valid() && !aborted; sg.next()) {
      const XItem& it = sg.it;
      const int q = it.mt * 2 * kXM + static_cast<int>(rank) * kXM + row;
      const int L = it.s1 - it.s0;
      const int n_ch = chain_count(L, p.sub);
      float acc[kMaxPadN];          // 0 + v = v: the first chain lands unchanged
#pragma unroll
      for (int j = 0; j < kMaxPadN; ++j) acc[j] = 0.0f;
      for (int k = 0; k < n_ch; ++k) {
        if (!warp_wait(smem_u32(&tfull[ab]), aph, tmo, s_abort)) {
          raise_device_error(p.status, s_abort, kStatusTimeout);
          aborted = true;
          break;
        }
        tc_fence_after();
        const uint32_t tbase = tmem + (static_cast<uint32_t>(32 * quarter) << 16) + ab * set_cols;
#pragma unroll
        for (int cb = 0; cb < kMaxPadN / 16; ++cb) {
          const int c = 16 * cb;
          if (c < p.n_pad) {
            // <x_b, y_q> ~= (y_hi + y_lo) x_hi + (y_hi + y_lo) x_lo; with two
            // issuers y_hi x_hi + y_hi x_lo + y_lo x_hi, the last in the set's
            // third part
            float v[16], w[16];
            tmem_ld16(tbase + c, v);
            tmem_ld16(tbase + p.n_pad + c, w);
            if constexpr (kTwo) {
              float u[16];
              tmem_ld16(tbase + 2 * p.n_pad + c, u);       // y_lo x_hi
#pragma unroll
              for (int jj = 0; jj < 16; ++jj) acc[c + jj] += (v[jj] + w[jj]) + u[jj];
            } else {
#pragma unroll
              for (int jj = 0; jj < 16; ++jj) acc[c + jj] += v[jj] + w[jj];
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(mapa_shared(smem_u32(&tempty[ab]), 0));
        if (++ab == 2) { ab = 0; aph ^= 1; }
      }
      if (aborted) break;
      if (q < p.Q) {
        float* dst = p.partial + static_cast<int64_t>(it.z) * p.B * p.Q + q;
#pragma unroll
        for (int cb = 0; cb < kMaxPadN / 16; ++cb) {
          const int c = 16 * cb;
          if (c < p.n_pad) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const int b = it.nt * p.n_pad + c + j;
              if (b < p.B) dst[static_cast<int64_t>(b) * p.Q] = acc[c + j];
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  cluster_sync();              // no MMA, commit or remote arrival is still in flight
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, p.tmem_cols);
  }
}

// s = sum over slices z (in order) of partial[z, b, q] (on pairs the planes
// of q's y tile, its segments in K order).  Cosine (xnorm given): scores[b, q]
// = s / sqrt(nx_b) / sqrt(ny_q), nx_b the sum over the row's chunks (in
// order) of xnorm[b, c], ny_q the sum over the same planes of ynorm[z, q] (0
// when either row is zero).  Otherwise scores[b, q] = alpha' s + beta scores[b, q] +
// gamma [b == q], alpha' = alpha * (*alpha_s) when alpha_s is given.
__global__ void finish_kernel(const float* __restrict__ partial, int S, int B, int Q,
                              const float* __restrict__ xnorm, int n_chunks,
                              const float* __restrict__ ynorm, int seg_clusters, int steps,
                              int y_rows, float alpha, const float* __restrict__ alpha_s,
                              float beta, float gamma, float* scores, int64_t ld) {
  griddep_wait();                 // partials, norms and alpha_s come from earlier grids
  const int64_t n = static_cast<int64_t>(B) * Q;
  const float al = alpha_s != nullptr ? alpha * *alpha_s : alpha;
  const int q = blockIdx.x * blockDim.x + threadIdx.x;     // grid: (Q / 256, rows of b)
  if (q >= Q) return;
  // planes of this row's y tile: all S, or on pairs the tile's segments
  const int n_mtiles = (Q + y_rows - 1) / y_rows;
  const int planes = seg_clusters > 0 ? seg_planes(q / y_rows, steps,
                                                   static_cast<int64_t>(n_mtiles) * steps,
                                                   seg_clusters)
                                      : S;
  for (int b = blockIdx.y; b < B; b += gridDim.y) {
    const int64_t i = static_cast<int64_t>(b) * Q + q;
    float s = 0.0f;
    for (int z = 0; z < planes; ++z) s += partial[z * n + i];
    float* dst = scores + b * ld + q;
    if (xnorm != nullptr) {
      float nx = 0.0f, ny = 0.0f;
      for (int c = 0; c < n_chunks; ++c) nx += xnorm[static_cast<int64_t>(b) * n_chunks + c];
      for (int z = 0; z < planes; ++z) ny += ynorm[static_cast<int64_t>(z) * Q + q];
      *dst = nx > 0.0f && ny > 0.0f ? s * (1.0f / sqrtf(nx)) * (1.0f / sqrtf(ny)) : 0.0f;
    } else {
      float v = al * s;
      if (beta != 0.0f) v = fmaf(beta, *dst, v);
      if (b == q) v += gamma;
      *dst = v;
    }
  }
}

size_t round_up256(size_t x) { return (x + 255) / 256 * 256; }

template <typename Kernel>
cudaError_t launch_product(Kernel kernel, PerDeviceOnce& attr, int threads, int grid, size_t smem,
                           cudaStream_t s, const CUtensorMap& tm_y, const CUtensorMap& tm_xh,
                           const CUtensorMap& tm_xl, const XGemmParams& p) {
  const cudaError_t e = smem_attr_once(attr, kernel, kXSmemBudget);
  if (e != cudaSuccess) return e;
  return launch_dependent(kernel, dim3(grid), dim3(threads), smem, s, tm_y, tm_xh, tm_xl, p);
}

template <typename Kernel>
cudaError_t launch_pair(Kernel kernel, PerDeviceOnce& attr, int grid, size_t smem, cudaStream_t s,
                        const CUtensorMap& tm_y, const CUtensorMap& tm_xh,
                        const CUtensorMap& tm_xl, const CUtensorMap& tm_xh2, const XGemmParams& p) {
  const cudaError_t e = smem_attr_once(attr, kernel, kXSmemBudget);
  if (e != cudaSuccess) return e;
  return launch_dependent(kernel, dim3(grid), dim3(kPThreads), smem, s, tm_y, tm_xh, tm_xl, tm_xh2,
                          p);
}

}  // namespace

cudaError_t launch_row_scales(const float* x, int n, int K, int64_t ld, int unit, float* scale,
                              cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  row_scales_kernel<<<n, kRowThreads, 0, s>>>(x, K, ld, unit, scale);
  return cudaGetLastError();
}

XGemmPlan xgemm_plan(int64_t B, int64_t Q, int64_t K) {
  XGemmPlan pl;
  const int64_t b1 = B > 0 ? B : 1;
  // Batches of up to 64 rows run on CTA pairs (256 rows of y per item, y in
  // TMEM); larger ones on single CTAs with y_lo in shared memory.
  pl.pair = b1 <= kMaxPadN;
  pl.n_pad = static_cast<int>(std::min<int64_t>(pl.pair ? kMaxPadN : kMaxPad, (b1 + 15) / 16 * 16));
  pl.y_rows = pl.pair ? 2 * kXM : kXM;
  pl.n_ntiles = static_cast<int>((b1 + pl.n_pad - 1) / pl.n_pad);
  pl.n_mtiles = static_cast<int>(std::max<int64_t>(1, (Q + pl.y_rows - 1) / pl.y_rows));
  pl.steps = static_cast<int>(std::max<int64_t>(1, (K + kXK - 1) / kXK));
  pl.sub = kSubSteps;
  pl.n_buf = 2;
  const int ring_budget = kXSmemBudget - 1024 - kXBarBytes;
  int stage_bytes;
  if (pl.pair) {
    // two accumulator sets of 2 n_pad columns (4 n_pad with two MMA issuers,
    // batch tiles up to 32 rows), then the y_hi / y_lo ring (64 columns a
    // stage)
    pl.tmem_cols = 512;
    pl.two_issuers = pl.n_pad <= 32;
    pl.a_base = pl.n_buf * (pl.two_issuers ? 3 : 2) * pl.n_pad;
    stage_bytes = kYBytes + pl.n_pad * 128 + (pl.two_issuers ? pl.n_pad * 64 : 0);
    pl.stages = std::min({kXMaxStages, (512 - pl.a_base) / (2 * kXK), ring_budget / stage_bytes});
    pl.a_slots = pl.stages;
  } else {
    pl.tmem_cols = 32;
    while (pl.tmem_cols < pl.n_buf * 2 * pl.n_pad) pl.tmem_cols <<= 1;
    pl.a_base = 0;
    stage_bytes = 2 * kYBytes + 2 * pl.n_pad * 128;
    pl.stages = std::min(kXMaxStages, ring_budget / stage_bytes);
  }
  const int units = kPlanCTAs;
  // Pairs: the (y tile, step) space split evenly over the clusters; S = the
  // most segments (partial planes) any tile gets.
  if (pl.pair) {
    const int64_t W = static_cast<int64_t>(pl.n_mtiles) * pl.steps;
    pl.n_clusters = static_cast<int>(std::min<int64_t>(kPlanCTAs / 2, W));
    pl.S = 1;
    for (int mt = 0; mt < pl.n_mtiles; ++mt)
      pl.S = std::max(pl.S, seg_planes(mt, pl.steps, W, pl.n_clusters));
  }
  // Single CTAs: K slices, the fewest waves of persistent CTAs for the y
  // stream plus the partials each slice adds (written and read back once).
  const int64_t tiles = static_cast<int64_t>(pl.n_mtiles) * pl.n_ntiles;
  double best = -1.0;
  if (!pl.pair) pl.S = 1;
  for (int S = 1; S <= std::min(pl.steps, kMaxSlices) && !pl.pair; ++S) {
    if (tiles * S > (1ll << 30)) break;
    const int64_t waves = (tiles * S + units - 1) / units;
    const int64_t per_item = (pl.steps + S - 1) / S;
    const double cost = static_cast<double>(waves) * (per_item + 2) * stage_bytes +
                        8.0 * S * static_cast<double>(b1) * static_cast<double>(Q) / kPlanCTAs;
    if (best < 0.0 || cost < best) {
      best = cost;
      pl.S = S;
    }
  }
  size_t off = 0;
  pl.n_chunks = static_cast<int>(std::max<int64_t>(1, (K + kSplitChunk - 1) / kSplitChunk));
  pl.xnorm_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(b1) * pl.n_chunks);
  pl.ynorm_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(pl.S) * std::max<int64_t>(Q, 1));
  pl.partial_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(pl.S) * b1 * std::max<int64_t>(Q, 1));
  pl.xh_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(b1) * K);
  pl.xl_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(b1) * K);
  pl.total = off;
  return pl;
}

cudaError_t xgemm_run(const XGemmArgs& a, int sms, cudaStream_t s) {
  if (a.B == 0 || a.Q == 0) return cudaSuccess;
  const XGemmPlan pl = xgemm_plan(a.B, a.Q, a.K);
  CUtensorMap tm_y, tm_xh, tm_xl, tm_xh2;
  if (encode_tmap_2d(&tm_y, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.y, a.K, a.Q, a.ldy * 4, kXK, kXM) !=
          CUDA_SUCCESS ||
      encode_tmap_2d(&tm_xh, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.ws + pl.xh_off, a.K, a.B,
                     static_cast<int64_t>(a.K) * 4, kXK, pl.n_pad) != CUDA_SUCCESS ||
      encode_tmap_2d(&tm_xl, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.ws + pl.xl_off, a.K, a.B,
                     static_cast<int64_t>(a.K) * 4, kXK, pl.n_pad) != CUDA_SUCCESS ||
      (pl.two_issuers &&
       encode_tmap_2d(&tm_xh2, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.ws + pl.xh_off, a.K, a.B,
                      static_cast<int64_t>(a.K) * 4, kXK, pl.n_pad / 2) != CUDA_SUCCESS))
    return cudaErrorInvalidValue;
  float* xnorm = reinterpret_cast<float*>(a.ws + pl.xnorm_off);
  float* xh = reinterpret_cast<float*>(a.ws + pl.xh_off);
  float* xl = reinterpret_cast<float*>(a.ws + pl.xl_off);
  const dim3 sgrid(a.B, std::min(pl.n_chunks, 65535));
  split_rows_kernel<<<sgrid, kRowThreads, 0, s>>>(a.x, a.K, a.ldx, a.unit, pl.n_chunks, xh, xl,
                                                  xnorm);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;

  XGemmParams p;
  p.B = a.B;
  p.Q = a.Q;
  p.n_pad = pl.n_pad;
  p.n_mtiles = pl.n_mtiles;
  p.S = pl.S;
  p.steps = pl.steps;
  p.stages = pl.stages;
  p.n_items = pl.n_mtiles * pl.n_ntiles * pl.S;
  p.tmem_cols = pl.tmem_cols;
  p.sub = pl.sub;
  p.a_base = pl.a_base;
  p.n_clusters = pl.n_clusters;
  p.unit = a.unit;
  p.partial = reinterpret_cast<float*>(a.ws + pl.partial_off);
  p.ynorm = reinterpret_cast<float*>(a.ws + pl.ynorm_off);
  p.status = a.status;
  p.timeout_ns = a.timeout_ns;
  const size_t stage_bytes =
      pl.pair ? kYBytes + pl.n_pad * 128 + (pl.two_issuers ? pl.n_pad * 64 : 0)
              : 2 * kYBytes + 2 * pl.n_pad * 128;
  const size_t smem = 1024 + pl.stages * stage_bytes + kXBarBytes;
  static PerDeviceOnce attr_pair[4], attr_m;
  if (pl.pair) {
    const int grid = 2 * pl.n_clusters;        // the segmentation assumes exactly these
    if (!pl.two_issuers) tm_xh2 = tm_xh;        // not read
    if (pl.two_issuers)
      e = a.unit ? launch_pair(xgemm_pair_kernel<true, true>, attr_pair[0], grid, smem, s, tm_y,
                               tm_xh, tm_xl, tm_xh2, p)
                 : launch_pair(xgemm_pair_kernel<false, true>, attr_pair[1], grid, smem, s, tm_y,
                               tm_xh, tm_xl, tm_xh2, p);
    else
      e = a.unit ? launch_pair(xgemm_pair_kernel<true, false>, attr_pair[2], grid, smem, s, tm_y,
                               tm_xh, tm_xl, tm_xh2, p)
                 : launch_pair(xgemm_pair_kernel<false, false>, attr_pair[3], grid, smem, s, tm_y,
                               tm_xh, tm_xl, tm_xh2, p);
  } else {
    const int grid = std::max(1, std::min(sms > 0 ? sms : 1, p.n_items));
    e = launch_product(xgemm_kernel, attr_m, kXThreads, grid, smem, s, tm_y, tm_xh, tm_xl, p);
  }
  if (e != cudaSuccess) return e;

  const dim3 fgrid((a.Q + 255) / 256, std::min(a.B, 65535));
  const float* xn = a.unit ? xnorm : nullptr;
  return launch_dependent(finish_kernel, fgrid, dim3(256), 0, s, p.partial, pl.S, a.B, a.Q, xn,
                          pl.n_chunks, p.ynorm, pl.pair ? pl.n_clusters : 0, pl.steps, pl.y_rows,
                          a.alpha, a.alpha_s, a.beta, a.gamma, a.scores, a.ld_scores);
}

}  // namespace bergson
