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
// loads 32-column fp32 tiles of y (128-byte swizzle) into a shared-memory
// ring; the tile itself is y_hi (the tensor cores truncate it) and converter
// warps compute its y_lo (the swizzle permutes 16-byte chunks, so an
// elementwise map keeps the layout) and, for cosine scores, the rows' squared
// norms from the same tile.  x is split by a pre-pass into x_hi and x_lo (and
// its norms) in workspace, and its tiles come from L2.  Two kernels:
//
//  * batch tiles of up to 64 rows (the common case: a training batch, a
//    handful of query rows): y on the MMA's N side.  A = [x_hi; x_lo] (M =
//    twice the batch tile, 64 or 128 rows), B = 256 rows of y (N = 256), so
//    one MMA covers 32 KB of y for 8 columns: a tcgen05 MMA has a fixed issue
//    cost of roughly 150 cycles whatever its N, and eight MMAs of N = 32 on a
//    16 KB stage (y on the M side) cap the stream near half the HBM rate.
//    Per 32-column step: four MMAs read y as y_hi; the converter warps then
//    overwrite the stage with y_lo in place (they read the tile as soon as it
//    lands and store once those MMAs are done) and four more MMAs read y_lo
//    into the same accumulator.  Rows [0, n) of D are x_hi (y_hi + y_lo),
//    rows [n, 2n) x_lo (y_hi + y_lo); the two halves sit in different TMEM
//    lane quarters, so each goes to its own partial plane.
//  * larger batch tiles (up to 128 rows): y on the M side (M = 128 rows of y,
//    N = twice the batch tile), y_lo written next to y in shared memory.
//
// Work items are (tile of y, batch tile, K slice), handed out round-robin to
// persistent CTAs (all items have the same cost); every item writes fp32
// partial planes that a finishing kernel sums in order and scales
// (deterministic result).  Every wait is bounded.

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
constexpr int kNY = 256;                   // rows of y per tile, N side (MMA N)
constexpr int kNYBytes = kNY * 128;        // one y tile, N side
constexpr int kNLookahead = 2;             // y_hi steps issued ahead of the y_lo step (at most)
constexpr int kNStages = 3;                // N side: y stages
constexpr int kNLoSlots = 2;               // N side: y_lo slots
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
constexpr int kMaxPadN = 64;                 // largest batch tile with y on the N side

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
  int lookahead;      // N side: y_hi steps the MMA thread may issue ahead of y_lo
  int lo_slots;       // N side: y_lo slots
  int x_slots;        // N side: x slots
  int unit;
  float* partial;     // [planes, B, Q]
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

// Accumulation chains of the N-side kernel: an item of L steps is cut into
// ceil(L / sub) chains of near-equal length (floor or ceil of L / chains).
__device__ __forceinline__ int chain_count(int L, int sub) { return (L + sub - 1) / sub; }
__device__ __forceinline__ int chain_start(int L, int n_ch, int k) { return k * L / n_ch; }

// One thread's walk over the 32-column steps of the CTA's items, in order,
// with the chain the current step belongs to.
struct StepCursor {
  int item;
  XItem it;
  int st;
  int n_ch, ck, c_lo, c_hi;      // chains of the item, current chain [c_lo, c_hi)
  __device__ __forceinline__ void set_chain(int k) {
    const int L = it.s1 - it.s0;
    ck = k;
    c_lo = it.s0 + chain_start(L, n_ch, k);
    c_hi = it.s0 + chain_start(L, n_ch, k + 1);
  }
  __device__ __forceinline__ void load(const XGemmParams& p) {
    if (item < p.n_items) {
      it = decode_xitem(p, item);
      st = it.s0;
      n_ch = chain_count(it.s1 - it.s0, p.sub);
      set_chain(0);
    }
  }
  __device__ __forceinline__ void start(const XGemmParams& p) {
    item = blockIdx.x;
    load(p);
  }
  __device__ __forceinline__ bool valid(const XGemmParams& p) const { return item < p.n_items; }
  __device__ __forceinline__ bool chain_first() const { return st == c_lo; }
  __device__ __forceinline__ bool chain_last() const { return st + 1 == c_hi; }
  __device__ __forceinline__ void next(const XGemmParams& p) {
    if (++st < c_hi) return;
    if (st < it.s1) {
      set_chain(ck + 1);
    } else {
      item += gridDim.x;
      load(p);
    }
  }
};

// y on the N side, batch tiles of kPad = 32 or 64 rows (see the top of the
// file).  Three rings in shared memory, each released as soon as its last
// reader is done, so that y tiles are requested as early as possible:
//   y stages (p.stages x 32 KB): TMA -> four y_hi MMAs and the converters'
//     reads -> free;
//   y_lo slots (p.lo_slots x 32 KB): converters' stores -> four y_lo MMAs ->
//     free;
//   x slots (p.x_slots x 2 kPad rows): TMA (with the step's y tile, on the
//     same barrier) -> all eight MMAs -> free.
// The MMA thread issues, in a fixed order (the accumulation order, hence the
// result, never depends on timing), the y_hi MMAs of a step and then the y_lo
// MMAs of the step p.lookahead - 1 before it.  A chain's first y_hi step waits
// for the epilogue to release the accumulator set two chains back; that
// chain's last y_lo step has been issued by then when every chain has at
// least lookahead - 1 steps (the planner caps the lookahead accordingly).
//
// Accumulator D (M = 2 kPad rows, N = 256 columns, two sets in 512 TMEM
// columns): an M = 128 accumulator keeps row r in TMEM lane r; an M = 64 one
// keeps rows 16 j .. 16 j + 15 in lanes 32 j .. 32 j + 15 and leaves lanes
// 32 j + 16 .. 32 j + 31 untouched (measured).  Either way lane quarters 0
// and 1 hold the x_hi rows and quarters 2 and 3 the x_lo rows, in the same
// order; the two go to separate partial planes.  The epilogue warps add an
// item's chains in registers (64 values a thread) and store each item's
// planes once.
template <int kPad>
struct NSide {
  static constexpr int kEpiWarps = kPad == 32 ? 8 : 16;
  static constexpr int kThreads = 32 * (6 + kEpiWarps);  // producer, MMA, 4 converter, epilogue
  static constexpr int kRowsQ = kPad == 32 ? 16 : 32;     // accumulator rows per lane quarter
  static constexpr int kXBytes = 2 * kPad * 128;           // x_hi and x_lo rows of one step
};

// Shared-memory bytes of the N-side rings (before the barriers).
__host__ __device__ constexpr int nside_ring_bytes(int n_pad, int stages, int lo_slots,
                                                   int x_slots) {
  return (stages + lo_slots) * kNYBytes + x_slots * 2 * n_pad * 128;
}

template <int kPad, bool kUnit>
__global__ void __launch_bounds__(NSide<kPad>::kThreads, 1)
    xgemm_n_kernel(const __grid_constant__ CUtensorMap tm_y, const __grid_constant__ CUtensorMap tm_xh,
                   const __grid_constant__ CUtensorMap tm_xl, const XGemmParams p) {
  using C = NSide<kPad>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const int lo_off = p.stages * kNYBytes;                    // y_lo slots after the y stages
  const int x_off = lo_off + p.lo_slots * kNYBytes;          // x slots after those
  uint64_t* yfull = reinterpret_cast<uint64_t*>(
      smem + nside_ring_bytes(kPad, p.stages, p.lo_slots, p.x_slots));
  uint64_t* yempty = yfull + p.stages;
  uint64_t* lfull = yempty + p.stages;
  uint64_t* lempty = lfull + p.lo_slots;
  uint64_t* xempty = lempty + p.lo_slots;
  uint64_t* tfull = xempty + p.x_slots;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* s_abort = reinterpret_cast<volatile int*>(s_tmem + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < p.stages; ++s) {
      mbar_init(smem_u32(&yfull[s]), 1);
      mbar_init(smem_u32(&yempty[s]), 1 + 4);      // the y_hi MMAs' commit, 4 converter warps
    }
    for (int s = 0; s < p.lo_slots; ++s) {
      mbar_init(smem_u32(&lfull[s]), 128);
      mbar_init(smem_u32(&lempty[s]), 1);
    }
    for (int s = 0; s < p.x_slots; ++s) mbar_init(smem_u32(&xempty[s]), 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), C::kEpiWarps);
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
    // y tiles at once; x tiles (the row split's output) only after
    // griddep_wait(), so the first steps stream y while the split finishes.
    if (lane == 0) {
      prefetch_tmap(&tm_y);
      prefetch_tmap(&tm_xh);
      prefetch_tmap(&tm_xl);
      const uint64_t pol_y = policy_evict_first();    // streamed once
      const uint64_t pol_x = policy_evict_last();     // re-read by every tile
      int ys = 0, xs = 0;
      uint32_t yph = 0, xph = 0;
      uint32_t issued = 0, issued_par = 0;            // y stages with loads in flight
      bool ok = true, dep = false;
      const int n_first = min(p.stages, p.x_slots);
      int n_def = 0;
      int def_st[kXMaxStages], def_nt[kXMaxStages], def_ys[kXMaxStages], def_xs[kXMaxStages];
      auto load_x = [&](int y_stage, int x_slot, int st, int nt) {
        const uint32_t fb = smem_u32(&yfull[y_stage]);
        const uint32_t dst = sbase + x_off + x_slot * C::kXBytes;
        tma_load_2d_hint(dst, &tm_xh, fb, st * kXK, nt * kPad, pol_x);
        tma_load_2d_hint(dst + kPad * 128, &tm_xl, fb, st * kXK, nt * kPad, pol_x);
      };
      auto release = [&]() {
        griddep_wait();
        dep = true;
        for (int d = 0; d < n_def; ++d) load_x(def_ys[d], def_xs[d], def_st[d], def_nt[d]);
        n_def = 0;
      };
      for (int item = blockIdx.x; item < p.n_items && ok; item += gridDim.x) {
        const XItem it = decode_xitem(p, item);
        for (int st = it.s0; st < it.s1; ++st) {
          if (!dep && n_def == n_first) release();
          if (!mbar_wait(smem_u32(&yempty[ys]), yph ^ 1, tmo, s_abort) ||
              !mbar_wait(smem_u32(&xempty[xs]), xph ^ 1, tmo, s_abort)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&yfull[ys]);
          mbar_arrive_expect_tx(fb, kNYBytes + C::kXBytes);
          tma_load_2d_hint(sbase + ys * kNYBytes, &tm_y, fb, st * kXK, it.mt * kNY, pol_y);
          if (dep) {
            load_x(ys, xs, st, it.nt);
          } else {
            def_st[n_def] = st;
            def_nt[n_def] = it.nt;
            def_ys[n_def] = ys;
            def_xs[n_def] = xs;
            ++n_def;
          }
          issued |= 1u << ys;
          issued_par = (issued_par & ~(1u << ys)) | (yph << ys);
          if (++ys == p.stages) { ys = 0; yph ^= 1; }
          if (++xs == p.x_slots) { xs = 0; xph ^= 1; }
        }
      }
      if (!dep) release();
      griddep_launch_dependents();   // every load issued: the finishing grid may launch
      if (!ok) {
        raise_device_error(p.status, s_abort, kStatusTimeout);
        for (int s = 0; s < p.stages; ++s)
          if (issued >> s & 1)
            mbar_wait(smem_u32(&yfull[s]), (issued_par >> s) & 1, kXDrainTimeoutNs, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = make_idesc_tf32(2 * kPad, kNY);   // [x_hi; x_lo] y^T
      StepCursor hc, lc;                 // next y_hi step, next y_lo step
      hc.start(p);
      lc.start(p);
      int hy = 0, hx = 0, ll = 0, lx = 0;          // ring positions of the two cursors
      uint32_t hyph = 0, llph = 0;
      int hset = 0, lset = 0;                      // their accumulator sets
      uint32_t hsph = 0;
      int ahead = 0;
      bool ok = true;
      while (lc.valid(p)) {
        if (hc.valid(p) && ahead < p.lookahead) {
          const bool first = hc.chain_first();
          if (first && !mbar_wait(smem_u32(&tempty[hset]), hsph ^ 1, tmo, s_abort)) { ok = false; break; }
          if (!mbar_wait(smem_u32(&yfull[hy]), hyph, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          const uint64_t dx = sw128_desc(sbase + x_off + hx * C::kXBytes);
          const uint64_t dy = sw128_desc(sbase + hy * kNYBytes);
          const uint32_t d = tmem + hset * kNY;
#pragma unroll
          for (int kk = 0; kk < kXK / 8; ++kk)      // 8 tf32 = 32 bytes: +2 in the address field
            umma_tf32(d, dx + 2 * kk, dy + 2 * kk, idesc, first && kk == 0 ? 0u : 1u);
          umma_commit(smem_u32(&yempty[hy]));
          if (hc.chain_last() && ++hset == 2) { hset = 0; hsph ^= 1; }
          hc.next(p);
          if (++hy == p.stages) { hy = 0; hyph ^= 1; }
          if (++hx == p.x_slots) hx = 0;
          ++ahead;
        } else {
          if (!mbar_wait(smem_u32(&lfull[ll]), llph, tmo, s_abort)) { ok = false; break; }
          tc_fence_after();
          const uint64_t dx = sw128_desc(sbase + x_off + lx * C::kXBytes);
          const uint64_t dl = sw128_desc(sbase + lo_off + ll * kNYBytes);
          const uint32_t d = tmem + lset * kNY;
#pragma unroll
          for (int kk = 0; kk < kXK / 8; ++kk) umma_tf32(d, dx + 2 * kk, dl + 2 * kk, idesc, 1u);
          umma_commit(smem_u32(&lempty[ll]));
          umma_commit(smem_u32(&xempty[lx]));
          if (lc.chain_last()) {
            umma_commit(smem_u32(&tfull[lset]));
            lset ^= 1;
          }
          lc.next(p);
          if (++ll == p.lo_slots) { ll = 0; llph ^= 1; }
          if (++lx == p.x_slots) lx = 0;
          --ahead;
        }
      }
      if (!ok) raise_device_error(p.status, s_abort, kStatusTimeout);
      umma_commit(smem_u32(drain));
      mbar_wait(smem_u32(drain), 0, kXDrainTimeoutNs, nullptr);
    }
    __syncwarp();
  } else if (warp < 6) {
    // ------------------------------------------------------------ converter
    // Thread ct owns 16-byte chunks ct + 128 i (i < 16) of each tile: rows
    // ct / 8 + 16 i.  It reads them as soon as the tile lands (then frees the
    // y stage for its part) and stores their y_lo at the same places of a
    // y_lo slot.
    const int ct = threadIdx.x - 64;
    int ys = 0, ls = 0;
    uint32_t yph = 0, lph = 0;
    bool aborted = false;
    for (int item = blockIdx.x; item < p.n_items && !aborted; item += gridDim.x) {
      const XItem it = decode_xitem(p, item);
      KahanSum nrm[kUnit ? 16 : 1];
      for (int st = it.s0; st < it.s1; ++st) {
        if (!warp_wait(smem_u32(&yfull[ys]), yph, tmo, s_abort)) {
          aborted = true;
          break;
        }
        const float4* yb = reinterpret_cast<const float4*>(smem + ys * kNYBytes);
        float4* lb = reinterpret_cast<float4*>(smem + lo_off + ls * kNYBytes);
        if constexpr (kPad == 32) {
          float4 lo[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float4 v = yb[ct + 128 * i];
            lo[i] = tf32_remainder(v);
            if constexpr (kUnit) nrm[i].add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&yempty[ys]));
          if (!warp_wait(smem_u32(&lempty[ls]), lph ^ 1, tmo, s_abort)) {
            aborted = true;
            break;
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) lb[ct + 128 * i] = lo[i];
        } else {
          // (a smaller register budget per thread: convert straight into the slot)
          if (!warp_wait(smem_u32(&lempty[ls]), lph ^ 1, tmo, s_abort)) {
            aborted = true;
            break;
          }
#pragma unroll 4
          for (int i = 0; i < 16; ++i) {
            const float4 v = yb[ct + 128 * i];
            lb[ct + 128 * i] = tf32_remainder(v);
            if constexpr (kUnit) nrm[i].add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&yempty[ys]));
        }
        if (++ys == p.stages) { ys = 0; yph ^= 1; }
        fence_proxy_async_smem();
        mbar_arrive(smem_u32(&lfull[ls]));
        if (++ls == p.lo_slots) { ls = 0; lph ^= 1; }
      }
      if (aborted) break;
      if constexpr (kUnit) {
        if (it.nt == 0) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            float s = nrm[i].s;                      // the 8 lanes of a row, in a fixed order
            s += __shfl_xor_sync(0xffffffffu, s, 1);
            s += __shfl_xor_sync(0xffffffffu, s, 2);
            s += __shfl_xor_sync(0xffffffffu, s, 4);
            const int q = it.mt * kNY + ct / 8 + 16 * i;
            if ((ct & 7) == 0 && q < p.Q) p.ynorm[static_cast<int64_t>(it.z) * p.Q + q] = s;
          }
        }
      }
    }
    if (aborted) raise_device_error(p.status, s_abort, kStatusTimeout);
  } else {
    // ------------------------------------------------------------ epilogue
    // Warp e = warp - 6 reads lane quarter warp % 4.  kPad = 32: columns
    // 128 (e / 4) .. + 127 of a set with the 16x32bx2 shape, thread t holding
    // row 16 quarter + t % 16 and columns 64 (t / 16) .. + 63 of those;
    // kPad = 64: columns 64 (e / 4) .. + 63 with the 32x32b shape, thread t
    // holding row 32 quarter + t.
    const int e = warp - 6;
    const int quarter = warp & 3;
    const int r_in_q = kPad == 32 ? (lane & 15) : lane;
    const int tcol = kPad == 32 ? 128 * (e >> 2) : 64 * (e >> 2);           // TMEM column of the load
    const int col0 = kPad == 32 ? tcol + 64 * (lane >> 4) : tcol;          // this thread's first column
    const int plane = quarter >> 1;
    const int bl = C::kRowsQ * (quarter & 1) + r_in_q;
    int ab = 0;
    uint32_t aph = 0;
    bool aborted = false;
    for (int item = blockIdx.x; item < p.n_items && !aborted; item += gridDim.x) {
      const XItem it = decode_xitem(p, item);
      float acc[64];                 // the item's chains, added in order (0 + v = v)
#pragma unroll
      for (int j = 0; j < 64; ++j) acc[j] = 0.0f;
      const int n_ch = chain_count(it.s1 - it.s0, p.sub);
      for (int k = 0; k < n_ch; ++k) {
        if (!warp_wait(smem_u32(&tfull[ab]), aph, tmo, s_abort)) {
          raise_device_error(p.status, s_abort, kStatusTimeout);
          aborted = true;
          break;
        }
        tc_fence_after();
        const uint32_t tb = tmem + (static_cast<uint32_t>(32 * quarter) << 16) + ab * kNY + tcol;
#pragma unroll
        for (int blk = 0; blk < 4; ++blk) {
          float v[16];
          if constexpr (kPad == 32)
            tmem_ld16_x2<64>(tb + 16 * blk, v);
          else
            tmem_ld16(tb + 16 * blk, v);
#pragma unroll
          for (int jj = 0; jj < 16; ++jj)
            acc[16 * blk + jj] += v[jj];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&tempty[ab]));
        if (++ab == 2) { ab = 0; aph ^= 1; }
      }
      if (aborted) break;
      const int b = it.nt * kPad + bl;
      const int q0 = it.mt * kNY + col0;
      if (b < p.B && q0 < p.Q) {
        float* dst = p.partial + (static_cast<int64_t>(2 * it.z + plane) * p.B + b) * p.Q + q0;
        if ((p.Q & 3) == 0 && q0 + 64 <= p.Q) {
#pragma unroll
          for (int j = 0; j < 16; ++j)
            *reinterpret_cast<float4*>(dst + 4 * j) =
                make_float4(acc[4 * j], acc[4 * j + 1], acc[4 * j + 2], acc[4 * j + 3]);
        } else {
#pragma unroll
          for (int j = 0; j < 64; ++j)
            if (q0 + j < p.Q) dst[j] = acc[j];
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

// s = sum over planes z (in order) of partial[z, b, q].  Cosine (xnorm
// given): scores[b, q] = s / sqrt(nx_b) / sqrt(ny_q), nx_b the sum over the
// row's chunks (in order) of xnorm[b, c], ny_q the sum over the S slices of
// ynorm[z, q] (0 when either row is zero).  Otherwise scores[b, q] = alpha' s +
// beta scores[b, q] + gamma [b == q], alpha' = alpha * (*alpha_s) when alpha_s
// is given.
__global__ void finish_kernel(const float* __restrict__ partial, int planes, int S, int B, int Q,
                              const float* __restrict__ xnorm, int n_chunks,
                              const float* __restrict__ ynorm,
                              float alpha, const float* __restrict__ alpha_s, float beta,
                              float gamma, float* scores, int64_t ld) {
  griddep_wait();                 // partials, norms and alpha_s come from earlier grids
  const int64_t n = static_cast<int64_t>(B) * Q;
  const float al = alpha_s != nullptr ? alpha * *alpha_s : alpha;
  const int q = blockIdx.x * blockDim.x + threadIdx.x;     // grid: (Q / 256, rows of b)
  if (q >= Q) return;
  for (int b = blockIdx.y; b < B; b += gridDim.y) {
    const int64_t i = static_cast<int64_t>(b) * Q + q;
    float s = 0.0f;
    for (int z = 0; z < planes; ++z) s += partial[z * n + i];
    float* dst = scores + b * ld + q;
    if (xnorm != nullptr) {
      float nx = 0.0f, ny = 0.0f;
      for (int c = 0; c < n_chunks; ++c) nx += xnorm[static_cast<int64_t>(b) * n_chunks + c];
      for (int z = 0; z < S; ++z) ny += ynorm[static_cast<int64_t>(z) * Q + q];
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
  // Batches of up to 64 rows put y on the MMA's N side (one batch tile of 32
  // or 64 rows: M = 64 or 128); larger ones keep y on the M side.
  pl.n_side = b1 <= kMaxPadN;
  if (pl.n_side) {
    pl.n_pad = b1 <= 32 ? 32 : 64;
    pl.y_rows = kNY;
    pl.planes = 2;
  } else {
    pl.n_pad = static_cast<int>(std::min<int64_t>(kMaxPad, (b1 + 15) / 16 * 16));
    pl.y_rows = kXM;
    pl.planes = 1;
  }
  pl.n_ntiles = static_cast<int>((b1 + pl.n_pad - 1) / pl.n_pad);
  pl.n_mtiles = static_cast<int>(std::max<int64_t>(1, (Q + pl.y_rows - 1) / pl.y_rows));
  pl.steps = static_cast<int>(std::max<int64_t>(1, (K + kXK - 1) / kXK));
  pl.sub = kSubSteps;
  pl.n_buf = 2;
  const int ring_budget = kXSmemBudget - 1024 - kXBarBytes;
  int stage_bytes;
  if (pl.n_side) {
    // three y stages, two y_lo slots, and as many x slots as fit (up to 8):
    // the x slots live from a step's load to its y_lo MMAs, a few steps longer
    // than the y stages
    pl.tmem_cols = 2 * kNY;
    pl.stages = kNStages;
    pl.lo_slots = kNLoSlots;
    const int xb = 2 * pl.n_pad * 128;
    pl.x_slots = std::min(kXMaxStages, (ring_budget - (pl.stages + pl.lo_slots) * kNYBytes) / xb);
    stage_bytes = kNYBytes + xb;
  } else {
    pl.tmem_cols = 32;
    while (pl.tmem_cols < pl.n_buf * 2 * pl.n_pad) pl.tmem_cols <<= 1;
    stage_bytes = 2 * kYBytes + 2 * pl.n_pad * 128;
    pl.stages = std::min(kXMaxStages, ring_budget / stage_bytes);
  }
  // K slices: fewest waves of persistent CTAs for the y stream, plus the
  // partial planes each slice adds (written and read back once).
  const int64_t tiles = static_cast<int64_t>(pl.n_mtiles) * pl.n_ntiles;
  double best = -1.0;
  pl.S = 1;
  for (int S = 1; S <= std::min(pl.steps, kMaxSlices); ++S) {
    if (tiles * S > (1ll << 30)) break;
    const int64_t waves = (tiles * S + kPlanCTAs - 1) / kPlanCTAs;
    const int64_t per_item = (pl.steps + S - 1) / S;
    const double cost = static_cast<double>(waves) * (per_item + 2) * stage_bytes +
                        8.0 * pl.planes * S * static_cast<double>(b1) * static_cast<double>(Q) /
                            kPlanCTAs;
    if (best < 0.0 || cost < best) {
      best = cost;
      pl.S = S;
    }
  }
  // N side: y_hi steps ahead of y_lo, at most the shortest chain + 1 (items
  // have floor or ceil of steps / S steps, cut into near-equal chains) and
  // short of the ring
  int min_chain = pl.sub;
  for (int L : {pl.steps / pl.S, (pl.steps + pl.S - 1) / pl.S}) {
    const int n_ch = (L + pl.sub - 1) / pl.sub;
    min_chain = std::min(min_chain, L / n_ch);
  }
  pl.lookahead = std::max(1, std::min(kNLookahead, min_chain + 1));
  size_t off = 0;
  pl.n_chunks = static_cast<int>(std::max<int64_t>(1, (K + kSplitChunk - 1) / kSplitChunk));
  pl.xnorm_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(b1) * pl.n_chunks);
  pl.ynorm_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(pl.S) * std::max<int64_t>(Q, 1));
  pl.partial_off = off;
  off += round_up256(sizeof(float) * static_cast<size_t>(pl.planes) * pl.S * b1 *
                     std::max<int64_t>(Q, 1));
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
  CUtensorMap tm_y, tm_xh, tm_xl;
  if (encode_tmap_2d(&tm_y, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.y, a.K, a.Q, a.ldy * 4, kXK,
                     pl.y_rows) != CUDA_SUCCESS ||
      encode_tmap_2d(&tm_xh, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.ws + pl.xh_off, a.K, a.B,
                     static_cast<int64_t>(a.K) * 4, kXK, pl.n_pad) != CUDA_SUCCESS ||
      encode_tmap_2d(&tm_xl, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, a.ws + pl.xl_off, a.K, a.B,
                     static_cast<int64_t>(a.K) * 4, kXK, pl.n_pad) != CUDA_SUCCESS)
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
  p.lookahead = pl.lookahead;
  p.lo_slots = pl.lo_slots;
  p.x_slots = pl.x_slots;
  p.unit = a.unit;
  p.partial = reinterpret_cast<float*>(a.ws + pl.partial_off);
  p.ynorm = reinterpret_cast<float*>(a.ws + pl.ynorm_off);
  p.status = a.status;
  p.timeout_ns = a.timeout_ns;
  const size_t rings =
      pl.n_side ? nside_ring_bytes(pl.n_pad, pl.stages, pl.lo_slots, pl.x_slots)
                : static_cast<size_t>(pl.stages) * (2 * kYBytes + 2 * pl.n_pad * 128);
  const size_t smem = 1024 + rings + kXBarBytes;
  const int grid = std::max(1, std::min(sms > 0 ? sms : 1, p.n_items));
  static PerDeviceOnce attr_n[4], attr_m;
  if (!pl.n_side)
    e = launch_product(xgemm_kernel, attr_m, kXThreads, grid, smem, s, tm_y, tm_xh, tm_xl, p);
  else if (pl.n_pad == 32)
    e = a.unit ? launch_product(xgemm_n_kernel<32, true>, attr_n[0], NSide<32>::kThreads, grid,
                                smem, s, tm_y, tm_xh, tm_xl, p)
               : launch_product(xgemm_n_kernel<32, false>, attr_n[1], NSide<32>::kThreads, grid,
                                smem, s, tm_y, tm_xh, tm_xl, p);
  else
    e = a.unit ? launch_product(xgemm_n_kernel<64, true>, attr_n[2], NSide<64>::kThreads, grid,
                                smem, s, tm_y, tm_xh, tm_xl, p)
               : launch_product(xgemm_n_kernel<64, false>, attr_n[3], NSide<64>::kThreads, grid,
                                smem, s, tm_y, tm_xh, tm_xl, p);
  if (e != cudaSuccess) return e;

  const dim3 fgrid((a.Q + 255) / 256, std::min(a.B, 65535));
  const float* xn = a.unit ? xnorm : nullptr;
  return launch_dependent(finish_kernel, fgrid, dim3(256), 0, s, p.partial, pl.planes * pl.S,
                          pl.S, a.B, a.Q, xn, pl.n_chunks, p.ynorm, a.alpha, a.alpha_s, a.beta,
                          a.gamma, a.scores, a.ld_scores);
}

}  // namespace bergson
