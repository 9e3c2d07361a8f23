// On-the-fly scores (Bergson Sec. 3.1, "bergson score"): projected training
// gradients scored directly against fixed query gradients, with no gradient
// store in between.  Table 3's grad-cosine (unit-normalised rows and queries)
// and grad-dot (raw inner products) are both served:
//   scores[b, q] = <x_b, y_q> * s_b * t_q,  s = 1/||x||, t = 1/||y|| (cosine) or 1.
//
// The inner products are a small fp32 GEMM [B x K] x [K x Q] (for a batch of
// 32 examples and 1024 queries at K = 12288, 0.8 GFLOP: ~0.5% of the batch's
// projection time), computed with CUDA-core FFMA in fp32 for full accuracy.
// Split-K gives enough CTAs for a 32-row batch; the partial sums are added in
// a fixed order, so the result is deterministic.

#include "internal.h"

namespace bergson {

namespace {

constexpr int kBM = 32;        // rows (examples) per CTA tile
constexpr int kBN = 128;       // queries per CTA tile
constexpr int kBK = 32;        // K per shared-memory step
constexpr int kThreads = 128;  // thread tile: 4 rows x 8 queries
constexpr int kRowThreads = 256;

// scale[i] = 1/||row_i|| (unit, 0 for a zero row) or 1.  One CTA per row,
// 16-byte loads, compensated fp32 sums per thread (fp64 is slow on this part).
__global__ void __launch_bounds__(kRowThreads) row_scales_kernel(
    const float* __restrict__ x, int K, int64_t ld, int unit, float* __restrict__ scale) {
  __shared__ float red[kRowThreads / 32];
  const float4* xr = reinterpret_cast<const float4*>(x + blockIdx.x * ld);
  float s = 0.0f, comp = 0.0f;
  for (int i = threadIdx.x; i < K / 4; i += kRowThreads) {
    const float4 v = xr[i];
    const float y = (v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w) - comp;
    const float t = s + y;
    comp = (t - s) - y;
    s = t;
  }
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

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  const int n = valid ? 16 : 0;                      // 0 source bytes -> zero fill
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(gmem), "r"(n)
               : "memory");
}

// partial[z, b, q] = sum over k in slice z of x[b, k] * y[q, k].
// Two shared-memory stages filled with cp.async; thread (tx, ty) owns rows
// 4ty..4ty+3 and queries tx + 16j (j < 8), which keeps the 16-byte shared
// loads of one warp on distinct banks.
__global__ void __launch_bounds__(kThreads) dot_partials_kernel(
    const float* __restrict__ x, int B, int64_t ldx, const float* __restrict__ y, int Q,
    int64_t ldy, int K, int kslice, float* __restrict__ partial) {
  __shared__ __align__(16) float xs[2][kBM][kBK + 4];
  __shared__ __align__(16) float ys[2][kBN][kBK + 4];
  const int tid = threadIdx.x;
  const int tx = tid % 16;
  const int ty = tid / 16;
  const int q0 = blockIdx.x * kBN;
  const int b0 = blockIdx.y * kBM;
  const int k_begin = blockIdx.z * kslice;
  const int k_end = min(K, k_begin + kslice);
  const int nsteps = (k_end - k_begin + kBK - 1) / kBK;

  auto load = [&](int st, int k0) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {   // x: 32 rows x 8 chunks of 16 B
      const int idx = tid + h * kThreads;
      const int r = idx / 8, c = (idx % 8) * 4;
      const bool ok = b0 + r < B && k0 + c < k_end;
      cp_async16(&xs[st][r][c], ok ? x + (b0 + r) * ldx + k0 + c : x, ok);
    }
#pragma unroll
    for (int h = 0; h < 8; ++h) {   // y: 128 rows x 8 chunks of 16 B
      const int idx = tid + h * kThreads;
      const int r = idx / 8, c = (idx % 8) * 4;
      const bool ok = q0 + r < Q && k0 + c < k_end;
      cp_async16(&ys[st][r][c], ok ? y + (q0 + r) * ldy + k0 + c : y, ok);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  float acc[4][8] = {};
  if (nsteps > 0) load(0, k_begin);
  for (int step = 0; step < nsteps; ++step) {
    const int st = step & 1;
    if (step + 1 < nsteps) {
      load(st ^ 1, k_begin + (step + 1) * kBK);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kBK; kk += 4) {
      float4 a[4], c[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = *reinterpret_cast<const float4*>(&xs[st][4 * ty + i][kk]);
#pragma unroll
      for (int j = 0; j < 8; ++j) c[j] = *reinterpret_cast<const float4*>(&ys[st][tx + 16 * j][kk]);
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          acc[i][j] = fmaf(a[i].x, c[j].x, acc[i][j]);
          acc[i][j] = fmaf(a[i].y, c[j].y, acc[i][j]);
          acc[i][j] = fmaf(a[i].z, c[j].z, acc[i][j]);
          acc[i][j] = fmaf(a[i].w, c[j].w, acc[i][j]);
        }
    }
    __syncthreads();
  }
  float* dst = partial + static_cast<int64_t>(blockIdx.z) * B * Q;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int b = b0 + 4 * ty + i;
    if (b >= B) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int q = q0 + tx + 16 * j;
      if (q < Q) dst[static_cast<int64_t>(b) * Q + q] = acc[i][j];
    }
  }
}

// scores[b, q] = (sum over slices, in order) * sx[b] * sy[q]
__global__ void finish_kernel(const float* __restrict__ partial, int S, int B, int Q,
                              const float* __restrict__ sx, const float* __restrict__ sy,
                              float* __restrict__ scores, int64_t ld) {
  const int64_t n = static_cast<int64_t>(B) * Q;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float s = 0.0f;
    for (int z = 0; z < S; ++z) s += partial[z * n + i];
    const int b = static_cast<int>(i / Q), q = static_cast<int>(i % Q);
    scores[b * ld + q] = sx != nullptr ? s * sx[b] * sy[q] : s;
  }
}

}  // namespace

cudaError_t launch_row_scales(const float* x, int n, int K, int64_t ld, int unit, float* scale,
                              cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  row_scales_kernel<<<n, kRowThreads, 0, s>>>(x, K, ld, unit, scale);
  return cudaGetLastError();
}

int onthefly_splits(int64_t B, int64_t Q, int64_t K) {
  const int64_t tiles = ((Q + kBN - 1) / kBN) * ((B + kBM - 1) / kBM);
  if (tiles == 0) return 1;                       // empty problem: nothing to split
  int64_t s = (kOnTheFlyTargetCTAs + tiles - 1) / tiles;
  const int64_t max_s = (K + kBK - 1) / kBK;
  if (s > max_s) s = max_s;
  if (s < 1) s = 1;
  const int64_t slice = ((K + s - 1) / s + kBK - 1) / kBK * kBK;
  return static_cast<int>((K + slice - 1) / slice);
}

cudaError_t launch_onthefly(const float* x, int B, int64_t ldx, const float* y, int Q,
                            int64_t ldy, int K, int unit, float* sx, float* sy, float* partial,
                            float* scores, int64_t ld_scores, cudaStream_t s) {
  if (B == 0 || Q == 0) return cudaSuccess;
  const int S = onthefly_splits(B, Q, K);
  const int slice = ((K + S - 1) / S + kBK - 1) / kBK * kBK;
  if (unit) {                  // plain products need no norms
    row_scales_kernel<<<B, kRowThreads, 0, s>>>(x, K, ldx, unit, sx);
    row_scales_kernel<<<Q, kRowThreads, 0, s>>>(y, K, ldy, unit, sy);
  } else {
    sx = sy = nullptr;
  }
  dim3 grid((Q + kBN - 1) / kBN, (B + kBM - 1) / kBM, S);
  dot_partials_kernel<<<grid, kThreads, 0, s>>>(x, B, ldx, y, Q, ldy, K, slice, partial);
  const int64_t n = static_cast<int64_t>(B) * Q;
  const int64_t blocks = (n + 255) / 256;
  finish_kernel<<<static_cast<unsigned>(blocks < 4096 ? blocks : 4096), 256, 0, s>>>(
      partial, S, B, Q, sx, sy, scores, ld_scores);
  return cudaGetLastError();
}

}  // namespace bergson
