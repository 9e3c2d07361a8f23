// Query aggregation (Bergson Sec. 3.2: a query formed as the mean or sum of
// the gradients of several generations or items, as LESS builds evaluation
// queries; Fig. 2 "unit_normalize: true, aggregation: mean"):
//   out[g] = agg over r in [offsets[g], offsets[g+1]) of  rows[r] * scale[r]
// with scale = 1/||rows[r]|| (normalise each) or 1, agg = sum or mean.
// One CTA per (group, 1024-column slice); each thread owns 4 columns and
// adds the group's rows in order (deterministic), reading rows once.

#include "internal.h"

namespace bergson {

namespace {

constexpr int kThreads = 256;
constexpr int kCols = 4 * kThreads;

__global__ void __launch_bounds__(kThreads) aggregate_kernel(
    const float* __restrict__ rows, int64_t n, int K, int64_t ld,
    const int64_t* __restrict__ offsets, int mode, const float* __restrict__ scale,
    float* __restrict__ out, int64_t ld_out) {
  const int g = blockIdx.x;
  const int c = blockIdx.y * kCols + 4 * threadIdx.x;
  if (c >= K) return;
  // Offsets are clamped to [0, n]; a decreasing pair is an empty group.
  int64_t a = offsets[g], b = offsets[g + 1];
  a = a < 0 ? 0 : (a > n ? n : a);
  b = b < a ? a : (b > n ? n : b);
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int64_t r = a; r < b; ++r) {
    const float4 v = *reinterpret_cast<const float4*>(rows + r * ld + c);
    const float w = scale != nullptr ? scale[r] : 1.0f;
    acc.x = fmaf(v.x, w, acc.x);
    acc.y = fmaf(v.y, w, acc.y);
    acc.z = fmaf(v.z, w, acc.z);
    acc.w = fmaf(v.w, w, acc.w);
  }
  if (mode == 1 && b > a) {
    const float inv = 1.0f / static_cast<float>(b - a);
    acc.x *= inv; acc.y *= inv; acc.z *= inv; acc.w *= inv;
  }
  *reinterpret_cast<float4*>(out + static_cast<int64_t>(g) * ld_out + c) = acc;
}

}  // namespace

cudaError_t launch_aggregate(const float* rows, int64_t n, int K, int64_t ld,
                             const int64_t* offsets, int G, int mode, const float* scale,
                             float* out, int64_t ld_out, cudaStream_t s) {
  if (G == 0) return cudaSuccess;
  dim3 grid(G, (K + kCols - 1) / kCols);
  aggregate_kernel<<<grid, kThreads, 0, s>>>(rows, n, K, ld, offsets, mode, scale, out, ld_out);
  return cudaGetLastError();
}

}  // namespace bergson
