// Gradient-store rows and query normalisation (Bergson Sec. 3.1: unit
// normalisation and the gradient store; grad-cosine = identity + unit norm).
//
// One CTA per row: the squared norm is accumulated from 16-byte vector loads
// (fp64 partial sums, so a 10^5-long row keeps fp32-level accuracy), reduced
// with warp shuffles, and the row is written back as fp16 (round to nearest
// even) with 16-byte vector stores.

#include "internal.h"

namespace bergson {

namespace {

constexpr int kRowThreads = 256;

__device__ __forceinline__ double block_sum(double v, double* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < (blockDim.x >> 5) ? red[lane] : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) red[0] = v;
  }
  __syncthreads();
  return red[0];
}

__device__ __forceinline__ uint4 pack8(float4 a, float4 b, float s) {
  const __half2 h0 = __floats2half2_rn(a.x * s, a.y * s);
  const __half2 h1 = __floats2half2_rn(a.z * s, a.w * s);
  const __half2 h2 = __floats2half2_rn(b.x * s, b.y * s);
  const __half2 h3 = __floats2half2_rn(b.z * s, b.w * s);
  uint4 u;
  u.x = *reinterpret_cast<const uint32_t*>(&h0);
  u.y = *reinterpret_cast<const uint32_t*>(&h1);
  u.z = *reinterpret_cast<const uint32_t*>(&h2);
  u.w = *reinterpret_cast<const uint32_t*>(&h3);
  return u;
}

// y[b, 0:K] = fp16(x[b, 0:K] * scale_b), scale_b = 1/||x_b|| (unit) or 1.
__global__ void __launch_bounds__(kRowThreads) normalize_rows_kernel(
    const float* __restrict__ x, int K, int64_t ldx, int unit, __half* __restrict__ y,
    int64_t ldy, float* __restrict__ norms) {
  __shared__ double red[kRowThreads / 32];
  const int64_t b = blockIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + b * ldx);
  double ss = 0.0;
  for (int i = threadIdx.x; i < K / 4; i += kRowThreads) {
    const float4 v = xr[i];
    ss += static_cast<double>(v.x) * v.x + static_cast<double>(v.y) * v.y +
          static_cast<double>(v.z) * v.z + static_cast<double>(v.w) * v.w;
  }
  const double tot = block_sum(ss, red);
  const float nrm = static_cast<float>(sqrt(tot));
  const float scale = unit ? (tot > 0.0 ? static_cast<float>(1.0 / sqrt(tot)) : 0.0f) : 1.0f;
  uint4* yr = reinterpret_cast<uint4*>(y + b * ldy);
  for (int i = threadIdx.x; i < K / 8; i += kRowThreads) yr[i] = pack8(xr[2 * i], xr[2 * i + 1], scale);
  if (norms != nullptr && threadIdx.x == 0) norms[b] = nrm;
}

// Queries may have any row stride; they are read with scalar loads.
__global__ void __launch_bounds__(kRowThreads) normalize_queries_kernel(
    const float* __restrict__ q, int K, int64_t ldq, __half* __restrict__ qh) {
  __shared__ double red[kRowThreads / 32];
  const int64_t r = blockIdx.x;
  const float* qr = q + r * ldq;
  double ss = 0.0;
  for (int i = threadIdx.x; i < K; i += kRowThreads) ss += static_cast<double>(qr[i]) * qr[i];
  const double tot = block_sum(ss, red);
  const float scale = tot > 0.0 ? static_cast<float>(1.0 / sqrt(tot)) : 0.0f;
  __half* out = qh + r * K;
  for (int i = threadIdx.x; i < K; i += kRowThreads) out[i] = __float2half_rn(qr[i] * scale);
}

}  // namespace

cudaError_t launch_build_store(const float* proj, int B, int K, int64_t ld_proj, int unit,
                               __half* store, int64_t ld_store, float* norms, cudaStream_t s) {
  if (B == 0) return cudaSuccess;
  normalize_rows_kernel<<<B, kRowThreads, 0, s>>>(proj, K, ld_proj, unit, store, ld_store, norms);
  return cudaGetLastError();
}

cudaError_t launch_normalize_queries(const float* q, int Q, int K, int64_t ld_q, __half* qh,
                                     cudaStream_t s) {
  if (Q == 0) return cudaSuccess;
  normalize_queries_kernel<<<Q, kRowThreads, 0, s>>>(q, K, ld_q, qh);
  return cudaGetLastError();
}

}  // namespace bergson
