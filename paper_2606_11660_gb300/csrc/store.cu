// Gradient-store rows and query normalisation (Bergson Sec. 3.1: unit
// normalisation and the gradient store; grad-cosine = identity + unit norm).
//
// One CTA per row: the squared norm is accumulated from 16-byte vector loads
// with compensated (Kahan) fp32 sums per thread -- fp64 arithmetic is slow on
// this part and unnecessary at this accuracy -- reduced with warp shuffles,
// and the row is written back as fp16 (round to nearest even) with 16-byte
// vector stores.

#include "internal.h"
#include "ptx.cuh"

namespace bergson {

namespace {

constexpr int kRowThreads = 256;

// Kahan-compensated running sum.
struct KahanSum {
  float s = 0.0f, c = 0.0f;
  __device__ __forceinline__ void add(float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
  }
};

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < (blockDim.x >> 5) ? red[lane] : 0.0f;
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
  __shared__ float red[kRowThreads / 32];
  griddep_wait();                // the rows are usually the preceding reduction's output
  const int64_t b = blockIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + b * ldx);
  KahanSum ss;
  for (int i = threadIdx.x; i < K / 4; i += kRowThreads) {
    const float4 v = xr[i];
    ss.add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
  }
  const float tot = block_sum(ss.s, red);
  const float nrm = sqrtf(tot);
  const float scale = unit ? (tot > 0.0f ? 1.0f / nrm : 0.0f) : 1.0f;
  uint4* yr = reinterpret_cast<uint4*>(y + b * ldy);
  for (int i = threadIdx.x; i < K / 8; i += kRowThreads) yr[i] = pack8(xr[2 * i], xr[2 * i + 1], scale);
  if (norms != nullptr && threadIdx.x == 0) norms[b] = nrm;
}

// Per-module unit normalisation: CTA (b, j) writes
//   y[b, o_j:o_{j+1}] = fp16(x[b, o_j:o_{j+1}] / ||x[b, o_j:o_{j+1}]||)
// (a zero block stays zero) and norms[b * n_blocks + j].  Offsets are
// multiples of 8, so every block starts on a 16-byte boundary of both rows.
__global__ void __launch_bounds__(kRowThreads) normalize_blocks_kernel(
    const float* __restrict__ x, int64_t ldx, const __grid_constant__ StoreBlocks bo,
    __half* __restrict__ y, int64_t ldy, float* __restrict__ norms) {
  __shared__ float red[kRowThreads / 32];
  griddep_wait();                // the rows are usually the preceding reduction's output
  const int64_t b = blockIdx.x;
  const int j = blockIdx.y;
  const int c0 = bo.offset[j], c1 = bo.offset[j + 1];
  const float4* xr = reinterpret_cast<const float4*>(x + b * ldx + c0);
  KahanSum ss;
  for (int i = threadIdx.x; i < (c1 - c0) / 4; i += kRowThreads) {
    const float4 v = xr[i];
    ss.add(v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w);
  }
  const float tot = block_sum(ss.s, red);
  const float scale = tot > 0.0f ? 1.0f / sqrtf(tot) : 0.0f;
  uint4* yr = reinterpret_cast<uint4*>(y + b * ldy + c0);
  for (int i = threadIdx.x; i < (c1 - c0) / 8; i += kRowThreads)
    yr[i] = pack8(xr[2 * i], xr[2 * i + 1], scale);
  if (norms != nullptr && threadIdx.x == 0) norms[b * bo.n + j] = sqrtf(tot);
}

// Queries may have any row stride; they are read with scalar loads.  With
// `negate` the row is written as -q / ||q|| (exactly the negation of the
// unit row: fp16 rounding is symmetric), which turns a top-k search into a
// bottom-k one.
__global__ void __launch_bounds__(kRowThreads) normalize_queries_kernel(
    const float* __restrict__ q, int K, int64_t ldq, int negate, __half* __restrict__ qh) {
  __shared__ float red[kRowThreads / 32];
  const int64_t r = blockIdx.x;
  const float* qr = q + r * ldq;
  KahanSum ss;
  for (int i = threadIdx.x; i < K; i += kRowThreads) ss.add(qr[i] * qr[i]);
  const float tot = block_sum(ss.s, red);
  const float inv = tot > 0.0f ? 1.0f / sqrtf(tot) : 0.0f;
  const float scale = negate ? -inv : inv;
  __half* out = qh + r * K;
  for (int i = threadIdx.x; i < K; i += kRowThreads) out[i] = __float2half_rn(qr[i] * scale);
}

}  // namespace

cudaError_t launch_build_store(const float* proj, int B, int K, int64_t ld_proj, int unit,
                               __half* store, int64_t ld_store, float* norms, cudaStream_t s) {
  if (B == 0) return cudaSuccess;
  return launch_dependent(normalize_rows_kernel, dim3(B), dim3(kRowThreads), 0, s, proj, K,
                          ld_proj, unit, store, ld_store, norms);
}

cudaError_t launch_build_store_blocks(const float* proj, int B, int64_t ld_proj,
                                      const StoreBlocks& blocks, __half* store, int64_t ld_store,
                                      float* norms, cudaStream_t s) {
  if (B == 0) return cudaSuccess;
  return launch_dependent(normalize_blocks_kernel, dim3(B, blocks.n), dim3(kRowThreads), 0, s,
                          proj, ld_proj, blocks, store, ld_store, norms);
}

cudaError_t launch_normalize_queries(const float* q, int Q, int K, int64_t ld_q, bool negate,
                                     __half* qh, cudaStream_t s) {
  if (Q == 0) return cudaSuccess;
  normalize_queries_kernel<<<Q, kRowThreads, 0, s>>>(q, K, ld_q, negate ? 1 : 0, qh);
  return cudaGetLastError();
}

}  // namespace bergson
