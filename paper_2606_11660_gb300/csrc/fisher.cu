// TrackStar's empirical-Fisher preconditioner (Bergson Sec. 3.1: the empirical
// Fisher used by TrackStar, stacked with optimizer normalisation and
// down-projection; Fig. 2: Fisher fitting and mixing before index building).
//
//   fit:    R = (1/n) X^T X over n projected gradient rows (K x K)
//   mix:    R = lam R1 + (1 - lam) R2 + damping * (tr(R)/K) * I
//   power:  M = R^-1/2 (or R^-1) by the coupled Newton-Schulz iteration
//           Y0 = R/c, Z0 = I, T = (3I - Z Y)/2, Y <- Y T, Z <- T Z, which
//           drives Y -> (R/c)^1/2 and Z -> (R/c)^-1/2 using only matrix
//           products (c = ||R||_F puts every eigenvalue of R/c in (0, 1]).
//   apply:  x' = M x for each row (bergson_precondition_rows, same GEMM as
//           the on-the-fly scores).
//
// All products are fp32 "NT" GEMMs C = alpha A B^T + beta C + gamma I, with A
// and B row-major and the reduction index contiguous: a 128 x 128 CTA tile,
// 8 x 8 outputs per thread over strided rows/columns (conflict-free 16-byte
// shared loads) and cp.async double buffering.  Products of the iteration
// are symmetric in exact arithmetic, so B^T = B there; each update is
// re-symmetrised so that rounding cannot build up an antisymmetric part.

#include "internal.h"

namespace bergson {

namespace {

constexpr int kTile = 128;
constexpr int kBK = 16;
constexpr int kThreads = 256;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(d), "l"(gmem),
               "r"(valid ? 16 : 0)
               : "memory");
}

// C[m, n] = alpha * sum_k A[m, k] B[n, k] + beta * C[m, n] + (m == n ? gamma : 0),
// alpha and gamma optionally scaled by a device scalar: alpha * (*alpha_s), gamma * (*gamma_s).
__global__ void __launch_bounds__(kThreads) gemm_nt_kernel(
    const float* __restrict__ A, int64_t lda, const float* __restrict__ B, int64_t ldb,
    float* C, int64_t ldc, int M, int N, int K, float alpha, float beta, float gamma,
    const float* __restrict__ alpha_s) {
  __shared__ __align__(16) float as[2][kTile][kBK + 4];
  __shared__ __align__(16) float bs[2][kTile][kBK + 4];
  const int tid = threadIdx.x;
  const int tx = tid % 16;
  const int ty = tid / 16;
  const int m0 = blockIdx.y * kTile;
  const int n0 = blockIdx.x * kTile;
  const int nsteps = (K + kBK - 1) / kBK;

  auto load = [&](int st, int k0) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {   // 128 rows x 4 chunks of 16 B, for A and for B
      const int idx = tid + h * kThreads;
      const int r = idx / 4, c = (idx % 4) * 4;
      const bool oka = m0 + r < M && k0 + c < K;
      cp_async16(&as[st][r][c], oka ? A + (m0 + r) * lda + k0 + c : A, oka);
      const bool okb = n0 + r < N && k0 + c < K;
      cp_async16(&bs[st][r][c], okb ? B + (n0 + r) * ldb + k0 + c : B, okb);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };

  float acc[8][8] = {};
  if (nsteps > 0) load(0, 0);
  for (int step = 0; step < nsteps; ++step) {
    const int st = step & 1;
    if (step + 1 < nsteps) {
      load(st ^ 1, (step + 1) * kBK);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kBK; kk += 4) {
      float4 a[8], b[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) a[i] = *reinterpret_cast<const float4*>(&as[st][ty + 16 * i][kk]);
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = *reinterpret_cast<const float4*>(&bs[st][tx + 16 * j][kk]);
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          acc[i][j] = fmaf(a[i].x, b[j].x, acc[i][j]);
          acc[i][j] = fmaf(a[i].y, b[j].y, acc[i][j]);
          acc[i][j] = fmaf(a[i].z, b[j].z, acc[i][j]);
          acc[i][j] = fmaf(a[i].w, b[j].w, acc[i][j]);
        }
    }
    __syncthreads();
  }
  const float al = alpha_s != nullptr ? alpha * *alpha_s : alpha;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = m0 + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n >= N) continue;
      float v = al * acc[i][j];
      if (beta != 0.0f) v = fmaf(beta, C[m * ldc + n], v);
      if (m == n) v += gamma;
      C[m * ldc + n] = v;
    }
  }
}

// xt[k, i] = x[i, k] for i < n, zero for n <= i < n_pad.
__global__ void transpose_kernel(const float* __restrict__ x, int n, int K, int64_t ldx,
                                 float* __restrict__ xt, int n_pad) {
  __shared__ float tile[32][33];
  const int i0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
  for (int r = threadIdx.y; r < 32; r += 8) {
    const int i = i0 + r, k = k0 + threadIdx.x;
    tile[r][threadIdx.x] = (i < n && k < K) ? x[i * ldx + k] : 0.0f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += 8) {
    const int k = k0 + r, i = i0 + threadIdx.x;
    if (k < K && i < n_pad) xt[k * static_cast<int64_t>(n_pad) + i] = tile[threadIdx.x][r];
  }
}

// scal[0] = sum_i (lam * R1[i,i] + (1 - lam) * R2[i,i])  (single CTA)
__global__ void mixed_trace_kernel(const float* __restrict__ r1, const float* __restrict__ r2,
                                   int64_t ld, int K, float lam, float* __restrict__ scal) {
  __shared__ float red[32];
  float s = 0.0f;
  for (int i = threadIdx.x; i < K; i += blockDim.x) {
    const float a = r1[i * ld + i];
    s += r2 != nullptr ? lam * a + (1.0f - lam) * r2[i * ld + i] : a;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += red[w];
    scal[0] = t;
  }
}

// out = lam R1 + (1 - lam) R2 + damping * trace / K * I   (R2 may be null: out = R1 + ...)
__global__ void mix_kernel(const float* __restrict__ r1, const float* __restrict__ r2, int64_t ld,
                           int K, float lam, float damping, const float* __restrict__ scal,
                           float* __restrict__ out, int64_t ldo) {
  const float d = damping * scal[0] / static_cast<float>(K);
  const int64_t n = static_cast<int64_t>(K) * K;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(e / K), j = static_cast<int>(e % K);
    float v = r1[i * ld + j];
    if (r2 != nullptr) v = lam * v + (1.0f - lam) * r2[i * ld + j];
    if (i == j) v += d;
    out[i * ldo + j] = v;
  }
}

constexpr int kFrobBlocks = 512;

// part[blockIdx] = compensated sum of squares over a grid-stride slice of R.
__global__ void frob_partial_kernel(const float* __restrict__ r, int64_t ld, int K,
                                    float* __restrict__ part) {
  __shared__ float red[32];
  float s = 0.0f, comp = 0.0f;
  const int64_t n = static_cast<int64_t>(K) * K;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const float x = r[(e / K) * ld + e % K];
    const float y = x * x - comp;
    const float t = s + y;
    comp = (t - s) - y;
    s = t;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += red[w];
    part[blockIdx.x] = t;
  }
}

// scal[1] = ||R||_F, scal[2] = 1/c, scal[3] = 1/sqrt(c), scal[4] = 1/c  (fixed-order sum)
__global__ void frob_final_kernel(const float* __restrict__ part, int n_part,
                                  float* __restrict__ scal) {
  if (threadIdx.x != 0) return;
  float t = 0.0f, comp = 0.0f;
  for (int i = 0; i < n_part; ++i) {
    const float y = part[i] - comp;
    const float u = t + y;
    comp = (u - t) - y;
    t = u;
  }
  const float c = sqrtf(t);
  scal[1] = c;
  scal[2] = 1.0f / c;
  scal[3] = 1.0f / sqrtf(c);
  scal[4] = 1.0f / c;
}

// y = r * scal[2] (R / c); z = I
__global__ void ns_init_kernel(const float* __restrict__ r, int64_t ld, int K,
                               const float* __restrict__ scal, float* __restrict__ y,
                               float* __restrict__ z) {
  const float inv_c = scal[2];
  const int64_t n = static_cast<int64_t>(K) * K;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(e / K), j = static_cast<int>(e % K);
    y[e] = r[i * ld + j] * inv_c;
    z[e] = i == j ? 1.0f : 0.0f;
  }
}

// x <- (x + x^T) / 2 in place (one thread per pair i < j).  The iterates are
// symmetric in exact arithmetic, but the products use B^T = B, which turns the
// rounding's antisymmetric part into a growing error unless it is removed.
__global__ void symmetrize_kernel(float* __restrict__ x, int K) {
  const int64_t n = static_cast<int64_t>(K) * K;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(e / K), j = static_cast<int>(e % K);
    if (i < j) {
      const float v = 0.5f * (x[e] + x[static_cast<int64_t>(j) * K + i]);
      x[e] = v;
      x[static_cast<int64_t>(j) * K + i] = v;
    }
  }
}

// dst[i, j] = src[i * K + j] * (*scale)
__global__ void scale_copy_kernel(const float* __restrict__ src, int K,
                                  const float* __restrict__ scale, float* __restrict__ dst,
                                  int64_t ldd) {
  const float sc = *scale;
  const int64_t n = static_cast<int64_t>(K) * K;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x)
    dst[(e / K) * ldd + e % K] = src[e] * sc;
}

cudaError_t gemm_nt(const float* A, int64_t lda, const float* B, int64_t ldb, float* C,
                    int64_t ldc, int M, int N, int K, float alpha, float beta, float gamma,
                    const float* alpha_s, cudaStream_t s) {
  dim3 grid((N + kTile - 1) / kTile, (M + kTile - 1) / kTile);
  gemm_nt_kernel<<<grid, kThreads, 0, s>>>(A, lda, B, ldb, C, ldc, M, N, K, alpha, beta, gamma,
                                           alpha_s);
  return cudaGetLastError();
}

unsigned elementwise_blocks(int64_t n) {
  const int64_t b = (n + 255) / 256;
  return static_cast<unsigned>(b < 8192 ? b : 8192);
}

}  // namespace

size_t fisher_fit_workspace(int64_t n, int64_t K) {
  const int64_t n_pad = (n + 3) / 4 * 4;
  return static_cast<size_t>(K) * n_pad * sizeof(float);
}

cudaError_t launch_fisher_fit(const float* x, int n, int K, int64_t ldx, float* r, int64_t ldr,
                              float* ws, cudaStream_t s) {
  const int n_pad = (n + 3) / 4 * 4;
  dim3 grid((n_pad + 31) / 32, (K + 31) / 32);
  transpose_kernel<<<grid, dim3(32, 8), 0, s>>>(x, n, K, ldx, ws, n_pad);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return gemm_nt(ws, n_pad, ws, n_pad, r, ldr, K, K, n_pad, 1.0f / static_cast<float>(n), 0.0f,
                 0.0f, nullptr, s);
}

size_t fisher_power_workspace(int64_t K) {
  return (4 * static_cast<size_t>(K) * K + 64 + kFrobBlocks) * sizeof(float);
}

cudaError_t launch_fisher_power(const float* r1, const float* r2, int K, int64_t ldr, float lam,
                                float damping, int inverse, int iterations, float* m, int64_t ldm,
                                float* ws, cudaStream_t s) {
  const int64_t kk = static_cast<int64_t>(K) * K;
  float* a = ws;            // mixed, damped R
  float* y = a + kk;
  float* z = y + kk;
  float* t = z + kk;
  float* scal = t + kk;     // trace, ||R||_F, 1/c, 1/sqrt(c), 1/c; [64, 64 + 512): partial sums
  mixed_trace_kernel<<<1, 1024, 0, s>>>(r1, r2, ldr, K, lam, scal);
  mix_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(r1, r2, ldr, K, lam, damping, scal, a, K);
  frob_partial_kernel<<<kFrobBlocks, 256, 0, s>>>(a, K, K, scal + 64);
  frob_final_kernel<<<1, 32, 0, s>>>(scal + 64, kFrobBlocks, scal);
  ns_init_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(a, K, K, scal, y, z);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  for (int it = 0; it < iterations; ++it) {
    // T = 1.5 I - 0.5 Z Y;  Y <- Y T;  Z <- T Z
    if ((e = gemm_nt(z, K, y, K, t, K, K, K, K, -0.5f, 0.0f, 1.5f, nullptr, s)) != cudaSuccess)
      return e;
    if ((e = gemm_nt(y, K, t, K, a, K, K, K, K, 1.0f, 0.0f, 0.0f, nullptr, s)) != cudaSuccess)
      return e;
    float* swap = y;      // new Y is in `a`; the old Y buffer becomes scratch
    y = a;
    a = swap;
    if ((e = gemm_nt(t, K, z, K, a, K, K, K, K, 1.0f, 0.0f, 0.0f, nullptr, s)) != cudaSuccess)
      return e;
    swap = z;
    z = a;
    a = swap;
    symmetrize_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(y, K);
    symmetrize_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(z, K);
  }
  // Z ~ (R/c)^-1/2:  R^-1/2 = Z / sqrt(c);  R^-1 = Z Z / c
  if (inverse) return gemm_nt(z, K, z, K, m, ldm, K, K, K, 1.0f, 0.0f, 0.0f, scal + 4, s);
  scale_copy_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(z, K, scal + 3, m, ldm);
  return cudaGetLastError();
}

}  // namespace bergson
