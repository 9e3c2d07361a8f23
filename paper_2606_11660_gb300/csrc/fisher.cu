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
// All products are "NT" GEMMs C = alpha A B^T + beta C + gamma I with A and B
// row-major and the reduction index contiguous, run by the tcgen05 skinny
// product of onthefly.cu (3xTF32: fp32 accuracy from tf32 tensor-core MMAs)
// with 128-row tiles on both sides.  Products of the iteration are
// symmetric in exact arithmetic, so B^T = B there; each update is
// re-symmetrised so that rounding cannot build up an antisymmetric part.

#include "internal.h"

namespace bergson {

namespace {

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

// part[blockIdx] = compensated sum of squares of (R - shift I) over a
// grid-stride slice of R.
__global__ void frob_partial_kernel(const float* __restrict__ r, int64_t ld, int K, float shift,
                                    float* __restrict__ part) {
  __shared__ float red[32];
  float s = 0.0f, comp = 0.0f;
  const int64_t n = static_cast<int64_t>(K) * K;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t i = e / K, j = e % K;
    const float x = r[i * ld + j] - (i == j ? shift : 0.0f);
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

// *out = scale * sqrt(fixed-order compensated sum of part[0, n_part))
__global__ void frob_norm_kernel(const float* __restrict__ part, int n_part, float scale,
                                 float* __restrict__ out) {
  if (threadIdx.x != 0) return;
  float t = 0.0f, comp = 0.0f;
  for (int i = 0; i < n_part; ++i) {
    const float y = part[i] - comp;
    const float u = t + y;
    comp = (u - t) - y;
    t = u;
  }
  *out = scale * sqrtf(t);
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

// x <- (x + x^T) / 2 in place.  The iterates are symmetric in exact
// arithmetic, but the products use B^T = B, which turns the rounding's
// antisymmetric part into a growing error unless it is removed.  One CTA per
// pair of 32 x 32 tiles (ti <= tj): both tiles are read row by row into shared
// memory and written back row by row, so every global access is coalesced.
__global__ void __launch_bounds__(256) symmetrize_kernel(float* __restrict__ x, int K) {
  __shared__ float a[32][33], b[32][33];
  const int ti = blockIdx.y, tj = blockIdx.x;
  if (ti > tj) return;
  const int i0 = ti * 32, j0 = tj * 32, c = threadIdx.x;
  for (int r = threadIdx.y; r < 32; r += 8) {
    a[r][c] = (i0 + r < K && j0 + c < K) ? x[static_cast<int64_t>(i0 + r) * K + j0 + c] : 0.0f;
    b[r][c] = (j0 + r < K && i0 + c < K) ? x[static_cast<int64_t>(j0 + r) * K + i0 + c] : 0.0f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += 8) {
    if (i0 + r < K && j0 + c < K)
      x[static_cast<int64_t>(i0 + r) * K + j0 + c] = 0.5f * (a[r][c] + b[c][r]);
    if (ti != tj && j0 + r < K && i0 + c < K)
      x[static_cast<int64_t>(j0 + r) * K + i0 + c] = 0.5f * (b[r][c] + a[c][r]);
  }
}

// x <- x^T in place (K x K, leading dimension K).  One CTA per pair of 32 x 32
// tiles (ti <= tj), both read row by row into shared memory and written back
// swapped, so every global access is coalesced.
__global__ void __launch_bounds__(256) transpose_inplace_kernel(float* __restrict__ x, int K) {
  __shared__ float a[32][33], b[32][33];
  const int ti = blockIdx.y, tj = blockIdx.x;
  if (ti > tj) return;
  const int i0 = ti * 32, j0 = tj * 32, c = threadIdx.x;
  for (int r = threadIdx.y; r < 32; r += 8) {
    a[r][c] = (i0 + r < K && j0 + c < K) ? x[static_cast<int64_t>(i0 + r) * K + j0 + c] : 0.0f;
    b[r][c] = (j0 + r < K && i0 + c < K) ? x[static_cast<int64_t>(j0 + r) * K + i0 + c] : 0.0f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += 8) {
    if (i0 + r < K && j0 + c < K) x[static_cast<int64_t>(i0 + r) * K + j0 + c] = b[c][r];
    if (ti != tj && j0 + r < K && i0 + c < K)
      x[static_cast<int64_t>(j0 + r) * K + i0 + c] = a[c][r];
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

// C[m, n] = alpha' sum_k A[m, k] B[n, k] + beta C[m, n] + gamma [m == n] for
// M x K A and N x K B (alpha' = alpha * (*alpha_s) when alpha_s is given);
// `ws` holds xgemm_plan(M, N, K).
cudaError_t gemm_nt(const float* A, int64_t lda, const float* B, int64_t ldb, float* C,
                    int64_t ldc, int M, int N, int K, float alpha, float beta, float gamma,
                    const float* alpha_s, uint8_t* ws, int* status, int sms, cudaStream_t s) {
  XGemmArgs a;
  a.x = A;
  a.ldx = lda;
  a.y = B;
  a.ldy = ldb;
  a.B = M;
  a.Q = N;
  a.K = K;
  a.unit = 0;
  a.alpha = alpha;
  a.alpha_s = alpha_s;
  a.beta = beta;
  a.gamma = gamma;
  a.scores = C;
  a.ld_scores = ldc;
  a.ws = ws;
  a.status = status;
  a.timeout_ns = kWaitTimeoutNs;
  return xgemm_run(a, sms, s);
}

size_t round_up256(size_t x) { return (x + 255) / 256 * 256; }

unsigned elementwise_blocks(int64_t n) {
  const int64_t b = (n + 255) / 256;
  return static_cast<unsigned>(b < 8192 ? b : 8192);
}

}  // namespace

size_t fisher_fit_workspace(int64_t n, int64_t K) {
  const int64_t n_pad = (n + 3) / 4 * 4;
  return round_up256(static_cast<size_t>(K) * n_pad * sizeof(float)) +
         xgemm_plan(K, K, n_pad).total;
}

cudaError_t launch_fisher_fit(const float* x, int n, int K, int64_t ldx, float* r, int64_t ldr,
                              float* ws, int* status, int sms, cudaStream_t s) {
  const int n_pad = (n + 3) / 4 * 4;
  dim3 grid((n_pad + 31) / 32, (K + 31) / 32);
  transpose_kernel<<<grid, dim3(32, 8), 0, s>>>(x, n, K, ldx, ws, n_pad);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  uint8_t* gws = reinterpret_cast<uint8_t*>(ws) +
                 round_up256(static_cast<size_t>(K) * n_pad * sizeof(float));
  return gemm_nt(ws, n_pad, ws, n_pad, r, ldr, K, K, n_pad, 1.0f / static_cast<float>(n), 0.0f,
                 0.0f, nullptr, gws, status, sms, s);
}

size_t fisher_power_workspace(int64_t K) {
  return round_up256((4 * static_cast<size_t>(K) * K + 64 + kFrobBlocks) * sizeof(float)) +
         xgemm_plan(K, K, K).total;
}

cudaError_t launch_fisher_power(const float* r1, const float* r2, int K, int64_t ldr, float lam,
                                float damping, int inverse, int iterations, float tol,
                                float* residuals, int* iterations_done, float* m, int64_t ldm,
                                float* ws, int* status, int sms, cudaStream_t s) {
  const int64_t kk = static_cast<int64_t>(K) * K;
  uint8_t* gws = reinterpret_cast<uint8_t*>(ws) +
                 round_up256((4 * static_cast<size_t>(K) * K + 64 + kFrobBlocks) * sizeof(float));
  float* a = ws;            // mixed, damped R
  float* y = a + kk;
  float* z = y + kk;
  float* t = z + kk;
  float* scal = t + kk;     // trace, ||R||_F, 1/c, 1/sqrt(c), 1/c, residual;
                            // [64, 64 + 512): partial sums
  const bool track = residuals != nullptr || tol > 0.0f;
  if (iterations_done != nullptr) *iterations_done = 0;
  mixed_trace_kernel<<<1, 1024, 0, s>>>(r1, r2, ldr, K, lam, scal);
  mix_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(r1, r2, ldr, K, lam, damping, scal, a, K);
  frob_partial_kernel<<<kFrobBlocks, 256, 0, s>>>(a, K, K, 0.0f, scal + 64);
  frob_final_kernel<<<1, 32, 0, s>>>(scal + 64, kFrobBlocks, scal);
  ns_init_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(a, K, K, scal, y, z);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const dim3 tiles((K + 31) / 32, (K + 31) / 32);
  for (int it = 0;; ++it) {
    if (!track && it == iterations) break;
    // T = 1.5 I - 0.5 Z Y;  Z <- T Z;  Y <- Y T.
    // Z Y is not symmetric in floating point, so T != T^T: the Y update must
    // use T itself.  The products are NT (C = A B^T), so T Z = nt(T, Z) (Z is
    // symmetric) and Y T = nt(Y, T^T): T is transposed in place between them.
    // (Taking Y T^T instead is unstable: to first order, a symmetric
    // perturbation of the iterates along eigenvectors i, j of R grows by
    // (rho - 1) / 2 per step, rho = (s_i / s_j + s_j / s_i) / 2 with s the
    // eigenvalues of R^1/2, so once R's condition number exceeds ~34
    // (s_i / s_j > 3 + sqrt(8)) the converged iterates drift away again.
    // With Y T the same perturbation maps to a fixed point: stable.)
    if ((e = gemm_nt(z, K, y, K, t, K, K, K, K, -0.5f, 0.0f, 1.5f, nullptr, gws, status, sms,
                     s)) != cudaSuccess)
      return e;
    if (track) {
      // ||I - Z Y||_F / sqrt(K) = 2 ||T - I||_F / sqrt(K): the current iterate's
      // residual (Z Y = Z (R/c) Z = M R M while the iteration keeps Y = (R/c) Z).
      frob_partial_kernel<<<kFrobBlocks, 256, 0, s>>>(t, K, K, 1.0f, scal + 64);
      frob_norm_kernel<<<1, 32, 0, s>>>(scal + 64, kFrobBlocks,
                                        2.0f / sqrtf(static_cast<float>(K)), scal + 5);
      float res = 0.0f;
      if ((e = cudaMemcpyAsync(&res, scal + 5, sizeof(float), cudaMemcpyDeviceToHost, s)) !=
              cudaSuccess ||
          (e = cudaStreamSynchronize(s)) != cudaSuccess)
        return e;
      if (residuals != nullptr) residuals[it] = res;
      if (res <= tol) break;
    }
    if (it == iterations) break;
    if ((e = gemm_nt(t, K, z, K, a, K, K, K, K, 1.0f, 0.0f, 0.0f, nullptr, gws, status, sms,
                     s)) != cudaSuccess)            // a = T Z (new Z)
      return e;
    transpose_inplace_kernel<<<tiles, dim3(32, 8), 0, s>>>(t, K);     // t = T^T
    if ((e = gemm_nt(y, K, t, K, z, K, K, K, K, 1.0f, 0.0f, 0.0f, nullptr, gws, status, sms,
                     s)) != cudaSuccess)            // old Z buffer = Y T (new Y)
      return e;
    float* old_y = y;
    y = z;
    z = a;
    a = old_y;
    symmetrize_kernel<<<tiles, dim3(32, 8), 0, s>>>(y, K);
    symmetrize_kernel<<<tiles, dim3(32, 8), 0, s>>>(z, K);
    if (iterations_done != nullptr) *iterations_done = it + 1;
  }
  // Z ~ (R/c)^-1/2:  R^-1/2 = Z / sqrt(c);  R^-1 = Z Z / c
  if (inverse)
    return gemm_nt(z, K, z, K, m, ldm, K, K, K, 1.0f, 0.0f, 0.0f, scal + 4, gws, status, sms, s);
  scale_copy_kernel<<<elementwise_blocks(kk), 256, 0, s>>>(z, K, scal + 3, m, ldm);
  return cudaGetLastError();
}

}  // namespace bergson
