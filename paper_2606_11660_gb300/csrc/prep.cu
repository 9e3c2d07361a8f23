// Projection preparation (Fig. 1: random down-projection; App. "Gradients":
// double-sided projection), mask tile flags and the bounded-wait probe.
//
// The Gaussian projection is generated on the fly from its seed: entry
// (i, j) of P in R^{d x k} is z(seed, i*k + j) / sqrt(k), where z is a
// stateless counter-based normal draw: SplitMix64's finaliser (Steele, Lea
// and Flood, OOPSLA 2014) hashes the pair counter into two 53-bit uniforms
// and the Box-Muller transform (Box and Muller, 1958) turns them into a
// cosine draw (even counter) and a sine draw (odd counter).  The arithmetic is
// fp32 with the logarithm taken in the form that keeps relative accuracy near
// u1 = 1; the result agrees with an fp64 evaluation to a few fp32 ulps.
//
// The factored second moments are folded into P:  P_in' = diag(c^-1/2) P_in,
// P_out' = diag(r^-1/2) P_out, because
//   P_out^T (W / sqrt(r c^T)) P_in = P_out'^T W P_in'.
// P' is stored transposed ([k, d], K-major for the tensor cores) and split
// into two bf16 terms hi + lo, so A and G (exact bf16) meet a projection that
// is accurate to ~2^-16 relative instead of bf16's 2^-8.

#include "internal.h"
#include "ptx.cuh"

namespace bergson {

__device__ __forceinline__ uint64_t mix64(uint64_t x) {
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

// Standard normal draw number `e` of stream `seed`.
__device__ __forceinline__ float gaussian_draw(uint64_t seed, uint64_t e) {
  const uint64_t p = e >> 1;
  const uint64_t h1 = mix64(seed ^ mix64(2 * p));
  const uint64_t h2 = mix64(seed ^ mix64(2 * p + 1));
  const uint64_t n1 = (h1 >> 11) + 1;            // u1 = n1 * 2^-53 in (0, 1]
  float ln_u1;
  if (n1 > (1ull << 52)) {
    // u1 > 1/2: ln(u1) = log1p(-(1 - u1)) with 1 - u1 = (2^53 - n1) 2^-53 exact.
    ln_u1 = log1pf(-static_cast<float>((1ull << 53) - n1) * 0x1p-53f);
  } else {
    ln_u1 = logf(static_cast<float>(n1) * 0x1p-53f);
  }
  const float rho = sqrtf(-2.0f * ln_u1);
  const float two_u2 = static_cast<float>(h2 >> 11) * 0x1p-52f;   // 2 u2 in [0, 2)
  float s, c;
  sincospif(two_u2, &s, &c);                                       // angle 2 pi u2
  return (e & 1) ? rho * s : rho * c;
}

// Entry (i, j) of P' = diag(scale) P, fp32.
__device__ __forceinline__ float projection_entry(uint64_t seed, int i, int j, int k, int kind,
                                                  const float* moment) {
  float v;
  if (kind == 1) {
    v = (i == j) ? 1.0f : 0.0f;
  } else {
    const float inv_sqrt_k = 1.0f / sqrtf(static_cast<float>(k));
    v = gaussian_draw(seed, static_cast<uint64_t>(i) * k + j) * inv_sqrt_k;
  }
  if (moment != nullptr) v = v * (1.0f / sqrtf(moment[i]));
  return v;
}

__global__ void prep_kernel(const PrepSeg* __restrict__ segs, int n_segs, int64_t total) {
  for (int64_t f = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; f < total;
       f += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    int lo = 0, hi = n_segs - 1;               // last segment with begin <= f
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (segs[mid].begin <= f) lo = mid; else hi = mid - 1;
    }
    const PrepSeg& sg = segs[lo];
    const int64_t local = f - sg.begin;        // ordered (j, i): i fastest for coalesced stores
    const int i = static_cast<int>(local % sg.d);
    const int j = static_cast<int>(local / sg.d);
    const float v = projection_entry(sg.seed, i, j, sg.k, sg.kind, sg.moment);
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    const __nv_bfloat16 l = __float2bfloat16_rn(v - __bfloat162float(h));
    sg.dst[static_cast<int64_t>(j) * sg.d + i] = h;
    sg.dst[static_cast<int64_t>(sg.k + j) * sg.d + i] = l;
  }
}

__global__ void projection_matrix_kernel(uint64_t seed, int d, int k, int kind,
                                         const float* __restrict__ moment, float* __restrict__ out) {
  const int64_t n = static_cast<int64_t>(d) * k;
  for (int64_t f = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; f < n;
       f += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(f / k);
    const int j = static_cast<int>(f % k);
    out[f] = projection_entry(seed, i, j, k, kind, moment);
  }
}

// tile_valid[b, t] = 1 if any token of 128-token tile t of example b is valid.
__global__ void tile_valid_kernel(const uint8_t* __restrict__ mask, int B, int T, int n_tiles,
                                  uint8_t* __restrict__ tile_valid) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= B * n_tiles) return;
  const int b = warp / n_tiles;
  const int t0 = (warp % n_tiles) * kTileTokens;
  int any = 0;
  for (int t = t0 + lane; t < min(T, t0 + kTileTokens); t += 32)
    any |= mask[static_cast<int64_t>(b) * T + t] != 0;
  any = __any_sync(0xffffffffu, any);
  if (lane == 0) tile_valid[warp] = any ? 1 : 0;
}

// Waits on an mbarrier that nothing completes; exercises the timeout path.
__global__ void wait_probe_kernel(int* status, uint64_t timeout_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ volatile int abort_flag;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(smem_u32(&bar), 1);
    fence_barrier_init();
    if (!mbar_wait(smem_u32(&bar), 0, timeout_ns, &abort_flag))
      raise_device_error(status, &abort_flag, kStatusTimeout);
  }
}

cudaError_t launch_prep(const PrepSeg* segs, int n_segs, int64_t total, cudaStream_t s) {
  if (total <= 0) return cudaSuccess;
  const int threads = 256;
  const int64_t blocks = (total + threads - 1) / threads;
  prep_kernel<<<static_cast<unsigned>(blocks < 65535 * 8 ? blocks : 65535 * 8), threads, 0, s>>>(
      segs, n_segs, total);
  return cudaGetLastError();
}

cudaError_t launch_projection_matrix(uint64_t seed, int d, int k, int kind, const float* moment,
                                     float* out, cudaStream_t s) {
  const int64_t n = static_cast<int64_t>(d) * k;
  const int threads = 256;
  const int64_t blocks = (n + threads - 1) / threads;
  projection_matrix_kernel<<<static_cast<unsigned>(blocks < 65535 ? blocks : 65535), threads, 0,
                             s>>>(seed, d, k, kind, moment, out);
  return cudaGetLastError();
}

cudaError_t launch_tile_valid(const uint8_t* mask, int B, int T, int n_tiles, uint8_t* tile_valid,
                              cudaStream_t s) {
  const int64_t warps = static_cast<int64_t>(B) * n_tiles;
  if (warps == 0) return cudaSuccess;
  const int threads = 256;
  const int64_t blocks = (warps * 32 + threads - 1) / threads;
  tile_valid_kernel<<<static_cast<unsigned>(blocks), threads, 0, s>>>(mask, B, T, n_tiles,
                                                                      tile_valid);
  return cudaGetLastError();
}

cudaError_t launch_wait_probe(int* status, uint64_t timeout_ns, cudaStream_t s) {
  wait_probe_kernel<<<1, 32, 0, s>>>(status, timeout_ns);
  return cudaGetLastError();
}

}  // namespace bergson
