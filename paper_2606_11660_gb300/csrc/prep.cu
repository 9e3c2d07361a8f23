// Projection preparation (Fig. 1: random down-projection; App. B, "Gradients":
// double-sided projection), mask tile flags and the bounded-wait probe.
//
// The projection is generated on the fly from its seed: entry
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

#include "bergson.h"
#include "internal.h"
#include "ptx.cuh"

namespace bergson {

__device__ __forceinline__ uint64_t mix64(uint64_t x) {
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

// The two standard normal draws of pair `p` of stream `seed`: counter 2p takes
// the cosine branch (*zc), counter 2p + 1 the sine branch (*zs).
__device__ __forceinline__ void gaussian_pair(uint64_t seed, uint64_t p, float* zc, float* zs) {
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
  *zc = rho * c;
  *zs = rho * s;
}

// Rademacher and uniform draws (App. B names both) take one hash per counter,
// h_e = mix(seed ^ mix(e)).  Rademacher: +1 when the top bit of h_e is set,
// else -1.  Uniform on (-1, 1): the top 24 bits v of h_e give the cell
// midpoint (2v + 1 - 2^24) 2^-24, exact in fp32; sqrt(3) brings the variance
// from 1/3 to 1.
__device__ __forceinline__ float counter_draw(uint64_t seed, uint64_t e, int kind) {
  const uint64_t h = mix64(seed ^ mix64(e));
  if (kind == BERGSON_PROJ_RADEMACHER) return (h >> 63) ? 1.0f : -1.0f;
  const int v = static_cast<int>(h >> 40);
  return static_cast<float>(2 * v + 1 - (1 << 24)) * 0x1p-24f * 1.7320508075688772f;
}

// Entries (i, j) and (i, j + 1), j even, of P' = diag(scale) P, fp32.  They
// are counters e = i*k + j and e + 1, i.e. both draws of pair e / 2.  The
// factored second moments must be positive (the scale is moment_i^-1/2): an
// entry that is not (zero, negative or NaN) is recorded as BERGSON_EMOMENT in
// the device status word, and the values computed from it (inf or NaN) are
// stored as they come.
__device__ __forceinline__ void projection_pair(uint64_t seed, int i, int j, int k, int kind,
                                                const float* moment, int* status, float* v0,
                                                float* v1) {
  const float inv_sqrt_k = 1.0f / sqrtf(static_cast<float>(k));
  const uint64_t e = static_cast<uint64_t>(i) * k + j;
  if (kind == BERGSON_PROJ_IDENTITY) {
    *v0 = (i == j) ? 1.0f : 0.0f;
    *v1 = (i == j + 1) ? 1.0f : 0.0f;
  } else if (kind == BERGSON_PROJ_GAUSSIAN) {
    float zc, zs;
    gaussian_pair(seed, e >> 1, &zc, &zs);
    *v0 = zc * inv_sqrt_k;
    *v1 = zs * inv_sqrt_k;
  } else {
    *v0 = counter_draw(seed, e, kind) * inv_sqrt_k;
    *v1 = counter_draw(seed, e + 1, kind) * inv_sqrt_k;
  }
  if (moment != nullptr) {
    const float m = moment[i];
    if (!(m > 0.0f) && j == 0 && status != nullptr) atomicCAS(status, 0, kStatusMoment);
    const float sc = 1.0f / sqrtf(m);
    *v0 = *v0 * sc;
    *v1 = *v1 * sc;
  }
}

__device__ __forceinline__ void store_hi_lo(__nv_bfloat16* dst, int64_t hi_idx, int64_t lo_idx,
                                            float v) {
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  dst[hi_idx] = h;
  dst[lo_idx] = __float2bfloat16_rn(v - __bfloat162float(h));
}

// Entry pair q = (i, j / 2) of a segment: both values of P'[i, j..j+1] as bf16
// hi + lo, written transposed.
__device__ __forceinline__ void prep_pair(const PrepSeg& sg, int i, int j, int* status) {
  float v0, v1;
  projection_pair(sg.seed, i, j, sg.k, sg.kind, sg.moment, status, &v0, &v1);
  const int64_t d = sg.d;
  store_hi_lo(sg.dst, j * d + i, (sg.k + j) * d + i, v0);
  store_hi_lo(sg.dst, (j + 1) * d + i, (sg.k + j + 1) * d + i, v1);
}

// blockIdx.y = segment; threads walk the segment's d*k/2 entry pairs with the
// input index i fastest, so the transposed bf16 stores are coalesced.  The
// index arithmetic is 32-bit when the segment allows it (the common case).
__global__ void prep_kernel(const PrepSeg* __restrict__ segs, int* status) {
  griddep_launch_dependents();   // the projection kernel may set itself up meanwhile
  const PrepSeg sg = segs[blockIdx.y];
  const int64_t npairs = static_cast<int64_t>(sg.d) * sg.k / 2;
  if (npairs <= 0x7fffffff) {
    const uint32_t n = static_cast<uint32_t>(npairs), d = static_cast<uint32_t>(sg.d);
    for (uint32_t q = blockIdx.x * blockDim.x + threadIdx.x; q < n; q += gridDim.x * blockDim.x)
      prep_pair(sg, static_cast<int>(q % d), 2 * static_cast<int>(q / d), status);
  } else {
    for (int64_t q = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; q < npairs;
         q += static_cast<int64_t>(gridDim.x) * blockDim.x)
      prep_pair(sg, static_cast<int>(q % sg.d), 2 * static_cast<int>(q / sg.d), status);
  }
}

__global__ void projection_matrix_kernel(uint64_t seed, int d, int k, int kind,
                                         const float* __restrict__ moment, int* status,
                                         float* __restrict__ out) {
  const int64_t npairs = static_cast<int64_t>(d) * k / 2;
  for (int64_t q = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; q < npairs;
       q += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>((2 * q) / k);
    const int j = static_cast<int>((2 * q) % k);
    float v0, v1;
    projection_pair(seed, i, j, k, kind, moment, status, &v0, &v1);
    out[2 * q] = v0;
    out[2 * q + 1] = v1;
  }
}

// tile_valid[b, t] bit q (q = 0..3) = 1 if any token of the 32-token slice
// [128 t + 32 q, 128 t + 32 q + 32) of example b is valid.  One warp per tile.
__global__ void tile_valid_kernel(const uint8_t* __restrict__ mask, int B, int T, int n_tiles,
                                  uint8_t* __restrict__ tile_valid) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= B * n_tiles) return;
  const int b = warp / n_tiles;
  const int t0 = (warp % n_tiles) * kTileTokens;
  uint32_t bits = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int t = t0 + 32 * q + lane;
    const int v = t < T && mask[static_cast<int64_t>(b) * T + t] != 0;
    if (__any_sync(0xffffffffu, v)) bits |= 1u << q;
  }
  if (lane == 0) tile_valid[warp] = static_cast<uint8_t>(bits);
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

cudaError_t launch_prep(const PrepSeg* segs, int n_segs, int64_t max_pairs, int* status,
                        cudaStream_t s) {
  if (n_segs <= 0 || max_pairs <= 0) return cudaSuccess;
  const int threads = 256;
  int64_t bx = (max_pairs + 4 * threads - 1) / (4 * threads);   // ~4 pairs per thread
  if (bx > 4096) bx = 4096;
  prep_kernel<<<dim3(static_cast<unsigned>(bx), static_cast<unsigned>(n_segs)), threads, 0, s>>>(
      segs, status);
  return cudaGetLastError();
}

cudaError_t launch_projection_matrix(uint64_t seed, int d, int k, int kind, const float* moment,
                                     int* status, float* out, cudaStream_t s) {
  const int64_t npairs = static_cast<int64_t>(d) * k / 2;
  const int threads = 256;
  const int64_t blocks = (npairs + threads - 1) / threads;
  projection_matrix_kernel<<<static_cast<unsigned>(blocks < 65535 ? blocks : 65535), threads, 0,
                             s>>>(seed, d, k, kind, moment, status, out);
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
