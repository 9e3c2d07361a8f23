// bergson_project_grads_noalloc: the projected-gradient entry point for
// callers that cannot hand the library a workspace.
//
// Some callers have no way to allocate device memory at the point where they
// call us: plugin and callback interfaces of host frameworks that pass only
// the input and output buffers, runtimes that own every byte of device memory
// through their own pool and forbid outside allocations, and latency-critical
// loops where a cudaMalloc (which can synchronise the device, and can fail
// when memory is short or fragmented) is not acceptable.  For them this file
// keeps a fixed scratch area in static device memory and runs the regular
// bergson_project_grads path on it.  Nothing here calls cudaMalloc, cudaFree
// or any allocating library routine; the array's memory is reserved by the
// CUDA driver when it loads this file's module on a device (see below).
//
// Properties a caller must know:
//   * The scratch is a file-scope __device__ array of BERGSON_NOALLOC_SCRATCH_BYTES
//     (32 MiB).  Every GPU that loads this part of the library keeps it until
//     the process exits.  Requests whose workspace would exceed it are
//     rejected with BERGSON_EWORKSPACE before anything is enqueued.
//   * All calls share that one array.  It keeps whatever the last call left
//     there; every call rewrites everything it reads (descriptors, counters,
//     projection slices, partial sums) before reading it.  Calls whose work
//     overlaps on the GPU (e.g. on two streams at once) race on the array and
//     must be ordered by the caller.
//   * The device address of the array is looked up once per device, on the
//     first call that runs on that device (with that device current).  This
//     file has no kernels, so under lazy module loading (CUDA's default) that
//     lookup is what loads its module on the device, and the driver reserves
//     the 32 MiB array then: the first call can fail with BERGSON_ECUDA when
//     the device has no 32 MiB left.  A warm-up call with B = 0 and
//     out = NULL (any valid layer array) does the lookup on the current
//     device and enqueues nothing, so a caller can take that step early.
//     Make the first call on each device before any stream capture begins.
//   * The kernels it runs set their shared-memory limits once per device, so
//     one process may call this on several GPUs (one scratch array each).

#include <mutex>

#include "bergson.h"
#include "internal.h"

namespace {

constexpr size_t kScratchBytes = BERGSON_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// Host code must not use this name as an address: it is a host-side stand-in.
// The device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// Device address of the scratch array on `dev` (which must be current), or
// nullptr if the lookup failed.
void* scratch_address(int dev) {
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  std::lock_guard<std::mutex> lk(mu);
  if (dev < 0 || dev >= kMaxDevices) return nullptr;
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
    addr[dev] = p;
  }
  return addr[dev];
}

}  // namespace

extern "C" BERGSON_API int bergson_project_grads_noalloc(const bergson_layer* layers, int n_layers,
                                                         int64_t B, int64_t T,
                                                         const uint8_t* mask, float* out,
                                                         int64_t ld_out, void* stream) {
  size_t need = 0;
  const int st = bergson_project_grads_workspace(layers, n_layers, B, T, &need);
  if (st != BERGSON_OK) return st;
  if (need > kScratchBytes)
    return bergson::record_error(
        BERGSON_EWORKSPACE,
        "bergson_project_grads_noalloc: this request needs %zu bytes of scratch but the "
        "allocation-free entry point has a fixed %zu bytes; split the modules over several "
        "calls or call bergson_project_grads with a workspace",
        need, kScratchBytes);
  // The work runs on the device that owns `out` (the current device if there is no output).
  int dev = -1;
  if (out != nullptr) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, out) != cudaSuccess ||
        (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged))
      return bergson::record_error(BERGSON_EINVAL,
                                   "bergson_project_grads_noalloc: out is not device memory");
    dev = at.device;
  } else if (cudaGetDevice(&dev) != cudaSuccess) {
    return bergson::record_error(BERGSON_ECUDA, "bergson_project_grads_noalloc: no CUDA device");
  }
  int prev = -1;
  if (cudaGetDevice(&prev) != cudaSuccess || (prev != dev && cudaSetDevice(dev) != cudaSuccess))
    return bergson::record_error(BERGSON_ECUDA, "bergson_project_grads_noalloc: cannot select "
                                                "device %d", dev);
  void* scratch = scratch_address(dev);
  if (prev != dev) cudaSetDevice(prev);
  if (scratch == nullptr)
    return bergson::record_error(BERGSON_ECUDA, "bergson_project_grads_noalloc: "
                                                "cudaGetSymbolAddress of the scratch array failed");
  return bergson_project_grads(layers, n_layers, B, T, mask, out, ld_out, scratch, kScratchBytes,
                               stream);
}
