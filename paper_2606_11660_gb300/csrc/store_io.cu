// On-disk gradient store (Bergson Sec. 3.1: gradient stores persisted to disk
// and read back as memory maps).  The file is the store itself: N rows of K
// fp16 values, row-major, no header, so numpy.memmap(path, float16, shape=(N, K))
// opens it.  Rows are moved through a host bounce buffer in 64 MiB pieces.

#include <fcntl.h>
#include <unistd.h>

#include <cstdio>
#include <vector>

#include "bergson.h"
#include "internal.h"

namespace {

constexpr size_t kPiece = size_t{64} << 20;

bool write_all(int fd, const void* buf, size_t n, off_t off) {
  const char* p = static_cast<const char*>(buf);
  while (n > 0) {
    const ssize_t w = pwrite(fd, p, n, off);
    if (w <= 0) return false;
    p += w;
    n -= static_cast<size_t>(w);
    off += w;
  }
  return true;
}

bool read_all(int fd, void* buf, size_t n, off_t off) {
  char* p = static_cast<char*>(buf);
  while (n > 0) {
    const ssize_t r = pread(fd, p, n, off);
    if (r <= 0) return false;
    p += r;
    n -= static_cast<size_t>(r);
    off += r;
  }
  return true;
}

int check_store_args(const void* store, int64_t rows, int64_t K, int64_t ld, const char* path,
                     int64_t row_offset) {
  if (path == nullptr || path[0] == 0) return bergson::record_error(BERGSON_EINVAL, "path is empty");
  if (rows < 0 || row_offset < 0 || K < 1 || ld < K)
    return bergson::record_error(BERGSON_EINVAL, "need rows >= 0, row_offset >= 0, K >= 1, ld >= K");
  if (rows > 0 && store == nullptr) return bergson::record_error(BERGSON_EINVAL, "store is NULL");
  return BERGSON_OK;
}

}  // namespace

extern "C" BERGSON_API int bergson_store_save(const void* store, int64_t rows, int64_t K,
                                              int64_t ld_store, const char* path,
                                              int64_t file_row_offset, void* stream) {
  int st = check_store_args(store, rows, K, ld_store, path, file_row_offset);
  if (st != BERGSON_OK) return st;
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess)
    return bergson::record_error(BERGSON_ECUDA, "stream synchronisation: %s", cudaGetErrorString(e));
  const int fd = open(path, O_WRONLY | O_CREAT, 0644);
  if (fd < 0) return bergson::record_error(BERGSON_EINVAL, "cannot open %s for writing", path);
  const size_t row_bytes = static_cast<size_t>(K) * 2;
  const int64_t rows_per_piece = static_cast<int64_t>(kPiece / row_bytes > 0 ? kPiece / row_bytes : 1);
  std::vector<char> buf(static_cast<size_t>(rows_per_piece) * row_bytes);
  for (int64_t r0 = 0; r0 < rows; r0 += rows_per_piece) {
    const int64_t n = rows - r0 < rows_per_piece ? rows - r0 : rows_per_piece;
    e = cudaMemcpy2D(buf.data(), row_bytes,
                     static_cast<const char*>(store) + static_cast<size_t>(r0) * ld_store * 2,
                     static_cast<size_t>(ld_store) * 2, row_bytes, static_cast<size_t>(n),
                     cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) {
      close(fd);
      return bergson::record_error(BERGSON_ECUDA, "device-to-host copy: %s", cudaGetErrorString(e));
    }
    if (!write_all(fd, buf.data(), static_cast<size_t>(n) * row_bytes,
                   static_cast<off_t>((file_row_offset + r0) * static_cast<int64_t>(row_bytes)))) {
      close(fd);
      return bergson::record_error(BERGSON_EINVAL, "write to %s failed", path);
    }
  }
  if (close(fd) != 0) return bergson::record_error(BERGSON_EINVAL, "closing %s failed", path);
  return BERGSON_OK;
}

extern "C" BERGSON_API int bergson_store_load(const char* path, int64_t file_row_offset,
                                              int64_t rows, int64_t K, void* store,
                                              int64_t ld_store, void* stream) {
  int st = check_store_args(store, rows, K, ld_store, path, file_row_offset);
  if (st != BERGSON_OK) return st;
  const int fd = open(path, O_RDONLY);
  if (fd < 0) return bergson::record_error(BERGSON_EINVAL, "cannot open %s", path);
  const size_t row_bytes = static_cast<size_t>(K) * 2;
  const off_t end = lseek(fd, 0, SEEK_END);
  if (end < 0 || (file_row_offset + rows) * static_cast<int64_t>(row_bytes) > end) {
    close(fd);
    return bergson::record_error(BERGSON_EINVAL, "%s holds fewer than %lld rows of %lld values",
                                 path, (long long)(file_row_offset + rows), (long long)K);
  }
  const int64_t rows_per_piece = static_cast<int64_t>(kPiece / row_bytes > 0 ? kPiece / row_bytes : 1);
  std::vector<char> buf(static_cast<size_t>(rows_per_piece) * row_bytes);
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  for (int64_t r0 = 0; e == cudaSuccess && r0 < rows; r0 += rows_per_piece) {
    const int64_t n = rows - r0 < rows_per_piece ? rows - r0 : rows_per_piece;
    if (!read_all(fd, buf.data(), static_cast<size_t>(n) * row_bytes,
                  static_cast<off_t>((file_row_offset + r0) * static_cast<int64_t>(row_bytes)))) {
      close(fd);
      return bergson::record_error(BERGSON_EINVAL, "read from %s failed", path);
    }
    e = cudaMemcpy2D(static_cast<char*>(store) + static_cast<size_t>(r0) * ld_store * 2,
                     static_cast<size_t>(ld_store) * 2, buf.data(), row_bytes, row_bytes,
                     static_cast<size_t>(n), cudaMemcpyHostToDevice);
  }
  close(fd);
  if (e != cudaSuccess)
    return bergson::record_error(BERGSON_ECUDA, "host-to-device copy: %s", cudaGetErrorString(e));
  return BERGSON_OK;
}
