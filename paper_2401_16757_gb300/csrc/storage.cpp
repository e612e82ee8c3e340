// Storage tier (Sec. 4.2.1 "Direct Block Fetch"): the weights file writer,
// its validating reader, and the direct-I/O read of a block's file runs
// that an engine loaded from a file issues for every swap-in.
//
// Blocks are read with O_DIRECT, so the page cache keeps no second copy of
// a block (the paper's reason for bypassing `read`): the file offset, the
// length and the destination of every read are multiples of kFileAlign.
// The format is documented beside swapnet_weights_file_write in swapnet.h.
#include <fcntl.h>
#include <sys/stat.h>
#include <unistd.h>

#include <algorithm>
#include <cerrno>
#include <cstdlib>
#include <cstring>
#include <memory>
#include <new>

#include "internal.h"

namespace swapnet {
namespace {

constexpr char kMagic[8] = {'S', 'W', 'N', 'W', 'G', 'T', '0', '1'};
constexpr uint32_t kVersion = 1;
constexpr uint64_t kHeadFixed = 8 + 4 + 4 + 8;  // magic, version, count, data offset
constexpr uint64_t kBounce = 16ull << 20;       // host read: bounce window

std::string errno_text(const std::string& what, int e) { return what + ": " + std::strerror(e); }

// Whole positional read: retries short reads and EINTR; EIO at end of file.
int pread_all(int fd, char* dst, uint64_t len, uint64_t off) {
  while (len > 0) {
    const ssize_t r = ::pread(fd, dst, (size_t)std::min<uint64_t>(len, 1ull << 30), (off_t)off);
    if (r < 0) {
      if (errno == EINTR) continue;
      return errno;
    }
    if (r == 0) return EIO;
    dst += r;
    off += (uint64_t)r;
    len -= (uint64_t)r;
  }
  return 0;
}

int pwrite_all(int fd, const char* src, uint64_t len, uint64_t off) {
  while (len > 0) {
    const ssize_t r = ::pwrite(fd, src, (size_t)std::min<uint64_t>(len, 1ull << 30), (off_t)off);
    if (r < 0) {
      if (errno == EINTR) continue;
      return errno;
    }
    if (r == 0) return EIO;
    src += r;
    off += (uint64_t)r;
    len -= (uint64_t)r;
  }
  return 0;
}

struct AlignedBuf {
  void* p = nullptr;
  explicit AlignedBuf(uint64_t bytes) {
    if (posix_memalign(&p, kFileAlign, (size_t)std::max<uint64_t>(bytes, kFileAlign)) != 0) p = nullptr;
  }
  ~AlignedBuf() { std::free(p); }
  char* data() const { return static_cast<char*>(p); }
};

template <typename T> void put(char* at, T v) { std::memcpy(at, &v, sizeof(T)); }
template <typename T> T get(const char* at) {
  T v;
  std::memcpy(&v, at, sizeof(T));
  return v;
}

}  // namespace

int file_read_runs(const swapnet_weights_file* f, const FileRun* runs, size_t n, char* stage) {
  for (size_t i = 0; i < n; ++i) {
    const int e = pread_all(f->fd, stage + runs[i].stage_off, runs[i].len, runs[i].file_off);
    if (e) return e;
  }
  return 0;
}

}  // namespace swapnet

using namespace swapnet;

extern "C" {

int swapnet_weights_file_write(const char* path, const swapnet_model_desc* desc, const void* const* host_weights,
                               uint32_t n_tensors) {
  return swapnet::guard_abi([&]() -> int {
    if (!path || !desc || (n_tensors && !host_weights)) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    Model m;
    int rc = analyse_model(desc, &m);
    if (rc) return rc;
    if ((int)n_tensors != m.n_tensors)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "expected " + std::to_string(m.n_tensors) + " host tensors");
    const uint64_t table = kHeadFixed + 16ull * n_tensors;
    const uint64_t data0 = align_up(table, kFileAlign);
    std::vector<uint64_t> off(n_tensors), len(n_tensors);
    uint64_t cur = data0;
    for (uint32_t t = 0; t < n_tensors; ++t) {
      len[t] = m.tensor_raw[t];
      if (len[t] && !host_weights[t]) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null host weight pointer");
      off[t] = cur;
      cur = align_up(cur + len[t], kFileAlign);
    }
    std::vector<char> head(data0, 0);
    std::memcpy(head.data(), kMagic, 8);
    put<uint32_t>(head.data() + 8, kVersion);
    put<uint32_t>(head.data() + 12, n_tensors);
    put<uint64_t>(head.data() + 16, data0);
    for (uint32_t t = 0; t < n_tensors; ++t) {
      put<uint64_t>(head.data() + kHeadFixed + 16ull * t, off[t]);
      put<uint64_t>(head.data() + kHeadFixed + 16ull * t + 8, len[t]);
    }
    const int fd = ::open(path, O_WRONLY | O_CREAT | O_TRUNC | O_CLOEXEC, 0644);
    if (fd < 0) SN_FAIL(SWAPNET_ERR_IO, errno_text(std::string("open ") + path, errno));
    int e = pwrite_all(fd, head.data(), head.size(), 0);
    for (uint32_t t = 0; t < n_tensors && !e; ++t)
      if (len[t]) e = pwrite_all(fd, static_cast<const char*>(host_weights[t]), len[t], off[t]);
    if (!e && ::ftruncate(fd, (off_t)cur) != 0) e = errno;
    if (!e && ::fsync(fd) != 0) e = errno;
    if (::close(fd) != 0 && !e) e = errno;
    if (e) SN_FAIL(SWAPNET_ERR_IO, errno_text(std::string("write ") + path, e));
    return SWAPNET_OK;
  });
}

int swapnet_weights_file_open(const char* path, uint32_t flags, swapnet_weights_file** out) {
  return swapnet::guard_abi([&]() -> int {
    if (!path || !out) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    if (flags & ~(uint32_t)SWAPNET_FILE_ALLOW_BUFFERED) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "unknown flags");
    std::unique_ptr<swapnet_weights_file> f(new (std::nothrow) swapnet_weights_file());
    if (!f) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    f->fd = ::open(path, O_RDONLY | O_CLOEXEC | O_DIRECT);
    f->direct = true;
    if (f->fd < 0 && errno == EINVAL && (flags & SWAPNET_FILE_ALLOW_BUFFERED)) {
      f->fd = ::open(path, O_RDONLY | O_CLOEXEC);
      f->direct = false;
    }
    if (f->fd < 0) SN_FAIL(SWAPNET_ERR_IO, errno_text(std::string("open ") + path, errno));
    struct stat st;
    if (::fstat(f->fd, &st) != 0) SN_FAIL(SWAPNET_ERR_IO, errno_text("fstat", errno));
    f->file_bytes = (uint64_t)st.st_size;
    if (f->file_bytes < kFileAlign || f->file_bytes % kFileAlign)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "not a weights file (length is not a positive multiple of 4096)");
    AlignedBuf first(kFileAlign);
    if (!first.p) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    int e = pread_all(f->fd, first.data(), kFileAlign, 0);
    if (e) SN_FAIL(SWAPNET_ERR_IO, errno_text("read header", e));
    if (std::memcmp(first.data(), kMagic, 8) != 0) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "not a weights file (magic)");
    if (get<uint32_t>(first.data() + 8) != kVersion) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "unsupported weights file version");
    const uint32_t n = get<uint32_t>(first.data() + 12);
    const uint64_t data0 = get<uint64_t>(first.data() + 16);
    const uint64_t table = kHeadFixed + 16ull * n;
    if (data0 % kFileAlign || data0 < table || data0 > f->file_bytes)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "weights file: bad data offset");
    AlignedBuf head(data0);
    if (!head.p) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    e = pread_all(f->fd, head.data(), data0, 0);
    if (e) SN_FAIL(SWAPNET_ERR_IO, errno_text("read header", e));
    f->n = n;
    f->off.resize(n);
    f->bytes.resize(n);
    uint64_t prev_end = data0;
    for (uint32_t t = 0; t < n; ++t) {
      const uint64_t o = get<uint64_t>(head.data() + kHeadFixed + 16ull * t);
      const uint64_t b = get<uint64_t>(head.data() + kHeadFixed + 16ull * t + 8);
      if (o % kFileAlign || o < prev_end || b > f->file_bytes || o > f->file_bytes - b)
        SN_FAIL(SWAPNET_ERR_INVALID_ARG, "weights file: tensor " + std::to_string(t) + " out of place");
      f->off[t] = o;
      f->bytes[t] = b;
      prev_end = o + b;
    }
    *out = f.release();
    return SWAPNET_OK;
  });
}

int swapnet_weights_file_info(const swapnet_weights_file* f, uint32_t* n_tensors, int32_t* direct) {
  return swapnet::guard_abi([&]() -> int {
    if (!f) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null file");
    if (n_tensors) *n_tensors = f->n;
    if (direct) *direct = f->direct ? 1 : 0;
    return SWAPNET_OK;
  });
}

int swapnet_weights_file_read(swapnet_weights_file* f, uint32_t tensor, uint64_t offset, uint64_t bytes, void* dst) {
  return swapnet::guard_abi([&]() -> int {
    if (!f || (bytes && !dst)) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "null argument");
    if (tensor >= f->n) SN_FAIL(SWAPNET_ERR_INVALID_ARG, "tensor index out of range");
    if (offset > f->bytes[tensor] || bytes > f->bytes[tensor] - offset)
      SN_FAIL(SWAPNET_ERR_INVALID_ARG, "range outside the tensor");
    AlignedBuf bounce(kBounce + kFileAlign);
    if (!bounce.p) SN_FAIL(SWAPNET_ERR_OOM, "host allocation failed");
    uint64_t a = f->off[tensor] + offset;
    char* d = static_cast<char*>(dst);
    while (bytes > 0) {
      const uint64_t lo = a / kFileAlign * kFileAlign;
      const uint64_t take = std::min<uint64_t>(bytes, kBounce - (a - lo));
      const uint64_t hi = align_up(a + take, kFileAlign);
      const int e = pread_all(f->fd, bounce.data(), hi - lo, lo);
      if (e) SN_FAIL(SWAPNET_ERR_IO, errno_text("read", e));
      std::memcpy(d, bounce.data() + (a - lo), take);
      d += take;
      a += take;
      bytes -= take;
    }
    return SWAPNET_OK;
  });
}

void swapnet_weights_file_close(swapnet_weights_file* f) {
  if (!f) return;
  if (f->fd >= 0) ::close(f->fd);
  delete f;
}

}  // extern "C"
