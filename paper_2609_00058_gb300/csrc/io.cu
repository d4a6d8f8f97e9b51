// io.cu -- the test-data I/O of sv_io.h: the scaffold's read and write
// helpers (Sec. 4.1.2) made dtype-correct (Sec. 5.2.3).
//
// A file moves in chunks through SV_IO_SLOTS pinned host buffers.  A pool of
// host threads reads the stripes of one chunk in parallel while the chunks
// before it cross the NVLink-C2C link with cudaMemcpyAsync and, when the
// element types differ, are converted on the GPU (convert.cu) from a
// two-chunk staging area in the caller's workspace.  Writes run the other
// way, one writer thread per chunk while later chunks come back from the GPU.
// A pinned buffer is reused only after an event shows that the copy out of
// (or into) it is done.
#include <cuda_runtime.h>
#include <errno.h>
#include <fcntl.h>
#include <sys/stat.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <condition_variable>
#include <cstring>
#include <functional>
#include <mutex>
#include <thread>
#include <vector>

#include "../../include/sv_io.h"
#include "sv_kernels.h"

namespace sv {
namespace {

static_assert(sizeof(sv_tensor_header) == SV_TENSOR_HEADER_BYTES, "tensor header layout");

constexpr uint64_t kStripeMin = 1u << 20;  // smallest file stripe given to one host thread
constexpr uint64_t kStageAlign = 256;

int dtype_bytes(int t) {
  switch (t) {
    case SV_F32: case SV_I32: case SV_U32: return 4;
    case SV_F16: case SV_BF16: case SV_I16: case SV_U16: return 2;
    case SV_I64: case SV_U64: case SV_F64: return 8;
    case SV_U8: case SV_I8: return 1;
    default: return 0;
  }
}

bool is_float_type(int t) { return t == SV_F32 || t == SV_F16 || t == SV_BF16 || t == SV_F64; }

// ---- a pool of host threads; the caller works too ----
class Pool {
 public:
  Pool() {
    const unsigned hc = std::thread::hardware_concurrency();
    const unsigned n = hc > 1 ? std::min(hc - 1, 15u) : 0u;
    for (unsigned i = 0; i < n; ++i) th_.emplace_back([this] { loop(); });
    for (auto& t : th_) t.detach();  // the pool lives as long as the process
  }
  int threads() const { return (int)th_.size() + 1; }

  // fn(i) for every i in [0, tasks); returns when all have run
  void run(int tasks, const std::function<void(int)>& fn) {
    std::unique_lock<std::mutex> lk(mu_);
    idle_.wait(lk, [&] { return active_ == 0; });  // no worker still holds the previous job
    fn_ = &fn;
    tasks_ = tasks;
    done_ = 0;
    next_.store(0);
    ++gen_;
    lk.unlock();
    wake_.notify_all();
    int finished = 0;
    for (int i; (i = next_.fetch_add(1)) < tasks;) {
      fn(i);
      ++finished;
    }
    lk.lock();
    done_ += finished;
    idle_.wait(lk, [&] { return done_ == tasks && active_ == 0; });
  }

 private:
  void loop() {
    uint64_t seen = 0;
    std::unique_lock<std::mutex> lk(mu_);
    for (;;) {
      wake_.wait(lk, [&] { return gen_ != seen; });
      seen = gen_;
      const std::function<void(int)>* fn = fn_;
      const int tasks = tasks_;
      ++active_;
      lk.unlock();
      int finished = 0;
      for (int i; (i = next_.fetch_add(1)) < tasks;) {  // a late worker finds nothing left
        (*fn)(i);
        ++finished;
      }
      lk.lock();
      done_ += finished;
      --active_;
      idle_.notify_all();
    }
  }

  std::vector<std::thread> th_;
  std::mutex mu_;
  std::condition_variable wake_, idle_;
  const std::function<void(int)>* fn_ = nullptr;
  int tasks_ = 0, done_ = 0, active_ = 0;
  uint64_t gen_ = 0;
  std::atomic<int> next_{0};
};

Pool& pool() {
  static Pool* p = new Pool();
  return *p;
}

// ---- pinned chunk buffers (process lifetime) ----
std::mutex g_io;  // one I/O call at a time: the buffers and the pool are shared
std::atomic<uint64_t> g_chunk{SV_IO_CHUNK_BYTES};

struct Pinned {
  uint8_t* base = nullptr;
  uint8_t* slot(int i) const { return base + (size_t)i * SV_IO_CHUNK_BYTES; }
  unsigned long long* lost() const {
    return reinterpret_cast<unsigned long long*>(base + (size_t)SV_IO_SLOTS * SV_IO_CHUNK_BYTES);
  }
};

bool pinned(Pinned& out) {  // under g_io
  static Pinned p;
  if (!p.base) {
    void* b = nullptr;
    if (cudaHostAlloc(&b, (size_t)SV_IO_SLOTS * SV_IO_CHUNK_BYTES + 64, cudaHostAllocPortable) != cudaSuccess) {
      cudaGetLastError();
      return false;
    }
    p.base = static_cast<uint8_t*>(b);
  }
  out = p;
  return true;
}

struct Fd {
  int fd = -1;
  ~Fd() {
    if (fd >= 0) close(fd);
  }
};

struct Events {
  cudaEvent_t ev[SV_IO_SLOTS + 1] = {};
  bool ok = true;
  Events() {
    for (auto& e : ev) ok = ok && cudaEventCreateWithFlags(&e, cudaEventDisableTiming) == cudaSuccess;
  }
  ~Events() {
    for (auto& e : ev)
      if (e) cudaEventDestroy(e);
  }
};

int pread_all(int fd, uint8_t* dst, uint64_t off, uint64_t len) {
  while (len) {
    const ssize_t r = pread(fd, dst, (size_t)std::min<uint64_t>(len, 1u << 30), (off_t)off);
    if (r < 0 && errno == EINTR) continue;
    if (r <= 0) return SV_EIO;  // an error, or the file ended early
    dst += r;
    off += (uint64_t)r;
    len -= (uint64_t)r;
  }
  return SV_OK;
}

int pwrite_all(int fd, const uint8_t* src, uint64_t off, uint64_t len) {
  while (len) {
    const ssize_t r = pwrite(fd, src, (size_t)std::min<uint64_t>(len, 1u << 30), (off_t)off);
    if (r < 0 && errno == EINTR) continue;
    if (r <= 0) return SV_EIO;
    src += r;
    off += (uint64_t)r;
    len -= (uint64_t)r;
  }
  return SV_OK;
}

// one chunk's bytes moved by the pool in stripes of at least kStripeMin.
// Writes take one thread: file systems serialise writers of one file (one and
// sixteen pwrite threads reached the same rate where this was measured).
int parallel_io(bool write, int fd, uint8_t* buf, uint64_t off, uint64_t len) {
  if (write) return pwrite_all(fd, buf, off, len);
  const uint64_t want = std::max<uint64_t>(1, len / kStripeMin);
  const int stripes = (int)std::min<uint64_t>(want, (uint64_t)pool().threads());
  const uint64_t stripe = ((len + stripes - 1) / stripes + 4095) / 4096 * 4096;
  std::atomic<int> err{SV_OK};
  pool().run(stripes, [&](int i) {
    const uint64_t b = (uint64_t)i * stripe;
    if (b >= len) return;
    const uint64_t l = std::min(stripe, len - b);
    const int rc = pread_all(fd, buf + b, off + b, l);
    if (rc != SV_OK) err.store(rc);
  });
  return err.load();
}

bool mul_ok(uint64_t a, uint64_t b, uint64_t* out) {
  if (a != 0 && b > UINT64_MAX / a) return false;
  *out = a * b;
  return true;
}

// read and check the header of an open tensor file of `fsize` bytes
int read_header(int fd, uint64_t fsize, sv_tensor_header* h) {
  if (fsize < SV_TENSOR_HEADER_BYTES) return SV_EFORMAT;
  if (pread_all(fd, reinterpret_cast<uint8_t*>(h), 0, SV_TENSOR_HEADER_BYTES) != SV_OK) return SV_EIO;
  if (h->magic != SV_TENSOR_MAGIC || h->header_bytes != SV_TENSOR_HEADER_BYTES) return SV_EFORMAT;
  const int sz = dtype_bytes((int)h->dtype);
  if (sz == 0 || h->ndim > SV_TENSOR_MAX_DIMS) return SV_EFORMAT;
  uint64_t n = 1;
  for (uint32_t i = 0; i < SV_TENSOR_MAX_DIMS; ++i) {
    if (i >= h->ndim) {
      if (h->shape[i] != 0) return SV_EFORMAT;
    } else if (!mul_ok(n, h->shape[i], &n)) {
      return SV_EFORMAT;
    }
  }
  for (uint64_t r : h->reserved)
    if (r != 0) return SV_EFORMAT;
  uint64_t bytes = 0;
  if (h->n != n || !mul_ok(n, (uint64_t)sz, &bytes) || h->data_bytes != bytes) return SV_EFORMAT;
  if (fsize != SV_TENSOR_HEADER_BYTES + bytes) return SV_EFORMAT;
  return SV_OK;
}

int open_regular(const char* path, int flags, Fd& f, uint64_t* size) {
  f.fd = open(path, flags | O_CLOEXEC, 0644);
  if (f.fd < 0) return SV_EIO;
  struct stat st;
  if (fstat(f.fd, &st) != 0 || !S_ISREG(st.st_mode)) return SV_EIO;
  if (size) *size = (uint64_t)st.st_size;
  return SV_OK;
}

uint64_t stage_bytes(uint64_t total) {  // one half of the conversion staging area
  return std::min<uint64_t>(SV_IO_CHUNK_BYTES, (total + kStageAlign - 1) / kStageAlign * kStageAlign);
}

}  // namespace
}  // namespace sv

using namespace sv;

extern "C" {

int sv_dtype_bytes(int dtype) { return dtype_bytes(dtype); }

int sv_debug_io_chunk_bytes(size_t bytes) {
  if (bytes == 0) bytes = SV_IO_CHUNK_BYTES;
  if (bytes % 4096 != 0 || bytes > SV_IO_CHUNK_BYTES) return SV_EINVAL;
  g_chunk.store(bytes);
  return SV_OK;
}

int sv_tensor_probe(const char* path, sv_tensor_header* out) {
  if (!path || !out) return SV_EINVAL;
  Fd f;
  uint64_t size = 0;
  int rc = open_regular(path, O_RDONLY, f, &size);
  if (rc != SV_OK) return rc;
  sv_tensor_header h;
  rc = read_header(f.fd, size, &h);
  if (rc == SV_OK) *out = h;
  return rc;
}

size_t sv_io_workspace_bytes(int src_dtype, int dst_dtype, uint64_t n) {
  const int ss = dtype_bytes(src_dtype);
  if (ss == 0 || dtype_bytes(dst_dtype) == 0) return 0;
  if (src_dtype == dst_dtype || n == 0 || n > SV_MAX_LOGICAL_N) return 0;
  return (size_t)(kStageAlign + 2 * stage_bytes(n * (uint64_t)ss));
}

int sv_convert(int src_dtype, const void* d_src, uint64_t n, int dst_dtype, void* d_dst, uint64_t* d_lost,
               sv_stream_t stream) {
  const int ss = dtype_bytes(src_dtype), ds = dtype_bytes(dst_dtype);
  if (ss == 0 || ds == 0) return SV_EINVAL;
  if (is_float_type(src_dtype) && !is_float_type(dst_dtype)) return SV_EINVAL;
  if (n > SV_MAX_LOGICAL_N) return SV_ERANGE;
  if (n == 0) return SV_OK;
  if (!d_src || !d_dst) return SV_EINVAL;
  if (reinterpret_cast<uintptr_t>(d_src) % 16 || reinterpret_cast<uintptr_t>(d_dst) % 16 ||
      reinterpret_cast<uintptr_t>(d_lost) % 8)
    return SV_EALIGN;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (src_dtype == dst_dtype) {
    e = cudaMemcpyAsync(d_dst, d_src, n * (uint64_t)ss, cudaMemcpyDeviceToDevice, st);
  } else {
    if (!d_lost) return SV_EINVAL;
    e = launch_convert(src_dtype, dst_dtype, d_src, d_dst, n, reinterpret_cast<unsigned long long*>(d_lost), st);
  }
  return e == cudaSuccess ? SV_OK : SV_ECUDA;
}

int sv_read_tensor(const char* path, uint32_t flags, int file_dtype, uint64_t n_expect, int dst_dtype, void* d_dst,
                   size_t dst_bytes, void* d_ws, size_t ws_bytes, sv_stream_t stream, sv_tensor_header* out_header,
                   uint64_t* n_lost) {
  if (n_lost) *n_lost = 0;
  if (!path || (flags & ~(uint32_t)(SV_IO_RAW | SV_IO_STRICT)) || dtype_bytes(dst_dtype) == 0) return SV_EINVAL;
  const bool raw = flags & SV_IO_RAW;
  if (raw ? dtype_bytes(file_dtype) == 0 : (file_dtype != -1 && dtype_bytes(file_dtype) == 0)) return SV_EINVAL;
  std::lock_guard<std::mutex> lk(g_io);
  Fd f;
  uint64_t fsize = 0;
  int rc = open_regular(path, O_RDONLY, f, &fsize);
  if (rc != SV_OK) return rc;
  sv_tensor_header h;
  std::memset(&h, 0, sizeof h);
  uint64_t data_off = 0;
  if (raw) {
    const uint64_t sz = (uint64_t)dtype_bytes(file_dtype);
    if (fsize % sz != 0) return SV_EFORMAT;
    h.magic = SV_TENSOR_MAGIC;
    h.header_bytes = SV_TENSOR_HEADER_BYTES;
    h.dtype = (uint32_t)file_dtype;
    h.ndim = 1;
    h.shape[0] = h.n = fsize / sz;
    h.data_bytes = fsize;
  } else {
    rc = read_header(f.fd, fsize, &h);
    if (rc != SV_OK) return rc;
    if (file_dtype != -1 && (int)h.dtype != file_dtype) return SV_EFORMAT;
    data_off = SV_TENSOR_HEADER_BYTES;
  }
  if (n_expect != 0 && h.n != n_expect) return SV_EFORMAT;
  const int s = (int)h.dtype;
  if ((flags & SV_IO_STRICT) && s != dst_dtype) return SV_EFORMAT;
  if (is_float_type(s) && !is_float_type(dst_dtype)) return SV_EINVAL;
  const uint64_t n = h.n, ss = (uint64_t)dtype_bytes(s), ds = (uint64_t)dtype_bytes(dst_dtype);
  if (n > SV_MAX_LOGICAL_N) return SV_ERANGE;
  if (n && !d_dst) return SV_EINVAL;
  if (reinterpret_cast<uintptr_t>(d_dst) % 16) return SV_EALIGN;
  if (n * ds > dst_bytes) return SV_ERANGE;
  const bool conv = s != dst_dtype;
  const uint64_t total = n * ss;
  if (conv && n) {
    if (!d_ws || reinterpret_cast<uintptr_t>(d_ws) % kStageAlign ||
        ws_bytes < sv_io_workspace_bytes(s, dst_dtype, n))
      return SV_EWORKSPACE;
  }
  if (out_header) *out_header = h;
  if (n == 0) return SV_OK;

  Pinned P;
  if (!pinned(P)) return SV_ECUDA;
  Events E;
  if (!E.ok) return SV_ECUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint8_t* dst = static_cast<uint8_t*>(d_dst);
  uint8_t* ws = static_cast<uint8_t*>(d_ws);
  unsigned long long* lost_dev = conv ? reinterpret_cast<unsigned long long*>(ws) : nullptr;
  const uint64_t chunk = g_chunk.load(), half = stage_bytes(total);
  cudaError_t ce = cudaSuccess;
  if (conv) ce = cudaMemsetAsync(lost_dev, 0, sizeof(unsigned long long), st);
  uint64_t k = 0;
  for (uint64_t off = 0; off < total && ce == cudaSuccess && rc == SV_OK; off += chunk, ++k) {
    const int slot = (int)(k % SV_IO_SLOTS);
    if (k >= SV_IO_SLOTS && (ce = cudaEventSynchronize(E.ev[slot])) != cudaSuccess) break;  // its copy is done
    const uint64_t len = std::min(chunk, total - off);
    rc = parallel_io(false, f.fd, P.slot(slot), data_off + off, len);
    if (rc != SV_OK) break;
    if (!conv) {
      ce = cudaMemcpyAsync(dst + off, P.slot(slot), len, cudaMemcpyHostToDevice, st);
    } else {
      uint8_t* stage = ws + kStageAlign + (k % 2) * half;
      ce = cudaMemcpyAsync(stage, P.slot(slot), len, cudaMemcpyHostToDevice, st);
      if (ce == cudaSuccess) ce = launch_convert(s, dst_dtype, stage, dst + off / ss * ds, len / ss, lost_dev, st);
    }
    if (ce == cudaSuccess) ce = cudaEventRecord(E.ev[slot], st);
  }
  // always drain: no copy out of a pinned buffer may outlive the call
  if (conv && ce == cudaSuccess && rc == SV_OK)
    ce = cudaMemcpyAsync(P.lost(), lost_dev, sizeof(unsigned long long), cudaMemcpyDeviceToHost, st);
  cudaError_t de = cudaEventRecord(E.ev[SV_IO_SLOTS], st);
  if (de == cudaSuccess) de = cudaEventSynchronize(E.ev[SV_IO_SLOTS]);
  if (de != cudaSuccess) cudaStreamSynchronize(st);
  if (ce != cudaSuccess || de != cudaSuccess) {
    cudaGetLastError();
    return SV_ECUDA;
  }
  if (rc != SV_OK) return rc;
  if (conv) {
    const uint64_t lost = *P.lost();
    if (n_lost) *n_lost = lost;
    if (lost) return SV_ELOSSY;
  }
  return SV_OK;
}

int sv_write_tensor(const char* path, uint32_t flags, int dtype, const uint64_t* shape, int ndim, const void* d_src,
                    size_t src_bytes, sv_stream_t stream) {
  const int sz = dtype_bytes(dtype);
  if (!path || sz == 0 || (flags & ~(uint32_t)SV_IO_RAW) || ndim < 0 || ndim > SV_TENSOR_MAX_DIMS ||
      (ndim > 0 && !shape))
    return SV_EINVAL;
  sv_tensor_header h;
  std::memset(&h, 0, sizeof h);
  h.magic = SV_TENSOR_MAGIC;
  h.header_bytes = SV_TENSOR_HEADER_BYTES;
  h.dtype = (uint32_t)dtype;
  h.ndim = (uint32_t)ndim;
  uint64_t n = 1;
  for (int i = 0; i < ndim; ++i) {
    h.shape[i] = shape[i];
    if (!mul_ok(n, shape[i], &n)) return SV_ERANGE;
  }
  if (n > SV_MAX_LOGICAL_N) return SV_ERANGE;
  h.n = n;
  h.data_bytes = n * (uint64_t)sz;
  if (n && !d_src) return SV_EINVAL;
  if (reinterpret_cast<uintptr_t>(d_src) % 16) return SV_EALIGN;
  if (h.data_bytes > src_bytes) return SV_ERANGE;
  std::lock_guard<std::mutex> lk(g_io);
  Fd f;
  int rc = open_regular(path, O_WRONLY | O_CREAT | O_TRUNC, f, nullptr);
  if (rc != SV_OK) return rc;
  const uint64_t data_off = (flags & SV_IO_RAW) ? 0 : SV_TENSOR_HEADER_BYTES;
  if (data_off && (rc = pwrite_all(f.fd, reinterpret_cast<const uint8_t*>(&h), 0, sizeof h)) != SV_OK) return rc;
  if (n == 0) {
    const int fd = f.fd;
    f.fd = -1;
    return close(fd) == 0 ? (int)SV_OK : (int)SV_EIO;
  }

  Pinned P;
  if (!pinned(P)) return SV_ECUDA;
  Events E;
  if (!E.ok) return SV_ECUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const uint8_t* src = static_cast<const uint8_t*>(d_src);
  const uint64_t total = h.data_bytes, chunk = g_chunk.load();
  const uint64_t n_chunks = (total + chunk - 1) / chunk;
  cudaError_t ce = cudaSuccess;
  auto issue = [&](uint64_t k) {
    const int slot = (int)(k % SV_IO_SLOTS);
    const uint64_t off = k * chunk, len = std::min(chunk, total - off);
    ce = cudaMemcpyAsync(P.slot(slot), src + off, len, cudaMemcpyDeviceToHost, st);
    if (ce == cudaSuccess) ce = cudaEventRecord(E.ev[slot], st);
  };
  for (uint64_t k = 0; k < std::min<uint64_t>(SV_IO_SLOTS, n_chunks) && ce == cudaSuccess; ++k) issue(k);
  for (uint64_t k = 0; k < n_chunks && ce == cudaSuccess && rc == SV_OK; ++k) {
    const int slot = (int)(k % SV_IO_SLOTS);
    if ((ce = cudaEventSynchronize(E.ev[slot])) != cudaSuccess) break;
    const uint64_t off = k * chunk, len = std::min(chunk, total - off);
    rc = parallel_io(true, f.fd, P.slot(slot), data_off + off, len);
    if (rc == SV_OK && k + SV_IO_SLOTS < n_chunks) issue(k + SV_IO_SLOTS);
  }
  cudaError_t de = cudaEventRecord(E.ev[SV_IO_SLOTS], st);  // drain the copies still in flight
  if (de == cudaSuccess) de = cudaEventSynchronize(E.ev[SV_IO_SLOTS]);
  if (de != cudaSuccess) cudaStreamSynchronize(st);
  if (ce != cudaSuccess || de != cudaSuccess) {
    cudaGetLastError();
    return SV_ECUDA;
  }
  if (rc != SV_OK) return rc;
  const int fd = f.fd;
  f.fd = -1;
  return close(fd) == 0 ? (int)SV_OK : (int)SV_EIO;
}

}  // extern "C"
