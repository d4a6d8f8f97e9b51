// abi.cu -- the C ABI of synverify.h: host-side validation, workspace
// layout, table upload and kernel launches.  No device memory is allocated
// here; every device buffer comes from the caller.  Entry tables larger than
// the launch parameters go up from pinned host staging buffers that the
// library allocates on first need and reuses for the life of the process.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>
#include <new>
#include <vector>

#include "sv_device.cuh"
#include "../../include/sv_io.h"
#include "sv_kernels.h"

namespace sv {

static_assert(sizeof(sv_perturb) == 40, "sv_perturb layout");
static_assert(sizeof(vc_tiles) == 88, "vc_tiles layout");
static_assert(sizeof(syn_spec) == 224, "syn_spec layout");
static_assert(sizeof(vc_pair) == 48, "vc_pair layout");
static_assert(sizeof(vc_result) == 80, "vc_result layout");
static_assert(sizeof(Partial) == 64, "partial record layout");
static_assert(sizeof(DevSpec) == 248, "spec table entry layout");
static_assert(sizeof(DevPair) == 80, "pair table entry layout");

constexpr size_t kAlign = 256;
static size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// ---------------------------------------------------------------------------
// per-device launch shape: one resident wave of each kernel, so every CTA of
// a persistent grid runs at once and the contiguous chunks finish together
// ---------------------------------------------------------------------------
namespace {
struct CapEntry {
  int dev;
  const void* fn;
  uint32_t cap;
};
std::mutex g_mu;
std::vector<CapEntry> g_caps;
}  // namespace

namespace {
std::atomic<uint64_t> g_launches{0};
}
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

namespace {
std::atomic<int> g_fail_launches{0};
}
unsigned launch_block() {
  int n = g_fail_launches.load(std::memory_order_relaxed);
  while (n > 0 && !g_fail_launches.compare_exchange_weak(n, n - 1, std::memory_order_relaxed)) {
  }
  return n > 0 ? 0u : (unsigned)kThreads;
}

uint32_t grid_cap_for(const void* fn, size_t dyn_smem, int block) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 152;
  std::lock_guard<std::mutex> lk(g_mu);
  for (const CapEntry& c : g_caps)
    if (c.dev == dev && c.fn == fn) return c.cap;
  int sms = 0, per_sm = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) sms = 152;
  if (dyn_smem > 0)  // opt in to dynamic shared memory beyond the default 48 KB, once per device
    cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn_smem);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, block, dyn_smem) != cudaSuccess || per_sm <= 0)
    per_sm = 1;
  const uint32_t cap = (uint32_t)std::min<int>(sms * per_sm, (int)kGridCap);
  g_caps.push_back(CapEntry{dev, fn, cap});
  return cap;
}

LaunchShape shape_for(uint64_t units, uint64_t tiles, uint32_t cap, uint64_t align) {
  LaunchShape s{0, 1};
  if (units == 0) return s;
  const uint64_t g = std::min<uint64_t>(std::min<uint64_t>(units, std::max<uint64_t>(tiles, 1)),
                                        std::max<uint32_t>(cap, 1));
  s.chunk = (units + g - 1) / g;
  s.chunk = (s.chunk + align - 1) / align * align;  // slices start on whole loop iterations
  s.grid = (uint32_t)((units + s.chunk - 1) / s.chunk);
  return s;
}

// ---------------------------------------------------------------------------
// validation
// ---------------------------------------------------------------------------
static bool add_ok(uint64_t a, uint64_t b, uint64_t limit) { return a <= limit && b <= limit - a; }

static int check_range(uint64_t off, uint64_t bytes, uint64_t buf) {
  if (off % 16) return SV_EALIGN;
  if (!add_ok(off, bytes, buf)) return SV_ERANGE;
  return SV_OK;
}

static bool valid_rate(double r) { return r >= 0.0 && r <= 1.0; }  // false for NaN

static int check_spec(const syn_spec& s, uint64_t arena) {
  if (s.dtype > SV_U32 || s.dist > SV_FROM_ARENA) return SV_EINVAL;
  const bool fl = is_float((int)s.dtype);
  switch (s.dist) {
    case SV_UNIFORM: case SV_NORMAL: case SV_DOTLIKE: if (!fl) return SV_EINVAL; break;
    case SV_INT_RANGE: case SV_PERMUTATION: if (fl) return SV_EINVAL; break;
    default: break;
  }
  if (s.ref_offset == SV_NO_OUTPUT && s.cand_offset == SV_NO_OUTPUT) return SV_EINVAL;
  if (s.elem_offset % 4) return SV_EALIGN;
  if (!add_ok(s.elem_offset, s.n, SV_MAX_LOGICAL_N)) return SV_ERANGE;
  const uint64_t N = s.logical_n ? s.logical_n : s.elem_offset + s.n;
  if (N > SV_MAX_LOGICAL_N) return SV_ERANGE;
  if (s.elem_offset + s.n > N) return SV_EINVAL;
  const uint64_t bytes = s.n * elem_bytes((int)s.dtype);
  int rc;
  if (s.ref_offset != SV_NO_OUTPUT && (rc = check_range(s.ref_offset, bytes, arena))) return rc;
  if (s.cand_offset != SV_NO_OUTPUT && (rc = check_range(s.cand_offset, bytes, arena))) return rc;
  const uint32_t fmask = SV_SP_NAN | SV_SP_PINF | SV_SP_NINF | SV_SP_DENORM | SV_SP_ZERO | SV_SP_DUP | SV_SP_EXACT;
  const uint32_t imask = SV_SP_ZERO | SV_SP_IMIN | SV_SP_IMAX | SV_SP_DUP | SV_SP_EXACT;
  if (s.special_mask & ~(fl ? fmask : imask)) return SV_EINVAL;
  if (!valid_rate(s.special_rate)) return SV_EINVAL;
  if (exact_special_count(s) > SV_MAX_COUNT) return SV_ERANGE;  // strata indices stay below 2^21
  if ((s.dist == SV_UNIFORM || s.dist == SV_NORMAL) && !(std::isfinite(s.p0) && std::isfinite(s.p1)))
    return SV_EINVAL;  // finite parameters keep every drawn value finite
  if (s.dist == SV_UNIFORM && !(s.p1 >= s.p0)) return SV_EINVAL;
  if (s.dist == SV_INT_RANGE) {
    if (s.i1 < s.i0) return SV_EINVAL;
    if (s.dtype == SV_I32 && (s.i0 < INT32_MIN || s.i1 > INT32_MAX)) return SV_EINVAL;
    if (s.dtype == SV_U32 && (s.i0 < 0 || s.i1 > (int64_t)UINT32_MAX)) return SV_EINVAL;
  }
  if (s.dist == SV_PERMUTATION) {
    if (s.dtype == SV_I32 && N > (1ull << 31)) return SV_ERANGE;
    if (s.dtype == SV_U32 && N > (1ull << 32)) return SV_ERANGE;
  }
  if (s.dist == SV_DOTLIKE) {
    if (s.cols == 0 || s.rows == 0 || s.cols % 4 || s.dot_k == 0 || s.dot_k > (1u << 20)) return SV_EINVAL;
    if (s.rows > N / s.cols || s.rows * s.cols != N) return SV_EINVAL;
    if (s.rows > (1ull << 40) / s.dot_k || s.cols > (1ull << 40) / s.dot_k) return SV_ERANGE;
    if ((rc = check_range(s.a_offset, 4 * s.rows * s.dot_k, arena))) return rc;
    if ((rc = check_range(s.b_offset, 4 * s.dot_k * s.cols, arena))) return rc;
  }
  if (s.dist == SV_FROM_ARENA) {  // the source: the whole logical array, apart from the outputs
    const uint64_t src = N * elem_bytes((int)s.dtype);
    if ((rc = check_range(s.a_offset, src, arena))) return rc;
    auto overlaps = [&](uint64_t off) {
      return off != SV_NO_OUTPUT && bytes && src && off < s.a_offset + src && s.a_offset < off + bytes;
    };
    if (overlaps(s.ref_offset) || overlaps(s.cand_offset)) return SV_EINVAL;
  }
  const sv_perturb& pe = s.pelem;
  if (pe.kind != SV_PERT_NONE && pe.kind != SV_PERT_RATE_ADD_PM && pe.kind != SV_PERT_REL_NOISE) return SV_EINVAL;
  if (pe.kind == SV_PERT_REL_NOISE && !fl) return SV_EINVAL;
  if (pe.kind == SV_PERT_RATE_ADD_PM && !valid_rate(pe.rate)) return SV_EINVAL;
  const sv_perturb& pc = s.pcount;
  if (pc.kind != SV_PERT_NONE && pc.kind != SV_PERT_COUNT_SET && pc.kind != SV_PERT_COUNT_ADD &&
      pc.kind != SV_PERT_SWAP_PAIRS)
    return SV_EINVAL;
  if (pc.kind != SV_PERT_NONE) {
    if (pc.count == 0 || pc.count > SV_MAX_COUNT) return SV_EINVAL;
    const uint64_t strata = pc.kind == SV_PERT_SWAP_PAIRS ? 2 * pc.count : pc.count;
    if (strata > N) return SV_EINVAL;
  }
  return SV_OK;
}

static int check_pair(const vc_pair& p, uint64_t cand_bytes, uint64_t ref_bytes) {
  if (p.dtype > SV_U32) return SV_EINVAL;
  if (p.flags & ~(uint32_t)SV_EQUAL_NAN) return SV_EINVAL;
  if (p.n > SV_MAX_LOGICAL_N) return SV_ERANGE;
  if (is_float((int)p.dtype) && !(p.atol >= 0.0 && p.rtol >= 0.0)) return SV_EINVAL;  // NaN fails too
  const uint64_t bytes = p.n * elem_bytes((int)p.dtype);
  int rc;
  if ((rc = check_range(p.cand_offset, bytes, cand_bytes))) return rc;
  if ((rc = check_range(p.ref_offset, bytes, ref_bytes))) return rc;
  return SV_OK;
}

// a shaped output: geometry, alignment and both operands inside their buffers
static int check_tiles(const vc_tiles& t, uint64_t cand_bytes, uint64_t ref_bytes, uint64_t* n_tiles) {
  if (t.dtype > SV_U32 || (t.flags & ~(uint32_t)SV_EQUAL_NAN)) return SV_EINVAL;
  if (is_float((int)t.dtype) && !(t.atol >= 0.0 && t.rtol >= 0.0)) return SV_EINVAL;
  if (t.tile_rows == 0 || t.tile_cols == 0) return SV_EINVAL;
  if (t.cand_pitch < t.cols || t.ref_pitch < t.cols) return SV_EINVAL;
  const uint64_t sz = elem_bytes((int)t.dtype);
  *n_tiles = 0;
  if (t.rows == 0 || t.cols == 0) return SV_OK;
  const uint64_t th = t.tile_rows < t.rows ? t.tile_rows : t.rows;
  const uint64_t tw = t.tile_cols < t.cols ? t.tile_cols : t.cols;
  if (th > 0x7FFFFFFFull || tw > 0x7FFFFFFFull) return SV_EINVAL;
  if (t.cand_offset % 16 || t.ref_offset % 16) return SV_EALIGN;
  if (t.rows > 1 && ((t.cand_pitch * sz) % 16 || (t.ref_pitch * sz) % 16)) return SV_EALIGN;
  if (t.tile_cols < t.cols && (t.tile_cols * sz) % 16) return SV_EALIGN;
  // a tile that spans rows steps between them with 32-bit byte pitches
  if (th > 1 && (t.cand_pitch * sz > 0xFFFFFFFFull || t.ref_pitch * sz > 0xFFFFFFFFull)) return SV_ERANGE;
  // the last element of each operand: offset + ((rows - 1) * pitch + cols) * size, without overflow
  for (int k = 0; k < 2; ++k) {
    const uint64_t pitch = k ? t.ref_pitch : t.cand_pitch, off = k ? t.ref_offset : t.cand_offset;
    const uint64_t buf = k ? ref_bytes : cand_bytes;
    if (pitch > UINT64_MAX / sz / t.rows) return SV_ERANGE;
    if (!add_ok(off, ((t.rows - 1) * pitch + t.cols) * sz, buf)) return SV_ERANGE;
  }
  const uint64_t ntr = (t.rows + t.tile_rows - 1) / t.tile_rows, ntc = (t.cols + t.tile_cols - 1) / t.tile_cols;
  if (ntr > SV_MAX_TILES || ntc > SV_MAX_TILES || ntr * ntc > SV_MAX_TILES) return SV_ERANGE;
  *n_tiles = ntr * ntc;
  return SV_OK;
}

static int check_specs(const syn_spec* specs, int n, size_t arena) {
  if (n < 0 || n > SV_MAX_ENTRIES || (n > 0 && !specs)) return SV_EINVAL;
  for (int i = 0; i < n; ++i)
    if (int rc = check_spec(specs[i], arena)) return rc;
  return SV_OK;
}

static int check_pairs(const vc_pair* pairs, int n, size_t cb, size_t rb) {
  if (n < 0 || n > SV_MAX_ENTRIES || (n > 0 && !pairs)) return SV_EINVAL;
  for (int i = 0; i < n; ++i)
    if (int rc = check_pair(pairs[i], cb, rb)) return rc;
  return SV_OK;
}

// ---------------------------------------------------------------------------
// tables and workspace layout
//   generate: [spec table, if n > SV_INLINE_ENTRIES]
//   compare:  [pair table, if n > SV_INLINE_ENTRIES][partial slots]
// Entries are stored grouped by kind (stable), one launch per group.
// ---------------------------------------------------------------------------
struct Group {
  uint32_t key;
  int begin, end;  // range in the grouped table
  uint64_t units, tiles;
  LaunchShape sh;
};

// stable grouping by a small key (< kMaxKey; validated dtypes and
// distributions): a counting sort, linear in n
constexpr uint32_t kMaxKey = 64;
template <class KeyFn>
static void group_by(int n, KeyFn key, std::vector<int>& order, std::vector<Group>& groups) {
  uint32_t count[kMaxKey] = {0}, start[kMaxKey];
  for (int i = 0; i < n; ++i) ++count[key(i) % kMaxKey];
  groups.clear();
  uint32_t at = 0;
  for (uint32_t k = 0; k < kMaxKey; ++k) {
    start[k] = at;
    if (count[k]) groups.push_back(Group{k, (int)at, (int)(at + count[k]), 0, 0, {0, 1}});
    at += count[k];
  }
  order.resize(n);
  for (int i = 0; i < n; ++i) order[start[key(i) % kMaxKey]++] = i;
}

// ---------------------------------------------------------------------------
// pinned host staging for entry tables: a buffer is reused once the copy last
// issued from it has completed (an event recorded after that copy); tables
// beyond kMaxStaging, or when pinned memory is unavailable, go up from
// ordinary host memory instead
// ---------------------------------------------------------------------------
namespace {
constexpr size_t kMaxStaging = size_t(16) << 20;
constexpr size_t kMaxStagingBuffers = 64;
struct StagingBuf {
  int dev;
  void* host;
  size_t cap;
  cudaEvent_t done;
  bool claimed;
};
std::mutex g_stage_mu;
std::vector<StagingBuf*> g_stage;  // kept for the life of the process

bool copy_finished(cudaEvent_t e) {
  const cudaError_t q = cudaEventQuery(e);
  if (q == cudaErrorNotReady && cudaPeekAtLastError() == cudaErrorNotReady) cudaGetLastError();
  return q == cudaSuccess;
}

StagingBuf* claim_staging(size_t bytes) {
  int dev = 0;
  if (bytes == 0 || bytes > kMaxStaging || cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  std::lock_guard<std::mutex> lk(g_stage_mu);
  for (StagingBuf* b : g_stage)
    if (b->dev == dev && !b->claimed && b->cap >= bytes && copy_finished(b->done)) {
      b->claimed = true;
      return b;
    }
  if (g_stage.size() >= kMaxStagingBuffers) return nullptr;
  size_t cap = size_t(64) << 10;
  while (cap < bytes) cap *= 2;
  void* h = nullptr;
  if (cudaHostAlloc(&h, cap, cudaHostAllocPortable) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  cudaEvent_t e;
  if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    cudaFreeHost(h);
    return nullptr;
  }
  StagingBuf* b = new StagingBuf{dev, h, cap, e, true};
  g_stage.push_back(b);
  return b;
}

// a host table of n entries of T: pinned when it will be uploaded and fits a
// staging buffer, else ordinary memory; upload() copies it to the device and
// marks the buffer busy until that copy completes
template <class T>
class HostTable {
 public:
  HostTable(int n, bool upload) : n_(n) {
    if (upload) buf_ = claim_staging(sizeof(T) * (size_t)n);
    if (buf_) {
      p_ = static_cast<T*>(buf_->host);
    } else {
      vec_.resize(n);
      p_ = vec_.data();
    }
  }
  ~HostTable() {  // the host copy is read until the call returns
    if (buf_) {
      std::lock_guard<std::mutex> lk(g_stage_mu);
      buf_->claimed = false;
    }
  }
  T* data() { return p_; }
  T& operator[](int i) { return p_[i]; }
  cudaError_t upload(void* dst, cudaStream_t st) {
    const cudaError_t e = cudaMemcpyAsync(dst, p_, sizeof(T) * (size_t)n_, cudaMemcpyHostToDevice, st);
    if (e != cudaSuccess || !buf_) return e;
    return cudaEventRecord(buf_->done, st);
  }

 private:
  int n_;
  StagingBuf* buf_ = nullptr;
  T* p_ = nullptr;
  std::vector<T> vec_;
};
}  // namespace

static size_t spec_table_bytes(int n) { return n > SV_INLINE_ENTRIES ? align_up(sizeof(DevSpec) * (size_t)n) : 0; }
static size_t pair_table_bytes(int n) { return n > SV_INLINE_ENTRIES ? align_up(sizeof(DevPair) * (size_t)n) : 0; }

// partial slots of one group: CTA b of the group writes slot base + b + e for
// its e-th pair, so a group needs grid + n - 1 slots; bounded without a device
// by min(tiles, kGridCap) + n
static size_t compare_partial_bytes(const vc_pair* pairs, int n) {
  uint64_t tiles[8] = {0}, count[8] = {0};
  for (int i = 0; i < n; ++i) {
    tiles[pairs[i].dtype & 7] += cmp_tiles(pairs[i]);
    count[pairs[i].dtype & 7] += 1;
  }
  uint64_t slots = 0;
  for (int d = 0; d < 8; ++d)
    if (count[d]) slots += std::min<uint64_t>(tiles[d], kGridCap) + count[d];
  return align_up(sizeof(Partial) * (size_t)std::max<uint64_t>(slots, 1));
}

static int status_of(cudaError_t e) { return e == cudaSuccess ? SV_OK : SV_ECUDA; }

// base addresses the kernels read and write with vector accesses: element
// buffers 16-byte aligned (128-bit loads and stores at 16-byte offsets),
// result records 8-byte aligned (64-bit fields), the ladder's flag 4-byte
// aligned.  A misaligned base is refused before anything is enqueued, so a
// byte view with an odd storage offset cannot fault the GPU.
static bool misaligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) != 0; }
static int check_bases(const void* cand, const void* ref, const void* results) {
  if (misaligned(cand, 16) || misaligned(ref, 16) || misaligned(results, 8)) return SV_EALIGN;
  return SV_OK;
}

static bool ws_ok(const void* ws, size_t have, size_t need) {
  if (need == 0) return true;
  return ws && have >= need && reinterpret_cast<uintptr_t>(ws) % kAlign == 0;
}

// the plan of one verify_compare: the pair table grouped (many small segments
// to one warp-per-segment launch, key kSmallKey; the rest one launch per
// dtype), each group's launch shape, and every pair's units and partial slots
constexpr uint32_t kSmallKey = 8;

template <class Tab>
static void build_pair_plan(const vc_pair* pairs, int n_pairs, Tab& tab, std::vector<Group>& groups) {
  int n_small = 0;
  for (int i = 0; i < n_pairs; ++i) n_small += cmp_vectors(pairs[i]) <= kSmallVectors;
  const bool split = n_small >= kSmallMinPairs;
  std::vector<int> order;
  group_by(n_pairs, [&](int i) {
    return split && cmp_vectors(pairs[i]) <= kSmallVectors ? kSmallKey : pairs[i].dtype;
  }, order, groups);
  uint64_t slot_base = 0;
  for (Group& g : groups) {
    if (g.key == kSmallKey) {  // one slot each; the combine reads just slot0
      // the warps start in table order: largest segments first (by the
      // power of two of their vector count, a stable linear pass), so that
      // the longest ones do not start last
      std::vector<int> by_size;
      by_size.reserve((size_t)(g.end - g.begin));
      for (int b = 11; b >= 0; --b)
        for (int k = g.begin; k < g.end; ++k) {
          const uint64_t v = cmp_vectors(pairs[order[k]]);
          if ((v == 0 ? 0 : 64 - __builtin_clzll(v)) == b) by_size.push_back(order[k]);
        }
      std::copy(by_size.begin(), by_size.end(), order.begin() + g.begin);
      for (int k = g.begin; k < g.end; ++k) {
        DevPair& d = tab[k];
        d.p = pairs[order[k]];
        d.work_begin = 0;
        d.chunk = ~0ull >> 1;
        d.slot0 = slot_base++;
        d.orig = (uint32_t)order[k];
        d.pad = 0;
      }
      continue;
    }
    for (int k = g.begin; k < g.end; ++k) {
      g.tiles += cmp_tiles(pairs[order[k]]);
      g.units += cmp_units(pairs[order[k]]);
    }
    g.sh = compare_shape(g.key, g.units, g.tiles);
    uint64_t u = 0;
    for (int k = g.begin; k < g.end; ++k) {
      DevPair& d = tab[k];
      d.p = pairs[order[k]];
      d.work_begin = u;
      d.chunk = g.sh.chunk;
      d.slot0 = slot_base + (uint64_t)(k - g.begin);
      d.orig = (uint32_t)order[k];
      d.pad = 0;
      u += cmp_units(d.p);
    }
    slot_base += g.sh.grid + (uint64_t)(g.end - g.begin) - 1;  // slots slot0 + b, b < grid
  }
}

// the launches of a plan: one per group, then the combine
static int run_pair_plan(const DevPair* host, const DevPair* dev, int n_pairs, const std::vector<Group>& groups,
                         Partial* partials, const uint8_t* cand, const uint8_t* ref, vc_result* results,
                         cudaStream_t st) {
  for (const Group& g : groups) {
    const DevPair* h = host + g.begin;
    const DevPair* d = dev ? dev + g.begin : nullptr;
    const cudaError_t e = g.key == kSmallKey
                              ? launch_compare_small(h, d, g.end - g.begin, cand, ref, partials, st)
                              : launch_compare_group(g.key, h, d, g.end - g.begin, g.units, g.sh, cand, ref, partials,
                                                     nullptr, st);
    if (e != cudaSuccess) return SV_ECUDA;
  }
  return status_of(launch_combine(host, dev, n_pairs, partials, results, nullptr, 0, st));
}

// the plan of one syn_generate: the spec table grouped by dtype x
// distribution (stable), each group's weighted units and launch shape, every
// spec's first unit, and its exact-count fixup threads -- edits are applied by
// the generating warps where a warp's slice (at most 4 x chunk elements) meets
// few strata, else by the fixup kernel.  Returns the fixup threads.
template <class Tab>
static uint64_t build_spec_plan(const syn_spec* specs, int n_specs, Tab& tab, std::vector<Group>& groups) {
  std::vector<int> order;
  group_by(n_specs, [&](int i) { return specs[i].dtype * 8u + specs[i].dist; }, order, groups);
  for (Group& g : groups) {
    for (int k = g.begin; k < g.end; ++k) {
      const syn_spec& s = specs[order[k]];
      tab[k].s = s;
      tab[k].work_begin = g.units;
      tab[k].fused = 0;
      tab[k].pad = 0;
      g.units += gen_units(s);
      g.tiles += gen_tiles(s);
    }
    if (g.units) g.sh = generate_shape(tab[g.begin].s.dtype, tab[g.begin].s.dist, g.units, g.tiles);
  }
  uint64_t fixes = 0;
  for (const Group& g : groups) {
    for (int k = g.begin; k < g.end; ++k) {
      DevSpec& d = tab[k];
      d.fix_begin = fixes;
      fixes += fix_special_units(d.s);  // dot-like exact specials: fixup threads
      const uint64_t units = fix_units(d.s);
      if (units == 0) continue;
      const uint64_t N = d.s.logical_n ? d.s.logical_n : d.s.elem_offset + d.s.n;
      if (d.s.dist != SV_DOTLIKE && 4 * g.sh.chunk / N * fix_strata(d.s) +
                                            (4 * g.sh.chunk % N) * fix_strata(d.s) / N + 2 <= kMaxFusedEdits) {
        d.fused = 1;
        continue;
      }
      fixes += units;
    }
  }
  return fixes;
}

// the launches of a generator plan: one per group (one per spec for dot-like
// values), then the fixup
static int run_spec_plan(const DevSpec* host, const DevSpec* dev, int n_specs, const std::vector<Group>& groups,
                         uint64_t fixes, uint8_t* arena, cudaStream_t st) {
  cudaError_t e = cudaSuccess;
  for (const Group& g : groups) {
    const DevSpec& first = host[g.begin];
    if (first.s.dist == SV_DOTLIKE) {
      for (int k = g.begin; e == cudaSuccess && k < g.end; ++k) e = launch_dotlike(host[k], arena, st);
    } else {
      e = launch_generate_group(first.s.dtype, first.s.dist, host + g.begin, dev ? dev + g.begin : nullptr,
                                g.end - g.begin, g.units, g.sh, arena, st);
    }
    if (e != cudaSuccess) return SV_ECUDA;
  }
  return status_of(launch_fixup(host, dev, n_specs, fixes, arena, st));
}

}  // namespace sv

// a prepared syn_generate (synverify.h): the grouped spec table, kept on the
// host for the launch parameters and, beyond SV_INLINE_ENTRIES specs, in the
// caller's workspace for the kernels
struct sv_generate_plan {
  int n = 0;
  size_t arena_bytes = 0;
  int device = -1;
  std::vector<sv::DevSpec> tab;
  std::vector<sv::Group> groups;
  uint64_t fixes = 0;
  const sv::DevSpec* dev_tab = nullptr;
};

// a prepared verify_compare (synverify.h): the grouped table, kept on the host
// for the launch parameters and, beyond SV_INLINE_ENTRIES pairs, in the
// caller's workspace for the kernels
struct sv_compare_plan {
  int n = 0;
  size_t cand_bytes = 0, ref_bytes = 0;
  int device = -1;
  std::vector<sv::DevPair> tab;
  std::vector<sv::Group> groups;
  const sv::DevPair* dev_tab = nullptr;
  sv::Partial* partials = nullptr;
};

using namespace sv;

extern "C" {

int sv_abi_version(void) { return SV_ABI_VERSION; }

uint64_t sv_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

int sv_debug_fail_launches(int n) {
  if (n < 0) return SV_EINVAL;
  g_fail_launches.store(n, std::memory_order_relaxed);
  return SV_OK;
}

int syn_box_muller(const uint32_t* d_words, size_t n_pairs, float* d_z, sv_stream_t stream) {
  if (n_pairs == 0) return SV_OK;
  if (!d_words || !d_z) return SV_EINVAL;
  if (n_pairs > SV_MAX_LOGICAL_N / 2) return SV_ERANGE;
  if ((reinterpret_cast<uintptr_t>(d_words) | reinterpret_cast<uintptr_t>(d_z)) & 7) return SV_EALIGN;
  return status_of(launch_box_muller(d_words, n_pairs, d_z, reinterpret_cast<cudaStream_t>(stream)));
}

int sv_check_tiles(const vc_tiles* tiles, size_t cand_bytes, size_t ref_bytes, uint64_t* n_tiles) {
  uint64_t n = 0;
  if (!tiles) return SV_EINVAL;
  const int rc = check_tiles(*tiles, cand_bytes, ref_bytes, &n);
  if (n_tiles) *n_tiles = rc == SV_OK ? n : 0;
  return rc;
}

int verify_compare_tiles(const vc_tiles* tiles, const void* d_cand, size_t cand_bytes, const void* d_ref,
                         size_t ref_bytes, vc_result* d_results, sv_stream_t stream) {
  if (!tiles) return SV_EINVAL;
  uint64_t n = 0;
  if (int rc = check_tiles(*tiles, cand_bytes, ref_bytes, &n)) return rc;
  if (n == 0) return SV_OK;
  if (!d_cand || !d_ref || !d_results) return SV_EINVAL;
  if ((reinterpret_cast<uintptr_t>(d_cand) | reinterpret_cast<uintptr_t>(d_ref)) & 15) return SV_EALIGN;
  if (reinterpret_cast<uintptr_t>(d_results) & 7) return SV_EALIGN;
  const uint64_t ntc = (tiles->cols + tiles->tile_cols - 1) / tiles->tile_cols;
  return status_of(launch_compare_tiles(*tiles, ntc, n, static_cast<const uint8_t*>(d_cand),
                                        static_cast<const uint8_t*>(d_ref), d_results,
                                        reinterpret_cast<cudaStream_t>(stream)));
}

const char* sv_strerror(int status) {
  switch (status) {
    case SV_OK: return "ok";
    case SV_EINVAL: return "invalid argument (enum, count, tolerance, rate or dtype/dist pairing)";
    case SV_EALIGN: return "misaligned offset (byte offsets must be multiples of 16, elem_offset of 4)";
    case SV_ERANGE: return "data beyond its buffer, or a size beyond the library limits";
    case SV_EWORKSPACE: return "workspace missing, misaligned or too small";
    case SV_ECUDA: return "a CUDA launch or copy failed";
    case SV_EIO: return "a file could not be opened, read, written or sized";
    case SV_EFORMAT: return "bad tensor header, or the file's type, count or size is not the one stated";
    case SV_ELOSSY: return "data loaded, but values were clamped or overflowed by the type conversion";
    default: return "unknown status";
  }
}

int sv_check_specs(const syn_spec* specs, int n_specs, size_t arena_bytes) {
  return check_specs(specs, n_specs, arena_bytes);
}

int sv_check_pairs(const vc_pair* pairs, int n_pairs, size_t cand_bytes, size_t ref_bytes) {
  return check_pairs(pairs, n_pairs, cand_bytes, ref_bytes);
}

size_t sv_generate_workspace_bytes(const syn_spec* specs, int n_specs) {
  if (n_specs < 0 || n_specs > SV_MAX_ENTRIES || (n_specs > 0 && !specs)) return 0;
  return spec_table_bytes(n_specs);
}

size_t sv_compare_workspace_bytes(const vc_pair* pairs, int n_pairs) {
  if (n_pairs < 0 || n_pairs > SV_MAX_ENTRIES || (n_pairs > 0 && !pairs)) return 0;
  for (int i = 0; i < n_pairs; ++i)
    if (pairs[i].dtype > SV_U32) return 0;
  return pair_table_bytes(n_pairs) + compare_partial_bytes(pairs, n_pairs);
}

// Progressive stages run in groups: consecutive stages of one dtype, at most
// SV_INLINE_ENTRIES of them and kStageGroupBytes of data together (a larger
// stage is a group of its own), share one compare launch and one ordered
// combine.  Reading a few small stages together costs less than the launches
// it saves; the fail-fast order is applied inside the group.
constexpr uint64_t kStageGroupBytes = 64ull << 20;

static void stage_groups(const vc_pair* stages, int n, std::vector<std::pair<int, int>>& out) {
  out.clear();
  int b = 0;
  while (b < n) {
    int e = b + 1;
    uint64_t bytes = 2 * stages[b].n * elem_bytes((int)stages[b].dtype);
    while (e < n && e - b < SV_INLINE_ENTRIES && stages[e].dtype == stages[b].dtype) {
      const uint64_t more = 2 * stages[e].n * elem_bytes((int)stages[e].dtype);
      if (bytes + more > kStageGroupBytes) break;
      bytes += more;
      ++e;
    }
    out.emplace_back(b, e);
    b = e;
  }
}

size_t sv_progressive_workspace_bytes(const vc_pair* stages, int n_stages) {
  if (n_stages < 0 || n_stages > SV_MAX_ENTRIES || (n_stages > 0 && !stages)) return 0;
  for (int i = 0; i < n_stages; ++i)
    if (stages[i].dtype > SV_U32) return 0;
  std::vector<std::pair<int, int>> groups;
  stage_groups(stages, n_stages, groups);
  size_t mx = 0;
  for (const auto& g : groups) mx = std::max(mx, compare_partial_bytes(stages + g.first, g.second - g.first));
  return mx;
}

int syn_generate(const syn_spec* specs, int n_specs, void* d_arena, size_t arena_bytes, void* d_ws,
                 size_t ws_bytes, sv_stream_t stream) {
  if (int rc = check_specs(specs, n_specs, arena_bytes)) return rc;
  if (n_specs == 0) return SV_OK;
  if (!d_arena) return SV_EINVAL;
  if (misaligned(d_arena, 16)) return SV_EALIGN;
  const size_t need = spec_table_bytes(n_specs);
  if (!ws_ok(d_ws, ws_bytes, need)) return SV_EWORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  std::vector<Group> groups;
  HostTable<DevSpec> tab(n_specs, need != 0);
  const uint64_t fixes = build_spec_plan(specs, n_specs, tab, groups);
  const DevSpec* dev = nullptr;
  if (need) {
    if (tab.upload(d_ws, st) != cudaSuccess) return SV_ECUDA;
    dev = static_cast<const DevSpec*>(d_ws);
  }
  return run_spec_plan(tab.data(), dev, n_specs, groups, fixes, static_cast<uint8_t*>(d_arena), st);
}

int sv_generate_plan_create(const syn_spec* specs, int n_specs, size_t arena_bytes, void* d_ws, size_t ws_bytes,
                            sv_stream_t stream, sv_generate_plan** plan) {
  if (!plan) return SV_EINVAL;
  *plan = nullptr;
  if (int rc = check_specs(specs, n_specs, arena_bytes)) return rc;
  const size_t need = spec_table_bytes(n_specs);
  if (!ws_ok(d_ws, ws_bytes, need)) return SV_EWORKSPACE;
  sv_generate_plan* p = new (std::nothrow) sv_generate_plan();
  if (!p) return SV_ERANGE;
  p->n = n_specs;
  p->arena_bytes = arena_bytes;
  if (cudaGetDevice(&p->device) != cudaSuccess) p->device = -1;
  if (n_specs > 0) {
    p->tab.resize((size_t)n_specs);
    p->fixes = build_spec_plan(specs, n_specs, p->tab, p->groups);
    if (need) {  // the table goes up once; the plan's launches read it from the workspace
      cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
      if (cudaMemcpyAsync(d_ws, p->tab.data(), sizeof(DevSpec) * (size_t)n_specs, cudaMemcpyHostToDevice, st) !=
              cudaSuccess ||
          cudaStreamSynchronize(st) != cudaSuccess) {
        cudaGetLastError();
        delete p;
        return SV_ECUDA;
      }
      p->dev_tab = static_cast<const DevSpec*>(d_ws);
    }
  }
  *plan = p;
  return SV_OK;
}

int syn_generate_planned(const sv_generate_plan* plan, void* d_arena, sv_stream_t stream) {
  if (!plan) return SV_EINVAL;
  if (plan->n == 0) return SV_OK;
  if (!d_arena) return SV_EINVAL;
  if (misaligned(d_arena, 16)) return SV_EALIGN;
  return run_spec_plan(plan->tab.data(), plan->dev_tab, plan->n, plan->groups, plan->fixes,
                       static_cast<uint8_t*>(d_arena), reinterpret_cast<cudaStream_t>(stream));
}

void sv_generate_plan_destroy(sv_generate_plan* plan) { delete plan; }

int verify_compare(const vc_pair* pairs, int n_pairs, const void* d_cand, size_t cand_bytes, const void* d_ref,
                   size_t ref_bytes, vc_result* d_results, void* d_ws, size_t ws_bytes, sv_stream_t stream) {
  if (int rc = check_pairs(pairs, n_pairs, cand_bytes, ref_bytes)) return rc;
  if (n_pairs == 0) return SV_OK;
  if (!d_results || (cand_bytes && !d_cand) || (ref_bytes && !d_ref)) return SV_EINVAL;
  if (int rc = check_bases(d_cand, d_ref, d_results)) return rc;
  const size_t tb = pair_table_bytes(n_pairs);
  if (!ws_ok(d_ws, ws_bytes, tb + compare_partial_bytes(pairs, n_pairs))) return SV_EWORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  std::vector<Group> groups;
  HostTable<DevPair> tab(n_pairs, tb != 0);
  build_pair_plan(pairs, n_pairs, tab, groups);
  uint8_t* ws = static_cast<uint8_t*>(d_ws);
  const DevPair* dev = nullptr;
  if (tb) {
    if (tab.upload(ws, st) != cudaSuccess) return SV_ECUDA;
    dev = reinterpret_cast<const DevPair*>(ws);
  }
  return run_pair_plan(tab.data(), dev, n_pairs, groups, reinterpret_cast<Partial*>(ws + tb),
                       static_cast<const uint8_t*>(d_cand), static_cast<const uint8_t*>(d_ref), d_results, st);
}

int sv_compare_plan_create(const vc_pair* pairs, int n_pairs, size_t cand_bytes, size_t ref_bytes, void* d_ws,
                           size_t ws_bytes, sv_stream_t stream, sv_compare_plan** plan) {
  if (!plan) return SV_EINVAL;
  *plan = nullptr;
  if (int rc = check_pairs(pairs, n_pairs, cand_bytes, ref_bytes)) return rc;
  const size_t tb = pair_table_bytes(n_pairs);
  if (n_pairs > 0 && !ws_ok(d_ws, ws_bytes, tb + compare_partial_bytes(pairs, n_pairs))) return SV_EWORKSPACE;
  sv_compare_plan* p = new (std::nothrow) sv_compare_plan();
  if (!p) return SV_ERANGE;
  p->n = n_pairs;
  p->cand_bytes = cand_bytes;
  p->ref_bytes = ref_bytes;
  if (cudaGetDevice(&p->device) != cudaSuccess) p->device = -1;
  if (n_pairs > 0) {
    p->tab.resize((size_t)n_pairs);
    build_pair_plan(pairs, n_pairs, p->tab, p->groups);
    uint8_t* ws = static_cast<uint8_t*>(d_ws);
    p->partials = reinterpret_cast<Partial*>(ws + tb);
    if (tb) {  // the table goes up once; the plan's launches read it from the workspace
      cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
      if (cudaMemcpyAsync(ws, p->tab.data(), sizeof(DevPair) * (size_t)n_pairs, cudaMemcpyHostToDevice, st) !=
              cudaSuccess ||
          cudaStreamSynchronize(st) != cudaSuccess) {
        cudaGetLastError();
        delete p;
        return SV_ECUDA;
      }
      p->dev_tab = reinterpret_cast<const DevPair*>(ws);
    }
  }
  *plan = p;
  return SV_OK;
}

int verify_compare_planned(const sv_compare_plan* plan, const void* d_cand, const void* d_ref, vc_result* d_results,
                           sv_stream_t stream) {
  if (!plan) return SV_EINVAL;
  if (plan->n == 0) return SV_OK;
  if (!d_results || (plan->cand_bytes && !d_cand) || (plan->ref_bytes && !d_ref)) return SV_EINVAL;
  if (int rc = check_bases(d_cand, d_ref, d_results)) return rc;
  return run_pair_plan(plan->tab.data(), plan->dev_tab, plan->n, plan->groups, plan->partials,
                       static_cast<const uint8_t*>(d_cand), static_cast<const uint8_t*>(d_ref), d_results,
                       reinterpret_cast<cudaStream_t>(stream));
}

void sv_compare_plan_destroy(sv_compare_plan* plan) { delete plan; }

int verify_progressive(const vc_pair* stages, int n_stages, const void* d_cand, size_t cand_bytes,
                       const void* d_ref, size_t ref_bytes, vc_result* d_results, int32_t* d_first_failed,
                       void* d_ws, size_t ws_bytes, sv_stream_t stream) {
  if (int rc = check_pairs(stages, n_stages, cand_bytes, ref_bytes)) return rc;
  if (!d_first_failed) return SV_EINVAL;
  if (n_stages > 0 && (!d_results || (cand_bytes && !d_cand) || (ref_bytes && !d_ref))) return SV_EINVAL;
  if (misaligned(d_first_failed, 4)) return SV_EALIGN;
  if (int rc = check_bases(d_cand, d_ref, d_results)) return rc;
  if (!ws_ok(d_ws, ws_bytes, sv_progressive_workspace_bytes(stages, n_stages))) return SV_EWORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // the first group's combine sets the flag (failing stage or -1); an empty
  // ladder only clears it
  if (n_stages == 0) return cudaMemsetAsync(d_first_failed, 0xFF, sizeof(int32_t), st) == cudaSuccess ? SV_OK
                                                                                                        : SV_ECUDA;
  Partial* partials = static_cast<Partial*>(d_ws);
  const uint8_t* cand = static_cast<const uint8_t*>(d_cand);
  const uint8_t* ref = static_cast<const uint8_t*>(d_ref);
  std::vector<std::pair<int, int>> groups;
  stage_groups(stages, n_stages, groups);
  for (const auto& g : groups) {
    DevPair tab[SV_INLINE_ENTRIES];
    const int ng = g.second - g.first;
    uint64_t tiles = 0, units = 0;
    for (int k = 0; k < ng; ++k) {
      tiles += cmp_tiles(stages[g.first + k]);
      units += cmp_units(stages[g.first + k]);
    }
    const uint32_t dtype = stages[g.first].dtype;
    const LaunchShape sh = compare_shape(dtype, units, tiles);
    uint64_t u = 0;
    for (int k = 0; k < ng; ++k) {
      tab[k].p = stages[g.first + k];
      tab[k].work_begin = u;
      tab[k].chunk = sh.chunk;
      tab[k].slot0 = (uint64_t)k;
      tab[k].orig = (uint32_t)(g.first + k);
      tab[k].pad = 0;
      u += cmp_units(tab[k].p);
    }
    // the compare of a later group returns at once when an earlier group
    // failed; the combine then reports the group as skipped
    const bool first = g.first == 0;
    cudaError_t e = launch_compare_group(dtype, tab, nullptr, ng, units, sh, cand, ref, partials,
                                         first ? nullptr : d_first_failed, st);
    if (e == cudaSuccess) e = launch_combine(tab, nullptr, ng, partials, d_results, d_first_failed, first, st);
    if (e != cudaSuccess) return SV_ECUDA;
  }
  return SV_OK;
}

}  // extern "C"
