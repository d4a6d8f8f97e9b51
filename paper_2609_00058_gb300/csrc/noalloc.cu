// noalloc.cu -- verify_compare_noalloc: the verify_compare verdicts for
// callers that cannot allocate device memory.
//
// verify_compare needs a caller workspace for its per-CTA partial records.
// Some callers have no way to provide one: code loaded into a host process
// whose device memory is owned and budgeted by another component (a
// framework's caching allocator, a serving runtime that pre-reserves the
// GPU), or code on a latency-critical path that must not pay for an
// allocation and the synchronisation it can imply.  Such a caller only holds
// its inputs and outputs.  This entry point takes exactly those and keeps its
// scratch in a fixed array in this library's device memory instead.
//
// The scratch is a file-scope __device__ array of SV_NOALLOC_SLOTS 64-byte
// partial records (262,656 bytes).  Every GPU that loads the library holds
// one copy of it until the process exits.  Host code cannot use the array's
// name as a device address (on the host it names a stand-in object), so the
// first call on each device looks the address up with cudaGetSymbolAddress,
// with that device current, and caches it.  Every later call on the device
// reuses the same array: calls whose work overlaps on the GPU (different
// streams, or different host threads without ordering) race on it and must
// be serialised by the caller.  Nothing in it needs clearing between calls:
// every partial record a call reads was written earlier in that same call.
// No cudaMalloc, cudaFree or other allocating routine is called.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "sv_kernels.h"

namespace sv {
namespace {

__device__ __align__(256) Partial g_noalloc_scratch[SV_NOALLOC_SLOTS];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
Partial* g_scratch_ptr[kMaxDevices];  // device address per device, nullptr until looked up

// the device address of this device's scratch array (looked up once per device)
int scratch_for_current_device(Partial** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SV_ECUDA;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return SV_ECUDA;
    g_scratch_ptr[dev] = static_cast<Partial*>(p);
  }
  *out = g_scratch_ptr[dev];
  return SV_OK;
}

}  // namespace
}  // namespace sv

extern "C" int verify_compare_noalloc(const vc_pair* pairs, int n_pairs, const void* d_cand, size_t cand_bytes,
                                      const void* d_ref, size_t ref_bytes, vc_result* d_results,
                                      sv_stream_t stream) {
  using namespace sv;
  if (int rc = sv_check_pairs(pairs, n_pairs, cand_bytes, ref_bytes)) return rc;
  if (n_pairs == 0) return SV_OK;
  if (n_pairs > SV_NOALLOC_MAX_PAIRS) return SV_ERANGE;
  if (!d_results || (cand_bytes && !d_cand) || (ref_bytes && !d_ref)) return SV_EINVAL;

  // pairs grouped by dtype (stable), one compare launch per group; a group
  // uses at most min(tiles, kGridCap) CTAs and one slot per (CTA, pair)
  std::vector<int> order(n_pairs);
  for (int i = 0; i < n_pairs; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return pairs[a].dtype < pairs[b].dtype; });
  struct Run {
    uint32_t dtype;
    int begin, end;
    uint64_t tiles, units;
  };
  std::vector<Run> runs;
  for (int k = 0; k < n_pairs; ++k) {
    const vc_pair& p = pairs[order[k]];
    if (runs.empty() || runs.back().dtype != p.dtype) runs.push_back(Run{p.dtype, k, k, 0, 0});
    runs.back().end = k + 1;
    runs.back().tiles += cmp_tiles(p);
    runs.back().units += cmp_units(p);
  }
  uint64_t slots = 0;
  for (const Run& r : runs) slots += std::min<uint64_t>(r.tiles, kGridCap) + (uint64_t)(r.end - r.begin);
  if (slots > SV_NOALLOC_SLOTS) return SV_ERANGE;
  // 128-bit loads from the operands, 64-bit fields in the results: a
  // misaligned base is refused here, before the scratch lookup or any launch
  const uintptr_t operands = reinterpret_cast<uintptr_t>(d_cand) | reinterpret_cast<uintptr_t>(d_ref);
  if ((operands & 15) || (reinterpret_cast<uintptr_t>(d_results) & 7)) return SV_EALIGN;

  Partial* scratch = nullptr;
  if (int rc = scratch_for_current_device(&scratch)) return rc;

  DevPair tab[SV_NOALLOC_MAX_PAIRS];
  std::vector<LaunchShape> shapes(runs.size());
  uint64_t slot_base = 0;
  for (size_t g = 0; g < runs.size(); ++g) {
    const Run& r = runs[g];
    shapes[g] = compare_shape(r.dtype, r.units, r.tiles);
    uint64_t t = 0;
    for (int k = r.begin; k < r.end; ++k) {
      DevPair& d = tab[k];
      d.p = pairs[order[k]];
      d.work_begin = t;
      d.chunk = shapes[g].chunk;
      d.slot0 = slot_base + (uint64_t)(k - r.begin);
      d.orig = (uint32_t)order[k];
      d.pad = 0;
      t += cmp_units(d.p);
    }
    slot_base += shapes[g].grid + (uint64_t)(r.end - r.begin) - 1;  // slots slot0 + b, b < grid
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const uint8_t* cand = static_cast<const uint8_t*>(d_cand);
  const uint8_t* ref = static_cast<const uint8_t*>(d_ref);
  for (size_t g = 0; g < runs.size(); ++g) {
    const Run& r = runs[g];
    if (launch_compare_group(r.dtype, tab + r.begin, nullptr, r.end - r.begin, r.units, shapes[g], cand, ref,
                             scratch, nullptr, st) != cudaSuccess)
      return SV_ECUDA;
  }
  return launch_combine(tab, nullptr, n_pairs, scratch, d_results, nullptr, 0, st) == cudaSuccess ? SV_OK
                                                                                                    : SV_ECUDA;
}
