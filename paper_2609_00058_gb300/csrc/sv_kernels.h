// sv_kernels.h -- launch interface between the C-ABI layer (abi.cu) and the
// kernels (generate.cu, compare.cu).  Internal to the library.
//
// Table entries are grouped by kind on the host (dtype for the compare,
// dtype x distribution for the generator) so that every launch runs one
// template instantiation with its own register budget and occupancy.
#pragma once

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "../../include/synverify.h"

#ifdef __CUDACC__
#define SV_HD __host__ __device__
#else
#define SV_HD
#endif

namespace sv {

constexpr int kThreads = 256;              // threads per CTA of every kernel
constexpr uint32_t kGenTileElems = 8192;   // elements per generator tile
constexpr uint32_t kCmpTileBytes = 16384;  // bytes per operand per compare tile
constexpr uint32_t kGridCap = 4096;        // most persistent CTAs per launch
constexpr int kStagedStarts = 2048;        // tables up to this size are searched in shared memory

// Work is scheduled in weighted units: every entry costs a fixed overhead
// (staging it, building its context, flushing its statistics) plus its
// elements, and each CTA of a persistent grid takes an equal contiguous slice
// of the units, so many small entries spread as evenly as a few large ones.
#ifndef SV_GEN_ENTRY_UNITS
#define SV_GEN_ENTRY_UNITS 2048
#endif
#ifndef SV_CMP_ENTRY_UNITS
#define SV_CMP_ENTRY_UNITS 2048
#endif
constexpr uint64_t kGenEntryUnits = SV_GEN_ENTRY_UNITS;  // generator: units are 4-element quanta
constexpr uint64_t kCmpEntryUnits = SV_CMP_ENTRY_UNITS;  // compare: units are 16-byte vectors

// generator table entry: the caller's spec plus scheduling data
struct DevSpec {
  syn_spec s;
  uint64_t work_begin;  // first unit inside its group's unit range
  uint64_t fix_begin;   // first thread in the exact-count fixup's list
  uint32_t fused;       // exact-count edits applied by the generator CTAs (no fixup threads)
  uint32_t pad;
};

// compare table entry: the caller's pair plus scheduling data
struct DevPair {
  vc_pair p;
  uint64_t work_begin;  // first unit inside its group's unit range
  uint64_t chunk;       // tiles per CTA of its group's launch
  uint64_t slot0;       // partial slot of CTA 0 for this pair (slot0 + b for CTA b)
  uint32_t orig;        // index of the pair in the caller's table (result slot)
  uint32_t pad;
};

// per-CTA partial statistics of one compare segment (64 bytes)
struct Partial {
  uint64_t mism, nan_d, inf_d;
  uint64_t nonfin;  // float types: elements with a NaN or an infinity on a side
  uint64_t first;   // lowest mismatching index, UINT64_MAX if none
  double ssq;       // sum of squared differences
  uint64_t maxabs;  // float types: fp32 bits of max |x-y|; integers: max |x-y|
  double maxrel;
};

struct LaunchShape {
  uint32_t grid;   // CTAs with work
  uint64_t chunk;  // tiles per CTA
};

// persistent grid over `units` weighted units: at most min(cap, tiles) CTAs
// (tiles: 8192-element generator or 16 KiB compare tiles, which bounds the
// grid and so the compare's partial slots), contiguous chunks of units
// (align: the chunk is rounded up to a multiple of it, one loop iteration of
// the kernel, so every slice starts on an iteration boundary)
LaunchShape shape_for(uint64_t units, uint64_t tiles, uint32_t cap, uint64_t align);
// SMs x resident CTAs of this kernel at `block` threads per CTA (cached per
// device), at most kGridCap
uint32_t grid_cap_for(const void* kernel, size_t dyn_smem = 0, int block = kThreads);
// a launch in a chain of this library's kernels (programmatic dependent
// launch, sm_90+): the kernel may be scheduled while the previous kernel of
// the stream still runs, so its launch latency and ramp overlap that
// kernel's tail; it starts with pdl_wait() (griddepcontrol.wait), which
// returns once the previous kernel has completed and its stores are visible,
// so no data dependency changes.  Errors as for <<<>>>.
template <typename P>
inline cudaError_t launch_chained(void (*kernel)(P), unsigned grid, unsigned block, cudaStream_t st, const P& p) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, p);
  const cudaError_t last = cudaGetLastError();  // clears what the launch left
  return e != cudaSuccess ? e : last;
}
// one more kernel launched by this library (the sv_kernel_launches counter)
void count_launch();
// the block size of every launch: kThreads, or 0 (an invalid configuration,
// so the launch fails and no kernel runs) while sv_debug_fail_launches has
// failures pending
unsigned launch_block();

SV_HD inline uint64_t cmp_tiles(const vc_pair& p) {
  const uint64_t sz = p.dtype == SV_I64 ? 8 : ((p.dtype == SV_F16 || p.dtype == SV_BF16) ? 2 : 4);
  return (p.n * sz + kCmpTileBytes - 1) / kCmpTileBytes;
}
SV_HD inline uint64_t cmp_vectors(const vc_pair& p) {
  const uint64_t sz = p.dtype == SV_I64 ? 8 : ((p.dtype == SV_F16 || p.dtype == SV_BF16) ? 2 : 4);
  return (p.n * sz + 15) / 16;
}
SV_HD inline uint64_t cmp_units(const vc_pair& p) { return kCmpEntryUnits + cmp_vectors(p); }
SV_HD inline uint64_t gen_tiles(const syn_spec& s) {
  return s.dist == SV_DOTLIKE ? 0 : (s.n + kGenTileElems - 1) / kGenTileElems;
}
SV_HD inline uint64_t gen_units(const syn_spec& s) {
  return s.dist == SV_DOTLIKE ? 0 : kGenEntryUnits + (s.n + 3) / 4;
}
// exact-count edits a generator CTA applies itself, at most, per entry it
// touches (more strata than this in a CTA's slice: the fixup kernel does them)
constexpr int kMaxFusedEdits = 64;

SV_HD inline uint64_t fix_units(const syn_spec& s) {
  if (s.cand_offset == SV_NO_OUTPUT) return 0;
  const uint32_t k = s.pcount.kind;
  return (k == SV_PERT_COUNT_SET || k == SV_PERT_COUNT_ADD || k == SV_PERT_SWAP_PAIRS) ? s.pcount.count : 0;
}


// exact-count special values of a spec: round(rate * N), at most N (the
// same fp64 steps on the host and the device); 0 in the Bernoulli mode or
// with no kind in the mask
SV_HD inline uint64_t exact_special_count(const syn_spec& s) {
  if (!(s.special_mask & SV_SP_EXACT) || !(s.special_mask & SV_SP_KINDS) || !(s.special_rate > 0.0)) return 0;
  const uint64_t N = s.logical_n ? s.logical_n : s.elem_offset + s.n;
  const double k = floor(s.special_rate * (double)N + 0.5);
  return k >= (double)N ? N : (uint64_t)k;
}

// fixup threads that write exact-count special values: the dot-like values'
// (their generator writes none); the streaming generator's CTAs write their own
SV_HD inline uint64_t fix_special_units(const syn_spec& s) {
  return s.dist == SV_DOTLIKE ? exact_special_count(s) : 0;
}

// strata the exact-count edits cut [0, N) into (two per swapped pair)
SV_HD inline uint64_t fix_strata(const syn_spec& s) {
  return s.pcount.kind == SV_PERT_SWAP_PAIRS ? 2 * s.pcount.count : s.pcount.count;
}

// ---- generator ----
LaunchShape generate_shape(uint32_t dtype, uint32_t dist, uint64_t units, uint64_t tiles);
// entries: either host (n <= SV_INLINE_ENTRIES, copied into the launch) or device
cudaError_t launch_generate_group(uint32_t dtype, uint32_t dist, const DevSpec* host, const DevSpec* dev, int n,
                                  uint64_t units, LaunchShape sh, uint8_t* arena, cudaStream_t st);
cudaError_t launch_fixup(const DevSpec* host, const DevSpec* dev, int n, uint64_t units, uint8_t* arena,
                         cudaStream_t st);
cudaError_t launch_dotlike(const DevSpec& spec, uint8_t* arena, cudaStream_t st);
cudaError_t launch_box_muller(const uint32_t* words, uint64_t n_pairs, float* z, cudaStream_t st);

// ---- compare ----
LaunchShape compare_shape(uint32_t dtype, uint64_t units, uint64_t tiles);
cudaError_t launch_compare_group(uint32_t dtype, const DevPair* host, const DevPair* dev, int n, uint64_t units,
                                 LaunchShape sh, const uint8_t* cand, const uint8_t* ref, Partial* partials,
                                 const int32_t* flag, cudaStream_t st);
// many small segments of any dtypes, one warp each (at most kSmallVectors vectors per segment)
constexpr uint64_t kSmallVectors = 1024;
constexpr int kSmallMinPairs = 64;  // below this many, small segments stay in their dtype groups
cudaError_t launch_compare_small(const DevPair* host, const DevPair* dev, int n, const uint8_t* cand,
                                 const uint8_t* ref, Partial* partials, cudaStream_t st);
cudaError_t launch_combine(const DevPair* host, const DevPair* dev, int n, const Partial* partials,
                           vc_result* results, int32_t* flag, int first_group, cudaStream_t st);

// shaped outputs: one CTA per tile (grid-stride); ntc tiles per tile row
cudaError_t launch_compare_tiles(const vc_tiles& t, uint64_t ntc, uint64_t n_tiles, const uint8_t* cand,
                                 const uint8_t* ref, vc_result* results, cudaStream_t st);

// ---- value conversion of test data (convert.cu) ----
// n elements of type s at src become n elements of type d at dst (16-byte
// aligned, s != d, not float -> integer); clamped or overflowed values are
// added to *lost
cudaError_t launch_convert(int s, int d, const void* src, void* dst, uint64_t n, unsigned long long* lost,
                           cudaStream_t st);

}  // namespace sv
