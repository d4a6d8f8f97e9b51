// compare.cu -- verify_compare / verify_progressive kernels: functional
// validation by Eq. 1 of CUDA-Harness (Sec. 4.2.1), per segment, sm_103a.
//
//   cmp_kernel      persistent; CTA b owns the contiguous slice
//                   [b*chunk, (b+1)*chunk) of the weighted work units (a fixed
//                   cost per segment plus its 16-byte vectors; 16 KiB per
//                   operand per loop iteration).  Four 128-bit loads per operand per
//                   thread are issued before any arithmetic; each element is
//                   tested with explicit fp32 round-to-nearest operations.
//                   Statistics stay in registers until the segment ends in
//                   this CTA's run, then warp shuffles and one shared-memory
//                   pass give one 64-byte partial, written to slot b + segment
//                   (unique: runs are contiguous and ordered).  No atomics.
//   combine_kernel  one warp per segment folds its partials in CTA order
//                   (deterministic) and writes the vc_result.
//
// For the progressive ladder (Sec. 4.2.2) both kernels take a device flag:
// once a stage has failed, later stages return at once.
//
// Bound: HBM reads, 2 * n * sizeof(element) per segment.
#include <float.h>

#include "sv_device.cuh"
#include "sv_kernels.h"

namespace sv {

struct CmpParams {
  const DevPair* tab;  // device table, or nullptr: use inl
  DevPair inl[SV_INLINE_ENTRIES];
  int n;
  uint64_t total, chunk;
  const uint8_t* cand;
  const uint8_t* ref;
  Partial* partials;
  const int32_t* flag;  // progressive: skip when *flag >= 0
};

struct CombParams {
  const DevPair* tab;
  DevPair inl[SV_INLINE_ENTRIES];
  int n;
  const Partial* partials;
  vc_result* results;
  int32_t* flag;
  int first_group;  // progressive: the ladder's first group (the flag is not yet set)
};

template <class P>
__device__ __forceinline__ const DevPair* pentry(const P& p, int i) { return p.tab ? p.tab + i : p.inl + i; }

// ---------------------------------------------------------------------------
// per-thread accumulators
// ---------------------------------------------------------------------------
struct Acc {
  uint32_t mism, nan_d, inf_d, nonfin;  // nonfin: float elements outside the both-finite set
  uint64_t first;
  double ssq;
  float maxabs_f, maxrel_f;  // float types
  float relthr;              // float types: a max |x-y|/|y| already reached (the warp's), see float_vector
  uint64_t maxabs_u;         // integer types
  double maxrel_d;           // integer types
};

__device__ __forceinline__ void acc_reset(Acc& a) {
  a.mism = a.nan_d = a.inf_d = a.nonfin = 0;
  a.first = ~0ull;
  a.ssq = 0.0;
  a.maxabs_f = a.maxrel_f = a.relthr = 0.0f;
  a.maxabs_u = 0;
  a.maxrel_d = 0.0;
}

struct Tol {
  float atol, rtol;
  bool eqnan;
};

// Float pairs: Eq. 1 in fp32 with explicit round-to-nearest operations.
//
// The hot loop handles the common case of every element: d = |x - y| <= FLT_MAX
// (both values finite), where x == y implies d = 0 <= tol, so the verdict is
// d <= tol alone; d and d^2 feed the per-vector max and sum.  Anything else in
// a 16-byte vector -- a mismatch, a NaN or an infinity, a difference that
// overflows, or an element that might raise max |x-y|/|y| -- sets one
// predicate, and the whole vector is then re-evaluated under the full rule by
// an out-of-line handler (float_vector_rare) that does the bookkeeping.  The
// handler takes and returns the accumulators by value, so they never leave
// registers on the hot path.
//
// max |x-y|/|y| stays exact without a division per element: fl(d/|y|) is
// monotone in the exact quotient, so an element can raise a maximum M already
// reached only if d/|y| > M, that is d - M |y| > 0, and one fused
// multiply-add gives the sign of d - M |y| exactly (one rounding of the exact
// value); only those elements are divided.
//
// The sum of squares (a statistic, not part of the verdict) accumulates with a
// fused multiply-add per element, then per 16-byte vector into fp64.
template <int DT>
__device__ __forceinline__ void unpack_vector(const uint4& v, float (&f)[16 / elem_bytes(DT)]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (DT == SV_F32) {
#pragma unroll
    for (int j = 0; j < 4; ++j) f[j] = __uint_as_float(w[j]);
  } else if constexpr (DT == SV_BF16) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      f[2 * j] = __uint_as_float(w[j] << 16);
      f[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 h = __half22float2(*reinterpret_cast<const __half2*>(&w[j]));
      f[2 * j] = h.x;
      f[2 * j + 1] = h.y;
    }
  }
}

// the full rule on one element, for the rare handler and the segment tail
__device__ __forceinline__ void float_elem_full(Acc& a, const Tol& t, float x, float y, uint64_t idx) {
  const float ay = fabsf(y);
  const float d = fabsf(__fsub_rn(x, y));
  const float tol = __fadd_rn(t.atol, __fmul_rn(t.rtol, ay));
  const bool xn = x != x, yn = y != y;
  const bool fin = (fabsf(x) <= FLT_MAX) & (ay <= FLT_MAX);
  const bool match = (x == y) | (fin & (d <= tol)) | (xn & yn & t.eqnan);
  if (!match) {
    a.mism++;
    if (a.first == ~0ull) a.first = idx;
    if (xn != yn) a.nan_d++;
    else if (!xn && (isinf(x) || ay > FLT_MAX)) a.inf_d++;
  }
  if (!fin) {
    a.nonfin++;
  } else if (!(d <= FLT_MAX)) {  // both finite, the difference overflowed
    a.maxabs_f = d;
    a.ssq = (double)d;
    a.maxrel_f = d;
    a.relthr = d;
  } else if (ay != 0.0f && __fmaf_rn(-a.relthr, ay, d) > 0.0f) {
    a.maxrel_f = fmaxf(a.maxrel_f, __fdiv_rn(d, ay));
    a.relthr = a.maxrel_f;
  }
}

template <int DT>
__device__ __noinline__ Acc float_vector_rare(Acc a, Tol t, uint4 xv, uint4 yv, uint64_t idx0) {
  constexpr int VE = 16 / elem_bytes(DT);
  float x[VE], y[VE];
  unpack_vector<DT>(xv, x);
  unpack_vector<DT>(yv, y);
  for (int j = 0; j < VE; ++j) float_elem_full(a, t, x[j], y[j], idx0 + j);
  return a;
}

// fold one vector's sum of squares: kept in fp32 while it can neither overflow
// nor lose its terms to underflow, otherwise recomputed exactly in fp64
template <int VE>
__device__ __forceinline__ void fold_vector(Acc& a, float vsum, float vmax, const float (&dk)[VE]) {
  a.maxabs_f = fmaxf(a.maxabs_f, vmax);
  if (vsum <= 0x1p120f && (vsum >= 0x1p-100f || vmax == 0.0f)) {
    a.ssq += (double)vsum;
  } else {
    double s = 0.0;
#pragma unroll
    for (int j = 0; j < VE; ++j) s += (double)dk[j] * (double)dk[j];
    a.ssq += s;
  }
}

// A vector of matching, finite elements whose only trigger is that some of
// them may raise the running max |x-y|/|y|: the max part of float_elem_full
// over its elements in order (the verdict and the other statistics need
// nothing more).  Returns the updated (max, threshold).
template <int DT>
__device__ __noinline__ float2 float_vector_ratio(float maxrel, float relthr, uint4 xv, uint4 yv) {
  constexpr int VE = 16 / elem_bytes(DT);
  float x[VE], y[VE];
  unpack_vector<DT>(xv, x);
  unpack_vector<DT>(yv, y);
  for (int j = 0; j < VE; ++j) {
    const float ay = fabsf(y[j]);
    const float d = fabsf(__fsub_rn(x[j], y[j]));
    if (ay != 0.0f && __fmaf_rn(-relthr, ay, d) > 0.0f) {
      maxrel = fmaxf(maxrel, __fdiv_rn(d, ay));
      relthr = maxrel;
    }
  }
  return make_float2(maxrel, relthr);
}

template <int DT>
__device__ __forceinline__ void float_vector(Acc& a, const Tol& t, const uint4& xv, const uint4& yv, uint64_t idx0) {
  constexpr int VE = 16 / elem_bytes(DT);
  float x[VE], y[VE], dk[VE];
  unpack_vector<DT>(xv, x);
  unpack_vector<DT>(yv, y);
  float vsum = 0.0f, vmax = 0.0f;
  bool rare = false, rel = false;
#pragma unroll
  for (int j = 0; j < VE; ++j) {
    const float ay = fabsf(y[j]);
    const float d = fabsf(__fsub_rn(x[j], y[j]));
    const float tol = __fadd_rn(t.atol, __fmul_rn(t.rtol, ay));
    const bool fin = d <= FLT_MAX;
    rare |= !(d <= tol) | !fin;
    rel |= __fmaf_rn(-a.relthr, ay, d) > 0.0f;
    dk[j] = fin ? d : 0.0f;
    vmax = fmaxf(vmax, dk[j]);
    vsum = __fmaf_rn(dk[j], dk[j], vsum);
  }
  fold_vector<VE>(a, vsum, vmax, dk);
  if (rare) {
    a = float_vector_rare<DT>(a, t, xv, yv, idx0);
  } else if (rel) {
    const float2 m = float_vector_ratio<DT>(a.maxrel_f, a.relthr, xv, yv);
    a.maxrel_f = m.x;
    a.relthr = m.y;
  }
}

// integers: exact equality; statistics only for the (rare) unequal elements,
// handled out of line with the accumulators passed by value
template <int DT>
__device__ __noinline__ Acc int_vector_rare(Acc a, uint4 xv, uint4 yv, uint64_t idx0) {
  constexpr int VE = 16 / elem_bytes(DT);
  int64_t x[VE], y[VE];
  if constexpr (DT == SV_I64) {
    x[0] = (int64_t)(((uint64_t)xv.y << 32) | xv.x);
    x[1] = (int64_t)(((uint64_t)xv.w << 32) | xv.z);
    y[0] = (int64_t)(((uint64_t)yv.y << 32) | yv.x);
    y[1] = (int64_t)(((uint64_t)yv.w << 32) | yv.z);
  } else {
    const uint32_t xs[4] = {xv.x, xv.y, xv.z, xv.w}, ys[4] = {yv.x, yv.y, yv.z, yv.w};
    for (int j = 0; j < 4; ++j) {
      x[j] = DT == SV_I32 ? (int64_t)(int32_t)xs[j] : (int64_t)xs[j];
      y[j] = DT == SV_I32 ? (int64_t)(int32_t)ys[j] : (int64_t)ys[j];
    }
  }
  for (int j = 0; j < VE; ++j) {
    if (x[j] == y[j]) continue;
    a.mism++;
    if (a.first == ~0ull) a.first = idx0 + j;
    const uint64_t d = x[j] >= y[j] ? (uint64_t)x[j] - (uint64_t)y[j] : (uint64_t)y[j] - (uint64_t)x[j];
    a.maxabs_u = d > a.maxabs_u ? d : a.maxabs_u;
    const double dd = (double)d;
    a.ssq += dd * dd;
    if (y[j] != 0) a.maxrel_d = fmax(a.maxrel_d, dd / fabs((double)y[j]));
  }
  return a;
}

template <int DT>
__device__ __forceinline__ void int_vector(Acc& a, const uint4& xv, const uint4& yv, uint64_t idx0) {
  const bool differ = (xv.x != yv.x) | (xv.y != yv.y) | (xv.z != yv.z) | (xv.w != yv.w);
  if (differ) a = int_vector_rare<DT>(a, xv, yv, idx0);
}

template <int DT>
__device__ __forceinline__ void do_vector(Acc& a, const Tol& t, const uint4& xv, const uint4& yv, uint64_t idx0) {
  if constexpr (is_float(DT)) float_vector<DT>(a, t, xv, yv, idx0);
  else int_vector<DT>(a, xv, yv, idx0);
}

// the elements of a segment's last, partial vector, one at a time
template <int DT>
__device__ void do_tail(Acc& a, const Tol& t, const uint8_t* xb, const uint8_t* yb, uint64_t i0, uint64_t i1) {
  constexpr uint32_t sz = elem_bytes(DT);
  for (uint64_t i = i0; i < i1; ++i) {
    if constexpr (is_float(DT)) {
      uint32_t xr, yr;
      if constexpr (sz == 4) {
        xr = reinterpret_cast<const uint32_t*>(xb)[i];
        yr = reinterpret_cast<const uint32_t*>(yb)[i];
      } else {
        xr = reinterpret_cast<const uint16_t*>(xb)[i];
        yr = reinterpret_cast<const uint16_t*>(yb)[i];
      }
      const float x = to_f32<DT>(xr), y = to_f32<DT>(yr);
      float_elem_full(a, t, x, y, i);
      const float d = fabsf(__fsub_rn(x, y));
      if (d <= FLT_MAX && (fabsf(x) <= FLT_MAX) && (fabsf(y) <= FLT_MAX)) {
        a.maxabs_f = fmaxf(a.maxabs_f, d);
        a.ssq += (double)d * (double)d;
      }
    } else {
      int64_t x, y;
      if constexpr (DT == SV_I64) {
        x = reinterpret_cast<const int64_t*>(xb)[i];
        y = reinterpret_cast<const int64_t*>(yb)[i];
      } else if constexpr (DT == SV_I32) {
        x = reinterpret_cast<const int32_t*>(xb)[i];
        y = reinterpret_cast<const int32_t*>(yb)[i];
      } else {
        x = reinterpret_cast<const uint32_t*>(xb)[i];
        y = reinterpret_cast<const uint32_t*>(yb)[i];
      }
      if (x != y) {
        a.mism++;
        if (a.first == ~0ull) a.first = i;
        const uint64_t d = x >= y ? (uint64_t)x - (uint64_t)y : (uint64_t)y - (uint64_t)x;
        a.maxabs_u = d > a.maxabs_u ? d : a.maxabs_u;
        const double dd = (double)d;
        a.ssq += dd * dd;
        if (y != 0) a.maxrel_d = fmax(a.maxrel_d, dd / fabs((double)y));
      }
    }
  }
}

__device__ __forceinline__ uint4 ldg_stream(const uint4* p) { return __ldcs(p); }

// elements [i0, i1) of one segment by a team of NT threads (the CTA, or one
// warp), `tid` the thread's rank in it: i0 is vector-aligned, i1 a loop
// boundary or n
template <int DT, int NT = kThreads>
__device__ void cmp_run(Acc& a, const vc_pair& pr, const uint8_t* cand, const uint8_t* ref, uint64_t i0,
                        uint64_t i1, int tid = threadIdx.x) {
  constexpr uint32_t sz = elem_bytes(DT), VE = 16 / sz;
  constexpr int U = kCmpTileBytes / 16 / kThreads;  // vectors per thread per loop iteration (4)
  const Tol t{__double2float_rn(pr.atol), __double2float_rn(pr.rtol), (pr.flags & SV_EQUAL_NAN) != 0};
  const uint8_t* xb = cand + pr.cand_offset;
  const uint8_t* yb = ref + pr.ref_offset;
  const uint4* xv = reinterpret_cast<const uint4*>(xb);
  const uint4* yv = reinterpret_cast<const uint4*>(yb);
  const uint64_t v0 = i0 / VE, vfull = i1 / VE;  // whole vectors in [i0, i1)
  for (uint64_t base = v0; base < vfull; base += (uint64_t)U * NT) {
    uint4 x[U], y[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint64_t v = base + (uint64_t)u * NT + tid;
      if (v < vfull) {
        x[u] = ldg_stream(xv + v);
        y[u] = ldg_stream(yv + v);
      }
    }

#pragma unroll
    for (int u = 0; u < U; ++u) {
      const uint64_t v = base + (uint64_t)u * NT + tid;
      if (v < vfull) do_vector<DT>(a, t, x[u], y[u], v * VE);
    }
    if constexpr (is_float(DT)) {
      // share the running max |x-y|/|y| across the warp: a lane only needs
      // the exact path for an element that could raise the warp's maximum
      // (the segment's maximum is the max over all lanes' own maxima, and an
      // element below the warp's maximum cannot change it)
      float m = a.maxrel_f;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
      a.relthr = m;
    }
  }
  const uint64_t tail0 = vfull * VE;
  if (tail0 < i1 && tid == 0) do_tail<DT>(a, t, xb, yb, tail0, i1);
}

// fold of the accumulators over aligned groups of `width` lanes (a power of
// two; 32: the whole warp), in fixed order; each group's result is in its
// first lane
template <bool FLOAT>
__device__ __forceinline__ Partial warp_fold(const Acc& a, int width = 32) {
  uint64_t mism = a.mism, nan_d = a.nan_d, inf_d = a.inf_d, nonfin = a.nonfin, first = a.first;
  double ssq = a.ssq;
  uint64_t maxabs = FLOAT ? (uint64_t)__float_as_uint(a.maxabs_f) : a.maxabs_u;
  double maxrel = FLOAT ? (double)a.maxrel_f : a.maxrel_d;
  for (int o = width >> 1; o > 0; o >>= 1) {
    mism += __shfl_down_sync(0xFFFFFFFFu, mism, o);
    nan_d += __shfl_down_sync(0xFFFFFFFFu, nan_d, o);
    inf_d += __shfl_down_sync(0xFFFFFFFFu, inf_d, o);
    nonfin += __shfl_down_sync(0xFFFFFFFFu, nonfin, o);
    const uint64_t f2 = __shfl_down_sync(0xFFFFFFFFu, first, o);
    first = f2 < first ? f2 : first;
    ssq += __shfl_down_sync(0xFFFFFFFFu, ssq, o);
    const uint64_t m2 = __shfl_down_sync(0xFFFFFFFFu, maxabs, o);
    maxabs = m2 > maxabs ? m2 : maxabs;  // non-negative fp32 bits order like the values
    maxrel = fmax(maxrel, __shfl_down_sync(0xFFFFFFFFu, maxrel, o));
  }
  return Partial{mism, nan_d, inf_d, nonfin, first, ssq, maxabs, maxrel};
}

// block-wide fold of the accumulators into one partial (fixed order)
template <bool FLOAT>
__device__ void flush(Acc& a, Partial* out) {
  __shared__ Partial wp[kThreads / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const Partial f = warp_fold<FLOAT>(a);
  if (lane == 0) wp[w] = f;
  __syncthreads();
  if (threadIdx.x == 0) {
    Partial r = wp[0];
    for (int i = 1; i < kThreads / 32; ++i) {
      const Partial& q = wp[i];
      r.mism += q.mism;
      r.nan_d += q.nan_d;
      r.inf_d += q.inf_d;
      r.nonfin += q.nonfin;
      r.first = q.first < r.first ? q.first : r.first;
      r.ssq += q.ssq;
      r.maxabs = q.maxabs > r.maxabs ? q.maxabs : r.maxabs;
      r.maxrel = fmax(r.maxrel, q.maxrel);
    }
    *out = r;
  }
  __syncthreads();
  acc_reset(a);
}

// one instantiation per dtype; the host groups the pairs by dtype
template <int DT>
__global__ void __launch_bounds__(kThreads, 3) cmp_kernel(const __grid_constant__ CmpParams p) {
  pdl_wait();
  pdl_trigger();
  if (p.flag && *p.flag >= 0) return;  // an earlier stage failed
  __shared__ uint64_t staged[kStagedStarts];
  const uint64_t u0 = (uint64_t)blockIdx.x * p.chunk;
  const uint64_t u1 = umin(u0 + p.chunk, p.total);
  if (u0 >= u1) return;
  const int lo = find_start(pentry(p, 0), p.n, u0, staged);  // segment containing u0
  Acc a;
  acc_reset(a);
  constexpr uint64_t VE = 16 / elem_bytes(DT);
  for (int e = lo; e < p.n; ++e) {
    // every thread reads the segment from the table (no staging, no barrier)
    const DevPair* te = pentry(p, e);
    const uint64_t wb = te->work_begin;
    if (wb >= u1) break;
    const vc_pair pr = te->p;
    const uint64_t we = wb + cmp_units(pr);
    if (we <= u0) continue;
    // this CTA overlaps the segment's units: it writes a partial for it (the
    // combine reads one from every overlapping CTA), covering the segment's
    // vectors that fall in [u0, u1) -- units [wb + overhead, we)
    const uint64_t v_base = wb + kCmpEntryUnits;
    const uint64_t vlo = umax(u0, v_base), vhi = umin(u1, we);
    if (vhi > vlo) cmp_run<DT>(a, pr, p.cand, p.ref, (vlo - v_base) * VE, umin((vhi - v_base) * VE, pr.n));
    flush<is_float(DT)>(a, p.partials + te->slot0 + blockIdx.x);
  }
}

// ---------------------------------------------------------------------------
// many small segments (at most kSmallVectors vectors each): one warp per
// segment, any dtype, no block barriers; the warp writes the segment's only
// partial at its slot0 (the combine reads that one slot: work_begin 0 and a
// chunk beyond the segment's units)
// ---------------------------------------------------------------------------
template <int DT>
__device__ __forceinline__ void warp_segment(const vc_pair& pr, const uint8_t* cand, const uint8_t* ref, Partial* out,
                                             int lane) {
  Acc a;
  acc_reset(a);
  cmp_run<DT, 32>(a, pr, cand, ref, 0, pr.n, lane);
  const Partial f = warp_fold<is_float(DT)>(a);
  if (lane == 0) *out = f;
}

__global__ void __launch_bounds__(kThreads) cmp_small_kernel(const __grid_constant__ CmpParams p) {
  pdl_wait();
  pdl_trigger();
  const int w = (int)(blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5)), lane = threadIdx.x & 31;
  if (w >= p.n) return;
  const DevPair* dp = pentry(p, w);
  const vc_pair& pr = dp->p;
  Partial* out = p.partials + dp->slot0;
  switch (pr.dtype) {  // uniform over the warp
    case SV_F32: warp_segment<SV_F32>(pr, p.cand, p.ref, out, lane); break;
    case SV_F16: warp_segment<SV_F16>(pr, p.cand, p.ref, out, lane); break;
    case SV_BF16: warp_segment<SV_BF16>(pr, p.cand, p.ref, out, lane); break;
    case SV_I32: warp_segment<SV_I32>(pr, p.cand, p.ref, out, lane); break;
    case SV_I64: warp_segment<SV_I64>(pr, p.cand, p.ref, out, lane); break;
    default: warp_segment<SV_U32>(pr, p.cand, p.ref, out, lane); break;
  }
}

// ---------------------------------------------------------------------------
// pass 2: one warp per segment folds the partials of CTAs b_first..b_last in
// order (deterministic) into a vc_result
// ---------------------------------------------------------------------------
__device__ vc_result fold_pair(const DevPair& dp, const Partial* partials, int lane) {
  const vc_pair& pr = dp.p;
  const bool fl = is_float(pr.dtype);
  uint64_t mism = 0, nan_d = 0, inf_d = 0, nonfin = 0, first = ~0ull, maxabs = 0;
  double ssq = 0.0, maxrel = 0.0;
  {
    // every CTA whose unit slice overlaps [work_begin, work_begin + units)
    const uint64_t b0 = dp.work_begin / dp.chunk, b1 = (dp.work_begin + cmp_units(pr) - 1) / dp.chunk;
#pragma unroll 4  // independent record loads in flight together
    for (uint64_t b = b0 + lane; b <= b1; b += 32) {
      const Partial q = partials[dp.slot0 + b];
      mism += q.mism;
      nan_d += q.nan_d;
      inf_d += q.inf_d;
      nonfin += q.nonfin;
      first = q.first < first ? q.first : first;
      ssq += q.ssq;
      maxabs = q.maxabs > maxabs ? q.maxabs : maxabs;
      maxrel = fmax(maxrel, q.maxrel);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mism += __shfl_down_sync(0xFFFFFFFFu, mism, o);
    nan_d += __shfl_down_sync(0xFFFFFFFFu, nan_d, o);
    inf_d += __shfl_down_sync(0xFFFFFFFFu, inf_d, o);
    nonfin += __shfl_down_sync(0xFFFFFFFFu, nonfin, o);
    const uint64_t f2 = __shfl_down_sync(0xFFFFFFFFu, first, o);
    first = f2 < first ? f2 : first;
    ssq += __shfl_down_sync(0xFFFFFFFFu, ssq, o);
    const uint64_t m2 = __shfl_down_sync(0xFFFFFFFFu, maxabs, o);
    maxabs = m2 > maxabs ? m2 : maxabs;
    maxrel = fmax(maxrel, __shfl_down_sync(0xFFFFFFFFu, maxrel, o));
  }
  vc_result r;  // meaningful in lane 0
  r.mismatches = mism;
  r.nan_disagree = nan_d;
  r.inf_disagree = inf_d;
  r.n_finite = fl ? pr.n - nonfin : pr.n;
  r.first_mismatch = first == ~0ull ? -1 : (int64_t)first;
  r.max_abs_u64 = fl ? 0 : maxabs;
  r.max_abs = fl ? (double)__uint_as_float((uint32_t)maxabs) : (double)maxabs;
  r.max_rel = maxrel;
  r.rms = r.n_finite ? sqrt(ssq / (double)r.n_finite) : 0.0;
  r.pass = mism == 0;
  r.state = SV_STAGE_RUN;
  return r;
}

__device__ __forceinline__ vc_result skipped_result() {
  vc_result r = {};
  r.first_mismatch = -1;
  r.state = SV_STAGE_SKIPPED;
  return r;
}

__global__ void __launch_bounds__(kThreads) combine_kernel(const __grid_constant__ CombParams p) {
  pdl_wait();
  pdl_trigger();
  const int e = (int)((blockIdx.x * (uint64_t)kThreads + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (e >= p.n) return;
  const DevPair dp = *pentry(p, e);
  const vc_result r = fold_pair(dp, p.partials, lane);
  if (lane == 0) p.results[dp.orig] = r;
}

// progressive ladder: one CTA folds a group of up to eight consecutive stages
// (one warp each), then applies the fail-fast order inside the group: stages
// after the first failing one are reported as skipped, and the flag records
// the failing stage so that later groups do not run.  Stages of a group are
// compared in one pass; the verdicts equal those of running them one by one.
__global__ void __launch_bounds__(kThreads) combine_stages_kernel(const __grid_constant__ CombParams p) {
  pdl_wait();
  pdl_trigger();
  __shared__ vc_result res[SV_INLINE_ENTRIES];
  const int e = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (!p.first_group && *p.flag >= 0) {  // an earlier group failed: nothing of this group ran
    if (threadIdx.x < p.n) p.results[pentry(p, threadIdx.x)->orig] = skipped_result();
    return;
  }
  if (e < p.n) {
    const vc_result r = fold_pair(*pentry(p, e), p.partials, lane);
    if (lane == 0) res[e] = r;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int failed = -1;
    for (int i = 0; i < p.n; ++i) {
      const DevPair* dp = pentry(p, i);
      if (failed >= 0) {
        p.results[dp->orig] = skipped_result();
        continue;
      }
      p.results[dp->orig] = res[i];
      if (!res[i].pass) failed = (int)dp->orig;
    }
    if (failed >= 0 || p.first_group) *p.flag = failed;  // the first group also clears it
  }
}

// ---------------------------------------------------------------------------
// shaped outputs: a rows x cols output with row pitches, tile by tile.  One
// CTA owns a whole tile at a time (grid-stride over the tiles): its threads
// walk the tile's whole 16-byte vectors in row-major order, U per step, with
// row / column counters that advance by a constant (no division per vector),
// then the ragged ends of the rows one element each; the CTA folds the tile
// and writes its vc_result.  Reported indices are output-wide, row * cols + col.
// ---------------------------------------------------------------------------
struct TileParams {
  vc_tiles t;
  uint64_t ntc, n_tiles;  // tiles per tile row, tiles in all
  const uint8_t* cand;
  const uint8_t* ref;
  vc_result* results;
  // warp teams only: groups of G full-width tiles side by side (G = 32 / the
  // tile width in 16-byte vectors; 0: no groups), gpr groups per tile row,
  // n_groups in all; the other `left` tiles of each tile row one by one
  uint32_t G;
  uint64_t gpr, n_groups, left;
};

// fold b (statistics of other elements) into a; first by minimum
__device__ __forceinline__ void acc_merge(Acc& a, const Acc& b) {
  a.mism += b.mism;
  a.nan_d += b.nan_d;
  a.inf_d += b.inf_d;
  a.nonfin += b.nonfin;
  a.first = b.first < a.first ? b.first : a.first;
  a.ssq += b.ssq;
  a.maxabs_f = fmaxf(a.maxabs_f, b.maxabs_f);
  a.maxrel_f = fmaxf(a.maxrel_f, b.maxrel_f);
  a.relthr = fmaxf(a.relthr, b.relthr);
  a.maxabs_u = b.maxabs_u > a.maxabs_u ? b.maxabs_u : a.maxabs_u;
  a.maxrel_d = fmax(a.maxrel_d, b.maxrel_d);
}

__device__ __forceinline__ vc_result tile_result(const Partial& q, uint64_t n, bool fl) {
  vc_result r;
  r.mismatches = q.mism;
  r.nan_disagree = q.nan_d;
  r.inf_disagree = q.inf_d;
  r.n_finite = fl ? n - q.nonfin : n;
  r.first_mismatch = q.first == ~0ull ? -1 : (int64_t)q.first;
  r.max_abs_u64 = fl ? 0 : q.maxabs;
  r.max_abs = fl ? (double)__uint_as_float((uint32_t)q.maxabs) : (double)q.maxabs;
  r.max_rel = q.maxrel;
  r.rms = r.n_finite ? sqrt(q.ssq / (double)r.n_finite) : 0.0;
  r.pass = q.mism == 0;
  r.state = SV_STAGE_RUN;
  return r;
}

// A team of NT threads owns one tile at a time: the whole CTA (NT = 256) when
// tiles are few and large, or one warp (NT = 32) when there are many, so that
// the warps of an SM stream their tiles independently (a warp's fold needs no
// block barrier, and no tile boundary drains the memory pipeline).
#ifndef SV_TILE_MINB
#define SV_TILE_MINB 3  // resident CTAs per SM the tile kernel's register budget must allow
#endif
#ifndef SV_TILE_U
#define SV_TILE_U 2  // 16-byte vectors per operand a tile-kernel thread loads per step
#endif
#ifndef SV_TILE_GROUP_RING
#define SV_TILE_GROUP_RING 2  // steps a tile-group lane keeps in flight through its shared-memory ring (0: none)
#endif
__device__ __forceinline__ void cp_async16_tile(void* dst, const void* src) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit_tile() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_tile() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

#ifndef SV_TILE_GROUP_U
#define SV_TILE_GROUP_U 4  // rows a tile-group lane loads per step (one 16-byte vector per operand each)
#endif
// G side-by-side tiles of one tile row for one warp: lane l owns vector
// column l of the group (tile l / (32 / G)) and walks down the rows, so every
// row of the group is one 512-byte run per operand, and the address and the
// element index advance by one add per row.  The running max |x-y|/|y| is
// shared within a tile's lanes only (its threshold must not exceed that
// tile's own maximum).
template <int DT>
__device__ __forceinline__ void tile_group(const TileParams& p, uint64_t item, int lane, const Tol& tol) {
  constexpr uint32_t sz = elem_bytes(DT), VE = 16 / sz;
  constexpr int U = SV_TILE_GROUP_U;
  const vc_tiles& t = p.t;
  const int vr = 32 / (int)p.G;  // lanes per tile
  const uint64_t ti = item / p.gpr, gj = item - ti * p.gpr;
  const uint64_t r0 = ti * t.tile_rows, col = gj * p.G * t.tile_cols + (uint64_t)lane * VE;
  const uint32_t h = (uint32_t)(umin(r0 + t.tile_rows, t.rows) - r0);
  const uint64_t xpb = t.cand_pitch * sz, ypb = t.ref_pitch * sz;
  const uint8_t* xp = p.cand + t.cand_offset + (r0 * t.cand_pitch + col) * sz;
  const uint8_t* yp = p.ref + t.ref_offset + (r0 * t.ref_pitch + col) * sz;
  uint64_t idx = r0 * t.cols + col;
  Acc a;
  acc_reset(a);
#if SV_TILE_GROUP_RING
  // the rows of the next kRing steps are in flight as cp.async copies into
  // this thread's own slots of a shared-memory ring (one 16-byte vector per
  // operand and row; slot-major with the threads innermost, so a warp's
  // copies and reads are contiguous): step st waits for its own copies,
  // reads them and refills its slot with step st + kRing
  constexpr int kRing = SV_TILE_GROUP_RING;
  extern __shared__ __align__(16) uint4 tring[];
  const uint32_t steps = (h + U - 1) / U;
  auto at = [&](uint32_t st, int u, int op) { return tring + ((int)((st % kRing) * U + u) * 2 + op) * kThreads + threadIdx.x; };
  auto fill = [&](uint32_t st) {
    if (st < steps) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t row = st * U + u;
        if (row < h) {
          cp_async16_tile(at(st, u, 0), xp + row * xpb);
          cp_async16_tile(at(st, u, 1), yp + row * ypb);
        }
      }
    }
    cp_async_commit_tile();  // one group per step, empty past the end: uniform counting
  };
#pragma unroll
  for (int s0 = 0; s0 < kRing; ++s0) fill((uint32_t)s0);
  for (uint32_t st = 0, r = 0; r < h; ++st, r += U) {  // h is the same for every lane
    cp_async_wait_tile<kRing - 1>();
    uint4 x[U], y[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (r + u < h) {
        x[u] = *at(st, u, 0);
        y[u] = *at(st, u, 1);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (r + u < h) do_vector<DT>(a, tol, x[u], y[u], idx + (uint64_t)u * t.cols);
    idx += U * t.cols;
    fill(st + kRing);  // the slot's values are in registers
#else
  for (uint32_t r = 0; r < h; r += U) {  // h is the same for every lane
    uint4 x[U], y[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (r + u < h) {
        x[u] = ldg_stream(reinterpret_cast<const uint4*>(xp + u * xpb));
        y[u] = ldg_stream(reinterpret_cast<const uint4*>(yp + u * ypb));
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (r + u < h) do_vector<DT>(a, tol, x[u], y[u], idx + (uint64_t)u * t.cols);
    xp += U * xpb;
    yp += U * ypb;
    idx += U * t.cols;
#endif
    if constexpr (is_float(DT)) {
      float m = a.maxrel_f;
      for (int o = vr >> 1; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
      a.relthr = m;
    }
  }
#if SV_TILE_GROUP_RING
  cp_async_wait_tile<0>();
#endif
  const Partial f = warp_fold<is_float(DT)>(a, vr);
  if (lane % vr == 0)
    p.results[ti * p.ntc + gj * p.G + (uint64_t)(lane / vr)] = tile_result(f, (uint64_t)h * t.tile_cols, is_float(DT));
}

template <int DT, int NT>
__global__ void __launch_bounds__(kThreads, SV_TILE_MINB) tile_kernel(const __grid_constant__ TileParams p) {
  constexpr uint32_t sz = elem_bytes(DT), VE = 16 / sz;
  constexpr int U = SV_TILE_U;                        // vectors per thread per step
  constexpr uint32_t kStep = (uint32_t)U * NT;
  constexpr int kTeams = kThreads / NT;               // teams per CTA
  __shared__ Partial tile_sum;
  const int tid = (int)(threadIdx.x % NT);
  const uint64_t team = (uint64_t)blockIdx.x * kTeams + threadIdx.x / NT;
  const uint64_t teams = (uint64_t)gridDim.x * kTeams;
  const vc_tiles& t = p.t;
  const Tol tol{__double2float_rn(t.atol), __double2float_rn(t.rtol), (t.flags & SV_EQUAL_NAN) != 0};
  const uint8_t* xb = p.cand + t.cand_offset;
  const uint8_t* yb = p.ref + t.ref_offset;
  // every team runs the same number of rounds (a CTA's barrier needs all its threads)
  const uint64_t rounds = NT == kThreads ? (p.n_tiles + teams - 1) / teams : 0;
  // warp teams take the tiles outside the groups (all tiles when there are none)
  const uint64_t items = NT == kThreads ? p.n_tiles : p.n_tiles - p.n_groups * p.G;
  for (uint64_t k = 0, item = team; NT == kThreads ? k < rounds : item < items; ++k, item += teams) {
    uint64_t tile = item;
    if constexpr (NT != kThreads) {
      const uint64_t tr = item / p.left;
      tile = tr * p.ntc + p.gpr * p.G + (item - tr * p.left);
    }
    const bool live = tile < p.n_tiles;
    const uint64_t ti = live ? tile / p.ntc : 0, tj = live ? tile - ti * p.ntc : 0;
    const uint64_t r0 = ti * t.tile_rows, c0 = tj * t.tile_cols;
    const uint32_t h = live ? (uint32_t)(umin(r0 + t.tile_rows, t.rows) - r0) : 0;
    const uint32_t w = live ? (uint32_t)(umin(c0 + t.tile_cols, t.cols) - c0) : 0;
    const uint32_t vr = w / VE;  // whole vectors per row of the tile
    // the tile's origin in each operand; a row step is a 32 x 32 -> 64-bit
    // multiply (row pitches under 4 GiB when a tile spans rows: validated)
    const uint8_t* xt = xb + (r0 * t.cand_pitch + c0) * sz;
    const uint8_t* yt = yb + (r0 * t.ref_pitch + c0) * sz;
    const uint32_t xpb = (uint32_t)(t.cand_pitch * sz), ypb = (uint32_t)(t.ref_pitch * sz);
    Acc a;
    acc_reset(a);
    if (vr > 0) {
      uint32_t rr[U], cc[U];  // row and vector column (in the tile) of this thread's u-th vector
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const uint32_t v = (uint32_t)tid + (uint32_t)u * NT;
        rr[u] = v / vr;
        cc[u] = v - rr[u] * vr;
      }
      const uint32_t dq = kStep / vr, dr = kStep - dq * vr;
      const uint64_t nvec = (uint64_t)h * vr;
      for (uint64_t base = 0; base < nvec; base += kStep) {  // uniform trip count: the shuffles below need the warp
        uint4 x[U], y[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (rr[u] < h) {
            const uint32_t cb = cc[u] * 16u;
            x[u] = ldg_stream(reinterpret_cast<const uint4*>(xt + (uint64_t)rr[u] * xpb + cb));
            y[u] = ldg_stream(reinterpret_cast<const uint4*>(yt + (uint64_t)rr[u] * ypb + cb));
          }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (rr[u] < h) do_vector<DT>(a, tol, x[u], y[u], (r0 + rr[u]) * t.cols + c0 + (uint64_t)cc[u] * VE);
          cc[u] += dr;
          rr[u] += dq;
          if (cc[u] >= vr) {
            cc[u] -= vr;
            ++rr[u];
          }
        }
        if constexpr (is_float(DT)) {  // share the running max |x-y|/|y| across the warp (as cmp_run)
          float m = a.maxrel_f;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
          a.relthr = m;
        }
      }
    }
    if (vr * VE < w) {  // the ragged end of every row: one thread per row, elements in order
      Acc b;
      acc_reset(b);
      for (uint32_t r = (uint32_t)tid; r < h; r += NT) {
        const uint64_t row = r0 + r, cs = c0 + (uint64_t)vr * VE;
        Acc e;
        acc_reset(e);
        do_tail<DT>(e, tol, xb + (row * t.cand_pitch + cs) * sz, yb + (row * t.ref_pitch + cs) * sz, 0,
                    w - vr * VE);
        if (e.first != ~0ull) e.first += row * t.cols + cs;  // do_tail reports indices from 0
        acc_merge(b, e);
      }
      acc_merge(a, b);
    }
    if constexpr (NT == kThreads) {
      flush<is_float(DT)>(a, &tile_sum);  // block fold; ends with a barrier
      if (threadIdx.x == 0 && live) p.results[tile] = tile_result(tile_sum, (uint64_t)h * w, is_float(DT));
    } else {
      const Partial f = warp_fold<is_float(DT)>(a);
      if (tid == 0) p.results[tile] = tile_result(f, (uint64_t)h * w, is_float(DT));
    }
  }
}

// the groups of side-by-side tiles, one group per warp at a time (a kernel of
// its own: few registers, so 3 CTAs per SM keep 4 rows of loads in flight)
template <int DT>
__global__ void __launch_bounds__(kThreads, 3) tile_group_kernel(const __grid_constant__ TileParams p) {
  const vc_tiles& t = p.t;
  const Tol tol{__double2float_rn(t.atol), __double2float_rn(t.rtol), (t.flags & SV_EQUAL_NAN) != 0};
  const int lane = (int)(threadIdx.x & 31);
  const uint64_t warps = (uint64_t)gridDim.x * (kThreads / 32);
  for (uint64_t item = (uint64_t)blockIdx.x * (kThreads / 32) + threadIdx.x / 32; item < p.n_groups; item += warps)
    tile_group<DT>(p, item, lane, tol);
}

static const void* tile_group_kernel_for(uint32_t dtype) {
  switch (dtype) {
    case SV_F32: return reinterpret_cast<const void*>(&tile_group_kernel<SV_F32>);
    case SV_F16: return reinterpret_cast<const void*>(&tile_group_kernel<SV_F16>);
    case SV_BF16: return reinterpret_cast<const void*>(&tile_group_kernel<SV_BF16>);
    case SV_I32: return reinterpret_cast<const void*>(&tile_group_kernel<SV_I32>);
    case SV_I64: return reinterpret_cast<const void*>(&tile_group_kernel<SV_I64>);
    default: return reinterpret_cast<const void*>(&tile_group_kernel<SV_U32>);
  }
}

// dynamic shared memory of a tile-group CTA: its threads' rings
constexpr size_t kTileRingSmem = (size_t)SV_TILE_GROUP_RING * SV_TILE_GROUP_U * 2 * kThreads * 16;

static void launch_tile_groups(const TileParams& tp, uint32_t grid, cudaStream_t st) {
  switch (tp.t.dtype) {
    case SV_F32: tile_group_kernel<SV_F32><<<grid, launch_block(), kTileRingSmem, st>>>(tp); break;
    case SV_F16: tile_group_kernel<SV_F16><<<grid, launch_block(), kTileRingSmem, st>>>(tp); break;
    case SV_BF16: tile_group_kernel<SV_BF16><<<grid, launch_block(), kTileRingSmem, st>>>(tp); break;
    case SV_I32: tile_group_kernel<SV_I32><<<grid, launch_block(), kTileRingSmem, st>>>(tp); break;
    case SV_I64: tile_group_kernel<SV_I64><<<grid, launch_block(), kTileRingSmem, st>>>(tp); break;
    default: tile_group_kernel<SV_U32><<<grid, launch_block(), kTileRingSmem, st>>>(tp); break;
  }
}

template <int NT>
static const void* tile_kernel_for(uint32_t dtype) {
  switch (dtype) {
    case SV_F32: return reinterpret_cast<const void*>(&tile_kernel<SV_F32, NT>);
    case SV_F16: return reinterpret_cast<const void*>(&tile_kernel<SV_F16, NT>);
    case SV_BF16: return reinterpret_cast<const void*>(&tile_kernel<SV_BF16, NT>);
    case SV_I32: return reinterpret_cast<const void*>(&tile_kernel<SV_I32, NT>);
    case SV_I64: return reinterpret_cast<const void*>(&tile_kernel<SV_I64, NT>);
    default: return reinterpret_cast<const void*>(&tile_kernel<SV_U32, NT>);
  }
}

template <int NT>
static void launch_tiles(const TileParams& tp, uint32_t grid, cudaStream_t st) {
  switch (tp.t.dtype) {
    case SV_F32: tile_kernel<SV_F32, NT><<<grid, launch_block(), 0, st>>>(tp); break;
    case SV_F16: tile_kernel<SV_F16, NT><<<grid, launch_block(), 0, st>>>(tp); break;
    case SV_BF16: tile_kernel<SV_BF16, NT><<<grid, launch_block(), 0, st>>>(tp); break;
    case SV_I32: tile_kernel<SV_I32, NT><<<grid, launch_block(), 0, st>>>(tp); break;
    case SV_I64: tile_kernel<SV_I64, NT><<<grid, launch_block(), 0, st>>>(tp); break;
    default: tile_kernel<SV_U32, NT><<<grid, launch_block(), 0, st>>>(tp); break;
  }
}

cudaError_t launch_compare_tiles(const vc_tiles& t, uint64_t ntc, uint64_t n_tiles, const uint8_t* cand,
                                 const uint8_t* ref, vc_result* results, cudaStream_t st) {
  if (n_tiles == 0) return cudaSuccess;
  TileParams tp;
  tp.t = t;
  tp.ntc = ntc;
  tp.n_tiles = n_tiles;
  tp.cand = cand;
  tp.ref = ref;
  tp.results = results;
  tp.G = 0;
  tp.gpr = 0;
  tp.n_groups = 0;
  tp.left = ntc;
  // one warp per tile once there are enough tiles for every resident warp to
  // hold a few; otherwise the whole CTA shares each tile
  const uint32_t cap_w = grid_cap_for(tile_kernel_for<32>(t.dtype));
  const bool warps = n_tiles >= 4ull * cap_w * (kThreads / 32);
  if (warps) {
    // tiles narrower than the output whose width in 16-byte vectors divides
    // 32 go to the warps in groups of 32 / width side by side
    const uint64_t vr = t.tile_cols * elem_bytes((int)t.dtype) / 16;  // whole vectors (validated)
    if (t.tile_cols < t.cols && vr >= 1 && vr <= 32 && 32 % vr == 0) {
      tp.G = (uint32_t)(32 / vr);
      tp.gpr = (t.cols / t.tile_cols) / tp.G;
      tp.left = ntc - tp.gpr * tp.G;
      tp.n_groups = (n_tiles / ntc) * tp.gpr;
    }
    if (tp.n_groups) {  // the groups, then the other tiles one warp each
      const uint64_t want = (tp.n_groups + kThreads / 32 - 1) / (kThreads / 32);
      launch_tile_groups(tp, (uint32_t)umin(want, grid_cap_for(tile_group_kernel_for(t.dtype), kTileRingSmem)), st);
      count_launch();
    }
    const uint64_t rest = n_tiles - tp.n_groups * tp.G;
    if (rest == 0) return cudaGetLastError();
    const uint64_t want = (rest + kThreads / 32 - 1) / (kThreads / 32);
    launch_tiles<32>(tp, (uint32_t)umin(want, cap_w), st);
  } else {
    launch_tiles<kThreads>(tp, (uint32_t)umin(n_tiles, grid_cap_for(tile_kernel_for<kThreads>(t.dtype))), st);
  }
  count_launch();
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// host launchers
// ---------------------------------------------------------------------------
static const void* cmp_kernel_for(uint32_t dtype) {
  switch (dtype) {
    case SV_F32: return reinterpret_cast<const void*>(&cmp_kernel<SV_F32>);
    case SV_F16: return reinterpret_cast<const void*>(&cmp_kernel<SV_F16>);
    case SV_BF16: return reinterpret_cast<const void*>(&cmp_kernel<SV_BF16>);
    case SV_I32: return reinterpret_cast<const void*>(&cmp_kernel<SV_I32>);
    case SV_I64: return reinterpret_cast<const void*>(&cmp_kernel<SV_I64>);
    default: return reinterpret_cast<const void*>(&cmp_kernel<SV_U32>);
  }
}

LaunchShape compare_shape(uint32_t dtype, uint64_t units, uint64_t tiles) {
  return shape_for(units, tiles, grid_cap_for(cmp_kernel_for(dtype)), kCmpTileBytes / 16);
}

template <class P>
static void fill_pairs(P& cp, const DevPair* host, const DevPair* dev, int n) {
  cp.tab = dev;
  cp.n = n;
  if (!dev)
    for (int i = 0; i < n; ++i) cp.inl[i] = host[i];
}

cudaError_t launch_compare_group(uint32_t dtype, const DevPair* host, const DevPair* dev, int n, uint64_t units,
                                 LaunchShape sh, const uint8_t* cand, const uint8_t* ref, Partial* partials,
                                 const int32_t* flag, cudaStream_t st) {
  if (units == 0 || n == 0) return cudaSuccess;
  CmpParams cp;
  fill_pairs(cp, host, dev, n);
  cp.total = units;
  cp.chunk = sh.chunk;
  cp.cand = cand;
  cp.ref = ref;
  cp.partials = partials;
  cp.flag = flag;
  cudaError_t e;
  switch (dtype) {
    case SV_F32: e = launch_chained(cmp_kernel<SV_F32>, sh.grid, launch_block(), st, cp); break;
    case SV_F16: e = launch_chained(cmp_kernel<SV_F16>, sh.grid, launch_block(), st, cp); break;
    case SV_BF16: e = launch_chained(cmp_kernel<SV_BF16>, sh.grid, launch_block(), st, cp); break;
    case SV_I32: e = launch_chained(cmp_kernel<SV_I32>, sh.grid, launch_block(), st, cp); break;
    case SV_I64: e = launch_chained(cmp_kernel<SV_I64>, sh.grid, launch_block(), st, cp); break;
    default: e = launch_chained(cmp_kernel<SV_U32>, sh.grid, launch_block(), st, cp); break;
  }
  count_launch();
  return e;
}

cudaError_t launch_compare_small(const DevPair* host, const DevPair* dev, int n, const uint8_t* cand,
                                 const uint8_t* ref, Partial* partials, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  CmpParams cp;
  fill_pairs(cp, host, dev, n);
  cp.total = 0;
  cp.chunk = 0;
  cp.cand = cand;
  cp.ref = ref;
  cp.partials = partials;
  cp.flag = nullptr;
  const unsigned blocks = (unsigned)((n + kThreads / 32 - 1) / (kThreads / 32));
  const cudaError_t e = launch_chained(cmp_small_kernel, blocks, launch_block(), st, cp);
  count_launch();
  return e;
}

cudaError_t launch_combine(const DevPair* host, const DevPair* dev, int n, const Partial* partials,
                           vc_result* results, int32_t* flag, int first_group, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  CombParams cp;
  fill_pairs(cp, host, dev, n);
  cp.partials = partials;
  cp.results = results;
  cp.flag = flag;
  cp.first_group = first_group;
  cudaError_t e;
  if (flag) {  // a progressive group: one CTA, stages in order
    if (n > SV_INLINE_ENTRIES || dev) return cudaErrorInvalidValue;
    e = launch_chained(combine_stages_kernel, 1u, launch_block(), st, cp);
  } else {
    const uint64_t blocks = ((uint64_t)n * 32 + kThreads - 1) / kThreads;
    e = launch_chained(combine_kernel, (unsigned)blocks, launch_block(), st, cp);
  }
  count_launch();
  return e;
}

}  // namespace sv
