// convert.cu -- dtype-correct value conversion of test data on the GPU.
//
// The scaffold's helpers load the prepared test inputs (Sec. 4.1.2); a loader
// that reads every file as float turns uint8 or int32 data into wrong values
// (the defect behind 31.4% of the false positives in Sec. 5.2.3).  Loading
// into a buffer of another element type therefore converts VALUES:
// integer -> integer exactly (clamped, and counted, out of range); anything
// -> float rounded once to nearest-even (overflow to +-Inf counted; NaN made
// canonical); float -> integer is refused by the caller before a launch.
//
// The kernel streams 16-byte source vectors (one per thread and step of a
// persistent grid, several steps in flight), converts their 16/sizeof(S)
// elements in registers and stores the results with 16-byte (or narrower)
// stores; it is bound by HBM bandwidth: sizeof(S) + sizeof(D) bytes per
// element.
//
// Rounding to the 16-bit float types from wider sources goes through fp32
// rounded to odd: the value truncated toward zero with the last bit set when
// that lost anything.  A second rounding to nearest-even into a format with
// at least two fewer significant bits than fp32 then equals one direct
// rounding (Boldo and Melquiond, "Emulation of FMA and correctly rounded
// sums: proved algorithms using rounding to odd", IEEE Trans. Computers 57(4),
// 2008); fp16 and bf16 keep 11 and 8 bits against fp32's 24, and fp32's
// exponent range covers both, subnormals included.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <type_traits>

#include "../../include/sv_io.h"
#include "sv_kernels.h"

namespace sv {
namespace {

struct F16 { uint16_t b; };
struct BF16 { uint16_t b; };

template <class T> struct Info;
#define SV_INFO(T, FLOAT, SIGNED, LO, HI)                               \
  template <> struct Info<T> {                                          \
    static constexpr bool kFloat = FLOAT;                               \
    static constexpr bool kSigned = SIGNED;                             \
    static constexpr long long kLo = LO;                                \
    static constexpr unsigned long long kHi = HI;                       \
  };
SV_INFO(uint8_t, false, false, 0, 0xFFull)
SV_INFO(int8_t, false, true, -128, 127ull)
SV_INFO(uint16_t, false, false, 0, 0xFFFFull)
SV_INFO(int16_t, false, true, -32768, 32767ull)
SV_INFO(uint32_t, false, false, 0, 0xFFFFFFFFull)
SV_INFO(int32_t, false, true, -2147483647ll - 1, 2147483647ull)
SV_INFO(uint64_t, false, false, 0, 0xFFFFFFFFFFFFFFFFull)
SV_INFO(int64_t, false, true, -9223372036854775807ll - 1, 9223372036854775807ull)
#undef SV_INFO
template <> struct Info<F16> { static constexpr bool kFloat = true; };
template <> struct Info<BF16> { static constexpr bool kFloat = true; };
template <> struct Info<float> { static constexpr bool kFloat = true; };
template <> struct Info<double> { static constexpr bool kFloat = true; };

constexpr uint32_t kNanF32 = 0x7FC00000u;
constexpr unsigned long long kNanF64 = 0x7FF8000000000000ull;
constexpr uint16_t kNanF16 = 0x7E00u;
constexpr uint16_t kNanBF16 = 0x7FC0u;

// ---- source classification ----
template <class S> __device__ __forceinline__ bool src_nan(S) { return false; }
template <> __device__ __forceinline__ bool src_nan<F16>(F16 x) { return (x.b & 0x7FFFu) > 0x7C00u; }
template <> __device__ __forceinline__ bool src_nan<BF16>(BF16 x) { return (x.b & 0x7FFFu) > 0x7F80u; }
template <> __device__ __forceinline__ bool src_nan<float>(float x) { return x != x; }
template <> __device__ __forceinline__ bool src_nan<double>(double x) { return x != x; }
template <class S> __device__ __forceinline__ bool src_inf(S) { return false; }
template <> __device__ __forceinline__ bool src_inf<F16>(F16 x) { return (x.b & 0x7FFFu) == 0x7C00u; }
template <> __device__ __forceinline__ bool src_inf<BF16>(BF16 x) { return (x.b & 0x7FFFu) == 0x7F80u; }
template <> __device__ __forceinline__ bool src_inf<float>(float x) { return isinf(x); }
template <> __device__ __forceinline__ bool src_inf<double>(double x) { return isinf(x); }

__device__ __forceinline__ float set_odd(float r, bool inexact) {
  return inexact ? __uint_as_float(__float_as_uint(r) | 1u) : r;
}

// ---- the source value in fp32, rounded to odd (exact where it fits) ----
template <class S> __device__ __forceinline__ float odd32(S x) { return (float)x; }  // 8/16-bit integers: exact
template <> __device__ __forceinline__ float odd32<F16>(F16 x) { return __half2float(__ushort_as_half(x.b)); }
template <> __device__ __forceinline__ float odd32<BF16>(BF16 x) { return __uint_as_float((uint32_t)x.b << 16); }
template <> __device__ __forceinline__ float odd32<float>(float x) { return x; }
template <> __device__ __forceinline__ float odd32<double>(double x) {
  const float r = __double2float_rz(x);
  return set_odd(r, (double)r != x);
}
template <> __device__ __forceinline__ float odd32<int32_t>(int32_t x) {
  const float r = __int2float_rz(x);
  return set_odd(r, __float2int_rz(r) != x);
}
template <> __device__ __forceinline__ float odd32<uint32_t>(uint32_t x) {
  const float r = __uint2float_rz(x);
  return set_odd(r, __float2uint_rz(r) != x);
}
template <> __device__ __forceinline__ float odd32<int64_t>(int64_t x) {
  const float r = __ll2float_rz(x);
  return set_odd(r, __float2ll_rz(r) != x);
}
template <> __device__ __forceinline__ float odd32<uint64_t>(uint64_t x) {
  const float r = __ull2float_rz(x);
  return set_odd(r, __float2ull_rz(r) != x);
}

// ---- the source value rounded once to fp32 ----
template <class S> __device__ __forceinline__ float rn32(S x) { return odd32(x); }  // exact cases
template <> __device__ __forceinline__ float rn32<double>(double x) { return __double2float_rn(x); }
template <> __device__ __forceinline__ float rn32<int32_t>(int32_t x) { return __int2float_rn(x); }
template <> __device__ __forceinline__ float rn32<uint32_t>(uint32_t x) { return __uint2float_rn(x); }
template <> __device__ __forceinline__ float rn32<int64_t>(int64_t x) { return __ll2float_rn(x); }
template <> __device__ __forceinline__ float rn32<uint64_t>(uint64_t x) { return __ull2float_rn(x); }

// ---- the source value rounded once to fp64 ----
template <class S> __device__ __forceinline__ double rn64(S x) {
  if constexpr (std::is_same<S, int64_t>::value) return __ll2double_rn(x);
  else if constexpr (std::is_same<S, uint64_t>::value) return __ull2double_rn(x);
  else if constexpr (Info<S>::kFloat) return (double)odd32(x);  // fp16 / bf16 / fp32: exact
  else return (double)x;                                        // integers up to 32 bits: exact
}

template <class D, class S> __device__ __forceinline__ D convert(S x, uint32_t& lost) {
  if constexpr (std::is_same<D, double>::value) {
    return src_nan(x) ? __longlong_as_double((long long)kNanF64) : rn64(x);
  } else if constexpr (std::is_same<D, float>::value) {
    if (src_nan(x)) return __uint_as_float(kNanF32);
    const float r = rn32(x);
    lost += (isinf(r) && !src_inf(x)) ? 1u : 0u;
    return r;
  } else if constexpr (std::is_same<D, F16>::value) {
    if (src_nan(x)) return F16{kNanF16};
    const uint16_t h = __half_as_ushort(__float2half_rn(odd32(x)));
    lost += ((h & 0x7FFFu) == 0x7C00u && !src_inf(x)) ? 1u : 0u;
    return F16{h};
  } else if constexpr (std::is_same<D, BF16>::value) {
    if (src_nan(x)) return BF16{kNanBF16};
    const uint16_t h = __bfloat16_as_ushort(__float2bfloat16_rn(odd32(x)));
    lost += ((h & 0x7FFFu) == 0x7F80u && !src_inf(x)) ? 1u : 0u;
    return BF16{h};
  } else {  // integer -> integer, clamped to D's range
    static_assert(!Info<S>::kFloat, "float -> integer is refused before a launch");
    if constexpr (Info<S>::kSigned) {
      const long long v = (long long)x;
      if (v < Info<D>::kLo) { ++lost; return (D)Info<D>::kLo; }
      if (v > 0 && (unsigned long long)v > Info<D>::kHi) { ++lost; return (D)Info<D>::kHi; }
      return (D)v;
    } else {
      const unsigned long long v = (unsigned long long)x;
      if (v > Info<D>::kHi) { ++lost; return (D)Info<D>::kHi; }
      return (D)v;
    }
  }
}

// store `bytes` (a power of two from 2 to 128) of a thread's converted
// elements; 16-byte pieces where the run is that long
template <int kBytes> __device__ __forceinline__ void store_run(uint8_t* dst, const uint8_t* src) {
  if constexpr (kBytes >= 16) {
#pragma unroll
    for (int i = 0; i < kBytes / 16; ++i)
      __stcs(reinterpret_cast<uint4*>(dst) + i, reinterpret_cast<const uint4*>(src)[i]);
  } else if constexpr (kBytes == 8) {
    __stcs(reinterpret_cast<uint2*>(dst), *reinterpret_cast<const uint2*>(src));
  } else if constexpr (kBytes == 4) {
    __stcs(reinterpret_cast<unsigned int*>(dst), *reinterpret_cast<const unsigned int*>(src));
  } else {
    *reinterpret_cast<unsigned short*>(dst) = *reinterpret_cast<const unsigned short*>(src);
  }
}

template <class S, class D>
__global__ void __launch_bounds__(kThreads) cvt_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                                       uint64_t n, unsigned long long* __restrict__ lost) {
  constexpr int kE = 16 / (int)sizeof(S);              // elements per source vector
  constexpr int kOut = kE * (int)sizeof(D);            // bytes they become
  constexpr int kU = kOut <= 32 ? 4 : (kOut <= 64 ? 2 : 1);  // vectors in flight per thread
  const uint64_t nv = n / kE;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  uint64_t v = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t my_lost = 0;
  for (; v + (kU - 1) * stride < nv; v += kU * stride) {
    uint4 in[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) in[u] = __ldcs(reinterpret_cast<const uint4*>(src) + v + u * stride);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      S e[kE];
      memcpy(e, &in[u], 16);
      alignas(16) D o[kE];
#pragma unroll
      for (int i = 0; i < kE; ++i) o[i] = convert<D>(e[i], my_lost);
      store_run<kOut>(dst + (v + u * stride) * kOut, reinterpret_cast<const uint8_t*>(o));
    }
  }
  for (; v < nv; v += stride) {
    const uint4 in = __ldcs(reinterpret_cast<const uint4*>(src) + v);
    S e[kE];
    memcpy(e, &in, 16);
    alignas(16) D o[kE];
#pragma unroll
    for (int i = 0; i < kE; ++i) o[i] = convert<D>(e[i], my_lost);
    store_run<kOut>(dst + v * kOut, reinterpret_cast<const uint8_t*>(o));
  }
  // the ragged tail (fewer than kE elements): one element per thread
  const uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t < n - nv * kE) {  // typed accesses: both arrays are aligned to their element size
    const uint64_t i = nv * kE + t;
    reinterpret_cast<D*>(dst)[i] = convert<D>(reinterpret_cast<const S*>(src)[i], my_lost);
  }
  // lost values: one atomic per warp that saw any (rare)
  const unsigned warp_lost = __reduce_add_sync(0xFFFFFFFFu, my_lost);
  if (warp_lost && (threadIdx.x & 31) == 0) atomicAdd(lost, (unsigned long long)warp_lost);
}

template <class S, class D>
cudaError_t launch_cvt(const void* src, void* dst, uint64_t n, unsigned long long* lost, cudaStream_t st) {
  if constexpr (std::is_same<S, D>::value || (Info<S>::kFloat && !Info<D>::kFloat)) {
    return cudaErrorInvalidValue;  // same type: a copy; float -> integer: refused
  } else {
    constexpr int kE = 16 / (int)sizeof(S);
    const uint64_t nv = n / kE;
    const uint64_t want = (nv + kThreads - 1) / kThreads;
    const uint32_t cap = grid_cap_for(reinterpret_cast<const void*>(&cvt_kernel<S, D>));
    const uint32_t grid = (uint32_t)(want < 1 ? 1 : (want < cap ? want : cap));
    count_launch();
    cvt_kernel<S, D><<<grid, launch_block(), 0, st>>>(static_cast<const uint8_t*>(src), static_cast<uint8_t*>(dst),
                                                     n, lost);
    return cudaGetLastError();
  }
}

template <class S>
cudaError_t launch_from(int d, const void* src, void* dst, uint64_t n, unsigned long long* lost, cudaStream_t st) {
  switch (d) {
    case SV_F32: return launch_cvt<S, float>(src, dst, n, lost, st);
    case SV_F16: return launch_cvt<S, F16>(src, dst, n, lost, st);
    case SV_BF16: return launch_cvt<S, BF16>(src, dst, n, lost, st);
    case SV_F64: return launch_cvt<S, double>(src, dst, n, lost, st);
    case SV_I32: return launch_cvt<S, int32_t>(src, dst, n, lost, st);
    case SV_I64: return launch_cvt<S, int64_t>(src, dst, n, lost, st);
    case SV_U32: return launch_cvt<S, uint32_t>(src, dst, n, lost, st);
    case SV_U8: return launch_cvt<S, uint8_t>(src, dst, n, lost, st);
    case SV_I8: return launch_cvt<S, int8_t>(src, dst, n, lost, st);
    case SV_I16: return launch_cvt<S, int16_t>(src, dst, n, lost, st);
    case SV_U16: return launch_cvt<S, uint16_t>(src, dst, n, lost, st);
    case SV_U64: return launch_cvt<S, uint64_t>(src, dst, n, lost, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_convert(int s, int d, const void* src, void* dst, uint64_t n, unsigned long long* lost,
                           cudaStream_t st) {
  switch (s) {
    case SV_F32: return launch_from<float>(d, src, dst, n, lost, st);
    case SV_F16: return launch_from<F16>(d, src, dst, n, lost, st);
    case SV_BF16: return launch_from<BF16>(d, src, dst, n, lost, st);
    case SV_F64: return launch_from<double>(d, src, dst, n, lost, st);
    case SV_I32: return launch_from<int32_t>(d, src, dst, n, lost, st);
    case SV_I64: return launch_from<int64_t>(d, src, dst, n, lost, st);
    case SV_U32: return launch_from<uint32_t>(d, src, dst, n, lost, st);
    case SV_U8: return launch_from<uint8_t>(d, src, dst, n, lost, st);
    case SV_I8: return launch_from<int8_t>(d, src, dst, n, lost, st);
    case SV_I16: return launch_from<int16_t>(d, src, dst, n, lost, st);
    case SV_U16: return launch_from<uint16_t>(d, src, dst, n, lost, st);
    case SV_U64: return launch_from<uint64_t>(d, src, dst, n, lost, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace sv
