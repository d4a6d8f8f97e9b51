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
template <> __device__ __forceinline__ bool src_nan<double>(double x) {  // integer tests: no fp64 instruction
  const unsigned long long b = (unsigned long long)__double_as_longlong(x);
  return (b & 0x7FFFFFFFFFFFFFFFull) > 0x7FF0000000000000ull;
}
template <class S> __device__ __forceinline__ bool src_inf(S) { return false; }
template <> __device__ __forceinline__ bool src_inf<F16>(F16 x) { return (x.b & 0x7FFFu) == 0x7C00u; }
template <> __device__ __forceinline__ bool src_inf<BF16>(BF16 x) { return (x.b & 0x7FFFu) == 0x7F80u; }
template <> __device__ __forceinline__ bool src_inf<float>(float x) { return isinf(x); }
template <> __device__ __forceinline__ bool src_inf<double>(double x) {
  const unsigned long long b = (unsigned long long)__double_as_longlong(x);
  return (b & 0x7FFFFFFFFFFFFFFFull) == 0x7FF0000000000000ull;
}

// ---- rounding with integer steps ----
// GB300's fp64 pipe is narrow, so no fp64 instruction takes part: a value
// (-1)^sign * M * 2^E (M > 0 an integer) is rounded on the integer pipes.
enum Mode { kNearestEven, kOdd };

// to fp32 bits; *over set when a finite value rounds past the largest float
template <Mode kMode>
__device__ __forceinline__ uint32_t round_f32(uint32_t sign, uint64_t M, int E, uint32_t& over) {
  const int p = 63 - __clzll((long long)M);  // top bit of M
  const int fe = p + E + 127;                // biased exponent of a normal result
  if (fe >= 255) {
    ++over;
    return sign | 0x7F800000u;
  }
  const int shift = fe >= 1 ? p - 23 : p - 23 + (1 - fe);  // bits of M below the last kept place
  uint64_t kept, rest = 0, half = 0;
  if (shift <= 0) {
    kept = M << (-shift);
  } else if (shift < 64) {
    kept = M >> shift;
    rest = M & ((1ull << shift) - 1);
    half = 1ull << (shift - 1);
  } else {  // below half of the smallest subnormal (shift 64: M < 2^64 = 2 * half)
    kept = 0;
    rest = M;
    half = shift == 64 ? (1ull << 63) : ~0ull;
  }
  // the exponent field and the kept bits add up, so a carry moves to the next binade
  uint32_t bits = (fe >= 1 ? (uint32_t)(fe - 1) << 23 : 0u) + (uint32_t)kept;
  if (kMode == kNearestEven) {
    bits += (rest > half || (rest == half && rest != 0 && (bits & 1u))) ? 1u : 0u;
    if (bits >= 0x7F800000u) ++over;
  } else {
    bits |= rest != 0 ? 1u : 0u;
  }
  return sign | bits;
}

// to fp64 bits, to nearest even; every source here is inside fp64's normal range
__device__ __forceinline__ unsigned long long round_f64(uint64_t sign, uint64_t M, int E) {
  const int p = 63 - __clzll((long long)M);
  const int fe = p + E + 1023;
  const int shift = p - 52;
  uint64_t bits;
  if (shift <= 0) {
    bits = ((uint64_t)(fe - 1) << 52) + (M << (-shift));
  } else {
    const uint64_t kept = M >> shift, rest = M & ((1ull << shift) - 1), half = 1ull << (shift - 1);
    bits = ((uint64_t)(fe - 1) << 52) + kept;
    bits += (rest > half || (rest == half && (bits & 1u))) ? 1u : 0u;
  }
  return sign | bits;
}

// ---- a source element as (NaN, infinity, sign, M, E) ----
struct Parts {
  bool nan, inf;
  uint32_t neg;  // 1 for a negative value (or -0)
  uint64_t M;    // 0 for a zero
  int E;
};

template <class S> __device__ __forceinline__ Parts parts(S x) {  // integers
  if constexpr (Info<S>::kSigned) {
    const long long v = (long long)x;
    return Parts{false, false, v < 0 ? 1u : 0u, v < 0 ? 0ull - (unsigned long long)v : (unsigned long long)v, 0};
  } else {
    return Parts{false, false, 0u, (unsigned long long)x, 0};
  }
}
__device__ __forceinline__ Parts float_parts(uint64_t b, int frac_bits, int exp_bits) {
  const int width = 1 + exp_bits + frac_bits;
  const uint64_t frac = b & ((1ull << frac_bits) - 1);
  const int e = (int)((b >> frac_bits) & ((1u << exp_bits) - 1));
  const int bias = (1 << (exp_bits - 1)) - 1;
  Parts r;
  r.neg = (uint32_t)(b >> (width - 1)) & 1u;
  r.nan = e == (1 << exp_bits) - 1 && frac != 0;
  r.inf = e == (1 << exp_bits) - 1 && frac == 0;
  r.M = e ? (frac | (1ull << frac_bits)) : frac;
  r.E = (e ? e : 1) - bias - frac_bits;
  return r;
}
template <> __device__ __forceinline__ Parts parts<F16>(F16 x) { return float_parts(x.b, 10, 5); }
template <> __device__ __forceinline__ Parts parts<BF16>(BF16 x) { return float_parts(x.b, 7, 8); }
template <> __device__ __forceinline__ Parts parts<float>(float x) { return float_parts(__float_as_uint(x), 23, 8); }
template <> __device__ __forceinline__ Parts parts<double>(double x) {
  return float_parts((uint64_t)__double_as_longlong(x), 52, 11);
}

// the source value in fp32: exact where it fits, else rounded (to nearest
// even, or to odd as the first step toward a 16-bit float)
template <Mode kMode, class S> __device__ __forceinline__ float to_f32(S x, uint32_t& over) {
  if constexpr (std::is_same<S, float>::value) {
    return x;
  } else if constexpr (std::is_same<S, F16>::value) {
    return __half2float(__ushort_as_half(x.b));  // exact
  } else if constexpr (std::is_same<S, BF16>::value) {
    return __uint_as_float((uint32_t)x.b << 16);  // exact
  } else if constexpr (!Info<S>::kFloat && sizeof(S) <= 2) {
    return (float)x;  // exact
  } else if constexpr (std::is_same<S, int32_t>::value || std::is_same<S, uint32_t>::value) {
    // one 32-bit conversion instruction; to odd: truncate, and mark it when
    // the truncated value converts back to another integer
    if constexpr (kMode == kNearestEven) {
      return std::is_same<S, int32_t>::value ? __int2float_rn((int)x) : __uint2float_rn((unsigned)x);
    } else if constexpr (std::is_same<S, int32_t>::value) {
      const float r = __int2float_rz((int)x);
      return __uint_as_float(__float_as_uint(r) | (__float2int_rz(r) != (int)x ? 1u : 0u));
    } else {
      const float r = __uint2float_rz((unsigned)x);
      return __uint_as_float(__float_as_uint(r) | (__float2uint_rz(r) != (unsigned)x ? 1u : 0u));
    }
  } else if constexpr (kMode == kNearestEven && (std::is_same<S, int64_t>::value ||
                                                  std::is_same<S, uint64_t>::value)) {
    // to nearest: the 64-bit integer conversion instruction
    return std::is_same<S, int64_t>::value ? __ll2float_rn((long long)x) : __ull2float_rn((unsigned long long)x);
  } else {  // 64-bit integers (to odd) and fp64: integer rounding
    if constexpr (std::is_same<S, double>::value) {
      // fast path, 32-bit steps: a result in fp32's normal range (biased fp64
      // exponent 897 ... 1150); the top 35 bits of the fp64 encoding less the
      // exponent offset are the truncated fp32 encoding, the low 29 bits decide
      // the rounding
      const unsigned long long b = (unsigned long long)__double_as_longlong(x);
      const uint32_t hi = (uint32_t)(b >> 32), lo = (uint32_t)b;
      const uint32_t e = (hi >> 20) & 0x7FFu;
      if (e - 897u <= 253u) {
        uint32_t bits = (((hi & 0x7FFFFFFFu) - (896u << 20)) << 3) | (lo >> 29);
        const uint32_t rest = lo & 0x1FFFFFFFu;
        if (kMode == kNearestEven) {
          bits += (rest > 0x10000000u || (rest == 0x10000000u && (bits & 1u))) ? 1u : 0u;
          if (bits >= 0x7F800000u) ++over;
        } else {
          bits |= rest != 0 ? 1u : 0u;
        }
        return __uint_as_float((hi & 0x80000000u) | bits);
      }
    }
    const Parts q = parts(x);  // the general case
    const uint32_t sign = q.neg << 31;
    if (q.inf) return __uint_as_float(sign | 0x7F800000u);
    if (q.M == 0) return __uint_as_float(sign);
    return __uint_as_float(round_f32<kMode>(sign, q.M, q.E, over));
  }
}

template <class D, class S> __device__ __forceinline__ D convert(S x, uint32_t& lost) {
  if constexpr (std::is_same<D, double>::value) {
    if (src_nan(x)) return __longlong_as_double((long long)kNanF64);
    if constexpr (std::is_same<S, float>::value) {  // fast path: a normal fp32 widens by moving its fields
      const uint32_t b = __float_as_uint(x), e = (b >> 23) & 0xFFu;
      if (e - 1u <= 253u) {
        const uint32_t hi = (b & 0x80000000u) | ((e + 896u) << 20) | ((b & 0x7FFFFFu) >> 3);
        return __longlong_as_double((long long)(((unsigned long long)hi << 32) | (unsigned long long)(b << 29)));
      }
    } else if constexpr (std::is_same<S, int32_t>::value || std::is_same<S, uint32_t>::value) {
      return (double)x;  // exact: one 32-bit to fp64 conversion
    }
    const Parts q = parts(x);
    const uint64_t sign = (uint64_t)q.neg << 63;
    if (q.inf) return __longlong_as_double((long long)(sign | 0x7FF0000000000000ull));
    if (q.M == 0) return __longlong_as_double((long long)sign);
    return __longlong_as_double((long long)round_f64(sign, q.M, q.E));
  } else if constexpr (std::is_same<D, float>::value) {
    if (src_nan(x)) return __uint_as_float(kNanF32);
    uint32_t over = 0;
    const float r = to_f32<kNearestEven>(x, over);
    lost += over;
    return r;
  } else if constexpr (std::is_same<D, F16>::value) {
    if (src_nan(x)) return F16{kNanF16};
    uint32_t unused = 0;
    const uint16_t h = __half_as_ushort(__float2half_rn(to_f32<kOdd>(x, unused)));
    lost += ((h & 0x7FFFu) == 0x7C00u && !src_inf(x)) ? 1u : 0u;
    return F16{h};
  } else if constexpr (std::is_same<D, BF16>::value) {
    if (src_nan(x)) return BF16{kNanBF16};
    uint32_t unused = 0;
    const uint16_t h = __bfloat16_as_ushort(__float2bfloat16_rn(to_f32<kOdd>(x, unused)));
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

// a thread's run of kBytes (a power of two, 2 to 16) of consecutive bytes:
// adjacent lanes hold adjacent runs, so every warp access is coalesced
template <int kBytes> struct Run;
template <> struct Run<16> { using T = uint4; };
template <> struct Run<8> { using T = uint2; };
template <> struct Run<4> { using T = unsigned int; };
template <> struct Run<2> { using T = unsigned short; };

template <class S, class D>
__global__ void __launch_bounds__(kThreads) cvt_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst,
                                                       uint64_t n, unsigned long long* __restrict__ lost) {
  constexpr int kE = 16 / (int)(sizeof(S) > sizeof(D) ? sizeof(S) : sizeof(D));  // elements per thread step
  constexpr int kIn = kE * (int)sizeof(S), kOut = kE * (int)sizeof(D);          // at most 16 bytes each
  constexpr int kU = 4;                                                          // steps in flight per thread
  using In = typename Run<kIn>::T;
  using Out = typename Run<kOut>::T;
  const uint64_t nv = n / kE;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  uint64_t v = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t my_lost = 0;
  const In* in = reinterpret_cast<const In*>(src);
  Out* out = reinterpret_cast<Out*>(dst);
  for (; v + (kU - 1) * stride < nv; v += kU * stride) {
    In r[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) r[u] = __ldcs(in + v + u * stride);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      S e[kE];
      memcpy(e, &r[u], kIn);
      D o[kE];
#pragma unroll
      for (int i = 0; i < kE; ++i) o[i] = convert<D>(e[i], my_lost);
      Out w;
      memcpy(&w, o, kOut);
      __stcs(out + v + u * stride, w);
    }
  }
  for (; v < nv; v += stride) {
    const In r = __ldcs(in + v);
    S e[kE];
    memcpy(e, &r, kIn);
    D o[kE];
#pragma unroll
    for (int i = 0; i < kE; ++i) o[i] = convert<D>(e[i], my_lost);
    Out w;
    memcpy(&w, o, kOut);
    __stcs(out + v, w);
  }
  // the ragged tail (fewer than kE elements): one element per thread, typed
  // accesses (both arrays are aligned to their element size)
  const uint64_t t = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t < n - nv * kE) {
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
    constexpr int kE = 16 / (int)(sizeof(S) > sizeof(D) ? sizeof(S) : sizeof(D));
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
