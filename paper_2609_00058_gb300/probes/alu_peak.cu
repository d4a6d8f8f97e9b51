// alu_peak.cu -- measures the ALU rates that bound the generator on this GPU:
// Philox-4x32-10 blocks (two interleaved under one key, as the generator
// draws them), Box-Muller pairs (the generator's own fp32 transform) and fp32
// fused multiply-adds (scalar and packed), each run alone at full occupancy
// with no memory traffic, per SM per cycle at the maximum clock.  The
// generator's ALU roofline for a quantum is the sum of its blocks', pairs'
// and FMAs' cycle costs.  Prints one JSON line.  Not part of the library.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>

#include "../csrc/sv_device.cuh"

namespace {
constexpr int kIter = 256;
constexpr int kFmaIter = 4096;  // long enough (about 0.5 ms a launch) for a steady clock

__global__ void philox_kernel(uint32_t* out, uint32_t k0, uint32_t k1) {
  const sv::RoundKeys rk = sv::round_keys(sv::Key{k0, k1});
  uint32_t acc = 0;
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  for (int i = 0; i < kIter; i += 2) {
    uint4 a = make_uint4(t, i, 7, 0), b = make_uint4(t, i + 1, 7, 0);
    sv::philox2_rk(a, b, rk);
    acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w;
  }
  if (acc == 0x12345678u) out[t] = acc;  // keeps the work live
}

__global__ void box_muller_kernel(uint32_t* out) {
  float acc = 0.f;
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  const uint32_t wa = t * 2654435761u, wb = t * 40503u + 17u;
  for (int i = 0; i < kIter; i += 2) {
    float a0, a1, b0, b1;
    sv::box_muller(wa + i * 0x9E3779B9u, wb ^ (i * 0x85EBCA6Bu), a0, a1);
    sv::box_muller(wa ^ (i * 0xC2B2AE35u), wb + i * 0x27D4EB2Fu, b0, b1);
    acc += a0 + a1 + b0 + b1;
  }
  if (acc == 12345.0f) out[t] = 1;
}

// fp32 fused multiply-adds, scalar and packed pairs (fma.rn.f32x2): 16
// independent accumulators per thread, counted in single FMAs
__global__ void ffma_kernel(float* out, float x) {
  float acc[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) acc[j] = (float)(threadIdx.x + j);
  const float y = x * 0.5f;
  for (int i = 0; i < kFmaIter; i += 16) {
#pragma unroll
    for (int u = 0; u < 16; ++u)
#pragma unroll
      for (int j = 0; j < 16; ++j) acc[j] = __fmaf_rn(acc[j], x, y);
  }
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 16; ++j) s += acc[j];
  if (s == 12345.0f) out[threadIdx.x] = s;
}

__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

__global__ void ffma2_kernel(float* out, float x) {
  uint64_t acc[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const float lo = (float)(threadIdx.x + j), hi = (float)(threadIdx.x + 2 * j);
    acc[j] = ((uint64_t)__float_as_uint(hi) << 32) | __float_as_uint(lo);
  }
  const uint64_t xx = ((uint64_t)__float_as_uint(x) << 32) | __float_as_uint(x);
  const uint64_t yy = ((uint64_t)__float_as_uint(x * 0.5f) << 32) | __float_as_uint(x * 0.5f);
  for (int i = 0; i < kFmaIter; i += 16) {
#pragma unroll
    for (int u = 0; u < 16; ++u)
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = fma2(acc[j], xx, yy);
  }
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) s += __uint_as_float((uint32_t)acc[j]) + __uint_as_float((uint32_t)(acc[j] >> 32));
  if (s == 12345.0f) out[threadIdx.x] = s;
}

template <class F>
double per_sm_cycle(F launch, double units, int sms, int clk_khz) {
  cudaEvent_t a, b;
  cudaEventCreate(&a);
  cudaEventCreate(&b);
  launch();
  cudaEventRecord(a);
  for (int r = 0; r < 5; ++r) launch();
  cudaEventRecord(b);
  cudaEventSynchronize(b);
  float ms = 0;
  cudaEventElapsedTime(&ms, a, b);
  ms /= 5;
  const double cycles = ms * 1e-3 * clk_khz * 1e3;
  return units / sms / cycles;
}
}  // namespace

int main() {
  int sms = 0, clk = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0);
  cudaDeviceGetAttribute(&clk, cudaDevAttrClockRate, 0);
  uint32_t* out = nullptr;
  if (cudaMalloc(&out, (size_t)sms * 8 * 256 * sizeof(uint32_t)) != cudaSuccess) return 1;
  const int blocks = sms * 8, threads = 256;
  const double work = (double)blocks * threads * kIter;
  const double philox = per_sm_cycle([&] { philox_kernel<<<blocks, threads>>>(out, 1, 2); }, work, sms, clk);
  const double bm = per_sm_cycle([&] { box_muller_kernel<<<blocks, threads>>>(out); }, work, sms, clk);
  float* fout = reinterpret_cast<float*>(out);
  const double fwork = (double)blocks * threads * kFmaIter * 16;
  const double ffma = per_sm_cycle([&] { ffma_kernel<<<blocks, threads>>>(fout, 0.999f); }, fwork, sms, clk);
  const double ffma2 = per_sm_cycle([&] { ffma2_kernel<<<blocks, threads>>>(fout, 0.999f); }, fwork, sms, clk);
  cudaFree(out);
  if (cudaGetLastError() != cudaSuccess) return 1;
  printf("{\"philox_blocks_per_sm_cycle\": %.4f, \"box_muller_pairs_per_sm_cycle\": %.4f, "
         "\"ffma_per_sm_cycle\": %.2f, \"ffma2_fmas_per_sm_cycle\": %.2f, \"sms\": %d, \"clock_mhz\": %d}\n",
         philox, bm, ffma, ffma2, sms, clk / 1000);
  return 0;
}
