// alu_peak.cu -- measures the two ALU rates that bound the normal-value
// generator on this GPU: Philox-4x32-10 blocks and Box-Muller pairs per SM
// per cycle, each run alone at full occupancy with no memory traffic.  The
// generator's ALU roofline for a quantum is the sum of its blocks' and
// pairs' cycle costs.  Prints one JSON line.  Not part of the library.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>

namespace {
constexpr uint32_t kM0 = 0xD2511F53u, kM1 = 0xCD9E8D57u, kW0 = 0x9E3779B9u, kW1 = 0xBB67AE85u;
constexpr int kIter = 256;

__device__ __forceinline__ uint4 block(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint64_t p0 = (uint64_t)kM0 * c.x, p1 = (uint64_t)kM1 * c.z;
    c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ (k0 + r * kW0), (uint32_t)p1, (uint32_t)(p0 >> 32) ^ c.w ^ (k1 + r * kW1),
                   (uint32_t)p0);
  }
  return c;
}

__global__ void philox_kernel(uint32_t* out, uint32_t k0, uint32_t k1) {
  uint32_t acc = 0;
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  for (int i = 0; i < kIter; i += 2) {
    const uint4 a = block(make_uint4(t, i, 7, 0), k0, k1), b = block(make_uint4(t, i + 1, 7, 0), k0, k1);
    acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w;
  }
  if (acc == 0x12345678u) out[t] = acc;  // keeps the work live
}

__device__ __forceinline__ void pair(uint32_t wa, uint32_t wb, float& z0, float& z1) {
  const float u1 = __fmul_rn(__uint2float_rn((wa >> 8) + 1u), 0x1p-24f);
  const float r = sqrtf(__fmul_rn(-2.0f, logf(u1)));
  float s, c;
  sincospif(__fmul_rn(__uint2float_rn(wb >> 8), 0x1p-23f), &s, &c);
  z0 = __fmul_rn(r, c);
  z1 = __fmul_rn(r, s);
}

__global__ void box_muller_kernel(uint32_t* out) {
  float acc = 0.f;
  const uint32_t t = blockIdx.x * blockDim.x + threadIdx.x;
  const uint32_t wa = t * 2654435761u, wb = t * 40503u + 17u;
  for (int i = 0; i < kIter; i += 2) {
    float a0, a1, b0, b1;
    pair(wa + i * 0x9E3779B9u, wb ^ (i * 0x85EBCA6Bu), a0, a1);
    pair(wa ^ (i * 0xC2B2AE35u), wb + i * 0x27D4EB2Fu, b0, b1);
    acc += a0 + a1 + b0 + b1;
  }
  if (acc == 12345.0f) out[t] = 1;
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
  cudaFree(out);
  if (cudaGetLastError() != cudaSuccess) return 1;
  printf("{\"philox_blocks_per_sm_cycle\": %.4f, \"box_muller_pairs_per_sm_cycle\": %.4f, \"sms\": %d, "
         "\"clock_mhz\": %d}\n", philox, bm, sms, clk / 1000);
  return 0;
}
