// bench_alu_peak.cu -- hardware ALU issue rates of the GPU, for bench.py's
// ALU roofline of the dot-like synthesis (K fp32 fused multiply-adds per
// output, which no memory bound limits).
//
// Four plain kernels, none of them the library's code:
//   ffma   8 independent fma.rn.f32 chains per thread     -> fp32 FMA / s
//   ffma2  8 independent fma.rn.f32x2 chains per thread   -> fp32 FMA / s (2 per instruction)
//   imad   8 independent mad.lo.u32 chains per thread     -> 32-bit IMAD / s
//   wide   8 independent mad.wide.u32 chains per thread   -> 32x32->64 IMAD / s
// Grid: 8 CTAs of 256 threads per SM, every thread the same fixed number of
// steps (no data-dependent bound, nothing waits on anything), one store per
// thread at the end so no chain is dead code.  Each kernel runs three times
// after one warm-up; the best time counts.  SM cycles come from clock64 read
// by the first thread of every CTA.
//
// Output: one JSON line on stdout.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>
#include <cstdlib>

constexpr int kThreads = 256, kCtasPerSm = 8, kChains = 8, kUnroll = 8;
constexpr int kIters = 32768;  // steps of kChains x kUnroll operations per thread

__global__ void __launch_bounds__(kThreads) ffma_kernel(float* out, float a, float b, long long* cycles) {
  const long long t0 = clock64();
  float c[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) c[j] = (float)(threadIdx.x + j);
  for (int i = 0; i < kIters; ++i) {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) asm volatile("fma.rn.f32 %0, %0, %1, %2;" : "+f"(c[j]) : "f"(a), "f"(b));
  }
  float s = 0.0f;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s += c[j];
  out[(size_t)blockIdx.x * kThreads + threadIdx.x] = s;
  if (threadIdx.x == 0) cycles[blockIdx.x] = clock64() - t0;
}

// packed pairs: one fma.rn.f32x2 is two fp32 fused multiply-adds
__global__ void __launch_bounds__(kThreads) ffma2_kernel(float* out, float a, float b, long long* cycles) {
  const long long t0 = clock64();
  unsigned long long c[kChains];
  unsigned long long a2, b2;
  asm("mov.b64 %0, {%1, %2};" : "=l"(a2) : "f"(a), "f"(a));
  asm("mov.b64 %0, {%1, %2};" : "=l"(b2) : "f"(b), "f"(b));
#pragma unroll
  for (int j = 0; j < kChains; ++j) {
    const float lo = (float)(threadIdx.x + j), hi = (float)(threadIdx.x + 2 * j);
    asm("mov.b64 %0, {%1, %2};" : "=l"(c[j]) : "f"(lo), "f"(hi));
  }
  for (int i = 0; i < kIters; ++i) {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) asm volatile("fma.rn.f32x2 %0, %0, %1, %2;" : "+l"(c[j]) : "l"(a2), "l"(b2));
  }
  float s = 0.0f;
#pragma unroll
  for (int j = 0; j < kChains; ++j) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(c[j]));
    s += lo + hi;
  }
  out[(size_t)blockIdx.x * kThreads + threadIdx.x] = s;
  if (threadIdx.x == 0) cycles[blockIdx.x] = clock64() - t0;
}

__global__ void __launch_bounds__(kThreads) imad_kernel(uint32_t* out, uint32_t a, uint32_t b, long long* cycles) {
  const long long t0 = clock64();
  uint32_t c[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) c[j] = threadIdx.x + j;
  for (int i = 0; i < kIters; ++i) {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) asm volatile("mad.lo.u32 %0, %0, %1, %2;" : "+r"(c[j]) : "r"(a), "r"(b));
  }
  uint32_t s = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s ^= c[j];
  out[(size_t)blockIdx.x * kThreads + threadIdx.x] = s;
  if (threadIdx.x == 0) cycles[blockIdx.x] = clock64() - t0;
}

__global__ void __launch_bounds__(kThreads) wide_kernel(uint64_t* out, uint32_t a, long long* cycles) {
  const long long t0 = clock64();
  uint64_t c[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) c[j] = threadIdx.x + j;
  for (int i = 0; i < kIters; ++i) {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
#pragma unroll
      for (int j = 0; j < kChains; ++j) {
        // the 64-bit product of the chain's low word and a, plus the chain
        uint32_t lo = (uint32_t)c[j];
        asm volatile("mad.wide.u32 %0, %1, %2, %0;" : "+l"(c[j]) : "r"(lo), "r"(a));
      }
  }
  uint64_t s = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s ^= c[j];
  out[(size_t)blockIdx.x * kThreads + threadIdx.x] = s;
  if (threadIdx.x == 0) cycles[blockIdx.x] = clock64() - t0;
}

#define CHECK(x)                                                          \
  do {                                                                    \
    cudaError_t e_ = (x);                                                 \
    if (e_ != cudaSuccess) {                                              \
      fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));            \
      return 1;                                                           \
    }                                                                     \
  } while (0)

struct Rate {
  double ops_per_s, ops_per_sm_cycle, mhz;
};

// best of three timed runs of `launch` (one warm-up first)
template <class F>
static int time_kernel(F launch, int grid, long long* d_cycles, int sms, Rate* r) {
  const double ops = (double)grid * kThreads * kIters * kUnroll * kChains;
  cudaEvent_t e0, e1;
  CHECK(cudaEventCreate(&e0));
  CHECK(cudaEventCreate(&e1));
  launch();
  CHECK(cudaGetLastError());
  CHECK(cudaDeviceSynchronize());
  float best = 1e30f;
  long long* h = (long long*)malloc(sizeof(long long) * grid);
  double best_cycles = 0.0;
  for (int rep = 0; rep < 3; ++rep) {
    CHECK(cudaEventRecord(e0));
    launch();
    CHECK(cudaEventRecord(e1));
    CHECK(cudaEventSynchronize(e1));
    float ms = 0.0f;
    CHECK(cudaEventElapsedTime(&ms, e0, e1));
    if (ms < best) {
      best = ms;
      CHECK(cudaMemcpy(h, d_cycles, sizeof(long long) * grid, cudaMemcpyDeviceToHost));
      long long mx = 0;
      for (int i = 0; i < grid; ++i) mx = h[i] > mx ? h[i] : mx;
      best_cycles = (double)mx;
    }
  }
  free(h);
  r->ops_per_s = ops / (best * 1e-3);
  // every SM runs the same share: ops per SM over the longest CTA's cycles
  r->ops_per_sm_cycle = best_cycles > 0 ? ops / sms / best_cycles : 0.0;
  r->mhz = best_cycles / (best * 1e-3) / 1e6;
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  return 0;
}

int main() {
  int dev = 0, sms = 0;
  CHECK(cudaGetDevice(&dev));
  CHECK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int grid = sms * kCtasPerSm;
  void* buf = nullptr;
  long long* cyc = nullptr;
  CHECK(cudaMalloc(&buf, (size_t)grid * kThreads * sizeof(uint64_t)));
  CHECK(cudaMalloc(&cyc, (size_t)grid * sizeof(long long)));
  Rate f{}, f2{}, m{}, w{};
  if (time_kernel([&] { ffma_kernel<<<grid, kThreads>>>((float*)buf, 0.999999f, 1e-7f, cyc); }, grid, cyc, sms, &f))
    return 1;
  if (time_kernel([&] { ffma2_kernel<<<grid, kThreads>>>((float*)buf, 0.999999f, 1e-7f, cyc); }, grid, cyc, sms,
                  &f2))
    return 1;
  f2.ops_per_s *= 2;  // two FMAs per packed instruction
  f2.ops_per_sm_cycle *= 2;
  if (time_kernel([&] { imad_kernel<<<grid, kThreads>>>((uint32_t*)buf, 0x9E3779B9u, 7u, cyc); }, grid, cyc, sms, &m))
    return 1;
  if (time_kernel([&] { wide_kernel<<<grid, kThreads>>>((uint64_t*)buf, 0xD2511F53u, cyc); }, grid, cyc, sms, &w))
    return 1;
  CHECK(cudaFree(buf));
  CHECK(cudaFree(cyc));
  printf("{\"sms\": %d, \"ffma_per_s\": %.6g, \"ffma_per_sm_cycle\": %.4f, \"ffma_mhz\": %.1f, "
         "\"ffma2_fma_per_s\": %.6g, \"ffma2_fma_per_sm_cycle\": %.4f, "
         "\"imad_per_s\": %.6g, \"imad_per_sm_cycle\": %.4f, \"imad_wide_per_s\": %.6g, "
         "\"imad_wide_per_sm_cycle\": %.4f}\n",
         sms, f.ops_per_s, f.ops_per_sm_cycle, f.mhz, f2.ops_per_s, f2.ops_per_sm_cycle, m.ops_per_s,
         m.ops_per_sm_cycle, w.ops_per_s, w.ops_per_sm_cycle);
  return 0;
}
