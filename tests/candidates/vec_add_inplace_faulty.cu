// Candidate for the in-place vector add task with a planted fault: elements at
// and beyond index 2^20 get a * b added instead of b, so small stages pass and
// the first stage larger than 2^20 elements fails.
#include <cuda_runtime.h>

__global__ void vec_add_faulty(float* a, const float* b, long long n) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  a[i] = i < (1LL << 20) ? __fadd_rn(a[i], b[i]) : __fadd_rn(a[i], __fmul_rn(a[i], b[i]));
}

extern "C" int candidate_launch(float* a, const float* b, long long n, void* stream) {
  if (n <= 0) return 0;
  vec_add_faulty<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(a, b, n);
  return (int)cudaGetLastError();
}
