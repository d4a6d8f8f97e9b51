// Candidate for the in-place vector add task that does not compile (an
// undeclared identifier), for the compilation tool's failure path.
#include <cuda_runtime.h>

__global__ void vec_add_broken(float* a, const float* b, long long n) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) a[i] = a[i] + b[i] * scale_factor;
}

extern "C" int candidate_launch(float* a, const float* b, long long n, void* stream) {
  vec_add_broken<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(a, b, n);
  return (int)cudaGetLastError();
}
