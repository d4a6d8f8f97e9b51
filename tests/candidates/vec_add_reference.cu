// Trusted reference for the in-place vector add task: a[i] = a[i] + b[i].
// One thread per element; the plainest form of the operation.
#include <cuda_runtime.h>

__global__ void vec_add_ref(float* a, const float* b, long long n) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) a[i] = __fadd_rn(a[i], b[i]);
}

extern "C" int candidate_launch(float* a, const float* b, long long n, void* stream) {
  if (n <= 0) return 0;
  const long long blocks = (n + 255) / 256;
  vec_add_ref<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(a, b, n);
  return (int)cudaGetLastError();
}
