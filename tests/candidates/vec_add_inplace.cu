// Candidate for the in-place vector add task: a grid-stride loop over float4
// vectors with a scalar tail (a correct, faster form).
#include <cuda_runtime.h>

__global__ void vec_add_v4(float* a, const float* b, long long n) {
  const long long nv = n / 4;
  const long long stride = (long long)gridDim.x * blockDim.x;
  float4* a4 = reinterpret_cast<float4*>(a);
  const float4* b4 = reinterpret_cast<const float4*>(b);
  for (long long v = (long long)blockIdx.x * blockDim.x + threadIdx.x; v < nv; v += stride) {
    float4 x = a4[v];
    const float4 y = b4[v];
    x.x = __fadd_rn(x.x, y.x);
    x.y = __fadd_rn(x.y, y.y);
    x.z = __fadd_rn(x.z, y.z);
    x.w = __fadd_rn(x.w, y.w);
    a4[v] = x;
  }
  for (long long i = 4 * nv + (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    a[i] = __fadd_rn(a[i], b[i]);
}

extern "C" int candidate_launch(float* a, const float* b, long long n, void* stream) {
  if (n <= 0) return 0;
  int sms = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0);
  long long blocks = (n / 4 + 255) / 256;
  if (blocks > 8LL * sms) blocks = 8LL * sms;
  if (blocks < 1) blocks = 1;
  vec_add_v4<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(a, b, n);
  return (int)cudaGetLastError();
}
