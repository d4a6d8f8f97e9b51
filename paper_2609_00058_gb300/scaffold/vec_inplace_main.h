// vec_inplace_main.h -- main() of a self-contained program for an in-place
// binary fp32 vector task, a <- f(a, b) (the running example of CUDA-Harness,
// vecAddInplace): it reads the prepared inputs with the scaffold's helpers,
// calls the launcher the candidate source defines, writes the output and
// times the launcher (Sec. 4.1.2 scaffold; Eq. 3 latency).  Compiled in front
// of the candidate's source (nvcc -include vec_inplace_main.h candidate.cu).
#pragma once

#include <cuda_runtime.h>

#include <cstdio>
#include <cstdlib>
#include <vector>

#include "sv_scaffold.h"

extern "C" int candidate_launch(float* a, const float* b, long long n, void* stream);

namespace sv_scaffold {
inline void check(cudaError_t e, const char* what) {
  if (e != cudaSuccess) {
    std::fprintf(stderr, "sv_scaffold: %s: %s\n", what, cudaGetErrorString(e));
    std::exit(4);
  }
}
}  // namespace sv_scaffold

int main(int argc, char** argv) {
#pragma message("Calling convention: PROGRAM A.svt B.svt OUT.svt [RUNS]; A, B: float32 [n] tensor files; OUT: float32 [n], A after the in-place launch; with RUNS, also prints 'latency_ms <mean of RUNS launches>' timed on a scratch copy of A")
  using namespace sv_scaffold;
  if (argc < 4) {
    std::fprintf(stderr, "usage: %s A.svt B.svt OUT.svt [RUNS]\n", argv[0]);
    return 2;
  }
  std::vector<uint64_t> shape_a, shape_b;
  std::vector<float> a = read_binary_file<float>(argv[1], &shape_a);
  std::vector<float> b = read_binary_file<float>(argv[2], &shape_b);
  if (a.size() != b.size()) fail(argv[2], "B does not have A's element count");
  const long long n = (long long)a.size();
  float *da = nullptr, *db = nullptr;
  cudaStream_t st;
  check(cudaStreamCreate(&st), "stream");
  check(cudaMalloc(&da, (size_t)n * sizeof(float) + 16), "allocation");
  check(cudaMalloc(&db, (size_t)n * sizeof(float) + 16), "allocation");
  check(cudaMemcpy(da, a.data(), (size_t)n * sizeof(float), cudaMemcpyHostToDevice), "copy");
  check(cudaMemcpy(db, b.data(), (size_t)n * sizeof(float), cudaMemcpyHostToDevice), "copy");
  if (candidate_launch(da, db, n, st) != 0) fail(argv[0], "the launcher returned an error");
  check(cudaStreamSynchronize(st), "launch");
  std::vector<float> out((size_t)n);
  check(cudaMemcpy(out.data(), da, (size_t)n * sizeof(float), cudaMemcpyDeviceToHost), "copy");
  write_binary_file<float>(argv[3], out.data(), shape_a);
  if (argc > 4) {
    const int runs = std::atoi(argv[4]) > 0 ? std::atoi(argv[4]) : 1;
    check(cudaMemcpy(da, a.data(), (size_t)n * sizeof(float), cudaMemcpyHostToDevice), "copy");
    for (int i = 0; i < 3; ++i) candidate_launch(da, db, n, st);
    cudaEvent_t e0, e1;
    check(cudaEventCreate(&e0), "event");
    check(cudaEventCreate(&e1), "event");
    check(cudaEventRecord(e0, st), "event");
    for (int i = 0; i < runs; ++i) candidate_launch(da, db, n, st);
    check(cudaEventRecord(e1, st), "event");
    check(cudaEventSynchronize(e1), "timing");
    float ms = 0.f;
    check(cudaEventElapsedTime(&ms, e0, e1), "timing");
    std::printf("latency_ms %.6f\n", ms / runs);
  }
  cudaFree(da);
  cudaFree(db);
  return 0;
}
