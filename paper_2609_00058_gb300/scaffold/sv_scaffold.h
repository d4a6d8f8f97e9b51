// sv_scaffold.h -- the test-data helpers of a self-contained CUDA program in
// the harness: read_binary_file reads a prepared test input, write_binary_file
// writes an output (the scaffold of CUDA-Harness, Sec. 4.1.2).  Header only,
// host code, no dependency on the synverify library.
//
// Files are tensor files: a 128-byte little-endian header ("SVT1", header
// size, element type, rank, eight extents, element count, data bytes, four
// reserved words) followed by the elements.  A file is read only as the
// element type it holds: asking for float from a uint8 or int32 file is an
// error, not a reinterpretation of its bytes (the loading defect behind
// 31.4% of the false positives analysed in Sec. 5.2.3).  Every error prints
// one line on stderr and ends the program with exit status 3.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <vector>

namespace sv_scaffold {

// element type codes of the tensor file header
template <class T> struct dtype_of;
template <> struct dtype_of<float> { static constexpr uint32_t code = 0; static constexpr const char* name = "float32"; };
template <> struct dtype_of<__half> { static constexpr uint32_t code = 1; static constexpr const char* name = "float16"; };
template <> struct dtype_of<__nv_bfloat16> { static constexpr uint32_t code = 2; static constexpr const char* name = "bfloat16"; };
template <> struct dtype_of<int32_t> { static constexpr uint32_t code = 3; static constexpr const char* name = "int32"; };
template <> struct dtype_of<int64_t> { static constexpr uint32_t code = 4; static constexpr const char* name = "int64"; };
template <> struct dtype_of<uint32_t> { static constexpr uint32_t code = 5; static constexpr const char* name = "uint32"; };
template <> struct dtype_of<uint8_t> { static constexpr uint32_t code = 6; static constexpr const char* name = "uint8"; };
template <> struct dtype_of<int8_t> { static constexpr uint32_t code = 7; static constexpr const char* name = "int8"; };
template <> struct dtype_of<int16_t> { static constexpr uint32_t code = 8; static constexpr const char* name = "int16"; };
template <> struct dtype_of<uint16_t> { static constexpr uint32_t code = 9; static constexpr const char* name = "uint16"; };
template <> struct dtype_of<uint64_t> { static constexpr uint32_t code = 10; static constexpr const char* name = "uint64"; };
template <> struct dtype_of<double> { static constexpr uint32_t code = 11; static constexpr const char* name = "float64"; };

inline const char* dtype_name(uint32_t code) {
  static const char* names[] = {"float32", "float16", "bfloat16", "int32", "int64", "uint32",
                                "uint8", "int8", "int16", "uint16", "uint64", "float64"};
  return code < 12 ? names[code] : "unknown";
}

struct header {
  uint32_t magic, header_bytes, dtype, ndim;
  uint64_t shape[8];
  uint64_t n, data_bytes;
  uint64_t reserved[4];
};
static_assert(sizeof(header) == 128, "tensor file header");
constexpr uint32_t kMagic = 0x31545653u;  // "SVT1"

[[noreturn]] inline void fail(const char* path, const char* what, const char* detail = "") {
  std::fprintf(stderr, "sv_scaffold: %s: %s%s\n", path, what, detail);
  std::exit(3);
}

// The elements of a tensor file of element type T, row-major; its extents go
// to *shape when shape is not null.
template <class T> std::vector<T> read_binary_file(const char* path, std::vector<uint64_t>* shape = nullptr) {
  FILE* f = std::fopen(path, "rb");
  if (!f) fail(path, "cannot open");
  header h;
  if (std::fread(&h, sizeof h, 1, f) != 1 || h.magic != kMagic || h.header_bytes != sizeof h || h.ndim > 8)
    fail(path, "not a tensor file");
  if (h.dtype != dtype_of<T>::code) {
    char msg[96];
    std::snprintf(msg, sizeof msg, "%s, the program reads %s", dtype_name(h.dtype), dtype_of<T>::name);
    fail(path, "element type is ", msg);
  }
  uint64_t n = 1;
  for (uint32_t i = 0; i < h.ndim; ++i) {
    if (h.shape[i] != 0 && n > UINT64_MAX / h.shape[i]) fail(path, "extents overflow");
    n *= h.shape[i];
  }
  if (n != h.n || h.data_bytes != n * sizeof(T)) fail(path, "inconsistent header");
  std::vector<T> v(n);
  if (n && std::fread(v.data(), sizeof(T), n, f) != n) fail(path, "file shorter than its header says");
  if (std::fgetc(f) != EOF) fail(path, "bytes after the data");
  std::fclose(f);
  if (shape) shape->assign(h.shape, h.shape + h.ndim);
  return v;
}

// Writes n = prod(shape) elements of type T from host memory as a tensor file.
template <class T> void write_binary_file(const char* path, const T* data, const std::vector<uint64_t>& shape) {
  if (shape.size() > 8) fail(path, "rank above 8");
  header h = {};
  h.magic = kMagic;
  h.header_bytes = sizeof h;
  h.dtype = dtype_of<T>::code;
  h.ndim = (uint32_t)shape.size();
  uint64_t n = 1;
  for (size_t i = 0; i < shape.size(); ++i) {
    h.shape[i] = shape[i];
    n *= shape[i];
  }
  h.n = n;
  h.data_bytes = n * sizeof(T);
  FILE* f = std::fopen(path, "wb");
  if (!f) fail(path, "cannot create");
  if (std::fwrite(&h, sizeof h, 1, f) != 1 || (n && std::fwrite(data, sizeof(T), n, f) != n) || std::fclose(f) != 0)
    fail(path, "write failed");
}

}  // namespace sv_scaffold
