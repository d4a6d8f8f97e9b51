// Host-only probe of the scaffold's file helpers: reads IN as the element type
// named by the first argument and writes it back to OUT with the same shape.
#include <cstdio>
#include <cstring>
#include <vector>

#include "sv_scaffold.h"

template <class T> static int copy(const char* in, const char* out) {
  std::vector<uint64_t> shape;
  std::vector<T> v = sv_scaffold::read_binary_file<T>(in, &shape);
  sv_scaffold::write_binary_file<T>(out, v.data(), shape);
  std::printf("%zu\n", v.size());
  return 0;
}

int main(int argc, char** argv) {
  if (argc != 4) return 2;
  const char* t = argv[1];
  if (!std::strcmp(t, "float32")) return copy<float>(argv[2], argv[3]);
  if (!std::strcmp(t, "uint8")) return copy<uint8_t>(argv[2], argv[3]);
  if (!std::strcmp(t, "int32")) return copy<int32_t>(argv[2], argv[3]);
  if (!std::strcmp(t, "bfloat16")) return copy<__nv_bfloat16>(argv[2], argv[3]);
  if (!std::strcmp(t, "float64")) return copy<double>(argv[2], argv[3]);
  return 2;
}
