// append_common.cuh -- small device helpers shared by the append kernels:
// vector loads, the 128-byte swizzled operand layout, and the ordered top-k
// insertion used by the candidate selection.
#pragma once
#include "ptx_sm103.cuh"

namespace qwm {
namespace {

__device__ __forceinline__ uint4 ldg16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ uint4 lds16(const uint8_t* p) { return *reinterpret_cast<const uint4*>(p); }
// 32-byte read-only global load (address 32-byte aligned): one whole sector.
__device__ __forceinline__ void ldg32(const void* p, uint32_t (&r)[8]) {
  asm volatile("ld.global.nc.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
               : "l"(p));
}

// Byte offset of 16-byte chunk `ch` (channels 8ch..8ch+7) of row `row` in a
// pair of 128-byte-swizzled blocks of `rows` rows x 64 two-byte elements.
__device__ __forceinline__ int sw_off(int rows, int row, int ch) {
  return (ch >> 3) * rows * 128 + row * 128 + (((ch & 7) ^ (row & 7)) << 4);
}

// Insert (v, j) into the ascending list of the n smallest (value, index)
// pairs; indices arrive in ascending order, so an equal value stays behind.
template <int CAP>
__device__ __forceinline__ void insert_top(float (&tv)[CAP], int (&tj)[CAP], int n, float v, int j) {
#pragma unroll
  for (int s = 0; s < CAP; ++s) {
    if (s < n && v < tv[s]) {
      const float ov = tv[s];
      const int oj = tj[s];
      tv[s] = v;
      tj[s] = j;
      v = ov;
      j = oj;
    }
  }
}
template <int CAP>
__device__ __forceinline__ float sel_at(const float (&tv)[CAP], int i) {
  float k = tv[0];
#pragma unroll
  for (int s = 1; s < CAP; ++s)
    if (s == i) k = tv[s];
  return k;
}

__device__ __forceinline__ float sel4(const float (&a)[4], int g) {
  return g == 0 ? a[0] : (g == 1 ? a[1] : (g == 2 ? a[2] : a[3]));
}

constexpr float kMagic = 12582912.0f;   // 1.5 * 2^23: (y + kMagic) - kMagic = rint(y) for |y| < 2^22
constexpr float kTwo23 = 8388608.0f;

}  // namespace
}  // namespace qwm
