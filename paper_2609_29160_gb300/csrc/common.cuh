// Internal helpers shared by the library's CUDA translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "tre.h"

namespace tre {

// ---------------------------------------------------------------------------
// IEEE arithmetic with explicit rounding, one operation at a time. The library
// is compiled with -fmad=false as well, but the intrinsics make the intent
// (no contraction, correctly rounded) explicit at every step.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float mul_rn(float a, float b) { return __fmul_rn(a, b); }
__device__ __forceinline__ double mul_rn(double a, double b) { return __dmul_rn(a, b); }
__device__ __forceinline__ float add_rn(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ double add_rn(double a, double b) { return __dadd_rn(a, b); }
__device__ __forceinline__ float div_rn(float a, float b) { return __fdiv_rn(a, b); }
__device__ __forceinline__ double div_rn(double a, double b) { return __ddiv_rn(a, b); }
template <class T> __device__ __forceinline__ T from_i32(int32_t v);
template <> __device__ __forceinline__ float from_i32<float>(int32_t v) { return __int2float_rn(v); }
template <> __device__ __forceinline__ double from_i32<double>(int32_t v) { return __int2double_rn(v); }

// bit pattern of a non-negative value as an order-preserving unsigned key
__device__ __forceinline__ uint32_t key_of(float v) { return __float_as_uint(v); }
__device__ __forceinline__ unsigned long long key_of(double v) {
  return (unsigned long long)__double_as_longlong(v);
}

constexpr int kMaxModels = 1024;

__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }
constexpr uint8_t kCrit = TRE_CRIT, kNom = TRE_NOM, kSurp = TRE_SURP, kIdle = TRE_IDLE;

// floor and remainder of x / d for 0 <= x < 2^63, 1 <= d < 2^31 (32-bit path
// when the dividend fits, which is the common case)
__device__ __forceinline__ void divmod(unsigned long long x, uint32_t d, unsigned long long& q,
                                       unsigned long long& r) {
  if (x <= 0xffffffffull) {
    const uint32_t xx = (uint32_t)x;
    const uint32_t qq = xx / d;
    q = qq;
    r = xx - qq * d;
  } else {
    q = x / d;
    r = x - q * d;
  }
}

// Division of an unsigned 32-bit value by a divisor fixed for the launch,
// without a divide instruction (round-up multiply-high method of Granlund and
// Montgomery): exact for every 32-bit dividend and 1 <= d < 2^31.
struct FastDiv {
  uint32_t d, m, s1, s2;
  FastDiv() = default;
  __host__ __device__ explicit FastDiv(uint32_t div) : d(div) {
    uint32_t l = 0;
    while ((1ull << l) < div) ++l;
    m = (uint32_t)(((1ull << 32) * ((1ull << l) - div)) / div + 1);
    s1 = l > 0 ? 1 : 0;
    s2 = l > 0 ? l - 1 : 0;
  }
  __device__ __forceinline__ uint32_t div(uint32_t x) const {
    const uint32_t t = __umulhi(x, m);
    return (t + ((x - t) >> s1)) >> s2;
  }
};

// Largest i in [0, n) with base[i] * scale <= v, for a non-decreasing table
// (prefix sums of per-series counts) with base[0] * scale <= v: a binary
// search, so a lookup in a 64-entry kernel-parameter table costs six steps.
__device__ __forceinline__ int prefix_index(const int32_t* base, int n, int64_t v,
                                            int64_t scale = 1) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if ((int64_t)base[mid] * scale <= v) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// warp-level sum of a 64-bit counter, one atomic per warp when non-zero
__device__ __forceinline__ void warp_add_counter(unsigned long long* dst, unsigned long long v) {
  const unsigned full = 0xffffffffu;
  for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(full, v, o);
  if ((threadIdx.x & 31) == 0 && v) atomicAdd(dst, v);
}

// Smoothing state carried through a window range: S and whether the model has
// had a non-idle window yet. Summaries compose as affine maps (see score.cu).
template <class T> struct EmaState {
  T S;
  int init;
};

}  // namespace tre
