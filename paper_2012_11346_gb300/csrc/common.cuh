// Shared device/host helpers of libslim (no attention arithmetic here).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/slim.h"

namespace slim {

// ---------------------------------------------------------------- dtype I/O
template <typename T> struct Io;
template <> struct Io<float> {
  static __device__ __forceinline__ float load(const float* p, size_t i) { return p[i]; }
  static __device__ __forceinline__ void store(float* p, size_t i, float x) { p[i] = x; }
};
template <> struct Io<__nv_bfloat16> {
  static __device__ __forceinline__ float load(const __nv_bfloat16* p, size_t i) {
    return __bfloat162float(p[i]);
  }
  // round to nearest even
  static __device__ __forceinline__ void store(__nv_bfloat16* p, size_t i, float x) {
    p[i] = __float2bfloat16_rn(x);
  }
};

// ---------------------------------------------------------------- error-free sums
// Knuth's TwoSum: s + e == a + b exactly (round-to-nearest, no FMA contraction
// of these adds -- the intrinsics keep the compiler from reassociating).
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  float bb = __fsub_rn(s, a);
  e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// (hi, lo) += x, then renormalise so |lo| <= ulp(hi)/2.
__device__ __forceinline__ void pair_add(float& hi, float& lo, float x) {
  float s, e;
  two_sum(hi, x, s, e);
  float t = __fadd_rn(lo, e);
  float h2, l2;
  two_sum(s, t, h2, l2);
  hi = h2;
  lo = l2;
}

// ---------------------------------------------------------------- workspace carving
struct Carver {
  char* base;
  size_t off;
  explicit Carver(void* b) : base(static_cast<char*>(b)), off(0) {}
  template <typename T>
  T* take(size_t count) {
    off = (off + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
  size_t bytes() const { return (off + 255) & ~size_t(255); }
};

// One-time, per-device set-up (kernel attributes such as the dynamic
// shared-memory limit belong to the device that was current when they were
// set).  Returns the current device's flag, or null when it cannot be told.
constexpr int kMaxDevices = 64;
inline bool* device_flag(bool (&flags)[kMaxDevices]) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  return &flags[dev];
}

struct Problem {
  int B, H, L, d, M, C;
  slim_dtype dtype;
  slim_feature feature;
  int chains() const { return B * H; }
  int slice_len() const { return C < L ? C : L; }  // C > L behaves as C = L
  int num_slices() const { int c = slice_len(); return L == 0 ? 0 : (L + c - 1) / c; }
};

// Final state handed from the forward to the backward: fp32 values plus the
// optional low-order residuals of the carried value/error pair.
struct StateOut {
  float *S, *z, *S_lo, *z_lo;
};
struct StateIn {
  const float *S, *z, *S_lo, *z_lo;
};
// The state a forward sweep starts from, B^(0) (all null: zero), and the
// state gradient a backward sweep starts from, G^(N) (null: zero), and
// returns, G^(0) (null: not returned) -- the values a sequence cut into
// segments hands from one call to the next (Sec. 3.2, eq. 16; Sec. 3.3, eq. 18).
struct StateInit {
  const float *S, *z, *S_lo, *z_lo;
};
struct GradIO {
  const float *S_in, *z_in;
  float *S_out, *z_out;
};

}  // namespace slim
