// Per-thread body of the carried-state scans (see scan.h); shared by the scan
// kernel and the multiplexed small kernels of the tensor-core path.
#pragma once
#include "common.cuh"
#include "scan.h"

namespace slim {

__device__ __forceinline__ void pair_add4(float4& h, float4& l, const float4& x) {
  pair_add(h.x, l.x, x.x);
  pair_add(h.y, l.y, x.y);
  pair_add(h.z, l.z, x.z);
  pair_add(h.w, l.w, x.w);
}
__device__ __forceinline__ float4 pair_val4(const float4& h, const float4& l) {
  return make_float4(h.x + l.x, h.y + l.y, h.z + l.z, h.w + l.w);
}
__device__ __forceinline__ float4 neg4(const float4& x) { return make_float4(-x.x, -x.y, -x.z, -x.w); }

// One thread per (chain, 4 consecutive state elements); tiles are loaded in
// batches of KB so their latencies overlap, then folded in order.
constexpr int KB = 8;
__device__ __forceinline__ void scan_thread(float4* buf, float4* hi_p, float4* lo_p, int chains,
                                            int nt, int E4, int mode, long long idx) {
  if (idx >= (long long)chains * E4) return;
  const int c = (int)(idx / E4), e = (int)(idx % E4);
  float4 hi = hi_p[idx], lo = lo_p[idx];
  float4* col = buf + (size_t)c * nt * E4 + e;
  float4 x[KB];
  if (mode == SCAN_GREV) {
    // G_t = G + sum_{t' > t} Gd_t'  (reversed prefix sum), then G += all
    for (int t0 = nt - 1; t0 >= 0; t0 -= KB) {
#pragma unroll
      for (int k = 0; k < KB; ++k)
        if (t0 - k >= 0) x[k] = col[(size_t)(t0 - k) * E4];
#pragma unroll
      for (int k = 0; k < KB; ++k)
        if (t0 - k >= 0) {
          col[(size_t)(t0 - k) * E4] = pair_val4(hi, lo);
          pair_add4(hi, lo, x[k]);
        }
    }
    hi_p[idx] = hi;
    lo_p[idx] = lo;
    return;
  }
  if (mode == SCAN_ROLLBACK) {
    // eq. 17: B^(n-1) = B^(n) - sum_t Delta_t, undone in reverse order
    for (int t0 = nt - 1; t0 >= 0; t0 -= KB) {
#pragma unroll
      for (int k = 0; k < KB; ++k)
        if (t0 - k >= 0) x[k] = col[(size_t)(t0 - k) * E4];
#pragma unroll
      for (int k = 0; k < KB; ++k)
        if (t0 - k >= 0) pair_add4(hi, lo, neg4(x[k]));
    }
    hi_p[idx] = hi;
    lo_p[idx] = lo;
  }
  for (int t0 = 0; t0 < nt; t0 += KB) {
#pragma unroll
    for (int k = 0; k < KB; ++k)
      if (t0 + k < nt) x[k] = col[(size_t)(t0 + k) * E4];
#pragma unroll
    for (int k = 0; k < KB; ++k)
      if (t0 + k < nt) {
        col[(size_t)(t0 + k) * E4] = pair_val4(hi, lo);
        pair_add4(hi, lo, x[k]);
      }
  }
  if (mode == SCAN_FWD) {
    hi_p[idx] = hi;
    lo_p[idx] = lo;
  }
}


}  // namespace slim
