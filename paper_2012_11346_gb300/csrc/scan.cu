// Carried-state scans over the tiles of one slice; see scan.h.
//
// One thread per (chain, state element).  The state B = (S, z) and its
// gradient G are carried across tiles and slices as an fp32 value/error pair
// (TwoSum), so rolling back by subtraction (eq. 17) in the reverse order of
// the forward additions returns the forward's state to within the pair's
// precision.
#include "common.cuh"
#include "scan.h"

namespace slim {

// State scans over the tiles of one slice, one thread per (chain, element).
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
__global__ void k_scan(float4* buf, float4* hi_p, float4* lo_p, int chains, int nt, int E4,
                       int mode) {
  // the tile totals come from the kernel just before (programmatic launch)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
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

cudaError_t launch_scan(cudaStream_t s, float* buf, float* hi, float* lo, int chains, int nt,
                        int E, ScanMode mode, prof::Kid kid) {
  // E is a multiple of 4 for every supported shape (M % 16 == 0) and every
  // buffer is 256-byte aligned, so the state is scanned 4 floats at a time.
  const int E4 = E / 4;
  const long long n = (long long)chains * E4;
  // bytes: the tile totals read and rewritten, the pair read and written
  prof::Scope ps(kid, s, 0.0, (double)chains * E * 4.0 * (2.0 * nt + 4.0));
  // launched as a programmatic dependent of the previous kernel in the stream
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((n + 255) / 256));
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_scan, reinterpret_cast<float4*>(buf),
                            reinterpret_cast<float4*>(hi), reinterpret_cast<float4*>(lo), chains, nt,
                            E4, (int)mode);
}

}  // namespace slim
