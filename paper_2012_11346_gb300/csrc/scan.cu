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
__global__ void k_scan(float* buf, float* hi_p, float* lo_p, int chains, int nt, int E, int mode) {
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (long long)chains * E) return;
  const int c = (int)(idx / E), e = (int)(idx % E);
  float hi = hi_p[idx], lo = lo_p[idx];
  float* col = buf + (size_t)c * nt * E + e;
  if (mode == SCAN_GREV) {
    // G_t = G + sum_{t' > t} Gd_t'  (reversed prefix sum), then G += all
    for (int t = nt - 1; t >= 0; --t) {
      float x = col[(size_t)t * E];
      col[(size_t)t * E] = hi + lo;
      pair_add(hi, lo, x);
    }
    hi_p[idx] = hi;
    lo_p[idx] = lo;
    return;
  }
  if (mode == SCAN_ROLLBACK) {
    // eq. 17: B^(n-1) = B^(n) - sum_t Delta_t, undone in reverse order
    for (int t = nt - 1; t >= 0; --t) pair_add(hi, lo, -col[(size_t)t * E]);
    hi_p[idx] = hi;
    lo_p[idx] = lo;
  }
  for (int t = 0; t < nt; ++t) {
    float x = col[(size_t)t * E];
    col[(size_t)t * E] = hi + lo;
    pair_add(hi, lo, x);
  }
  if (mode == SCAN_FWD) {
    hi_p[idx] = hi;
    lo_p[idx] = lo;
  }
}


cudaError_t launch_scan(cudaStream_t s, float* buf, float* hi, float* lo, int chains, int nt,
                        int E, ScanMode mode, prof::Kid kid) {
  const long long n = (long long)chains * E;
  prof::Scope ps(kid, s);
  k_scan<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(buf, hi, lo, chains, nt, E, (int)mode);
  return cudaGetLastError();
}

}  // namespace slim
