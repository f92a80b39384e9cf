// Carried-state scans over the tiles of one slice; see scan.h.
//
// One thread per (chain, state element).  The state B = (S, z) and its
// gradient G are carried across tiles and slices as an fp32 value/error pair
// (TwoSum), so rolling back by subtraction (eq. 17) in the reverse order of
// the forward additions returns the forward's state to within the pair's
// precision.
#include "common.cuh"
#include "scan.h"
#include "scan_dev.cuh"

namespace slim {

// State scans over the tiles of one slice, one thread per (chain, element).
__global__ void k_scan(float4* buf, float4* hi_p, float4* lo_p, int chains, int nt, int E4,
                       int mode) {
  // the tile totals come from the kernel just before (programmatic launch)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  scan_thread(buf, hi_p, lo_p, chains, nt, E4, mode,
              (long long)blockIdx.x * blockDim.x + threadIdx.x);
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
