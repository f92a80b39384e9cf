// Carried-state scans over the tiles of one slice (shared by both paths).
#pragma once
#include <cuda_runtime.h>

#include "profiler.h"

namespace slim {

enum ScanMode {
  SCAN_FWD = 0,       // P_t = B + sum_{t'<t} D_t' (in place), then B += sum_t D_t
  SCAN_ROLLBACK = 1,  // B -= sum_t D_t (eq. 17), then P_t as SCAN_FWD, B left rolled back
  SCAN_GREV = 2       // G_t = G + sum_{t'>t} D_t' (in place), then G += sum_t D_t
};

// buf: [chains][nt][E] fp32 tile totals, rewritten in place with the per-tile
// state; hi/lo: [chains][E] fp32 value/error pair of the carried state.
cudaError_t launch_scan(cudaStream_t s, float* buf, float* hi, float* lo, int chains, int nt,
                        int E, ScanMode mode, prof::Kid kid);

}  // namespace slim
