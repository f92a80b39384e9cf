// slim_fwd_noalloc: the forward sweep with its scratch in a fixed device array
// owned by the library, for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) at the point
// where they run the forward: code running inside an allocator callback or a
// memory-pool hook, a host that forbids allocation after start-up (fixed
// memory budgets, certified or real-time deployments), or a plug-in whose host
// owns every allocation.  For them this entry point uses SLIM_NOALLOC_SCRATCH_BYTES
// of scratch that the library reserves in a file-scope __device__ array; the
// caller still provides every input and output buffer.
#include <mutex>

#include "../../include/slim.h"
#include "common.cuh"
#include "simt_path.h"
#include "tc_path.h"

namespace slim {
slim_status fwd_unreported(const void* q, const void* k, const void* v, const float* omega,
                           int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                           slim_feature feature, void* out, float* S_state, float* z_state,
                           float* S_state_lo, float* z_state_lo, void* workspace,
                           size_t workspace_bytes, cudaStream_t stream);
}

namespace {

// Reserved in a GPU's memory when this library's device code is loaded on that
// GPU, and held until the process exits.  CUDA loads device code lazily: the
// first libslim call that reaches a device (the first slim_fwd_noalloc there
// looks up this array's address) loads it and reserves the array.
static __device__ __align__(256) unsigned char g_noalloc_scratch[SLIM_NOALLOC_SCRATCH_BYTES];

std::mutex g_mu;
void* g_scratch_ptr[slim::kMaxDevices] = {nullptr};

// The array's name in host code is only a host-side stand-in; the kernels need
// its device address, looked up once per device with that device current.
slim_status scratch_for_current_device(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= slim::kMaxDevices) return SLIM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr)
      return SLIM_ERR_CUDA;
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return SLIM_OK;
}

}  // namespace

extern "C" slim_status slim_fwd_noalloc(const void* q, const void* k, const void* v,
                                        const float* omega, int B, int H, int L, int d, int M,
                                        int C, slim_dtype dtype, slim_feature feature, void* out,
                                        float* S_state, float* z_state, float* S_state_lo,
                                        float* z_state_lo, void* stream) {
  // Same argument rules as slim_fwd.
  if (B < 1 || H < 1 || L < 0 || C < 1 || d < 1 || M < 1) return SLIM_ERR_INVALID_ARG;
  if (dtype != SLIM_F32 && dtype != SLIM_BF16) return SLIM_ERR_INVALID_ARG;
  if (feature != SLIM_FEAT_EXP && feature != SLIM_FEAT_RELU && feature != SLIM_FEAT_SQUARE)
    return SLIM_ERR_INVALID_ARG;
  size_t need = 0;
  slim_status st = slim_fwd_workspace_size(B, H, L, d, M, C, dtype, feature, &need);
  if (st != SLIM_OK) return st;
  if (need > (size_t)SLIM_NOALLOC_SCRATCH_BYTES) return SLIM_ERR_WORKSPACE;  // too large here
  void* scratch = nullptr;
  st = scratch_for_current_device(&scratch);
  if (st != SLIM_OK) return st;
  // The forward validates the pointers and clears, on the stream, every part
  // of the scratch that must start at zero (error word, flags, carried state);
  // the rest is written before it is read, so stale contents from an earlier
  // call do not leak into this one.  It runs without the timeout report,
  // which would pin a page of host memory on its first call.
  return slim::fwd_unreported(q, k, v, omega, B, H, L, d, M, C, dtype, feature, out, S_state,
                              z_state, S_state_lo, z_state_lo, scratch,
                              (size_t)SLIM_NOALLOC_SCRATCH_BYTES,
                              static_cast<cudaStream_t>(stream));
}
