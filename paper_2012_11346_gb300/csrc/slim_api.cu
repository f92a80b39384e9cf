// C ABI of libslim: argument validation, workspace sizing, dispatch.
// Declarations and the contract of every entry point: include/slim.h.
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "common.cuh"
#include "report.h"
#include "simt_path.h"
#include "stack.h"
#include "tc_path.h"

using slim::Problem;

namespace {

constexpr int kVersion = 100;  // 0.1.0

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool pointers_ok(const void* const* ptrs, int n, bool null_allowed) {
  for (int i = 0; i < n; ++i) {
    if (ptrs[i] == nullptr) {
      if (!null_allowed) return false;
    } else if (!aligned16(ptrs[i])) {
      return false;
    }
  }
  return true;
}

slim_status check_problem(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                          slim_feature feature, Problem* out) {
  if (B < 1 || H < 1 || L < 0 || C < 1) return SLIM_ERR_INVALID_ARG;
  if (dtype != SLIM_F32 && dtype != SLIM_BF16) return SLIM_ERR_INVALID_ARG;
  if (feature != SLIM_FEAT_EXP && feature != SLIM_FEAT_RELU && feature != SLIM_FEAT_SQUARE)
    return SLIM_ERR_INVALID_ARG;
  if (d < 1 || M < 1) return SLIM_ERR_INVALID_ARG;
  if (feature == SLIM_FEAT_SQUARE && M != d) return SLIM_ERR_INVALID_ARG;  // g(x)_i = x_i^2
  // element counts must stay far inside 64-bit range, chains inside int
  const long long chains = (long long)B * H;
  if (chains > (1LL << 24)) return SLIM_ERR_INVALID_ARG;
  if ((long long)L * d > (1LL << 40) / chains) return SLIM_ERR_INVALID_ARG;
  if (!(d == 16 || d == 32 || d == 64 || d == 128)) return SLIM_ERR_UNSUPPORTED;
  if (M % 16 != 0 || M > 256) return SLIM_ERR_UNSUPPORTED;
  *out = Problem{B, H, L, d, M, C, dtype, feature};
  return SLIM_OK;
}

// Path selection: the tensor-core path where it applies, else the fp32-compute
// path.  SLIM_PATH=simt in the environment (read on every call) forces the
// fp32-compute path.
bool use_tc(const Problem& p) {
  const char* e = getenv("SLIM_PATH");
  if (e && strcmp(e, "simt") == 0) return false;
  return slim::tc::supports(p);
}

size_t ws_bytes(const Problem& p, bool bwd) {
  return use_tc(p) ? slim::tc::workspace_bytes(p, bwd) : slim::simt::workspace_bytes(p, bwd);
}

slim_status check_workspace(const Problem& p, bool bwd, void* ws, size_t bytes) {
  const size_t need = ws_bytes(p, bwd);
  if (need == 0) return SLIM_OK;
  if (ws == nullptr || bytes < need) return SLIM_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return SLIM_ERR_INVALID_ARG;
  return SLIM_OK;
}

// Both halves of a pair (value, normaliser) given, or neither.
bool pair_ok(const void* a, const void* b) { return (a == nullptr) == (b == nullptr); }

cudaError_t copy_or_zero(float* dst, const float* src, size_t n, cudaStream_t s) {
  if (src) return cudaMemcpyAsync(dst, src, n * sizeof(float), cudaMemcpyDeviceToDevice, s);
  return cudaMemsetAsync(dst, 0, n * sizeof(float), s);
}

// The forward sweep behind slim_fwd, slim_fwd_from and slim_fwd_noalloc.
// report: the non-blocking timeout report of report.cu (off for the
// allocation-free entry point).
slim_status forward(const void* q, const void* k, const void* v, const float* omega, int B,
                    int H, int L, int d, int M, int C, slim_dtype dtype, slim_feature feature,
                    const float* S_init, const float* z_init, const float* S_init_lo,
                    const float* z_init_lo, void* out, float* S_state, float* z_state,
                    float* S_state_lo, float* z_state_lo, void* workspace,
                    size_t workspace_bytes, cudaStream_t s, bool report) {
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  // [B,H,L,d] tensors are empty when L = 0 and may then be null; the quadratic
  // map does not use Omega
  const void* seq[] = {q, k, v, out};
  const void* fixed[] = {S_state, z_state};
  const void* opt[] = {S_state_lo, z_state_lo, S_init, z_init, S_init_lo, z_init_lo, omega};
  if (!pointers_ok(seq, 4, L == 0) || !pointers_ok(fixed, 2, false) || !pointers_ok(opt, 7, true))
    return SLIM_ERR_INVALID_ARG;
  if (omega == nullptr && feature != SLIM_FEAT_SQUARE) return SLIM_ERR_INVALID_ARG;
  if (!pair_ok(S_init, z_init) || (S_init == nullptr && (S_init_lo || z_init_lo)))
    return SLIM_ERR_INVALID_ARG;
  st = check_workspace(p, false, workspace, workspace_bytes);
  if (st != SLIM_OK) return st;
  cudaStream_t s_ = s;
  if (L == 0) {
    // no rows: the state passes through unchanged
    const size_t n = (size_t)p.chains() * M;
    if (copy_or_zero(S_state, S_init, n * d, s_) != cudaSuccess) return SLIM_ERR_CUDA;
    if (copy_or_zero(z_state, z_init, n, s_) != cudaSuccess) return SLIM_ERR_CUDA;
    if (S_state_lo && copy_or_zero(S_state_lo, S_init_lo, n * d, s_) != cudaSuccess)
      return SLIM_ERR_CUDA;
    if (z_state_lo && copy_or_zero(z_state_lo, z_init_lo, n, s_) != cudaSuccess)
      return SLIM_ERR_CUDA;
    return SLIM_OK;
  }
  // the fp32-compute kernels have no device-side waits; only the tensor-core
  // calls take part in the timeout report
  const bool tc = use_tc(p);
  unsigned* counter = nullptr;
  st = slim::report::begin(workspace, report && tc, &counter);
  if (st != SLIM_OK) return st;
  const slim::StateOut so{S_state, z_state, S_state_lo, z_state_lo};
  const slim::StateInit si{S_init, z_init, S_init_lo, z_init_lo};
  if (tc) return slim::tc::fwd(p, q, k, v, omega, out, so, si, counter, workspace, s_);
  return slim::simt::fwd(p, q, k, v, omega, out, so, si, workspace, s_);
}

slim_status backward(const void* q, const void* k, const void* v, const float* omega,
                     const void* out, const void* dout, const float* S_state,
                     const float* z_state, const float* S_state_lo, const float* z_state_lo,
                     const float* G_S_in, const float* g_z_in, int B, int H, int L, int d,
                     int M, int C, slim_dtype dtype, slim_feature feature, void* dq, void* dk,
                     void* dv, float* domega, float* G_S_out, float* g_z_out, void* workspace,
                     size_t workspace_bytes, cudaStream_t s) {
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  const void* seq[] = {q, k, v, out, dout, dq, dk, dv};
  const void* fixed[] = {S_state, z_state};
  const void* opt[] = {S_state_lo, z_state_lo, G_S_in, g_z_in, G_S_out, g_z_out, omega, domega};
  if (!pointers_ok(seq, 8, L == 0) || !pointers_ok(fixed, 2, false) || !pointers_ok(opt, 8, true))
    return SLIM_ERR_INVALID_ARG;
  if ((omega == nullptr || domega == nullptr) && feature != SLIM_FEAT_SQUARE)
    return SLIM_ERR_INVALID_ARG;
  if (!pair_ok(G_S_in, g_z_in) || !pair_ok(G_S_out, g_z_out)) return SLIM_ERR_INVALID_ARG;
  st = check_workspace(p, true, workspace, workspace_bytes);
  if (st != SLIM_OK) return st;
  if (L == 0) {
    if (domega && cudaMemsetAsync(domega, 0, (size_t)M * d * sizeof(float), s) != cudaSuccess)
      return SLIM_ERR_CUDA;
    const size_t n = (size_t)p.chains() * M;
    if (G_S_out && (copy_or_zero(G_S_out, G_S_in, n * d, s) != cudaSuccess ||
                    copy_or_zero(g_z_out, g_z_in, n, s) != cudaSuccess))
      return SLIM_ERR_CUDA;
    return SLIM_OK;
  }
  const bool tc = use_tc(p);
  unsigned* counter = nullptr;
  st = slim::report::begin(workspace, tc, &counter);
  if (st != SLIM_OK) return st;
  const slim::StateIn si{S_state, z_state, S_state_lo, z_state_lo};
  const slim::GradIO gio{G_S_in, g_z_in, G_S_out, g_z_out};
  if (tc)
    return slim::tc::bwd(p, q, k, v, omega, out, dout, si, gio, dq, dk, dv, domega, counter,
                         workspace, s);
  return slim::simt::bwd(p, q, k, v, omega, out, dout, si, gio, dq, dk, dv, domega, workspace, s);
}

}  // namespace

namespace slim {
// slim_fwd without the timeout report (for the allocation-free entry point,
// which must not pin memory on its first call).
slim_status fwd_unreported(const void* q, const void* k, const void* v, const float* omega,
                           int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                           slim_feature feature, void* out, float* S_state, float* z_state,
                           float* S_state_lo, float* z_state_lo, void* workspace,
                           size_t workspace_bytes, cudaStream_t stream) {
  return forward(q, k, v, omega, B, H, L, d, M, C, dtype, feature, nullptr, nullptr, nullptr,
                 nullptr, out, S_state, z_state, S_state_lo, z_state_lo, workspace,
                 workspace_bytes, stream, false);
}
}  // namespace slim

extern "C" {

const char* slim_status_string(slim_status s) {
  switch (s) {
    case SLIM_OK: return "SLIM_OK";
    case SLIM_ERR_INVALID_ARG: return "SLIM_ERR_INVALID_ARG: invalid argument";
    case SLIM_ERR_UNSUPPORTED: return "SLIM_ERR_UNSUPPORTED: unsupported (d, M, dtype, feature)";
    case SLIM_ERR_WORKSPACE: return "SLIM_ERR_WORKSPACE: workspace missing or too small";
    case SLIM_ERR_CUDA: return "SLIM_ERR_CUDA: a CUDA launch or runtime call failed";
    case SLIM_ERR_TIMEOUT: return "SLIM_ERR_TIMEOUT: a bounded device-side wait gave up";
  }
  return "unknown slim_status";
}

int slim_version(void) { return kVersion; }

slim_status slim_fwd_workspace_size(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                                    slim_feature feature, size_t* bytes) {
  if (!bytes) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  *bytes = ws_bytes(p, false);
  return SLIM_OK;
}

slim_status slim_bwd_workspace_size(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                                    slim_feature feature, size_t* bytes) {
  if (!bytes) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  *bytes = ws_bytes(p, true);
  return SLIM_OK;
}

slim_status slim_fwd(const void* q, const void* k, const void* v, const float* omega, int B,
                     int H, int L, int d, int M, int C, slim_dtype dtype, slim_feature feature,
                     void* out, float* S_state, float* z_state, float* S_state_lo,
                     float* z_state_lo, void* workspace, size_t workspace_bytes, void* stream) {
  return forward(q, k, v, omega, B, H, L, d, M, C, dtype, feature, nullptr, nullptr, nullptr,
                 nullptr, out, S_state, z_state, S_state_lo, z_state_lo, workspace,
                 workspace_bytes, static_cast<cudaStream_t>(stream), true);
}

slim_status slim_fwd_from(const void* q, const void* k, const void* v, const float* omega, int B,
                          int H, int L, int d, int M, int C, slim_dtype dtype,
                          slim_feature feature, const float* S_init, const float* z_init,
                          const float* S_init_lo, const float* z_init_lo, void* out,
                          float* S_state, float* z_state, float* S_state_lo, float* z_state_lo,
                          void* workspace, size_t workspace_bytes, void* stream) {
  return forward(q, k, v, omega, B, H, L, d, M, C, dtype, feature, S_init, z_init, S_init_lo,
                 z_init_lo, out, S_state, z_state, S_state_lo, z_state_lo, workspace,
                 workspace_bytes, static_cast<cudaStream_t>(stream), true);
}

slim_status slim_bwd(const void* q, const void* k, const void* v, const float* omega,
                     const void* out, const void* dout, const float* S_state,
                     const float* z_state, const float* S_state_lo, const float* z_state_lo,
                     int B, int H, int L, int d, int M, int C,
                     slim_dtype dtype, slim_feature feature, void* dq, void* dk, void* dv,
                     float* domega, void* workspace, size_t workspace_bytes, void* stream) {
  return backward(q, k, v, omega, out, dout, S_state, z_state, S_state_lo, z_state_lo, nullptr,
                  nullptr, B, H, L, d, M, C, dtype, feature, dq, dk, dv, domega, nullptr,
                  nullptr, workspace, workspace_bytes, static_cast<cudaStream_t>(stream));
}

slim_status slim_bwd_from(const void* q, const void* k, const void* v, const float* omega,
                          const void* out, const void* dout, const float* S_state,
                          const float* z_state, const float* S_state_lo,
                          const float* z_state_lo, const float* G_S_in, const float* g_z_in,
                          int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                          slim_feature feature, void* dq, void* dk, void* dv, float* domega,
                          float* G_S_out, float* g_z_out, void* workspace,
                          size_t workspace_bytes, void* stream) {
  return backward(q, k, v, omega, out, dout, S_state, z_state, S_state_lo, z_state_lo, G_S_in,
                  g_z_in, B, H, L, d, M, C, dtype, feature, dq, dk, dv, domega, G_S_out, g_z_out,
                  workspace, workspace_bytes, static_cast<cudaStream_t>(stream));
}

slim_status slim_bidir_workspace_size(int B, int H, int L, int d, int M, int C,
                                      slim_dtype dtype, slim_feature feature, int backward,
                                      size_t* bytes) {
  if (!bytes) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  *bytes = slim::simt::workspace_bytes(p, backward != 0);
  return SLIM_OK;
}

slim_status slim_fwd_bidir(const void* q, const void* k, const void* v, const float* omega,
                           int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                           slim_feature feature, void* out, float* S_state, float* z_state,
                           void* workspace, size_t workspace_bytes, void* stream) {
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  const void* seq[] = {q, k, v, out};
  const void* fixed[] = {S_state, z_state};
  const void* opt[] = {omega};
  if (!pointers_ok(seq, 4, L == 0) || !pointers_ok(fixed, 2, false) || !pointers_ok(opt, 1, true))
    return SLIM_ERR_INVALID_ARG;
  if (omega == nullptr && feature != SLIM_FEAT_SQUARE) return SLIM_ERR_INVALID_ARG;
  const size_t need = slim::simt::workspace_bytes(p, false);
  if (workspace == nullptr || workspace_bytes < need) return SLIM_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SLIM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (L == 0) {
    const size_t n = (size_t)p.chains() * M;
    if (cudaMemsetAsync(S_state, 0, n * d * sizeof(float), s) != cudaSuccess ||
        cudaMemsetAsync(z_state, 0, n * sizeof(float), s) != cudaSuccess)
      return SLIM_ERR_CUDA;
    return SLIM_OK;
  }
  return slim::simt::fwd_bidir(p, q, k, v, omega, out, slim::StateOut{S_state, z_state, nullptr,
                                                                       nullptr},
                               workspace, s);
}

slim_status slim_bwd_bidir(const void* q, const void* k, const void* v, const float* omega,
                           const void* out, const void* dout, const float* S_state,
                           const float* z_state, int B, int H, int L, int d, int M, int C,
                           slim_dtype dtype, slim_feature feature, void* dq, void* dk, void* dv,
                           float* domega, void* workspace, size_t workspace_bytes,
                           void* stream) {
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  const void* seq[] = {q, k, v, out, dout, dq, dk, dv};
  const void* fixed[] = {S_state, z_state};
  const void* opt[] = {omega, domega};
  if (!pointers_ok(seq, 8, L == 0) || !pointers_ok(fixed, 2, false) || !pointers_ok(opt, 2, true))
    return SLIM_ERR_INVALID_ARG;
  if ((omega == nullptr || domega == nullptr) && feature != SLIM_FEAT_SQUARE)
    return SLIM_ERR_INVALID_ARG;
  const size_t need = slim::simt::workspace_bytes(p, true);
  if (workspace == nullptr || workspace_bytes < need) return SLIM_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SLIM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (L == 0) {
    if (domega && cudaMemsetAsync(domega, 0, (size_t)M * d * sizeof(float), s) != cudaSuccess)
      return SLIM_ERR_CUDA;
    return SLIM_OK;
  }
  return slim::simt::bwd_bidir(p, q, k, v, omega, out, dout,
                               slim::StateIn{S_state, z_state, nullptr, nullptr}, dq, dk, dv,
                               domega, workspace, s);
}

slim_status slim_stack_workspace_size(int B, int H, int L, int d, int M, int C, int layers,
                                      slim_dtype dtype, slim_feature feature, int backward,
                                      size_t* bytes) {
  if (!bytes || layers < 1 || layers > 64) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  *bytes = L == 0 ? 0 : slim::stack::workspace_bytes(p, layers, backward != 0);
  return SLIM_OK;
}

slim_status slim_stack_fwd(const void* x, const float* omegas, int B, int H, int L, int d,
                           int M, int C, int layers, slim_dtype dtype, slim_feature feature,
                           void* y, float* S_state, float* z_state, float* S_state_lo,
                           float* z_state_lo, void* workspace, size_t workspace_bytes,
                           void* stream) {
  if (layers < 1 || layers > 64) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  const void* seq[] = {x, y};
  const void* fixed[] = {S_state, z_state};
  const void* opt[] = {S_state_lo, z_state_lo, omegas};
  if (!pointers_ok(seq, 2, L == 0) || !pointers_ok(fixed, 2, false) || !pointers_ok(opt, 3, true))
    return SLIM_ERR_INVALID_ARG;
  if (omegas == nullptr && feature != SLIM_FEAT_SQUARE) return SLIM_ERR_INVALID_ARG;
  if (!pair_ok(S_state_lo, z_state_lo)) return SLIM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t n = (size_t)layers * p.chains() * M;
  if (L == 0) {
    if (cudaMemsetAsync(S_state, 0, n * d * 4, s) != cudaSuccess ||
        cudaMemsetAsync(z_state, 0, n * 4, s) != cudaSuccess ||
        (S_state_lo && cudaMemsetAsync(S_state_lo, 0, n * d * 4, s) != cudaSuccess) ||
        (z_state_lo && cudaMemsetAsync(z_state_lo, 0, n * 4, s) != cudaSuccess))
      return SLIM_ERR_CUDA;
    return SLIM_OK;
  }
  const size_t need = slim::stack::workspace_bytes(p, layers, false);
  if (workspace == nullptr || workspace_bytes < need) return SLIM_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SLIM_ERR_INVALID_ARG;
  return slim::stack::fwd(p, layers, x, omegas, y, S_state, z_state, S_state_lo, z_state_lo,
                          workspace, s);
}

slim_status slim_stack_bwd(const void* x, const float* omegas, const void* dy,
                           const float* S_state, const float* z_state, const float* S_state_lo,
                           const float* z_state_lo, int B, int H, int L, int d, int M, int C,
                           int layers, slim_dtype dtype, slim_feature feature, void* dx,
                           float* domegas, void* workspace, size_t workspace_bytes,
                           void* stream) {
  if (layers < 1 || layers > 64) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  const void* seq[] = {x, dy, dx};
  const void* fixed[] = {S_state, z_state};
  const void* opt[] = {S_state_lo, z_state_lo, omegas, domegas};
  if (!pointers_ok(seq, 3, L == 0) || !pointers_ok(fixed, 2, false) || !pointers_ok(opt, 4, true))
    return SLIM_ERR_INVALID_ARG;
  if ((omegas == nullptr || domegas == nullptr) && feature != SLIM_FEAT_SQUARE)
    return SLIM_ERR_INVALID_ARG;
  if (!pair_ok(S_state_lo, z_state_lo)) return SLIM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (L == 0) {
    if (domegas &&
        cudaMemsetAsync(domegas, 0, (size_t)layers * M * d * 4, s) != cudaSuccess)
      return SLIM_ERR_CUDA;
    return SLIM_OK;
  }
  const size_t need = slim::stack::workspace_bytes(p, layers, true);
  if (workspace == nullptr || workspace_bytes < need) return SLIM_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SLIM_ERR_INVALID_ARG;
  return slim::stack::bwd(p, layers, x, omegas, dy, S_state, z_state, S_state_lo, z_state_lo, dx,
                          domegas, workspace, s);
}

slim_status slim_path_for(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                          slim_feature feature, int* path) {
  if (!path) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  *path = use_tc(p) ? 1 : 0;
  return SLIM_OK;
}

slim_status slim_bwd_schedule(int B, int H, int L, int d, int M, int C, slim_dtype dtype,
                              slim_feature feature, int* items, int cap, int* count,
                              int* ring) {
  if (!count || cap < 0 || (cap > 0 && !items)) return SLIM_ERR_INVALID_ARG;
  Problem p;
  slim_status st = check_problem(B, H, L, d, M, C, dtype, feature, &p);
  if (st != SLIM_OK) return st;
  if (!use_tc(p) || L == 0) return SLIM_ERR_UNSUPPORTED;
  *count = slim::tc::bwd_schedule(p, items, cap, ring);
  return SLIM_OK;
}

slim_status slim_check_device_error(void* workspace, void* stream) {
  if (workspace == nullptr) return SLIM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int word = 0;
  if (cudaMemcpyAsync(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return SLIM_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return SLIM_ERR_CUDA;
  // the stream is drained: every failure counted on this workspace is in the
  // word just read, so the next call need not report it again
  slim::report::mark_seen(workspace);
  if (word != 0) {
    if (cudaMemsetAsync(workspace, 0, sizeof(int), s) != cudaSuccess) return SLIM_ERR_CUDA;
    return SLIM_ERR_TIMEOUT;
  }
  return SLIM_OK;
}

}  // extern "C"
