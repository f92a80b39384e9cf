// Diagnostic: one CTA computes D[128 x N] = A[128 x K] B[K x N] with tcgen05
// from swizzled shared-memory tiles in the requested operand layouts, so the
// descriptor conventions of tc_common.cuh can be checked against a reference.
#include "../../include/slim.h"
#include "common.cuh"
#include "profiler.h"
#include "report.h"
#include "tc_common.cuh"

namespace slim {
namespace tc {

__global__ void __launch_bounds__(128) k_tc_selftest(const __nv_bfloat16* A, const __nv_bfloat16* Bm,
                                                     float* D, int K, int N, int a_mn, int b_mn,
                                                     int* err) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = base;                  // 128 x K
  uint8_t* sB = base + 128 * K * 2;    // K x N
  __shared__ __align__(8) uint64_t mbar;
  __shared__ uint32_t tmem_base;
  const int tid = threadIdx.x, warp = tid / 32;

  for (int e = tid; e < 128 * K; e += 128) {
    const int m = e / K, k = e % K;
    const uint32_t off = a_mn ? tile_off(K, k, m) : tile_off(128, m, k);
    *reinterpret_cast<__nv_bfloat16*>(sA + off) = A[e];
  }
  for (int e = tid; e < K * N; e += 128) {
    const int k = e / N, n = e % N;
    const uint32_t off = b_mn ? tile_off(K, k, n) : tile_off(N, n, k);
    *reinterpret_cast<__nv_bfloat16*>(sB + off) = Bm[e];
  }
  if (tid == 0) {
    mbar_init(smem_u32(&mbar), 1);
    mbar_fence_init();
  }
  if (warp == 0) tmem_alloc(smem_u32(&tmem_base), 256);
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  if (tid == 0) {
    const uint32_t a0 = smem_u32(sA), b0 = smem_u32(sB);
    const uint32_t id = idesc_bf16(128, N, a_mn, b_mn);
    for (int k0 = 0; k0 < K; k0 += 16) {
      const uint64_t ad = a_mn ? mnmaj(a0, k0, (uint32_t)K * 128) : kmaj(a0, 128, k0);
      const uint64_t bd = b_mn ? mnmaj(b0, k0, (uint32_t)K * 128) : kmaj(b0, N, k0);
      mma(tmem, ad, bd, id, k0 > 0);
    }
    mma_commit(smem_u32(&mbar));
  }
  const bool ok = mbar_wait(smem_u32(&mbar), 0, err, false);  // err: a plain int
  tc_fence_after();
  if (ok) {
    const int row = tid;
    for (int c0 = 0; c0 < N; c0 += 32) {
      float v[32];
      tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + c0, v);
      for (int i = 0; i < 32; ++i) D[(size_t)row * N + c0 + i] = v[i];
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

// A bounded wait on an mbarrier that nothing arrives at: it gives up after
// its iteration limit, records the failure in the error word and returns --
// the same path every kernel takes when a wait gives up.
__global__ void k_wait_timeout(int* err, unsigned* rep) {
  __shared__ __align__(8) uint64_t mbar;
  if (threadIdx.x == 0) {
    *err = 0;
    set_report(err, rep);
    mbar_init(smem_u32(&mbar), 1);
    mbar_fence_init();
  }
  __syncthreads();
  mbar_wait(smem_u32(&mbar), 0, err);
}

}  // namespace tc
}  // namespace slim

extern "C" slim_status slim_diag_wait_timeout(void* workspace, void* stream) {
  if (!workspace) return SLIM_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the same error word and report counter as the tensor-core calls
  unsigned* counter = nullptr;
  const slim_status st = slim::report::begin(workspace, true, &counter);
  if (st != SLIM_OK) return st;
  slim::prof::Scope ps(slim::prof::K_TC_SELFTEST, s);
  slim::tc::k_wait_timeout<<<1, 32, 0, s>>>(static_cast<int*>(workspace), counter);
  return cudaGetLastError() == cudaSuccess ? SLIM_OK : SLIM_ERR_CUDA;
}

extern "C" slim_status slim_tc_selftest(int a_mn, int b_mn, int K, int N, const void* A,
                                        const void* B, float* D, int* err, void* stream) {
  if (!(K == 64 || K == 128 || K == 256) || !(N == 64 || N == 128 || N == 256))
    return SLIM_ERR_INVALID_ARG;
  if (!A || !B || !D || !err || (a_mn & ~1) || (b_mn & ~1)) return SLIM_ERR_INVALID_ARG;
  const size_t smem = 1024 + (size_t)128 * K * 2 + (size_t)K * N * 2;
  if (cudaFuncSetAttribute(slim::tc::k_tc_selftest, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return SLIM_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  slim::prof::Scope ps(slim::prof::K_TC_SELFTEST, s);
  slim::tc::k_tc_selftest<<<1, 128, smem, s>>>(static_cast<const __nv_bfloat16*>(A),
                                               static_cast<const __nv_bfloat16*>(B), D, K, N,
                                               a_mn, b_mn, err);
  return cudaGetLastError() == cudaSuccess ? SLIM_OK : SLIM_ERR_CUDA;
}
