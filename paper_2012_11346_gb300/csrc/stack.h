// A stack of residual layers by Algorithm 1 (slices outer, layers inner); see stack.cu.
#pragma once
#include "common.cuh"

namespace slim {
namespace stack {

size_t workspace_bytes(const Problem& p, int layers, bool bwd);

slim_status fwd(const Problem& p, int layers, const void* x, const float* omegas, void* y,
                float* S_state, float* z_state, float* S_lo, float* z_lo, void* workspace,
                cudaStream_t s);

slim_status bwd(const Problem& p, int layers, const void* x, const float* omegas, const void* dy,
                const float* S_state, const float* z_state, const float* S_lo,
                const float* z_lo, void* dx, float* domegas, void* workspace, cudaStream_t s);

}  // namespace stack
}  // namespace slim
