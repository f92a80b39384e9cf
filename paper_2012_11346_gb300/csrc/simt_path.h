// fp32-compute path of libslim (fp32 operands, warp-MMA contractions); see simt_path.cu.
#pragma once
#include "common.cuh"

namespace slim {
namespace simt {

size_t workspace_bytes(const Problem& p, bool bwd);

slim_status fwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, void* out, const StateOut& st, const StateInit& init,
                void* workspace, cudaStream_t s);

slim_status bwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, const void* out, const void* dout, const StateIn& st,
                const GradIO& gio, void* dq, void* dk, void* dv, float* domega, void* workspace,
                cudaStream_t s);

// The non-causal form (no mask, one global state; S_state/z_state are that
// state), on the same workspace layout as the causal sweeps.
slim_status fwd_bidir(const Problem& p, const void* q, const void* k, const void* v,
                      const float* omega, void* out, const StateOut& st, void* workspace,
                      cudaStream_t s);
slim_status bwd_bidir(const Problem& p, const void* q, const void* k, const void* v,
                      const float* omega, const void* out, const void* dout, const StateIn& st,
                      void* dq, void* dk, void* dv, float* domega, void* workspace,
                      cudaStream_t s);

}  // namespace simt
}  // namespace slim
