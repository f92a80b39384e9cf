// Tensor-core (tcgen05) path of libslim; see tc_path.cu.
#pragma once
#include "common.cuh"

namespace slim {
namespace tc {

// bf16, d = 64, M in {128, 256}, the exp or ReLU map, slices of at least 64 rows.
bool supports(const Problem& p);
size_t workspace_bytes(const Problem& p, bool bwd);
// The backward launch's item order: items[3 x] = (role, slice, index) of
// ticket x, for x < min(count, cap), and (if ring is not null) the number of
// hand-off ring slots.  Returns the item count.
int bwd_schedule(const Problem& p, int* items, int cap, int* ring);

// report: the device address of the call's timeout-report counter, or null
// (see report.h); the first kernel of the call stores it in the workspace.
slim_status fwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, void* out, const StateOut& st, const StateInit& init,
                unsigned* report, void* workspace, cudaStream_t s);

slim_status bwd(const Problem& p, const void* q, const void* k, const void* v,
                const float* omega, const void* out, const void* dout, const StateIn& st,
                const GradIO& gio, void* dq, void* dk, void* dv, float* domega,
                unsigned* report, void* workspace, cudaStream_t s);

}  // namespace tc
}  // namespace slim
