// Launch accounting and CUDA-event timing of every libslim kernel launch.
#pragma once
#include <cuda_runtime.h>

namespace slim {
namespace prof {

// Every kernel of the library, by name.
enum Kid {
  K_GEMM = 0,
  K_PREP,
  K_SCAN,
  K_FINALIZE,
  K_DSTAT,
  K_VJP,
  K_STORE,
  K_REDUCE,
  K_STATE,
  K_TC_FWD,
  K_TC_BWD,
  K_TC_DELTA,
  K_TC_SCAN,
  K_TC_BWD_Q,
  K_TC_BWD_KV,
  K_TC_REDUCE,
  K_TC_SELFTEST,
  K_TC_PREP,
  K_STACK,
  K_COUNT
};

bool enabled();
void count_launch();
void record(Kid k, cudaEvent_t* start, cudaEvent_t* stop, double flops, double bytes);

// Brackets one launch: records a start event in the constructor and a stop
// event in the destructor when profiling is on; always counts the launch.
class Scope {
 public:
  Scope(Kid k, cudaStream_t s, double flops = 0.0, double bytes = 0.0);
  ~Scope();

 private:
  Kid k_;
  cudaStream_t s_;
  double flops_, bytes_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
};

}  // namespace prof
}  // namespace slim
