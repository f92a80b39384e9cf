// Launch accounting and CUDA-event timing; see profiler.h and include/slim.h.
#include <string.h>

#include <atomic>
#include <vector>

#include "../../include/slim.h"
#include "profiler.h"

namespace slim {
namespace prof {
namespace {

const char* kNames[K_COUNT] = {
    "mma_gemm",    "simt_prep",     "simt_scan",      "simt_finalize", "simt_dstat",
    "simt_vjp",    "simt_store",    "simt_reduce",    "simt_state",    "tc_fwd",
    "tc_bwd",      "tc_delta",      "tc_scan",        "tc_bwd_q",      "tc_bwd_kv",
    "tc_reduce",   "tc_selftest",   "tc_prep",        "stack_rows"};

struct Rec {
  Kid k;
  cudaEvent_t a, b;
  double flops, bytes;
};

struct Totals {
  unsigned long long launches = 0;
  double ms = 0, flops = 0, bytes = 0;
};

std::atomic<unsigned long long> g_launches{0};
bool g_on = false;
std::vector<Rec> g_recs;
std::vector<cudaEvent_t> g_free;
Totals g_tot[K_COUNT];

cudaEvent_t get_event() {
  if (!g_free.empty()) {
    cudaEvent_t e = g_free.back();
    g_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

}  // namespace

bool enabled() { return g_on; }
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

Scope::Scope(Kid k, cudaStream_t s, double flops, double bytes)
    : k_(k), s_(s), flops_(flops), bytes_(bytes) {
  count_launch();
  if (g_on) {
    a_ = get_event();
    b_ = get_event();
    if (a_ && b_) cudaEventRecord(a_, s_);
  }
}

Scope::~Scope() {
  if (a_ && b_) {
    cudaEventRecord(b_, s_);
    g_recs.push_back(Rec{k_, a_, b_, flops_, bytes_});
  }
}

}  // namespace prof
}  // namespace slim

using namespace slim::prof;

extern "C" {

unsigned long long slim_launch_count(void) { return g_launches.load(); }

void slim_profiler_enable(int on) { g_on = on != 0; }

void slim_profiler_reset(void) {
  for (auto& r : g_recs) {
    cudaEventSynchronize(r.b);
    g_free.push_back(r.a);
    g_free.push_back(r.b);
  }
  g_recs.clear();
  for (auto& t : g_tot) t = Totals{};
}

int slim_profiler_read(slim_kernel_stats* stats, int cap) {
  for (auto& r : g_recs) {
    if (cudaEventSynchronize(r.b) != cudaSuccess) return -1;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) return -1;
    Totals& t = g_tot[r.k];
    t.launches += 1;
    t.ms += ms;
    t.flops += r.flops;
    t.bytes += r.bytes;
    g_free.push_back(r.a);
    g_free.push_back(r.b);
  }
  g_recs.clear();
  int n = 0;
  for (int k = 0; k < K_COUNT; ++k) {
    if (g_tot[k].launches == 0) continue;
    if (stats && n < cap) {
      slim_kernel_stats& s = stats[n];
      memset(s.name, 0, sizeof(s.name));
      strncpy(s.name, kNames[k], sizeof(s.name) - 1);
      s.launches = g_tot[k].launches;
      s.total_ms = g_tot[k].ms;
      s.flops = g_tot[k].flops;
      s.bytes = g_tot[k].bytes;
    }
    ++n;
  }
  return n;
}

}  // extern "C"
