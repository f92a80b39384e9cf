// Non-blocking report of bounded device waits that gave up.
//
// A wait that gives up (see give_up in tc_common.cuh) sets word 0 of the
// call's workspace -- which the other CTAs of the call poll, to leave early --
// and increments a counter in host-visible memory whose address the call's
// first kernel stored in bytes 8..15 of the workspace.  The counters live in one page of
// this library's own static storage, pinned and mapped once per process
// (cudaHostRegister), one counter per workspace slot.  At its start every
// call compares its workspace's counter with the count it last reported: a
// plain host read, no event query and no synchronisation.  A difference means
// that a wait of an earlier call on this workspace gave up after the earlier
// report; the call returns SLIM_ERR_TIMEOUT without launching anything.
//
// Slots are assigned to (workspace, device) pairs as they are seen, at most
// kSlots at a time; the least recently used is reassigned.  A call still
// running on a workspace whose slot was reassigned could then count against
// the new owner, which needs more than kSlots workspaces in flight at once.
#include <stdint.h>
#include <string.h>

#include <mutex>

#include "report.h"

namespace slim {
namespace report {
namespace {

constexpr int kSlots = 256;

// counters [0, kSlots), then each slot's counter address as a 64-bit value
struct alignas(4096) Page {
  unsigned counter[kSlots];
  unsigned long long addr[kSlots];
};
static_assert(sizeof(Page) == 4096, "one page");
Page g_page;

std::mutex g_mu;
int g_state = 0;  // 0: not yet registered, 1: registered, -1: registration failed
const void* g_ws[kSlots];
int g_dev[kSlots];
unsigned long long g_used[kSlots];
unsigned g_seen[kSlots];
unsigned long long g_tick = 0;

unsigned load_counter(int slot) {
  return __atomic_load_n(&g_page.counter[slot], __ATOMIC_ACQUIRE);
}

bool ensure_registered() {
  if (g_state == 0) {
    memset(&g_page, 0, sizeof(g_page));
    g_state = -1;
    if (cudaHostRegister(&g_page, sizeof(g_page),
                         cudaHostRegisterMapped | cudaHostRegisterPortable) == cudaSuccess) {
      void* dptr = nullptr;
      if (cudaHostGetDevicePointer(&dptr, &g_page, 0) == cudaSuccess && dptr != nullptr) {
        for (int i = 0; i < kSlots; ++i)
          g_page.addr[i] = reinterpret_cast<unsigned long long>(
              static_cast<char*>(dptr) + (reinterpret_cast<char*>(&g_page.counter[i]) -
                                          reinterpret_cast<char*>(&g_page)));
        g_state = 1;
      } else {
        cudaHostUnregister(&g_page);
      }
    }
    cudaGetLastError();  // a failed registration leaves no sticky error behind
  }
  return g_state == 1;
}

int find_slot(const void* ws, int dev) {
  for (int i = 0; i < kSlots; ++i)
    if (g_ws[i] == ws && g_dev[i] == dev) return i;
  return -1;
}

int take_slot(const void* ws, int dev) {
  int slot = find_slot(ws, dev);
  if (slot < 0) {
    slot = 0;
    for (int i = 0; i < kSlots; ++i) {
      if (g_ws[i] == nullptr) {
        slot = i;
        break;
      }
      if (g_used[i] < g_used[slot]) slot = i;
    }
    g_ws[slot] = ws;
    g_dev[slot] = dev;
    g_seen[slot] = load_counter(slot);  // counts from before belong to others
  }
  g_used[slot] = ++g_tick;
  return slot;
}

}  // namespace

slim_status begin(const void* workspace, bool enabled, unsigned** counter) {
  *counter = nullptr;
  if (!enabled) return SLIM_OK;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return SLIM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!ensure_registered()) return SLIM_OK;
  const int slot = take_slot(workspace, dev);
  const unsigned now = load_counter(slot);
  if (now != g_seen[slot]) {
    g_seen[slot] = now;
    return SLIM_ERR_TIMEOUT;
  }
  *counter = reinterpret_cast<unsigned*>(g_page.addr[slot]);
  return SLIM_OK;
}

void mark_seen(const void* workspace) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_state != 1) return;
  const int slot = find_slot(workspace, dev);
  if (slot >= 0) g_seen[slot] = load_counter(slot);
}

}  // namespace report
}  // namespace slim
