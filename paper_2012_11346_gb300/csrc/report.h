// Reporting of device waits that gave up to the next call on the same
// workspace, without synchronising the device; see report.cu.
#pragma once
#include "common.cuh"

namespace slim {
namespace report {

// Called by an entry point after its arguments are validated and before it
// enqueues anything; host-only (it enqueues nothing).  With enabled = true:
// returns SLIM_ERR_TIMEOUT if a bounded wait of an earlier call on this
// workspace has given up since that was last reported; otherwise returns
// SLIM_OK and sets *counter to the device address of the workspace's report
// counter, which the call's first kernel stores in bytes 8..15 of the
// workspace (see give_up in tc_common.cuh).  With enabled = false (the
// allocation-free entry point), or when the counters could not be set up,
// *counter is null: a wait that gives up is then counted nowhere.
slim_status begin(const void* workspace, bool enabled, unsigned** counter);

// After a blocking read of a workspace's error word: every failure counted on
// that workspace so far has been seen, so the next call does not report it
// again.
void mark_seen(const void* workspace);

}  // namespace report
}  // namespace slim
