// Tracked bounded waits on mbarriers, for kernels that wait CTA-wide and may have to give
// up (the attention kernels).
#pragma once
#include "ptx.cuh"

// Phase bookkeeping of one mbarrier for CTA-wide bounded waits: `done` counts the phases
// waited for (every thread keeps the same count), `pend` marks a phase armed by the issuing
// thread (a copy's expect_tx or an MMA commit) and not yet waited for.  After a wait gave
// up, the issuing thread drains: it waits (bounded again) for what it armed, so that no
// copy or product is still writing the CTA's shared memory or TMEM when it leaves.
struct BarTrack {
  uint32_t done = 0;
  bool pend = false;
};
FL_DEV bool track_wait_all(uint64_t* bar, BarTrack& t) {
  const bool ok = __syncthreads_and(mbar_wait(bar, t.done & 1));
  if (ok) {
    ++t.done;
    t.pend = false;
  }
  return ok;
}
FL_DEV void track_drain(uint64_t* bar, BarTrack& t) {
  if (t.pend && mbar_wait(bar, t.done & 1)) {
    ++t.done;
    t.pend = false;
  }
}
