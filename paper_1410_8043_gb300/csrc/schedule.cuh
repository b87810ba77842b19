// The read-version rule v_p(c) of one worker (Sec. 2.2 SSP condition and
// ESSP; Sec. 3 formal SSP bound; Sec. 4 READ guarantee and server push; the
// Sec. 2.1 VAP value bound).  SSP and ESSP are integer-only, so they are
// bit-exact against any other implementation of the same rule; VAP compares
// fp32 max-norms of the table against its bound.
#pragma once

#include "internal.h"
#include "ptx.cuh"

namespace esspt {

__device__ __forceinline__ void schedule_worker(const ScheduleArgs& a, int32_t p) {
  const int32_t lo = max(0, a.c - 1 - a.s);
  int32_t v = a.v[p];
  if (a.model == ESSPT_SSP_LAZY) {
    // Lazy pull: refresh only when the cached version would fall out of the
    // bound, so the staleness (c-1) - v cycles through 0..s.
    uint32_t phi = 0;
    if (a.phased) {
      const uint64_t h = ctr_u64(a.seed, kStreamPhase, (uint64_t)p);
      phi = (uint32_t)(((h >> 32) * (uint64_t)(a.s + 1)) >> 32);
    }
    v = (a.c - 1) - (int32_t)(((uint32_t)(a.c - 1) + phi) % (uint32_t)(a.s + 1));
    v = max(v, 0);
  } else if (a.model == ESSPT_ESSP_EAGER) {
    // Eager push of version c-1, arriving after d ~ Geometric clock(s):
    // d >= k iff u < thr[k] (thresholds decrease with k).
    const uint32_t u = (uint32_t)(ctr_u64(a.seed, kStreamDelay, ((uint64_t)(uint32_t)a.c << 32) | (uint32_t)p) >> 32);
    int32_t d = 0;
    for (int32_t k = 1; k <= a.dmax; ++k) d += (u < a.thr[k]) ? 1 : 0;
    v = max(max(v, a.c - 1 - d), 0);
  } else if (a.model == ESSPT_SSP_ROW) {
    // Reads are per row (the row refresh); the worker's nominal version is
    // the newest one it may read.
    v = a.c - 1;
  } else if (a.model == ESSPT_VAP) {
    // Stalest version in the window whose in-transit max-norm is in bound.
    v = a.c - 1;
    for (int32_t k = min(a.s, a.c - 1); k >= 1; --k) {
      if ((double)__uint_as_float(a.vap_norm[k]) <= a.vap_bound) {
        v = a.c - 1 - k;
        break;
      }
    }
  }
  // ESSPT_EXTERNAL: v was written by the host; only the check below runs.
  if (v < lo || v > a.c - 1) atomicOr(a.status, kErrStale);
  a.v[p] = v;
}

}  // namespace esspt
