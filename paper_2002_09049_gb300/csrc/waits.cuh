// Bounded waits of the tensor-core kernels (output error, clipping search, integer inference): the
// clock budget of one wait, the per-device word where a kernel records a wait that gave up, and a
// test hook that makes every wait of the output-error contraction run out.
//
// A kernel whose wait gives up sets its CTA's abort flag, records its MPQ_TIMEOUT_* bit, and
// unwinds: every role stops issuing work, the roles that issued copies or MMAs wait for them to
// finish (drain_wait), tensor memory is released, and the outputs read NaN.  The host reads the
// word with mpq_device_status.
#pragma once

#include <stdint.h>

#include "mpq.h"
#include "sm100.cuh"

namespace mpq {

struct WaitCtl {
    unsigned *status;    // this device's timeout word (MPQ_TIMEOUT_* bits, atomicOr)
    long long budget;    // SM clocks one wait may take before it gives up
    int withhold;        // test hook: the contraction's copy thread issues no copies
};

// Host: the control block for a launch on the current device (the word's address is looked up
// once per device).  MPQ_ERR_CUDA if that lookup fails.
mpq_status wait_ctl(WaitCtl *out);

__device__ __forceinline__ void note_timeout(const WaitCtl &w, unsigned bits)
{
    atomicOr(w.status, bits);
}

// A wait for work this CTA issued itself (its tile copies or its MMAs) to finish before tensor
// memory is released or the CTA exits: it is given 16 budgets, since that work always ends.  A
// drain that still gives up is recorded with MPQ_TIMEOUT_DRAIN.
__device__ __forceinline__ bool drain_wait(uint64_t *bar, uint32_t parity, const WaitCtl &w,
                                           unsigned kernel)
{
    for (int i = 0; i < 16; ++i)
        if (sm100::mbar_wait(bar, parity, w.budget)) return true;
    note_timeout(w, kernel | MPQ_TIMEOUT_DRAIN);
    return false;
}

__device__ __forceinline__ bool drain_wait_cluster(uint64_t *bar, uint32_t parity,
                                                   const WaitCtl &w, unsigned kernel)
{
    for (int i = 0; i < 16; ++i)
        if (sm100::mbar_wait_cluster(bar, parity, w.budget)) return true;
    note_timeout(w, kernel | MPQ_TIMEOUT_DRAIN);
    return false;
}

}  // namespace mpq
