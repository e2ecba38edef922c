// Bounds checks of the checked build (compiled with -DMPQ_CHECK_BOUNDS; include/mpq.h:
// mpq_build_options, MPQ_FAULT_BOUNDS).
//
// MPQ_CHECK(cond) guards one access whose index the kernel computed: in the checked build a false
// condition counts a violation, records the source line of the first one, and evaluates to false
// so that the caller skips the access -- nothing traps, and the launch runs to its end.  In the
// normal build it is the constant true and the condition is not evaluated (so it must have no side
// effects).  Every translation unit is its own device module, so each keeps its own two words;
// MPQ_CHECKED_UNIT(name) registers the unit with the host, and mpq_device_status takes every
// registered unit's words (reads and clears them on the device) and reports MPQ_FAULT_BOUNDS.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "mpq.h"

namespace mpq {

// Host: the units of the checked build, filled at load time (status.cu).
using BoundsTake = cudaError_t (*)(cudaStream_t s, unsigned *count, unsigned *line);
void register_bounds_unit(const char *name, BoundsTake take);

}  // namespace mpq

#ifdef MPQ_CHECK_BOUNDS

namespace mpq {
namespace {   // one copy per translation unit

__device__ unsigned bnd_count;     // violations since the last take
__device__ unsigned bnd_line;      // the source line of the first one (0: none)
__device__ unsigned bnd_taken[2];  // the last take's count and line, copied to the host

__global__ void bnd_take_kernel()
{
    bnd_taken[0] = atomicExch(&bnd_count, 0u);
    bnd_taken[1] = atomicExch(&bnd_line, 0u);
}

__device__ __noinline__ bool bnd_fail(unsigned line)
{
    atomicAdd(&bnd_count, 1u);
    atomicCAS(&bnd_line, 0u, line);
    return false;
}

// The dynamic shared memory this launch was given (bytes).
__device__ __forceinline__ unsigned bnd_dynamic_smem()
{
    unsigned r;
    asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(r));
    return r;
}

cudaError_t bnd_take(cudaStream_t s, unsigned *count, unsigned *line)
{
    bnd_take_kernel<<<1, 1, 0, s>>>();
    cudaError_t e = cudaGetLastError();
    unsigned h[2] = {0u, 0u};
    if (e == cudaSuccess)
        e = cudaMemcpyFromSymbolAsync(h, bnd_taken, sizeof(h), 0, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    *count = h[0];
    *line = h[1];
    return e;
}

struct BoundsRegistrar {
    explicit BoundsRegistrar(const char *name) { register_bounds_unit(name, &bnd_take); }
};

}  // namespace
}  // namespace mpq

#define MPQ_CHECK(cond) ((cond) ? true : ::mpq::bnd_fail(__LINE__))
// end (a byte address relative to the start of dynamic shared memory) within the launch's share
#define MPQ_CHECK_SMEM_END(end) MPQ_CHECK((size_t)(end) <= (size_t)::mpq::bnd_dynamic_smem())
#define MPQ_CHECKED_UNIT(name) static ::mpq::BoundsRegistrar mpq_bounds_unit_(name)

#else

// the condition is an unevaluated operand: named (so no variable it alone uses goes unreferenced)
// but neither evaluated nor compiled into code
#define MPQ_CHECK(cond) (sizeof((cond) ? 1 : 0) != 0)
#define MPQ_CHECK_SMEM_END(end) (sizeof(end) != 0)
#define MPQ_CHECKED_UNIT(name) static_assert(true, "")

#endif

// index i of an array of n elements
#define MPQ_IN(i, n) MPQ_CHECK((size_t)(i) < (size_t)(n))
