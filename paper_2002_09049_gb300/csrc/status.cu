// Device-side status (include/mpq.h: mpq_device_status, mpq_set_wait_limit,
// mpq_test_withhold_copies, mpq_build_options).  One word per device collects the MPQ_TIMEOUT_*
// bits of kernels whose bounded waits gave up; mpq_device_status takes it (reads and clears it in
// one atomic exchange on the device).  The word's device address is looked up once per device,
// with that device current, and handed to every tensor-core launch.  In the checked build
// (MPQ_CHECK_BOUNDS) every kernel unit also keeps a count of the accesses its bounds checks
// skipped, taken by the same call.
#include <atomic>
#include <mutex>
#include <vector>

#include "checks.cuh"
#include "mpq_internal.cuh"
#include "waits.cuh"

namespace mpq {

static __device__ unsigned g_timeouts;   // MPQ_TIMEOUT_* bits since the last take
static __device__ unsigned g_taken;      // the last take's value, copied to the host

__global__ void take_timeouts_kernel() { g_taken = atomicExch(&g_timeouts, 0u); }

constexpr long long kDefaultWaitBudget = 1LL << 31;   // SM clocks, about 1 s at 2 GHz
static std::atomic<long long> g_budget{kDefaultWaitBudget};
static std::atomic<int> g_withhold{0};
static unsigned *g_word[kMaxDevices];
static std::mutex g_mu;

static mpq_status timeout_word(unsigned **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_status(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) {
        set_error("device %d beyond %d devices", dev, kMaxDevices);
        return MPQ_ERR_UNSUPPORTED;
    }
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_word[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_timeouts);
        if (e != cudaSuccess) return cuda_status(e, "cudaGetSymbolAddress (timeout word)");
        g_word[dev] = static_cast<unsigned *>(p);
    }
    *out = g_word[dev];
    return MPQ_OK;
}

struct BoundsUnit {
    const char *name;
    BoundsTake take;
};

static std::vector<BoundsUnit> &bounds_units()
{
    static std::vector<BoundsUnit> units;   // filled while the library loads, read-only after
    return units;
}

void register_bounds_unit(const char *name, BoundsTake take)
{
    bounds_units().push_back({name, take});
}

mpq_status wait_ctl(WaitCtl *out)
{
    const mpq_status st = timeout_word(&out->status);
    if (st != MPQ_OK) return st;
    out->budget = g_budget.load(std::memory_order_relaxed);
    out->withhold = g_withhold.load(std::memory_order_relaxed);
    return MPQ_OK;
}

}  // namespace mpq

using namespace mpq;

extern "C" mpq_status mpq_device_status(void *stream, unsigned *flags)
{
    if (flags) *flags = 0;
    unsigned *word = nullptr;
    mpq_status st = timeout_word(&word);   // also loads the module on this device
    if (st != MPQ_OK) return st;
    const cudaStream_t s = (cudaStream_t)stream;
    take_timeouts_kernel<<<1, 1, 0, s>>>();
    cudaError_t e = cudaGetLastError();
    unsigned h = 0;
    if (e == cudaSuccess)
        e = cudaMemcpyFromSymbolAsync(&h, g_taken, sizeof(h), 0, cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    st = cuda_status(e, "reading the timeout word");
    if (st != MPQ_OK) return st;
    // the checked build's bounds counts, unit by unit (none are registered in the normal build)
    unsigned skipped = 0, first_line = 0;
    const char *first_unit = nullptr;
    for (const BoundsUnit &u : bounds_units()) {
        unsigned c = 0, line = 0;
        st = cuda_status(u.take(s, &c, &line), "reading the bounds-check words");
        if (st != MPQ_OK) return st;
        if (c != 0 && !first_unit) {
            first_unit = u.name;
            first_line = line;
        }
        skipped += c;
    }
    if (skipped != 0) h |= MPQ_FAULT_BOUNDS;
    if (flags) *flags = h;
    if (h & ~MPQ_FAULT_BOUNDS) {
        set_error("a bounded device-side wait gave up (MPQ_TIMEOUT bits 0x%x)",
                  h & ~MPQ_FAULT_BOUNDS);
        return MPQ_ERR_TIMEOUT;
    }
    if (skipped != 0) {
        set_error("bounds checks skipped %u accesses (the first at %s:%u)", skipped, first_unit,
                  first_line);
        return MPQ_ERR_BOUNDS;
    }
    return MPQ_OK;
}

extern "C" unsigned mpq_build_options(void)
{
#ifdef MPQ_CHECK_BOUNDS
    return MPQ_BUILD_CHECK_BOUNDS;
#else
    return 0u;
#endif
}

extern "C" mpq_status mpq_set_wait_limit(long long clocks)
{
    g_budget.store(clocks > 0 ? clocks : kDefaultWaitBudget, std::memory_order_relaxed);
    return MPQ_OK;
}

extern "C" mpq_status mpq_test_withhold_copies(int on)
{
    g_withhold.store(on ? 1 : 0, std::memory_order_relaxed);
    return MPQ_OK;
}
