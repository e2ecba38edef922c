// Per-channel point counts from the output-error table (Sec. 3.3, Algorithm 2).
//
// Budget mode.  The sequential rule -- hand each extra point to the channel whose next point has
// the largest gain e_k(n_k) - e_k(n_k+1), lowest k on ties, stop when no gain is positive -- is
// computed as one selection.  For channel k and n = 2..k_max let
//   gain_k(n) = e_k(n-1) - e_k(n)      (fp32 subtraction; NaN reads as -inf)
//   p_k(n)    = min_{2<=m<=n} gain_k(m) (prefix minimum)
// and order the pairs (k, n) by (p desc, k asc, n asc).  The sequential loop takes exactly the
// first `extra` pairs of this order that have p > 0: a channel's (n+1)-th gain becomes its head
// only after the n-th was taken, its priority never exceeds the priorities before it, and a head
// at or above every other head is taken next -- so both rules visit the pairs in the same order.
// Each pair becomes one unique 64-bit key (~bits(p) in the high word, k*(k_max-1)+(n-2) in the
// low word); an MSB-first radix select finds the extra-th smallest key T, and
// n_k = 1 + #{n : key(k, n) <= T}.  The keys live in shared memory when they fit (they are
// recomputed from the error table on every pass otherwise); no global scratch is used.
#include <math.h>

#include "mpq_internal.cuh"

MPQ_CHECKED_UNIT("allocate.cu");

namespace mpq {
namespace {

constexpr int AB_THREADS = 1024;
constexpr unsigned long long NO_KEY = ~0ULL;

// The keys of channel k for n = 2..k_max, in n order, via callback.
template <typename F>
__device__ __forceinline__ void channel_keys(const float *__restrict__ err, int k, int k_max, F f)
{
    const float *e = err + (size_t)k * (k_max + 1);
    float p = INFINITY;
    float prev = e[1];
    for (int n = 2; n <= k_max; ++n) {
        const float cur = e[n];
        float g = __fsub_rn(prev, cur);
        if (isnan(g)) g = -INFINITY;
        p = fminf(p, g);
        prev = cur;
        unsigned long long key = NO_KEY;
        if (p > 0.0f) {
            const unsigned hi = ~__float_as_uint(p);
            const unsigned lo = (unsigned)((unsigned long long)k * (k_max - 1) + (n - 2));
            key = ((unsigned long long)hi << 32) | lo;
        }
        f(n, key);
    }
}

constexpr int KEY_CACHE = 12288;   // keys held in shared memory (96 KB) when they fit

// Radix select of the rank-th smallest selectable key, MSB first, 8 bits per pass.  A pass whose
// target bucket holds one key ends the search with that key (recorded as the bucket's witness).
// One CTA of AB_THREADS threads allocates one layer; skeys: dynamic shared memory for its keys.
__device__ __forceinline__ void allocate_budget_cta(const float *__restrict__ err, int C, int k_max,
                                                    long long extra, int *__restrict__ npoints,
                                                    int *__restrict__ points_used, bool cached,
                                                    unsigned long long *skeys)
{
    __shared__ unsigned int hist[256];
    __shared__ unsigned long long witness[256];
    __shared__ unsigned long long s_prefix, s_T, s_total;
    __shared__ long long s_rem;
    __shared__ int s_done, s_used;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int KM1 = k_max - 1;
    // the cached keys within the launch's shared memory, else read again from err
    if (cached && !MPQ_CHECK_SMEM_END(8 * (size_t)C * KM1)) cached = false;

    if (tid == 0) {
        s_total = 0;
        s_used = 0;
        s_done = 0;
        s_prefix = 0;
    }
    __syncthreads();
    unsigned long long mine = 0;
    for (int k = tid; k < C; k += AB_THREADS)
        channel_keys(err, k, k_max, [&](int n, unsigned long long key) {
            if (cached) skeys[(size_t)k * KM1 + (n - 2)] = key;
            mine += key != NO_KEY;
        });
    atomicAdd(&s_total, mine);
    __syncthreads();
    const long long total = (long long)s_total;
    const long long take = extra < total ? extra : total;

    // visit every selectable key
    auto for_keys = [&](auto f) {
        if (cached) {
            const long long nk = (long long)C * KM1;
            for (long long i = tid; i < nk; i += AB_THREADS) {
                const unsigned long long key = skeys[i];
                if (key != NO_KEY) f(key);
            }
        } else {
            for (int k = tid; k < C; k += AB_THREADS)
                channel_keys(err, k, k_max, [&](int, unsigned long long key) {
                    if (key != NO_KEY) f(key);
                });
        }
    };

    unsigned long long T = 0;   // selected = keys <= T (when take > 0)
    if (take > 0 && take == total) {
        T = NO_KEY - 1;
    } else if (take > 0) {
        if (tid == 0) s_rem = take;   // 1-based rank of the key we look for
        for (int shift = 56; shift >= 0; shift -= 8) {
            for (int b = tid; b < 256; b += AB_THREADS) hist[b] = 0;
            __syncthreads();
            const unsigned long long prefix = s_prefix;
            const int hs = shift + 8;
            for_keys([&](unsigned long long key) {
                if (hs < 64 && ((key ^ prefix) >> hs) != 0) return;
                const unsigned b = (unsigned)(key >> shift) & 255u;
                atomicAdd(&hist[b], 1u);
                witness[b] = key;   // meaningful only when the bucket ends with one key
            });
            __syncthreads();
            if (warp == 0) {
                // warp-parallel search for the bucket that holds the rem-th key
                const long long rem = s_rem;
                unsigned int loc = 0;
#pragma unroll
                for (int i = 0; i < 8; ++i) loc += hist[lane * 8 + i];
                unsigned long long incl = loc;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const unsigned long long excl = incl - loc;
                const unsigned hit = __ballot_sync(0xffffffffu,
                                                   (long long)excl < rem && rem <= (long long)incl);
                const int src = __ffs(hit) - 1;
                if (lane == src) {
                    long long cum = (long long)excl;
                    int b = lane * 8;
                    for (; b < lane * 8 + 7; ++b) {
                        if (cum + (long long)hist[b] >= rem) break;
                        cum += hist[b];
                    }
                    s_rem = rem - cum;
                    s_prefix = prefix | ((unsigned long long)b << shift);
                    if (hist[b] == 1) {
                        s_T = witness[b];
                        s_done = 1;
                    }
                }
            }
            __syncthreads();
            if (s_done) break;
        }
        T = s_done ? s_T : s_prefix;
    }

    // n_k = 1 + number of selected keys of channel k (a prefix n = 2..n_k, since p is monotone)
    int used = 0;
    for (int k = tid; k < C; k += AB_THREADS) {
        int n_k = 1;
        if (take > 0) {
            if (cached) {
                for (int n = 0; n < KM1; ++n) {
                    const unsigned long long key = skeys[(size_t)k * KM1 + n];
                    if (key != NO_KEY && key <= T) ++n_k;
                }
            } else {
                channel_keys(err, k, k_max, [&](int, unsigned long long key) {
                    if (key != NO_KEY && key <= T) ++n_k;
                });
            }
        }
        npoints[k] = n_k;
        used += n_k;
    }
    if (points_used) {
        for (int o = 16; o > 0; o >>= 1) used += __shfl_xor_sync(0xffffffffu, used, o);
        if (lane == 0) atomicAdd(&s_used, used);   // integer sum: order-free
        __syncthreads();
        if (tid == 0) *points_used = s_used;
    }
}

__global__ void __launch_bounds__(AB_THREADS)
allocate_budget_kernel(const float *__restrict__ err, int C, int k_max, long long extra,
                       int *__restrict__ npoints, int *__restrict__ points_used, bool cached)
{
    extern __shared__ unsigned long long skeys[];   // [C * (k_max - 1)] when cached
    allocate_budget_cta(err, C, k_max, extra, npoints, points_used, cached, skeys);
}

// Threshold mode (Algorithm 2 as printed) for one layer by one CTA, the total by a block sum.
__device__ __forceinline__ void allocate_threshold_cta(const float *__restrict__ err, int C,
                                                       int k_max, double eps,
                                                       int *__restrict__ npoints,
                                                       int *__restrict__ points_used)
{
    __shared__ int s_used;
    if (threadIdx.x == 0) s_used = 0;
    __syncthreads();
    int used = 0;
    for (int k = threadIdx.x; k < C; k += blockDim.x) {
        const float *e = err + (size_t)k * (k_max + 1);
        int n = k_max;
        for (int m = 1; m <= k_max; ++m) {
            if ((double)e[m] < eps) {
                n = m;
                break;
            }
        }
        npoints[k] = n;
        used += n;
    }
    if (points_used) {
        for (int o = 16; o > 0; o >>= 1) used += __shfl_xor_sync(0xffffffffu, used, o);
        if ((threadIdx.x & 31) == 0) atomicAdd(&s_used, used);   // integer sum: order-free
        __syncthreads();
        if (threadIdx.x == 0) *points_used = s_used;
    }
}

// Several layers in one launch: CTA b allocates layer order[b] (largest first, so the longest
// CTAs start first).
struct AllocBatch {
    const float *err[MPQ_MAX_BATCH];
    int *npoints[MPQ_MAX_BATCH];
    int *points_used[MPQ_MAX_BATCH];
    double param[MPQ_MAX_BATCH];     // threshold mode: eps
    long long extra[MPQ_MAX_BATCH];  // budget mode
    int C[MPQ_MAX_BATCH];
    unsigned char cached[MPQ_MAX_BATCH];
    unsigned char order[MPQ_MAX_BATCH];
};

__global__ void __launch_bounds__(AB_THREADS)
allocate_batch_kernel(const __grid_constant__ AllocBatch b, int k_max, int mode)
{
    extern __shared__ unsigned long long skeys[];
    if (!MPQ_IN(blockIdx.x, MPQ_MAX_BATCH) || !MPQ_IN(b.order[blockIdx.x], MPQ_MAX_BATCH)) return;
    const int l = b.order[blockIdx.x];
    if (mode == MPQ_ALLOC_BUDGET)
        allocate_budget_cta(b.err[l], b.C[l], k_max, b.extra[l], b.npoints[l], b.points_used[l],
                            b.cached[l] != 0, skeys);
    else
        allocate_threshold_cta(b.err[l], b.C[l], k_max, b.param[l], b.npoints[l],
                               b.points_used[l]);
}

constexpr int AT_THREADS = 256;

__global__ void __launch_bounds__(AT_THREADS)
allocate_threshold_kernel(const float *__restrict__ err, int C, int k_max, double eps,
                          int *__restrict__ npoints, int *__restrict__ points_used)
{
    int used = 0;
    for (int k = blockIdx.x * AT_THREADS + threadIdx.x; k < C; k += gridDim.x * AT_THREADS) {
        const float *e = err + (size_t)k * (k_max + 1);
        int n = k_max;
        for (int m = 1; m <= k_max; ++m) {
            if ((double)e[m] < eps) {
                n = m;
                break;
            }
        }
        npoints[k] = n;
        used += n;
    }
    if (points_used) {
        for (int o = 16; o > 0; o >>= 1) used += __shfl_xor_sync(0xffffffffu, used, o);
        if ((threadIdx.x & 31) == 0) atomicAdd(points_used, used);  // integer sum: order-free
    }
}

}  // namespace

mpq_status launch_allocate_budget(const float *err, int C, int k_max, long long extra,
                                  int *npoints, int *points_used, cudaStream_t stream)
{
    const long long nkeys = (long long)C * (k_max - 1);
    const bool cached = nkeys <= KEY_CACHE;
    const size_t smem = cached ? (size_t)nkeys * sizeof(unsigned long long) : 0;
    // always set: the kernel's static shared memory counts against the 48 KB default too
    cudaError_t e = cudaFuncSetAttribute(allocate_budget_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");
    allocate_budget_kernel<<<1, AB_THREADS, smem, stream>>>(err, C, k_max, extra, npoints,
                                                            points_used, cached);
    return cuda_status(cudaGetLastError(), "allocation kernel launch");
}

mpq_status launch_allocate_batch(int n, const float *const *err, const int *C, int k_max,
                                 int mode, const long long *extra, const double *eps,
                                 int *const *npoints, int *const *points_used, cudaStream_t stream)
{
    AllocBatch b;
    size_t smem = 0;
    int m = 0;
    for (int l = 0; l < n; ++l) {
        if (C[l] == 0) continue;   // nothing to allocate (points_used zeroed by the caller)
        b.err[l] = err[l];
        b.npoints[l] = npoints[l];
        b.points_used[l] = points_used ? points_used[l] : nullptr;
        b.C[l] = C[l];
        b.extra[l] = extra ? extra[l] : 0;
        b.param[l] = eps ? eps[l] : 0.0;
        const long long nkeys = (long long)C[l] * (k_max - 1);
        const bool cached = mode == MPQ_ALLOC_BUDGET && nkeys <= KEY_CACHE;
        b.cached[l] = cached;
        if (cached && (size_t)nkeys * sizeof(unsigned long long) > smem)
            smem = (size_t)nkeys * sizeof(unsigned long long);
        b.order[m++] = (unsigned char)l;
    }
    if (m == 0) return MPQ_OK;
    // largest layers first
    for (int i = 1; i < m; ++i)
        for (int j = i; j > 0 && b.C[b.order[j]] > b.C[b.order[j - 1]]; --j) {
            const unsigned char t = b.order[j];
            b.order[j] = b.order[j - 1];
            b.order[j - 1] = t;
        }
    const cudaError_t e = cudaFuncSetAttribute(allocate_batch_kernel,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)smem);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");
    allocate_batch_kernel<<<m, AB_THREADS, smem, stream>>>(b, k_max, mode);
    return cuda_status(cudaGetLastError(), "batched allocation kernel launch");
}

mpq_status launch_allocate_threshold(const float *err, int C, int k_max, double eps,
                                     int *npoints, int *points_used, cudaStream_t stream)
{
    if (points_used) {
        cudaError_t e = cudaMemsetAsync(points_used, 0, sizeof(int), stream);
        if (e != cudaSuccess) return cuda_status(e, "cudaMemsetAsync");
    }
    int blocks = (C + AT_THREADS - 1) / AT_THREADS;
    const int cap = sm_count() * 4;
    if (blocks > cap) blocks = cap;
    allocate_threshold_kernel<<<blocks, AT_THREADS, 0, stream>>>(err, C, k_max, eps, npoints,
                                                                  points_used);
    return cuda_status(cudaGetLastError(), "allocation kernel launch");
}

}  // namespace mpq
