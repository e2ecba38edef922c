// Host side of the C ABI (include/mpq.h): argument validation, error reporting, dispatch to the
// kernel launchers.  Nothing here allocates device memory or synchronizes.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <mutex>

#ifndef MPQ_NO_NVTX
#include <nvtx3/nvToolsExt.h>
#endif

#include "mpq_internal.cuh"

namespace mpq {

static thread_local char g_msg[512];

void set_error(const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
    va_end(ap);
}

mpq_status cuda_status(cudaError_t e, const char *what)
{
    if (e == cudaSuccess) return MPQ_OK;
    set_error("%s: %s (%s)", what, cudaGetErrorString(e), cudaGetErrorName(e));
    return MPQ_ERR_CUDA;
}

int sm_count()
{
    static int cache[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 148;
    if (cache[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = v > 0 ? v : 148;
    }
    return cache[dev];
}

int max_smem_optin()
{
    static int cache[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 48 * 1024;
    if (cache[dev] == 0) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
        cache[dev] = v > 0 ? v : 48 * 1024;
    }
    return cache[dev];
}

}  // namespace mpq

using namespace mpq;

// One NVTX range per C-ABI call (named after the entry point), so that a profiler's timeline shows
// which call enqueued which kernels; with no tool attached a range costs a few nanoseconds.
// Build with -DMPQ_NO_NVTX to leave them out.
namespace {
struct CallRange {
#ifndef MPQ_NO_NVTX
    explicit CallRange(const char *name) { nvtxRangePushA(name); }
    ~CallRange() { nvtxRangePop(); }
#else
    explicit CallRange(const char *) {}
#endif
};
}  // namespace

#define REQUIRE(cond, status, ...)  \
    do {                            \
        if (!(cond)) {              \
            set_error(__VA_ARGS__); \
            return (status);        \
        }                           \
    } while (0)

static mpq_status check_common(int C, int d, int k_max)
{
    REQUIRE(C >= 0, MPQ_ERR_INVALID_ARG, "C = %d must be >= 0", C);
    REQUIRE(d >= 1, MPQ_ERR_INVALID_ARG, "d = %d must be >= 1", d);
    REQUIRE(k_max >= 1, MPQ_ERR_INVALID_ARG, "k_max = %d must be >= 1", k_max);
    REQUIRE(k_max <= MPQ_MAX_POINTS, MPQ_ERR_UNSUPPORTED, "k_max = %d exceeds MPQ_MAX_POINTS = %d",
            k_max, MPQ_MAX_POINTS);
    REQUIRE((long long)C * d <= (1LL << 40), MPQ_ERR_UNSUPPORTED, "C*d = %lld too large",
            (long long)C * d);
    return MPQ_OK;
}

extern "C" mpq_status mpq_quantize_layer(const float *W, int C, int d, int bits, int G,
                                         const float *grid_frac, int k_max, int8_t *codes,
                                         float *scales, float *resid_sq, float *residuals,
                                         float *rmax, void *stream)
{
    CallRange range_("mpq_quantize_layer");
    g_msg[0] = 0;
    mpq_status st = check_common(C, d, k_max);
    if (st != MPQ_OK) return st;
    REQUIRE(bits >= MPQ_MIN_BITS && bits <= MPQ_MAX_BITS,
            (bits > MPQ_MAX_BITS ? MPQ_ERR_UNSUPPORTED : MPQ_ERR_INVALID_ARG),
            "bits = %d outside [%d, %d]", bits, MPQ_MIN_BITS, MPQ_MAX_BITS);
    REQUIRE(G >= 1, MPQ_ERR_INVALID_ARG, "G = %d must be >= 1", G);
    REQUIRE(G <= MPQ_MAX_GRID, MPQ_ERR_UNSUPPORTED, "G = %d exceeds MPQ_MAX_GRID = %d", G,
            MPQ_MAX_GRID);
    REQUIRE(d <= MPQ_MAX_DIM, MPQ_ERR_UNSUPPORTED, "d = %d exceeds MPQ_MAX_DIM = %d", d,
            MPQ_MAX_DIM);
    if (C == 0) return MPQ_OK;
    REQUIRE(W && codes && scales, MPQ_ERR_INVALID_ARG, "W, codes and scales must be non-NULL");

    GridFrac gf;
    if (grid_frac) {
        float prev = 0.0f;
        for (int g = 0; g < G; ++g) {
            float f = grid_frac[g];
            REQUIRE(isfinite(f) && f > 0.0f && f <= 1.0f, MPQ_ERR_INVALID_ARG,
                    "grid_frac[%d] = %g must be in (0, 1]", g, (double)f);
            REQUIRE(f > prev, MPQ_ERR_INVALID_ARG, "grid_frac must be strictly increasing at %d",
                    g);
            gf.f[g] = f;
            prev = f;
        }
    }
    int qmax = (1 << (bits - 1)) - 1;
    return launch_quantize(W, C, d, qmax, G, grid_frac ? &gf : nullptr, k_max, codes, scales,
                           resid_sq, residuals, rmax, (cudaStream_t)stream);
}

extern "C" mpq_status mpq_quantize_layer_adaptive(const float *W, int C, int d, int bits,
                                                  int k_max, double eta, long long max_cand,
                                                  int8_t *codes, float *scales, float *resid_sq,
                                                  long long *ncand, void *stream)
{
    CallRange range_("mpq_quantize_layer_adaptive");
    g_msg[0] = 0;
    mpq_status st = check_common(C, d, k_max);
    if (st != MPQ_OK) return st;
    REQUIRE(d <= MPQ_MAX_DIM, MPQ_ERR_UNSUPPORTED, "d = %d exceeds MPQ_MAX_DIM = %d", d,
            MPQ_MAX_DIM);
    REQUIRE(bits >= MPQ_MIN_BITS && bits <= MPQ_MAX_BITS,
            (bits > MPQ_MAX_BITS ? MPQ_ERR_UNSUPPORTED : MPQ_ERR_INVALID_ARG),
            "bits = %d outside [%d, %d]", bits, MPQ_MIN_BITS, MPQ_MAX_BITS);
    REQUIRE(isfinite(eta), MPQ_ERR_NONFINITE, "eta is not finite");
    REQUIRE(eta > 0.0, MPQ_ERR_INVALID_ARG, "eta = %g must be > 0", eta);
    REQUIRE(max_cand >= 1, MPQ_ERR_INVALID_ARG, "max_cand = %lld must be >= 1", max_cand);
    REQUIRE((long long)d * ((1 << (bits - 1)) - 1) <= MPQ_ADAPTIVE_MAX_THRESHOLDS,
            MPQ_ERR_UNSUPPORTED, "d * Qmax = %lld exceeds MPQ_ADAPTIVE_MAX_THRESHOLDS = %d",
            (long long)d * ((1 << (bits - 1)) - 1), MPQ_ADAPTIVE_MAX_THRESHOLDS);
    if (C == 0) return MPQ_OK;
    REQUIRE(W && codes && scales, MPQ_ERR_INVALID_ARG, "W, codes and scales must be non-NULL");
    return launch_adaptive(W, C, d, (1 << (bits - 1)) - 1, k_max, eta, max_cand, codes, scales,
                           resid_sq, ncand, (cudaStream_t)stream);
}

static mpq_status check_output_error(const float *X, int N, int groups, const float *W,
                                     const int8_t *codes, const float *scales, int C, int d,
                                     int k_max, float *err)
{
    mpq_status st = check_common(C, d, k_max);
    if (st != MPQ_OK) return st;
    REQUIRE(N >= 1, MPQ_ERR_INVALID_ARG, "N = %d must be >= 1", N);
    REQUIRE(groups == 1 || groups == C, MPQ_ERR_INVALID_ARG, "groups = %d must be 1 or C = %d",
            groups, C);
    REQUIRE((long long)N * d <= (1LL << 40), MPQ_ERR_UNSUPPORTED, "N*d too large");
    if (C == 0) return MPQ_OK;
    REQUIRE(X && W && codes && scales && err, MPQ_ERR_INVALID_ARG,
            "X, W, codes, scales and err must be non-NULL");
    return MPQ_OK;
}

extern "C" mpq_status mpq_output_error(const float *X, int N, int groups, const float *W,
                                       const int8_t *codes, const float *scales, const float *rmax,
                                       int C, int d, int k_max, float *err, void *stream)
{
    CallRange range_("mpq_output_error");
    g_msg[0] = 0;
    const mpq_status st = check_output_error(X, N, groups, W, codes, scales, C, d, k_max, err);
    if (st != MPQ_OK || C == 0) return st;
    return launch_output_error(X, N, groups, W, codes, scales, C, d, k_max, err,
                               (cudaStream_t)stream, nullptr, rmax);
}

// The fixed scratch of mpq_output_error_noalloc: one array for every call of that entry point
// (overlapping calls race on it, as its declaration states).  Host code cannot use the symbol
// itself as a device address: its address on each device is resolved once, with that device
// current, by the first call made there, and kept.
static __device__ __align__(256) unsigned g_noalloc_range[MPQ_NOALLOC_RANGE_WORDS];
static unsigned *g_noalloc_addr[kMaxDevices];
static std::mutex g_noalloc_mu;

static mpq_status noalloc_scratch(unsigned **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_status(e, "cudaGetDevice");
    REQUIRE(dev >= 0 && dev < kMaxDevices, MPQ_ERR_UNSUPPORTED, "device %d beyond %d devices", dev,
            kMaxDevices);
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_range);
        if (e != cudaSuccess) return cuda_status(e, "cudaGetSymbolAddress (fixed scratch)");
        g_noalloc_addr[dev] = static_cast<unsigned *>(p);
    }
    *out = g_noalloc_addr[dev];
    return MPQ_OK;
}

extern "C" mpq_status mpq_output_error_noalloc(const float *X, int N, int groups, const float *W,
                                               const int8_t *codes, const float *scales, int C,
                                               int d, int k_max, float *err, void *stream)
{
    CallRange range_("mpq_output_error_noalloc");
    g_msg[0] = 0;
    const mpq_status st = check_output_error(X, N, groups, W, codes, scales, C, d, k_max, err);
    if (st != MPQ_OK || C == 0) return st;
    const size_t words = output_error_scratch_words(X, groups, W, codes, C, d, k_max);
    REQUIRE(words <= (size_t)MPQ_NOALLOC_RANGE_WORDS, MPQ_ERR_UNSUPPORTED,
            "C = %d, k_max = %d need %zu scratch words; the fixed buffer holds %d", C, k_max, words,
            MPQ_NOALLOC_RANGE_WORDS);
    unsigned *range = nullptr;
    if (words > 0) {
        const mpq_status sa = noalloc_scratch(&range);
        if (sa != MPQ_OK) return sa;
    }
    return launch_output_error(X, N, groups, W, codes, scales, C, d, k_max, err,
                               (cudaStream_t)stream, range);
}

extern "C" mpq_status mpq_clip_search(const float *X, int N, int groups, const float *W, int C,
                                      int d, int bits, int n_cand, int mode, float *clip,
                                      float *err, int *best, void *stream)
{
    CallRange range_("mpq_clip_search");
    g_msg[0] = 0;
    mpq_status st = check_common(C, d, 1);
    if (st != MPQ_OK) return st;
    REQUIRE(d <= MPQ_MAX_DIM, MPQ_ERR_UNSUPPORTED, "d = %d exceeds MPQ_MAX_DIM = %d", d,
            MPQ_MAX_DIM);
    REQUIRE(bits >= MPQ_MIN_BITS && bits <= MPQ_MAX_BITS,
            (bits > MPQ_MAX_BITS ? MPQ_ERR_UNSUPPORTED : MPQ_ERR_INVALID_ARG),
            "bits = %d outside [%d, %d]", bits, MPQ_MIN_BITS, MPQ_MAX_BITS);
    REQUIRE(n_cand >= 1, MPQ_ERR_INVALID_ARG, "n_cand = %d must be >= 1", n_cand);
    REQUIRE(n_cand <= MPQ_MAX_CLIP_CANDIDATES, MPQ_ERR_UNSUPPORTED,
            "n_cand = %d exceeds MPQ_MAX_CLIP_CANDIDATES = %d", n_cand, MPQ_MAX_CLIP_CANDIDATES);
    REQUIRE(mode == MPQ_CLIP_PER_CHANNEL || mode == MPQ_CLIP_PER_LAYER, MPQ_ERR_INVALID_ARG,
            "mode = %d is not MPQ_CLIP_PER_CHANNEL or MPQ_CLIP_PER_LAYER", mode);
    REQUIRE(N >= 1, MPQ_ERR_INVALID_ARG, "N = %d must be >= 1", N);
    REQUIRE(groups == 1 || groups == C, MPQ_ERR_INVALID_ARG, "groups = %d must be 1 or C = %d",
            groups, C);
    REQUIRE((long long)N * d <= (1LL << 40), MPQ_ERR_UNSUPPORTED, "N*d too large");
    if (C == 0) return MPQ_OK;
    REQUIRE(X && W && clip && err && best, MPQ_ERR_INVALID_ARG,
            "X, W, clip, err and best must be non-NULL");
    return launch_clip(X, N, groups, W, C, d, (1 << (bits - 1)) - 1, n_cand, mode, clip, err, best,
                       (cudaStream_t)stream);
}

extern "C" mpq_status mpq_pack_layout(const int *npoints, int C, int d, int k_max, int bits, int p,
                                      int centered, mpq_packed_layout *layout)
{
    g_msg[0] = 0;
    mpq_status st = check_common(C, d, k_max);
    if (st != MPQ_OK) return st;
    REQUIRE(d <= MPQ_MAX_DIM, MPQ_ERR_UNSUPPORTED, "d = %d exceeds MPQ_MAX_DIM = %d", d,
            MPQ_MAX_DIM);
    REQUIRE(bits >= MPQ_MIN_BITS && bits <= MPQ_MAX_BITS,
            (bits > MPQ_MAX_BITS ? MPQ_ERR_UNSUPPORTED : MPQ_ERR_INVALID_ARG),
            "bits = %d outside [%d, %d]", bits, MPQ_MIN_BITS, MPQ_MAX_BITS);
    REQUIRE(p >= 0 && p <= 30, MPQ_ERR_INVALID_ARG, "p = %d outside [0, 30]", p);
    REQUIRE(layout, MPQ_ERR_INVALID_ARG, "layout must be non-NULL");
    REQUIRE(C == 0 || npoints, MPQ_ERR_INVALID_ARG, "npoints must be non-NULL");
    REQUIRE(centered == 0 || centered == 1, MPQ_ERR_INVALID_ARG, "centered = %d must be 0 or 1",
            centered);
    return make_pack_layout(npoints, C, d, k_max, bits, p, centered, layout);
}

extern "C" mpq_status mpq_pack_points(const int8_t *codes, const float *scales,
                                      const float *center, const int *npoints,
                                      const mpq_packed_layout *layout, void *packed, void *stream)
{
    CallRange range_("mpq_pack_points");
    g_msg[0] = 0;
    REQUIRE(layout, MPQ_ERR_INVALID_ARG, "layout must be non-NULL");
    mpq_status st = check_common(layout->C, layout->d, layout->k_max);
    if (st != MPQ_OK) return st;
    REQUIRE((center != nullptr) == (layout->centered == 1), MPQ_ERR_INVALID_ARG,
            "center must be given exactly when the layout is centered (centered = %d)",
            layout->centered);
    if (layout->C == 0) return MPQ_OK;
    REQUIRE(codes && scales && npoints && packed, MPQ_ERR_INVALID_ARG,
            "codes, scales, npoints and packed must be non-NULL");
    return launch_pack(codes, scales, center, npoints, layout, packed, (cudaStream_t)stream);
}

extern "C" mpq_status mpq_multipoint_linear(const int8_t *X, int T, const mpq_packed_layout *layout,
                                            const void *packed, int32_t *Y, void *stream)
{
    CallRange range_("mpq_multipoint_linear");
    g_msg[0] = 0;
    REQUIRE(layout, MPQ_ERR_INVALID_ARG, "layout must be non-NULL");
    mpq_status st = check_common(layout->C, layout->d, layout->k_max);
    if (st != MPQ_OK) return st;
    REQUIRE(T >= 1, MPQ_ERR_INVALID_ARG, "T = %d must be >= 1", T);
    REQUIRE((long long)T * layout->d <= (1LL << 40) && (long long)T * layout->C <= (1LL << 40),
            MPQ_ERR_UNSUPPORTED, "T too large");
    if (layout->C == 0) return MPQ_OK;
    REQUIRE(X && packed && Y, MPQ_ERR_INVALID_ARG, "X, packed and Y must be non-NULL");
    return launch_multipoint_linear(X, T, layout, packed, Y, (cudaStream_t)stream);
}

extern "C" mpq_status mpq_allocate_points(const float *err, int C, int k_max, int mode,
                                          double budget_or_eps, int *npoints, int *points_used,
                                          void *stream)
{
    CallRange range_("mpq_allocate_points");
    g_msg[0] = 0;
    mpq_status st = check_common(C, 1, k_max);
    if (st != MPQ_OK) return st;
    REQUIRE(mode == MPQ_ALLOC_BUDGET || mode == MPQ_ALLOC_THRESHOLD, MPQ_ERR_INVALID_ARG,
            "mode = %d must be MPQ_ALLOC_BUDGET (0) or MPQ_ALLOC_THRESHOLD (1)", mode);
    REQUIRE(!isnan(budget_or_eps), MPQ_ERR_NONFINITE, "budget_or_eps is NaN");
    if (mode == MPQ_ALLOC_BUDGET) {
        REQUIRE(isfinite(budget_or_eps), MPQ_ERR_NONFINITE, "budget must be finite");
        REQUIRE(budget_or_eps >= 0.0, MPQ_ERR_INVALID_ARG, "budget = %g must be >= 0",
                budget_or_eps);
    }
    if (C == 0) {
        if (points_used)
            return cuda_status(cudaMemsetAsync(points_used, 0, sizeof(int), (cudaStream_t)stream),
                               "cudaMemsetAsync");
        return MPQ_OK;
    }
    REQUIRE(err && npoints, MPQ_ERR_INVALID_ARG, "err and npoints must be non-NULL");
    if (mode == MPQ_ALLOC_THRESHOLD)
        return launch_allocate_threshold(err, C, k_max, budget_or_eps, npoints, points_used,
                                         (cudaStream_t)stream);
    long long total = (long long)floor(budget_or_eps * (double)C + 0.5);
    long long extra = total - (long long)C;
    long long cap = (long long)C * (k_max - 1);
    if (extra < 0) extra = 0;
    if (extra > cap) extra = cap;
    return launch_allocate_budget(err, C, k_max, extra, npoints, points_used,
                                  (cudaStream_t)stream);
}

extern "C" mpq_status mpq_allocate_points_batched(int n, const float *const *err, const int *C,
                                                  int k_max, int mode,
                                                  const double *budget_or_eps,
                                                  int *const *npoints, int *const *points_used,
                                                  void *stream)
{
    CallRange range_("mpq_allocate_points_batched");
    g_msg[0] = 0;
    REQUIRE(n >= 0, MPQ_ERR_INVALID_ARG, "n = %d must be >= 0", n);
    REQUIRE(n <= MPQ_MAX_BATCH, MPQ_ERR_UNSUPPORTED, "n = %d exceeds MPQ_MAX_BATCH = %d", n,
            MPQ_MAX_BATCH);
    if (n == 0) return MPQ_OK;
    REQUIRE(err && C && budget_or_eps && npoints, MPQ_ERR_INVALID_ARG,
            "err, C, budget_or_eps and npoints must be non-NULL host arrays");
    REQUIRE(mode == MPQ_ALLOC_BUDGET || mode == MPQ_ALLOC_THRESHOLD, MPQ_ERR_INVALID_ARG,
            "mode = %d must be MPQ_ALLOC_BUDGET (0) or MPQ_ALLOC_THRESHOLD (1)", mode);
    long long extra[MPQ_MAX_BATCH];
    for (int l = 0; l < n; ++l) {
        mpq_status st = check_common(C[l], 1, k_max);
        if (st != MPQ_OK) return st;
        const double v = budget_or_eps[l];
        REQUIRE(!isnan(v), MPQ_ERR_NONFINITE, "budget_or_eps[%d] is NaN", l);
        if (mode == MPQ_ALLOC_BUDGET) {
            REQUIRE(isfinite(v), MPQ_ERR_NONFINITE, "budget[%d] must be finite", l);
            REQUIRE(v >= 0.0, MPQ_ERR_INVALID_ARG, "budget[%d] = %g must be >= 0", l, v);
        }
        REQUIRE(C[l] == 0 || (err[l] && npoints[l]), MPQ_ERR_INVALID_ARG,
                "err[%d] and npoints[%d] must be non-NULL", l, l);
        long long e = (long long)floor(v * (double)C[l] + 0.5) - (long long)C[l];
        const long long cap = (long long)C[l] * (k_max - 1);
        extra[l] = e < 0 ? 0 : (e > cap ? cap : e);
    }
    for (int l = 0; l < n; ++l)   // empty layers: no CTA, a zero total
        if (C[l] == 0 && points_used && points_used[l]) {
            const mpq_status st = cuda_status(
                cudaMemsetAsync(points_used[l], 0, sizeof(int), (cudaStream_t)stream),
                "cudaMemsetAsync");
            if (st != MPQ_OK) return st;
        }
    return launch_allocate_batch(n, err, C, k_max, mode, extra, budget_or_eps, npoints,
                                 points_used, (cudaStream_t)stream);
}

extern "C" mpq_status mpq_reconstruct(const int8_t *codes, const float *scales, const int *npoints,
                                      const float *center, int C, int d, int k_max, float *W_hat,
                                      void *stream)
{
    CallRange range_("mpq_reconstruct");
    g_msg[0] = 0;
    mpq_status st = check_common(C, d, k_max);
    if (st != MPQ_OK) return st;
    if (C == 0) return MPQ_OK;
    REQUIRE(codes && scales && npoints && W_hat, MPQ_ERR_INVALID_ARG,
            "codes, scales, npoints and W_hat must be non-NULL");
    return launch_reconstruct(codes, scales, npoints, center, C, d, k_max, W_hat,
                              (cudaStream_t)stream);
}

extern "C" mpq_status mpq_center_weights(const float *W, int C, int d, int mode, float *center,
                                         float *Wc, void *stream)
{
    CallRange range_("mpq_center_weights");
    g_msg[0] = 0;
    mpq_status st = check_common(C, d, 1);
    if (st != MPQ_OK) return st;
    REQUIRE(mode == MPQ_CENTER_PER_CHANNEL || mode == MPQ_CENTER_PER_LAYER, MPQ_ERR_INVALID_ARG,
            "mode = %d is not MPQ_CENTER_PER_CHANNEL or MPQ_CENTER_PER_LAYER", mode);
    if (C == 0) return MPQ_OK;
    REQUIRE(W && center && Wc, MPQ_ERR_INVALID_ARG, "W, center and Wc must be non-NULL");
    return launch_center(W, C, d, mode, center, Wc, (cudaStream_t)stream);
}

extern "C" const char *mpq_status_string(mpq_status s)
{
    switch (s) {
    case MPQ_OK: return "MPQ_OK";
    case MPQ_ERR_INVALID_ARG: return "MPQ_ERR_INVALID_ARG";
    case MPQ_ERR_NONFINITE: return "MPQ_ERR_NONFINITE";
    case MPQ_ERR_UNSUPPORTED: return "MPQ_ERR_UNSUPPORTED";
    case MPQ_ERR_CUDA: return "MPQ_ERR_CUDA";
    case MPQ_ERR_TIMEOUT: return "MPQ_ERR_TIMEOUT";
    case MPQ_ERR_NOMEM: return "MPQ_ERR_NOMEM";
    case MPQ_ERR_BOUNDS: return "MPQ_ERR_BOUNDS";
    }
    return "MPQ_ERR_UNKNOWN";
}

extern "C" const char *mpq_last_error(void) { return g_msg; }

extern "C" int mpq_version(void) { return 200; }
