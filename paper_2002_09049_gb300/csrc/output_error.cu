// Output error of every channel for every point count (Sec. 3.3, Eq. 11):
//   err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2,  n = 0..k_max,
// with the residuals r_{k,n+1} regenerated on chip from W, codes and scales by the recursion of
// Eq. 7 (never materialised in global memory).
//
// Shared input (groups = 1) is a dense contraction and runs on the tensor cores: the CTA-pair kernel
// (output_error_pair.cu) when rows are 16-byte multiples, else the single-CTA one
// (output_error_tc.cu).  Per-channel input (groups = C, depthwise convolution, d = 9): one CTA per
// channel, its k_max+1 residuals in shared memory, the channel's own rows of X staged through
// shared memory with coalesced reads (each read once), threads over the rows.
#include <math.h>

#include "mpq_internal.cuh"

MPQ_CHECKED_UNIT("output_error.cu");

namespace mpq {
namespace {

constexpr int GR_THREADS = 256;

constexpr int GR_X_FLOATS = 4096;                 // 16 KB of calibration rows staged at a time

template <int KP1>
__global__ void __launch_bounds__(GR_THREADS)
output_error_grouped_kernel(const float *__restrict__ X, int N, const float *__restrict__ W,
                            const int8_t *__restrict__ codes, const float *__restrict__ scales,
                            int C, int d, float *__restrict__ err)
{
    extern __shared__ __align__(16) float Rsh[];   // [KP1][d], then rows of X [GR_X_FLOATS]
    __shared__ float red[GR_THREADS / 32][KP1];
    const int k = blockIdx.x;
    const int tid = threadIdx.x;
    const int k_max = KP1 - 1;
    const size_t plane = (size_t)C * d;
    // the residual rows and one staged chunk of X within the launch's shared memory
    if (!MPQ_IN(k, C) || !MPQ_CHECK(d <= GR_X_FLOATS) ||
        !MPQ_CHECK_SMEM_END(4 * ((size_t)((KP1 * d + 3) & ~3) + GR_X_FLOATS)))
        return;

    for (int j = tid; j < d; j += GR_THREADS) {
        float r = W[(size_t)k * d + j];
        Rsh[j] = r;
        for (int i = 0; i < k_max; ++i) {
            r = __fmaf_rn(-scales[(size_t)k * k_max + i], (float)codes[(size_t)i * plane + (size_t)k * d + j], r);
            Rsh[(size_t)(i + 1) * d + j] = r;
        }
    }
    __syncthreads();

    const float *Xk = X + (size_t)k * N * d;
    float *Xsh = Rsh + ((KP1 * d + 3) & ~3);
    const int chunk = GR_X_FLOATS / d;               // rows per staged chunk (d <= GR_X_FLOATS)
    // All in fp32 (the part's fp64 rate is a small fraction of its fp32 rate, and fp64 work per
    // row, or fp64 warp reductions, bound the kernel): squares summed over at most ERR_FOLD rows of
    // a thread, folded into a compensated (Kahan) sum, then a tree over the threads and one
    // division -- relative error below (ERR_FOLD + 2 + 8 + 1) * 2^-24 in all.
    constexpr int ERR_FOLD = 16;
    float acc[KP1], comp[KP1], part[KP1];
#pragma unroll
    for (int n = 0; n < KP1; ++n) {
        acc[n] = 0.0f;
        comp[n] = 0.0f;
        part[n] = 0.0f;
    }
    int rows = 0;
    for (int t0 = 0; t0 < N; t0 += chunk) {
        // the channel's next rows of X, read with consecutive threads on consecutive words
        const int nr = min(chunk, N - t0);
        __syncthreads();   // the previous chunk is no longer read
        for (int i = tid; i < nr * d; i += GR_THREADS) Xsh[i] = Xk[(size_t)t0 * d + i];
        __syncthreads();
        for (int t = tid; t < nr; t += GR_THREADS) {
            float y[KP1];
#pragma unroll
            for (int n = 0; n < KP1; ++n) y[n] = 0.0f;
            const float *x = Xsh + t * d;
            for (int j = 0; j < d; ++j) {
                const float xv = x[j];
#pragma unroll
                for (int n = 0; n < KP1; ++n) y[n] = fmaf(xv, Rsh[n * d + j], y[n]);
            }
#pragma unroll
            for (int n = 0; n < KP1; ++n) part[n] = fmaf(y[n], y[n], part[n]);
            if (++rows == ERR_FOLD) {
#pragma unroll
                for (int n = 0; n < KP1; ++n) {
                    kahan_add(acc[n], comp[n], part[n]);
                    part[n] = 0.0f;
                }
                rows = 0;
            }
        }
    }
    const int lane = tid & 31, wp = tid >> 5;
#pragma unroll
    for (int n = 0; n < KP1; ++n) {
        kahan_add(acc[n], comp[n], part[n]);
        float v = acc[n];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) red[wp][n] = v;
    }
    __syncthreads();
    if (tid < KP1) {
        float v[GR_THREADS / 32];
        for (int i = 0; i < GR_THREADS / 32; ++i) v[i] = red[i][tid];
        for (int w = GR_THREADS / 64; w > 0; w >>= 1)   // tree over the warps
            for (int i = 0; i < w; ++i) v[i] += v[i + w];
        if (MPQ_IN((size_t)k * KP1 + tid, (size_t)C * KP1))
            err[(size_t)k * KP1 + tid] = mean_of_sum(v[0], N);
    }
}

template <int KP1>
mpq_status launch_grouped(const float *X, int N, const float *W, const int8_t *codes,
                          const float *scales, int C, int d, float *err, cudaStream_t stream)
{
    const size_t smem = ((size_t)(KP1 * d + 3) / 4 * 4 + GR_X_FLOATS) * sizeof(float);
    if (d > GR_X_FLOATS || (long long)smem > max_smem_optin()) {
        set_error("groups = C with d = %d and k_max = %d needs %zu bytes of shared memory", d,
                  KP1 - 1, smem);
        return MPQ_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(output_error_grouped_kernel<KP1>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) {
        output_error_grouped_kernel<KP1><<<C, GR_THREADS, smem, stream>>>(X, N, W, codes, scales,
                                                                          C, d, err);
        e = cudaGetLastError();
    }
    return cuda_status(e, "grouped output-error kernel launch");
}

}  // namespace

size_t output_error_scratch_words(const float *X, int groups, const float *W,
                                  const int8_t *codes, int C, int d, int k_max)
{
    return (groups == 1 && output_error_pair_ok(X, W, codes, d)) ? 1 + (size_t)C * (k_max + 1) : 0;
}

mpq_status launch_output_error(const float *X, int N, int groups, const float *W,
                               const int8_t *codes, const float *scales, int C, int d, int k_max,
                               float *err, cudaStream_t stream, unsigned *range,
                               const float *rmax)
{
    if (groups == 1) {
        if (output_error_pair_ok(X, W, codes, d))
            return launch_output_error_pair(X, N, W, codes, scales, C, d, k_max, err, stream,
                                            range, rmax);
        return launch_output_error_tc(X, N, W, codes, scales, C, d, k_max, err, stream);
    }
    switch (k_max + 1) {
#define MPQ_CASE(n) \
    case n: return launch_grouped<n>(X, N, W, codes, scales, C, d, err, stream);
        MPQ_CASE(2) MPQ_CASE(3) MPQ_CASE(4) MPQ_CASE(5) MPQ_CASE(6) MPQ_CASE(7) MPQ_CASE(8)
        MPQ_CASE(9) MPQ_CASE(10) MPQ_CASE(11) MPQ_CASE(12) MPQ_CASE(13) MPQ_CASE(14) MPQ_CASE(15)
        MPQ_CASE(16) MPQ_CASE(17)
#undef MPQ_CASE
    }
    set_error("k_max = %d unsupported", k_max);
    return MPQ_ERR_UNSUPPORTED;
}

}  // namespace mpq
