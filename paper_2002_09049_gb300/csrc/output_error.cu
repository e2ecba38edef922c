// Output error of every channel for every point count (Sec. 3.3, Eq. 11):
//   err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2,  n = 0..k_max,
// with the residuals r_{k,n+1} regenerated on chip from W, codes and scales by the recursion of
// Eq. 7 (never materialised in global memory).
//
// Shared input (groups = 1) is a dense contraction and runs on the tensor cores
// (output_error_tc.cu).  Per-channel input (groups = C, depthwise convolution, d = 9): one CTA per
// channel, its k_max+1 residuals in shared memory, threads over the calibration rows; each
// channel's own X block is read once, so this path is bound by HBM.
#include <math.h>

#include "mpq_internal.cuh"

namespace mpq {
namespace {

constexpr int GR_THREADS = 256;

template <int KP1>
__global__ void __launch_bounds__(GR_THREADS)
output_error_grouped_kernel(const float *__restrict__ X, int N, const float *__restrict__ W,
                            const int8_t *__restrict__ codes, const float *__restrict__ scales,
                            int C, int d, float *__restrict__ err)
{
    extern __shared__ __align__(16) float Rsh[];   // [KP1][d]
    __shared__ double red[GR_THREADS / 32][KP1];
    const int k = blockIdx.x;
    const int tid = threadIdx.x;
    const int k_max = KP1 - 1;
    const size_t plane = (size_t)C * d;

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
    double acc[KP1];
#pragma unroll
    for (int n = 0; n < KP1; ++n) acc[n] = 0.0;
    for (int t = tid; t < N; t += GR_THREADS) {
        float y[KP1];
#pragma unroll
        for (int n = 0; n < KP1; ++n) y[n] = 0.0f;
        const float *x = Xk + (size_t)t * d;
        for (int j = 0; j < d; ++j) {
            const float xv = x[j];
#pragma unroll
            for (int n = 0; n < KP1; ++n) y[n] = fmaf(xv, Rsh[n * d + j], y[n]);
        }
#pragma unroll
        for (int n = 0; n < KP1; ++n) acc[n] += (double)y[n] * (double)y[n];
    }
    const int lane = tid & 31, wp = tid >> 5;
#pragma unroll
    for (int n = 0; n < KP1; ++n) {
        double v = acc[n];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) red[wp][n] = v;
    }
    __syncthreads();
    if (tid < KP1) {
        double s = 0.0;
        for (int i = 0; i < GR_THREADS / 32; ++i) s += red[i][tid];
        err[(size_t)k * KP1 + tid] = (float)(s / (double)N);
    }
}

template <int KP1>
mpq_status launch_grouped(const float *X, int N, const float *W, const int8_t *codes,
                          const float *scales, int C, int d, float *err, cudaStream_t stream)
{
    const size_t smem = (size_t)KP1 * d * sizeof(float);
    if ((long long)smem > max_smem_optin()) {
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

mpq_status launch_output_error(const float *X, int N, int groups, const float *W,
                               const int8_t *codes, const float *scales, int C, int d, int k_max,
                               float *err, cudaStream_t stream)
{
    if (groups == 1) {
        if (output_error_pair_ok(X, W, codes, d))
            return launch_output_error_pair(X, N, W, codes, scales, C, d, k_max, err, stream);
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
