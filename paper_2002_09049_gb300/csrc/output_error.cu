// Output error of every channel for every point count (Sec. 3.3, Eq. 11):
//   err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2,  n = 0..k_max,
// with the residuals r_{k,n+1} regenerated on chip from W, codes and scales by the recursion of
// Eq. 7 (never materialised in global memory).
//
// Shared input (groups = 1): a dense contraction Y = X R^T of X [N][d] with the C*(k_max+1)
// residual vectors, squared and averaged over the N rows in the epilogue.  One CTA owns 64 residual
// vectors and sweeps all N rows, so each err value is produced by exactly one CTA in a fixed order
// (deterministic, no atomics, no scratch memory).
//
// Per-channel input (groups = C, depthwise): one CTA per channel, its k_max+1 residuals in shared
// memory, threads over the calibration rows.
#include <math.h>
#include <stdlib.h>

#include "mpq_internal.cuh"

namespace mpq {
namespace {

constexpr int BM = 64;   // calibration rows per tile
constexpr int BN = 64;   // residual vectors per CTA
constexpr int BK = 16;   // d-chunk
constexpr int OE_THREADS = 256;

__global__ void __launch_bounds__(OE_THREADS)
output_error_shared_kernel(const float *__restrict__ X, int N, const float *__restrict__ W,
                           const int8_t *__restrict__ codes, const float *__restrict__ scales,
                           int C, int d, int k_max, float *__restrict__ err)
{
    __shared__ __align__(16) float Xs[BK][BM];
    __shared__ __align__(16) float Rs[BK][BN];
    __shared__ double red[16][BN];

    const int KP1 = k_max + 1;
    const long long V = (long long)C * KP1;
    const long long v0 = (long long)blockIdx.x * BN;
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;       // compute: vectors tx*4.., rows ty*4..
    const int lr = tid >> 2, lc = (tid & 3) * 4;  // load: row/vector lr, columns lc..lc+3
    const size_t plane = (size_t)C * d;

    const long long v = v0 + lr;
    const bool vvalid = v < V;
    const int kch = vvalid ? (int)(v / KP1) : 0;
    const int nn = vvalid ? (int)(v % KP1) : 0;
    const float *wrow = W + (size_t)kch * d;
    const float *srow = scales + (size_t)kch * k_max;
    const int8_t *crow = codes + (size_t)kch * d;

    double sq[4] = {0.0, 0.0, 0.0, 0.0};
    for (int t0 = 0; t0 < N; t0 += BM) {
        float acc[4][4];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[a][b] = 0.0f;

        for (int j0 = 0; j0 < d; j0 += BK) {
            const int t = t0 + lr;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int j = j0 + lc + c;
                Xs[lc + c][lr] = (t < N && j < d) ? X[(size_t)t * d + j] : 0.0f;
                float r = 0.0f;
                if (vvalid && j < d) {
                    r = wrow[j];
                    for (int i = 0; i < nn; ++i)
                        r = __fmaf_rn(-srow[i], (float)crow[(size_t)i * plane + j], r);
                }
                Rs[lc + c][lr] = r;
            }
            __syncthreads();
#pragma unroll
            for (int kk = 0; kk < BK; ++kk) {
                const float4 a = *reinterpret_cast<const float4 *>(&Xs[kk][ty * 4]);
                const float4 b = *reinterpret_cast<const float4 *>(&Rs[kk][tx * 4]);
                const float av[4] = {a.x, a.y, a.z, a.w};
                const float bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                for (int p = 0; p < 4; ++p)
#pragma unroll
                    for (int q = 0; q < 4; ++q) acc[p][q] = fmaf(av[p], bv[q], acc[p][q]);
            }
            __syncthreads();
        }
#pragma unroll
        for (int p = 0; p < 4; ++p) {
            if (t0 + ty * 4 + p < N) {
#pragma unroll
                for (int q = 0; q < 4; ++q) sq[q] += (double)acc[p][q] * (double)acc[p][q];
            }
        }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) red[ty][tx * 4 + q] = sq[q];
    __syncthreads();
    if (tid < BN && v0 + tid < V) {
        double s = 0.0;
        for (int y = 0; y < 16; ++y) s += red[y][tid];
        err[v0 + tid] = (float)(s / (double)N);
    }
}

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
    if (groups == 1 && !getenv("MPQ_DEBUG_SIMT_OUTPUT_ERROR"))
        return launch_output_error_tc(X, N, W, codes, scales, C, d, k_max, err, stream);
    if (groups == 1) {
        const long long V = (long long)C * (k_max + 1);
        const long long blocks = (V + BN - 1) / BN;
        output_error_shared_kernel<<<(unsigned)blocks, OE_THREADS, 0, stream>>>(
            X, N, W, codes, scales, C, d, k_max, err);
        return cuda_status(cudaGetLastError(), "output-error kernel launch");
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
