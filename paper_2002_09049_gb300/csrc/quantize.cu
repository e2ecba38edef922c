// Greedy multipoint construction (Sec. 3.2, Eq. 6-9, Algorithm 1) for every channel of a layer.
//
// One CTA owns one channel for all k_max steps: the residual row r (fp32) stays in shared memory
// from the first load of w to the last update, so global memory sees one read of w and one write
// of each step's codes (and of the optional residual / norm outputs).
//
// Scale search (Eq. 9).  For a candidate scale s with codes c_j = min(Qmax, rint(|r_j| / s)),
//   E(s) = ||r - s q||^2 = ||r||^2 - 2 s P + s^2 N,   P = sum_j |r_j| c_j,   N = sum_j c_j^2,
// so only D(s) = s (s N - 2 P) decides the argmin.  N is an exact integer.  P is accumulated
// exactly in 64-bit fixed point: |r_j| is scaled by 2^S (S chosen per step from max|r| so the sum
// cannot overflow), which is exact for every element whose code can be nonzero on the grid.  D is
// then evaluated once per candidate in double, so the decision carries ~1e-16 relative error --
// independent of d and of the summation order, hence deterministic.
#include <float.h>
#include <limits.h>
#include <math.h>

#include "mpq_internal.cuh"

namespace mpq {
namespace {

constexpr int QBLOCK = 256;
constexpr int QWARPS = QBLOCK / 32;

template <bool CUSTOM>
struct Grid;

template <>
struct Grid<false> {
    // f_g = g / G for the 1-based index g, one fp32 division
    __device__ __forceinline__ float frac(int g0, int G) const
    {
        return __fdiv_rn((float)(g0 + 1), (float)G);
    }
};

template <>
struct Grid<true> {
    GridFrac gf;
    __device__ __forceinline__ float frac(int g0, int) const { return gf.f[g0]; }
};

__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ double warp_sum(double v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

struct Reduce {
    float f[QWARPS];
    double dd[QWARPS];
    int g[QWARPS];
};

// Block-wide max of non-negative floats (exact).
__device__ float block_max(float v, Reduce &sh)
{
    v = warp_max(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) sh.f[w] = v;
    __syncthreads();
    float m = sh.f[0];
#pragma unroll
    for (int i = 1; i < QWARPS; ++i) m = fmaxf(m, sh.f[i]);
    return m;
}

// Block-wide sum in double, fixed reduction tree (deterministic).
__device__ double block_sum(double v, Reduce &sh)
{
    v = warp_sum(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) sh.dd[w] = v;
    __syncthreads();
    double s = 0.0;
#pragma unroll
    for (int i = 0; i < QWARPS; ++i) s += sh.dd[i];
    return s;
}

// Block-wide lexicographic min of (D, g): smallest D, lowest g among equal D.
__device__ int block_argmin(double D, int g, Reduce &sh)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        double D2 = __shfl_xor_sync(0xffffffffu, D, o);
        int g2 = __shfl_xor_sync(0xffffffffu, g, o);
        if (D2 < D || (D2 == D && g2 < g)) {
            D = D2;
            g = g2;
        }
    }
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) {
        sh.dd[w] = D;
        sh.g[w] = g;
    }
    __syncthreads();
    D = sh.dd[0];
    g = sh.g[0];
#pragma unroll
    for (int i = 1; i < QWARPS; ++i)
        if (sh.dd[i] < D || (sh.dd[i] == D && sh.g[i] < g)) {
            D = sh.dd[i];
            g = sh.g[i];
        }
    return g;
}

// Code magnitude of |r| at scale s > 0 (Eq. 8): nearest integer (ties to even) of the correctly
// rounded fp32 quotient, clipped to Qmax.
__device__ __forceinline__ int code_mag(float a, float s, float qmaxf)
{
    return (int)fminf(rintf(__fdiv_rn(a, s)), qmaxf);
}

// tsplit threads cooperate on one candidate (interleaved over j); QBLOCK / tsplit candidates are
// evaluated per pass.
template <bool CUSTOM>
__global__ void __launch_bounds__(QBLOCK)
quantize_direct_kernel(const float *__restrict__ W, int C, int d, int qmax, int G,
                       const Grid<CUSTOM> grid, int k_max, int8_t *__restrict__ codes,
                       float *__restrict__ scales, float *__restrict__ resid_sq,
                       float *__restrict__ residuals, int hbits, int tsplit)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    long long *sR = reinterpret_cast<long long *>(smem_raw);    // [d] fixed-point |r_j|
    float *sr = reinterpret_cast<float *>(sR + d);              // [d] residual r_j
    __shared__ Reduce red;

    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const float qmaxf = (float)qmax;
    const size_t plane = (size_t)C * d;
    const float *w = W + (size_t)k * d;

    int bad = 0;
    float part = 0.0f;
    for (int j = tid; j < d; j += QBLOCK) {
        float v = w[j];
        sr[j] = v;
        bad |= !isfinite(v);
        part = fmaf(v, v, part);
    }
    bad = __syncthreads_or(bad);
    double r2 = block_sum((double)part, red);
    if (resid_sq && tid == 0) resid_sq[(size_t)k * (k_max + 1)] = bad ? NAN : (float)r2;

    const int group = tid / tsplit, lane_in = tid % tsplit;
    const int per_pass = QBLOCK / tsplit;

    for (int i = 0; i < k_max; ++i) {
        int8_t *qi = codes + (size_t)i * plane + (size_t)k * d;
        float *ri = residuals ? residuals + (size_t)i * plane + (size_t)k * d : nullptr;
        if (bad) {
            for (int j = tid; j < d; j += QBLOCK) {
                qi[j] = 0;
                if (ri) ri[j] = sr[j];
            }
            if (tid == 0) {
                scales[(size_t)k * k_max + i] = NAN;
                if (resid_sq) resid_sq[(size_t)k * (k_max + 1) + i + 1] = NAN;
            }
            continue;
        }

        float am = 0.0f;
        for (int j = tid; j < d; j += QBLOCK) am = fmaxf(am, fabsf(sr[j]));
        const float m = block_max(am, red);

        float s_best = 0.0f;
        if (m > 0.0f) {
            const float smax = __fdiv_rn(m, qmaxf);
            int e;
            frexpf(m, &e);                      // m < 2^e
            const int S = 62 - e - hbits;       // sum_j R_j c_j < 2^62
            const double up = ldexp(1.0, S), down = ldexp(1.0, -S);
            for (int j = tid; j < d; j += QBLOCK) sR[j] = __double2ll_rn(fabs((double)sr[j]) * up);
            __syncthreads();

            double bestD = DBL_MAX;
            int bestg = INT_MAX;
            for (int gb = 0; gb < G; gb += per_pass) {
                const int g = gb + group;
                float s = 0.0f;
                long long P = 0;
                int N = 0;
                if (g < G) {
                    s = __fmul_rn(grid.frac(g, G), smax);
                    if (s > 0.0f) {
                        for (int j = lane_in; j < d; j += tsplit) {
                            const int c = code_mag(fabsf(sr[j]), s, qmaxf);
                            P += sR[j] * (long long)c;
                            N += c * c;
                        }
                    }
                }
                for (int o = tsplit >> 1; o > 0; o >>= 1) {
                    P += __shfl_xor_sync(0xffffffffu, P, o);
                    N += __shfl_xor_sync(0xffffffffu, N, o);
                }
                if (g < G && lane_in == 0) {
                    double D = 0.0;  // s == 0 (underflow): all codes 0, E = ||r||^2
                    if (s > 0.0f) {
                        const double sd = (double)s;
                        const double T = __fma_rn(sd, (double)N, -2.0 * ((double)P * down));
                        D = __dmul_rn(sd, T);
                    }
                    if (D < bestD) {
                        bestD = D;
                        bestg = g;
                    }
                }
            }
            int g = block_argmin(bestD, bestg, red);
            if (g < 0 || g >= G) g = G - 1;   // unreachable: every D is finite
            s_best = __fmul_rn(grid.frac(g, G), smax);
        }

        // residual update (Eq. 7) and code emission
        part = 0.0f;
        for (int j = tid; j < d; j += QBLOCK) {
            float v = sr[j];
            int q = 0;
            if (s_best > 0.0f) {
                const int c = code_mag(fabsf(v), s_best, qmaxf);
                q = (v < 0.0f) ? -c : c;
                v = __fmaf_rn(-s_best, (float)q, v);
            }
            qi[j] = (int8_t)q;
            sr[j] = v;
            if (ri) ri[j] = v;
            part = fmaf(v, v, part);
        }
        if (tid == 0) scales[(size_t)k * k_max + i] = s_best;
        r2 = block_sum((double)part, red);   // also orders the sr[] writes before the next step
        if (resid_sq && tid == 0) resid_sq[(size_t)k * (k_max + 1) + i + 1] = (float)r2;
    }
}

int ceil_log2(long long x)
{
    int b = 0;
    while ((1LL << b) < x) ++b;
    return b;
}

}  // namespace

mpq_status launch_quantize(const float *W, int C, int d, int qmax, int G, const GridFrac *grid,
                           int k_max, int8_t *codes, float *scales, float *resid_sq,
                           float *residuals, cudaStream_t stream)
{
    const size_t smem = (size_t)d * (sizeof(long long) + sizeof(float));
    if ((long long)smem > max_smem_optin()) {
        set_error("d = %d needs %zu bytes of shared memory", d, smem);
        return MPQ_ERR_UNSUPPORTED;
    }
    const int hbits = ceil_log2((long long)d * qmax) + 1;
    int tsplit = 1;
    while (tsplit < 32 && (long long)G * tsplit < QBLOCK) tsplit <<= 1;

    cudaError_t e;
    if (grid) {
        Grid<true> g;
        g.gf = *grid;
        e = cudaFuncSetAttribute(quantize_direct_kernel<true>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e == cudaSuccess) {
            quantize_direct_kernel<true><<<C, QBLOCK, smem, stream>>>(
                W, C, d, qmax, G, g, k_max, codes, scales, resid_sq, residuals, hbits, tsplit);
            e = cudaGetLastError();
        }
    } else {
        e = cudaFuncSetAttribute(quantize_direct_kernel<false>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e == cudaSuccess) {
            quantize_direct_kernel<false><<<C, QBLOCK, smem, stream>>>(
                W, C, d, qmax, G, Grid<false>(), k_max, codes, scales, resid_sq, residuals, hbits,
                tsplit);
            e = cudaGetLastError();
        }
    }
    return cuda_status(e, "quantize kernel launch");
}

}  // namespace mpq
