// Greedy multipoint construction (Sec. 3.2, Eq. 6-9, Algorithm 1) for every channel of a layer.
//
// One CTA owns one channel for all k_max steps: the residual row r (fp32) stays in shared memory
// from the first load of w to the last update, so global memory sees one read of w and one write
// of each step's codes (and of the optional residual / norm outputs).
//
// Scale search (Eq. 9).  For a candidate scale s with codes c_j = min(Qmax, rint(|r_j| / s)),
//   E(s) = ||r - s q||^2 = ||r||^2 - 2 s P + s^2 N,   P = sum_j |r_j| c_j,   N = sum_j c_j^2,
// so only D(s) = s (s N - 2 P) decides the argmin.  N is an exact integer and P is accumulated
// exactly in 64-bit fixed point (|r_j| scaled by 2^S, S chosen per step from max|r| so the sum
// cannot overflow; exact for every element whose code can be nonzero on the grid).  D is then
// formed once per candidate in double: the decision carries ~1e-16 relative error, independent
// of d and of summation order, hence deterministic.
//
// Event form.  The candidate scales increase with g, so every element's code c_j(g) is a
// non-increasing step function of g (the fp32 quotient, rint and the clamp are all monotone).
// For each level L, {g : c_j(g) >= L} is a prefix [0, T_{j,L}); hence
//   P_g = sum_{(j,L)} R_j [g < T_{j,L}],   N_g = sum_{(j,L)} (2L - 1) [g < T_{j,L}].
// Levels held at the largest scale (L <= c_j(G-1)) count for every g and are summed directly;
// every other level the element crosses adds (R_j, 2L-1) to a histogram bin T_{j,L}, found by a
// binary search on the scale table followed by an exact check with the same correctly rounded
// division and rint as the definition.  A suffix sum over the bins gives P_g and N_g for all g.
// Work per element and step is O(Qmax) instead of O(G).  (If a candidate scale underflows to 0
// the monotonicity argument fails; such steps evaluate every candidate directly.)
#include <float.h>
#include <limits.h>
#include <math.h>

#include "mpq_internal.cuh"

namespace mpq {
namespace {

constexpr int QBLOCK = 256;
constexpr int QWARPS = QBLOCK / 32;
constexpr int MPQ_QMAX_LIMIT = (1 << (MPQ_MAX_BITS - 1)) - 1;

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

template <typename T>
__device__ __forceinline__ T warp_sum(T v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

struct Reduce {
    float f[QWARPS];
    double dd[QWARPS];
    long long ll[QWARPS];
    int g[QWARPS];
    int flag;
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

// Block-wide max of non-negative floats and sum of doubles in one pass (fixed tree).
__device__ void block_max_sum(float &m, double &v, Reduce &sh)
{
    m = warp_max(m);
    v = warp_sum(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) {
        sh.f[w] = m;
        sh.dd[w] = v;
    }
    __syncthreads();
    m = sh.f[0];
    v = 0.0;
#pragma unroll
    for (int i = 0; i < QWARPS; ++i) {
        m = fmaxf(m, sh.f[i]);
        v += sh.dd[i];
    }
}

// Block-wide sums, fixed reduction tree (deterministic).
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

__device__ long long block_sum_ll(long long v, Reduce &sh)
{
    v = warp_sum(v);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) sh.ll[w] = v;
    __syncthreads();
    long long s = 0;
#pragma unroll
    for (int i = 0; i < QWARPS; ++i) s += sh.ll[i];
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

// |r| as a 64-bit fixed-point integer R = |r| * 2^S, from the fp32 bits (no fp64 work).  Exact
// whenever |r| * 2^S is an integer, i.e. for every element large enough to take a nonzero code;
// smaller elements are truncated (their P contribution is zero anyway).
__device__ __forceinline__ long long fixed_point(float a, int S)
{
    const uint32_t bits = __float_as_uint(a);
    const int E = (int)(bits >> 23);
    const long long M = (long long)((bits & 0x7FFFFFu) | (E ? 0x800000u : 0u));
    const int sh = (E ? E : 1) - 150 + S;   // a = M * 2^((E ? E : 1) - 150)
    if (sh >= 0) return M << sh;
    return sh > -40 ? (M >> -sh) : 0;
}

// Bound on |a * fl(1/s) - fl(a/s)| relative to the quotient, with margin: both roundings are
// 2^-24 each, so a fast quotient further than this from a rounding boundary decides exactly as
// the correctly rounded division would.
#define MPQ_FAST_REL 9.5367431640625e-07f   /* 2^-20 */

// rint(fl(a/s)) >= L, decided from q' = a * (1/s) unless q' is too close to L - 1/2.
__device__ __forceinline__ bool level_held(float a, float s, float inv_s, int L)
{
    const float qf = __fmul_rn(a, inv_s);
    const float h = (float)L - 0.5f;
    const float tol = MPQ_FAST_REL * (qf + 1.0f);
    if (qf > h + tol) return true;
    if (qf < h - tol) return false;
    return rintf(__fdiv_rn(a, s)) >= (float)L;
}

// min(Qmax, rint(fl(a/s))), decided from q' = a * (1/s) unless q' is too close to a half-integer.
__device__ __forceinline__ int code_fast(float a, float s, float inv_s, float qmaxf)
{
    const float qf = __fmul_rn(a, inv_s);
    const float tol = MPQ_FAST_REL * (qf + 1.0f);
    if (qf > qmaxf + 0.5f + tol) return (int)qmaxf;
    const float fl = floorf(qf);
    const float fr = qf - fl;   // exact
    if (fabsf(fr - 0.5f) > tol) return (int)fminf(fr > 0.5f ? fl + 1.0f : fl, qmaxf);
    return (int)fminf(rintf(__fdiv_rn(a, s)), qmaxf);
}

// Decision value D(s) = s (s N - 2 P) with P = Pfix * 2^-S, in double.
__device__ __forceinline__ double decision(float s, long long Pfix, long long N, double down)
{
    const double sd = (double)s;
    const double T = __fma_rn(sd, (double)N, -2.0 * ((double)Pfix * down));
    return __dmul_rn(sd, T);
}

template <bool CUSTOM>
__global__ void __launch_bounds__(QBLOCK, 4)
quantize_event_kernel(const float *__restrict__ W, int C, int d, int qmax, int G,
                      const Grid<CUSTOM> grid, int k_max, int8_t *__restrict__ codes,
                      float *__restrict__ scales, float *__restrict__ resid_sq,
                      float *__restrict__ residuals, int hbits)
{
    extern __shared__ __align__(16) unsigned char smem_raw[];
    // Event bins.  P bins are 64-bit values kept as two 32-bit words (32-bit shared atomics are
    // native; 64-bit ones are several times slower under contention): the low word takes an
    // atomic add whose returned old value shows every wrap-around exactly, and the high word
    // takes R >> 32 plus that carry.  After the events hP holds the combined 64-bit sums.
    long long *hP = reinterpret_cast<long long *>(smem_raw);    // [G + 1] P bins (lo | hi words)
    int *hN = reinterpret_cast<int *>(hP + (G + 1));             // [G + 1] event bins of N
    float *stab = reinterpret_cast<float *>(hN + (G + 1));       // [G] candidate scales
    float *sinv = stab + G;                                       // [G] fl(1 / scale)
    float *sr = sinv + G;                                         // [d] residual
    __shared__ Reduce red;
    __shared__ float s_hinv[MPQ_QMAX_LIMIT + 1];   // 1 / (L - 1/2): threshold estimates only

    const int tid = threadIdx.x;
    const int k = blockIdx.x;
    const float qmaxf = (float)qmax;
    for (int L = tid; L <= qmax; L += QBLOCK) s_hinv[L] = 1.0f / ((float)L - 0.5f);
    const size_t plane = (size_t)C * d;
    const float *w = W + (size_t)k * d;

    int bad = 0;
    float part = 0.0f;
    float am = 0.0f;
    for (int j = tid; j < d; j += QBLOCK) {
        float v = w[j];
        sr[j] = v;
        bad |= !isfinite(v);
        part = fmaf(v, v, part);
        am = fmaxf(am, fabsf(v));
    }
    bad = __syncthreads_or(bad);
    float m = am;                 // max |r| of the current residual (exact)
    double r2 = (double)part;
    block_max_sum(m, r2, red);
    if (resid_sq && tid == 0) resid_sq[(size_t)k * (k_max + 1)] = bad ? NAN : (float)r2;

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

        float s_best = 0.0f, inv_best = 0.0f;
        if (m > 0.0f) {
            const float smax = __fdiv_rn(m, qmaxf);
            int e;
            frexpf(m, &e);                      // m < 2^e
            const int S = 62 - e - hbits;       // sum_j R_j c_j < 2^62
            const double down = ldexp(1.0, -S);
            int zero_scale = 0;
            for (int g = tid; g < G; g += QBLOCK) {
                const float s = __fmul_rn(grid.frac(g, G), smax);
                stab[g] = s;
                sinv[g] = (s > 0.0f) ? __frcp_rn(s) : 0.0f;
                zero_scale |= (s == 0.0f);
            }
            for (int t = tid; t <= G; t += QBLOCK) {
                hP[t] = 0;
                hN[t] = 0;
            }
            zero_scale = __syncthreads_or(zero_scale);

            double bestD = DBL_MAX;
            int bestg = INT_MAX;
            if (!zero_scale) {
                // ---- events: one per (element, level crossed inside the grid)
                const float s0 = stab[0], sG = stab[G - 1];
                const float i0 = sinv[0], iG = sinv[G - 1];
                const float g_per_a = __fdiv_rn((float)G, smax);   // default grid: s_g ~ (g+1)/G*smax
                unsigned int *hPw = reinterpret_cast<unsigned int *>(hP);   // [2*(G+1)] lo, hi
                long long Pb = 0;
                long long Nb = 0;
                for (int j = tid; j < d; j += QBLOCK) {
                    const float a = fabsf(sr[j]);
                    if (a == 0.0f) continue;
                    const int c_hi = code_fast(a, s0, i0, qmaxf);
                    if (c_hi == 0) continue;   // code 0 at every scale: no contribution
                    const int c_lo = code_fast(a, sG, iG, qmaxf);
                    const long long R = fixed_point(a, S);
                    Pb += R * (long long)c_lo;
                    Nb += (long long)c_lo * c_lo;
                    const unsigned int Rlo = (unsigned int)R;
                    const unsigned int Rhi = (unsigned int)((unsigned long long)R >> 32);
                    const float ag = a * g_per_a;
                    for (int L = c_lo + 1; L <= c_hi; ++L) {
                        // first g whose code is below L: estimate where s_g crosses a/(L - 1/2),
                        // then settle with the exact rule (level_held is monotone in g)
                        int T;
                        if (CUSTOM) {
                            const float s_est = a * s_hinv[L];
                            int lo = 1, hi = G - 1;
                            while (lo < hi) {
                                const int mid = (lo + hi) >> 1;
                                if (stab[mid] < s_est) lo = mid + 1; else hi = mid;
                            }
                            T = lo;
                        } else {
                            // s_g = (g+1)/G * smax up to two fp32 roundings and x is a*G/(smax*h)
                            // up to 2^-22, so unless x is within 2^-20 x of an integer, level L
                            // is held exactly for g + 1 < x: T = floor(x) with no further check.
                            const float x = ag * s_hinv[L];
                            const float fx = floorf(x);
                            const float tolx = MPQ_FAST_REL * x;
                            T = (int)fminf(fmaxf(fx, 1.0f), (float)(G - 1));
                            if (x - fx > tolx && fx + 1.0f - x > tolx && fx >= 1.0f &&
                                fx <= (float)(G - 1)) {
                                const unsigned int old = atomicAdd(&hPw[2 * T], Rlo);
                                const unsigned int carry = (old + Rlo < old) ? 1u : 0u;
                                if (Rhi + carry) atomicAdd(&hPw[2 * T + 1], Rhi + carry);
                                atomicAdd(&hN[T], 2 * L - 1);
                                continue;
                            }
                        }
                        const bool up = (T < G - 1) && level_held(a, stab[T], sinv[T], L);
                        const bool down = !up && (T > 1) && !level_held(a, stab[T - 1], sinv[T - 1], L);
                        if (up) {
                            ++T;
                            while (T < G - 1 && level_held(a, stab[T], sinv[T], L)) ++T;
                        } else if (down) {
                            --T;
                            while (T > 1 && !level_held(a, stab[T - 1], sinv[T - 1], L)) --T;
                        }
                        const unsigned int old = atomicAdd(&hPw[2 * T], Rlo);
                        const unsigned int carry = (old + Rlo < old) ? 1u : 0u;
                        if (Rhi + carry) atomicAdd(&hPw[2 * T + 1], Rhi + carry);
                        atomicAdd(&hN[T], 2 * L - 1);
                    }
                }
                const long long Pbase = block_sum_ll(Pb, red);
                const long long Nbase = block_sum_ll(Nb, red);   // also orders the bin updates
                // ---- suffix sums over the bins (warp 0), in place: bin t <- sum_{u >= t}, so
                // that P_g = Pbase + hP[g + 1].  Each lane owns bins (b0, b1].
                if (tid < 32) {
                    const int per = (G + 31) / 32;
                    const int b0 = min(G, tid * per), b1 = min(G, b0 + per);
                    long long sp = 0;
                    long long sn = 0;
                    for (int t = b0 + 1; t <= b1; ++t) {
                        sp += hP[t];
                        sn += hN[t];
                    }
                    // inclusive scan toward lower lanes: lane l gets the totals of lanes >= l
                    long long xp = sp, xn = sn;
#pragma unroll
                    for (int o = 1; o < 32; o <<= 1) {
                        const long long yp = __shfl_down_sync(0xffffffffu, xp, o);
                        const long long yn = __shfl_down_sync(0xffffffffu, xn, o);
                        if (tid + o < 32) {
                            xp += yp;
                            xn += yn;
                        }
                    }
                    long long rp = xp - sp, rn = xn - sn;   // bins beyond b1
                    for (int t = b1; t > b0; --t) {
                        rp += hP[t];
                        rn += hN[t];
                        hP[t] = rp;
                        hN[t] = (int)rn;
                    }
                }
                __syncthreads();
                for (int g = tid; g < G; g += QBLOCK) {
                    const double D = decision(stab[g], Pbase + hP[g + 1],
                                              Nbase + (long long)hN[g + 1], down);
                    if (D < bestD) {
                        bestD = D;
                        bestg = g;
                    }
                }
            } else {
                // ---- direct evaluation (a candidate scale underflowed to 0)
                for (int g = tid; g < G; g += QBLOCK) {
                    const float s = stab[g];
                    double D = 0.0;  // s == 0: all codes 0, E = ||r||^2
                    if (s > 0.0f) {
                        long long P = 0, N = 0;
                        for (int j = 0; j < d; ++j) {
                            const float a = fabsf(sr[j]);
                            const int c = code_mag(a, s, qmaxf);
                            P += fixed_point(a, S) * (long long)c;
                            N += (long long)c * c;
                        }
                        D = decision(s, P, N, down);
                    }
                    if (D < bestD) {
                        bestD = D;
                        bestg = g;
                    }
                }
            }
            int g = block_argmin(bestD, bestg, red);
            if (g < 0 || g >= G) g = G - 1;   // unreachable: every D is finite
            s_best = stab[g];
            inv_best = sinv[g];
        }

        // residual update (Eq. 7) and code emission; also the next step's max |r|
        part = 0.0f;
        am = 0.0f;
        for (int j = tid; j < d; j += QBLOCK) {
            float v = sr[j];
            int q = 0;
            if (s_best > 0.0f) {
                const int c = (inv_best > 0.0f) ? code_fast(fabsf(v), s_best, inv_best, qmaxf)
                                                : code_mag(fabsf(v), s_best, qmaxf);
                q = (v < 0.0f) ? -c : c;
                v = __fmaf_rn(-s_best, (float)q, v);
            }
            qi[j] = (int8_t)q;
            sr[j] = v;
            if (ri) ri[j] = v;
            part = fmaf(v, v, part);
            am = fmaxf(am, fabsf(v));
        }
        if (tid == 0) scales[(size_t)k * k_max + i] = s_best;
        m = am;
        r2 = (double)part;
        block_max_sum(m, r2, red);   // also orders the sr[] writes before the next step
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
    const size_t smem = (size_t)(G + 1) * (sizeof(long long) + sizeof(int)) +
                        (size_t)2 * G * sizeof(float) + (size_t)d * sizeof(float);
    if ((long long)smem > max_smem_optin()) {
        set_error("d = %d, G = %d need %zu bytes of shared memory", d, G, smem);
        return MPQ_ERR_UNSUPPORTED;
    }
    const int hbits = ceil_log2((long long)d * qmax) + 1;

    cudaError_t e;
    if (grid) {
        Grid<true> g;
        g.gf = *grid;
        e = cudaFuncSetAttribute(quantize_event_kernel<true>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e == cudaSuccess) {
            quantize_event_kernel<true><<<C, QBLOCK, smem, stream>>>(
                W, C, d, qmax, G, g, k_max, codes, scales, resid_sq, residuals, hbits);
            e = cudaGetLastError();
        }
    } else {
        e = cudaFuncSetAttribute(quantize_event_kernel<false>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e == cudaSuccess) {
            quantize_event_kernel<false><<<C, QBLOCK, smem, stream>>>(
                W, C, d, qmax, G, Grid<false>(), k_max, codes, scales, resid_sq, residuals, hbits);
            e = cudaGetLastError();
        }
    }
    return cuda_status(e, "quantize kernel launch");
}

}  // namespace mpq
