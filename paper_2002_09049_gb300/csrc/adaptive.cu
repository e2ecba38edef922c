// Algorithm 1 with the adaptive grid of Eq. 10 (Definition 1) for short channels.
//
// Step i of channel k: Delta = the minimal gap of r_i (Definition 1, pairs of distinct
// magnitudes), gamma = min(Delta / Qmax, eta) (eta when r_i has one distinct magnitude), and the
// grid search of a over I = [0, 2 Qmax ||r_i||] with step gamma: a_m = m gamma, m = 1..M,
// M = floor(2 Qmax ||r_i|| / gamma), each taken as the fp32 point scale s_m = fl(a_m / Qmax)
// (s q = a [r/a]_Q, Eq. 1).  Codes q = clamp(rint(fl(r / s)), -Qmax, Qmax) (Eq. 8), objective
// ||r - s q||^2 in double in index order (Eq. 9), the first minimiser, r <- fmaf(-s, q, r) (Eq. 7).
//
// The grid of a step is enumerated: one CTA per channel, its threads striding over m.  Every
// double operation of the objective, of ||r||^2 and of the grid arithmetic is written out
// (__dmul_rn, __dadd_rn, ...), so none is contracted into a fused multiply-add and each step takes
// the same decision as a plain sequential evaluation of the definition.  A step whose grid would
// exceed max_cand candidates is refused: its scale and every later one read NaN, codes 0, and
// ncand holds -1.  Short channels only (d <= 64): on longer ones the minimal gap makes grids of
// 1e8 candidates and more.
#include <climits>
#include <math.h>

#include "mpq_internal.cuh"

namespace mpq {
namespace {

constexpr int AD_THREADS = 256;

__device__ __forceinline__ int ad_code(float r, float s, int qmax)
{
    if (s == 0.0f) return 0;
    float t = rintf(__fdiv_rn(r, s));
    t = fminf(fmaxf(t, (float)(-qmax)), (float)qmax);
    return (int)t;
}

__device__ __forceinline__ float ad_scale(long long m, double gamma, int qmax)
{
    return __double2float_rn(__ddiv_rn(__dmul_rn((double)m, gamma), (double)qmax));
}

__global__ void __launch_bounds__(AD_THREADS)
adaptive_kernel(const float *__restrict__ W, int C, int d, int qmax, int k_max, double eta,
                long long max_cand, int8_t *__restrict__ codes, float *__restrict__ scales,
                float *__restrict__ resid_sq, long long *__restrict__ ncand)
{
    __shared__ float r[MPQ_ADAPTIVE_MAX_DIM];
    __shared__ double mag[MPQ_ADAPTIVE_MAX_DIM];
    __shared__ double s_r2, s_gamma;
    __shared__ long long s_M;
    __shared__ int s_state;                       // 0 search, 1 null point, 2 refused or non-finite
    __shared__ double red_E[AD_THREADS / 32];
    __shared__ long long red_m[AD_THREADS / 32];
    __shared__ long long s_best;

    const int k = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const size_t plane = (size_t)C * d;
    for (int j = tid; j < d; j += AD_THREADS) r[j] = W[(size_t)k * d + j];
    __syncthreads();
    int dead = 0;                                  // refused or non-finite: NaN from here on
    if (tid == 0) {
        double r2 = 0.0;
        int finite = 1;
        for (int j = 0; j < d; ++j) {
            finite &= isfinite(r[j]);
            r2 = __dadd_rn(r2, __dmul_rn((double)r[j], (double)r[j]));
        }
        s_r2 = r2;
        s_M = 0;
        s_state = finite ? 0 : 2;
        if (resid_sq) resid_sq[(size_t)k * (k_max + 1)] = finite ? (float)r2 : NAN;
    }
    __syncthreads();
    dead = (s_state == 2);

    for (int i = 0; i < k_max; ++i) {
        int8_t *qi = codes + (size_t)i * plane + (size_t)k * d;
        if (!dead && tid == 0) {
            const double r2 = s_r2;
            if (r2 == 0.0) {
                s_state = 1;
                s_M = 0;
                s_gamma = 0.0;
            } else {
                // Definition 1: sorted magnitudes (insertion sort, d <= 64), distinct neighbours
                for (int j = 0; j < d; ++j) {
                    const double v = fabs((double)r[j]);
                    int p = j;
                    while (p > 0 && mag[p - 1] > v) {
                        mag[p] = mag[p - 1];
                        --p;
                    }
                    mag[p] = v;
                }
                double delta = INFINITY;
                for (int j = 1; j < d; ++j)
                    if (mag[j] != mag[j - 1]) {
                        const double x = __ddiv_rn(__dsub_rn(mag[j], mag[j - 1]), 2.0);
                        if (x < delta) delta = x;
                    }
                double g = __ddiv_rn(delta, (double)qmax);
                if (!(g < eta)) g = eta;
                const double top = __dmul_rn(__dmul_rn(2.0, (double)qmax), __dsqrt_rn(r2));
                const double mf = floor(__ddiv_rn(top, g));
                s_gamma = g;
                if (mf > (double)max_cand) {
                    s_state = 2;
                    s_M = -1;
                } else {
                    s_state = 0;
                    s_M = (long long)mf;
                }
            }
        }
        __syncthreads();
        if (!dead && s_state == 2) dead = 1;   // refused at this step
        if (dead) {
            for (int j = tid; j < d; j += AD_THREADS) qi[j] = 0;
            if (tid == 0) {
                scales[(size_t)k * k_max + i] = NAN;
                if (ncand) ncand[(size_t)k * k_max + i] = (s_M < 0) ? -1 : 0;
                if (resid_sq) resid_sq[(size_t)k * (k_max + 1) + i + 1] = NAN;
                s_M = 0;   // later steps of a dead channel report 0 candidates
            }
            __syncthreads();
            continue;
        }
        float sbest = 0.0f;   // a null point, or a grid without candidates: scale 0, codes 0
        if (s_state == 0 && s_M > 0) {
            const long long M = s_M;
            const double g = s_gamma;
            double bE = INFINITY;
            long long bm = LLONG_MAX;
            for (long long m = tid + 1; m <= M; m += AD_THREADS) {   // increasing m: strict <
                const float s = ad_scale(m, g, qmax);
                double E = 0.0;
                for (int j = 0; j < d; ++j) {
                    const int q = ad_code(r[j], s, qmax);
                    const double e = __dsub_rn((double)r[j], __dmul_rn((double)s, (double)q));
                    E = __dadd_rn(E, __dmul_rn(e, e));
                }
                if (E < bE) {
                    bE = E;
                    bm = m;
                }
            }
            // first minimiser: smallest E, then smallest m
            for (int o = 16; o > 0; o >>= 1) {
                const double oE = __shfl_down_sync(0xffffffffu, bE, o);
                const long long om = __shfl_down_sync(0xffffffffu, bm, o);
                if (oE < bE || (oE == bE && om < bm)) {
                    bE = oE;
                    bm = om;
                }
            }
            if (lane == 0) {
                red_E[warp] = bE;
                red_m[warp] = bm;
            }
            __syncthreads();
            if (tid == 0) {
                double E1 = red_E[0];
                long long m1 = red_m[0];
                for (int w = 1; w < AD_THREADS / 32; ++w)
                    if (red_E[w] < E1 || (red_E[w] == E1 && red_m[w] < m1)) {
                        E1 = red_E[w];
                        m1 = red_m[w];
                    }
                s_best = m1;
            }
            __syncthreads();
            sbest = ad_scale(s_best, g, qmax);
        }
        // update (a null point leaves codes 0 and r unchanged)
        for (int j = tid; j < d; j += AD_THREADS) {
            const int q = ad_code(r[j], sbest, qmax);
            qi[j] = (int8_t)q;
            r[j] = __fmaf_rn(-sbest, (float)q, r[j]);
        }
        __syncthreads();
        if (tid == 0) {
            scales[(size_t)k * k_max + i] = sbest;
            if (ncand) ncand[(size_t)k * k_max + i] = s_M;
            double r2 = 0.0;
            for (int j = 0; j < d; ++j) r2 = __dadd_rn(r2, __dmul_rn((double)r[j], (double)r[j]));
            s_r2 = r2;
            if (resid_sq) resid_sq[(size_t)k * (k_max + 1) + i + 1] = (float)r2;
        }
        __syncthreads();
    }
}

}  // namespace

mpq_status launch_adaptive(const float *W, int C, int d, int qmax, int k_max, double eta,
                           long long max_cand, int8_t *codes, float *scales, float *resid_sq,
                           long long *ncand, cudaStream_t stream)
{
    adaptive_kernel<<<C, AD_THREADS, 0, stream>>>(W, C, d, qmax, k_max, eta, max_cand, codes,
                                                  scales, resid_sq, ncand);
    return cuda_status(cudaGetLastError(), "adaptive-grid kernel launch");
}

}  // namespace mpq
