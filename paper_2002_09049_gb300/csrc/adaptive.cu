// Algorithm 1 with the adaptive grid of Eq. 10 (Definition 1), for channels of any length.
//
// Step i of channel k: Delta = the minimal gap of r_i (Definition 1, pairs of distinct
// magnitudes), gamma = min(Delta / Qmax, eta) (eta when r_i has one distinct magnitude), and the
// grid search of a over I = [0, 2 Qmax ||r_i||] with step gamma: a_m = m gamma, m = 1..M,
// M = floor(2 Qmax ||r_i|| / gamma), each taken as the fp32 point scale s_m = fl(a_m / Qmax)
// (s q = a [r/a]_Q, Eq. 1).  Codes q = clamp(rint(fl(r / s)), -Qmax, Qmax) (Eq. 8), the objective
// ||r - s q||^2 (Eq. 9), its first minimiser over m, r <- fmaf(-s, q, r) (Eq. 7).
//
// The grid is not enumerated (Definition 1 makes it 1e8..1e10 points long on real channels).
// Every element's code magnitude is a non-increasing step function of the scale, so for each
// element a = |r_j| and level L the set of fp32 scales where the code is at least L is
// {s <= tau_{j,L}}, with tau the largest such fp32 value (found with the correctly rounded
// division itself).  Sorted, the thresholds cut the scale axis into pieces with constant codes,
// on which the objective is the quadratic R2 - 2 s P + s^2 N (P = sum a_j c_j exact in 64-bit
// fixed point, N = sum c_j^2 exact).  An fp32 screen bounds every piece's minimum from below; the
// pieces whose bound can reach the best exact value are settled in double at their grid points
// next to the quadratic's minimiser (grid indices found by bisection on the exact s_m).  Equal
// values go to the smaller scale, i.e. the first m.  The decision is the exact minimiser of the
// objective; the oracle's double sum of squares differs from it only by rounding, so the two can
// differ only at a near tie.
//
// ||r||^2 (for M and the squared-norm output) is summed in double in index order by one thread,
// exactly as the definition, and Delta from the sorted magnitudes: the grid sizes are bit-exact.
// One CTA per channel at a time (persistent over the layer), the threshold lists in global
// scratch from the stream-ordered pool, sorted by a CTA radix sort.
#include <float.h>
#include <limits.h>
#include <math.h>

#include <algorithm>

#include "mpq_internal.cuh"

MPQ_CHECKED_UNIT("adaptive.cu");

namespace mpq {
namespace {

constexpr int AW = 16;                 // warps per CTA
constexpr int AT = AW * 32;
constexpr int A_CTAS_PER_SM = 2;
constexpr int A_MAX_EVENTS = 1 << 16;  // d * Qmax (the thresholds of one step)

// ---- the definition's scalar arithmetic -------------------------------------------------------
__device__ __forceinline__ int ad_code_mag(float a, float s, int qmax)
{
    if (s == 0.0f) return 0;
    return (int)fminf(rintf(__fdiv_rn(a, s)), (float)qmax);
}

// the grid's point scale s_m = fl32(fl64(m gamma) / Qmax), each operation rounded once
__device__ __forceinline__ float ad_scale(long long m, double gamma, int qmax)
{
    return __double2float_rn(__ddiv_rn(__dmul_rn((double)m, gamma), (double)qmax));
}

// code magnitude >= L (1 <= L <= Qmax) at scale s: rint(fl(a/s)) >= L
__device__ __forceinline__ bool ad_held(float a, float s, int L)
{
    return s > 0.0f && rintf(__fdiv_rn(a, s)) >= (float)L;
}

// tau_{a,L}: the largest fp32 scale with code >= L, 0 if no positive scale has it.  fl(a/s) is
// non-increasing in s, so the set is a prefix of the positive floats; the start a / (L - 1/2) is
// within a few ulps of its end.  Each loop is bounded (64 steps; the start is never that far off).
__device__ __forceinline__ float ad_threshold(float a, int L)
{
    float s = __fdiv_rn(a, (float)L - 0.5f);
    if (!(s < FLT_MAX)) s = FLT_MAX;
    if (ad_held(a, s, L)) {
        for (int it = 0; it < 64 && s < FLT_MAX; ++it) {
            const float u = nextafterf(s, FLT_MAX);
            if (!ad_held(a, u, L)) break;
            s = u;
        }
        return s;
    }
    for (int it = 0; it < 64; ++it) {
        s = nextafterf(s, 0.0f);
        if (s == 0.0f || ad_held(a, s, L)) return s;
    }
    return s;
}

// Smallest m in [lo, M] with s_m >= f (an fp32 value); M + 1 if none.  s_m = fl32(y_m) is
// non-decreasing in m and reaches f once y_m passes the midpoint between f's predecessor and f,
// which y_m = m gamma / Qmax (1 + O(2^-52)) crosses within a couple of indices of
// midpoint * Qmax / gamma: the answer is bracketed there by two exact s_m and bisected (about
// five exact scales in all); a failed bracket falls back to bisecting [lo, M].
__device__ long long ad_first_m_ge(float f, long long lo, long long M, double gamma, int qmax)
{
    auto ok = [&](long long m) { return ad_scale(m, gamma, qmax) >= f; };
    if (lo > M) return M + 1;
    if (ok(lo)) return lo;
    if (!ok(M)) return M + 1;
    long long a = lo, b = M;   // ok(a) false, ok(b) true
    const double h = 0.5 * ((double)nextafterf(f, 0.0f) + (double)f);   // exact
    const double est = __dmul_rn(h, __ddiv_rn((double)qmax, gamma));
    if (est > (double)lo && est < (double)M) {
        const long long c = (long long)est;
        const long long a2 = c - 2 > lo ? c - 2 : lo;
        const long long b2 = c + 3 < M ? c + 3 : M;
        if (!ok(a2) && ok(b2)) {
            a = a2;
            b = b2;
        }
    }
    for (int it = 0; it < 80 && b - a > 1; ++it) {
        const long long mid = a + (b - a) / 2;
        if (ok(mid)) b = mid; else a = mid;
    }
    return b;
}

// the smallest fp32 value >= x, and the one after the fp32 value x
__device__ __forceinline__ float ad_ceil_f(double x)
{
    float f = __double2float_rn(x);
    if ((double)f < x) f = nextafterf(f, INFINITY);
    return f;
}
__device__ __forceinline__ float ad_next_f(float x) { return nextafterf(x, INFINITY); }

// ---- CTA-wide building blocks (all AT threads call them) -------------------------------------
struct ASort {
    unsigned hist[AW][256];   // per-warp digit counts, then scatter offsets
    unsigned wsum[AW];
    unsigned keys_or, keys_and;
};

// exclusive prefix over the 256 digit totals (threads 0..255 each hold one), through wsum
__device__ __forceinline__ unsigned ad_scan256(unsigned v, ASort &st)
{
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    unsigned x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (t < 256 && lane == 31) st.wsum[w] = x;
    __syncthreads();
    unsigned base = 0;
    if (t < 256)
        for (int i = 0; i < w; ++i) base += st.wsum[i];
    __syncthreads();
    return base + x - v;
}

// Sorts n (key, val) pairs ascending by key: stable LSD radix sort, 8-bit digits, ping-pong between
// a and b; digits on which every key agrees are skipped.  Each warp owns a contiguous segment and
// ranks equal digits inside a 32-element tile with __match_any_sync, so the order is stable.
// Returns the buffer that holds the result.
__device__ uint2 *ad_sort(uint2 *a, uint2 *b, int n, ASort &st)
{
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    if (t == 0) {
        st.keys_or = 0u;
        st.keys_and = 0xffffffffu;
    }
    __syncthreads();
    unsigned o = 0u, an = 0xffffffffu;
    for (int i = t; i < n; i += AT) {
        const unsigned k = a[i].x;
        o |= k;
        an &= k;
    }
    atomicOr(&st.keys_or, o);
    atomicAnd(&st.keys_and, an);
    __syncthreads();
    const unsigned diff = st.keys_or ^ st.keys_and;
    const int seg = ((n + AW - 1) / AW + 31) / 32 * 32;
    const int w0 = min(n, w * seg), w1 = min(n, w * seg + seg);
    const unsigned lt = (1u << lane) - 1u;
    for (int shift = 0; shift < 32; shift += 8) {
        if (((diff >> shift) & 255u) == 0u) continue;   // uniform across the CTA
        for (int i = t; i < AW * 256; i += AT) (&st.hist[0][0])[i] = 0u;
        __syncthreads();
        for (int t0 = w0; t0 < w1; t0 += 32) {
            const int i = t0 + lane;
            const unsigned dg = i < w1 ? (a[i].x >> shift) & 255u : 256u;
            const unsigned m = __match_any_sync(0xffffffffu, dg);
            if (dg < 256u && (m & lt) == 0u) st.hist[w][dg] += __popc(m);
            __syncwarp();
        }
        __syncthreads();
        unsigned tot = 0;
        if (t < 256)
            for (int ww = 0; ww < AW; ++ww) tot += st.hist[ww][t];
        const unsigned base = ad_scan256(tot, st);
        if (t < 256) {
            unsigned run = base;
            for (int ww = 0; ww < AW; ++ww) {
                const unsigned c = st.hist[ww][t];
                st.hist[ww][t] = run;
                run += c;
            }
        }
        __syncthreads();
        for (int t0 = w0; t0 < w1; t0 += 32) {
            const int i = t0 + lane;
            uint2 e = make_uint2(0u, 0u);
            if (i < w1) e = a[i];
            const unsigned dg = i < w1 ? (e.x >> shift) & 255u : 256u;
            const unsigned m = __match_any_sync(0xffffffffu, dg);
            if (dg < 256u && MPQ_IN(st.hist[w][dg] + __popc(m & lt), n))
                b[st.hist[w][dg] + __popc(m & lt)] = e;
            __syncwarp();
            if (dg < 256u && (m & lt) == 0u) st.hist[w][dg] += __popc(m);
            __syncwarp();
        }
        __syncthreads();
        uint2 *x = a;
        a = b;
        b = x;
    }
    return a;
}

// Order-preserving image of a double (total order on non-NaN values).
__device__ __forceinline__ unsigned long long ad_ordered(double x)
{
    const unsigned long long v = (unsigned long long)__double_as_longlong(x);
    return (v >> 63) ? ~v : (v | 0x8000000000000000ull);
}

__device__ __forceinline__ unsigned ad_ordered_f(float x)
{
    const unsigned v = __float_as_uint(x);
    return (v >> 31) ? ~v : (v | 0x80000000u);
}


// |r| as a 64-bit fixed-point integer a * 2^S from its fp32 bits (exact whenever a * 2^S is an
// integer: for every element that can take a nonzero code; smaller ones truncate, and their code
// is 0 at every positive grid scale on which P is used).
__device__ __forceinline__ long long ad_fixed(float a, int S)
{
    const uint32_t bits = __float_as_uint(a);
    const int E = (int)(bits >> 23);
    const long long Mt = (long long)((bits & 0x7FFFFFu) | (E ? 0x800000u : 0u));
    const int sh = (E ? E : 1) - 150 + S;
    if (sh >= 0) return Mt << sh;
    return sh > -40 ? (Mt >> -sh) : 0;
}

// Decision value D(s) = s (s N - 2 P) = ||r - s q||^2 - ||r||^2, P = Pfix 2^-S, in double.
__device__ __forceinline__ double ad_decision(float s, long long Pfix, long long N, double down)
{
    const double sd = (double)s;
    return __dmul_rn(sd, __fma_rn(sd, (double)N, -2.0 * ((double)Pfix * down)));
}

constexpr int A_LIST = 512;   // candidate pieces settled by the whole CTA

struct APiece {
    float lo, hi;
    long long P, N;
};

struct AShared {
    ASort sort;
    APiece list[A_LIST];
    int nlist;
    int finite;
    double r2;                  // ||r||^2, double, index order
    double gamma;
    long long M, mpos;
    unsigned long long gap;     // Definition 1: bits of the smallest half-gap (non-negative double)
    unsigned long long lbkey;   // (ordered fp32 lower bound, piece) of the best piece
    unsigned long long dkey;    // ordered D of the best settled grid point
    unsigned skey;              // its scale's bits, among equal D
    double U;                   // best exact D of the first settled piece
    unsigned amax;              // max |r| as bits
    int state;                  // 0 search, 1 scale 0 (null point or no positive grid scale), 2 dead
    int nev;
    float spos, slast, sbest;
    long long part[AW][2];
};

// The (P, N) prefix of this thread's block of sorted events, by a block exclusive scan.
__device__ __forceinline__ void ad_block_prefix(long long &p, long long &n, AShared &sh)
{
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    long long xp = p, xn = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long yp = __shfl_up_sync(0xffffffffu, xp, o);
        const long long yn = __shfl_up_sync(0xffffffffu, xn, o);
        if (lane >= o) {
            xp += yp;
            xn += yn;
        }
    }
    if (lane == 31) {
        sh.part[w][0] = xp;
        sh.part[w][1] = xn;
    }
    __syncthreads();
    long long bp = 0, bn = 0;
    for (int i = 0; i < w; ++i) {
        bp += sh.part[i][0];
        bn += sh.part[i][1];
    }
    __syncthreads();
    p = bp + xp - p;
    n = bn + xn - n;
}

// The smallest objective over the grid points of one piece (lo, hi] with constant (P, N): the
// grid points on either side of the quadratic's minimiser P / N, clipped to the piece.  Returns
// false when no grid point falls inside.
__device__ bool ad_settle_piece(float lo, float hi, long long Pfix, long long N, double down,
                                double gamma, int qmax, long long mpos, long long M, double &D,
                                float &s)
{
    const long long m1 = ad_first_m_ge(ad_next_f(lo), mpos, M, gamma, qmax);
    if (m1 > M) return false;
    const long long m2 = ad_first_m_ge(ad_next_f(hi), m1, M, gamma, qmax) - 1;
    if (m1 > m2) return false;
    if (N == 0) {   // every code 0: D = 0 on the whole piece, its smallest scale first
        D = 0.0;
        s = ad_scale(m1, gamma, qmax);
        return true;
    }
    const double sbar = __ddiv_rn((double)Pfix * down, (double)N);
    long long mb = ad_first_m_ge(ad_ceil_f(sbar), m1, m2, gamma, qmax);
    if (mb > m2) mb = m2;
    const long long ma = mb > m1 ? mb - 1 : m1;
    const float sa = ad_scale(ma, gamma, qmax), sb = ad_scale(mb, gamma, qmax);
    const double Da = ad_decision(sa, Pfix, N, down), Db = ad_decision(sb, Pfix, N, down);
    if (Db < Da) {
        D = Db;
        s = sb;
    } else {
        D = Da;
        s = sa;
    }
    return true;
}

// fp32 lower bound of D' = D 2^-2e over the scales [lo, hi] of a piece (continuous, so it also
// bounds the piece's grid points), with a margin for the fp32 roundings (at most ~8 of 2^-24).
__device__ __forceinline__ float ad_piece_lb(float lo, float hi, float Pn, float N, int e)
{
    if (N == 0.0f) return 0.0f;
    const float l = ldexpf(lo, -e), h = ldexpf(hi, -e);
    const float sb = __fdiv_rn(Pn, N);
    constexpr float REL = 9.5367431640625e-07f;   // 2^-20
    if (sb >= l * (1.0f - REL) && sb <= h * (1.0f + REL)) return -(Pn * sb) * (1.0f + REL);
    const float dl = l * (l * N - 2.0f * Pn) - REL * l * (l * N + 2.0f * Pn);
    const float dh = h * (h * N - 2.0f * Pn) - REL * h * (h * N + 2.0f * Pn);
    return fminf(dl, dh);
}


// sum_j x_j in double, in index order, one rounding per addition (the definition's ||r||^2 once
// the exact squares are in x); the loads run ahead of the dependent additions
__device__ __forceinline__ double ad_serial_sum(const double *__restrict__ x, int d)
{
    double s = 0.0;
    int j = 0;
    for (; j + 8 <= d; j += 8) {
        double v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = x[j + u];
#pragma unroll
        for (int u = 0; u < 8; ++u) s = __dadd_rn(s, v[u]);
    }
    for (; j < d; ++j) s = __dadd_rn(s, x[j]);
    return s;
}

__global__ void __launch_bounds__(AT, A_CTAS_PER_SM)
adaptive_kernel(const float *__restrict__ W, int C, int d, int qmax, int k_max, double eta,
                long long max_cand, int hbits, int8_t *__restrict__ codes,
                float *__restrict__ scales, float *__restrict__ resid_sq,
                long long *__restrict__ ncand, uint2 *__restrict__ scratch, int cap)
{
    extern __shared__ __align__(16) float r[];   // the residual row, d floats
    __shared__ AShared sh;
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    uint2 *bufA = scratch + (size_t)blockIdx.x * 2 * cap;
    uint2 *bufB = bufA + cap;
    double *sq = reinterpret_cast<double *>(bufB);   // r_j^2 for the serial sum (cap >= d)
    const size_t plane = (size_t)C * d;
    const size_t n_codes = (size_t)k_max * plane, n_sc = (size_t)C * k_max;
    const size_t n_rs = (size_t)C * (k_max + 1);
    if (!MPQ_CHECK_SMEM_END(4 * (size_t)d) || !MPQ_CHECK(d <= cap)) return;

    for (int k = blockIdx.x; k < C; k += gridDim.x) {
        if (t == 0) sh.finite = 1;
        __syncthreads();
        int fin = 1;
        for (int j = t; j < d; j += AT) {
            const float v = MPQ_IN((size_t)k * d + j, plane) ? W[(size_t)k * d + j] : 0.0f;
            r[j] = v;
            sq[j] = __dmul_rn((double)v, (double)v);   // exact: 24-bit times 24-bit
            fin &= isfinite(v);
        }
        if (!fin) atomicAnd(&sh.finite, 0);
        __syncthreads();
        if (t == 0) {
            const double r2 = ad_serial_sum(sq, d);
            sh.r2 = r2;
            sh.state = sh.finite ? 0 : 2;
            if (resid_sq && MPQ_IN((size_t)k * (k_max + 1), n_rs))
                resid_sq[(size_t)k * (k_max + 1)] = sh.finite ? (float)r2 : NAN;
        }
        __syncthreads();
        bool dead = sh.state == 2;
        for (int i = 0; i < k_max; ++i) {
            int8_t *qi = codes + (size_t)i * plane + (size_t)k * d;
            bool refused_now = false;
            if (!dead) {
                // ---- Definition 1: the sorted magnitudes' smallest half-gap; max |r|
                if (t == 0) {
                    sh.gap = 0x7FF0000000000000ull;   // +inf
                    sh.amax = 0u;
                    sh.nev = 0;
                    sh.lbkey = ~0ull;
                    sh.dkey = ~0ull;
                    sh.skey = ~0u;
                    sh.nlist = 0;
                }
                __syncthreads();
                unsigned am = 0u;
                for (int j = t; j < d; j += AT) {
                    const unsigned b = __float_as_uint(fabsf(r[j]));
                    bufA[j] = make_uint2(b, 0u);
                    am = max(am, b);
                }
                atomicMax(&sh.amax, am);
                __syncthreads();
                const uint2 *mag = ad_sort(bufA, bufB, d, sh.sort);
                unsigned long long gl = 0x7FF0000000000000ull;
                for (int j = t + 1; j < d; j += AT) {
                    const unsigned a0 = mag[j - 1].x, a1 = mag[j].x;
                    if (a0 != a1) {
                        const double x = __ddiv_rn(__dsub_rn((double)__uint_as_float(a1),
                                                             (double)__uint_as_float(a0)), 2.0);
                        gl = min(gl, (unsigned long long)__double_as_longlong(x));
                    }
                }
                atomicMin(&sh.gap, gl);
                __syncthreads();
                // ---- the grid of Eq. 10
                if (t == 0) {
                    const double r2 = sh.r2;
                    sh.M = 0;
                    if (r2 == 0.0) {
                        sh.state = 1;   // null point
                    } else {
                        double g = __ddiv_rn(__longlong_as_double((long long)sh.gap), (double)qmax);
                        if (!(g < eta)) g = eta;
                        const double top = __dmul_rn(__dmul_rn(2.0, (double)qmax), __dsqrt_rn(r2));
                        const double mf = floor(__ddiv_rn(top, g));
                        sh.gamma = g;
                        if (mf > (double)max_cand) {
                            sh.state = 2;
                            sh.M = -1;
                        } else {
                            const long long M = (long long)mf;
                            sh.M = M;
                            sh.state = 1;
                            if (M > 0) {
                                const long long mp = ad_first_m_ge(ad_next_f(0.0f), 1, M, g, qmax);
                                sh.mpos = mp;
                                sh.U = mp > 1 ? 0.0 : INFINITY;
                                if (mp <= M) {
                                    sh.state = 0;
                                    sh.spos = ad_scale(mp, g, qmax);
                                    sh.slast = ad_scale(M, g, qmax);
                                }
                            }
                        }
                    }
                }
                __syncthreads();
                if (sh.state == 2) {
                    dead = true;
                    refused_now = true;
                }
            }
            if (dead) {
                for (int j = t; j < d; j += AT)
                    if (MPQ_IN((size_t)i * plane + (size_t)k * d + j, n_codes)) qi[j] = 0;
                if (t == 0 && MPQ_IN((size_t)k * k_max + i, n_sc) &&
                    MPQ_IN((size_t)k * (k_max + 1) + i + 1, n_rs)) {
                    scales[(size_t)k * k_max + i] = NAN;
                    if (ncand) ncand[(size_t)k * k_max + i] = refused_now ? -1 : 0;
                    if (resid_sq) resid_sq[(size_t)k * (k_max + 1) + i + 1] = NAN;
                }
                __syncthreads();
                continue;
            }
            float sbest = 0.0f;   // null point, no grid point, or only scale-0 grid points
            if (sh.state == 0) {
                const double gamma = sh.gamma;
                const long long M = sh.M, mpos = sh.mpos;
                const float spos = sh.spos, slast = sh.slast;
                int e;
                frexpf(__uint_as_float(sh.amax), &e);   // max |r| < 2^e
                const int S = 62 - e - hbits;           // sum_j R_j c_j < 2^62
                const double down = __longlong_as_double((long long)(1023 - S) << 52);
                const float pscale = ldexpf(1.0f, hbits - 62);   // P 2^-S / 2^e
                // ---- thresholds tau_{j,L} >= spos: where code L of element j ends
                long long p0 = 0, n0 = 0;
                for (int j = t; j < d; j += AT) {
                    const float a = fabsf(r[j]);
                    if (a == 0.0f) continue;
                    const long long R = ad_fixed(a, S);
                    for (int L = 1; L <= qmax; ++L) {
                        const float tau = ad_threshold(a, L);
                        if (!(tau >= spos)) break;   // tau is non-increasing in L
                        const int pos = atomicAdd(&sh.nev, 1);
                        if (MPQ_IN(pos, cap))
                            bufA[pos] = make_uint2(__float_as_uint(tau),
                                                   ((unsigned)j << 8) | (unsigned)L);
                        p0 += R;
                        n0 += 2 * L - 1;
                    }
                }
                // totals: P and N at spos (every kept threshold is a level held there)
                long long P0 = p0, N0 = n0;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    P0 += __shfl_xor_sync(0xffffffffu, P0, o);
                    N0 += __shfl_xor_sync(0xffffffffu, N0, o);
                }
                if (lane == 0) {
                    sh.part[w][0] = P0;
                    sh.part[w][1] = N0;
                }
                __syncthreads();
                P0 = 0;
                N0 = 0;
                for (int x = 0; x < AW; ++x) {
                    P0 += sh.part[x][0];
                    N0 += sh.part[x][1];
                }
                __syncthreads();
                int n = sh.nev;
                if (!MPQ_CHECK(n <= cap)) n = cap;
                const uint2 *ev = ad_sort(bufA, bufB, n, sh.sort);
                // ---- pieces e = 0..n: scales (lo, hi] with the first e thresholds passed
                const int chunk = (n + 1 + AT - 1) / AT;
                const int e0 = min(n + 1, t * chunk), e1 = min(n + 1, e0 + chunk);
                long long pre_p = 0, pre_n = 0;
                for (int x = e0; x < min(e1, n); ++x) {
                    const unsigned v = ev[x].y;
                    if (!MPQ_IN(v >> 8, d)) continue;
                    pre_p += ad_fixed(fabsf(r[v >> 8]), S);
                    pre_n += 2 * (int)(v & 255u) - 1;
                }
                ad_block_prefix(pre_p, pre_n, sh);   // the thresholds before e0
                auto piece = [&](int x, float &lo, float &hi) -> bool {
                    lo = x == 0 ? nextafterf(spos, 0.0f) : __uint_as_float(ev[x - 1].x);
                    hi = x == n ? slast : fminf(__uint_as_float(ev[x].x), slast);
                    return lo < hi;
                };
                auto advance = [&](int x, long long &cp, long long &cn) {
                    if (x < n) {
                        const unsigned v = ev[x].y;
                        if (!MPQ_IN(v >> 8, d)) return;
                        cp += ad_fixed(fabsf(r[v >> 8]), S);
                        cn += 2 * (int)(v & 255u) - 1;
                    }
                };
                // screen: every piece's fp32 lower bound; the smallest one's piece is settled first
                unsigned long long mykey = ~0ull;
                long long bP = 0, bN = 0;
                float blo = 0.0f, bhi = 0.0f;
                {
                    long long cp = pre_p, cn = pre_n;
                    for (int x = e0; x < e1; ++x) {
                        float lo, hi;
                        if (piece(x, lo, hi)) {
                            const long long P = P0 - cp, N = N0 - cn;
                            const float lb = ad_piece_lb(lo, hi, (float)P * pscale, (float)N, e);
                            const unsigned long long key =
                                ((unsigned long long)ad_ordered_f(lb) << 32) | (unsigned)x;
                            if (key < mykey) {
                                mykey = key;
                                bP = P;
                                bN = N;
                                blo = lo;
                                bhi = hi;
                            }
                        }
                        advance(x, cp, cn);
                    }
                }
                atomicMin(&sh.lbkey, mykey);
                __syncthreads();
                if (mykey != ~0ull && mykey == sh.lbkey) {
                    double D;
                    float sv;
                    if (ad_settle_piece(blo, bhi, bP, bN, down, gamma, qmax, mpos, M, D, sv))
                        sh.U = fmin(sh.U, D);
                }
                __syncthreads();
                // pieces whose lower bound can reach the best settled value: settle them all
                const double U = sh.U;
                float Uf = INFINITY;
                if (U < INFINITY) {
                    const float u = (float)ldexp(U, -2 * e);
                    Uf = nextafterf(u, INFINITY) + fabsf(u) * 2.384185791015625e-07f;   // 2^-22
                }
                double bD = INFINITY;
                float bS = 0.0f;
                bool have = false;
                if (t == 0 && mpos > 1) {   // grid points of scale 0: every code 0, D = 0
                    bD = 0.0;
                    have = true;
                }
                {
                    long long cp = pre_p, cn = pre_n;
                    for (int x = e0; x < e1; ++x) {
                        float lo, hi;
                        if (piece(x, lo, hi)) {
                            const long long P = P0 - cp, N = N0 - cn;
                            const float lb = ad_piece_lb(lo, hi, (float)P * pscale, (float)N, e);
                            double D;
                            float sv;
                            if (lb <= Uf) {
                                const int slot = atomicAdd(&sh.nlist, 1);
                                if (slot < A_LIST) {
                                    sh.list[slot] = APiece{lo, hi, P, N};
                                } else if (ad_settle_piece(lo, hi, P, N, down, gamma, qmax, mpos, M,
                                                           D, sv) &&
                                           (!have || D < bD || (D == bD && sv < bS))) {
                                    bD = D;   // beyond the list: settled by its own thread
                                    bS = sv;
                                    have = true;
                                }
                            }
                        }
                        advance(x, cp, cn);
                    }
                }
                __syncthreads();
                // the queued pieces, spread over the CTA (neighbouring pieces share a thread above)
                for (int x = t; x < min(sh.nlist, A_LIST); x += AT) {
                    const APiece pc = sh.list[x];
                    double D;
                    float sv;
                    if (ad_settle_piece(pc.lo, pc.hi, pc.P, pc.N, down, gamma, qmax, mpos, M, D, sv) &&
                        (!have || D < bD || (D == bD && sv < bS))) {
                        bD = D;
                        bS = sv;
                        have = true;
                    }
                }
                const unsigned long long dk = have ? ad_ordered(bD) : ~0ull;
                atomicMin(&sh.dkey, dk);
                __syncthreads();
                if (have && dk == sh.dkey) atomicMin(&sh.skey, __float_as_uint(bS));
                __syncthreads();
                sbest = sh.skey != ~0u ? __uint_as_float(sh.skey) : spos;
            }
            // update (Eq. 7): codes at the chosen scale, r <- fmaf(-s, q, r)
            for (int j = t; j < d; j += AT) {
                const float v = r[j];
                int q = ad_code_mag(fabsf(v), sbest, qmax);
                q = v < 0.0f ? -q : q;
                if (MPQ_IN((size_t)i * plane + (size_t)k * d + j, n_codes)) qi[j] = (int8_t)q;
                const float nv = __fmaf_rn(-sbest, (float)q, v);
                r[j] = nv;
                sq[j] = __dmul_rn((double)nv, (double)nv);
            }
            __syncthreads();
            if (t == 0) {
                if (MPQ_IN((size_t)k * k_max + i, n_sc)) {
                    scales[(size_t)k * k_max + i] = sbest;
                    if (ncand) ncand[(size_t)k * k_max + i] = sh.M;
                }
                const double r2 = ad_serial_sum(sq, d);
                sh.r2 = r2;
                if (resid_sq && MPQ_IN((size_t)k * (k_max + 1) + i + 1, n_rs))
                    resid_sq[(size_t)k * (k_max + 1) + i + 1] = (float)r2;
            }
            __syncthreads();
        }
    }
}


int ad_ceil_log2(long long x)
{
    int b = 0;
    while ((1LL << b) < x) ++b;
    return b;
}

}  // namespace

mpq_status launch_adaptive(const float *W, int C, int d, int qmax, int k_max, double eta,
                           long long max_cand, int8_t *codes, float *scales, float *resid_sq,
                           long long *ncand, cudaStream_t stream)
{
    const long long ev = (long long)d * qmax;
    if (ev > A_MAX_EVENTS) {
        set_error("adaptive grid: d * Qmax = %lld exceeds %d thresholds per step", ev, A_MAX_EVENTS);
        return MPQ_ERR_UNSUPPORTED;
    }
    const int cap = (int)(ev > d ? ev : d);
    const int grid = (int)std::min<long long>(C, (long long)sm_count() * A_CTAS_PER_SM);
    const size_t smem = (size_t)d * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(adaptive_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute (adaptive grid)");
    uint2 *scratch = nullptr;
    const mpq_status st = pool_scratch(reinterpret_cast<void **>(&scratch),
                                       (size_t)grid * 2 * cap * sizeof(uint2), stream);
    if (st != MPQ_OK) return st;
    adaptive_kernel<<<grid, AT, smem, stream>>>(W, C, d, qmax, k_max, eta, max_cand,
                                                ad_ceil_log2(ev) + 1, codes, scales, resid_sq,
                                                ncand, scratch, cap);
    e = cudaGetLastError();
    const cudaError_t ef = cudaFreeAsync(scratch, stream);
    if (e == cudaSuccess) e = ef;
    return cuda_status(e, "adaptive-grid kernel launch");
}

}  // namespace mpq
