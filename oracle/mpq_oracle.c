/*
 * Multipoint quantization oracle -- plain, slow, single-threaded CPU restatement of the method
 * (Liu et al., "Post-training Quantization with Multiple Points", arXiv 2002.09049).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or calls this file: only the
 * tests, __graft_entry__.smoke() and bench.py's CPU-baseline / reference arm use it.  It shares no
 * code, header, table or helper with the CUDA path.
 *
 * Build: cc -std=c99 -O2 -ffp-contract=off -fno-fast-math -fPIC -shared (see oracle/__init__.py).
 * -ffp-contract=off keeps every a*b+c below as a rounded multiply followed by a rounded add, except
 * where fmaf() is written out on purpose.
 *
 * Notation follows the paper: residual r_i (Eq. 7), scale a and codes [r/a]_Q (Eq. 8), scale search
 * (Eq. 9), Algorithm 1 (greedy points), output error e(w, w~, D_L) (Eq. 11), Algorithm 2 (per-channel
 * point count), multipoint sum w~ = sum_i a_i w~_i (Eq. 4).  The paper's a_i [r/a_i]_{[-1:eps_b:1]}
 * is written here as s_i q_i with integer codes q_i in {-Qmax..Qmax}, Qmax = 2^(b-1)-1 and
 * s_i = a_i / Qmax (Eq. 1, symmetric set, B = 0).
 *
 * Readings where the paper is silent, ambiguous or garbled:
 *  - exact half-way ties of the nearest rounding (Eq. 2) go to the even integer (C nearbyintf);
 *  - r / a is one correctly rounded fp32 division (Eq. 8 writes a division);
 *  - the scale grid is G points s_g = f_g * (max|r| / Qmax), f_g = (g+1)/G in fp32 unless the caller
 *    gives its own increasing fractions in (0, 1] (replaces the adaptive grid of Eq. 10, which
 *    mpqo_quantize_channel_adaptive restates, with its own readings, for small channels);
 *  - the scale search keeps the FIRST (lowest g) minimiser;
 *  - a candidate whose fp32 scale underflows to 0 gives all-zero codes;
 *  - a residual that is exactly zero gives a "null point": scale 0, codes 0, residual unchanged;
 *  - a channel holding a NaN or Inf weight gets scales NaN, codes 0, residuals = w, errors NaN;
 *  - the residual update is r <- fmaf(-s, q, r), one correctly rounded fp32 operation;
 *  - the expectation of Eq. 11 is the sample mean over the N calibration rows, evaluated on the
 *    residual r_{n+1} = w - w~(n) produced by the same fp32 recursion;
 *  - the per-channel point budget: see mpqo_allocate_budget.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>
#include <stdlib.h>

/* Eq. 1 with b bits: the symmetric integer grid {-Qmax..Qmax}, Qmax = 2^(b-1) - 1. */
static int qmax_of(int bits) { return (1 << (bits - 1)) - 1; }

/* Eq. 2-3 and Eq. 8: nearest element of s * {-Qmax..Qmax} to r, returned as the integer code.
 * Rounding to the nearest integer and then clipping to [-Qmax, Qmax] gives the nearest grid
 * element because the grid is a contiguous run of integers. */
static int nearest_code(float r, float s, int qmax)
{
    if (s == 0.0f) return 0;
    float t = nearbyintf(r / s);
    if (t > (float)qmax) t = (float)qmax;
    if (t < (float)(-qmax)) t = (float)(-qmax);
    return (int)t;
}

/* The g-th candidate scale of the search grid (0-based g). */
static float candidate_scale(int g, int G, const float *grid_frac, float smax)
{
    float f = grid_frac ? grid_frac[g] : (float)(g + 1) / (float)G;
    return f * smax;
}

static int all_finite(const float *w, int d)
{
    for (int j = 0; j < d; ++j)
        if (!isfinite(w[j])) return 0;
    return 1;
}

/* The objective of Eq. 9 for one candidate scale: || r - s [r/s]_Q ||^2, summed in double in
 * index order.  s*q is exact in double (24-bit times <=8-bit). */
static double candidate_error(const float *r, int d, float s, int qmax)
{
    double E = 0.0;
    for (int j = 0; j < d; ++j) {
        int q = nearest_code(r[j], s, qmax);
        double e = (double)r[j] - (double)s * (double)q;
        E += e * e;
    }
    return E;
}

/* All G candidate errors of Eq. 9 for one residual (used by the brute-force tests).
 * E[g] and s[g] are written for g = 0..G-1.  A zero residual gives s = 0 and E = 0 everywhere. */
void mpqo_candidate_errors(const float *r, int d, int bits, int G, const float *grid_frac,
                           double *E, float *s)
{
    int qmax = qmax_of(bits);
    float m = 0.0f;
    for (int j = 0; j < d; ++j) {
        float a = fabsf(r[j]);
        if (a > m) m = a;
    }
    float smax = m / (float)qmax;
    for (int g = 0; g < G; ++g) {
        float sg = (m == 0.0f) ? 0.0f : candidate_scale(g, G, grid_frac, smax);
        s[g] = sg;
        E[g] = candidate_error(r, d, sg, qmax);
    }
}

/* Algorithm 1 for one channel w (length d), run to k_max points.
 *   codes     [k_max][code_stride]  int8  (row i holds q_{i+1}; only the first d entries are written)
 *   scales    [k_max]               fp32  (s_{i+1})
 *   resid_sq  [k_max+1]             double, ||r_{n+1}||^2 for n = 0..k_max (n = 0 is ||w||^2)
 *   residuals [k_max][res_stride]   fp32  r_{n+1} for n = 1..k_max, nullable
 *   gstar     [k_max]               chosen grid index, -1 for a null point, nullable
 *   best, second [k_max]            smallest and second smallest E_g of each step, nullable
 * Every step: m = max|r| (exact), smax = m / Qmax, candidates s_g, codes [r/s_g]_Q, the first g with
 * the smallest error (Eq. 9), then r <- r - s q (Eq. 7) as one fmaf per element. */
void mpqo_quantize_channel(const float *w, int d, int bits, int G, const float *grid_frac,
                           int k_max, int8_t *codes, long code_stride, float *scales,
                           double *resid_sq, float *residuals, long res_stride, float *r,
                           int *gstar, double *best, double *second)
{
    int qmax = qmax_of(bits);
    for (int j = 0; j < d; ++j) r[j] = w[j];
    int finite = all_finite(w, d);

    double r2 = 0.0;
    for (int j = 0; j < d; ++j) r2 += (double)r[j] * (double)r[j];
    if (resid_sq) resid_sq[0] = finite ? r2 : NAN;

    for (int i = 0; i < k_max; ++i) {
        int8_t *qi = codes + (long)i * code_stride;
        double E1 = INFINITY, E2 = INFINITY;
        int gbest = -1;
        float sbest = 0.0f;

        if (!finite) {
            for (int j = 0; j < d; ++j) qi[j] = 0;
            scales[i] = NAN;
        } else {
            float m = 0.0f;
            for (int j = 0; j < d; ++j) {
                float a = fabsf(r[j]);
                if (a > m) m = a;
            }
            if (m == 0.0f) {
                /* null point: nothing left to represent */
                for (int j = 0; j < d; ++j) qi[j] = 0;
                scales[i] = 0.0f;
                E1 = E2 = 0.0;
            } else {
                float smax = m / (float)qmax;
                for (int g = 0; g < G; ++g) {
                    float sg = candidate_scale(g, G, grid_frac, smax);
                    double E = candidate_error(r, d, sg, qmax);
                    if (E < E1) {
                        E2 = E1;
                        E1 = E;
                        gbest = g;
                        sbest = sg;
                    } else if (E < E2) {
                        E2 = E;
                    }
                }
                for (int j = 0; j < d; ++j) {
                    int q = nearest_code(r[j], sbest, qmax);
                    qi[j] = (int8_t)q;
                    r[j] = fmaf(-sbest, (float)q, r[j]);
                }
                scales[i] = sbest;
            }
        }
        if (gstar) gstar[i] = gbest;
        if (best) best[i] = E1;
        if (second) second[i] = E2;
        if (residuals) {
            float *ri = residuals + (long)i * res_stride;
            for (int j = 0; j < d; ++j) ri[j] = r[j];
        }
        if (resid_sq) {
            double s2 = 0.0;
            for (int j = 0; j < d; ++j) s2 += (double)r[j] * (double)r[j];
            resid_sq[i + 1] = finite ? s2 : NAN;
        }
    }
}

/* ---- The adaptive grid of Eq. 10 (Definition 1) ---------------------------------------------- */

static int cmp_double(const void *a, const void *b)
{
    const double x = *(const double *)a, y = *(const double *)b;
    return (x > y) - (x < y);
}

/* Definition 1: the minimal gap of t, half the smallest difference between two of its element
 * magnitudes.  Reading: the pair condition is |t_i| != |t_j| (as printed, t_i != t_j admits
 * t_i = -t_j, whose gap would be 0).  Magnitudes sorted in double; INFINITY when t has fewer than
 * two distinct magnitudes.  work: scratch of d doubles. */
double mpqo_minimal_gap(const float *t, int d, double *work)
{
    for (int j = 0; j < d; ++j) work[j] = fabs((double)t[j]);
    qsort(work, (size_t)d, sizeof(double), cmp_double);
    double g = INFINITY;
    for (int j = 1; j < d; ++j)
        if (work[j] != work[j - 1]) {
            const double x = (work[j] - work[j - 1]) / 2.0;
            if (x < g) g = x;
        }
    return g;
}

/* ---- The same grid search without enumerating the grid (long channels) ---------------------- */

static float adaptive_scale(long m, double gamma, int qmax)
{
    return (float)(((double)m * gamma) / (double)qmax);
}

/* Code magnitude of |r| = a at scale s, as nearest_code computes it (the rounding is symmetric). */
static int code_mag_at(float a, float s, int qmax)
{
    if (s == 0.0f) return 0;
    float t = nearbyintf(a / s);
    if (t > (float)qmax) t = (float)qmax;
    return (int)t;
}

struct ad_event {
    long m;      /* first grid index with the code below L */
    int j, L;
};

struct ad_piece {
    long ma, mb;     /* grid indices with the same codes */
    double P, N;     /* sum a_j c_j and sum c_j^2 there */
};

static int cmp_event(const void *x, const void *y)
{
    const struct ad_event *a = (const struct ad_event *)x, *b = (const struct ad_event *)y;
    return (a->m > b->m) - (a->m < b->m);
}

/* first m in [lo, hi] with s_m >= target (hi + 1 if none) */
static long first_scale_at_least(long lo, long hi, double target, double gamma, int qmax)
{
    long a = lo, b = hi + 1;
    while (a < b) {
        const long mid = a + (b - a) / 2;
        if ((double)adaptive_scale(mid, gamma, qmax) >= target) b = mid; else a = mid + 1;
    }
    return a;
}

/* The quadratic form of the objective and a bound on its distance from the definition's sum
 * (d double roundings of terms no larger than R2 + 2 s P + s^2 N, d <= 8192 < 2^13). */
static double quad(double R2, double P, double N, double s) { return R2 - 2.0 * s * P + s * s * N; }
static double quad_tol(double R2, double P, double N, double s)
{
    return 0x1p-36 * (R2 + 2.0 * s * P + s * s * N);
}

/* One step of the grid search of Eq. 10 taking the same decision as the enumeration (the first m
 * with the smallest objective), without enumerating the grid:
 *  - each element's code magnitude is a non-increasing step function of m (s_m and the correctly
 *    rounded division are monotone): its change points come from binary searches, and between
 *    them (pieces) the codes are constant and the objective is, up to rounding, the convex
 *    quadratic R2 - 2 s P + s^2 N of the fp32 scale s_m, smallest next to s = P / N;
 *  - pass 1 bounds the smallest objective from above with the grid points around each piece's
 *    minimiser; pass 2 evaluates by the definition, in m order, every grid point whose quadratic
 *    lower bound reaches that bound (the first of each run of equal scales).
 * ev: scratch of d Qmax events; pc: scratch of d Qmax + 1 pieces; c: scratch of d ints.
 * Returns the chosen m (0 when M = 0) and its objective in *E; -1 if more than max_eval points
 * would need the definition (never seen; a guard). */
static long adaptive_step_piecewise(const float *r, int d, int qmax, double gamma, long M,
                                    long max_eval, struct ad_event *ev, struct ad_piece *pc,
                                    int *c, double *E)
{
    *E = INFINITY;
    if (M <= 0) return 0;
    double R2 = 0.0;
    for (int j = 0; j < d; ++j) R2 += (double)r[j] * (double)r[j];
    long ne = 0;
    double P = 0.0, N = 0.0;
    const float s1 = adaptive_scale(1, gamma, qmax);
    for (int j = 0; j < d; ++j) {
        const float a = fabsf(r[j]);
        c[j] = code_mag_at(a, s1, qmax);
        P += (double)a * (double)c[j];
        N += (double)c[j] * (double)c[j];
        for (int L = c[j]; L >= 1; --L) {
            long lo = 2, hi = M + 1;         /* first m in [2, M] with code < L, or M + 1 */
            while (lo < hi) {
                const long mid = lo + (hi - lo) / 2;
                if (code_mag_at(a, adaptive_scale(mid, gamma, qmax), qmax) < L) hi = mid;
                else lo = mid + 1;
            }
            if (lo <= M) {
                ev[ne].m = lo;
                ev[ne].j = j;
                ev[ne].L = L;
                ++ne;
            }
        }
    }
    qsort(ev, (size_t)ne, sizeof(struct ad_event), cmp_event);
    /* pass 1: the pieces, and an upper bound of the smallest objective */
    long np = 0, e = 0, ma = 1;
    double upper = INFINITY;
    while (ma <= M) {
        const long mb = (e < ne) ? ev[e].m - 1 : M;
        if (mb >= ma) {
            pc[np].ma = ma;
            pc[np].mb = mb;
            pc[np].P = P;
            pc[np].N = N;
            ++np;
            long pick[3];
            int k = 0;
            pick[k++] = ma;
            if (N > 0.0) {
                const long g = first_scale_at_least(ma, mb, P / N, gamma, qmax);
                if (g <= mb) pick[k++] = g;
                if (g - 1 >= ma) pick[k++] = g - 1;
            }
            for (int t = 0; t < k; ++t) {
                const double sd = (double)adaptive_scale(pick[t], gamma, qmax);
                const double u = quad(R2, P, N, sd) + quad_tol(R2, P, N, sd);
                if (u < upper) upper = u;
            }
        }
        const long next = mb + 1;
        while (e < ne && ev[e].m == next) {
            P -= (double)fabsf(r[ev[e].j]);
            N -= (double)(2 * ev[e].L - 1);
            ++e;
        }
        ma = next;
    }
    /* pass 2: every grid point whose objective may reach the smallest, by the definition */
    long bestm = 0, evals = 0;
    double bestE = INFINITY;
    for (long t = 0; t < np; ++t) {
        const struct ad_piece *q = &pc[t];
        long lo = q->ma, hi = q->mb;
        if (q->N > 0.0) {
            /* N (s - P/N)^2 + R2 - P^2/N - tol <= upper, tol taken at the piece's largest scale */
            const double smax = (double)adaptive_scale(q->mb, gamma, qmax);
            const double tol = quad_tol(R2, q->P, q->N, smax);
            const double floor_q = R2 - q->P * q->P / q->N;
            const double room = (upper + 2.0 * tol - floor_q) / q->N;
            if (room < 0.0) continue;
            const double half = sqrt(room) * (1.0 + 0x1p-30) + 0x1p-60;
            const double tgt = q->P / q->N;
            lo = first_scale_at_least(q->ma, q->mb, tgt - half, gamma, qmax);
            hi = first_scale_at_least(q->ma, q->mb, tgt + half, gamma, qmax);   /* exclusive */
            if (hi <= q->mb) ++hi;   /* the first scale past the window too */
            hi -= 1;
            if (lo > hi) continue;
        } else {
            if (R2 - quad_tol(R2, 0.0, 0.0, 0.0) > upper) continue;
            hi = lo;              /* constant objective: the first index only */
        }
        float prev = -1.0f;
        for (long m = lo; m <= hi; ++m) {
            const float sm = adaptive_scale(m, gamma, qmax);
            if (sm == prev) continue;      /* same scale, same objective: the earlier m wins */
            prev = sm;
            if (++evals > max_eval) return -1;
            const double Em = candidate_error(r, d, sm, qmax);
            if (Em < bestE || (Em == bestE && m < bestm)) {
                bestE = Em;
                bestm = m;
            }
        }
    }
    *E = bestE;
    return bestm;
}

/* The objective of Eq. 9 at one scale s, by its definition (double, index order), and the codes
 * q = [r/s]_Q it takes (Eq. 8; nullable).  Used to judge a scale another implementation chose. */
double mpqo_objective(const float *r, int d, int bits, float s, int8_t *codes)
{
    const int qmax = qmax_of(bits);
    if (codes)
        for (int j = 0; j < d; ++j) codes[j] = (int8_t)nearest_code(r[j], s, qmax);
    return candidate_error(r, d, s, qmax);
}

/* Algorithm 1 with the grid of Eq. 10 for one channel w, run to k_max points.  Each step i:
 * Delta = minimal gap of r_i (Definition 1), gamma = min(Delta / Qmax, eta) (gamma = eta when
 * Delta is infinite), and the search over a in I = [0, 2 Qmax ||r_i||] with step gamma: the
 * candidates a_m = m * gamma, m = 1..M, M = floor(2 Qmax ||r_i|| / gamma) (a = 0 leaves [r/a]
 * undefined), each as the fp32 point scale s_m = fl(a_m / Qmax) (s q = a [r/a]_Q, Eq. 1).  The codes,
 * the error (double, index order), the first minimiser and the update r <- fmaf(-s, q, r) are those
 * of the fixed grid above.  A zero residual gives a null point (gamma = 0, no candidates).
 * Writes codes [k_max][d], scales [k_max], resid_sq [k_max+1], gamma [k_max], ncand [k_max],
 * best/second [k_max] (nullable).  A step whose grid would exceed max_cand candidates is refused:
 * its scale and every later one NaN, codes 0, squared norms NaN, ncand -1 for it and 0 after;
 * returns -1 then, else 0.  piecewise = 0 enumerates every grid point; 1 takes the same decisions
 * through adaptive_step_piecewise (best holds the chosen objective, second is NaN), for grids too
 * large to enumerate (-2 if its guard trips).  r: scratch of d floats; work: scratch of d doubles;
 * rin (nullable): [k_max][d], the residual each step starts from. */
int mpqo_quantize_channel_adaptive(const float *w, int d, int bits, int k_max, double eta,
                                   long max_cand, int8_t *codes, float *scales, double *resid_sq,
                                   double *gamma, long *ncand, double *best, double *second,
                                   float *r, double *work, int piecewise, float *rin)
{
    int qmax = qmax_of(bits);
    struct ad_event *ev = NULL;
    struct ad_piece *pc = NULL;
    int *cw = NULL;
    if (piecewise) {
        ev = (struct ad_event *)malloc(sizeof(struct ad_event) * ((size_t)d * qmax + 1));
        pc = (struct ad_piece *)malloc(sizeof(struct ad_piece) * ((size_t)d * qmax + 1));
        cw = (int *)malloc(sizeof(int) * (size_t)d);
        if (!ev || !pc || !cw) {
            free(ev);
            free(pc);
            free(cw);
            return -3;
        }
    }
    int status = 0;
    for (int j = 0; j < d; ++j) r[j] = w[j];
    int finite = all_finite(w, d);
    double r2 = 0.0;
    for (int j = 0; j < d; ++j) r2 += (double)r[j] * (double)r[j];
    resid_sq[0] = finite ? r2 : NAN;

    int refused = 0;
    for (int i = 0; i < k_max; ++i) {
        int8_t *qi = codes + (long)i * d;
        if (rin)
            for (int j = 0; j < d; ++j) rin[(long)i * d + j] = r[j];
        double E1 = INFINITY, E2 = INFINITY, g = 0.0;
        long M = 0;
        float sbest = 0.0f;
        if (!finite || refused) {
            for (int j = 0; j < d; ++j) qi[j] = 0;
            scales[i] = NAN;
            g = NAN;
        } else if (r2 == 0.0) {
            for (int j = 0; j < d; ++j) qi[j] = 0;   /* null point */
            scales[i] = 0.0f;
            E1 = E2 = 0.0;
        } else {
            const double delta = mpqo_minimal_gap(r, d, work);
            g = delta / (double)qmax;
            if (!(g < eta)) g = eta;
            const double top = 2.0 * (double)qmax * sqrt(r2);
            const double mf = floor(top / g);
            if (mf > (double)max_cand) {
                refused = 1;
                for (int j = 0; j < d; ++j) qi[j] = 0;
                scales[i] = NAN;
                gamma[i] = g;
                ncand[i] = -1;
                if (best) best[i] = NAN;
                if (second) second[i] = NAN;
                resid_sq[i + 1] = NAN;
                continue;
            }
            M = (long)mf;
            if (piecewise) {
                double Ebest;
                const long mb = adaptive_step_piecewise(r, d, qmax, g, M, 100000000L, ev, pc, cw,
                                                        &Ebest);
                if (mb < 0) {
                    status = -2;
                    break;
                }
                sbest = mb > 0 ? adaptive_scale(mb, g, qmax) : 0.0f;
                E1 = Ebest;
                E2 = NAN;
            } else {
                for (long m = 1; m <= M; ++m) {
                    const float sm = adaptive_scale(m, g, qmax);
                    const double E = candidate_error(r, d, sm, qmax);
                    if (E < E1) {
                        E2 = E1;
                        E1 = E;
                        sbest = sm;
                    } else if (E < E2) {
                        E2 = E;
                    }
                }
            }
            for (int j = 0; j < d; ++j) {
                int q = nearest_code(r[j], sbest, qmax);
                qi[j] = (int8_t)q;
                r[j] = fmaf(-sbest, (float)q, r[j]);
            }
            scales[i] = sbest;
        }
        gamma[i] = g;
        ncand[i] = M;
        if (best) best[i] = E1;
        if (second) second[i] = E2;
        r2 = 0.0;
        for (int j = 0; j < d; ++j) r2 += (double)r[j] * (double)r[j];
        resid_sq[i + 1] = (finite && !refused) ? r2 : NAN;
    }
    free(ev);
    free(pc);
    free(cw);
    if (status) return status;
    return refused ? -1 : 0;
}

/* Algorithm 1 for channels [c0, c1) of a C x d layer (row-major W).  Output layouts match the
 * library's: codes [k_max][C][d], scales [C][k_max], resid_sq [C][k_max+1] (double here),
 * residuals [k_max][C][d] (nullable), gstar/best/second [C][k_max] (nullable).
 * work: scratch of d floats. */
void mpqo_quantize_layer(const float *W, int C, int d, int bits, int G, const float *grid_frac,
                         int k_max, int8_t *codes, float *scales, double *resid_sq,
                         float *residuals, int *gstar, double *best, double *second, int c0, int c1,
                         float *work)
{
    long plane = (long)C * d;
    for (int k = c0; k < c1; ++k) {
        mpqo_quantize_channel(W + (long)k * d, d, bits, G, grid_frac, k_max,
                              codes + (long)k * d, plane, scales + (long)k * k_max,
                              resid_sq ? resid_sq + (long)k * (k_max + 1) : NULL,
                              residuals ? residuals + (long)k * d : NULL, plane, work,
                              gstar ? gstar + (long)k * k_max : NULL,
                              best ? best + (long)k * k_max : NULL,
                              second ? second + (long)k * k_max : NULL);
    }
}

/* Eq. 11 for channels [c0, c1): err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2, n = 0..k_max, with
 * r_{k,1} = w_k and r_{k,n+1} = fmaf(-s_{k,n}, q_{k,n}, r_{k,n}) (the recursion of Eq. 7).
 * groups = 1: X is N x d, shared by every channel.  groups = C: X is [C][N][d], channel k reads
 * its own N x d block (depthwise convolution: each channel sees its own input patches).
 * Dot products and the mean are taken in double.  work: scratch of d floats. */
void mpqo_output_error(const float *X, int N, int groups, const float *W, const int8_t *codes,
                       const float *scales, int C, int d, int k_max, double *err, int c0, int c1,
                       float *work)
{
    long plane = (long)C * d;
    for (int k = c0; k < c1; ++k) {
        const float *Xk = (groups == 1) ? X : X + (long)k * N * d;
        float *r = work;
        for (int j = 0; j < d; ++j) r[j] = W[(long)k * d + j];
        for (int n = 0; n <= k_max; ++n) {
            if (n > 0) {
                float s = scales[(long)k * k_max + (n - 1)];
                const int8_t *q = codes + (long)(n - 1) * plane + (long)k * d;
                for (int j = 0; j < d; ++j) r[j] = fmaf(-s, (float)q[j], r[j]);
            }
            double acc = 0.0;
            for (int t = 0; t < N; ++t) {
                const float *x = Xk + (long)t * d;
                double y = 0.0;
                for (int j = 0; j < d; ++j) y += (double)x[j] * (double)r[j];
                acc += y * y;
            }
            err[(long)k * (k_max + 1) + n] = acc / (double)N;
        }
    }
}

/* Gain of the (n+1)-th point of channel k: e_k(n) - e_k(n+1), one fp32 subtraction of the fp32
 * error table (the same table the GPU allocator receives).  NaN is read as "no gain". */
static float point_gain(const float *err, int k_max, int k, int n)
{
    const float *e = err + (long)k * (k_max + 1);
    float g = e[n] - e[n + 1];
    return isnan(g) ? -INFINITY : g;
}

/* Point allocation with a total budget (the marginal-gain reading of Algorithm 2).
 * Every channel starts with one point.  P_total = floor(beta*C + 0.5); the extra P_total - C points
 * (at most C*(k_max-1)) are handed out one at a time, each to the channel whose next point lowers
 * its output error the most (largest e_k(n_k) - e_k(n_k+1), lowest k on ties), among channels with
 * n_k < k_max.  The loop stops early when the best remaining gain is <= 0.
 * Writes npoints[C]; returns the total number of points used. */
long mpqo_allocate_budget(const float *err, int C, int k_max, double beta, int *npoints)
{
    long total = (long)floor(beta * (double)C + 0.5);
    long extra = total - C;
    long cap = (long)C * (k_max - 1);
    if (extra < 0) extra = 0;
    if (extra > cap) extra = cap;
    for (int k = 0; k < C; ++k) npoints[k] = 1;
    long used = C;
    for (long it = 0; it < extra; ++it) {
        float bestg = -INFINITY;
        int bk = -1;
        for (int k = 0; k < C; ++k) {
            if (npoints[k] >= k_max) continue;
            float g = point_gain(err, k_max, k, npoints[k]);
            if (bk < 0 || g > bestg) {
                bestg = g;
                bk = k;
            }
        }
        if (bk < 0 || !(bestg > 0.0f)) break;
        npoints[bk] += 1;
        used += 1;
    }
    return used;
}

/* Algorithm 2 with a threshold: n_k is the smallest n in 1..k_max with e_k(n) < eps (compared in
 * double), else k_max.  Returns the total number of points. */
long mpqo_allocate_threshold(const float *err, int C, int k_max, double eps, int *npoints)
{
    long used = 0;
    for (int k = 0; k < C; ++k) {
        int n = k_max;
        for (int m = 1; m <= k_max; ++m) {
            if ((double)err[(long)k * (k_max + 1) + m] < eps) {
                n = m;
                break;
            }
        }
        npoints[k] = n;
        used += n;
    }
    return used;
}

/* Eq. 4: w~_k = sum_{i=1..n_k} s_{k,i} q_{k,i}, accumulated as acc = fmaf(s_i, q_i, acc) from
 * acc = 0 in the order i = 1, 2, ...  n_k is clamped to [0, k_max]. */
void mpqo_reconstruct(const int8_t *codes, const float *scales, const int *npoints,
                      const float *center, int C, int d, int k_max, float *W_hat)
{
    long plane = (long)C * d;
    for (int k = 0; k < C; ++k) {
        int n = npoints[k];
        if (n < 0) n = 0;
        if (n > k_max) n = k_max;
        for (int j = 0; j < d; ++j) {
            float acc = center ? center[k] : 0.0f;   /* the set's centre B (Eq. 1), 0 if symmetric */
            for (int i = 0; i < n; ++i)
                acc = fmaf(scales[(long)k * k_max + i], (float)codes[(long)i * plane + (long)k * d + j],
                           acc);
            W_hat[(long)k * d + j] = acc;
        }
    }
}

/* ---- Eq. 1 with B != 0: asymmetric sets ---------------------------------------------------------
 * The quantization set K x [-1 : eps_b : 1] + B has the centre B.  Per channel (mode 0) every
 * channel has its own B; per layer (mode 1) one B serves all the layer's channels.  Readings (the
 * paper gives no formula for B): B is the midpoint of the weights' range, (max w + min w) / 2 rounded once to fp32,
 * so that K = (max w - min w) / 2 covers every weight without clipping (the per-channel
 * experiments clip nothing); the multipoint approximation takes B once and approximates the
 * centred weights w - B (one fp32 subtraction) with the greedy points, so that
 * w~ = B + sum_i s_i q_i; a non-finite weight makes B NaN for its channel (per layer: for all). */
void mpqo_center(const float *W, int C, int d, int mode, float *center, float *Wc)
{
    double lo = 0.0, hi = 0.0;
    int bad = 0, seen = 0;
    for (int k = 0; k < C; ++k) {
        const float *w = W + (long)k * d;
        double klo = 0.0, khi = 0.0;
        int kbad = !all_finite(w, d);
        for (int j = 0; j < d; ++j) {
            double v = (double)w[j];
            if (j == 0 || v < klo) klo = v;
            if (j == 0 || v > khi) khi = v;
        }
        if (mode == 0) {
            /* (hi + lo) / 2 is exact in double for two fp32 values of a weight range; one rounding */
            center[k] = kbad ? NAN : (d > 0 ? (float)((khi + klo) * 0.5) : 0.0f);
        } else if (d > 0) {
            if (!seen || klo < lo) lo = klo;
            if (!seen || khi > hi) hi = khi;
            seen = 1;
        }
        bad |= kbad;
    }
    if (mode == 1) {
        float b = bad ? NAN : (float)((hi + lo) * 0.5);
        for (int k = 0; k < C; ++k) center[k] = b;
    }
    for (int k = 0; k < C; ++k)
        for (int j = 0; j < d; ++j) {
            float v = W[(long)k * d + j] - center[k];   /* one fp32 subtraction */
            Wc[(long)k * d + j] = v;
        }
}

/* ---- Eq. 12: output-error-driven clipping factor ------------------------------------------------
 * The clipping factor K of the quantization set K x [-1 : eps_b : 1] (Eq. 1, B = 0) is chosen among
 * nc candidates by the output error of Eq. 11 instead of the weight error.  Readings (App. B gives
 * only the grid): the candidates are K_c = f_c * m with f_c = (c+1)/nc in fp32, c = 0..nc-1 (nc = 20 is
 * the experiments' uniform grid [0.05 : 0.05 : 1] x max|w|); m = max_j |w_kj| per channel
 * (mode 0) or the maximum over the whole layer (mode 1, one K for every channel); the set's
 * elements are s q with s = K / Qmax (fp32 division) and codes q = [w / s]_Q as in Eq. 8; the
 * residual is fmaf(-s, q, w); a non-finite weight makes m -- and so every K of that channel, or of
 * the layer in mode 1 -- NaN. */

/* Candidate clipping factors clip[k][c] of channels 0..C-1. */
void mpqo_clip_candidates(const float *W, int C, int d, int nc, int mode, float *clip)
{
    float layer_m = 0.0f;
    for (int k = 0; k < C; ++k) {
        const float *w = W + (long)k * d;
        float m = 0.0f;
        if (!all_finite(w, d)) {
            m = NAN;
        } else {
            for (int j = 0; j < d; ++j)
                if (fabsf(w[j]) > m) m = fabsf(w[j]);
        }
        if (mode == 0) {
            for (int c = 0; c < nc; ++c) clip[(long)k * nc + c] = ((float)(c + 1) / (float)nc) * m;
        }
        if (isnan(m) || isnan(layer_m)) layer_m = NAN;
        else if (m > layer_m) layer_m = m;
    }
    if (mode == 1)
        for (int k = 0; k < C; ++k)
            for (int c = 0; c < nc; ++c)
                clip[(long)k * nc + c] = ((float)(c + 1) / (float)nc) * layer_m;
}

/* The objective of Eq. 12 for every candidate of channels [c0, c1):
 * err[k][c] = (1/N) sum_t (x_t . r_{k,c})^2, r_{k,c} = fmaf(-s, [w_k / s]_Q, w_k), s = K_{k,c} / Qmax,
 * dot products and the mean in double.  groups as in mpqo_output_error.  work: d floats. */
void mpqo_clip_errors(const float *X, int N, int groups, const float *W, int C, int d, int bits,
                      int nc, const float *clip, double *err, int c0, int c1, float *work)
{
    const int qmax = qmax_of(bits);
    for (int k = c0; k < c1; ++k) {
        const float *Xk = (groups == 1) ? X : X + (long)k * N * d;
        const float *w = W + (long)k * d;
        for (int c = 0; c < nc; ++c) {
            const float s = clip[(long)k * nc + c] / (float)qmax;
            for (int j = 0; j < d; ++j)
                work[j] = fmaf(-s, (float)nearest_code(w[j], s, qmax), w[j]);
            double acc = 0.0;
            for (int t = 0; t < N; ++t) {
                const float *x = Xk + (long)t * d;
                double y = 0.0;
                for (int j = 0; j < d; ++j) y += (double)x[j] * (double)work[j];
                acc += y * y;
            }
            err[(long)k * nc + c] = acc / (double)N;
        }
    }
}

/* The argmin of Eq. 12 on an error table of fp32 values (as the device computes them):
 * mode 0, per channel: the lowest c with the smallest err[k][c];
 * mode 1, per layer: the lowest c with the smallest sum_k err[k][c] (double, k ascending), the same
 * c for every channel.  NaN never wins; no finite candidate gives -1. */
void mpqo_clip_select(const float *err, int C, int nc, int mode, int *best)
{
    if (mode == 0) {
        for (int k = 0; k < C; ++k) {
            int b = -1;
            float bv = 0.0f;
            for (int c = 0; c < nc; ++c) {
                const float v = err[(long)k * nc + c];
                if (isnan(v)) continue;
                if (b < 0 || v < bv) {
                    b = c;
                    bv = v;
                }
            }
            best[k] = b;
        }
        return;
    }
    int b = -1;
    double bv = 0.0;
    for (int c = 0; c < nc; ++c) {
        double e = 0.0;
        for (int k = 0; k < C; ++k) e += (double)err[(long)k * nc + c];
        if (isnan(e)) continue;
        if (b < 0 || e < bv) {
            b = c;
            bv = e;
        }
    }
    for (int k = 0; k < C; ++k) best[k] = b;
}

/* ---- Eq. 13 and Sec. 3.4: integer inference with multipoint weights -------------------------------
 * A layer whose channel k holds n_k points (s_{k,i}, q_{k,i}) computes, for integer inputs x_t,
 *   w~_k^T x_t = sum_i s_{k,i} (q_{k,i}^T x_t) ~ (sum_i A_{k,i} (q_{k,i}^T x_t)) / 2^p,
 *   A_{k,i} = [2^p s_{k,i}]  (Eq. 13),
 * in three steps: integer dot products (step 1), multiplication by the 32-bit coefficients and
 * summation (step 2), and a shift by p bits (step 3).  Readings of Sec. 3.4: the codes q are
 * the integers of the symmetric set, so the coefficient of q is s = a / Qmax and A = rint(2^p s)
 * (ties to even); "shifting p bits" is an arithmetic right shift, i.e. floor division by 2^p; the
 * products and sums are exact (64-bit); the result saturates to the 32-bit range; n_k = npoints[k]
 * clamped to [0, k_max]; a coefficient that does not fit 32 bits is an error. */

/* A = rint(2^p s); *ok = 0 when it does not fit a 32-bit integer (or s is not finite). */
long long mpqo_fixed_coeff(float s, int p, int *ok)
{
    double v = nearbyint(ldexp((double)s, p));
    if (!(fabs(v) < 2147483648.0)) {
        *ok = 0;
        return 0;
    }
    return (long long)v;
}

/* Y[k][t] for channels [c0, c1), X [T][d] int8, Y [C][T] int32.  With a centre B_k (asymmetric set,
 * Eq. 1; center may be NULL), w~ = B_k 1 + sum_i s_i q_i and the centre adds A_B (sum_j x_j) with
 * A_B = rint(2^p B_k) to the sum before the shift.  Returns 0, or 1 if a coefficient did not fit 32
 * bits (Y is then unspecified). */
int mpqo_multipoint_linear(const int8_t *X, int T, const int8_t *codes, const float *scales,
                           const int *npoints, const float *center, int C, int d, int k_max, int p,
                           int32_t *Y, int c0, int c1)
{
    long plane = (long)C * d;
    for (int k = c0; k < c1; ++k) {
        int n = npoints[k];
        if (n < 0) n = 0;
        if (n > k_max) n = k_max;
        long long A[64];
        for (int i = 0; i < n; ++i) {
            int ok = 1;
            A[i] = mpqo_fixed_coeff(scales[(long)k * k_max + i], p, &ok);
            if (!ok) return 1;
        }
        long long AB = 0;
        if (center) {
            int ok = 1;
            AB = mpqo_fixed_coeff(center[k], p, &ok);
            if (!ok) return 1;
        }
        for (int t = 0; t < T; ++t) {
            const int8_t *x = X + (long)t * d;
            long long sum = 0;
            if (center) {
                long long xs = 0;
                for (int j = 0; j < d; ++j) xs += (long long)x[j];
                sum += AB * xs;                                     /* the centre's term */
            }
            for (int i = 0; i < n; ++i) {
                const int8_t *q = codes + (long)i * plane + (long)k * d;
                long long acc = 0;                                  /* step 1 */
                for (int j = 0; j < d; ++j) acc += (long long)q[j] * (long long)x[j];
                sum += A[i] * acc;                                  /* step 2 */
            }
            long long y = sum >= 0 ? (sum >> p) : -((-sum + ((1LL << p) - 1)) >> p);  /* step 3: floor */
            if (y > 2147483647LL) y = 2147483647LL;
            if (y < -2147483648LL) y = -2147483648LL;
            Y[(long)k * T + t] = (int32_t)y;
        }
    }
    return 0;
}
