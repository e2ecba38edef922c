// Greedy multipoint construction (Sec. 3.2, Eq. 6-9, Algorithm 1) for every channel of a layer.
//
// A group of WPC warps (1, 2, 4 or 8; chosen per layer from C, d and shared memory) owns one
// channel for all k_max steps: the residual row r (fp32) stays in shared memory from the first
// load of w to the last update, so global memory sees one read of w and one write of each step's
// codes (and of the optional residual / norm outputs).  Short channels (depthwise 3x3, d = 9) get
// a single warp and synchronise with warp primitives only; long channels of layers with few
// channels get up to 8 warps and named barriers.
//
// Scale search (Eq. 9).  For a candidate scale s with codes c_j = min(Qmax, rint(|r_j| / s)),
//   E(s) = ||r - s q||^2 = ||r||^2 - 2 s P + s^2 N,   P = sum_j |r_j| c_j,   N = sum_j c_j^2,
// so only D(s) = s (s N - 2 P) decides the argmin.  N is an exact integer and P is accumulated
// exactly in 64-bit fixed point (|r_j| scaled by 2^S, S chosen per step from max|r| so the sum
// cannot overflow; exact for every element whose code can be nonzero on the grid).  Every D is
// first evaluated in fp32 together with a rigorous bound on its rounding error; only the
// candidates whose interval can hold the minimum are re-evaluated in double, and the lowest index
// among the exact minima wins.  The result is the argmin of the exact D values: deterministic and
// independent of d and of the summation order, with the narrow fp64 pipe touched a few times per
// step.
//
// Event form.  The candidate scales increase with g, so every element's code c_j(g) is a
// non-increasing step function of g (the fp32 quotient, rint and the clamp are all monotone).
// For each level L, {g : c_j(g) >= L} is a prefix [0, T_{j,L}); hence
//   P_g = sum_{(j,L)} R_j [g < T_{j,L}],   N_g = sum_{(j,L)} (2L - 1) [g < T_{j,L}].
// Levels held at the largest scale (L <= c_j(G-1)) count for every g and are summed directly;
// every other level the element crosses adds (R_j, 2L-1) to a histogram bin T_{j,L}.  T is found
// in closed form on the linear grid (exact unless the estimate falls within 2^-20 of a grid point,
// where the exact rule settles it) or by bisection on a caller's grid, then checked with the same
// correctly rounded division and rint as the definition.  A suffix sum over the bins gives P_g and
// N_g for all g.  Work per element and step is O(Qmax) instead of O(G).  (If a candidate scale
// underflows to 0 the monotonicity argument fails; such steps evaluate every candidate directly.)
#include <float.h>
#include <limits.h>
#include <math.h>

#include <algorithm>
#include <type_traits>
#include <vector>

#include "mpq_internal.cuh"
#include "rounding.cuh"
#include "sm100.cuh"

MPQ_CHECKED_UNIT("quantize.cu");

namespace mpq {
namespace {

constexpr int QTHREADS = 256;                                   // 8 warps per CTA
constexpr int QDIRECT_MAX_D = 32;                               // direct candidate evaluation up to here
constexpr int QMAX_LIMIT = (1 << (MPQ_MAX_BITS - 1)) - 1;

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

constexpr int QNEAR = 128;   // lattice-adjacent elements a group queues per step

// Per-group scratch for cross-warp reductions, and the queue of lattice-adjacent elements.
struct Scratch {
    float nearq[QNEAR];
    int nq;
    float f[8];
    float v[8];
    unsigned long long key[8];
    unsigned long long sp[8];
    long long sn[8];
    long long a[8];
    long long b[8];
    int g[8];
    int flag[8];
};

// Shared memory: a CTA-wide table of the grid fractions f_g and fl(1/f_g) (2G words; left out on
// the linear grid when that fits one more CTA per SM, f_g then computed where needed), then per
// channel group (all 4-byte words): `copies` copies of hLo[G+1], hHi[G+1] (64-bit P bins as two
// words) and hN[G+1], then r[d].  Without the lattice every warp has a private copy (so warps
// never contend on a bin); with the lattice form (below) events are rare and the group shares one
// copy, and the group also holds nb lattice buckets first, two words each: the low 32 bits of the
// bucket's fixed-point R sum, and its high bits plus the bucket's element count shifted to bit
// cnt_bit (the launcher checks that neither field can overflow).  (Two separate word arrays, low
// words on all 32 banks, measured no faster.)  Group regions stay 8-byte
// aligned.
__host__ __device__ constexpr size_t lattice_words(int nb) { return (size_t)2 * nb; }

// bytes of the CTA's bucket -> position-index table (uint16 per bucket, and 16 spare entries so
// that the largest element's bucket, at most nb - 1, needs no clamp), 16-byte multiple
__host__ __device__ constexpr size_t lut_bytes(int nb) { return ((size_t)(nb + 16) * 2 + 15) & ~(size_t)15; }

__host__ __device__ constexpr size_t group_words(int G, int d, int copies, int nb)
{
    return lattice_words(nb) + (((size_t)3 * (G + 1) * copies + (size_t)d + 1) & ~(size_t)1);
}

template <int WPC>
__device__ __forceinline__ void gsync(int grp)
{
    if (WPC == 1) {
        __syncwarp();
    } else if (WPC == 8) {
        __syncthreads();
    } else {
        asm volatile("bar.sync %0, %1;" ::"r"(grp + 1), "r"(WPC * 32) : "memory");
    }
}

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

__device__ __forceinline__ float warp_min(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Group-wide max (floats >= 0), fp32 sum (fixed tree) and OR, in one exchange.
template <int WPC>
__device__ __forceinline__ void group_max_sum_or(float &m, float &v, int &flag, Scratch &sc,
                                                 int gw, int lane, int grp)
{
    m = warp_max(m);
    v = warp_sum(v);
    flag = __any_sync(0xffffffffu, flag) ? 1 : 0;
    if (WPC > 1) {
        gsync<WPC>(grp);
        if (lane == 0) {
            sc.f[gw] = m;
            sc.v[gw] = v;
            sc.flag[gw] = flag;
        }
        gsync<WPC>(grp);
        m = sc.f[0];
        v = 0.0f;
        flag = 0;
#pragma unroll
        for (int i = 0; i < WPC; ++i) {
            m = fmaxf(m, sc.f[i]);
            v += sc.v[i];
            flag |= sc.flag[i];
        }
    }
}

template <int WPC>
__device__ __forceinline__ void group_sum2(long long &x, long long &y, Scratch &sc, int gw,
                                           int lane, int grp)
{
    x = warp_sum(x);
    y = warp_sum(y);
    gsync<WPC>(grp);   // also publishes this group's shared-memory updates
    if (WPC > 1) {
        if (lane == 0) {
            sc.a[gw] = x;
            sc.b[gw] = y;
        }
        gsync<WPC>(grp);
        x = 0;
        y = 0;
#pragma unroll
        for (int i = 0; i < WPC; ++i) {
            x += sc.a[i];
            y += sc.b[i];
        }
    }
}

template <int WPC>
__device__ __forceinline__ float group_min(float v, Scratch &sc, int gw, int lane, int grp)
{
    v = warp_min(v);
    if (WPC > 1) {
        gsync<WPC>(grp);
        if (lane == 0) sc.f[gw] = v;
        gsync<WPC>(grp);
        v = sc.f[0];
#pragma unroll
        for (int i = 1; i < WPC; ++i) v = fminf(v, sc.f[i]);
    }
    return v;
}

// Order-preserving map of a double to unsigned 64-bit (total order, -0 < +0 is harmless here).
__device__ __forceinline__ unsigned long long ordered_bits(double x)
{
    const unsigned long long b = (unsigned long long)__double_as_longlong(x);
    return (b >> 63) ? ~b : (b | 0x8000000000000000ull);
}

__device__ __forceinline__ unsigned long long umin64(unsigned long long a, unsigned long long b)
{
    return a < b ? a : b;
}

// Group-wide lexicographic min of (D, g): smallest D, lowest g among equal D.  The double is
// reduced as its order-preserving integer image (no fp64 compares), then the lowest g among the
// lanes that hold that minimum.
template <int WPC>
__device__ __forceinline__ int group_argmin(double D, int g, Scratch &sc, int gw, int lane,
                                            int grp)
{
    unsigned long long key = ordered_bits(D);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) key = umin64(key, __shfl_xor_sync(0xffffffffu, key, o));
    if (WPC > 1) {
        gsync<WPC>(grp);
        if (lane == 0) sc.key[gw] = key;
        gsync<WPC>(grp);
        key = sc.key[0];
#pragma unroll
        for (int i = 1; i < WPC; ++i) key = umin64(key, sc.key[i]);
    }
    int cand = (ordered_bits(D) == key) ? g : INT_MAX;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cand = min(cand, __shfl_xor_sync(0xffffffffu, cand, o));
    if (WPC > 1) {
        gsync<WPC>(grp);
        if (lane == 0) sc.g[gw] = cand;
        gsync<WPC>(grp);
        cand = sc.g[0];
#pragma unroll
        for (int i = 1; i < WPC; ++i) cand = min(cand, sc.g[i]);
    }
    return cand;
}

// In-place suffix sums over items t in [t0, t1) by the whole group: item t <- sum of items
// u >= t, for a 64-bit and a 32-bit quantity.  Each thread owns a contiguous block; block totals
// are combined with a shuffle scan inside each warp and scratch across warps.
template <int WPC, typename Load, typename Store>
__device__ __forceinline__ void group_suffix_scan(int t0, int t1, Load load, Store store,
                                                  Scratch &sc, int gw, int lane, int grp)
{
    constexpr int NT = WPC * 32;
    const int gt = gw * 32 + lane;
    const int n = t1 - t0;
    const int per = (n + NT - 1) / NT;
    const int b0 = t0 + min(n, gt * per), b1 = t0 + min(n, gt * per + per);
    unsigned long long sp = 0;
    long long sn = 0;
    for (int t = b0; t < b1; ++t) {
        unsigned long long p;
        long long q;
        load(t, p, q);
        sp += p;
        sn += q;
    }
    unsigned long long xp = sp;   // inclusive scan toward lower lanes
    long long xn = sn;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long yp = __shfl_down_sync(0xffffffffu, xp, o);
        const long long yn = __shfl_down_sync(0xffffffffu, xn, o);
        if (lane + o < 32) {
            xp += yp;
            xn += yn;
        }
    }
    unsigned long long rp = xp - sp;   // blocks of higher lanes in this warp
    long long rn = xn - sn;
    if (WPC > 1) {
        gsync<WPC>(grp);
        if (lane == 0) {
            sc.sp[gw] = xp;   // warp total
            sc.sn[gw] = xn;
        }
        gsync<WPC>(grp);
#pragma unroll
        for (int w = 0; w < WPC; ++w)
            if (w > gw) {
                rp += sc.sp[w];
                rn += sc.sn[w];
            }
    }
    for (int t = b1 - 1; t >= b0; --t) {
        unsigned long long p;
        long long q;
        load(t, p, q);
        rp += p;
        rn += q;
        store(t, rp, rn);
    }
}

// The same suffix sum by `nw` warps of a group (sw = 0..nw-1, contiguous blocks in warp order),
// which meet at named barrier `bar_id` (nw * 32 threads) to combine the warp totals in `sc`.
template <typename Load, typename Store>
__device__ __forceinline__ void warps_suffix_scan(int t0, int t1, Load load, Store store,
                                                  Scratch &sc, int nw, int sw, int lane, int bar_id)
{
    const int nt = nw * 32, st = sw * 32 + lane;
    const int n = t1 - t0;
    const int per = (n + nt - 1) / nt;
    const int b0 = t0 + min(n, st * per), b1 = t0 + min(n, st * per + per);
    unsigned long long sp = 0;
    long long sn = 0;
    for (int t = b0; t < b1; ++t) {
        unsigned long long p;
        long long q;
        load(t, p, q);
        sp += p;
        sn += q;
    }
    unsigned long long xp = sp;   // inclusive scan toward lower lanes
    long long xn = sn;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long yp = __shfl_down_sync(0xffffffffu, xp, o);
        const long long yn = __shfl_down_sync(0xffffffffu, xn, o);
        if (lane + o < 32) {
            xp += yp;
            xn += yn;
        }
    }
    unsigned long long rp = xp - sp;   // blocks of higher lanes in this warp
    long long rn = xn - sn;
    if (nw > 1) {
        asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "r"(nt) : "memory");
        if (lane == 0) {
            sc.sp[sw] = xp;   // warp total
            sc.sn[sw] = xn;
        }
        asm volatile("bar.sync %0, %1;" ::"r"(bar_id), "r"(nt) : "memory");
        for (int w = sw + 1; w < nw; ++w) {
            rp += sc.sp[w];
            rn += sc.sn[w];
        }
    }
    for (int t = b1 - 1; t >= b0; --t) {
        unsigned long long p;
        long long q;
        load(t, p, q);
        rp += p;
        rn += q;
        store(t, rp, rn);
    }
}

// |r| as a 64-bit fixed-point integer R = |r| * 2^S, from the fp32 bits.  Exact whenever
// |r| * 2^S is an integer, i.e. for every element large enough to take a nonzero code; smaller
// elements are truncated (their P contribution is zero anyway).
__device__ __forceinline__ long long fixed_point(float a, int S)
{
    const uint32_t bits = __float_as_uint(a);
    const int E = (int)(bits >> 23);
    const long long M = (long long)((bits & 0x7FFFFFu) | (E ? 0x800000u : 0u));
    const int sh = (E ? E : 1) - 150 + S;   // a = M * 2^((E ? E : 1) - 150)
    if (sh >= 0) return M << sh;
    return sh > -40 ? (M >> -sh) : 0;
}

// The same for a normal |r| whose shift is known to be in [0, 40) (lattice elements: |r| >=
// smax / 2G, scaled to lat_bits): no branches.
__device__ __forceinline__ unsigned long long fixed_point_lat(float a, int S)
{
    const uint32_t bits = __float_as_uint(a);
    const unsigned long long M = (unsigned long long)((bits & 0x7FFFFFu) | 0x800000u);
    return M << ((int)(bits >> 23) - 150 + S);
}

// 2^k as a double, built from its bits (k within the normal range).
__device__ __forceinline__ double pow2d(int k)
{
    return __longlong_as_double((long long)(1023 + k) << 52);
}

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

// Decision value D(s) = s (s N - 2 P) with P = Pfix * 2^-S, in double.
__device__ __forceinline__ double decision(float s, long long Pfix, long long N, double down)
{
    const double sd = (double)s;
    const double T = __fma_rn(sd, (double)N, -2.0 * ((double)Pfix * down));
    return __dmul_rn(sd, T);
}

__device__ __forceinline__ void kahan_add(float &sum, float &comp, float x)
{
    const float y = __fsub_rn(x, comp);
    const float t = __fadd_rn(sum, y);
    comp = __fsub_rn(__fsub_rn(t, sum), y);
    sum = t;
}

// Exact 64-bit shared-memory accumulation from two 32-bit atomics: the low word's returned old
// value shows whether it wrapped, and the carry goes into the high word with the high half.
__device__ __forceinline__ void add64(unsigned int *lo_word, unsigned int *hi_word,
                                      unsigned int Rlo, unsigned int Rhi)
{
    const unsigned int old = atomicAdd(lo_word, Rlo);
    const unsigned int carry = (old + Rlo < old) ? 1u : 0u;
    if (Rhi + carry) atomicAdd(hi_word, Rhi + carry);
}

__device__ __forceinline__ void add_event(unsigned int *hLo, unsigned int *hHi, int *hN, int T,
                                          unsigned int Rlo, unsigned int Rhi, int L, int G)
{
    if (!MPQ_IN(T, G + 1)) return;
    add64(&hLo[T], &hHi[T], Rlo, Rhi);
    atomicAdd(&hN[T], 2 * L - 1);
}

__device__ __forceinline__ long long bin64(const unsigned int *hLo, const unsigned int *hHi, int t)
{
    return (long long)(((unsigned long long)hHi[t] << 32) | hLo[t]);
}

// Int64 -> fp32 without the fp64 pipe: two exact 32-bit halves, three roundings in total.
__device__ __forceinline__ float i64_to_f32(long long x)
{
    const float hi = (float)(int)(x >> 32);
    const float lo = (float)(unsigned int)x;
    return __fmaf_rn(hi, 4294967296.0f, lo);
}

// Columns of tensor memory a CTA allocates for its groups' residual rows in the TM build: a power of
// two, at least 32.
__host__ __device__ constexpr uint32_t tm_alloc_cols(int cols)
{
    return cols <= 32 ? 32u : cols <= 64 ? 64u : cols <= 128 ? 128u : cols <= 256 ? 256u : 512u;
}
constexpr int TM_MAX_D = 4096;   // TM build: d a multiple of 4 x 128, at most 32 columns per group

// MINB: CTAs per SM the register budget allows (4: 64 registers per thread; 3: up to 85, for the
// layers whose shared memory holds an SM to 3 CTAs anyway).
// TM (4-warp groups on the lattice form): each channel's residual row lives in tensor memory, one
// lane per thread -- thread gt of the group holds elements gt + 128 c in columns c of its lane --
// instead of shared memory, which then holds only the lattice and bins (c5: 4 CTAs per SM instead
// of 3).  A group without a channel (the last CTA's) repeats the CTA's last channel without writing
// anything, so that every thread reaches the end, where tensor memory is released.
template <int WPC, bool CUSTOM, bool LAT, bool TABLE, int MINB = 4, bool TM = false>
__global__ void __launch_bounds__(QTHREADS, MINB)
quantize_kernel(const float *__restrict__ W, int C, int d, int qmax, int G, const Grid<CUSTOM> grid,
                int k_max, int8_t *__restrict__ codes, float *__restrict__ scales,
                float *__restrict__ resid_sq, float *__restrict__ residuals,
                float *__restrict__ rmax, int hbits,
                int lat_bits, int cnt_bit, int nc)
{
    const int nb = LAT ? 2 * G * qmax + 1 : 0;   // lattice buckets: floor(2u) in [0, 2 G Qmax]
    constexpr int NT = WPC * 32;
    constexpr int COPIES = LAT ? 1 : WPC;         // event bin copies per group
    constexpr int GPC = 8 / WPC;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    __shared__ Scratch scratch[GPC];
    __shared__ float s_hinv[QMAX_LIMIT + 1];   // 1 / (L - 1/2): threshold estimates only

    static_assert(!TM || (WPC == 4 && LAT && !CUSTOM), "tensor-memory rows: 4-warp lattice groups");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = warp / WPC, gw = warp % WPC, gt = gw * 32 + lane;
    const int k_own = blockIdx.x * GPC + grp;
    const bool ghost = TM && k_own >= C;          // TM: a group without a channel repeats C - 1
    const int k = ghost ? C - 1 : k_own;
    const int dsm = TM ? 0 : d;                   // residual words per group in shared memory
    const float qmaxf = (float)qmax;
    // the grid fractions f_g and fl(1 / f_g): a table, or (linear grid, when the table's 2G words
    // would cost a CTA per SM) computed where needed
    static_assert(TABLE || !CUSTOM, "a caller's grid needs the table");
    float *ftab = reinterpret_cast<float *>(smem_raw);   // [G] f_g, then [G] fl(1 / f_g)
    for (int L = threadIdx.x; L <= qmax; L += QTHREADS) s_hinv[L] = 1.0f / ((float)L - 0.5f);
    if (TABLE)
        for (int g = threadIdx.x; g < G; g += QTHREADS) {
            const float f = grid.frac(g, G);
            ftab[g] = f;
            ftab[G + g] = __frcp_rn(f);
        }
    // the last group's region ends the carve-up of dynamic shared memory
    if (!MPQ_CHECK_SMEM_END((TABLE ? 8 * (size_t)G : 0) + (LAT ? lut_bytes(nb) : 0) +
                            4 * (size_t)GPC * group_words(G, dsm, COPIES, nc)))
        return;
    auto fg = [&](int g) -> float { return TABLE ? ftab[g] : grid.frac(g, G); };
    auto fi = [&](int g) -> float { return TABLE ? ftab[G + g] : __frcp_rn(grid.frac(g, G)); };
    // Lattice compression: only the positions (g+1)(2L-1) are read, so bucket b is stored at the
    // index of the largest position <= b (lut[b]; nc positions in all): the suffix sum at a
    // position's index is the sum over the buckets at or above it, as before.
    unsigned short *lut = reinterpret_cast<unsigned short *>(ftab + (TABLE ? 2 * G : 0));
    if (LAT) {
        for (int b = threadIdx.x; b < nb; b += QTHREADS) lut[b] = 0;
        __syncthreads();
        for (int x = threadIdx.x; x < G * qmax; x += QTHREADS) {
            const int g = x / qmax, L = x - g * qmax + 1;
            if (MPQ_IN((g + 1) * (2 * L - 1), nb)) lut[(g + 1) * (2 * L - 1)] = 1;
        }
        __syncthreads();
        if (warp == 0) {   // inclusive count of positions, minus one
            int run = 0;
            for (int b0 = 0; b0 < nb; b0 += 32) {
                const int b = b0 + lane;
                const int bit = b < nb ? lut[b] : 0;
                const unsigned bal = __ballot_sync(0xffffffffu, bit);
                const int incl = run + __popc(bal & ((2u << lane) - 1u));
                if (b < nb) lut[b] = (unsigned short)(incl - 1);
                run += __popc(bal);
            }
        }
    }
    // TM: the CTA's tensor memory for its groups' rows (warp 0 allocates and releases it)
    __shared__ uint32_t s_tmem;
    const int tcg = TM ? d / NT : 0;               // columns per group
    const uint32_t tcols = tm_alloc_cols(GPC * tcg);
    if (TM && warp == 0) sm100::tmem_alloc(&s_tmem, tcols);
    if (TM) sm100::tc_fence_before();
    __syncthreads();
    if (TM) sm100::tc_fence_after();
    // this thread's lane (the warp's lane quarter) at the group's first column
    const uint32_t taddr = TM ? s_tmem + ((uint32_t)(gw * 32) << 16) + (uint32_t)(grp * tcg) : 0u;
    if (!TM && k >= C) return;   // whole group idle (group-uniform)

    unsigned int *gl = reinterpret_cast<unsigned int *>(
                           reinterpret_cast<unsigned char *>(lut) + (LAT ? lut_bytes(nb) : 0)) +
                       (size_t)grp * group_words(G, dsm, COPIES, nc);
    unsigned int *lat = gl;                         // [nc][2]: R low word, R high | count
    const unsigned cnt_one = 1u << cnt_bit, hmask = cnt_one - 1u;
    unsigned int *gbase = gl + lattice_words(nc);
    // this warp's private bins; copy 0 receives the merged suffix sums
    unsigned int *hLo = gbase + (size_t)(COPIES > 1 ? gw : 0) * 3 * (G + 1);
    unsigned int *hHi = hLo + (G + 1);
    int *hN = reinterpret_cast<int *>(hHi + (G + 1));
    unsigned int *mLo = gbase;
    unsigned int *mHi = mLo + (G + 1);
    int *mN = reinterpret_cast<int *>(mHi + (G + 1));
    float *sr = reinterpret_cast<float *>(gbase + (size_t)3 * (G + 1) * COPIES);
    Scratch &sc = scratch[grp];

    const size_t plane = (size_t)C * d;
    const float *w = W + (size_t)k * d;
    const bool short_share = d <= 64 * NT;
    // rows this short take every candidate directly: G*d code evaluations per step cost less than
    // the lattice's per-step clears, scans and fold over its 2 G Qmax + 1 buckets
    const bool direct = d <= QDIRECT_MAX_D;

    int bad = 0;
    float ssum = 0.0f, scomp = 0.0f, am = 0.0f;
    if constexpr (TM) {
        for (int cc = 0; cc < tcg; cc += 4) {
            float v4[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int j = gt + NT * (cc + u);
                const float v = MPQ_IN((size_t)k * d + j, plane) ? w[j] : 0.0f;
                v4[u] = v;
                bad |= !isfinite(v);
                kahan_add(ssum, scomp, v * v);
                am = fmaxf(am, fabsf(v));
            }
            __syncwarp();
            sm100::tmem_st_32x32b_x4(taddr + cc, v4);
        }
        sm100::tmem_wait_st();
    } else {
        for (int j = gt; j < d; j += NT) {
            const float v = MPQ_IN((size_t)k * d + j, plane) ? w[j] : 0.0f;
            sr[j] = v;
            bad |= !isfinite(v);
            kahan_add(ssum, scomp, v * v);
            am = fmaxf(am, fabsf(v));
        }
    }
    float m = am;
    float r2 = ssum;
    group_max_sum_or<WPC>(m, r2, bad, sc, gw, lane, grp);
    if (WPC == 1) __syncwarp();
    const size_t n_rs = (size_t)C * (k_max + 1), n_codes = (size_t)k_max * plane;
    if (resid_sq && gt == 0 && !ghost && MPQ_IN((size_t)k * (k_max + 1), n_rs))
        resid_sq[(size_t)k * (k_max + 1)] = bad ? NAN : r2;
    if (rmax && gt == 0 && !ghost && MPQ_IN((size_t)k * (k_max + 1), n_rs))
        rmax[(size_t)k * (k_max + 1)] = bad ? NAN : m;

    for (int i = 0; i < k_max; ++i) {
        int8_t *qi = codes + (size_t)i * plane + (size_t)k * d;
        float *ri = residuals ? residuals + (size_t)i * plane + (size_t)k * d : nullptr;
        if (bad) {
            if constexpr (TM) {
                for (int cc = 0; cc < tcg; cc += 4) {
                    float v4[4];
                    __syncwarp();
                    sm100::tmem_ld_32x32b_x4(taddr + cc, v4);
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int j = gt + NT * (cc + u);
                        if (ghost || !MPQ_IN((size_t)i * plane + (size_t)k * d + j, n_codes)) continue;
                        qi[j] = 0;
                        if (ri) ri[j] = v4[u];
                    }
                }
            } else {
                for (int j = gt; j < d; j += NT) {
                    if (!MPQ_IN((size_t)i * plane + (size_t)k * d + j, n_codes)) continue;
                    qi[j] = 0;
                    if (ri) ri[j] = sr[j];
                }
            }
            if (gt == 0 && !ghost) {
                const bool in_s = MPQ_IN((size_t)k * k_max + i, (size_t)C * k_max);
                const bool in_r = MPQ_IN((size_t)k * (k_max + 1) + i + 1, n_rs);
                if (in_s) scales[(size_t)k * k_max + i] = NAN;
                if (resid_sq && in_r) resid_sq[(size_t)k * (k_max + 1) + i + 1] = NAN;
                if (rmax && in_r) rmax[(size_t)k * (k_max + 1) + i + 1] = NAN;
            }
            continue;
        }

        float s_best = 0.0f, inv_best = 0.0f;
        if (m > 0.0f) {
            // candidate scales s_g = fl(f_g * smax) exactly as defined; fl(1/f_g) * fl(1/smax)
            // is within 2^-22 of 1/s_g, which the fast decisions' 2^-20 margin absorbs
            const float smax = __fdiv_rn(m, qmaxf);
            const float ism = __frcp_rn(smax);
            int e;
            frexpf(m, &e);                      // m < 2^e
            // fixed point R = |r| 2^S: on the lattice, exact for every |r| that can reach bucket 1
            // (|r| >= smax / 2G) and below 2^lat_bits; elsewhere sum_j R_j c_j < 2^62
            const bool zs = __fmul_rn(fg(0), smax) == 0.0f;
            const int S = (LAT && !zs) ? lat_bits - e : 62 - e - hbits;
            const float pscale = ldexpf(1.0f, -S - e);   // P 2^-S / 2^e for the fp32 screen
            // lattice elements (|r| >= smax / 2G >= 2^(e - 2 - log2(2 G Qmax))) are normal floats
            // unless max|r| itself is below ~2^-100
            const bool lat_normal = LAT && !zs && e > -100;
            const double down = pow2d(-S);
            const float smax_e = ldexpf(smax, -e);   // smax / 2^e for the fp32 screen
            if (!direct) {
                for (int t = COPIES > 1 ? lane : gt; t <= G; t += COPIES > 1 ? 32 : NT) {
                    hLo[t] = 0u;   // each warp clears its own copy, or the group the shared one
                    hHi[t] = 0u;
                    hN[t] = 0;
                }
                if (LAT) {
                    for (int t = gt; t < 2 * nc; t += NT) lat[t] = 0u;
                    if (gt == 0) sc.nq = 0;
                }
                gsync<WPC>(grp);
            }
            const bool zero_scale = __fmul_rn(fg(0), smax) == 0.0f;   // s_g increases with g

            double bestD = DBL_MAX;
            int bestg = INT_MAX;
            if (!zero_scale) {
                // ---- events: one per (element, level crossed inside the grid)
                const float s0 = __fmul_rn(fg(0), smax), sG = __fmul_rn(fg(G - 1), smax);
                const float i0 = fi(0) * ism, iG = fi(G - 1) * ism;
                const float g_per_a = __fdiv_rn((float)G, smax);   // linear grid: s_g ~ (g+1)/G*smax
                const float g2_per_a = 2.0f * g_per_a;   // 2 fl(a g_per_a) = fl(a g2_per_a) exactly
                long long Pb = 0;
                long long Nb = 0;
                // every level an element crosses inside the grid, one event each
                // the event of level L of an element (c_lo < L <= c_hi): the first g whose code is
                // below L, estimated where s_g crosses a/(L - 1/2), then settled with the exact
                // rule (level_held is monotone in g)
                auto event_level = [&](const float a, const int L, const unsigned int Rlo,
                                       const unsigned int Rhi, const float ag) {
                    int T;
                    if (CUSTOM) {
                        const float f_est = a * s_hinv[L] * ism;
                        int lo = 1, hi = G - 1;
                        while (lo < hi) {
                            const int mid = (lo + hi) >> 1;
                            if (fg(mid) < f_est) lo = mid + 1; else hi = mid;
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
                            add_event(hLo, hHi, hN, T, Rlo, Rhi, L, G);
                            return;
                        }
                    }
#define MPQ_HELD(t) level_held(a, __fmul_rn(fg(t), smax), fi(t) * ism, L)
                    const bool up = (T < G - 1) && MPQ_HELD(T);
                    const bool dn = !up && (T > 1) && !MPQ_HELD(T - 1);
                    if (up) {
                        ++T;
                        while (T < G - 1 && MPQ_HELD(T)) ++T;
                    } else if (dn) {
                        --T;
                        while (T > 1 && !MPQ_HELD(T - 1)) --T;
                    }
#undef MPQ_HELD
                    add_event(hLo, hHi, hN, T, Rlo, Rhi, L, G);
                };
                // every level an element crosses inside the grid, one event each; the levels held
                // at the largest scale go to the base sums
                auto events = [&](const float a) {
                    const int c_hi = code_fast(a, s0, i0, qmaxf);
                    if (c_hi == 0) return;   // code 0 at every scale: no contribution
                    const int c_lo = code_fast(a, sG, iG, qmaxf);
                    const long long R = fixed_point(a, S);
                    Pb += R * (long long)c_lo;
                    Nb += (long long)c_lo * c_lo;
                    const unsigned int Rlo = (unsigned int)R;
                    const unsigned int Rhi = (unsigned int)((unsigned long long)R >> 32);
                    const float ag = a * g_per_a;
                    for (int L = c_lo + 1; L <= c_hi; ++L) event_level(a, L, Rlo, Rhi, ag);
                };
                // 2u within 2^-20 (relative) of an integer: its bucket is not decided exactly
                auto near_lattice = [](float x) { return !(fabsf(x - rintf(x)) > MPQ_FAST_REL * x); };
                if (direct) {
                    // Short rows: every candidate's P_g and N_g straight from the codes, exact
                    // (the codes as the update emits them; P in the same fixed point), into the
                    // merged bins the screen reads, with Pbase = Nbase = 0.
                    for (int g = gt; g < G; g += NT) {
                        const float sg = __fmul_rn(fg(g), smax), ig = fi(g) * ism;
                        long long P = 0, N = 0;
                        for (int j = 0; j < d; ++j) {
                            const float a = fabsf(sr[j]);
                            const int c = code_fast(a, sg, ig, qmaxf);
                            P += fixed_point(a, S) * (long long)c;
                            N += (long long)c * c;
                        }
                        mLo[g + 1] = (unsigned int)P;
                        mHi[g + 1] = (unsigned int)((unsigned long long)P >> 32);
                        mN[g + 1] = (int)N;
                    }
                } else if (LAT) {
                    // Linear grid: level L is held at g iff u >= (g+1)(L - 1/2), u = aG/smax, i.e.
                    // iff floor(2u) >= (g+1)(2L-1), an integer.  Unless 2u lies within 2^-20
                    // (relative) of an integer, one bucket update records the element for every
                    // (g, L) exactly; near a lattice point the per-level events settle each
                    // threshold with the exact rule.  Two elements per pass, for overlap.
                    constexpr int U = TM ? 4 : 2;
                    for (int j0 = gt; j0 < d; j0 += U * NT) {
                        float av[U], u2[U];
                        if constexpr (TM) {   // columns (j0 - gt) / NT .. + 3 of this lane
                            float v4[4];
                            __syncwarp();   // tensor-memory accesses by the converged warp
                            sm100::tmem_ld_32x32b_x4(taddr + (uint32_t)((j0 - gt) / NT), v4);
#pragma unroll
                            for (int u = 0; u < U; ++u) {
                                av[u] = fabsf(v4[u]);
                                u2[u] = av[u] * g2_per_a;
                            }
                        } else {
#pragma unroll
                            for (int u = 0; u < U; ++u) {
                                const int j = j0 + u * NT;
                                av[u] = j < d ? fabsf(sr[j]) : 0.0f;
                                u2[u] = av[u] * g2_per_a;
                            }
                        }
#pragma unroll
                        for (int u = 0; u < U; ++u) {
                            if (av[u] == 0.0f) continue;
                            if (!near_lattice(u2[u])) {
                                const int b = (int)floorf(u2[u]);
                                if (b >= 1) {
                                    // b <= nb - 1: fl(max|r| G / smax) rounds to at most
                                    // G Qmax (1 + 2^-22), below the next integer
                                    if (!MPQ_IN(b, nb)) continue;
                                    const int bb = lut[b];
                                    if (!MPQ_IN(bb, nc)) continue;
                                    // two 32-bit atomics: the low word's old value gives
                                    // its carry, which the high word takes with the count
                                    const unsigned long long R =
                                        lat_normal ? fixed_point_lat(av[u], S)
                                                   : (unsigned long long)fixed_point(av[u], S);
                                    const unsigned Rlo = (unsigned)R;
                                    const unsigned old = atomicAdd(&lat[2 * bb], Rlo);
                                    atomicAdd(&lat[2 * bb + 1], (unsigned)(R >> 32) +
                                                                    (old + Rlo < old ? 1u : 0u) +
                                                                    cnt_one);
                                }
                            } else {
                                // within 2^-20 of a lattice point: queued, and settled level by
                                // level by the whole group after the pass, so that one lane's
                                // exact rule holds neither its warp nor the loop's registers
                                const int slot = atomicAdd(&sc.nq, 1);
                                if (slot < QNEAR) sc.nearq[slot] = av[u];
                            }
                        }
                    }
                    gsync<WPC>(grp);
                    const int nq = sc.nq;
                    if (nq <= QNEAR) {
                        // (queued element, level) pairs over the group's threads
                        for (int it = gt; it < nq * qmax; it += NT) {
                            const int q = it / qmax, L = it - q * qmax + 1;
                            if (!MPQ_IN(q, QNEAR)) continue;
                            const float a = sc.nearq[q];
                            const int c_hi = code_fast(a, s0, i0, qmaxf);
                            if (c_hi == 0) continue;
                            const int c_lo = code_fast(a, sG, iG, qmaxf);
                            const long long R = fixed_point(a, S);
                            if (L == 1) {
                                Pb += R * (long long)c_lo;
                                Nb += (long long)c_lo * c_lo;
                            }
                            if (L > c_lo && L <= c_hi)
                                event_level(a, L, (unsigned int)R,
                                            (unsigned int)((unsigned long long)R >> 32), a * g_per_a);
                        }
                    } else {   // the queue overflowed (never seen): every such element again
                        if constexpr (TM) {
                            for (int cc = 0; cc < tcg; cc += 4) {
                                float v4[4];
                                __syncwarp();
                                sm100::tmem_ld_32x32b_x4(taddr + cc, v4);
#pragma unroll
                                for (int u = 0; u < 4; ++u) {
                                    const float a = fabsf(v4[u]);
                                    if (a != 0.0f && near_lattice(2.0f * (a * g_per_a))) events(a);
                                }
                            }
                        } else {
                            for (int j = gt; j < d; j += NT) {
                                const float a = fabsf(sr[j]);
                                if (a != 0.0f && near_lattice(2.0f * (a * g_per_a))) events(a);
                            }
                        }
                    }
                } else {
                    for (int j = gt; j < d; j += NT) {
                        const float a = fabsf(sr[j]);
                        if (a != 0.0f) events(a);
                    }
                }
                group_sum2<WPC>(Pb, Nb, sc, gw, lane, grp);   // publishes the bins too
                const long long Pbase = Pb, Nbase = Nb;
                // ---- suffix sums over the event bins (private copies, if any, merged into
                // copy 0; warp 0), in place: bin t <- sum of bins u >= t, so P_g = Pbase +
                // bin(g + 1); and over the lattice buckets (warp 1 concurrently, or the whole
                // group afterwards when the lattice is large)
                auto bins_load = [&](int t, unsigned long long &p, long long &q) {
                    long long pp = bin64(mLo, mHi, t);
                    long long nn = mN[t];
#pragma unroll
                    for (int c = 1; c < COPIES; ++c) {
                        const unsigned int *cLo = mLo + (size_t)c * 3 * (G + 1);
                        pp += bin64(cLo, cLo + (G + 1), t);
                        nn += reinterpret_cast<const int *>(cLo + 2 * (G + 1))[t];
                    }
                    p = (unsigned long long)pp;
                    q = nn;
                };
                auto bins_store = [&](int t, unsigned long long p, long long q) {
                    mLo[t] = (unsigned int)p;
                    mHi[t] = (unsigned int)(p >> 32);
                    mN[t] = (int)q;
                };
                auto lat_load = [&](int t, unsigned long long &p, long long &q) {
                    const unsigned hi = lat[2 * t + 1];
                    p = ((unsigned long long)(hi & hmask) << 32) | lat[2 * t];
                    q = hi >> cnt_bit;
                };
                auto lat_store = [&](int t, unsigned long long p, long long q) {
                    lat[2 * t] = (unsigned)p;
                    lat[2 * t + 1] = (unsigned)(p >> 32) | ((unsigned)q << cnt_bit);
                };
                // with the lattice: warp 0 scans the bins while the other warps scan the lattice
                // together (named barrier 8 + grp: gsync takes 0 or 1..4), or one warp both;
                // event-form grids with many bins to merge: the whole group
                if (direct) {
                    // the bins already hold P_g, N_g (group_sum2 above ordered their writes)
                } else if (LAT) {
                    if (gw == 0)
                        group_suffix_scan<1>(1, G + 1, bins_load, bins_store, sc, 0, lane, grp);
                    if (WPC == 1)
                        group_suffix_scan<1>(0, nc, lat_load, lat_store, sc, 0, lane, grp);
                    else if (gw >= 1)
                        warps_suffix_scan(0, nc, lat_load, lat_store, sc, WPC - 1, gw - 1, lane,
                                          8 + grp);
                } else if (G * COPIES > 1024) {
                    group_suffix_scan<WPC>(1, G + 1, bins_load, bins_store, sc, gw, lane, grp);
                } else if (gw == 0) {
                    group_suffix_scan<1>(1, G + 1, bins_load, bins_store, sc, 0, lane, grp);
                }
                if (!direct) gsync<WPC>(grp);
                if (LAT && !direct) {
                    // fold the lattice into the merged bins: bin(g + 1) += sum_L bucket((g+1)(2L-1))
                    for (int g = gt; g < G; g += NT) {
                        long long p = bin64(mLo, mHi, g + 1);
                        long long n = mN[g + 1];
                        for (int L = 1; L <= qmax; ++L) {
                            const int b = lut[(g + 1) * (2 * L - 1)];
                            if (!MPQ_IN(b, nc)) continue;
                            const unsigned hi = lat[2 * b + 1];
                            p += (long long)(((unsigned long long)(hi & hmask) << 32) | lat[2 * b]);
                            n += (long long)(2 * L - 1) * (hi >> cnt_bit);
                        }
                        mLo[g + 1] = (unsigned int)p;
                        mHi[g + 1] = (unsigned int)((unsigned long long)p >> 32);
                        mN[g + 1] = (int)n;
                    }
                    gsync<WPC>(grp);
                }
                // ---- fp32 screen of D / 2^2e = s'(s'N - 2P') with s' = s / 2^e and
                // P' = P 2^-S / 2^e (both O(1) by construction): keep every candidate whose error
                // interval can contain the minimum, then decide among those in double.  The
                // inputs carry at most ~8 roundings of 2^-24, the bound allows 2^-20.
                float upper = FLT_MAX;
                for (int g = gt; g < G; g += NT) {
                    const float sh = fg(g) * smax_e;
                    const float Nf = (float)(int)(Nbase + mN[g + 1]);
                    const float Pf = i64_to_f32(Pbase + bin64(mLo, mHi, g + 1)) * pscale;
                    const float D32 = sh * (sh * Nf - 2.0f * Pf);
                    const float err = sh * (sh * Nf + 2.0f * Pf) * MPQ_FAST_REL;
                    upper = fminf(upper, D32 + err);
                }
                upper = group_min<WPC>(upper, sc, gw, lane, grp);
                for (int g = gt; g < G; g += NT) {
                    const float sh = fg(g) * smax_e;
                    const long long Pg = Pbase + bin64(mLo, mHi, g + 1);
                    const long long Ng = Nbase + mN[g + 1];
                    const float Nf = (float)(int)Ng;
                    const float Pf = i64_to_f32(Pg) * pscale;
                    const float D32 = sh * (sh * Nf - 2.0f * Pf);
                    const float err = sh * (sh * Nf + 2.0f * Pf) * MPQ_FAST_REL;
                    if (D32 - err <= upper) {
                        const double D = decision(__fmul_rn(fg(g), smax), Pg, Ng, down);
                        if (D < bestD) {
                            bestD = D;
                            bestg = g;
                        }
                    }
                }
            } else {
                // ---- direct evaluation (a candidate scale underflowed to 0)
                if constexpr (TM) {
                    // every candidate's P and N from each thread's own elements, summed over the
                    // group in the bins (cleared at the step's start), then decided as below
                    for (int g = 0; g < G; ++g) {
                        const float s = __fmul_rn(fg(g), smax);
                        if (!(s > 0.0f)) continue;   // the same for every thread
                        long long P = 0, N = 0;
                        for (int cc = 0; cc < tcg; cc += 4) {
                            float v4[4];
                            __syncwarp();
                            sm100::tmem_ld_32x32b_x4(taddr + cc, v4);
#pragma unroll
                            for (int u = 0; u < 4; ++u) {
                                const float a = fabsf(v4[u]);
                                const int c = code_mag(a, s, qmaxf);
                                P += fixed_point(a, S) * (long long)c;
                                N += (long long)c * c;
                            }
                        }
                        P = warp_sum(P);
                        N = warp_sum(N);
                        if (lane == 0) {
                            add64(&mLo[g + 1], &mHi[g + 1], (unsigned int)P,
                                  (unsigned int)((unsigned long long)P >> 32));
                            atomicAdd(&mN[g + 1], (int)N);
                        }
                    }
                    gsync<WPC>(grp);
                    for (int g = gt; g < G; g += NT) {
                        const float s = __fmul_rn(fg(g), smax);
                        const double D = s > 0.0f ? decision(s, bin64(mLo, mHi, g + 1), (long long)mN[g + 1], down)
                                                  : 0.0;   // s == 0: all codes 0, E = ||r||^2
                        if (D < bestD) {
                            bestD = D;
                            bestg = g;
                        }
                    }
                } else {
                    for (int g = gt; g < G; g += NT) {
                        const float s = __fmul_rn(fg(g), smax);
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
            }
            int g = group_argmin<WPC>(bestD, bestg, sc, gw, lane, grp);
            if (g < 0 || g >= G) g = G - 1;   // unreachable: every D is finite
            s_best = __fmul_rn(fg(g), smax);
            inv_best = zero_scale ? 0.0f : fi(g) * ism;
        }

        // residual update (Eq. 7) and code emission; also the next step's max |r|
        ssum = 0.0f;
        scomp = 0.0f;
        am = 0.0f;
        // one element: its code (stored), its new residual (returned), ||r||^2 and max |r|
        auto update = [&](float v, int j) -> float {
            int q = 0;
            if (s_best > 0.0f) {
                // the code of Eq. 8 as a float (an exact small integer) with the residual's sign
                const float c = (inv_best > 0.0f) ? code_fast_f(fabsf(v), s_best, inv_best, qmaxf)
                                                  : fminf(rintf(__fdiv_rn(fabsf(v), s_best)), qmaxf);
                const float qf = copysignf(c, v);
                q = (int)qf;
                v = __fmaf_rn(-s_best, qf, v);
            }
            const bool in = !ghost && MPQ_IN((size_t)i * plane + (size_t)k * d + j, n_codes);
            if (in) qi[j] = (int8_t)q;
            if (ri && in) ri[j] = v;
            // ||r||^2: a thread's share of at most 64 squares summed plainly (relative error
            // below 2^-18 with the group's tree), longer shares compensated
            if (short_share) ssum = __fmaf_rn(v, v, ssum);
            else kahan_add(ssum, scomp, v * v);
            am = fmaxf(am, fabsf(v));
            return v;
        };
        // Four elements at a time where the reciprocal is usable: their signed codes
        // clamp(rint(v (1/s))) without a branch, all four redone with the correctly rounded division
        // when any lane's quotient lies near a rounding boundary (a warp-uniform branch), so that the
        // four elements' arithmetic interleaves.  The codes are Eq. 8's either way.
        const bool fastq = s_best > 0.0f && inv_best > 0.0f;
        const float qlim = qmaxf + 1.0f, tband = 0.5f - MPQ_FAST_REL * (qlim + 1.0f);
        auto update4 = [&](float (&v4)[4], int j0) {   // elements j0 + NT u, every lane of the warp
            float q4[4];
            bool unsure = false;
#pragma unroll
            for (int u = 0; u < 4; ++u) q4[u] = code_signed_fast(v4[u], inv_best, qmaxf, qlim, tband, unsure);
            if (__any_sync(0xffffffffu, unsure)) {
#pragma unroll
                for (int u = 0; u < 4; ++u) q4[u] = code_signed_exact(v4[u], s_best, qmaxf);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int j = j0 + NT * u;
                const float v = __fmaf_rn(-s_best, q4[u], v4[u]);
                const bool in = !ghost && MPQ_IN((size_t)i * plane + (size_t)k * d + j, n_codes);
                if (in) qi[j] = (int8_t)(int)q4[u];
                if (ri && in) ri[j] = v;
                if (short_share) ssum = __fmaf_rn(v, v, ssum);
                else kahan_add(ssum, scomp, v * v);
                am = fmaxf(am, fabsf(v));
                v4[u] = v;
            }
        };
        if constexpr (TM) {
            for (int cc = 0; cc < tcg; cc += 4) {
                float v4[4];
                __syncwarp();
                sm100::tmem_ld_32x32b_x4(taddr + cc, v4);
                if (fastq) {
                    update4(v4, gt + NT * cc);
                } else {
#pragma unroll
                    for (int u = 0; u < 4; ++u) v4[u] = update(v4[u], gt + NT * (cc + u));
                }
                __syncwarp();
                sm100::tmem_st_32x32b_x4(taddr + cc, v4);
            }
            sm100::tmem_wait_st();
        } else {
            int j = gt;
            if (fastq) {
                // groups of four while the warp's last lane still has all four (warp-uniform)
                for (; j - lane + 31 + 3 * NT < d; j += 4 * NT) {
                    float v4[4] = {sr[j], sr[j + NT], sr[j + 2 * NT], sr[j + 3 * NT]};
                    update4(v4, j);
#pragma unroll
                    for (int u = 0; u < 4; ++u) sr[j + NT * u] = v4[u];
                }
            }
            for (; j < d; j += NT) sr[j] = update(sr[j], j);
        }
        if (gt == 0 && !ghost && MPQ_IN((size_t)k * k_max + i, (size_t)C * k_max))
            scales[(size_t)k * k_max + i] = s_best;
        m = am;
        r2 = ssum;
        int none = 0;
        group_max_sum_or<WPC>(m, r2, none, sc, gw, lane, grp);   // orders the sr[] writes too
        if (WPC == 1) __syncwarp();
        const bool in_r = MPQ_IN((size_t)k * (k_max + 1) + i + 1, n_rs);
        if (resid_sq && gt == 0 && !ghost && in_r) resid_sq[(size_t)k * (k_max + 1) + i + 1] = r2;
        if (rmax && gt == 0 && !ghost && in_r) rmax[(size_t)k * (k_max + 1) + i + 1] = m;
    }
    if constexpr (TM) {
        // every group is done with tensor memory before it is released
        sm100::tc_fence_before();
        __syncthreads();
        if (warp == 0) {
            sm100::tc_fence_after();
            sm100::tmem_dealloc(s_tmem, tcols);
        }
    }
}

int ceil_log2(long long x)
{
    int b = 0;
    while ((1LL << b) < x) ++b;
    return b;
}

// Bit layout of the lattice buckets (2 G Qmax + 1 of them): R = |r| 2^S < 2^lat_bits, exact for
// every |r| >= smax / 2G (the smallest magnitude that reaches bucket 1: its exponent is at least
// e - 2 - ceil(log2(2 G Qmax)) for max|r| < 2^e, so 25 + that many bits hold its mantissa, one
// more for margin); a bucket's high word holds its R sum's high part plus carries (at most
// d 2^(lat_bits - 32) + d) below bit cnt_bit and its count (at most d) above.  Returns false when
// the two fields do not fit one word (the event form runs then).
struct LatBits {
    int lat_bits, cnt_bit;
    int nc;   // distinct lattice positions (g+1)(2L-1)
};

int lattice_positions(int G, int qmax)
{
    std::vector<char> seen((size_t)2 * G * qmax + 1, 0);
    int n = 0;
    for (int g = 1; g <= G; ++g)
        for (int L = 1; L <= qmax; ++L) {
            char &c = seen[(size_t)g * (2 * L - 1)];
            if (!c) {
                c = 1;
                ++n;
            }
        }
    return n;
}

bool lattice_bits(int d, int qmax, int G, LatBits *lb)
{
    lb->lat_bits = 26 + ceil_log2(2LL * G * qmax);
    const long long hi_part = lb->lat_bits > 32 ? (1LL << (lb->lat_bits - 32)) - 1 : 0;
    const long long hi_max = (long long)d * hi_part + d;
    lb->cnt_bit = ceil_log2(hi_max + 1);
    return lb->cnt_bit + ceil_log2((long long)d + 1) <= 32;
}

template <int WPC, bool CUSTOM, bool LAT, bool TABLE, int MINB = 4, bool TM = false>
mpq_status launch_wpc(const float *W, int C, int d, int qmax, int G, const Grid<CUSTOM> &grid,
                      int k_max, int8_t *codes, float *scales, float *resid_sq, float *residuals,
                      float *rmax, int hbits, LatBits lb, size_t smem, cudaStream_t stream)
{
    constexpr int GPC = 8 / WPC;
    cudaError_t e = cudaFuncSetAttribute(quantize_kernel<WPC, CUSTOM, LAT, TABLE, MINB, TM>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess) {
        quantize_kernel<WPC, CUSTOM, LAT, TABLE, MINB, TM><<<(C + GPC - 1) / GPC, QTHREADS, smem, stream>>>(
            W, C, d, qmax, G, grid, k_max, codes, scales, resid_sq, residuals, rmax, hbits, lb.lat_bits,
            lb.cnt_bit, lb.nc);
        e = cudaGetLastError();
    }
    return cuda_status(e, "quantize kernel launch");
}

// CTAs of a quantize kernel that fit on one SM with `smem` bytes of dynamic shared memory.
template <int WPC, bool CUSTOM, bool LAT, bool TABLE, int MINB = 4, bool TM = false>
int quantize_ctas_per_sm(size_t smem)
{
    int n = 0;
    if (cudaFuncSetAttribute(quantize_kernel<WPC, CUSTOM, LAT, TABLE, MINB, TM>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, quantize_kernel<WPC, CUSTOM, LAT, TABLE, MINB, TM>,
                                                      QTHREADS, smem) != cudaSuccess)
        n = 0;
    (void)cudaGetLastError();
    return n;
}

template <int WPC, bool CUSTOM>
mpq_status launch_lat(bool lat, const float *W, int C, int d, int qmax, int G,
                      const Grid<CUSTOM> &grid, int k_max, int8_t *codes, float *scales,
                      float *resid_sq, float *residuals, float *rmax, int hbits, LatBits lb,
                      size_t smem, cudaStream_t stream)
{
    if constexpr (!CUSTOM) {
        if (lat) {
            // the lattice form on the linear grid: no grid table when that fits one more CTA on
            // an SM (it costs some arithmetic per candidate otherwise)
            const size_t notab = smem - (size_t)2 * G * sizeof(float);
            const int n_notab = quantize_ctas_per_sm<WPC, false, true, false>(notab);
            const int n_tab = quantize_ctas_per_sm<WPC, false, true, true>(smem);
            if constexpr (WPC == 4) {
                // residual rows in tensor memory where that fits more CTAs on an SM (their columns
                // included: at most 512 per SM)
                if (d % (4 * 128) == 0 && d <= TM_MAX_D) {
                    const size_t tm_smem = smem - (size_t)(8 / WPC) * 4 *
                                                      (group_words(G, d, 1, lb.nc) - group_words(G, 0, 1, lb.nc));
                    // (the occupancy query reports one CTA per SM for any kernel that allocates
                    // tensor memory, so the count is the same kernel's without it: registers and
                    // shared memory, then the columns)
                    const int cols = (int)tm_alloc_cols((8 / WPC) * d / 128);
                    const int n_tm = std::min(quantize_ctas_per_sm<WPC, false, true, true>(tm_smem), 512 / cols);
                    if (n_tm > n_tab && n_tm > n_notab)
                        return launch_wpc<WPC, false, true, true, 4, true>(W, C, d, qmax, G, grid, k_max,
                                                                           codes, scales, resid_sq, residuals,
                                                                           rmax, hbits, lb, tm_smem, stream);
                }
            }
            // where shared memory holds an SM to 3 CTAs or fewer, the build with more registers per
            // thread (no spills, more loads in flight) costs no occupancy (c5: 2 % faster)
            if (n_notab > n_tab) {
                if constexpr (WPC >= 4)
                    if (n_notab <= 3)
                        return launch_wpc<WPC, false, true, false, 3>(W, C, d, qmax, G, grid, k_max,
                                                                      codes, scales, resid_sq, residuals,
                                                                      rmax, hbits, lb, notab, stream);
                return launch_wpc<WPC, false, true, false>(W, C, d, qmax, G, grid, k_max, codes,
                                                           scales, resid_sq, residuals, rmax, hbits, lb,
                                                           notab, stream);
            }
            if constexpr (WPC >= 4)
                if (n_tab >= 1 && n_tab <= 3)
                    return launch_wpc<WPC, false, true, true, 3>(W, C, d, qmax, G, grid, k_max, codes,
                                                                 scales, resid_sq, residuals, rmax, hbits,
                                                                 lb, smem, stream);
            return launch_wpc<WPC, false, true, true>(W, C, d, qmax, G, grid, k_max, codes, scales,
                                                      resid_sq, residuals, rmax, hbits, lb, smem, stream);
        }
    }
    return launch_wpc<WPC, CUSTOM, false, true>(W, C, d, qmax, G, grid, k_max, codes, scales,
                                                resid_sq, residuals, rmax, hbits, lb, smem, stream);
}

template <bool CUSTOM>
mpq_status launch_grid(const float *W, int C, int d, int qmax, int G, const Grid<CUSTOM> &grid,
                       int k_max, int8_t *codes, float *scales, float *resid_sq, float *residuals,
                       float *rmax, cudaStream_t stream)
{
    const int hbits = ceil_log2((long long)d * qmax) + 1;
    // lattice form on the linear grid when its buckets fit (32 KB) and their fields one word
    LatBits lb;
    const bool lat = !CUSTOM && (long long)2 * G * qmax + 1 <= 4096 && lattice_bits(d, qmax, G, &lb);
    if (!lat) lb = LatBits{0, 31, 0};
    const int nb = lat ? 2 * G * qmax + 1 : 0;
    if (lat) lb.nc = lattice_positions(G, qmax);
    const int nc = lb.nc;
    const size_t per_group = group_words(G, d, 1, nc) * 4;
    const long long smem_cap = max_smem_optin();
    // Warps per channel: enough channels in flight to fill the GPU, at least ~2 elements per
    // lane, and enough warps per SM (24) for the shared memory the channels need -- on layers with
    // thousands of long channels, 4-warp groups (more channels per SM, barriers over fewer warps)
    // measured faster than 8-warp ones (c5's 11008 x 4096 layer: 2.28 -> 2.20 ms).
    const long long warps_gpu = (long long)sm_count() * 32;
    int wpc_c = 1;
    while (wpc_c < 8 && (long long)C * wpc_c < warps_gpu) wpc_c *= 2;
    int wpc_e = 1;
    while (wpc_e < 8 && wpc_e * 64 <= d) wpc_e *= 2;
    const long long groups_per_sm = (long long)(227 * 1024) / (long long)(per_group + 256);
    int wpc_s = 1;
    while (wpc_s < 8 && groups_per_sm * wpc_s < 24) wpc_s *= 2;
    int wpc = wpc_c < wpc_e ? wpc_c : wpc_e;
    if (wpc < wpc_s) wpc = wpc_s;
    for (; wpc <= 8; wpc *= 2) {
        const size_t smem = (size_t)(8 / wpc) * group_words(G, d, lat ? 1 : wpc, nc) * 4 +
                            (size_t)2 * G * sizeof(float) + (lat ? lut_bytes(nb) : 0);
        if ((long long)smem <= smem_cap) {
            switch (wpc) {
            case 1:
                return launch_lat<1, CUSTOM>(lat, W, C, d, qmax, G, grid, k_max, codes, scales,
                                             resid_sq, residuals, rmax, hbits, lb, smem, stream);
            case 2:
                return launch_lat<2, CUSTOM>(lat, W, C, d, qmax, G, grid, k_max, codes, scales,
                                             resid_sq, residuals, rmax, hbits, lb, smem, stream);
            case 4:
                return launch_lat<4, CUSTOM>(lat, W, C, d, qmax, G, grid, k_max, codes, scales,
                                             resid_sq, residuals, rmax, hbits, lb, smem, stream);
            default:
                return launch_lat<8, CUSTOM>(lat, W, C, d, qmax, G, grid, k_max, codes, scales,
                                             resid_sq, residuals, rmax, hbits, lb, smem, stream);
            }
        }
    }
    set_error("d = %d, G = %d need %zu bytes of shared memory per channel", d, G, per_group);
    return MPQ_ERR_UNSUPPORTED;
}

}  // namespace

mpq_status launch_quantize(const float *W, int C, int d, int qmax, int G, const GridFrac *grid,
                           int k_max, int8_t *codes, float *scales, float *resid_sq,
                           float *residuals, float *rmax, cudaStream_t stream)
{
    if (grid) {
        Grid<true> g;
        g.gf = *grid;
        return launch_grid<true>(W, C, d, qmax, G, g, k_max, codes, scales, resid_sq, residuals,
                                 rmax, stream);
    }
    return launch_grid<false>(W, C, d, qmax, G, Grid<false>(), k_max, codes, scales, resid_sq,
                              residuals, rmax, stream);
}

}  // namespace mpq
