// Output error (Sec. 3.3, Eq. 11) as a CTA-pair tcgen05 contraction:
//   err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2,  n = 0..k_max.
//
// This file holds the contraction for the output error entry point with a fixed range table (X
// split by the producers: it needs no scratch beyond that table); the output error with pooled
// scratch and the clipping search run output_error_f16.cu, the same contraction with X split
// ahead and the layout its measurements favoured.
//
// Y = R X^T with R the C*(k_max+1) residual vectors and X the N calibration rows (length d);
// err is the row-wise mean of Y^2.  Two CTAs on neighbouring SMs (cluster ranks 2p, 2p+1) form one
// UMMA of M = 256 residual vectors by N = 256 calibration rows: each CTA holds 128 vectors (whole
// channels: floor(128/(k_max+1)) of them) as its half of A and 128 calibration rows as its half of
// B, and receives its 128 vectors x all 256 rows in its own tensor memory.  Per flop, this halves
// the operand bytes each SM's tensor core reads and the residual vectors each SM regenerates,
// compared with one CTA computing 256 vectors x 128 rows alone.
//
// Precision.  Greedy residuals: pair_range_kernel first measures max|X| and max|r| of every residual
// vector; each operand is scaled by the power of two 2^e that puts its largest element in
// [2^14, 2^15) and split into fp16 hi = fl16(x) and lo = fl16(x - hi), and Y = hi*hi + hi*lo + lo*hi
// runs on kind::f16 (fp32 accumulate) -- 22 significant bits per operand like a tf32 hi/lo split,
// at twice the tf32 rate; the reduction multiplies each mean by 2^-2(e_X + e_v) exactly, in double.
// The accumulator restarts every 256 elements of d and the epilogue folds each segment into fp32
// running sums in tensor memory (columns [0, 256) segment, [256, 512) running sums), since the
// tensor core's accumulation truncates.
//
// Input: one thread per CTA streams each K chunk's X rows, W rows and codes into a ring of raw
// shared-memory slots with TMA tile copies (rows past N and channels past C read as zeros).  Eight
// producer warps split X into the B tiles and regenerate the residuals r_{n+1} = r_n - s_n q_n
// (Eq. 7) from W, codes and scales into the A tiles (128-byte swizzled, K-major); residuals never
// exist in global memory.  Two 64 KB tile sets hold the stages: a 32-element chunk fills a 64-byte
// half of every row (4 stages).
// Both CTAs' producers report a full stage to the even CTA, whose MMA
// thread issues the pair MMAs and signals both CTAs (multicast commits) when a stage or a segment
// is consumed.  Eight epilogue warps per CTA (one per TMEM lane quarter and column half) drain the
// segments; a segment is restarted only once both CTAs' epilogues have released it.
//
// Row tiles (256 rows) are split over the pairs of a cluster of up to 8 CTAs; ranks 0 and 1 add
// their peers' partial sums from distributed shared memory in rank order.  Every wait is bounded;
// on a timeout the kernel records MPQ_TIMEOUT_OUTPUT_ERROR, unwinds and the outputs read NaN.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>

#include "mpq_internal.cuh"
#include "pair_common.cuh"
#include "sm100.cuh"
#include "tf32_operands.cuh"
#include "waits.cuh"

MPQ_CHECKED_UNIT("output_error_pair.cu");

namespace mpq {
namespace {

using namespace sm100;

constexpr int P_VEC = 128;                      // residual vectors per CTA (TMEM lanes)
constexpr int P_ROWS = 128;                     // calibration rows per CTA
constexpr int P_N = 2 * P_ROWS;                 // rows per pair row tile (UMMA N)
constexpr int P_KC = 32;                        // fp32 per K chunk = one 128-byte swizzle row
constexpr int P_KC4 = P_KC / 4;
constexpr int P_TILE = 128 * P_KC * 4;          // 16 KB: one 128-row operand tile
constexpr int P_OFF_A_HI = 0;
constexpr int P_OFF_A_LO = P_TILE;
constexpr int P_OFF_B_HI = 2 * P_TILE;
constexpr int P_OFF_B_LO = 3 * P_TILE;
constexpr int P_STAGE_BYTES = 4 * P_TILE;       // 64 KB: one set of A hi/lo, B hi/lo tiles
constexpr int P_TILE_SETS = 2;
constexpr int P_MAX_STAGES = 4;
constexpr int P_EPI_WARPS = 8;                  // two per TMEM lane quarter, one per column half

// fp16 operands: a K chunk of 32 elements fills half of each 128-byte row (64 bytes), so the two
// tile sets hold 4 stages, and the accumulator restarts every 8 chunks (256 elements).
constexpr int P_STAGES = 4;
constexpr int P_SEG = 8;                        // chunks per accumulation segment

// Warp roles: producers first, then the epilogue warps (warp % 4 selects TMEM lanes, so the
// producer count is a multiple of 4), the MMA warp and the TMA warp.
struct PRoles {
    static constexpr int PROD_WARPS = 8;
    static constexpr int PROD_THREADS = PROD_WARPS * 32;
    static constexpr int EPI_WARP0 = PROD_WARPS;
    static constexpr int MMA_WARP = EPI_WARP0 + P_EPI_WARPS;
    static constexpr int TMA_WARP = MMA_WARP + 1;
    static constexpr int THREADS = (TMA_WARP + 1) * 32;   // 576
    static_assert(PROD_WARPS % 4 == 0, "epilogue warps start at a TMEM lane quarter boundary");
};
constexpr uint32_t P_TMEM_COLS = 512;
constexpr uint32_t P_RUN_COL = 256;
constexpr int P_MAX_RAW = 3;
constexpr int P_SMEM_LIMIT = 232448;            // opt-in shared memory per CTA on sm_100 parts

struct PairCtrl {
    uint64_t full[P_MAX_STAGES];  // even CTA: both CTAs' producer warps
    uint64_t empty[P_MAX_STAGES]; // both CTAs: pair MMA commit
    uint64_t raw_full[P_MAX_RAW];
    uint64_t raw_empty[P_MAX_RAW];
    uint64_t segfull;             // both CTAs: pair MMA commit
    uint64_t segempty;            // even CTA: both CTAs' epilogue warps (16 arrivals)
    uint64_t done;                // even CTA
    uint32_t tmem_base;
    int abort;
    double part[2][P_VEC];        // per column half: sum over the rows' y^2
    float vscale[P_VEC];          // 2^e per residual vector, 2^e for X
    int vexp[P_VEC];
    float xscale;
    int xexp;
};
constexpr int P_CTRL_BYTES = (sizeof(PairCtrl) + 1023) / 1024 * 1024;
constexpr int P_BASE_SMEM = 1024 /* alignment slack */ + P_CTRL_BYTES + P_TILE_SETS * P_STAGE_BYTES;

// Per-KP1 geometry and the raw slot layout, in the order the tile copies write it:
// X chunk [128 rows][32] fp32, W chunk [CH][32] fp32, codes [K][CH][32] int8.  KP1 = k_max + 1
// residual vectors per channel.
template <int KP1>
struct PGeo {
    static constexpr int K = KP1 - 1;
    static constexpr int CH = P_VEC / KP1;
    static constexpr int PT = PRoles::PROD_THREADS;
    static constexpr int ITEMS2 = (CH * (P_KC / 2) + PT - 1) / PT;
    static constexpr int X_ITEMS = (P_ROWS * P_KC4 + PT - 1) / PT;
    static constexpr int RAW_W = P_ROWS * P_KC * 4;
    static constexpr int RAW_Q = (RAW_W + CH * P_KC * 4 + 127) / 128 * 128;
    static constexpr uint32_t RAW_TX = P_ROWS * P_KC * 4 + CH * P_KC * 4 + K * CH * P_KC;
    static constexpr int RAW_BYTES = (RAW_Q + K * CH * P_KC + 1023) / 1024 * 1024;
    static constexpr int RAW_FIT = (P_SMEM_LIMIT - P_BASE_SMEM) / RAW_BYTES;
    static constexpr int RAW_STAGES = RAW_FIT < P_MAX_RAW ? RAW_FIT : P_MAX_RAW;
    static constexpr int SMEM = P_BASE_SMEM + RAW_STAGES * RAW_BYTES;
    static_assert(K >= 1, "at least one point");
    static_assert(RAW_STAGES >= 2, "raw ring needs two slots");
};

// fp16 operand stores fill 64-byte half rows, and the 128-byte swizzle puts a half row in banks
// 0-15 or 16-31 by bit 2 of its row.  A store wavefront serves 128 bytes: a half warp's 8-byte
// stores, or a whole warp's 4-byte stores.  So that each of them reaches both bank halves:
// X item q (8 bytes per operand half) of a warp's 32 items goes to rows r, r+4 (lanes 0-15) and
// r+1, r+5 (lanes 16-31) of an 8-row atom (the residual items' channels are paired by
// pair_channel for the same reason).
__device__ __forceinline__ int pair_x_item(int q)
{
    const int g = q >> 5, j = (q & 31) >> 3;
    const int row = (g >> 1) * 8 + (g & 1) * 2 + (j >> 1) + (j & 1) * 4;
    return row * P_KC4 + (q & 7);
}

// Raw slot -> operand stage (tile set `sb`, row half `hh`): X rows -> B tiles; for every (channel,
// element pair) item the residuals -> A tiles: r_0 = w, r_{n+1} = r_n - s_n q_n (Eq. 7).  Operands
// are scaled by 2^e first (xs for X, vf per residual vector), which the reduction undoes exactly.
template <int KP1>
__device__ __forceinline__ void pair_consume(uint32_t slot, uint32_t sb, int hh, int pt, int nch,
                                             const int (&chs)[PGeo<KP1>::ITEMS2],
                                             const float (&sc)[PGeo<KP1>::ITEMS2][KP1 - 1],
                                             const float (&vf)[PGeo<KP1>::ITEMS2][KP1], float xs)
{
    using G = PGeo<KP1>;
    constexpr int K = G::K;
    // every shared-memory read of a group before its stores (the accessors are ordered), so the
    // reads' latencies overlap instead of adding up
    constexpr int XN = P_ROWS * P_KC4;                  // 16-byte X items per chunk
    float4 xr[G::X_ITEMS];
#pragma unroll
    for (int i = 0; i < G::X_ITEMS; ++i) {
        const int q = pt + i * G::PT;
        const int qi = pair_x_item(q);
        if (G::X_ITEMS * G::PT == XN || q < XN) xr[i] = ld_shared_v4(slot + (uint32_t)qi * 16u);
    }
#pragma unroll
    for (int i = 0; i < G::X_ITEMS; ++i) {
        const int q = pt + i * G::PT;
        if (G::X_ITEMS * G::PT != XN && q >= XN) break;
        uint32_t h0, l0, h1, l1;
        split_f16x2(__fmul_rn(xr[i].x, xs), __fmul_rn(xr[i].y, xs), h0, l0);
        split_f16x2(__fmul_rn(xr[i].z, xs), __fmul_rn(xr[i].w, xs), h1, l1);
        const int qi = pair_x_item(q), q4 = qi % P_KC4;   // 4 elements = 8 bytes of a half row
        const uint32_t off = sw128_offset(qi / P_KC4, hh * 4 + (q4 >> 1)) + (uint32_t)(q4 & 1) * 8u;
        st_shared_v2u(sb + P_OFF_B_HI + off, h0, h1);
        st_shared_v2u(sb + P_OFF_B_LO + off, l0, l1);
    }
#pragma unroll
    for (int i = 0; i < G::ITEMS2; ++i) {
        const int p = pt + i * G::PT;
        if (p < nch * (P_KC / 2)) {
            const int ch = chs[i], e2 = p % (P_KC / 2);
            float2 r = ld_shared_v2(slot + G::RAW_W + (uint32_t)(ch * P_KC + e2 * 2) * 4u);
            uint32_t qb[K];
#pragma unroll
            for (int n = 0; n < K; ++n)
                qb[n] = ld_shared_u16(slot + G::RAW_Q + (uint32_t)((n * G::CH + ch) * P_KC + e2 * 2)) ^
                        0x8080u;
            const int hc = hh * 4 + (e2 >> 2);         // 2 elements = 4 bytes of a half row
            const uint32_t cofs = (uint32_t)(e2 & 3) * 4u;
#pragma unroll
            for (int n = 0; n < KP1; ++n) {
                uint32_t hi, lo;
                split_f16x2(__fmul_rn(r.x, vf[i][n]), __fmul_rn(r.y, vf[i][n]), hi, lo);
                const uint32_t off = sw128_offset(ch * KP1 + n, hc) + cofs;
                st_shared_u32(sb + P_OFF_A_HI + off, hi);
                st_shared_u32(sb + P_OFF_A_LO + off, lo);
                if (n < K) {
                    const float sn = sc[i][n];
                    r.x = __fmaf_rn(-sn, code_from_biased(qb[n], 0), r.x);
                    r.y = __fmaf_rn(-sn, code_from_biased(qb[n], 1), r.y);
                }
            }
        }
    }
}

// scales: [C][k_max] point scales; xrange, vrange: max|X| and max|r| per residual vector, as
// float bits (pair_range_kernel).
template <int KP1>
__global__ void __launch_bounds__(PRoles::THREADS, 1)
output_error_pair_kernel(const float *__restrict__ scales, int C, int N, int d,
                         const unsigned *__restrict__ xrange, const unsigned *__restrict__ vrange,
                         float *__restrict__ err, int split,
                         const WaitCtl wc, const __grid_constant__ CUtensorMap tmX,
                         const __grid_constant__ CUtensorMap tmW,
                         const __grid_constant__ CUtensorMap tmQ)
{
    using G = PGeo<KP1>;
    using PR = PRoles;
    constexpr unsigned KBIT = MPQ_TIMEOUT_OUTPUT_ERROR;
    constexpr int NST = P_STAGES, SEG = P_SEG;
    constexpr int R = G::RAW_STAGES;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw_u32 & 1023u)) & 1023u;
    PairCtrl &ctl = *reinterpret_cast<PairCtrl *>(smem_raw + pad);
    const uint32_t stages_u32 = raw_u32 + pad + P_CTRL_BYTES;
    const uint32_t ring_u32 = stages_u32 + P_TILE_SETS * P_STAGE_BYTES;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t crank = cluster_ctarank();
    const int half = (int)(crank & 1u);              // 0: even CTA (issues the MMAs), 1: its peer
    const uint32_t leader = crank & ~1u;
    const uint16_t pair_mask = (uint16_t)(3u << leader);
    const int pr = (int)(crank >> 1);                // pair index in the cluster: row-tile phase
    const int pair_tile = blockIdx.x / (2 * split);
    const int k0 = (pair_tile * 2 + half) * G::CH;   // first channel of this CTA
    const int nch = max(0, min(G::CH, C - k0));
    const int nvec = nch * KP1;
    const int n_rt = (N + P_N - 1) / P_N;
    const int my_rt = (n_rt - pr + split - 1) / split;
    const int n_kc = (d + P_KC - 1) / P_KC;
    const int nseg = (n_kc + SEG - 1) / SEG;
    const int total = my_rt * n_kc;
    // control block, tile sets and the raw-tile ring within the launch's shared memory (the same
    // in every CTA, so the whole cluster leaves together)
    if (!MPQ_CHECK_SMEM_END((size_t)pad + P_CTRL_BYTES + (size_t)P_TILE_SETS * P_STAGE_BYTES +
                            (size_t)R * G::RAW_BYTES))
        return;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) {
            mbar_init(&ctl.full[s], 2 * PR::PROD_WARPS);
            mbar_init(&ctl.empty[s], 1);
        }
        for (int r = 0; r < P_MAX_RAW; ++r) {
            mbar_init(&ctl.raw_full[r], 1);
            mbar_init(&ctl.raw_empty[r], PR::PROD_WARPS);
        }
        mbar_init(&ctl.segfull, 1);
        mbar_init(&ctl.segempty, 2 * P_EPI_WARPS);
        mbar_init(&ctl.done, 1);
        ctl.abort = 0;
        fence_barrier_init();
    }
    for (int i = threadIdx.x; i < nvec; i += PR::THREADS) {
        if (!MPQ_IN((size_t)k0 * KP1 + i, (size_t)C * KP1)) continue;
        const int e = f16_scale_exp(__uint_as_float(__ldg(vrange + (size_t)k0 * KP1 + i)));
        ctl.vexp[i] = e;
        ctl.vscale[i] = pow2f(e);
    }
    if (threadIdx.x == 0) {
        const int e = f16_scale_exp(__uint_as_float(__ldg(xrange)));
        ctl.xexp = e;
        ctl.xscale = pow2f(e);
    }
    if (warp == PR::MMA_WARP) {
        tmem_alloc_pair(&ctl.tmem_base, P_TMEM_COLS);
        tc_fence_before();
    }
    cluster_sync();                     // barriers of both CTAs initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem = ctl.tmem_base;
    volatile int *abort_flag = &ctl.abort;

    if (warp < PR::PROD_WARPS) {
        // ---------------------------------------------------------------- producers
        const int pt = threadIdx.x;
        float sc[G::ITEMS2][KP1 - 1];   // scales of this thread's items, the same for every chunk
        float vf[G::ITEMS2][KP1];       // 2^e of the items' residual vectors
        int chs[G::ITEMS2];             // channel of each item
#pragma unroll
        for (int i = 0; i < G::ITEMS2; ++i) {
            const int p = pt + i * PR::PROD_THREADS;
            chs[i] = pair_channel<KP1>(p / (P_KC / 2), nch);
            const int k = k0 + chs[i];
            const bool own = p < nch * (P_KC / 2);
#pragma unroll
            for (int n = 0; n < KP1 - 1; ++n)
                sc[i][n] = own ? __ldg(scales + (size_t)k * (KP1 - 1) + n) : 0.0f;
#pragma unroll
            for (int n = 0; n < KP1; ++n)
                vf[i][n] = own ? ctl.vscale[chs[i] * KP1 + n] : 0.0f;
        }
        const float xs = ctl.xscale;
        for (int it = 0; it < total; ++it) {
            const int s = it % NST, slot = it % R;
            const uint32_t ph = (uint32_t)(it / NST) & 1u;
            const bool ok = mbar_wait(&ctl.raw_full[slot], (uint32_t)(it / R) & 1u, wc.budget) &&
                            mbar_wait_cluster(&ctl.empty[s], ph ^ 1u, wc.budget);
            if (!ok) {
                *abort_flag = 1;
                note_timeout(wc, KBIT);
            }
            if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;   // warp-uniform
            pair_consume<KP1>(ring_u32 + slot * G::RAW_BYTES, stages_u32 + (s >> 1) * P_STAGE_BYTES,
                              s & 1, pt, nch, chs, sc, vf, xs);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive_cluster(&ctl.full[s], leader);
                mbar_arrive(&ctl.raw_empty[slot]);
            }
        }
    } else if (warp < PR::MMA_WARP) {
        // ---------------------------------------------------------------- epilogue
        // lane quarter q (the TMEM lanes this warp may access) and column half h
        const int ew = warp - PR::EPI_WARP0, q = ew & 3, h = ew >> 2;
        const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(h * (P_N / 2));
        double acc = 0.0;
        int g = 0;
        bool stop = false;
        for (int lt = 0; lt < my_rt && !stop; ++lt) {
            for (int sg = 0; sg < nseg; ++sg, ++g) {
                const bool ok = mbar_wait_cluster(&ctl.segfull, (uint32_t)g & 1u, wc.budget);
                if (!ok) {
                    *abort_flag = 1;
                    note_timeout(wc, KBIT);
                }
                stop = __any_sync(0xffffffffu, !ok || *abort_flag);   // warp-uniform
                if (stop) break;
                tc_fence_after();
                const bool first = (sg == 0), last = (sg == nseg - 1);
                // the previous drain's running-sum stores land before they are read back (the MMA
                // never writes those columns, so the segment was released without waiting)
                if (!first) tmem_wait_st();
#pragma unroll 1
                for (int cb = 0; cb < P_N / 64; ++cb) {
                    const uint32_t col = (uint32_t)(cb * 32);
                    float v[32];
                    if (first) {
                        tmem_ld_32x32b_x32(lane_base + col, v);
                    } else {   // segment and running sums loaded together
                        float r[32];
                        tmem_ld2_32x32b_x32(lane_base + col, lane_base + P_RUN_COL + col, v, r);
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = __fadd_rn(v[i], r[i]);
                    }
                    if (last) {
                        float p = 0.0f;
#pragma unroll
                        for (int i = 0; i < 32; ++i) p = fmaf(v[i], v[i], p);
                        acc += (double)p;
                    } else {
                        tmem_st_32x32b_x32(lane_base + P_RUN_COL + col, v);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(&ctl.segempty, leader);
            }
        }
        tmem_wait_st();   // nothing of this warp's is in flight when tensor memory is released
        ctl.part[h][q * 32 + lane] = *abort_flag ? (double)NAN : acc;
    } else if (warp == PR::MMA_WARP) {
        // ---------------------------------------------------------------- MMA issuer (even CTA)
        if (half == 0 && lane == 0) {
            constexpr uint32_t idesc = idesc_f16(2 * P_VEC, P_N);
            int g = 0;
            for (int lt = 0; lt < my_rt && !*abort_flag; ++lt) {
                for (int kc = 0; kc < n_kc; ++kc) {
                    const bool seg_start = (kc % SEG) == 0;
                    if (seg_start) {
                        // both CTAs' epilogues must have drained the previous segment
                        if (!mbar_wait_cluster(&ctl.segempty, ((uint32_t)g & 1u) ^ 1u, wc.budget)) {
                            *abort_flag = 1;
                            note_timeout(wc, KBIT);
                        }
                        if (*abort_flag) break;
                        tc_fence_after();
                    }
                    const int it = lt * n_kc + kc;
                    const int s = it % NST;
                    const uint32_t ph = (uint32_t)(it / NST) & 1u;
                    if (!mbar_wait_cluster(&ctl.full[s], ph, wc.budget)) {
                        *abort_flag = 1;
                        note_timeout(wc, KBIT);
                    }
                    if (*abort_flag) break;
                    tc_fence_after();
                    const uint32_t sb = stages_u32 + (s >> 1) * P_STAGE_BYTES;
                    const uint64_t ah = smem_desc_sw128(sb + P_OFF_A_HI);
                    const uint64_t al = smem_desc_sw128(sb + P_OFF_A_LO);
                    const uint64_t bh = smem_desc_sw128(sb + P_OFF_B_HI);
                    const uint64_t bl = smem_desc_sw128(sb + P_OFF_B_LO);
                    // 32 fp16 elements of this stage's row half = two K = 16 steps of 32 bytes
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk) {
                        const uint64_t o = (uint64_t)(((s & 1) * 2 + kk) * 2);   // 16 B units
                        mma_f16_pair(tmem, al + o, bh + o, idesc, (seg_start && kk == 0) ? 0u : 1u);
                        mma_f16_pair(tmem, ah + o, bl + o, idesc, 1u);
                        mma_f16_pair(tmem, ah + o, bh + o, idesc, 1u);
                    }
                    mma_commit_pair(&ctl.empty[s], pair_mask);
                    if ((kc % SEG) == SEG - 1 || kc == n_kc - 1) {
                        mma_commit_pair(&ctl.segfull, pair_mask);
                        ++g;
                    }
                }
            }
            // drain: every MMA issued above completes before TMEM is released
            mma_commit_pair(&ctl.done, (uint16_t)(1u << leader));
            drain_wait_cluster(&ctl.done, 0, wc, KBIT);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------------- raw tile copies
        if (lane == 0) {
            prefetch_tensormap(&tmX);
            prefetch_tensormap(&tmW);
            prefetch_tensormap(&tmQ);
            int issued = 0;
            for (int f = 0; f < (wc.withhold ? 0 : total); ++f) {
                const int slot = f % R;
                if (f >= R &&
                    !mbar_wait(&ctl.raw_empty[slot], (uint32_t)(f / R - 1) & 1u, wc.budget)) {
                    *abort_flag = 1;
                    note_timeout(wc, KBIT);
                }
                if (*abort_flag) break;
                const uint32_t dst = ring_u32 + slot * G::RAW_BYTES;
                const int x = (f % n_kc) * P_KC;
                const int row0 = (pr + (f / n_kc) * split) * P_N + half * P_ROWS;
                // a tile copy starts 16-byte aligned (x counts int8 codes in the code map) into a
                // 16-byte aligned destination; a copy that would not is not issued, and the
                // consumers' bounded waits end the launch
                if (!MPQ_CHECK((x & 15) == 0 && (dst & 15u) == 0u && x < d)) {
                    *abort_flag = 1;
                    break;
                }
                mbar_arrive_expect_tx(&ctl.raw_full[slot], G::RAW_TX);
                tma_load_2d(dst, &tmX, x, row0, &ctl.raw_full[slot]);
                tma_load_2d(dst + G::RAW_W, &tmW, x, k0, &ctl.raw_full[slot]);
                tma_load_3d(dst + G::RAW_Q, &tmQ, x, k0, 0, &ctl.raw_full[slot]);
                issued = f + 1;
            }
            // no copy may land after the CTA is gone: wait for the last copies of every slot
            for (int f = issued - R > 0 ? issued - R : 0; f < issued; ++f)
                drain_wait(&ctl.raw_full[f % R], (uint32_t)(f / R) & 1u, wc, KBIT);
        }
        __syncwarp();
    }

    // ---------------------------------------------------------------- cluster reduction
    cluster_sync();
    if (crank < 2 && warp >= PR::EPI_WARP0 && warp < PR::EPI_WARP0 + 4) {
        const int m = (warp - PR::EPI_WARP0) * 32 + lane;
        if (m < nvec) {
            double s = 0.0;
            for (int j = 0; j < split; ++j) {
                s += ld_dsmem_f64(&ctl.part[0][m], crank + 2u * (uint32_t)j);
                s += ld_dsmem_f64(&ctl.part[1][m], crank + 2u * (uint32_t)j);
            }
            double v = s / (double)N;
            v *= pow2d(-2 * (ctl.xexp + ctl.vexp[m]));   // exact: undo the operand scales
            if (MPQ_IN((size_t)k0 * KP1 + m, (size_t)C * KP1)) err[(size_t)k0 * KP1 + m] = (float)v;
        }
    }
    cluster_sync();
    if (warp == PR::MMA_WARP) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, P_TMEM_COLS);
    }
}

__device__ __forceinline__ float max_abs4(float4 v)
{
    return fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w)));
}

// Ranges for the fp16 operand scales, folded with atomicMax into a zeroed range[] (float bits of
// non-negative values order like unsigned integers): blocks [0, xb) take max|X| into range[0], four
// independent 16-byte loads in flight per thread; the other blocks give each channel `split`
// warps, each over a 1/split share of the row, for max_j |r_{k,n+1,j}| of every residual vector
// (the same fp32 recursion of Eq. 7 as the contraction's producers) into
// range[1 + k (k_max + 1) + n].  d % 4 == 0, rows and code planes 16-byte aligned.
template <int KP1>
__device__ __forceinline__ void range_step(float4 r, const int8_t *__restrict__ codes, size_t plane,
                                           size_t row, int j, const float (&sc)[KP1 > 1 ? KP1 - 1 : 1],
                                           float (&mx)[KP1])
{
    mx[0] = fmaxf(mx[0], max_abs4(r));
#pragma unroll
    for (int n = 0; n < KP1 - 1; ++n) {
        const char4 q = __ldg(reinterpret_cast<const char4 *>(codes + n * plane + row) + j);
        r.x = __fmaf_rn(-sc[n], (float)q.x, r.x);
        r.y = __fmaf_rn(-sc[n], (float)q.y, r.y);
        r.z = __fmaf_rn(-sc[n], (float)q.z, r.z);
        r.w = __fmaf_rn(-sc[n], (float)q.w, r.w);
        mx[n + 1] = fmaxf(mx[n + 1], max_abs4(r));
    }
}

template <int KP1>
__global__ void __launch_bounds__(256)
pair_range_kernel(const float4 *__restrict__ X, long long nx4, int xb, const float *__restrict__ W,
                  const int8_t *__restrict__ codes, const float *__restrict__ scales, int C, int d,
                  int split, unsigned *__restrict__ range)
{
    constexpr int K = KP1 - 1;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if ((int)blockIdx.x < xb) {
        float m = 0.0f;
        const long long stride = (long long)xb * blockDim.x;
        long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
        for (; i + 3 * stride < nx4; i += 4 * stride) {
            const float4 a = __ldg(X + i), b = __ldg(X + i + stride);
            const float4 c = __ldg(X + i + 2 * stride), e = __ldg(X + i + 3 * stride);
            m = fmaxf(m, fmaxf(fmaxf(max_abs4(a), max_abs4(b)), fmaxf(max_abs4(c), max_abs4(e))));
        }
        for (; i < nx4; i += stride) m = fmaxf(m, max_abs4(__ldg(X + i)));
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (lane == 0) atomicMax(range, __float_as_uint(m));
        return;
    }
    const int gw = ((int)blockIdx.x - xb) * 8 + warp;
    const int k = gw / split, part = gw - k * split;
    if (k >= C) return;
    // 16-byte row loads and 4-byte code loads need d % 4 == 0 and aligned bases
    if (!MPQ_CHECK((d & 3) == 0 && ((uintptr_t)W & 15) == 0 && ((uintptr_t)codes & 3) == 0))
        return;
    float sc[K > 0 ? K : 1], mx[KP1];
#pragma unroll
    for (int n = 0; n < K; ++n) sc[n] = __ldg(scales + (size_t)k * K + n);
#pragma unroll
    for (int n = 0; n < KP1; ++n) mx[n] = 0.0f;
    const float4 *w4 = reinterpret_cast<const float4 *>(W + (size_t)k * d);
    const size_t plane = (size_t)C * d, row = (size_t)k * d;
    const int d4 = d / 4, step = 32 * split;
    int j = part * 32 + lane;
    for (; j + step < d4; j += 2 * step) {          // two rows' worth of loads in flight
        const float4 a = __ldg(w4 + j), b = __ldg(w4 + j + step);
        range_step<KP1>(a, codes, plane, row, j, sc, mx);
        range_step<KP1>(b, codes, plane, row, j + step, sc, mx);
    }
    if (j < d4) range_step<KP1>(__ldg(w4 + j), codes, plane, row, j, sc, mx);
#pragma unroll
    for (int n = 0; n < KP1; ++n) {
        float m = mx[n];
        for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (lane == 0 && MPQ_IN((size_t)k * KP1 + n, (size_t)C * KP1))
            atomicMax(range + 1 + (size_t)k * KP1 + n, __float_as_uint(m));
    }
}

// The range pre-pass into `range` (zeroed here): max|X| into range[0] and, with `residuals`, max|r|
// of every residual vector into range[1 + k (k_max+1) + n].
template <int KP1>
cudaError_t launch_ranges(const float *X, int N, const float *W, const int8_t *codes,
                          const float *scales, int C, int d, bool residuals, unsigned *range,
                          cudaStream_t stream)
{
    const size_t words = residuals ? 1 + (size_t)C * KP1 : 1;
    const long long nx4 = (long long)N * d / 4;
    const int xb = (int)std::min<long long>((nx4 + 1023) / 1024, 4LL * sm_count());
    const int rsplit = std::min(8, std::max(1, (d / 4 + 255) / 256));   // >= 8 loads per lane
    const long long cb = residuals ? ((long long)C * rsplit + 7) / 8 : 0;
    cudaError_t e = cudaMemsetAsync(range, 0, words * sizeof(unsigned), stream);
    if (e != cudaSuccess) return e;
    pair_range_kernel<KP1><<<(unsigned)(xb + cb), 256, 0, stream>>>(
        reinterpret_cast<const float4 *>(X), nx4, xb, W, codes, scales, C, d, rsplit, range);
    return cudaGetLastError();
}

// The greedy residuals' output error with scratch from the stream-ordered pool: the range table
// and the split X planes (2 N d fp16) in one block, the range pre-pass, then output_error_f16.cu's
// contraction.
template <int KP1>
mpq_status launch_pooled_f16(const float *X, int N, const float *W, const int8_t *codes,
                             const float *scales, int C, int d, float *err, cudaStream_t stream,
                             const float *rmax)
{
    const size_t words = rmax ? 1 : 1 + (size_t)C * KP1;
    const size_t range_bytes = (words * sizeof(unsigned) + 255) / 256 * 256;
    const size_t xs_bytes = (size_t)N * d * 2 * sizeof(uint16_t);
    void *scratch = nullptr;
    const mpq_status st = pool_scratch(&scratch, range_bytes + xs_bytes, stream);
    if (st != MPQ_OK) return st;
    unsigned *range = static_cast<unsigned *>(scratch);
    uint16_t *xs = reinterpret_cast<uint16_t *>(static_cast<char *>(scratch) + range_bytes);
    const cudaError_t e =
        launch_ranges<KP1>(X, N, W, codes, scales, C, d, rmax == nullptr, range, stream);
    mpq_status r = cuda_status(e, "output-error range pre-pass");
    if (r == MPQ_OK) {
        const unsigned *vr = rmax ? reinterpret_cast<const unsigned *>(rmax) : range + 1;
        r = launch_output_error_f16(X, N, W, codes, scales, C, d, KP1 - 1, err, range, vr, xs,
                                    stream);
    }
    const cudaError_t ef = cudaFreeAsync(scratch, stream);
    if (r == MPQ_OK) r = cuda_status(ef, "scratch release (cudaFreeAsync)");
    return r;
}

// ext_range: caller-provided range scratch (this kernel), or NULL (the pooled path of
// output_error_f16.cu).
template <int KP1>
mpq_status launch_pair(const float *X, int N, const float *W, const int8_t *codes,
                       const float *scales, int C, int d, float *err, cudaStream_t stream,
                       unsigned *ext_range, const float *rmax)
{
    if (!ext_range) return launch_pooled_f16<KP1>(X, N, W, codes, scales, C, d, err, stream, rmax);
    using G = PGeo<KP1>;
    const int n_pairs = (C + 2 * G::CH - 1) / (2 * G::CH);
    const int n_rt = (N + P_N - 1) / P_N;

    CUtensorMap tmX, tmW, tmQ;
    memset(&tmX, 0, sizeof(tmX));
    memset(&tmW, 0, sizeof(tmW));
    memset(&tmQ, 0, sizeof(tmQ));
    const cuuint64_t dx[2] = {(cuuint64_t)d, (cuuint64_t)N}, sx[1] = {(cuuint64_t)d * 4};
    const cuuint32_t bx[2] = {P_KC, P_ROWS};
    const cuuint64_t dw[2] = {(cuuint64_t)d, (cuuint64_t)C}, sw[1] = {(cuuint64_t)d * 4};
    const cuuint32_t bw[2] = {P_KC, (cuuint32_t)G::CH};
    const cuuint64_t dq[3] = {(cuuint64_t)d, (cuuint64_t)C, (cuuint64_t)G::K};
    const cuuint64_t sq[2] = {(cuuint64_t)d, (cuuint64_t)C * d};
    const cuuint32_t bq[3] = {P_KC, (cuuint32_t)G::CH, (cuuint32_t)G::K};
    if (!encode_tile_map(&tmX, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, X, dx, sx, bx) ||
        !encode_tile_map(&tmW, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, W, dw, sw, bw) ||
        !encode_tile_map(&tmQ, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, codes, dq, sq, bq)) {
        set_error("output error: tensor map encoding failed");
        return MPQ_ERR_CUDA;
    }
    if ((long long)G::SMEM > max_smem_optin()) {
        set_error("pair output error needs %d bytes of shared memory", G::SMEM);
        return MPQ_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(output_error_pair_kernel<KP1>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");

    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(PRoles::THREADS, 1, 1);
    cfg.dynamicSmemBytes = (size_t)G::SMEM;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;

    // Row tiles split over `split` pairs per cluster (clusters of 2 * split CTAs).  Larger clusters
    // fit fewer at a time on the GPU (SMs are grouped), so pick the split with the least
    // (waves of resident clusters) x (row tiles per CTA), ties to the smaller cluster.
    // resident clusters per cluster size, queried once per process (one device per process)
    static std::atomic<int> resident[3] = {{0}, {0}, {0}};
    int split = 1;
    long long best = -1;
    for (int sp = 1, i = 0; sp <= 4 && sp <= n_rt; sp *= 2, ++i) {
        attr[0].val.clusterDim.x = (unsigned)(2 * sp);
        cfg.gridDim = dim3((unsigned)(n_pairs * 2 * sp), 1, 1);
        int active = resident[i].load(std::memory_order_relaxed);
        if (active == 0) {
            if (cudaOccupancyMaxActiveClusters(&active, output_error_pair_kernel<KP1>, &cfg) !=
                cudaSuccess)
                active = -1;
            (void)cudaGetLastError();
            resident[i].store(active, std::memory_order_relaxed);
        }
        if (active < 1) continue;
        const long long waves = (n_pairs + active - 1) / active;
        const long long cost = waves * ((n_rt + sp - 1) / sp);
        if (best < 0 || cost < best) {
            best = cost;
            split = sp;
        }
    }
    attr[0].val.clusterDim.x = (unsigned)(2 * split);
    cfg.gridDim = dim3((unsigned)(n_pairs * 2 * split), 1, 1);
    WaitCtl wc;
    mpq_status wst = wait_ctl(&wc);
    if (wst != MPQ_OK) return wst;
    // the ranges of X and of every residual vector first, into the caller's table (the residual
    // vectors' from rmax when the greedy search gave them: then the pre-pass reads X alone)
    e = launch_ranges<KP1>(X, N, W, codes, scales, C, d, rmax == nullptr, ext_range, stream);
    const unsigned *vr = rmax ? reinterpret_cast<const unsigned *>(rmax) : ext_range + 1;
    if (e == cudaSuccess)
        e = cudaLaunchKernelEx(&cfg, output_error_pair_kernel<KP1>, scales, C, N, d,
                               (const unsigned *)ext_range, vr, err, split, wc, tmX, tmW, tmQ);
    return cuda_status(e, "pair output-error kernel launch");
}

}  // namespace

namespace {
PFN_cuTensorMapEncodeTiled_v12000 tile_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        return (PFN_cuTensorMapEncodeTiled_v12000) nullptr;
    }();
    return fn;
}
}  // namespace

bool encode_tile_map(CUtensorMap *m, CUtensorMapDataType type, int rank, const void *base,
                     const cuuint64_t *dims, const cuuint64_t *strides, const cuuint32_t *box,
                     CUtensorMapSwizzle swizzle)
{
    PFN_cuTensorMapEncodeTiled_v12000 enc = tile_map_encoder();
    if (!enc) return false;
    const cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, type, (cuuint32_t)rank, const_cast<void *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Scratch (the fp16 contraction's range table, the adaptive grid's event lists) comes from the device's stream-ordered pool (allocated and
// freed on the call's stream, so concurrent calls on other streams never share it; inside a CUDA
// graph capture these become the graph's own allocation nodes).  Freed blocks stay cached in the
// pool instead of going back to the driver at every synchronisation (set on the first call made
// outside a stream capture, where a pool attribute may not be changed).
mpq_status pool_scratch(void **p, size_t bytes, cudaStream_t stream)
{
    static std::atomic<int> pool_set{0};
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusActive;
    if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess) {
        (void)cudaGetLastError();
        cs = cudaStreamCaptureStatusActive;
    }
    if (cs == cudaStreamCaptureStatusNone && !pool_set.exchange(1)) {
        int dev = 0;
        cudaMemPool_t pool;
        if (cudaGetDevice(&dev) == cudaSuccess && cudaDeviceGetDefaultMemPool(&pool, dev) == cudaSuccess) {
            uint64_t keep = UINT64_MAX;
            (void)cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
        }
        (void)cudaGetLastError();
    }
    const cudaError_t e = cudaMallocAsync(p, bytes, stream);
    if (e == cudaErrorMemoryAllocation) {
        (void)cudaGetLastError();
        set_error("no %zu bytes of scratch in the stream-ordered pool", bytes);
        return MPQ_ERR_NOMEM;
    }
    return cuda_status(e, "scratch allocation (cudaMallocAsync)");
}

bool output_error_pair_ok(const float *X, const float *W, const int8_t *codes, int d)
{
    return (d % 16 == 0) && ((uintptr_t)X % 16 == 0) && ((uintptr_t)W % 16 == 0) &&
           ((uintptr_t)codes % 16 == 0);
}

mpq_status launch_output_error_pair(const float *X, int N, const float *W, const int8_t *codes,
                                    const float *scales, int C, int d, int k_max, float *err,
                                    cudaStream_t stream, unsigned *range, const float *rmax)
{
    switch (k_max + 1) {
#define MPQ_CASE(n) \
    case n: return launch_pair<n>(X, N, W, codes, scales, C, d, err, stream, range, rmax);
        MPQ_CASE(2) MPQ_CASE(3) MPQ_CASE(4) MPQ_CASE(5) MPQ_CASE(6) MPQ_CASE(7) MPQ_CASE(8)
        MPQ_CASE(9) MPQ_CASE(10) MPQ_CASE(11) MPQ_CASE(12) MPQ_CASE(13) MPQ_CASE(14) MPQ_CASE(15)
        MPQ_CASE(16) MPQ_CASE(17)
#undef MPQ_CASE
    }
    set_error("k_max = %d unsupported", k_max);
    return MPQ_ERR_UNSUPPORTED;
}

mpq_status launch_x_range(const float *X, int N, int d, unsigned *range, cudaStream_t stream)
{
    return cuda_status(launch_ranges<2>(X, N, nullptr, nullptr, nullptr, 0, d, false, range, stream),
                       "X range pass");
}

}  // namespace mpq
