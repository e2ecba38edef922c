// Output error (Sec. 3.3, Eq. 11) of the greedy residuals on the tensor cores, with X split ahead:
//   err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2,  n = 0..k_max.
//
// The contraction Y = R X^T is the CTA-pair one of output_error_pair.cu's fp16 mode: M = 256
// residual vectors (128 per CTA: whole channels) by N = 256 calibration rows per pair tile, each
// operand scaled by a power of two and split into fp16 hi/lo halves, Y = hi*hi + hi*lo + lo*hi on
// kind::f16 with fp32 accumulation restarted every 256 elements of d, the segments added into
// fp32 running sums, err = mean of Y^2 with the scales undone exactly.  What differs is the
// layout, set by shared-memory traffic, by the segment hand-off and by the cost of issuing tile
// copies and barrier operations:
//
// * X is scaled and split once per call (f16_split_kernel) into fp16 hi and lo planes in global
//   memory ([2][N][d]); tile copies put each 64-element step of a CTA's 128 rows straight into its
//   B operand tiles (128-byte swizzle).  The producer warps only regenerate the residuals
//   r_{n+1} = r_n - s_n q_n (Eq. 7) from W, codes and scales into the A tiles.
// * Work advances in steps of 64 elements (one 128-byte row of fp16 per operand row): one stage
//   hand-off, one W copy, one code copy and one X copy per step.
// * Two accumulators in tensor memory (columns [0, 256) and [256, 512)) take alternate segments,
//   and the running sums live in the epilogue warps' registers (one TMEM lane x 128 columns per
//   thread; setmaxnreg moves registers from warpgroups 0-1 to the epilogue's), so the MMA thread
//   starts the next segment in the other accumulator while the epilogue folds the last one.
// * The tile copies are issued by one epilogue warp, which is idle between its folds: neither the
//   producers (a stage waits for its slowest producer warp) nor the MMA thread carry them.
//
// The clipping search (Eq. 12, CLIP) runs the same contraction over every channel's n_cand
// candidate residuals r = w - s q: clip_planes_kernel writes them once as fp16 hi/lo planes like
// X's, and the A tiles are tile-copied from those planes like the B tiles (128 vectors per CTA,
// regardless of channel boundaries), so no producer work remains in that mode.
//
// Warps: 0-6 producers (224 threads: one (channel, 4 elements) item per step each when
// k_max + 1 = 9; in the clipping search warp 0 only relays that a stage's tiles have landed), 7
// the MMA issuer (lane 0 of the even CTA), 8-15 the epilogue (lane quarter warp % 4, column half;
// warp 15 also issues this CTA's tile copies).  Results are
// bit-identical to the fp16 mode of output_error_pair.cu: the same operands, MMAs in the same
// order (zero-filled elements past d add exact zeros), the same fp32 additions and the same
// reduction.  Every wait is bounded; on a timeout the kernel records MPQ_TIMEOUT_OUTPUT_ERROR (or
// MPQ_TIMEOUT_CLIP), waits for what it issued, and the outputs read NaN.
#include <cuda.h>
#include <cuda_fp16.h>
#include <math.h>
#include <string.h>

#include <algorithm>
#include <atomic>

#include "mpq_internal.cuh"
#include "pair_common.cuh"
#include "rounding.cuh"
#include "sm100.cuh"
#include "tf32_operands.cuh"
#include "waits.cuh"

MPQ_CHECKED_UNIT("output_error_f16.cu");

namespace mpq {
namespace {

using namespace sm100;

constexpr int F_VEC = 128;                 // residual vectors per CTA (TMEM lanes)
constexpr int F_ROWS = 128;                // calibration rows per CTA
constexpr int F_N = 2 * F_ROWS;            // rows per pair row tile (UMMA N)
constexpr int F_KS = 64;                   // elements per step: one 128-byte fp16 row
constexpr int F_ASETS = 2;                 // A operand stages (tile sets) at least (the producers')
constexpr int F_MAX_ASETS = 3;             // at most: where two raw slots still fit beside them
constexpr int F_PRE_ASETS = 3;             // A operand stages filled by tile copies (clipping search)
constexpr int F_BSLOTS = 3;                // B operand slots
constexpr int F_SEG = 4;                   // steps per accumulation segment (256 elements)
constexpr int F_PROD_WARPS = 7;
constexpr int F_PT = F_PROD_WARPS * 32;    // producer threads
constexpr int F_MMA_WARP = 7;              // MMA issuer (shares warpgroup 1 with producers 4-6)
constexpr int F_EPI_WARP0 = 8;             // a multiple of 4: warp % 4 is the TMEM lane quarter
constexpr int F_EPI_WARPS = 8;
constexpr int F_COPY_WARP = 15;            // an epilogue warp that also issues the tile copies
constexpr int F_THREADS = 512;
// registers per thread after setmaxnreg: warpgroups 0-1 (producers, MMA issuer) and 2-3
// (epilogue); together they use exactly what the launch holds (512 threads x 128)
constexpr int F_REGS_LOW = 88;
constexpr int F_REGS_HIGH = 168;
static_assert(256 * F_REGS_LOW + 256 * F_REGS_HIGH == F_THREADS * 128, "register split");
constexpr int F_TILE = 128 * 128;          // 16 KB: 128 rows of 128 bytes (128-byte swizzle)
constexpr int F_SET = 2 * F_TILE;          // hi and lo tiles of one operand stage
constexpr int F_MAX_RAW = 4;
constexpr uint32_t F_TMEM_COLS = 512;
constexpr int F_SMEM_LIMIT = 232448;       // opt-in shared memory per CTA on sm_100 parts

struct F16Ctrl {
    uint64_t full[F_MAX_ASETS];    // even CTA: both CTAs' producer warps (A written, B landed)
    uint64_t empty[F_MAX_ASETS];   // both CTAs: pair MMA commit (A stage free)
    uint64_t afull[F_MAX_ASETS];   // this CTA's A tile copy (clipping search)
    uint64_t bfull[F_BSLOTS];      // this CTA's B tile copy
    uint64_t bempty[F_BSLOTS];     // both CTAs: pair MMA commit (B slot free)
    uint64_t raw_full[F_MAX_RAW];  // this CTA's W and code tile copies
    uint64_t raw_empty[F_MAX_RAW]; // this CTA's producer warps
    uint64_t segfull[2];           // both CTAs: pair MMA commit, per accumulator
    uint64_t segempty[2];          // even CTA: both CTAs' epilogue warps, per accumulator
    uint64_t done;                 // even CTA: every MMA complete
    uint32_t tmem_base;
    int abort;
    double part[2][F_VEC];         // per column half: sum over the rows' y^2
    float vscale[F_VEC];           // 2^e per residual vector
    int vexp[F_VEC];
    int xexp;
};
constexpr int F_CTRL_BYTES = (sizeof(F16Ctrl) + 1023) / 1024 * 1024;
constexpr int F_BASE_SMEM = 1024 /* alignment slack */ + F_CTRL_BYTES + F_ASETS * F_SET +
                            F_BSLOTS * F_SET;

// Raw slot: W step [CH][64] fp32, then codes [K][CH][64] int8, as the tile copies write them.
// A third A stage where two raw slots still fit beside it (it gives the producers a step of slack:
// k_max = 8 2.80 -> 2.75 ms, k_max = 6 2.39 -> 2.27 ms on an 11008 x 4096 layer), else two.
template <int KP1>
struct FGeo {
    static constexpr int K = KP1 - 1;
    static constexpr int CH = F_VEC / KP1;
    static constexpr int ITEMS = (CH * 16 + F_PT - 1) / F_PT;   // 16 items of 4 elements per step
    static constexpr int RAW_Q = CH * F_KS * 4;
    static constexpr uint32_t RAW_TX = CH * F_KS * 4 + K * CH * F_KS;
    static constexpr int RAW_BYTES = (RAW_Q + K * CH * F_KS + 1023) / 1024 * 1024;
    static constexpr int NA =
        (F_BASE_SMEM + F_SET + 2 * RAW_BYTES <= F_SMEM_LIMIT) ? F_MAX_ASETS : F_ASETS;
    static constexpr int BASE = F_BASE_SMEM + (NA - F_ASETS) * F_SET;
    static constexpr int RAW_FIT = (F_SMEM_LIMIT - BASE) / RAW_BYTES;
    static constexpr int RAW = RAW_FIT < F_MAX_RAW ? RAW_FIT : F_MAX_RAW;
    static constexpr int SMEM = BASE + RAW * RAW_BYTES;
    static_assert(K >= 1, "at least one point");
    static_assert(RAW >= 2, "raw ring needs two slots");
};

// Per-launch sizes.  Greedy residuals: whole channels of k_max + 1 vectors per CTA, W and codes
// through the raw ring, A written by the producers.  Clipping search: 128 residual vectors per CTA
// whatever their channel, A tiles copied from the residual planes (no raw ring).
template <int KP1, bool CLIP>
struct FShape {
    static constexpr int kp1 = KP1, ch = FGeo<KP1>::CH, raw = FGeo<KP1>::RAW, na = FGeo<KP1>::NA;
    static constexpr int raw_bytes = FGeo<KP1>::RAW_BYTES, smem = FGeo<KP1>::SMEM;
    static constexpr uint32_t raw_tx = FGeo<KP1>::RAW_TX;
};

template <int KP1>
struct FShape<KP1, true> {
    static constexpr int kp1 = 1, ch = F_VEC, raw = 0, na = F_PRE_ASETS, raw_bytes = 0;
    static constexpr int smem = 1024 + F_CTRL_BYTES + (F_PRE_ASETS + F_BSLOTS) * F_SET;
};
static_assert(FShape<1, true>::smem <= F_SMEM_LIMIT, "clipping search: shared memory");

template <int N>
__device__ __forceinline__ void setmaxnreg_inc()
{
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}

template <int N>
__device__ __forceinline__ void setmaxnreg_dec()
{
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}

// Raw slot -> A tiles of one step (tile set `aset`): for every (channel, 4 contiguous elements)
// item the residuals r_0 = w, r_{n+1} = r_n - s_n q_n (Eq. 7), each scaled by its vector's 2^e
// (vf) and split into fp16 hi/lo halves.  W as one 16-byte load, each point's codes as one 4-byte
// load, 8-byte operand stores: a half warp's 16 items fill one 128-byte row.  Every shared-memory
// read of an item before its stores.
template <int KP1>
__device__ __forceinline__ void f16_make_a(uint32_t slot, uint32_t aset, int pt, int nch,
                                           const int (&chs)[FGeo<KP1>::ITEMS],
                                           const float (&sc)[FGeo<KP1>::ITEMS][KP1 - 1],
                                           const float (&vf)[FGeo<KP1>::ITEMS][KP1])
{
    using G = FGeo<KP1>;
    constexpr int K = G::K;
#pragma unroll
    for (int i = 0; i < G::ITEMS; ++i) {
        const int p = pt + i * F_PT;
        if (p < nch * 16) {
            const int ch = chs[i], e4 = p % 16;
            float4 r = ld_shared_v4(slot + (uint32_t)(ch * F_KS + e4 * 4) * 4u);
            uint32_t qb[K];
#pragma unroll
            for (int n = 0; n < K; ++n)
                qb[n] = ld_shared_u32(slot + G::RAW_Q + (uint32_t)((n * G::CH + ch) * F_KS + e4 * 4)) ^
                        0x80808080u;
            const uint32_t cofs = (uint32_t)(e4 & 1) * 8u;   // 4 elements = 8 bytes of a 16-byte chunk
#pragma unroll
            for (int n = 0; n < KP1; ++n) {
                uint32_t h0, l0, h1, l1;
                split_f16x2(__fmul_rn(r.x, vf[i][n]), __fmul_rn(r.y, vf[i][n]), h0, l0);
                split_f16x2(__fmul_rn(r.z, vf[i][n]), __fmul_rn(r.w, vf[i][n]), h1, l1);
                const uint32_t off = sw128_offset(ch * KP1 + n, e4 >> 1) + cofs;
                st_shared_v2u(aset + off, h0, h1);
                st_shared_v2u(aset + F_TILE + off, l0, l1);
                if (n < K) {
                    const float sn = sc[i][n];
                    r.x = __fmaf_rn(-sn, code_from_biased(qb[n], 0), r.x);
                    r.y = __fmaf_rn(-sn, code_from_biased(qb[n], 1), r.y);
                    r.z = __fmaf_rn(-sn, code_from_biased(qb[n], 2), r.z);
                    r.w = __fmaf_rn(-sn, code_from_biased(qb[n], 3), r.w);
                }
            }
        }
    }
}

// Greedy residuals (CLIP false): scales [C][k_max] point scales; vrange: max|r| per residual
// vector ([C][k_max+1], float bits); tmW: W; tmQ: the codes.  Clipping search (CLIP, KP1 unused):
// C residual vectors, given as fp16 hi/lo planes (tmW: [2][C][d], clip_planes_kernel); vrange:
// the bound on each vector's elements that set its operand scale.  Both: xrange[0]: max|X| as
// float bits; tmX: the split X planes [2][N][d] fp16.
template <int KP1, bool CLIP>
__global__ void __launch_bounds__(F_THREADS, 1)
output_error_f16_kernel(const float *__restrict__ scales, int C, int N, int d,
                        const unsigned *__restrict__ xrange, const unsigned *__restrict__ vrange,
                        float *__restrict__ err, int split, const WaitCtl wc,
                        const __grid_constant__ CUtensorMap tmX,
                        const __grid_constant__ CUtensorMap tmW,
                        const __grid_constant__ CUtensorMap tmQ)
{
    using S = FShape<KP1, CLIP>;
    constexpr int NA = S::na, NB = F_BSLOTS, SEG = F_SEG, R = S::raw, kp1 = S::kp1;
    constexpr unsigned KBIT = CLIP ? MPQ_TIMEOUT_CLIP : MPQ_TIMEOUT_OUTPUT_ERROR;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw_u32 & 1023u)) & 1023u;
    F16Ctrl &ctl = *reinterpret_cast<F16Ctrl *>(smem_raw + pad);
    const uint32_t a_u32 = raw_u32 + pad + F_CTRL_BYTES;
    const uint32_t b_u32 = a_u32 + NA * F_SET;
    const uint32_t ring_u32 = b_u32 + NB * F_SET;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t crank = cluster_ctarank();
    const int half = (int)(crank & 1u);              // 0: even CTA (issues the MMAs), 1: its peer
    const uint32_t leader = crank & ~1u;
    const uint16_t pair_mask = (uint16_t)(3u << leader);
    const int pr = (int)(crank >> 1);                // pair index in the cluster: row-tile phase
    const int pair_tile = blockIdx.x / (2 * split);
    const int k0 = (pair_tile * 2 + half) * S::ch;    // first channel (clip: vector) of this CTA
    const int nch = max(0, min(S::ch, C - k0));
    const int nvec = nch * kp1;
    const int n_rt = (N + F_N - 1) / F_N;
    const int my_rt = (n_rt - pr + split - 1) / split;
    const int n_ks = (d + F_KS - 1) / F_KS;          // steps per row tile
    const int nseg = (n_ks + SEG - 1) / SEG;
    const int total = my_rt * n_ks;
    // control block, operand tiles and the raw ring within the launch's shared memory (the same in
    // every CTA, so the whole cluster leaves together)
    if (!MPQ_CHECK_SMEM_END((size_t)pad + F_CTRL_BYTES + (size_t)(NA + NB) * F_SET +
                            (size_t)R * S::raw_bytes))
        return;

    if (threadIdx.x == 0) {
        for (int s = 0; s < NA; ++s) {
            // both CTAs' producer warps, or (CLIP) one relay warp per CTA
            mbar_init(&ctl.full[s], CLIP ? 2 : 2 * F_PROD_WARPS);
            mbar_init(&ctl.empty[s], 1);
            mbar_init(&ctl.afull[s], 1);
        }
        for (int s = 0; s < NB; ++s) {
            mbar_init(&ctl.bfull[s], 1);
            mbar_init(&ctl.bempty[s], 1);
        }
        for (int r = 0; r < F_MAX_RAW; ++r) {
            mbar_init(&ctl.raw_full[r], 1);
            mbar_init(&ctl.raw_empty[r], F_PROD_WARPS);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&ctl.segfull[b], 1);
            mbar_init(&ctl.segempty[b], 2 * F_EPI_WARPS);
        }
        mbar_init(&ctl.done, 1);
        ctl.abort = 0;
        fence_barrier_init();
    }
    for (int i = threadIdx.x; i < nvec; i += F_THREADS) {
        if (!MPQ_IN((size_t)k0 * kp1 + i, (size_t)C * kp1)) continue;
        const int e = f16_scale_exp(__uint_as_float(__ldg(vrange + (size_t)k0 * kp1 + i)));
        ctl.vexp[i] = e;
        ctl.vscale[i] = pow2f(e);
    }
    if (threadIdx.x == 0) ctl.xexp = f16_scale_exp(__uint_as_float(__ldg(xrange)));
    if (warp == F_MMA_WARP) {
        tmem_alloc_pair(&ctl.tmem_base, F_TMEM_COLS);
        tc_fence_before();
    }
    cluster_sync();                     // barriers of both CTAs initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem = ctl.tmem_base;
    volatile int *abort_flag = &ctl.abort;

    // one setmaxnreg per warpgroup: 0-1 (producers, MMA issuer) give registers to 2-3 (epilogue)
    if (warp < F_EPI_WARP0) {
        setmaxnreg_dec<F_REGS_LOW>();
        if (CLIP && warp == 0) {
            // ------------------------------------------------------------ relay (clipping search)
            // a step's A and B tiles of this CTA have landed: report the stage full
            int s = 0, sb = 0;
            uint32_t aph = 0, bph = 0;
            for (int it = 0; it < total; ++it) {
                const bool ok = mbar_wait(&ctl.afull[s], aph, wc.budget) &&
                                mbar_wait(&ctl.bfull[sb], bph, wc.budget);
                if (!ok) {
                    *abort_flag = 1;
                    note_timeout(wc, KBIT);
                }
                if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;   // warp-uniform
                if (lane == 0) mbar_arrive_cluster(&ctl.full[s], leader);
                if (++s == NA) {
                    s = 0;
                    aph ^= 1u;
                }
                if (++sb == NB) {
                    sb = 0;
                    bph ^= 1u;
                }
            }
        } else if (!CLIP && warp < F_PROD_WARPS) {
            // ------------------------------------------------------------ producers
            using G = FGeo<CLIP ? 2 : KP1>;   // (CLIP never gets here; FGeo<2> keeps it well-formed)
            constexpr int K = G::K;
            const int pt = threadIdx.x;
            float sc[G::ITEMS][K];      // scales of this thread's items, the same for every step
            float vf[G::ITEMS][K + 1];  // 2^e of the items' residual vectors
            int chs[G::ITEMS];          // channel of each item
#pragma unroll
            for (int i = 0; i < G::ITEMS; ++i) {
                const int p = pt + i * F_PT;
                chs[i] = p / 16;
                const bool own = p < nch * 16;
                const int k = k0 + chs[i];
#pragma unroll
                for (int n = 0; n < K; ++n) sc[i][n] = own ? __ldg(scales + (size_t)k * K + n) : 0.0f;
#pragma unroll
                for (int n = 0; n <= K; ++n) vf[i][n] = own ? ctl.vscale[chs[i] * (K + 1) + n] : 0.0f;
            }
            int s = 0, slot = 0, sb = 0;
            uint32_t aph = 0, rph = 0, bph = 0;    // phase parities of stage s, slot, B slot sb
            for (int it = 0; it < total; ++it) {
                bool ok = mbar_wait(&ctl.raw_full[slot], rph, wc.budget) &&
                          mbar_wait_cluster(&ctl.empty[s], aph ^ 1u, wc.budget);
                if (!ok) {
                    *abort_flag = 1;
                    note_timeout(wc, KBIT);
                }
                if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;   // warp-uniform
                f16_make_a<K + 1>(ring_u32 + slot * G::RAW_BYTES, a_u32 + s * F_SET, pt, nch, chs,
                                  sc, vf);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&ctl.raw_empty[slot]);
                // the step's B tiles have landed too before the stage is reported full
                ok = mbar_wait(&ctl.bfull[sb], bph, wc.budget);
                if (!ok) {
                    *abort_flag = 1;
                    note_timeout(wc, KBIT);
                }
                if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;
                if (lane == 0) mbar_arrive_cluster(&ctl.full[s], leader);
                if (++s == NA) {
                    s = 0;
                    aph ^= 1u;
                }
                if (++slot == G::RAW) {
                    slot = 0;
                    rph ^= 1u;
                }
                if (++sb == NB) {
                    sb = 0;
                    bph ^= 1u;
                }
            }
        } else if (warp == F_MMA_WARP && half == 0 && lane == 0) {
            // ------------------------------------------------------------ MMA issuer (even CTA)
            constexpr uint32_t idesc = idesc_f16(2 * F_VEC, F_N);
            bool ok = true;
            // step it = (row tile, step ks), stage s, B slot sb, segment g (accumulator g & 1)
            int ks = 0, s = 0, sb = 0, g = 0, sk = 0;
            uint32_t aph = 0;
            for (int it = 0; it < total && ok && !*abort_flag; ++it) {
                const bool seg_start = sk == 0;
                const uint32_t b = (uint32_t)g & 1u;
                if (seg_start) {
                    // this accumulator's previous segment has been folded by both epilogues
                    if (!mbar_wait_cluster(&ctl.segempty[b], ((uint32_t)(g >> 1) & 1u) ^ 1u,
                                           wc.budget)) {
                        note_timeout(wc, KBIT);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                }
                if (!mbar_wait_cluster(&ctl.full[s], aph, wc.budget)) {
                    note_timeout(wc, KBIT);
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t aset = a_u32 + s * F_SET, bset = b_u32 + sb * F_SET;
                const uint64_t ah = smem_desc_sw128(aset), al = smem_desc_sw128(aset + F_TILE);
                const uint64_t bh = smem_desc_sw128(bset), bl = smem_desc_sw128(bset + F_TILE);
                const uint32_t dt = tmem + b * (F_TMEM_COLS / 2);
                // 64 fp16 elements = four K = 16 steps, 32 bytes apart in the 128-byte rows
                // (16-byte units); per K step the passes lo*hi, hi*lo, hi*hi
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t o = (uint64_t)(kk * 2);
                    mma_f16_pair(dt, al + o, bh + o, idesc, (seg_start && kk == 0) ? 0u : 1u);
                    mma_f16_pair(dt, ah + o, bl + o, idesc, 1u);
                    mma_f16_pair(dt, ah + o, bh + o, idesc, 1u);
                }
                mma_commit_pair(&ctl.empty[s], pair_mask);
                mma_commit_pair(&ctl.bempty[sb], pair_mask);
                ++ks;
                if (++sk == SEG || ks == n_ks) {
                    mma_commit_pair(&ctl.segfull[b], pair_mask);
                    sk = 0;
                    ++g;
                }
                if (ks == n_ks) ks = 0;
                if (++s == NA) {
                    s = 0;
                    aph ^= 1u;
                }
                if (++sb == NB) sb = 0;
            }
            if (!ok) *abort_flag = 1;
            // drain: every MMA issued above completes before tensor memory is released
            mma_commit_pair(&ctl.done, (uint16_t)(1u << leader));
            drain_wait_cluster(&ctl.done, 0, wc, KBIT);
        }
        __syncwarp();
    } else {
        setmaxnreg_inc<F_REGS_HIGH>();
        // ---------------------------------------------------------------- epilogue
        // lane quarter q (the TMEM lanes this warp may access) and column half h; the running sums
        // of this thread's TMEM lane over the half's 128 columns stay in registers
        const int ew = warp - F_EPI_WARP0, q = ew & 3, h = ew >> 2;
        const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(h * (F_N / 2));
        const int nseg_all = my_rt * nseg;
        float sums[F_N / 2];
        double acc = 0.0;
        // Warp F_COPY_WARP also issues the CTA's tile copies, step by step: W and codes of step f
        // into raw slot f % R once the producers have released step f - R, X rows of step f into B
        // slot f % NB once the MMAs of step f - NB have completed.  It goes on copying until the
        // next segment has ended, then folds it like the other epilogue warps (a segment ends
        // every SEG steps, and its fold is needed only SEG steps later, when its accumulator is
        // taken again).
        const bool copier = warp == F_COPY_WARP && wc.withhold == 0;
        int next = 0, raw_issued = 0, b_issued = 0;
        if (copier && lane == 0) {
            prefetch_tensormap(&tmX);
            prefetch_tensormap(&tmW);
            if constexpr (!CLIP) prefetch_tensormap(&tmQ);
        }
        for (int g = 0; g < nseg_all; ++g) {
            const uint32_t b = (uint32_t)g & 1u, par = (uint32_t)(g >> 1) & 1u;
            bool ok = true;
            if (copier) {
                while (next < total) {
                    if (lane == 0) {
                        const int f = next, x = (f % n_ks) * F_KS;
                        const int bslot = f % NB;
                        const uint32_t bdst = b_u32 + bslot * F_SET;
                        const int row0 = (pr + (f / n_ks) * split) * F_N + half * F_ROWS;
                        // a tile copy starts 16-byte aligned (x counts int8 codes in the code
                        // map, fp16 elements in the planes) into a 1024-byte aligned destination
                        // (128-byte swizzle), or is not issued and the launch ends through the
                        // bounded waits
                        if constexpr (CLIP) {
                            // A tiles of step f (residual planes) into stage f % NA once the
                            // MMAs of step f - NA have completed
                            const int as = f % NA;
                            const uint32_t adst = a_u32 + as * F_SET;
                            ok = MPQ_CHECK((x & 15) == 0 && (adst & 1023u) == 0u &&
                                           (bdst & 1023u) == 0u && x < d);
                            if (ok && f >= NA)
                                ok = mbar_wait_cluster(&ctl.empty[as], (uint32_t)((f - NA) / NA) & 1u,
                                                       wc.budget);
                            if (ok) {
                                mbar_arrive_expect_tx(&ctl.afull[as], 2 * F_TILE);
                                tma_load_3d(adst, &tmW, x, k0, 0, &ctl.afull[as]);
                                raw_issued = f + 1;
                            }
                        } else {
                            // the raw slot takes W rows and the codes of the greedy residuals
                            const int rslot = f % R;
                            const uint32_t rdst = ring_u32 + rslot * S::raw_bytes;
                            ok = MPQ_CHECK((x & 15) == 0 && (rdst & 15u) == 0u &&
                                           (bdst & 1023u) == 0u && x < d);
                            if (ok && f >= R)
                                ok = mbar_wait(&ctl.raw_empty[rslot], (uint32_t)((f - R) / R) & 1u,
                                               wc.budget);
                            if (ok) {
                                mbar_arrive_expect_tx(&ctl.raw_full[rslot], S::raw_tx);
                                tma_load_2d(rdst, &tmW, x, k0, &ctl.raw_full[rslot]);
                                tma_load_3d(rdst + FGeo<KP1>::RAW_Q, &tmQ, x, k0, 0,
                                            &ctl.raw_full[rslot]);
                                raw_issued = f + 1;
                            }
                        }
                        if (ok && f >= NB)
                            ok = mbar_wait_cluster(&ctl.bempty[bslot], (uint32_t)((f - NB) / NB) & 1u,
                                                   wc.budget);
                        if (ok) {
                            mbar_arrive_expect_tx(&ctl.bfull[bslot], 2 * F_TILE);
                            tma_load_3d(bdst, &tmX, x, row0, 0, &ctl.bfull[bslot]);
                            b_issued = f + 1;
                        }
                    }
                    ++next;
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) break;
                    // stop copying once segment g has ended
                    const bool ended = mbar_test_cluster(&ctl.segfull[b], par);
                    if (__shfl_sync(0xffffffffu, ended, 0)) break;
                }
            }
            ok = ok && mbar_wait_cluster(&ctl.segfull[b], par, wc.budget);
            if (!ok) {
                *abort_flag = 1;
                note_timeout(wc, KBIT);
            }
            if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;   // warp-uniform
            // fold segment g (accumulator b) into the sums; the last segment of a row tile adds
            // the rows' y^2 into acc
            tc_fence_after();
            const int sg = g % nseg;
            // a row tile's sums start from zero (0 + v = v, up to the sign of a zero, which the
            // squares below do not see)
            if (sg == 0) {
#pragma unroll
                for (int i = 0; i < F_N / 2; ++i) sums[i] = 0.0f;
            }
#pragma unroll
            for (int cb = 0; cb < F_N / 64; ++cb) {
                float v[32];
                tmem_ld_32x32b_x32(lane_base + b * (F_TMEM_COLS / 2) + (uint32_t)(cb * 32), v);
#pragma unroll
                for (int i = 0; i < 32; ++i) sums[cb * 32 + i] = __fadd_rn(v[i], sums[cb * 32 + i]);
            }
            // the accumulator is free again (the loads have completed)
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(&ctl.segempty[b], leader);
            if (sg == nseg - 1) {
#pragma unroll
                for (int cb = 0; cb < F_N / 64; ++cb) {
                    float p = 0.0f;
#pragma unroll
                    for (int i = 0; i < 32; ++i) p = fmaf(sums[cb * 32 + i], sums[cb * 32 + i], p);
                    acc += (double)p;
                }
            }
        }
        // no copy lands after the CTA is gone: the last copy of every slot
        if (copier && lane == 0) {
            if constexpr (CLIP) {
                for (int f = raw_issued - NA > 0 ? raw_issued - NA : 0; f < raw_issued; ++f)
                    drain_wait(&ctl.afull[f % NA], (uint32_t)(f / NA) & 1u, wc, KBIT);
            } else {
                for (int f = raw_issued - R > 0 ? raw_issued - R : 0; f < raw_issued; ++f)
                    drain_wait(&ctl.raw_full[f % R], (uint32_t)(f / R) & 1u, wc, KBIT);
            }
            for (int f = b_issued - NB > 0 ? b_issued - NB : 0; f < b_issued; ++f)
                drain_wait(&ctl.bfull[f % NB], (uint32_t)(f / NB) & 1u, wc, KBIT);
        }
        __syncwarp();
        ctl.part[h][q * 32 + lane] = *abort_flag ? (double)NAN : acc;
    }

    // ---------------------------------------------------------------- cluster reduction
    cluster_sync();
    if (crank < 2 && warp >= F_EPI_WARP0 && warp < F_EPI_WARP0 + 4) {
        const int m = (warp - F_EPI_WARP0) * 32 + lane;
        if (m < nvec) {
            double s = 0.0;
            for (int j = 0; j < split; ++j) {
                s += ld_dsmem_f64(&ctl.part[0][m], crank + 2u * (uint32_t)j);
                s += ld_dsmem_f64(&ctl.part[1][m], crank + 2u * (uint32_t)j);
            }
            double v = s / (double)N;
            v *= pow2d(-2 * (ctl.xexp + ctl.vexp[m]));   // exact: undo the operand scales
            if (MPQ_IN((size_t)k0 * kp1 + m, (size_t)C * kp1)) err[(size_t)k0 * kp1 + m] = (float)v;
        }
    }
    cluster_sync();
    if (warp == F_MMA_WARP) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, F_TMEM_COLS);
    }
}

// X * 2^e split into fp16 hi and lo planes ([2][N][d]: hi at 0, lo at N d), 8 elements a thread
// per step, e from max|X| (xrange[0]) as the contraction's operand scale.
__global__ void __launch_bounds__(256)
f16_split_kernel(const float4 *__restrict__ X, long long n8, const unsigned *__restrict__ xrange,
                 uint4 *__restrict__ hi, uint4 *__restrict__ lo)
{
    const float xs = pow2f(f16_scale_exp(__uint_as_float(__ldg(xrange))));
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n8; i += stride) {
        const float4 a = __ldg(X + 2 * i), b = __ldg(X + 2 * i + 1);
        uint4 H, L;
        split_f16x2(__fmul_rn(a.x, xs), __fmul_rn(a.y, xs), H.x, L.x);
        split_f16x2(__fmul_rn(a.z, xs), __fmul_rn(a.w, xs), H.y, L.y);
        split_f16x2(__fmul_rn(b.x, xs), __fmul_rn(b.y, xs), H.z, L.z);
        split_f16x2(__fmul_rn(b.z, xs), __fmul_rn(b.w, xs), H.w, L.w);
        hi[i] = H;
        lo[i] = L;
    }
}

// Clipping search (Eq. 12): the residual r = w - s q of channel c0 + v / n_cand under candidate
// v mod n_cand (s = K / Qmax, the codes q of Eq. 8 with the sign of w, q = 0 where s is 0 or NaN),
// scaled by 2^e and split into fp16 hi/lo planes ([2][M][d] as hi and lo).  One CTA per vector v,
// 8 elements a thread per step.  e comes from a bound on the vector's elements,
// max(min(max|w|, s/2), max|w| - Qmax s): an element with code 0 keeps r = w, one with a nearest
// nonzero code |r| <= s/2, a clamped one |r| = |w| - Qmax s (a residual a rounding above the bound
// still fits fp16, whose range reaches 2^16); kept in vrange[v] (float bits) for the contraction.
// (With max|w| below s/2, as for a small channel under a layer-wide K, every code is 0 and the
// bound is max|r| itself.)
__global__ void __launch_bounds__(128)
clip_planes_kernel(const float *__restrict__ W, int d, const float *__restrict__ clip,
                   const float *__restrict__ chmax, int c0, int n_cand, int qmax, int M,
                   uint4 *__restrict__ hi, uint4 *__restrict__ lo, unsigned *__restrict__ vrange)
{
    const int v = blockIdx.x, d8 = d / 8;
    if (v >= M) return;
    const long long k = c0 + v / n_cand;
    const float qmaxf = (float)qmax, qlim = qmaxf + 1.0f;
    const float tband = 0.5f - MPQ_FAST_REL * (qlim + 1.0f);
    // clip row of channel k, candidate v mod n_cand: index c0 n_cand + v
    const float sv = __fdiv_rn(__ldg(clip + (long long)c0 * n_cand + v), qmaxf);
    const float inv = sv > 0.0f ? __frcp_rn(sv) : 0.0f;
    const float m = __ldg(chmax + k);
    const float bound = fmaxf(fminf(m, __fmul_rn(0.5f, sv)), __fmaf_rn(-qmaxf, sv, m));
    const float vf = pow2f(f16_scale_exp(bound));
    if (threadIdx.x == 0) vrange[v] = __float_as_uint(bound);
    const float4 *w4 = reinterpret_cast<const float4 *>(W + k * d);
    const long long row = (long long)v * d8;
    for (int j = threadIdx.x; j < d8; j += blockDim.x) {
        const float4 a = __ldg(w4 + 2 * j), b = __ldg(w4 + 2 * j + 1);
        const float w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        float q[8];
        bool unsure = false;
#pragma unroll
        for (int e = 0; e < 8; ++e) q[e] = code_signed_fast(w[e], inv, qmaxf, qlim, tband, unsure);
        if (unsure) {
#pragma unroll
            for (int e = 0; e < 8; ++e) q[e] = code_signed_exact(w[e], sv, qmaxf);
        }
        uint32_t h[4], l[4];
#pragma unroll
        for (int e = 0; e < 4; ++e)
            split_f16x2(__fmul_rn(__fmaf_rn(-sv, q[2 * e], w[2 * e]), vf),
                        __fmul_rn(__fmaf_rn(-sv, q[2 * e + 1], w[2 * e + 1]), vf), h[e], l[e]);
        hi[row + j] = make_uint4(h[0], h[1], h[2], h[3]);
        lo[row + j] = make_uint4(l[0], l[1], l[2], l[3]);
    }
}

// X split into the fp16 planes xs ([2][N][d]) on `stream`.
cudaError_t launch_x_split(const float *X, int N, int d, const unsigned *xrange, uint16_t *xs,
                           cudaStream_t stream)
{
    const long long n8 = (long long)N * d / 8;
    const int sb = (int)std::min<long long>((n8 + 255) / 256, 4LL * sm_count());
    f16_split_kernel<<<(unsigned)std::max(sb, 1), 256, 0, stream>>>(
        reinterpret_cast<const float4 *>(X), n8, xrange, reinterpret_cast<uint4 *>(xs),
        reinterpret_cast<uint4 *>(xs + (size_t)N * d));
    return cudaGetLastError();
}

// The contraction, X already split into xs.  Greedy residuals: A = W, with codes and scales.
// Clipping search: A = the residual planes of C vectors.
template <int KP1, bool CLIP>
mpq_status launch_f16(const void *A, int N, const int8_t *codes, const float *scales, int C,
                      int d, float *err, const unsigned *xrange, const unsigned *vrange,
                      const uint16_t *xs, cudaStream_t stream)
{
    using S = FShape<KP1, CLIP>;
    const int n_pairs = (C + 2 * S::ch - 1) / (2 * S::ch);
    const int n_rt = (N + F_N - 1) / F_N;

    CUtensorMap tmX, tmW, tmQ;
    memset(&tmX, 0, sizeof(tmX));
    memset(&tmW, 0, sizeof(tmW));
    memset(&tmQ, 0, sizeof(tmQ));
    const cuuint64_t dx[3] = {(cuuint64_t)d, (cuuint64_t)N, 2};
    const cuuint64_t sx[2] = {(cuuint64_t)d * 2, (cuuint64_t)N * d * 2};
    const cuuint32_t bx[3] = {F_KS, F_ROWS, 2};
    bool maps = encode_tile_map(&tmX, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, xs, dx, sx, bx,
                                CU_TENSOR_MAP_SWIZZLE_128B);
    if constexpr (CLIP) {
        const cuuint64_t da[3] = {(cuuint64_t)d, (cuuint64_t)C, 2};
        const cuuint64_t sa[2] = {(cuuint64_t)d * 2, (cuuint64_t)C * d * 2};
        const cuuint32_t ba[3] = {F_KS, F_VEC, 2};
        maps = maps && encode_tile_map(&tmW, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, A, da, sa, ba,
                                       CU_TENSOR_MAP_SWIZZLE_128B);
    } else {
        using G = FGeo<KP1>;
        const cuuint64_t dw[2] = {(cuuint64_t)d, (cuuint64_t)C}, sw[1] = {(cuuint64_t)d * 4};
        const cuuint32_t bw[2] = {F_KS, (cuuint32_t)G::CH};
        const cuuint64_t dq[3] = {(cuuint64_t)d, (cuuint64_t)C, (cuuint64_t)G::K};
        const cuuint64_t sq[2] = {(cuuint64_t)d, (cuuint64_t)C * d};
        const cuuint32_t bq[3] = {F_KS, (cuuint32_t)G::CH, (cuuint32_t)G::K};
        maps = maps && encode_tile_map(&tmW, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, A, dw, sw, bw) &&
               encode_tile_map(&tmQ, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, codes, dq, sq, bq);
    }
    if (!maps) {
        set_error("output error: tensor map encoding failed");
        return MPQ_ERR_CUDA;
    }
    if ((long long)S::smem > max_smem_optin()) {
        set_error("fp16 output error needs %d bytes of shared memory", S::smem);
        return MPQ_ERR_UNSUPPORTED;
    }
    cudaError_t e = cudaFuncSetAttribute(output_error_f16_kernel<KP1, CLIP>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, S::smem);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");

    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(F_THREADS, 1, 1);
    cfg.dynamicSmemBytes = (size_t)S::smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;

    // Row tiles split over `split` pairs per cluster (clusters of 2 * split CTAs): the split with
    // the least (waves of resident clusters) x (row tiles per CTA), ties to the smaller cluster --
    // or, where A is copied from global memory, to the larger one, whose pairs read the same A
    // tiles at about the same time (from L2); resident clusters per cluster size queried once per
    // process (one device per process).
    static std::atomic<int> resident[3] = {{0}, {0}, {0}};
    int split = 1;
    long long best = -1;
    for (int sp = 1, i = 0; sp <= 4 && sp <= n_rt; sp *= 2, ++i) {
        attr[0].val.clusterDim.x = (unsigned)(2 * sp);
        cfg.gridDim = dim3((unsigned)(n_pairs * 2 * sp), 1, 1);
        int active = resident[i].load(std::memory_order_relaxed);
        if (active == 0) {
            if (cudaOccupancyMaxActiveClusters(&active, output_error_f16_kernel<KP1, CLIP>, &cfg) !=
                cudaSuccess)
                active = -1;
            (void)cudaGetLastError();
            resident[i].store(active, std::memory_order_relaxed);
        }
        if (active < 1) continue;
        const long long waves = (n_pairs + active - 1) / active;
        const long long cost = waves * ((n_rt + sp - 1) / sp);
        if (best < 0 || cost < best || (CLIP && cost == best)) {
            best = cost;
            split = sp;
        }
    }
    attr[0].val.clusterDim.x = (unsigned)(2 * split);
    cfg.gridDim = dim3((unsigned)(n_pairs * 2 * split), 1, 1);
    WaitCtl wc;
    mpq_status wst = wait_ctl(&wc);
    if (wst != MPQ_OK) return wst;
    e = cudaLaunchKernelEx(&cfg, output_error_f16_kernel<KP1, CLIP>, scales, C, N, d, xrange,
                           vrange, err, split, wc, tmX, tmW, tmQ);
    return cuda_status(e, "fp16 output-error kernel launch");
}

}  // namespace

mpq_status launch_output_error_f16(const float *X, int N, const float *W, const int8_t *codes,
                                   const float *scales, int C, int d, int k_max, float *err,
                                   const unsigned *xrange, const unsigned *vrange, uint16_t *xs,
                                   cudaStream_t stream)
{
    if (k_max < 1 || k_max > 16) {
        set_error("k_max = %d unsupported", k_max);
        return MPQ_ERR_UNSUPPORTED;
    }
    const cudaError_t e = launch_x_split(X, N, d, xrange, xs, stream);
    if (e != cudaSuccess) return cuda_status(e, "X split kernel launch");
    switch (k_max + 1) {
#define MPQ_CASE(n) \
    case n: return launch_f16<n, false>(W, N, codes, scales, C, d, err, xrange, vrange, xs, stream);
        MPQ_CASE(2) MPQ_CASE(3) MPQ_CASE(4) MPQ_CASE(5) MPQ_CASE(6) MPQ_CASE(7) MPQ_CASE(8)
        MPQ_CASE(9) MPQ_CASE(10) MPQ_CASE(11) MPQ_CASE(12) MPQ_CASE(13) MPQ_CASE(14) MPQ_CASE(15)
        MPQ_CASE(16) MPQ_CASE(17)
#undef MPQ_CASE
    }
    return MPQ_ERR_UNSUPPORTED;
}

// Channels per chunk of residual planes: whole channels, at most 4 GiB of planes at a time.
static int clip_chunk_channels(int C, int d, int n_cand)
{
    return (int)std::min<long long>(C, std::max(1LL, (1LL << 32) / (4LL * d * n_cand)));
}

size_t clip_f16_scratch_bytes(int C, int N, int d, int n_cand)
{
    const long long m_max = (long long)clip_chunk_channels(C, d, n_cand) * n_cand;
    return 256 /* X range */ + (size_t)N * d * 4 /* X planes */ + (size_t)m_max * d * 4 /* planes */ +
           ((size_t)m_max * 4 + 255) / 256 * 256 /* bounds */;
}

mpq_status launch_clip_f16(const float *X, int N, const float *W, const float *clip,
                           const float *chmax, int C, int d, int qmax, int n_cand, float *err,
                           void *scratch, cudaStream_t stream)
{
    // scratch: the X range word, X's planes, the residual planes of one chunk, their bounds
    const int cc = clip_chunk_channels(C, d, n_cand);
    char *p = static_cast<char *>(scratch);
    unsigned *xrange = reinterpret_cast<unsigned *>(p);
    uint16_t *xs = reinterpret_cast<uint16_t *>(p + 256);
    uint16_t *planes = reinterpret_cast<uint16_t *>(p + 256 + (size_t)N * d * 4);
    unsigned *vrange = reinterpret_cast<unsigned *>(p + 256 + (size_t)N * d * 4 +
                                                    (size_t)cc * n_cand * d * 4);
    mpq_status st = launch_x_range(X, N, d, xrange, stream);
    if (st != MPQ_OK) return st;
    cudaError_t e = launch_x_split(X, N, d, xrange, xs, stream);
    if (e != cudaSuccess) return cuda_status(e, "X split kernel launch");
    for (int c0 = 0; c0 < C && st == MPQ_OK; c0 += cc) {
        const int cn = std::min(cc, C - c0);
        const int M = cn * n_cand;
        const int threads = std::min(128, (d / 8 + 31) / 32 * 32);
        uint4 *hi = reinterpret_cast<uint4 *>(planes);
        clip_planes_kernel<<<(unsigned)M, (unsigned)threads, 0, stream>>>(
            W, d, clip, chmax, c0, n_cand, qmax, M, hi, hi + (size_t)M * (d / 8), vrange);
        e = cudaGetLastError();
        st = cuda_status(e, "clip residual planes kernel launch");
        if (st == MPQ_OK)
            st = launch_f16<1, true>(planes, N, nullptr, nullptr, M, d,
                                     err + (size_t)c0 * n_cand, xrange, vrange, xs, stream);
    }
    return st;
}

}  // namespace mpq
