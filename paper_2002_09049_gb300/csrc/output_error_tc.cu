// Output error (Sec. 3.3, Eq. 11) on the 5th-generation tensor cores, single-CTA form:
//   err[k][n] = (1/N) sum_t (x_t . r_{k,n+1})^2,  n = 0..k_max.
// It serves the shapes the CTA-pair kernel's TMA tile copies cannot address (rows whose byte
// length is not a multiple of 16, or unaligned buffers); producers read global memory directly.
//
// As a contraction: Y = R X^T with R the C*(k_max+1) residual vectors (rows) and X the N
// calibration rows, both of length d; err is the row-wise mean of Y^2.  Mapping:
//   * A operand = residual vectors, 256 per CTA as two M = 128 halves (TMEM lanes = vectors),
//     whole channels per CTA (floor(256/(k_max+1)) channels);
//   * B operand = 128 calibration rows per row tile (UMMA N = 128);
//   * K = d in chunks of 32 fp32 (one 128-byte swizzle row).
// fp32-grade products with tcgen05 kind::tf32: each operand x is split exactly into
// hi = x with the 13 low mantissa bits cleared (a tf32 value) and lo = x - hi, and
// Y = hi*hi + hi*lo + lo*hi (the dropped lo*lo term is ~2^-22 relative).
//
// Accumulation.  The tensor core adds each product into the fp32 accumulator truncated at the
// accumulator's precision, so one long K chain biases |Y| low by a relative amount that grows with
// the chain length and the accumulator magnitude.  The chain is therefore restarted every
// SEG_CHUNKS chunks (128 elements of d, 48 MMA steps); the epilogue warps add each segment into a
// running sum kept in tensor memory with round-to-nearest fp32 additions.  TMEM columns:
// [0, 256) segment accumulators of the two halves, [256, 512) running sums.
//
// Warp roles (416 threads): warps 0-7 produce operand stages in shared memory (X rows and the
// residuals, which are regenerated from W, codes and scales by the recursion of Eq. 7 and never
// exist in global memory), prefetching the next stage's global data into registers with guarded
// loads while the current one is consumed; warps 8-11 fold segments into the running sums and
// square-sum the finished row tiles; warp 12 owns TMEM and one of its threads issues the MMAs.
// Each warp reports a stage with one arrival, and stops only on a warp-uniform decision.
//
// Row tiles are split over the CTAs of a thread-block cluster; rank 0 adds the partial sums of
// its peers from distributed shared memory in rank order, so every result is written once, in a
// fixed order, with no global scratch and no atomics.  Every wait is bounded; on a timeout the
// CTA unwinds and its outputs read NaN.
#include <math.h>

#include "mpq_internal.cuh"
#include "sm100.cuh"
#include "tf32_operands.cuh"
#include "waits.cuh"

MPQ_CHECKED_UNIT("output_error_tc.cu");

namespace mpq {
namespace {

using namespace sm100;

constexpr int TC_M = 128;                       // vectors per accumulator (TMEM lanes)
constexpr int TC_HALVES = 2;                    // accumulators per CTA
constexpr int TC_VEC = TC_M * TC_HALVES;        // 256 vectors per CTA
constexpr int TC_ROWS = 128;                    // calibration rows per row tile (UMMA N)
constexpr int TC_KC = 32;                       // fp32 per K chunk = one 128-byte row
constexpr int SEG_CHUNKS = 4;                   // accumulator restart period (chunks)
constexpr int TC_STAGES = 2;
constexpr int A_TILE = TC_M * TC_KC * 4;        // 16 KB
constexpr int B_TILE = TC_ROWS * TC_KC * 4;     // 16 KB
constexpr int OFF_A_HI = 0;                     // + h * A_TILE
constexpr int OFF_A_LO = TC_HALVES * A_TILE;    // + h * A_TILE
constexpr int OFF_B_HI = 2 * TC_HALVES * A_TILE;
constexpr int OFF_B_LO = OFF_B_HI + B_TILE;
constexpr int STAGE_BYTES = OFF_B_LO + B_TILE;  // 96 KB
constexpr int PRODUCER_WARPS = 8;
constexpr int PRODUCER_THREADS = PRODUCER_WARPS * 32;
constexpr int X_PER_THREAD = TC_ROWS * TC_KC / 4 / PRODUCER_THREADS;   // float4 per thread
constexpr int EPI_WARP0 = PRODUCER_WARPS;       // warps 8..11: warp % 4 selects TMEM lanes
constexpr int MMA_WARP = EPI_WARP0 + 4;
constexpr int TC_THREADS = (MMA_WARP + 1) * 32; // 416
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t RUN_COL = 256;               // running sums start here

struct Ctrl {
    uint64_t full[TC_STAGES];
    uint64_t empty[TC_STAGES];
    uint64_t segfull;
    uint64_t segempty;
    uint64_t done;
    uint32_t tmem_base;
    int abort;
    double part[TC_VEC];
};
constexpr int CTRL_BYTES = (sizeof(Ctrl) + 1023) / 1024 * 1024;
constexpr int TC_SMEM = 1024 /* alignment slack */ + CTRL_BYTES + TC_STAGES * STAGE_BYTES;

__device__ __forceinline__ float4 load4_guarded(const float *__restrict__ p, int j, int d,
                                                bool vec_ok)
{
    if (vec_ok && j + 3 < d && MPQ_CHECK(((uintptr_t)(p + j) & 15) == 0))
        return __ldg(reinterpret_cast<const float4 *>(p + j));
    float4 v;
    v.x = (j + 0 < d) ? __ldg(p + j + 0) : 0.0f;
    v.y = (j + 1 < d) ? __ldg(p + j + 1) : 0.0f;
    v.z = (j + 2 < d) ? __ldg(p + j + 2) : 0.0f;
    v.w = (j + 3 < d) ? __ldg(p + j + 3) : 0.0f;
    return v;
}

// Four int8 codes packed in a word (zeros past the end of the row).
__device__ __forceinline__ uint32_t codes4_guarded(const int8_t *__restrict__ p, int j, int d,
                                                   bool vec_ok)
{
    if (vec_ok && j + 3 < d && MPQ_CHECK(((uintptr_t)(p + j) & 3) == 0))
        return __ldg(reinterpret_cast<const unsigned int *>(p + j));
    uint32_t w = 0;
#pragma unroll
    for (int b = 0; b < 4; ++b)
        if (j + b < d) w |= (uint32_t)(uint8_t)__ldg(p + j + b) << (8 * b);
    return w;
}

__device__ __forceinline__ float code_byte(uint32_t w, int b)
{
    return (float)(int8_t)((w >> (8 * b)) & 0xFFu);
}

// Global data one producer thread needs for one stage.
template <int KP1>
struct Prefetch {
    static constexpr int K = KP1 - 1;
    static constexpr int CH = TC_VEC / KP1;                                // channels per CTA
    static constexpr int PAIRS = (CH * 8 + PRODUCER_THREADS - 1) / PRODUCER_THREADS;
    float4 x[X_PER_THREAD];
    float4 w[PAIRS];
    uint32_t q[PAIRS][K > 0 ? K : 1];
    float s[PAIRS][K > 0 ? K : 1];
};

template <int KP1>
__device__ __forceinline__ void prefetch(Prefetch<KP1> &pf, int pt, int rt, int kc,
                                         const float *__restrict__ X, int N,
                                         const float *__restrict__ W,
                                         const int8_t *__restrict__ codes,
                                         const float *__restrict__ scales, int k0, int nch, int d,
                                         size_t plane, bool vec_ok)
{
    constexpr int K = KP1 - 1;
    const int jc = kc * TC_KC;
#pragma unroll
    for (int i = 0; i < X_PER_THREAD; ++i) {
        const int q = pt + i * PRODUCER_THREADS;
        const int row = q >> 3, c = q & 7;
        const int t = rt * TC_ROWS + row;
        pf.x[i] = (t < N) ? load4_guarded(X + (size_t)t * d, jc + c * 4, d, vec_ok)
                          : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < Prefetch<KP1>::PAIRS; ++i) {
        const int p = pt + i * PRODUCER_THREADS;
        if (p < nch * 8) {
            const int ch = p >> 3, c = p & 7;
            const int k = k0 + ch;
            const int j = jc + c * 4;
            pf.w[i] = load4_guarded(W + (size_t)k * d, j, d, vec_ok);
#pragma unroll
            for (int n = 0; n < K; ++n) {
                pf.q[i][n] = codes4_guarded(codes + (size_t)n * plane + (size_t)k * d, j, d, vec_ok);
                pf.s[i][n] = __ldg(scales + (size_t)k * K + n);
            }
        }
    }
}

template <int KP1>
__device__ __forceinline__ void store_stage(const Prefetch<KP1> &pf, int pt, uint32_t sb, int nch)
{
    constexpr int K = KP1 - 1;
#pragma unroll
    for (int i = 0; i < X_PER_THREAD; ++i) {
        const int q = pt + i * PRODUCER_THREADS;
        const int row = q >> 3, c = q & 7;
        float4 hi, lo;
        split4(pf.x[i], hi, lo);
        const uint32_t off = sw128_offset(row, c);
        st_shared_v4(sb + OFF_B_HI + off, hi);
        st_shared_v4(sb + OFF_B_LO + off, lo);
    }
#pragma unroll
    for (int i = 0; i < Prefetch<KP1>::PAIRS; ++i) {
        const int p = pt + i * PRODUCER_THREADS;
        if (p < nch * 8) {
            const int ch = p >> 3, c = p & 7;
            float4 r = pf.w[i];
#pragma unroll
            for (int n = 0; n < KP1; ++n) {
                const int m = ch * KP1 + n;
                const int h = m >> 7, row = m & 127;
                float4 hi, lo;
                split4(r, hi, lo);
                const uint32_t off = sw128_offset(row, c);
                st_shared_v4(sb + OFF_A_HI + h * A_TILE + off, hi);
                st_shared_v4(sb + OFF_A_LO + h * A_TILE + off, lo);
                if (n < K) {
                    const float sn = pf.s[i][n];
                    const uint32_t qw = pf.q[i][n];
                    r.x = __fmaf_rn(-sn, code_byte(qw, 0), r.x);
                    r.y = __fmaf_rn(-sn, code_byte(qw, 1), r.y);
                    r.z = __fmaf_rn(-sn, code_byte(qw, 2), r.z);
                    r.w = __fmaf_rn(-sn, code_byte(qw, 3), r.w);
                }
            }
        }
    }
}

template <int KP1>
__global__ void __launch_bounds__(TC_THREADS, 1)
output_error_tc_kernel(const float *__restrict__ X, int N, const float *__restrict__ W,
                       const int8_t *__restrict__ codes, const float *__restrict__ scales, int C,
                       int d, float *__restrict__ err, int split, bool vec_ok, const WaitCtl wc)
{
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw_u32 & 1023u)) & 1023u;
    Ctrl &ctl = *reinterpret_cast<Ctrl *>(smem_raw + pad);
    const uint32_t stages_u32 = raw_u32 + pad + CTRL_BYTES;

    constexpr int CH = TC_VEC / KP1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile = blockIdx.x / split;
    const int crank = (int)cluster_ctarank();
    const int k0 = tile * CH;
    const int nch = min(CH, C - k0);
    const int nvec = nch * KP1;
    const int n_row_tiles = (N + TC_ROWS - 1) / TC_ROWS;
    const int my_rt = (n_row_tiles - crank + split - 1) / split;
    const int n_kc = (d + TC_KC - 1) / TC_KC;
    const int nseg = (n_kc + SEG_CHUNKS - 1) / SEG_CHUNKS;
    const int total = my_rt * n_kc;
    const size_t plane = (size_t)C * d;
    // control block and stages within the launch's shared memory (uniform over the cluster)
    if (!MPQ_CHECK_SMEM_END((size_t)pad + CTRL_BYTES + (size_t)TC_STAGES * STAGE_BYTES)) return;

    if (threadIdx.x == 0) {
        for (int s = 0; s < TC_STAGES; ++s) {
            mbar_init(&ctl.full[s], PRODUCER_WARPS);
            mbar_init(&ctl.empty[s], 1);
        }
        mbar_init(&ctl.segfull, 1);
        mbar_init(&ctl.segempty, 4);
        mbar_init(&ctl.done, 1);
        ctl.abort = 0;
        fence_barrier_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc(&ctl.tmem_base, TMEM_COLS);
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = ctl.tmem_base;
    volatile int *abort_flag = &ctl.abort;

    if (warp < PRODUCER_WARPS) {
        // ---------------------------------------------------------------- producers
        const int pt = threadIdx.x;
        Prefetch<KP1> pf;
        if (total > 0)
            prefetch<KP1>(pf, pt, crank, 0, X, N, W, codes, scales, k0, nch, d, plane, vec_ok);
        for (int it = 0; it < total; ++it) {
            const int s = it % TC_STAGES;
            const uint32_t ph = (uint32_t)(it / TC_STAGES) & 1u;
            const bool ok = mbar_wait(&ctl.empty[s], ph ^ 1u, wc.budget);
            if (!ok) {
                *abort_flag = 1;
                note_timeout(wc, MPQ_TIMEOUT_OUTPUT_ERROR);
            }
            if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;   // warp-uniform
            store_stage<KP1>(pf, pt, stages_u32 + s * STAGE_BYTES, nch);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.full[s]);
            const int nx = it + 1;
            if (nx < total) {
                const int lt = nx / n_kc, kc = nx % n_kc;
                prefetch<KP1>(pf, pt, crank + lt * split, kc, X, N, W, codes, scales, k0, nch,
                              d, plane, vec_ok);
            }
        }
    } else if (warp < MMA_WARP) {
        // ---------------------------------------------------------------- epilogue
        const int ew = warp - EPI_WARP0;
        const uint32_t lane_base = tmem + ((uint32_t)(ew * 32) << 16);
        double acc[TC_HALVES] = {0.0, 0.0};
        int g = 0;
        bool stop = false;
        for (int lt = 0; lt < my_rt && !stop; ++lt) {
            for (int sg = 0; sg < nseg; ++sg, ++g) {
                const bool ok = mbar_wait(&ctl.segfull, (uint32_t)g & 1u, wc.budget);
                if (!ok) {
                    *abort_flag = 1;
                    note_timeout(wc, MPQ_TIMEOUT_OUTPUT_ERROR);
                }
                stop = __any_sync(0xffffffffu, !ok || *abort_flag);   // warp-uniform
                if (stop) break;
                tc_fence_after();
                const bool first = (sg == 0), last = (sg == nseg - 1);
#pragma unroll
                for (int h = 0; h < TC_HALVES; ++h) {
#pragma unroll 1
                    for (int cb = 0; cb < TC_ROWS / 32; ++cb) {
                        const uint32_t col = (uint32_t)(h * TC_ROWS + cb * 32);
                        float v[32];
                        tmem_ld_32x32b_x32(lane_base + col, v);
                        if (!first) {
                            float r[32];
                            tmem_ld_32x32b_x32(lane_base + RUN_COL + col, r);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = __fadd_rn(v[i], r[i]);
                        }
                        if (last) {
                            float p = 0.0f;
#pragma unroll
                            for (int i = 0; i < 32; ++i) p = fmaf(v[i], v[i], p);
                            acc[h] += (double)p;
                        } else {
                            tmem_st_32x32b_x32(lane_base + RUN_COL + col, v);
                        }
                    }
                }
                if (!last) tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&ctl.segempty);
            }
        }
        const int m0 = ew * 32 + lane;
        const bool ok = !*abort_flag;
        ctl.part[m0] = ok ? acc[0] : (double)NAN;
        ctl.part[TC_M + m0] = ok ? acc[1] : (double)NAN;
    } else {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_tf32(TC_M, TC_ROWS);
            int g = 0;
            for (int lt = 0; lt < my_rt && !*abort_flag; ++lt) {
                for (int kc = 0; kc < n_kc; ++kc) {
                    const bool seg_start = (kc % SEG_CHUNKS) == 0;
                    if (seg_start) {
                        // the epilogue must have drained the previous segment
                        if (!mbar_wait(&ctl.segempty, ((uint32_t)g & 1u) ^ 1u, wc.budget)) {
                            *abort_flag = 1;
                            note_timeout(wc, MPQ_TIMEOUT_OUTPUT_ERROR);
                        }
                        if (*abort_flag) break;
                        tc_fence_after();
                    }
                    const int it = lt * n_kc + kc;
                    const int s = it % TC_STAGES;
                    const uint32_t ph = (uint32_t)(it / TC_STAGES) & 1u;
                    if (!mbar_wait(&ctl.full[s], ph, wc.budget)) {
                        *abort_flag = 1;
                        note_timeout(wc, MPQ_TIMEOUT_OUTPUT_ERROR);
                    }
                    if (*abort_flag) break;
                    tc_fence_after();
                    const uint32_t sb = stages_u32 + s * STAGE_BYTES;
                    const uint64_t bh = smem_desc_sw128(sb + OFF_B_HI);
                    const uint64_t bl = smem_desc_sw128(sb + OFF_B_LO);
#pragma unroll
                    for (int h = 0; h < TC_HALVES; ++h) {
                        const uint64_t ah = smem_desc_sw128(sb + OFF_A_HI + h * A_TILE);
                        const uint64_t al = smem_desc_sw128(sb + OFF_A_LO + h * A_TILE);
                        const uint32_t dt = tmem + (uint32_t)(h * TC_ROWS);
#pragma unroll
                        for (int kk = 0; kk < TC_KC / 8; ++kk) {
                            const uint64_t o = (uint64_t)(kk * 2);  // 32 bytes, in 16 B units
                            mma_tf32(dt, al + o, bh + o, idesc, (seg_start && kk == 0) ? 0u : 1u);
                            mma_tf32(dt, ah + o, bl + o, idesc, 1u);
                            mma_tf32(dt, ah + o, bh + o, idesc, 1u);
                        }
                    }
                    mma_commit(&ctl.empty[s]);
                    if ((kc % SEG_CHUNKS) == SEG_CHUNKS - 1 || kc == n_kc - 1) {
                        mma_commit(&ctl.segfull);
                        ++g;
                    }
                }
            }
            // drain: every MMA issued above completes before TMEM is released
            mma_commit(&ctl.done);
            drain_wait(&ctl.done, 0, wc, MPQ_TIMEOUT_OUTPUT_ERROR);
        }
        __syncwarp();
    }

    // ---------------------------------------------------------------- cluster reduction
    cluster_sync();
    if (crank == 0 && warp >= EPI_WARP0 && warp < MMA_WARP) {
        const int m0 = (warp - EPI_WARP0) * 32 + lane;
        for (int h = 0; h < TC_HALVES; ++h) {
            const int m = h * TC_M + m0;
            if (m < nvec) {
                double s = 0.0;
                for (int c = 0; c < split; ++c) s += ld_dsmem_f64(&ctl.part[m], (uint32_t)c);
                if (MPQ_IN((size_t)k0 * KP1 + m, (size_t)C * KP1))
                    err[(size_t)k0 * KP1 + m] = (float)(s / (double)N);
            }
        }
    }
    cluster_sync();
    __syncthreads();
    if (warp == MMA_WARP) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

template <int KP1>
mpq_status launch_tc(const float *X, int N, const float *W, const int8_t *codes,
                     const float *scales, int C, int d, float *err, cudaStream_t stream)
{
    const int ch_per_tile = TC_VEC / KP1;
    const int n_tiles = (C + ch_per_tile - 1) / ch_per_tile;
    const int n_row_tiles = (N + TC_ROWS - 1) / TC_ROWS;
    int split = 1;
    const int sms = sm_count();
    while (split < 8 && split * 2 <= n_row_tiles && (long long)n_tiles * split < 2LL * sms)
        split *= 2;
    const bool vec_ok = (d % 4 == 0) && ((uintptr_t)X % 16 == 0) && ((uintptr_t)W % 16 == 0) &&
                        ((uintptr_t)codes % 4 == 0);

    cudaError_t e = cudaFuncSetAttribute(output_error_tc_kernel<KP1>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, TC_SMEM);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(n_tiles * split), 1, 1);
    cfg.blockDim = dim3(TC_THREADS, 1, 1);
    cfg.dynamicSmemBytes = TC_SMEM;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)split;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    WaitCtl wc;
    const mpq_status wst = wait_ctl(&wc);
    if (wst != MPQ_OK) return wst;
    e = cudaLaunchKernelEx(&cfg, output_error_tc_kernel<KP1>, X, N, W, codes, scales, C, d, err,
                           split, vec_ok, wc);
    return cuda_status(e, "tensor-core output-error kernel launch");
}

}  // namespace

mpq_status launch_output_error_tc(const float *X, int N, const float *W, const int8_t *codes,
                                  const float *scales, int C, int d, int k_max, float *err,
                                  cudaStream_t stream)
{
    if ((long long)TC_SMEM > max_smem_optin()) {
        set_error("tensor-core output error needs %d bytes of shared memory", TC_SMEM);
        return MPQ_ERR_UNSUPPORTED;
    }
    switch (k_max + 1) {
#define MPQ_CASE(n) \
    case n: return launch_tc<n>(X, N, W, codes, scales, C, d, err, stream);
        MPQ_CASE(2) MPQ_CASE(3) MPQ_CASE(4) MPQ_CASE(5) MPQ_CASE(6) MPQ_CASE(7) MPQ_CASE(8)
        MPQ_CASE(9) MPQ_CASE(10) MPQ_CASE(11) MPQ_CASE(12) MPQ_CASE(13) MPQ_CASE(14) MPQ_CASE(15)
        MPQ_CASE(16) MPQ_CASE(17)
#undef MPQ_CASE
    }
    set_error("k_max = %d unsupported", k_max);
    return MPQ_ERR_UNSUPPORTED;
}

}  // namespace mpq
