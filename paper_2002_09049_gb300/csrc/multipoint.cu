// Integer inference with multipoint weights (Sec. 3.4, Eq. 13):
//   Y[k][t] = sat32( floor( sum_{i<n_k} A_{k,i} (q_{k,i} . x_t) / 2^p ) ),  A_{k,i} = rint(2^p s_{k,i}),
// in the paper's three steps: integer dot products of every point's codes with the integer input
// (step 1), multiplication by the 32-bit coefficients and summation (step 2), and the shift by p
// (step 3).
//
// Packing (offline, mpq_pack_points).  Each channel's n_k code rows become consecutive rows of one
// operand: channels are grouped by R = the power of two >= n_k (a channel with no point gets one
// zero row), and every 128-row tile holds 128/R channels of one group, so a channel's rows are R
// aligned TMEM lanes of one warp.  Rows past n_k and empty slots are zero with coefficient 0.  The
// codes are stored as bf16 (every int8 value is exact), rows padded to a multiple of 64 elements.
//
// Step 1 on the tensor cores.  tcgen05.mma kind::f16 with bf16 operands: the codes (TMA straight
// into 128-byte-swizzled K-major tiles) against the input rows (int8 by TMA into a raw ring, turned
// into bf16 exactly by eight producer warps through the fp32 exponent bias).  Products are exact
// and every partial sum is an integer of magnitude below 2^24 when d * Qmax * 128 < 2^24, so the
// fp32 accumulator holds the exact dot products (checked on the host; other layers take the
// integer kernel below).  A CTA takes RT 128-row tiles against 256 inputs (RT accumulators of 256
// TMEM columns): two on large layers, so each converted input tile feeds both, one on small layers
// for more CTAs; K chunks of 64.  The inputs vary fastest in the grid, so the CTAs that share a row
// tile run together and read its codes from L2.  Codes tiles, raw input tiles and bf16 input tiles
// have rings of their own, so each kind of load runs as far ahead as its latency needs: a raw tile
// is handed back as soon as the producers have read it, the others when the MMAs reading them
// complete.
// Steps 2 and 3 in the epilogue: each lane turns its accumulator into an integer, multiplies by its
// row's coefficient in 64 bits, the R lanes of a channel add with warp shuffles, and the first lane
// shifts (arithmetic: floor), saturates and writes 32 consecutive outputs.  Every wait is bounded.
// Asymmetric sets (a centre B_k, Eq. 1): the producers also sum each input row's int8 values while
// they convert it, and the first lane adds A_B,k (sum_j x_tj), A_B,k = rint(2^p B_k), before the
// shift.
//
// Rows that TMA cannot address (d not a multiple of 16, unaligned input) and layers beyond the
// exactness bound use a CUDA-core kernel with the same integer arithmetic.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>
#include <math.h>
#include <string.h>

#include <vector>

#include "mpq_internal.cuh"
#include "sm100.cuh"
#include "tf32_operands.cuh"
#include "waits.cuh"

MPQ_CHECKED_UNIT("multipoint.cu");

namespace mpq {
namespace {

using namespace sm100;

constexpr int L_M = 128;                        // packed rows per tile (TMEM lanes)
constexpr int L_N = 256;                        // inputs per tile (UMMA N)
constexpr int L_KC = 64;                        // bf16 per K chunk = one 128-byte swizzle row
constexpr int L_A_BYTES = L_M * L_KC * 2;       // 16 KB codes tile
constexpr int L_B_BYTES = L_N * L_KC * 2;       // 32 KB input tile (bf16)
constexpr int L_RAW_BYTES = L_N * L_KC;         // 16 KB input tile (int8, as loaded)
constexpr int L_MAX_RT = 2;

// Three rings, each as deep as its own latency needs: codes tiles (TMA, freed by the MMAs), raw
// int8 input tiles (TMA, freed as soon as the producers have read them) and bf16 input tiles
// (written by the producers, freed by the MMAs).  208 KB for RT = 1 and RT = 2.
constexpr int L_MAX_SLOTS = 4;
template <int RT>
struct LGeo {
    static constexpr int A_SLOTS = RT == 1 ? 4 : 3;
    static constexpr int A_SLOT = RT * L_A_BYTES;
    static constexpr int B_SLOTS = RT == 1 ? 3 : 2;
    static constexpr int R_SLOTS = 3;
    static constexpr int OFF_B = A_SLOTS * A_SLOT;
    static constexpr int OFF_RAW = OFF_B + B_SLOTS * L_B_BYTES;
    static constexpr int BYTES = OFF_RAW + R_SLOTS * L_RAW_BYTES;
    static constexpr uint32_t TMEM_COLS = RT * L_N;
};
constexpr int L_PROD_WARPS = 8;
constexpr int L_PROD_THREADS = L_PROD_WARPS * 32;
constexpr int L_EPI_WARP0 = L_PROD_WARPS;       // warps 8..11: warp % 4 selects TMEM lanes
constexpr int L_MMA_WARP = L_EPI_WARP0 + 4;
constexpr int L_TMA_A_WARP = L_MMA_WARP + 1;    // codes tiles
constexpr int L_TMA_X_WARP = L_TMA_A_WARP + 1;  // raw input tiles
constexpr int L_THREADS = (L_TMA_X_WARP + 1) * 32;   // 480

struct LinCtrl {
    uint64_t a_full[L_MAX_SLOTS];     // a codes slot has landed
    uint64_t a_empty[L_MAX_SLOTS];    // the MMAs reading a codes slot completed
    uint64_t b_full[L_MAX_SLOTS];     // producers wrote a bf16 input slot
    uint64_t b_empty[L_MAX_SLOTS];    // the MMAs reading a bf16 input slot completed
    uint64_t r_full[L_MAX_SLOTS];     // a raw input slot has landed
    uint64_t r_empty[L_MAX_SLOTS];    // producers read a raw input slot
    uint64_t done;                    // every MMA completed
    uint64_t xs_ready;                // producers stored the input-row sums
    uint32_t tmem_base;
    int abort;
    int coef[L_MAX_RT][L_M];          // the row coefficients A of this CTA's tiles
    int xsum[L_N];                    // sum_j x_tj of this CTA's inputs (centred layers)
    int kch[4][32];                   // per epilogue warp: the channel of each lane's row (-1: none)
};
constexpr int L_CTRL_BYTES = (sizeof(LinCtrl) + 1023) / 1024 * 1024;
template <int RT>
constexpr int lin_smem() { return 1024 + L_CTRL_BYTES + LGeo<RT>::BYTES; }
// the epilogue's staging (4 warps x 32 x 33 ints) reuses the bf16 input ring once every MMA is done
static_assert(4 * 32 * 33 * 4 <= 2 * L_B_BYTES, "epilogue staging fits the bf16 ring");

// Row r of a packed buffer: (channel, point) or channel -1 / point -1 for padding.
struct PackView {
    int *coef;
    int *chan;
    int *point;
    int *tile_R;
    int *center;                  // A_B of each channel, or null
    __nv_bfloat16 *codes;
    int *flag;
};

PackView view(const mpq_packed_layout *L, void *packed)
{
    unsigned char *b = static_cast<unsigned char *>(packed);
    PackView v;
    v.coef = reinterpret_cast<int *>(b + L->off_coef);
    v.chan = reinterpret_cast<int *>(b + L->off_chan);
    v.point = reinterpret_cast<int *>(b + L->off_point);
    v.tile_R = reinterpret_cast<int *>(b + L->off_tile);
    v.center = L->centered ? reinterpret_cast<int *>(b + L->off_center) : nullptr;
    v.codes = reinterpret_cast<__nv_bfloat16 *>(b + L->off_codes);
    v.flag = reinterpret_cast<int *>(b);   // header word 0: coefficient overflow
    return v;
}

// rint(2^p v) (ties to even) as a 32-bit coefficient; sets *flag when it does not fit (NaN included).
__device__ __forceinline__ int fixed_coeff(float v, int p, int *flag)
{
    const double x = nearbyint(ldexp((double)v, p));
    if (fabs(x) < 2147483648.0) return (int)x;
    atomicExch(flag, 1);
    return 0;
}

// A_B = rint(2^p B_k) of every channel.
__global__ void pack_center_kernel(const float *__restrict__ center, int C, int p, PackView v)
{
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k < C) v.center[k] = fixed_coeff(center[k], p, v.flag);
}

// A = rint(2^p s) (ties to even) and the bf16 codes of every packed row.
__global__ void pack_kernel(const int8_t *__restrict__ codes, const float *__restrict__ scales,
                            int C, int d, int d_pad, int k_max, int p, int rows, PackView v)
{
    const int r = blockIdx.x;
    const int k = v.chan[r], i = v.point[r];
    const bool live = k >= 0 && i >= 0 && MPQ_IN(k, C) && MPQ_IN(i, k_max);
    if (threadIdx.x == 0) v.coef[r] = live ? fixed_coeff(scales[(size_t)k * k_max + i], p, v.flag) : 0;
    const int8_t *q = live ? codes + (size_t)i * C * d + (size_t)k * d : nullptr;
    for (int j = threadIdx.x; j < d_pad; j += blockDim.x)
        v.codes[(size_t)r * d_pad + j] = __float2bfloat16_rn(live && j < d ? (float)q[j] : 0.0f);
}

// Two int8 -> two bf16 packed in a word (exact: |v| <= 128 has at most 8 significant bits).
__device__ __forceinline__ uint32_t bf16x2_from_biased(uint32_t biased, int b0)
{
    const uint32_t lo = __float_as_uint(code_from_biased(biased, b0));
    const uint32_t hi = __float_as_uint(code_from_biased(biased, b0 + 1));
    return __byte_perm(lo, hi, 0x7632u);
}

template <int RT>
__global__ void __launch_bounds__(L_THREADS, 1)
multipoint_linear_kernel(int T, int C, int tiles, int n_kc, int p, const int *__restrict__ coef,
                         const int *__restrict__ chan, const int *__restrict__ tile_R,
                         const int *__restrict__ center_coef,
                         int32_t *__restrict__ Y, const WaitCtl wc,
                         const __grid_constant__ CUtensorMap tmA,
                         const __grid_constant__ CUtensorMap tmX)
{
    using G = LGeo<RT>;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw_u32 = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (raw_u32 & 1023u)) & 1023u;
    LinCtrl &ctl = *reinterpret_cast<LinCtrl *>(smem_raw + pad);
    unsigned char *ring = smem_raw + pad + L_CTRL_BYTES;
    const uint32_t ring_u32 = raw_u32 + pad + L_CTRL_BYTES;
    const uint32_t a_u32 = ring_u32, b_u32 = ring_u32 + G::OFF_B, x_u32 = ring_u32 + G::OFF_RAW;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // inputs vary fastest: the CTAs sharing a row tile run together and read its codes from L2
    const int tile0 = blockIdx.y * RT, n0 = blockIdx.x * L_N;
    const int nt = min(RT, tiles - tile0);          // row tiles of this CTA (the last may hold one)
    if (!MPQ_CHECK_SMEM_END((size_t)pad + L_CTRL_BYTES + (size_t)G::BYTES)) return;

    if (threadIdx.x == 0) {
        for (int i = 0; i < G::A_SLOTS; ++i) {
            mbar_init(&ctl.a_full[i], 1);
            mbar_init(&ctl.a_empty[i], 1);
        }
        for (int i = 0; i < G::B_SLOTS; ++i) {
            mbar_init(&ctl.b_full[i], L_PROD_WARPS);
            mbar_init(&ctl.b_empty[i], 1);
        }
        for (int i = 0; i < G::R_SLOTS; ++i) {
            mbar_init(&ctl.r_full[i], 1);
            mbar_init(&ctl.r_empty[i], L_PROD_WARPS);
        }
        mbar_init(&ctl.done, 1);
        mbar_init(&ctl.xs_ready, L_PROD_WARPS);
        ctl.abort = 0;
        fence_barrier_init();
    }
    for (int r = threadIdx.x; r < RT * L_M; r += L_THREADS)
        ctl.coef[r / L_M][r % L_M] = r / L_M < nt ? coef[(size_t)tile0 * L_M + r] : 0;
    if (warp == L_MMA_WARP) {
        tmem_alloc(&ctl.tmem_base, G::TMEM_COLS);
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = ctl.tmem_base;
    volatile int *abort_flag = &ctl.abort;

    const bool centered = center_coef != nullptr;
    if (warp < L_PROD_WARPS) {
        // ---------------------------------------------------------------- producers: int8 -> bf16
        constexpr int ITEMS = L_N * (L_KC / 16) / L_PROD_THREADS;
        int xs[ITEMS];   // this thread's 16-byte share of each input row's sum
#pragma unroll
        for (int it = 0; it < ITEMS; ++it) xs[it] = 0;
        for (int kc = 0; kc < n_kc; ++kc) {
            const int rs = kc % G::R_SLOTS, bs = kc % G::B_SLOTS;
            bool ok = mbar_wait(&ctl.r_full[rs], (uint32_t)(kc / G::R_SLOTS) & 1u, wc.budget);
            if (ok && kc >= G::B_SLOTS)
                ok = mbar_wait(&ctl.b_empty[bs], (uint32_t)(kc / G::B_SLOTS - 1) & 1u, wc.budget);
            if (!ok) {
                *abort_flag = 1;
                note_timeout(wc, MPQ_TIMEOUT_INFERENCE);
            }
            if (__any_sync(0xffffffffu, !ok || *abort_flag)) break;   // warp-uniform
            // 16 input bytes (one input row, 16 K elements) per item, 4 items per thread: all
            // reads first, then the raw slot goes back to the TMA thread
            float4 raw[ITEMS];
#pragma unroll
            for (int it = 0; it < ITEMS; ++it)
                raw[it] = ld_shared_v4(x_u32 + rs * L_RAW_BYTES +
                                       (uint32_t)(threadIdx.x + it * L_PROD_THREADS) * 16u);
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.r_empty[rs]);
            const uint32_t bb = b_u32 + bs * L_B_BYTES;
#pragma unroll
            for (int it = 0; it < ITEMS; ++it) {
                const int q = threadIdx.x + it * L_PROD_THREADS;
                const int row = q >> 2, c16 = q & 3;
                if (centered) {   // signed bytes summed exactly (|sum| <= 128 d)
                    xs[it] = __dp4a(__float_as_int(raw[it].x), 0x01010101, xs[it]);
                    xs[it] = __dp4a(__float_as_int(raw[it].y), 0x01010101, xs[it]);
                    xs[it] = __dp4a(__float_as_int(raw[it].z), 0x01010101, xs[it]);
                    xs[it] = __dp4a(__float_as_int(raw[it].w), 0x01010101, xs[it]);
                }
                const uint32_t w[4] = {__float_as_uint(raw[it].x) ^ 0x80808080u,
                                       __float_as_uint(raw[it].y) ^ 0x80808080u,
                                       __float_as_uint(raw[it].z) ^ 0x80808080u,
                                       __float_as_uint(raw[it].w) ^ 0x80808080u};
                float4 o0, o1;
                o0.x = __uint_as_float(bf16x2_from_biased(w[0], 0));
                o0.y = __uint_as_float(bf16x2_from_biased(w[0], 2));
                o0.z = __uint_as_float(bf16x2_from_biased(w[1], 0));
                o0.w = __uint_as_float(bf16x2_from_biased(w[1], 2));
                o1.x = __uint_as_float(bf16x2_from_biased(w[2], 0));
                o1.y = __uint_as_float(bf16x2_from_biased(w[2], 2));
                o1.z = __uint_as_float(bf16x2_from_biased(w[3], 0));
                o1.w = __uint_as_float(bf16x2_from_biased(w[3], 2));
                st_shared_v4(bb + sw128_offset(row, 2 * c16), o0);
                st_shared_v4(bb + sw128_offset(row, 2 * c16 + 1), o1);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.b_full[bs]);
        }
        if (centered) {
            // the 4 threads of an input row (lanes 4m..4m+3) hold its 4 column shares
#pragma unroll
            for (int it = 0; it < ITEMS; ++it) {
                int v = xs[it];
                v += __shfl_xor_sync(0xffffffffu, v, 1);
                v += __shfl_xor_sync(0xffffffffu, v, 2);
                if ((threadIdx.x & 3) == 0) ctl.xsum[(threadIdx.x + it * L_PROD_THREADS) >> 2] = v;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&ctl.xs_ready);   // also after an abort: no wait is left open
        }
    } else if (warp < L_MMA_WARP) {
        // ---------------------------------------------------------------- epilogue
        const int ew = warp - L_EPI_WARP0;
        bool ok = mbar_wait(&ctl.done, 0, wc.budget);
        if (ok && centered) ok = mbar_wait(&ctl.xs_ready, 0, wc.budget);
        if (!ok) {
            *abort_flag = 1;
            note_timeout(wc, MPQ_TIMEOUT_INFERENCE);
        }
        const bool good = !__any_sync(0xffffffffu, !ok || *abort_flag);
        tc_fence_after();
        // staging for the stores: the bf16 input ring, idle once every MMA has completed
        int (*out)[33] = reinterpret_cast<int (*)[33]>(ring + G::OFF_B) + ew * 32;
        for (int u = 0; u < nt && good; ++u) {
            const int R = tile_R[tile0 + u];
            const int r = ew * 32 + lane;
            const int k = chan[(size_t)(tile0 + u) * L_M + r];
            const long long a = ctl.coef[u][r];
            const long long ab =
                centered && k >= 0 && MPQ_IN(k, C) ? (long long)center_coef[k] : 0;
            const uint32_t lane_base = tmem + ((uint32_t)(ew * 32) << 16) + (uint32_t)(u * L_N);
            // the rows this warp writes: one per channel (its first lane), -1 for none
            ctl.kch[ew][lane] = (lane & (R - 1)) == 0 ? k : -1;
            __syncwarp();
#pragma unroll 1
            for (int cb = 0; cb < L_N / 32; ++cb) {
                float v[32];
                tmem_ld_32x32b_x32(lane_base + (uint32_t)(cb * 32), v);
                long long sum[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) sum[j] = a * (long long)__float2int_rz(v[j]);
                for (int o = 1; o < R; o <<= 1) {   // the channel's R lanes (R-aligned)
#pragma unroll
                    for (int j = 0; j < 32; ++j) sum[j] += __shfl_xor_sync(0xffffffffu, sum[j], o);
                }
                if (centered) {   // the row sums first: no shared-memory store comes before them
                    int xs[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) xs[j] = ctl.xsum[cb * 32 + j];
#pragma unroll
                    for (int j = 0; j < 32; ++j) sum[j] += ab * (long long)xs[j];
                }
                int zr[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) {
                    long long z = sum[j] >> p;   // arithmetic shift: floor division by 2^p
                    z = z > 2147483647LL ? 2147483647LL : (z < -2147483648LL ? -2147483648LL : z);
                    zr[j] = (int)z;
                }
#pragma unroll
                for (int j = 0; j < 32; ++j) out[lane][j] = zr[j];
                __syncwarp();
                // one channel's 32 consecutive outputs per store: 128 contiguous bytes; every
                // shared-memory read is issued before the first store
                int kv[32], ov[32];
#pragma unroll
                for (int L = 0; L < 32; ++L) {
                    kv[L] = ctl.kch[ew][L];
                    ov[L] = out[L][lane];
                }
                __syncwarp();
                const int t = n0 + cb * 32 + lane;
                if (t < T) {
#pragma unroll
                    for (int L = 0; L < 32; ++L)
                        if (kv[L] >= 0 && MPQ_IN(kv[L], C)) Y[(size_t)kv[L] * T + t] = ov[L];
                }
            }
        }
    } else if (warp == L_MMA_WARP) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(L_M, L_N);
            for (int kc = 0; kc < n_kc; ++kc) {
                const int as = kc % G::A_SLOTS, bs = kc % G::B_SLOTS;
                bool ok = mbar_wait(&ctl.a_full[as], (uint32_t)(kc / G::A_SLOTS) & 1u, wc.budget);
                if (ok) ok = mbar_wait(&ctl.b_full[bs], (uint32_t)(kc / G::B_SLOTS) & 1u, wc.budget);
                if (!ok) {
                    *abort_flag = 1;
                    note_timeout(wc, MPQ_TIMEOUT_INFERENCE);
                }
                if (*abort_flag) break;
                tc_fence_after();
                const uint64_t bd = smem_desc_sw128(b_u32 + bs * L_B_BYTES);
                for (int u = 0; u < nt; ++u) {
                    const uint64_t ad = smem_desc_sw128(a_u32 + as * G::A_SLOT + u * L_A_BYTES);
#pragma unroll
                    for (int kk = 0; kk < L_KC / 16; ++kk) {
                        const uint64_t o = (uint64_t)(kk * 2);   // 32 bytes, in 16 B units
                        mma_bf16(tmem + (uint32_t)(u * L_N), ad + o, bd + o, idesc,
                                 (kc > 0 || kk > 0) ? 1u : 0u);
                    }
                }
                mma_commit(&ctl.a_empty[as]);
                mma_commit(&ctl.b_empty[bs]);
            }
            mma_commit(&ctl.done);
        }
        __syncwarp();
    } else if (warp == L_TMA_A_WARP) {
        // ---------------------------------------------------------------- TMA: codes tiles
        if (lane == 0) {
            prefetch_tensormap(&tmA);
            int issued = 0;
            for (int kc = 0; kc < n_kc; ++kc) {
                const int as = kc % G::A_SLOTS;
                if (kc >= G::A_SLOTS &&
                    !mbar_wait(&ctl.a_empty[as], (uint32_t)(kc / G::A_SLOTS - 1) & 1u, wc.budget)) {
                    *abort_flag = 1;
                    note_timeout(wc, MPQ_TIMEOUT_INFERENCE);
                }
                if (*abort_flag) break;
                // 16-byte aligned tile copies (bf16 codes: x a multiple of 8)
                if (!MPQ_CHECK(((kc * L_KC) & 7) == 0 && ((a_u32 + as * G::A_SLOT) & 15u) == 0u)) {
                    *abort_flag = 1;
                    break;
                }
                mbar_arrive_expect_tx(&ctl.a_full[as], (uint32_t)(nt * L_A_BYTES));
                for (int u = 0; u < nt; ++u)
                    tma_load_2d(a_u32 + as * G::A_SLOT + u * L_A_BYTES, &tmA, kc * L_KC,
                                (tile0 + u) * L_M, &ctl.a_full[as]);
                issued = kc + 1;
            }
            // no copy may land after the CTA is gone
            for (int kc = issued - G::A_SLOTS > 0 ? issued - G::A_SLOTS : 0; kc < issued; ++kc)
                drain_wait(&ctl.a_full[kc % G::A_SLOTS], (uint32_t)(kc / G::A_SLOTS) & 1u, wc,
                           MPQ_TIMEOUT_INFERENCE);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------------- TMA: raw input tiles
        if (lane == 0) {
            prefetch_tensormap(&tmX);
            int issued = 0;
            for (int kc = 0; kc < n_kc; ++kc) {
                const int rs = kc % G::R_SLOTS;
                if (kc >= G::R_SLOTS &&
                    !mbar_wait(&ctl.r_empty[rs], (uint32_t)(kc / G::R_SLOTS - 1) & 1u, wc.budget)) {
                    *abort_flag = 1;
                    note_timeout(wc, MPQ_TIMEOUT_INFERENCE);
                }
                if (*abort_flag) break;
                // 16-byte aligned tile copies (int8 inputs: x a multiple of 16)
                if (!MPQ_CHECK(((kc * L_KC) & 15) == 0 && ((x_u32 + rs * L_RAW_BYTES) & 15u) == 0u)) {
                    *abort_flag = 1;
                    break;
                }
                mbar_arrive_expect_tx(&ctl.r_full[rs], (uint32_t)L_RAW_BYTES);
                tma_load_2d(x_u32 + rs * L_RAW_BYTES, &tmX, kc * L_KC, n0, &ctl.r_full[rs]);
                issued = kc + 1;
            }
            for (int kc = issued - G::R_SLOTS > 0 ? issued - G::R_SLOTS : 0; kc < issued; ++kc)
                drain_wait(&ctl.r_full[kc % G::R_SLOTS], (uint32_t)(kc / G::R_SLOTS) & 1u, wc,
                           MPQ_TIMEOUT_INFERENCE);
        }
        __syncwarp();
    }

    __syncthreads();
    if (warp == L_MMA_WARP) {
        // every MMA has completed: the epilogue waited for `done` (or the wait timed out)
        if (lane == 0 && *abort_flag) drain_wait(&ctl.done, 0, wc, MPQ_TIMEOUT_INFERENCE);
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, G::TMEM_COLS);
    }
}

// The same integer arithmetic on CUDA cores: one thread per (channel, input).
__global__ void multipoint_linear_simt(const int8_t *__restrict__ X, int T, int C, int d, int d_pad,
                                       int rows,
                                       int p, const int *__restrict__ coef,
                                       const int *__restrict__ chan,
                                       const __nv_bfloat16 *__restrict__ codes,
                                       const int *__restrict__ tile_R,
                                       const int *__restrict__ center_coef, int32_t *__restrict__ Y)
{
    const size_t idx = blockIdx.x * (size_t)blockDim.x + threadIdx.x;
    const int slot_row = (int)(idx / T), t = (int)(idx % T);   // slot_row: first row of a channel
    if (slot_row >= rows) return;
    const int R = tile_R[slot_row / L_M];
    if (slot_row % R != 0) return;
    const int k = chan[slot_row];
    if (k < 0 || !MPQ_IN(k, C)) return;
    const int8_t *x = X + (size_t)t * d;
    long long sum = 0;
    for (int i = 0; i < R; ++i) {
        const int r = slot_row + i;
        const __nv_bfloat16 *q = codes + (size_t)r * d_pad;
        long long acc = 0;
        for (int j = 0; j < d; ++j) acc += (long long)__bfloat162float(q[j]) * (long long)x[j];
        sum += (long long)coef[r] * acc;
    }
    if (center_coef) {
        long long xs = 0;
        for (int j = 0; j < d; ++j) xs += x[j];
        sum += (long long)center_coef[k] * xs;
    }
    long long z = sum >> p;
    z = z > 2147483647LL ? 2147483647LL : (z < -2147483648LL ? -2147483648LL : z);
    Y[(size_t)k * T + t] = (int32_t)z;
}

PFN_cuTensorMapEncodeTiled_v12000 lin_map_encoder()
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

int pow2_at_least(int n)
{
    int r = 1;
    while (r < n) r <<= 1;
    return r;
}

}  // namespace

mpq_status make_pack_layout(const int *npoints, int C, int d, int k_max, int bits, int p,
                            int centered, mpq_packed_layout *L)
{
    memset(L, 0, sizeof(*L));
    L->C = C;
    L->d = d;
    L->k_max = k_max;
    L->bits = bits;
    L->p = p;
    L->centered = centered;
    L->d_pad = (d + L_KC - 1) / L_KC * L_KC;
    long long tiles = 0;
    for (int R = 1; R <= MPQ_MAX_POINTS; R <<= 1) {
        long long n = 0;
        for (int k = 0; k < C; ++k) {
            int nk = npoints[k] < 0 ? 0 : (npoints[k] > k_max ? k_max : npoints[k]);
            if (pow2_at_least(nk < 1 ? 1 : nk) == R) ++n;
        }
        tiles += (n + (L_M / R) - 1) / (L_M / R);
    }
    if (tiles * L_M > (1LL << 30)) {
        set_error("packed layer too large");
        return MPQ_ERR_UNSUPPORTED;
    }
    L->tiles = (int)tiles;
    L->rows = (int)(tiles * L_M);
    size_t off = 64;
    L->off_coef = off;
    off += (size_t)L->rows * 4;
    L->off_chan = off;
    off += (size_t)L->rows * 4;
    L->off_point = off;
    off += (size_t)L->rows * 4;
    L->off_tile = off;
    off += (size_t)L->tiles * 4;
    L->off_center = off;
    off += centered ? (size_t)C * 4 : 0;
    off = (off + 1023) / 1024 * 1024;
    L->off_codes = off;
    off += (size_t)L->rows * L->d_pad * 2;
    L->bytes = off;
    return MPQ_OK;
}

mpq_status launch_pack(const int8_t *codes, const float *scales, const float *center,
                       const int *npoints, const mpq_packed_layout *L, void *packed,
                       cudaStream_t stream)
{
    const int C = L->C, rows = L->rows;
    std::vector<int> chan((size_t)rows, -1), point((size_t)rows, -1), tR((size_t)L->tiles, 1);
    int t = 0;
    for (int R = 1; R <= MPQ_MAX_POINTS; R <<= 1) {
        int slot = 0, per = L_M / R;
        for (int k = 0; k < C; ++k) {
            int nk = npoints[k] < 0 ? 0 : (npoints[k] > L->k_max ? L->k_max : npoints[k]);
            if (pow2_at_least(nk < 1 ? 1 : nk) != R) continue;
            if (slot == per) {
                slot = 0;
                ++t;
            }
            tR[(size_t)t] = R;
            for (int i = 0; i < R; ++i) {
                const size_t r = (size_t)t * L_M + (size_t)slot * R + i;
                chan[r] = (i == 0 || i < nk) ? k : -1;   // the first row carries the channel
                point[r] = i < nk ? i : -1;
            }
            ++slot;
        }
        if (slot > 0) ++t;
    }
    if (t != L->tiles) {
        set_error("npoints differ from the ones the layout was made for");
        return MPQ_ERR_INVALID_ARG;
    }
    PackView v = view(L, packed);
    cudaError_t e = cudaMemsetAsync(packed, 0, 64, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(v.chan, chan.data(), (size_t)rows * 4, cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(v.point, point.data(), (size_t)rows * 4, cudaMemcpyHostToDevice, stream);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(v.tile_R, tR.data(), (size_t)L->tiles * 4, cudaMemcpyHostToDevice,
                            stream);
    if (e != cudaSuccess) return cuda_status(e, "packing copies");
    if (rows > 0) {
        pack_kernel<<<rows, 256, 0, stream>>>(codes, scales, C, L->d, L->d_pad, L->k_max, L->p, rows,
                                              v);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_status(e, "pack kernel launch");
    }
    if (L->centered) {
        pack_center_kernel<<<(C + 255) / 256, 256, 0, stream>>>(center, C, L->p, v);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_status(e, "pack center kernel launch");
    }
    int flag = 0;
    e = cudaMemcpyAsync(&flag, v.flag, sizeof(int), cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);   // host arrays above must outlive the copies
    if (e != cudaSuccess) return cuda_status(e, "packing");
    if (flag) {
        set_error("a coefficient rint(2^p * s) or rint(2^p * B) does not fit 32 bits (p = %d)", L->p);
        return MPQ_ERR_UNSUPPORTED;
    }
    return MPQ_OK;
}

mpq_status launch_multipoint_linear(const int8_t *X, int T, const mpq_packed_layout *L,
                                    const void *packed, int32_t *Y, cudaStream_t stream)
{
    PackView v = view(L, const_cast<void *>(packed));
    const int d = L->d, qmax = (1 << (L->bits - 1)) - 1;
    const bool exact = (double)d * qmax * 128.0 < 16777216.0;
    const bool tma = exact && d % 16 == 0 && (uintptr_t)X % 16 == 0 && L->rows > 0;
    if (tma) {
        PFN_cuTensorMapEncodeTiled_v12000 enc = lin_map_encoder();
        CUtensorMap tmA, tmX;
        memset(&tmA, 0, sizeof(tmA));
        memset(&tmX, 0, sizeof(tmX));
        const cuuint64_t da[2] = {(cuuint64_t)L->d_pad, (cuuint64_t)L->rows};
        const cuuint64_t sa[1] = {(cuuint64_t)L->d_pad * 2};
        const cuuint32_t ba[2] = {L_KC, L_M};
        const cuuint64_t dx[2] = {(cuuint64_t)d, (cuuint64_t)T};
        const cuuint64_t sx[1] = {(cuuint64_t)d};
        const cuuint32_t bx[2] = {L_KC, L_N};
        const cuuint32_t es[2] = {1, 1};
        if (!enc ||
            enc(&tmA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, v.codes, da, sa, ba, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
            enc(&tmX, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t *>(X), dx, sx, bx, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            set_error("multipoint linear: tensor map encoding failed");
            return MPQ_ERR_CUDA;
        }
        // two row tiles per CTA when that takes fewer waves of CTAs: such a CTA runs its K loop
        // near the tensor rate but takes ~1.4x as long as a one-tile CTA (measured)
        const long long tt = (T + L_N - 1) / L_N, sms = sm_count();
        const long long w1 = ((long long)L->tiles * tt + sms - 1) / sms;
        const long long w2 = ((long long)((L->tiles + 1) / 2) * tt + sms - 1) / sms;
        const bool two = 7 * w2 < 5 * w1;
        const int smem = two ? lin_smem<2>() : lin_smem<1>();
        if ((long long)smem > max_smem_optin()) {
            set_error("multipoint linear needs %d bytes of shared memory", smem);
            return MPQ_ERR_UNSUPPORTED;
        }
        auto kernel = two ? multipoint_linear_kernel<2> : multipoint_linear_kernel<1>;
        cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");
        const int rt = two ? 2 : 1;
        const dim3 grid((unsigned)tt, (unsigned)((L->tiles + rt - 1) / rt));
        WaitCtl wc;
        const mpq_status wst = wait_ctl(&wc);
        if (wst != MPQ_OK) return wst;
        kernel<<<grid, L_THREADS, smem, stream>>>(T, L->C, L->tiles, L->d_pad / L_KC, L->p, v.coef,
                                                  v.chan, v.tile_R, v.center, Y, wc, tmA, tmX);
        return cuda_status(cudaGetLastError(), "multipoint linear kernel launch");
    }
    const size_t n = (size_t)L->rows * T;
    if (n == 0) return MPQ_OK;
    multipoint_linear_simt<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(
        X, T, L->C, d, L->d_pad, L->rows, L->p, v.coef, v.chan, v.codes, v.tile_R, v.center, Y);
    return cuda_status(cudaGetLastError(), "multipoint linear (integer) kernel launch");
}

}  // namespace mpq
