// Output-error-driven clipping factor (Sec. 3.3, Eq. 12):
//   K* = argmin_K sum_{w in W} E_x (w^T x - w~^T x)^2,   w~ = [w]_Q,  Q = K x [-1 : eps_b : 1],
// over the candidate grid K_c = (c+1)/n_cand x max|w| (n_cand = 20: the experiments' grid
// [0.05 : 0.05 : 1] x max|w|), with W one channel (per-channel sets) or the whole layer (one K).
// The quantized weight is s q with s = K / Qmax and q the exact codes of Eq. 8, and its residual
// fmaf(-s, q, w) feeds the output error of Eq. 11.
//
// Three steps, all on the device:
//   1. candidates: one warp per channel takes max|w| (NaN if a weight is non-finite); per-layer
//      sets reduce the channels' maxima in one CTA;
//   2. errors: the CTA-pair tensor-core contraction with residuals generated from W and the
//      candidate scales on chip (output_error_f16.cu: fp16 hi/lo operands, each residual vector
//      scaled by a power of two from the bound max(min(max|w|, s/2), max|w| - Qmax s) on its
//      elements), or,
//      for rows that are not 16-byte multiples and for per-channel inputs, one CTA per channel
//      and candidate chunk with the residuals in shared memory and threads over the calibration
//      rows;
//   3. argmin: per channel, or per layer over the channel sums (double, channels in order).
#include <math.h>

#include "mpq_internal.cuh"
#include "rounding.cuh"

MPQ_CHECKED_UNIT("clip.cu");

namespace mpq {
namespace {

constexpr int CL_THREADS = 256;
constexpr int CL_CHUNK = 8;   // candidates per CTA in the shared-memory path

__device__ __forceinline__ float candidate_fraction(int c, int n_cand)
{
    return __fdiv_rn((float)(c + 1), (float)n_cand);
}

// One warp per channel: m = max|w| (NaN when a weight is not finite), also into chmax[k] when
// given.  Per channel, the candidate row K_c = f_c m; per layer, m is parked in column 0 for
// clip_layer_kernel.
__global__ void clip_channel_kernel(const float *__restrict__ W, int C, int d, int n_cand, int mode,
                                    float *__restrict__ clip, float *__restrict__ chmax)
{
    const int k = (int)((blockIdx.x * (size_t)blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (k >= C) return;
    const float *w = W + (size_t)k * d;
    float m = 0.0f;
    int bad = 0;
    for (int j = lane; j < d; j += 32) {
        const float v = w[j];
        bad |= !isfinite(v);
        m = fmaxf(m, fabsf(v));
    }
    for (int o = 16; o > 0; o >>= 1) {
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    if (bad) m = NAN;
    if (chmax && lane == 0) chmax[k] = m;
    if (mode == MPQ_CLIP_PER_CHANNEL) {
        for (int c = lane; c < n_cand; c += 32)
            clip[(size_t)k * n_cand + c] = __fmul_rn(candidate_fraction(c, n_cand), m);
    } else if (lane == 0) {
        clip[(size_t)k * n_cand] = m;
    }
}

// One CTA: the layer's m = max over the channels (NaN if any channel's is), then every row.
__global__ void clip_layer_kernel(int C, int n_cand, float *__restrict__ clip)
{
    __shared__ float wm[32];
    __shared__ int wb[32];
    float m = 0.0f;
    int bad = 0;
    for (int k = threadIdx.x; k < C; k += blockDim.x) {
        const float v = clip[(size_t)k * n_cand];
        bad |= isnan(v);
        m = fmaxf(m, v);
    }
    for (int o = 16; o > 0; o >>= 1) {
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        wm[warp] = m;
        wb[warp] = bad;
    }
    __syncthreads();   // every read of column 0 is done before the rows are written
    m = 0.0f;
    bad = 0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
        m = fmaxf(m, wm[i]);
        bad |= wb[i];
    }
    if (bad) m = NAN;
    for (size_t i = threadIdx.x; i < (size_t)C * n_cand; i += blockDim.x)
        clip[i] = __fmul_rn(candidate_fraction((int)(i % n_cand), n_cand), m);
}

// One CTA per (channel, chunk of CL_CHUNK candidates): residuals r_c = fmaf(-s_c, q_c, w) in
// shared memory, threads over the calibration rows, fp32 dot products, squares summed in fp32
// (16-row partial sums, a compensated sum per thread, a tree over the threads).
__global__ void __launch_bounds__(CL_THREADS)
clip_errors_kernel(const float *__restrict__ X, int N, int groups, const float *__restrict__ W,
                   int C, int d, int qmax, int n_cand, const float *__restrict__ clip,
                   float *__restrict__ err)
{
    extern __shared__ __align__(16) float R[];   // [CL_CHUNK][d]
    __shared__ float red[CL_THREADS / 32][CL_CHUNK];
    const int k = blockIdx.x, c0 = blockIdx.y * CL_CHUNK;
    const int nc = min(CL_CHUNK, n_cand - c0);
    if (!MPQ_IN(k, C) || !MPQ_CHECK(nc >= 1) || !MPQ_CHECK_SMEM_END(4 * (size_t)nc * d)) return;
    const float qmaxf = (float)qmax;
    const float *w = W + (size_t)k * d;
    for (int i = threadIdx.x; i < nc * d; i += CL_THREADS) {
        const int c = i / d, j = i % d;
        const float s = __fdiv_rn(clip[(size_t)k * n_cand + c0 + c], qmaxf);
        const float v = w[j];
        const float q = s > 0.0f ? copysignf((float)code_mag(fabsf(v), s, qmaxf), v) : 0.0f;
        R[i] = __fmaf_rn(-s, q, v);
    }
    __syncthreads();
    const float *Xk = groups == 1 ? X : X + (size_t)k * N * d;
    // all in fp32 (fp64 throughput is a small fraction of fp32's on this part): squares summed over
    // at most 16 rows of a thread, folded into a compensated sum, then a tree over the threads
    float acc[CL_CHUNK], comp[CL_CHUNK], part[CL_CHUNK];
#pragma unroll
    for (int c = 0; c < CL_CHUNK; ++c) {
        acc[c] = 0.0f;
        comp[c] = 0.0f;
        part[c] = 0.0f;
    }
    int rows = 0;
    for (int t = threadIdx.x; t < N; t += CL_THREADS) {
        const float *x = Xk + (size_t)t * d;
        float y[CL_CHUNK];
#pragma unroll
        for (int c = 0; c < CL_CHUNK; ++c) y[c] = 0.0f;
        for (int j = 0; j < d; ++j) {
            const float xv = x[j];
#pragma unroll
            for (int c = 0; c < CL_CHUNK; ++c)
                if (c < nc) y[c] = fmaf(xv, R[c * d + j], y[c]);
        }
#pragma unroll
        for (int c = 0; c < CL_CHUNK; ++c) part[c] = fmaf(y[c], y[c], part[c]);
        if (++rows == 16) {
#pragma unroll
            for (int c = 0; c < CL_CHUNK; ++c) {
                kahan_add(acc[c], comp[c], part[c]);
                part[c] = 0.0f;
            }
            rows = 0;
        }
    }
    const int lane = threadIdx.x & 31, wp = threadIdx.x >> 5;
#pragma unroll
    for (int c = 0; c < CL_CHUNK; ++c) {
        kahan_add(acc[c], comp[c], part[c]);
        float v = acc[c];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) red[wp][c] = v;
    }
    __syncthreads();
    if (threadIdx.x < nc) {
        float v[CL_THREADS / 32];
        for (int i = 0; i < CL_THREADS / 32; ++i) v[i] = red[i][threadIdx.x];
        for (int w = CL_THREADS / 64; w > 0; w >>= 1)   // tree over the warps
            for (int i = 0; i < w; ++i) v[i] += v[i + w];
        if (MPQ_IN((size_t)k * n_cand + c0 + threadIdx.x, (size_t)C * n_cand))
            err[(size_t)k * n_cand + c0 + threadIdx.x] = mean_of_sum(v[0], N);
    }
}

// Per channel: the lowest c with the smallest err[k][c]; NaN never wins, none finite gives -1.
__global__ void clip_select_channel_kernel(const float *__restrict__ err, int C, int n_cand,
                                           int *__restrict__ best)
{
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= C) return;
    int b = -1;
    float bv = 0.0f;
    for (int c = 0; c < n_cand; ++c) {
        const float v = err[(size_t)k * n_cand + c];
        if (isnan(v)) continue;
        if (b < 0 || v < bv) {
            b = c;
            bv = v;
        }
    }
    best[k] = b;
}

// Per layer (one CTA): lane c sums column c over the channels in order (double); the lowest c with
// the smallest sum goes to every channel.
__global__ void clip_select_layer_kernel(const float *__restrict__ err, int C, int n_cand,
                                         int *__restrict__ best)
{
    __shared__ int pick;
    if (threadIdx.x < 32) {
        const int c = threadIdx.x;
        double e = 0.0;
        if (c < n_cand)
            for (int k = 0; k < C; ++k) e += (double)err[(size_t)k * n_cand + c];
        const bool ok = c < n_cand && !isnan(e);
        int b = -1;
        double bv = 0.0;
        for (int i = 0; i < n_cand; ++i) {   // in candidate order: the lowest index keeps ties
            const double ei = __shfl_sync(0xffffffffu, e, i);
            const int oki = __shfl_sync(0xffffffffu, (int)ok, i);
            if (oki && (b < 0 || ei < bv)) {
                b = i;
                bv = ei;
            }
        }
        if (threadIdx.x == 0) pick = b;
    }
    __syncthreads();
    for (int k = threadIdx.x; k < C; k += blockDim.x) best[k] = pick;
}

}  // namespace

mpq_status launch_clip(const float *X, int N, int groups, const float *W, int C, int d, int qmax,
                       int n_cand, int mode, float *clip, float *err, int *best,
                       cudaStream_t stream)
{
    // the tensor-core path takes all its scratch from the stream-ordered pool before anything is
    // enqueued: channel maxima, then the contraction's (X range and planes, residual planes)
    const bool tc = groups == 1 && output_error_pair_ok(X, W, reinterpret_cast<const int8_t *>(W), d);
    const size_t max_bytes = ((size_t)C * sizeof(float) + 255) / 256 * 256;
    char *scratch = nullptr;
    if (tc) {
        const mpq_status st = pool_scratch(reinterpret_cast<void **>(&scratch),
                                           max_bytes + clip_f16_scratch_bytes(C, N, d, n_cand),
                                           stream);
        if (st != MPQ_OK) return st;
    }
    float *chmax = reinterpret_cast<float *>(scratch);
    const unsigned blocks = (unsigned)(((size_t)C * 32 + CL_THREADS - 1) / CL_THREADS);
    clip_channel_kernel<<<blocks, CL_THREADS, 0, stream>>>(W, C, d, n_cand, mode, clip, chmax);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess && mode == MPQ_CLIP_PER_LAYER) {
        clip_layer_kernel<<<1, 1024, 0, stream>>>(C, n_cand, clip);
        e = cudaGetLastError();
    }
    if (tc) {
        mpq_status st = cuda_status(e, "clip candidate kernel launch");
        if (st == MPQ_OK)
            st = launch_clip_f16(X, N, W, clip, chmax, C, d, qmax, n_cand, err, scratch + max_bytes,
                                 stream);
        const cudaError_t ef = cudaFreeAsync(scratch, stream);
        if (st == MPQ_OK) st = cuda_status(ef, "scratch release (cudaFreeAsync)");
        if (st != MPQ_OK) return st;
    } else {
        if (e != cudaSuccess) return cuda_status(e, "clip candidate kernel launch");
        const size_t smem = (size_t)CL_CHUNK * d * sizeof(float);
        if ((long long)smem > max_smem_optin()) {
            set_error("clip search with d = %d needs %zu bytes of shared memory", d, smem);
            return MPQ_ERR_UNSUPPORTED;
        }
        e = cudaFuncSetAttribute(clip_errors_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute");
        const dim3 grid((unsigned)C, (unsigned)((n_cand + CL_CHUNK - 1) / CL_CHUNK));
        clip_errors_kernel<<<grid, CL_THREADS, smem, stream>>>(X, N, groups, W, C, d, qmax, n_cand,
                                                              clip, err);
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_status(e, "clip error kernel launch");
    }

    if (mode == MPQ_CLIP_PER_CHANNEL)
        clip_select_channel_kernel<<<(C + CL_THREADS - 1) / CL_THREADS, CL_THREADS, 0, stream>>>(
            err, C, n_cand, best);
    else
        clip_select_layer_kernel<<<1, 1024, 0, stream>>>(err, C, n_cand, best);
    e = cudaGetLastError();
    return cuda_status(e, "clip select kernel launch");
}

}  // namespace mpq
