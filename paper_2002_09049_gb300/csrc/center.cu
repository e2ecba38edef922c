// Asymmetric quantization sets (Eq. 1 with B != 0): the centre B of K x [-1 : eps_b : 1] + B is the
// midpoint of the weights' range, (max w + min w) / 2 rounded once to fp32, per channel or for the
// whole layer, and the centred weights Wc = fl(w - B) are what the greedy points approximate.
// One warp per channel reads its row twice (the second time from L1/L2): range, then Wc.  Per
// layer: the channels' ranges, one CTA for the layer's B, then Wc.  Memory-bound: 4 B read and 4 B
// written per weight.
#include <math.h>

#include "mpq_internal.cuh"

MPQ_CHECKED_UNIT("center.cu");

namespace mpq {
namespace {

constexpr int CT_THREADS = 256;

// (hi + lo) / 2 in double, then one rounding to fp32 (the exact midpoint of two fp32 values of a
// weight range is representable in double).
__device__ __forceinline__ float midpoint(float hi, float lo)
{
    return (float)(((double)hi + (double)lo) * 0.5);
}

// Channel k's range (warp-wide), with `bad` set if a weight is not finite.
__device__ __forceinline__ void channel_range(const float *w, int d, int lane, float &hi, float &lo,
                                              int &bad)
{
    hi = -INFINITY;
    lo = INFINITY;
    bad = 0;
    for (int j = lane; j < d; j += 32) {
        const float v = w[j];
        bad |= !isfinite(v);
        hi = fmaxf(hi, v);
        lo = fminf(lo, v);
    }
    for (int o = 16; o > 0; o >>= 1) {
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
}

enum { PASS_CHANNEL = 0, PASS_RANGE = 1, PASS_APPLY = 2 };

// PASS_CHANNEL: B_k and Wc in one pass.  PASS_RANGE (per layer, first): each channel's maximum
// goes to center[k] and its minimum to Wc[k] (NaN for a non-finite channel) for
// center_layer_kernel.  PASS_APPLY (per layer, last): Wc from the layer's B in center[k].
__global__ void __launch_bounds__(CT_THREADS)
center_channel_kernel(const float *__restrict__ W, int C, int d, int pass, float *__restrict__ center,
                      float *__restrict__ Wc)
{
    const int k = (int)((blockIdx.x * (size_t)blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (k >= C) return;
    const float *w = W + (size_t)k * d;
    float b;
    if (pass == PASS_APPLY) {
        b = center[k];
    } else {
        float hi, lo;
        int bad;
        channel_range(w, d, lane, hi, lo, bad);
        if (pass == PASS_RANGE) {
            if (lane == 0) {
                center[k] = bad ? NAN : hi;
                Wc[k] = bad ? NAN : lo;
            }
            return;
        }
        b = bad ? NAN : midpoint(hi, lo);
        if (lane == 0) center[k] = b;
    }
    float *out = Wc + (size_t)k * d;
    for (int j = lane; j < d; j += 32)
        if (MPQ_IN((size_t)k * d + j, (size_t)C * d)) out[j] = __fsub_rn(w[j], b);
}

// One CTA: the layer's B from the channels' ranges, written to every center[k].
__global__ void center_layer_kernel(int C, float *__restrict__ center, const float *__restrict__ lo_in)
{
    __shared__ float sh[32], sl[32];
    __shared__ int sb[32];
    float hi = -INFINITY, lo = INFINITY;
    int bad = 0;
    for (int k = threadIdx.x; k < C; k += blockDim.x) {
        const float h = center[k], l = lo_in[k];
        bad |= isnan(h);
        hi = fmaxf(hi, h);
        lo = fminf(lo, l);
    }
    for (int o = 16; o > 0; o >>= 1) {
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        sh[warp] = hi;
        sl[warp] = lo;
        sb[warp] = bad;
    }
    __syncthreads();   // every read of the ranges is done before center is overwritten
    hi = -INFINITY;
    lo = INFINITY;
    bad = 0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
        hi = fmaxf(hi, sh[i]);
        lo = fminf(lo, sl[i]);
        bad |= sb[i];
    }
    const float b = bad ? NAN : midpoint(hi, lo);
    for (int k = threadIdx.x; k < C; k += blockDim.x) center[k] = b;
}

}  // namespace

mpq_status launch_center(const float *W, int C, int d, int mode, float *center, float *Wc,
                         cudaStream_t stream)
{
    const unsigned blocks = (unsigned)(((size_t)C * 32 + CT_THREADS - 1) / CT_THREADS);
    const bool layer = mode == MPQ_CENTER_PER_LAYER;
    center_channel_kernel<<<blocks, CT_THREADS, 0, stream>>>(W, C, d, layer ? PASS_RANGE : PASS_CHANNEL,
                                                             center, Wc);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !layer) return cuda_status(e, "center kernel launch");
    center_layer_kernel<<<1, 1024, 0, stream>>>(C, center, Wc);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_status(e, "center layer kernel launch");
    center_channel_kernel<<<blocks, CT_THREADS, 0, stream>>>(W, C, d, PASS_APPLY, center, Wc);
    return cuda_status(cudaGetLastError(), "center apply kernel launch");
}

}  // namespace mpq
