// Pieces shared by the CTA-pair output-error kernels (Sec. 3.3, Eq. 11): the power-of-two scaling
// and fp16 hi/lo split of the contraction's operands, the pairing of a warp's two channels for
// conflict-free operand stores, and tile-map encoding for the TMA copies.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <math.h>
#include <stdint.h>

#include "mpq.h"

namespace mpq {

// fp16 operands: exponent e with m * 2^e in [2^14, 2^15) for the largest magnitude m of a residual
// vector or of X, so that the vector's hi and lo halves are normal fp16 numbers down to 2^-7 of its
// largest element (and nothing overflows).  0 for m = 0, NaN or inf (which then propagate); capped
// at 126 so that 2^e stays a normal float (only vectors below 2^-111 are scaled less).
__device__ __forceinline__ int f16_scale_exp(float m)
{
    if (!(m > 0.0f) || !isfinite(m)) return 0;
    int E;
    (void)frexpf(m, &E);              // m = f 2^E, f in [0.5, 1)
    return min(15 - E, 126);
}

__device__ __forceinline__ float pow2f(int e) { return __int_as_float((127 + e) << 23); }

__device__ __forceinline__ double pow2d(int e)
{
    return __longlong_as_double((long long)(1023 + e) << 52);
}

// x * 2^e (exact) split into fp16 hi + lo: hi = fl16(x), lo = fl16(x - hi) (x - hi is exact in fp32).
__device__ __forceinline__ void split_f16x2(float a, float b, uint32_t &hi, uint32_t &lo)
{
    const __half2 h = __floats2half2_rn(a, b);
    const float2 hf = __half22float2(h);
    const __half2 l = __floats2half2_rn(__fsub_rn(a, hf.x), __fsub_rn(b, hf.y));
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

// fp16 operand stores fill 64-byte half rows of a 128-byte-swizzled tile, and the swizzle puts a
// half row in banks 0-15 or 16-31 by bit 2 of its row.  The two channels of a warp's residual
// items (slots j = 2t, 2t+1: lanes 0-15 and 16-31) are D apart, with D (k_max+1) = 4 (mod 8) where
// possible, so that their rows differ in bit 2.  A bijection of the slots 0..nch-1: blocks of 2D
// slots pair channel i with i + D; a last partial block of T slots pairs its first T - D channels
// so and keeps the rest in place.
template <int KP1>
__device__ __forceinline__ int pair_channel(int j, int nch)
{
    constexpr int D = (KP1 & 1) ? 4 : ((KP1 & 3) == 2 ? 2 : 1);
    const int F = nch / (2 * D) * (2 * D);
    if (j < F) {
        const int w = j % (2 * D);
        return j - w + (w >> 1) + (w & 1) * D;
    }
    const int T = nch - F, m = T > D ? T - D : 0, s = j - F;
    return s < 2 * m ? F + (s >> 1) + (s & 1) * D : F + m + (s - 2 * m);
}

// Host: tile map over a row-major tensor (dims[0] contiguous, byte strides for dims 1..), zero
// fill out of range, the given shared-memory swizzle.  False if the driver entry point is missing
// or rejects the arguments.
bool encode_tile_map(CUtensorMap *m, CUtensorMapDataType type, int rank, const void *base,
                     const cuuint64_t *dims, const cuuint64_t *strides, const cuuint32_t *box,
                     CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_NONE);

// Host: max|X| (float bits) into range[0], zeroed first (N d a multiple of 4, X 16-byte aligned).
mpq_status launch_x_range(const float *X, int N, int d, unsigned *range, cudaStream_t stream);

// Host: the output error of the greedy residuals on output_error_f16.cu's kernel, with its range
// table ready on `stream` (xrange[0] = max|X|, vrange = max|r| per residual vector, float bits)
// and `xs` scratch of 2 N d fp16 for the split X planes.
mpq_status launch_output_error_f16(const float *X, int N, const float *W, const int8_t *codes,
                                   const float *scales, int C, int d, int k_max, float *err,
                                   const unsigned *xrange, const unsigned *vrange, uint16_t *xs,
                                   cudaStream_t stream);

}  // namespace mpq
