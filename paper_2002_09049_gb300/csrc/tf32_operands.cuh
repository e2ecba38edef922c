// Operand preparation shared by the tensor-core output-error kernels: the exact fp32 -> tf32 hi/lo
// split of Sec. 3.3's contraction operands, exact int8 code -> float conversion and the byte
// offsets of the K-major swizzled shared-memory tiles the UMMA descriptors describe.
#pragma once

#include <stdint.h>

namespace mpq {

// x = hi + lo exactly: hi keeps sign, exponent and the top 10 mantissa bits (a tf32 value).
__device__ __forceinline__ void split4(const float4 x, float4 &hi, float4 &lo)
{
    hi.x = __uint_as_float(__float_as_uint(x.x) & 0xFFFFE000u);
    hi.y = __uint_as_float(__float_as_uint(x.y) & 0xFFFFE000u);
    hi.z = __uint_as_float(__float_as_uint(x.z) & 0xFFFFE000u);
    hi.w = __uint_as_float(__float_as_uint(x.w) & 0xFFFFE000u);
    lo.x = __fsub_rn(x.x, hi.x);
    lo.y = __fsub_rn(x.y, hi.y);
    lo.z = __fsub_rn(x.z, hi.z);
    lo.w = __fsub_rn(x.w, hi.w);
}

// Code byte b (0..3) of `biased` (int8 codes XOR 0x80 per byte) as an exact float: the byte
// becomes the low mantissa byte of 2^23, and subtracting 2^23 + 128 is exact.
__device__ __forceinline__ float code_from_biased(uint32_t biased, int b)
{
    return __fsub_rn(__uint_as_float(__byte_perm(biased, 0x4B000000u, 0x7650u + (uint32_t)b)),
                     8388736.0f);
}

// Byte offset of 16-byte chunk `chunk` (0..7) of row `row` of a K-major tile with 128-byte rows in
// the 128-byte swizzle layout: 8-row atoms of 1024 bytes, chunk XOR the row within the atom.
__device__ __forceinline__ uint32_t sw128_offset(int row, int chunk)
{
    return (uint32_t)((row >> 3) * 1024 + (row & 7) * 128 + ((chunk ^ (row & 7)) << 4));
}

}  // namespace mpq
