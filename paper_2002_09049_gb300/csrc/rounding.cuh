// Exact codes of Eq. 8 for a symmetric b-bit set: c = min(Qmax, rint(fl(a / s))) for a = |r| >= 0 and
// scale s > 0, with fl the correctly rounded fp32 division and rint ties-to-even -- and a fast path
// that reaches the same integer from a multiply by a reciprocal whenever the quotient is not too
// close to a rounding boundary.  Shared by the greedy search and the clipping-factor search.
#pragma once

namespace mpq {

// Code magnitude of |r| at scale s > 0 (Eq. 8): nearest integer (ties to even) of the correctly
// rounded fp32 quotient, clipped to Qmax.
__device__ __forceinline__ int code_mag(float a, float s, float qmaxf)
{
    return (int)fminf(rintf(__fdiv_rn(a, s)), qmaxf);
}

// Bound on |a * fl(1/s) - fl(a/s)| relative to the quotient, with margin: both roundings are
// 2^-24 each, so a fast quotient further than this from a rounding boundary decides exactly as
// the correctly rounded division would.
#define MPQ_FAST_REL 9.5367431640625e-07f /* 2^-20 */

// min(Qmax, rint(fl(a/s))), decided from q' = a * (1/s) unless q' is too close to a half-integer:
// then q' and the exact quotient round to the same integer (no tie can lie between them).
__device__ __forceinline__ int code_fast(float a, float s, float inv_s, float qmaxf)
{
    const float qf = __fmul_rn(a, inv_s);
    const float rq = rintf(qf);
    if (0.5f - fabsf(qf - rq) > MPQ_FAST_REL * (qf + 1.0f)) return (int)fminf(rq, qmaxf);
    return (int)fminf(rintf(__fdiv_rn(a, s)), qmaxf);
}

// code_fast as a float (the same integer value).
__device__ __forceinline__ float code_fast_f(float a, float s, float inv_s, float qmaxf)
{
    const float qf = __fmul_rn(a, inv_s);
    const float rq = rintf(qf);
    if (0.5f - fabsf(qf - rq) > MPQ_FAST_REL * (qf + 1.0f)) return fminf(rq, qmaxf);
    return fminf(rintf(__fdiv_rn(a, s)), qmaxf);
}

// Signed code clamp(rint(w (1/s)), -Qmax, Qmax) without a branch, for clamp(rint(fl(w/s)), ...)
// (Eq. 8 with the sign of w; rint and fl are symmetric).  `unsure` is set where the two may differ:
// |q'| < Qmax + 1 = qlim and q' within 0.5 - tband of a half-integer, tband = 0.5 - 2^-20 (qlim + 1)
// (at least MPQ_FAST_REL (|q'| + 1) for every |q'| < qlim).  At |q'| >= qlim both clamp to +-Qmax.
// inv_s = 0 gives q = 0 (scales 0 or NaN).
__device__ __forceinline__ float code_signed_fast(float w, float inv_s, float qmaxf, float qlim,
                                                  float tband, bool &unsure)
{
    const float qf = __fmul_rn(w, inv_s);
    const float rq = rintf(qf);
    unsure |= fabsf(__fsub_rn(qf, rq)) >= tband && fabsf(qf) < qlim;
    return fminf(fmaxf(rq, -qmaxf), qmaxf);
}

// The exact signed code clamp(rint(fl(w/s)), -Qmax, Qmax) for s > 0, 0 otherwise.
__device__ __forceinline__ float code_signed_exact(float w, float s, float qmaxf)
{
    return s > 0.0f ? fminf(fmaxf(rintf(__fdiv_rn(w, s)), -qmaxf), qmaxf) : 0.0f;
}

}  // namespace mpq
