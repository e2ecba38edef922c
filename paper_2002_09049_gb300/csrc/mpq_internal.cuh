// Internal declarations shared by the CUDA translation units of libmpq.so (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "checks.cuh"
#include "mpq.h"

namespace mpq {

// Devices whose per-device state (cached attributes, resolved symbol addresses) is kept.
constexpr int kMaxDevices = 64;

// acc + comp += v, compensated (Kahan): the rounding error of each addition is carried in comp.
__device__ __forceinline__ void kahan_add(float &acc, float &comp, float v)
{
    const float y = __fsub_rn(v, comp);
    const float t = __fadd_rn(acc, y);
    comp = __fsub_rn(__fsub_rn(t, acc), y);
    acc = t;
}

// sum / N rounded once to fp32 (N exactly representable below 2^24, else in double).
__device__ __forceinline__ float mean_of_sum(float sum, int N)
{
    return N < (1 << 24) ? __fdiv_rn(sum, (float)N) : (float)((double)sum / (double)N);
}


// Records a formatted failure message for mpq_last_error() on the calling thread.
void set_error(const char *fmt, ...);

// Maps a CUDA error to MPQ_ERR_CUDA (recording its text), cudaSuccess to MPQ_OK.
mpq_status cuda_status(cudaError_t e, const char *what);

// `bytes` of device scratch from the current device's default stream-ordered pool, allocated on
// `stream` (free it with cudaFreeAsync on the same stream).  MPQ_ERR_NOMEM if the pool has no room.
mpq_status pool_scratch(void **p, size_t bytes, cudaStream_t stream);

// Multiprocessor count of the current device (cached per device).
int sm_count();

// Opt-in dynamic shared memory limit per block of the current device (cached per device).
int max_smem_optin();

struct GridFrac {
    float f[MPQ_MAX_GRID];
};

// --- launchers, one per kernel family; arguments are already validated ----------------------
mpq_status launch_quantize(const float *W, int C, int d, int qmax, int G, const GridFrac *grid,
                           int k_max, int8_t *codes, float *scales, float *resid_sq,
                           float *residuals, float *rmax, cudaStream_t stream);

// range: scratch of output_error_scratch_words() words for the pair kernel's operand ranges, or
// NULL to take it from the device's stream-ordered pool on `stream`.  rmax (nullable): max |r| of
// every residual vector ([C][k_max+1], from mpq_quantize_layer); the range pre-pass then reads X
// alone and the table holds one word.
mpq_status launch_output_error(const float *X, int N, int groups, const float *W,
                               const int8_t *codes, const float *scales, int C, int d, int k_max,
                               float *err, cudaStream_t stream, unsigned *range = nullptr,
                               const float *rmax = nullptr);
// Words of range scratch a call needs (0 where it takes no scratch).
size_t output_error_scratch_words(const float *X, int groups, const float *W,
                                  const int8_t *codes, int C, int d, int k_max);

mpq_status launch_output_error_tc(const float *X, int N, const float *W, const int8_t *codes,
                                  const float *scales, int C, int d, int k_max, float *err,
                                  cudaStream_t stream);

// CTA-pair tensor-core kernel: needs d % 16 == 0 and 16-byte aligned X, W and codes.
bool output_error_pair_ok(const float *X, const float *W, const int8_t *codes, int d);
mpq_status launch_output_error_pair(const float *X, int N, const float *W, const int8_t *codes,
                                    const float *scales, int C, int d, int k_max, float *err,
                                    cudaStream_t stream, unsigned *range, const float *rmax);

// Clipping-search errors on the CTA-pair fp16 contraction (output_error_f16.cu): chmax = max|w|
// per channel; scratch of clip_f16_scratch_bytes() bytes, 256-byte aligned, on `stream`.  Needs
// output_error_pair_ok(X, W, W, d).
size_t clip_f16_scratch_bytes(int C, int N, int d, int n_cand);
mpq_status launch_clip_f16(const float *X, int N, const float *W, const float *clip,
                           const float *chmax, int C, int d, int qmax, int n_cand, float *err,
                           void *scratch, cudaStream_t stream);
mpq_status launch_clip(const float *X, int N, int groups, const float *W, int C, int d, int qmax,
                       int n_cand, int mode, float *clip, float *err, int *best,
                       cudaStream_t stream);

mpq_status make_pack_layout(const int *npoints, int C, int d, int k_max, int bits, int p,
                            int centered, mpq_packed_layout *L);
mpq_status launch_pack(const int8_t *codes, const float *scales, const float *center,
                       const int *npoints, const mpq_packed_layout *L, void *packed,
                       cudaStream_t stream);
mpq_status launch_multipoint_linear(const int8_t *X, int T, const mpq_packed_layout *L,
                                    const void *packed, int32_t *Y, cudaStream_t stream);

mpq_status launch_allocate_budget(const float *err, int C, int k_max, long long extra,
                                  int *npoints, int *points_used, cudaStream_t stream);

// Several layers, one CTA each (n <= MPQ_MAX_BATCH; extra for budget mode, eps for threshold mode).
mpq_status launch_allocate_batch(int n, const float *const *err, const int *C, int k_max,
                                 int mode, const long long *extra, const double *eps,
                                 int *const *npoints, int *const *points_used, cudaStream_t stream);

mpq_status launch_allocate_threshold(const float *err, int C, int k_max, double eps,
                                     int *npoints, int *points_used, cudaStream_t stream);

mpq_status launch_reconstruct(const int8_t *codes, const float *scales, const int *npoints,
                              const float *center, int C, int d, int k_max, float *W_hat,
                              cudaStream_t stream);
mpq_status launch_adaptive(const float *W, int C, int d, int qmax, int k_max, double eta,
                           long long max_cand, int8_t *codes, float *scales, float *resid_sq,
                           long long *ncand, cudaStream_t stream);

mpq_status launch_center(const float *W, int C, int d, int mode, float *center, float *Wc,
                         cudaStream_t stream);

}  // namespace mpq
