// Multipoint weights (Eq. 4): W_hat[k][j] = B_k + sum_{i=1..n_k} s_{k,i} q_{k,i,j}, accumulated as
// acc = fmaf(s_{k,i}, q_{k,i,j}, acc) from the set's centre B_k (Eq. 1; 0 for symmetric sets) in
// the order i = 1, 2, ...; n_k clamped to [0, k_max].
// Memory-bound: each element reads n_k code bytes and writes one fp32; four elements per thread
// when d allows 16-byte stores.
#include "mpq_internal.cuh"

MPQ_CHECKED_UNIT("reconstruct.cu");

namespace mpq {
namespace {

constexpr int RC_THREADS = 256;

__global__ void __launch_bounds__(RC_THREADS)
reconstruct_kernel(const int8_t *__restrict__ codes, const float *__restrict__ scales,
                   const int *__restrict__ npoints, const float *__restrict__ center, int C, int d,
                   int k_max, float *__restrict__ W_hat)
{
    const size_t plane = (size_t)C * d;
    const size_t total = plane;
    for (size_t idx = (size_t)blockIdx.x * RC_THREADS + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * RC_THREADS) {
        const int k = (int)(idx / d);
        if (!MPQ_IN(k, C)) continue;
        int n = npoints[k];
        n = n < 0 ? 0 : (n > k_max ? k_max : n);
        float acc = center ? center[k] : 0.0f;
        for (int i = 0; i < n; ++i)
            acc = __fmaf_rn(scales[(size_t)k * k_max + i], (float)codes[(size_t)i * plane + idx], acc);
        W_hat[idx] = acc;
    }
}

// d % 4 == 0: four consecutive elements of one channel per thread (char4 code loads, float4
// stores).
__global__ void __launch_bounds__(RC_THREADS)
reconstruct_vec4_kernel(const int8_t *__restrict__ codes, const float *__restrict__ scales,
                        const int *__restrict__ npoints, const float *__restrict__ center, int C,
                        int d, int k_max, float *__restrict__ W_hat)
{
    const size_t plane = (size_t)C * d;
    const size_t total4 = plane / 4;
    for (size_t q = (size_t)blockIdx.x * RC_THREADS + threadIdx.x; q < total4;
         q += (size_t)gridDim.x * RC_THREADS) {
        const size_t idx = q * 4;
        const int k = (int)(idx / d);
        // four elements of one channel, 4-byte code and 16-byte output alignment
        if (!MPQ_IN(k, C) || !MPQ_IN(idx + 3, plane) || !MPQ_CHECK(idx / d == (idx + 3) / d) ||
            !MPQ_CHECK(((uintptr_t)codes & 3) == 0 && ((uintptr_t)(W_hat + idx) & 15) == 0))
            continue;
        int n = npoints[k];
        n = n < 0 ? 0 : (n > k_max ? k_max : n);
        const float b = center ? center[k] : 0.0f;
        float a0 = b, a1 = b, a2 = b, a3 = b;
        for (int i = 0; i < n; ++i) {
            const float s = scales[(size_t)k * k_max + i];
            const char4 c = *reinterpret_cast<const char4 *>(codes + (size_t)i * plane + idx);
            a0 = __fmaf_rn(s, (float)c.x, a0);
            a1 = __fmaf_rn(s, (float)c.y, a1);
            a2 = __fmaf_rn(s, (float)c.z, a2);
            a3 = __fmaf_rn(s, (float)c.w, a3);
        }
        *reinterpret_cast<float4 *>(W_hat + idx) = make_float4(a0, a1, a2, a3);
    }
}

}  // namespace

mpq_status launch_reconstruct(const int8_t *codes, const float *scales, const int *npoints,
                              const float *center, int C, int d, int k_max, float *W_hat,
                              cudaStream_t stream)
{
    const size_t total = (size_t)C * d;
    const bool vec = (d % 4 == 0) && ((uintptr_t)codes % 4 == 0) && ((uintptr_t)W_hat % 16 == 0);
    const size_t items = vec ? total / 4 : total;
    size_t blocks = (items + RC_THREADS - 1) / RC_THREADS;
    const size_t cap = (size_t)sm_count() * 8;
    if (blocks > cap) blocks = cap;
    if (vec)
        reconstruct_vec4_kernel<<<(unsigned)blocks, RC_THREADS, 0, stream>>>(
            codes, scales, npoints, center, C, d, k_max, W_hat);
    else
        reconstruct_kernel<<<(unsigned)blocks, RC_THREADS, 0, stream>>>(
            codes, scales, npoints, center, C, d, k_max, W_hat);
    return cuda_status(cudaGetLastError(), "reconstruct kernel launch");
}

}  // namespace mpq
