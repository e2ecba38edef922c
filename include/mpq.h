/*
 * mpq.h -- C ABI of the GB300 multipoint post-training quantization library (libmpq.so).
 *
 * Method: Liu et al., "Post-training Quantization with Multiple Points: Mixed Precision without
 * Mixed Precision" (arXiv 2002.09049).  A weight channel w (d values) is approximated by
 * n points, w~ = sum_i a_i w~_i (Eq. 4), built greedily one point at a time from the residual
 * (Eq. 6-9, Algorithm 1); the number of points of each channel is chosen from its output error on
 * calibration inputs (Eq. 11, Algorithm 2).
 *
 * Representation.  A point i of channel k is a pair (s_{k,i}, q_{k,i}): an fp32 scale and a
 * vector of d integer codes in {-Qmax..Qmax}, Qmax = 2^(b-1) - 1, stored as int8.  The paper's
 * a_i * [r/a_i]_Q with Q = [-1 : 1/Qmax : 1] (Eq. 1) is s_i * q_i with s_i = a_i / Qmax.
 *
 * Conventions shared by every entry point:
 *  - All array arguments are DEVICE pointers, allocated and owned by the caller, row-major,
 *    on the device that is current when the call is made, unless an argument says "host".
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).  Every call
 *    only enqueues work on `stream` and returns; results are ready when the stream reaches them.
 *    No entry point synchronizes, and none allocates device memory except the scratch of
 *    mpq_output_error, mpq_clip_search and mpq_quantize_layer_adaptive, which comes from the
 *    device's stream-ordered pool on `stream` and goes back to it on `stream` (see there).
 *  - Arguments are validated on the host before anything is enqueued; an invalid argument
 *    returns MPQ_ERR_INVALID_ARG / MPQ_ERR_UNSUPPORTED and leaves every output untouched.
 *    A failed kernel launch returns MPQ_ERR_CUDA.  mpq_last_error() gives a message for the
 *    most recent failure on the calling thread.  No C++ exception crosses this boundary.
 *  - Outputs must not alias inputs.  C = 0 is a valid empty call that enqueues nothing.
 *  - Non-finite data cannot be checked on the host without a synchronization, so it is handled
 *    on the device, visibly: a channel with a NaN/Inf weight gets NaN scales and zero codes, and
 *    NaN propagates into its output errors; the allocator treats a NaN gain as "no gain".
 */
#ifndef MPQ_H
#define MPQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MPQ_OK = 0,
    MPQ_ERR_INVALID_ARG = 1,  /* a size, pointer or parameter is out of its documented range */
    MPQ_ERR_NONFINITE = 2,    /* a host-side numeric parameter is NaN/Inf */
    MPQ_ERR_UNSUPPORTED = 3,  /* valid for the method but beyond this library's limits below */
    MPQ_ERR_CUDA = 4,         /* a CUDA runtime call or kernel launch failed */
    MPQ_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up (mpq_device_status) */
    MPQ_ERR_NOMEM = 6,        /* mpq_output_error's stream-ordered scratch allocation failed */
    MPQ_ERR_BOUNDS = 7        /* the checked build skipped an out-of-range access (mpq_device_status) */
} mpq_status;

/* Library limits. */
#define MPQ_MIN_BITS 2        /* b = 2 gives Q = {-1, 0, 1}, the smallest set of Eq. 1 */
#define MPQ_MAX_BITS 8        /* codes are stored as int8 */
#define MPQ_MAX_POINTS 16     /* k_max */
#define MPQ_MAX_GRID 1024     /* G, candidate scales per greedy step */
#define MPQ_MAX_DIM 8192      /* d for mpq_quantize_layer: one channel's residual lives on chip */

/* Allocation modes of mpq_allocate_points. */
#define MPQ_ALLOC_BUDGET 0
#define MPQ_ALLOC_THRESHOLD 1

/* Centres of mpq_center_weights: one B per channel, or one B for the whole layer. */
#define MPQ_CENTER_PER_CHANNEL 0
#define MPQ_CENTER_PER_LAYER 1

/* Clipping-factor sets of mpq_clip_search: one K per channel, or one K for the whole layer. */
#define MPQ_CLIP_PER_CHANNEL 0
#define MPQ_CLIP_PER_LAYER 1
#define MPQ_MAX_CLIP_CANDIDATES 32

/*
 * mpq_quantize_layer -- greedy multipoint construction (Sec. 3.2, Eq. 6-9, Algorithm 1) for every
 * channel of one layer, run to k_max points.
 *
 * For each channel k and step i = 1..k_max, with residual r (r_1 = w_k, Eq. 7):
 *   m = max_j |r_j|; smax = m / Qmax (fp32 division);
 *   candidate scales s_g = f_g * smax (fp32), g = 1..G, where f_g = g/G (fp32 division) when
 *     grid_frac is NULL, else f_g = grid_frac[g-1];
 *   codes of candidate g: q_j = clamp(rint(r_j / s_g), -Qmax, Qmax) (Eq. 8; fp32 division,
 *     ties of rint to even);
 *   the chosen candidate minimises ||r - s_g q||^2 (Eq. 9), the lowest g on ties;
 *   r <- fmaf(-s*, q*, r) elementwise (Eq. 7).
 * A residual that is exactly zero yields a null point (scale 0, codes 0).
 *
 *   W          [C][d] fp32, the layer's weights, one output channel per row.
 *   C, d       channels and weights per channel; 1 <= d <= MPQ_MAX_DIM.
 *   bits       b in [MPQ_MIN_BITS, MPQ_MAX_BITS]; Qmax = 2^(b-1) - 1.
 *   G          candidate scales per step, 1..MPQ_MAX_GRID.
 *   grid_frac  HOST array of G fp32 fractions, strictly increasing, in (0, 1]; or NULL for the
 *              linear grid g/G.  Copied into the launch; the caller may free it on return.
 *   k_max      points per channel, 1..MPQ_MAX_POINTS.
 *   codes      out [k_max][C][d] int8: codes[i][k][:] = q_{k,i+1}.
 *   scales     out [C][k_max] fp32: scales[k][i] = s_{k,i+1}.
 *   resid_sq   out [C][k_max+1] fp32, nullable: ||r_{k,n+1}||^2 for n = 0..k_max points
 *              (n = 0 is ||w_k||^2).
 *   residuals  out [k_max][C][d] fp32, nullable: residuals[i][k][:] = r_{k,i+2}.
 *   rmax       out [C][k_max+1] fp32, nullable: max_j |r_{k,n+1,j}| for n = 0..k_max points
 *              (n = 0 is max_j |w_kj|; NaN for a channel with a non-finite weight) -- the
 *              operand ranges mpq_output_error can take instead of measuring them.
 */
mpq_status mpq_quantize_layer(const float *W, int C, int d, int bits, int G,
                              const float *grid_frac, int k_max, int8_t *codes, float *scales,
                              float *resid_sq, float *residuals, float *rmax, void *stream);

/*
 * mpq_output_error -- output error of every channel for every point count (Sec. 3.3, Eq. 11):
 *   err[k][n] = (1/N) sum_{t=1..N} (x_t . (w_k - w~_k(n)))^2,  n = 0..k_max,
 * where w_k - w~_k(n) is the residual r_{k,n+1} regenerated from W, codes and scales by the
 * recursion of Eq. 7 (r_{k,1} = w_k, r_{k,i+1} = fmaf(-s_{k,i}, q_{k,i}, r_{k,i})).
 *
 *   X       calibration inputs D_L.  groups == 1: [N][d], shared by all channels.
 *           groups == C: [C][N][d], channel k uses its own block (depthwise convolution, where
 *           each output channel sees only its own input patches).
 *   N       calibration rows, >= 1.
 *   groups  1 or C.
 *   W, codes, scales, C, d, k_max   as produced by / passed to mpq_quantize_layer.
 *   rmax    [C][k_max+1] fp32 or NULL: the rmax output of the mpq_quantize_layer call that made
 *           codes and scales (max |r| of every residual vector).  Given, the tensor-core path's
 *           range pass reads X alone instead of X, W and every code plane; NULL, it measures the
 *           ranges itself.  The results are the same either way.
 *   err     out [C][k_max+1] fp32.
 *
 * Scratch: with groups == 1, d a multiple of 16 and X, W, codes 16-byte aligned (the tensor-core
 * path with scaled fp16 operands), the call takes 4 (1 + C (k_max+1)) bytes (4 bytes with rmax),
 * rounded up to 256, plus 4 N d bytes for X's fp16 hi/lo planes
 * from the current device's default stream-ordered memory pool with cudaMallocAsync on `stream`
 * and returns them with cudaFreeAsync on `stream` -- concurrent calls on other streams each get
 * their own, and a CUDA graph capture records them as the graph's allocation nodes.
 * MPQ_ERR_NOMEM if that allocation fails (nothing else is enqueued then).  The first such call in
 * a process made outside a stream capture raises that pool's release threshold
 * (cudaMemPoolAttrReleaseThreshold) to keep freed blocks cached in the pool instead of returning
 * them to the driver at every synchronization; a process that manages the default pool itself
 * can call mpq_output_error_noalloc instead.
 */
mpq_status mpq_output_error(const float *X, int N, int groups, const float *W,
                            const int8_t *codes, const float *scales, const float *rmax, int C,
                            int d, int k_max, float *err, void *stream);

/* Most code-level thresholds (d * Qmax) one step of mpq_quantize_layer_adaptive sorts. */
#define MPQ_ADAPTIVE_MAX_THRESHOLDS 65536

/*
 * mpq_quantize_layer_adaptive -- Algorithm 1 with the adaptive grid of Eq. 10 (Sec. 3.2,
 * Definition 1) instead of a fixed grid.  Step i of channel k, with r = r_{k,i} (r_1 = w_k):
 *   Delta = the minimal gap of r (Definition 1): half the smallest difference between two distinct
 *     element magnitudes |r_j| (the printed pair condition t_i != t_j read as |t_i| != |t_j|);
 *   gamma = min(Delta / Qmax, eta), or eta when r has fewer than two distinct magnitudes;
 *   grid search of a over I = [0, 2 Qmax ||r||] with step gamma (Eq. 10): a_m = m gamma for
 *     m = 1..M, M = floor(2 Qmax ||r|| / gamma) (double, ||r||^2 summed in index order), as fp32
 *     point scales s_m = fl(a_m / Qmax);
 *   codes as mpq_quantize_layer; the chosen m minimises ||r - s_m q||^2 (the first m on ties);
 *   r <- fmaf(-s, q, r).
 * A zero residual gives a null point (scale 0, codes 0); so does a grid without candidates.
 * The grid is not enumerated: the thresholds where each element's code changes are sorted and the
 * objective, a quadratic in s between them, is minimised exactly; the work per step is
 * O(d Qmax log(d Qmax)) whatever M is (Definition 1 makes M 1e8..1e10 on real channels).
 *
 *   W          [C][d] fp32; 1 <= d <= MPQ_MAX_DIM and d * Qmax <= MPQ_ADAPTIVE_MAX_THRESHOLDS.
 *   bits, k_max, codes, scales, resid_sq   as for mpq_quantize_layer (resid_sq nullable).
 *   eta        the largest grid step (the paper's experiments: 2^-10); finite, > 0.
 *   max_cand   the largest grid a step may have (>= 1).  A step whose grid is larger is refused on
 *              the device: its scale and every later scale of that channel read NaN, their codes
 *              0, and ncand holds -1 for it (0 for the later steps).
 *   ncand      out [C][k_max] int64, nullable: M of every step (0 for a null point).
 * Scratch: the threshold lists, 16 d Qmax bytes per resident CTA (at most 2 per SM), come from the
 * current device's stream-ordered pool on `stream` (as for mpq_output_error; MPQ_ERR_NOMEM if it
 * has no room).
 */
mpq_status mpq_quantize_layer_adaptive(const float *W, int C, int d, int bits, int k_max,
                                       double eta, long long max_cand, int8_t *codes,
                                       float *scales, float *resid_sq, long long *ncand,
                                       void *stream);

/* Words of mpq_output_error_noalloc's fixed scratch buffer (4 MiB). */
#define MPQ_NOALLOC_RANGE_WORDS (1 << 20)

/*
 * mpq_output_error_noalloc -- mpq_output_error that allocates nothing.  The paper has no
 * counterpart: it is an engineering variant of the Eq. 11 call for callers that cannot allocate
 * device memory while they run -- a process whose memory is budgeted up front by its owner, a
 * framework whose allocator owns the stream-ordered pool, or a pool that is switched off.
 *
 * Same arguments (without rmax: the ranges are always measured), layouts, validation, results
 * (bit for bit) and errors as mpq_output_error, except for the scratch: the tensor-core path's range table (1 + C (k_max+1) words) lives in one
 * fixed device array of MPQ_NOALLOC_RANGE_WORDS words (4 MiB) inside the library, which every
 * device that loads the library's module keeps until the process exits.  The call zeroes the
 * part of the table it uses before filling it.  Therefore:
 *  - a call whose table would exceed MPQ_NOALLOC_RANGE_WORDS words is rejected with
 *    MPQ_ERR_UNSUPPORTED before anything is enqueued;
 *  - the first call on a device (made with that device current) looks up the array's device
 *    address (cudaGetSymbolAddress) and keeps it; under CUDA's default lazy module loading that
 *    lookup is also what loads the module, and so the array, on that device.  Make this first
 *    call before any stream capture begins;
 *  - overlapping calls race: every call of this entry point uses the same array, so two calls
 *    whose kernels can run at the same time (on different streams or from different threads)
 *    overwrite each other's ranges and return wrong errors.  Order them (one stream, or events
 *    between streams).  mpq_output_error has no such limit.
 */
mpq_status mpq_output_error_noalloc(const float *X, int N, int groups, const float *W,
                                    const int8_t *codes, const float *scales, int C, int d,
                                    int k_max, float *err, void *stream);

/*
 * mpq_allocate_points -- per-channel point counts from the output-error table (Sec. 3.3,
 * Algorithm 2).
 *
 * mode MPQ_ALLOC_THRESHOLD (Algorithm 2 as printed): npoints[k] = the smallest n in 1..k_max with
 *   err[k][n] < eps (compared in double), else k_max.  budget_or_eps = eps (not NaN).
 * mode MPQ_ALLOC_BUDGET: a total of P = floor(beta*C + 0.5) points (beta = budget_or_eps, finite,
 *   >= 0).  Every channel starts with one point; the P - C extra points (clamped to
 *   [0, C*(k_max-1)]) go one at a time to the channel whose next point lowers its output error
 *   most: gain_k = err[k][n_k] - err[k][n_k+1] (fp32 subtraction; NaN counts as no gain), lowest k
 *   on ties, stopping early when the best remaining gain is <= 0.  Computed in one device-wide
 *   selection that gives exactly the result of that sequential loop.
 *
 *   err          [C][k_max+1] fp32 (from mpq_output_error).
 *   npoints      out [C] int32.
 *   points_used  out, nullable: one device int32, the total sum_k npoints[k].
 */
mpq_status mpq_allocate_points(const float *err, int C, int k_max, int mode, double budget_or_eps,
                               int *npoints, int *points_used, void *stream);

/* Most layers one mpq_allocate_points_batched call takes. */
#define MPQ_MAX_BATCH 64

/*
 * mpq_allocate_points_batched -- mpq_allocate_points for n layers in one launch, one CTA per layer
 * (a network's small layers each leave most of the GPU idle on their own).  Every layer gets
 * exactly what mpq_allocate_points gives it for the same arguments (each layer has its own budget
 * or threshold; Algorithm 2 per layer).
 *
 *   n              number of layers, 0..MPQ_MAX_BATCH.
 *   err            HOST array of n device pointers: layer l's [C[l]][k_max+1] fp32 error table.
 *   C              HOST array of n channel counts (0 is an empty layer).
 *   k_max, mode    shared by every layer (mode as for mpq_allocate_points).
 *   budget_or_eps  HOST array of n values: each layer's beta (budget mode) or eps (threshold).
 *   npoints        HOST array of n device pointers: out [C[l]] int32.
 *   points_used    HOST array of n device pointers (each nullable), or NULL.
 * Arguments are validated for every layer before anything is enqueued.
 */
mpq_status mpq_allocate_points_batched(int n, const float *const *err, const int *C, int k_max,
                                       int mode, const double *budget_or_eps,
                                       int *const *npoints, int *const *points_used,
                                       void *stream);

/*
 * mpq_reconstruct -- multipoint weights (Eq. 4): W_hat[k][j] = B_k + sum_{i=1..n_k} s_{k,i} q_{k,i,j},
 * accumulated as acc = fmaf(s_{k,i}, q_{k,i,j}, acc) from acc = B_k (the centre of an asymmetric
 * set, from mpq_center_weights; 0 when center is NULL) in the order i = 1, 2, ...
 * n_k = npoints[k] clamped to [0, k_max] (npoints lives on the device and is not checked on the
 * host).
 *
 *   codes [k_max][C][d] int8, scales [C][k_max] fp32, npoints [C] int32.
 *   center [C] fp32 or NULL.
 *   W_hat out [C][d] fp32.
 */
mpq_status mpq_reconstruct(const int8_t *codes, const float *scales, const int *npoints,
                           const float *center, int C, int d, int k_max, float *W_hat,
                           void *stream);

/*
 * mpq_center_weights -- asymmetric quantization sets (Eq. 1 with B != 0; per-channel and per-layer
 * settings of Sec. 3.1 and App. B).  The set K x [-1 : eps_b : 1] + B has the centre
 *   B = (max w + min w) / 2, rounded once to fp32,
 * over the channel's weights (MPQ_CENTER_PER_CHANNEL) or over the whole layer
 * (MPQ_CENTER_PER_LAYER, one B for every channel), so that K = (max w - min w) / 2 covers every
 * weight.  The multipoint approximation takes B once and approximates the centred weights with
 * the greedy points: Wc = fl(w - B) (one fp32 subtraction) is the W to give mpq_quantize_layer,
 * mpq_output_error and mpq_clip_search, and center is the B to give mpq_reconstruct and
 * mpq_pack_points, so that w~ = B + sum_i s_i q_i.  A non-finite weight makes B NaN for its
 * channel (per layer: for every channel), and so that channel's Wc.
 *
 *   W, C, d   [C][d] fp32 weights; d >= 1.
 *   mode      MPQ_CENTER_PER_CHANNEL or MPQ_CENTER_PER_LAYER.
 *   center    out [C] fp32.
 *   Wc        out [C][d] fp32 (per layer, its first C values also serve as working storage).
 */
mpq_status mpq_center_weights(const float *W, int C, int d, int mode, float *center, float *Wc,
                              void *stream);

/*
 * mpq_clip_search -- output-error-driven clipping factor (Sec. 3.3, Eq. 12; candidate grid of
 * App. B): the clipping factor K of the quantization set K x [-1 : eps_b : 1] (Eq. 1, B = 0) that
 * minimises the output error of the quantized weights, chosen among n_cand candidates
 *   K_c = f_c * m,  f_c = (c+1)/n_cand (fp32 division), c = 0..n_cand-1
 * (n_cand = 20 is the experiments' grid [0.05 : 0.05 : 1] x max|w|), with m = max_j |w_kj| of
 * channel k (MPQ_CLIP_PER_CHANNEL) or of the whole layer (MPQ_CLIP_PER_LAYER, one K for every
 * channel).  The quantized channel is s q with s = K / Qmax (fp32 division) and
 * q_j = clamp(rint(w_j / s), -Qmax, Qmax) as in Eq. 8; its output error is
 *   err[k][c] = (1/N) sum_t (x_t . r_{k,c})^2,  r_{k,c} = fmaf(-s, q, w_k)   (Eq. 11's form).
 * best[k] = the lowest c with the smallest err[k][c] (per channel), or the lowest c with the
 * smallest sum_k err[k][c] summed in double over the channels in order (per layer, the same c for
 * every channel).  A non-finite weight makes that channel's K (per layer: every K) NaN, its errors
 * NaN, and NaN never wins; best is -1 where no candidate is finite.
 *
 *   X, N, groups  calibration inputs as for mpq_output_error.
 *   W, C, d       [C][d] fp32 weights; 1 <= d <= MPQ_MAX_DIM.
 *   bits          b in [MPQ_MIN_BITS, MPQ_MAX_BITS].
 *   n_cand        1..MPQ_MAX_CLIP_CANDIDATES.
 *   mode          MPQ_CLIP_PER_CHANNEL or MPQ_CLIP_PER_LAYER.
 *   clip          out [C][n_cand] fp32: K_c of each channel (also used as working storage).
 *   err           out [C][n_cand] fp32.
 *   best          out [C] int32; the chosen factor of channel k is clip[k][best[k]].
 * Scratch: with groups == 1, d a multiple of 16 and X, W 16-byte aligned (the tensor-core path),
 * 4 C + 4 N d bytes (channel maxima, X's fp16 hi/lo planes) and the fp16 hi/lo planes of the
 * candidates' residuals, 4 d n_cand bytes per channel for at most max(1, 2^32 / (4 d n_cand))
 * channels at a time (larger layers run in chunks of whole channels), come from the current
 * device's stream-ordered pool on `stream` in one allocation (as for mpq_output_error;
 * MPQ_ERR_NOMEM if it has no room, and nothing else is enqueued then).
 */
mpq_status mpq_clip_search(const float *X, int N, int groups, const float *W, int C, int d,
                           int bits, int n_cand, int mode, float *clip, float *err, int *best,
                           void *stream);

/*
 * Integer inference with multipoint weights (Sec. 3.4, Eq. 13).  For integer inputs x_t (int8),
 * channel k with n_k points (s_{k,i}, q_{k,i}) computes
 *   Y[k][t] = sat32( floor( sum_{i<n_k} A_{k,i} (q_{k,i} . x_t) / 2^p ) ),  A_{k,i} = rint(2^p s_{k,i})
 * (ties to even): integer dot products (step 1), multiplication by the 32-bit coefficients and
 * summation (step 2), and the shift by p bits (step 3; an arithmetic right shift, i.e. floor), with
 * exact 64-bit products and sums and saturation to the int32 range.  n_k = npoints[k] clamped to
 * [0, k_max]; a channel with no point outputs 0 (with a centre, its A_B term alone).  The q are the
 * integer codes of mpq_quantize_layer, so the coefficient of q is s = a / Qmax.  With asymmetric
 * sets (a centre B_k per channel, from mpq_center_weights), w~ = B_k 1 + sum_i s_i q_i and the sum
 * before the shift also holds A_{B,k} (sum_j x_tj), A_{B,k} = rint(2^p B_k).
 *
 * Deployment is split as in the paper: the coefficients and a packed copy of the used points are
 * made once, offline (mpq_pack_layout on the host, then mpq_pack_points), and
 * mpq_multipoint_linear runs per input batch.
 */
typedef struct {
    int C, d, k_max, bits, p;
    int centered;        /* 1: the layer has centres B_k (asymmetric sets) */
    int d_pad;           /* d rounded up to a multiple of 64 */
    int rows;            /* packed code rows, a multiple of 128 */
    int tiles;           /* rows / 128 */
    size_t off_coef, off_chan, off_point, off_tile, off_center, off_codes;   /* byte offsets */
    size_t bytes;        /* size of the device buffer to allocate */
} mpq_packed_layout;

/*
 * mpq_pack_layout -- HOST only: the layout of a packed layer for the given point counts.
 *   npoints  HOST [C] int32 (e.g. copied back from mpq_allocate_points).
 *   bits     the codes' width (their magnitude is at most 2^(bits-1) - 1).
 *   p        coefficient precision, 0..30.
 *   centered 1 if the layer has centres (mpq_pack_points then takes them), else 0.
 *   layout   out.
 */
mpq_status mpq_pack_layout(const int *npoints, int C, int d, int k_max, int bits, int p,
                           int centered, mpq_packed_layout *layout);

/*
 * mpq_pack_points -- fill a packed layer: coefficients A = rint(2^p s) of the used points and their
 * codes (as bf16, exact), and A_B = rint(2^p B) of the centres.  Synchronous: returns after the
 * device has finished with the host arrays.
 *   codes [k_max][C][d] int8 and scales [C][k_max] fp32 on the device (from mpq_quantize_layer);
 *   center  [C] fp32 on the device (from mpq_center_weights) if layout->centered, else NULL;
 *   npoints HOST [C], the same as given to mpq_pack_layout;
 *   packed  device buffer of layout->bytes bytes, written here.
 * MPQ_ERR_UNSUPPORTED if a coefficient (or a centre's) does not fit 32 bits, NaN included.
 */
mpq_status mpq_pack_points(const int8_t *codes, const float *scales, const float *center,
                           const int *npoints, const mpq_packed_layout *layout, void *packed,
                           void *stream);

/*
 * mpq_multipoint_linear -- Y [C][T] int32 (channel-major: one channel's T outputs are contiguous)
 * for X [T][d] int8 inputs (row-major), from a packed layer.  T >= 1.
 */
mpq_status mpq_multipoint_linear(const int8_t *X, int T, const mpq_packed_layout *layout,
                                 const void *packed, int32_t *Y, void *stream);

/*
 * Bounded device-side waits.  The tensor-core kernels (mpq_output_error and its _noalloc variant,
 * mpq_clip_search, mpq_multipoint_linear) hand work between their warps through shared-memory
 * barriers, and every wait on one is bounded by a clock budget.  A kernel whose wait gives up
 * stops issuing work, waits for the copies and MMAs it has already issued to finish, releases its
 * tensor memory and returns, with NaN in its output errors (its inference outputs unspecified);
 * it records which kernel it was in a word kept per device.  A NaN error can therefore mean a
 * non-finite input or a timeout: mpq_device_status tells them apart.
 */
#define MPQ_TIMEOUT_OUTPUT_ERROR 0x1u   /* mpq_output_error / mpq_output_error_noalloc */
#define MPQ_TIMEOUT_CLIP 0x2u           /* mpq_clip_search */
#define MPQ_TIMEOUT_INFERENCE 0x4u      /* mpq_multipoint_linear */
#define MPQ_TIMEOUT_DRAIN 0x100u        /* a wait for the kernel's own copies or MMAs also gave up */

/*
 * The checked build.  Compiled with -DMPQ_CHECK_BOUNDS (paper_2002_09049_gb300._build:
 * build(checked=True) -> libmpq_checked.so), every kernel checks the indices it computes before
 * it uses them: each global store against the extent its arguments give the output, the
 * data-dependent shared-memory indices (lattice buckets, event bins, queue slots, sort keys)
 * against their arrays, the carve-up of dynamic shared memory against the launch's share, and
 * every tile copy's coordinates against the rule that its first element be 16-byte aligned.  A
 * failed check is counted and the access skipped -- the kernel never traps -- so a bad index
 * shows as MPQ_FAULT_BOUNDS from mpq_device_status (with the first failing source line in
 * mpq_last_error) and as wrong or NaN outputs, never as a fault.  A skipped tile copy leaves its
 * barrier unsatisfied, so that kernel's bounded wait gives up too (MPQ_TIMEOUT_*).  The checks
 * cost time: the checked build is for tests, the normal build's kernels carry none.
 */
#define MPQ_FAULT_BOUNDS 0x10000u        /* mpq_device_status: the checked build skipped accesses */
#define MPQ_BUILD_CHECK_BOUNDS 0x1u      /* mpq_build_options: this is the checked build */

/*
 * mpq_device_status -- synchronizes `stream`, then takes the current device's timeout word
 * (reads and clears it in one atomic exchange on the device), and in the checked build every
 * kernel unit's count of skipped accesses likewise: MPQ_OK if no bounded wait gave up and no
 * check failed since the last call; else MPQ_ERR_TIMEOUT if a wait gave up (it takes precedence),
 * else MPQ_ERR_BOUNDS.  *flags (nullable; 0 on MPQ_OK) receives the MPQ_TIMEOUT_* bits, plus
 * MPQ_FAULT_BOUNDS if a check failed.  It covers the kernels that have finished when the exchange
 * runs: synchronize the other streams first to include their calls.  Synchronous.
 */
mpq_status mpq_device_status(void *stream, unsigned *flags);

/*
 * mpq_set_wait_limit -- the clock budget of every bounded wait of the kernels launched after
 * this call (process-wide), in SM clocks; clocks <= 0 restores the default of 2^31 (about one
 * second at the maximum SM clock).  A budget far below a kernel's normal waits makes healthy
 * launches give up: it is meant for tests.
 */
mpq_status mpq_set_wait_limit(long long clocks);

/*
 * mpq_test_withhold_copies -- TEST HOOK, process-wide: while on (1), the tile-copy thread of the
 * output-error contraction (mpq_output_error's tensor-core path) issues no copies, so that every
 * wait of that kernel runs out with nothing in flight and the call reports MPQ_TIMEOUT_OUTPUT_ERROR
 * through mpq_device_status.  Off (0) by default; never on outside tests of the timeout path.
 */
mpq_status mpq_test_withhold_copies(int on);

/* MPQ_BUILD_* bits of the options this library was compiled with (0 for the normal build). */
unsigned mpq_build_options(void);

/* Name of a status code (static string). */
const char *mpq_status_string(mpq_status s);

/* Message describing the most recent failure on the calling thread ("" if none). */
const char *mpq_last_error(void);

/* Library version, major*10000 + minor*100 + patch. */
int mpq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MPQ_H */
