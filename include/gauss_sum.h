/*
 * gauss_sum.h -- C ABI of the GB300 (sm_103a) Gauss kernel sum library.
 *
 * The library evaluates the Gauss kernel sum of arXiv 2609.04910, Sec. 1,
 * Eq. 1:
 *
 *     s_m = sum_{n=1..N} exp(-tau/2 * ||q_m - k_n||^2) * v_n  in R^C,
 *                                                      m = 1..M,
 *
 * for query points q (M x D), key points k (N x D), signed values v (N x C)
 * and bandwidth tau > 0, and the gradient of s_m with respect to q_m for
 * scalar weights (Sec. 3, MMD flows and SVGD):
 *
 *     grad_m = tau * ( sum_n Phi(q_m,k_n) v_n k_n  -  q_m sum_n Phi(q_m,k_n) v_n ),
 *
 * which the library evaluates as one Gauss sum with the augmented values
 * (v_n k_n, v_n) in R^{D+1}, and the vector-Jacobian product of Eq. 1
 * (gauss_sum_vjp: the gradients of sum_m g_m . s_m in q, k and v).
 *
 * Conventions shared by every entry point:
 *  - Array arguments are DEVICE pointers to contiguous row-major arrays,
 *    owned by the caller and not retained after the call returns.  q, k and
 *    v share one element type (gs_dtype); q may alias k (the MMD form q = k
 *    of Sec. 3).  Outputs are float32 and are overwritten, not accumulated.
 *  - Base pointers must be 16-byte aligned.
 *  - `stream` is a cudaStream_t passed as void* (NULL: the legacy default
 *    stream).  Calls are asynchronous and stream ordered; the status return
 *    covers argument checks, allocation and launch errors.  A device-side
 *    wait that runs out of time is reported by gauss_sum_device_status().
 *  - Without a caller workspace the library allocates its workspace on
 *    `stream` (cudaMallocFromPoolAsync) and frees it on the same stream
 *    (cudaFreeAsync), from a stream-ordered memory pool of its own per
 *    device that keeps up to 1 GiB of freed workspace mapped between calls.
 *  - M = 0 is a no-op; N = 0 writes zeros.
 *  - fp16/bf16 inputs run on the tensor-core kernels (tcgen05, sm_103a) and
 *    need D <= 256 and C <= 256 (gradients: D <= 256, any C).  fp32 inputs
 *    run on the fp32 SIMT kernel (D <= 128 forward, D <= 64 gradients, any
 *    C) or, for forward sums with C <= 4 and D <= 32, on the tensor cores
 *    with three tf32 MMAs per product (q^ k^T ~ hi.hi + hi.lo + lo.hi of the
 *    tf32 splits x = hi + lo, fp32-level accuracy): chosen automatically
 *    from 2^25 pairs (per call, summed over a batch), or forced with
 *    GS_PATH_TENSOR / GS_PATH_SIMT.
 *  - On a non-OK return gauss_sum_last_error() describes the failure.
 */
#ifndef GAUSS_SUM_H
#define GAUSS_SUM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element type of q, k and v. */
typedef enum { GS_FP32 = 0, GS_FP16 = 1, GS_BF16 = 2 } gs_dtype;

typedef enum {
    GS_OK = 0,
    GS_ERR_INVALID_ARGUMENT = 1, /* null pointer, negative size, bad tau, misalignment */
    GS_ERR_UNSUPPORTED = 2,      /* shape or dtype outside the supported range, or no sm_103 GPU */
    GS_ERR_OUT_OF_MEMORY = 3,    /* workspace allocation failed / caller workspace too small */
    GS_ERR_CUDA = 4,             /* a CUDA runtime call or a kernel launch failed */
    GS_ERR_DEVICE_TIMEOUT = 5    /* a bounded device-side wait ran out (see device_status) */
} gs_status;

/* Which kernel family evaluates the sum. */
typedef enum { GS_PATH_AUTO = 0, GS_PATH_TENSOR = 1, GS_PATH_SIMT = 2 } gs_path;

/*
 * Options of the _ex entry points.  Initialise with gauss_sum_default_options.
 *  center          1: shift q and k by their common mean before rounding to
 *                     the MMA type (the overflow/cancellation safeguard of
 *                     Remark 2, Sec. 2); 0: use the raw points.
 *  split_n         number of key splits per row tile (0: chosen from the
 *                  SM count; on the FMA-pipe kernel (C <= 2, or C <= 4
 *                  below 2^28 pairs or with rows too wide for the augmented
 *                  layout) one persistent block per SM takes an equal run
 *                  of (row tile, key tile) pairs); partial sums
 *                  over splits are added in a fixed order, so results are
 *                  deterministic for a fixed split and GPU.
 *  workspace       caller-owned device buffer of workspace_bytes bytes
 *                  (256-byte aligned) used instead of an allocation; its
 *                  required size is gauss_sum_workspace_size().
 *  path            GS_PATH_AUTO picks the tensor-core kernels for fp16/bf16
 *                  and, for fp32, the 3xTF32 tensor-core variant for large
 *                  forward sums with C <= 4 and D <= 32, else the SIMT
 *                  kernel; GS_PATH_TENSOR takes fp32 only within that
 *                  range (GS_ERR_UNSUPPORTED otherwise); GS_PATH_SIMT
 *                  rejects fp16/bf16.
 *  main_events     measurement hook: two cudaEvent_t handles (or NULL) that
 *                  the call records on `stream` immediately before and after
 *                  the launch of its main kernel (the fused tensor-core
 *                  kernel, or the fp32 SIMT kernel), so a caller can time
 *                  that kernel alone.  The caller owns the events.
 *  exp2_fma        0 (default): every kernel value 2^x is computed by the
 *                  MUFU ex2 unit.  1..4: a fixed share of them (1/32, 1/16,
 *                  1/8, 1/4) is computed on the FMA pipe instead (Cody-Waite
 *                  range reduction and a degree-4 minimax polynomial for
 *                  2^f, relative error < 3e-6), the exponential-throughput
 *                  variant for SFU-bound shapes.  Only forward fp16/bf16
 *                  sums with C = 1 and D + 4 (fp16) or D + 6 (bf16) <= 128
 *                  take it (GS_ERR_UNSUPPORTED otherwise).
 */
typedef struct gs_options {
    int center;
    int split_n;
    void* workspace;
    size_t workspace_bytes;
    int path;
    void* main_events[2];
    int exp2_fma;
} gs_options;

/* Fill *opt with the defaults (center = 1, split_n = 0, no workspace, auto
 * path, no events, exp2_fma = 0). */
void gauss_sum_default_options(gs_options* opt);

/*
 * Eq. 1.  q: M x D, k: N x D, v: N x C (all `dtype`); out: M x C float32.
 */
gs_status gauss_sum(const void* q, const void* k, const void* v, double tau, int64_t M,
                    int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out, void* stream);

/* Eq. 1 with options (opt may be NULL for the defaults). */
gs_status gauss_sum_ex(const void* q, const void* k, const void* v, double tau, int64_t M,
                       int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out,
                       void* stream, const gs_options* opt);

/*
 * q-gradient of Sec. 3 for scalar weights: v is N x 1.
 * grad: M x D float32, grad[m] = d/dq_m sum_n Phi(q_m, k_n) v_n.
 * s_out: M x 1 float32 forward sum s_m, or NULL.
 */
gs_status gauss_sum_grad_q(const void* q, const void* k, const void* v, double tau, int64_t M,
                           int64_t N, int64_t D, gs_dtype dtype, float* grad, float* s_out,
                           void* stream);

gs_status gauss_sum_grad_q_ex(const void* q, const void* k, const void* v, double tau,
                              int64_t M, int64_t N, int64_t D, gs_dtype dtype, float* grad,
                              float* s_out, void* stream, const gs_options* opt);

/*
 * Vector-Jacobian product of Eq. 1 (reverse-mode derivative, as used by the
 * gradient flows of Sec. 3): for an upstream gradient g (M x C, float32) of
 * L = sum_m g_m . s_m,
 *
 *     grad_q[m] = tau sum_n Phi(q_m, k_n) (g_m . v_n) (k_n - q_m)   M x D
 *     grad_k[n] = tau sum_m Phi(q_m, k_n) (g_m . v_n) (q_m - k_n)   N x D
 *     grad_v[n] =     sum_m Phi(q_m, k_n) g_m                       N x C
 *
 * (all float32).  q, k, v as for gauss_sum (dtype); any of grad_q, grad_k,
 * grad_v may be NULL to skip it.  k^ and q^ below are shifted by the common
 * mean.  Evaluation:
 *  - fp16/bf16 with 2 <= C <= 8 and D + 1 <= 128 (weighted single pass):
 *    with the pair weights w_mn = g_m . v_n multiplied into the kernel
 *    values in float32 (before the rounding to fp16), grad_q is one Gauss
 *    sum over the keys with the D + 1 values (k^_n, 1), grad_k one over the
 *    queries with (q^_m, 1), and grad_v the forward sum over the queries
 *    with the values g (three passes in all, each exponential computed once
 *    per pass).
 *  - otherwise: grad_q is a Gauss sum over the keys with the C (D + 1)
 *    values (v_nc k^_n, v_nc) contracted with g_m; grad_k and grad_v are one
 *    Gauss sum over the queries with the values (g_mc q^_m, g_mc)
 *    contracted with v_n (its unweighted channels are grad_v).  On the
 *    tensor-core path the channels are evaluated in launches of at most 256
 *    channels (ceil(C (D + 1) / 256) launches per sum, each recomputing the
 *    kernel values), with the values rounded to fp16 after a per-channel
 *    power-of-two scale; the fp32 path makes C launches per sum.
 * g must be 16-byte aligned.  Default options; the workspace is allocated
 * on `stream`.
 */
gs_status gauss_sum_vjp(const void* q, const void* k, const void* v, const float* g, double tau,
                        int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype,
                        float* grad_q, float* grad_k, float* grad_v, void* stream);

/*
 * Workspace bytes that gauss_sum_ex (grad = 0, C channels) or
 * gauss_sum_grad_q_ex (grad = 1, C ignored) needs for these sizes and
 * options (opt may be NULL).  Returns 0 for a no-op call and (size_t)-1 for
 * arguments the call would reject.
 */
size_t gauss_sum_workspace_size(int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype,
                                int grad, const gs_options* opt);

/*
 * A batch of B independent problems of Eq. 1 with equal sizes (the paper
 * benchmarks batches of independent point clouds, Sec. 4), stored
 * contiguously: q is B x M x D, k is B x N x D, v is B x N x C and out is
 * B x M x C (float32).  Problem b uses only its own points; centring (the
 * shift of Remark 2) is per problem.  Default options.  For C <= 4 (fp16 /
 * bf16) the whole batch runs in one launch of each kernel; otherwise the
 * problems run one after another on `stream`, and every problem's q, k, v
 * and out must then start 16-byte aligned (GS_ERR_INVALID_ARGUMENT
 * otherwise).  B = 0 is a no-op.
 */
gs_status gauss_sum_batched(const void* q, const void* k, const void* v, double tau, int64_t B,
                            int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out,
                            void* stream);

/*
 * Squared maximum mean discrepancy of Sec. 3 for B problems: for points
 * x (B x N x D) carrying the signed weights v (B x N) of the difference of
 * two discrete measures,
 *     mmd2[b] = sum_{m,n} v[b,m] Phi(x[b,m], x[b,n]) v[b,n] = v_b^T s_b,
 * with s_b the Gauss sum of Eq. 1 for q = k = x_b and C = 1.  Since the
 * kernel matrix is symmetric, fp16 / bf16 points with D + 4 (fp16) or
 * D + 6 (bf16) <= 128 are evaluated over the upper triangle of 128 x 128
 * tile pairs only, off-diagonal tiles counted twice (half the
 * exponentials); other inputs use the full sum.  mmd2 is a device array of
 * B floats (16-byte aligned); the final sum over m runs in float64 in a
 * fixed order.  Allocates B x N floats and a few float64 partial sums on
 * `stream` (cudaMallocAsync) besides the Gauss sum's workspace.
 */
gs_status gauss_sum_mmd2(const void* x, const void* v, double tau, int64_t B, int64_t N,
                         int64_t D, gs_dtype dtype, float* mmd2, void* stream);

/*
 * Synchronise `stream`, then return and clear the device status word of the
 * current device: GS_OK, or GS_ERR_DEVICE_TIMEOUT if a kernel gave up a
 * bounded wait since the last call (its outputs are then invalid;
 * gauss_sum_last_error() names the block, warp and barrier of the first
 * wait that gave up), or GS_ERR_CUDA if the synchronisation itself failed.
 */
gs_status gauss_sum_device_status(void* stream);

/* Description of the last non-OK status returned on this host thread. */
const char* gauss_sum_last_error(void);

/* Static name of a status code. */
const char* gauss_sum_status_string(gs_status status);

/* Size of the static scratch array used by gauss_sum_noalloc: 32 MiB. */
#define GS_NOALLOC_SCRATCH_BYTES (32u * 1024u * 1024u)

/*
 * Eq. 1 like gauss_sum (default options), but without allocating device
 * memory.  The paper has no counterpart: this is for callers that cannot
 * allocate at the point of the call, e.g. code inside a framework that owns
 * every device allocation through its own pool, or code that has reserved
 * all free device memory up front.  The scratch memory is a static device
 * array of GS_NOALLOC_SCRATCH_BYTES bytes inside the library, held by every
 * GPU that loads the library until the process exits.
 *  - Arguments, layouts and ownership are those of gauss_sum.
 *  - Calls that need more scratch than the array holds return
 *    GS_ERR_UNSUPPORTED (see gauss_sum_last_error) without any GPU work;
 *    the M = N = 65536, D = 64, C = 1 fp16 MMD workload fits (it needs
 *    21 MiB).  The scratch a call needs is that of the kernel gauss_sum
 *    would run: calls of 2^28 or more pairs with three or four channels
 *    on rows of D + 4 <= 128 (fp16; D + 6 for bf16) take the two-MMA
 *    kernel, whose transposed values and per-split partial sums need more
 *    than the FMA-pipe kernel that smaller calls use
 *    (gauss_sum_workspace_size gives the figure).
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress with that device current) and keeps it for the
 *    life of the process; make that first call before any stream capture.
 *    The kept address assumes the device's primary context is never reset:
 *    after cudaDeviceReset on that device the library's cached addresses
 *    (this array and the device status word) are stale, and calls on that
 *    device fail or misbehave.
 *  - All calls on a device share the array and leave their data in it:
 *    calls whose GPU work can overlap (unordered streams, several host
 *    threads) race and must be ordered by the caller.
 *  - No cudaMalloc, cudaMallocAsync, cudaFree or allocating library call is
 *    made; each call clears the few scratch words it accumulates into
 *    (cudaMemsetAsync) before using them.
 */
gs_status gauss_sum_noalloc(const void* q, const void* k, const void* v, double tau, int64_t M,
                            int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out,
                            void* stream);

/*
 * Measurement helper (not part of Eq. 1): sustained MUFU exp2 throughput of
 * the current device in exponentials per second, measured with CUDA events
 * by a kernel of independent ex2.approx chains on every SM.  Synchronises
 * `stream`.  Used as the SFU roofline of the fused kernel.
 */
gs_status gauss_sum_probe_ex2_rate(void* stream, double* exp2_per_second);

/*
 * Measurement helper (not part of Eq. 1): the exp2 rate that the instruction
 * mix of the fused FMA kernel's exponent loop can reach, in exponentials
 * per second: per key pair and two query rows two paired multiplies by c,
 * four ex2.approx, one broadcast shared-memory load of the pair's values and
 * two paired FMAs, on four warps per SMSP like the kernel's exponent warps,
 * without its tensor-memory loads, barriers or MMAs.  Synchronises
 * `stream`.  Reported beside the MUFU rate as the ceiling of that loop.
 */
gs_status gauss_sum_probe_ex2_mix_rate(void* stream, double* exp2_per_second);

/*
 * Accounting helper (not part of Eq. 1): number of CUDA kernels this
 * library has launched in this process, over all devices and streams,
 * counted on the host at each launch.  Never fails.
 */
uint64_t gauss_sum_kernel_launches(void);

#ifdef __cplusplus
}
#endif

#endif /* GAUSS_SUM_H */
