// Internal interfaces between the C ABI (api.cu) and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>

#include "gauss_sum.h"

namespace gs {

enum class InType { F32 = 0, F16 = 1, BF16 = 2 };

// Kernel launches of one library call, back to back on the caller's stream.
// A kernel launched right after another kernel of the same call carries the
// programmatic-stream-serialization attribute: it may be scheduled while its
// predecessor drains, and every library kernel waits (pdl_wait, ptx.cuh)
// for the previous kernel's completion before it reads that kernel's
// outputs.  The first kernel of a call, and a kernel after any other stream
// operation (memset, event record), is launched without it: t_pdl_next is
// cleared by pdl_reset() at those points and set by every kernel launch.
inline thread_local bool t_pdl_next = false;
inline void pdl_reset() { t_pdl_next = false; }

template <typename... K, typename... A>
cudaError_t launch_kernel(void (*kern)(K...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                          A... args) {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = t_pdl_next ? 1u : 0u;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, static_cast<K>(args)...);
    t_pdl_next = e == cudaSuccess;
    return e;
}

// Largest value-channel count evaluated on the FMA pipe (the P.v product of
// tc_gauss_fma.cu); more channels use the two-MMA kernel of tc_gauss.cu.
constexpr int kFmaMaxChannels = 4;
// Calls of at least this many pairs take the two-MMA kernel for three or
// four channels when the augmented rows fit (plan_tensor, tc_gauss.cu).
constexpr int64_t kTwoMmaMinPairs = int64_t(1) << 28;

// Workspace plan of the tensor-core path.  All offsets are bytes from the
// workspace base and are 1024-byte aligned.
struct TcPlan {
    int64_t M, N, D, Cv;     // Cv: value channels of one launch (C, or a chunk of the
                             // C (D + 1) gradient channels)
    int64_t Mpad, Npad;      // rows padded to the row tile / key tile
    int Dp, Cp;              // D and Cv rounded up to 16
    int BN;                  // key tile width (128, or 64 when Cp > 128)
    int splits;              // key splits per row tile (two-MMA kernel: of the tail row
                             // tiles, see main_tiles)
    // Two-MMA kernel: the first main_tiles row tiles (whole waves of one
    // CTA per SM) run unsplit in a first launch; the remaining row tiles
    // run with `splits` key splits in a second launch, so that the last
    // wave is not left part-empty.
    int64_t main_tiles;
    // Row tiles per wave of the main launch (the SM count): waves of odd
    // index walk the keys in reverse order, so that the keys the previous
    // wave read last are still in L2 when this wave starts.
    int wave_tiles;
    int stages;              // shared-memory pipeline depth
    size_t smem_bytes;       // dynamic shared memory of the fused kernel
    int mean_blocks;
    bool alias;              // q and k are the same array (M == N): prep once
    bool center;
    bool fma;                // kernel of tc_gauss_fma.cu (C <= kFmaMaxChannels, forward)
    bool aug;                // FMA kernel with augmented operands (Dp = D + 2 aug_norm_terms
                             // rounded to 16)
    bool tf;                 // fp32 inputs on the FMA kernel with 3xTF32 MMAs: q^ and k^
                             // rows are [hi | lo] of Dp (a multiple of 32) floats each
    int nq;                  // query tiles of 128 rows per CTA (FMA kernel)
    bool early_s;            // two-MMA kernel: S buffers handed back as soon as they are
                             // in registers (exponent-bound shapes), else with P
    // FMA kernel over the upper triangle of tile pairs (q = k, one value
    // channel; for v^T K v only): pair P of query tiles takes the key tiles
    // from 2P on, those past its own two with kernel values doubled, so the
    // row sums s'_m satisfy sum_m v_m s'_m = v^T K v.  tri_units: units per
    // problem, sum over pairs P of (key tiles - 2P).
    bool tri;
    int64_t tri_units;
    // Two-MMA kernel: q^ in tensor memory (MMA1 reads A from TMEM), so that
    // its shared memory goes to a fourth key stage.
    bool qtm;
    // FMA kernel work split: units = (pairs of query tiles) x key tiles, in
    // row-major order; CTA i takes units [i unit_len, (i + 1) unit_len); the
    // partial sums of a pair of query tiles have one slot per contributing
    // CTA (`splits` = the largest number of contributors).
    int64_t units, unit_len;
    int grid;
    // Banded order of the FMA kernel for keys larger than L2 (band_len > 0):
    // runs of band_len key tiles of one pair of query tiles, band-major, so
    // that the CTAs read the same bands at the same time; `splits` is then
    // the number of bands (one partial-sum slot per band).
    int band_len;
    int64_t nruns;
    // FMA kernel with short segments (runs of at most kOverlapMaxTiles key
    // tiles per pair of query tiles): the control warps start the next
    // segment's copies and MMAs while the exponent warps finish the current
    // one, instead of meeting them at a CTA barrier at every segment end.
    bool overlap;
    // FMA kernel, C = 1 with fp16 values on augmented operands: the value
    // magnitudes are folded into the key operands' norm terms
    // (log2(|v| 2^-16) / c) and the key records hold only signs (VF).
    bool vfold;
    // FMA kernel with augmented fp16 operands: the exponent scale c is folded
    // into the query rows (rn(c q^)), so the exponent loop has no multiply;
    // implied by vfold.
    bool cfold;
    // Problems of a batch handled by one launch (the FMA kernel stacks them:
    // q^ batch x Mpad rows, k^ batch x Npad rows); 1 for the other paths.
    int64_t batch;
    // FMA kernel: share of the exponentials computed on the FMA pipe
    // (gs_options.exp2_fma: 0 none, 1..4 = 1/32 .. 1/4).
    int exp2_fma;
    // Weighted vector-Jacobian pass (two-MMA kernel): the kernel values are
    // multiplied by pair weights w_mn = sum_c r[m, c] k[n, c] of wt (padded)
    // channels, computed from float32 factors in the exponent warps; 0: none.
    int wt;
    size_t off_rowf, off_colT, off_wmax;
    size_t off_mean_part, off_mu, off_qh, off_kh, off_A, off_B, off_vt, off_vmax, off_inv,
        off_rec, off_part, total;
};

struct SimtPlan {
    int64_t M, N, D, Cv;
    int dmax;          // register tile of the query row (16, 32, 64 or 128)
    int cblk;          // channels per launch slice
    int splits;
    int64_t keys_per_split;
    size_t off_part, total;
};

int device_sm_count(int device);
bool device_is_sm103(int device);

bool plan_tensor(InType t, int64_t M, int64_t N, int64_t D, int64_t C, bool grad, bool center,
                 bool alias, int split_override, int sms, TcPlan* p, const char** why,
                 int64_t batch = 1, bool tri = false, int wt = 0);
bool plan_simt(int64_t M, int64_t N, int64_t D, int64_t C, bool grad, int split_override,
               int sms, SimtPlan* p, const char** why);

// prep.cu --------------------------------------------------------------
// Key records of the FMA kernel that the mean launch may write alongside
// (values only: augmented operands, no norm terms in the records).
struct RecordArgs {
    const void* v;       // N x C values per problem, 16-bit like q, or fp32 (v_f32)
    bool v_f32;
    int64_t N, Npad;
    int C;
    float* out;          // Npad / 2 pairs x 2C floats per problem
    bool signs;          // sign records of folded value magnitudes (fp16 values, C = 1;
                         // per key tile of 128 keys: 128 signed 2^16 and 4 group words)
};
// Common mean of q and k per problem.  With `rec`, the launch also writes
// those key records where it can (the vectorised path); *rec_done says
// whether it did.
cudaError_t launch_mean(InType t, const void* q, const void* k, int64_t M, int64_t N, int D,
                        int blocks, float* partial, float* mu, cudaStream_t s, int batch = 1,
                        const RecordArgs* rec = nullptr, bool* rec_done = nullptr);
// (cf > 0 with vw: the exponent scale c folds into the query rows and the
// magnitudes of the fp16 values vw into the key rows' norm terms;
// vf_rec: sign records already written, whose per-problem flags the launch
// then also computes where it can, *flags_done saying whether it did.)
// Centred, rounded MMA operands of q (M rows, padded to Mpad) and, with
// with_k, of k (N rows, padded to Npad), in one launch where the vector
// path applies (16-bit inputs, D a multiple of 8).  aug: the augmented
// layout (Dp >= D + 2 aug_norm_terms(t)) into qh, and into qh_as_key (the
// key layout of the same points, for q = k; may be null) and kh; plain:
// x^ into qh / kh and the norm terms -(c/2)||x^||^2 into nrm_q / nrm_k
// (pad_value for padded rows).
cudaError_t launch_operands(InType t, bool aug, const void* q, int64_t M, int64_t Mpad,
                            void* qh, void* qh_as_key, float* nrm_q, bool with_k, const void* k,
                            int64_t N, int64_t Npad, void* kh, float* nrm_k, int D, int Dp,
                            const float* mu, float half_c, float pad_value, cudaStream_t s,
                            int batch = 1, const void* vw = nullptr, float cf = 0.f,
                            float* vf_rec = nullptr, bool* flags_done = nullptr);
// Transposed fp16 value operand of the two-MMA kernel for the channels
// ch0 .. ch0 + Cc - 1 (Cp >= Cc rows of Npad keys), with per-channel
// power-of-two scales.  Forward: channel ch of key n is w[n, ch] (w has the
// input dtype, Cw = channels).  grad: channel c (D + 1) + d is
// w[n, c] (x[n, d] - mu_d) for d < D and w[n, c] for d = D (w is N x Cw,
// float32 when w_f32, else the input dtype; x is N x D).
cudaError_t launch_value_prep(InType t, bool grad, bool w_f32, const void* w, const void* x,
                              const float* mu, int64_t N, int64_t Npad, int D, int Cw, int ch0,
                              int Cc, int Cp, unsigned* vmax_bits, void* vt, float* inv_scale,
                              cudaStream_t s);
// Factors of the pair weights w_mn = sum_c r[m, c] k[n, c] of the weighted
// vector-Jacobian pass (see prep.cu): row factors rsrc (R x C) into rowf
// (Rpad x WT float32), column factors csrc (Ncol x C) into colT (per key
// tile of BN keys, channel-major), their per-channel maxima into wmax
// (2 WT float bits).  One side is float32 (r_f32 / c_f32), the other has the
// inputs' dtype t.
cudaError_t launch_weight_prep(InType t, const void* rsrc, bool r_f32, int64_t R, int64_t Rpad,
                               const void* csrc, bool c_f32, int64_t Ncol, int64_t Npad, int C,
                               int WT, int BN, float* rowf, float* colT, unsigned* wmax,
                               cudaStream_t s);
// Forward: out (M x Cv) = inv_scale (when given) x the split partials summed
// in split order; rows below main_rows have one split.
cudaError_t launch_finalize(const float* part, int splits, int64_t split_stride_rows,
                            int64_t M, int Cv, int part_ld, const float* inv_scale, float* out,
                            cudaStream_t s, int64_t main_rows = 0);
// Gradient contraction of one launch's channels ch0 .. ch0 + Cc - 1 (see
// prep.cu): out[m, d] (+)= tau sum_c u[m, c] (S_{c,d} - x^_{m,d} S_{c,D}),
// s_out[m, c] = S_{c,D}.  direct: fp32 kernel partials (difference form).
cudaError_t launch_finalize_points(bool direct, InType t, bool u_f32, const float* part,
                                   int splits, int64_t split_stride_rows, int64_t M, int part_ld,
                                   const float* inv_scale, const void* x, const float* mu,
                                   float tau, int D, int Cw, int ch0, int Cc, const void* u,
                                   int accumulate, float* out, float* s_out, cudaStream_t s,
                                   int64_t main_rows = 0);
// MMD^2 of Sec. 3 per problem of a batch: out[b] = sum_n v[b, n] s[b, n]
// (float64 accumulation, fixed order), through float64 chunk partials in
// `partial` (mmd2_partial_bytes(B, N) bytes).
size_t mmd2_partial_bytes(int64_t B, int64_t N);
cudaError_t launch_mmd2_reduce(InType t, const float* s, const void* v, int64_t B, int64_t N,
                               double* partial, float* out, cudaStream_t st);
// Forward sum of the FMA kernel's contributor slots, added in slot order:
// every row has slots 0 .. fixed_slots - 1 when fixed_slots > 0 (banded
// order); otherwise rows of the pair of query tiles r = m / rows_per_unit
// have slots 0 .. last(r) - first(r), with first(r) = r key_tiles /
// unit_len and last(r) = ((r + 1) key_tiles - 1) / unit_len; with
// tri_key_tiles = T > 0 (upper-triangle order, rows of T + 2 units: pair s,
// then pair T / 2 - 1 - s) pair r = b (T / 2) + P holds T - 2P units.
cudaError_t launch_finalize_slots(const float* part, int64_t Mpad, int64_t M, int C,
                                  int rows_per_unit, int64_t key_tiles, int64_t unit_len,
                                  float* out, cudaStream_t s, int batch = 1,
                                  int fixed_slots = 0, int64_t tri_key_tiles = 0);

// simt_fp32.cu ---------------------------------------------------------
// grad: keys weighted by channel wch of v (N x Cw); partials have D + 1
// channels (sum Phi w (k - q), sum Phi w).
cudaError_t launch_simt(const SimtPlan& p, bool grad, const float* q, const float* k,
                        const float* v, int Cw, int wch, float half_c, float* part,
                        cudaStream_t s);

// Key records of the FMA kernel: per key pair (2t, 2t+1) the floats
// B_2t, B_2t+1 (omitted when B is null), v_2t[0], v_2t+1[0], ...,
// v_2t[C-1], v_2t+1[C-1].
cudaError_t launch_key_records(InType t, const void* v, const float* B, int64_t N, int64_t Npad,
                               int C, float* rec, cudaStream_t s, int batch = 1, bool signs = false);
// 3xTF32 operands of fp32 inputs (see prep.cu): rows of 2 Dp floats
// [hi | lo] into out, nrm = -(c/2)||x - mu||^2 (pad_value for padded rows).
cudaError_t launch_tf32_split(const float* x, int64_t rows, int64_t rows_pad, int D, int Dp,
                              const float* mu, float half_c, float* out, float* nrm,
                              float pad_value, cudaStream_t s, int batch = 1);
constexpr int aug_norm_terms(InType t) { return t == InType::BF16 ? 3 : 2; }

// tc_gauss.cu ----------------------------------------------------------
cudaError_t launch_tc(const TcPlan& p, InType t, float c, char* ws, unsigned* status,
                      cudaStream_t s, const char** why);

// tc_gauss_fma.cu ------------------------------------------------------
// Largest (augmented) Dp for which the FMA kernel keeps q^ in shared memory
// and folds the norms into the MMA.
constexpr int kAugMaxDp = 128;
// Largest D of the 3xTF32 (fp32) variant: q^ hi and lo tiles of two query
// tiles stay in shared memory next to the key stages.
constexpr int kTf32MaxDp = 32;
bool plan_fma_kernel(int Dp, int C, bool aug, bool tf, int* nq, int* stages, size_t* smem);
// vf_pass (plans with vfold): 1 = the problems whose 32-key groups all have
// values of one sign, 2 = the others (launched after pass 1); 0 otherwise.
cudaError_t launch_tc_fma(const TcPlan& p, InType t, float c, char* ws, unsigned* status,
                          cudaStream_t s, const char** why, int vf_pass = 0);
// Per-problem words after the sign records (rec: batch x (Npad / 128) tiles
// of 132 floats): 1 where every 32-key group of the problem has values of
// one sign, else 0.
cudaError_t launch_vf_flags(float* rec, int64_t Npad, int batch, cudaStream_t s);

// probe
// Best of three timed runs of the ex2 probe kernel: independent ex2 chains
// (mix false), or the FMA kernel's exponent-loop instruction mix (true).
cudaError_t run_ex2_probe(cudaStream_t s, double* rate, bool mix);

// api.cu: workspace bytes that a forward call with exactly these arguments
// and default options needs (through *bytes), or the status the call
// would fail with; and recording a message for gauss_sum_last_error().
gs_status forward_workspace_bytes(const void* q, const void* k, const void* v, double tau,
                                  int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype,
                                  float* out, size_t* bytes);
gs_status set_last_error(gs_status st, const char* msg);
// Adds n to the count behind gauss_sum_kernel_launches(); called right
// after each kernel launch of the library.
void note_launches(int n);
// Records the variant of the last fused FMA-kernel launch (bit flags of
// gauss_sum_testing_last_fma_variant).
void note_fma_variant(int flags);

}  // namespace gs
