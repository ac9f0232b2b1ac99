// Preparation and finalisation kernels of the Gauss-sum path.
//
//  * common mean of all query and key points (the shift safeguard of
//    Remark 2, Sec. 2: the kernel depends on q - k only, so any common shift
//    is exact and only changes rounding), rounded to the input format's
//    grid so that the shift itself adds no rounding near the mean;
//  * centring, rounding to the MMA operand type and the scaled squared norms
//    A_m = -(c/2)||q^_m||^2, B_n = -(c/2)||k^_n||^2 (c = tau log2 e) taken
//    from the ROUNDED points, so that c q^.k^ + A_m + B_n is exactly
//    -(c/2)||q^_m - k^_n||^2 up to fp32 rounding (the norm factors of Alg. 1,
//    folded into one exponent);
//  * the value operand: per-channel power-of-two scaling of v (or of the
//    gradient values (v_n k_n, v_n) of Sec. 3) rounded to fp16 and stored
//    transposed (channel-major) so that both MMAs read K-major operands;
//  * the fixed-order sum of key-split partials and the final scaling, or
//    the gradient tau (S[:D] - q_m S[D]) of Sec. 3.
#include <algorithm>
#include <type_traits>

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <math_constants.h>

#include "internal.h"
#include "ptx.cuh"

namespace gs {
namespace {

template <typename T> __device__ __forceinline__ float to_f(T x);
template <> __device__ __forceinline__ float to_f<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f<__half>(__half x) { return __half2float(x); }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) {
    return __bfloat162float(x);
}

// a / b for a non-negative a below 2^32 with 32-bit division (much
// cheaper than the 64-bit one), else 64-bit.
__device__ __forceinline__ int64_t div_nonneg(int64_t a, int b) {
    if (a <= 0xffffffffLL)
        return static_cast<int64_t>(static_cast<uint32_t>(a) / static_cast<uint32_t>(b));
    return a / b;
}

template <typename H> __device__ __forceinline__ H from_f(float x);
template <> __device__ __forceinline__ __half from_f<__half>(float x) { return __float2half_rn(x); }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

// ---------------------------------------------------------------- mean
// Block (32, 8): 32 consecutive coordinates x 8 row lanes; each block sums
// a contiguous chunk of the stacked rows [q; k] and writes, per coordinate,
// its partial sum (partial[block][d]) and largest magnitude
// (partial[G + block][d]).
template <typename T>
__global__ void mean_partial_kernel(const T* __restrict__ q, const T* __restrict__ k, int64_t M,
                                    int64_t N, int D, int64_t rows_per_block,
                                    float* __restrict__ partial) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[8][33];
    __shared__ float big[8][33];
    // Problem blockIdx.y of a batch: its own points and partial rows.
    q += static_cast<int64_t>(blockIdx.y) * M * D;
    k += static_cast<int64_t>(blockIdx.y) * N * D;
    partial += static_cast<int64_t>(blockIdx.y) * 2 * gridDim.x * D;
    const int64_t r0 = static_cast<int64_t>(blockIdx.x) * rows_per_block;
    const int64_t r1 = min(r0 + rows_per_block, M + N);
    for (int d0 = 0; d0 < D; d0 += 32) {
        const int d = d0 + threadIdx.x;
        float acc = 0.f, mx = 0.f;
        if (d < D) {
            for (int64_t r = r0 + threadIdx.y; r < r1; r += 8) {
                const float x = to_f(r < M ? q[r * D + d] : k[(r - M) * D + d]);
                acc += x;
                mx = fmaxf(mx, fabsf(x));
            }
        }
        red[threadIdx.y][threadIdx.x] = acc;
        big[threadIdx.y][threadIdx.x] = mx;
        __syncthreads();
        if (threadIdx.y == 0 && d < D) {
            float sum = 0.f, m = 0.f;
#pragma unroll
            for (int y = 0; y < 8; ++y) {
                sum += red[y][threadIdx.x];
                m = fmaxf(m, big[y][threadIdx.x]);
            }
            partial[static_cast<int64_t>(blockIdx.x) * D + d] = sum;
            partial[static_cast<int64_t>(gridDim.x + blockIdx.x) * D + d] = m;
        }
        __syncthreads();
    }
}

// Vectorised variant for 16-bit inputs with D a power of two in [8, 2048]:
// 256 threads read 16-byte vectors (8 coordinates) of a contiguous run of
// rows; a block advances by 2048 elements, a multiple of D, so every thread
// always sees the same 8 coordinates and keeps their sums and maxima in
// registers.  Blocks [0, Gq) cover rows of q, blocks [Gq, G) rows of k
// (none when q and k are the same points).  Same partial layout as above.
// Blocks from G on, when given a record job, write the FMA kernel's key
// records instead (see key_record_kernel): they depend on the values only,
// so they ride along in this first launch of the call rather than taking
// a launch of their own later in the chain.
constexpr int kMeanVecThreads = 256;

template <typename TV>
struct RecordJob {
    const TV* v;         // N x C values per problem (batch-stacked)
    int64_t N, pairs;    // keys and key pairs (Npad / 2) per problem
    int C;
    float* rec;          // pairs x 2C floats per problem
    bool signs;          // sign records (see sign_record) instead of values
};

// Sign records of the FMA kernel with folded value magnitudes (C = 1, the
// magnitudes sit in the key operands): per key tile of kRecTile keys, the
// floats s_n = sign(v_n) 2^16 in key order (0 for v_n = 0 and for padded
// keys), then one word per group of 32 keys: -2^16 if the group's nonzero
// values are all negative, 0 if it has values of both signs, else 2^16.
// One thread per key n < Npad of problem `problem`, whole warps per group.
constexpr int kRecTile = 128;
constexpr int kRecTileFloats = kRecTile + kRecTile / 32;

__device__ __forceinline__ void write_sign_record(const __half* v, int64_t N, float* rec, int64_t n,
                                                  int problem, int64_t npad) {
    const float x = n < N ? __half2float(v[static_cast<int64_t>(problem) * N + n]) : 0.f;
    const float sg = x > 0.f ? 65536.f : x < 0.f ? -65536.f : 0.f;
    float* r = rec + (static_cast<int64_t>(problem) * (npad / kRecTile) + n / kRecTile) * kRecTileFloats;
    const int kn = static_cast<int>(n % kRecTile);
    r[kn] = sg;
    // Zero values and padded keys contribute nothing whatever the group's
    // sign (their folded exponent flushes), so only the signs of the
    // nonzero values decide.
    const bool any_pos = __any_sync(0xffffffffu, x > 0.f);
    const bool any_neg = __any_sync(0xffffffffu, x < 0.f);
    if ((kn & 31) == 0) r[kRecTile + kn / 32] = any_pos && any_neg ? 0.f : any_neg ? -65536.f : 65536.f;
}

// One block per problem b: the AND over its 32-key groups of "values of
// one sign" (group word != 0), into the word after all problems' records.
// Every thread of the block calls this.
__device__ __forceinline__ void write_vf_flag(float* __restrict__ rec, int64_t tiles, int batch, int b) {
    const float* gw = rec + static_cast<int64_t>(b) * tiles * kRecTileFloats + kRecTile;
    bool mixed = false;
    for (int64_t i = threadIdx.x; i < tiles * (kRecTile / 32); i += blockDim.x)
        mixed |= gw[(i / (kRecTile / 32)) * kRecTileFloats + i % (kRecTile / 32)] == 0.f;
    const int any_mixed = __syncthreads_or(mixed ? 1 : 0);
    if (threadIdx.x == 0)
        reinterpret_cast<unsigned*>(rec + static_cast<int64_t>(batch) * tiles * kRecTileFloats)[b] =
            any_mixed ? 0u : 1u;
}

__global__ void __launch_bounds__(256)
vf_flags_kernel(float* __restrict__ rec, int64_t tiles, int batch) {
    pdl_trigger();
    pdl_wait();
    write_vf_flag(rec, tiles, batch, blockIdx.x);
}

__global__ void sign_record_kernel(const __half* __restrict__ v, int64_t N, int64_t npad,
                                   float* __restrict__ rec) {
    pdl_trigger();
    pdl_wait();
    const int64_t n = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (n < npad) write_sign_record(v, N, rec, n, blockIdx.y, npad);
}

template <typename TV>
__device__ __forceinline__ void write_key_record(const RecordJob<TV>& j, int64_t t, int problem) {
    const int64_t n0 = 2 * t, n1 = 2 * t + 1;
    const TV* v = j.v + static_cast<int64_t>(problem) * j.N * j.C;
    float* out = j.rec + (static_cast<int64_t>(problem) * j.pairs + t) * (2 * j.C);
    for (int c = 0; c < j.C; ++c) {
        out[2 * c] = n0 < j.N ? to_f(v[n0 * j.C + c]) : 0.f;
        out[2 * c + 1] = n1 < j.N ? to_f(v[n1 * j.C + c]) : 0.f;
    }
}

template <typename T, typename TV>
__global__ void __launch_bounds__(kMeanVecThreads)
mean_partial_vec_kernel(const T* __restrict__ q, const T* __restrict__ k, int64_t M, int64_t N,
                        int D, int64_t rows_per_block, int Gq, int G, float* __restrict__ partial,
                        const RecordJob<TV> rj) {
    pdl_trigger();
    pdl_wait();
    if (static_cast<int>(blockIdx.x) >= G) {
        const int64_t t = static_cast<int64_t>(blockIdx.x - G) * kMeanVecThreads + threadIdx.x;
        if (rj.signs) {
            if constexpr (std::is_same<TV, __half>::value) {
                if (t < 2 * rj.pairs) write_sign_record(rj.v, rj.N, rj.rec, t, blockIdx.y, 2 * rj.pairs);
            }
        } else if (t < rj.pairs) {
            write_key_record(rj, t, blockIdx.y);
        }
        return;
    }
    __shared__ float s_sum[kMeanVecThreads][9];
    __shared__ float s_max[kMeanVecThreads][9];
    const int t = threadIdx.x;
    // Problem blockIdx.y of a batch: its own points and partial rows.
    q += static_cast<int64_t>(blockIdx.y) * M * D;
    k += static_cast<int64_t>(blockIdx.y) * N * D;
    partial += static_cast<int64_t>(blockIdx.y) * 2 * G * D;
    const bool on_q = static_cast<int>(blockIdx.x) < Gq;
    const int64_t b = on_q ? blockIdx.x : blockIdx.x - Gq;
    const int64_t rows = on_q ? M : N;
    const T* x = on_q ? q : k;
    const int64_t r0 = b * rows_per_block;
    const int64_t r1 = min(r0 + rows_per_block, rows);
    const int64_t v0 = r0 * D / 8, v1 = r1 * D / 8;      // 8-element vectors
    const uint4* xv = reinterpret_cast<const uint4*>(x);
    float sum[8], mx[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) sum[e] = mx[e] = 0.f;
    // Four vectors in flight per thread, then the remainder one at a time
    // (each thread's vectors are accumulated in index order either way).
    auto add = [&](const uint4 u) {
        const T* h = reinterpret_cast<const T*>(&u);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float f = to_f(h[e]);
            sum[e] += f;
            mx[e] = fmaxf(mx[e], fabsf(f));
        }
    };
    int64_t v = v0 + t;
    for (; v + 3 * kMeanVecThreads < v1; v += 4 * kMeanVecThreads) {
        uint4 u[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) u[r] = xv[v + r * kMeanVecThreads];
#pragma unroll
        for (int r = 0; r < 4; ++r) add(u[r]);
    }
    for (; v < v1; v += kMeanVecThreads) add(xv[v]);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        s_sum[t][e] = sum[e];
        s_max[t][e] = mx[e];
    }
    __syncthreads();
    // Thread t holds coordinates 8 (t mod NG) .. +7, NG = D / 8 groups.
    const int NG = D / 8;
    for (int d = t; d < D; d += kMeanVecThreads) {
        const int g = d >> 3, e = d & 7;
        float a = 0.f, m = 0.f;
        for (int u = g; u < kMeanVecThreads; u += NG) {
            a += s_sum[u][e];
            m = fmaxf(m, s_max[u][e]);
        }
        partial[static_cast<int64_t>(blockIdx.x) * D + d] = a;
        partial[static_cast<int64_t>(G + blockIdx.x) * D + d] = m;
    }
}

// mu_d = the mean of coordinate d rounded to a multiple of g_d, the spacing
// of the input format at max |x_d| (2^(e - mant_bits) for max |x_d| in
// [2^e, 2^(e+1)), at least the subnormal spacing 2^min_exp).  Every input
// x_d is a multiple of its own spacing, which divides g_d, so x_d - mu_d is
// a multiple of the spacing of x_d: it is exact in the input format
// whenever |x_d - mu_d| stays below 2^(e_x + 1) (x_d in [2^e_x, 2^(e_x+1))),
// i.e. the shift adds no rounding for points near the mean.  Any common
// shift leaves the Gauss sum unchanged.
constexpr int kMeanFinalThreads = 256;

// The grid-rounded mean of the folded sum s and largest magnitude mx.
__device__ __forceinline__ float rounded_mean(float s, float mx, float total, int mant_bits,
                                              int min_exp) {
    // float32 throughout: any shift is exact for the Gauss sum, so the mean
    // needs no more precision than that, and float64 is slow on this GPU.
    float m = s / total;
    if (mx > 0.f) {
        int e;
        frexpf(mx, &e);                                   // mx in [2^(e-1), 2^e)
        const float g = ldexpf(1.f, max(e - 1 - mant_bits, min_exp));
        m = rintf(m / g) * g;
    }
    return m;
}

// Many partials per coordinate (G > kMeanFinalThreadMax): one block per
// (coordinate d, problem blockIdx.y); thread t folds partials t, t + 256,
// ... in order, a fixed butterfly adds the lanes of each warp and thread 0
// the warps in order (deterministic).
constexpr int kMeanFinalThreadMax = 32;

__global__ void __launch_bounds__(kMeanFinalThreads)
mean_final_block_kernel(const float* __restrict__ partial, int G, int D, float total,
                        int mant_bits, int min_exp, float* __restrict__ mu) {
    pdl_trigger();
    pdl_wait();
    constexpr int W = kMeanFinalThreads / 32;
    __shared__ float red_s[W];
    __shared__ float red_m[W];
    const int d = blockIdx.x;
    const int t = threadIdx.x;
    partial += static_cast<int64_t>(blockIdx.y) * 2 * G * D;
    mu += static_cast<int64_t>(blockIdx.y) * D;
    float s = 0.f;
    float mx = 0.f;
    for (int g = t; g < G; g += kMeanFinalThreads) {
        s += partial[static_cast<int64_t>(g) * D + d];
        mx = fmaxf(mx, partial[static_cast<int64_t>(G + g) * D + d]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        s += __shfl_xor_sync(0xffffffffu, s, o);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if ((t & 31) == 0) {
        red_s[t >> 5] = s;
        red_m[t >> 5] = mx;
    }
    __syncthreads();
    if (t == 0) {
        float a = 0.f, m = 0.f;
        for (int w = 0; w < W; ++w) {
            a += red_s[w];
            m = fmaxf(m, red_m[w]);
        }
        mu[d] = rounded_mean(a, m, total, mant_bits, min_exp);
    }
}

// Few partials per coordinate (the small problems of a batch): one thread
// per item = (problem b, coordinate d), folding the G partials in order.
__global__ void __launch_bounds__(kMeanFinalThreads)
mean_final_kernel(const float* __restrict__ partial, int G, int D, int64_t items, float total,
                  int mant_bits, int min_exp, float* __restrict__ mu) {
    pdl_trigger();
    pdl_wait();
    const int64_t it = static_cast<int64_t>(blockIdx.x) * kMeanFinalThreads + threadIdx.x;
    if (it >= items) return;
    const int64_t b = it / D;
    const int d = static_cast<int>(it - b * D);
    partial += b * 2 * G * D;                      // problem b
    float s = 0.f;
    float mx = 0.f;
    for (int g = 0; g < G; ++g) {
        s += partial[static_cast<int64_t>(g) * D + d];
        mx = fmaxf(mx, partial[static_cast<int64_t>(G + g) * D + d]);
    }
    mu[it] = rounded_mean(s, mx, total, mant_bits, min_exp);
}

// ---------------------------------------------------------------- MMA operands
// Both operand layouts are written by one kernel that stages kRowsPerBlock
// rows through shared memory: the block's input rows are one contiguous
// run of rows x D elements (16-byte vector loads), and its output rows one
// contiguous run of rows x Dp elements (16-byte vector stores).  One warp
// per row inside the block.
//
// Plain layout (AUG = false): centred points rounded to the MMA type,
// x^ = rn(x - mu), zero padded to Dp columns, and the scaled squared norm
// nrm = -(c/2)||x^||^2 (c = tau log2 e) taken from the ROUNDED point, so that
// c q^.k^ + A_m + B_n is exactly -(c/2)||q^_m - k^_n||^2 up to fp32
// rounding (the norm factors of Alg. 1 folded into one exponent).  Rows in
// [rows, rows_pad) become zero rows with norm `pad_value` (-inf for padded
// keys, so their kernel value is 0).
//
// Augmented layout (AUG = true): x^ followed by 2 NT columns that make the
// MMA produce the whole exponent up to the factor c:
//   query rows  [q^, F, 1, .., 1, a_0, a_1, .., a_NT-1, 0 ...]
//   key rows    [k^, b_0, b_1, .., b_NT-1, F, 1, .., 1, 0 ...]
// with a = -||q^||^2 / 2 and b = -||k^||^2 / 2 taken from the rounded
// points in fp32 and written as F t_0 + t_1 + ... + t_NT-1, each t_i a
// rounded remainder, so that
//   q^_aug . k^_aug = q^.k^ + a + b = -||q^ - k^||^2 / 2
// up to the split error (|a| 2^-22 for two fp16 terms, |a| 2^-24 for three
// bf16 terms) and the fp32 accumulation; the kernel value is 2^(c S).  The
// power of two F (1024 for fp16) keeps norms up to 6.7e7 inside the fp16
// range.  Padded key rows get b_0 = -30000 / F (their values are zero as
// well); padded query rows are zero.  `out_q` and/or `out_k` may be given
// (both for q = k).
//
// Folded exponent scale and value magnitudes (cf = c > 0, one fp16 value
// per key in vw): the query rows hold u = rn(c q^), with a = -||u||^2/(2c),
// and the key rows b = -c ||k^||^2 / 2 + log2(|v_n| 2^-16), so that the MMA
// yields S = u.k^ + a + b = -(1/(2c)) ||u - c k^||^2 + log2(|v_n| 2^-16):
// the exponent of Phi |v_n| 2^-16 itself, at the query point u / c (within
// 2^-12 of q^ per coordinate), and never above log2(|v_n| 2^-16) in exact
// arithmetic.  The FMA kernel then needs no multiply by c and only the
// signs of the values (see write_sign_record).  |v_n| < 2^16 for every
// finite fp16 value.  Keys with v_n = 0 get -256: their 2^S flushes to
// zero, so they may sit in a group of either sign (padded keys have
// -30000 already).
constexpr float kZeroWeightLog2 = -256.f;

__device__ __forceinline__ float log_weight(const __half* vw) {
    if (!vw) return 0.f;
    const float a = fabsf(__half2float(*vw));
    return a > 0.f ? log2f(a * (1.f / 65536.f)) : kZeroWeightLog2;
}

constexpr int kRowsPerBlock = 32;
constexpr int kOperandThreads = 128;
constexpr int kOperandMaxCols = 256;

template <typename T, bool AUG>
__global__ void __launch_bounds__(kOperandThreads)
operand_kernel(const T* __restrict__ x, int64_t rows, int64_t rows_pad, int D, int Dp, int nt, float F,
               const float* __restrict__ mu, float half_c, float pad_value,
               T* __restrict__ out_q, T* __restrict__ out_k, float* __restrict__ nrm,
               const __half* __restrict__ vw, float cf) {
    pdl_trigger();
    pdl_wait();
    constexpr int R = kRowsPerBlock;
    // Dynamic shared memory sized to this call: s_out holds R x Dp
    // elements per written layout (AUG: q rows, then k rows), s_in the R x D
    // input elements (rounded up to 16 bytes), then D floats of mu.
    extern __shared__ __align__(16) uint8_t operand_smem[];
    const bool wq = AUG ? out_q != nullptr : true;
    const bool wk = AUG && out_k != nullptr;
    const int nout = (wq ? 1 : 0) + (wk ? 1 : 0);
    T* s_out = reinterpret_cast<T*>(operand_smem);
    T* s_in = s_out + nout * R * Dp;
    float* s_mu = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(s_in) +
                                           ((R * D * static_cast<int>(sizeof(T)) + 15) & ~15));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // Problem blockIdx.y of a batch: its own rows, mean and outputs.
    {
        const int64_t b = blockIdx.y;
        x += b * rows * D;
        if (mu) mu += b * D;
        if (out_q) out_q += b * rows_pad * Dp;
        if (out_k) out_k += b * rows_pad * Dp;
        if (nrm) nrm += b * rows_pad;
        if (vw) vw += b * rows;
    }
    const int64_t r0 = static_cast<int64_t>(blockIdx.x) * R;
    for (int d = tid; d < D; d += kOperandThreads) s_mu[d] = mu ? mu[d] : 0.f;
    const int64_t left = rows - r0;
    const int rin = left <= 0 ? 0 : left >= R ? R : static_cast<int>(left);
    {
        // The block's rows are one run of rin x D elements.  Within one
        // problem its start (r0 D sizeof(T), r0 a multiple of 32) is 16-byte
        // aligned; a later problem of a batch may start anywhere, so the
        // vector loads are used only when the run is 16-byte aligned.
        const int n_el = rin * D;
        constexpr int PER_VEC = 16 / static_cast<int>(sizeof(T));
        const T* src = x + r0 * D;
        const int nvec = (reinterpret_cast<uintptr_t>(src) & 15u) == 0 ? n_el / PER_VEC : 0;
        for (int i = tid; i < nvec; i += kOperandThreads)
            reinterpret_cast<uint4*>(s_in)[i] = reinterpret_cast<const uint4*>(src)[i];
        for (int i = nvec * PER_VEC + tid; i < n_el; i += kOperandThreads) s_in[i] = src[i];
    }
    __syncthreads();
    T* sq = s_out;
    T* sk = s_out + (wq ? R * Dp : 0);
    const T zero = from_f<T>(0.f);
    for (int row = warp; row < R; row += kOperandThreads / 32) {
        const bool valid = row < rin;
        T* oq = sq + row * Dp;
        T* ok = sk + row * Dp;
        float acc = 0.f, accu = 0.f;
        const bool fold = AUG && cf > 0.f;
        const int dend = AUG ? D : Dp;
        for (int d = lane; d < dend; d += 32) {
            const float val = (valid && d < D) ? to_f(s_in[row * D + d]) - s_mu[d] : 0.f;
            const T h = from_f<T>(val);
            const float hf = to_f(h);
            if (fold) {
                const T hs = from_f<T>(cf * hf);   // folded scale: the query row holds rn(c x^)
                if (wq) oq[d] = hs;
                accu = fmaf(to_f(hs), to_f(hs), accu);
            } else if (wq) {
                oq[d] = h;
            }
            if (wk) ok[d] = h;
            acc = fmaf(hf, hf, acc);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            acc += __shfl_xor_sync(0xffffffffu, acc, o);
            accu += __shfl_xor_sync(0xffffffffu, accu, o);
        }
        if (!AUG) {
            if (lane == 0) nrm[r0 + row] = valid ? -half_c * acc : pad_value;
            continue;
        }
        for (int d = D + 2 * nt + lane; d < Dp; d += 32) {
            if (wq) oq[d] = zero;
            if (wk) ok[d] = zero;
        }
        if (lane < nt) {
            // Lane i writes term i of the split and its partner column (the
            // key side with its log weight, when values are folded).
            auto split_term = [&](float r) {
                T t = from_f<T>(r / F);
                r -= F * to_f(t);
                for (int i = 1; i <= lane; ++i) {
                    t = from_f<T>(r);
                    r -= to_f(t);
                }
                return t;
            };
            T t = zero, tk = zero, one = zero;
            if (valid) {
                if (fold) {
                    t = split_term(-0.5f * accu / cf);
                    tk = split_term(-0.5f * cf * acc + log_weight(vw ? vw + r0 + row : nullptr));
                } else {
                    t = tk = split_term(-0.5f * acc);
                }
                one = from_f<T>(lane == 0 ? F : 1.f);
            } else if (lane == 0) {
                t = tk = from_f<T>(-30000.f / F);
            }
            if (wq) {
                oq[D + lane] = valid ? one : zero;
                oq[D + nt + lane] = valid ? t : zero;
            }
            if (wk) {
                ok[D + lane] = tk;
                ok[D + nt + lane] = one;
            }
        }
    }
    __syncthreads();
    // r0 Dp sizeof(T) is a multiple of 16 (Dp is a multiple of 16).
    const int nvec = R * Dp * static_cast<int>(sizeof(T)) / 16;
    if (wq) {
        uint4* dst = reinterpret_cast<uint4*>(out_q + r0 * Dp);
        for (int i = tid; i < nvec; i += kOperandThreads) dst[i] = reinterpret_cast<const uint4*>(sq)[i];
    }
    if (wk) {
        uint4* dst = reinterpret_cast<uint4*>(out_k + r0 * Dp);
        for (int i = tid; i < nvec; i += kOperandThreads) dst[i] = reinterpret_cast<const uint4*>(sk)[i];
    }
}

// 3xTF32 operands (fp32 inputs on the tensor cores).  Row r of problem b
// becomes 2 Dp floats [hi_0 .. hi_Dp-1, lo_0 .. lo_Dp-1] with
// x^ = x - mu (fp32), hi = x^ rounded to tf32 and lo = (x^ - hi) rounded to
// tf32, zero padded; q^.k^ is then hi.hi + hi.lo + lo.hi up to the dropped
// lo.lo term (2^-22 relative).  nrm = -(c/2) ||x^||^2 from the fp32 x^;
// rows in [rows, rows_pad) are zero with norm pad_value.  One warp per row,
// over all problems of a batch.
__global__ void tf32_split_kernel(const float* __restrict__ x, int64_t rows, int64_t rows_pad,
                                  int64_t total_rows, int D, int Dp,
                                  const float* __restrict__ mu, float half_c, float pad_value,
                                  float* __restrict__ out, float* __restrict__ nrm) {
    pdl_trigger();
    pdl_wait();
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= total_rows) return;
    const int64_t b = w / rows_pad;
    const int64_t r = w - b * rows_pad;
    const bool valid = r < rows;
    const float* xr = x + (b * rows + r) * D;
    const float* mb = mu ? mu + b * D : nullptr;
    float* o = out + w * 2 * Dp;
    float acc = 0.f;
    for (int d = lane; d < Dp; d += 32) {
        const float xv = (valid && d < D) ? xr[d] - (mb ? mb[d] : 0.f) : 0.f;
        const float hi = round_tf32(xv);
        o[d] = hi;
        o[Dp + d] = round_tf32(xv - hi);
        acc = fmaf(xv, xv, acc);
    }
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, s);
    if (lane == 0) nrm[w] = valid ? -half_c * acc : pad_value;
}

__global__ void finalize_slots_kernel(const float* __restrict__ part, int64_t Mpad, int64_t M,
                                      int C, int rows_per_unit, int64_t key_tiles,
                                      int64_t unit_len, int64_t batch, int fixed_slots,
                                      int64_t tri_kt, float* __restrict__ out) {
    pdl_trigger();
    pdl_wait();
    // out: batch x M x C; partial rows are batch-stacked with Mpad rows per
    // problem and batch Mpad rows per slot.
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= batch * M * C) return;
    const int64_t bm = div_nonneg(idx, C);
    const int c = static_cast<int>(idx - bm * C);
    const int64_t b = M <= 0x7fffffff ? div_nonneg(bm, static_cast<int>(M)) : bm / M;
    const int64_t m = (bm - b * M) + b * Mpad;
    int64_t nslots = fixed_slots;
    if (nslots == 0 && tri_kt > 0) {
        // Upper-triangle order (folded rows of tri_kt + 2 units: pair s,
        // then pair ppb - 1 - s): pair P of problem b holds tri_kt - 2P units.
        const int64_t r = m / rows_per_unit;
        const int64_t ppb = tri_kt / 2;
        const int64_t bb = r / ppb, P = r - bb * ppb;
        const int64_t U = ppb * tri_kt - ppb * (ppb - 1);
        const int64_t s = 2 * P <= ppb - 1 ? P : ppb - 1 - P;
        const int64_t start = bb * U + s * (tri_kt + 2) + (s == P ? 0 : tri_kt - 2 * s);
        const int64_t first = start / unit_len;
        const int64_t last = (start + tri_kt - 2 * P - 1) / unit_len;
        nslots = last - first + 1;
    } else if (nslots == 0) {
        const int64_t r = m / rows_per_unit;
        const int64_t first = r * key_tiles / unit_len;
        const int64_t last = ((r + 1) * key_tiles - 1) / unit_len;
        nslots = last - first + 1;
    }
    float acc = 0.f;
    for (int64_t sl = 0; sl < nslots; ++sl) acc += part[(sl * batch * Mpad + m) * C + c];
    out[idx] = acc;
}

// Vectorised variant of operand_kernel for D a multiple of 8: G lanes
// (G = the power of two >= D / 8) share a row, each converting one 16-byte
// vector of 8 coordinates straight from global memory to global memory;
// the squared norm is reduced over the G lanes and the group's first lane
// writes the columns past D (norm terms or zeros).  Same outputs as
// operand_kernel.
constexpr int kOperandVecThreads = 256;

template <typename T> __device__ __forceinline__ T bits_to(unsigned short b);
template <> __device__ __forceinline__ __half bits_to<__half>(unsigned short b) {
    return __ushort_as_half(b);
}
template <> __device__ __forceinline__ __nv_bfloat16 bits_to<__nv_bfloat16>(unsigned short b) {
    return __ushort_as_bfloat16(b);
}
template <typename T> __device__ __forceinline__ unsigned short to_bits(T h);
template <> __device__ __forceinline__ unsigned short to_bits<__half>(__half h) {
    return __half_as_ushort(h);
}
template <> __device__ __forceinline__ unsigned short to_bits<__nv_bfloat16>(__nv_bfloat16 h) {
    return __bfloat16_as_ushort(h);
}

// Packed 16-bit pair arithmetic of the operand conversion.  x - mu of two
// 16-bit inputs and a mean on the input grid (see rounded_mean), rounded
// once to the input format (the MMA operand type), and the pair as floats.
template <typename T> struct Pair;
template <> struct Pair<__half> {
    using P = __half2;
    static __device__ __forceinline__ P sub(P a, P b) { return __hsub2(a, b); }
    static __device__ __forceinline__ float2 to_f2(P a) { return __half22float2(a); }
    static __device__ __forceinline__ P from_f2(float lo, float hi) { return __floats2half2_rn(lo, hi); }
};
template <> struct Pair<__nv_bfloat16> {
    using P = __nv_bfloat162;
    static __device__ __forceinline__ P sub(P a, P b) { return __hsub2(a, b); }
    static __device__ __forceinline__ float2 to_f2(P a) { return __bfloat1622float2(a); }
    static __device__ __forceinline__ P from_f2(float lo, float hi) { return __floats2bfloat162_rn(lo, hi); }
};

// One output row of the operand layouts, converted by the G lanes of a
// row group: lane vi holds the row's 16-byte input vectors vi, vi + G, ...
// (in[e] = vector vi + G e, 8 coordinates each, for vi + G e < D / 8; up to
// kOperandVecs of them) and smean the problem's mean as packed pairs of the
// input format in shared memory (exact: the mean lies on the input grid).
// out_q / out_k: the row in either layout (either may be null; AUG only).
// Every lane of the warp must call this together (the squared norm is
// reduced with shuffles over the G lanes); rows outside the output (in_pad
// false) write nothing.  Returns the norm term written for the row (plain
// layout: -(c/2)||x^||^2, or pad_value) in every lane.
constexpr int kOperandVecs = 8;

template <typename T, bool AUG, int G>
__device__ __forceinline__ float operand_row(const uint4 (&in)[kOperandVecs],
                                             const uint4* __restrict__ smean, int vi,
                                             bool in_pad, bool valid, int D, int Dp, int nt,
                                             float F, float half_c, float pad_value,
                                             T* __restrict__ out_q, T* __restrict__ out_k,
                                             float cf, const __half* vw) {
    using PT = Pair<T>;
    const int V = D / 8;
    const bool fold = AUG && cf > 0.f;
    float acc = 0.f, accu = 0.f;
    if (in_pad) {
        uint64_t acc2 = 0ull, accu2 = 0ull;
#pragma unroll
        for (int e = 0; e < kOperandVecs; ++e) {
            const int v = vi + G * e;
            if (v >= V) break;
            uint4 u = make_uint4(0u, 0u, 0u, 0u), us = u;
            if (valid) {
                const uint4 m2 = smean[v];
                const typename PT::P* x2 = reinterpret_cast<const typename PT::P*>(&in[e]);
                const typename PT::P* mm = reinterpret_cast<const typename PT::P*>(&m2);
                typename PT::P h[4], hs[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    h[k] = PT::sub(x2[k], mm[k]);
                    const float2 f = PT::to_f2(h[k]);
                    const uint64_t f2 = f32x2_pack(f.x, f.y);
                    acc2 = f32x2_fma(f2, f2, acc2);
                    if (fold) {
                        // Folded scale: the query row holds rn(c x^).
                        hs[k] = PT::from_f2(cf * f.x, cf * f.y);
                        const float2 g = PT::to_f2(hs[k]);
                        const uint64_t g2 = f32x2_pack(g.x, g.y);
                        accu2 = f32x2_fma(g2, g2, accu2);
                    }
                }
                u = *reinterpret_cast<const uint4*>(h);
                us = fold ? *reinterpret_cast<const uint4*>(hs) : u;
            }
            if (out_q) *reinterpret_cast<uint4*>(out_q + 8 * v) = fold ? us : u;
            if (out_k) *reinterpret_cast<uint4*>(out_k + 8 * v) = u;
        }
        float lo, hi;
        f32x2_unpack(acc2, lo, hi);
        acc = lo + hi;
        f32x2_unpack(accu2, lo, hi);
        accu = lo + hi;
    }
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xffffffffu, acc, o, G);
        if (fold) accu += __shfl_xor_sync(0xffffffffu, accu, o, G);
    }
    const float nrm = valid ? -half_c * acc : pad_value;
    if (!in_pad || vi != 0) return nrm;
    if (!AUG) {
        for (int c = D; c < Dp; c += 8)
            *reinterpret_cast<uint4*>(out_q + c) = make_uint4(0u, 0u, 0u, 0u);
        return nrm;
    }
    // Norm terms: a (or b) = -||x^||^2 / 2 = F t_0 + t_1 + ... (rounded
    // remainders, nt <= 3 of them), partners F, 1, 1 on the other side.
    // Built in registers: element e of the query tail is the partner
    // (F, 1, 1) for e < nt and t_(e - nt) for nt <= e < 2 nt; the key tail
    // the other way round; zeros after that.
    unsigned short t0 = 0, t1 = 0, t2 = 0, k0 = 0, k1 = 0, k2 = 0;
    auto split = [&](float r, unsigned short& z0, unsigned short& z1, unsigned short& z2) {
        const T a0 = from_f<T>(r * (1.f / F));   // F is a power of two: exact
        r -= F * to_f(a0);
        const T a1 = from_f<T>(r);
        r -= to_f(a1);
        const T a2 = from_f<T>(r);
        z0 = to_bits(a0);
        z1 = to_bits(a1);
        z2 = nt > 2 ? to_bits(a2) : 0;
    };
    if (valid) {
        if (fold) {
            // Folded: a = -||u||^2 / (2c) from the rounded scaled row, and
            // b = -c ||k^||^2 / 2 + log2(|v| 2^-16) (see log_weight).
            split(-0.5f * accu / cf, t0, t1, t2);
            split(-0.5f * cf * acc + log_weight(vw), k0, k1, k2);
        } else {
            split(-0.5f * acc, t0, t1, t2);
            k0 = t0; k1 = t1; k2 = t2;
        }
    }
    const unsigned short oneF = valid ? to_bits(from_f<T>(F)) : 0;
    const unsigned short one1 = valid ? to_bits(from_f<T>(1.f)) : 0;
    const unsigned short pad_b = valid ? k0 : to_bits(from_f<T>(-30000.f / F));
    auto term = [&](int i) { return i == 0 ? pad_b : i == 1 ? k1 : k2; };
    auto qterm = [&](int i) { return i == 0 ? t0 : i == 1 ? t1 : t2; };
    auto partner = [&](int i) { return i == 0 ? oneF : one1; };
    auto tail_q = [&](int e) -> unsigned {
        return e < nt ? partner(e) : e < 2 * nt ? qterm(e - nt) : 0u;
    };
    auto tail_k = [&](int e) -> unsigned {
        return e < nt ? term(e) : e < 2 * nt ? partner(e - nt) : 0u;
    };
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = D + 8 * h;
        if (c >= Dp) break;
        uint32_t wq[4], wk[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            wq[e] = tail_q(8 * h + 2 * e) | (tail_q(8 * h + 2 * e + 1) << 16);
            wk[e] = tail_k(8 * h + 2 * e) | (tail_k(8 * h + 2 * e + 1) << 16);
        }
        if (out_q) *reinterpret_cast<uint4*>(out_q + c) = make_uint4(wq[0], wq[1], wq[2], wq[3]);
        if (out_k) *reinterpret_cast<uint4*>(out_k + c) = make_uint4(wk[0], wk[1], wk[2], wk[3]);
    }
    for (int c = D + 16; c < Dp; c += 8) {
        if (out_q) *reinterpret_cast<uint4*>(out_q + c) = make_uint4(0u, 0u, 0u, 0u);
        if (out_k) *reinterpret_cast<uint4*>(out_k + c) = make_uint4(0u, 0u, 0u, 0u);
    }
    return nrm;
}

// One array's operand rows: x (batch x rows x D) into out_q / out_k
// (batch x rows_pad x Dp; either may be null, AUG only) and, for the plain
// layout, the norm terms nrm (batch x rows_pad).
struct OperandJob {
    const void* x;
    int64_t rows, rows_pad;
    void* out_q;
    void* out_k;
    float* nrm;
    const void* vw;      // fp16 values of the rows written to out_k (folded magnitudes), or null
};

// Vector path of the operand preparation (D a multiple of 8): G lanes per
// row (G = 1 up to D = 64, 2 up to 128, 4 up to 256), each lane converting
// up to eight 16-byte vectors of its row, all loaded before any is
// converted; so every lane of a warp does its own row's work (no lanes idle
// during the norm split) and has up to 128 bytes of loads in flight.  The
// block's output rows are staged in shared memory (a row stride of an odd
// number of 16-byte vectors, so that the lanes' row stores do not share
// banks) and then written as one contiguous run of 16-byte vectors, one per
// thread and step, instead of one row per lane.
// Blocks [0, blocks0) of grid row b convert rows of job j0 of problem b,
// the rest those of j1 (the keys, when they are not the queries), so that
// both arrays of every problem take one launch; a block never straddles
// two problems.  The problem's mean is staged once per block in shared
// memory as packed pairs of the input format.
template <typename T, bool AUG, int G>
__global__ void __launch_bounds__(kOperandVecThreads)
operand_vec_kernel(const OperandJob j0, const OperandJob j1, unsigned blocks0, int D, int Dp,
                   int nt, float F, const float* __restrict__ mu, float half_c, float pad_value,
                   float cf, unsigned op_blocks, float* __restrict__ vf_rec, int64_t vf_tiles) {
    using PT = Pair<T>;
    pdl_trigger();
    pdl_wait();
    if (blockIdx.x >= op_blocks) {
        // Folded values: the per-problem flag of the sign records (written
        // by an earlier launch of the call), one extra block per problem.
        write_vf_flag(vf_rec, vf_tiles, static_cast<int>(gridDim.y), blockIdx.y);
        return;
    }
    constexpr int SLOTS = kOperandVecThreads / G;   // rows of a block
    __shared__ uint4 smean[kOperandMaxCols / 8];
    extern __shared__ uint4 staged[];                // SLOTS rows of each output
    const int b = blockIdx.y;                        // problem of the batch
    const bool second = blockIdx.x >= blocks0;
    const OperandJob j = second ? j1 : j0;
    const int blk = static_cast<int>(second ? blockIdx.x - blocks0 : blockIdx.x);
    const int vi = threadIdx.x % G;                  // first vector of this lane
    const int slot = threadIdx.x / G;
    const int V = D / 8;
    const int rows_pad = static_cast<int>(j.rows_pad);
    const int rows = static_cast<int>(j.rows);
    const int i = blk * SLOTS + slot;                // row of problem b
    const T* xr = static_cast<const T*>(j.x) + (static_cast<int64_t>(b) * rows + i) * D;
    uint4 in[kOperandVecs];
#pragma unroll
    for (int e = 0; e < kOperandVecs; ++e) {
        const int v = vi + G * e;
        in[e] = (i < rows && v < V) ? *reinterpret_cast<const uint4*>(xr + 8 * v)
                                    : make_uint4(0u, 0u, 0u, 0u);
    }
    const float* mb = mu ? mu + static_cast<int64_t>(b) * D : nullptr;
    typename PT::P* sm = reinterpret_cast<typename PT::P*>(smean);
    for (int c = threadIdx.x; c < D / 2; c += kOperandVecThreads)
        sm[c] = mb ? PT::from_f2(mb[2 * c], mb[2 * c + 1]) : PT::from_f2(0.f, 0.f);
    __syncthreads();
    const bool wq = AUG ? j.out_q != nullptr : true;
    const bool wk = AUG && j.out_k != nullptr;
    const bool in_pad = i < rows_pad;
    const int64_t row = static_cast<int64_t>(b) * rows_pad + i;   // batch-stacked output row
    const __half* vw = (wk && j.vw && i < rows)
                           ? static_cast<const __half*>(j.vw) + static_cast<int64_t>(b) * rows + i
                           : nullptr;
    const int nv = Dp / 8;                           // 16-byte vectors per output row
    const int sv = nv | 1;                           // staged row stride (odd)
    uint4* stage_q = staged;
    uint4* stage_k = staged + (wq ? SLOTS * sv : 0);
    const float n = operand_row<T, AUG, G>(
        in, smean, vi, in_pad, i < rows, D, Dp, nt, F, half_c, pad_value,
        wq ? reinterpret_cast<T*>(stage_q + slot * sv) : nullptr,
        wk ? reinterpret_cast<T*>(stage_k + slot * sv) : nullptr, cf, vw);
    if (!AUG && in_pad && vi == 0) j.nrm[row] = n;
    __syncthreads();
    // The block's rows [i0, i0 + nrows) are consecutive output rows.
    const int i0 = blk * SLOTS;
    const int nrows = min(SLOTS, rows_pad - i0);
    const int total = nrows * nv;
    const int64_t base = (static_cast<int64_t>(b) * rows_pad + i0) * Dp;
    uint4* gq = wq ? reinterpret_cast<uint4*>(static_cast<T*>(j.out_q) + base) : nullptr;
    uint4* gk = wk ? reinterpret_cast<uint4*>(static_cast<T*>(j.out_k) + base) : nullptr;
    for (int u = threadIdx.x; u < total; u += kOperandVecThreads) {
        const int r = u / nv;
        const int s = r * sv + (u - r * nv);
        if (wq) gq[u] = stage_q[s];
        if (wk) gk[u] = stage_k[s];
    }
}

template <typename T, bool AUG>
cudaError_t operand_typed(const OperandJob& j0, const OperandJob* j1, int D, int Dp, int nt,
                          float F, const float* mu, float half_c, float pad_value, cudaStream_t s,
                          int batch, float cf, float* vf_rec, int64_t vf_tiles, bool* flags_done) {
    const OperandJob none = {nullptr, 0, 0, nullptr, nullptr, nullptr, nullptr};
    for (const OperandJob* j : {&j0, j1}) {
        if (j && (j->rows_pad % kRowsPerBlock != 0)) return cudaErrorInvalidValue;
    }
    if (Dp % 16 != 0 || Dp > kOperandMaxCols || (AUG && 2 * Dp > kOperandMaxCols))
        return cudaErrorInvalidValue;
    // The vector path indexes rows with 32-bit integers.
    const int64_t most_rows = std::max(j0.rows_pad, j1 ? j1->rows_pad : int64_t(0)) * batch;
    if (D % 8 == 0 && D >= 8 && (!AUG || Dp - D >= 2 * nt) && most_rows < (int64_t(1) << 30)) {
        // Vector path: G lanes per row (up to kOperandVecs vectors each),
        // both arrays in one launch.
        const int V = D / 8;
        const int G = V <= kOperandVecs ? 1 : V <= 2 * kOperandVecs ? 2 : 4;
        const int64_t per_block = kOperandVecThreads / G;
        const int64_t b0 = (j0.rows_pad + per_block - 1) / per_block;
        const int64_t b1 = j1 ? (j1->rows_pad + per_block - 1) / per_block : 0;
        if (b0 + b1 == 0 || batch == 0) return cudaSuccess;
        const unsigned op_blocks = static_cast<unsigned>(b0 + b1);
        // Staged output rows: one or two outputs per job (AUG with q = k
        // writes both layouts of the same rows).
        auto nout = [](const OperandJob* j) {
            return j ? (AUG ? (j->out_q ? 1 : 0) + (j->out_k ? 1 : 0) : 1) : 0;
        };
        const size_t smem = static_cast<size_t>(std::max(nout(&j0), nout(j1))) * per_block *
                            ((Dp / 8) | 1) * 16;
        auto go = [&](auto kern) {
            cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            launch_kernel(kern, dim3(op_blocks + (vf_rec ? 1u : 0u), static_cast<unsigned>(batch)),
                          kOperandVecThreads, smem, s, j0, j1 ? *j1 : none, static_cast<unsigned>(b0),
                          D, Dp, nt, F, mu, half_c, pad_value, cf, op_blocks, vf_rec, vf_tiles);
            return cudaSuccess;
        };
        if (flags_done) *flags_done = vf_rec != nullptr;
        cudaError_t e;
        switch (G) {
            case 1: e = go(operand_vec_kernel<T, AUG, 1>); break;
            case 2: e = go(operand_vec_kernel<T, AUG, 2>); break;
            default: e = go(operand_vec_kernel<T, AUG, 4>); break;
        }
        if (e != cudaSuccess) return e;
        note_launches(1);
        return cudaGetLastError();
    }
    for (const OperandJob* j : {&j0, j1}) {
        if (!j) continue;
        const int64_t blocks = j->rows_pad / kRowsPerBlock;
        if (blocks == 0) continue;
        const int nout = AUG ? (j->out_q ? 1 : 0) + (j->out_k ? 1 : 0) : 1;
        const size_t smem = static_cast<size_t>(nout) * kRowsPerBlock * Dp * sizeof(T) +
                            ((static_cast<size_t>(kRowsPerBlock) * D * sizeof(T) + 15) & ~size_t(15)) +
                            static_cast<size_t>(D) * sizeof(float);
        launch_kernel(operand_kernel<T, AUG>, dim3(static_cast<unsigned>(blocks), batch),
                      kOperandThreads, smem, s, static_cast<const T*>(j->x), j->rows, j->rows_pad,
                      D, Dp, nt, F, mu, half_c, pad_value, static_cast<T*>(j->out_q),
                      static_cast<T*>(j->out_k), j->nrm, static_cast<const __half*>(j->vw), cf);
        note_launches(1);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// ---------------------------------------------------------------- values
// Value of channel ch of key n.  Forward (Eq. 1): w[n, ch] (Cw = channels).
// Gradients (Sec. 3, and the vector-Jacobian product of Eq. 1): channel
// ch = c (D + 1) + d holds w[n, c] (x[n, d] - mu_d) for d < D and w[n, c]
// for d = D, one group of D + 1 channels per weight channel c < Cw; a null
// w means unit weights (the weighted vector-Jacobian pass, whose weights
// enter through the kernel values instead).
template <typename T, typename W, bool GRAD>
__device__ __forceinline__ float value_at(const W* __restrict__ w, const T* __restrict__ x,
                                          const float* __restrict__ mu, int64_t n, int ch, int D,
                                          int Cw) {
    if (GRAD) {
        const int c = ch / (D + 1);
        const int d = ch - c * (D + 1);
        const float wn = w ? to_f(w[n * Cw + c]) : 1.f;
        if (d < D) return wn * (to_f(x[n * D + d]) - (mu ? mu[d] : 0.f));
        return wn;
    }
    return to_f(w[n * Cw + ch]);
}

// Per-channel max |value| over the keys for channels ch0 .. ch0 + Cc - 1;
// block (32, 8) as in the mean.
template <typename T, typename W, bool GRAD>
__global__ void value_max_kernel(const W* __restrict__ w, const T* __restrict__ x,
                                 const float* __restrict__ mu, int64_t N, int D, int Cw, int ch0,
                                 int Cc, int64_t rows_per_block, unsigned* __restrict__ vmax_bits) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[8][33];
    const int64_t r0 = static_cast<int64_t>(blockIdx.x) * rows_per_block;
    const int64_t r1 = min(r0 + rows_per_block, N);
    for (int c0 = 0; c0 < Cc; c0 += 32) {
        const int c = c0 + threadIdx.x;
        float mx = 0.f;
        if (c < Cc)
            for (int64_t n = r0 + threadIdx.y; n < r1; n += 8)
                mx = fmaxf(mx, fabsf(value_at<T, W, GRAD>(w, x, mu, n, ch0 + c, D, Cw)));
        red[threadIdx.y][threadIdx.x] = mx;
        __syncthreads();
        if (threadIdx.y == 0 && c < Cc) {
            float m = 0.f;
#pragma unroll
            for (int y = 0; y < 8; ++y) m = fmaxf(m, red[y][threadIdx.x]);
            // Non-negative floats order like their bit patterns.
            atomicMax(&vmax_bits[c], __float_as_uint(m));
        }
        __syncthreads();
    }
}

// Power-of-two channel scale 2^e with e = -floor(log2 max|value|), so that
// the scaled channel's largest magnitude lies in [1, 2); e is clamped to
// [-126, 126] and is 0 for an all-zero channel.  Exact bit construction.
__device__ __forceinline__ int channel_exponent(unsigned max_bits) {
    if (max_bits == 0u) return 0;
    int E = static_cast<int>((max_bits >> 23) & 0xffu);
    if (E == 0) E = 1;             // subnormal maximum: clamp
    if (E == 0xff) return 0;       // inf / nan: leave unscaled
    int e = 127 - E;               // -floor(log2 max)
    return max(-126, min(126, e));
}

__device__ __forceinline__ float pow2f(int e) { return __uint_as_float(static_cast<unsigned>(e + 127) << 23); }

// Transposed, scaled fp16 value operand vt[j][n] = value of channel ch0 + j
// (Cp x Npad, zero padded), through a 32 x 32 shared-memory tile; block
// (32, 8).
template <typename T, typename W, bool GRAD>
__global__ void value_prep_kernel(const W* __restrict__ w, const T* __restrict__ x,
                                  const float* __restrict__ mu, int64_t N, int64_t Npad, int D,
                                  int Cw, int ch0, int Cc, int Cp,
                                  const unsigned* __restrict__ vmax_bits, __half* __restrict__ vt,
                                  float* __restrict__ inv_scale) {
    pdl_trigger();
    pdl_wait();
    // A block transposes 64 keys x 32 channels; each thread stores two
    // adjacent keys of one channel as a half2 (Npad is a multiple of 128).
    __shared__ float tile[64][33];
    const int64_t n0 = static_cast<int64_t>(blockIdx.x) * 64;
    const int c0 = blockIdx.y * 32;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t n = n0 + threadIdx.y + 8 * i;
        const int c = c0 + threadIdx.x;
        float val = 0.f;
        if (n < N && c < Cc) val = value_at<T, W, GRAD>(w, x, mu, n, ch0 + c, D, Cw);
        tile[threadIdx.y + 8 * i][threadIdx.x] = val;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int c = c0 + threadIdx.y + 8 * i;
        const int64_t n = n0 + 2 * threadIdx.x;
        if (c < Cp && n < Npad) {
            const float sc = c < Cc ? pow2f(channel_exponent(vmax_bits[c])) : 0.f;
            const int cl = threadIdx.y + 8 * i;
            *reinterpret_cast<__half2*>(vt + static_cast<int64_t>(c) * Npad + n) =
                __floats2half2_rn(tile[2 * threadIdx.x][cl] * sc, tile[2 * threadIdx.x + 1][cl] * sc);
        }
    }
    if (blockIdx.x == 0 && threadIdx.y == 0) {
        const int c = c0 + threadIdx.x;
        if (c < Cp) inv_scale[c] = c < Cc ? pow2f(-channel_exponent(vmax_bits[c])) : 0.f;
    }
}

// ---------------------------------------------------------------- key records
// One thread per key pair t: B_2t, B_2t+1 (only when B is given), then the
// values of both keys channel by channel, in fp32 (zero for padded keys).
template <typename T>
__global__ void key_record_kernel(const T* __restrict__ v, const float* __restrict__ B, int64_t N,
                                  int64_t pairs, int C, float* __restrict__ rec) {
    pdl_trigger();
    pdl_wait();
    const int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (t >= pairs) return;
    const int64_t n0 = 2 * t, n1 = 2 * t + 1;
    const int head = B ? 2 : 0;
    // Problem blockIdx.y of a batch (2 pairs keys per problem).
    v += static_cast<int64_t>(blockIdx.y) * N * C;
    if (B) B += static_cast<int64_t>(blockIdx.y) * 2 * pairs;
    rec += static_cast<int64_t>(blockIdx.y) * pairs * (head + 2 * C);
    float* out = rec + t * (head + 2 * C);
    if (B) {
        out[0] = B[n0];
        out[1] = B[n1];
    }
    for (int c = 0; c < C; ++c) {
        out[head + 2 * c] = n0 < N ? to_f(v[n0 * C + c]) : 0.f;
        out[head + 1 + 2 * c] = n1 < N ? to_f(v[n1 * C + c]) : 0.f;
    }
}

// ---------------------------------------------------------------- pair weights
// Factors of the pair weights w_mn = sum_c r[m, c] k[n, c] of the weighted
// vector-Jacobian pass (row factors r: the rows of the Gauss sum, column
// factors k: its keys; C <= WT channels, zero padded to WT).  Blocks
// [0, rblocks) write the row factors row-major in float32,
// rowf[m WT + c] (Rpad rows, zero past R); the other blocks write the
// column factors per key tile of BN keys, channel-major inside the tile,
// colT[(n / BN) WT BN + c BN + n % BN] (Npad keys, zero past Ncol), so that
// one bulk copy brings a key tile's factors into shared memory.  wmax[c]
// and wmax[WT + c] receive the largest |r[., c]| and |k[., c]| (float bits,
// atomicMax over blocks; the caller zeroes them).  One thread per (row or
// key, channel), 256 threads per block.
constexpr int kWeightThreads = 256;

template <typename TR, typename TC>
__global__ void __launch_bounds__(kWeightThreads)
weight_prep_kernel(const TR* __restrict__ rsrc, int64_t R, int64_t Rpad,
                   const TC* __restrict__ csrc, int64_t Ncol, int64_t Npad, int C, int WT, int BN,
                   unsigned rblocks, float* __restrict__ rowf, float* __restrict__ colT,
                   unsigned* __restrict__ wmax) {
    pdl_trigger();
    pdl_wait();
    __shared__ float red[kWeightThreads];
    const bool on_rows = blockIdx.x < rblocks;
    const int64_t blk = on_rows ? blockIdx.x : blockIdx.x - rblocks;
    const int64_t idx = blk * kWeightThreads + threadIdx.x;
    const int64_t i = idx / WT;                 // row or key
    const int c = static_cast<int>(idx - i * WT);
    float val = 0.f;
    if (on_rows) {
        if (i < Rpad) {
            if (i < R && c < C) val = to_f(rsrc[i * C + c]);
            rowf[idx] = val;
        }
    } else if (i < Npad) {
        if (i < Ncol && c < C) val = to_f(csrc[i * C + c]);
        colT[(i / BN) * WT * BN + static_cast<int64_t>(c) * BN + i % BN] = val;
    }
    // Channel c of this block: threads t with t % WT == c (WT divides 256).
    red[threadIdx.x] = fabsf(val);
    __syncthreads();
    if (threadIdx.x < WT) {
        float m = 0.f;
        for (int t = threadIdx.x; t < kWeightThreads; t += WT) m = fmaxf(m, red[t]);
        // Non-negative floats order like their bit patterns.
        atomicMax(&wmax[(on_rows ? 0 : WT) + threadIdx.x], __float_as_uint(m));
    }
}

// ---------------------------------------------------------------- finalise
// Forward: out[m, c] = inv_scale[c] sum_s part[s][m][c] (splits added in
// order).  part: splits blocks of split_stride_rows rows x part_ld floats.
__global__ void finalize_kernel(const float* __restrict__ part, int splits,
                                int64_t split_stride_rows, int64_t M, int Cv, int part_ld,
                                const float* __restrict__ inv_scale, float* __restrict__ out,
                                int64_t main_rows) {
    pdl_trigger();
    pdl_wait();
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= M * Cv) return;
    const int64_t m = div_nonneg(idx, Cv);
    const int c = static_cast<int>(idx - m * Cv);
    float acc = 0.f;
    const int ns = m < main_rows ? 1 : splits;
    for (int s = 0; s < ns; ++s)
        acc += part[(static_cast<int64_t>(s) * split_stride_rows + m) * part_ld + c];
    out[idx] = acc * (inv_scale ? inv_scale[c] : 1.f);
}

// Gradient contraction for the channels ch0 .. ch0 + Cc - 1 of one launch
// (channel ch = c (D + 1) + d, as in value_at).  With S_j the sum over
// splits of partial channel j (times inv_scale[j] when given):
//   out[m, d] (+)= tau sum_c u[m, c] (S_{c,d} - x^_{m,d} S_{c,D})
//   s_out[m, c]   = S_{c,D}
// where x^ = x - mu is the row's centred point.  DIRECT: the partials
// already hold sum Phi w (k - x) (the fp32 kernel's difference form), so the
// x^ S_{c,D} term is left out.  Terms whose channel lies outside this launch
// are added by the launch that holds it (accumulate = 1 adds to out).  u
// null means u = 1; out may be null when only s_out is wanted.  One thread
// per (m, d) for d < max(D, 1).
template <bool DIRECT, typename T, typename U>
__global__ void finalize_points_kernel(const float* __restrict__ part, int splits,
                                       int64_t split_stride_rows, int64_t M, int part_ld,
                                       const float* __restrict__ inv_scale,
                                       const T* __restrict__ x, const float* __restrict__ mu,
                                       float tau, int D, int Cw, int ch0, int Cc,
                                       const U* __restrict__ u, int accumulate,
                                       float* __restrict__ out, float* __restrict__ s_out,
                                       int64_t main_rows) {
    pdl_trigger();
    pdl_wait();
    const int width = D > 0 ? D : 1;
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= M * width) return;
    const int64_t m = div_nonneg(idx, width);
    const int d = static_cast<int>(idx - m * width);
    const int ns = m < main_rows ? 1 : splits;
    auto S = [&](int j) {
        float acc = 0.f;
        // Unrolled so that the loads of several splits are in flight
        // together (the sum keeps the split order): 71 -> 58 us on the
        // 131072-point gradient with four splits.
#pragma unroll 4
        for (int s = 0; s < ns; ++s)
            acc += part[(static_cast<int64_t>(s) * split_stride_rows + m) * part_ld + j];
        return inv_scale ? acc * inv_scale[j] : acc;
    };
    const int G = D + 1;
    const int c_lo = ch0 / G, c_hi = (ch0 + Cc - 1) / G;
    const float xd = (DIRECT || d >= D) ? 0.f : to_f(x[m * D + d]) - (mu ? mu[d] : 0.f);
    float acc = 0.f;
    for (int c = c_lo; c <= c_hi; ++c) {
        const int jd = c * G + d - ch0;
        const int js = c * G + D - ch0;
        const bool has_d = d < D && jd >= 0 && jd < Cc;
        const bool has_s = js >= 0 && js < Cc;
        if (!has_d && !(has_s && (d == 0 || !DIRECT))) continue;
        const float ss = has_s ? S(js) : 0.f;
        if (d == 0 && has_s && s_out) s_out[m * Cw + c] = ss;
        if (d >= D) continue;
        float t = has_d ? S(jd) : 0.f;
        if (!DIRECT && has_s) t -= xd * ss;
        acc += (u ? to_f(u[m * Cw + c]) : 1.f) * t;
    }
    if (out && d < D) out[m * D + d] = (accumulate ? out[m * D + d] : 0.f) + tau * acc;
}

template <typename T, typename W, bool GRAD>
cudaError_t value_prep_typed(const void* w, const void* x, const float* mu, int64_t N,
                             int64_t Npad, int D, int Cw, int ch0, int Cc, int Cp,
                             unsigned* vmax_bits, void* vt, float* inv_scale, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(vmax_bits, 0, sizeof(unsigned) * Cp, s);
    if (e != cudaSuccess) return e;
    pdl_reset();   // the next kernel follows a memset
    // 64 rows per block: several blocks per SM even for N of a few 10^4.
    const int64_t rows_per_block = 64;
    const int64_t blocks = N > 0 ? (N + rows_per_block - 1) / rows_per_block : 0;
    if (blocks > 0) {
        launch_kernel(value_max_kernel<T, W, GRAD>, static_cast<unsigned>(blocks), dim3(32, 8), 0, s, 
            static_cast<const W*>(w), static_cast<const T*>(x), mu, N, D, Cw, ch0, Cc,
            rows_per_block, vmax_bits);
        note_launches(1);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    dim3 grid(static_cast<unsigned>((Npad + 63) / 64), static_cast<unsigned>((Cp + 31) / 32));
    launch_kernel(value_prep_kernel<T, W, GRAD>, grid, dim3(32, 8), 0, s, 
        static_cast<const W*>(w), static_cast<const T*>(x), mu, N, Npad, D, Cw, ch0, Cc, Cp,
        vmax_bits, static_cast<__half*>(vt), inv_scale);
    note_launches(1);
    return cudaGetLastError();
}

template <bool DIRECT, typename T, typename U>
cudaError_t finalize_points_typed(const float* part, int splits, int64_t stride_rows, int64_t M,
                                  int part_ld, const float* inv_scale, const void* x,
                                  const float* mu, float tau, int D, int Cw, int ch0, int Cc,
                                  const void* u, int accumulate, float* out, float* s_out,
                                  cudaStream_t s, int64_t main_rows) {
    const int64_t total = M * (D > 0 ? D : 1);
    if (total == 0) return cudaSuccess;
    const int threads = 256;
    const int64_t blocks = (total + threads - 1) / threads;
    launch_kernel(finalize_points_kernel<DIRECT, T, U>, static_cast<unsigned>(blocks), threads, 0, s, 
        part, splits, stride_rows, M, part_ld, inv_scale, static_cast<const T*>(x), mu, tau, D,
        Cw, ch0, Cc, static_cast<const U*>(u), accumulate, out, s_out, main_rows);
    note_launches(1);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_mean(InType t, const void* q, const void* k, int64_t M, int64_t N, int D,
                        int blocks, float* partial, float* mu, cudaStream_t s, int batch,
                        const RecordArgs* rec, bool* rec_done) {
    if (rec_done) *rec_done = false;
    // q and k the same points: the mean of [q; q] is the mean of q.
    if (q == k && M == N) N = 0;
    const int64_t total = M + N;
    int G = 0;
    const bool vec = t != InType::F32 && D >= 8 && D <= 2048 && (D & (D - 1)) == 0 &&
                     2048 % D == 0 && blocks >= 4;
    if (vec) {
        // At most `blocks` blocks over both arrays (the partial buffer holds
        // `blocks` rows of 2 D floats).
        const int64_t rpb = std::max<int64_t>(1, (total + blocks - 3) / (blocks - 2));
        const int Gq = static_cast<int>((M + rpb - 1) / rpb);
        const int Gk = static_cast<int>((N + rpb - 1) / rpb);
        G = Gq + Gk;
        // Key records (see RecordJob) in blocks G .. G + rblocks - 1.
        const int64_t pairs = rec ? rec->Npad / 2 : 0;
        // One thread per key pair, or per key for sign records.
        const int64_t rthreads = rec && rec->signs ? 2 * pairs : pairs;
        const int rblocks = static_cast<int>((rthreads + kMeanVecThreads - 1) / kMeanVecThreads);
        auto go = [&](auto tag, auto vtag) {
            using T = decltype(tag);
            using TV = decltype(vtag);
            const RecordJob<TV> rj = {rec ? static_cast<const TV*>(rec->v) : nullptr, rec ? rec->N : 0,
                                      pairs, rec ? rec->C : 0, rec ? rec->out : nullptr,
                                      rec && rec->signs};
            launch_kernel(mean_partial_vec_kernel<T, TV>, dim3(G + rblocks, batch), kMeanVecThreads, 0,
                          s, static_cast<const T*>(q), static_cast<const T*>(k), M, N, D, rpb, Gq, G,
                          partial, rj);
        };
        const bool vf = rec && rec->v_f32;
        if (t == InType::F16) {
            if (vf) go(__half(), float()); else go(__half(), __half());
        } else {
            if (vf) go(__nv_bfloat16(), float()); else go(__nv_bfloat16(), __nv_bfloat16());
        }
        if (rec_done) *rec_done = rec != nullptr;
        note_launches(1);
    } else {
        const int64_t rpb = (total + blocks - 1) / blocks;
        G = static_cast<int>((total + rpb - 1) / rpb);
        switch (t) {
            case InType::F16:
                launch_kernel(mean_partial_kernel<__half>, dim3(G, batch), dim3(32, 8), 0, s, 
                    static_cast<const __half*>(q), static_cast<const __half*>(k), M, N, D, rpb,
                    partial);
                break;
            case InType::BF16:
                launch_kernel(mean_partial_kernel<__nv_bfloat16>, dim3(G, batch), dim3(32, 8), 0, s, 
                    static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(k), M, N,
                    D, rpb, partial);
                break;
            default:
                launch_kernel(mean_partial_kernel<float>, dim3(G, batch), dim3(32, 8), 0, s, 
                    static_cast<const float*>(q), static_cast<const float*>(k), M, N, D, rpb,
                    partial);
        }
        note_launches(1);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int mant_bits = t == InType::F16 ? 10 : t == InType::BF16 ? 7 : 23;
    const int min_exp = t == InType::F16 ? -24 : t == InType::BF16 ? -133 : -149;
    if (G > kMeanFinalThreadMax) {
        launch_kernel(mean_final_block_kernel, dim3(D, batch), kMeanFinalThreads, 0, s, partial,
                      G, D, static_cast<float>(total), mant_bits, min_exp, mu);
    } else {
        const int64_t items = static_cast<int64_t>(batch) * D;
        launch_kernel(mean_final_kernel,
                      dim3(static_cast<unsigned>((items + kMeanFinalThreads - 1) / kMeanFinalThreads)),
                      kMeanFinalThreads, 0, s, partial, G, D, items, static_cast<float>(total),
                      mant_bits, min_exp, mu);
    }
    note_launches(1);
    return cudaGetLastError();
}

namespace {

// Sec. 3: MMD^2 = v^T s for s = K v (q = k).  Block g of problem b folds
// the products v_n s_n of its chunk of kMmdChunk points (n = chunk start + t,
// + 256, ...) in float64, a fixed tree adds the threads, and
// mmd2_final_kernel adds the chunks of each problem in order
// (deterministic).
constexpr int64_t kMmdChunk = 4096;

template <typename T>
__global__ void __launch_bounds__(256)
mmd2_reduce_kernel(const float* __restrict__ s, const T* __restrict__ v, int64_t N,
                   double* __restrict__ partial) {
    pdl_trigger();
    pdl_wait();
    __shared__ double red[256];
    const int t = threadIdx.x;
    const int64_t b = blockIdx.y;
    const int64_t n0 = static_cast<int64_t>(blockIdx.x) * kMmdChunk;
    const int64_t n1 = min(N, n0 + kMmdChunk);
    double acc = 0.0;
    for (int64_t n = n0 + t; n < n1; n += 256)
        acc += static_cast<double>(to_f(v[b * N + n])) * static_cast<double>(s[b * N + n]);
    red[t] = acc;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if (t < w) red[t] += red[t + w];
        __syncthreads();
    }
    if (t == 0) partial[b * gridDim.x + blockIdx.x] = red[0];
}

__global__ void mmd2_final_kernel(const double* __restrict__ partial, int chunks, int64_t B,
                                  float* __restrict__ out) {
    pdl_trigger();
    pdl_wait();
    const int64_t b = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (b >= B) return;
    double acc = 0.0;
    for (int g = 0; g < chunks; ++g) acc += partial[b * chunks + g];
    out[b] = static_cast<float>(acc);
}

}  // namespace

size_t mmd2_partial_bytes(int64_t B, int64_t N) {
    const int64_t chunks = std::max<int64_t>(1, (N + kMmdChunk - 1) / kMmdChunk);
    return static_cast<size_t>(B * chunks) * sizeof(double);
}

cudaError_t launch_mmd2_reduce(InType t, const float* s, const void* v, int64_t B, int64_t N,
                               double* partial, float* out, cudaStream_t st) {
    if (B == 0) return cudaSuccess;
    const int64_t chunks = std::max<int64_t>(1, (N + kMmdChunk - 1) / kMmdChunk);
    const dim3 grid(static_cast<unsigned>(chunks), static_cast<unsigned>(B));
    switch (t) {
        case InType::F16:
            launch_kernel(mmd2_reduce_kernel<__half>, grid, 256, 0, st, s, static_cast<const __half*>(v), N,
                                                             partial);
            break;
        case InType::BF16:
            launch_kernel(mmd2_reduce_kernel<__nv_bfloat16>, grid, 256, 0, st, 
                s, static_cast<const __nv_bfloat16*>(v), N, partial);
            break;
        default:
            launch_kernel(mmd2_reduce_kernel<float>, grid, 256, 0, st, s, static_cast<const float*>(v), N,
                                                            partial);
    }
    note_launches(1);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    launch_kernel(mmd2_final_kernel, static_cast<unsigned>((B + 127) / 128), 128, 0, st, 
        partial, static_cast<int>(chunks), B, out);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_finalize_slots(const float* part, int64_t Mpad, int64_t M, int C,
                                  int rows_per_unit, int64_t key_tiles, int64_t unit_len,
                                  float* out, cudaStream_t s, int batch, int fixed_slots,
                                  int64_t tri_key_tiles) {
    const int64_t total = static_cast<int64_t>(batch) * M * C;
    if (total == 0) return cudaSuccess;
    const int threads = 256;
    launch_kernel(finalize_slots_kernel, static_cast<unsigned>((total + threads - 1) / threads), threads, 0, s, 
        part, Mpad, M, C, rows_per_unit, key_tiles, unit_len, static_cast<int64_t>(batch),
        fixed_slots, tri_key_tiles, out);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_operands(InType t, bool aug, const void* q, int64_t M, int64_t Mpad,
                            void* qh, void* qh_as_key, float* nrm_q, bool with_k, const void* k,
                            int64_t N, int64_t Npad, void* kh, float* nrm_k, int D, int Dp,
                            const float* mu, float half_c, float pad_value, cudaStream_t s,
                            int batch, const void* vw, float cf, float* vf_rec, bool* flags_done) {
    if (flags_done) *flags_done = false;
    const int64_t vf_tiles = Npad / kRecTile;
    OperandJob jq, jk;
    if (aug) {
        // vw: folded value magnitudes on the key rows (the q job writes the
        // key rows too when q is k).
        jq = {q, M, Mpad, qh, qh_as_key, nullptr, qh_as_key ? vw : nullptr};
        jk = {k, N, Npad, nullptr, kh, nullptr, vw};
    } else {
        jq = {q, M, Mpad, qh, nullptr, nrm_q, nullptr};
        jk = {k, N, Npad, kh, nullptr, nrm_k, nullptr};
    }
    if (!aug) cf = 0.f;
    // (k itself may be null: an empty array when D = 0.)
    const OperandJob* j1 = with_k ? &jk : nullptr;
    const int nt = aug ? aug_norm_terms(t) : 0;
    if (t == InType::BF16) {
        return aug ? operand_typed<__nv_bfloat16, true>(jq, j1, D, Dp, nt, 1.f, mu, 0.f, 0.f, s, batch,
                                                        cf, vf_rec, vf_tiles, flags_done)
                   : operand_typed<__nv_bfloat16, false>(jq, j1, D, Dp, 0, 1.f, mu, half_c,
                                                         pad_value, s, batch, cf, vf_rec,
                                                         vf_tiles, flags_done);
    }
    return aug ? operand_typed<__half, true>(jq, j1, D, Dp, nt, 1024.f, mu, 0.f, 0.f, s, batch,
                                             cf, vf_rec, vf_tiles, flags_done)
               : operand_typed<__half, false>(jq, j1, D, Dp, 0, 1.f, mu, half_c, pad_value, s,
                                              batch, cf, vf_rec, vf_tiles, flags_done);
}

cudaError_t launch_tf32_split(const float* x, int64_t rows, int64_t rows_pad, int D, int Dp,
                              const float* mu, float half_c, float* out, float* nrm,
                              float pad_value, cudaStream_t s, int batch) {
    const int64_t total = rows_pad * batch;
    if (total == 0) return cudaSuccess;
    const int threads = 256;
    const int64_t blocks = (total * 32 + threads - 1) / threads;
    launch_kernel(tf32_split_kernel, static_cast<unsigned>(blocks), threads, 0, s, 
        x, rows, rows_pad, total, D, Dp, mu, half_c, pad_value, out, nrm);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_value_prep(InType t, bool grad, bool w_f32, const void* w, const void* x,
                              const float* mu, int64_t N, int64_t Npad, int D, int Cw, int ch0,
                              int Cc, int Cp, unsigned* vmax_bits, void* vt, float* inv_scale,
                              cudaStream_t s) {
#define GS_VALUE_PREP(T, W, G) \
    value_prep_typed<T, W, G>(w, x, mu, N, Npad, D, Cw, ch0, Cc, Cp, vmax_bits, vt, inv_scale, s)
    if (t == InType::BF16) {
        if (!grad)
            return w_f32 ? GS_VALUE_PREP(__nv_bfloat16, float, false)
                         : GS_VALUE_PREP(__nv_bfloat16, __nv_bfloat16, false);
        return w_f32 ? GS_VALUE_PREP(__nv_bfloat16, float, true)
                     : GS_VALUE_PREP(__nv_bfloat16, __nv_bfloat16, true);
    }
    if (!grad) return w_f32 ? GS_VALUE_PREP(__half, float, false) : GS_VALUE_PREP(__half, __half, false);
    return w_f32 ? GS_VALUE_PREP(__half, float, true) : GS_VALUE_PREP(__half, __half, true);
#undef GS_VALUE_PREP
}


cudaError_t launch_key_records(InType t, const void* v, const float* B, int64_t N, int64_t Npad,
                               int C, float* rec, cudaStream_t s, int batch, bool signs) {
    if (signs) {
        // Sign records (fp16 values, C = 1): one thread per key, 256 per block.
        if (t != InType::F16 || C != 1 || B || Npad % kRecTile != 0) return cudaErrorInvalidValue;
        if (Npad == 0) return cudaSuccess;
        launch_kernel(sign_record_kernel, dim3(static_cast<unsigned>((Npad + 255) / 256), batch), 256, 0,
                      s, static_cast<const __half*>(v), N, Npad, rec);
        note_launches(1);
        return cudaGetLastError();
    }
    const int64_t pairs = Npad / 2;
    if (pairs == 0) return cudaSuccess;
    const int threads = 256;
    const unsigned blocks = static_cast<unsigned>((pairs + threads - 1) / threads);
    if (t == InType::BF16)
        launch_kernel(key_record_kernel<__nv_bfloat16>, dim3(blocks, batch), threads, 0, s, 
            static_cast<const __nv_bfloat16*>(v), B, N, pairs, C, rec);
    else if (t == InType::F32)
        launch_kernel(key_record_kernel<float>, dim3(blocks, batch), threads, 0, s, 
            static_cast<const float*>(v), B, N, pairs, C, rec);
    else
        launch_kernel(key_record_kernel<__half>, dim3(blocks, batch), threads, 0, s, static_cast<const __half*>(v), B, N,
                                                             pairs, C, rec);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_vf_flags(float* rec, int64_t Npad, int batch, cudaStream_t s) {
    if (batch <= 0) return cudaSuccess;
    launch_kernel(vf_flags_kernel, dim3(static_cast<unsigned>(batch)), 256, 0, s, rec, Npad / kRecTile,
                  batch);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_weight_prep(InType t, const void* rsrc, bool r_f32, int64_t R, int64_t Rpad,
                               const void* csrc, bool c_f32, int64_t Ncol, int64_t Npad, int C,
                               int WT, int BN, float* rowf, float* colT, unsigned* wmax,
                               cudaStream_t s) {
    if (WT <= 0 || kWeightThreads % WT != 0 || C > WT) return cudaErrorInvalidValue;
    cudaError_t e = cudaMemsetAsync(wmax, 0, sizeof(unsigned) * 2 * WT, s);
    if (e != cudaSuccess) return e;
    pdl_reset();   // the next kernel follows a memset
    const int64_t rb = (Rpad * WT + kWeightThreads - 1) / kWeightThreads;
    const int64_t cb = (Npad * WT + kWeightThreads - 1) / kWeightThreads;
    if (rb + cb == 0) return cudaSuccess;
    const dim3 grid(static_cast<unsigned>(rb + cb));
    const unsigned rbu = static_cast<unsigned>(rb);
#define GS_WPREP(TR, TC)                                                                        \
    launch_kernel(weight_prep_kernel<TR, TC>, grid, kWeightThreads, 0, s,                      \
                  static_cast<const TR*>(rsrc), R, Rpad, static_cast<const TC*>(csrc), Ncol,   \
                  Npad, C, WT, BN, rbu, rowf, colT, wmax)
    // One side is the float32 upstream gradient, the other the inputs' dtype.
    if (t == InType::BF16) {
        if (r_f32 && !c_f32) GS_WPREP(float, __nv_bfloat16);
        else if (!r_f32 && c_f32) GS_WPREP(__nv_bfloat16, float);
        else return cudaErrorInvalidValue;
    } else if (t == InType::F16) {
        if (r_f32 && !c_f32) GS_WPREP(float, __half);
        else if (!r_f32 && c_f32) GS_WPREP(__half, float);
        else return cudaErrorInvalidValue;
    } else {
        return cudaErrorInvalidValue;
    }
#undef GS_WPREP
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_finalize(const float* part, int splits, int64_t split_stride_rows,
                            int64_t M, int Cv, int part_ld, const float* inv_scale, float* out,
                            cudaStream_t s, int64_t main_rows) {
    const int64_t total = M * Cv;
    if (total == 0) return cudaSuccess;
    const int threads = 256;
    const int64_t blocks = (total + threads - 1) / threads;
    launch_kernel(finalize_kernel, static_cast<unsigned>(blocks), threads, 0, s, 
        part, splits, split_stride_rows, M, Cv, part_ld, inv_scale, out, main_rows);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_finalize_points(bool direct, InType t, bool u_f32, const float* part,
                                   int splits, int64_t split_stride_rows, int64_t M, int part_ld,
                                   const float* inv_scale, const void* x, const float* mu,
                                   float tau, int D, int Cw, int ch0, int Cc, const void* u,
                                   int accumulate, float* out, float* s_out, cudaStream_t s,
                                   int64_t main_rows) {
#define GS_FIN(DIR, T, U)                                                                     \
    finalize_points_typed<DIR, T, U>(part, splits, split_stride_rows, M, part_ld, inv_scale, x, \
                                     mu, tau, D, Cw, ch0, Cc, u, accumulate, out, s_out, s,      \
                                     main_rows)
    if (direct) return GS_FIN(true, float, float);
    if (t == InType::BF16)
        return u_f32 ? GS_FIN(false, __nv_bfloat16, float)
                     : GS_FIN(false, __nv_bfloat16, __nv_bfloat16);
    return u_f32 ? GS_FIN(false, __half, float) : GS_FIN(false, __half, __half);
#undef GS_FIN
}

}  // namespace gs
