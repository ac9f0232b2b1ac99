// fp32 SIMT Gauss-sum kernel (the single-precision regime of the paper's
// appendix, where tensor-core attention is not available).
//
// Each thread owns one query row, held in registers and zero padded to
// DMAX coordinates.  Keys stream through shared memory in tiles of KT keys
// (zero padded to DMAX, so padded coordinates add (0 - 0)^2 = 0).  For each
// pair the squared distance is formed in the direct-difference form
// sum_d (q_d - k_d)^2 (no Gram identity, hence no cancellation), the kernel
// value is 2^(-(c/2) d^2) with c = tau log2 e, and the values are
// accumulated with fp32 FMAs:
//   forward (Eq. 1):     acc[j] += Phi v[n, c0 + j]       for CBLK channels
//   gradient (Sec. 3):   acc[d] += Phi w_n (k_d - q_d),   acc[D] += Phi w_n
//                        with w_n = v[n, c] for one weight channel c
// The key range is split over gridDim.y; partial sums go to a workspace and
// are added in a fixed order by the finalise kernel.  Coordinates are
// handled in pairs with the packed f32x2 subtract / FMA of sm_100+ (the
// squared distance accumulates even and odd coordinates separately and
// adds the two at the end).
#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

namespace gs {
namespace {

constexpr int KT = 64;       // keys per shared-memory tile
constexpr int THREADS = 128; // query rows per block

template <int DMAX, int CBLK, bool GRAD>
__global__ void __launch_bounds__(THREADS)
simt_gauss_kernel(const float* __restrict__ q, const float* __restrict__ k,
                  const float* __restrict__ v, int64_t M, int64_t N, int D, int Cv,
                  int wch, float half_c, int64_t keys_per_split, float* __restrict__ part) {
    pdl_trigger();
    pdl_wait();
    __shared__ __align__(16) float ks[KT][DMAX];
    __shared__ float vs[KT][GRAD ? 1 : CBLK];

    const int64_t m = static_cast<int64_t>(blockIdx.x) * THREADS + threadIdx.x;
    const int split = blockIdx.y;
    const int c0 = GRAD ? 0 : blockIdx.z * CBLK;
    const int64_t n_begin = static_cast<int64_t>(split) * keys_per_split;
    const int64_t n_end = min(N, n_begin + keys_per_split);

    uint64_t qr[DMAX / 2];   // coordinate pairs of the query row
#pragma unroll
    for (int d = 0; d < DMAX; d += 2)
        qr[d / 2] = f32x2_pack((m < M && d < D) ? q[m * D + d] : 0.f,
                               (m < M && d + 1 < D) ? q[m * D + d + 1] : 0.f);
    float acc[GRAD ? 1 : CBLK];      // forward channels; gradient: sum of w
    uint64_t acc2[GRAD ? DMAX / 2 : 1];   // gradient coordinates, in pairs
#pragma unroll
    for (int j = 0; j < (GRAD ? 1 : CBLK); ++j) acc[j] = 0.f;
#pragma unroll
    for (int j = 0; j < (GRAD ? DMAX / 2 : 1); ++j) acc2[j] = 0ull;

    for (int64_t t0 = n_begin; t0 < n_end; t0 += KT) {
        const int cnt = static_cast<int>(min(static_cast<int64_t>(KT), n_end - t0));
        __syncthreads();
        for (int i = threadIdx.x; i < KT * DMAX; i += THREADS) {
            const int kk = i / DMAX, d = i - kk * DMAX;
            ks[kk][d] = (kk < cnt && d < D) ? k[(t0 + kk) * D + d] : 0.f;
        }
        if (GRAD) {
            // v is N x Cv here; the weight is its channel wch.
            for (int i = threadIdx.x; i < KT; i += THREADS)
                vs[i][0] = i < cnt ? v[(t0 + i) * Cv + wch] : 0.f;
        } else {
            for (int i = threadIdx.x; i < KT * CBLK; i += THREADS) {
                const int kk = i / CBLK, j = i - kk * CBLK;
                vs[kk][j] = (kk < cnt && c0 + j < Cv) ? v[(t0 + kk) * Cv + c0 + j] : 0.f;
            }
        }
        __syncthreads();
        for (int kk = 0; kk < cnt; ++kk) {
            uint64_t d2p = 0ull;   // (even, odd) partial squared distances
#pragma unroll
            for (int d = 0; d < DMAX; d += 4) {
                const float4 kv = *reinterpret_cast<const float4*>(&ks[kk][d]);
                const uint64_t t0 = f32x2_sub(qr[d / 2], f32x2_pack(kv.x, kv.y));
                const uint64_t t1 = f32x2_sub(qr[d / 2 + 1], f32x2_pack(kv.z, kv.w));
                d2p = f32x2_fma(t0, t0, d2p);
                d2p = f32x2_fma(t1, t1, d2p);
            }
            float d2e, d2o;
            f32x2_unpack(d2p, d2e, d2o);
            const float phi = ex2_approx(-half_c * (d2e + d2o));
            if (GRAD) {
                const float w = phi * vs[kk][0];
                const uint64_t w2 = f32x2_pack(w, w);
#pragma unroll
                for (int d = 0; d < DMAX; d += 4) {
                    const float4 kv = *reinterpret_cast<const float4*>(&ks[kk][d]);
                    acc2[d / 2] = f32x2_fma(w2, f32x2_sub(f32x2_pack(kv.x, kv.y), qr[d / 2]), acc2[d / 2]);
                    acc2[d / 2 + 1] =
                        f32x2_fma(w2, f32x2_sub(f32x2_pack(kv.z, kv.w), qr[d / 2 + 1]), acc2[d / 2 + 1]);
                }
                acc[0] += w;
            } else {
#pragma unroll
                for (int j = 0; j < CBLK; ++j) acc[j] = fmaf(phi, vs[kk][j], acc[j]);
            }
        }
    }
    if (m >= M) return;
    if (GRAD) {
        float* out = part + (static_cast<int64_t>(split) * M + m) * (D + 1);
#pragma unroll
        for (int d = 0; d < DMAX; d += 2) {
            float lo, hi;
            f32x2_unpack(acc2[d / 2], lo, hi);
            if (d < D) out[d] = lo;
            if (d + 1 < D) out[d + 1] = hi;
        }
        out[D] = acc[0];
    } else {
        float* out = part + (static_cast<int64_t>(split) * M + m) * Cv + c0;
#pragma unroll
        for (int j = 0; j < CBLK; ++j)
            if (c0 + j < Cv) out[j] = acc[j];
    }
}

template <int DMAX, int CBLK, bool GRAD>
cudaError_t launch_cblk(const SimtPlan& p, const float* q, const float* k, const float* v,
                        int Cw, int wch, float half_c, float* part, cudaStream_t s) {
    dim3 grid(static_cast<unsigned>((p.M + THREADS - 1) / THREADS), p.splits,
              GRAD ? 1u : static_cast<unsigned>((p.Cv + CBLK - 1) / CBLK));
    launch_kernel(simt_gauss_kernel<DMAX, CBLK, GRAD>, grid, THREADS, 0, s, 
        q, k, v, p.M, p.N, static_cast<int>(p.D), GRAD ? Cw : static_cast<int>(p.Cv), wch,
        half_c, p.keys_per_split, part);
    note_launches(1);
    return cudaGetLastError();
}

// Channel blocks of 4, or of 1 for a single channel (no idle FMAs).
template <int DMAX, bool GRAD>
cudaError_t launch_dmax(const SimtPlan& p, const float* q, const float* k, const float* v,
                        int Cw, int wch, float half_c, float* part, cudaStream_t s) {
    if (!GRAD && p.Cv == 1) return launch_cblk<DMAX, 1, GRAD>(p, q, k, v, Cw, wch, half_c, part, s);
    return launch_cblk<DMAX, 4, GRAD>(p, q, k, v, Cw, wch, half_c, part, s);
}

}  // namespace

bool plan_simt(int64_t M, int64_t N, int64_t D, int64_t C, bool grad, int split_override,
               int sms, SimtPlan* p, const char** why) {
    p->M = M;
    p->N = N;
    p->D = D;
    p->Cv = grad ? D + 1 : C;
    const int64_t dlimit = grad ? 64 : 128;
    if (D > dlimit) {
        *why = grad ? "fp32 gradient supports D <= 64" : "fp32 path supports D <= 128";
        return false;
    }
    p->dmax = D <= 16 ? 16 : D <= 32 ? 32 : D <= 64 ? 64 : 128;
    p->cblk = 4;
    const int64_t rowblocks = (M + THREADS - 1) / THREADS;
    const int64_t chunks = grad ? 1 : (p->Cv + 3) / 4;
    const int64_t key_tiles = (N + KT - 1) / KT;
    int64_t splits = split_override > 0 ? split_override
                                        : (4LL * sms + rowblocks * chunks - 1) / (rowblocks * chunks);
    splits = std::max<int64_t>(1, std::min<int64_t>(splits, std::max<int64_t>(1, key_tiles)));
    splits = std::min<int64_t>(splits, 65535);
    const int64_t tiles_per_split = (key_tiles + splits - 1) / splits;
    p->keys_per_split = std::max<int64_t>(KT, tiles_per_split * KT);
    p->splits = static_cast<int>((N + p->keys_per_split - 1) / p->keys_per_split);
    if (p->splits < 1) p->splits = 1;
    p->off_part = 0;
    p->total = static_cast<size_t>(p->splits) * M * p->Cv * sizeof(float);
    p->total = (p->total + 1023) & ~static_cast<size_t>(1023);
    return true;
}

cudaError_t launch_simt(const SimtPlan& p, bool grad, const float* q, const float* k,
                        const float* v, int Cw, int wch, float half_c, float* part,
                        cudaStream_t s) {
    if (grad) {
        switch (p.dmax) {
            case 16: return launch_dmax<16, true>(p, q, k, v, Cw, wch, half_c, part, s);
            case 32: return launch_dmax<32, true>(p, q, k, v, Cw, wch, half_c, part, s);
            default: return launch_dmax<64, true>(p, q, k, v, Cw, wch, half_c, part, s);
        }
    }
    switch (p.dmax) {
        case 16: return launch_dmax<16, false>(p, q, k, v, 0, 0, half_c, part, s);
        case 32: return launch_dmax<32, false>(p, q, k, v, 0, 0, half_c, part, s);
        case 64: return launch_dmax<64, false>(p, q, k, v, 0, 0, half_c, part, s);
        default: return launch_dmax<128, false>(p, q, k, v, 0, 0, half_c, part, s);
    }
}

}  // namespace gs
