// Fused tensor-core Gauss-sum kernel for sm_103a (tcgen05 + TMA + TMEM).
//
// For one tile of 128 query rows and a range of key tiles of BN keys the
// kernel evaluates Eq. 1 on the flash-attention schedule, without any
// softmax normalisation: in exact arithmetic the exponent
//     x_mn = c q^_m . k^_n + A_m + B_n = -(c/2) ||q^_m - k^_n||^2 <= 0,
//     c = tau log2 e,  A_m = -(c/2)||q^_m||^2,  B_n = -(c/2)||k^_n||^2
// is never positive (Phi <= 1, proof of Prop. 1), so 2^x needs no running
// maximum.  This is the algebra of Alg. 1 (prescale by the key norms, rescale
// by the query norms) folded into one fp32 exponent per pair instead of
// scaling the values and the output.
//
//   MMA1  S   = q^ k^T          tcgen05.mma kind::f16, A,B from shared memory,
//                               fp32 accumulator in TMEM (128 x BN)
//   exp   P   = fp16(2^(c S + A_m + B_n + 15))   TMEM -> registers -> TMEM
//   MMA2  O  += P v~            tcgen05.mma kind::f16, A = P from TMEM,
//                               B = value tile from shared memory, fp32 TMEM
//
// Warp roles ((NEXP + 4) x 32 threads; NEXP = 16 for BN = 128, 8 for BN = 64):
//   warps 0 .. NEXP-1  exponent warps in two groups of NEXP/2; group g
//              handles the key tiles j = g (mod 2).  Warp w owns TMEM lanes
//              32 (w % 4) .. +31 (its hardware lane quarter) and a share of
//              the key columns; all of them run the epilogue (TMEM O -> fp32
//              partial sums).
//   warp NEXP  TMA producer: q^ tile once, then k^ / v~ / B tiles into a
//              ring of `stages` shared-memory stages.
//   warp NEXP+1  TMEM allocator and MMA1 issuer (one elected thread).
//   warp NEXP+2  MMA2 issuer (EARLY; one elected thread); warp NEXP+3 idle.
// TMEM columns: S double buffer [0, 2 BN), P double buffer [2 BN, 3 BN)
// (fp16 pairs packed in 32-bit columns), O accumulator [3 BN, 3 BN + Cp);
// buffer g of S and of P belongs to exponent group g.
//
// Schedule (EARLY, exponent-bound shapes).  A group hands its S buffer
// back (s_free) as soon as the tile is in registers, so MMA1 of the group's
// next tile but one runs under the exponent work of the current tile; its P
// buffer comes back (p_free) when MMA2 of that tile has read it.  MMA1 and
// MMA2 are issued by two warps, each in key-tile order: the MMA1 stream
// waits for the keys and the S buffer, the MMA2 stream for P, so that a
// stage reload that MMA1 waits for never holds back an MMA2 that a group
// needs.  Tensor-bound shapes keep one MMA warp issuing MMA1 of tile j + 1
// after MMA2 of tile j - 1 (S handed back with P), which measured faster
// there.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "internal.h"
#include "ptx.cuh"
#include "tensor_map.h"

namespace gs {
namespace {

constexpr int BM = 128;           // query rows per CTA (MMA M)
constexpr int KB = 64;            // 16-bit elements per 128-byte swizzled row
constexpr uint32_t TMEM_COLS = 512;
// P is stored as fp16(2^(x + P_SHIFT)) with P_SHIFT = 15: kernel values
// down to 2^-29 stay normal fp16 numbers (instead of 2^-14), a kernel value
// of 1 is stored exactly (2^15), and the epilogue multiplies O by
// 2^-P_SHIFT.  The exponent is <= 0 in exact arithmetic.  A rounding-
// positive x is not clamped: 2^(15 + x) differs from the clamped 2^15 by
// less than x ln 2 relative, no more than the rounding error of x itself
// (and below 2^-12, half an fp16 ulp at 2^15, it rounds to 2^15 anyway);
// the saturating conversion keeps P finite for any x.
constexpr float P_SHIFT = 15.f;
constexpr float P_UNSHIFT = 1.f / 32768.f;

struct TcParams {
    const float* A;      // Mpad: -(c/2)||q^_m||^2
    const float* B;      // Npad: -(c/2)||k^_n||^2 (-inf for padded keys)
    float* part;         // splits x Mpad x Cp partial sums (unscaled)
    unsigned* status;    // device status word
    int64_t Mpad;
    int tile_off;        // row tile of blockIdx.x = 0 (main launch 0, tail launch main_tiles)
    int wave_tiles;      // > 0: blocks of odd waves (blockIdx.x / wave_tiles) take their key
                         // tiles in reverse order
    int key_tiles;
    int tiles_per_split;
    int nkb;             // 64-element K blocks of q^/k^
    int ksteps1;         // Dp / 16
    int Cp;
    int stages;
    uint32_t stage_bytes;
    uint32_t kh_bytes;   // k^ part of a stage
    uint32_t vt_bytes;   // v~ part of a stage
    uint32_t tx_bytes;   // bytes a stage's TMA copies deliver
    float c;
    uint32_t idesc1, idesc2;
    const uint32_t* qh;  // QTM: q^ rows (packed 16-bit pairs, Dp / 2 per row)
    // WT: factors of the pair weights (see launch_weight_prep): row factors
    // (Mpad x WT), column factors per key tile (WT x BN), and their
    // per-channel maxima (2 WT float bits).
    const float* rowf;
    const float* colT;
    const unsigned* wmax;
};

struct __align__(8) Barriers {
    uint64_t q_full;
    uint64_t o_full;
    uint64_t drain;       // MMA1 warp: its MMAs are complete
    uint64_t drain2;      // MMA2 warp: its MMAs are complete
    uint64_t s_full[2];   // S buffer g computed (MMA1 commit)
    uint64_t s_free[2];   // S buffer g in the registers of group g
    uint64_t p_full[2];   // P buffer g written by group g
    uint64_t p_free[2];   // P buffer g read by MMA2 (MMA2 commit)
    uint64_t kv_full[8];
    uint64_t kv_empty[8];
    uint32_t tmem_base;
    int abort_flag;
};

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned* status) {
    const bool ok = mbar_wait_bounded(bar, parity, abort_flag, status);
    return __all_sync(0xffffffffu, ok);
}

// Threads of a CTA with NEXP exponent warps plus one warpgroup holding the
// producer and MMA warps (and two idle warps, so that the register split
// below applies to whole warpgroups).
template <int NEXP>
constexpr int cta_threads() { return (NEXP + 4) * 32; }

// Register split for NEXP = 16 (launched with 640 x 96 registers).
constexpr uint32_t kExpRegs2 = 112;
constexpr uint32_t kCtrlRegs2 = 32;
static_assert(16 * 32 * kExpRegs2 + 4 * 32 * kCtrlRegs2 <= 640 * 96, "register split");

// AUG: augmented operands (S = -||q^ - k^||^2 / 2, no B records).
// EARLY: S buffers handed back right after the TMEM loads, MMA1 and MMA2
// issued by two warps (exponent-bound shapes); otherwise one MMA warp in
// P-then-S order (tensor-bound shapes).  QTM: q^ in TMEM (columns
// [3 BN + Cp, 3 BN + Cp + Dp / 2), copied there by the exponent warps; MMA1
// reads A from TMEM), which leaves its shared memory to the key stages.
// WT > 0: weighted vector-Jacobian pass: the kernel values are multiplied
// by the pair weights w_mn = sum_c r[m, c] k[n, c] (WT channels) before the
// rounding to fp16; see the exponent warps.
template <int BN, int NEXP, bool AUG, bool EARLY, bool QTM = false, int WT = 0>
__global__ void __launch_bounds__(cta_threads<NEXP>(), 1)
tc_gauss_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                const __grid_constant__ CUtensorMap tm_v, const TcParams p) {
    static_assert(NEXP % 4 == 0, "exponent warps cover the four TMEM lane quarters");
    constexpr int PRODUCER_WARP = NEXP;
    constexpr int MMA_WARP = NEXP + 1;     // MMA1 issuer, TMEM allocator
    constexpr int MMA2_WARP = NEXP + 2;    // MMA2 issuer
    // The exponent warps form two groups; group g handles the key tiles
    // j = g (mod 2), i.e. S/P buffer g, so that one group's TMEM and MMA
    // latency overlaps the other group's exp2 work.
    constexpr int GROUP_WARPS = NEXP / 2;
    constexpr int COLS = BN * 4 / GROUP_WARPS;  // key columns per exponent warp and tile
    static_assert(GROUP_WARPS % 4 == 0, "each group covers the four TMEM lane quarters");
    static_assert(COLS % 32 == 0, "exponent warps load whole 32-column chunks");
    static_assert(COLS == 64, "one 64-column TMEM load per warp and tile");

    extern __shared__ uint8_t smem_raw[];
    // 1024-byte aligned base for the 128-byte swizzle atoms.
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
    uint8_t* q_smem = smem;
    uint8_t* stage0 = smem + (QTM ? 0 : p.nkb * (BM * 128));
    Barriers* bars = reinterpret_cast<Barriers*>(stage0 + p.stages * p.stage_bytes);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int tile_m = p.tile_off + static_cast<int>(blockIdx.x);
    const int split = blockIdx.y;
    const int kt0 = split * p.tiles_per_split;
    const int kt1 = min(p.key_tiles, kt0 + p.tiles_per_split);
    const int T = kt1 - kt0;
    volatile int* abort_flag = &bars->abort_flag;

    pdl_trigger();
    if (tid == 0) {
        mbar_init(&bars->q_full, QTM ? NEXP : 1);   // TMA copy, or one arrival per exponent warp
        mbar_init(&bars->o_full, 1);
        mbar_init(&bars->drain, 1);
        mbar_init(&bars->drain2, 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->s_full[b], 1);
            mbar_init(&bars->s_free[b], GROUP_WARPS);  // one arrival per warp
            mbar_init(&bars->p_full[b], GROUP_WARPS);  // one arrival per warp
            mbar_init(&bars->p_free[b], 1);
        }
        for (int s = 0; s < p.stages; ++s) {
            mbar_init(&bars->kv_full[s], 1);
            mbar_init(&bars->kv_empty[s], 1);
        }
        bars->abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // The prologue above may overlap the previous kernel of the call; its
    // outputs (operands, values, norms) are read only from here on.
    pdl_wait();
    const uint32_t tmem = bars->tmem_base;
    const uint32_t S_col0 = 0, P_col0 = 2 * BN, O_col = 3 * BN;
    const uint32_t Q_col = 3 * BN + static_cast<uint32_t>(p.Cp);   // QTM

    auto kh_smem = [&](int s) { return stage0 + s * p.stage_bytes; };
    auto vt_smem = [&](int s) { return stage0 + s * p.stage_bytes + p.kh_bytes; };
    auto b_smem = [&](int s) {
        return reinterpret_cast<const float*>(stage0 + s * p.stage_bytes + p.kh_bytes + p.vt_bytes);
    };
    // WT: the key tile's column factors, channel-major (WT x BN floats).
    auto cw_smem = [&](int s) {
        return reinterpret_cast<const float*>(stage0 + s * p.stage_bytes + p.kh_bytes + p.vt_bytes +
                                              BN * 4);
    };

    if (warp == PRODUCER_WARP) {
        if (NEXP == 16) reg_dealloc<kCtrlRegs2>();
        // The whole warp runs the loop (warp-uniform operands); the elected
        // lane issues the copies.
        if (T > 0) {
            const bool leader = elect_one();
            if (leader) {
                tma_prefetch_desc(&tm_k);
                tma_prefetch_desc(&tm_v);
                if (!QTM) {
                    tma_prefetch_desc(&tm_q);
                    mbar_arrive_expect_tx(&bars->q_full, static_cast<uint32_t>(p.nkb * BM * 128));
                    for (int kb = 0; kb < p.nkb; ++kb)
                        tma_load_2d(q_smem + kb * (BM * 128), &tm_q, &bars->q_full, kb * KB, tile_m * BM);
                }
            }
            __syncwarp();
            int issued = 0;
            // Waves of one block per SM stream the same keys at about the
            // same time; every other wave streams them backwards, starting
            // with the keys the previous wave read last (still in L2)
            // instead of those it read first (evicted by then).  The sum of
            // a row is then taken in the reverse key order, a fixed order
            // all the same.
            const bool reverse = p.wave_tiles > 0 && ((blockIdx.x / p.wave_tiles) & 1u);
            RingPos st;
            for (int j = 0; j < T; ++j, st.advance(p.stages)) {
                const int s = st.idx;
                if (!warp_wait(&bars->kv_empty[s], st.phase ^ 1u, abort_flag, p.status)) break;
                if (leader) {
                    mbar_arrive_expect_tx(&bars->kv_full[s], p.tx_bytes);
                    const int n0 = (reverse ? kt1 - 1 - j : kt0 + j) * BN;
                    for (int kb = 0; kb < p.nkb; ++kb)
                        tma_load_2d(kh_smem(s) + kb * (BN * 128), &tm_k, &bars->kv_full[s], kb * KB, n0);
                    for (int h = 0; h < BN / KB; ++h)
                        tma_load_2d(vt_smem(s) + h * (p.Cp * 128), &tm_v, &bars->kv_full[s], n0 + h * KB, 0);
                    if (!AUG) bulk_load(const_cast<float*>(b_smem(s)), p.B + n0, BN * 4, &bars->kv_full[s]);
                    if (WT > 0)
                        bulk_load(const_cast<float*>(cw_smem(s)), p.colT + static_cast<int64_t>(n0) * WT,
                                  BN * WT * 4, &bars->kv_full[s]);
                }
                __syncwarp();
                issued = j + 1;
            }
            // Let every copy this CTA started land before the CTA can exit.
            mbar_wait_bounded(&bars->q_full, 0, nullptr, p.status);
            for (int j = max(0, issued - p.stages); j < issued; ++j)
                mbar_wait_bounded(&bars->kv_full[j % p.stages],
                                  static_cast<uint32_t>(j / p.stages) & 1u, nullptr, p.status);
            __syncwarp();
        }
    } else if (EARLY && warp == MMA_WARP) {
        if (NEXP == 16) reg_dealloc<kCtrlRegs2>();
        // MMA1 stream: S of key tile j into buffer j % 2, as soon as the
        // keys are loaded and group j % 2 holds tile j - 2 in registers.  The
        // whole warp runs the loop (warp-uniform descriptors); the elected
        // lane issues the MMAs and commits.
        if (T > 0) {
            const bool leader = elect_one();
            const uint32_t q_base = smem_u32(q_smem);
            bool ok = warp_wait(&bars->q_full, 0, abort_flag, p.status);
            RingPos st;
            for (int j = 0; ok && j < T; ++j, st.advance(p.stages)) {
                const int b = j & 1;
                ok = warp_wait(&bars->kv_full[st.idx], st.phase, abort_flag, p.status);
                if (ok && j >= 2)
                    ok = warp_wait(&bars->s_free[b], static_cast<uint32_t>((j - 2) >> 1) & 1u, abort_flag,
                                   p.status);
                if (!ok) break;
                tc_fence_after();
                const uint32_t kh_base = smem_u32(kh_smem(st.idx));
                if (leader) {
                    for (int kk = 0; kk < p.ksteps1; ++kk) {
                        const uint32_t koff = static_cast<uint32_t>(kk & 3) * 32;
                        const uint64_t bd = smem_desc_kmajor_sw128(kh_base + (kk >> 2) * (BN * 128) + koff);
                        if (QTM) {
                            mma_ts_f16(tmem + S_col0 + b * BN, tmem + Q_col + kk * 8, bd, p.idesc1,
                                       kk > 0 ? 1u : 0u);
                        } else {
                            const uint64_t ad = smem_desc_kmajor_sw128(q_base + (kk >> 2) * (BM * 128) + koff);
                            mma_ss_f16(tmem + S_col0 + b * BN, ad, bd, p.idesc1, kk > 0 ? 1u : 0u);
                        }
                    }
                    mma_commit(&bars->s_full[b]);
                }
                __syncwarp();
            }
            // No MMA of this warp may still be running when TMEM is released.
            if (leader) mma_commit(&bars->drain);
            __syncwarp();
            mbar_wait_bounded(&bars->drain, 0, nullptr, p.status);
            __syncwarp();
        }
    } else if (EARLY && warp == MMA2_WARP) {
        if (NEXP == 16) reg_dealloc<kCtrlRegs2>();
        // MMA2 stream: O += P v~ for key tile j once group j % 2 has written
        // P; its commits hand back the P buffer and the stage.  (MMA1 of
        // tile j completed before the group could write P of tile j, so the
        // stage is released after both MMAs that read it.)
        if (T > 0) {
            const bool leader = elect_one();
            bool ok = true;
            RingPos st;
            for (int j = 0; ok && j < T; ++j, st.advance(p.stages)) {
                const int b = j & 1;
                ok = warp_wait(&bars->p_full[b], static_cast<uint32_t>(j >> 1) & 1u, abort_flag, p.status);
                // The values of tile j landed before MMA1 of tile j was issued;
                // this wait (already complete) also orders them for this warp.
                if (ok) ok = warp_wait(&bars->kv_full[st.idx], st.phase, abort_flag, p.status);
                if (!ok) break;
                tc_fence_after();
                const uint32_t vt_base = smem_u32(vt_smem(st.idx));
                if (leader) {
                    for (int kk = 0; kk < BN / 16; ++kk) {
                        const uint64_t bd = smem_desc_kmajor_sw128(vt_base + (kk >> 2) * (p.Cp * 128) + (kk & 3) * 32);
                        mma_ts_f16(tmem + O_col, tmem + P_col0 + b * (BN / 2) + kk * 8, bd, p.idesc2,
                                   (j > 0 || kk > 0) ? 1u : 0u);
                    }
                    mma_commit(&bars->p_free[b]);
                    mma_commit(&bars->kv_empty[st.idx]);
                }
                __syncwarp();
            }
            if (leader) {
                if (ok) mma_commit(&bars->o_full);
                mma_commit(&bars->drain2);
            }
            __syncwarp();
            mbar_wait_bounded(&bars->drain2, 0, nullptr, p.status);
            __syncwarp();
        }
    } else if (!EARLY && warp == MMA_WARP) {
        if (NEXP == 16) reg_dealloc<kCtrlRegs2>();
        // Both streams in one warp, P-then-S order: MMA1 of tile j, then
        // (once P of tile j - 1 is written) MMA2 of tile j - 1.  MMA1 of tile
        // j + 1 thus enters the tensor queue behind MMA2 of tile j - 1, S
        // buffer (j + 1) % 2 is free then (P of tile j - 1 is written), and
        // the completion of S of a tile implies that MMA2 of the tile two
        // before it has read its P buffer.  The whole warp runs the loop
        // (warp-uniform descriptors); the elected lane issues the MMAs and
        // commits.
        if (T > 0) {
            const bool leader = elect_one();
            const uint32_t q_base = smem_u32(q_smem);
            bool ok = warp_wait(&bars->q_full, 0, abort_flag, p.status);
            RingPos st, stp;   // stage of tile j (MMA1) and of tile j - 1 (MMA2)
            for (int j = 0; ok && j <= T; ++j) {
                if (j < T) {
                    const int s = st.idx;
                    const int b = j & 1;
                    ok = warp_wait(&bars->kv_full[s], st.phase, abort_flag, p.status);
                    if (!ok) break;
                    tc_fence_after();
                    const uint32_t kh_base = smem_u32(kh_smem(s));
                    if (leader) {
                        for (int kk = 0; kk < p.ksteps1; ++kk) {
                            const uint32_t koff = static_cast<uint32_t>(kk & 3) * 32;
                            const uint64_t bd = smem_desc_kmajor_sw128(kh_base + (kk >> 2) * (BN * 128) + koff);
                            if (QTM) {
                                mma_ts_f16(tmem + S_col0 + b * BN, tmem + Q_col + kk * 8, bd, p.idesc1,
                                           kk > 0 ? 1u : 0u);
                            } else {
                                const uint64_t ad = smem_desc_kmajor_sw128(q_base + (kk >> 2) * (BM * 128) + koff);
                                mma_ss_f16(tmem + S_col0 + b * BN, ad, bd, p.idesc1, kk > 0 ? 1u : 0u);
                            }
                        }
                        mma_commit(&bars->s_full[b]);
                    }
                    __syncwarp();
                    st.advance(p.stages);
                }
                if (j >= 1) {
                    const int jp = j - 1;
                    const int bp = jp & 1;
                    const int sp = stp.idx;
                    ok = warp_wait(&bars->p_full[bp], static_cast<uint32_t>(jp >> 1) & 1u,
                                   abort_flag, p.status);
                    if (!ok) break;
                    tc_fence_after();
                    const uint32_t vt_base = smem_u32(vt_smem(sp));
                    if (leader) {
                        for (int kk = 0; kk < BN / 16; ++kk) {
                            const uint64_t bd = smem_desc_kmajor_sw128(vt_base + (kk >> 2) * (p.Cp * 128) + (kk & 3) * 32);
                            mma_ts_f16(tmem + O_col, tmem + P_col0 + bp * (BN / 2) + kk * 8, bd, p.idesc2,
                                       (jp > 0 || kk > 0) ? 1u : 0u);
                        }
                        mma_commit(&bars->kv_empty[sp]);
                    }
                    __syncwarp();
                    stp.advance(p.stages);
                }
            }
            if (leader) {
                if (ok) mma_commit(&bars->o_full);
                // No MMA may still be running when TMEM is released.
                mma_commit(&bars->drain);
            }
            __syncwarp();
            mbar_wait_bounded(&bars->drain, 0, nullptr, p.status);
            __syncwarp();
        }
    } else if (warp >= MMA_WARP) {
        // Idle warps completing the control warpgroup.
        if (NEXP == 16) reg_dealloc<kCtrlRegs2>();
    } else {
        if (NEXP == 16) reg_alloc<kExpRegs2>();
        // ------------------------------------------------ exponent warps
        // Warp w of group g = w / GROUP_WARPS reads TMEM lanes 32 (w % 4) ..
        // +31 (rows of the tile) and key columns [COLS part, COLS (part + 1))
        // of S buffer g, part = (w % GROUP_WARPS) / 4.
        const int group = warp / GROUP_WARPS;
        const int quarter = warp & 3;
        const int part = (warp % GROUP_WARPS) >> 2;
        const int col0 = part * COLS;
        const int row_local = quarter * 32 + lane;
        const int64_t row = static_cast<int64_t>(tile_m) * BM + row_local;
        const float a_m = (AUG ? 0.f : p.A[row]) + (WT > 0 ? 0.f : P_SHIFT);
        const uint64_t a2 = f32x2_pack(a_m, a_m);
        // WT: this row's factors of the pair weights, times 2^sw, and the
        // epilogue's inverse scale.  With Wb = sum_c max|r_c| max|k_c| >=
        // |w_mn| and sw = 15 - ceil(log2 Wb), |2^sw w_mn| <= 2^15, so the
        // products 2^x 2^sw w_mn (x <= 0) fit fp16 like the unweighted
        // P = 2^(x + 15), and small weights keep their precision.
        float unshift = P_UNSHIFT;
        uint64_t rw2[WT > 0 ? WT : 1];
        if (WT > 0) {
            float wb = 0.f;
#pragma unroll
            for (int c = 0; c < WT; ++c)
                wb = fmaf(__uint_as_float(p.wmax[c]), __uint_as_float(p.wmax[WT + c]), wb);
            int e = 0;
            if (wb > 0.f) frexpf(wb, &e);                // wb <= 2^e
            const int sw = max(-100, min(100, 15 - e));
            const float sc = ldexpf(1.f, sw);
            unshift = ldexpf(1.f, -sw);
#pragma unroll
            for (int c = 0; c < WT; ++c) {
                const float r = p.rowf[row * WT + c] * sc;
                rw2[c] = f32x2_pack(r, r);
            }
        }
        const uint64_t c2 = f32x2_pack(p.c, p.c);
        const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
        if (QTM) {
            // q^ rows of this lane quarter -> TMEM (MMA1's A operand): the
            // NEXP / 4 warps of a quarter take every (NEXP / 4)-th chunk of 8
            // columns (16 coordinates).
            const uint32_t* src = p.qh + row * (p.ksteps1 * 8);
            for (int ck = warp >> 2; ck < p.ksteps1; ck += NEXP / 4) {
                const uint4 lo = *reinterpret_cast<const uint4*>(src + ck * 8);
                const uint4 hi = *reinterpret_cast<const uint4*>(src + ck * 8 + 4);
                const uint32_t r8[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
                tmem_st_32x32b_x8(tmem + lane_base + Q_col + ck * 8, r8);
            }
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars->q_full);
        }
        bool ok = true;
        RingPos st;   // stage of key tile j
        if (group) st.advance(p.stages);
        for (int j = group; j < T; j += 2, st.advance(p.stages), st.advance(p.stages)) {
            const int b = group;
            const int s = st.idx;
            // The B records and the column factors of the stage are read
            // from shared memory (without augmented operands / with pair
            // weights); S itself is ordered by s_full.
            if (!AUG || WT > 0) ok = warp_wait(&bars->kv_full[s], st.phase, abort_flag, p.status);
            if (ok && !__all_sync(0xffffffffu, mbar_test_wait(&bars->s_full[b],
                                                               static_cast<uint32_t>(j >> 1) & 1u)))
                ok = warp_wait(&bars->s_full[b], static_cast<uint32_t>(j >> 1) & 1u, abort_flag,
                               p.status);
            if (!ok) break;
            tc_fence_after();
            // The warp's 64 S columns in one TMEM load, and below its P
            // columns in one TMEM store: each tcgen05 instruction takes a
            // slot of the queue that the MUFU exp2 instructions share, and
            // halving their number (from two x32 loads and two x16 stores)
            // measured 8 % faster on the 131072^2 gradient (3.030 -> 2.780
            // ms).  The wait names the loaded registers, so that no use of
            // them is scheduled above it (the loads land asynchronously).
            uint32_t r[64];
            tmem_ld_32x32b_x64(tmem + lane_base + S_col0 + b * BN + col0, r);
            tmem_wait_ld_regs(r);
            // S buffer b is in registers: MMA1 of tile j + 2 may overwrite it
            // (EARLY; otherwise MMA1 of tile j + 2 follows P of tile j).
            if (EARLY) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&bars->s_free[b]);
            }
            const float* Bs = b_smem(s) + col0;
            uint32_t pk[32];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                // x = c S + (A_m + 15) + B_n for four keys, two per f32x2 op
                // (with augmented operands S already holds the norm terms:
                // x = c S + 15).
                uint64_t t01 = a2, t23 = a2;
                if (!AUG) {
                    const float4 bb = *reinterpret_cast<const float4*>(Bs + 4 * i);
                    t01 = f32x2_add(f32x2_pack(bb.x, bb.y), a2);
                    t23 = f32x2_add(f32x2_pack(bb.z, bb.w), a2);
                }
                const uint64_t s01 = f32x2_pack(__uint_as_float(r[4 * i + 0]), __uint_as_float(r[4 * i + 1]));
                const uint64_t s23 = f32x2_pack(__uint_as_float(r[4 * i + 2]), __uint_as_float(r[4 * i + 3]));
                float x0, x1, x2, x3;
                f32x2_unpack(f32x2_fma(s01, c2, t01), x0, x1);
                f32x2_unpack(f32x2_fma(s23, c2, t23), x2, x3);
                if (WT > 0) {
                    // P' = 2^min(x, 0) (2^sw w_mn) for the four keys: the
                    // weights from the row factors (registers) and the key
                    // tile's column factors (shared memory, one broadcast
                    // 16-byte load per channel), in float32.
                    const float* cws = cw_smem(s) + col0 + 4 * i;
                    uint64_t w01 = 0ull, w23 = 0ull;
#pragma unroll
                    for (int c = 0; c < WT; ++c) {
                        const float4 kc = *reinterpret_cast<const float4*>(cws + c * BN);
                        w01 = f32x2_fma(rw2[c], f32x2_pack(kc.x, kc.y), w01);
                        w23 = f32x2_fma(rw2[c], f32x2_pack(kc.z, kc.w), w23);
                    }
                    float p0, p1, p2, p3;
                    f32x2_unpack(f32x2_mul(f32x2_pack(ex2_nonpos(x0), ex2_nonpos(x1)), w01), p0, p1);
                    f32x2_unpack(f32x2_mul(f32x2_pack(ex2_nonpos(x2), ex2_nonpos(x3)), w23), p2, p3);
                    pk[2 * i + 0] = pack_half2_satfinite(p0, p1);
                    pk[2 * i + 1] = pack_half2_satfinite(p2, p3);
                } else {
                    pk[2 * i + 0] = pack_half2_satfinite(ex2_approx(x0), ex2_approx(x1));
                    pk[2 * i + 1] = pack_half2_satfinite(ex2_approx(x2), ex2_approx(x3));
                }
            }
            if (EARLY && j >= 2) {
                // P buffer b: MMA2 of tile j - 2 has read it.  (With one MMA
                // warp the completion of S of tile j implies it.)
                ok = warp_wait(&bars->p_free[b], static_cast<uint32_t>((j - 2) >> 1) & 1u, abort_flag,
                               p.status);
                if (!ok) break;
                tc_fence_after();
            }
            tmem_st_32x32b_x32(tmem + lane_base + P_col0 + b * (BN / 2) + col0 / 2, pk);
            if (!ok) break;
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars->p_full[b]);
        }
        if (ok && T > 0 && warp_wait(&bars->o_full, 0, abort_flag, p.status)) {
            tc_fence_after();
            float* out = p.part + (static_cast<int64_t>(split) * p.Mpad + row) * p.Cp;
            constexpr int PARTS = NEXP / 4;
            const int epart = warp >> 2;
            for (int c8 = epart * 8; c8 < p.Cp; c8 += 8 * PARTS) {
                uint32_t r[8];
                tmem_ld_32x32b_x8(tmem + lane_base + O_col + c8, r);
                tmem_wait_ld_regs(r);
                float4 lo = make_float4(__uint_as_float(r[0]) * unshift, __uint_as_float(r[1]) * unshift,
                                        __uint_as_float(r[2]) * unshift, __uint_as_float(r[3]) * unshift);
                float4 hi = make_float4(__uint_as_float(r[4]) * unshift, __uint_as_float(r[5]) * unshift,
                                        __uint_as_float(r[6]) * unshift, __uint_as_float(r[7]) * unshift);
                *reinterpret_cast<float4*>(out + c8) = lo;
                *reinterpret_cast<float4*>(out + c8 + 4) = hi;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == MMA_WARP) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

// ---------------------------------------------------------------- host side
size_t align1k(size_t x) { return (x + 1023) & ~static_cast<size_t>(1023); }

template <int BN, int NEXP, bool AUG, bool EARLY, bool QTM = false, int WT = 0>
cudaError_t launch_bn(const TcPlan& pl, InType t, float c, char* ws, unsigned* status,
                      cudaStream_t s, const char** why, int tile_off, int tiles, int splits) {
    const CUtensorMapDataType hdt =
        t == InType::BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    CUtensorMap tm_q, tm_k, tm_v;
    if (!encode_tile_map_2d(&tm_q, hdt, ws + pl.off_qh, pl.Dp, pl.Mpad, pl.Dp * 2ull, KB, BM) ||
        !encode_tile_map_2d(&tm_k, hdt, ws + pl.off_kh, pl.Dp, pl.Npad, pl.Dp * 2ull, KB, BN) ||
        !encode_tile_map_2d(&tm_v, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, ws + pl.off_vt, pl.Npad,
                            pl.Cp, pl.Npad * 2ull, KB, pl.Cp)) {
        *why = "cuTensorMapEncodeTiled failed or is unavailable";
        return cudaErrorInvalidValue;
    }
    TcParams p;
    p.A = AUG ? nullptr : reinterpret_cast<const float*>(ws + pl.off_A);
    p.B = AUG ? nullptr : reinterpret_cast<const float*>(ws + pl.off_B);
    p.part = reinterpret_cast<float*>(ws + pl.off_part);
    p.status = status;
    p.Mpad = pl.Mpad;
    p.tile_off = tile_off;
    p.wave_tiles = splits == 1 ? pl.wave_tiles : 0;
    p.key_tiles = static_cast<int>(pl.Npad / BN);
    p.tiles_per_split = (p.key_tiles + splits - 1) / splits;
    p.nkb = (pl.Dp + KB - 1) / KB;
    p.ksteps1 = pl.Dp / 16;
    p.Cp = pl.Cp;
    p.stages = pl.stages;
    p.kh_bytes = static_cast<uint32_t>(p.nkb * BN * 128);
    p.vt_bytes = static_cast<uint32_t>((BN / KB) * pl.Cp * 128);
    p.tx_bytes = p.kh_bytes + p.vt_bytes + (AUG ? 0 : BN * 4) + BN * WT * 4;
    p.stage_bytes = static_cast<uint32_t>(align1k(p.kh_bytes + p.vt_bytes + BN * 4 + BN * WT * 4));
    p.c = c;
    const uint32_t hb = t == InType::BF16 ? 1u : 0u;
    p.idesc1 = idesc_f16(BM, BN, hb, hb);
    p.idesc2 = idesc_f16(BM, static_cast<uint32_t>(pl.Cp), 0u, 0u);

    // Per-device function attribute; cheap enough to set on every launch.
    p.qh = reinterpret_cast<const uint32_t*>(ws + pl.off_qh);
    p.rowf = WT > 0 ? reinterpret_cast<const float*>(ws + pl.off_rowf) : nullptr;
    p.colT = WT > 0 ? reinterpret_cast<const float*>(ws + pl.off_colT) : nullptr;
    p.wmax = WT > 0 ? reinterpret_cast<const unsigned*>(ws + pl.off_wmax) : nullptr;
    cudaError_t e = cudaFuncSetAttribute(tc_gauss_kernel<BN, NEXP, AUG, EARLY, QTM, WT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(pl.smem_bytes));
    if (e != cudaSuccess) return e;
    dim3 grid(static_cast<unsigned>(tiles), static_cast<unsigned>(splits));
    launch_kernel(tc_gauss_kernel<BN, NEXP, AUG, EARLY, QTM, WT>, grid, cta_threads<NEXP>(), pl.smem_bytes, s, tm_q, tm_k, tm_v, p);
    note_launches(1);
    return cudaGetLastError();
}

}  // namespace

// Banded order of the FMA kernel (see plan_tensor).
constexpr double kBandMinKeyBytes = 64.0 * 1024 * 1024;
constexpr int64_t kBandTiles = 64;
constexpr int64_t kMaxBands = 256;
// Longest segment (key tiles of one pair of query tiles in a row) that the
// FMA kernel runs with overlapped segment transitions.
constexpr int64_t kOverlapMaxTiles = 64;

bool plan_tensor(InType t, int64_t M, int64_t N, int64_t D, int64_t C, bool grad, bool center,
                 bool alias, int split_override, int sms, TcPlan* p, const char** why,
                 int64_t batch, bool tri, int wt) {
    p->M = M;
    p->N = N;
    p->D = D;
    // grad: C is the channel count of one launch (a chunk of C_w (D + 1)).
    p->Cv = C;
    p->Dp = static_cast<int>(std::max<int64_t>(16, (D + 15) / 16 * 16));
    p->Cp = static_cast<int>((p->Cv + 15) / 16 * 16);
    if (D > 256) { *why = "tensor-core path supports D <= 256"; return false; }
    if (p->Cp > 256) { *why = "tensor-core path supports C <= 256"; return false; }
    p->alias = alias;
    p->center = center;
    p->tf = false;
    p->early_s = false;
    p->tri = false;
    p->tri_units = 0;
    p->qtm = false;
    p->wt = wt;
    if (wt != 0 && !(grad && t != InType::F32 && (wt == 2 || wt == 4 || wt == 8))) {
        *why = "pair weights need a 16-bit gradient pass with 2, 4 or 8 weight channels";
        return false;
    }
    size_t fma_smem = 0;
    int fma_stages = 0, nq = 1;
    if (t == InType::F32) {
        // fp32 inputs on the tensor cores: the FMA kernel with 3xTF32 MMAs
        // (forward sum, few channels, small D).
        if (grad || p->Cv > kFmaMaxChannels || D > kTf32MaxDp) {
            *why = "the fp32 tensor-core path takes the forward sum with C <= 4 and D <= 32";
            return false;
        }
        p->tf = true;
        p->aug = false;
        p->Dp = 32;
        if (!plan_fma_kernel(p->Dp, static_cast<int>(p->Cv), false, true, &nq, &fma_stages,
                             &fma_smem)) {
            *why = "shared-memory budget exceeded";
            return false;
        }
    }
    // Few channels: FMA-pipe kernel.  When the augmented rows fit in 128
    // columns it takes the augmented operands (q^ in shared memory, norms
    // folded into the MMA).
    const int dp_aug = static_cast<int>((D + 2 * aug_norm_terms(t) + 15) / 16 * 16);
    // Three or four channels: on the FMA pipe their P.v costs the exponent
    // warps more than a second MMA costs the tensor cores, once a call is
    // large enough to repay the two-MMA path's value preparation (one
    // GB300, whole calls, 65536^2 pairs: D = 32, C = 4 1.16 ms on the FMA
    // kernel against 0.70 ms for C = 5 on the two-MMA kernel; D = 64, C = 3
    // and 4 0.94 and 1.16 against 0.87 ms).  Not with rows too wide for the
    // augmented layout (q^ in tensor memory: at D = 256, C = 4 the FMA
    // kernel took 6.4 ms against 12.8 ms for C = 5), nor for batches of
    // problems (their one-launch path) or the MMD^2 upper triangle.
    const bool channels_on_mma = p->Cv >= 3 && batch == 1 && !tri && dp_aug <= kAugMaxDp &&
                                 M * N >= kTwoMmaMinPairs;
    if (p->tf) {
        p->fma = true;
    } else {
        p->aug = !grad && p->Cv <= kFmaMaxChannels && dp_aug <= kAugMaxDp;
        const int dp_fma = p->aug ? dp_aug : p->Dp;
        p->fma = !grad && p->Cv <= kFmaMaxChannels && !channels_on_mma &&
                 plan_fma_kernel(dp_fma, static_cast<int>(p->Cv), p->aug, false, &nq, &fma_stages,
                                 &fma_smem);
        if (!p->fma) p->aug = false;
    }
    if (p->fma) {
        if (!p->tf) p->Dp = p->aug ? dp_aug : p->Dp;
        p->BN = 128;
        p->nq = nq;
        p->stages = fma_stages;
        p->smem_bytes = fma_smem;
    } else {
        // Two-MMA kernel: augmented operands when the extra MMA work stays
        // small next to the exponentials (the norm terms then cost the
        // exponent warps nothing).
        if (dp_aug + p->Cp <= 128) {
            p->aug = true;
            p->Dp = dp_aug;
        }
        const int nkb = (p->Dp + KB - 1) / KB;
        p->BN = p->Cp <= 128 ? 128 : 64;
        p->nq = 1;
        if (wt > 0 && p->BN != 128) {
            *why = "pair weights need D + 1 <= 128 value channels";
            return false;
        }

        const size_t stage = align1k(static_cast<size_t>(nkb) * p->BN * 128 +
                                     static_cast<size_t>(p->BN / KB) * p->Cp * 128 + p->BN * 4 +
                                     static_cast<size_t>(p->BN) * wt * 4);
        const size_t qbytes = static_cast<size_t>(nkb) * BM * 128;
        size_t fixed = 1024 /*alignment slack*/ + qbytes + sizeof(Barriers) + 64;
        const size_t budget = 232448;
        int stages = static_cast<int>(std::min<size_t>(6, (budget - fixed) / stage));
        // Fewer than four stages: q^ moves to tensor memory when its Dp / 2
        // columns fit beside S, P and O (3 BN + Cp + Dp / 2 <= 512), and its
        // shared memory buys another stage.
        if (stages < 4 && !p->aug && p->BN == 128 && 3 * 128 + p->Cp + p->Dp / 2 <= static_cast<int>(TMEM_COLS)) {
            const int st_t = static_cast<int>(std::min<size_t>(6, (budget - (fixed - qbytes)) / stage));
            if (st_t > stages) {
                p->qtm = true;
                fixed -= qbytes;
                stages = st_t;
            }
        }
        if (stages < 2) { *why = "shared-memory budget exceeded"; return false; }
        p->stages = stages;
        // Early S release with two MMA warps lets MMA1 run up to two key
        // tiles ahead of the exponent work, which needs stages to load them
        // into: with four or more stages it measured faster on every shape
        // tried (fp16 forward C = 8..128, gradients, VJP: 3-16 %), with three
        // (bf16 D = 128, C = 64) the P-then-S order of one MMA warp is 8 %
        // faster.
        p->early_s = stages >= 4;
        // At least ~116 KB so that one CTA (which owns all 512 TMEM columns)
        // runs per SM.
        p->smem_bytes = std::max<size_t>(fixed + stages * stage, 118 * 1024);
    }
    const int64_t rows_per_cta = static_cast<int64_t>(BM) * p->nq;
    p->Mpad = (M + rows_per_cta - 1) / rows_per_cta * rows_per_cta;
    p->Npad = alias ? p->Mpad : (N + 127) / 128 * 128;

    // Only the FMA kernel takes a batch in one launch; the caller loops over
    // the problems of a batch for the other kernels.
    p->batch = p->fma ? std::max<int64_t>(1, batch) : 1;
    const int64_t B = p->batch;
    const int64_t tiles = B * (p->Mpad / rows_per_cta);
    const int64_t key_tiles = p->Npad / p->BN;
    int best_s = 1;
    if (split_override > 0) {
        best_s = static_cast<int>(std::min<int64_t>(split_override, key_tiles));
    } else {
        double best = 1e300;
        for (int s = 1; s <= 64 && s <= key_tiles; ++s) {
            const int64_t tps = (key_tiles + s - 1) / s;
            const int64_t s_eff = (key_tiles + tps - 1) / tps;
            const int64_t waves = (tiles * s_eff + sms - 1) / sms;
            const double cost = static_cast<double>(waves) * (tps + 2);
            if (cost < best * 0.99) { best = cost; best_s = static_cast<int>(s_eff); }
        }
    }
    {
        const int64_t tps = (key_tiles + best_s - 1) / best_s;
        best_s = static_cast<int>((key_tiles + tps - 1) / tps);
    }
    p->splits = std::max(1, best_s);
    p->main_tiles = 0;
    if (!p->fma && split_override == 0 && tiles >= sms) {
        // Two-MMA kernel: whole waves of row tiles (one CTA per SM) take
        // their full key range in one launch (no partial sums to add, each
        // q^ tile read once, all CTAs of a wave streaming the same keys);
        // the tail row tiles, fewer than the SMs, split their key range so
        // that the last wave is filled: s key splits for the fewest waves of
        // the tail per key tile (about ceil(tail s / sms) / s of a tile).
        const int64_t main = tiles / sms * sms;
        const int64_t tail = tiles - main;
        int ts = 1;
        double best_t = tail > 0 ? 1e300 : 0.0;
        for (int s = 1; tail > 0 && s <= 64 && s <= key_tiles; ++s) {
            const int64_t tps = (key_tiles + s - 1) / s;
            const int64_t s_eff = (key_tiles + tps - 1) / tps;
            const double cost = static_cast<double>((tail * s_eff + sms - 1) / sms) * (tps + 2);
            if (cost < best_t * 0.99) { best_t = cost; ts = static_cast<int>(s_eff); }
        }
        p->main_tiles = main;
        p->splits = ts;
        p->wave_tiles = sms;
    }
    if (p->fma || split_override != 0 || tiles < sms) p->wave_tiles = 0;
    p->units = p->unit_len = 0;
    p->grid = 0;
    p->band_len = 0;
    p->nruns = 0;
    if (p->fma) {
        // Persistent split: one CTA per SM, each taking an equal run of
        // (pair of query tiles, key tile) units; with a forced split count
        // each pair of query tiles is cut into that many runs instead.
        const int64_t units = tiles * key_tiles;
        if (units >= (int64_t(1) << 31)) {
            *why = "too many query/key tile pairs for the FMA kernel";
            return false;
        }
        int64_t len = split_override > 0
                          ? (key_tiles + std::min<int64_t>(split_override, key_tiles) - 1) /
                                std::min<int64_t>(split_override, key_tiles)
                          : (units + sms - 1) / sms;
        len = std::max<int64_t>(1, len);
        p->units = units;
        p->unit_len = len;
        p->grid = static_cast<int>((units + len - 1) / len);
        int64_t most = 1;
        for (int64_t r = 0; r < tiles; ++r)
            most = std::max(most, ((r + 1) * key_tiles - 1) / len - r * key_tiles / len + 1);
        p->splits = static_cast<int>(most);
        // v^T K v with q = k and one channel: the upper triangle of tile
        // pairs only (pair P of query tiles takes key tiles 2P ..), half the
        // exponentials.
        if (tri && alias && p->aug && !p->tf && p->Cv == 1 && split_override == 0 &&
            p->Mpad == p->Npad && key_tiles % 2 == 0 && key_tiles / 2 == p->Mpad / (BM * 2)) {
            const int64_t ppb = key_tiles / 2;
            const int64_t U = ppb * key_tiles - ppb * (ppb - 1);
            const int64_t tunits = B * U;
            if (tunits < (int64_t(1) << 31)) {
                const int64_t tlen = std::max<int64_t>(1, (tunits + sms - 1) / sms);
                int64_t tmost = 1;
                for (int64_t r = 0; r < B * ppb; ++r) {
                    // Folded rows of key_tiles + 2 units: pair s, then pair ppb - 1 - s.
                    const int64_t b = r / ppb, P = r - b * ppb;
                    const int64_t s = 2 * P <= ppb - 1 ? P : ppb - 1 - P;
                    const int64_t start = b * U + s * (key_tiles + 2) + (s == P ? 0 : key_tiles - 2 * s);
                    tmost = std::max(tmost, (start + key_tiles - 2 * P - 1) / tlen - start / tlen + 1);
                }
                p->tri = true;
                p->tri_units = U;
                p->units = tunits;
                p->unit_len = tlen;
                p->grid = static_cast<int>((tunits + tlen - 1) / tlen);
                p->splits = static_cast<int>(tmost);
            }
        }
        // Keys (operand rows and records) larger than half the L2: in the
        // contiguous order the CTAs stand at evenly spread key tiles, so
        // every pair of query tiles reads all keys from DRAM again.  The
        // banded order keeps all CTAs within a few bands of 64 key tiles,
        // which stay in L2 while the pairs of query tiles pass over them.
        const double key_bytes =
            static_cast<double>(B) * p->Npad *
            ((p->tf ? 8.0 : 2.0) * p->Dp + 2.0 * ((p->aug ? 0 : 1) + p->Cv));
        if (!p->tri && split_override == 0 && key_bytes > kBandMinKeyBytes && key_tiles > kBandTiles) {
            const int64_t blen = std::max<int64_t>(kBandTiles, (key_tiles + kMaxBands - 1) / kMaxBands);
            const int64_t nbands = (key_tiles + blen - 1) / blen;
            const int64_t nruns = tiles * nbands;
            if (nruns < (int64_t(1) << 31)) {
                p->band_len = static_cast<int>(blen);
                p->nruns = nruns;
                p->grid = static_cast<int>(std::min<int64_t>(sms, nruns));
                p->splits = static_cast<int>(nbands);
                p->units = p->unit_len = 0;
            }
        }
    }
    // Short segments restart the pipeline often (q^ copy, first MMAs, the
    // segment barrier); with at most kOverlapMaxTiles key tiles per segment
    // the FMA kernel overlaps the restart with the previous segment's tail
    // (forward sums with augmented operands; measured on one GB300: B = 256
    // problems of 1024 points 0.205 -> 0.137 ms per call, B = 64 x 16384
    // 3.06 -> 2.96 ms).  Long segments keep the barrier, whose code measured
    // faster there.
    p->overlap = false;
    if (p->fma && p->aug && !p->tf && !p->tri) {
        const int64_t seg = p->band_len > 0 ? p->band_len : std::min<int64_t>(key_tiles, p->unit_len);
        p->overlap = seg <= kOverlapMaxTiles;
    }
    // ~256 rows per block of the mean kernel, so that every SM has work.
    p->mean_blocks = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(4096, (M + N + 255) / 256)));

    size_t off = 0;
    auto take = [&](size_t bytes) { size_t o = off; off = align1k(off + bytes); return o; };
    p->off_mean_part = take(static_cast<size_t>(B) * p->mean_blocks * D * 2 * 4);
    p->off_mu = take(static_cast<size_t>(B) * D * 4);
    // Operand rows: Dp 16-bit values, or (3xTF32) hi and lo halves of Dp floats.
    const size_t row_bytes = p->tf ? static_cast<size_t>(p->Dp) * 8 : static_cast<size_t>(p->Dp) * 2;
    p->off_qh = take(static_cast<size_t>(B) * p->Mpad * row_bytes);
    // Augmented query and key operands differ in their extra columns, so
    // they are separate arrays even when q and k are the same points.
    p->off_kh = (alias && !p->aug) ? p->off_qh
                                   : take(static_cast<size_t>(B) * p->Npad * row_bytes);
    if (p->aug) {
        p->off_A = p->off_B = 0;   // the norms live in the augmented columns
    } else {
        p->off_A = take(static_cast<size_t>(B) * p->Mpad * 4);
        p->off_B = alias ? p->off_A : take(static_cast<size_t>(B) * p->Npad * 4);
    }
    if (p->fma) {
        p->off_vt = p->off_vmax = p->off_inv = 0;
        // Key records: value pairs, or (one channel on augmented operands,
        // when the value magnitudes are folded) 132 floats per key tile.
        size_t rec_floats = static_cast<size_t>(p->Npad / 2) * ((p->aug ? 0 : 2) + 2 * p->Cv);
        if (p->aug && p->Cv == 1) rec_floats = std::max<size_t>(rec_floats, (p->Npad / 128) * 132);
        // (+ one word per problem: the folded-value pass flags.)
        p->off_rec = take(static_cast<size_t>(B) * (rec_floats + 1) * 4);
        p->off_part = take(static_cast<size_t>(p->splits) * B * p->Mpad * p->Cv * 4);
    } else {
        p->off_rec = 0;
        p->off_vt = take(static_cast<size_t>(p->Cp) * p->Npad * 2);
        p->off_vmax = take(static_cast<size_t>(p->Cp) * 4);
        p->off_inv = take(static_cast<size_t>(p->Cp) * 4);
        p->off_part = take(static_cast<size_t>(p->splits) * p->Mpad * p->Cp * 4);
    }
    p->off_rowf = p->off_colT = p->off_wmax = 0;
    if (wt > 0) {
        p->off_rowf = take(static_cast<size_t>(p->Mpad) * wt * 4);
        p->off_colT = take(static_cast<size_t>(p->Npad) * wt * 4);
        p->off_wmax = take(static_cast<size_t>(2) * wt * 4);
    }
    p->total = off;
    return true;
}

namespace {

cudaError_t launch_tc_range(const TcPlan& p, InType t, float c, char* ws, unsigned* status,
                            cudaStream_t s, const char** why, int off, int tiles, int splits) {
#define GS_TC(BN_, NE_, AUG_, EARLY_, QTM_) \
    launch_bn<BN_, NE_, AUG_, EARLY_, QTM_>(p, t, c, ws, status, s, why, off, tiles, splits)
#define GS_TCW(AUG_, EARLY_, QTM_)                                                               \
    (p.wt == 2   ? launch_bn<128, 16, AUG_, EARLY_, QTM_, 2>(p, t, c, ws, status, s, why, off,   \
                                                             tiles, splits)                      \
     : p.wt == 4 ? launch_bn<128, 16, AUG_, EARLY_, QTM_, 4>(p, t, c, ws, status, s, why, off,   \
                                                             tiles, splits)                      \
                 : launch_bn<128, 16, AUG_, EARLY_, QTM_, 8>(p, t, c, ws, status, s, why, off,   \
                                                             tiles, splits))
    if (p.wt > 0) {
        // Weighted vector-Jacobian pass (BN = 128 only, see plan_tensor).
        if (p.BN != 128) return cudaErrorInvalidValue;
        if (p.aug) return p.early_s ? GS_TCW(true, true, false) : GS_TCW(true, false, false);
        if (p.qtm) return p.early_s ? GS_TCW(false, true, true) : GS_TCW(false, false, true);
        return p.early_s ? GS_TCW(false, true, false) : GS_TCW(false, false, false);
    }
    if (p.aug) {
        if (p.BN == 128) return p.early_s ? GS_TC(128, 16, true, true, false) : GS_TC(128, 16, true, false, false);
        return p.early_s ? GS_TC(64, 8, true, true, false) : GS_TC(64, 8, true, false, false);
    }
    if (p.BN == 128 && p.qtm)
        return p.early_s ? GS_TC(128, 16, false, true, true) : GS_TC(128, 16, false, false, true);
    if (p.BN == 128) return p.early_s ? GS_TC(128, 16, false, true, false) : GS_TC(128, 16, false, false, false);
    return p.early_s ? GS_TC(64, 8, false, true, false) : GS_TC(64, 8, false, false, false);
#undef GS_TCW
#undef GS_TC
}

}  // namespace

cudaError_t launch_tc(const TcPlan& p, InType t, float c, char* ws, unsigned* status,
                      cudaStream_t s, const char** why) {
    // Whole waves of row tiles unsplit, then the tail row tiles with their
    // key range split (see plan_tensor).
    const int tiles = static_cast<int>(p.Mpad / BM);
    const int main = static_cast<int>(p.main_tiles);
    cudaError_t e = cudaSuccess;
    if (main > 0) e = launch_tc_range(p, t, c, ws, status, s, why, 0, main, 1);
    if (e == cudaSuccess && tiles > main)
        e = launch_tc_range(p, t, c, ws, status, s, why, main, tiles - main, p.splits);
    return e;
}

}  // namespace gs
