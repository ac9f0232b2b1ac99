// Fused Gauss-sum kernel for few value channels (C <= 4), sm_103a.
//
// Only the dense contraction runs on the tensor cores: tcgen05 MMAs form
// S = q^ k^T (fp16/bf16 operands, fp32 accumulator in TMEM) for 128 x 128
// tiles.  The exponent warps turn each S tile into kernel values
// Phi(q_m, k_n) = 2^(c S + A_m + B_n) (the exponent is <= 0, so no running
// maximum is needed; see tc_gauss.cu) and accumulate sum_n Phi v_n in fp32
// on the FMA pipe.  With augmented operands (prep.cu) the MMA already adds
// the norm terms, S = -||q^ - k^||^2 / 2, and Phi = 2^(c S).  For one or
// two channels this costs fewer issue slots than a second MMA with N = 16,
// and it keeps kernel values and values in fp32; three or four channels
// come here for calls below 2^28 pairs and for rows too wide for the
// augmented layout (larger calls of three or four channels on augmented
// rows run faster on the two-MMA kernel, whose value preparation they
// repay).
//
// Layout choices:
//   * A CTA owns two query tiles (256 rows), which halves the L2 -> shared
//     memory traffic of the key tiles; every exponent warp handles the same
//     key columns of both query tiles, so one broadcast load of a key
//     record serves two kernel values.
//   * One barrier handshake per key tile: the 2 x (Dp / 16) MMAs of a key
//     tile are issued back to back and committed once; the exponent warps
//     release both S buffers and the stage of the key tile with one
//     (predicated) arrival per warp on each barrier once the tile is done,
//     and, on the two-slot fp16/bf16 path, query the next key tile's
//     barriers before exponentiating the current one.
//   * Work order: persistent CTAs over (pair of query tiles, key tile)
//     units, contiguous runs or (keys beyond half the L2) bands of key
//     tiles; for v^T K v with q = k (TRI) only the upper triangle of tile
//     pairs, folded into rows of equal length.  A CTA's work is a sequence
//     of segments (one pair of query tiles, consecutive key tiles).  With
//     short segments (OVL) the control warps move on to the next segment
//     without a CTA barrier: they reload q^ once the last two S tiles of
//     the segment are complete and release each stage when they next load
//     it, so the next segment's copies and MMAs run while the exponent
//     warps finish the current one.
//   * TMEM holds SL slots of two 128-column S buffers (one per query
//     tile); key tile j uses slot j % SL, so the MMAs of key tile j only
//     wait for the release of key tile j - SL.  With Dp <= 128 the query
//     tiles q^ stay in shared memory (A operand read by the MMA from shared
//     memory) and SL = 2; with larger Dp they would not fit next to the key
//     stages, so q^ is copied into TMEM (A operand from TMEM) and SL = 1.
//   * The kernel is bound by instruction dispatch next to the MUFU pipe,
//     and TMEM lane quarters tie every row to one SMSP, so each SMSP must
//     carry the same extra work: the MMA issue and key loads are split over
//     one control warp per SMSP (round robin over key tiles) rather than
//     given to one MMA warp, whose SMSP would otherwise pace all others.
//
// Warp roles (20 warps):
//   warps 0-15   exponent warps.  Warp w reads TMEM lanes 32 (w % 4) .. +31
//                (rows of both query tiles) and key columns 32 (w / 4) .. +31
//                of the two S buffers of each key tile.
//   warps 16-19  control warps, one per SMSP.  Control warp k owns shared-
//                memory stage k and key tiles j = k (mod stages): it loads
//                their k^ rows and key records (TMA) and issues and commits
//                their MMAs.  Warp 16 also allocates TMEM and loads q^.
// Key records: for each pair of keys (2t, 2t + 1) the floats
//   [B_2t, B_2t+1,] v_2t[0], v_2t+1[0], ..., v_2t[C-1], v_2t+1[C-1]
// (B only without augmented operands).  With folded values (VF: C = 1,
// fp16 values, augmented operands whose query rows carry the exponent
// scale c and whose key norm terms carry log2(|v_n| 2^-16), so that
// 2^S = Phi |v_n| 2^-16 with no multiply), the records of a key tile are
// the signs s_n = sign(v_n) 2^16 in key order and one word per 32-key
// column group, +-2^16 where all the group's values share a sign, else 0:
// such a group's exponent loop then reads no record at all (the broadcast
// record load per key pair was a fifth of its MIO work).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"
#include "tensor_map.h"

namespace gs {
namespace {

constexpr int BM = 128;            // rows per query tile (MMA M)
constexpr int NQ = 2;              // query tiles per CTA
constexpr int BN = 128;            // keys per key tile (MMA N)
constexpr int KB = 64;             // 16-bit elements per 128-byte swizzled row
constexpr int NEXP = 16;
// Exponentials on the FMA pipe (exp2_fma_x2) instead of MUFU (augmented
// operands, template parameter SOFT = 1..4): the kernel values of row 0 of
// key pair t take the FMA route when (t & soft_mask(SOFT)) == 0, which moves
// 1/32, 1/16, 1/8 or 1/4 of the exponentials; SOFT = 0: none.
__host__ __device__ constexpr int soft_mask(int soft) {
    return soft == 1 ? 15 : soft == 2 ? 7 : soft == 3 ? 3 : 1;
}
constexpr int CTRL_WARP0 = 16;     // control warps 16..19, one per SMSP
constexpr int NCTRL_MAX = 4;
constexpr int THREADS = (NEXP + NCTRL_MAX) * 32;
constexpr int NPART = 4;           // column groups (partial sums) per row
constexpr int MAX_SL = 2;          // TMEM slots of two S buffers
constexpr uint32_t TMEM_COLS = 512;
constexpr int MAX_STAGES = NCTRL_MAX;   // one stage per control warp
// Augmented operands keep q^ in shared memory (two TMEM slots of S).
constexpr bool kAugQsm = true;
// Register split between the roles (setmaxnreg); the sum stays within the
// registers the CTA is launched with (THREADS x 96).
constexpr uint32_t kExpRegs = 112;
constexpr uint32_t kCtrlRegs = 32;
static_assert(NEXP * 32 * kExpRegs + NCTRL_MAX * 32 * kCtrlRegs <= THREADS * 96, "register split");

struct FmaParams {
    const uint32_t* qh;  // Mpad x Dp/2 packed 16-bit pairs (centred, rounded q)
    const float* A;      // Mpad: -(c/2)||q^_m||^2
    const float* rec;    // key records, Npad / 2 pairs
    float* part;         // contributor slots x Mpad x C partial sums
    unsigned* status;
    int64_t Mpad;
    int units;           // work units: (pair of query tiles, key tile), row major
    int unit_len;        // units per CTA (CTA i: units [i unit_len, (i + 1) unit_len))
    // Banded order (band_len > 0, for keys larger than L2): run r = (band
    // r / pairs_total, pair of query tiles r % pairs_total) covers band_len
    // key tiles; CTA i takes runs i, i + grid, ...; the slot is the band.
    int band_len;
    int nruns;           // banded order: runs; upper-triangle order (TRI): units per problem
    int pairs_total;
    int key_tiles;       // key tiles per problem
    int pairs_per_batch; // pairs of query tiles per problem of a batch
    int npad;            // k^ rows per problem of a batch
    int Dp;
    int nkb;             // 128-byte K blocks of a q^ / k^ row (TF: hi blocks, then lo)
    int kb_elems;        // elements per K block (64 16-bit, 32 fp32)
    int ksteps;          // MMA K steps over the coordinates (16 fp16/bf16, 8 tf32 each)
    int stages;
    uint32_t q_bytes;    // shared-memory q^ tiles (0 when q^ is in TMEM)
    uint32_t stage_bytes;
    uint32_t kh_bytes;
    uint32_t rec_bytes;  // key-record bytes of one key tile
    uint32_t red_offset; // byte offset of the reduction area
    float c;
    uint32_t idesc;
};

struct __align__(8) FmaBarriers {
    uint64_t qa_ready;          // q^ available to the MMAs
    uint64_t q_free;            // OVL: every MMA of the segment has read q^ (one arrival per control warp)
    uint64_t s_full[MAX_SL];    // slot phase: both S tiles of a key tile computed
    uint64_t s_free[MAX_SL];    // slot phase: both S tiles of a key tile in registers
    uint64_t kv_full[MAX_STAGES];
    uint64_t kv_empty[MAX_STAGES];
    uint64_t stall;             // test hook: a barrier nothing arrives on
    uint64_t drain[NCTRL_MAX];  // control warp k: its MMAs are complete
    uint32_t tmem_base;
    int abort_flag;
};

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned* status) {
    const bool ok = mbar_wait_bounded(bar, parity, abort_flag, status);
    return __all_sync(0xffffffffu, ok);
}

// One segment of a CTA's work: the pair of query tiles tile_m and T
// consecutive key tiles from kt0, and the partial-sum slot it writes.
struct Segment {
    int tile_m, kt0, T, slot;
};

// Next segment of this CTA, or false after its last one.  Contiguous order:
// the CTA's run of units [u, u_end) split at query-pair boundaries, slot =
// rank of this CTA among the CTAs of that pair.  Banded order: runs
// blockIdx.x, blockIdx.x + gridDim.x, ..., slot = band.
template <bool TRI>
__device__ __forceinline__ bool next_segment(const FmaParams& p, int u_end, int& u, int& run,
                                             Segment& sg) {
    if (TRI) {
        // Upper-triangle order: pair P of query tiles takes the key tiles
        // 2P .. KT - 1 (KT - 2P units).  Pairs are folded into rows of equal
        // length KT + 2: row s holds pair s, then pair PPB - 1 - s (2s + 2
        // units); with PPB odd the middle pair forms a last, shorter row.
        // Every CTA thus walks about the same number of pairs.
        if (u >= u_end) return false;
        const int64_t U = p.nruns;
        const int64_t KT = p.key_tiles;
        const int64_t PPB = p.pairs_per_batch;
        const int64_t b = u / U;
        const int64_t r = u - b * U;
        const int64_t s = r / (KT + 2);
        const int64_t o = r - s * (KT + 2);
        int64_t P, start, j0;
        if (o < KT - 2 * s) {
            P = s;                                   // first pair of the row
            start = s * (KT + 2);
            j0 = o;
        } else {
            P = PPB - 1 - s;                         // second pair of the row
            start = s * (KT + 2) + (KT - 2 * s);
            j0 = o - (KT - 2 * s);
        }
        sg.tile_m = static_cast<int>(b * PPB + P);
        sg.kt0 = static_cast<int>(2 * P + j0);
        sg.T = min(p.key_tiles - sg.kt0, u_end - u);
        sg.slot = static_cast<int>(blockIdx.x) - static_cast<int>((b * U + start) / p.unit_len);
        u += sg.T;
        return true;
    }
    if (p.band_len == 0) {
        if (u >= u_end) return false;
        sg.tile_m = u / p.key_tiles;
        sg.kt0 = u - sg.tile_m * p.key_tiles;
        sg.T = min(p.key_tiles - sg.kt0, u_end - u);
        sg.slot = static_cast<int>(blockIdx.x) -
                  static_cast<int>(static_cast<int64_t>(sg.tile_m) * p.key_tiles / p.unit_len);
        u += sg.T;
        return true;
    }
    const int r = static_cast<int>(blockIdx.x) + run * static_cast<int>(gridDim.x);
    if (r >= p.nruns) return false;
    const int band = r / p.pairs_total;
    sg.tile_m = r - band * p.pairs_total;
    sg.kt0 = band * p.band_len;
    sg.T = min(p.band_len, p.key_tiles - sg.kt0);
    sg.slot = band;
    ++run;
    return true;
}

// Folded values (VF): per-problem words after the sign records of all
// problems, 1 where every 32-key group of the problem has values of one
// sign (written by vf_flags_kernel).  Pass VF = 1 takes those problems
// (the exponent loop reads no records), pass VF = 2 the others.
template <int VF>
__device__ __forceinline__ bool vf_takes(const FmaParams& p, int tile_m) {
    if (VF == 0 || VF == 3) return true;
    const int problem = tile_m / p.pairs_per_batch;
    const int batch = p.pairs_total / p.pairs_per_batch;
    const unsigned* flags = reinterpret_cast<const unsigned*>(
        p.rec + static_cast<int64_t>(batch) * (p.npad / BN) * (BN + BN / 32));
    return (flags[problem] != 0u) == (VF == 1);
}

__device__ __forceinline__ void exp_warps_sync() {
    asm volatile("bar.sync 1, %0;" ::"r"(NEXP * 32) : "memory");
}

// The OR of v over all exponent warps, and a barrier of theirs: every
// exponent warp gets the same answer (so that they leave their segment
// loop together and never leave one of them waiting at a named barrier).
__device__ __forceinline__ bool exp_warps_any(bool v) {
    unsigned r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, %2, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(v ? 1u : 0u), "r"(NEXP * 32)
        : "memory");
    return r != 0u;
}

// AUG: augmented operands (S = -||q^ - k^||^2 / 2; no norm terms in the
// key records).  QSM: q^ tiles in shared memory (A operand from shared
// memory, SL = 2); otherwise q^ in TMEM (A operand from TMEM, SL = 1).
// TRI: upper-triangle order for v^T K v (q = k, C = 1, augmented
// operands): key tiles past the pair's own two get the weight 2, applied as
// +1 in the exponent.
template <int C, bool AUG, bool QSM, bool TF, bool TRI, int SOFT, bool OVL, int VF>
__global__ void __launch_bounds__(THREADS, 1)
tc_gauss_fma_kernel(const __grid_constant__ CUtensorMap tm_q,
                    const __grid_constant__ CUtensorMap tm_k, const FmaParams p) {
    // TF (3xTF32): q^ in shared memory, norm terms from A and the records.
    static_assert(!TF || (QSM && !AUG), "3xTF32 runs with q^ in shared memory");
    static_assert(!OVL || QSM, "overlapped segments keep q^ in shared memory");
    static_assert(VF == 0 || (AUG && SOFT == 0 && !TF), "folded operands: augmented fp16 rows");
    static_assert(VF != 1 || C == 1, "folded values: one channel");
    static_assert(VF != 2 || C == 1, "folded values: one channel");
    static_assert(SOFT == 0 || (AUG && !TRI), "FMA-pipe exponentials: augmented operands");
    constexpr int kSoftMask = soft_mask(SOFT);
    constexpr int REC_PAIR = (AUG ? 0 : 2) + 2 * C;   // floats per key pair
    constexpr int SL = QSM ? 2 : 1;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + (((raw_addr + 1023u) & ~1023u) - raw_addr);
    uint8_t* q_smem = smem;                            // QSM: NQ x nkb x 16 KB
    uint8_t* stage0 = smem + p.q_bytes;
    float* red = reinterpret_cast<float*>(smem + p.red_offset);    // NPART x 256 x C
    FmaBarriers* bars = reinterpret_cast<FmaBarriers*>(smem + p.red_offset + NPART * NQ * BM * C * 4);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    volatile int* abort_flag = &bars->abort_flag;

    pdl_trigger();
    if (VF == 2) {
        // The second folded-value pass often has nothing to do (every problem
        // of the call went to the first): a CTA none of whose segments is of
        // this pass leaves before allocating tensor memory.  (The flags come
        // from an earlier launch, hence the wait first.)
        pdl_wait();
        const int ub = static_cast<int>(blockIdx.x) * p.unit_len;
        const int ue = p.units < ub + p.unit_len ? p.units : ub + p.unit_len;
        int u = ub, run = 0;
        Segment sg;
        bool any = false;
        while (!any && next_segment<TRI>(p, ue, u, run, sg)) any = vf_takes<VF>(p, sg.tile_m);
        if (!any) return;   // uniform over the block: every thread reads the same flags
    }
    if (tid == 0) bars->abort_flag = 0;
    if (warp == CTRL_WARP0) {
        tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    const uint32_t qa_col = static_cast<uint32_t>(2 * SL * BN);   // TMEM q^ (not QSM)

    auto kh_smem = [&](int s) { return stage0 + s * p.stage_bytes; };
    auto rec_smem = [&](int s) {
        return reinterpret_cast<const float*>(stage0 + s * p.stage_bytes + p.kh_bytes);
    };

    // The CTA's work is a sequence of segments (next_segment): consecutive
    // key tiles of one pair of query tiles.  The barriers are initialised
    // once and keep running across segments: every stage, slot and phase
    // follows the CTA-local running tile index g (tiles of all earlier
    // segments plus the index within the segment), and qa_ready completes
    // once per segment.  Each segment writes its partial sums to its slot.
    if (tid == 0) {
        mbar_init(&bars->qa_ready, QSM ? 1 : NEXP);
        mbar_init(&bars->q_free, NCTRL_MAX);
        mbar_init(&bars->stall, 1);
        for (int k = 0; k < NCTRL_MAX; ++k) mbar_init(&bars->drain[k], 1);
        for (int sl = 0; sl < SL; ++sl) {
            mbar_init(&bars->s_full[sl], 1);
            mbar_init(&bars->s_free[sl], NEXP);        // one arrival per exponent warp
        }
        for (int s = 0; s < p.stages; ++s) {
            mbar_init(&bars->kv_full[s], 1);
            mbar_init(&bars->kv_empty[s], 1 + NEXP);  // MMA commit + exponent warps
        }
        fence_mbar_init();
    }
    __syncthreads();
    // The prologue above may overlap the previous kernel of the call; its
    // outputs (operands, key records) are read only from here on.
    pdl_wait();
    // Unit indices fit in 32 bits (the plan checks units < 2^31).
    const int u_begin = static_cast<int>(blockIdx.x) * p.unit_len;
    const int u_end = p.units < u_begin + p.unit_len ? p.units : u_begin + p.unit_len;
    // Segment barrier of both role loops (a non-aligned barrier, since the
    // two roles reach it from different loops).
    // Segment end of both role loops (not OVL; a non-aligned barrier, since
    // the two roles reach it from different loops), with the OR of the
    // threads' abort observations: all roles leave the loop together.
    auto segment_sync_any = [&](bool v) -> bool {
        tc_fence_before();
        unsigned r;
        asm volatile(
            "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
            "barrier.red.or.pred q, 2, %2, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
            : "=r"(r)
            : "r"(v ? 1u : 0u), "r"(THREADS)
            : "memory");
        tc_fence_after();
        return r != 0u;
    };
    if (warp >= CTRL_WARP0) {
        // Control warps need few registers; the exponent warps take them
        // (16 x 32 x kExpRegs + 4 x 32 x kCtrlRegs <= 640 x 96 at launch).
        reg_dealloc<kCtrlRegs>();
        // The lane that issues this warp's copies, MMAs and commits (the
        // warp is converged here; the same lane for the whole kernel).
        const bool leader = elect_one();
        bool issued = false;       // this warp has issued MMAs (warp-uniform)
        uint32_t seg_parity = 0;   // parity of the qa_ready phase of this segment
        int u = u_begin, run = 0, g0 = 0;   // g0: running index of the segment's first tile
        Segment sg;
        for (; next_segment<TRI>(p, u_end, u, run, sg); ) {
        // Segments of the other folded-value pass are skipped, and the
        // running tile index and the q^ phase count only this pass's tiles.
        if (!vf_takes<VF>(p, sg.tile_m)) continue;
        // (Not OVL: the abort decision is taken at the segment-end barrier.)
        if (OVL && __any_sync(0xffffffffu, *abort_flag != 0)) break;
        const int tile_m = sg.tile_m;         // query tiles 2 tile_m, 2 tile_m + 1
        // First k^ row of this pair's problem (batch-stacked operands).
        const int kbase = (tile_m / p.pairs_per_batch) * p.npad;
        const int kt0 = sg.kt0;
        const int T = sg.T;

            // ------------------------------------------------ control warps
            // Control warp k (on SMSP k) owns shared-memory stage k and the key
            // tiles with running index g = k (mod nctrl): it loads their keys and
            // records and issues their MMAs, so that the MMA issue work is spread over the
            // SMSPs instead of slowing the exponent warps of one of them.  The
            // whole warp runs the loop (warp-uniform operands); the elected lane
            // issues copies, MMAs and commits.
            const int k = warp - CTRL_WARP0;
            const int nctrl = p.stages;
            // This warp's tiles: running index g = g0 + j with g = k (mod nctrl).
            const int j_first = (k - g0 % nctrl + nctrl) % nctrl;
            const bool has_tiles = k < nctrl && j_first < T;
            bool ok = true;
            if (OVL && k == 0 && g0 > 0) {
                // q^ of this segment overwrites that of the previous one once
                // every MMA that read it is complete (q_free of the previous
                // segment), while the exponent warps may still be working on
                // that segment's last tiles.
                ok = warp_wait(&bars->q_free, seg_parity ^ 1u, abort_flag, p.status);
            }
            const bool q_issued = QSM && k == 0 && ok;   // warp-uniform
            if (q_issued && leader) {
                // q^ of this segment.
                tma_prefetch_desc(&tm_q);
                mbar_arrive_expect_tx(&bars->qa_ready, p.q_bytes);
                for (int h = 0; h < NQ; ++h)
                    for (int kb = 0; kb < p.nkb; ++kb)
                        tma_load_2d(q_smem + (h * p.nkb + kb) * (BM * 128), &tm_q, &bars->qa_ready,
                                    kb * p.kb_elems, (tile_m * NQ + h) * BM);
            }
            __syncwarp();
            if (has_tiles && ok) {
                auto load_keys = [&](int j) {
                    mbar_arrive_expect_tx(&bars->kv_full[k], p.kh_bytes + p.rec_bytes);
                    const int n0 = kbase + (kt0 + j) * BN;
                    for (int kb = 0; kb < p.nkb; ++kb)
                        tma_load_2d(kh_smem(k) + kb * (BN * 128), &tm_k, &bars->kv_full[k],
                                    kb * p.kb_elems, n0);
                    bulk_load(const_cast<float*>(rec_smem(k)),
                              p.rec + ((VF == 1 || VF == 2) ? static_cast<int64_t>(n0 / BN) * (BN + BN / 32)
                                          : static_cast<int64_t>(n0 / 2) * REC_PAIR),
                              p.rec_bytes, &bars->kv_full[k]);
                };
                // Parity of stage k's barriers for tile j: stage k completes once
                // per tile g = k (mod nctrl).
                uint32_t ph = static_cast<uint32_t>((g0 + j_first) / nctrl) & 1u;
                // OVL: the stage's previous tile (the last one of an earlier
                // segment) is released here rather than waited for at the end
                // of that segment, so that the next segment's loads and MMAs
                // overlap the exponent work on the last tiles.
                if (OVL && g0 + j_first >= nctrl)
                    ok = warp_wait(&bars->kv_empty[k], ph ^ 1u, abort_flag, p.status);
                if (leader && ok) {
                    tma_prefetch_desc(&tm_k);
                    load_keys(j_first);
                }
                __syncwarp();
                if (ok) ok = warp_wait(&bars->qa_ready, seg_parity, abort_flag, p.status);
                // Test hook (status word 6 set by the host): control warp 0 of
                // CTA 0 waits on a barrier that nothing arrives on, so its
                // bounded wait runs out and every role takes the abort path.
                if (ok && k == 0 && blockIdx.x == 0 && g0 == 0 &&
                    *reinterpret_cast<volatile unsigned*>(p.status + kDevStallRequest) != 0u)
                    ok = warp_wait(&bars->stall, 0, abort_flag, p.status);
                const int ksteps = p.ksteps;
                // Shared-memory descriptors of stage k and of q^ tile 0; query
                // tile h and K step kk add byte offsets / 16 to the start-address
                // field.
                const uint64_t kdesc = smem_desc_kmajor_sw128(smem_u32(kh_smem(k)));
                const uint64_t qdesc0 = smem_desc_kmajor_sw128(smem_u32(q_smem));
                const uint32_t qdesc_h = static_cast<uint32_t>((p.nkb * BM * 128) >> 4);
                const uint32_t a0 = tmem + qa_col, a1 = a0 + (p.Dp / 2);
                bool pending = ok;            // keys of tile j requested, not yet waited for
                int j = j_first;
                for (; ok && j < T; j += nctrl, ph ^= 1u) {
                    // S slot of tile j and the parities of its barriers: s_full
                    // completes once per tile of the slot, and tile g reuses the
                    // slot that tile g - SL released.
                    const int g = g0 + j;
                    const int sl = SL == 2 ? (g & 1) : 0;
                    const uint32_t full_parity = static_cast<uint32_t>(SL == 2 ? (g >> 1) : g) & 1u;
                    const uint32_t free_parity = full_parity ^ 1u;
                    const bool ready = __all_sync(
                        0xffffffffu, g < SL ? mbar_test_wait(&bars->kv_full[k], ph)
                                            : mbar_test_wait2(&bars->s_free[sl], free_parity,
                                                              &bars->kv_full[k], ph));
                    if (!ready) {
                        if (g >= SL) {
                            ok = warp_wait(&bars->s_free[sl], free_parity, abort_flag, p.status);
                            if (!ok) break;
                        }
                        ok = warp_wait(&bars->kv_full[k], ph, abort_flag, p.status);
                        if (!ok) break;
                    }
                    pending = false;
                    tc_fence_after();
                    const uint32_t d0 = tmem + sl * (2 * BN), d1 = d0 + BN;
                    if (leader && TF) {
                        // 3xTF32: per K step of 8 coordinates (32 bytes),
                        // hi.lo + lo.hi + hi.hi; the lo blocks follow the
                        // hi blocks (nkb / 2 of each).
                        const uint32_t klo = static_cast<uint32_t>((p.nkb / 2) * (BN * 128 / 16));
                        const uint32_t qlo = static_cast<uint32_t>((p.nkb / 2) * (BM * 128 / 16));
                        for (int h = 0; h < NQ; ++h) {
                            for (int kk = 0; kk < ksteps; ++kk) {
                                const uint32_t step = static_cast<uint32_t>((kk & 3) * 2);
                                const uint64_t kd = kdesc + (kk >> 2) * (BN * 128 / 16) + step;
                                const uint64_t qd = qdesc0 + h * qdesc_h + (kk >> 2) * (BM * 128 / 16) + step;
                                const uint32_t d = h ? d1 : d0;
                                mma_ss_tf32(d, qd, kd + klo, p.idesc, kk > 0 ? 1u : 0u);
                                mma_ss_tf32(d, qd + qlo, kd, p.idesc, 1u);
                                mma_ss_tf32(d, qd, kd, p.idesc, 1u);
                            }
                        }
                        mma_commit(&bars->s_full[sl]);
                        mma_commit(&bars->kv_empty[k]);
                        if (OVL && j + nctrl >= T) mma_commit(&bars->q_free);
                    } else if (leader) {
                        for (int h = 0; h < NQ; ++h) {
                            for (int kk = 0; kk < ksteps; ++kk) {
                                const uint32_t koff = static_cast<uint32_t>((kk >> 2) * (BN * 128 / 16) + (kk & 3) * 2);
                                if (QSM) {
                                    const uint32_t qoff = h * qdesc_h + static_cast<uint32_t>((kk >> 2) * (BM * 128 / 16) + (kk & 3) * 2);
                                    mma_ss_f16(h ? d1 : d0, qdesc0 + qoff, kdesc + koff, p.idesc, kk > 0 ? 1u : 0u);
                                } else {
                                    mma_ts_f16(h ? d1 : d0, (h ? a1 : a0) + kk * 8, kdesc + koff, p.idesc,
                                               kk > 0 ? 1u : 0u);
                                }
                            }
                        }
                        mma_commit(&bars->s_full[sl]);
                        mma_commit(&bars->kv_empty[k]);
                        // OVL, the warp's last tile of the segment: q_free
                        // arrives once these MMAs, and so all of this warp's
                        // MMAs that read the segment's q^, are complete.
                        if (OVL && j + nctrl >= T) mma_commit(&bars->q_free);
                    }
                    __syncwarp();
                    issued = true;
                    // Stage k is free again once these MMAs and the exponent
                    // warps are done with tile j.  OVL: the release of a
                    // segment's last tile on this stage is waited for when the
                    // stage is next loaded (above); otherwise the segment ends
                    // with it.
                    if (!OVL || j + nctrl < T) {
                        ok = warp_wait(&bars->kv_empty[k], ph, abort_flag, p.status);
                        if (!ok) break;
                    }
                    if (j + nctrl < T) {
                        if (leader) load_keys(j + nctrl);
                        __syncwarp();
                        pending = true;
                    }
                }
                // Every copy this warp started must be complete before the
                // CTA moves on: copies still in flight after an abort are
                // waited for here (MMAs in flight after an abort are drained
                // once, before TMEM is freed).  These waits poll per lane, so
                // the warp reconverges after them.
                if (pending) mbar_wait_bounded(&bars->kv_full[k], ph, nullptr, p.status);
                __syncwarp();
            } else if (OVL && ok) {
                // A control warp without tiles in this segment arrives on
                // q_free once the segment's q^ has landed: that orders the
                // arrival after the completion of the previous q_free phase,
                // which the q^ copy waited for.
                ok = warp_wait(&bars->qa_ready, seg_parity, abort_flag, p.status);
                if (leader && ok) mbar_arrive(&bars->q_free);
                __syncwarp();
            }
            if (q_issued) {
                // The q^ copy of this segment must have landed before the
                // CTA moves on (the next segment overwrites q^; after an
                // abort the copy may still be in flight).
                mbar_wait_bounded(&bars->qa_ready, seg_parity, nullptr, p.status);
                __syncwarp();
            }
            // Segment end (not OVL): every MMA, copy and TMEM read of this
            // segment is done (control warps waited for their last stage
            // release and copies).
            if (!OVL && segment_sync_any(*abort_flag != 0)) break;
            seg_parity ^= 1u;
            g0 += sg.T;
        }
        // No MMA of this warp may still run when TMEM is freed.  Without an
        // abort the last stage-release wait has already seen them complete;
        // after an abort a tile's MMAs may still be in flight.  The commit
        // arrives on this warp's own drain barrier once every tcgen05
        // operation the leader issued is done, so the wait ends by itself.
        if (issued) {
            const int k = warp - CTRL_WARP0;
            if (leader) mma_commit(&bars->drain[k]);
            __syncwarp();
            mbar_wait_bounded(&bars->drain[k], 0, nullptr, p.status);
            __syncwarp();
        }
    } else {
        reg_alloc<kExpRegs>();
        uint32_t seg_parity = 0;
        int u = u_begin, run = 0, g0 = 0;
        Segment sg;
        for (; next_segment<TRI>(p, u_end, u, run, sg); ) {
        if (!vf_takes<VF>(p, sg.tile_m)) continue;   // the other folded-value pass
        // (The abort decision is taken at the end of each segment, at a
        // barrier of all exponent warps.)
        const int tile_m = sg.tile_m;         // query tiles 2 tile_m, 2 tile_m + 1
        const int T = sg.T;
        // TRI: tiles j >= w_from of this segment lie past the pair's own two
        // key tiles; their kernel values count twice.
        const int w_from = TRI ? 2 * (tile_m % p.pairs_per_batch) + 2 - sg.kt0 : 0;
        const int slot = sg.slot;

            // ------------------------------------------------ exponent warps
            const int quarter = warp & 3;
            const int cg = warp >> 2;                  // column group: keys 32 cg .. 32 cg + 31
            const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
            const int row_t = quarter * 32 + lane;     // row inside each query tile
            const int64_t row0 = static_cast<int64_t>(tile_m) * NQ * BM + row_t;
            const int64_t row1 = row0 + BM;

            if (!QSM) {
                // q^ rows -> TMEM (A operand).  Column group cg copies query tile
                // cg / 2, 8-column chunks ck = cg % 2 (mod 2) of its Dp / 2 columns.
                const int h = cg >> 1;
                const uint32_t* src = p.qh + (row0 + h * BM) * (p.Dp / 2);
                for (int ck = cg & 1; ck < p.Dp / 16; ck += 2) {
                    const uint4 lo = *reinterpret_cast<const uint4*>(src + ck * 8);
                    const uint4 hi = *reinterpret_cast<const uint4*>(src + ck * 8 + 4);
                    const uint32_t r[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
                    tmem_st_32x32b_x8(tmem + lane_base + qa_col + h * (p.Dp / 2) + ck * 8, r);
                }
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&bars->qa_ready);
            }

            // Row terms of the exponent (only without augmented operands).
            const float am0 = AUG ? 0.f : p.A[row0];
            const float am1 = AUG ? 0.f : p.A[row1];
            const uint64_t a2_0 = f32x2_pack(am0, am0);
            const uint64_t a2_1 = f32x2_pack(am1, am1);
            const uint64_t c2 = f32x2_pack(p.c, p.c);
            const float s_min = -127.0f / p.c;   // exp2_fma_x2 range limit
            uint64_t acc0[C], acc1[C];
    #pragma unroll
            for (int cc = 0; cc < C; ++cc) acc0[cc] = acc1[cc] = 0ull;
            bool ok = true;
            bool ready = false;   // both barriers of key tile j already seen complete
            RingPos st, sl;       // stage and TMEM slot of key tile j (running index g0 + j)
            st.idx = g0 % p.stages;
            st.phase = static_cast<uint32_t>(g0 / p.stages) & 1u;
            sl.idx = g0 % SL;
            sl.phase = static_cast<uint32_t>(g0 / SL) & 1u;
            // The key-tile loop; FAST (folded values, pass 1): every 32-key
            // group of the problem has values of one sign, and the exponent
            // loop reads no records.  (One kernel holding both versions of the
            // loop measured 3 % slower on the fast one than a kernel with the
            // fast one alone.)
            auto tile_loop = [&](auto fast_tag) {
                constexpr bool FAST = decltype(fast_tag)::value;
                for (int j = 0; j < T; ++j, st.advance(p.stages), sl.advance(SL)) {
                    const int s = st.idx;
                    const uint32_t col0 = static_cast<uint32_t>(sl.idx * 2 * BN);
                    if (!__all_sync(0xffffffffu, ready || mbar_test_wait2(&bars->kv_full[s], st.phase,
                                                                          &bars->s_full[sl.idx], sl.phase))) {
                        ok = warp_wait(&bars->kv_full[s], st.phase, abort_flag, p.status);
                        if (ok) ok = warp_wait(&bars->s_full[sl.idx], sl.phase, abort_flag, p.status);
                        if (!ok) break;
                    }
                    tc_fence_after();
                    uint32_t r0[32], r1[32];
                    tmem_ld_32x32b_x32(tmem + lane_base + col0 + cg * 32, r0);
                    tmem_ld_32x32b_x32(tmem + lane_base + col0 + BN + cg * 32, r1);
                    // The wait names r0 and r1, so that no use of the loaded
                    // values is scheduled above it (the loads land asynchronously).
                    tmem_wait_ld_regs(r0, r1);
                    // When and where the S slot is handed back: with two slots
                    // (q^ in shared memory) only after the exponent work of this
                    // tile (with the stage, below), because releasing it right
                    // after the loads let the next MMAs into the slot corrupt S
                    // values of this tile in some warps when the MMAs were long
                    // (measured with 3xTF32 operands and three or more stages,
                    // also with the loads' registers named in the wait; the early
                    // release was no faster on the 65536^2, D = 64 sum either:
                    // 0.6428 against 0.6418 ms).
                    // With one slot (q^ in TMEM) a late release would serialise
                    // the MMAs and the exponent work, so it is released here; no
                    // corruption was seen there in repeated runs (regression
                    // test: repeated calls agree bit for bit).
                    if (!QSM) {
                        tc_fence_before();
                        __syncwarp();
                        mbar_arrive_if_zero(&bars->s_free[sl.idx], lane);
                    }
                    // Query the barriers of key tile j + 1 now and read the answer
                    // after the exponent work of tile j: the query latency overlaps
                    // the arithmetic instead of stalling all exponent warps at once.
                    // A phase seen complete stays complete until this warp releases
                    // that stage and slot.  Two slots only: with one, tile j + 1
                    // needs the slot this warp has just handed back, so the query
                    // would always fail (and skipping it measured 4 % faster on
                    // the D = 256, 1M-key workload).  Not with 3xTF32 operands
                    // either: their three MMAs per K step make the next tile rarely
                    // ready this early (skipping the query: fp32 65536^2 sums 4-5 %
                    // faster).
                    if (QSM && !TF) {
                        RingPos st2 = st, sl2 = sl;
                        st2.advance(p.stages);
                        sl2.advance(SL);
                        ready = j + 1 < T && mbar_test_wait2(&bars->kv_full[st2.idx], st2.phase,
                                                             &bars->s_full[sl2.idx], sl2.phase);
                    }
                    const float* rec = rec_smem(s) + (cg * 16) * REC_PAIR;
                    const uint64_t w2 = (TRI && j >= w_from) ? f32x2_pack(1.f, 1.f) : 0ull;
                    if constexpr (FAST) {
                        // Folded values, every group of this problem of one sign:
                        // P = Phi |v| 2^-16 from the MMA's exponent, times this
                        // column group's sign word +-2^16; no per-key records.
                        const float uw = rec_smem(s)[BN + cg];
                        const uint64_t u2 = f32x2_pack(uw, uw);
        #pragma unroll
                        for (int t = 0; t < 16; ++t) {
                            float x0, x1, y0, y1;
                            const uint64_t sx = f32x2_pack(__uint_as_float(r0[2 * t]), __uint_as_float(r0[2 * t + 1]));
                            const uint64_t sy = f32x2_pack(__uint_as_float(r1[2 * t]), __uint_as_float(r1[2 * t + 1]));
                            f32x2_unpack(TRI ? f32x2_add(sx, w2) : sx, x0, x1);   // the operands carry c
                            f32x2_unpack(TRI ? f32x2_add(sy, w2) : sy, y0, y1);
                            const uint64_t px = f32x2_pack(TRI ? ex2_approx(x0) : ex2_nonpos(x0),
                                                           TRI ? ex2_approx(x1) : ex2_nonpos(x1));
                            const uint64_t py = f32x2_pack(TRI ? ex2_approx(y0) : ex2_nonpos(y0),
                                                           TRI ? ex2_approx(y1) : ex2_nonpos(y1));
                            acc0[0] = f32x2_fma(px, u2, acc0[0]);
                            acc1[0] = f32x2_fma(py, u2, acc1[0]);
                        }
                    } else if (AUG) {
                        // Augmented operands: S = -||q^ - k^||^2 / 2, so Phi = 2^(c S)
                        // (VF: Phi |v| 2^-16, the records holding the signs 2^16).
                        // Keys 32 cg + 2t and + 1, rows row0 (S0) and row1 (S1).
        #pragma unroll
                        for (int t = 0; t < 16; ++t) {
                            const float* pr = rec + t * REC_PAIR;
                            uint64_t px, py;
                            if (SOFT > 0 && (t & kSoftMask) == 0) {
                                px = exp2_fma_x2(__uint_as_float(r0[2 * t]), __uint_as_float(r0[2 * t + 1]), c2, s_min);
                            } else {
                                float x0, x1;
                                const uint64_t sx = f32x2_pack(__uint_as_float(r0[2 * t]), __uint_as_float(r0[2 * t + 1]));
                                f32x2_unpack(VF != 0 ? (TRI ? f32x2_add(sx, w2) : sx)
                                                      : (TRI ? f32x2_fma(sx, c2, w2) : f32x2_mul(sx, c2)),
                                             x0, x1);
                                px = f32x2_pack(TRI ? ex2_approx(x0) : ex2_nonpos(x0),
                                                TRI ? ex2_approx(x1) : ex2_nonpos(x1));
                            }
                            {
                                float y0, y1;
                                const uint64_t sy = f32x2_pack(__uint_as_float(r1[2 * t]), __uint_as_float(r1[2 * t + 1]));
                                f32x2_unpack(VF != 0 ? (TRI ? f32x2_add(sy, w2) : sy)
                                                      : (TRI ? f32x2_fma(sy, c2, w2) : f32x2_mul(sy, c2)),
                                             y0, y1);
                                py = f32x2_pack(TRI ? ex2_approx(y0) : ex2_nonpos(y0),
                                                TRI ? ex2_approx(y1) : ex2_nonpos(y1));
                            }
        #pragma unroll
                            for (int cc = 0; cc < C; ++cc) {
                                const float2 vc = *reinterpret_cast<const float2*>(pr + 2 * cc);
                                const uint64_t vv = f32x2_pack(vc.x, vc.y);
                                acc0[cc] = f32x2_fma(px, vv, acc0[cc]);
                                acc1[cc] = f32x2_fma(py, vv, acc1[cc]);
                            }
                        }
                    } else {
        #pragma unroll
                    for (int t = 0; t < 16; ++t) {
                        // Keys 32 cg + 2t and + 1, rows row0 (S0) and row1 (S1).
                        const float* pr = rec + t * REC_PAIR;
                        float2 bb, v0;
                        if (C == 1) {
                            const float4 bv = *reinterpret_cast<const float4*>(pr);
                            bb = make_float2(bv.x, bv.y);
                            v0 = make_float2(bv.z, bv.w);
                        } else {
                            bb = *reinterpret_cast<const float2*>(pr);
                            v0 = *reinterpret_cast<const float2*>(pr + 2);
                        }
                        const uint64_t b2 = f32x2_pack(bb.x, bb.y);
                        const uint64_t x01 = f32x2_fma(f32x2_pack(__uint_as_float(r0[2 * t]), __uint_as_float(r0[2 * t + 1])),
                                                       c2, f32x2_add(b2, a2_0));
                        const uint64_t y01 = f32x2_fma(f32x2_pack(__uint_as_float(r1[2 * t]), __uint_as_float(r1[2 * t + 1])),
                                                       c2, f32x2_add(b2, a2_1));
                        float x0, x1, y0, y1;
                        f32x2_unpack(x01, x0, x1);
                        f32x2_unpack(y01, y0, y1);
                        const uint64_t px = f32x2_pack(ex2_nonpos(x0), ex2_nonpos(x1));
                        const uint64_t py = f32x2_pack(ex2_nonpos(y0), ex2_nonpos(y1));
                        const uint64_t vv0 = f32x2_pack(v0.x, v0.y);
                        acc0[0] = f32x2_fma(px, vv0, acc0[0]);
                        acc1[0] = f32x2_fma(py, vv0, acc1[0]);
        #pragma unroll
                        for (int cc = 1; cc < C; ++cc) {
                            const float2 vc = *reinterpret_cast<const float2*>(pr + 2 + 2 * cc);
                            const uint64_t vv = f32x2_pack(vc.x, vc.y);
                            acc0[cc] = f32x2_fma(px, vv, acc0[cc]);
                            acc1[cc] = f32x2_fma(py, vv, acc1[cc]);
                        }
                    }
                    }
                    tc_fence_before();
                    __syncwarp();
                    // Lane 0 hands back the slot (two-slot path) and the stage,
                    // predicated rather than branched: a divergent branch here
                    // cost 0.7 % of the kernel time.
                    if (QSM) mbar_arrive2_if_zero(&bars->s_free[sl.idx], &bars->kv_empty[s], lane);
                    else mbar_arrive_if_zero(&bars->kv_empty[s], lane);
                }
            };
            tile_loop(std::integral_constant<bool, VF == 1>{});
            // Fixed-order reduction of the NPART column-group partial sums.
            // (The reduction area of the previous segment has been read by
            // every warp: they met at its end.)
    #pragma unroll
            for (int cc = 0; cc < C; ++cc) {
                float lo, hi;
                f32x2_unpack(acc0[cc], lo, hi);
                red[(cg * NQ * BM + row_t) * C + cc] = lo + hi;
                f32x2_unpack(acc1[cc], lo, hi);
                red[(cg * NQ * BM + BM + row_t) * C + cc] = lo + hi;
            }
            exp_warps_sync();
            if (cg < NQ && T > 0 && *abort_flag == 0) {
                // Column group cg writes the rows of query tile cg.
                const int rt = cg * BM + row_t;
                float* out = p.part + (static_cast<int64_t>(slot) * p.Mpad + row0 + cg * BM) * C;
    #pragma unroll
                for (int cc = 0; cc < C; ++cc) {
                    float sum = 0.f;
    #pragma unroll
                    for (int q = 0; q < NPART; ++q) sum += red[(q * NQ * BM + rt) * C + cc];
                    out[cc] = sum;
                }
            }
        // Segment end: every exponent warp is done with the reduction area;
        // not OVL also every MMA, copy and TMEM read of the segment (with q^
        // in TMEM, before the exponent warps copy the next q^).  The abort
        // decision is the same for all warps that meet here.
        if (OVL ? exp_warps_any(*abort_flag != 0) : segment_sync_any(*abort_flag != 0)) break;
        seg_parity ^= 1u;
        g0 += sg.T;
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == CTRL_WARP0) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

size_t align1k(size_t x) { return (x + 1023) & ~static_cast<size_t>(1023); }

// Floats per key pair in the key records: (B_2t, B_2t+1 unless the norms
// are folded into augmented operands) + both keys' values.
int rec_pair_floats(int C, bool aug) { return (aug ? 0 : 2) + 2 * C; }

// Key-record bytes of one key tile (VF: the signs and four group words).
size_t rec_bytes_for(int C, bool aug, bool vf) {
    return vf ? static_cast<size_t>(BN + BN / 32) * 4
              : static_cast<size_t>(BN / 2) * rec_pair_floats(C, aug) * 4;
}

size_t stage_bytes_for(int nkb, int C, bool aug, bool vf = false) {
    return align1k(static_cast<size_t>(nkb) * BN * 128 + rec_bytes_for(C, aug, vf));
}

size_t fixed_bytes_for(int C, size_t q_bytes) {
    return 1024 /*alignment slack*/ + q_bytes + static_cast<size_t>(NPART) * NQ * BM * C * 4 +
           sizeof(FmaBarriers) + 64;
}

// 128-byte K blocks of an operand row: 16-bit elements, or (TF) the hi and
// lo fp32 halves of Dp columns each.
int nkb_for(int Dp, bool tf) { return tf ? 2 * ((Dp + 31) / 32) : (Dp + KB - 1) / KB; }

// Shared-memory bytes of the q^ tiles when they live in shared memory.
size_t q_bytes_for(int nkb, bool qsm) {
    return qsm ? static_cast<size_t>(NQ) * nkb * BM * 128 : 0;
}

template <int C, bool AUG, bool QSM, bool TF, bool TRI = false, int SOFT = 0, bool OVL = false,
          int VF = 0>
cudaError_t launch_typed(const TcPlan& pl, InType t, float c, char* ws, unsigned* status,
                         cudaStream_t s, const char** why) {
    const CUtensorMapDataType hdt =
        TF ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
           : t == InType::BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    // Row elements and bytes: Dp 16-bit values, or (TF) 2 Dp floats.
    const uint64_t row_el = TF ? 2ull * pl.Dp : static_cast<uint64_t>(pl.Dp);
    const uint64_t row_bytes = TF ? row_el * 4 : row_el * 2;
    const uint32_t kb_elems = TF ? 32u : static_cast<uint32_t>(KB);
    CUtensorMap tm_q, tm_k;
    if (!encode_tile_map_2d(&tm_k, hdt, ws + pl.off_kh, row_el, pl.Npad * pl.batch, row_bytes, kb_elems, BN) ||
        !encode_tile_map_2d(&tm_q, hdt, ws + pl.off_qh, row_el, pl.Mpad * pl.batch, row_bytes, kb_elems, BM)) {
        *why = "cuTensorMapEncodeTiled failed or is unavailable";
        return cudaErrorInvalidValue;
    }
    FmaParams p;
    p.qh = reinterpret_cast<const uint32_t*>(ws + pl.off_qh);
    p.A = AUG ? nullptr : reinterpret_cast<const float*>(ws + pl.off_A);
    p.rec = reinterpret_cast<const float*>(ws + pl.off_rec);
    p.part = reinterpret_cast<float*>(ws + pl.off_part);
    p.status = status;
    p.Mpad = pl.Mpad * pl.batch;   // partial-sum rows per contributor slot
    p.key_tiles = static_cast<int>(pl.Npad / BN);
    p.pairs_per_batch = static_cast<int>(pl.Mpad / (NQ * BM));
    p.npad = static_cast<int>(pl.Npad);
    p.units = static_cast<int>(pl.units);
    p.unit_len = static_cast<int>(pl.unit_len);
    p.band_len = pl.band_len;
    p.nruns = static_cast<int>(pl.tri ? pl.tri_units : pl.nruns);
    p.pairs_total = static_cast<int>((pl.Mpad / (NQ * BM)) * pl.batch);
    p.Dp = pl.Dp;
    p.nkb = nkb_for(pl.Dp, TF);
    p.kb_elems = static_cast<int>(kb_elems);
    p.ksteps = TF ? static_cast<int>(std::max<int64_t>(1, (pl.D + 7) / 8)) : pl.Dp / 16;
    p.stages = pl.stages;
    p.q_bytes = static_cast<uint32_t>(q_bytes_for(p.nkb, QSM));
    p.kh_bytes = static_cast<uint32_t>(p.nkb * BN * 128);
    p.rec_bytes = static_cast<uint32_t>(rec_bytes_for(C, AUG, VF == 1 || VF == 2));
    p.stage_bytes = static_cast<uint32_t>(stage_bytes_for(p.nkb, C, AUG, VF == 1 || VF == 2));
    p.red_offset = p.q_bytes + static_cast<uint32_t>(pl.stages * p.stage_bytes);
    p.c = c;
    const uint32_t hb = t == InType::BF16 ? 1u : 0u;
    p.idesc = TF ? idesc_tf32(BM, BN) : idesc_f16(BM, BN, hb, hb);
    cudaError_t e = cudaFuncSetAttribute(tc_gauss_fma_kernel<C, AUG, QSM, TF, TRI, SOFT, OVL, VF>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(pl.smem_bytes));
    if (e != cudaSuccess) return e;
    dim3 grid(static_cast<unsigned>(pl.grid));
    launch_kernel(tc_gauss_fma_kernel<C, AUG, QSM, TF, TRI, SOFT, OVL, VF>, grid, THREADS, pl.smem_bytes, s, tm_q, tm_k, p);
    note_launches(1);
    return cudaGetLastError();
}

template <int C>
cudaError_t launch_c(const TcPlan& pl, InType t, float c, char* ws, unsigned* status,
                     cudaStream_t s, const char** why, int vf_pass) {
    if (pl.tf) return launch_typed<C, false, true, true>(pl, t, c, ws, status, s, why);
    // Folded operands (template parameter VF): 1 / 2 = folded values, the
    // pass of the problems whose groups all share a sign / of the others;
    // 3 = only the exponent scale folded, value records as usual.
    const int vf = pl.vfold ? vf_pass : pl.cfold ? 3 : 0;
    if constexpr (C == 1 && kAugQsm) {
        if (pl.tri && pl.aug) {
            switch (vf) {
                case 1: return launch_typed<1, true, true, false, true, 0, false, 1>(pl, t, c, ws, status, s, why);
                case 2: return launch_typed<1, true, true, false, true, 0, false, 2>(pl, t, c, ws, status, s, why);
                case 3: return launch_typed<1, true, true, false, true, 0, false, 3>(pl, t, c, ws, status, s, why);
                default: return launch_typed<1, true, true, false, true>(pl, t, c, ws, status, s, why);
            }
        }
        if (pl.aug && vf == 1)
            return launch_typed<1, true, true, false, false, 0, false, 1>(pl, t, c, ws, status, s, why);
        if (pl.aug && vf == 2)
            return launch_typed<1, true, true, false, false, 0, false, 2>(pl, t, c, ws, status, s, why);
        if (pl.aug && pl.exp2_fma > 0) {
            switch (pl.exp2_fma) {
                case 1: return launch_typed<1, true, true, false, false, 1>(pl, t, c, ws, status, s, why);
                case 2: return launch_typed<1, true, true, false, false, 2>(pl, t, c, ws, status, s, why);
                case 3: return launch_typed<1, true, true, false, false, 3>(pl, t, c, ws, status, s, why);
                default: return launch_typed<1, true, true, false, false, 4>(pl, t, c, ws, status, s, why);
            }
        }
    }
    if (pl.aug && kAugQsm && pl.overlap) {
        if (vf == 3) return launch_typed<C, true, true, false, false, 0, true, 3>(pl, t, c, ws, status, s, why);
        return launch_typed<C, true, true, false, false, 0, true>(pl, t, c, ws, status, s, why);
    }
    if (pl.aug && vf == 3)
        return launch_typed<C, true, kAugQsm, false, false, 0, false, 3>(pl, t, c, ws, status, s, why);
    if (pl.aug) return launch_typed<C, true, kAugQsm, false>(pl, t, c, ws, status, s, why);
    return launch_typed<C, false, false, false>(pl, t, c, ws, status, s, why);
}

}  // namespace

bool plan_fma_kernel(int Dp, int C, bool aug, bool tf, int* nq, int* stages, size_t* smem) {
    if (C < 1 || C > kFmaMaxChannels || Dp > 256) return false;
    if (aug && Dp > kAugMaxDp) return false;
    if (tf && (aug || Dp > kTf32MaxDp)) return false;
    // TMEM: q^ in TMEM needs Dp columns beside one slot of two S buffers.
    const bool qsm = tf || (aug && kAugQsm);
    if (!qsm && static_cast<int>(TMEM_COLS) - 2 * BN < Dp) return false;
    const int nkb = nkb_for(Dp, tf);
    const size_t budget = 232448;
    const size_t stage = stage_bytes_for(nkb, C, aug);
    const size_t fixed = fixed_bytes_for(C, q_bytes_for(nkb, qsm));
    if (fixed >= budget) return false;
    // Control warp k owns stage k (stages = control warps) and checks the
    // S-slot release of key tile j - SL before the MMAs of tile j.  An
    // mbarrier parity test is only unambiguous while the barrier is at most
    // one phase behind the phase it asks about; the warp knows every key
    // tile up to j - stages is done (its previous stage release), and the
    // slot's previous phase is tile j - 2 SL, so stages <= 2 SL.
    const int sl = qsm ? 2 : 1;
    const int st = static_cast<int>(
        std::min<size_t>(std::min(MAX_STAGES, 2 * sl), (budget - fixed) / stage));
    if (st < 2) return false;
    *nq = NQ;
    *stages = st;
    *smem = std::max<size_t>(fixed + st * stage, 118 * 1024);
    return true;
}

cudaError_t launch_tc_fma(const TcPlan& p, InType t, float c, char* ws, unsigned* status,
                          cudaStream_t s, const char** why, int vf_pass) {
    const bool qsm = p.tf || (p.aug && kAugQsm);
    note_fma_variant((p.aug && kAugQsm && p.overlap && !p.tri && p.exp2_fma == 0 ? 1 : 0) |
                     (p.band_len > 0 ? 2 : 0) | (qsm ? 0 : 4) |
                     (p.vfold ? 8 : 0) | (p.cfold || p.vfold ? 16 : 0));
    switch (p.Cv) {
        case 1: return launch_c<1>(p, t, c, ws, status, s, why, vf_pass);
        case 2: return launch_c<2>(p, t, c, ws, status, s, why, vf_pass);
        case 3: return launch_c<3>(p, t, c, ws, status, s, why, vf_pass);
        default: return launch_c<4>(p, t, c, ws, status, s, why, vf_pass);
    }
}

}  // namespace gs
