// C ABI of the Gauss-sum library: argument checks, workspace handling,
// kernel sequencing and error reporting.  See include/gauss_sum.h.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <atomic>
#include <mutex>

#include "gauss_sum.h"
#include "gauss_sum_testing.h"
#include "internal.h"
#include "ptx.cuh"

namespace {

thread_local char g_last_error[512] = "no error";
std::atomic<uint64_t> g_launches{0};
std::atomic<int> g_last_fma_variant{-1};

gs_status fail(gs_status st, const char* fmt, const char* detail = nullptr) {
    if (detail)
        std::snprintf(g_last_error, sizeof(g_last_error), fmt, detail);
    else
        std::snprintf(g_last_error, sizeof(g_last_error), "%s", fmt);
    return st;
}

gs_status cuda_fail(cudaError_t e, const char* where) {
    char buf[256];
    std::snprintf(buf, sizeof(buf), "%s: %s", where, cudaGetErrorString(e));
    return fail(e == cudaErrorMemoryAllocation ? GS_ERR_OUT_OF_MEMORY : GS_ERR_CUDA, "%s", buf);
}

// Device status word: a kernel that gives up a bounded wait records the
// reason here; gauss_sum_device_status() reads and clears it.
// Device status word and, after a timeout, where the first wait gave up.
__device__ unsigned g_device_status[8];

constexpr int kMaxDevices = 64;
std::mutex g_dev_mu;
unsigned* g_status_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};
int g_is_sm103[kMaxDevices] = {};  // 0 unknown, 1 yes, 2 no

cudaError_t device_info(int* dev, unsigned** status) {
    cudaError_t e = cudaGetDevice(dev);
    if (e != cudaSuccess) return e;
    if (*dev < 0 || *dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_dev_mu);
    if (!g_status_ptr[*dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_device_status);
        if (e != cudaSuccess) return e;
        int sms = 0, major = 0, minor = 0;
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, *dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, *dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, *dev);
        g_sm_count[*dev] = sms > 0 ? sms : 1;
        g_is_sm103[*dev] = (major == 10 && minor == 3) ? 1 : 2;
        g_status_ptr[*dev] = static_cast<unsigned*>(p);
    }
    *status = g_status_ptr[*dev];
    return cudaSuccess;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Workspaces come from a stream-ordered memory pool of the library's own,
// one per device, which keeps up to kPoolKeepBytes of freed workspace
// mapped between calls (the device's default pool gives freed memory back to
// the driver at every synchronisation, so that a caller who synchronises
// between calls would pay a new mapping per call).
constexpr uint64_t kPoolKeepBytes = uint64_t(1) << 30;
cudaMemPool_t g_pool[kMaxDevices] = {};

cudaError_t workspace_pool(int dev, cudaMemPool_t* pool) {
    std::lock_guard<std::mutex> lk(g_dev_mu);
    if (!g_pool[dev]) {
        cudaMemPoolProps props = {};
        props.allocType = cudaMemAllocationTypePinned;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        cudaMemPool_t p = nullptr;
        cudaError_t e = cudaMemPoolCreate(&p, &props);
        if (e != cudaSuccess) return e;
        uint64_t keep = kPoolKeepBytes;
        e = cudaMemPoolSetAttribute(p, cudaMemPoolAttrReleaseThreshold, &keep);
        if (e != cudaSuccess) {
            cudaMemPoolDestroy(p);
            return e;
        }
        g_pool[dev] = p;
    }
    *pool = g_pool[dev];
    return cudaSuccess;
}

// Stream-ordered allocation from the library's pool of the current device.
cudaError_t pool_alloc(void** ptr, size_t bytes, cudaStream_t s) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    cudaMemPool_t pool = nullptr;
    e = workspace_pool(dev, &pool);
    if (e != cudaSuccess) return e;
    return cudaMallocFromPoolAsync(ptr, bytes, pool, s);
}

struct Call {
    const void* q;
    const void* k;
    const void* v;
    double tau;
    int64_t M, N, D, C;
    gs_dtype dtype;
    bool grad;
    float* out;    // M x C (forward) or M x D (grad)
    float* s_out;  // grad only, M x C, nullable
    cudaStream_t stream;
    gs_options opt;
    int64_t B = 1;  // problems of a batch: q B x M x D, k B x N x D, v B x N x C, out B x M x ..
    // Gradient mode: v holds the key weights w (N x C; float32 when w_f32,
    // else the input dtype) and u the weights of the query rows that the C
    // channels are contracted with (M x C; float32 when u_f32; null: ones).
    // out (M x D) may be null when only s_out is wanted.
    bool w_f32 = false;
    const void* u = nullptr;
    bool u_f32 = false;
    // Only v^T out is wanted (q = k, C = 1): the FMA kernel may evaluate the
    // upper triangle of tile pairs, and out then holds row sums s' with
    // sum_m v_m s'_m = v^T K v instead of K v.
    bool tri = false;
    // Weighted vector-Jacobian pass (gradient mode with C = 1 and v null):
    // the kernel values are multiplied by the pair weights
    // w_mn = sum_c r[m, c] k[n, c] of wc channels, r = rw (M x wc, float32
    // when rw_f32, else the input dtype) and k = kw (N x wc, likewise); the
    // value channels are the unit-weight group (k^_n, 1).
    int wc = 0;
    const void* rw = nullptr;
    bool rw_f32 = false;
    const void* kw = nullptr;
    bool kw_f32 = false;
};

// Padded weight channels of a weighted pass (the kernel's instances).
int weight_channels(int64_t wc) { return wc <= 2 ? 2 : wc <= 4 ? 4 : 8; }

gs_status validate(const Call& c) {
    if (c.dtype != GS_FP32 && c.dtype != GS_FP16 && c.dtype != GS_BF16)
        return fail(GS_ERR_INVALID_ARGUMENT, "unknown dtype");
    if (c.M < 0 || c.N < 0 || c.D < 0 || c.C < 0 || c.B < 0)
        return fail(GS_ERR_INVALID_ARGUMENT, "negative size");
    if (!(std::isfinite(c.tau) && c.tau > 0.0))
        return fail(GS_ERR_INVALID_ARGUMENT, "tau must be finite and > 0");
    const bool any = c.B > 0;   // an empty batch reads and writes nothing
    if (!c.grad && any && c.M > 0 && c.C > 0 && !c.out)
        return fail(GS_ERR_INVALID_ARGUMENT, "null output pointer");
    if (any && c.M > 0 && c.D > 0 && !c.q) return fail(GS_ERR_INVALID_ARGUMENT, "null q pointer");
    if (any && c.N > 0 && c.D > 0 && !c.k) return fail(GS_ERR_INVALID_ARGUMENT, "null k pointer");
    if (any && c.N > 0 && c.C > 0 && !c.v && c.wc == 0)
        return fail(GS_ERR_INVALID_ARGUMENT, "null v pointer");
    if (!aligned16(c.q) || !aligned16(c.k) || !aligned16(c.v) || !aligned16(c.out) ||
        !aligned16(c.s_out) || !aligned16(c.u))
        return fail(GS_ERR_INVALID_ARGUMENT, "base pointers must be 16-byte aligned");
    if (c.opt.path == GS_PATH_SIMT && c.dtype != GS_FP32)
        return fail(GS_ERR_UNSUPPORTED, "the SIMT path takes fp32 inputs");
    if (c.opt.path == GS_PATH_TENSOR && c.dtype == GS_FP32 &&
        (c.grad || c.C > gs::kFmaMaxChannels || c.D > gs::kTf32MaxDp))
        return fail(GS_ERR_UNSUPPORTED,
                    "the fp32 tensor-core path takes the forward sum with C <= 4 and D <= 32");
    if (c.opt.path < 0 || c.opt.path > 2) return fail(GS_ERR_INVALID_ARGUMENT, "unknown path");
    if (c.opt.split_n < 0) return fail(GS_ERR_INVALID_ARGUMENT, "split_n must be >= 0");
    if (c.opt.workspace && (reinterpret_cast<uintptr_t>(c.opt.workspace) & 255u))
        return fail(GS_ERR_INVALID_ARGUMENT, "caller workspace must be 256-byte aligned");
    if (c.opt.exp2_fma < 0 || c.opt.exp2_fma > 4)
        return fail(GS_ERR_INVALID_ARGUMENT, "exp2_fma must be 0..4");
    return GS_OK;
}

// Gradient channels on the tensor-core path: the C (D + 1) channels of
// value_prep are split into *n launches of equal width (at most 256, the
// widest value operand of the two-MMA kernel); returns that width.
int64_t grad_chunk(int64_t D, int64_t C, int64_t* n) {
    const int64_t total = std::max<int64_t>(1, C * (D + 1));
    *n = (total + 255) / 256;
    return (total + *n - 1) / *n;
}

gs::InType in_type(gs_dtype d) {
    return d == GS_FP16 ? gs::InType::F16 : d == GS_BF16 ? gs::InType::BF16 : gs::InType::F32;
}

// fp32 inputs go to the tensor cores (3xTF32) when the path is chosen
// explicitly, or automatically for forward sums that the variant covers
// and that are large enough to repay its extra operand kernels (measured
// on a GB300 at D = 16, C = 1: 4096^2 pairs take 0.157 ms through the
// tensor-core path and 0.136 ms through the SIMT kernel; 16384^2 pairs
// 0.197 ms and 0.571 ms).
constexpr int64_t kFp32TensorMinPairs = int64_t(1) << 25;

bool fp32_on_tensor_cores(const Call& c) {
    if (c.opt.path == GS_PATH_TENSOR) return true;
    if (c.opt.path != GS_PATH_AUTO) return false;
    return !c.grad && c.C <= gs::kFmaMaxChannels && c.D <= gs::kTf32MaxDp &&
           c.B * c.M * c.N >= kFp32TensorMinPairs;
}

// Plans the call; returns GS_OK and the workspace size, or an error.
gs_status plan(const Call& c, int sms, bool* tensor, gs::TcPlan* tp, gs::SimtPlan* sp,
               size_t* bytes) {
    const char* why = "unsupported shape";
    *tensor = c.dtype != GS_FP32 || fp32_on_tensor_cores(c);
    if (*tensor) {
        const bool alias = c.q == c.k && c.M == c.N && c.q != nullptr;
        int64_t nch = 1;
        const int64_t width = c.grad ? grad_chunk(c.D, c.C, &nch) : c.C;
        if (!gs::plan_tensor(in_type(c.dtype), c.M, c.N, c.D, width, c.grad, c.opt.center != 0,
                             alias, c.opt.split_n, sms, tp, &why, c.B, c.tri && !c.grad,
                             c.wc > 0 ? weight_channels(c.wc) : 0))
            return fail(GS_ERR_UNSUPPORTED, "%s", why);
        tp->exp2_fma = c.opt.exp2_fma;
        if (tp->exp2_fma > 0 && !(tp->fma && tp->aug && !tp->tri && tp->Cv == 1))
            return fail(GS_ERR_UNSUPPORTED,
                        "exp2_fma needs a forward fp16/bf16 sum with C = 1 on augmented operands");
        // One fp16 value channel on augmented operands: the value magnitudes
        // go into the key operands and the key records keep the signs.  Not
        // for short segments (small problems), where the flag kernel and the
        // second pass of the fused kernel cost more than they save (B = 256
        // problems of 1024 points: 0.135 -> 0.144 ms per call).
        // The exponent scale c folds into the query rows with them (rn(c q^)
        // must stay a normal fp16 number for points of any spread: c <= 1/2,
        // and not far below it: c >= 2^-14).
        const double cx = c.tau * 1.4426950408889634;
        tp->cfold = tp->fma && tp->aug && !tp->tf && c.dtype == GS_FP16 && tp->exp2_fma == 0 &&
                    cx <= 0.5 && cx >= 1.0 / 16384.0;
        tp->vfold = tp->cfold && tp->Cv == 1 && !c.w_f32 && c.C == 1 && !tp->overlap;
        *bytes = tp->total;
    } else {
        if (c.opt.exp2_fma > 0)
            return fail(GS_ERR_UNSUPPORTED,
                        "exp2_fma needs a forward fp16/bf16 sum with C = 1 on augmented operands");
        if (!gs::plan_simt(c.M, c.N, c.D, c.C, c.grad, c.opt.split_n, sms, sp, &why))
            return fail(GS_ERR_UNSUPPORTED, "%s", why);
        *bytes = sp->total;
    }
    return GS_OK;
}

// Records a measurement event; the next kernel then launches without the
// programmatic-serialization attribute (it follows an event, not a kernel).
cudaError_t record_event(void* ev, cudaStream_t s) {
    if (!ev) return cudaSuccess;
    gs::pdl_reset();
    return cudaEventRecord(static_cast<cudaEvent_t>(ev), s);
}

// Test hook (gauss_sum_testing_fail_allocations): workspace allocations
// fail.  A relaxed atomic load per allocating call; nothing else reads it.
std::atomic<int> g_fail_allocations{0};

bool forced_alloc_failure() { return g_fail_allocations.load(std::memory_order_relaxed) != 0; }

gs_status run(Call c) {
    // The first kernel of a call follows whatever the caller queued before.
    gs::pdl_reset();
    gs_status st = validate(c);
    if (st != GS_OK) return st;
    if (c.M == 0 || c.B == 0) return GS_OK;
    if (c.grad && c.D == 0) c.out = nullptr;   // the gradient has no coordinates
    if (c.grad ? !(c.out || c.s_out) : c.C == 0) return GS_OK;

    if (c.N == 0 || c.C == 0) {
        // No keys, or no weight channels (gradient): every sum is empty.
        cudaError_t e = cudaSuccess;
        const int64_t out_w = c.grad ? c.D : c.C;
        if (c.out && out_w > 0)
            e = cudaMemsetAsync(c.out, 0, sizeof(float) * c.B * c.M * out_w, c.stream);
        if (e == cudaSuccess && c.grad && c.s_out && c.C > 0)
            e = cudaMemsetAsync(c.s_out, 0, sizeof(float) * c.B * c.M * c.C, c.stream);
        return e == cudaSuccess ? GS_OK : cuda_fail(e, "cudaMemsetAsync");
    }

    int dev = 0;
    unsigned* status = nullptr;
    cudaError_t e = device_info(&dev, &status);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
    bool tensor = false;
    gs::TcPlan tp{};
    gs::SimtPlan sp{};
    size_t bytes = 0;
    st = plan(c, g_sm_count[dev], &tensor, &tp, &sp, &bytes);
    if (st != GS_OK) return st;
    if (tensor && g_is_sm103[dev] != 1)
        return fail(GS_ERR_UNSUPPORTED, "the tensor-core kernel needs an sm_103 (GB300) GPU");
    if (c.B > 1 && !(tensor && tp.fma)) {
        // Only the FMA kernel takes a batch in one launch: the problems of a
        // batch run one after another on the stream.
        const int64_t es = c.dtype == GS_FP32 ? 4 : 2;
        const int64_t ws_ = c.w_f32 ? 4 : es, us = c.u_f32 ? 4 : es;
        const int64_t out_w1 = c.grad ? c.D : c.C;
        for (int64_t b = 0; b < c.B; ++b) {
            Call cb = c;
            cb.B = 1;
            cb.q = static_cast<const char*>(c.q) + b * c.M * c.D * es;
            cb.k = static_cast<const char*>(c.k) + b * c.N * c.D * es;
            cb.v = static_cast<const char*>(c.v) + b * c.N * c.C * ws_;
            if (c.u) cb.u = static_cast<const char*>(c.u) + b * c.M * c.C * us;
            if (c.out) cb.out = c.out + b * c.M * out_w1;
            if (c.s_out) cb.s_out = c.s_out + b * c.M * c.C;
            st = run(cb);
            if (st != GS_OK) return st;
        }
        return GS_OK;
    }
    const int batch = static_cast<int>(tp.batch > 0 ? tp.batch : 1);

    char* ws = static_cast<char*>(c.opt.workspace);
    bool owned = false;
    if (ws) {
        if (c.opt.workspace_bytes < bytes)
            return fail(GS_ERR_OUT_OF_MEMORY, "caller workspace is smaller than gauss_sum_workspace_size()");
    } else if (bytes > 0) {
        if (forced_alloc_failure()) return fail(GS_ERR_OUT_OF_MEMORY, "workspace allocation failed (test hook)");
        e = pool_alloc(reinterpret_cast<void**>(&ws), bytes, c.stream);
        if (e != cudaSuccess) return cuda_fail(e, "workspace allocation");
        owned = true;
    }

    const double log2e = 1.4426950408889634;
    const float cexp = static_cast<float>(c.tau * log2e);
    const float half_c = static_cast<float>(0.5 * c.tau * log2e);
    const char* why = "";
    const char* where = "kernel launch";
    if (tensor) {
        const gs::InType t = in_type(c.dtype);
        float* mu = (tp.center && c.D > 0) ? reinterpret_cast<float*>(ws + tp.off_mu) : nullptr;
        // Key records of the FMA kernel with augmented operands depend on the
        // values only: the mean launch writes them where it can.
        bool records_done = false;
        bool flags_done = false;   // folded values: per-problem flags written by the operand launch
        if (mu) {
            const gs::RecordArgs rec = {c.v, c.w_f32, c.N, tp.Npad, static_cast<int>(tp.Cv),
                                        reinterpret_cast<float*>(ws + tp.off_rec), tp.vfold};
            e = gs::launch_mean(t, c.q, c.k, c.M, c.N, static_cast<int>(c.D), tp.mean_blocks,
                                reinterpret_cast<float*>(ws + tp.off_mean_part), mu, c.stream,
                                batch, (tp.fma && tp.aug) ? &rec : nullptr, &records_done);
            where = "mean kernel";
        }
        const float ninf = -INFINITY;
        if (e != cudaSuccess) {
            // an error: nothing more is launched
        } else if (tp.tf) {
            // 3xTF32 operands: hi / lo tf32 halves and the norm terms.
            e = gs::launch_tf32_split(static_cast<const float*>(c.q), c.M, tp.Mpad,
                                      static_cast<int>(c.D), tp.Dp, mu, half_c,
                                      reinterpret_cast<float*>(ws + tp.off_qh),
                                      reinterpret_cast<float*>(ws + tp.off_A), ninf, c.stream,
                                      batch);
            where = "tf32 split kernel (q)";
            if (e == cudaSuccess && !tp.alias) {
                e = gs::launch_tf32_split(static_cast<const float*>(c.k), c.N, tp.Npad,
                                          static_cast<int>(c.D), tp.Dp, mu, half_c,
                                          reinterpret_cast<float*>(ws + tp.off_kh),
                                          reinterpret_cast<float*>(ws + tp.off_B), ninf,
                                          c.stream, batch);
                where = "tf32 split kernel (k)";
            }
        } else {
            // Centred, rounded operands of q and (unless q is k) k in one
            // launch: augmented rows (norms folded into the MMA), or plain
            // rows with the norm terms A and B.
            e = gs::launch_operands(
                t, tp.aug, c.q, c.M, tp.Mpad, ws + tp.off_qh,
                (tp.aug && tp.alias) ? ws + tp.off_kh : nullptr,
                tp.aug ? nullptr : reinterpret_cast<float*>(ws + tp.off_A),
                !tp.alias, c.k, c.N, tp.Npad, ws + tp.off_kh,
                tp.aug ? nullptr : reinterpret_cast<float*>(ws + tp.off_B), static_cast<int>(c.D),
                tp.Dp, mu, half_c, ninf, c.stream, batch, tp.vfold ? c.v : nullptr,
                (tp.vfold || tp.cfold) ? cexp : 0.f,
                (tp.vfold && records_done) ? reinterpret_cast<float*>(ws + tp.off_rec) : nullptr,
                &flags_done);
            where = tp.aug ? "augmented-operand kernel" : "centre/cast kernel";
        }
        if (e == cudaSuccess && tp.fma) {
            if (!records_done) {
                e = gs::launch_key_records(
                    c.w_f32 ? gs::InType::F32 : t, c.v,
                    tp.aug ? nullptr : reinterpret_cast<const float*>(ws + tp.off_B), c.N,
                    tp.Npad, static_cast<int>(tp.Cv), reinterpret_cast<float*>(ws + tp.off_rec),
                    c.stream, batch, tp.vfold);
                where = "key-record kernel";
            }
            if (e == cudaSuccess && tp.vfold && !flags_done) {
                e = gs::launch_vf_flags(reinterpret_cast<float*>(ws + tp.off_rec), tp.Npad, batch,
                                        c.stream);
                where = "folded-value flag kernel";
            }
            if (e == cudaSuccess) e = record_event(c.opt.main_events[0], c.stream);
            if (e == cudaSuccess) {
                // Folded values: two passes of the fused kernel, for the
                // problems whose 32-key groups all have values of one sign
                // (no record loads) and for the others; each pass skips the
                // other's problems.
                e = gs::launch_tc_fma(tp, t, cexp, ws, status, c.stream, &why, tp.vfold ? 1 : 0);
                if (e == cudaSuccess && tp.vfold)
                    e = gs::launch_tc_fma(tp, t, cexp, ws, status, c.stream, &why, 2);
                where = "fused tensor-core kernel";
            }
            if (e == cudaSuccess) e = record_event(c.opt.main_events[1], c.stream);
            if (e == cudaSuccess) {
                e = gs::launch_finalize_slots(reinterpret_cast<float*>(ws + tp.off_part), tp.Mpad,
                                              c.M, static_cast<int>(tp.Cv), 128 * tp.nq,
                                              tp.Npad / tp.BN, tp.unit_len, c.out, c.stream,
                                              batch, tp.band_len > 0 ? tp.splits : 0,
                                              tp.tri ? tp.Npad / tp.BN : 0);
                where = "finalise kernel";
            }
        } else if (e == cudaSuccess) {
            // Two-MMA kernel, once per chunk of value channels (one chunk for
            // the forward sum; C (D + 1) channels in chunks for gradients).
            const int64_t total = c.grad ? c.C * (c.D + 1) : c.C;
            const int64_t width = tp.Cv;
            float* part = reinterpret_cast<float*>(ws + tp.off_part);
            float* inv = reinterpret_cast<float*>(ws + tp.off_inv);
            for (int64_t ch0 = 0; ch0 < total && e == cudaSuccess; ch0 += width) {
                const int cc = static_cast<int>(std::min(width, total - ch0));
                e = gs::launch_value_prep(t, c.grad, c.w_f32, c.v, c.k, mu, c.N, tp.Npad,
                                          static_cast<int>(c.D), static_cast<int>(c.C),
                                          static_cast<int>(ch0), cc, tp.Cp,
                                          reinterpret_cast<unsigned*>(ws + tp.off_vmax),
                                          ws + tp.off_vt, inv, c.stream);
                where = "value kernel";
                if (e == cudaSuccess && tp.wt > 0) {
                    e = gs::launch_weight_prep(t, c.rw, c.rw_f32, c.M, tp.Mpad, c.kw, c.kw_f32, c.N,
                                               tp.Npad, static_cast<int>(c.wc), tp.wt, tp.BN,
                                               reinterpret_cast<float*>(ws + tp.off_rowf),
                                               reinterpret_cast<float*>(ws + tp.off_colT),
                                               reinterpret_cast<unsigned*>(ws + tp.off_wmax),
                                               c.stream);
                    where = "pair-weight kernel";
                }
                if (e == cudaSuccess && ch0 == 0) e = record_event(c.opt.main_events[0], c.stream);
                if (e == cudaSuccess) {
                    e = gs::launch_tc(tp, t, cexp, ws, status, c.stream, &why);
                    where = "fused tensor-core kernel";
                }
                if (e == cudaSuccess && ch0 + width >= total)
                    e = record_event(c.opt.main_events[1], c.stream);
                if (e == cudaSuccess) {
                    // Rows of the unsplit row tiles have one partial sum.
                    const int64_t main_rows = tp.main_tiles * 128;
                    if (c.grad)
                        e = gs::launch_finalize_points(
                            false, t, c.u_f32, part, tp.splits, tp.Mpad, c.M, tp.Cp, inv, c.q, mu,
                            static_cast<float>(c.tau), static_cast<int>(c.D),
                            static_cast<int>(c.C), static_cast<int>(ch0), cc, c.u, ch0 > 0,
                            c.out, c.s_out, c.stream, main_rows);
                    else
                        e = gs::launch_finalize(part, tp.splits, tp.Mpad, c.M, cc, tp.Cp, inv,
                                                c.out, c.stream, main_rows);
                    where = "finalise kernel";
                }
            }
        }
    } else {
        float* part = reinterpret_cast<float*>(ws + sp.off_part);
        const float* qf = static_cast<const float*>(c.q);
        const float* kf = static_cast<const float*>(c.k);
        const float* vf = static_cast<const float*>(c.v);
        // Forward: one launch over all channels.  Gradient: one launch per
        // weight channel, contracted into out by the finalise kernel.
        const int64_t passes = c.grad ? c.C : 1;
        for (int64_t wc = 0; wc < passes && e == cudaSuccess; ++wc) {
            if (wc == 0) e = record_event(c.opt.main_events[0], c.stream);
            if (e == cudaSuccess)
                e = gs::launch_simt(sp, c.grad, qf, kf, vf, static_cast<int>(c.C),
                                    static_cast<int>(wc), half_c, part, c.stream);
            where = "fp32 kernel";
            if (e == cudaSuccess && wc + 1 == passes) e = record_event(c.opt.main_events[1], c.stream);
            if (e == cudaSuccess) {
                const int G = static_cast<int>(c.D + 1);
                if (c.grad)
                    e = gs::launch_finalize_points(
                        true, gs::InType::F32, true, part, sp.splits, c.M, c.M, G, nullptr,
                        nullptr, nullptr, static_cast<float>(c.tau), static_cast<int>(c.D),
                        static_cast<int>(c.C), static_cast<int>(wc) * G, G, c.u, wc > 0, c.out,
                        c.s_out, c.stream);
                else
                    e = gs::launch_finalize(part, sp.splits, c.M, c.M, static_cast<int>(sp.Cv),
                                            static_cast<int>(sp.Cv), nullptr, c.out, c.stream);
                where = "finalise kernel";
            }
        }
    }
    if (owned) {
        cudaError_t ef = cudaFreeAsync(ws, c.stream);
        if (e == cudaSuccess && ef != cudaSuccess) return cuda_fail(ef, "workspace cudaFreeAsync");
    }
    if (e != cudaSuccess) {
        if (why && why[0]) return fail(GS_ERR_CUDA, "%s", why);
        return cuda_fail(e, where);
    }
    return GS_OK;
}

gs_options defaults() {
    gs_options o;
    o.center = 1;
    o.split_n = 0;
    o.workspace = nullptr;
    o.workspace_bytes = 0;
    o.path = GS_PATH_AUTO;
    o.main_events[0] = nullptr;
    o.main_events[1] = nullptr;
    o.exp2_fma = 0;
    return o;
}

// ---------------------------------------------------------------- ex2 probe
template <int CH>
__global__ void ex2_probe_kernel(float* out, int iters) {
    float x[CH];
#pragma unroll
    for (int i = 0; i < CH; ++i) x[i] = -0.001f * static_cast<float>(threadIdx.x + i);
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < CH; ++i) x[i] = gs::ex2_approx(x[i]) - 1.0f;
    }
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < CH; ++i) s += x[i];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

// The FMA kernel's exponent loop without its tiles: per key pair and two
// query rows two paired multiplies by c (here paired FMAs that also add a
// per-iteration offset, so that no exponential is loop invariant and none
// can be hoisted out of the loop), four ex2.approx (-|x| form), one
// broadcast 8-byte shared-memory load of the pair's values and two paired
// FMAs, on 16 warps per SM (the kernel's exponent warps: four per SMSP), no
// tensor-memory traffic or barriers.  Measures the exp2 rate this
// instruction mix can reach.

constexpr int kMixProbeThreads = 512;

__global__ void __launch_bounds__(kMixProbeThreads, 1) ex2_mix_probe_kernel(float* out, int iters,
                                                                            float c) {
    __shared__ float2 vals[64];
    if (threadIdx.x < 64)
        vals[threadIdx.x] = make_float2(1e-3f * threadIdx.x, -1e-3f * threadIdx.x);
    __syncthreads();
    float s0[16], s1[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        s0[i] = -0.01f * static_cast<float>(threadIdx.x + i);
        s1[i] = -0.02f * static_cast<float>(threadIdx.x + i);
    }
    const uint64_t c2 = gs::f32x2_pack(c, c);
    uint64_t a0 = 0ull, a1 = 0ull;
    float off = 0.f;
    for (int it = 0; it < iters; ++it) {
        off -= 1e-7f;
        const uint64_t o2 = gs::f32x2_pack(off, off);
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            float x0, x1, y0, y1;
            gs::f32x2_unpack(gs::f32x2_fma(gs::f32x2_pack(s0[2 * t], s0[2 * t + 1]), c2, o2), x0, x1);
            gs::f32x2_unpack(gs::f32x2_fma(gs::f32x2_pack(s1[2 * t], s1[2 * t + 1]), c2, o2), y0, y1);
            const uint64_t px = gs::f32x2_pack(gs::ex2_nonpos(x0), gs::ex2_nonpos(x1));
            const uint64_t py = gs::f32x2_pack(gs::ex2_nonpos(y0), gs::ex2_nonpos(y1));
            const float2 v = vals[(t + it) & 63];
            const uint64_t vv = gs::f32x2_pack(v.x, v.y);
            a0 = gs::f32x2_fma(px, vv, a0);
            a1 = gs::f32x2_fma(py, vv, a1);
        }
    }
    float u0, u1, w0, w1;
    gs::f32x2_unpack(a0, u0, u1);
    gs::f32x2_unpack(a1, w0, w1);
    out[blockIdx.x * blockDim.x + threadIdx.x] = u0 + u1 + w0 + w1;
}

}  // namespace

namespace gs {

gs_status forward_workspace_bytes(const void* q, const void* k, const void* v, double tau,
                                  int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype,
                                  float* out, size_t* bytes) {
    Call c{q, k, v, tau, M, N, D, C, dtype, false, out, nullptr, nullptr, defaults()};
    *bytes = 0;
    gs_status st = validate(c);
    if (st != GS_OK) return st;
    if (M == 0 || N == 0 || C == 0) return GS_OK;
    int dev = 0;
    unsigned* status = nullptr;
    cudaError_t e = device_info(&dev, &status);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
    bool tensor = false;
    TcPlan tp{};
    SimtPlan sp{};
    return plan(c, g_sm_count[dev], &tensor, &tp, &sp, bytes);
}

gs_status set_last_error(gs_status st, const char* msg) { return fail(st, "%s", msg); }

void note_launches(int n) { g_launches.fetch_add(static_cast<uint64_t>(n), std::memory_order_relaxed); }
void note_fma_variant(int flags) { g_last_fma_variant.store(flags, std::memory_order_relaxed); }

cudaError_t run_ex2_probe(cudaStream_t s, double* rate, bool mix) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int sms = 1;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // Plain: independent ex2 chains on 64 warps per SM; mix: the FMA
    // kernel's loop on one block of 16 warps per SM.
    const int blocks = mix ? sms : sms * 4, threads = mix ? kMixProbeThreads : 512;
    const int iters = mix ? 2048 : 4096;
    float* out = nullptr;
    e = cudaMallocAsync(reinterpret_cast<void**>(&out), sizeof(float) * blocks * threads, s);
    if (e != cudaSuccess) return e;
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    double best = 0.0;
    for (int rep = 0; rep < 4; ++rep) {
        cudaEventRecord(e0, s);
        if (mix)
            ex2_mix_probe_kernel<<<blocks, threads, 0, s>>>(out, iters, 0.0225f);
        else
            ex2_probe_kernel<8><<<blocks, threads, 0, s>>>(out, iters);
        note_launches(1);
        cudaEventRecord(e1, s);
        e = cudaEventSynchronize(e1);
        if (e != cudaSuccess) break;
        float ms = 0.f;
        cudaEventElapsedTime(&ms, e0, e1);
        const double n = static_cast<double>(blocks) * threads * iters * (mix ? 32 : 8);
        if (rep > 0 && ms > 0.f) best = std::max(best, n / (ms * 1e-3));
    }
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    cudaFreeAsync(out, s);
    cudaError_t e2 = cudaStreamSynchronize(s);
    *rate = best;
    return e != cudaSuccess ? e : e2;
}
}  // namespace gs

extern "C" {

void gauss_sum_default_options(gs_options* opt) {
    if (opt) *opt = defaults();
}

gs_status gauss_sum_ex(const void* q, const void* k, const void* v, double tau, int64_t M,
                       int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out, void* stream,
                       const gs_options* opt) {
    Call c{q, k, v, tau, M, N, D, C, dtype, false, out, nullptr,
           static_cast<cudaStream_t>(stream), opt ? *opt : defaults()};
    return run(c);
}

gs_status gauss_sum(const void* q, const void* k, const void* v, double tau, int64_t M,
                    int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out, void* stream) {
    return gauss_sum_ex(q, k, v, tau, M, N, D, C, dtype, out, stream, nullptr);
}

gs_status gauss_sum_batched(const void* q, const void* k, const void* v, double tau, int64_t B,
                            int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype, float* out,
                            void* stream) {
    Call c{q, k, v, tau, M, N, D, C, dtype, false, out, nullptr,
           static_cast<cudaStream_t>(stream), defaults()};
    c.B = B;
    return run(c);
}

gs_status gauss_sum_mmd2(const void* x, const void* v, double tau, int64_t B, int64_t N,
                         int64_t D, gs_dtype dtype, float* mmd2, void* stream) {
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (B < 0 || N < 0 || D < 0) return fail(GS_ERR_INVALID_ARGUMENT, "negative size");
    if (B > 0 && !mmd2) return fail(GS_ERR_INVALID_ARGUMENT, "null output pointer");
    if (!aligned16(mmd2)) return fail(GS_ERR_INVALID_ARGUMENT, "base pointers must be 16-byte aligned");
    if (B == 0) return GS_OK;
    if (N == 0) {
        cudaError_t e = cudaMemsetAsync(mmd2, 0, sizeof(float) * B, st);
        return e == cudaSuccess ? GS_OK : cuda_fail(e, "cudaMemsetAsync");
    }
    // s = K v for every problem (q = k = x), then v^T s.  The arguments are
    // validated with mmd2 standing in for the s buffer allocated below.  The
    // FMA kernel (fp16 / bf16, augmented operands) evaluates only the upper
    // triangle of tile pairs (K is symmetric): s then holds row sums s' with
    // v^T s' = v^T K v, at half the exponentials.
    Call c{x, x, v, tau, N, N, D, 1, dtype, false, mmd2, nullptr, st, defaults()};
    c.B = B;
    c.tri = true;
    gs_status status = validate(c);
    if (status != GS_OK) return status;
    if (forced_alloc_failure()) return fail(GS_ERR_OUT_OF_MEMORY, "workspace allocation failed (test hook)");
    float* s_buf = nullptr;
    // s (B x N float32), then the float64 chunk partials of the reduction.
    const size_t s_bytes = (sizeof(float) * B * N + 255) & ~static_cast<size_t>(255);
    cudaError_t e = pool_alloc(reinterpret_cast<void**>(&s_buf),
                                    s_bytes + gs::mmd2_partial_bytes(B, N), st);
    if (e != cudaSuccess) return cuda_fail(e, "workspace allocation");
    c.out = s_buf;
    status = run(c);
    if (status == GS_OK) {
        e = gs::launch_mmd2_reduce(in_type(dtype), s_buf, v, B, N,
                                   reinterpret_cast<double*>(reinterpret_cast<char*>(s_buf) + s_bytes),
                                   mmd2, st);
        if (e != cudaSuccess) status = cuda_fail(e, "MMD reduction kernel");
    }
    cudaError_t ef = cudaFreeAsync(s_buf, st);
    if (status == GS_OK && ef != cudaSuccess) return cuda_fail(ef, "cudaFreeAsync");
    return status;
}

gs_status gauss_sum_grad_q_ex(const void* q, const void* k, const void* v, double tau,
                              int64_t M, int64_t N, int64_t D, gs_dtype dtype, float* grad,
                              float* s_out, void* stream, const gs_options* opt) {
    Call c{q, k, v, tau, M, N, D, 1, dtype, true, grad, s_out,
           static_cast<cudaStream_t>(stream), opt ? *opt : defaults()};
    if (M > 0 && D > 0 && !grad) return fail(GS_ERR_INVALID_ARGUMENT, "null output pointer");
    return run(c);
}

gs_status gauss_sum_vjp(const void* q, const void* k, const void* v, const float* g, double tau,
                        int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype,
                        float* grad_q, float* grad_k, float* grad_v, void* stream) {
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    // dL/dq: queries q, keys k weighted by v, contracted with g.
    Call a{q, k, v, tau, M, N, D, C, dtype, true, grad_q, nullptr, st, defaults()};
    a.u = g;
    a.u_f32 = true;
    // dL/dk and dL/dv: queries k, keys q weighted by g, contracted with v;
    // the unweighted channel of each group is dL/dv.
    Call b{k, q, g, tau, N, M, D, C, dtype, true, grad_k, grad_v, st, defaults()};
    b.w_f32 = true;
    b.u = v;
    b.u_f32 = dtype == GS_FP32;
    if (M > 0 && C > 0 && !g) return fail(GS_ERR_INVALID_ARGUMENT, "null g pointer");
    gs_status status = validate(a);
    if (status == GS_OK) status = validate(b);
    if (status != GS_OK) return status;
    if (C >= 2 && C <= 8 && dtype != GS_FP32 && D >= 1 && D + 1 <= 128) {
        // Weighted single pass per side: with the pair weights
        // w_mn = g_m . v_n folded into the kernel values,
        //   grad_q[m] = tau (sum_n Phi w k^_n - q^_m sum_n Phi w)
        //   grad_k[n] = tau (sum_m Phi w q^_m - k^_n sum_m Phi w)
        // are Gauss sums of the D + 1 unit-weight channels (x^, 1), and
        // grad_v[n] = sum_m Phi_mn g_m is the forward sum with the values g.
        Call wa{q, k, nullptr, tau, M, N, D, 1, dtype, true, grad_q, nullptr, st, defaults()};
        wa.wc = static_cast<int>(C);
        wa.rw = g;
        wa.rw_f32 = true;
        wa.kw = v;
        Call wb{k, q, nullptr, tau, N, M, D, 1, dtype, true, grad_k, nullptr, st, defaults()};
        wb.wc = static_cast<int>(C);
        wb.rw = v;
        wb.kw = g;
        wb.kw_f32 = true;
        Call wv{k, q, g, tau, N, M, D, C, dtype, false, grad_v, nullptr, st, defaults()};
        wv.w_f32 = true;
        status = validate(wa);
        if (status == GS_OK) status = validate(wb);
        if (status == GS_OK && grad_v) status = validate(wv);
        if (status != GS_OK) return status;
        if (grad_q) status = run(wa);
        if (status == GS_OK && grad_k) status = run(wb);
        if (status == GS_OK && grad_v) status = run(wv);
        return status;
    }
    if (grad_q) status = run(a);
    if (status == GS_OK && (grad_k || grad_v)) status = run(b);
    return status;
}

gs_status gauss_sum_grad_q(const void* q, const void* k, const void* v, double tau, int64_t M,
                           int64_t N, int64_t D, gs_dtype dtype, float* grad, float* s_out,
                           void* stream) {
    return gauss_sum_grad_q_ex(q, k, v, tau, M, N, D, dtype, grad, s_out, stream, nullptr);
}

size_t gauss_sum_workspace_size(int64_t M, int64_t N, int64_t D, int64_t C, gs_dtype dtype,
                                int grad, const gs_options* opt) {
    const gs_options o = opt ? *opt : defaults();
    // Distinct stand-in pointers: the size returned covers q and k being
    // different arrays (an aliased call needs less).
    static const char dummy[64] __attribute__((aligned(16))) = {0};
    Call c{dummy, dummy + 16, dummy + 32, 1.0, M, N, D, grad ? 1 : C, dtype, grad != 0,
           reinterpret_cast<float*>(const_cast<char*>(dummy + 48)), nullptr, nullptr, o};
    c.opt.workspace = nullptr;
    if (validate(c) != GS_OK) return static_cast<size_t>(-1);
    if (M == 0 || N == 0) return 0;
    int sms = 152;
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess) {
        int s = 0;
        if (cudaDeviceGetAttribute(&s, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && s > 0) sms = s;
    } else {
        cudaGetLastError();
    }
    bool tensor = false;
    gs::TcPlan tp{};
    gs::SimtPlan sp{};
    size_t bytes = 0;
    if (plan(c, sms, &tensor, &tp, &sp, &bytes) != GS_OK) return static_cast<size_t>(-1);
    return bytes;
}

gs_status gauss_sum_device_status(void* stream) {
    int dev = 0;
    unsigned* status = nullptr;
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    e = device_info(&dev, &status);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
    unsigned v[8] = {0};
    e = cudaMemcpy(v, status, sizeof(v), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "status read");
    const unsigned zero[8] = {0};
    e = cudaMemcpy(status, zero, sizeof(zero), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "status clear");
    if (v[0] == gs::kDevTimeout) {
        char where[160];
        std::snprintf(where, sizeof(where),
                      "block (%u, %u), warp %u, barrier at shared address %u, parity %u", v[1],
                      v[2], v[3], v[4], v[5]);
        return fail(GS_ERR_DEVICE_TIMEOUT, "a device-side wait ran out of time: %s", where);
    }
    return GS_OK;
}

const char* gauss_sum_last_error(void) { return g_last_error; }

const char* gauss_sum_status_string(gs_status s) {
    switch (s) {
        case GS_OK: return "GS_OK";
        case GS_ERR_INVALID_ARGUMENT: return "GS_ERR_INVALID_ARGUMENT";
        case GS_ERR_UNSUPPORTED: return "GS_ERR_UNSUPPORTED";
        case GS_ERR_OUT_OF_MEMORY: return "GS_ERR_OUT_OF_MEMORY";
        case GS_ERR_CUDA: return "GS_ERR_CUDA";
        case GS_ERR_DEVICE_TIMEOUT: return "GS_ERR_DEVICE_TIMEOUT";
    }
    return "unknown status";
}

uint64_t gauss_sum_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

int gauss_sum_testing_last_fma_variant(void) { return g_last_fma_variant.load(std::memory_order_relaxed); }

void gauss_sum_testing_fail_allocations(int on) {
    g_fail_allocations.store(on ? 1 : 0, std::memory_order_relaxed);
}

gs_status gauss_sum_testing_request_stall(void* stream) {
    int dev = 0;
    unsigned* status = nullptr;
    cudaError_t e = device_info(&dev, &status);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
    static const unsigned one = 1u;
    e = cudaMemcpyAsync(status + gs::kDevStallRequest, &one, sizeof(one), cudaMemcpyHostToDevice,
                        static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "stall request");
    e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? GS_OK : cuda_fail(e, "stall request");
}

gs_status gauss_sum_probe_ex2_rate(void* stream, double* exp2_per_second) {
    if (!exp2_per_second) return fail(GS_ERR_INVALID_ARGUMENT, "null output pointer");
    cudaError_t e = gs::run_ex2_probe(static_cast<cudaStream_t>(stream), exp2_per_second, false);
    if (e != cudaSuccess) return cuda_fail(e, "ex2 probe");
    return GS_OK;
}

gs_status gauss_sum_probe_ex2_mix_rate(void* stream, double* exp2_per_second) {
    if (!exp2_per_second) return fail(GS_ERR_INVALID_ARGUMENT, "null output pointer");
    cudaError_t e = gs::run_ex2_probe(static_cast<cudaStream_t>(stream), exp2_per_second, true);
    if (e != cudaSuccess) return cuda_fail(e, "ex2 mix probe");
    return GS_OK;
}

}  // extern "C"
