// api.cu -- the C ABI (include/memoroid.h): argument validation, workspace
// checks, launches and device-error read-back.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <map>
#include <mutex>
#include <utility>

#include "internal.cuh"

namespace memoroid {

namespace {
constexpr uint64_t kDefaultWaitNs = 1000000000ull;  // 1 s
std::atomic<uint64_t> g_wait_ns{kDefaultWaitNs};
std::atomic<int64_t> g_withhold{-1};
std::atomic<int> g_lnorm_padded{0};
// Launch counter: bits 0..30 are the launch's tag, the bits above count the
// times the tag has wrapped ("generation").
std::atomic<uint64_t> g_epoch{1};
// Per (device, workspace address): the generation in which this process last
// cleared the workspace's tagged region, and how far that clear reached.
struct Cleared {
    uint64_t generation;
    size_t end;
};
std::mutex g_cleared_mutex;
std::map<std::pair<int, uintptr_t>, Cleared> g_cleared;
constexpr size_t kMaxClearedEntries = 4096;

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }
}  // namespace

DebugKnobs debug_knobs() { return DebugKnobs{g_wait_ns.load(), g_withhold.load(), g_lnorm_padded.load()}; }

EncodeTiledFn encode_tiled() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

uint32_t tagged_epoch(const void* workspace, size_t region_end, cudaStream_t stream, bool* clear) {
    uint64_t c = 0;
    while ((c & 0x7fffffffull) == 0) c = g_epoch.fetch_add(1u);
    // a call captured into a graph replays this tag every time: its region is
    // cleared on every replay, and the registry, which records clears already
    // done, is left as it is (the captured clear has not run)
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cap) != cudaSuccess || cap != cudaStreamCaptureStatusNone) {
        *clear = true;
        return static_cast<uint32_t>(c & 0x7fffffffull);
    }
    const uint64_t generation = c >> 31;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) dev = -1;
    const std::pair<int, uintptr_t> key{dev, reinterpret_cast<uintptr_t>(workspace)};
    std::lock_guard<std::mutex> lock(g_cleared_mutex);
    auto it = g_cleared.find(key);
    *clear = it == g_cleared.end() || it->second.generation != generation || it->second.end < region_end;
    if (*clear) {
        if (it == g_cleared.end() && g_cleared.size() >= kMaxClearedEntries) g_cleared.clear();  // forget, clear again later
        g_cleared[key] = Cleared{generation, region_end};
    }
    return static_cast<uint32_t>(c & 0x7fffffffull);
}

}  // namespace memoroid

using namespace memoroid;

extern "C" {

const char* memoroid_status_string(memoroid_status_t s) {
    switch (s) {
        case MEMOROID_OK: return "ok";
        case MEMOROID_ERR_INVALID_ARG: return "invalid argument";
        case MEMOROID_ERR_UNSUPPORTED: return "unsupported shape or mode";
        case MEMOROID_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case MEMOROID_ERR_CUDA: return "CUDA error";
        case MEMOROID_ERR_TIMEOUT: return "device-side wait timed out";
        case MEMOROID_ERR_BAD_DATA: return "device-side data check failed";
    }
    return "unknown status";
}

int memoroid_version(void) { return 100; }

void memoroid_debug_set_wait_limit_ns(uint64_t ns) { g_wait_ns.store(ns == 0 ? kDefaultWaitNs : ns); }

void memoroid_debug_withhold_tile(int64_t ticket) { g_withhold.store(ticket); }

void memoroid_debug_lnorm_padded(int on) { g_lnorm_padded.store(on != 0 ? 1 : 0); }

memoroid_status_t memoroid_get_device_error(const void* workspace, void* stream) {
    if (workspace == nullptr) return MEMOROID_ERR_INVALID_ARG;
    uint32_t code = 0;
    cudaStream_t s = as_stream(stream);
    if (cudaMemcpyAsync(&code, workspace, sizeof(code), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (code == DEV_OK) return MEMOROID_OK;
    return code == DEV_BAD_DATA ? MEMOROID_ERR_BAD_DATA : MEMOROID_ERR_TIMEOUT;
}

// ---------------------------------------------------------------------------
// diagonal scan
// ---------------------------------------------------------------------------

size_t memoroid_scan_diag_workspace_bytes(int64_t B, int64_t L, int64_t D) {
    if (B < 0 || L < 0 || D < 0 || (D % 2) != 0) return 0;
    return diag::workspace_bytes(B, L, D);
}

int memoroid_scan_diag_kernels_per_call(int64_t B, int64_t L, int64_t D, int lambda_per_step,
                                        int backward, int with_grad_lambda) {
    if (B < 0 || L < 0 || D < 0 || (D % 2) != 0) return -1;
    return diag::kernels_per_call(B, L, D, lambda_per_step != 0, backward != 0, with_grad_lambda != 0);
}

static memoroid_status_t check_ws(int64_t B, int64_t L, int64_t D, const void* ws, size_t bytes) {
    if (ws == nullptr || !aligned(ws, 256)) return MEMOROID_ERR_WORKSPACE;
    if (bytes < diag::workspace_bytes(B, L, D)) return MEMOROID_ERR_WORKSPACE;
    return MEMOROID_OK;
}

memoroid_status_t memoroid_scan_diag_fwd(const void* lambda, int lambda_per_step, const void* u,
                                         const uint8_t* start, const void* h0, void* h,
                                         void* h_last, int64_t B, int64_t L, int64_t D,
                                         void* workspace, size_t workspace_bytes, void* stream) {
    if (B < 0 || L < 0 || D < 0 || (D % 2) != 0) return MEMOROID_ERR_INVALID_ARG;
    if (lambda_per_step != 0 && lambda_per_step != 1) return MEMOROID_ERR_INVALID_ARG;
    const bool work = B > 0 && L > 0 && D > 0;
    if (work) {
        if (!lambda || !u || !start || !h) return MEMOROID_ERR_INVALID_ARG;
        if (!aligned(lambda, 16) || !aligned(u, 16) || !aligned(h, 16)) return MEMOROID_ERR_INVALID_ARG;
    }
    if ((h0 && !aligned(h0, 16)) || (h_last && !aligned(h_last, 16))) return MEMOROID_ERR_INVALID_ARG;
    cudaStream_t s = as_stream(stream);
    if (!work) {
        // empty tape: h_last = h0 (or the identity)
        if (h_last && B > 0 && D > 0) {
            const size_t bytes = static_cast<size_t>(B) * D * 8;
            const cudaError_t e = h0 ? cudaMemcpyAsync(h_last, h0, bytes, cudaMemcpyDeviceToDevice, s)
                                     : cudaMemsetAsync(h_last, 0, bytes, s);
            if (e != cudaSuccess) return MEMOROID_ERR_CUDA;
        }
        return MEMOROID_OK;
    }
    const memoroid_status_t w = check_ws(B, L, D, workspace, workspace_bytes);
    if (w != MEMOROID_OK) return w;
    diag::Args a{};
    a.lambda = lambda;
    a.lambda_per_step = lambda_per_step;
    a.u = u;
    a.start = start;
    a.h0 = h0;
    a.out = h;
    a.out_last = h_last;
    a.B = B;
    a.L = L;
    a.D = D;
    a.workspace = workspace;
    a.workspace_bytes = workspace_bytes;
    return diag::launch_fwd(a, s);
}

memoroid_status_t memoroid_scan_diag_bwd(const void* lambda, int lambda_per_step,
                                         const uint8_t* start, const void* h0, const void* h,
                                         const void* grad_h, const void* grad_h_last, void* grad_u,
                                         void* grad_lambda, void* grad_h0, int64_t B, int64_t L,
                                         int64_t D, void* workspace, size_t workspace_bytes,
                                         void* stream) {
    if (B < 0 || L < 0 || D < 0 || (D % 2) != 0) return MEMOROID_ERR_INVALID_ARG;
    if (lambda_per_step != 0 && lambda_per_step != 1) return MEMOROID_ERR_INVALID_ARG;
    const bool work = B > 0 && L > 0 && D > 0;
    cudaStream_t s = as_stream(stream);
    if ((h0 && !aligned(h0, 16)) || (grad_h_last && !aligned(grad_h_last, 16)) ||
        (grad_lambda && !aligned(grad_lambda, 16)) || (grad_h0 && !aligned(grad_h0, 16)))
        return MEMOROID_ERR_INVALID_ARG;
    if (work) {
        if (!lambda || !start || !h || !grad_h || !grad_u) return MEMOROID_ERR_INVALID_ARG;
        if (!aligned(lambda, 16) || !aligned(h, 16) || !aligned(grad_h, 16) || !aligned(grad_u, 16))
            return MEMOROID_ERR_INVALID_ARG;
        if (grad_u == h) return MEMOROID_ERR_INVALID_ARG;
    }
    if (!work) {
        if (D > 0 && grad_lambda && !lambda_per_step &&
            cudaMemsetAsync(grad_lambda, 0, static_cast<size_t>(D) * 8, s) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
        if (grad_h0 && B > 0 && D > 0) {
            const size_t bytes = static_cast<size_t>(B) * D * 8;
            const cudaError_t e = grad_h_last
                                      ? cudaMemcpyAsync(grad_h0, grad_h_last, bytes, cudaMemcpyDeviceToDevice, s)
                                      : cudaMemsetAsync(grad_h0, 0, bytes, s);
            if (e != cudaSuccess) return MEMOROID_ERR_CUDA;
        }
        return MEMOROID_OK;
    }
    const memoroid_status_t w = check_ws(B, L, D, workspace, workspace_bytes);
    if (w != MEMOROID_OK) return w;
    diag::Args a{};
    a.lambda = lambda;
    a.lambda_per_step = lambda_per_step;
    a.u = grad_h;
    a.start = start;
    a.h0 = h0;
    a.out = grad_u;
    a.h = h;
    a.g_last = grad_h_last;
    a.grad_lambda = grad_lambda;
    a.grad_h0 = grad_h0;
    a.B = B;
    a.L = L;
    a.D = D;
    a.workspace = workspace;
    a.workspace_bytes = workspace_bytes;
    return diag::launch_bwd(a, s);
}

// ---------------------------------------------------------------------------
// episode index list <-> begin flags
// ---------------------------------------------------------------------------

memoroid_status_t memoroid_starts_from_offsets(const int64_t* offsets, int64_t E, int64_t L,
                                               uint8_t* start, void* stream) {
    if (E < 0 || L < 0) return MEMOROID_ERR_INVALID_ARG;
    if ((L > 0 && !start) || (E > 0 && !offsets)) return MEMOROID_ERR_INVALID_ARG;
    return tape::launch_starts_from_offsets(offsets, E, L, start, as_stream(stream));
}

size_t memoroid_offsets_workspace_bytes(int64_t L) {
    if (L < 0) return 0;
    return tape::offsets_workspace_bytes(L);
}

memoroid_status_t memoroid_offsets_from_starts(const uint8_t* start, int64_t L, int64_t* offsets,
                                               int64_t* count, void* workspace,
                                               size_t workspace_bytes, void* stream) {
    if (L < 0 || !count) return MEMOROID_ERR_INVALID_ARG;
    if (L > 0 && (!start || !offsets)) return MEMOROID_ERR_INVALID_ARG;
    if (!aligned(count, 8) || (offsets && !aligned(offsets, 8))) return MEMOROID_ERR_INVALID_ARG;
    if (L > 0) {
        if (!workspace || !aligned(workspace, 256)) return MEMOROID_ERR_WORKSPACE;
        if (workspace_bytes < tape::offsets_workspace_bytes(L)) return MEMOROID_ERR_WORKSPACE;
    }
    return tape::launch_offsets_from_starts(start, L, offsets, count, workspace, workspace_bytes,
                                            as_stream(stream));
}


// ---------------------------------------------------------------------------
// decayed linear attention
// ---------------------------------------------------------------------------

static bool la_shape_ok(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, int64_t chunk) {
    if (B < 0 || L < 0 || H < 0) return false;
    if (dk != dv || (dk != 64 && dk != 128)) return false;
    return chunk == 64 || chunk == 128;
}

size_t memoroid_scan_linattn_workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv,
                                             int64_t chunk) {
    if (!la_shape_ok(B, L, H, dk, dv, chunk)) return 0;
    return la::workspace_bytes(B, L, H, dk);
}

int memoroid_scan_linattn_kernels_per_call(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, int backward,
                                           int with_dgamma_per_head) {
    if (!la_shape_ok(B, L, H, dk, dv, 64)) return -1;
    return la::kernels_per_call(B, L, H, backward != 0, with_dgamma_per_head != 0);
}

memoroid_status_t memoroid_scan_linattn_fwd(const void* q, const void* k, const void* v, int in_dtype,
                                            const float* gamma, int gamma_per_step, const uint8_t* start,
                                            const float* S0, float* y, float* S_last, int64_t B, int64_t L,
                                            int64_t H, int64_t dk, int64_t dv, int64_t chunk, void* workspace,
                                            size_t workspace_bytes, void* stream) {
    if (B < 0 || L < 0 || H < 0 || dk < 0 || dv < 0) return MEMOROID_ERR_INVALID_ARG;
    if (gamma_per_step != 0 && gamma_per_step != 1) return MEMOROID_ERR_INVALID_ARG;
    if (in_dtype != MEMOROID_BF16 && in_dtype != MEMOROID_F32) return MEMOROID_ERR_INVALID_ARG;
    if (!la_shape_ok(B, L, H, dk, dv, chunk) || in_dtype != MEMOROID_BF16) return MEMOROID_ERR_UNSUPPORTED;
    const bool work = B > 0 && L > 0 && H > 0;
    if (work) {
        if (!q || !k || !v || !gamma || !start || !y) return MEMOROID_ERR_INVALID_ARG;
        if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(y, 16) || !aligned(gamma, 4))
            return MEMOROID_ERR_INVALID_ARG;
    }
    if ((S0 && !aligned(S0, 16)) || (S_last && !aligned(S_last, 16))) return MEMOROID_ERR_INVALID_ARG;
    cudaStream_t s = as_stream(stream);
    if (!work) {
        // empty tape: S_last = S0 (or zero)
        if (S_last && B > 0 && H > 0) {
            const size_t bytes = static_cast<size_t>(B * H) * dk * dv * sizeof(float);
            const cudaError_t e = S0 ? cudaMemcpyAsync(S_last, S0, bytes, cudaMemcpyDeviceToDevice, s)
                                     : cudaMemsetAsync(S_last, 0, bytes, s);
            if (e != cudaSuccess) return MEMOROID_ERR_CUDA;
        }
        return MEMOROID_OK;
    }
    if (workspace == nullptr || !aligned(workspace, 256) ||
        workspace_bytes < la::fwd_workspace_bytes(B, L, H, dk))
        return MEMOROID_ERR_WORKSPACE;
    la::Args a{};
    a.q = q;
    a.k = k;
    a.v = v;
    a.gamma = gamma;
    a.gamma_per_step = gamma_per_step;
    a.start = start;
    a.S0 = S0;
    a.y = y;
    a.S_last = S_last;
    a.B = B;
    a.L = L;
    a.H = H;
    a.D = dk;
    a.workspace = workspace;
    a.workspace_bytes = workspace_bytes;
    return la::launch_fwd(a, s);
}

memoroid_status_t memoroid_scan_linattn_bwd(const void* q, const void* k, const void* v, int in_dtype,
                                            const float* gamma, int gamma_per_step, const uint8_t* start,
                                            const float* S0, const float* grad_y, const float* grad_S_last,
                                            float* dq, float* dk_out, float* dv_out, float* dgamma, float* dS0,
                                            int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, int64_t chunk,
                                            void* workspace, size_t workspace_bytes, void* stream) {
    if (B < 0 || L < 0 || H < 0 || dk < 0 || dv < 0) return MEMOROID_ERR_INVALID_ARG;
    if (gamma_per_step != 0 && gamma_per_step != 1) return MEMOROID_ERR_INVALID_ARG;
    if (in_dtype != MEMOROID_BF16 && in_dtype != MEMOROID_F32) return MEMOROID_ERR_INVALID_ARG;
    if (!la_shape_ok(B, L, H, dk, dv, chunk) || in_dtype != MEMOROID_BF16) return MEMOROID_ERR_UNSUPPORTED;
    const bool work = B > 0 && L > 0 && H > 0;
    if (work) {
        if (!q || !k || !v || !gamma || !start || !grad_y || !dq || !dk_out || !dv_out) return MEMOROID_ERR_INVALID_ARG;
        if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(grad_y, 16) || !aligned(dq, 16) ||
            !aligned(dk_out, 16) || !aligned(dv_out, 16) || !aligned(gamma, 4))
            return MEMOROID_ERR_INVALID_ARG;
        if (dgamma && !aligned(dgamma, 4)) return MEMOROID_ERR_INVALID_ARG;
    }
    if ((S0 && !aligned(S0, 16)) || (grad_S_last && !aligned(grad_S_last, 16)) || (dS0 && !aligned(dS0, 16)))
        return MEMOROID_ERR_INVALID_ARG;
    cudaStream_t s = as_stream(stream);
    if (!work) {
        // empty tape: dS0 = grad_S_last (or zero), dgamma = 0
        if (dS0 && B > 0 && H > 0) {
            const size_t bytes = static_cast<size_t>(B * H) * dk * dv * sizeof(float);
            const cudaError_t e = grad_S_last ? cudaMemcpyAsync(dS0, grad_S_last, bytes, cudaMemcpyDeviceToDevice, s)
                                              : cudaMemsetAsync(dS0, 0, bytes, s);
            if (e != cudaSuccess) return MEMOROID_ERR_CUDA;
        }
        if (dgamma && !gamma_per_step && H > 0) {
            if (cudaMemsetAsync(dgamma, 0, static_cast<size_t>(H) * sizeof(float), s) != cudaSuccess)
                return MEMOROID_ERR_CUDA;
        }
        return MEMOROID_OK;
    }
    if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < la::workspace_bytes(B, L, H, dk))
        return MEMOROID_ERR_WORKSPACE;
    la::Args a{};
    a.q = q;
    a.k = k;
    a.v = v;
    a.gamma = gamma;
    a.gamma_per_step = gamma_per_step;
    a.start = start;
    a.S0 = S0;
    a.grad_y = grad_y;
    a.dS_last = grad_S_last;
    a.dq = dq;
    a.dk = dk_out;
    a.dv = dv_out;
    a.dgamma = dgamma;
    a.dS0 = dS0;
    a.B = B;
    a.L = L;
    a.H = H;
    a.D = dk;
    a.workspace = workspace;
    a.workspace_bytes = workspace_bytes;
    return la::launch_bwd(a, s);
}

size_t memoroid_bench_linattn_intra_scratch_bytes(int64_t d) {
    if (d != 64 && d != 128) return 0;
    return la::intra_bench_scratch_bytes(d);
}

memoroid_status_t memoroid_bench_linattn_intra(int64_t d, int64_t reps, int64_t ctas, void* scratch,
                                               size_t scratch_bytes, void* stream) {
    if (d != 64 && d != 128) return MEMOROID_ERR_UNSUPPORTED;
    if (reps < 1 || ctas < 1 || ctas > (1 << 20)) return MEMOROID_ERR_INVALID_ARG;
    if (scratch == nullptr || !aligned(scratch, 256) || scratch_bytes < la::intra_bench_scratch_bytes(d))
        return MEMOROID_ERR_WORKSPACE;
    return la::launch_intra_bench(d, reps, ctas, scratch, as_stream(stream));
}

// ---------------------------------------------------------------------------
// Fast and Forgetful Memory
// ---------------------------------------------------------------------------

static bool ffm_shape_ok(int64_t B, int64_t L, int64_t m, int64_t c) {
    if (B < 0 || L < 0 || m <= 0 || (m % 4) != 0) return false;
    return c == 1 || c == 2 || c == 4 || c == 8 || c == 16;
}

size_t memoroid_ffm_workspace_bytes(int64_t B, int64_t L, int64_t m, int64_t c) {
    if (!ffm_shape_ok(B, L, m, c)) return 0;
    return diag::ffm_workspace_bytes(B, L, m, c);
}

int memoroid_ffm_kernels_per_call(int64_t B, int64_t L, int64_t m, int64_t c, int backward,
                                  int with_param_grads) {
    if (!ffm_shape_ok(B, L, m, c)) return -1;
    return diag::ffm_kernels_per_call(B, L, m, c, backward != 0, with_param_grads != 0);
}

static memoroid_status_t ffm_check_ws(int64_t B, int64_t L, int64_t m, int64_t c, const void* ws, size_t bytes) {
    if (ws == nullptr || !aligned(ws, 256)) return MEMOROID_ERR_WORKSPACE;
    if (bytes < diag::ffm_workspace_bytes(B, L, m, c)) return MEMOROID_ERR_WORKSPACE;
    return MEMOROID_OK;
}

memoroid_status_t memoroid_ffm_fwd(const float* x, const float* alpha, const float* omega, const uint8_t* start,
                                   const void* S0, float* z, void* S_last, int64_t B, int64_t L, int64_t m,
                                   int64_t c, void* workspace, size_t workspace_bytes, void* stream) {
    if (!ffm_shape_ok(B, L, m, c)) return MEMOROID_ERR_INVALID_ARG;
    const bool work = B > 0 && L > 0;
    if ((S0 && !aligned(S0, 16)) || (S_last && !aligned(S_last, 16))) return MEMOROID_ERR_INVALID_ARG;
    cudaStream_t s = as_stream(stream);
    if (!work) {
        // empty tape: S_last = S0 (or e_I = 0)
        if (S_last && B > 0) {
            const size_t bytes = static_cast<size_t>(B) * m * c * 8;
            const cudaError_t e = S0 ? cudaMemcpyAsync(S_last, S0, bytes, cudaMemcpyDeviceToDevice, s)
                                     : cudaMemsetAsync(S_last, 0, bytes, s);
            if (e != cudaSuccess) return MEMOROID_ERR_CUDA;
        }
        return MEMOROID_OK;
    }
    if (!x || !alpha || !omega || !start || !z) return MEMOROID_ERR_INVALID_ARG;
    if (!aligned(x, 16) || !aligned(z, 16) || !aligned(alpha, 4) || !aligned(omega, 4))
        return MEMOROID_ERR_INVALID_ARG;
    const memoroid_status_t w = ffm_check_ws(B, L, m, c, workspace, workspace_bytes);
    if (w != MEMOROID_OK) return w;
    diag::FfmArgs f{};
    f.backward = false;
    f.x = x;
    f.alpha = alpha;
    f.omega = omega;
    f.start = start;
    f.S0 = S0;
    f.z = z;
    f.S_last = S_last;
    f.B = B;
    f.L = L;
    f.m = m;
    f.c = c;
    f.workspace = workspace;
    f.workspace_bytes = workspace_bytes;
    return diag::launch_ffm(f, s);
}

memoroid_status_t memoroid_ffm_bwd(const float* alpha, const float* omega, const uint8_t* start, const void* S0,
                                   const float* z, const float* grad_z, const void* grad_S_last, float* grad_x,
                                   float* grad_alpha, float* grad_omega, void* grad_S0, int64_t B, int64_t L,
                                   int64_t m, int64_t c, void* workspace, size_t workspace_bytes, void* stream) {
    if (!ffm_shape_ok(B, L, m, c)) return MEMOROID_ERR_INVALID_ARG;
    const bool work = B > 0 && L > 0;
    if ((S0 && !aligned(S0, 16)) || (grad_S_last && !aligned(grad_S_last, 16)) || (grad_S0 && !aligned(grad_S0, 16)) ||
        (grad_alpha && !aligned(grad_alpha, 4)) || (grad_omega && !aligned(grad_omega, 4)))
        return MEMOROID_ERR_INVALID_ARG;
    cudaStream_t s = as_stream(stream);
    if (!work) {
        if (grad_alpha && cudaMemsetAsync(grad_alpha, 0, static_cast<size_t>(m) * 4, s) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
        if (grad_omega && cudaMemsetAsync(grad_omega, 0, static_cast<size_t>(c) * 4, s) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
        if (grad_S0 && B > 0) {
            const size_t bytes = static_cast<size_t>(B) * m * c * 8;
            const cudaError_t e = grad_S_last
                                      ? cudaMemcpyAsync(grad_S0, grad_S_last, bytes, cudaMemcpyDeviceToDevice, s)
                                      : cudaMemsetAsync(grad_S0, 0, bytes, s);
            if (e != cudaSuccess) return MEMOROID_ERR_CUDA;
        }
        return MEMOROID_OK;
    }
    if (!alpha || !omega || !start || !z || !grad_z || !grad_x) return MEMOROID_ERR_INVALID_ARG;
    if (static_cast<const void*>(grad_x) == z || static_cast<const void*>(grad_x) == grad_z)
        return MEMOROID_ERR_INVALID_ARG;
    if (!aligned(z, 16) || !aligned(grad_z, 16) || !aligned(grad_x, 16) || !aligned(alpha, 4) || !aligned(omega, 4))
        return MEMOROID_ERR_INVALID_ARG;
    const memoroid_status_t w = ffm_check_ws(B, L, m, c, workspace, workspace_bytes);
    if (w != MEMOROID_OK) return w;
    diag::FfmArgs f{};
    f.backward = true;
    f.alpha = alpha;
    f.omega = omega;
    f.start = start;
    f.S0 = S0;
    f.z = const_cast<float*>(z);
    f.grad_z = grad_z;
    f.grad_S_last = grad_S_last;
    f.grad_x = grad_x;
    f.grad_alpha = grad_alpha;
    f.grad_omega = grad_omega;
    f.grad_S0 = grad_S0;
    f.B = B;
    f.L = L;
    f.m = m;
    f.c = c;
    f.workspace = workspace;
    f.workspace_bytes = workspace_bytes;
    return diag::launch_ffm(f, s);
}

// ---------------------------------------------------------------------------
// the Linear Transformer with phi = 1 + ELU and its normalizer
// ---------------------------------------------------------------------------

static bool lnorm_shape_ok(int64_t B, int64_t L, int64_t H, int64_t d) {
    return B >= 0 && L >= 0 && H >= 0 && d >= 8 && d <= 120 && (d % 8) == 0;
}

size_t memoroid_linattn_norm_workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t d) {
    if (!lnorm_shape_ok(B, L, H, d)) return 0;
    return lnorm::workspace_bytes(B, L, H);
}

int memoroid_linattn_norm_kernels_per_call(int64_t B, int64_t L, int64_t H, int64_t d, int backward,
                                           int with_dgamma_per_head, int with_states) {
    if (!lnorm_shape_ok(B, L, H, d)) return -1;
    return lnorm::kernels_per_call(B, L, H, d, backward != 0, with_dgamma_per_head != 0, with_states != 0);
}

static memoroid_status_t lnorm_common(lnorm::Args& a, const float* gamma, int gamma_per_step, const uint8_t* start,
                                      size_t workspace_bytes, void* stream) {
    if (!lnorm_shape_ok(a.B, a.L, a.H, a.d)) return MEMOROID_ERR_INVALID_ARG;
    if (gamma_per_step != 0 && gamma_per_step != 1) return MEMOROID_ERR_INVALID_ARG;
    if (a.B == 0 || a.L == 0 || a.H == 0) {
        // nothing to scan: the outgoing state is the incoming one (and its gradient passes back)
        cudaStream_t s = as_stream(stream);
        const size_t nS = static_cast<size_t>(a.B * a.H * a.d * a.d) * 4, nz = static_cast<size_t>(a.B * a.H * a.d) * 4;
        auto pass = [&](void* dst, const void* src, size_t bytes) {
            if (dst == nullptr || bytes == 0) return cudaSuccess;
            return src ? cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, s) : cudaMemsetAsync(dst, 0, bytes, s);
        };
        cudaError_t e = cudaSuccess;
        if (!a.backward) {
            if (e == cudaSuccess) e = pass(a.S_last, a.S0, nS);
            if (e == cudaSuccess) e = pass(a.z_last, a.z0, nz);
        } else {
            if (e == cudaSuccess) e = pass(a.dS0, a.dS_last, nS);
            if (e == cudaSuccess) e = pass(a.dz0, a.dz_last, nz);
            if (e == cudaSuccess && a.dgamma != nullptr) {
                const size_t ng = static_cast<size_t>(gamma_per_step ? a.B * a.L * a.H : a.H) * 4;
                if (ng) e = cudaMemsetAsync(a.dgamma, 0, ng, s);
            }
        }
        return e == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
    }
    if (!a.q || !a.k || !a.v || !gamma || !start || !a.y) return MEMOROID_ERR_INVALID_ARG;
    if (!aligned(a.q, 16) || !aligned(a.k, 16) || !aligned(a.v, 16) || !aligned(a.y, 4) || !aligned(gamma, 4))
        return MEMOROID_ERR_INVALID_ARG;
    if (a.backward && (!aligned(a.dq, 16) || !aligned(a.dk, 16) || !aligned(a.dv, 16)))
        return MEMOROID_ERR_INVALID_ARG;
    if (a.B * a.L * a.H * a.d >= (int64_t{1} << 32)) return MEMOROID_ERR_UNSUPPORTED;  // 32-bit element indices
    if (a.workspace == nullptr || !aligned(a.workspace, 256) ||
        workspace_bytes < lnorm::workspace_bytes(a.B, a.L, a.H))
        return MEMOROID_ERR_WORKSPACE;
    a.gamma = gamma;
    a.gamma_per_step = gamma_per_step;
    a.start = start;
    return lnorm::launch(a, as_stream(stream));
}

memoroid_status_t memoroid_linattn_norm_fwd(const void* q, const void* k, const void* v, const float* gamma,
                                            int gamma_per_step, const uint8_t* start, const float* S0,
                                            const float* z0, float* y, float* den, float* S_last, float* z_last,
                                            int64_t B, int64_t L, int64_t H, int64_t d, void* workspace,
                                            size_t workspace_bytes, void* stream) {
    lnorm::Args a{};
    a.backward = false;
    a.q = q;
    a.k = k;
    a.v = v;
    a.S0 = S0;
    a.z0 = z0;
    a.y = y;
    a.den = den;
    a.S_last = S_last;
    a.z_last = z_last;
    a.B = B;
    a.L = L;
    a.H = H;
    a.d = d;
    a.workspace = workspace;
    return lnorm_common(a, gamma, gamma_per_step, start, workspace_bytes, stream);
}

memoroid_status_t memoroid_linattn_norm_bwd(const void* q, const void* k, const void* v, const float* gamma,
                                            int gamma_per_step, const uint8_t* start, const float* S0,
                                            const float* z0, const float* y, const float* den, const float* grad_y,
                                            const float* grad_S_last, const float* grad_z_last, float* dq, float* dk,
                                            float* dv, float* dgamma, float* dS0, float* dz0, int64_t B, int64_t L,
                                            int64_t H, int64_t d, void* workspace, size_t workspace_bytes,
                                            void* stream) {
    if (B > 0 && L > 0 && H > 0 && (!den || !grad_y || !dq || !dk || !dv)) return MEMOROID_ERR_INVALID_ARG;
    lnorm::Args a{};
    a.backward = true;
    a.q = q;
    a.k = k;
    a.v = v;
    a.S0 = S0;
    a.z0 = z0;
    a.y = const_cast<float*>(y);
    a.den = const_cast<float*>(den);
    a.grad_y = grad_y;
    a.dS_last = grad_S_last;
    a.dz_last = grad_z_last;
    a.dq = dq;
    a.dk = dk;
    a.dv = dv;
    a.dgamma = dgamma;
    a.dS0 = dS0;
    a.dz0 = dz0;
    a.B = B;
    a.L = L;
    a.H = H;
    a.d = d;
    a.workspace = workspace;
    return lnorm_common(a, gamma, gamma_per_step, start, workspace_bytes, stream);
}

// ---------------------------------------------------------------------------
// tape-based batching: sampling and row gather
// ---------------------------------------------------------------------------

size_t memoroid_tbb_workspace_bytes(int64_t K) {
    if (K < 0) return 0;
    return tbb::workspace_bytes(K);
}

memoroid_status_t memoroid_tbb_sample(const int64_t* begin, int64_t E, int64_t N, const int64_t* draws, int64_t K,
                                      int64_t B, uint8_t* start, int64_t* src, int64_t* n_used, void* workspace,
                                      size_t workspace_bytes, void* stream) {
    if (E < 0 || N < 0 || K < 0 || B < 0) return MEMOROID_ERR_INVALID_ARG;
    if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < tbb::workspace_bytes(K))
        return MEMOROID_ERR_WORKSPACE;
    cudaStream_t s = as_stream(stream);
    if (B == 0) {
        if (cudaMemsetAsync(workspace, 0, kHeaderBytes, s) != cudaSuccess) return MEMOROID_ERR_CUDA;
        if (n_used && cudaMemsetAsync(n_used, 0, sizeof(int64_t), s) != cudaSuccess) return MEMOROID_ERR_CUDA;
        return MEMOROID_OK;
    }
    if (!start || !src || (K > 0 && (!begin || !draws))) return MEMOROID_ERR_INVALID_ARG;
    if (!aligned(src, 8) || (begin && !aligned(begin, 8)) || (draws && !aligned(draws, 8)) ||
        (n_used && !aligned(n_used, 8)))
        return MEMOROID_ERR_INVALID_ARG;
    return tbb::launch_sample(begin, E, N, draws, K, B, start, src, n_used, workspace, s);
}

memoroid_status_t memoroid_gather_rows(const void* rows, int64_t N, int64_t row_bytes, const int64_t* src, int64_t B,
                                       void* out, void* workspace, size_t workspace_bytes, void* stream) {
    if (N < 0 || row_bytes <= 0 || B < 0) return MEMOROID_ERR_INVALID_ARG;
    if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < kHeaderBytes)
        return MEMOROID_ERR_WORKSPACE;
    cudaStream_t s = as_stream(stream);
    if (B == 0) return cudaMemsetAsync(workspace, 0, kHeaderBytes, s) == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
    if (!src || !out || (N > 0 && !rows) || !aligned(src, 8)) return MEMOROID_ERR_INVALID_ARG;
    return tbb::launch_gather(rows, N, row_bytes, src, B, out, workspace, s);
}

// ---------------------------------------------------------------------------
// discounted return and GAE
// ---------------------------------------------------------------------------

size_t memoroid_returns_workspace_bytes(int64_t B, int64_t L) {
    if (B < 0 || L < 0) return 0;
    return ret::workspace_bytes(B, L);
}

static memoroid_status_t returns_common(const float* r, const float* v, const uint8_t* start, float c, float gamma,
                                        const float* boot, float* out, int64_t B, int64_t L, void* workspace,
                                        size_t workspace_bytes, void* stream) {
    if (B < 0 || L < 0) return MEMOROID_ERR_INVALID_ARG;
    if (B == 0 || L == 0) return MEMOROID_OK;
    if (!r || !start || !out) return MEMOROID_ERR_INVALID_ARG;
    if (!aligned(r, 4) || !aligned(out, 4) || (v && !aligned(v, 4)) || (boot && !aligned(boot, 4)))
        return MEMOROID_ERR_INVALID_ARG;
    if (workspace == nullptr || !aligned(workspace, 256) || workspace_bytes < ret::workspace_bytes(B, L))
        return MEMOROID_ERR_WORKSPACE;
    return ret::launch(r, v, start, c, gamma, boot, out, B, L, workspace, as_stream(stream));
}

memoroid_status_t memoroid_discounted_return(const float* r, const uint8_t* start, float gamma, const float* boot,
                                             float* G, int64_t B, int64_t L, void* workspace,
                                             size_t workspace_bytes, void* stream) {
    return returns_common(r, nullptr, start, gamma, gamma, boot, G, B, L, workspace, workspace_bytes, stream);
}

memoroid_status_t memoroid_gae(const float* r, const float* v, const uint8_t* start, float gamma, float lambda,
                               const float* v_boot, float* A, int64_t B, int64_t L, void* workspace,
                               size_t workspace_bytes, void* stream) {
    if (v == nullptr && B > 0 && L > 0) return MEMOROID_ERR_INVALID_ARG;
    return returns_common(r, v, start, gamma * lambda, gamma, v_boot, A, B, L, workspace, workspace_bytes, stream);
}

}  // extern "C"
