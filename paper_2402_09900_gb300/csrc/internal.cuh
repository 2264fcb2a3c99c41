// internal.cuh -- declarations shared by the C-ABI layer and the kernel files.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "memoroid.h"

namespace memoroid {

// Device-side error codes written to the first word of a workspace header.
enum DeviceError : uint32_t {
    DEV_OK = 0,
    DEV_LOOKBACK_TIMEOUT = 1,  // a look-back wait on a predecessor's summary ran out
    DEV_TMA_TIMEOUT = 2,       // a wait for staged data (TMA completion) ran out
    DEV_STAGE_TIMEOUT = 3,     // the producer's wait for a free stage ran out
    DEV_AGG_TIMEOUT = 4,       // the look-back warp's wait for warp aggregates ran out
    DEV_CARRY_TIMEOUT = 5,     // a compute warp's wait for its carry ran out
    DEV_ACC_TIMEOUT = 6,       // the wait for grad_lambda partials ran out
    DEV_DRAIN_TIMEOUT = 7,     // the final wait for in-flight copies ran out
    DEV_MMA_TIMEOUT = 8,       // a wait for tensor-core completion ran out
    DEV_BAD_DATA = 9,          // device-side data check failed (index out of range, too few draws)
};

// Workspace header (256 bytes): [0] error code, [1] tile ticket counter,
// [2..3] ticket of the tile that recorded the error (u64).
constexpr size_t kHeaderBytes = 256;

// Process-wide debug knobs (set through memoroid_debug_*).
struct DebugKnobs {
    uint64_t wait_ns;
    int64_t withhold_ticket;
    int lnorm_padded;  // the normalised calls always take the padded-operand path
};
DebugKnobs debug_knobs();

// A fresh 31-bit, non-zero tag for a launch whose look-back summaries, in
// the bytes [kHeaderBytes, region_end) of `workspace`, carry it.  Tags are
// handed out in sequence and repeat only after 2^31 launches (a new
// "generation").  *clear is set when the caller must zero that region before
// the launch: the first time this process uses the workspace address on the
// current device, the first time in each generation, or when the region
// reaches further than the last clear.  So a summary word with this launch's
// tag was written by this launch: every earlier write of the same tag is in a
// past generation, and the region was cleared since.
// Under stream capture (a graph replays the tag), *clear is always true.
uint32_t tagged_epoch(const void* workspace, size_t region_end, cudaStream_t stream, bool* clear);

// Launches a kernel that follows another kernel on the stream with programmatic
// stream serialization: it may be scheduled before that kernel completes and
// waits for it at its first statement (ptx::grid_dependency_wait), which hides
// the launch latency between the two.  Only for kernels whose predecessor on
// the stream is a kernel.
template <typename... KArgs, typename... Args>
cudaError_t launch_after(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                         Args... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// cuTensorMapEncodeTiled, taken from the driver at run time (the library does
// not link libcuda); null if the driver does not provide it.
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled();

namespace diag {

struct Args {
    const void* lambda;
    int lambda_per_step;
    const void* u;  // fwd: u; bwd: grad_h
    const uint8_t* start;
    const void* h0;
    void* out;       // fwd: h; bwd: grad_u
    void* out_last;  // fwd: h_last
    const void* h;   // bwd: forward output
    const void* g_last;
    void* grad_lambda;
    void* grad_h0;
    int64_t B, L, D;
    void* workspace;
    size_t workspace_bytes;
    // Fast and Forgetful Memory layout (ffm_c > 0): forward input x~ [B, L, m]
    // in place of u, planar Re || Im states and gradients, backward output
    // grad_x~ [B, L, m] in place of grad_u
    const float* ffm_x = nullptr;
    float* ffm_gx = nullptr;
    int64_t ffm_m = 0;
    int ffm_c = 0;
};

// FFM call: lambda_ij = exp(-|alpha_i| + i omega_j) built in the workspace,
// then the scan in the FFM layout (and, backward, the parameter gradients)
struct FfmArgs {
    bool backward;
    const float* x;  // fwd: x~ [B, L, m]
    const float* alpha;
    const float* omega;
    const uint8_t* start;
    const void* S0;           // [B, m*c] complex or null
    float* z;                 // fwd output / bwd input: [B, L, 2*m*c]
    void* S_last;             // fwd: [B, m*c] complex or null
    const float* grad_z;      // bwd
    const void* grad_S_last;  // bwd, or null
    float* grad_x;            // bwd: [B, L, m]
    float* grad_alpha;        // bwd: [m] or null
    float* grad_omega;        // bwd: [c] or null
    void* grad_S0;            // bwd: [B, m*c] complex or null
    int64_t B, L, m, c;
    void* workspace;
    size_t workspace_bytes;
};

size_t ffm_workspace_bytes(int64_t B, int64_t L, int64_t m, int64_t c);
int ffm_kernels_per_call(int64_t B, int64_t L, int64_t m, int64_t c, int backward, int with_param_grads);
memoroid_status_t launch_ffm(const FfmArgs& a, cudaStream_t stream);

size_t workspace_bytes(int64_t B, int64_t L, int64_t D);
int kernels_per_call(int64_t B, int64_t L, int64_t D, int per_step, int backward, int with_grad_lambda);
memoroid_status_t launch_fwd(const Args& a, cudaStream_t stream);
memoroid_status_t launch_bwd(const Args& a, cudaStream_t stream);

}  // namespace diag

namespace la {

struct Args {
    const void* q;  // bf16 [B, L, H, D]
    const void* k;
    const void* v;
    const float* gamma;  // [H] or [B, L, H]
    int gamma_per_step;
    const uint8_t* start;  // [B, L]
    const float* S0;       // [B, H, D, D] or null
    float* y;              // fwd: [B, L, H, D]
    float* S_last;         // fwd: [B, H, D, D] or null
    const float* grad_y;   // bwd: [B, L, H, D]
    const float* dS_last;  // bwd: [B, H, D, D] or null
    float* dq;             // bwd outputs: [B, L, H, D]
    float* dk;
    float* dv;
    float* dgamma;  // [H] or [B, L, H], or null
    float* dS0;     // [B, H, D, D] or null
    int64_t B, L, H, D;
    void* workspace;
    size_t workspace_bytes;
    // norm = 1: the Linear Transformer with phi and its normalizer for
    // 64-channel heads at D = 128, with q, k, v the unpadded [B, L, H, 64]
    // tensors.  Forward: y [B, L, H, 64] and den [B, L, H] (or null); S0 and
    // S_last in the padded [B, H, 128, 128] layout.  Backward: the padded bf16
    // upstream gradient in grad_y16 and out_cols = 64; dq, dk, dv [B, L, H, 64]
    // are the gradients with respect to the raw q, k, v (the epilogues apply
    // phi'(q) and phi'(k) to the padded gradients' first 64 columns).
    int norm = 0;
    float* den = nullptr;
    // backward only: grad_y already in bf16 [B, L, H, D] (exact values), used as
    // the operand directly instead of the workspace copy
    const uint16_t* grad_y16 = nullptr;
    // backward only: 64 (with D = 128) writes only the first 64 columns of dq,
    // dk, dv, as [B, L, H, 64] arrays; 0 writes all D
    int64_t out_cols = 0;
    // backward only: >= 0 adds column fold_col of dq to every column of dq (the
    // normalised backward's sum channel); -1 = off
    int64_t fold_col = -1;
};

size_t workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t D);      // forward and backward
size_t fwd_workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t D);  // forward only
int kernels_per_call(int64_t B, int64_t L, int64_t H, int backward, int with_dgamma_per_head);
memoroid_status_t launch_fwd(const Args& a, cudaStream_t stream);
memoroid_status_t launch_bwd(const Args& a, cudaStream_t stream);
size_t intra_bench_scratch_bytes(int64_t D);
memoroid_status_t launch_intra_bench(int64_t D, int64_t reps, int64_t ctas, void* scratch, cudaStream_t stream);

}  // namespace la

namespace ret {
size_t workspace_bytes(int64_t B, int64_t L);
// v == null: discounted return (c = gamma, boot = value after the tape);
// otherwise GAE (c = gamma * lambda, boot = v_boot)
memoroid_status_t launch(const float* r, const float* v, const uint8_t* start, float c, float gamma,
                         const float* boot, float* out, int64_t B, int64_t L, void* workspace, cudaStream_t s);
}  // namespace ret

namespace lnorm {
// the Linear Transformer with phi and normalizer, by the padded-operand
// construction over the d = 128 linear-attention kernels
struct Args {
    bool backward;
    const void *q, *k, *v;  // bf16 [B, L, H, d]
    const float* gamma;     // [H] or [B, L, H]
    int gamma_per_step;
    const uint8_t* start;
    const float *S0, *z0;        // [B, H, d, d], [B, H, d] or null
    float* y;                    // fwd output / bwd input: [B, L, H, d]
    float* den;                  // fwd output (or null) / bwd input: [B, L, H]
    float *S_last, *z_last;      // fwd outputs or null
    const float* grad_y;         // bwd
    const float *dS_last, *dz_last;
    float *dq, *dk, *dv, *dgamma, *dS0, *dz0;
    int64_t B, L, H, d;
    void* workspace;
};
size_t workspace_bytes(int64_t B, int64_t L, int64_t H);
int kernels_per_call(int64_t B, int64_t L, int64_t H, int64_t d, int backward, int with_dgamma_per_head,
                     int with_states);
memoroid_status_t launch(const Args& a, cudaStream_t s);
}  // namespace lnorm

namespace tbb {
size_t workspace_bytes(int64_t K);
memoroid_status_t launch_sample(const int64_t* begin, int64_t E, int64_t N, const int64_t* ep, int64_t K, int64_t B,
                                uint8_t* start, int64_t* src, int64_t* n_used, void* workspace, cudaStream_t s);
memoroid_status_t launch_gather(const void* rows, int64_t N, int64_t row_bytes, const int64_t* src, int64_t B,
                                void* out, void* workspace, cudaStream_t s);
}  // namespace tbb

namespace tape {
size_t offsets_workspace_bytes(int64_t L);
memoroid_status_t launch_starts_from_offsets(const int64_t* offsets, int64_t E, int64_t L,
                                             uint8_t* start, cudaStream_t stream);
memoroid_status_t launch_offsets_from_starts(const uint8_t* start, int64_t L, int64_t* offsets,
                                             int64_t* count, void* workspace, size_t ws_bytes,
                                             cudaStream_t stream);
}  // namespace tape

}  // namespace memoroid
