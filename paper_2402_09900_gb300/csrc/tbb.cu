// tbb.cu -- tape-based batching on the device: the sampling step of
// Algorithm 2 ("Sampling transitions using TBB") and the row gather that
// builds the sampled tape from a buffer of transitions.
//
// Algorithm 2 appends the episode D[I[i] : I[i+1]] of a drawn index i while
// the batch is shorter than B, then cuts the batch to B transitions.  With
// the draws given (ep[0..K), from the caller's generator) the batch is fixed:
// piece k is episode ep[k], it starts at tape step off[k] = sum of the
// earlier pieces' lengths, and the draws used are the fewest n with
// off[n-1] + len(ep[n-1]) >= B.  The episode of the last index runs to the end
// of the buffer (I[E] reads as N).
//
//   offsets_kernel  one CTA: chunked block-wide prefix sum of the drawn
//                   episodes' lengths, stopping at the chunk that covers B
//   fill_kernel     one warp per piece: begin flag and source index of each
//                   of its steps (start[off[k]] = 1, src[off[k] + j] = I[ep[k]] + j)
//   gather_kernel   out[t] = rows[src[t]] for rows of any byte size (16-byte
//                   streaming copies when the rows allow it)
// Integer work only: results are exact.  Bad data (an index out of range, an
// empty episode, too few draws, a source index outside the buffer) is
// recorded in the workspace header and read back with
// memoroid_get_device_error; the kernels never trap.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"
#include "ptx.cuh"

namespace memoroid {
namespace tbb {

namespace {

constexpr int kScanThreads = 1024;
constexpr int kPer = 4;  // draws per thread per chunk
constexpr int kChunk = kScanThreads * kPer;
constexpr int kFillCtas = 152 * 4;
constexpr int kGatherCtas = 152 * 8;

__device__ __forceinline__ void bad_data(uint32_t* hdr) { atomicCAS(hdr, 0u, static_cast<uint32_t>(DEV_BAD_DATA)); }

// length of episode i of the buffer, or -1 (bad index or empty episode)
__device__ __forceinline__ int64_t episode(const int64_t* begin, int64_t E, int64_t N, int64_t i, int64_t* lo) {
    if (i < 0 || i >= E) return -1;
    const int64_t a = begin[i], b = (i + 1 < E) ? begin[i + 1] : N;
    *lo = a;
    return (a >= 0 && b > a && b <= N) ? b - a : -1;
}

__global__ void __launch_bounds__(kScanThreads) offsets_kernel(const int64_t* __restrict__ begin, int64_t E, int64_t N,
                                                               const int64_t* __restrict__ ep, int64_t K, int64_t B,
                                                               int64_t* __restrict__ off, int64_t* __restrict__ meta,
                                                               uint32_t* __restrict__ hdr,
                                                               int64_t* __restrict__ n_used) {
    __shared__ int64_t warp_sum[kScanThreads / 32];
    __shared__ int64_t s_carry;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        s_carry = 0;
        meta[0] = 0;  // draws used
        *hdr = 0u;    // this call's error word (this kernel runs first)
    }
    __syncthreads();
    for (int64_t c0 = 0; c0 < K; c0 += kChunk) {
        int64_t len[kPer], sum = 0;
        bool bad = false;
#pragma unroll
        for (int j = 0; j < kPer; ++j) {
            const int64_t k = c0 + static_cast<int64_t>(tid) * kPer + j;
            len[j] = 0;
            if (k < K) {
                int64_t lo;
                const int64_t l = episode(begin, E, N, ep[k], &lo);
                if (l < 0) bad = true;
                else len[j] = l;
            }
            sum += len[j];
        }
        if (bad) bad_data(hdr);
        // exclusive block scan of the per-thread sums (warp shuffles, then the warp totals)
        int64_t inc = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t v = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += v;
        }
        if (lane == 31) warp_sum[warp] = inc;
        __syncthreads();
        if (warp == 0) {
            int64_t w = warp_sum[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int64_t v = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += v;
            }
            warp_sum[lane] = w;  // inclusive over warps
        }
        __syncthreads();
        const int64_t carry = s_carry;
        int64_t o = carry + (warp > 0 ? warp_sum[warp - 1] : 0) + (inc - sum);
#pragma unroll
        for (int j = 0; j < kPer; ++j) {
            const int64_t k = c0 + static_cast<int64_t>(tid) * kPer + j;
            if (k < K) {
                off[k] = o;
                if (o < B && o + len[j] >= B) meta[0] = k + 1;  // the piece that covers step B - 1
            }
            o += len[j];
        }
        const int64_t total = carry + warp_sum[kScanThreads / 32 - 1];
        __syncthreads();  // every thread has read s_carry and warp_sum
        if (tid == 0) s_carry = total;
        __syncthreads();
        if (total >= B) break;
    }
    __syncthreads();  // meta[0] is written by the thread that holds the last piece
    if (tid == 0) {
        if (s_carry < B) {  // the draws do not fill the batch
            bad_data(hdr);
            meta[0] = K;
        }
        meta[1] = s_carry < B ? s_carry : B;  // steps covered by pieces
        if (n_used != nullptr) *n_used = meta[0];
    }
}

__global__ void __launch_bounds__(256) fill_kernel(const int64_t* __restrict__ begin, int64_t E, int64_t N,
                                                   const int64_t* __restrict__ ep, int64_t B,
                                                   const int64_t* __restrict__ off, const int64_t* __restrict__ meta,
                                                   uint8_t* __restrict__ start, int64_t* __restrict__ src) {
    ptx::grid_dependency_wait();  // the episode offsets
    const int lane = threadIdx.x & 31;
    const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const int64_t n = meta[0], covered = meta[1];
    for (int64_t k = gw; k < n; k += nw) {
        int64_t lo = 0;
        const int64_t l = episode(begin, E, N, ep[k], &lo);
        if (l < 0) continue;  // recorded by offsets_kernel
        const int64_t o = off[k];
        const int64_t m = l < B - o ? l : B - o;
        for (int64_t j = lane; j < m; j += 32) {
            start[o + j] = j == 0 ? 1 : 0;
            src[o + j] = lo + j;
        }
    }
    // steps no piece reaches (too few draws): no source
    for (int64_t t = covered + gw * 32 + lane; t < B; t += nw * 32) {
        start[t] = 0;
        src[t] = -1;
    }
}

// out[t] = rows[src[t]]: U units of `Unit` bytes per row; one warp per row for
// wide rows, one thread per row for narrow ones (consecutive steps of a piece
// then read consecutive rows).
template <typename Unit>
__global__ void __launch_bounds__(256) gather_kernel(const Unit* __restrict__ rows, int64_t N, int64_t U,
                                                     const int64_t* __restrict__ src, int64_t B,
                                                     Unit* __restrict__ out, uint32_t* __restrict__ hdr) {
    const int lane = threadIdx.x & 31;
    const int64_t gt = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    const int64_t nt = static_cast<int64_t>(gridDim.x) * blockDim.x;
    bool bad = false;
    if (U >= 8) {
        const int64_t gw = gt >> 5, nw = nt >> 5;
        for (int64_t t = gw; t < B; t += nw) {
            const int64_t s = src[t];
            const bool ok = s >= 0 && s < N;
            bad |= !ok;
            Unit* o = out + t * U;
            if (!ok) {  // the same for the whole warp
                for (int64_t u = lane; u < U; u += 32) o[u] = Unit{};
                continue;
            }
            const Unit* in = rows + s * U;
            int64_t u = lane;
            for (; u + 96 < U; u += 128) {  // four units in flight per lane
                const Unit a = __ldcs(in + u), b = __ldcs(in + u + 32), c = __ldcs(in + u + 64), d = __ldcs(in + u + 96);
                __stcs(o + u, a);
                __stcs(o + u + 32, b);
                __stcs(o + u + 64, c);
                __stcs(o + u + 96, d);
            }
            for (; u < U; u += 32) __stcs(o + u, __ldcs(in + u));
        }
    } else {
        for (int64_t t = gt; t < B; t += nt) {
            const int64_t s = src[t];
            const bool ok = s >= 0 && s < N;
            bad |= !ok;
            for (int64_t u = 0; u < U; ++u) out[t * U + u] = ok ? rows[s * U + u] : Unit{};
        }
    }
    if (bad) bad_data(hdr);
}

}  // namespace

// workspace: header | draws used, steps covered | off[K]
size_t workspace_bytes(int64_t K) { return kHeaderBytes + align_up(static_cast<size_t>(K + 2) * 8, 256); }

memoroid_status_t launch_sample(const int64_t* begin, int64_t E, int64_t N, const int64_t* ep, int64_t K, int64_t B,
                                uint8_t* start, int64_t* src, int64_t* n_used, void* workspace, cudaStream_t s) {
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    uint32_t* hdr = reinterpret_cast<uint32_t*>(ws);
    int64_t* meta = reinterpret_cast<int64_t*>(ws + kHeaderBytes);
    int64_t* off = meta + 2;
    offsets_kernel<<<1, kScanThreads, 0, s>>>(begin, E, N, ep, K, B, off, meta, hdr, n_used);
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    return launch_after(fill_kernel, dim3(kFillCtas), dim3(256), 0, s, begin, E, N, ep, B,
                        static_cast<const int64_t*>(off), static_cast<const int64_t*>(meta), start, src) == cudaSuccess
               ? MEMOROID_OK
               : MEMOROID_ERR_CUDA;
}

memoroid_status_t launch_gather(const void* rows, int64_t N, int64_t row_bytes, const int64_t* src, int64_t B,
                                void* out, void* workspace, cudaStream_t s) {
    uint32_t* hdr = static_cast<uint32_t*>(workspace);
    if (cudaMemsetAsync(workspace, 0, kHeaderBytes, s) != cudaSuccess) return MEMOROID_ERR_CUDA;
    auto al = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; };
    if (row_bytes % 16 == 0 && al(rows, 16) && al(out, 16))
        gather_kernel<uint4><<<kGatherCtas, 256, 0, s>>>(static_cast<const uint4*>(rows), N, row_bytes / 16, src, B,
                                                         static_cast<uint4*>(out), hdr);
    else if (row_bytes % 4 == 0 && al(rows, 4) && al(out, 4))
        gather_kernel<uint32_t><<<kGatherCtas, 256, 0, s>>>(static_cast<const uint32_t*>(rows), N, row_bytes / 4, src,
                                                            B, static_cast<uint32_t*>(out), hdr);
    else
        gather_kernel<uint8_t><<<kGatherCtas, 256, 0, s>>>(static_cast<const uint8_t*>(rows), N, row_bytes, src, B,
                                                           static_cast<uint8_t*>(out), hdr);
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

}  // namespace tbb
}  // namespace memoroid
