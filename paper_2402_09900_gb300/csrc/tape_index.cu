// tape_index.cu -- exact conversion between the episode begin-index list I and
// the per-step begin flags b_t of a tape.  Algorithm 1 keeps I = where(b);
// Figure 2 shows a tape with I = [0, 4, 6, 7].
#include <cuda_runtime.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace memoroid {
namespace tape {

constexpr int CHUNK_THREADS = 256;
constexpr int CHUNK_PER_THREAD = 16;
constexpr int64_t CHUNK = CHUNK_THREADS * CHUNK_PER_THREAD;  // flags per block

__global__ void scatter_starts_kernel(const int64_t* __restrict__ offsets, int64_t E, int64_t L,
                                      uint8_t* __restrict__ start) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i < E) {
        const int64_t o = offsets[i];
        if (o >= 0 && o < L) start[o] = 1;
    }
}

// Number of non-zero flags in each CHUNK.
__global__ void __launch_bounds__(CHUNK_THREADS) count_kernel(const uint8_t* __restrict__ start,
                                                              int64_t L,
                                                              int64_t* __restrict__ counts) {
    __shared__ int s[CHUNK_THREADS / 32];
    const int64_t base = static_cast<int64_t>(blockIdx.x) * CHUNK;
    int c = 0;
    for (int k = 0; k < CHUNK_PER_THREAD; ++k) {
        const int64_t t = base + static_cast<int64_t>(k) * CHUNK_THREADS + threadIdx.x;
        if (t < L && start[t] != 0) ++c;
    }
    for (int o = 16; o > 0; o >>= 1) c += __shfl_down_sync(0xffffffffu, c, o);
    if ((threadIdx.x & 31) == 0) s[threadIdx.x >> 5] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
        int tot = 0;
        for (int w = 0; w < CHUNK_THREADS / 32; ++w) tot += s[w];
        counts[blockIdx.x] = tot;
    }
}

// In-place exclusive scan of the per-chunk counts (one block); writes the
// total to *count.
__global__ void __launch_bounds__(1024) scan_counts_kernel(int64_t* __restrict__ counts, int64_t nb,
                                                           int64_t* __restrict__ count) {
    __shared__ int64_t s[1024];
    ptx::grid_dependency_wait();  // the chunk counts
    __shared__ int64_t s_carry;
    if (threadIdx.x == 0) s_carry = 0;
    __syncthreads();
    for (int64_t base = 0; base < nb; base += 1024) {
        const int64_t i = base + threadIdx.x;
        const int64_t v = (i < nb) ? counts[i] : 0;
        s[threadIdx.x] = v;
        __syncthreads();
        for (int o = 1; o < 1024; o <<= 1) {  // Hillis-Steele inclusive scan
            const int64_t add = (threadIdx.x >= o) ? s[threadIdx.x - o] : 0;
            __syncthreads();
            s[threadIdx.x] += add;
            __syncthreads();
        }
        const int64_t incl = s[threadIdx.x] + s_carry;
        if (i < nb) counts[i] = incl - v;
        __syncthreads();
        if (threadIdx.x == 1023) s_carry = incl;
        __syncthreads();
    }
    if (threadIdx.x == 0) *count = s_carry;
}

// Writes the indices of each chunk's flags at the chunk's scanned offset,
// in increasing order: thread k handles flags [k*16, k*16+16) of the chunk.
__global__ void __launch_bounds__(CHUNK_THREADS) write_offsets_kernel(
    const uint8_t* __restrict__ start, int64_t L, const int64_t* __restrict__ base_off,
    int64_t* __restrict__ offsets) {
    __shared__ int s[CHUNK_THREADS];
    ptx::grid_dependency_wait();  // the chunk offsets
    const int64_t base = static_cast<int64_t>(blockIdx.x) * CHUNK;
    const int64_t t0 = base + static_cast<int64_t>(threadIdx.x) * CHUNK_PER_THREAD;
    int c = 0;
    for (int k = 0; k < CHUNK_PER_THREAD; ++k) {
        const int64_t t = t0 + k;
        if (t < L && start[t] != 0) ++c;
    }
    s[threadIdx.x] = c;
    __syncthreads();
    for (int o = 1; o < CHUNK_THREADS; o <<= 1) {
        const int add = (threadIdx.x >= o) ? s[threadIdx.x - o] : 0;
        __syncthreads();
        s[threadIdx.x] += add;
        __syncthreads();
    }
    int64_t pos = base_off[blockIdx.x] + s[threadIdx.x] - c;
    for (int k = 0; k < CHUNK_PER_THREAD; ++k) {
        const int64_t t = t0 + k;
        if (t < L && start[t] != 0) offsets[pos++] = t;
    }
}

size_t offsets_workspace_bytes(int64_t L) {
    const int64_t nb = (L + CHUNK - 1) / CHUNK;
    return align_up(kHeaderBytes + static_cast<size_t>(nb > 0 ? nb : 1) * 8, 256);
}

memoroid_status_t launch_starts_from_offsets(const int64_t* offsets, int64_t E, int64_t L,
                                             uint8_t* start, cudaStream_t s) {
    if (L > 0 && cudaMemsetAsync(start, 0, static_cast<size_t>(L), s) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    if (E > 0 && L > 0) {
        const int64_t nb = (E + 255) / 256;
        if (nb > 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;
        scatter_starts_kernel<<<static_cast<unsigned>(nb), 256, 0, s>>>(offsets, E, L, start);
        if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    }
    return MEMOROID_OK;
}

memoroid_status_t launch_offsets_from_starts(const uint8_t* start, int64_t L, int64_t* offsets,
                                             int64_t* count, void* workspace, size_t ws_bytes,
                                             cudaStream_t s) {
    (void)ws_bytes;
    const int64_t nb = (L + CHUNK - 1) / CHUNK;
    if (nb > 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;
    if (L == 0) {
        if (cudaMemsetAsync(count, 0, sizeof(int64_t), s) != cudaSuccess) return MEMOROID_ERR_CUDA;
        return MEMOROID_OK;
    }
    int64_t* counts = reinterpret_cast<int64_t*>(static_cast<unsigned char*>(workspace) + kHeaderBytes);
    count_kernel<<<static_cast<unsigned>(nb), CHUNK_THREADS, 0, s>>>(start, L, counts);
    if (cudaGetLastError() != cudaSuccess ||
        launch_after(scan_counts_kernel, dim3(1), dim3(1024), 0, s, counts, nb, count) != cudaSuccess ||
        launch_after(write_offsets_kernel, dim3(static_cast<unsigned>(nb)), dim3(CHUNK_THREADS), 0, s, start, L,
                     static_cast<const int64_t*>(counts), offsets) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    return MEMOROID_OK;
}

}  // namespace tape
}  // namespace memoroid
