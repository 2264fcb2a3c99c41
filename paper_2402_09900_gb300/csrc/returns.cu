// returns.cu -- per-step discounted return and GAE with resets at episode
// boundaries: the memoroids of the appendices "The Discounted Return as a
// Memoroid" and "The Generalized Advantage Estimate as a Memoroid",
// (a, r) . (a', r') = (a a', a r' + r) with f = (gamma, r_t) resp.
// (gamma lambda, delta_t), evaluated for every step.  Per step this is the
// reverse recurrence
//   G_t = x_t + m_t G_{t+1},   m_t = c [b_{t+1} = 0]   (c = gamma or gamma lambda)
// with x_t = r_t (return) or delta_t = r_t + gamma V_{t+1} - V_t (GAE, V after
// an episode's last step 0, after the tape's last step v_boot).
//
// A step whose successor starts an episode has m_t = 0, so a segment of the
// tape that ends right before a begin flag does not depend on later steps.
// Segment boundaries are therefore moved to begin flags (the linear-attention
// planner) and every CTA scans its segment backwards on its own, in blocks of
// kThreads * kElems steps: each thread folds its kElems steps into an affine
// map G_first = X + A G_in, a block-wide suffix scan of these maps (fixed
// order) gives each thread its incoming value, and the block's result is the
// carry into the block before it.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"

namespace memoroid {
namespace ret {

constexpr int kThreads = 256;
constexpr int kElems = 8;
constexpr int kBlock = kThreads * kElems;
constexpr int kTargetCtas = 152 * 8;

struct Plan {
    int64_t G, seg_len;
};

Plan make_plan(int64_t B, int64_t L) {
    Plan p;
    int64_t G = B > 0 ? kTargetCtas / B : 1;
    const int64_t max_g = (L + kBlock - 1) / kBlock;
    if (G > max_g) G = max_g;
    if (G < 1) G = 1;
    p.seg_len = L > 0 ? (L + G - 1) / G : 1;
    p.G = L > 0 ? (L + p.seg_len - 1) / p.seg_len : 1;
    return p;
}

size_t workspace_bytes(int64_t B, int64_t L) {
    const Plan p = make_plan(B, L);
    return kHeaderBytes + align_up(static_cast<size_t>(B * p.G) * sizeof(int64_t), 256);
}

struct Params {
    const float* r;
    const float* v;  // GAE: values; null for the return
    const uint8_t* start;
    const float* boot;  // return: value after the tape's last step; GAE: v_boot
    float* out;
    const int64_t* seg_first;
    int64_t B, L;
    int G;
    float c;      // per-step multiplier: gamma or gamma * lambda
    float gamma;  // GAE: the discount inside delta
};

// (A, X) maps G_in -> X + A G_in; compose(earlier, later) applies `later` first.
struct Aff {
    float a, x;
};
__device__ __forceinline__ Aff compose(Aff e, Aff l) { return Aff{e.a * l.a, fmaf(e.a, l.x, e.x)}; }

template <bool GAE>
__global__ void __launch_bounds__(kThreads) scan_kernel(const Params p) {
    __shared__ Aff warp_agg[kThreads / 32];
    __shared__ float s_carry;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t b = blockIdx.x / p.G;
    const int g = static_cast<int>(blockIdx.x % p.G);
    const int64_t* sf = p.seg_first + b * p.G;
    const int64_t lo = sf[g];
    if (lo < 0) return;  // covered by an earlier segment
    int64_t hi = p.L;
    for (int g2 = g + 1; g2 < p.G; ++g2) {
        if (sf[g2] >= 0) {
            hi = sf[g2];
            break;
        }
    }
    const float* r = p.r + b * p.L;
    const float* v = GAE ? p.v + b * p.L : nullptr;
    const uint8_t* st = p.start + b * p.L;
    const float boot = p.boot != nullptr ? p.boot[b] : 0.f;
    // value entering the segment's last step from after it: the bootstrap at the
    // tape's end (return only; the advantage after the tape is 0)
    float carry = (!GAE && hi == p.L) ? boot : 0.f;

    for (int64_t b1 = hi; b1 > lo; b1 -= kBlock) {
        const int64_t b0 = b1 - kBlock > lo ? b1 - kBlock : lo;
        const int64_t t0 = b0 + static_cast<int64_t>(tid) * kElems;
        float x[kElems], m[kElems];
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
            const int64_t t = t0 + e;
            if (t < b1) {
                const bool last = t + 1 >= p.L;
                const bool cont = !last && st[t + 1] == 0;  // the next step is in the same episode
                m[e] = last ? p.c : (cont ? p.c : 0.f);
                if (GAE) {
                    const float nv = last ? boot : (cont ? v[t + 1] : 0.f);
                    x[e] = fmaf(p.gamma, nv, r[t]) - v[t];
                } else {
                    x[e] = r[t];
                }
            } else {
                m[e] = 1.f;  // identity past the block
                x[e] = 0.f;
            }
        }
        // this thread's map: G at its first step as a function of G after its last
        Aff mine{1.f, 0.f};
#pragma unroll
        for (int e = kElems - 1; e >= 0; --e) mine = Aff{m[e] * mine.a, fmaf(m[e], mine.x, x[e])};
        // inclusive suffix over the lanes (lane + 1 is later in time)
        Aff suf = mine;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float oa = __shfl_down_sync(0xffffffffu, suf.a, off);
            const float ox = __shfl_down_sync(0xffffffffu, suf.x, off);
            if (lane + off < 32) suf = compose(suf, Aff{oa, ox});
        }
        if (lane == 0) warp_agg[warp] = suf;
        if (tid == 0) s_carry = carry;
        __syncthreads();
        // map of everything after this thread's last step within the block
        Aff after{1.f, 0.f};
        {
            const float na = __shfl_down_sync(0xffffffffu, suf.a, 1);
            const float nx = __shfl_down_sync(0xffffffffu, suf.x, 1);
            if (lane < 31) after = Aff{na, nx};
        }
        for (int w = warp + 1; w < kThreads / 32; ++w) after = compose(after, warp_agg[w]);
        float gin = fmaf(after.a, s_carry, after.x);
        // the block's value at its first step is the carry into the block before it
        Aff whole = warp_agg[0];
#pragma unroll
        for (int w = 1; w < kThreads / 32; ++w) whole = compose(whole, warp_agg[w]);
        carry = fmaf(whole.a, s_carry, whole.x);
        // outputs, last step first
        float out[kElems];
#pragma unroll
        for (int e = kElems - 1; e >= 0; --e) {
            gin = fmaf(m[e], gin, x[e]);
            out[e] = gin;
        }
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
            const int64_t t = t0 + e;
            if (t < b1) p.out[b * p.L + t] = out[e];
        }
        __syncthreads();  // warp_agg and s_carry are rewritten by the next block
    }
}

memoroid_status_t launch(const float* r, const float* v, const uint8_t* start, float c, float gamma,
                         const float* boot, float* out, int64_t B, int64_t L, void* workspace, cudaStream_t s) {
    const Plan pl = make_plan(B, L);
    int64_t* seg_first = reinterpret_cast<int64_t*>(static_cast<unsigned char*>(workspace) + kHeaderBytes);
    if (cudaMemsetAsync(workspace, 0, kHeaderBytes, s) != cudaSuccess) return MEMOROID_ERR_CUDA;
    const memoroid_status_t st = la::launch_segment_plan(start, B, L, pl.seg_len, pl.G, seg_first, s);
    if (st != MEMOROID_OK) return st;
    Params p{r, v, start, boot, out, seg_first, B, L, static_cast<int>(pl.G), c, gamma};
    const unsigned grid = static_cast<unsigned>(B * pl.G);
    if (v != nullptr)
        scan_kernel<true><<<grid, kThreads, 0, s>>>(p);
    else
        scan_kernel<false><<<grid, kThreads, 0, s>>>(p);
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

}  // namespace ret
}  // namespace memoroid
