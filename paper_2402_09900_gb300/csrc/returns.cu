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
// A step whose successor starts an episode has m_t = 0, so a stretch of the
// tape that ends right before a begin flag does not depend on later steps.
// Each tape is cut into G nominal ranges of seg_len steps, one warp each; a
// warp's segment runs from the first begin flag in its range (step 0 for the
// first range) to the first begin flag after its range (or the tape's end),
// found by the warp itself, so no planning pass, carry or fix-up is needed.
// The warp walks its segment backwards in chunks of 32 * kElems steps on
// absolute chunk boundaries (16-byte loads and stores when the tape length is
// a multiple of 8 and the buffers are aligned), loading the chunk before
// while it scans the current one: each lane folds its kElems steps into an
// affine map G_first = X + A G_in, a shuffle suffix scan (fixed order) gives
// each lane its incoming value, and the chunk's result is the carry into the
// chunk before it.  The successor of a lane's last step is the next lane's
// first step, taken by shuffle.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"

namespace memoroid {
namespace ret {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kElems = 8;
constexpr int kChunk = 32 * kElems;
// upper bound on the warps of one launch
constexpr int64_t kMaxWarps = 152 * 64;

size_t workspace_bytes(int64_t, int64_t) { return kHeaderBytes; }

struct Params {
    const float* r;
    const float* v;  // GAE: values; null for the return
    const uint8_t* start;
    const float* boot;  // return: value after the tape's last step; GAE: v_boot
    float* out;
    int64_t B, L, G, seg_len;
    int vec;      // 16-byte loads and stores: L % 8 == 0 and aligned base pointers
    float c;      // per-step multiplier: gamma or gamma * lambda
    float gamma;  // GAE: the discount inside delta
};

// (A, X) maps G_in -> X + A G_in; compose(earlier, later) applies `later` first.
struct Aff {
    float a, x;
};
__device__ __forceinline__ Aff compose(Aff e, Aff l) { return Aff{e.a * l.a, fmaf(e.a, l.x, e.x)}; }

// first nonzero flag of st in [a, e), or -1; the same value in every lane.
// Each round trip covers 4 * 32 * 8 bytes (byte loads: no alignment needed).
__device__ int64_t find_flag(const uint8_t* st, int64_t a, int64_t e, int lane) {
    constexpr int kSpan = 4 * 32 * 8;
    for (int64_t base = a; base < e; base += kSpan) {
        int first = kSpan;
#pragma unroll
        for (int j = 4 * 8 - 1; j >= 0; --j) {
            // lane covers bytes [q * 256 + lane * 8, + 8) of this span for q = j / 8
            const int off = (j >> 3) * 256 + lane * 8 + (j & 7);
            const int64_t t = base + off;
            if (t < e && st[t] != 0) first = min(first, off);
        }
        // smallest offset over the lanes
#pragma unroll
        for (int s = 16; s > 0; s >>= 1) first = min(first, __shfl_xor_sync(0xffffffffu, first, s));
        if (first < kSpan) return base + first;
    }
    return -1;
}

// one lane's kElems steps of one chunk
struct Blk {
    float r[kElems], v[kElems];
    uint32_t s[kElems / 4];  // begin flags, packed 4 per word
};

template <bool GAE>
__device__ __forceinline__ void load_blk(Blk& d, const Params& p, const float* r, const float* v, const uint8_t* st,
                                         int64_t t0) {
    if (p.vec && t0 + kElems <= p.L) {
        const float4 r0 = __ldcs(reinterpret_cast<const float4*>(r + t0));
        const float4 r1 = __ldcs(reinterpret_cast<const float4*>(r + t0 + 4));
        d.r[0] = r0.x; d.r[1] = r0.y; d.r[2] = r0.z; d.r[3] = r0.w;
        d.r[4] = r1.x; d.r[5] = r1.y; d.r[6] = r1.z; d.r[7] = r1.w;
        const uint2 sw = __ldcs(reinterpret_cast<const uint2*>(st + t0));
        d.s[0] = sw.x;
        d.s[1] = sw.y;
        if (GAE) {
            const float4 v0 = __ldcs(reinterpret_cast<const float4*>(v + t0));
            const float4 v1 = __ldcs(reinterpret_cast<const float4*>(v + t0 + 4));
            d.v[0] = v0.x; d.v[1] = v0.y; d.v[2] = v0.z; d.v[3] = v0.w;
            d.v[4] = v1.x; d.v[5] = v1.y; d.v[6] = v1.z; d.v[7] = v1.w;
        }
    } else {
        d.s[0] = d.s[1] = 0;
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
            const int64_t t = t0 + e;
            const bool in = t < p.L;
            d.r[e] = in ? r[t] : 0.f;
            d.s[e >> 2] |= static_cast<uint32_t>(in ? st[t] : 1) << (8 * (e & 3));
            if (GAE) d.v[e] = in ? v[t] : 0.f;
        }
    }
}

__device__ __forceinline__ bool flag_of(const Blk& d, int e) { return ((d.s[e >> 2] >> (8 * (e & 3))) & 0xffu) != 0; }

template <bool GAE>
__global__ void __launch_bounds__(kThreads) scan_kernel(const Params p) {
    const int lane = threadIdx.x & 31;
    const int64_t wid = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    if (wid >= p.B * p.G) return;
    const int64_t b = wid / p.G, g = wid % p.G;
    const int64_t a = g * p.seg_len;
    if (a >= p.L) return;
    const int64_t e_nom = min(a + p.seg_len, p.L);
    const uint8_t* st = p.start + b * p.L;
    // segment [lo, hi): lo the first begin flag of the range (step 0 for the
    // first range), hi the first begin flag after the range, else the tape's end
    const int64_t lo = g == 0 ? 0 : find_flag(st, a, e_nom, lane);
    if (lo < 0) return;  // no episode starts here: the segment before covers the range
    int64_t hi = e_nom < p.L ? find_flag(st, e_nom, p.L, lane) : -1;
    if (hi < 0) hi = p.L;

    const float* r = p.r + b * p.L;
    const float* v = GAE ? p.v + b * p.L : nullptr;
    float* o = p.out + b * p.L;
    const float boot = p.boot != nullptr ? p.boot[b] : 0.f;
    // value entering the segment's last step from after it: the bootstrap at the
    // tape's end (return only; the advantage after the tape is 0)
    float carry = (!GAE && hi == p.L) ? boot : 0.f;
    // begin flag and value of the step after the current chunk (lane 31's successor):
    // for the segment's last chunk that step is hi, a begin flag or past the tape
    bool next_flag = true;
    float next_v = 0.f;

    const int64_t k_last = (hi - 1) / kChunk, k_first = lo / kChunk;
    Blk cur;
    load_blk<GAE>(cur, p, r, v, st, k_last * kChunk + lane * kElems);
    for (int64_t k = k_last; k >= k_first; --k) {
        const int64_t t0 = k * kChunk + lane * kElems;
        Blk nxt;
        if (k > k_first) load_blk<GAE>(nxt, p, r, v, st, t0 - kChunk);
        // successor of this lane's last step: the next lane's first step
        const bool f_up = __shfl_down_sync(0xffffffffu, flag_of(cur, 0) ? 1 : 0, 1) != 0;
        const float v_up = GAE ? __shfl_down_sync(0xffffffffu, cur.v[0], 1) : 0.f;
        const bool succ_flag = lane == 31 ? next_flag : f_up;
        const float succ_v = lane == 31 ? next_v : v_up;
        next_flag = __shfl_sync(0xffffffffu, flag_of(cur, 0) ? 1 : 0, 0) != 0;
        if (GAE) next_v = __shfl_sync(0xffffffffu, cur.v[0], 0);

        float x[kElems], m[kElems];
#pragma unroll
        for (int e = 0; e < kElems; ++e) {
            const int64_t t = t0 + e;
            if (t >= lo && t < hi) {
                const bool last = t + 1 >= p.L;
                const bool sflag = e + 1 < kElems ? flag_of(cur, e + 1) : succ_flag;
                const bool cont = !last && !sflag;  // the next step is in the same episode
                m[e] = (last || cont) ? p.c : 0.f;
                if (GAE) {
                    const float vn = e + 1 < kElems ? cur.v[e + 1] : succ_v;
                    const float nv = last ? boot : (cont ? vn : 0.f);
                    x[e] = fmaf(p.gamma, nv, cur.r[e]) - cur.v[e];
                } else {
                    x[e] = cur.r[e];
                }
            } else {
                m[e] = 1.f;  // identity outside the segment
                x[e] = 0.f;
            }
        }
        // this lane's map: G at its first step as a function of G after its last
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
        // map of everything after this lane's last step within the chunk
        const float na = __shfl_down_sync(0xffffffffu, suf.a, 1);
        const float nx = __shfl_down_sync(0xffffffffu, suf.x, 1);
        const Aff after = lane < 31 ? Aff{na, nx} : Aff{1.f, 0.f};
        float gin = fmaf(after.a, carry, after.x);
        // the chunk's value at its first step is the carry into the chunk before it
        const float wa = __shfl_sync(0xffffffffu, suf.a, 0);
        const float wx = __shfl_sync(0xffffffffu, suf.x, 0);
        carry = fmaf(wa, carry, wx);
        float out[kElems];
#pragma unroll
        for (int e = kElems - 1; e >= 0; --e) {
            gin = fmaf(m[e], gin, x[e]);
            out[e] = gin;
        }
        if (p.vec && t0 >= lo && t0 + kElems <= hi) {
            __stcs(reinterpret_cast<float4*>(o + t0), make_float4(out[0], out[1], out[2], out[3]));
            __stcs(reinterpret_cast<float4*>(o + t0 + 4), make_float4(out[4], out[5], out[6], out[7]));
        } else {
#pragma unroll
            for (int e = 0; e < kElems; ++e) {
                const int64_t t = t0 + e;
                if (t >= lo && t < hi) o[t] = out[e];
            }
        }
        cur = nxt;
    }
}

memoroid_status_t launch(const float* r, const float* v, const uint8_t* start, float c, float gamma,
                         const float* boot, float* out, int64_t B, int64_t L, void*, cudaStream_t s) {
    // one wave: as many warps as fit on the device at once, split evenly over the tapes
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    const cudaError_t oe = v != nullptr
        ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, scan_kernel<true>, kThreads, 0)
        : cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, scan_kernel<false>, kThreads, 0);
    if (oe != cudaSuccess) return MEMOROID_ERR_CUDA;
    int64_t warps = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1) * kWarps;
    if (warps > kMaxWarps) warps = kMaxWarps;
    int64_t G = warps / B;
    const int64_t max_g = (L + kChunk - 1) / kChunk;  // at least one chunk per segment
    if (G > max_g) G = max_g;
    if (G < 1) G = 1;
    const int64_t seg_len = (L + G - 1) / G;
    G = (L + seg_len - 1) / seg_len;

    auto aligned = [](const void* q, uintptr_t al) { return (reinterpret_cast<uintptr_t>(q) & (al - 1)) == 0; };
    // every tape then starts on a 32-byte boundary of r, v and out and an 8-byte one of start
    const bool vec = (L & 7) == 0 && aligned(r, 16) && (v == nullptr || aligned(v, 16)) && aligned(start, 8) &&
                     aligned(out, 16);
    const Params p{r, v, start, boot, out, B, L, G, seg_len, vec ? 1 : 0, c, gamma};
    const int64_t blocks = (B * G + kWarps - 1) / kWarps;
    if (blocks > 0x7fffffff) return MEMOROID_ERR_INVALID_ARG;
    if (v != nullptr)
        scan_kernel<true><<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(p);
    else
        scan_kernel<false><<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(p);
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

}  // namespace ret
}  // namespace memoroid
