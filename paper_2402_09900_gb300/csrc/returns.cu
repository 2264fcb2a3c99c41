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
// Each tape is cut into G ranges of seg_len steps, one warp each, which
// scans its range from the value entering it from the right.  Those values
// come from a resettable scan over the ranges.  Every range publishes its
// affine map G_start = X + A G_after, where only the steps up to its first
// cut matter (a step whose successor starts an episode has m_t = 0, so X
// stops there and A = 0), and composes, in a fixed order, the maps of the
// ranges after it up to the first cut (or the tape's end and its bootstrap).
// Warps take tickets in order and ranges are handed out from each tape's end,
// so a warp only ever waits for maps of warps that started before it.  With a
// cut, the steps before it are final from a zero value (they are written
// while the map is formed) and the rest are scanned once the carry is known:
// one pass over the tape.  Without one, the range is read twice (for its map,
// then for its outputs).  So a tape without begin flags runs on as many warps
// as any other.
// A warp walks its range backwards in chunks of 32 * kElems steps on
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
#include "ptx.cuh"

namespace memoroid {
namespace ret {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kElems = 8;
constexpr int kChunk = 32 * kElems;
// upper bound on the warps of one launch
constexpr int64_t kMaxWarps = 152 * 64;

// header (error word, ticket counter), then the ranges' maps (A, X) as two
// tagged 64-bit words each: at most kMaxWarps of them (with more than one
// range per tape, B * G <= the warps of one launch)
constexpr size_t kMapBytes = static_cast<size_t>(kMaxWarps) * 16;
size_t workspace_bytes(int64_t, int64_t) { return kHeaderBytes + kMapBytes; }

struct Params {
    const float* r;
    const float* v;  // GAE: values; null for the return
    const uint8_t* start;
    const float* boot;  // return: value after the tape's last step; GAE: v_boot
    float* out;
    unsigned long long* maps;  // [B * G][2]: (A, X) of each range, each value next to the launch's tag
    uint32_t* hdr;             // [0] error word, [1] ticket counter
    int64_t B, L, G, seg_len;
    int vec;      // 16-byte loads and stores: L % 8 == 0 and aligned base pointers
    float c;      // per-step multiplier: gamma or gamma * lambda
    float gamma;  // GAE: the discount inside delta
    uint32_t epoch;
    uint64_t wait_ns;
};

// (A, X) maps G_in -> X + A G_in; compose(earlier, later) applies `later` first.
struct Aff {
    float a, x;
};
__device__ __forceinline__ Aff compose(Aff e, Aff l) { return Aff{e.a * l.a, fmaf(e.a, l.x, e.x)}; }

// first nonzero flag of st in [a, e), or -1; the same value in every lane.
// Each round trip covers 4 * 32 * 8 bytes.  With `vec` (st 8-byte aligned)
// every lane loads four aligned 8-byte words from a base rounded down to 8
// bytes, and the bytes outside [a, e) are masked; otherwise byte loads.
__device__ int64_t find_flag(const uint8_t* st, int64_t a, int64_t e, int lane, bool vec) {
    constexpr int kSpan = 4 * 32 * 8;
    for (int64_t base = vec ? (a & ~int64_t{7}) : a; base < e; base += kSpan) {
        int first = kSpan;
        if (vec) {
#pragma unroll
            for (int q = 3; q >= 0; --q) {
                // lane covers bytes [q * 256 + lane * 8, + 8) of this span
                const int off = q * 256 + lane * 8;
                const int64_t t = base + off;
                if (t < e) {
                    unsigned long long w = *reinterpret_cast<const unsigned long long*>(st + t);
                    // bytes before a or at / after e do not count
                    if (t < a) w &= ~0ull << (8 * (a - t));
                    if (t + 8 > e) w &= ~0ull >> (8 * (t + 8 - e));
                    if (w != 0ull) first = min(first, off + (__ffsll(static_cast<long long>(w)) - 1) / 8);
                }
            }
        } else {
#pragma unroll
            for (int j = 4 * 8 - 1; j >= 0; --j) {
                const int off = (j >> 3) * 256 + lane * 8 + (j & 7);
                const int64_t t = base + off;
                if (t < e && st[t] != 0) first = min(first, off);
            }
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

// Walks steps [lo, hi) of tape b backwards from the value `carry` entering step
// hi - 1 from after it; next_flag / next_v: the begin flag and V of step hi
// (true / 0 past the tape).  OUT: writes every step's value.  Returns the
// value at step lo.  Warp-wide.
template <bool GAE, bool OUT>
__device__ float walk(const Params& p, int64_t b, int64_t lo, int64_t hi, float carry, bool next_flag, float next_v,
                      int lane) {
    const float* r = p.r + b * p.L;
    const float* v = GAE ? p.v + b * p.L : nullptr;
    const uint8_t* st = p.start + b * p.L;
    float* o = p.out + b * p.L;
    const float boot = p.boot != nullptr ? p.boot[b] : 0.f;
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
        // the step after this chunk's last one: hi (the caller's) for the range's
        // last chunk, else the first step of the chunk after it
        const bool succ_flag = lane == 31 ? next_flag : f_up;
        const float succ_v = lane == 31 ? next_v : v_up;
        next_flag = __shfl_sync(0xffffffffu, flag_of(cur, 0) ? 1 : 0, 0) != 0;
        if (GAE) next_v = __shfl_sync(0xffffffffu, cur.v[0], 0);

        float x[kElems], m[kElems];
        // a chunk inside [lo, hi) that ends before the tape's last step: no per-step range
        // or tape-end tests (the same values as the general loop below)
        const int64_t c0 = k * kChunk;
        if (c0 >= lo && c0 + kChunk <= hi && c0 + kChunk < p.L) {
#pragma unroll
            for (int e = 0; e < kElems; ++e) {
                const bool sflag = e + 1 < kElems ? flag_of(cur, e + 1) : succ_flag;
                m[e] = sflag ? 0.f : p.c;
                if (GAE) {
                    const float vn = e + 1 < kElems ? cur.v[e + 1] : succ_v;
                    x[e] = fmaf(p.gamma, sflag ? 0.f : vn, cur.r[e]) - cur.v[e];
                } else {
                    x[e] = cur.r[e];
                }
            }
        } else {
#pragma unroll
            for (int e = 0; e < kElems; ++e) {
                const int64_t t = t0 + e;
                if (t >= lo && t < hi) {
                    const bool last = t + 1 >= p.L;
                    // the successor: inside the lane's block (loaded from memory even past hi),
                    // or for the block's last step the next lane's first (hi for lane 31)
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
                    m[e] = 1.f;  // identity outside the range
                    x[e] = 0.f;
                }
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
        if (OUT) {
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
        }
        cur = nxt;
    }
    return carry;
}

__device__ __forceinline__ unsigned long long tagged(uint32_t epoch, float v) {
    return (static_cast<unsigned long long>(epoch) << 32) | __float_as_uint(v);
}

// 4 (return) or 3 (GAE) CTAs per SM: the GAE variant would otherwise take 89
// registers and fit 2
template <bool GAE>
__global__ void __launch_bounds__(kThreads, GAE ? 3 : 4) scan_kernel(const Params p) {
    const int lane = threadIdx.x & 31;
    // ticket -> (tape, range): position 0 is each tape's last range
    uint32_t tk = 0;
    if (lane == 0) tk = atomicAdd(p.hdr + 1, 1u);
    tk = __shfl_sync(0xffffffffu, tk, 0);
    if (static_cast<int64_t>(tk) >= p.B * p.G) return;
    const int64_t b = tk % p.B, g = p.G - 1 - static_cast<int64_t>(tk / p.B);
    const int64_t a = g * p.seg_len;
    const int64_t e = min(a + p.seg_len, p.L);
    const uint8_t* st = p.start + b * p.L;
    const bool nf_e = e < p.L ? st[e] != 0 : true;  // begin flag of the step after the range
    const float nv_e = (GAE && e < p.L) ? p.v[b * p.L + e] : 0.f;
    // the first cut: the first begin flag in (a, e] (step f - 1 does not see step f)
    const int64_t f = p.G > 1 ? find_flag(st, a + 1, min(e + 1, p.L), lane, p.vec != 0) : -1;
    const bool cut = f >= 0;
    if (p.G > 1) {
        // the range's map; with a cut its steps before f are final (written now)
        float x, A;
        if (cut) {
            x = walk<GAE, true>(p, b, a, f, 0.f, true, 0.f, lane);
            A = 0.f;
        } else {
            x = walk<GAE, false>(p, b, a, e, 0.f, nf_e, nv_e, lane);
            A = powf(p.c, static_cast<float>(e - a));
        }
        if (lane == 0) {
            unsigned long long* m = p.maps + 2 * (b * p.G + g);
            __stcg(m, tagged(p.epoch, A));
            __stcg(m + 1, tagged(p.epoch, x));
        }
    }
    // the value entering step e - 1 from after the range: the maps of the ranges
    // after it composed in order, batches of 32 from the nearest, up to the first
    // cut, applied to the value after the tape (the return's bootstrap; the
    // advantage after the tape is 0)
    const float after_tape = (!GAE && p.boot != nullptr) ? p.boot[b] : 0.f;
    Aff tot{1.f, 0.f};
    for (int64_t j0 = g + 1; j0 < p.G; j0 += 32) {
        const int64_t j = j0 + lane;
        Aff mj{1.f, 0.f};
        bool ok = true;
        if (j < p.G) {
            // published by a warp with an earlier ticket
            const unsigned long long* m = p.maps + 2 * (b * p.G + j);
            uint64_t t0 = 0;
            for (uint32_t it = 0;; ++it) {
                const unsigned long long wa = __ldcg(m), wx = __ldcg(m + 1);
                if (static_cast<uint32_t>(wa >> 32) == p.epoch && static_cast<uint32_t>(wx >> 32) == p.epoch) {
                    mj = Aff{__uint_as_float(static_cast<uint32_t>(wa)), __uint_as_float(static_cast<uint32_t>(wx))};
                    break;
                }
                if (it == 0) t0 = ptx::globaltimer();
                if ((it & 15u) == 15u && ptx::globaltimer() - t0 > p.wait_ns) {
                    ok = false;
                    break;
                }
            }
        }
        if (!__all_sync(0xffffffffu, ok)) {
            if (lane == 0) atomicCAS(p.hdr, 0u, static_cast<uint32_t>(DEV_LOOKBACK_TIMEOUT));
            return;
        }
        const unsigned cuts = __ballot_sync(0xffffffffu, j < p.G && mj.a == 0.f);
        // maps after the first cut do not reach this range
        if (cuts != 0u && lane > __ffs(cuts) - 1) mj = Aff{1.f, 0.f};
        // their composition in a fixed order (lane 0 earliest)
        Aff suf = mj;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float oa = __shfl_down_sync(0xffffffffu, suf.a, off);
            const float ox = __shfl_down_sync(0xffffffffu, suf.x, off);
            if (lane + off < 32) suf = compose(suf, Aff{oa, ox});
        }
        tot = compose(tot, Aff{__shfl_sync(0xffffffffu, suf.a, 0), __shfl_sync(0xffffffffu, suf.x, 0)});
        if (cuts != 0u) break;
    }
    const float carry = fmaf(tot.a, after_tape, tot.x);
    walk<GAE, true>(p, b, cut ? f : a, e, carry, nf_e, nv_e, lane);
}

memoroid_status_t launch(const float* r, const float* v, const uint8_t* start, float c, float gamma,
                         const float* boot, float* out, int64_t B, int64_t L, void* workspace, cudaStream_t s) {
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
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    const int64_t blocks = (B * G + kWarps - 1) / kWarps;
    if (blocks > 0x7fffffff || B * G >= 0xffffffffLL) return MEMOROID_ERR_INVALID_ARG;
    // B * G <= warps <= kMaxWarps whenever G > 1: the maps fit the workspace.  The
    // maps' tag; their region is zeroed where an old word could carry it.
    bool clear = false;
    const uint32_t epoch = tagged_epoch(workspace, kHeaderBytes + kMapBytes, s, &clear);
    if (cudaMemsetAsync(ws, 0, clear ? kHeaderBytes + kMapBytes : kHeaderBytes, s) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    const Params p{r, v, start, boot, out, reinterpret_cast<unsigned long long*>(ws + kHeaderBytes),
                   reinterpret_cast<uint32_t*>(ws), B, L, G, seg_len, vec ? 1 : 0, c, gamma, epoch,
                   debug_knobs().wait_ns};
    if (v != nullptr)
        scan_kernel<true><<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(p);
    else
        scan_kernel<false><<<static_cast<unsigned>(blocks), kThreads, 0, s>>>(p);
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

}  // namespace ret
}  // namespace memoroid
