// diag_scan.cu -- single-pass resettable diagonal scan (forward and reverse)
// for sm_103a.
//
// Semantics: the S5 / LRU memoroid with diagonal X (paper appendix,
// "Simplified State Space Models" / "Linear Recurrent Unit"),
//     (X, x) . (X', x') = (X' X, X' x + x'),   e_I = (1, 0),
// made resettable by Theorem 3.2: an element whose begin flag is set discards
// everything to its left, (A, b) o (A', 1) = (A', 1).  Per step the lifted
// element is ((lambda_t, u_t), b_t), so h_t = b_t ? u_t : lambda_t h_{t-1} + u_t.
// The backward pass is the same scan run right to left over
//     delta_t = grad_h_t + [b_{t+1} = 0] conj(lambda_{t+1}) delta_{t+1},
// i.e. the element of step t is (conj(lambda_{t+1}), grad_h_t, b_{t+1}), plus
// grad_lambda = sum_{b_t = 0} delta_t conj(h_{t-1}).
//
// Design (GB300-first; the paper itself ships no kernels):
//   * The tape [B, L, D] is cut into tiles of T steps x 64 complex channels
//     (a 512-byte row slab).  A "chain" is one (tape, slab) pair.  Tiles are
//     handed out in order by an atomic ticket, so a tile only ever waits on
//     tiles whose tickets were taken earlier by running CTAs.
//   * One CTA per tile, several CTAs resident per SM.  A CTA has W scan
//     warps and two look-back warps.  Each scan warp owns R consecutive steps
//     and each lane two complex channels (one 16-byte vector): a lane scans
//     its steps serially from the identity, then rescans them from its carry
//     and streams the outputs out with 16-byte stores.  HBM traffic is one
//     read of the inputs and one write of the outputs.
//   * Look-back warp 1 stages the tile into shared memory (one TMA tensor
//     load of T rows per staged array), folds the summaries it needs from earlier tiles while the
//     copies are in flight, and publishes the tile's own summary as soon as
//     the scan warps' partial aggregates are in; look-back warp 2 derives the
//     carry into the tile from earlier tiles' summaries, also starting at
//     once.  A summary never waits on a carry: if it did, every tile of a
//     chain would wait on the one before it.
//   * The look-back is deterministic: tile j publishes the aggregate of the
//     fixed range of tiles covered by Fenwick-tree node j+1, folded from its
//     Fenwick children in a fixed order, and its carry is the fixed
//     right-to-left fold of the Fenwick prefix nodes of position j.  Every
//     value is a function of the inputs alone, not of the order in which
//     CTAs happen to run: repeated calls are bit-identical, and changing one
//     episode leaves every other episode's outputs bit-identical.
//   * A summary is self-validating: each fp32 value is stored in a 64-bit
//     word next to a per-launch tag (and the summary's begin-flag bit), and
//     64-bit accesses are single-copy atomic, so a reader needs no separate
//     status flag and a writer no fence: a summary is complete once every
//     word carries this launch's tag.  Under a saturated memory system each
//     dependent round trip costs microseconds, so this halves the look-back
//     latency.
//   * Each chain is cut into G segments that are scanned as independent
//     chains from the identity, and tiles are handed out position-major over
//     all segments: the tile before a given tile in its chain was handed out
//     (chains x G) tickets earlier, long enough for its summary to be visible
//     when it is needed.  A small second pass then adds the true state
//     entering each segment to the steps of that segment before its first
//     begin flag (only those depend on it): for the step-t output the
//     correction is (product of the multipliers from the segment start to t)
//     times that state.  With episodes much shorter than a segment this
//     touches a few percent of the tape.
//   * A begin flag inside a summary's range discards everything to its left,
//     so folds stop at the first such summary; a tile whose first step is a
//     begin flag needs no carry at all.
//   * Every wait (TMA completion, look-back flags) is bounded by the global
//     timer; on expiry the kernel records an error in the workspace and
//     returns.
// grad_lambda (per-channel lambda) is accumulated per tile and reduced in a
// fixed order by two small kernels (fp32 within a part of a few dozen tiles,
// fp64 across parts), so it is deterministic as well.
#include <cuda_runtime.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace memoroid {
namespace diag {

constexpr int SLAB = 64;  // complex channels per slab
// 64-bit words per lane in a summary: (a, x) = 8 floats with a per-step lambda;
// x alone (4 floats) with a per-channel lambda, whose a is lambda^(steps in
// the summary's range) and is recomputed by the reader.
constexpr int NODE_WORDS = 8;
constexpr int NB_READ = 1;  // summaries read per round trip in a look-back fold
// Unroll factors of the per-step loops (measured: unrolling helps the
// backward scan and slows the forward one; the FFM forward, whose loops carry
// an x~ load and two planar stores per step, gains from 8: 0.499 -> 0.477 ms at
// L = 2^20, m = 64, c = 4, against 0.485 / 0.479 / 0.492 ms for 2 / 4 / 31).
constexpr int UNROLL_FWD = 1;
constexpr int UNROLL_FFM_FWD = 8;
constexpr int UNROLL_BWD = 32;
constexpr int RED_PARTS = 512;  // first-stage parts of the grad_lambda reduction


struct Params {
    // 3-D tensor maps {row floats, L, B} of the staged arrays, boxes of T rows:
    // the input (u / grad_h, or FFM x~ / grad_z), the forward states (backward)
    // and the per-step lambda
    CUtensorMap map_in, map_h, map_l;
    const float4* lambda;  // [D/2] or [B, L, D/2]; one float4 = two complex channels
    const float4* in;      // fwd: u; bwd: grad_h
    const uint8_t* start;  // [B, L]
    const float4* h0;      // [B, D/2] or null
    float4* out;           // fwd: h; bwd: grad_u
    float4* out_last;      // fwd: h_last or null
    const float4* h;       // bwd: forward states
    const float4* g_last;  // bwd: grad_h_last or null
    float4* grad_lambda;   // bwd, per-step lambda: [B, L, D/2] or null
    float4* grad_h0;       // bwd: [B, D/2] or null
    int64_t B, L, D2, n_slabs, n_tt, n_chains, n_tiles;
    int64_t n_seg, q_seg, n_sc;  // segments per chain, tiles per segment, segment chains
    uint32_t* hdr;               // workspace header: [0] error, [1] ticket counter, [4] fix-up list length
    unsigned long long* node;    // [n_sc * q_seg * 32 * NODE_WORDS] tagged Fenwick nodes
    float4* gpart;               // [n_chains * n_tt * 32]      per-tile grad_lambda
    uint32_t* fix;               // [n_chains * n_tt] tiles that need their segment's carry added (n_seg > 1),
                                 // a list of hdr[4] tile indices in completion order
    float4* pin;                 // [n_chains * n_tt * 32] product of multipliers from the segment start
    float4* segc;                // [n_chains * n_seg * 32] true state entering each segment
    float4* sega;                // [n_chains * n_seg * 32 * 2] each segment's aggregate (a, x)
    uint32_t* segb;              // [n_chains * n_seg] each segment holds a begin flag
    uint64_t wait_ns;
    int64_t withhold;
    uint32_t epoch;              // this launch's tag (31 bits, non-zero)
    int full_nodes;              // summaries store a (per-step lambda) or only x
    int T;                       // steps per tile
    int rag;                     // steps missing from the chain's first tile in processing order
    // Fast and Forgetful Memory layout (FFM configurations only): the forward
    // input is x~ [B, L, m], one real value per row i of the m x c state,
    // repeated over its c columns (channel i * c + j); states and their
    // gradients are stored as Re || Im halves [B, L, 2D] (same row size as
    // the interleaved layout); the backward writes grad_x~ [B, L, m] = the
    // sum over the c columns of Re(delta) instead of grad_u.
    const float* ffm_x;
    float* ffm_gx;
    int64_t ffm_m;
    int ffm_lc;  // log2 c
};

__host__ __device__ __forceinline__ int64_t lmin(int64_t a, int64_t b) { return a < b ? a : b; }

__host__ __device__ __forceinline__ int64_t lmax(int64_t a, int64_t b) { return a > b ? a : b; }

// ---- FFM layout: one lane's two channels (2 lane, 2 lane + 1 of the slab) ----
// The staged forward input holds x~ of the slab's rows i (rows of 64 / c
// floats, packed); channel 2 lane reads element (2 lane) >> log2 c of its row.
// Staged planar rows of a T-step tile: the Re halves of all rows (64 floats
// each), then the Im halves.
template <int T>
__device__ __forceinline__ float4 ffm_planar_pair(const float4* buf, int r, int lane) {
    const float2* b = reinterpret_cast<const float2*>(buf);
    const float2 re = b[r * 32 + lane], im = b[T * 32 + r * 32 + lane];
    return make_float4(re.x, im.x, re.y, im.y);
}
// global planar row (D2 float4 = 2D floats): float2 index col of Re, D2 + col of Im
__device__ __forceinline__ float4 ffm_load_planar(const float4* rowbase, int64_t D2, int64_t col) {
    const float2* r = reinterpret_cast<const float2*>(rowbase);
    const float2 re = r[col], im = r[D2 + col];
    return make_float4(re.x, im.x, re.y, im.y);
}
__device__ __forceinline__ void ffm_store_planar(float4* rowbase, int64_t D2, int64_t col, float4 v, bool stream) {
    float2* r = reinterpret_cast<float2*>(rowbase);
    if (stream) {
        __stcs(r + col, make_float2(v.x, v.z));
        __stcs(r + D2 + col, make_float2(v.y, v.w));
    } else {
        r[col] = make_float2(v.x, v.z);
        r[D2 + col] = make_float2(v.y, v.w);
    }
}
// grad_x~ of step row: Re of this lane's two channels summed over the c
// columns of their row i (a fixed butterfly over groups of c/2 lanes; lanes of
// a group are all active or all inactive, `mask` holds the active ones), then
// stored (accumulate = add to the stored value) by the group's first lane.
__device__ __forceinline__ void ffm_grad_x(const Params& p, int64_t row, int64_t col, float4 d, unsigned mask,
                                           bool active, bool accumulate, bool stream) {
    const int lane = threadIdx.x & 31;
    float* gx = p.ffm_gx + row * p.ffm_m;
    if (p.ffm_lc == 0) {  // c = 1: the two channels are two rows i
        if (active) {
            float2* g2 = reinterpret_cast<float2*>(gx + 2 * col);
            float2 v = make_float2(d.x, d.z);
            if (accumulate) {
                const float2 o = *g2;
                v = make_float2(o.x + v.x, o.y + v.y);
            }
            if (stream) __stcs(g2, v);
            else *g2 = v;
        }
        return;
    }
    float v = d.x + d.z;
    const int group = 1 << (p.ffm_lc - 1);  // lanes per row i
    for (int o = 1; o < group; o <<= 1) v += __shfl_xor_sync(mask, v, o);
    if (active && (lane & (group - 1)) == 0) {
        float* g = gx + ((2 * col) >> p.ffm_lc);
        if (accumulate) v += *g;
        if (stream) __stcs(g, v);
        else *g = v;
    }
}

// ---- two complex numbers per float4: (re0, im0, re1, im1) -------------------
__device__ __forceinline__ float4 one2() { return make_float4(1.f, 0.f, 1.f, 0.f); }
__device__ __forceinline__ float4 zero2() { return make_float4(0.f, 0.f, 0.f, 0.f); }
__device__ __forceinline__ float4 cmul2(float4 a, float4 b) {
    return make_float4(fmaf(a.x, b.x, -a.y * b.y), fmaf(a.x, b.y, a.y * b.x),
                       fmaf(a.z, b.z, -a.w * b.w), fmaf(a.z, b.w, a.w * b.z));
}
// a * b + c
__device__ __forceinline__ float4 cfma2(float4 a, float4 b, float4 c) {
    return make_float4(fmaf(a.x, b.x, fmaf(-a.y, b.y, c.x)), fmaf(a.x, b.y, fmaf(a.y, b.x, c.y)),
                       fmaf(a.z, b.z, fmaf(-a.w, b.w, c.z)), fmaf(a.z, b.w, fmaf(a.w, b.z, c.w)));
}
__device__ __forceinline__ float4 conj2(float4 a) { return make_float4(a.x, -a.y, a.z, -a.w); }
__device__ __forceinline__ float4 add2(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}

// ---- tile shapes -------------------------------------------------------------
// W warps x R steps per warp; REV = backward; PS = per-step lambda; FFM = the
// Fast and Forgetful Memory layout (broadcast input, planar states); LC =
// log2 c fixed at compile time (the FFM forward), -1 = taken from the parameters.
template <int W_, int R_, bool REV_, bool PS_, bool FFM_ = false, int LC_ = -1>
struct Cfg {
    static constexpr int W = W_, R = R_, T = W_ * R_;
    static constexpr bool REV = REV_, PS = PS_, FFM = FFM_;
    static constexpr int LC = LC_;
    static_assert(!(PS_ && FFM_), "the FFM multiplier is per channel");
    static constexpr int UNROLL = REV_ ? UNROLL_BWD : (FFM_ ? UNROLL_FFM_FWD : UNROLL_FWD);
    // arrays staged per tile: input [, h (backward)] [, lambda (per step)]
    static constexpr int NB = 1 + (REV_ ? 1 : 0) + (PS_ ? 1 : 0);
    // float4 per staged array: a 512-byte row per step, or for the FFM forward
    // the row's x~ (at most 64 floats, c = 1)
    static constexpr int BUF_F4 = (FFM_ && !REV_) ? T * 16 : T * 32;
    static constexpr int THREADS = (W_ + 2) * 32;  // W scan warps + 2 look-back warps
    static constexpr int NSYNC = (W_ + 1) * 32;    // scan warps + one look-back warp
    // shared memory layout (bytes)
    static constexpr size_t OFF_WA = size_t(NB) * BUF_F4 * 16;
    static constexpr size_t OFF_WX = OFF_WA + W_ * 32 * 16;
    static constexpr size_t OFF_CARRY = OFF_WX + W_ * 32 * 16;
    static constexpr size_t OFF_ACC = OFF_CARRY + 32 * 16;
    static constexpr size_t OFF_WR = OFF_ACC + ((REV_ && !PS_) ? W_ * 32 * 16 : 0);
    static constexpr size_t OFF_MISC = (OFF_WR + W_ * 4 + 15) / 16 * 16;  // bar, ticket, abort, h bar
    static constexpr size_t SMEM = OFF_MISC + 32;
    static_assert(R_ < 32, "R + 1 begin flags are read by one warp");
};

struct Tile {
    int64_t tk;      // ticket
    int64_t b, c2;   // tape, first float4 column of the slab
    int64_t chain;   // tape * n_slabs + slab
    int64_t g;       // segment of the chain
    int64_t pos;     // position in the segment (left-to-right forward, right-to-left backward)
    int64_t jt;      // time tile
    int64_t t0;      // first step
    int64_t fbase;   // first node of the segment chain
    int width2;      // float4 columns in the slab
    int nrows;       // steps in the tile
    bool valid;      // the ticket maps to a tile (the last segment may be shorter)
};

// Tickets are position-major over the segment chains: ticket = pos * n_sc + sc,
// sc = g * n_chains + chain, so the slabs of the same steps are handed out
// together (their rows share DRAM pages).
template <class C>
__device__ __forceinline__ Tile decode(const Params& p, int64_t tk) {
    Tile t{};
    t.tk = tk;
    const int64_t q = tk / p.n_sc;
    const int64_t sc = tk - q * p.n_sc;
    t.g = sc / p.n_chains;
    t.chain = sc - t.g * p.n_chains;
    t.pos = q;
    const int64_t jg = t.g * p.q_seg + q;  // position in the whole chain
    t.valid = (q < p.q_seg) && (jg < p.n_tt);
    t.jt = C::REV ? p.n_tt - 1 - jg : jg;
    t.b = t.chain / p.n_slabs;
    t.c2 = (t.chain - t.b * p.n_slabs) * (SLAB / 2);
    t.width2 = static_cast<int>(lmin(SLAB / 2, p.D2 - t.c2));
    t.t0 = t.jt * C::T;
    t.nrows = static_cast<int>(lmin(C::T, p.L - t.t0));
    t.fbase = sc * p.q_seg;
    return t;
}

// ---- errors and bounded waits -------------------------------------------------
__device__ __forceinline__ void record_error(const Params& p, uint32_t code, int64_t ticket) {
    if (atomicCAS(p.hdr, 0u, code) == 0u) {
        *reinterpret_cast<volatile unsigned long long*>(p.hdr + 2) =
            static_cast<unsigned long long>(ticket);
    }
}

// Publishes this lane's part of a Fenwick node (tile index idx): [a,] x and
// the begin-flag bit, each value tagged with the launch's epoch.
__device__ __forceinline__ void store_node(const Params& p, int64_t idx, float4 a, float4 x, bool b) {
    const int lane = threadIdx.x & 31;
    unsigned long long* dst = p.node + (idx * 32 + lane) * NODE_WORDS;
    const unsigned long long hi = static_cast<unsigned long long>((p.epoch << 1) | (b ? 1u : 0u)) << 32;
    auto w = [&](float v) { return hi | static_cast<unsigned long long>(__float_as_uint(v)); };
    ptx::st_relaxed_v2u64(dst + 0, w(x.x), w(x.y));
    ptx::st_relaxed_v2u64(dst + 2, w(x.z), w(x.w));
    if (p.full_nodes) {
        ptx::st_relaxed_v2u64(dst + 4, w(a.x), w(a.y));
        ptx::st_relaxed_v2u64(dst + 6, w(a.z), w(a.w));
    }
}

// m^n for the two complex numbers of a float4, by repeated squaring.
__device__ __forceinline__ float4 cpow2(float4 m, int64_t n) {
    float4 r = one2();
    while (n > 0) {
        if (n & 1) r = cmul2(r, m);
        m = cmul2(m, m);
        n >>= 1;
    }
    return r;
}

// Reads this lane's part of Fenwick node `pos` (1-based) of a segment chain.
// Returns true if all of its words carry this launch's tag (then b holds the
// node's begin-flag bit).  Without stored a, a = mul^(steps in the node's
// range); rag = steps missing from the segment chain's first tile.
__device__ __forceinline__ bool load_node(const Params& p, int64_t fbase, int64_t pos, float4 mul,
                                          int rag, float4& a, float4& x, bool& b) {
    const int lane = threadIdx.x & 31;
    const unsigned long long* src = p.node + ((fbase + pos - 1) * 32 + lane) * NODE_WORDS;
    unsigned long long w[NODE_WORDS];
    ptx::ld_relaxed_v2u64(src + 0, w[0], w[1]);
    ptx::ld_relaxed_v2u64(src + 2, w[2], w[3]);
    const int nw = p.full_nodes ? 8 : 4;
    if (p.full_nodes) {
        ptx::ld_relaxed_v2u64(src + 4, w[4], w[5]);
        ptx::ld_relaxed_v2u64(src + 6, w[6], w[7]);
    }
    bool ok = true;
#pragma unroll
    for (int i = 0; i < NODE_WORDS; ++i) ok = ok && (i >= nw || static_cast<uint32_t>(w[i] >> 33) == p.epoch);
    b = (w[0] >> 32) & 1u;
    auto f = [&](int i) { return __uint_as_float(static_cast<uint32_t>(w[i])); };
    x = make_float4(f(0), f(1), f(2), f(3));
    if (p.full_nodes) {
        a = make_float4(f(4), f(5), f(6), f(7));
    } else {
        const int64_t lb = pos & (-pos);
        const int64_t steps = lb * p.T - ((pos == lb) ? rag : 0);
        a = b ? one2() : cpow2(mul, steps);  // a of a range holding a begin flag is never used
    }
    return ok;
}

// Folds the Fenwick nodes whose positions lanes 0..n-1 hold in `mypos`
// (lane 0 the right-most) onto the left of (Ra, Rx, Rb) in that order:
// node o R = (R.a * node.a, R.a * node.x + R.x, node.b) while R holds no begin
// flag.  The fold stops after the first node whose range holds one (every
// node further left would be discarded by the select of Theorem 3.2, so
// stopping changes no bit).  Nodes are read NB_READ at a time and re-read
// until every lane sees them complete.  Warp-wide; false on timeout / error.
__device__ bool fold_nodes(const Params& p, int64_t fbase, int64_t mypos, int n, float4 mul, int rag,
                           float4& Ra, float4& Rx, bool& Rb, int64_t ticket) {
    for (int m0 = 0; m0 < n && !Rb; m0 += NB_READ) {
        int64_t pk[NB_READ];
#pragma unroll
        for (int k = 0; k < NB_READ; ++k) pk[k] = __shfl_sync(0xffffffffu, mypos, (m0 + k) & 31);
        const int cnt = n - m0 < NB_READ ? n - m0 : NB_READ;
        uint32_t pending = (1u << cnt) - 1u;
        float4 a[NB_READ], x[NB_READ];
        bool rb[NB_READ];
        uint64_t t0 = 0;
        for (uint32_t it = 0; pending != 0u; ++it) {
#pragma unroll
            for (int k = 0; k < NB_READ; ++k) {
                if ((pending >> k) & 1u) {
                    const bool ok = load_node(p, fbase, pk[k], mul, rag, a[k], x[k], rb[k]);
                    if (__all_sync(0xffffffffu, ok)) pending &= ~(1u << k);
                }
            }
            if (pending == 0u) break;
            if (it == 0) t0 = ptx::globaltimer();
            if ((it & 15u) == 15u) {
                if (ptx::ld_relaxed(p.hdr) != 0u) return false;
                if (ptx::globaltimer() - t0 > p.wait_ns) {
                    if ((threadIdx.x & 31) == 0) record_error(p, DEV_LOOKBACK_TIMEOUT, ticket);
                    return false;
                }
            }
        }
#pragma unroll
        for (int k = 0; k < NB_READ; ++k) {
            if (k < cnt && !Rb) {
                Rx = cfma2(Ra, x[k], Rx);
                Ra = cmul2(Ra, a[k]);
                Rb = rb[k];
            }
        }
    }
    return true;
}

// Fenwick node pos (1-based; tile pos-1 of the chain) covers tiles
// [pos - lowbit(pos), pos - 1].  Its children are the nodes pos - k for
// k = 1, 2, 4, .. < lowbit(pos); they cover the same range minus tile pos-1.
// Returns the children folded right to left, C = child(pos - lowbit/2) o ...
// o child(pos - 1) (the identity if there are none).
__device__ bool fenwick_children(const Params& p, int64_t fbase, int64_t pos, float4 mul, int rag,
                                 float4& Ca, float4& Cx, bool& Cb, int64_t ticket) {
    const int lane = threadIdx.x & 31;
    const int64_t lb = pos & (-pos);
    const int nc = 63 - __clzll(static_cast<long long>(lb));  // log2(lowbit(pos))
    Ca = one2();
    Cx = zero2();
    Cb = false;
    if (nc == 0) return true;
    const int64_t child = pos - (int64_t(1) << (lane < nc ? lane : 0));
    return fold_nodes(p, fbase, child, nc, mul, rag, Ca, Cx, Cb, ticket);
}

// Publishes node j+1 = C o T (T: the tile's own aggregate) unless !ok or the
// debug knob withholds it.  Warp-wide.
__device__ void fenwick_publish(const Params& p, int64_t fbase, int64_t j, float4 Ca, float4 Cx, bool Cb,
                                float4 Ta, float4 Tx, bool Tb, bool ok, bool skip) {
    if (!ok || skip) return;
    const float4 Na = Tb ? Ta : cmul2(Ta, Ca);
    const float4 Nx = Tb ? Tx : cfma2(Ta, Cx, Tx);
    store_node(p, fbase + j, Na, Nx, Tb || Cb);
}

// State entering segment position j > 0: the Fenwick prefix nodes of
// position j (j, j - lowbit(j), ...) folded right to left into (Ra, Rx, Rb)
// and applied to `base` (the state before the segment's first step) unless a
// begin flag intervenes.  Warp-wide.
__device__ bool fenwick_carry(const Params& p, int64_t fbase, int64_t j, float4 mul, int rag, float4 base,
                              float4& carry, float4& Ra, float4& Rx, bool& Rb, int64_t ticket) {
    const int lane = threadIdx.x & 31;
    int64_t q = j;  // lane i holds the i-th prefix node position
    for (int k = 0; k < lane && q > 0; ++k) q -= q & (-q);
    const int nq = __popcll(static_cast<unsigned long long>(j));
    Rx = zero2();
    Ra = one2();
    Rb = false;
    if (!fold_nodes(p, fbase, q, nq, mul, rag, Ra, Rx, Rb, ticket)) return false;
    carry = Rb ? Rx : cfma2(Ra, base, Rx);
    return true;
}

// ============================================================================
// the scan kernel (forward: REV = false; backward: REV = true), one tile per CTA
// ============================================================================
template <class C>
__global__ void __launch_bounds__(C::THREADS) diag_scan_kernel(const __grid_constant__ Params p) {
    constexpr int W = C::W, R = C::R;
    constexpr int LB_PUBLISH = W, LB_CARRY = W + 1;  // the two look-back warps
    // named barriers: 1 aggregates ready (scan warps -> publisher),
    // 2 carry ready (carry warp <-> scan warps), 3 grad_lambda parts ready
    constexpr int BAR_AGG = 1, BAR_CARRY = 2, BAR_ACC = 3;
    extern __shared__ __align__(128) unsigned char smem[];
    float4* s_in = reinterpret_cast<float4*>(smem);                     // [T][32] input rows
    float4* s_h = s_in + C::BUF_F4;                                       // [T][32] h_{t-1} (backward)
    float4* s_l = s_in + (C::NB - 1) * C::BUF_F4;                         // [T][32] lambda (per step)
    float4* s_wa = reinterpret_cast<float4*>(smem + C::OFF_WA);          // [W][32] warp aggregate a
    float4* s_wx = reinterpret_cast<float4*>(smem + C::OFF_WX);          // [W][32] warp aggregate x
    float4* s_carry = reinterpret_cast<float4*>(smem + C::OFF_CARRY);    // [32] carry into the tile
    float4* s_acc = reinterpret_cast<float4*>(smem + C::OFF_ACC);        // [W][32] grad_lambda parts
    uint32_t* s_wr = reinterpret_cast<uint32_t*>(smem + C::OFF_WR);      // [W] warp holds a reset
    uint64_t* bar = reinterpret_cast<uint64_t*>(smem + C::OFF_MISC);
    uint64_t* bar_h = reinterpret_cast<uint64_t*>(smem + C::OFF_MISC + 24);  // h_{t-1} rows (backward)
    long long* s_tk = reinterpret_cast<long long*>(smem + C::OFF_MISC + 8);
    volatile int* s_abort = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 16);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        *s_tk = static_cast<long long>(atomicAdd(p.hdr + 1, 1u));
        *s_abort = 0;
        ptx::mbar_init(bar, 1);
        if (C::REV) ptx::mbar_init(bar_h, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    const int64_t tk = *s_tk;
    const Tile t = decode<C>(p, tk);
    if (!t.valid) return;  // uniform over the CTA: the ticket has no tile
    const bool lane_ok = lane < t.width2;
    // multiplier whose powers rebuild the a of summaries stored without it
    float4 node_mul = one2();
    if (!C::PS && lane_ok) node_mul = C::REV ? conj2(p.lambda[t.c2 + lane]) : p.lambda[t.c2 + lane];
    const int node_rag = (t.g == 0) ? p.rag : 0;

    if (warp == LB_PUBLISH) {
        // ----------------------------------------- stage the tile, publish its summary
        // one box of T rows per staged array; rows past the tape (and the row
        // before step 0) read as zeros, and every box counts in full.  The
        // backward's h_{t-1} rows complete on a barrier of their own: only the
        // rescan reads them, so the first pass starts as soon as grad_h is in
        if (lane == 0) {
            const int x = static_cast<int>(4 * t.c2), y = static_cast<int>(t.t0), z = static_cast<int>(t.b);
            constexpr uint32_t BOX = C::T * 512u;  // a full 512-byte row per step
            if (C::FFM && !C::REV) {
                ptx::mbar_arrive_expect_tx(bar, static_cast<uint32_t>(C::T) * static_cast<uint32_t>(256 >> p.ffm_lc));
                ptx::tma_load_3d(ptx::smem_addr(s_in), &p.map_in, static_cast<int>((2 * t.c2) >> p.ffm_lc), y, z, bar);
            } else if (C::FFM) {
                // Re halves at x = 2 c2, Im halves at x = D + 2 c2 (floats), T x 256 bytes each
                const int re = static_cast<int>(2 * t.c2), im = static_cast<int>(2 * p.D2 + 2 * t.c2);
                ptx::mbar_arrive_expect_tx(bar, BOX);
                ptx::tma_load_3d(ptx::smem_addr(s_in), &p.map_in, re, y, z, bar);
                ptx::tma_load_3d(ptx::smem_addr(s_in + C::T * 16), &p.map_in, im, y, z, bar);
                ptx::mbar_arrive_expect_tx(bar_h, BOX);
                ptx::tma_load_3d(ptx::smem_addr(s_h), &p.map_h, re, y - 1, z, bar_h);
                ptx::tma_load_3d(ptx::smem_addr(s_h + C::T * 16), &p.map_h, im, y - 1, z, bar_h);
            } else {
                ptx::mbar_arrive_expect_tx(bar, BOX * (C::NB - (C::REV ? 1 : 0)));
                ptx::tma_load_3d(ptx::smem_addr(s_in), &p.map_in, x, y, z, bar);
                if (C::PS) ptx::tma_load_3d(ptx::smem_addr(s_l), &p.map_l, x, y + (C::REV ? 1 : 0), z, bar);
                if (C::REV) {
                    ptx::mbar_arrive_expect_tx(bar_h, BOX);
                    ptx::tma_load_3d(ptx::smem_addr(s_h), &p.map_h, x, y - 1, z, bar_h);
                }
            }
        }
        __syncwarp();
        float4 Ca, Cx;
        bool Cb;
        bool ok = fenwick_children(p, t.fbase, t.pos + 1, node_mul, node_rag, Ca, Cx, Cb, tk);
        ptx::named_sync(BAR_AGG, C::NSYNC);
        // the tile's aggregate: the scan warps' aggregates folded in processing order
        float4 Ta = one2(), Tx = zero2();
        bool Tb = false;
        for (int k = 0; k < W; ++k) {
            const int v = C::REV ? W - 1 - k : k;
            const float4 wa = s_wa[v * 32 + lane], wx = s_wx[v * 32 + lane];
            if (s_wr[v]) {
                Ta = wa;
                Tx = wx;
                Tb = true;
            } else {
                Tx = cfma2(wa, Tx, wx);
                Ta = cmul2(wa, Ta);
            }
        }
        ok = ok && (*s_abort == 0);
        fenwick_publish(p, t.fbase, t.pos, Ca, Cx, Cb, Ta, Tx, Tb, ok, tk == p.withhold);
        return;
    }

    if (warp == LB_CARRY) {
        // ------------------------------------------------- carry into the tile
        bool need_carry;
        float4 base = zero2();
        if (!C::REV) {
            need_carry = p.start[t.b * p.L + t.t0] == 0;
            if (p.h0 != nullptr && lane_ok) base = p.h0[t.b * p.D2 + t.c2 + lane];
        } else {
            // the first step processed is t0 + nrows - 1; its carry is cut if b_{t0+nrows} = 1
            const int64_t tn = t.t0 + t.nrows;
            need_carry = !(tn < p.L && p.start[t.b * p.L + tn] != 0);
            if (p.g_last != nullptr && lane_ok) base = p.g_last[t.b * p.D2 + t.c2 + lane];
        }
        if (t.g > 0) base = zero2();  // later segments start from the identity; fixed up afterwards
        float4 carry = base, Ra = one2(), Rx = zero2();
        bool Rb = false, ok = true;
        if (need_carry && t.pos > 0)
            ok = fenwick_carry(p, t.fbase, t.pos, node_mul, node_rag, base, carry, Ra, Rx, Rb, tk);
        if (p.fix != nullptr) {
            // steps of this tile before its first begin flag miss the state entering the segment
            const int64_t tid = t.chain * p.n_tt + t.jt;
            const bool partial = (t.g > 0) && need_carry && !Rb;
            if (partial) {
                p.pin[tid * 32 + lane] = Ra;
                if (lane == 0) p.fix[atomicAdd(p.hdr + 4, 1u)] = static_cast<uint32_t>(tid);
            }
        }
        s_carry[lane] = carry;
        if (!ok && lane == 0) *s_abort = 1;
        ptx::named_sync(BAR_CARRY, C::NSYNC);
        if (p.fix != nullptr && *s_abort == 0 && t.pos == lmin(p.q_seg, p.n_tt - t.g * p.q_seg) - 1) {
            // last tile of its segment: the segment's aggregate, T o R, for the carry pass
            // (the scan warps' aggregates are visible here: they were written before BAR_CARRY)
            float4 Ta = one2(), Tx = zero2();
            bool Tb = false;
            for (int k = 0; k < W; ++k) {
                const int v = C::REV ? W - 1 - k : k;
                const float4 wa = s_wa[v * 32 + lane], wx = s_wx[v * 32 + lane];
                if (s_wr[v]) {
                    Ta = wa;
                    Tx = wx;
                    Tb = true;
                } else {
                    Tx = cfma2(wa, Tx, wx);
                    Ta = cmul2(wa, Ta);
                }
            }
            const int64_t si = t.chain * p.n_seg + t.g;
            p.sega[si * 64 + lane] = Tb ? Ta : cmul2(Ta, Ra);
            p.sega[si * 64 + 32 + lane] = Tb ? Tx : cfma2(Ta, Rx, Tx);
            if (lane == 0) p.segb[si] = (Tb || Rb) ? 1u : 0u;
        }
        if (C::REV && !C::PS && *s_abort == 0) {
            // grad_lambda partial of this tile, summed over warps in a fixed order
            ptx::named_sync(BAR_ACC, C::NSYNC);
            float4 sum = zero2();
            for (int v = 0; v < W; ++v) sum = add2(sum, s_acc[v * 32 + lane]);
            p.gpart[(t.chain * p.n_tt + t.jt) * 32 + lane] = sum;
        }
        return;
    }

    // ----------------------------------------------------------------- scan warps
    const int64_t ts = t.t0 + static_cast<int64_t>(warp) * R;
    const int nv = static_cast<int>(lmax(0, lmin(R, p.L - ts)));
    uint32_t rmask, bmask;
    if (!C::REV) {
        const uint32_t bit = (lane < nv) ? (p.start[t.b * p.L + ts + lane] != 0) : 0u;
        rmask = bmask = __ballot_sync(0xffffffffu, bit);
    } else {
        // bit k of bmask: b_{ts+k} for k <= R (0 past the tape end);
        // bit k of rmask: b_{ts+k+1}, the reset of the reverse element of step ts+k
        const uint32_t bit = (lane <= R && ts + lane < p.L) ? (p.start[t.b * p.L + ts + lane] != 0) : 0u;
        bmask = __ballot_sync(0xffffffffu, bit);
        rmask = bmask >> 1;
    }
    const float4 lam = (!C::PS && lane_ok) ? p.lambda[t.c2 + lane] : one2();
    const float4 mlam = conj2(lam);
    const float4* sin = s_in + warp * R * 32 + lane;
    const float4* sl = s_l + warp * R * 32 + lane;

    bool landed = true;
    {
        const uint64_t w0 = ptx::globaltimer();
        while (!ptx::mbar_try_wait(bar, 0)) {
            if (ptx::globaltimer() - w0 > p.wait_ns) {
                record_error(p, DEV_TMA_TIMEOUT, tk);
                landed = false;
                break;
            }
        }
    }
    if (!landed && lane == 0) *s_abort = 1;

    // FFM forward: this lane's two x~ values per staged row (rows of 64 / c
    // floats); from c = 2 on, both channels of a lane belong to the same row i
    const int lcx = C::LC >= 0 ? C::LC : p.ffm_lc;
    const int xrow = 64 >> lcx;
    const float* xs = reinterpret_cast<const float*>(s_in) + warp * R * xrow;
    const int xi0 = (2 * lane) >> lcx, xi1 = lcx >= 1 ? xi0 : xi0 + 1;
    auto xpair = [&](int k) { return make_float4(xs[k * xrow + xi0], 0.f, xs[k * xrow + xi1], 0.f); };
    // loops without per-step tests (a per-channel lambda): a whole warp range with
    // no begin flag; in reverse also no flag at the step after it (bits 0..R of
    // bmask), and neither the tape's first nor its last step inside it
    const bool plain = !C::PS && nv == R &&
                       (C::REV ? ((bmask & ((2u << R) - 1u)) == 0u && ts > 0 && ts + R < p.L) : rmask == 0u);

    // phase 1: aggregate of this warp's steps, from the identity, in processing order
    float4 a = one2(), x = zero2();
    if (landed && !C::PS) {
        // a constant lambda per channel: the aggregate's multiplier is lambda^n over the
        // n steps after the last reset in processing order (lambda -> 1 at the tape's
        // last step in reverse), taken once by repeated squaring
        const uint32_t rv = rmask & ((nv >= 32) ? 0xffffffffu : ((1u << nv) - 1u));
        if (!C::REV) {
            if (plain) {
#pragma unroll C::UNROLL
                for (int k = 0; k < R; ++k) x = cfma2(lam, x, C::FFM ? xpair(k) : sin[k * 32]);
            } else {
#pragma unroll C::UNROLL
                for (int k = 0; k < R; ++k) {
                    if (k < nv) {
                        const float4 uu = C::FFM ? xpair(k) : sin[k * 32];
                        x = ((rmask >> k) & 1u) ? uu : cfma2(lam, x, uu);
                    }
                }
            }
            a = cpow2(lam, rv ? nv - (31 - __clz(rv)) : nv);
        } else if (plain) {
#pragma unroll C::UNROLL
            for (int kk = 0; kk < R; ++kk) {
                const int k = R - 1 - kk;
                x = cfma2(mlam, x, C::FFM ? ffm_planar_pair<C::T>(s_in, warp * R + k, lane) : sin[k * 32]);
            }
            a = cpow2(mlam, nv);
        } else {
#pragma unroll C::UNROLL
            for (int kk = 0; kk < R; ++kk) {
                const int k = R - 1 - kk;
                if (k < nv) {
                    const float4 gg = C::FFM ? ffm_planar_pair<C::T>(s_in, warp * R + k, lane) : sin[k * 32];
                    const float4 m = (ts + k == p.L - 1) ? one2() : mlam;
                    x = ((rmask >> k) & 1u) ? gg : cfma2(m, x, gg);
                }
            }
            const int cnt = rv ? __ffs(rv) : nv;  // steps k < cnt multiply the carry
            const int64_t kl = p.L - 1 - ts;      // the tape's last step, if in this warp
            a = cpow2(mlam, cnt - ((kl >= 0 && kl < cnt) ? 1 : 0));
        }
    } else if (landed) {
        // a lambda per step: the multiplier is the running product
        if (!C::REV) {
#pragma unroll C::UNROLL
            for (int k = 0; k < R; ++k) {
                if (k < nv) {
                    const float4 uu = sin[k * 32];
                    const float4 ll = sl[k * 32];
                    if ((rmask >> k) & 1u) {
                        a = ll;
                        x = uu;
                    } else {
                        x = cfma2(ll, x, uu);
                        a = cmul2(ll, a);
                    }
                }
            }
        } else {
#pragma unroll C::UNROLL
            for (int kk = 0; kk < R; ++kk) {
                const int k = R - 1 - kk;
                if (k < nv) {
                    const float4 gg = sin[k * 32];
                    const float4 m = (ts + k == p.L - 1) ? one2() : conj2(sl[k * 32]);
                    if ((rmask >> k) & 1u) {
                        a = m;
                        x = gg;
                    } else {
                        x = cfma2(m, x, gg);
                        a = cmul2(m, a);
                    }
                }
            }
        }
    }
    const uint32_t vmask = (nv >= 32) ? 0xffffffffu : ((1u << nv) - 1u);
    s_wa[warp * 32 + lane] = a;
    s_wx[warp * 32 + lane] = x;
    if (lane == 0) s_wr[warp] = ((rmask & vmask) != 0u);
    ptx::named_arrive(BAR_AGG, C::NSYNC);
    ptx::named_sync(BAR_CARRY, C::NSYNC);
    if (*s_abort) return;

    // carry into this warp: the tile's carry through the warps before it (in processing order)
    float4 c = s_carry[lane];
    for (int k = 0; k < W; ++k) {
        const int v = C::REV ? W - 1 - k : k;
        if (v == warp) break;
        const float4 wa = s_wa[v * 32 + lane], wx = s_wx[v * 32 + lane];
        c = s_wr[v] ? wx : cfma2(wa, c, wx);
    }

    // phase 3: rescan from the carry and stream the outputs
    if (!C::REV) {
        if (lane_ok) {
            float4* dst = p.out + (t.b * p.L + ts) * p.D2 + t.c2 + lane;
            // FFM: planar rows (Re half, then Im half, D2 float2 each)
            float2* pre = reinterpret_cast<float2*>(p.out + (t.b * p.L + ts) * p.D2) + t.c2 + lane;
            const int64_t prow = 2 * p.D2;  // float2 per planar row
            if (plain) {
#pragma unroll C::UNROLL
                for (int k = 0; k < R; ++k) {
                    c = cfma2(lam, c, C::FFM ? xpair(k) : sin[k * 32]);
                    if (C::FFM) {
                        __stcs(pre + k * prow, make_float2(c.x, c.z));
                        __stcs(pre + k * prow + p.D2, make_float2(c.y, c.w));
                    } else {
                        __stcs(dst + static_cast<int64_t>(k) * p.D2, c);
                    }
                }
            } else {
#pragma unroll C::UNROLL
                for (int k = 0; k < R; ++k) {
                    if (k < nv) {
                        const float4 uu = C::FFM ? xpair(k) : sin[k * 32];
                        const float4 ll = C::PS ? sl[k * 32] : lam;
                        c = ((rmask >> k) & 1u) ? uu : cfma2(ll, c, uu);
                        if (C::FFM) {
                            __stcs(pre + k * prow, make_float2(c.x, c.z));
                            __stcs(pre + k * prow + p.D2, make_float2(c.y, c.w));
                        } else {
                            __stcs(dst + static_cast<int64_t>(k) * p.D2, c);
                        }
                    }
                }
            }
            if (p.out_last != nullptr && nv > 0 && ts + nv == p.L) p.out_last[t.b * p.D2 + t.c2 + lane] = c;
        }
    } else {
        const float4* sh = s_h + warp * R * 32 + lane;
        float4 acc = zero2();
        // the h_{t-1} rows have their own barrier: the first pass did not wait for them
        {
            const uint64_t w0 = ptx::globaltimer();
            while (!ptx::mbar_try_wait(bar_h, 0)) {
                if (ptx::globaltimer() - w0 > p.wait_ns) {
                    record_error(p, DEV_TMA_TIMEOUT, tk);
                    break;
                }
            }
        }
        // FFM: every lane runs the loop (grad_x~ is reduced across lanes); the
        // lanes past the slab's width touch no global memory
        if (C::FFM || lane_ok) {
            float4* dst = p.out + (t.b * p.L + ts) * p.D2 + t.c2 + lane;
            // FFM: this lane's grad_x~ element in row ts (rows of m floats): its two
            // channels' row i for c = 1, else the row i of its group of c / 2 lanes
            const int lc = p.ffm_lc;
            const int grp = lc > 0 ? 1 << (lc - 1) : 1;  // lanes per row i (c > 1)
            const bool gx_writer = lane_ok && (lane & (grp - 1)) == 0;
            float* gxw = C::FFM ? p.ffm_gx + (t.b * p.L + ts) * p.ffm_m + ((2 * (t.c2 + lane)) >> lc) : nullptr;
            const int64_t gxrow = p.ffm_m;
            // step k's output: grad_u, or the FFM's grad_x~ (summed over the row's lanes)
            auto emit = [&](int k) {
                if (C::FFM) {
                    float* g = gxw + k * gxrow;
                    if (lc == 0) {
                        if (lane_ok) __stcs(reinterpret_cast<float2*>(g), make_float2(c.x, c.z));
                    } else {
                        float v = c.x + c.z;
                        if (grp > 1) v += __shfl_xor_sync(0xffffffffu, v, 1);
                        if (grp > 2) v += __shfl_xor_sync(0xffffffffu, v, 2);
                        if (grp > 4) v += __shfl_xor_sync(0xffffffffu, v, 4);
                        if (gx_writer) __stcs(g, v);
                    }
                } else {
                    __stcs(dst + static_cast<int64_t>(k) * p.D2, c);
                }
            };
            if (plain) {
#pragma unroll C::UNROLL
                for (int kk = 0; kk < R; ++kk) {
                    const int k = R - 1 - kk;
                    c = cfma2(mlam, c, C::FFM ? ffm_planar_pair<C::T>(s_in, warp * R + k, lane) : sin[k * 32]);
                    emit(k);
                    if (lane_ok) {
                        const float4 hp = C::FFM ? ffm_planar_pair<C::T>(s_h, warp * R + k, lane) : sh[k * 32];
                        acc = cfma2(c, conj2(hp), acc);
                    }
                }
            } else {
#pragma unroll C::UNROLL
                for (int kk = 0; kk < R; ++kk) {
                    const int k = R - 1 - kk;
                    if (k >= nv) continue;
                    const int64_t tt = ts + k;
                    const float4 gg = C::FFM ? ffm_planar_pair<C::T>(s_in, warp * R + k, lane) : sin[k * 32];
                    const float4 m = (tt == p.L - 1) ? one2() : (C::PS ? conj2(sl[k * 32]) : mlam);
                    c = ((rmask >> k) & 1u) ? gg : cfma2(m, c, gg);
                    emit(k);
                    float4 gl = zero2();
                    if (!((bmask >> k) & 1u) && lane_ok) {
                        float4 hp;
                        if (tt > 0) hp = C::FFM ? ffm_planar_pair<C::T>(s_h, warp * R + k, lane) : sh[k * 32];
                        else hp = (p.h0 != nullptr) ? p.h0[t.b * p.D2 + t.c2 + lane] : zero2();
                        if (C::PS) gl = cmul2(c, conj2(hp));
                        else acc = cfma2(c, conj2(hp), acc);  // the same fused form as the loop above
                    }
                    if (C::PS && p.grad_lambda != nullptr)
                        __stcs(p.grad_lambda + (t.b * p.L + tt) * p.D2 + t.c2 + lane, gl);
                    if (tt == 0 && p.grad_h0 != nullptr && lane_ok) {
                        const float4 l0 = C::PS ? p.lambda[(t.b * p.L) * p.D2 + t.c2 + lane] : lam;
                        p.grad_h0[t.b * p.D2 + t.c2 + lane] = (bmask & 1u) ? zero2() : cmul2(conj2(l0), c);
                    }
                }
            }
        }
        if (!C::PS) {
            s_acc[warp * 32 + lane] = acc;
            ptx::named_arrive(BAR_ACC, C::NSYNC);
        }
    }
}

// ============================================================================
// segment fix-up
// ============================================================================
// State entering each segment, one CTA per chain: each warp folds a range of
// the segments' aggregates (published by their last tiles) from the identity,
// the warps' aggregates are folded in order from the chain's initial state,
// and each warp then walks its range again from its own entering state.  A
// begin flag inside a fold discards what is left of it, exactly.
constexpr int CARRY_WARPS = 8;
constexpr int CARRY_BATCH = 8;
__global__ void __launch_bounds__(CARRY_WARPS * 32) segment_carry_kernel(const Params p, bool rev) {
    __shared__ float4 s_a[CARRY_WARPS][32], s_x[CARRY_WARPS][32];
    __shared__ uint32_t s_b[CARRY_WARPS];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t chain = blockIdx.x;
    ptx::grid_dependency_wait();  // the scan's summaries
    if (ptx::ld_relaxed(p.hdr) != 0u) return;  // uniform over the CTA
    const int64_t G = p.n_seg;
    const int64_t b = chain / p.n_slabs;
    const int64_t c2 = (chain - b * p.n_slabs) * (SLAB / 2);
    const bool lane_ok = lane < lmin(SLAB / 2, p.D2 - c2);
    const int64_t per = (G + CARRY_WARPS - 1) / CARRY_WARPS;
    const int64_t g_lo = lmin(G, warp * per), g_hi = lmin(G, g_lo + per);
    // this warp's range folded from the identity
    float4 A = one2(), X = zero2();
    bool Bf = false;
    for (int64_t g0 = g_lo; g0 < g_hi; g0 += CARRY_BATCH) {
        float4 a[CARRY_BATCH], x[CARRY_BATCH];
        uint32_t bb[CARRY_BATCH];
#pragma unroll
        for (int k = 0; k < CARRY_BATCH; ++k) {
            const int64_t si = chain * G + g0 + k;
            if (g0 + k < g_hi) {
                a[k] = p.sega[si * 64 + lane];
                x[k] = p.sega[si * 64 + 32 + lane];
                bb[k] = p.segb[si];
            }
        }
#pragma unroll
        for (int k = 0; k < CARRY_BATCH; ++k) {
            if (g0 + k < g_hi) {
                if (bb[k]) {
                    A = a[k];
                    X = x[k];
                    Bf = true;
                } else {
                    X = cfma2(a[k], X, x[k]);
                    A = cmul2(a[k], A);
                }
            }
        }
    }
    s_a[warp][lane] = A;
    s_x[warp][lane] = X;
    if (lane == 0) s_b[warp] = Bf ? 1u : 0u;
    __syncthreads();
    // state entering this warp's range: the initial state through the warps before it
    const float4* base_src = rev ? p.g_last : p.h0;
    float4 c = (base_src != nullptr && lane_ok) ? base_src[b * p.D2 + c2 + lane] : zero2();
    for (int w = 0; w < warp; ++w) c = s_b[w] ? s_x[w][lane] : cfma2(s_a[w][lane], c, s_x[w][lane]);
    for (int64_t g0 = g_lo; g0 < g_hi; g0 += CARRY_BATCH) {
        float4 a[CARRY_BATCH], x[CARRY_BATCH];
        uint32_t bb[CARRY_BATCH];
#pragma unroll
        for (int k = 0; k < CARRY_BATCH; ++k) {
            const int64_t si = chain * G + g0 + k;
            if (g0 + k < g_hi) {
                a[k] = p.sega[si * 64 + lane];
                x[k] = p.sega[si * 64 + 32 + lane];
                bb[k] = p.segb[si];
            }
        }
#pragma unroll
        for (int k = 0; k < CARRY_BATCH; ++k) {
            if (g0 + k < g_hi) {
                p.segc[(chain * G + g0 + k) * 32 + lane] = c;
                c = bb[k] ? x[k] : cfma2(a[k], c, x[k]);
            }
        }
    }
}

// Adds the state entering its segment to the outputs of a tile that the
// scan computed from the identity, up to the tile's first begin flag: the
// CTAs walk the list of such tiles the scan wrote (each tile touches only
// its own rows, so the list's order does not matter).  The rows to fix are
// counted first, so their loads can be issued in batches.  With a
// per-channel lambda the rows are split over `nparts` warps: part w starts
// from the carry times m^k (m = lambda, or conj(lambda) in reverse; k = the
// rows before the part, by repeated squaring) and leaves its grad_lambda
// partial in gl_out[w] for a fixed-order sum; with a per-step lambda one
// warp takes the whole tile (nparts = 1).
template <class C>
__device__ void segment_fix_tile(const Params& p, int64_t tid, int part, int nparts, float4* gl_out) {
    constexpr int BATCH = 8;
    const int lane = threadIdx.x & 31;
    const int64_t chain = tid / p.n_tt, jt = tid - chain * p.n_tt;
    const int64_t b = chain / p.n_slabs;
    const int64_t c2 = (chain - b * p.n_slabs) * (SLAB / 2);
    const int64_t jg = C::REV ? p.n_tt - 1 - jt : jt;
    const int64_t g = jg / p.q_seg;
    const int64_t t0 = jt * C::T;
    const int nrows = static_cast<int>(lmin(C::T, p.L - t0));
    // steps to fix, in processing order, before the first begin flag that cuts the carry
    int nfix = nrows;
    for (int r0 = 0; r0 < nrows; r0 += 32) {
        const int r = r0 + lane;
        bool cut = false;
        if (r < nrows) {
            if (!C::REV) {
                cut = p.start[b * p.L + t0 + r] != 0;
            } else {
                const int64_t t = t0 + nrows - 1 - r;  // r-th step processed
                cut = (t + 1 < p.L) && p.start[b * p.L + t + 1] != 0;
            }
        }
        const uint32_t m = __ballot_sync(0xffffffffu, cut);
        if (m != 0u) {
            nfix = r0 + __ffs(m) - 1;
            break;
        }
    }
    // lanes of the slab (FFM: the butterfly over a row's lanes uses this mask;
    // a row's lanes are all in the slab or all past it)
    const bool active = lane < lmin(SLAB / 2, p.D2 - c2);
    const unsigned act = __ballot_sync(0xffffffffu, active);
    float4 gl = zero2();
    if (!active) return;
    const int64_t col = c2 + lane;
    float4 corr = cmul2(p.pin[tid * 32 + lane], p.segc[(chain * p.n_seg + g) * 32 + lane]);
    const float4 lam = C::PS ? one2() : p.lambda[col];
    const int per = (nfix + nparts - 1) / nparts;
    const int k_lo = min(nfix, part * per), k_hi = min(nfix, k_lo + per);
    if (k_lo > 0) {
        // the rows before this part: every one multiplies the carry by m, except
        // that in reverse the tape's last step (processed first) multiplies by 1
        const int skip = (C::REV && t0 + nrows == p.L) ? 1 : 0;
        corr = cmul2(cpow2(C::REV ? conj2(lam) : lam, k_lo - skip), corr);
    }
    for (int k0 = k_lo; k0 < k_hi; k0 += BATCH) {
        // forward, per-step lambda: the batch's multipliers load with its outputs (a
        // load behind the previous row's store would wait for it)
        float4 v[BATCH], aux[BATCH], mul[(!C::REV && C::PS) ? BATCH : 1];
#pragma unroll
        for (int k = 0; k < BATCH; ++k) {
            if (k0 + k < k_hi) {
                const int64_t t = C::REV ? t0 + nrows - 1 - (k0 + k) : t0 + k0 + k;
                if constexpr (!C::REV && C::PS) mul[k] = p.lambda[(b * p.L + t) * p.D2 + col];
                if (!C::FFM) v[k] = p.out[(b * p.L + t) * p.D2 + col];
                else if (!C::REV) v[k] = ffm_load_planar(p.out + (b * p.L + t) * p.D2, p.D2, col);
                if (C::REV) {
                    if (t > 0)
                        aux[k] = C::FFM ? ffm_load_planar(p.h + (b * p.L + t - 1) * p.D2, p.D2, col)
                                        : p.h[(b * p.L + t - 1) * p.D2 + col];
                    else
                        aux[k] = (p.h0 != nullptr) ? p.h0[b * p.D2 + col] : zero2();
                }
            }
        }
#pragma unroll
        for (int k = 0; k < BATCH; ++k) {
            if (k0 + k >= k_hi) break;
            const int64_t t = C::REV ? t0 + nrows - 1 - (k0 + k) : t0 + k0 + k;
            if (!C::REV) {
                float4 l = lam;
                if constexpr (C::PS) l = mul[k];
                corr = cmul2(l, corr);
            } else {
                const float4 m = (t == p.L - 1) ? one2()
                                                : conj2(C::PS ? p.lambda[(b * p.L + t + 1) * p.D2 + col] : lam);
                corr = cmul2(m, corr);
            }
            if (!C::FFM)
                p.out[(b * p.L + t) * p.D2 + col] = add2(v[k], corr);
            else if (!C::REV)
                ffm_store_planar(p.out + (b * p.L + t) * p.D2, p.D2, col, add2(v[k], corr), false);
            else
                ffm_grad_x(p, b * p.L + t, col, corr, act, true, true, false);
            if (!C::REV) {
                if (t == p.L - 1 && p.out_last != nullptr) {
                    float4* ol = p.out_last + b * p.D2 + col;
                    *ol = add2(*ol, corr);
                }
            } else if (p.start[b * p.L + t] == 0) {
                const float4 d = cmul2(corr, conj2(aux[k]));
                if (C::PS) {
                    if (p.grad_lambda != nullptr) {
                        float4* gp = p.grad_lambda + (b * p.L + t) * p.D2 + col;
                        *gp = add2(*gp, d);
                    }
                } else {
                    gl = add2(gl, d);
                }
                if (t == 0 && p.grad_h0 != nullptr) {
                    const float4 l0 = C::PS ? p.lambda[(b * p.L) * p.D2 + col] : lam;
                    float4* g0 = p.grad_h0 + b * p.D2 + col;
                    *g0 = add2(*g0, cmul2(conj2(l0), corr));
                }
            }
        }
    }
    if (gl_out != nullptr) gl_out[part * 32 + lane] = gl;
    else if (C::REV && !C::PS) p.gpart[tid * 32 + lane] = add2(p.gpart[tid * 32 + lane], gl);
}

template <class C>
__global__ void __launch_bounds__(128) segment_fix_kernel(const Params p) {
    ptx::grid_dependency_wait();  // the segment carries
    if (ptx::ld_relaxed(p.hdr) != 0u) return;
    const int64_t n_fix = static_cast<int64_t>(ptx::ld_relaxed(p.hdr + 4));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if constexpr (C::PS) {
        // per-step lambda: one warp per tile
        const int64_t nw = static_cast<int64_t>(gridDim.x) * 4;
        for (int64_t f = static_cast<int64_t>(blockIdx.x) * 4 + warp; f < n_fix; f += nw)
            segment_fix_tile<C>(p, static_cast<int64_t>(p.fix[f]), 0, 1, nullptr);
    } else {
        // per-channel lambda: the four warps of a CTA split a tile's rows
        __shared__ float4 gl[4 * 32];
        for (int64_t f = blockIdx.x; f < n_fix; f += gridDim.x) {
            const int64_t tid = static_cast<int64_t>(p.fix[f]);
            segment_fix_tile<C>(p, tid, warp, 4, C::REV ? gl : nullptr);
            if (C::REV) {
                __syncthreads();
                const int64_t c2 = (tid / p.n_tt % p.n_slabs) * (SLAB / 2);
                if (warp == 0 && lane < lmin(SLAB / 2, p.D2 - c2)) {
                    const float4 sum = add2(add2(gl[lane], gl[32 + lane]), add2(gl[64 + lane], gl[96 + lane]));
                    p.gpart[tid * 32 + lane] = add2(p.gpart[tid * 32 + lane], sum);
                }
                __syncthreads();
            }
        }
    }
}

// ============================================================================
// grad_lambda reduction (per-channel lambda): fixed-order sums (fp32 within a part, fp64 across parts)
// ============================================================================
__global__ void __launch_bounds__(256) reduce_parts_kernel(const float4* __restrict__ gpart,
                                                           double* __restrict__ rpart, int64_t B,
                                                           int64_t n_slabs, int64_t n_tt) {
    __shared__ double s[8][32][4];
    ptx::grid_dependency_wait();  // the tile partials, fixed up
    const int slab = blockIdx.x, part = blockIdx.y;
    const int grp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t total = B * n_tt;
    const int64_t per = (total + RED_PARTS - 1) / RED_PARTS;
    const int64_t k0 = part * per, k1 = lmin(total, k0 + per);
    // fp32 within a part (a few dozen tile partials), fp64 across parts and in the final tree
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    // this group's tiles k0 + grp, k0 + grp + 8, ...: loads issued in batches of 8, summed in that order
    constexpr int RB = 8;
    for (int64_t k = k0 + grp; k < k1; k += 8 * RB) {
        float4 v[RB];
#pragma unroll
        for (int u = 0; u < RB; ++u) {
            const int64_t kk = k + 8 * u;
            if (kk < k1) {
                const int64_t bb = kk / n_tt, jj = kk - bb * n_tt;
                v[u] = gpart[((bb * n_slabs + slab) * n_tt + jj) * 32 + lane];
            }
        }
#pragma unroll
        for (int u = 0; u < RB; ++u) {
            if (k + 8 * u < k1) {
                acc[0] += v[u].x;
                acc[1] += v[u].y;
                acc[2] += v[u].z;
                acc[3] += v[u].w;
            }
        }
    }
    for (int c = 0; c < 4; ++c) s[grp][lane][c] = static_cast<double>(acc[c]);
    __syncthreads();
    if (grp == 0) {
        double r[4] = {0.0, 0.0, 0.0, 0.0};
        for (int g = 0; g < 8; ++g)
            for (int c = 0; c < 4; ++c) r[c] += s[g][lane][c];
        double* o = rpart + ((static_cast<int64_t>(slab) * RED_PARTS + part) * 32 + lane) * 4;
        for (int c = 0; c < 4; ++c) o[c] = r[c];
    }
}

// One block of RED_PARTS threads per (slab, lane): thread p holds part p, then
// a shared-memory tree with a fixed pairing sums the parts.
__global__ void __launch_bounds__(RED_PARTS) reduce_final_kernel(const double* __restrict__ rpart,
                                                                 float4* __restrict__ grad_lambda, int64_t D2) {
    __shared__ double2 s[2][RED_PARTS];
    ptx::grid_dependency_wait();  // the parts
    const int slab = blockIdx.x >> 5, lane = blockIdx.x & 31, p = threadIdx.x;
    const double2* o =
        reinterpret_cast<const double2*>(rpart + ((static_cast<int64_t>(slab) * RED_PARTS + p) * 32 + lane) * 4);
    s[0][p] = o[0];
    s[1][p] = o[1];
    __syncthreads();
#pragma unroll
    for (int w = RED_PARTS / 2; w > 0; w >>= 1) {
        if (p < w) {
            s[0][p].x += s[0][p + w].x;
            s[0][p].y += s[0][p + w].y;
            s[1][p].x += s[1][p + w].x;
            s[1][p].y += s[1][p + w].y;
        }
        __syncthreads();
    }
    const int64_t col = static_cast<int64_t>(slab) * 32 + lane;
    if (p == 0 && col < D2)
        grad_lambda[col] = make_float4(static_cast<float>(s[0][0].x), static_cast<float>(s[0][0].y),
                                       static_cast<float>(s[1][0].x), static_cast<float>(s[1][0].y));
}

// ============================================================================
// host side
// ============================================================================
namespace {

// Tile shapes (scan warps, steps per warp): the measured best on GB300.
// The forward (per-channel lambda) takes 5 x 20 tiles where every chain is one
// segment and 5 x 24 where chains are cut into segments (measured: the
// 2^20-step, 256-channel tape 0.696 ms with 4 x 24, 0.689 with 5 x 20, 0.680
// with 5 x 24; 64 tapes x 16384 steps x 128 channels 0.349 / 0.347 / 0.364 ms).
using FwdC = Cfg<5, 20, false, false>;
using FwdL = Cfg<5, 24, false, false>;
// per-step lambda (two staged arrays forward, three backward)
using FwdS = Cfg<4, 12, false, true>;
// The backward likewise: 8 x 12 where every chain is one segment, 7 x 14 where
// chains are cut into segments (measured: 1.006 / 1.001 ms on the 2^20-step,
// 256-channel tape; 0.559 / 0.562 ms on the 64 tapes).
using BwdC = Cfg<8, 12, true, false>;
using BwdL = Cfg<7, 14, true, false>;
using BwdS = Cfg<8, 8, true, true>;
// The FFM forward stages only x~ (a few bytes per step), so larger tiles pay:
// 6 x 31 (186-step tiles) was the measured best on GB300.
// The forward is compiled for each c (log2 c = LC), so the lanes' x~ offsets
// are constants.
template <int LC>
using FwdF = Cfg<6, 31, false, false, true, LC>;
using BwdF = Cfg<8, 12, true, false, true>;

// Segments per chain: enough segment chains that a tile's predecessor was
// handed out long before it (target), at least MIN_SEG_TILES tiles each.  From
// CHAINS_NO_SEG chains on, the chains themselves interleave enough, and one
// segment per chain saves the fix-up of every segment's steps before its first
// begin flag, all of its steps on a tape without flags (measured on 64 tapes x
// 16384 steps x 128 channels, half of them one episode: fwd 0.474 -> 0.361 ms,
// bwd 0.703 -> 0.600 ms; 4 chains keep their segments: with a quarter of the
// target the 2^20-step, 256-channel tape took 0.733 / 1.162 instead of 0.700 /
// 1.089 ms).  The targets were swept again with the current tiles on that tape:
// the times move by up to 2% between neighbouring counts (forward 384 / 416 /
// 448 / 480 / 512 segment chains: 0.675 / 0.674 / 0.676 / 0.695 / 0.680 ms;
// backward 208 / 224 / 228 / 240 / 256: 1.010 / 0.994 / 1.014 / 1.014 / 1.001 ms).
// With a per-step lambda (other tiles, another CTA count per SM) the earlier
// 512 / 256 stay: with 416 / 224 its forward took 1.114 instead of 1.036 ms.
constexpr int64_t TARGET_SC = 416;
constexpr int64_t TARGET_SC_BWD = 224;
constexpr int64_t TARGET_SC_PS = 512;
constexpr int64_t TARGET_SC_PS_BWD = 256;
constexpr int64_t MAX_SEG = 192;
constexpr int64_t MIN_SEG_TILES = 8;
constexpr int64_t CHAINS_NO_SEG = 128;

struct Segs {
    int64_t G, Q;
};
Segs choose_segments(int64_t n_chains, int64_t n_tt, bool rev, bool ps) {
    if (n_chains >= CHAINS_NO_SEG) return Segs{1, n_tt};
    const int64_t target = ps ? (rev ? TARGET_SC_PS_BWD : TARGET_SC_PS) : (rev ? TARGET_SC_BWD : TARGET_SC);
    int64_t G = (target + n_chains - 1) / n_chains;
    G = lmin(G, lmin(MAX_SEG, n_tt / MIN_SEG_TILES));
    if (G < 1) G = 1;
    const int64_t Q = (n_tt + G - 1) / G;
    return Segs{(n_tt + Q - 1) / Q, Q};
}

struct Layout {
    int64_t n_slabs, n_chains, n_tt;
    Segs sg;
    size_t node_off, gpart_off, fix_off, pin_off, segc_off, sega_off, segb_off, rpart_off, total;
};

// Workspace layout for tiles of T steps (rev, ps: the segment target of the
// backward scan, of a per-step lambda).
Layout layout(int64_t B, int64_t L, int64_t D, int T, bool rev, bool ps) {
    Layout l{};
    l.n_slabs = (D + SLAB - 1) / SLAB;
    l.n_chains = B * l.n_slabs;
    l.n_tt = (L + T - 1) / T;
    l.sg = choose_segments(l.n_chains, l.n_tt, rev, ps);
    const size_t tiles = static_cast<size_t>(l.n_chains) * static_cast<size_t>(l.n_tt);
    const size_t nodes = static_cast<size_t>(l.n_chains) * static_cast<size_t>(l.sg.G * l.sg.Q);
    l.node_off = kHeaderBytes;
    l.gpart_off = align_up(l.node_off + nodes * 32 * NODE_WORDS * 8, 256);
    l.fix_off = align_up(l.gpart_off + tiles * 32 * 16, 256);
    l.pin_off = align_up(l.fix_off + tiles * 4, 256);
    l.segc_off = align_up(l.pin_off + tiles * 32 * 16, 256);
    const size_t nseg = static_cast<size_t>(l.n_chains * l.sg.G);
    l.sega_off = align_up(l.segc_off + nseg * 32 * 16, 256);
    l.segb_off = align_up(l.sega_off + nseg * 64 * 16, 256);
    l.rpart_off = align_up(l.segb_off + nseg * 4, 256);
    l.total = align_up(l.rpart_off + static_cast<size_t>(l.n_slabs) * RED_PARTS * 32 * 32, 256);
    return l;
}

Params make_params(const Args& a, const Layout& l, int T, bool backward) {
    const int64_t n_tt = l.n_tt;
    const Segs sg = l.sg;
    Params p{};
    p.lambda = static_cast<const float4*>(a.lambda);
    p.in = static_cast<const float4*>(a.u);
    p.start = a.start;
    p.h0 = static_cast<const float4*>(a.h0);
    p.out = static_cast<float4*>(a.out);
    p.out_last = static_cast<float4*>(a.out_last);
    p.h = static_cast<const float4*>(a.h);
    p.g_last = static_cast<const float4*>(a.g_last);
    p.grad_lambda = static_cast<float4*>(a.grad_lambda);
    p.grad_h0 = static_cast<float4*>(a.grad_h0);
    p.B = a.B;
    p.L = a.L;
    p.D2 = a.D / 2;
    p.n_slabs = l.n_slabs;
    p.n_tt = n_tt;
    p.n_chains = l.n_chains;
    p.n_tiles = n_tt * l.n_chains;
    p.n_seg = sg.G;
    p.q_seg = sg.Q;
    p.n_sc = l.n_chains * sg.G;
    unsigned char* ws = static_cast<unsigned char*>(a.workspace);
    p.hdr = reinterpret_cast<uint32_t*>(ws);
    p.node = reinterpret_cast<unsigned long long*>(ws + l.node_off);
    p.gpart = reinterpret_cast<float4*>(ws + l.gpart_off);
    p.fix = sg.G > 1 ? reinterpret_cast<uint32_t*>(ws + l.fix_off) : nullptr;
    p.pin = reinterpret_cast<float4*>(ws + l.pin_off);
    p.segc = reinterpret_cast<float4*>(ws + l.segc_off);
    p.sega = reinterpret_cast<float4*>(ws + l.sega_off);
    p.segb = reinterpret_cast<uint32_t*>(ws + l.segb_off);
    const DebugKnobs k = debug_knobs();
    p.wait_ns = k.wait_ns;
    p.withhold = k.withhold_ticket;
    p.epoch = 0;  // set at launch (tagged_epoch)
    p.full_nodes = a.lambda_per_step ? 1 : 0;
    p.T = T;
    // backward: the chain's first tile (processing order) is the ragged last
    // time tile, and its step L-1 has multiplier 1 rather than conj(lambda)
    p.rag = backward ? static_cast<int>(n_tt * T - a.L) + 1 : 0;
    p.ffm_x = a.ffm_x;
    p.ffm_gx = a.ffm_gx;
    p.ffm_m = a.ffm_m;
    p.ffm_lc = 0;
    while ((int64_t{1} << p.ffm_lc) < a.ffm_c) ++p.ffm_lc;
    return p;
}

// A [B, L, row] fp32 array as a 3-D map {row, L, B} with boxes of `box_x`
// floats x T rows x 1 tape (no swizzle; out-of-range elements read as 0).
bool map3(CUtensorMap* m, const void* base, int64_t B, int64_t L, int64_t row, int box_x, int T) {
    const EncodeTiledFn fn = encode_tiled();
    if (fn == nullptr || base == nullptr) return fn != nullptr;
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(row), static_cast<cuuint64_t>(L), static_cast<cuuint64_t>(B)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(row * 4), static_cast<cuuint64_t>(L * row * 4)};
    const cuuint32_t box[3] = {static_cast<cuuint32_t>(box_x), static_cast<cuuint32_t>(T), 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The staging maps of a launch (see Params::map_in).
bool make_maps(Params& p, const Args& a, int T, bool backward) {
    const int64_t row = 4 * p.D2;  // floats per step: D complex, or Re || Im
    if (a.ffm_c > 0 && !backward) return map3(&p.map_in, a.ffm_x, a.B, a.L, a.ffm_m, 64 >> p.ffm_lc, T);
    const int bx = a.ffm_c > 0 ? 64 : 128;
    bool ok = map3(&p.map_in, a.u, a.B, a.L, row, bx, T);
    if (backward) ok = ok && map3(&p.map_h, a.h, a.B, a.L, row, bx, T);
    if (a.lambda_per_step) ok = ok && map3(&p.map_l, a.lambda, a.B, a.L, row, 128, T);
    return ok;
}

// One CTA per ticket; tickets are claimed in order by the CTAs as they
// start.  With more than one segment per chain, two small kernels then add the
// state entering each segment where it is missing.
template <class C>
memoroid_status_t launch(const Args& a, cudaStream_t s, Layout* out_layout) {
    const Layout l = layout(a.B, a.L, a.D, C::T, C::REV, C::PS);
    const Segs sg = l.sg;
    const int64_t n_tickets = sg.Q * l.n_chains * sg.G;
    if (n_tickets >= 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;
    if (l.total > a.workspace_bytes) return MEMOROID_ERR_WORKSPACE;  // this tile shape's layout must fit
    if (cudaMemsetAsync(a.workspace, 0, kHeaderBytes, s) != cudaSuccess) return MEMOROID_ERR_CUDA;
    auto kernel = diag_scan_kernel<C>;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(C::SMEM)) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    Params p = make_params(a, l, C::T, C::REV);
    if (!make_maps(p, a, C::T, C::REV)) return MEMOROID_ERR_CUDA;
    // the summaries' tag; their region is zeroed where an old word could carry it
    bool clear = false;
    p.epoch = tagged_epoch(a.workspace, l.gpart_off, s, &clear);
    if (clear && cudaMemsetAsync(static_cast<unsigned char*>(a.workspace) + l.node_off, 0, l.gpart_off - l.node_off, s) !=
                     cudaSuccess)
        return MEMOROID_ERR_CUDA;
    kernel<<<static_cast<unsigned>(n_tickets), C::THREADS, C::SMEM, s>>>(p);
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (sg.G > 1) {
        if (launch_after(segment_carry_kernel, dim3(static_cast<unsigned>(l.n_chains)), dim3(CARRY_WARPS * 32), 0, s, p,
                         C::REV) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
        const int64_t n_tiles = l.n_chains * l.n_tt;
        // the CTAs (per-channel lambda) or warps (per-step lambda) walk the list of tiles to fix
        const int64_t fix_ctas = lmin(C::PS ? (n_tiles + 3) / 4 : n_tiles, 152 * 8);
        if (launch_after(segment_fix_kernel<C>, dim3(static_cast<unsigned>(fix_ctas)), dim3(128), 0, s, p) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
        if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    }
    if (out_layout) *out_layout = l;
    return MEMOROID_OK;
}

}  // namespace

size_t workspace_bytes(int64_t B, int64_t L, int64_t D) {
    size_t m = 0;
    const int Ts[6] = {FwdC::T, FwdL::T, FwdS::T, BwdC::T, BwdL::T, BwdS::T};
    const bool revs[6] = {false, false, false, true, true, true};
    const bool pss[6] = {false, false, true, false, false, true};
    for (int i = 0; i < 6; ++i) {
        const size_t t = layout(B, L, D, Ts[i], revs[i], pss[i]).total;
        if (t > m) m = t;
    }
    return m;
}


// the tiles for a per-channel lambda: the longer ones where chains are cut into segments
static bool long_tiles(int64_t B, int64_t D) { return B * ((D + SLAB - 1) / SLAB) < CHAINS_NO_SEG; }

int kernels_per_call(int64_t B, int64_t L, int64_t D, int per_step, int backward, int with_grad_lambda) {
    if (B <= 0 || L <= 0 || D <= 0) return 0;
    const bool lt = long_tiles(B, D);
    const int T = backward ? (per_step ? BwdS::T : (lt ? BwdL::T : BwdC::T))
                           : (per_step ? FwdS::T : (lt ? FwdL::T : FwdC::T));
    const Layout l = layout(B, L, D, T, backward != 0, per_step != 0);
    int n = l.sg.G > 1 ? 3 : 1;  // scan [+ segment carries + fix-up]
    if (backward && !per_step && with_grad_lambda) n += 2;  // grad_lambda reduction
    return n;
}

memoroid_status_t launch_fwd(const Args& a, cudaStream_t s) {
    switch (a.ffm_c) {
        case 0: break;
        case 1: return launch<FwdF<0>>(a, s, nullptr);
        case 2: return launch<FwdF<1>>(a, s, nullptr);
        case 4: return launch<FwdF<2>>(a, s, nullptr);
        case 8: return launch<FwdF<3>>(a, s, nullptr);
        case 16: return launch<FwdF<4>>(a, s, nullptr);
        default: return MEMOROID_ERR_INVALID_ARG;
    }
    if (a.lambda_per_step) return launch<FwdS>(a, s, nullptr);
    return long_tiles(a.B, a.D) ? launch<FwdL>(a, s, nullptr) : launch<FwdC>(a, s, nullptr);
}

memoroid_status_t launch_bwd(const Args& a, cudaStream_t s) {
    const bool ps = a.lambda_per_step != 0;
    Layout l{};
    const memoroid_status_t st = a.ffm_c > 0 ? launch<BwdF>(a, s, &l)
                                 : ps        ? launch<BwdS>(a, s, &l)
                                 : long_tiles(a.B, a.D) ? launch<BwdL>(a, s, &l)
                                                        : launch<BwdC>(a, s, &l);
    if (st != MEMOROID_OK) return st;
    if (!ps && a.grad_lambda != nullptr) {
        unsigned char* ws = static_cast<unsigned char*>(a.workspace);
        const float4* gpart = reinterpret_cast<const float4*>(ws + l.gpart_off);
        double* rpart = reinterpret_cast<double*>(ws + l.rpart_off);
        if (launch_after(reduce_parts_kernel, dim3(static_cast<unsigned>(l.n_slabs), RED_PARTS), dim3(256), 0, s, gpart,
                         rpart, a.B, l.n_slabs, l.n_tt) != cudaSuccess ||
            launch_after(reduce_final_kernel, dim3(static_cast<unsigned>(l.n_slabs * 32)), dim3(RED_PARTS), 0, s,
                         static_cast<const double*>(rpart), static_cast<float4*>(a.grad_lambda), a.D / 2) !=
                cudaSuccess)
            return MEMOROID_ERR_CUDA;
    }
    return MEMOROID_OK;
}

// ============================================================================
// Fast and Forgetful Memory: lambda_ij = exp(-|alpha_i| + i omega_j) per
// channel, then the diagonal scan in the FFM layout
// ============================================================================
namespace {

// one thread per channel i * c + j; computed in fp64 and rounded once
__global__ void __launch_bounds__(256) ffm_lambda_kernel(const float* __restrict__ alpha,
                                                         const float* __restrict__ omega, int64_t m, int64_t c,
                                                         float2* __restrict__ lam) {
    const int64_t ij = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (ij >= m * c) return;
    const int64_t i = ij / c, j = ij - i * c;
    const double mag = exp(-fabs(static_cast<double>(alpha[i])));
    double sn, cs;
    sincos(static_cast<double>(omega[j]), &sn, &cs);
    lam[ij] = make_float2(static_cast<float>(mag * cs), static_cast<float>(mag * sn));
}

// grad_alpha_i = sum_j Re(conj(g_ij) (-sign(alpha_i)) lambda_ij) and
// grad_omega_j = sum_i Re(conj(g_ij) i lambda_ij), one thread per output,
// fixed-order fp64 sums (lambda as the forward used it)
__global__ void __launch_bounds__(256) ffm_param_grad_kernel(const float2* __restrict__ glam,
                                                             const float2* __restrict__ lam,
                                                             const float* __restrict__ alpha, int64_t m, int64_t c,
                                                             float* __restrict__ grad_alpha,
                                                             float* __restrict__ grad_omega) {
    ptx::grid_dependency_wait();  // the grad_lambda reduction
    const int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (k < m) {
        if (grad_alpha == nullptr) return;
        const double sg = alpha[k] > 0.f ? 1.0 : (alpha[k] < 0.f ? -1.0 : 0.0);
        double acc = 0.0;
        for (int64_t j = 0; j < c; ++j) {
            const float2 g = glam[k * c + j], l = lam[k * c + j];
            acc += -sg * (static_cast<double>(g.x) * l.x + static_cast<double>(g.y) * l.y);
        }
        grad_alpha[k] = static_cast<float>(acc);
    } else if (k < m + c) {
        if (grad_omega == nullptr) return;
        const int64_t j = k - m;
        double acc = 0.0;
        for (int64_t i = 0; i < m; ++i) {
            // Re(conj(g) * i * l) = g.x * (-l.y) + g.y * l.x
            const float2 g = glam[i * c + j], l = lam[i * c + j];
            acc += static_cast<double>(g.y) * l.x - static_cast<double>(g.x) * l.y;
        }
        grad_omega[j] = static_cast<float>(acc);
    }
}

size_t ffm_lambda_off(int64_t B, int64_t L, int64_t D) { return align_up(workspace_bytes(B, L, D), 256); }
size_t ffm_glam_off(int64_t B, int64_t L, int64_t D) {
    return align_up(ffm_lambda_off(B, L, D) + static_cast<size_t>(D) * 8, 256);
}

}  // namespace

size_t ffm_workspace_bytes(int64_t B, int64_t L, int64_t m, int64_t c) {
    const int64_t D = m * c;
    return align_up(ffm_glam_off(B, L, D) + static_cast<size_t>(D) * 8, 256);
}

int ffm_kernels_per_call(int64_t B, int64_t L, int64_t m, int64_t c, int backward, int with_param_grads) {
    if (B <= 0 || L <= 0 || m <= 0 || c <= 0) return 0;
    const int64_t D = m * c;
    const Layout l = layout(B, L, D, backward ? BwdF::T : FwdF<0>::T, backward != 0, false);
    int n = 1 + (l.sg.G > 1 ? 3 : 1);  // lambda + scan [+ segment carries + fix-up]
    if (backward && with_param_grads) n += 3;  // grad_lambda reduction + parameter gradients
    return n;
}

memoroid_status_t launch_ffm(const FfmArgs& f, cudaStream_t s) {
    const int64_t D = f.m * f.c;
    unsigned char* ws = static_cast<unsigned char*>(f.workspace);
    float2* lam = reinterpret_cast<float2*>(ws + ffm_lambda_off(f.B, f.L, D));
    float2* glam = reinterpret_cast<float2*>(ws + ffm_glam_off(f.B, f.L, D));
    ffm_lambda_kernel<<<static_cast<unsigned>((D + 255) / 256), 256, 0, s>>>(f.alpha, f.omega, f.m, f.c, lam);
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    const bool param = f.backward && (f.grad_alpha != nullptr || f.grad_omega != nullptr);
    Args a{};
    a.lambda = lam;
    a.lambda_per_step = 0;
    a.start = f.start;
    a.h0 = f.S0;
    a.B = f.B;
    a.L = f.L;
    a.D = D;
    a.workspace = f.workspace;
    a.workspace_bytes = ffm_lambda_off(f.B, f.L, D);  // the scan's part, before lambda and its gradient
    a.ffm_c = static_cast<int>(f.c);
    a.ffm_m = f.m;
    if (!f.backward) {
        a.ffm_x = f.x;
        a.out = f.z;
        a.out_last = f.S_last;
        return launch_fwd(a, s);
    }
    a.u = f.grad_z;
    a.h = f.z;
    a.g_last = f.grad_S_last;
    a.ffm_gx = f.grad_x;
    a.grad_lambda = param ? glam : nullptr;
    a.grad_h0 = f.grad_S0;
    const memoroid_status_t st = launch_bwd(a, s);
    if (st != MEMOROID_OK || !param) return st;
    return launch_after(ffm_param_grad_kernel, dim3(static_cast<unsigned>((f.m + f.c + 255) / 256)), dim3(256), 0, s,
                        static_cast<const float2*>(glam), static_cast<const float2*>(lam), f.alpha, f.m, f.c,
                        f.grad_alpha, f.grad_omega) == cudaSuccess
               ? MEMOROID_OK
               : MEMOROID_ERR_CUDA;
}

}  // namespace diag
}  // namespace memoroid
