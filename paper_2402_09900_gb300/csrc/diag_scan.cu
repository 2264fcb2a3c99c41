// diag_scan.cu -- single-pass resettable diagonal scan (forward and reverse)
// for sm_103a.
//
// Semantics: the S5 / LRU memoroid with diagonal X (paper appendix,
// "Simplified State Space Models" / "Linear Recurrent Unit"),
//     (X, x) . (X', x') = (X' X, X' x + x'),   e_I = (1, 0),
// made resettable by Theorem 3.2: an element whose begin flag is set discards
// everything to its left, (A, b) o (A', 1) = (A', 1).  Per step the lifted
// element is ((lambda_t, u_t), b_t), so h_t = b_t ? u_t : lambda_t h_{t-1} + u_t.
//
// Design (GB300-first; the paper itself ships no kernels):
//   * The tape [B, L, D] is cut into tiles of T steps x 64 complex channels
//     (a 512-byte row slab).  A "chain" is one (tape, slab) pair; its tiles
//     are scanned left to right in a single pass with a look-back over
//     already-published tile summaries.
//   * One CTA per tile.  Tiles are handed out by an atomic ticket so that a
//     CTA only ever waits on tiles whose CTAs are already resident.
//   * The look-back is deterministic: tile j publishes the aggregate of the
//     fixed range of tiles covered by Fenwick-tree node j+1, folded from its
//     Fenwick children in a fixed order, and its carry is the fixed
//     right-to-left fold of the Fenwick prefix nodes of position j.  Every
//     value is therefore a function of the inputs alone, not of the order in
//     which CTAs happen to run: repeated calls are bit-identical, and changing
//     one episode leaves every other episode's outputs bit-identical.  Each
//     tile reads at most ~2 log2(#tiles) summaries.
//   * The tile is staged into shared memory with one TMA bulk copy per row;
//     each warp owns R consecutive steps, each lane two complex channels
//     (one 16-byte vector).  A lane scans its R steps serially, warps are
//     combined through shared memory, and tiles through the look-back.
//   * A begin flag inside a summary's range discards everything to its left,
//     so folds stop at the first such summary (episode boundaries cut the
//     look-back short); a tile whose first step is a begin flag needs no
//     carry at all.
//   * Outputs are recomputed from the carry with the plain recurrence and
//     written with streaming 16-byte stores; HBM traffic is one read of the
//     inputs and one write of the outputs.
//   * Every wait (TMA completion, look-back) is bounded by the global timer;
//     on expiry the kernel records an error in the workspace and returns.
//
// The backward pass is the same machinery run right to left over
//     delta_t = grad_h_t + [b_{t+1} = 0] conj(lambda_{t+1}) delta_{t+1},
// i.e. the element of step t is (conj(lambda_{t+1}), grad_h_t, b_{t+1}), plus
// grad_lambda = sum_{b_t = 0} delta_t conj(h_{t-1}) (per-tile partials reduced
// in a fixed order by a second kernel, so results are deterministic).
#include <cuda_runtime.h>

#include <algorithm>

#include "internal.cuh"
#include "ptx.cuh"

namespace memoroid {
namespace diag {

constexpr int SLAB = 64;                    // complex channels per slab
// look-back status words: empty, Fenwick node published (its range holds no
// begin flag / holds one), error
constexpr uint32_t ST_EMPTY = 0, ST_NODE = 1, ST_NODE_RESET = 2, ST_ERROR = 3;
constexpr int RED_PARTS = 64;               // first-stage parts of the grad_lambda reduction
constexpr int MIN_T = 32;                   // smallest tile used (sizes the workspace)

// tile shapes: W warps x R steps per warp
constexpr int FWD_W = 8, FWD_R = 16;        // per-channel lambda: T = 128, 64 KB smem
constexpr int FWDS_W = 8, FWDS_R = 8;       // per-step lambda:    T = 64, 64 KB smem
constexpr int BWD_W = 8, BWD_R = 8;         // per-channel lambda: T = 64, 64 KB smem
constexpr int BWDS_W = 4, BWDS_R = 8;       // per-step lambda:    T = 32, 48 KB smem

struct Params {
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
    int64_t B, L, D2, n_slabs, n_tt, n_chains;
    int64_t D;
    uint32_t* hdr;         // workspace header
    uint32_t* flags;       // [n_chains * n_tt]
    float4* node;          // [n_chains * n_tt * 32 * 2]  Fenwick node (a, x) per lane
    float4* gpart;         // [n_chains * n_tt * 32]      per-tile grad_lambda
    uint64_t wait_ns;
    int64_t withhold;
};

__host__ __device__ __forceinline__ int64_t lmin(int64_t a, int64_t b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ int64_t lmax(int64_t a, int64_t b) { return a > b ? a : b; }

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

// ---- errors and bounded waits -------------------------------------------------
__device__ __forceinline__ void record_error(const Params& p, uint32_t code, int64_t ticket) {
    if (atomicCAS(p.hdr, 0u, code) == 0u) {
        *reinterpret_cast<volatile unsigned long long*>(p.hdr + 2) =
            static_cast<unsigned long long>(ticket);
    }
}

// Lane-0 wait on a look-back flag; returns the published status, or
// ST_ERROR after recording a timeout (or seeing another tile's error).
__device__ uint32_t wait_flag(const Params& p, const uint32_t* f, uint64_t t_begin,
                              int64_t ticket) {
    uint32_t v = ptx::ld_acquire(f);
    unsigned ns = 32;
    while (v == ST_EMPTY) {
        if (ptx::ld_relaxed(p.hdr) != 0u) return ST_ERROR;
        if (ptx::globaltimer() - t_begin > p.wait_ns) {
            record_error(p, DEV_LOOKBACK_TIMEOUT, ticket);
            return ST_ERROR;
        }
        __nanosleep(ns);
        if (ns < 1024) ns <<= 1;
        v = ptx::ld_acquire(f);
    }
    return v;
}

// Bounded wait on the TMA mbarrier (all threads).
__device__ bool wait_tma(const Params& p, uint64_t* bar, uint64_t t_begin, int64_t ticket) {
    while (!ptx::mbar_try_wait(bar, 0)) {
        if (ptx::globaltimer() - t_begin > p.wait_ns) {
            record_error(p, DEV_TMA_TIMEOUT, ticket);
            return false;
        }
    }
    return true;
}

// Publishes a status word after this warp's payload stores (all lanes call).
__device__ __forceinline__ void publish(uint32_t* f, uint32_t status, bool skip) {
    __threadfence();
    __syncwarp();
    if (!skip && (threadIdx.x & 31) == 0) ptx::st_release(f, status);
}

// Waits for the Fenwick node of chain position `pos` (1-based; stored at
// tile index pos-1) and folds it onto the left of (Ra, Rx, Rb), which must
// hold no begin flag yet:  node o R = (R.a * node.a, R.a * node.x + R.x, node.b).
// Warp-wide; returns false on timeout / error.
__device__ bool fold_node(const Params& p, int64_t fbase, int64_t pos, float4& Ra, float4& Rx,
                          bool& Rb, uint64_t t_begin, int64_t ticket) {
    const int lane = threadIdx.x & 31;
    const uint32_t* f = p.flags + fbase + pos - 1;
    uint32_t st = 0;
    if (lane == 0) st = wait_flag(p, f, t_begin, ticket);
    st = __shfl_sync(0xffffffffu, st, 0);
    if (st == ST_ERROR) return false;
    (void)ptx::ld_acquire(f);  // every lane acquires before reading the payload
    const int64_t idx = (fbase + pos - 1) * 32 + lane;
    const float4 a = __ldcg(p.node + 2 * idx);
    const float4 x = __ldcg(p.node + 2 * idx + 1);
    Rx = cfma2(Ra, x, Rx);
    Ra = cmul2(Ra, a);
    Rb = (st == ST_NODE_RESET);
    return true;
}

// Look-back of chain position j (0-based) for a tile whose aggregate is
// (Ta, Tx, Tb) (warp-wide, warp 0).
//  1. Publishes Fenwick node j+1, the aggregate of tiles [j+1-lowbit(j+1), j]:
//     its children j, j-1, j-3, ... (positions j+1-k, k = 1, 2, 4, .. <
//     lowbit) folded right to left onto the tile's own aggregate.
//  2. If need_carry, returns the state entering tile j: the Fenwick prefix
//     nodes of position j folded right to left, applied to `base` (the state
//     before the chain's first step) unless a begin flag intervenes.
// Folds stop early at a begin flag: everything to its left is discarded by
// the select of Theorem 3.2, so stopping changes no bit of the result.
__device__ bool fenwick_lookback(const Params& p, int64_t fbase, int64_t j, float4 Ta, float4 Tx,
                                 bool Tb, bool need_carry, float4 base, float4& carry,
                                 uint64_t t_begin, int64_t ticket, bool skip) {
    const int lane = threadIdx.x & 31;
    const int64_t pos = j + 1;
    const int64_t lb = pos & (-pos);
    bool ok = true;
    float4 Na = Ta, Nx = Tx;
    bool Nb = Tb;
    for (int64_t k = 1; k < lb && !Nb; k <<= 1) {
        if (!fold_node(p, fbase, pos - k, Na, Nx, Nb, t_begin, ticket)) {
            ok = false;
            break;
        }
    }
    uint32_t* myflag = p.flags + fbase + j;
    if (ok) {
        const int64_t idx = (fbase + j) * 32 + lane;
        __stcg(p.node + 2 * idx, Na);
        __stcg(p.node + 2 * idx + 1, Nx);
        publish(myflag, Nb ? ST_NODE_RESET : ST_NODE, skip);
    } else {
        if (lane == 0 && !skip) ptx::st_release(myflag, ST_ERROR);
        return false;
    }
    carry = base;
    if (!need_carry) return true;
    float4 Ra = one2(), Rx = zero2();
    bool Rb = false;
    for (int64_t q = j; q > 0 && !Rb; q -= (q & (-q))) {
        if (!fold_node(p, fbase, q, Ra, Rx, Rb, t_begin, ticket)) return false;
    }
    carry = Rb ? Rx : cfma2(Ra, base, Rx);
    return true;
}

// ============================================================================
// forward
// ============================================================================
template <int W, int R, bool PER_STEP>
__global__ void __launch_bounds__(W * 32) diag_fwd_kernel(const Params p) {
    constexpr int T = W * R;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    float4* s_u = reinterpret_cast<float4*>(smem_raw);  // [T][32]
    float4* s_l = s_u + T * 32;                         // [T][32] (per-step lambda)
    __shared__ float4 s_wa[W][32], s_wx[W][32];
    __shared__ uint32_t s_wr[W];
    __shared__ float4 s_carry[32];
    __shared__ __align__(8) uint64_t s_bar;
    __shared__ long long s_ticket;
    __shared__ int s_abort;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        s_ticket = static_cast<long long>(atomicAdd(p.hdr + 1, 1u));
        s_abort = 0;
        ptx::mbar_init(&s_bar, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    const int64_t ticket = s_ticket;
    const int64_t j = ticket / p.n_chains;       // position in chain = time tile
    const int64_t chain = ticket - j * p.n_chains;
    const int64_t b = chain / p.n_slabs;
    const int64_t slab = chain - b * p.n_slabs;
    const int64_t t0 = j * T;
    const int64_t c2 = slab * (SLAB / 2);        // first float4 column of the slab
    const int width2 = static_cast<int>(lmin(SLAB / 2, p.D2 - c2));  // float4 columns
    const int nrows = static_cast<int>(lmin(T, p.L - t0));
    const uint64_t t_begin = ptx::globaltimer();

    if (warp == 0) {
        const uint32_t rb = static_cast<uint32_t>(width2) * 16u;
        if (lane == 0) ptx::mbar_arrive_expect_tx(&s_bar, rb * nrows * (PER_STEP ? 2u : 1u));
        __syncwarp();
        for (int r = lane; r < nrows; r += 32) {
            const int64_t g = (b * p.L + t0 + r) * p.D2 + c2;
            ptx::bulk_g2s(s_u + r * 32, p.in + g, rb, &s_bar);
            if (PER_STEP) ptx::bulk_g2s(s_l + r * 32, p.lambda + g, rb, &s_bar);
        }
    }

    // begin flags of this warp's steps (overlaps the copies)
    const int64_t ts = t0 + static_cast<int64_t>(warp) * R;
    const int nv = static_cast<int>(lmax(0, lmin(R, p.L - ts)));
    const uint32_t bit = (lane < nv) ? (p.start[b * p.L + ts + lane] != 0) : 0u;
    const uint32_t rmask = __ballot_sync(0xffffffffu, bit);
    const bool lane_ok = lane < width2;
    const float4 lam = (!PER_STEP && lane_ok) ? p.lambda[c2 + lane] : one2();

    if (!wait_tma(p, &s_bar, t_begin, ticket)) return;

    // phase 1: aggregate of this warp's R steps (from the identity)
    float4 a = one2(), x = zero2();
    for (int i = 0; i < nv; ++i) {
        const float4 uu = s_u[(warp * R + i) * 32 + lane];
        const float4 ll = PER_STEP ? s_l[(warp * R + i) * 32 + lane] : lam;
        if ((rmask >> i) & 1u) {
            a = ll;
            x = uu;
        } else {
            x = cfma2(ll, x, uu);
            a = cmul2(ll, a);
        }
    }
    s_wa[warp][lane] = a;
    s_wx[warp][lane] = x;
    if (lane == 0) s_wr[warp] = (rmask != 0u);
    __syncthreads();

    // phase 2: tile aggregate, publish, look back (warp 0)
    if (warp == 0) {
        float4 Ta = one2(), Tx = zero2();
        bool Tb = false;
        for (int v = 0; v < W; ++v) {
            const float4 wa = s_wa[v][lane], wx = s_wx[v][lane];
            if (s_wr[v]) {
                Ta = wa;
                Tx = wx;
                Tb = true;
            } else {
                Tx = cfma2(wa, Tx, wx);
                Ta = cmul2(wa, Ta);
            }
        }
        const int64_t fbase = chain * p.n_tt;
        const bool skip = (ticket == p.withhold);
        const bool first_is_start = (rmask & 1u) != 0u;
        // state before the chain's first step: h0 (or the identity's 0)
        const float4 base = (p.h0 != nullptr && lane_ok) ? p.h0[b * p.D2 + c2 + lane] : zero2();
        float4 carry = zero2();
        const bool ok = fenwick_lookback(p, fbase, j, Ta, Tx, Tb, !first_is_start, base, carry,
                                         t_begin, ticket, skip);
        s_carry[lane] = carry;
        if (lane == 0 && !ok) s_abort = 1;
    }
    __syncthreads();
    if (s_abort) return;

    // phase 3: carry into this warp, recompute and store
    float4 Ea = one2(), Ex = zero2();
    bool Eb = false;
    for (int v = 0; v < warp; ++v) {
        const float4 wa = s_wa[v][lane], wx = s_wx[v][lane];
        if (s_wr[v]) {
            Ea = wa;
            Ex = wx;
            Eb = true;
        } else {
            Ex = cfma2(wa, Ex, wx);
            Ea = cmul2(wa, Ea);
        }
    }
    float4 hc = Eb ? Ex : cfma2(Ea, s_carry[lane], Ex);
    if (lane_ok) {
        float4* dst = p.out + (b * p.L + ts) * p.D2 + c2 + lane;
        for (int i = 0; i < nv; ++i) {
            const float4 uu = s_u[(warp * R + i) * 32 + lane];
            const float4 ll = PER_STEP ? s_l[(warp * R + i) * 32 + lane] : lam;
            hc = ((rmask >> i) & 1u) ? uu : cfma2(ll, hc, uu);
            __stcs(dst + static_cast<int64_t>(i) * p.D2, hc);
        }
        if (p.out_last != nullptr && nv > 0 && ts + nv == p.L) p.out_last[b * p.D2 + c2 + lane] = hc;
    }
}

// ============================================================================
// backward (right-to-left)
// ============================================================================
template <int W, int R, bool PER_STEP>
__global__ void __launch_bounds__(W * 32) diag_bwd_kernel(const Params p) {
    static_assert(R < 32, "R + 1 begin flags are read by one warp");
    constexpr int T = W * R;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    float4* s_g = reinterpret_cast<float4*>(smem_raw);  // row i: grad_h_{t0+i}
    float4* s_h = s_g + T * 32;                          // row i: h_{t0+i-1}
    float4* s_l = s_h + T * 32;                          // row i: lambda_{t0+i+1} (per step)
    __shared__ float4 s_wa[W][32], s_wx[W][32];
    __shared__ uint32_t s_wr[W];
    __shared__ float4 s_carry[32];
    __shared__ float4 s_acc[W][32];
    __shared__ __align__(8) uint64_t s_bar;
    __shared__ long long s_ticket;
    __shared__ int s_abort;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        s_ticket = static_cast<long long>(atomicAdd(p.hdr + 1, 1u));
        s_abort = 0;
        ptx::mbar_init(&s_bar, 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    const int64_t ticket = s_ticket;
    const int64_t jr = ticket / p.n_chains;  // position in chain (right to left)
    const int64_t chain = ticket - jr * p.n_chains;
    const int64_t j = p.n_tt - 1 - jr;       // time tile
    const int64_t b = chain / p.n_slabs;
    const int64_t slab = chain - b * p.n_slabs;
    const int64_t t0 = j * T;
    const int64_t c2 = slab * (SLAB / 2);
    const int width2 = static_cast<int>(lmin(SLAB / 2, p.D2 - c2));
    const int nrows = static_cast<int>(lmin(T, p.L - t0));
    const uint64_t t_begin = ptx::globaltimer();

    if (warp == 0) {
        const uint32_t rb = static_cast<uint32_t>(width2) * 16u;
        const int h_rows = nrows - (t0 == 0 ? 1 : 0);                               // rows t0-1 .. t0+nrows-2
        const int l_rows = PER_STEP ? static_cast<int>(lmin(nrows, p.L - 1 - t0)) : 0;  // rows t0+1 ..
        if (lane == 0) ptx::mbar_arrive_expect_tx(&s_bar, rb * (nrows + h_rows + l_rows));
        __syncwarp();
        for (int r = lane; r < nrows; r += 32) {
            const int64_t g = (b * p.L + t0 + r) * p.D2 + c2;
            ptx::bulk_g2s(s_g + r * 32, p.in + g, rb, &s_bar);
            if (t0 + r >= 1) ptx::bulk_g2s(s_h + r * 32, p.h + g - p.D2, rb, &s_bar);
            if (PER_STEP && r < l_rows) ptx::bulk_g2s(s_l + r * 32, p.lambda + g + p.D2, rb, &s_bar);
        }
    }

    const int64_t ts = t0 + static_cast<int64_t>(warp) * R;
    const int nv = static_cast<int>(lmax(0, lmin(R, p.L - ts)));
    // bit i of bmask: b_{ts+i} for i <= R (0 past the tape end)
    const uint32_t bit = (lane <= R && ts + lane < p.L) ? (p.start[b * p.L + ts + lane] != 0) : 0u;
    const uint32_t bmask = __ballot_sync(0xffffffffu, bit);
    const uint32_t rmask = bmask >> 1;  // bit i: b_{ts+i+1}, the reset of the reverse element
    const bool lane_ok = lane < width2;
    const float4 lam = (!PER_STEP && lane_ok) ? p.lambda[c2 + lane] : one2();
    const float4 mlam = conj2(lam);

    if (!wait_tma(p, &s_bar, t_begin, ticket)) return;

    // phase 1: aggregate over this warp's steps, right to left
    float4 a = one2(), x = zero2();
    for (int i = nv - 1; i >= 0; --i) {
        const int64_t t = ts + i;
        const float4 gg = s_g[(warp * R + i) * 32 + lane];
        const float4 m = (t == p.L - 1) ? one2() : (PER_STEP ? conj2(s_l[(warp * R + i) * 32 + lane]) : mlam);
        if ((rmask >> i) & 1u) {
            a = m;
            x = gg;
        } else {
            x = cfma2(m, x, gg);
            a = cmul2(m, a);
        }
    }
    const uint32_t vmask = (nv >= 32) ? 0xffffffffu : ((1u << nv) - 1u);
    s_wa[warp][lane] = a;
    s_wx[warp][lane] = x;
    if (lane == 0) s_wr[warp] = ((rmask & vmask) != 0u);
    __syncthreads();

    if (warp == 0) {
        float4 Ta = one2(), Tx = zero2();
        bool Tb = false;
        for (int v = W - 1; v >= 0; --v) {
            const float4 wa = s_wa[v][lane], wx = s_wx[v][lane];
            if (s_wr[v]) {
                Ta = wa;
                Tx = wx;
                Tb = true;
            } else {
                Tx = cfma2(wa, Tx, wx);
                Ta = cmul2(wa, Ta);
            }
        }
        const int64_t fbase = chain * p.n_tt;
        const bool skip = (ticket == p.withhold);
        // the first step processed is t0 + nrows - 1; its carry is cut if b_{t0+nrows} = 1
        const int64_t tn = t0 + nrows;
        const bool first_cut = (tn < p.L) && (p.start[b * p.L + tn] != 0);
        // adjoint entering the chain's first (right-most) step: grad_h_last (or 0)
        const float4 base = (p.g_last != nullptr && lane_ok) ? p.g_last[b * p.D2 + c2 + lane] : zero2();
        float4 carry = zero2();
        const bool ok = fenwick_lookback(p, fbase, jr, Ta, Tx, Tb, !first_cut, base, carry,
                                         t_begin, ticket, skip);
        s_carry[lane] = carry;
        if (lane == 0 && !ok) s_abort = 1;
    }
    __syncthreads();
    if (s_abort) return;

    // carry into this warp from the warps to its right
    float4 Ea = one2(), Ex = zero2();
    bool Eb = false;
    for (int v = W - 1; v > warp; --v) {
        const float4 wa = s_wa[v][lane], wx = s_wx[v][lane];
        if (s_wr[v]) {
            Ea = wa;
            Ex = wx;
            Eb = true;
        } else {
            Ex = cfma2(wa, Ex, wx);
            Ea = cmul2(wa, Ea);
        }
    }
    float4 delta = Eb ? Ex : cfma2(Ea, s_carry[lane], Ex);
    float4 acc = zero2();
    if (lane_ok) {
        float4* dst = p.out + (b * p.L + ts) * p.D2 + c2 + lane;
        for (int i = nv - 1; i >= 0; --i) {
            const int64_t t = ts + i;
            const float4 gg = s_g[(warp * R + i) * 32 + lane];
            const float4 m = (t == p.L - 1) ? one2() : (PER_STEP ? conj2(s_l[(warp * R + i) * 32 + lane]) : mlam);
            delta = ((rmask >> i) & 1u) ? gg : cfma2(m, delta, gg);
            __stcs(dst + static_cast<int64_t>(i) * p.D2, delta);
            float4 gl = zero2();
            if (!((bmask >> i) & 1u)) {
                float4 hp;
                if (t > 0) hp = s_h[(warp * R + i) * 32 + lane];
                else hp = (p.h0 != nullptr) ? p.h0[b * p.D2 + c2 + lane] : zero2();
                gl = cmul2(delta, conj2(hp));
            }
            if (PER_STEP) {
                if (p.grad_lambda != nullptr) __stcs(p.grad_lambda + (b * p.L + t) * p.D2 + c2 + lane, gl);
            } else {
                acc = add2(acc, gl);
            }
            if (t == 0 && p.grad_h0 != nullptr) {
                float4 l0 = lam;
                if (PER_STEP) l0 = p.lambda[(b * p.L) * p.D2 + c2 + lane];
                p.grad_h0[b * p.D2 + c2 + lane] = (bmask & 1u) ? zero2() : cmul2(conj2(l0), delta);
            }
        }
    }
    if (!PER_STEP) {
        s_acc[warp][lane] = acc;
        __syncthreads();
        if (warp == 0) {
            float4 s = zero2();
            for (int v = 0; v < W; ++v) s = add2(s, s_acc[v][lane]);
            p.gpart[(chain * p.n_tt + j) * 32 + lane] = s;
        }
    }
}

// ============================================================================
// grad_lambda reduction (per-channel lambda): fixed-order fp64 sums
// ============================================================================
__global__ void __launch_bounds__(256) reduce_parts_kernel(const float4* __restrict__ gpart,
                                                           double* __restrict__ rpart, int64_t B,
                                                           int64_t n_slabs, int64_t n_tt) {
    __shared__ double s[8][32][4];
    const int slab = blockIdx.x, part = blockIdx.y;
    const int grp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t total = B * n_tt;
    const int64_t per = (total + RED_PARTS - 1) / RED_PARTS;
    const int64_t k0 = part * per, k1 = lmin(total, k0 + per);
    double acc[4] = {0.0, 0.0, 0.0, 0.0};
    for (int64_t k = k0 + grp; k < k1; k += 8) {
        const int64_t bb = k / n_tt, jj = k - bb * n_tt;
        const float4 v = gpart[((bb * n_slabs + slab) * n_tt + jj) * 32 + lane];
        acc[0] += v.x;
        acc[1] += v.y;
        acc[2] += v.z;
        acc[3] += v.w;
    }
    for (int c = 0; c < 4; ++c) s[grp][lane][c] = acc[c];
    __syncthreads();
    if (grp == 0) {
        double r[4] = {0.0, 0.0, 0.0, 0.0};
        for (int g = 0; g < 8; ++g)
            for (int c = 0; c < 4; ++c) r[c] += s[g][lane][c];
        double* o = rpart + ((static_cast<int64_t>(slab) * RED_PARTS + part) * 32 + lane) * 4;
        for (int c = 0; c < 4; ++c) o[c] = r[c];
    }
}

__global__ void reduce_final_kernel(const double* __restrict__ rpart, float4* __restrict__ grad_lambda,
                                    int64_t D2) {
    const int slab = blockIdx.x, lane = threadIdx.x;
    double r[4] = {0.0, 0.0, 0.0, 0.0};
    for (int part = 0; part < RED_PARTS; ++part) {
        const double* o = rpart + ((static_cast<int64_t>(slab) * RED_PARTS + part) * 32 + lane) * 4;
        for (int c = 0; c < 4; ++c) r[c] += o[c];
    }
    const int64_t col = static_cast<int64_t>(slab) * 32 + lane;
    if (col < D2)
        grad_lambda[col] = make_float4(static_cast<float>(r[0]), static_cast<float>(r[1]),
                                       static_cast<float>(r[2]), static_cast<float>(r[3]));
}

// ============================================================================
// host side
// ============================================================================
namespace {

struct Layout {
    int64_t n_slabs, n_tt_max, n_chains;
    size_t flags_off, node_off, gpart_off, rpart_off, total;
};

Layout layout(int64_t B, int64_t L, int64_t D) {
    Layout l{};
    l.n_slabs = (D + SLAB - 1) / SLAB;
    l.n_tt_max = (L + MIN_T - 1) / MIN_T;
    l.n_chains = B * l.n_slabs;
    const size_t tiles = static_cast<size_t>(l.n_chains) * static_cast<size_t>(l.n_tt_max);
    l.flags_off = kHeaderBytes;
    l.node_off = align_up(l.flags_off + tiles * 4, 256);
    l.gpart_off = align_up(l.node_off + tiles * 32 * 32, 256);
    l.rpart_off = align_up(l.gpart_off + tiles * 32 * 16, 256);
    l.total = align_up(l.rpart_off + static_cast<size_t>(l.n_slabs) * RED_PARTS * 32 * 32, 256);
    return l;
}

template <typename K>
cudaError_t set_smem(K kernel, int bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

Params make_params(const Args& a, const Layout& l, int64_t n_tt) {
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
    p.D = a.D;
    p.D2 = a.D / 2;
    p.n_slabs = l.n_slabs;
    p.n_tt = n_tt;
    p.n_chains = l.n_chains;
    unsigned char* ws = static_cast<unsigned char*>(a.workspace);
    p.hdr = reinterpret_cast<uint32_t*>(ws);
    p.flags = reinterpret_cast<uint32_t*>(ws + l.flags_off);
    p.node = reinterpret_cast<float4*>(ws + l.node_off);
    p.gpart = reinterpret_cast<float4*>(ws + l.gpart_off);
    const DebugKnobs k = debug_knobs();
    p.wait_ns = k.wait_ns;
    p.withhold = k.withhold_ticket;
    return p;
}

cudaError_t clear_status(const Args& a, const Layout& l, int64_t n_tt, cudaStream_t s) {
    const size_t bytes = l.flags_off + static_cast<size_t>(l.n_chains) * n_tt * 4;
    return cudaMemsetAsync(a.workspace, 0, bytes, s);
}

}  // namespace

size_t workspace_bytes(int64_t B, int64_t L, int64_t D) { return layout(B, L, D).total; }

memoroid_status_t launch_fwd(const Args& a, cudaStream_t s) {
    const Layout l = layout(a.B, a.L, a.D);
    const bool ps = a.lambda_per_step != 0;
    const int T = ps ? FWDS_W * FWDS_R : FWD_W * FWD_R;
    const int64_t n_tt = (a.L + T - 1) / T;
    const int64_t n_tiles = n_tt * l.n_chains;
    if (n_tiles > 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;
    if (clear_status(a, l, n_tt, s) != cudaSuccess) return MEMOROID_ERR_CUDA;
    const Params p = make_params(a, l, n_tt);
    cudaError_t e;
    if (ps) {
        const int smem = 2 * T * 32 * 16;
        auto k = diag_fwd_kernel<FWDS_W, FWDS_R, true>;
        e = set_smem(k, smem);
        if (e == cudaSuccess) k<<<static_cast<unsigned>(n_tiles), FWDS_W * 32, smem, s>>>(p);
    } else {
        const int smem = T * 32 * 16;
        auto k = diag_fwd_kernel<FWD_W, FWD_R, false>;
        e = set_smem(k, smem);
        if (e == cudaSuccess) k<<<static_cast<unsigned>(n_tiles), FWD_W * 32, smem, s>>>(p);
    }
    if (e != cudaSuccess || cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    return MEMOROID_OK;
}

memoroid_status_t launch_bwd(const Args& a, cudaStream_t s) {
    const Layout l = layout(a.B, a.L, a.D);
    const bool ps = a.lambda_per_step != 0;
    const int T = ps ? BWDS_W * BWDS_R : BWD_W * BWD_R;
    const int64_t n_tt = (a.L + T - 1) / T;
    const int64_t n_tiles = n_tt * l.n_chains;
    if (n_tiles > 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;
    if (clear_status(a, l, n_tt, s) != cudaSuccess) return MEMOROID_ERR_CUDA;
    const Params p = make_params(a, l, n_tt);
    cudaError_t e;
    if (ps) {
        const int smem = 3 * T * 32 * 16;
        auto k = diag_bwd_kernel<BWDS_W, BWDS_R, true>;
        e = set_smem(k, smem);
        if (e == cudaSuccess) k<<<static_cast<unsigned>(n_tiles), BWDS_W * 32, smem, s>>>(p);
    } else {
        const int smem = 2 * T * 32 * 16;
        auto k = diag_bwd_kernel<BWD_W, BWD_R, false>;
        e = set_smem(k, smem);
        if (e == cudaSuccess) k<<<static_cast<unsigned>(n_tiles), BWD_W * 32, smem, s>>>(p);
    }
    if (e != cudaSuccess || cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (!ps && a.grad_lambda != nullptr) {
        unsigned char* ws = static_cast<unsigned char*>(a.workspace);
        double* rpart = reinterpret_cast<double*>(ws + l.rpart_off);
        reduce_parts_kernel<<<dim3(static_cast<unsigned>(l.n_slabs), RED_PARTS), 256, 0, s>>>(
            p.gpart, rpart, a.B, l.n_slabs, n_tt);
        reduce_final_kernel<<<static_cast<unsigned>(l.n_slabs), 32, 0, s>>>(
            rpart, static_cast<float4*>(a.grad_lambda), p.D2);
        if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    }
    return MEMOROID_OK;
}

}  // namespace diag
}  // namespace memoroid
