// linattn.cu -- the decayed, resettable linear-attention memoroid on tcgen05.
//
// Recurrence: the Linear Transformer memoroid (appendix "Rewriting Sequence
// Models as Memoroids") with a decay gamma_t, reset by the begin-of-episode
// flag b_t (Section 2.1) through the resettable monoid of Theorem 3.2:
//   S_t = [b_t = 0] gamma_t S_{t-1} + k_t v_t^T        (S: dk x dv, fp32)
//   y_t = S_t^T q_t
// The tape is cut into 128-step tiles.  Inside a tile the recurrence is the
// masked, decayed quadratic form
//   y_t = sum_{r <= t, same episode} exp(Lam_t - Lam_r) (q_t . k_r) v_r
//         + [no start in tile up to t] exp(Lam_t) S_prev^T q_t
// with Lam the running sum of log gamma over the tile, and the tile's state is
//   S_tile = [no start in tile] exp(Lam_end) S_prev + sum_{r >= last start} exp(Lam_end - Lam_r) k_r v_r^T.
// Both are dense bf16 contractions with fp32 accumulators in tensor memory.
//
// Parallel structure: the tape of each (tape, head) is cut into G segments of
// tps whole tiles, one CTA each, which walks its tiles in order carrying the
// state in TMEM from the state entering the segment.  Those entry states come
// from a resettable scan over the segments (Theorem 3.2 applied to segment
// aggregates): a summary kernel computes, per segment, the state its rows
// after the last begin flag leave behind from a zero start (rows whose decay
// weight underflows are skipped), and a carry kernel folds the summaries in
// order, S_exit(g) = [no flag in g] a_g S_exit(g-1) + X_g.  The backward
// runs the same scan in reverse for the reverse state.  The amount of work
// therefore does not depend on where the begin flags fall: a tape with one
// episode runs on as many CTAs as one with many.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <mutex>

#include <cstdint>

#include "internal.cuh"
#include "ptx.cuh"

namespace memoroid {
namespace la {

using namespace ptx;

constexpr int T = 128;         // steps per tile = the M of the tile contractions
// After a wait has run out, in-flight TMA loads and tensor-core batches are
// drained with this fixed limit before the CTA frees its TMEM and exits.
constexpr uint64_t kDrainNs = 1000000000ull;
constexpr int kThreads = 256;   // forward / pass F: 8 warps, warp w reads TMEM lane quarter w % 4, column half w / 4
constexpr int kRThreads = 512;  // pass R: 16 warps, warp w reads lane quarter w % 4, column quarter w / 4
constexpr int kTargetCtas = 152;

// Per-tile decay and reset summary, computed once per (tape, head, tile).
struct __align__(16) TileMeta {
    float lam2[T];        // running sum of log2(gamma) over the tile's rows; start rows and rows past L add 0
    int8_t seg[T];        // index of the last start row <= r within the tile, -1 if none
    float a;              // decay of the whole tile: 0 if it holds a start, else exp2(lam2[T-1])
    int32_t has_start;
    int32_t first_start;  // T if none
    int32_t last_start;   // -1 if none
};
static_assert(sizeof(TileMeta) == 656, "TileMeta is copied as 41 16-byte chunks");

// ---------------------------------------------------------------------------
// segment plan and workspace layout
// ---------------------------------------------------------------------------
// Segment g of a (tape, head) holds tiles [g * tps, min((g + 1) * tps, n_tiles)).
struct Plan {
    int64_t n_tiles, tps, G;  // tiles per tape, tiles per segment, segments per (tape, head)
};

Plan make_plan(int64_t B, int64_t L, int64_t H) {
    Plan p;
    p.n_tiles = (L + T - 1) / T;
    const int64_t bh = B * H;
    int64_t G = bh > 0 ? kTargetCtas / bh : 1;
    if (G < 1) G = 1;
    if (G > p.n_tiles) G = p.n_tiles;
    if (G < 1) G = 1;
    p.tps = p.n_tiles > 0 ? (p.n_tiles + G - 1) / G : 1;
    p.G = p.n_tiles > 0 ? (p.n_tiles + p.tps - 1) / p.tps : 1;
    return p;
}

struct Layout {
    size_t meta, info, carry_f, fwd_total;
    size_t dy16, states, dlam_f, gpart, carry_r, total;  // backward only
};

Layout make_layout(int64_t B, int64_t L, int64_t H, int64_t D) {
    const Plan pl = make_plan(B, L, H);
    const size_t nseg = static_cast<size_t>(B * H * pl.G);
    Layout ly;
    size_t off = kHeaderBytes;
    ly.meta = off;
    off = align_up(off + static_cast<size_t>(B * H * pl.n_tiles) * sizeof(TileMeta), 256);
    ly.info = off;  // per segment: (begin flag in the segment, log2 of its decay)
    off = align_up(off + nseg * sizeof(float2), 256);
    ly.carry_f = off;  // per segment: its summary, then (carry) the state leaving it
    off = align_up(off + nseg * static_cast<size_t>(D * D) * sizeof(float), 256);
    ly.fwd_total = off;
    ly.dy16 = off;
    off = align_up(off + static_cast<size_t>(B * L * H * D) * sizeof(uint16_t), 256);
    ly.states = off;
    off = align_up(off + static_cast<size_t>(B * H * pl.n_tiles * D * D) * sizeof(uint16_t), 256);
    ly.dlam_f = off;
    off = align_up(off + static_cast<size_t>(B * L * H) * sizeof(float), 256);
    ly.gpart = off;
    off = align_up(off + static_cast<size_t>(B * H * pl.G) * sizeof(float), 256);
    ly.carry_r = off;  // per segment: its reverse summary, then the reverse state leaving it
    off = align_up(off + nseg * static_cast<size_t>(D * D) * sizeof(float), 256);
    ly.total = off;
    return ly;
}

// ---------------------------------------------------------------------------
// kernel 1: tile metadata (log-decay prefix sums, start positions)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) meta_kernel(const float* __restrict__ gamma, int per_step,
                                                   const uint8_t* __restrict__ start, int64_t B, int64_t L,
                                                   int64_t H, int64_t n_tiles, TileMeta* __restrict__ meta) {
    const int64_t wid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (wid >= B * n_tiles * H) return;
    // (tape, tile, head) with the head fastest: the warps of a block read the
    // same gamma rows
    const int64_t h = wid % H;
    const int64_t tile = (wid / H) % n_tiles;
    const int64_t b = wid / (H * n_tiles);
    float lg[4];
    int sg[4];
    int first = T;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int r = lane * 4 + k;
        const int64_t t = tile * T + r;
        const bool valid = t < L;
        const bool st = valid && start[b * L + t] != 0;
        float l = 0.f;
        if (valid && !st) {
            const float g = per_step ? gamma[(b * L + t) * H + h] : gamma[h];
            // gamma is a decay: clamped to [2^-126, 1] (gamma = 0 gives a weight of at
            // most 2^-126 instead of 0)
            l = fminf(fmaxf(log2f(g), -126.f), 0.f);
        }
        lg[k] = l;
        sg[k] = st ? r : -1;
        if (st && r < first) first = r;
    }
#pragma unroll
    for (int k = 1; k < 4; ++k) {
        lg[k] += lg[k - 1];
        sg[k] = max(sg[k], sg[k - 1]);
    }
    float tot = lg[3];
    int mx = sg[3];
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float o = __shfl_up_sync(0xffffffffu, tot, off);
        const int om = __shfl_up_sync(0xffffffffu, mx, off);
        if (lane >= off) {
            tot += o;
            mx = max(mx, om);
        }
    }
    float ex = __shfl_up_sync(0xffffffffu, tot, 1);
    int exm = __shfl_up_sync(0xffffffffu, mx, 1);
    if (lane == 0) {
        ex = 0.f;
        exm = -1;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) first = min(first, __shfl_xor_sync(0xffffffffu, first, off));

    TileMeta* m = meta + (b * H + h) * n_tiles + tile;
    float4 l4;
    l4.x = lg[0] + ex;
    l4.y = lg[1] + ex;
    l4.z = lg[2] + ex;
    l4.w = lg[3] + ex;
    reinterpret_cast<float4*>(m->lam2)[lane] = l4;
    char4 s4;
    s4.x = static_cast<signed char>(max(sg[0], exm));
    s4.y = static_cast<signed char>(max(sg[1], exm));
    s4.z = static_cast<signed char>(max(sg[2], exm));
    s4.w = static_cast<signed char>(max(sg[3], exm));
    reinterpret_cast<char4*>(m->seg)[lane] = s4;
    if (lane == 31) {
        m->has_start = mx >= 0 ? 1 : 0;
        m->a = mx >= 0 ? 0.f : exp2f(tot);
        m->first_start = first;
        m->last_start = mx;
    }
}

// ---------------------------------------------------------------------------
// shared-memory operand layout
// ---------------------------------------------------------------------------
// Every [rows x cols] bf16 operand tile uses the no-swizzle core-matrix layout
//   byte(row, col) = (row / 8) * (cols * 16) + (col / 8) * 128 + (row % 8) * 16 + (col % 8) * 2
// i.e. 8x8 core matrices (8 rows of 16 contiguous bytes), col-groups adjacent.
// Read with rows as M/N and cols as K (K-major): LBO = 128, SBO = cols * 16,
// K step of 16 = +256 bytes.  Read with cols as M/N and rows as K (MN-major):
// LBO = cols * 16, SBO = 128, K step of 16 = +2 * cols * 16 bytes.
__device__ __forceinline__ uint32_t core_off(int row, int col, int cols) {
    return static_cast<uint32_t>((row >> 3) * (cols * 16) + (col >> 3) * 128 + (row & 7) * 16 + (col & 7) * 2);
}
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t base, int cols, int kk) {
    return tc::smem_desc(base + kk * 256, 128, cols * 16);
}
__device__ __forceinline__ uint64_t desc_mnmajor(uint32_t base, int cols, int kk) {
    return tc::smem_desc(base + kk * 2 * cols * 16, cols * 16, 128);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ float2 unpack_bf16x2(uint32_t w) {
    __nv_bfloat162 v;
    *reinterpret_cast<uint32_t*>(&v) = w;
    return __bfloat1622float2(v);
}

// Operand tiles of T steps x D channels are loaded by TMA with 128-byte
// swizzling: one box per 64 channels ("chunk", T rows of 128 bytes, chunk m at
// m * T * 128), and within a chunk the 16-byte unit u of row r stored at unit
// u ^ (r % 8):
//   byte(row, col) = (col / 64) * T * 128 + row * 128 + (((col % 64) / 8) ^ (row % 8)) * 16 + (col % 8) * 2.
// Read with rows as M/N and cols as K (K-major): SBO = 1024 (8-row groups),
// the K step of 16 moves the start by 32 bytes inside a chunk.  Read with cols
// as M/N and rows as K (MN-major): LBO = T * 128 (the next 64 columns), SBO =
// 1024, K step of 16 rows = +2048 bytes.  Chunks are 1024-byte aligned.
__device__ __forceinline__ uint32_t sw_off(int row, int col) {
    return static_cast<uint32_t>((col >> 6) * (T * 128) + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4) +
                                 (col & 7) * 2);
}
__device__ __forceinline__ uint64_t sw_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
    return tc::smem_desc(addr, lbo, sbo) | (static_cast<uint64_t>(2) << 61);  // layout: 128-byte swizzle
}
__device__ __forceinline__ uint64_t desc_sw_k(uint32_t base, int kk) {
    return sw_desc(base + (kk >> 2) * (T * 128) + (kk & 3) * 32, 16, 1024);
}
__device__ __forceinline__ uint64_t desc_sw_mn(uint32_t base, int kk) {
    return sw_desc(base + kk * 2048, T * 128, 1024);
}

// One [T x D] bf16 tile, steps t0..t0+T-1 of head h of tape b, from a 4-D
// tensor map {D, H, L, B} with 128-byte swizzling: D/64 boxes of {64, 1, T, 1}.
// Steps past L read as 0.
template <int D>
__device__ __forceinline__ void tma_tile(uint32_t dst, const CUtensorMap* map, int64_t h, int64_t t0, int64_t b,
                                         uint64_t* bar) {
#pragma unroll
    for (int m = 0; m < D / 64; ++m)
        tma_load_4d(dst + m * T * 128, map, 64 * m, static_cast<int>(h), static_cast<int>(t0), static_cast<int>(b), bar);
}

// Scales row r of a 128-byte swizzled [T x D] bf16 tile by w[r] in place: one
// thread per (row, 64-channel chunk) while there are enough threads, each
// with one weight and eight 16-byte units (conflict-free: the swizzle spreads
// the same unit of 8 consecutive rows over 8 bank groups).  SELECT: rows of
// weight 0 become exact zeros (the forward's, so that a non-finite q or k stays
// in its episode).
template <int D, int NT = kThreads, bool SELECT = false, typename WFn>
__device__ __forceinline__ void scale_rows_sw(unsigned char* tile, int tid, WFn weight) {
    constexpr int CHUNKS = D / 64;
    constexpr int UNITS = 8 * CHUNKS * T / NT;  // units per thread (NT threads)
    static_assert(UNITS >= 1, "at most one thread per 16-byte unit");
    const int r = tid & (T - 1);
    const float w = weight(r);
    if (w == 1.f) return;
    unsigned char* row = tile + r * 128;
#pragma unroll
    for (int i = 0; i < UNITS; ++i) {
        // thread tid covers units (tid / T) * UNITS + i of its row (chunk = unit / 8)
        const int unit = (tid / T) * UNITS + i;
        unsigned char* a = row + (unit >> 3) * (T * 128) + (((unit & 7) ^ (r & 7)) << 4);
        uint4 u = *reinterpret_cast<uint4*>(a);
        float2 f;
        f = unpack_bf16x2(u.x);
        u.x = pack_bf16x2(f.x * w, f.y * w);
        f = unpack_bf16x2(u.y);
        u.y = pack_bf16x2(f.x * w, f.y * w);
        f = unpack_bf16x2(u.z);
        u.z = pack_bf16x2(f.x * w, f.y * w);
        f = unpack_bf16x2(u.w);
        u.w = pack_bf16x2(f.x * w, f.y * w);
        if (SELECT && w == 0.f) u = make_uint4(0u, 0u, 0u, 0u);
        *reinterpret_cast<uint4*>(a) = u;
    }
}

// phi'(z) of the raw input (1 above 0, else e^z, by the SFU exponential: a
// few ulp of fp32): the chain rule of the normalised backward, applied to dq
// and dk in the epilogues
__device__ __forceinline__ float phi_prime(float z) { return z > 0.f ? 1.f : __expf(z); }
__device__ __forceinline__ float4 times_phi_prime(float4 o, uint2 raw) {
    const float2 a = unpack_bf16x2(raw.x), b = unpack_bf16x2(raw.y);
    return make_float4(o.x * phi_prime(a.x), o.y * phi_prime(a.y), o.z * phi_prime(b.x), o.w * phi_prime(b.y));
}

// phi(z) = 1 + ELU(z) in place on the first 64-channel box of a [T x 128]
// operand slot (bf16, round to nearest, the SFU exponential); rows at or past
// `valid` become 0, as rows past the tape end of padded operands are.  NT
// threads, one 16-byte unit (8 channels) of one row per step.
template <int NT>
__device__ __forceinline__ void phi_box(unsigned char* slot, int tid, int64_t valid) {
#pragma unroll
    for (int i = 0; i < T * 8 / NT; ++i) {
        const int unit = i * NT + tid, row = unit / 8;
        uint4* a = reinterpret_cast<uint4*>(slot + unit * 16);
        uint4 u = *a;
        uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = unpack_bf16x2(w[e]);
            w[e] = row < valid ? pack_bf16x2(f.x > 0.f ? 1.f + f.x : __expf(f.x), f.y > 0.f ? 1.f + f.y : __expf(f.y))
                               : 0u;
        }
        *a = u;
    }
}

// psi(z) = ELU(z) = phi(z) - 1 in place on the first 64-channel box (the
// normalised backward's key operand; rows at or past `valid` become 0).
template <int NT>
__device__ __forceinline__ void psi_box(unsigned char* slot, int tid, int64_t valid) {
#pragma unroll
    for (int i = 0; i < T * 8 / NT; ++i) {
        const int unit = i * NT + tid, row = unit / 8;
        uint4* a = reinterpret_cast<uint4*>(slot + unit * 16);
        uint4 u = *a;
        uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = unpack_bf16x2(w[e]);
            w[e] = row < valid ? pack_bf16x2(f.x > 0.f ? f.x : __expf(f.x) - 1.f, f.y > 0.f ? f.y : __expf(f.y) - 1.f)
                               : 0u;
        }
        *a = u;
    }
}

// Sum of the 8 values of a 16-byte unit of bf16, in channel order.
__device__ __forceinline__ float unit_sum(const uint4& u) {
    const uint32_t* w = reinterpret_cast<const uint32_t*>(&u);
    float acc = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float2 f = unpack_bf16x2(w[e]);
        acc += f.x;
        acc += f.y;
    }
    return acc;
}

// The normalised backward's query operand in place: phi on the first box (as
// phi_box) and, in channels 64 and 65 of the second box, sigma = sum of the
// row's 64 phi values as a bf16 pair (hi, lo = bf16(sigma - hi)); the rest of
// that 16-byte unit is 0 (the other units of the box are zeros already).  The
// 8 units of a row are 8 consecutive threads: unit sums in channel order,
// then a fixed butterfly over the units (the same association as the padded
// operands' builder, whatever the swizzle).
template <int NT>
__device__ __forceinline__ void phiq_box(unsigned char* slot, int tid, int64_t valid) {
#pragma unroll
    for (int i = 0; i < T * 8 / NT; ++i) {
        const int unit = i * NT + tid, row = unit / 8;
        uint4* a = reinterpret_cast<uint4*>(slot + unit * 16);
        uint4 u = *a;
        uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = unpack_bf16x2(w[e]);
            w[e] = row < valid ? pack_bf16x2(f.x > 0.f ? 1.f + f.x : __expf(f.x), f.y > 0.f ? 1.f + f.y : __expf(f.y))
                               : 0u;
        }
        *a = u;
        float sg = unit_sum(u);
        sg += __shfl_xor_sync(0xffffffffu, sg, 1);
        sg += __shfl_xor_sync(0xffffffffu, sg, 2);
        sg += __shfl_xor_sync(0xffffffffu, sg, 4);
        if ((unit & 7) == 0) {
            const float hi = __bfloat162float(__float2bfloat16_rn(sg));
            *reinterpret_cast<uint4*>(slot + T * 128 + row * 128 + ((row & 7) << 4)) =
                make_uint4(pack_bf16x2(hi, sg - hi), 0u, 0u, 0u);
        }
    }
}

// The second 64-channel box of a [T x 128] operand slot as a constant: zeros,
// or (ones) channels 64 and 65 of every row 1 and the rest 0.  Unit u of row r
// holds channels 8 (u ^ (r % 8)) .. + 7 of the box.
template <int NT>
__device__ __forceinline__ void const_box(unsigned char* slot, int tid, bool ones) {
    const uint32_t one2 = pack_bf16x2(1.f, 1.f);
    for (int i = tid; i < T * 8; i += NT) {
        const int r = i / 8, u = i % 8;
        *reinterpret_cast<uint4*>(slot + T * 128 + i * 16) = make_uint4(ones && (u ^ (r & 7)) == 0 ? one2 : 0u, 0u, 0u, 0u);
    }
}

__device__ __forceinline__ bool wait_mbar(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer() - t0 > limit_ns) return false;
    }
    return true;
}

__device__ __forceinline__ void record_error(uint32_t* hdr, uint32_t code) {
    if (hdr != nullptr) atomicCAS(hdr, 0u, code);
}

// ---------------------------------------------------------------------------
// kernel 2: forward main kernel
// ---------------------------------------------------------------------------
template <int D>
struct FwdSmem {
    static constexpr int TILE = T * D * 2;
    static constexpr int PM = T * T * 2;
    static constexpr int STAGE = 3 * TILE;       // Q, K, V
    static constexpr int OFF_SB = 2 * STAGE;     // bf16 state operand of the inter-tile term
    // d = 128: the masked scores live in the state operand's buffer, free from the
    // end of the first contractions to the epilogue, which writes the next state
    static constexpr bool PM_IN_SB = D * D * 2 >= PM;
    static constexpr int OFF_PM = PM_IN_SB ? OFF_SB : OFF_SB + D * D * 2;
    static constexpr int NMETA = 3;  // metadata ring: tiles c, c+1 in use, c+2 loading
    static constexpr int OFF_META = PM_IN_SB ? OFF_SB + D * D * 2 : OFF_PM + PM;
    static constexpr int OFF_Z = OFF_META + NMETA * static_cast<int>(sizeof(TileMeta));  // [2][T] fp32 (pass F)
    static constexpr int OFF_BAR = OFF_Z + 2 * T * 4;
    static constexpr int BYTES = OFF_BAR + 64;
    // the fp32 output tile is staged in the K and V slots of the finished stage
    // in the 128-byte swizzled layout of its TMA store (32 channels per 128-byte
    // row, chunk of 32 channels at m * T * 128); pass F loads the q tile into the
    // Q slot once the first contractions are done and then stages its stored state there
    static constexpr int OFF_Y = TILE;
    static_assert(T * D * 4 <= 2 * TILE, "output staging fits in the K and V slots of one stage");
    static_assert(D * D * 2 <= TILE, "pass F's stored state is staged in the Q slot of the same stage");
    // TMEM columns: scores P, intra output, inter output, state S
    static constexpr uint32_t COL_P = 0, COL_YA = 128, COL_YI = 128 + D, COL_S = 128 + 2 * D;
    static constexpr uint32_t TMEM_COLS = 512;
    static_assert(COL_S + D <= TMEM_COLS, "tensor memory budget");
};

struct FwdParams {
    CUtensorMap map_q, map_k, map_v;  // the q, k, v operands (4-D {D, H, L, B}, box {64, 1, 128, 1})
    CUtensorMap map_y;                // the fp32 output (4-D {D, H, L, B}, box {32, 1, 128, 1})
    CUtensorMap map_zq;               // pass F: q for the z term (as map_q)
    float* den;                       // normalised forward: the normalizer [B, L, H] (or null)
    const uint16_t* q;
    const uint16_t* k;
    const uint16_t* v;
    const float* S0;
    float* y;
    const TileMeta* meta;
    const float* carry;  // [B * H * G][D][D]: the state leaving each segment (g < G - 1)
    float* S_last;
    uint32_t* hdr;
    int64_t B, L, H, n_tiles, tps;
    int G;
    uint64_t wait_ns;
    int64_t fail_cta;  // test knob: this CTA reports its first tensor-core wait as timed out (-1: none)
    // backward pass F only (see fwd_kernel<D, true>)
    float* dlam_f;       // [B, L, H]: the state-side terms of dL/dlog(gamma_t)
    uint16_t* states;    // [B, H, n_tiles, D, D] bf16: S_{c-1}^T before tiles without a begin flag
    int fold_col;        // >= 0: output column added to every output column (pass F, normalised), else -1
};


// Thread -> row of a D x D state accumulator in TMEM.  With M = 128 the row
// is the TMEM lane; with M = 64 rows 16q..16q+15 sit in lanes 32q..32q+15 and
// the upper 16 lanes of each quarter hold nothing (-1).
// Byte offset of element (row, col) in the stored image of a D x D bf16
// state: rows of 2D bytes whose 16-byte unit u sits at u ^ (row % (D / 8)),
// so that eight consecutive rows written 16 bytes at a time (pass F), and one
// row read 2 bytes at a time by 32 consecutive columns (pass R), touch
// distinct bank groups of shared memory.
template <int D>
__device__ __forceinline__ uint32_t state_off(int row, int col) {
    return static_cast<uint32_t>(row * (2 * D) + ((((col >> 3) ^ (row & (D / 8 - 1)))) << 4) + (col & 7) * 2);
}

// 16 bf16 values of row `row` (columns j0..j0+15, j0 a multiple of 16) of a
// stored state image at `base` (global or shared memory).
template <int D>
__device__ __forceinline__ void store_state_row(unsigned char* base, int row, int j0, const float* v) {
    uint4 w0, w1;
    w0.x = pack_bf16x2(v[0], v[1]);
    w0.y = pack_bf16x2(v[2], v[3]);
    w0.z = pack_bf16x2(v[4], v[5]);
    w0.w = pack_bf16x2(v[6], v[7]);
    w1.x = pack_bf16x2(v[8], v[9]);
    w1.y = pack_bf16x2(v[10], v[11]);
    w1.z = pack_bf16x2(v[12], v[13]);
    w1.w = pack_bf16x2(v[14], v[15]);
    *reinterpret_cast<uint4*>(base + state_off<D>(row, j0)) = w0;
    *reinterpret_cast<uint4*>(base + state_off<D>(row, j0 + 8)) = w1;
}
template <int D>
__device__ __forceinline__ unsigned char* state_image(uint16_t* states, int64_t bh, int64_t n_tiles, int64_t tile) {
    return reinterpret_cast<unsigned char*>(states + (bh * n_tiles + tile) * D * D);
}

template <int D>
__device__ __forceinline__ int state_row(int quarter, int lane) {
    if (D == 128) return 32 * quarter + lane;
    return lane < 16 ? 16 * quarter + lane : -1;
}

__device__ __forceinline__ void store_bf16x16(unsigned char* base, uint32_t off0, uint32_t off1, const float* v) {
    uint4 w0, w1;
    w0.x = pack_bf16x2(v[0], v[1]);
    w0.y = pack_bf16x2(v[2], v[3]);
    w0.z = pack_bf16x2(v[4], v[5]);
    w0.w = pack_bf16x2(v[6], v[7]);
    w1.x = pack_bf16x2(v[8], v[9]);
    w1.y = pack_bf16x2(v[10], v[11]);
    w1.z = pack_bf16x2(v[12], v[13]);
    w1.w = pack_bf16x2(v[14], v[15]);
    *reinterpret_cast<uint4*>(base + off0) = w0;
    *reinterpret_cast<uint4*>(base + off1) = w1;
}

// BWD = false: the forward pass, y = S^T q.
// BWD = true: pass F of the backward.  Called with (q, k, v) = (dy, v, k) and
// S0^T, it carries S'_t = S_t^T and its output is dq_t = S_t dy_t.  It also
// writes, per step s, the sum over t >= s in the tile of
//   z_t = w_in_t q_t^T S_{c-1} dy_t
// (the term of dL/dlog(gamma_s) that pairs the incoming state with the tile's
// outputs), and stores S'_{c-1} as bf16 for every tile without a begin flag,
// for pass R.
template <int D, bool BWD, bool NORM = false, bool HALF_OUT = false, bool FOLD = false>
__global__ void __launch_bounds__(kThreads, 1) fwd_kernel(const __grid_constant__ FwdParams p) {
    // FOLD (pass F of the normalised backward): column p.fold_col of the output is
    // added to every output column (see the epilogue); compiled out elsewhere
    static_assert(!FOLD || BWD, "the fold is pass F's");
    static_assert(!NORM || (D == 128 && (!BWD || HALF_OUT)), "the normalised operands run the d = 128 kernels");
    // HALF_OUT (pass F at d = 128): only the first 64 output columns are written,
    // to a [B, L, H, 64] output (the normalised path needs no more of dq')
    static_assert(!HALF_OUT || (D == 128 && BWD), "half-width output for pass F at d = 128");
    using S = FwdSmem<D>;
    // NORM without BWD: the forward of the Linear Transformer with phi and its
    // normalizer for heads of 64 channels.  q, k, v are the unpadded [B, L, H, 64] tensors; each operand
    // slot holds them in its first 64 channels (one TMA box), phi is applied to
    // q and k in shared memory, the contractions over the q/k channels stop at
    // 64, the second half of the K slot holds zeros and that of the V slot the
    // columns [1, 1, 0, ...], so the 128-wide state is [[X, x, x], [0]] and
    // column 64 of the output is the normalizer; the epilogue writes
    // y = y'[:64] / y'[64] and the normalizer.
    // NORM with BWD: pass F of the normalised backward for 64-channel heads, on
    // (dy', v', k'') with dy' padded by the caller and v' = [v, 1, 1, 0],
    // k'' = [psi(k), 1, 1, 0] (psi = phi - 1) built in the K and V slots the same
    // way, and q'' = [phi(q), sigma_hi, sigma_lo, 0] for the z term (phi applied
    // as the tile is read, sigma = sum of phi(q) formed by the upper half of the
    // threads).  The output rows are staged in the K slot, whose constant half is
    // written again once they drain.  Column 64 of the output (the gradient of
    // the sum channel) is added to the other columns (fold_col).
    constexpr bool NF = NORM && !BWD, NB = NORM && BWD;
    constexpr int KQ = NF ? 64 : D;          // channels of the first contractions
    constexpr int BQ = NF ? 64 : D;          // channels loaded into the Q slot
    constexpr int BKV = NORM ? 64 : D;       // channels loaded into the K and V slots
    constexpr int DOUT = (NORM || HALF_OUT) ? 64 : D;  // output channels written
    constexpr int Y_OFF = NF ? 0 : S::OFF_Y;  // output staging: the Q slot (NF) or the K and V slots
    extern __shared__ __align__(1024) unsigned char smem[];
    grid_dependency_wait();  // the kernel before this one on the stream (metadata, carries)
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int quarter = warp & 3, half = warp >> 2;
    const int64_t bh = blockIdx.x / p.G;
    const int g = static_cast<int>(blockIdx.x % p.G);
    const int64_t b = bh / p.H, h = bh % p.H;
    // this segment: tiles [tile0, tile0 + nt), steps up to seg_hi (the tape end for the last)
    const int64_t tile0 = static_cast<int64_t>(g) * p.tps;
    const int nt = static_cast<int>(min(p.tps, p.n_tiles - tile0));
    const int64_t seg_hi = min(p.L, (tile0 + nt) * T);
    // the state entering the segment: S0 for the first, else the carry
    const float* s_in = g == 0 ? (p.S0 != nullptr ? p.S0 + bh * D * D : nullptr)
                               : p.carry + (bh * p.G + g - 1) * D * D;

    uint64_t* bar1 = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);
    uint64_t* bar2 = bar1 + 1;
    uint64_t* full = bar1 + 2;  // [2]: stage s loaded
    uint32_t* tslot = reinterpret_cast<uint32_t*>(bar1 + 4);
    uint64_t* qbar = bar1 + 5;  // pass F: the q tile of the z term
    TileMeta* metas = reinterpret_cast<TileMeta*>(smem + S::OFF_META);
    const uint32_t sbase = smem_addr(smem);
    const uint32_t sSb = sbase + S::OFF_SB;
    const TileMeta* gmeta = p.meta + bh * p.n_tiles + tile0;

    auto stage_q = [&](int s) { return sbase + s * S::STAGE; };
    auto stage_k = [&](int s) { return sbase + s * S::STAGE + S::TILE; };
    auto stage_v = [&](int s) { return sbase + s * S::STAGE + 2 * S::TILE; };
    const uint32_t sPm = sbase + S::OFF_PM;
    // thread 0: TMA loads of tile c into stage s and of metadata tiles m0 (and
    // m1 >= 0) into their ring slots, all completing on full[s]
    auto issue_tile = [&](int c, int s, int m0, int m1) {
        const uint32_t meta_bytes = (m0 >= 0 ? sizeof(TileMeta) : 0) + (m1 >= 0 ? sizeof(TileMeta) : 0);
        mbar_arrive_expect_tx(&full[s], T * BQ * 2 + 2 * (T * BKV * 2) + meta_bytes);
        const int64_t t0 = (tile0 + c) * T;
        tma_tile<BQ>(stage_q(s), &p.map_q, h, t0, b, &full[s]);
        tma_tile<BKV>(stage_k(s), &p.map_k, h, t0, b, &full[s]);
        tma_tile<BKV>(stage_v(s), &p.map_v, h, t0, b, &full[s]);
        if (m0 >= 0) bulk_g2s(&metas[m0 % S::NMETA], gmeta + m0, sizeof(TileMeta), &full[s]);
        if (m1 >= 0) bulk_g2s(&metas[m1 % S::NMETA], gmeta + m1, sizeof(TileMeta), &full[s]);
    };

    if (tid == 0) {
        mbar_init(bar1, 1);
        mbar_init(bar2, 1);
        mbar_init(&full[0], 1);
        mbar_init(&full[1], 1);
        mbar_init(qbar, 1);
        fence_mbar_init();
        prefetch_tensormap(&p.map_q);
        prefetch_tensormap(&p.map_k);
        prefetch_tensormap(&p.map_v);
        prefetch_tensormap(&p.map_y);
        if (BWD) prefetch_tensormap(&p.map_zq);
    }
    if (warp == 0) tc::alloc(tslot, S::TMEM_COLS);
    if (NORM) {
        // the constant second halves of the K and V slots of both stages (the forward:
        // zeros for k, [1, 1, 0, ...] for v; pass F: the v' constants in the K slot,
        // zeros for k in the V slot); the loads only ever write the first halves
        for (int st = 0; st < 2; ++st) {
            const_box<kThreads>(smem + st * S::STAGE + S::TILE, tid, NB);
            const_box<kThreads>(smem + st * S::STAGE + 2 * S::TILE, tid, true);
        }
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (tid == 0) issue_tile(0, 0, 0, nt > 1 ? 1 : -1);
    const bool first_ok = wait_mbar(&full[0], 0, p.wait_ns);
    const uint32_t tm = *tslot;

    const int srow = state_row<D>(quarter, lane);
    constexpr int SC = D / 2;  // state and output columns per thread
    const uint32_t lane_base = tm + (static_cast<uint32_t>(32 * quarter) << 16);

    // 16 values of row `row` of the bf16 state operand.  The normalised backward
    // keeps column fold_col + 1 (a copy of column fold_col: both key channels are 1)
    // as the bf16 rounding remainder of column fold_col instead, so the two
    // inter-tile output columns sum to the sum channel's value to about 16 bits.
    auto sb_store16 = [&](int row, int j0, const float* v) {
        if (FOLD && p.fold_col >= j0 && p.fold_col + 1 < j0 + 16) {
            const int f = p.fold_col - j0;
            float vf = 0.f;
#pragma unroll
            for (int x = 0; x < 16; ++x)
                if (x == f) vf = v[x];
            const float rem = vf - __bfloat162float(__float2bfloat16_rn(vf));
            float w[16];
#pragma unroll
            for (int x = 0; x < 16; ++x) w[x] = x == f + 1 ? rem : v[x];
            store_bf16x16(smem + S::OFF_SB, core_off(row, j0, D), core_off(row, j0 + 8, D), w);
        } else {
            store_bf16x16(smem + S::OFF_SB, core_off(row, j0, D), core_off(row, j0 + 8, D), v);
        }
    };

    // ---- incoming state (unless the segment's first step begins an episode) ----
    bool have_prev = false, have_state = false;
    if (s_in != nullptr && metas[0].first_start != 0) {
        have_prev = true;
        const bool scale = metas[0].has_start == 0;
        have_state = scale;
        const float a0 = metas[0].a;
        const float* s0 = s_in;
#pragma unroll 1
        for (int cc = 0; cc < SC / 16; ++cc) {
            const int j0 = half * SC + cc * 16;
            float v[16];
            if (srow >= 0) {
                if (BWD) {
#pragma unroll
                    for (int x = 0; x < 16; ++x) v[x] = s0[(j0 + x) * D + srow];
                } else {
#pragma unroll
                    for (int x = 0; x < 16; x += 4) {
                        const float4 f = *reinterpret_cast<const float4*>(s0 + srow * D + j0 + x);
                        v[x] = f.x;
                        v[x + 1] = f.y;
                        v[x + 2] = f.z;
                        v[x + 3] = f.w;
                    }
                }
                sb_store16(srow, j0, v);
                if (BWD && metas[0].has_start == 0)
                    store_state_row<D>(state_image<D>(p.states, bh, p.n_tiles, tile0), srow, j0, v);
            } else {
#pragma unroll
                for (int x = 0; x < 16; ++x) v[x] = 0.f;
            }
            if (scale) {
#pragma unroll
                for (int x = 0; x < 16; ++x) v[x] *= a0;
                tc::st16(lane_base + S::COL_S + j0, v);
            }
        }
    }

    if (BWD && !have_prev && metas[0].has_start == 0 && srow >= 0) {
        // the zero state before the tape's first tile (no S0)
        float zero[16];
#pragma unroll
        for (int x = 0; x < 16; ++x) zero[x] = 0.f;
        for (int j0 = half * SC; j0 < half * SC + SC; j0 += 16)
            store_state_row<D>(state_image<D>(p.states, bh, p.n_tiles, tile0), srow, j0, zero);
    }

    constexpr uint32_t ID_QS = tc::idesc_bf16(128, D, false, true);
    constexpr uint32_t ID_QK = tc::idesc_bf16(128, T, false, false);
    constexpr uint32_t ID_PV = tc::idesc_bf16(128, D, false, true);
    constexpr uint32_t ID_KV = tc::idesc_bf16(D, D, true, true);

    bool failed = __syncthreads_or(!first_ok);
    int pending = 0;       // the last issued tile whose load may still be in flight (-1: none)
    int drain_bar = 0;     // 1 / 2: the batch on bar1 / bar2 was issued but not seen complete
    uint32_t drain_par = 0;
    bool q_pending = false;  // pass F: a q tile load not seen complete
    uint32_t q_par = 0;
#pragma unroll 1
    for (int c = 0; c < nt && !failed; ++c) {
        const int s = c & 1;
        const TileMeta& mc = metas[c % S::NMETA];
        // tile c's loads (issued during the previous tile) are complete
        bool ok = wait_mbar(&full[s], (c >> 1) & 1, p.wait_ns);
        tc::fence_smem_to_async();
        tc::fence_before();
        if (__syncthreads_or(!ok)) {
            failed = true;
            break;
        }
        pending = -1;
        tc::fence_after();
        if (NORM) {
            // phi on the loaded q and k (the forward) or k (pass F), in place
            const int64_t valid = p.L - (tile0 + c) * T;
            if (NF) {
                phi_box<kThreads>(smem + s * S::STAGE, tid, valid);
                phi_box<kThreads>(smem + s * S::STAGE + S::TILE, tid, valid);
            } else {
                psi_box<kThreads>(smem + s * S::STAGE + 2 * S::TILE, tid, valid);
            }
            tc::fence_smem_to_async();
            tc::fence_before();
            __syncthreads();
            tc::fence_after();
        }

        // ---- P = Q K^T and (with an incoming state) Y_inter = Q S_prev ----
        if (tid == 0) {
            const uint32_t sq = stage_q(s), sk = stage_k(s);
            if (have_prev) {
#pragma unroll
                for (int kk = 0; kk < KQ / 16; ++kk)
                    tc::mma(tm + S::COL_YI, desc_sw_k(sq, kk), desc_mnmajor(sSb, D, kk), ID_QS, kk > 0);
            }
#pragma unroll
            for (int kk = 0; kk < KQ / 16; ++kk)
                tc::mma(tm + S::COL_P, desc_sw_k(sq, kk), desc_sw_k(sk, kk), ID_QK, kk > 0);
            tc::commit(bar1);
        }
        ok = wait_mbar(bar1, c & 1, p.wait_ns) && !(c == 0 && static_cast<int64_t>(blockIdx.x) == p.fail_cta);
        if (__syncthreads_or(!ok)) {
            failed = true;
            drain_bar = 1;
            drain_par = c & 1;
            break;
        }
        tc::fence_after();
        // pass F: the Q slot (dy) is free once the first contractions are done; the
        // q tile of the z term goes there
        const bool zload = BWD && have_prev;
        // the normalised backward also reads q in the epilogue: dq = dphi(q) (.) phi'(q)
        const bool qload = zload || NB;
        if (qload) {
            if (tid == 0) {
                mbar_arrive_expect_tx(qbar, T * BKV * 2);
                tma_tile<BKV>(stage_q(s), &p.map_zq, h, (tile0 + c) * T, b, qbar);
            }
            q_pending = true;
        }

        // ---- mask: Pm[t][r] = [seg_t <= r <= t] exp2(lam2_t - lam2_r) P[t][r] ----
        {
            const int t = 32 * quarter + lane;
            const float lt = mc.lam2[t];
            const int st = mc.seg[t];
            unsigned char* pm = smem + S::OFF_PM;
            uint32_t raw[64];
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) tc::ld16_nowait(lane_base + S::COL_P + half * 64 + cc * 16, raw + cc * 16);
            tc::ld_wait();
            float rs = 0.f;  // the normalised backward: fp32 row sum of the masked scores (this half)
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
                const int r0 = half * 64 + cc * 16;
                float v[16];
#pragma unroll
                for (int x = 0; x < 16; ++x) {
                    const int r = r0 + x;
                    const bool in = r <= t && r >= st;
                    v[x] = in ? __uint_as_float(raw[cc * 16 + x]) * fast_exp2(lt - mc.lam2[r]) : 0.f;
                    if (FOLD) rs += v[x];
                }
                store_bf16x16(pm, core_off(t, r0, T), core_off(t, r0 + 8, T), v);
            }
            // read at the start of the epilogue, before the z terms take the same slots
            if (FOLD) reinterpret_cast<float*>(smem + S::OFF_Z)[half * T + t] = rs;
        }
        // ---- K~[r] = exp2(lam2_end - lam2_r) K[r] for rows of the last episode ----
        {
            const float lend = mc.lam2[T - 1];
            const int ls = mc.last_start;
            scale_rows_sw<D, kThreads, !BWD>(smem + (stage_k(s) - sbase), tid,
                             [&](int r) { return r >= ls ? fast_exp2(lend - mc.lam2[r]) : 0.f; });
        }
        // the previous tile's output stores, which read stage s ^ 1, have drained
        // behind this tile's first contractions and mask pass
        if (warp == 0) bulk_wait_read();
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        tc::fence_after();
        // pass F (normalised): the output rows were staged over the v' constants of stage s ^ 1
        if (NB) const_box<kThreads>(smem + (s ^ 1) * S::STAGE + S::TILE, tid, true);
        // the next tile's loads into stage s ^ 1
        if (c + 1 < nt) {
            if (tid == 32) issue_tile(c + 1, s ^ 1, c + 2 < nt ? c + 2 : -1, -1);
            pending = c + 1;
        }

        // ---- Y_intra = Pm V and S = a S + K~^T V ----
        if (tid == 0) {
            const uint32_t spm = sPm, sk = stage_k(s), sv = stage_v(s);
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_YA, desc_kmajor(spm, T, kk), desc_sw_mn(sv, kk), ID_PV, kk > 0);
            const bool acc = have_state && mc.has_start == 0;
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_S, desc_sw_mn(sk, kk), desc_sw_mn(sv, kk), ID_KV, acc || kk > 0);
            tc::commit(bar2);
        }
        const int64_t t0 = (tile0 + c) * T;
        ok = wait_mbar(bar2, c & 1, p.wait_ns);
        if (__syncthreads_or(!ok)) {
            failed = true;
            drain_bar = 2;
            drain_par = c & 1;
            break;
        }
        tc::fence_after();
        if (qload) {
            ok = wait_mbar(qbar, q_par, p.wait_ns);
            if (__syncthreads_or(!ok)) {
                failed = true;
                break;
            }
            q_pending = false;
            q_par ^= 1;
        }

        // ---- y = Y_intra + w_in * Y_inter, staged as fp32 rows in stage s ----
        // rows of this tile inside the tape
        const int r_hi = static_cast<int>(min(static_cast<int64_t>(T), seg_hi - t0));
        if (NF) {
            // y = y'[:64] / y'[64]: every thread reads the normalizer (column 64) of
            // its row and divides its 32 of the 64 output columns
            const int t = 32 * quarter + lane;
            const float w_in = (have_prev && mc.seg[t] < 0) ? fast_exp2(mc.lam2[t]) : 0.f;
            const int j0 = half * 32;
            uint32_t ya[32], yi[32], na[16], ni[16];
            tc::ld16_nowait(lane_base + S::COL_YA + 64, na);
            tc::ld16_nowait(lane_base + S::COL_YA + j0, ya);
            tc::ld16_nowait(lane_base + S::COL_YA + j0 + 16, ya + 16);
            if (have_prev) {
                tc::ld16_nowait(lane_base + S::COL_YI + 64, ni);
                tc::ld16_nowait(lane_base + S::COL_YI + j0, yi);
                tc::ld16_nowait(lane_base + S::COL_YI + j0 + 16, yi + 16);
            }
            tc::ld_wait();
            // rows whose episode began in this tile take no inter-tile term (a select:
            // a non-finite incoming state does not cross the begin flag)
            const bool inter = w_in != 0.f;
            const float dn = have_prev && inter ? fmaf(w_in, __uint_as_float(ni[0]), __uint_as_float(na[0]))
                                                : __uint_as_float(na[0]);
            if (half == 0 && p.den != nullptr && t < r_hi) p.den[(b * p.L + t0 + t) * p.H + h] = dn;
            const float inv = 1.f / dn;
            unsigned char* yst = smem + s * S::STAGE + Y_OFF + t * 128;  // row t of chunk 0
#pragma unroll
            for (int x = 0; x < 32; x += 4) {
                float o[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    o[e] = __uint_as_float(ya[x + e]);
                    if (have_prev) o[e] = inter ? fmaf(w_in, __uint_as_float(yi[x + e]), o[e]) : o[e];
                    o[e] *= inv;
                }
                const int j = j0 + x;
                *reinterpret_cast<float4*>(yst + (j >> 5) * (T * 128) + ((((j & 31) >> 2) ^ (t & 7)) << 4)) =
                    make_float4(o[0], o[1], o[2], o[3]);
            }
        } else {
            const int t = 32 * quarter + lane;
            const float w_in = (have_prev && mc.seg[t] < 0) ? fast_exp2(mc.lam2[t]) : 0.f;
            unsigned char* yst = smem + s * S::STAGE + Y_OFF + t * 128;  // row t of chunk 0
            const unsigned char* qs = smem + (stage_q(s) - sbase);  // pass F: the q tile
            const bool zrow = zload && w_in != 0.f;
            // HALF_OUT: the upper half of the threads writes no output, only its part of z
            const bool out_half = !(HALF_OUT && half == 1);
            // q' of the z term: the loaded values, or (normalised) phi of them rounded to bf16
            auto qpair = [](uint32_t w) {
                float2 f = unpack_bf16x2(w);
                if (NB) f = unpack_bf16x2(pack_bf16x2(f.x > 0.f ? 1.f + f.x : __expf(f.x), f.y > 0.f ? 1.f + f.y : __expf(f.y)));
                return f;
            };
            // the normalised backward: the output column of the sum channel, added to every
            // column.  Its intra-tile part is the row sum of the masked scores (the key
            // operand is 1 in that channel), taken in fp32 from the unrounded scores: that
            // sum cancels strongly, and the bf16 scores of the contraction would add their
            // rounding to it; the inter-tile part comes from the contraction.
            float ofold = 0.f;
            if (FOLD) {
                const float* rsp = reinterpret_cast<const float*>(smem + S::OFF_Z);
                const float rsum = rsp[t] + rsp[T + t];
                float vi = 0.f;  // the inter-tile part: the two columns (value and remainder)
                if (have_prev) {
                    const int fb = p.fold_col & ~15, fx = p.fold_col & 15;
                    float fi[16];
                    tc::ld16(lane_base + S::COL_YI + fb, fi);
                    float v0 = 0.f, v1 = 0.f;
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        if (e == fx) v0 = fi[e];
                        if (e == fx + 1) v1 = fi[e];
                    }
                    vi = v0 + v1;
                }
                ofold = (have_prev && w_in != 0.f) ? fmaf(w_in, vi, rsum) : rsum;
                __syncthreads();  // every row sum is read before the z terms overwrite the slots
            }
            // BWD: z_t = w_in_t q_t . (S_{c-1} dy_t), the inter output dotted with q
            float zacc = 0.f, zfold = 0.f;
#pragma unroll
            for (int cc = 0; cc < SC / 32; ++cc) {
                const int j0 = half * SC + cc * 32;
                uint32_t ya[32], yi[32];
                if (out_half) {
                    tc::ld16_nowait(lane_base + S::COL_YA + j0, ya);
                    tc::ld16_nowait(lane_base + S::COL_YA + j0 + 16, ya + 16);
                }
                if (have_prev) {
                    tc::ld16_nowait(lane_base + S::COL_YI + j0, yi);
                    tc::ld16_nowait(lane_base + S::COL_YI + j0 + 16, yi + 16);
                }
                tc::ld_wait();
                if (out_half) {
#pragma unroll
                    for (int x = 0; x < 32; x += 4) {
                        float4 o = make_float4(__uint_as_float(ya[x]), __uint_as_float(ya[x + 1]),
                                               __uint_as_float(ya[x + 2]), __uint_as_float(ya[x + 3]));
                        if (have_prev) {  // the forward: a select where w_in = 0, as above
                            const bool in2 = BWD || w_in != 0.f;
                            o.x = in2 ? fmaf(w_in, __uint_as_float(yi[x]), o.x) : o.x;
                            o.y = in2 ? fmaf(w_in, __uint_as_float(yi[x + 1]), o.y) : o.y;
                            o.z = in2 ? fmaf(w_in, __uint_as_float(yi[x + 2]), o.z) : o.z;
                            o.w = in2 ? fmaf(w_in, __uint_as_float(yi[x + 3]), o.w) : o.w;
                        }
                        if (FOLD) {
                            o.x += ofold;
                            o.y += ofold;
                            o.z += ofold;
                            o.w += ofold;
                        }
                        const int j = j0 + x;  // 4 channels = one 16-byte unit
                        *reinterpret_cast<float4*>(yst + (j >> 5) * (T * 128) + ((((j & 31) >> 2) ^ (t & 7)) << 4)) = o;
                    }
                }
                if (zrow && NB && half == 1) {
                    // q'' channels 64 and 65: sigma as a bf16 pair (the rest of the upper half is 0)
                    if (cc == 0) {
                        float su[8];
#pragma unroll
                        for (int u = 0; u < 8; ++u) {
                            const uint4 w = *reinterpret_cast<const uint4*>(qs + sw_off(t, 8 * u));
                            const float2 a = qpair(w.x), b2 = qpair(w.y), c2 = qpair(w.z), d2 = qpair(w.w);
                            float acc = 0.f;
                            acc += a.x;
                            acc += a.y;
                            acc += b2.x;
                            acc += b2.y;
                            acc += c2.x;
                            acc += c2.y;
                            acc += d2.x;
                            acc += d2.y;
                            su[u] = acc;
                        }
                        const float sg = ((su[0] + su[1]) + (su[2] + su[3])) + ((su[4] + su[5]) + (su[6] + su[7]));
                        const float hi = __bfloat162float(__float2bfloat16_rn(sg));
                        const float lo = __bfloat162float(__float2bfloat16_rn(sg - hi));
                        // the sum channel pair: (sigma_hi + sigma_lo) times (value + remainder)
                        zacc = fmaf(hi + lo, __uint_as_float(yi[0]) + __uint_as_float(yi[1]), zacc);
                    }
                } else if (zrow) {
#pragma unroll
                    for (int x = 0; x < 32; x += 8) {
                        const uint4 u = *reinterpret_cast<const uint4*>(qs + sw_off(t, j0 + x));
                        float2 q0 = qpair(u.x), q1 = qpair(u.y), q2 = qpair(u.z), q3 = qpair(u.w);
                        if (FOLD && p.fold_col >= j0 + x && p.fold_col < j0 + x + 8) {
                            // the sum channel pair (value, remainder columns) is taken below
                            const int f = p.fold_col - (j0 + x);  // 0 or 2, 4, 6 (even)
                            const float qs0 = f == 0 ? q0.x : (f == 2 ? q1.x : (f == 4 ? q2.x : q3.x));
                            const float qs1 = f == 0 ? q0.y : (f == 2 ? q1.y : (f == 4 ? q2.y : q3.y));
                            const float ys0 = __uint_as_float(yi[x + f]), ys1 = __uint_as_float(yi[x + f + 1]);
                            zfold = fmaf(qs0 + qs1, ys0 + ys1, 0.f);
                            if (f == 0) q0 = make_float2(0.f, 0.f);
                            if (f == 2) q1 = make_float2(0.f, 0.f);
                            if (f == 4) q2 = make_float2(0.f, 0.f);
                            if (f == 6) q3 = make_float2(0.f, 0.f);
                        }
                        zacc = fmaf(q0.x, __uint_as_float(yi[x]), zacc);
                        zacc = fmaf(q0.y, __uint_as_float(yi[x + 1]), zacc);
                        zacc = fmaf(q1.x, __uint_as_float(yi[x + 2]), zacc);
                        zacc = fmaf(q1.y, __uint_as_float(yi[x + 3]), zacc);
                        zacc = fmaf(q2.x, __uint_as_float(yi[x + 4]), zacc);
                        zacc = fmaf(q2.y, __uint_as_float(yi[x + 5]), zacc);
                        zacc = fmaf(q3.x, __uint_as_float(yi[x + 6]), zacc);
                        zacc = fmaf(q3.y, __uint_as_float(yi[x + 7]), zacc);
                    }
                }
            }
            if (FOLD) zacc += zfold;
            if (BWD) reinterpret_cast<float*>(smem + S::OFF_Z)[half * T + t] = w_in * zacc;
        }
        if (NB) {
            // dq = dphi(q) (.) phi'(q) on the staged rows, from the raw q tile: two
            // threads per row, one 32-channel chunk each
            __syncthreads();
            const int r = tid >> 1, m = tid & 1;
            unsigned char* row = smem + s * S::STAGE + Y_OFF + m * (T * 128) + r * 128;
            const unsigned char* qs = smem + (stage_q(s) - sbase);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                float4* o = reinterpret_cast<float4*>(row + ((u ^ (r & 7)) << 4));
                *o = times_phi_prime(*o, *reinterpret_cast<const uint2*>(qs + sw_off(r, 32 * m + 4 * u)));
            }
        }
        if (BWD) __syncthreads();  // every z term has read the q tile, where the state is staged next
        // ---- state: bf16 copy for the next tile, decay by the next tile's a ----
        if (c + 1 < nt) {
            const TileMeta& mn = metas[(c + 1) % S::NMETA];
            const bool scale = mn.has_start == 0 && mn.a != 1.f;
            const float an = mn.a;
#pragma unroll
            for (int cc = 0; cc < SC / 32; ++cc) {
                const int j0 = half * SC + cc * 32;
                uint32_t raw[32];
                tc::ld16_nowait(lane_base + S::COL_S + j0, raw);
                tc::ld16_nowait(lane_base + S::COL_S + j0 + 16, raw + 16);
                tc::ld_wait();
                float v[32];
#pragma unroll
                for (int x = 0; x < 32; ++x) v[x] = __uint_as_float(raw[x]);
                if (srow >= 0) {
                    sb_store16(srow, j0, v);
                    sb_store16(srow, j0 + 16, v + 16);
                    if (BWD && mn.has_start == 0) {
                        // staged in this stage's Q slot (the z term has read q) and
                        // bulk-stored with the output rows
                        unsigned char* img = smem + (stage_q(s) - sbase);
                        store_state_row<D>(img, srow, j0, v);
                        store_state_row<D>(img, srow, j0 + 16, v + 16);
                    }
                }
                if (scale) {
#pragma unroll
                    for (int x = 0; x < 32; ++x) v[x] *= an;
                    tc::st16(lane_base + S::COL_S + j0, v);
                    tc::st16(lane_base + S::COL_S + j0 + 16, v + 16);
                }
            }
        } else if (seg_hi == p.L && p.S_last != nullptr) {
            float* dst = p.S_last + bh * D * D;
#pragma unroll
            for (int cc = 0; cc < SC / 16; ++cc) {
                const int j0 = half * SC + cc * 16;
                float v[16];
                tc::ld16(lane_base + S::COL_S + j0, v);
                if (srow >= 0) {
#pragma unroll
                    for (int x = 0; x < 16; x += 4)
                        *reinterpret_cast<float4*>(dst + srow * D + j0 + x) = make_float4(v[x], v[x + 1], v[x + 2], v[x + 3]);
                }
            }
        }
        // ---- bulk-store the staged output rows ----
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        if (warp == 0) {
            // one TMA store per 32 channels (rows past L are clipped)
            if (lane == 0) {
#pragma unroll
                for (int m = 0; m < DOUT / 32; ++m)
                    tma_store_4d(&p.map_y, sbase + s * S::STAGE + Y_OFF + m * T * 128, 32 * m, static_cast<int>(h),
                                 static_cast<int>(t0), static_cast<int>(b));
            }
            if (BWD && lane == 0 && c + 1 < nt && metas[(c + 1) % S::NMETA].has_start == 0)
                bulk_s2g(state_image<D>(p.states, bh, p.n_tiles, tile0 + c + 1), stage_q(s), D * D * 2);
            bulk_commit();
        }
        if (BWD && warp == 1) {
            // suffix sums of z over the tile: dlam_f[t] = sum_{s >= t} z_s
            const float* zst = reinterpret_cast<const float*>(smem + S::OFF_Z);
            float zv[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) zv[x] = zst[4 * lane + x] + zst[T + 4 * lane + x];
#pragma unroll
            for (int x = 2; x >= 0; --x) zv[x] += zv[x + 1];
            float tot = zv[0];
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const float o = __shfl_down_sync(0xffffffffu, tot, off);
                if (lane + off < 32) tot += o;
            }
            float after = __shfl_down_sync(0xffffffffu, tot, 1);
            if (lane == 31) after = 0.f;
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                const int r = 4 * lane + x;
                if (r < r_hi) p.dlam_f[(b * p.L + t0 + r) * p.H + h] = zv[x] + after;
            }
        }
        have_prev = true;
        have_state = true;
    }
    if (failed) {
        if (tid == 0) record_error(p.hdr, DEV_MMA_TIMEOUT);
        // let work still in flight finish before the CTA's TMEM and shared memory go away
        if (drain_bar == 1) wait_mbar(bar1, drain_par, kDrainNs);
        if (drain_bar == 2) wait_mbar(bar2, drain_par, kDrainNs);
        if (pending >= 0) wait_mbar(&full[pending & 1], (pending >> 1) & 1, kDrainNs);
        if (q_pending) wait_mbar(qbar, q_par, kDrainNs);
    }
    if (warp == 0) bulk_wait_all();
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 0) tc::dealloc(tm, S::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// segment summaries and the carry between segments
// ---------------------------------------------------------------------------
// REV = false (the forward's "tail" summary, for segments g < G - 1): the state
// that the segment's rows after its last begin flag (all its rows if it has
// none) leave at its end from a zero start,
//   X_g = sum_r exp2(Lam_end - Lam_r) k_r v_r^T,
// REV = true (the backward's "head" summary, for segments g >= 1): the reverse
// state that the rows before its first begin flag pass to the segment before,
//   X_g = sum_s exp2(Lam_s - Lam_begin) q_s dy_s^T,
// with Lam the running sum of log2(gamma) over the segment.  Also per segment:
// info[g] = (1 if it holds a begin flag, log2 of its total decay).  Both are
// dense bf16 contractions K~^T V (or Q~^T dY) over the segment's tiles with
// fp32 accumulation in TMEM.  gamma <= 1, so the weights only shrink away from
// the segment's end (start); tiles whose weights all underflow to 0 are not
// read.
template <int D>
struct SegSmem {
    static constexpr int TILE = T * D * 2;
    static constexpr int NST = 3;  // stages: tile i computes while i + 1 and i + 2 load
    static constexpr int STAGE = 2 * TILE;  // X (k or q), Y (v or dy)
    static constexpr int OFF_META = NST * STAGE;
    static constexpr int OFF_RED = OFF_META + NST * static_cast<int>(sizeof(TileMeta));  // [256] floats + [256] ints
    static constexpr int OFF_BAR = OFF_RED + 256 * 8 + 64;
    static constexpr int BYTES = OFF_BAR + 64;
};

struct SegParams {
    CUtensorMap map_x, map_y;  // forward: k, v; reverse: q, dy
    const TileMeta* meta;
    float2* info;  // [B * H * G]
    float* out;    // [B * H * G][D][D]
    uint32_t* hdr;
    int64_t L, H, n_tiles, tps;
    int G;
    uint64_t wait_ns;
};

// log2 weights below this underflow to 0 in fast_exp2 (flush-to-zero), so
// every row of a tile past this offset contributes exactly nothing
constexpr float kUnderflowLog2 = -152.f;

template <int D, bool REV, bool NORM = false, bool PSI = false>
__global__ void __launch_bounds__(kThreads, 1) seg_state_kernel(const __grid_constant__ SegParams p) {
    // NORM: the Linear Transformer with phi for 64-channel heads, operands built
    // in shared memory as the tensor-core kernels build them: forward X = k' =
    // [phi(k), 0] (the forward's basis) or, PSI (the backward's), k'' = [psi(k),
    // 1, 1, 0]; reverse X = q'' = [phi(q), sigma_hi, sigma_lo, 0]; the forward's
    // Y holds v and the columns [1, 1, 0, ...]; the reverse Y is the padded dy'
    static_assert(!NORM || D == 128, "the normalised operands run at d = 128");
    grid_dependency_wait();  // the metadata (and, in the backward, the kernels before)
    static_assert(!REV || !NORM || PSI, "the reverse summary runs in the backward's basis");
    using S = SegSmem<D>;
    constexpr int BX = NORM ? 64 : D;
    constexpr int BY = (NORM && !REV) ? 64 : D;
    extern __shared__ __align__(1024) unsigned char smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int quarter = warp & 3, half = warp >> 2;
    const int per_bh = p.G - 1;
    const int64_t bh = blockIdx.x / per_bh;
    const int g = static_cast<int>(blockIdx.x % per_bh) + (REV ? 1 : 0);
    const int64_t b = bh / p.H, h = bh % p.H;
    const int64_t c0 = static_cast<int64_t>(g) * p.tps, c1 = min(p.n_tiles, c0 + p.tps);
    const TileMeta* gm = p.meta + bh * p.n_tiles;

    uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);  // [NST]
    uint64_t* mbar = full + S::NST;                                   // [NST]: the contraction reading stage s is done
    uint32_t* tslot = reinterpret_cast<uint32_t*>(mbar + S::NST);
    float* red_f = reinterpret_cast<float*>(smem + S::OFF_RED);
    int* red_i = reinterpret_cast<int*>(smem + S::OFF_RED + 256 * 4);
    int* bcast = reinterpret_cast<int*>(smem + S::OFF_RED + 256 * 8);
    TileMeta* metas = reinterpret_cast<TileMeta*>(smem + S::OFF_META);
    const uint32_t sbase = smem_addr(smem);

    if (tid == 0) {
        for (int i = 0; i < S::NST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&mbar[i], 1);
        }
        fence_mbar_init();
        prefetch_tensormap(&p.map_x);
        prefetch_tensormap(&p.map_y);
    }
    if (warp == 0) tc::alloc(tslot, 128);
    if (NORM) {
        for (int st = 0; st < S::NST; ++st) {
            const_box<kThreads>(smem + st * S::STAGE, tid, PSI && !REV);
            if (!REV) const_box<kThreads>(smem + st * S::STAGE + S::TILE, tid, true);
        }
    }

    // ---- which tiles: a pass over the segment's metadata ----
    // Each thread takes a run of consecutive tiles: the sum of their log2
    // decays (in order) and the latest (forward) / earliest (reverse) tile
    // holding a begin flag.
    const int64_t n = c1 - c0;
    const int64_t per = (n + kThreads - 1) / kThreads;
    const int64_t a0 = c0 + tid * per, a1 = min(c1, a0 + per);
    float run = 0.f;
    int flag_tile = REV ? 0x7fffffff : -1;
    for (int64_t c = a0; c < a1; ++c) {
        run += gm[c].lam2[T - 1];
        if (gm[c].has_start != 0) flag_tile = REV ? min(flag_tile, static_cast<int>(c - c0)) : static_cast<int>(c - c0);
    }
    red_f[tid] = run;
    red_i[tid] = flag_tile;
    __syncthreads();
    if (warp == 0) {
        // exclusive prefix of the runs' sums in thread order (fixed order), and the flag tile
        float v[8];
        float sum8 = 0.f;
        int ft = REV ? 0x7fffffff : -1;
#pragma unroll
        for (int x = 0; x < 8; ++x) {
            v[x] = red_f[lane * 8 + x];
            sum8 += v[x];
            const int f = red_i[lane * 8 + x];
            ft = REV ? min(ft, f) : max(ft, f);
        }
        float incl = sum8;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float o = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += o;
            const int of = __shfl_xor_sync(0xffffffffu, ft, off);
            ft = REV ? min(ft, of) : max(ft, of);
        }
        float pre = incl - sum8;
#pragma unroll
        for (int x = 0; x < 8; ++x) {
            red_f[lane * 8 + x] = pre;  // sum of the runs before thread lane * 8 + x
            pre += v[x];
        }
        const float total = __shfl_sync(0xffffffffu, incl, 31);
        if (lane == 0) {
            bcast[0] = ft;
            bcast[1] = __float_as_int(total);
            const bool has_flag = REV ? ft != 0x7fffffff : ft >= 0;
            p.info[bh * p.G + g] = make_float2(has_flag ? 1.f : 0.f, total);
        }
    }
    __syncthreads();
    const int ft = bcast[0];
    const float total = __int_as_float(bcast[1]);
    // the farthest tile (from the end forward, from the start reverse) whose
    // offset is still above the underflow bound: offsets only decrease
    {
        const float before = red_f[tid];  // the sum over tiles c0 .. a0 - 1
        int far = REV ? -1 : 0x7fffffff;
        if (REV) {
            float off = before;  // sum over tiles c0 .. c - 1
            for (int64_t c = a0; c < a1; ++c) {
                if (off >= kUnderflowLog2) far = static_cast<int>(c - c0);
                off += gm[c].lam2[T - 1];
            }
        } else {
            float off = total - before;  // sum over tiles a0 .. c1 - 1, then c + 1 .. c1 - 1
            for (int64_t c = a0; c < a1; ++c) {
                off -= gm[c].lam2[T - 1];
                if (off >= kUnderflowLog2 && far == 0x7fffffff) far = static_cast<int>(c - c0);
            }
        }
        red_i[tid] = far;
    }
    __syncthreads();
    if (warp == 0) {
        int far = REV ? -1 : 0x7fffffff;
#pragma unroll
        for (int x = 0; x < 8; ++x) far = REV ? max(far, red_i[lane * 8 + x]) : min(far, red_i[lane * 8 + x]);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const int o = __shfl_xor_sync(0xffffffffu, far, off);
            far = REV ? max(far, o) : min(far, o);
        }
        if (lane == 0) bcast[2] = far;
    }
    __syncthreads();
    const int far = bcast[2];
    // tiles processed, in order: forward c1 - 1 down to c0 + lo, reverse c0 up to c0 + hi
    int n_proc;
    if (REV) {
        const int hi = min(ft == 0x7fffffff ? static_cast<int>(n) - 1 : ft, far);
        n_proc = hi + 1;
    } else {
        const int lo = max(ft < 0 ? 0 : ft, far);
        n_proc = static_cast<int>(n) - lo;
    }
    auto tile_of = [&](int i) -> int64_t { return REV ? c0 + i : c1 - 1 - i; };

    // thread 0: TMA loads of processed tile i into stage i % NST
    auto issue = [&](int i) {
        const int st = i % S::NST;
        mbar_arrive_expect_tx(&full[st], T * BX * 2 + T * BY * 2 + sizeof(TileMeta));
        const int64_t c = tile_of(i);
        tma_tile<BX>(sbase + st * S::STAGE, &p.map_x, h, c * T, b, &full[st]);
        tma_tile<BY>(sbase + st * S::STAGE + S::TILE, &p.map_y, h, c * T, b, &full[st]);
        bulk_g2s(&metas[st], gm + c, sizeof(TileMeta), &full[st]);
    };
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tm = *tslot;
    int issued = 0;  // thread 0: tiles whose loads were issued
    if (tid == 0) {
        for (; issued < S::NST - 1 && issued < n_proc; ++issued) issue(issued);
    }
    constexpr uint32_t ID_XY = tc::idesc_bf16(D, D, true, true);
    bool failed = false;
    float off = 0.f;  // log2 decay between the segment's end (start) and this tile
    int i = 0;
#pragma unroll 1
    for (; i < n_proc; ++i) {
        const int st = i % S::NST;
        bool issue_ok = true;
        if (tid == 0 && issued < n_proc) {
            // the stage of tile i + NST - 1 held tile i - 1: free once its contraction is done
            if (i >= 1) issue_ok = wait_mbar(&mbar[(i - 1) % S::NST], ((i - 1) / S::NST) & 1, p.wait_ns);
            if (issue_ok) issue(issued++);
        }
        const bool ok = wait_mbar(&full[st], (i / S::NST) & 1, p.wait_ns);
        if (__syncthreads_or(!ok || !issue_ok)) {
            failed = true;
            break;
        }
        const TileMeta& mc = metas[st];
        const int64_t t0 = tile_of(i) * T;
        if (NORM) {
            if (REV) {
                phiq_box<kThreads>(smem + st * S::STAGE, tid, p.L - t0);
            } else if (PSI) {
                psi_box<kThreads>(smem + st * S::STAGE, tid, p.L - t0);
                // the constant half [1, 1, 0, ...]: this stage's last tile scaled it in place
                const_box<kThreads>(smem + st * S::STAGE, tid, true);
            } else {
                phi_box<kThreads>(smem + st * S::STAGE, tid, p.L - t0);
            }
            __syncthreads();
        }
        // X~ = w (.) X in place
        if (REV) {
            scale_rows_sw<D>(smem + st * S::STAGE, tid,
                             [&](int r) { return mc.seg[r] < 0 ? fast_exp2(off + mc.lam2[r]) : 0.f; });
        } else {
            const float lend = mc.lam2[T - 1];
            const int ls = mc.last_start;
            scale_rows_sw<D, kThreads, true>(smem + st * S::STAGE, tid,
                                             [&](int r) { return r >= ls ? fast_exp2(off + lend - mc.lam2[r]) : 0.f; });
        }
        off += mc.lam2[T - 1];
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        tc::fence_after();
        if (tid == 0) {
            const uint32_t sx = sbase + st * S::STAGE, sy = sx + S::TILE;
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm, desc_sw_mn(sx, kk), desc_sw_mn(sy, kk), ID_XY, i > 0 || kk > 0);
            tc::commit(&mbar[st]);
        }
    }
    // the last contraction (and with it every earlier one) is done
    const bool ok = !failed && wait_mbar(&mbar[(n_proc - 1) % S::NST], ((n_proc - 1) / S::NST) & 1, p.wait_ns);
    if (!ok && tid == 0) {
        record_error(p.hdr, DEV_MMA_TIMEOUT);
        // drain every issued load and contraction before TMEM and shared memory go away
        for (int j = i; j < issued; ++j) wait_mbar(&full[j % S::NST], (j / S::NST) & 1, kDrainNs);
        if (i >= 1) wait_mbar(&mbar[(i - 1) % S::NST], ((i - 1) / S::NST) & 1, kDrainNs);
    }
    __syncthreads();
    tc::fence_after();
    if (ok) {
        const int srow = state_row<D>(quarter, lane);
        const uint32_t lane_base = tm + (static_cast<uint32_t>(32 * quarter) << 16);
        float* dst = p.out + (bh * p.G + g) * D * D;
        constexpr int SC = D / 2;
#pragma unroll 1
        for (int cc = 0; cc < SC / 16; ++cc) {
            const int j0 = half * SC + cc * 16;
            float v[16];
            tc::ld16(lane_base + j0, v);
            if (srow >= 0) {
#pragma unroll
                for (int x = 0; x < 16; x += 4)
                    *reinterpret_cast<float4*>(dst + srow * D + j0 + x) = make_float4(v[x], v[x + 1], v[x + 2], v[x + 3]);
            }
        }
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 0) tc::dealloc(tm, 128);
}

// The resettable scan over the segments, in place (one thread per 4 state
// entries, segments in order):
//   forward: E_0 = S0 (or 0);  buf[g] <- [no flag in g] a_g E_g + X_g = E_{g+1}
//   reverse: R_{G-1} = dS_last (or 0);  buf[g] <- [no flag in g] a_g R_g + X_g = R_{g-1}
// with a_g = exp2(info[g].y) the segment's total decay; the flag selects, as
// in Theorem 3.2, so nothing from before a begin flag (NaN included) crosses it.
template <bool REV>
__global__ void __launch_bounds__(256) seg_carry_kernel(float* __restrict__ buf, const float2* __restrict__ info,
                                                       const float* __restrict__ init, int G, int DD) {
    grid_dependency_wait();  // the segment summaries
    const int64_t bh = blockIdx.y;
    const int e = (blockIdx.x * 256 + threadIdx.x) * 4;
    if (e >= DD) return;
    float* base = buf + bh * G * DD + e;
    const float2* inf = info + bh * G;
    float4 c = init != nullptr ? *reinterpret_cast<const float4*>(init + bh * DD + e) : make_float4(0.f, 0.f, 0.f, 0.f);
    // the segments' loads go out a batch at a time (the in-place stores would
    // otherwise hold every load back until the previous segment is folded)
    constexpr int NB = 8;
    for (int k0 = 0; k0 < G - 1; k0 += NB) {
        float4 x[NB];
        float2 f[NB];
#pragma unroll
        for (int j = 0; j < NB; ++j) {
            const int k = k0 + j;
            if (k < G - 1) {
                const int g = REV ? G - 1 - k : k;
                f[j] = inf[g];
                x[j] = *reinterpret_cast<const float4*>(base + static_cast<int64_t>(g) * DD);
            }
        }
#pragma unroll
        for (int j = 0; j < NB; ++j) {
            const int k = k0 + j;
            if (k < G - 1) {
                const int g = REV ? G - 1 - k : k;
                if (f[j].x != 0.f) {
                    c = x[j];
                } else {
                    const float a = exp2f(f[j].y);
                    c = make_float4(fmaf(a, c.x, x[j].x), fmaf(a, c.y, x[j].y), fmaf(a, c.z, x[j].z),
                                    fmaf(a, c.w, x[j].w));
                }
                *reinterpret_cast<float4*>(base + static_cast<int64_t>(g) * DD) = c;
            }
        }
    }
}

// ---------------------------------------------------------------------------
// backward pass R: reverse sweep for dk, dv, the reverse state and dL/dgamma
// ---------------------------------------------------------------------------
// Per tile c, with G_c = dL/dS_c (the state at the tile's end) in TMEM:
//   dk_r = sum_s M[s,r] (dy_s . v_r) q_s + w_out_r G_c v_r
//   dv_r = sum_s M[s,r] (q_s . k_r) dy_s + w_out_r G_c^T k_r
//   G_{c-1} = a_c G_c + sum_s w_in_s q_s dy_s^T
// and dL/dlog(gamma_t) (t not a begin flag) = gamma_t <dS_t, S_{t-1}>, split
// over the tile as
//   sum_{s >= t > r} E[s,r]                     E = M o (Q K^T) o (dY V^T)
//   + [no start in the tile up to t] sum_{s >= t} z_s      (pass F)
//   + sum_{r < t} x_r,  x_r = w_out_r k_r^T G_c v_r
//   + [no start in the tile] a_c <G_c, S_{c-1}>
// The first term is sum_{u < t} (colsum_u(E) - rowsum_u(E)): both sums come
// from the same fp32 E, so the telescoping cancels exactly up to fp32 rounding.
template <int D>
struct BwdSmem {
    static constexpr int TILE = T * D * 2;
    static constexpr int OFF_Q = 0, OFF_K = TILE, OFF_V = 2 * TILE, OFF_DY = 3 * TILE;
    static constexpr int OFF_PM = 4 * TILE, OFF_DPM = 4 * TILE + T * T * 2;
    static constexpr int OFF_GB = 4 * TILE + 2 * T * T * 2;
    // the stored state S_{c-1} (bf16, [j][i]) arrives with the tile in the dPm
    // buffer, which RP1 overwrites only after B1 is done
    static constexpr int OFF_SS = OFF_DPM;
    static_assert(D * D * 2 <= T * T * 2, "stored state fits in the dPm buffer");
    static constexpr int OFF_META = OFF_GB + D * D * 2;
    static constexpr int OFF_BAR = OFF_META + static_cast<int>(sizeof(TileMeta));
    static constexpr int BYTES = OFF_BAR + 64;
    // statistics, in the V tile (free once the first contractions are done)
    static constexpr int ST_COL = OFF_V;                // [4][T] column sums of E per lane quarter
    static constexpr int ST_ROW = ST_COL + 4 * T * 4;   // [4][T] row sums of E per column quarter
    static constexpr int ST_X = ST_ROW + 4 * T * 4;     // [4][T] x_r per column quarter
    static constexpr int ST_IV = ST_X + 4 * T * 4;      // [16] per-warp partial <G, S>, then [4] tile totals
    static constexpr int ST_INTRA = ST_IV + 128;        // [T] intra-tile term
    static constexpr int ST_WT = ST_INTRA + T * 4;      // [4] per-warp totals of x
    static_assert(ST_WT + 64 <= OFF_V + TILE, "statistics fit in the V tile");
    // fp32 dk / dv tiles staged for their TMA stores (128-byte swizzled, 32
    // channels x T rows = 16 KB per chunk), in buffers free once B2 is done:
    // d = 64: dk in Pm, dv in dPm; d = 128: dk in K | dPm (the buffers the next
    // tile's K and stored state go to, so that those loads wait only for the dk
    // stores), dv in Pm | G
    static constexpr int CHUNK = T * 128;
    __host__ __device__ static constexpr int dk_chunk(int m) {
        return D == 64 ? OFF_PM + m * CHUNK : (m < 2 ? OFF_K + m * CHUNK : OFF_DPM + (m - 2) * CHUNK);
    }
    __host__ __device__ static constexpr int dv_chunk(int m) {
        return D == 64 ? OFF_DPM + m * CHUNK : (m < 2 ? OFF_PM + m * CHUNK : OFF_GB + (m - 2) * CHUNK);
    }
    static_assert(D == 64 ? 2 * CHUNK <= T * T * 2 : 2 * CHUNK <= TILE && 2 * CHUNK <= T * T * 2 && 2 * CHUNK <= D * D * 2,
                  "output staging fits");
    // TMEM columns: P and dP, then dV and dK over them; V G^T; G
    static constexpr uint32_t COL_P = 0, COL_DP = 128, COL_DV = 0, COL_DK = 128, COL_DKI = 256,
                              COL_G = 256 + D, TMEM_COLS = 512;
    static_assert(COL_G + D <= TMEM_COLS, "tensor memory budget");
};

struct BwdParams {
    CUtensorMap map_q, map_k, map_v, map_dy;  // bf16 operands, box {64, 1, 128, 1}
    CUtensorMap map_dk, map_dv;               // fp32 outputs, box {32, 1, 128, 1}
    const uint16_t* q;
    const uint16_t* k;
    const uint16_t* v;
    const uint16_t* dy;  // bf16 copy of grad_y
    const float* gamma;
    int gamma_per_step;
    const float* dS_last;
    float* dk;
    float* dv;
    float* dgamma;      // per step: [B, L, H] output; per head: null (partials go to gpart)
    float* gpart;       // [B * H * G] per-segment sums of dL/dlog(gamma) (per-head mode)
    float* dS0;
    const TileMeta* meta;
    const float* carry;  // [B * H * G][D][D]: the reverse state leaving each segment (g >= 1)
    const float* dlam_f;
    const uint16_t* states;
    uint32_t* hdr;
    int64_t B, L, H, n_tiles, tps;
    int G;
    uint64_t wait_ns;
    int64_t fail_cta;  // test knob (see FwdParams)
};

// Reduces 32 values per lane over the warp's 32 lanes; lane l ends with the
// total of value l (a butterfly that halves the vector at each step).
__device__ __forceinline__ float warp_transpose_sum32(float (&v)[32], int lane) {
#pragma unroll
    for (int k = 16; k >= 1; k >>= 1) {
        const bool upper = (lane & k) != 0;
#pragma unroll
        for (int i = 0; i < k; ++i) {
            const float send = upper ? v[i] : v[i + k];
            const float keep = upper ? v[i + k] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, k);
        }
    }
    return v[0];
}

// Stores one thread's 16 fp32 values (columns j0..j0+15 of row r) into a
// 128-byte swizzled staging tile whose 32-channel chunks start at chunk(m).
template <typename ChunkFn>
__device__ __forceinline__ void stage_f32x16(unsigned char* smem, ChunkFn chunk, int r, int j0, const float* v) {
#pragma unroll
    for (int x = 0; x < 16; x += 4) {
        const int j = j0 + x;
        *reinterpret_cast<float4*>(smem + chunk(j >> 5) + r * 128 + ((((j & 31) >> 2) ^ (r & 7)) << 4)) =
            make_float4(v[x], v[x + 1], v[x + 2], v[x + 3]);
    }
}

template <int D, bool HALF_OUT = false, bool NORM = false>
__global__ void __launch_bounds__(kRThreads, 1) bwd_kernel(const __grid_constant__ BwdParams p) {
    static_assert(!HALF_OUT || D == 128, "half-width output at d = 128");
    static_assert(!NORM || HALF_OUT, "the normalised operands come with half-width outputs");
    // NORM: the normalised backward for 64-channel heads: q, k, v are the unpadded
    // [B, L, H, 64] tensors loaded into the first halves of their slots and built
    // in shared memory into q'' = [phi(q), sigma_hi, sigma_lo, 0], k'' = [psi(k),
    // 1, 1, 0] and v' = [v, 1, 1, 0]; dY is the caller's padded dy'.  K's
    // constant half, where dk rows are staged, is written again once they drain.
    constexpr int BKV = NORM ? 64 : D;  // channels loaded into the Q, K and V slots
    // HALF_OUT: only the first 64 columns of dk and dv are written, to [B, L, H, 64]
    // outputs (the normalised path needs no more of dk' and dv')
    constexpr int DOUT = HALF_OUT ? 64 : D;
    using S = BwdSmem<D>;
    extern __shared__ __align__(1024) unsigned char smem[];
    grid_dependency_wait();  // pass F (its tile states and dgamma terms)
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int quarter = warp & 3, cq = warp >> 2;  // TMEM lane quarter, column quarter
    const int64_t bh = blockIdx.x / p.G;
    const int g = static_cast<int>(blockIdx.x % p.G);
    const int64_t b = bh / p.H, h = bh % p.H;
    // this segment: tiles [tile_lo, tile_hi), steps up to seg_hi (the tape end for the last)
    const int64_t tile_lo = static_cast<int64_t>(g) * p.tps, tile_hi = min(p.n_tiles, tile_lo + p.tps);
    const int64_t seg_hi = min(p.L, tile_hi * T);
    // the reverse state entering the segment's last step: dS_last for the last
    // segment, else the carry
    const float* g_in = g == p.G - 1 ? (p.dS_last != nullptr ? p.dS_last + bh * D * D : nullptr)
                                     : p.carry + (bh * p.G + g + 1) * D * D;

    uint64_t* bar1 = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);
    uint64_t* bar2 = bar1 + 1;
    uint64_t* bar3 = bar1 + 2;
    uint64_t* full = bar1 + 3;
    uint32_t* tslot = reinterpret_cast<uint32_t*>(bar1 + 4);
    uint64_t* bar4 = bar1 + 5;  // V G^T of B1, committed apart from P and dP
    uint64_t* kbar = bar1 + 6;  // NORM: the raw k rows for phi'(k), in V's constant half
    const TileMeta& mc = *reinterpret_cast<const TileMeta*>(smem + S::OFF_META);
    const uint32_t sbase = smem_addr(smem);
    const uint32_t sQ = sbase + S::OFF_Q, sK = sbase + S::OFF_K, sV = sbase + S::OFF_V, sDY = sbase + S::OFF_DY;
    const uint32_t sPM = sbase + S::OFF_PM, sDPM = sbase + S::OFF_DPM, sGB = sbase + S::OFF_GB;
    float* st_col = reinterpret_cast<float*>(smem + S::ST_COL);
    float* st_row = reinterpret_cast<float*>(smem + S::ST_ROW);
    float* st_x = reinterpret_cast<float*>(smem + S::ST_X);
    float* st_iv = reinterpret_cast<float*>(smem + S::ST_IV);
    float* st_intra = reinterpret_cast<float*>(smem + S::ST_INTRA);
    float* st_wt = reinterpret_cast<float*>(smem + S::ST_WT);
    auto dk_chunk = [](int m) { return S::dk_chunk(m); };
    auto dv_chunk = [](int m) { return S::dv_chunk(m); };

    // thread 0: TMA loads of a tile, its metadata and (once a reverse state
    // exists) the stored forward state before it, completing on `full`.  The
    // state slot of a tile with a begin flag was never written: it is loaded
    // all the same and not read.
    constexpr uint32_t kTileBytes = 3 * (T * BKV * 2) + S::TILE;  // Q, K, V and dY
    auto issue_tile = [&](int64_t tile, bool with_state) {
        constexpr uint32_t kStateBytes = D * D * 2;
        mbar_arrive_expect_tx(full, kTileBytes + sizeof(TileMeta) + (with_state ? kStateBytes : 0u));
        const int64_t t0 = tile * T;
        tma_tile<BKV>(sQ, &p.map_q, h, t0, b, full);
        tma_tile<BKV>(sK, &p.map_k, h, t0, b, full);
        tma_tile<BKV>(sV, &p.map_v, h, t0, b, full);
        tma_tile<D>(sDY, &p.map_dy, h, t0, b, full);
        bulk_g2s(smem + S::OFF_META, p.meta + bh * p.n_tiles + tile, sizeof(TileMeta), full);
        if (with_state) bulk_g2s(smem + S::OFF_SS, p.states + (bh * p.n_tiles + tile) * D * D, kStateBytes, full);
    };
    // the same loads in two groups for every later tile: Q, V, dY and the metadata
    // as soon as B3 is done, K and the state once the staged output stores (in
    // K, G, Pm and dPm) have been read
    auto issue_tile_a = [&](int64_t tile) {
        mbar_arrive_expect_tx(full, kTileBytes + sizeof(TileMeta) + D * D * 2);
        const int64_t t0 = tile * T;
        tma_tile<BKV>(sQ, &p.map_q, h, t0, b, full);
        tma_tile<BKV>(sV, &p.map_v, h, t0, b, full);
        tma_tile<D>(sDY, &p.map_dy, h, t0, b, full);
        bulk_g2s(smem + S::OFF_META, p.meta + bh * p.n_tiles + tile, sizeof(TileMeta), full);
    };
    auto issue_tile_b = [&](int64_t tile) {
        tma_tile<BKV>(sK, &p.map_k, h, tile * T, b, full);
        bulk_g2s(smem + S::OFF_SS, p.states + (bh * p.n_tiles + tile) * D * D, D * D * 2, full);
    };
    bool have_g = g_in != nullptr;  // a reverse state enters the current tile

    if (tid == 0) {
        mbar_init(bar1, 1);
        mbar_init(bar2, 1);
        mbar_init(bar3, 1);
        mbar_init(full, 1);
        mbar_init(bar4, 1);
        if (NORM) mbar_init(kbar, 1);
        fence_mbar_init();
        prefetch_tensormap(&p.map_q);
        prefetch_tensormap(&p.map_k);
        prefetch_tensormap(&p.map_v);
        prefetch_tensormap(&p.map_dy);
        prefetch_tensormap(&p.map_dk);
        prefetch_tensormap(&p.map_dv);
    }
    if (warp == 0) tc::alloc(tslot, S::TMEM_COLS);
    if (NORM) {
        const_box<kRThreads>(smem + S::OFF_Q, tid, false);
        const_box<kRThreads>(smem + S::OFF_K, tid, true);
        const_box<kRThreads>(smem + S::OFF_V, tid, true);
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (tid == 0) issue_tile(tile_hi - 1, have_g);
    const uint32_t tm = *tslot;
    const uint32_t lane_base = tm + (static_cast<uint32_t>(32 * quarter) << 16);
    const int srow = state_row<D>(quarter, lane);
    constexpr int SC = D / 4;  // state and output columns per thread
    constexpr int PC = T / 4;  // score columns per thread

    // ---- incoming reverse state ----
    if (have_g) {
        const float* src = g_in;
#pragma unroll 1
        for (int cc = 0; cc < SC / 16; ++cc) {
            const int j0 = cq * SC + cc * 16;
            float v[16];
            if (srow >= 0) {
#pragma unroll
                for (int x = 0; x < 16; x += 4) {
                    const float4 f = *reinterpret_cast<const float4*>(src + srow * D + j0 + x);
                    v[x] = f.x;
                    v[x + 1] = f.y;
                    v[x + 2] = f.z;
                    v[x + 3] = f.w;
                }
                store_bf16x16(smem + S::OFF_GB, core_off(srow, j0, D), core_off(srow, j0 + 8, D), v);
            } else {
#pragma unroll
                for (int x = 0; x < 16; ++x) v[x] = 0.f;
            }
            tc::st16(lane_base + S::COL_G + j0, v);
        }
    }

    constexpr uint32_t ID_SCORE = tc::idesc_bf16(128, T, false, false);  // P, dP
    constexpr uint32_t ID_VG = tc::idesc_bf16(128, D, false, false);     // V G^T
    constexpr uint32_t ID_PTDY = tc::idesc_bf16(128, D, true, true);     // Pm^T dY, dPm^T Q
    constexpr uint32_t ID_KG = tc::idesc_bf16(128, D, false, true);      // K~ G
    constexpr uint32_t ID_QDY = tc::idesc_bf16(D, D, true, true);        // Q~^T dY

    float gsum = 0.f;  // per-head mode: sum of dL/dlog(gamma) over the segment's steps
    bool failed = false;
    bool pending = true;  // a tile load may be in flight
    uint64_t* drain = nullptr;  // a batch issued but not seen complete
    uint32_t drain_par = 0;
    uint32_t ph4 = 0;           // phase of bar4 (committed only on tiles with a reverse state)
    bool k_pending = false;     // NORM: a raw k load not seen complete
    int it = 0;
#pragma unroll 1
    for (int64_t tile = tile_hi - 1; tile >= tile_lo; --tile, ++it) {
        const int64_t t0 = tile * T;
        const int r_hi = static_cast<int>(min(static_cast<int64_t>(T), seg_hi - t0));  // rows inside the tape
        bool ok = wait_mbar(full, it & 1, p.wait_ns);
        tc::fence_smem_to_async();
        tc::fence_before();
        if (__syncthreads_or(!ok)) {
            failed = true;
            break;
        }
        pending = false;
        tc::fence_after();
        if (NORM) {
            const int64_t valid = p.L - t0;
            phiq_box<kRThreads>(smem + S::OFF_Q, tid, valid);
            psi_box<kRThreads>(smem + S::OFF_K, tid, valid);
            tc::fence_smem_to_async();
            __syncthreads();
        }
        const bool tile_start = mc.has_start != 0;

        // ---- B1: P = Q K^T, dP = dY V^T, dKi = V G^T ----
        if (tid == 0) {
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                tc::mma(tm + S::COL_P, desc_sw_k(sQ, kk), desc_sw_k(sK, kk), ID_SCORE, kk > 0);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                tc::mma(tm + S::COL_DP, desc_sw_k(sDY, kk), desc_sw_k(sV, kk), ID_SCORE, kk > 0);
            tc::commit(bar1);
            if (have_g) {
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    tc::mma(tm + S::COL_DKI, desc_sw_k(sV, kk), desc_kmajor(sGB, D, kk), ID_VG, kk > 0);
                tc::commit(bar4);
            }
        }
        // while B1 runs (it reads G only through its bf16 copy): this thread's row
        // of <G_c, S_{c-1}> and G *= a_c in tensor memory; pass F's dgamma term
        // and gamma for the rows of warps 0-3
        const bool need_iv = have_g && !tile_start;
        float ivp = 0.f;
        {
            const bool scale = have_g && !tile_start && mc.a != 1.f;
            if (need_iv || scale) {
                const unsigned char* ss = smem + S::OFF_SS;  // S_{c-1}: element [j][i] at state_off(j, i)
                uint32_t gv[SC];
#pragma unroll
                for (int cc = 0; cc < SC / 16; ++cc) tc::ld16_nowait(lane_base + S::COL_G + cq * SC + cc * 16, gv + cc * 16);
                tc::ld_wait();
                if (need_iv && srow >= 0) {
#pragma unroll
                    for (int x = 0; x < SC; ++x)
                        ivp = fmaf(__uint_as_float(gv[x]),
                                   __uint_as_float(static_cast<uint32_t>(*reinterpret_cast<const uint16_t*>(
                                                       ss + state_off<D>(cq * SC + x, srow))) << 16), ivp);
                }
                if (scale) {
#pragma unroll
                    for (int cc = 0; cc < SC / 16; ++cc) {
                        float v[16];
#pragma unroll
                        for (int x = 0; x < 16; ++x) v[x] = __uint_as_float(gv[cc * 16 + x]) * mc.a;
                        tc::st16(lane_base + S::COL_G + cq * SC + cc * 16, v);
                    }
                }
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) ivp += __shfl_xor_sync(0xffffffffu, ivp, off);
        }
        float dlf = 0.f, gmt = 1.f;
        if (warp < 4) {
            const int t = 32 * warp + lane;
            if (t < r_hi) {
                const int64_t idx = (b * p.L + t0 + t) * p.H + h;
                dlf = p.dlam_f[idx];
                if (p.dgamma != nullptr) gmt = p.gamma_per_step ? p.gamma[idx] : p.gamma[h];
            }
        }
        ok = wait_mbar(bar1, it & 1, p.wait_ns) && !(it == 0 && static_cast<int64_t>(blockIdx.x) == p.fail_cta);
        if (__syncthreads_or(!ok)) {
            failed = true;
            drain = have_g ? bar4 : bar1;  // bar4 completes after every batch before it
            drain_par = have_g ? ph4 : (it & 1);
            break;
        }
        tc::fence_after();

        // ---- RP1: masks and E statistics; x_r; <G_c, S_{c-1}> and G *= a ----
        {
            const int t = 32 * quarter + lane;  // the row s of P and dP this thread holds
            const float lt = mc.lam2[t];
            const int st = mc.seg[t];
            float rsum = 0.f;
            const int r0 = cq * PC;  // this warp's 32 score columns, in two batches of 16
            float e[PC];
            unsigned char* pmb = smem + S::OFF_PM;
            unsigned char* dpmb = smem + S::OFF_DPM;
#pragma unroll
            for (int cc = 0; cc < PC; cc += 16) {
                uint32_t rp[16], rd[16];
                tc::ld16_nowait(lane_base + S::COL_P + r0 + cc, rp);
                tc::ld16_nowait(lane_base + S::COL_DP + r0 + cc, rd);
                tc::ld_wait();
                float pm[16], dpm[16];
#pragma unroll
                for (int x = 0; x < 16; ++x) {
                    const int r = r0 + cc + x;
                    const float m = (r <= t && r >= st) ? fast_exp2(lt - mc.lam2[r]) : 0.f;
                    const float pv = __uint_as_float(rp[x]), dv = __uint_as_float(rd[x]);
                    pm[x] = m * pv;
                    dpm[x] = m * dv;
                    e[cc + x] = pm[x] * dv;
                    rsum += e[cc + x];
                }
                store_bf16x16(pmb, core_off(t, r0 + cc, T), core_off(t, r0 + cc + 8, T), pm);
                store_bf16x16(dpmb, core_off(t, r0 + cc, T), core_off(t, r0 + cc + 8, T), dpm);
            }
            static_assert(PC == 32, "one transposed warp sum per thread's score columns");
            const float cs = warp_transpose_sum32(e, lane);
            st_col[quarter * T + r0 + lane] = cs;
            st_row[cq * T + t] = rsum;

            // x_r = w_out_r k_r . (G_c v_r), from the unscaled K tile, once V G^T is done
            float xacc = 0.f;
            if (have_g) {
                ok = wait_mbar(bar4, ph4, p.wait_ns);
                tc::fence_after();
                const unsigned char* kt = smem + S::OFF_K;
                uint32_t gi[SC];  // this thread's quarter row of V G^T, all loads in flight at once
#pragma unroll
                for (int cc = 0; cc < SC / 16; ++cc) tc::ld16_nowait(lane_base + S::COL_DKI + cq * SC + cc * 16, gi + cc * 16);
                tc::ld_wait();
#pragma unroll
                for (int x = 0; x < SC; x += 8) {
                    const uint4 u = *reinterpret_cast<const uint4*>(kt + sw_off(t, cq * SC + x));
                    const float2 k0 = unpack_bf16x2(u.x), k1 = unpack_bf16x2(u.y), k2 = unpack_bf16x2(u.z),
                                 k3 = unpack_bf16x2(u.w);
                    xacc = fmaf(k0.x, __uint_as_float(gi[x]), xacc);
                    xacc = fmaf(k0.y, __uint_as_float(gi[x + 1]), xacc);
                    xacc = fmaf(k1.x, __uint_as_float(gi[x + 2]), xacc);
                    xacc = fmaf(k1.y, __uint_as_float(gi[x + 3]), xacc);
                    xacc = fmaf(k2.x, __uint_as_float(gi[x + 4]), xacc);
                    xacc = fmaf(k2.y, __uint_as_float(gi[x + 5]), xacc);
                    xacc = fmaf(k3.x, __uint_as_float(gi[x + 6]), xacc);
                    xacc = fmaf(k3.y, __uint_as_float(gi[x + 7]), xacc);
                }
                const float w_out = t >= mc.last_start ? fast_exp2(mc.lam2[T - 1] - mc.lam2[t]) : 0.f;
                xacc *= w_out;
            }
            st_x[cq * T + t] = xacc;
        }
        if (lane == 0) st_iv[warp] = ivp;
        if (__syncthreads_or(!ok)) {  // every x_r has read the unscaled K
            failed = true;
            drain = bar4;
            drain_par = ph4;
            break;
        }
        if (have_g) ph4 ^= 1;
        if (NORM && tid == 0) {
            // the first batch (V G^T included) is done with V: its constant half
            // takes the raw k rows of this tile for phi'(k) in the dk epilogue
            mbar_arrive_expect_tx(kbar, T * 64 * 2);
            tma_tile<64>(sV + T * 128, &p.map_k, h, t0, b, kbar);
        }
        if (NORM) k_pending = true;
        {
            // K~ = w_out (.) K in place (K is not read unscaled after this)
            const float lend = mc.lam2[T - 1];
            const int ls = mc.last_start;
            scale_rows_sw<D, kRThreads>(smem + S::OFF_K, tid,
                                        [&](int r) { return r >= ls ? fast_exp2(lend - mc.lam2[r]) : 0.f; });
        }
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        tc::fence_after();

        // ---- B2: dV = Pm^T dY + K~ G, dK = dPm^T Q ----
        if (tid == 0) {
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_DV, desc_mnmajor(sPM, T, kk), desc_sw_mn(sDY, kk), ID_PTDY, kk > 0);
            if (have_g) {
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    tc::mma(tm + S::COL_DV, desc_sw_k(sK, kk), desc_mnmajor(sGB, D, kk), ID_KG, true);
            }
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_DK, desc_mnmajor(sDPM, T, kk), desc_sw_mn(sQ, kk), ID_PTDY, kk > 0);
            tc::commit(bar2);
        }
        // intra-tile term while B2 runs: intra_t = sum_{u < t} (colsum_u - rowsum_u)
        if (warp == 7) {
            float d[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                const int u = 4 * lane + x;
                d[x] = (st_col[u] + st_col[T + u]) + (st_col[2 * T + u] + st_col[3 * T + u]) -
                       ((st_row[u] + st_row[T + u]) + (st_row[2 * T + u] + st_row[3 * T + u]));
            }
            float incl = d[0] + d[1] + d[2] + d[3];
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const float o = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += o;
            }
            float run = incl - (d[0] + d[1] + d[2] + d[3]);
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                st_intra[4 * lane + x] = run;
                run += d[x];
            }
        }
        // x prefix within each of warps 0-3 (rows 32w..32w+31) while B2 runs
        float xpre_in = 0.f;
        if (warp < 4) {
            const int t = 32 * warp + lane;
            const float xt = (st_x[t] + st_x[T + t]) + (st_x[2 * T + t] + st_x[3 * T + t]);
            float incl = xt;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const float o = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += o;
            }
            xpre_in = incl - xt;
            if (lane == 31) st_wt[warp] = incl;
        }
        ok = wait_mbar(bar2, it & 1, p.wait_ns);
        if (__syncthreads_or(!ok)) {
            failed = true;
            drain = bar2;
            drain_par = it & 1;
            break;
        }
        tc::fence_after();

        // ---- RP2: Q~ = w_in (.) Q in place, then B3: G += Q~^T dY ----
        scale_rows_sw<D, kRThreads>(smem + S::OFF_Q, tid,
                                    [&](int r) { return mc.seg[r] < 0 ? fast_exp2(mc.lam2[r]) : 0.f; });
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        tc::fence_after();
        if (tid == 0) {
            const bool acc = have_g && !tile_start;
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_G, desc_sw_mn(sQ, kk), desc_sw_mn(sDY, kk), ID_QDY, acc || kk > 0);
            tc::commit(bar3);
        }

        // ---- epilogue (while B3 runs): dk = dK + w_out dKi, then dv, each staged and
        // stored on its own, so that the dk stores drain while dv is staged ----
        // warp 0: one TMA store of the staged tile per 32 channels (rows past L are clipped)
        auto store_tile = [&](bool is_dv) {
            const CUtensorMap* map = is_dv ? &p.map_dv : &p.map_dk;
            if (lane == 0) {
#pragma unroll
                for (int m = 0; m < DOUT / 32; ++m)
                    tma_store_4d(map, sbase + (is_dv ? S::dv_chunk(m) : S::dk_chunk(m)), 32 * m, static_cast<int>(h),
                                 static_cast<int>(t0), static_cast<int>(b));
                bulk_commit();
            }
        };
        if (NORM) {
            ok = wait_mbar(kbar, it & 1, p.wait_ns);
            if (__syncthreads_or(!ok)) {
                failed = true;
                drain = bar3;
                drain_par = it & 1;
                break;
            }
            k_pending = false;
        }
        {
            const int r = 32 * quarter + lane;
            const float w_out = r >= mc.last_start ? fast_exp2(mc.lam2[T - 1] - mc.lam2[r]) : 0.f;
#pragma unroll
            for (int cc = 0; cc < SC / 16; ++cc) {
                const int j0 = cq * SC + cc * 16;
                uint32_t rk[16], ri[16];
                tc::ld16_nowait(lane_base + S::COL_DK + j0, rk);
                if (have_g) tc::ld16_nowait(lane_base + S::COL_DKI + j0, ri);
                tc::ld_wait();
                float vk[16];
#pragma unroll
                for (int x = 0; x < 16; ++x)
                    vk[x] = have_g ? fmaf(w_out, __uint_as_float(ri[x]), __uint_as_float(rk[x])) : __uint_as_float(rk[x]);
                stage_f32x16(smem, dk_chunk, r, j0, vk);
            }
        }
        if (NORM) {
            // dk = dk''[:64] (.) phi'(k) (psi' = phi') on the staged rows, from the
            // raw k rows: four threads per row, 16 channels each
            __syncthreads();
            const int r = tid >> 2, m = (tid >> 1) & 1, u0 = (tid & 1) * 4;
            const unsigned char* kraw = smem + S::OFF_V + T * 128;
            unsigned char* row = smem + S::dk_chunk(m) + r * 128;
#pragma unroll
            for (int u = u0; u < u0 + 4; ++u) {
                float4* o = reinterpret_cast<float4*>(row + ((u ^ (r & 7)) << 4));
                *o = times_phi_prime(*o, *reinterpret_cast<const uint2*>(kraw + sw_off(r, 32 * m + 4 * u)));
            }
        }
        tc::fence_smem_to_async();
        __syncthreads();
        if (warp == 0) store_tile(false);
        {
            const int r = 32 * quarter + lane;
#pragma unroll
            for (int cc = 0; cc < SC / 16; ++cc) {
                const int j0 = cq * SC + cc * 16;
                float vv[16];
                tc::ld16(lane_base + S::COL_DV + j0, vv);
                stage_f32x16(smem, dv_chunk, r, j0, vv);
            }
        }
        tc::fence_smem_to_async();
        __syncthreads();
        if (warp == 0) store_tile(true);
        // ---- dL/dlog(gamma_t) for the tile's rows (warps 0-3, one row per thread) ----
        if (warp < 4) {
            const int t = 32 * warp + lane;
            float lower = 0.f;
            for (int w2 = 0; w2 < warp; ++w2) lower += st_wt[w2];
            float iv = 0.f;
            if (!tile_start) {
#pragma unroll
                for (int w2 = 0; w2 < kRThreads / 32; ++w2) iv += st_iv[w2];
                iv *= mc.a;
            }
            const bool in = t < r_hi;
            const bool is_start = mc.seg[t] == t;
            float dl = 0.f;
            if (in && !is_start) dl = st_intra[t] + (lower + xpre_in) + iv + dlf;
            if (in && p.dgamma != nullptr) p.dgamma[(b * p.L + t0 + t) * p.H + h] = dl / gmt;
            // per-head mode: fixed-order tile total
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) dl += __shfl_xor_sync(0xffffffffu, dl, off);
            if (lane == 0) st_iv[16 + warp] = dl;
        }
        tc::fence_smem_to_async();  // the statistics in the V tile are overwritten by the next tile's load
        ok = wait_mbar(bar3, it & 1, p.wait_ns);
        if (__syncthreads_or(!ok)) {
            failed = true;
            drain = bar3;
            drain_par = it & 1;
            break;
        }
        tc::fence_after();
        const bool next = tile > tile_lo;
        if (tid == 0) {
            gsum += (st_iv[16] + st_iv[17]) + (st_iv[18] + st_iv[19]);
            // Q, V, dY and the metadata are free (B3 is done, the statistics are read):
            // their loads go out while the staged dk / dv stores drain
            if (next) {
                tc::fence_smem_to_async();
                issue_tile_a(tile - 1);
            }
            if (D == 128) {
                // K and dPm held the dk staging: once the dk stores (the older group)
                // have read it, the next tile's K and stored state go there
                bulk_wait_read_1();
                if (next) issue_tile_b(tile - 1);
            }
            bulk_wait_read();  // every staged store has been read (G is written next)
        }
        if (next) pending = true;
        have_g = true;
        __syncthreads();
        if (D == 64 && next && tid == 0) issue_tile_b(tile - 1);
        if (NORM) {
            const_box<kRThreads>(smem + S::OFF_K, tid, true);  // K's constant half held dk rows
            const_box<kRThreads>(smem + S::OFF_V, tid, true);  // V's held the raw k rows
        }

        // ---- G_{c-1} -> bf16 operand for the next tile (and dS0 at the tape start) ----
        {
            const bool last = tile == tile_lo;
            const bool write_ds0 = last && g == 0 && p.dS0 != nullptr;
            uint32_t gv[SC];
#pragma unroll
            for (int cc = 0; cc < SC / 16; ++cc) tc::ld16_nowait(lane_base + S::COL_G + cq * SC + cc * 16, gv + cc * 16);
            tc::ld_wait();
#pragma unroll
            for (int cc = 0; cc < SC / 16; ++cc) {
                const int j0 = cq * SC + cc * 16;
                float v[16];
#pragma unroll
                for (int x = 0; x < 16; ++x) v[x] = __uint_as_float(gv[cc * 16 + x]);
                if (srow >= 0) {
                    if (!last) store_bf16x16(smem + S::OFF_GB, core_off(srow, j0, D), core_off(srow, j0 + 8, D), v);
                    if (write_ds0) {
                        float* dst = p.dS0 + (bh * D + srow) * D + j0;
#pragma unroll
                        for (int x = 0; x < 16; x += 4)
                            *reinterpret_cast<float4*>(dst + x) = make_float4(v[x], v[x + 1], v[x + 2], v[x + 3]);
                    }
                }
            }
        }
        tc::fence_before();
        __syncthreads();
    }
    if (failed) {
        if (tid == 0) record_error(p.hdr, DEV_MMA_TIMEOUT);
        // let work still in flight finish before the CTA's TMEM and shared memory go away
        if (drain != nullptr) wait_mbar(drain, drain_par, kDrainNs);
        if (pending) wait_mbar(full, it & 1, kDrainNs);
        if (NORM && k_pending) wait_mbar(kbar, it & 1, kDrainNs);
    }
    if (tid == 0) bulk_wait_all();
    if (tid == 0 && p.gpart != nullptr) p.gpart[bh * p.G + g] = gsum;
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 0) tc::dealloc(tm, S::TMEM_COLS);
}

// grad_y (fp32) -> bf16 operand copy (round to nearest even), 8 values per thread
__global__ void __launch_bounds__(256) to_bf16_kernel(const float* __restrict__ x, uint16_t* __restrict__ y, int64_t n8) {
    grid_dependency_wait();  // the kernel before it on the stream
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n8;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const float4 a = reinterpret_cast<const float4*>(x)[2 * i];
        const float4 c = reinterpret_cast<const float4*>(x)[2 * i + 1];
        uint4 o;
        o.x = pack_bf16x2(a.x, a.y);
        o.y = pack_bf16x2(a.z, a.w);
        o.z = pack_bf16x2(c.x, c.y);
        o.w = pack_bf16x2(c.z, c.w);
        reinterpret_cast<uint4*>(y)[i] = o;
    }
}

// per-head dL/dgamma_h = (sum over tapes and segments of dL/dlog(gamma)) / gamma_h, fixed order
__global__ void dgamma_head_kernel(const float* __restrict__ gpart, const float* __restrict__ gamma,
                                   float* __restrict__ dgamma, int64_t B, int64_t H, int G) {
    grid_dependency_wait();  // pass R's per-segment sums
    const int64_t h = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (h >= H) return;
    double acc = 0.0;
    for (int64_t b = 0; b < B; ++b)
        for (int g = 0; g < G; ++g) acc += gpart[(b * H + h) * G + g];
    dgamma[h] = static_cast<float>(acc / gamma[h]);
}

// ---------------------------------------------------------------------------
// measurement: the intra-tile contraction alone, operands resident in smem
// ---------------------------------------------------------------------------
// Each CTA stages one Q, K, V tile and one masked-score tile (any bits; the
// values do not matter) and then issues `reps` times the two intra-tile
// contractions of the forward pass, P = Q K^T and Y = Pm V, with the same
// descriptors and instruction shapes as fwd_kernel, accumulating in TMEM.
// Executed flops per rep: 4 * T * T * D.  No HBM traffic after the staging.
template <int D>
__global__ void __launch_bounds__(128, 1) intra_bench_kernel(const uint4* __restrict__ src, int reps,
                                                            float* __restrict__ sink, uint32_t* hdr, uint64_t wait_ns) {
    constexpr int TILE = T * D * 2, PM = T * T * 2;
    extern __shared__ __align__(1024) unsigned char smem[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ uint32_t tslot;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int total16 = (3 * TILE + PM) / 16;
    for (int i = tid; i < total16; i += blockDim.x) {
        uint4 u = src[i];
        // keep the values finite and moderate: clear the exponent's top bits
        u.x &= 0x3fff3fffu;
        u.y &= 0x3fff3fffu;
        u.z &= 0x3fff3fffu;
        u.w &= 0x3fff3fffu;
        reinterpret_cast<uint4*>(smem)[i] = u;
    }
    if (tid == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    if (warp == 0) tc::alloc(&tslot, 256);
    tc::fence_smem_to_async();
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tm = tslot;
    const uint32_t sq = smem_addr(smem), sk = sq + TILE, sv = sq + 2 * TILE, spm = sq + 3 * TILE;
    constexpr uint32_t ID_QK = tc::idesc_bf16(128, T, false, false);
    constexpr uint32_t ID_PV = tc::idesc_bf16(128, D, false, true);
    if (tid == 0) {
        for (int r = 0; r < reps; ++r) {
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                tc::mma(tm, desc_sw_k(sq, kk), desc_sw_k(sk, kk), ID_QK, r > 0 || kk > 0);
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + 128, desc_kmajor(spm, T, kk), desc_sw_mn(sv, kk), ID_PV, r > 0 || kk > 0);
        }
        tc::commit(&bar);
    }
    const bool ok = wait_mbar(&bar, 0, wait_ns);
    if (!ok) wait_mbar(&bar, 0, kDrainNs);  // the contractions finish before TMEM is freed
    tc::fence_after();
    if (!ok && tid == 0) record_error(hdr, DEV_MMA_TIMEOUT);
    if (ok) {
        float v[16];
        tc::ld16(tm + (static_cast<uint32_t>(32 * warp) << 16), v);
        if (tid == 0) sink[blockIdx.x] = v[0];
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 0) tc::dealloc(tm, 256);
}

size_t intra_bench_scratch_bytes(int64_t D) {
    return kHeaderBytes + static_cast<size_t>(3 * T * D * 2 + T * T * 2) + 4096 * sizeof(float);
}

memoroid_status_t launch_intra_bench(int64_t D, int64_t reps, int64_t ctas, void* scratch, cudaStream_t stream) {
    unsigned char* ws = static_cast<unsigned char*>(scratch);
    uint32_t* hdr = reinterpret_cast<uint32_t*>(ws);
    const uint4* src = reinterpret_cast<const uint4*>(ws + kHeaderBytes);
    float* sink = reinterpret_cast<float*>(ws + kHeaderBytes + 3 * T * D * 2 + T * T * 2);
    const uint64_t wait_ns = debug_knobs().wait_ns;
    if (cudaMemsetAsync(scratch, 0, kHeaderBytes, stream) != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (D == 64) {
        const int bytes = 3 * T * 64 * 2 + T * T * 2;
        if (cudaFuncSetAttribute(intra_bench_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) !=
            cudaSuccess)
            return MEMOROID_ERR_CUDA;
        intra_bench_kernel<64><<<static_cast<unsigned>(ctas), 128, bytes, stream>>>(src, static_cast<int>(reps), sink,
                                                                                    hdr, wait_ns);
    } else if (D == 128) {
        const int bytes = 3 * T * 128 * 2 + T * T * 2;
        if (cudaFuncSetAttribute(intra_bench_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) !=
            cudaSuccess)
            return MEMOROID_ERR_CUDA;
        intra_bench_kernel<128><<<static_cast<unsigned>(ctas), 128, bytes, stream>>>(src, static_cast<int>(reps), sink,
                                                                                     hdr, wait_ns);
    } else {
        return MEMOROID_ERR_UNSUPPORTED;
    }
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {
template <typename K>
cudaError_t set_smem(K kernel, int bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

// A bf16 [B, L, H, D] tensor as a 4-D map {D, H, L, B} with 128-byte swizzled
// boxes of 64 channels x T steps of one head ({64, 1, T, 1}); steps past L
// read as zeros.
bool tile_map_y(CUtensorMap* m, const void* base, int64_t B, int64_t L, int64_t H, int64_t D);

bool tile_map(CUtensorMap* m, const void* base, int64_t B, int64_t L, int64_t H, int64_t D) {
    const EncodeTiledFn fn = encode_tiled();
    if (fn == nullptr) return false;
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(L),
                                static_cast<cuuint64_t>(B)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D * 2), static_cast<cuuint64_t>(H * D * 2),
                                   static_cast<cuuint64_t>(L * H * D * 2)};
    const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(T), 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// An fp32 [B, L, H, D] output as a 4-D map {D, H, L, B} with 128-byte swizzled
// boxes of 32 channels x T steps ({32, 1, T, 1}); stores past L are clipped.
bool tile_map_y(CUtensorMap* m, const void* base, int64_t B, int64_t L, int64_t H, int64_t D) {
    const EncodeTiledFn fn = encode_tiled();
    if (fn == nullptr) return false;
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(L),
                                static_cast<cuuint64_t>(B)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(D * 4), static_cast<cuuint64_t>(H * D * 4),
                                   static_cast<cuuint64_t>(L * H * D * 4)};
    const cuuint32_t box[4] = {32, 1, static_cast<cuuint32_t>(T), 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

namespace {
// Tile metadata (shared by the forward and backward passes).
memoroid_status_t launch_prep(const Args& a, const Plan& pl, TileMeta* meta, cudaStream_t stream) {
    const int64_t meta_blocks = (a.B * a.H * pl.n_tiles * 32 + 255) / 256;
    meta_kernel<<<static_cast<unsigned>(meta_blocks), 256, 0, stream>>>(a.gamma, a.gamma_per_step, a.start, a.B,
                                                                         a.L, a.H, pl.n_tiles, meta);
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

// The states entering the segments (REV = false, from the X = k, Y = v
// summaries and S0) or the reverse states entering them from the right
// (REV = true, from X = q, Y = dy and dS_last): the summary kernel, then the
// carry over the segments, in place in `buf`.  Nothing to do for one segment.
template <int D, bool REV, bool NORM, bool PSI>
memoroid_status_t launch_seg_carry(const Args& a, const Plan& pl, const TileMeta* meta, float2* info, float* buf,
                                   const CUtensorMap& map_x, const CUtensorMap& map_y, const float* init,
                                   uint32_t* hdr, cudaStream_t stream) {
    if (pl.G <= 1) return MEMOROID_OK;
    SegParams p;
    p.map_x = map_x;
    p.map_y = map_y;
    p.meta = meta;
    p.info = info;
    p.out = buf;
    p.hdr = hdr;
    p.L = a.L;
    p.H = a.H;
    p.n_tiles = pl.n_tiles;
    p.tps = pl.tps;
    p.G = static_cast<int>(pl.G);
    p.wait_ns = debug_knobs().wait_ns;
    if (set_smem(seg_state_kernel<D, REV, NORM, PSI>, SegSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (launch_after(seg_state_kernel<D, REV, NORM, PSI>, dim3(static_cast<unsigned>(a.B * a.H * (pl.G - 1))),
                     dim3(kThreads), SegSmem<D>::BYTES, stream, p) != cudaSuccess)
        return MEMOROID_ERR_CUDA;
    const dim3 grid(static_cast<unsigned>((D * D / 4 + 255) / 256), static_cast<unsigned>(a.B * a.H));
    return launch_after(seg_carry_kernel<REV>, grid, dim3(256), 0, stream, buf, static_cast<const float2*>(info), init,
                        static_cast<int>(pl.G), D * D) == cudaSuccess
               ? MEMOROID_OK
               : MEMOROID_ERR_CUDA;
}

template <int D, bool NORM = false>
memoroid_status_t launch_fwd_d(const Args& a, const Plan& pl, const Layout& ly, cudaStream_t stream) {
    unsigned char* ws = static_cast<unsigned char*>(a.workspace);
    TileMeta* meta = reinterpret_cast<TileMeta*>(ws + ly.meta);
    float2* info = reinterpret_cast<float2*>(ws + ly.info);
    float* carry = reinterpret_cast<float*>(ws + ly.carry_f);
    uint32_t* hdr = reinterpret_cast<uint32_t*>(ws);
    memoroid_status_t st = launch_prep(a, pl, meta, stream);
    if (st != MEMOROID_OK) return st;

    FwdParams p;
    constexpr int KQ = NORM ? 64 : D;  // channels of q, k, v (and of y) in memory
    if (!tile_map(&p.map_q, a.q, a.B, a.L, a.H, KQ) || !tile_map(&p.map_k, a.k, a.B, a.L, a.H, KQ) ||
        !tile_map(&p.map_v, a.v, a.B, a.L, a.H, KQ) || !tile_map_y(&p.map_y, a.y, a.B, a.L, a.H, KQ))
        return MEMOROID_ERR_CUDA;
    st = launch_seg_carry<D, false, NORM, false>(a, pl, meta, info, carry, p.map_k, p.map_v, a.S0, hdr, stream);
    if (st != MEMOROID_OK) return st;
    p.den = NORM ? a.den : nullptr;
    p.q = static_cast<const uint16_t*>(a.q);
    p.k = static_cast<const uint16_t*>(a.k);
    p.v = static_cast<const uint16_t*>(a.v);
    p.S0 = a.S0;
    p.y = a.y;
    p.meta = meta;
    p.carry = carry;
    p.S_last = a.S_last;
    p.hdr = hdr;
    p.B = a.B;
    p.L = a.L;
    p.H = a.H;
    p.n_tiles = pl.n_tiles;
    p.tps = pl.tps;
    p.G = static_cast<int>(pl.G);
    p.wait_ns = debug_knobs().wait_ns;
    p.fail_cta = debug_knobs().withhold_ticket;
    p.map_zq = p.map_q;  // not read by the forward
    p.dlam_f = nullptr;
    p.states = nullptr;
    p.fold_col = -1;
    if (set_smem(fwd_kernel<D, false, NORM>, FwdSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (launch_after(fwd_kernel<D, false, NORM>, dim3(static_cast<unsigned>(a.B * a.H * pl.G)), dim3(kThreads), FwdSmem<D>::BYTES, stream, p) !=
        cudaSuccess)
        return MEMOROID_ERR_CUDA;
    return MEMOROID_OK;
}
template <int D, bool HALF_OUT = false, bool NORM = false>
memoroid_status_t launch_bwd_d(const Args& a, const Plan& pl, const Layout& ly, cudaStream_t stream) {
    unsigned char* ws = static_cast<unsigned char*>(a.workspace);
    TileMeta* meta = reinterpret_cast<TileMeta*>(ws + ly.meta);
    float2* info = reinterpret_cast<float2*>(ws + ly.info);
    float* carry_f = reinterpret_cast<float*>(ws + ly.carry_f);
    float* carry_r = reinterpret_cast<float*>(ws + ly.carry_r);
    // the bf16 operand copy of grad_y, unless the caller passes grad_y in bf16 already
    const uint16_t* dy16 = a.grad_y16 != nullptr ? a.grad_y16 : reinterpret_cast<uint16_t*>(ws + ly.dy16);
    uint16_t* states = reinterpret_cast<uint16_t*>(ws + ly.states);
    float* dlam_f = reinterpret_cast<float*>(ws + ly.dlam_f);
    float* gpart = reinterpret_cast<float*>(ws + ly.gpart);
    uint32_t* hdr = reinterpret_cast<uint32_t*>(ws);
    memoroid_status_t st = launch_prep(a, pl, meta, stream);
    if (st != MEMOROID_OK) return st;

    if (a.grad_y16 == nullptr) {
        const int64_t n8 = a.B * a.L * a.H * D / 8;
        const int64_t cblocks = min((n8 + 255) / 256, static_cast<int64_t>(kTargetCtas) * 16);
        if (launch_after(to_bf16_kernel, dim3(static_cast<unsigned>(cblocks)), dim3(256), 0, stream, a.grad_y,
                         reinterpret_cast<uint16_t*>(ws + ly.dy16), n8) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
    }

    // the operand maps of pass R, also read by the segment summaries
    BwdParams r;
    constexpr int BKV = NORM ? 64 : D;  // channels of q, k, v in memory (the normalised path: unpadded)
    if (!tile_map(&r.map_q, a.q, a.B, a.L, a.H, BKV) || !tile_map(&r.map_k, a.k, a.B, a.L, a.H, BKV) ||
        !tile_map(&r.map_v, a.v, a.B, a.L, a.H, BKV) || !tile_map(&r.map_dy, dy16, a.B, a.L, a.H, D) ||
        !tile_map_y(&r.map_dk, a.dk, a.B, a.L, a.H, HALF_OUT ? 64 : D) ||
        !tile_map_y(&r.map_dv, a.dv, a.B, a.L, a.H, HALF_OUT ? 64 : D))
        return MEMOROID_ERR_CUDA;
    // the forward states entering the segments (for pass F) and the reverse
    // states entering them from the right (for pass R)
    st = launch_seg_carry<D, false, NORM, NORM>(a, pl, meta, info, carry_f, r.map_k, r.map_v, a.S0, hdr, stream);
    if (st != MEMOROID_OK) return st;
    st = launch_seg_carry<D, true, NORM, NORM>(a, pl, meta, info, carry_r, r.map_q, r.map_dy, a.dS_last, hdr, stream);
    if (st != MEMOROID_OK) return st;

    // pass F: dq = S dy, with (q, k, v) -> (dy, v, k)
    FwdParams f;
    if (!tile_map(&f.map_q, dy16, a.B, a.L, a.H, D) || !tile_map(&f.map_k, a.v, a.B, a.L, a.H, BKV) ||
        !tile_map(&f.map_v, a.k, a.B, a.L, a.H, BKV) ||
        !tile_map_y(&f.map_y, a.dq, a.B, a.L, a.H, HALF_OUT ? 64 : D) || !tile_map(&f.map_zq, a.q, a.B, a.L, a.H, BKV))
        return MEMOROID_ERR_CUDA;
    f.den = nullptr;
    f.q = dy16;
    f.k = static_cast<const uint16_t*>(a.v);
    f.v = static_cast<const uint16_t*>(a.k);
    f.S0 = a.S0;
    f.y = a.dq;
    f.meta = meta;
    f.carry = carry_f;
    f.S_last = nullptr;
    f.hdr = hdr;
    f.B = a.B;
    f.L = a.L;
    f.H = a.H;
    f.n_tiles = pl.n_tiles;
    f.tps = pl.tps;
    f.G = static_cast<int>(pl.G);
    f.wait_ns = debug_knobs().wait_ns;
    f.fail_cta = debug_knobs().withhold_ticket;
    f.dlam_f = dlam_f;
    f.states = states;
    f.fold_col = static_cast<int>(a.fold_col);
    // the normalised backward folds its sum channel (fold_col); the plain one never does
    if constexpr (NORM) {
        if (a.fold_col < 0) return MEMOROID_ERR_UNSUPPORTED;
        if (set_smem(fwd_kernel<D, true, NORM, HALF_OUT, true>, FwdSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
        if (launch_after(fwd_kernel<D, true, NORM, HALF_OUT, true>, dim3(static_cast<unsigned>(a.B * a.H * pl.G)), dim3(kThreads), FwdSmem<D>::BYTES,
                         stream, f) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
    } else if (a.fold_col >= 0) {
        if (set_smem(fwd_kernel<D, true, false, HALF_OUT, true>, FwdSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
        if (launch_after(fwd_kernel<D, true, false, HALF_OUT, true>, dim3(static_cast<unsigned>(a.B * a.H * pl.G)), dim3(kThreads), FwdSmem<D>::BYTES,
                         stream, f) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
    } else {
        if (set_smem(fwd_kernel<D, true, false, HALF_OUT>, FwdSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
        if (launch_after(fwd_kernel<D, true, false, HALF_OUT>, dim3(static_cast<unsigned>(a.B * a.H * pl.G)), dim3(kThreads), FwdSmem<D>::BYTES, stream,
                         f) != cudaSuccess)
            return MEMOROID_ERR_CUDA;
    }
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;

    // pass R: dk, dv, dgamma, dS0
    r.q = static_cast<const uint16_t*>(a.q);
    r.k = static_cast<const uint16_t*>(a.k);
    r.v = static_cast<const uint16_t*>(a.v);
    r.dy = dy16;
    r.gamma = a.gamma;
    r.gamma_per_step = a.gamma_per_step;
    r.dS_last = a.dS_last;
    r.dk = a.dk;
    r.dv = a.dv;
    r.dgamma = (a.dgamma != nullptr && a.gamma_per_step) ? a.dgamma : nullptr;
    r.gpart = (a.dgamma != nullptr && !a.gamma_per_step) ? gpart : nullptr;
    r.dS0 = a.dS0;
    r.meta = meta;
    r.carry = carry_r;
    r.dlam_f = dlam_f;
    r.states = states;
    r.hdr = hdr;
    r.B = a.B;
    r.L = a.L;
    r.H = a.H;
    r.n_tiles = pl.n_tiles;
    r.tps = pl.tps;
    r.G = static_cast<int>(pl.G);
    r.wait_ns = debug_knobs().wait_ns;
    r.fail_cta = debug_knobs().withhold_ticket;
    if (set_smem(bwd_kernel<D, HALF_OUT, NORM>, BwdSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
    if (launch_after(bwd_kernel<D, HALF_OUT, NORM>, dim3(static_cast<unsigned>(a.B * a.H * pl.G)), dim3(kRThreads), BwdSmem<D>::BYTES, stream, r) !=
        cudaSuccess)
        return MEMOROID_ERR_CUDA;
    if (r.gpart != nullptr) {
        if (launch_after(dgamma_head_kernel, dim3(static_cast<unsigned>((a.H + 127) / 128)), dim3(128), 0, stream,
                         static_cast<const float*>(gpart), a.gamma, a.dgamma, a.B, a.H, static_cast<int>(pl.G)) !=
            cudaSuccess)
            return MEMOROID_ERR_CUDA;
    }
    return MEMOROID_OK;
}
}  // namespace

size_t workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t D) { return make_layout(B, L, H, D).total; }
size_t fwd_workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t D) { return make_layout(B, L, H, D).fwd_total; }

int kernels_per_call(int64_t B, int64_t L, int64_t H, int backward, int with_dgamma_per_head) {
    if (B == 0 || L == 0 || H == 0) return 0;
    // the segment summary and carry kernels run once per direction when there are several segments
    const int carry = make_plan(B, L, H).G > 1 ? 2 : 0;
    if (!backward) return 2 + carry;  // meta, forward
    return 4 + 2 * carry + (with_dgamma_per_head ? 1 : 0);  // meta, bf16 copy, pass F, pass R
}

memoroid_status_t launch_bwd(const Args& a, cudaStream_t stream) {
    const Plan pl = make_plan(a.B, a.L, a.H);
    if (a.B * a.H * pl.G >= 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;  // one CTA per segment chain
    if (a.out_cols != 0 && !(a.out_cols == 64 && a.D == 128)) return MEMOROID_ERR_UNSUPPORTED;
    if (a.norm && (a.out_cols != 64 || a.grad_y16 == nullptr)) return MEMOROID_ERR_UNSUPPORTED;
    if (a.D != 64 && a.D != 128) return MEMOROID_ERR_UNSUPPORTED;
    if (cudaMemsetAsync(a.workspace, 0, kHeaderBytes, stream) != cudaSuccess) return MEMOROID_ERR_CUDA;
    const Layout ly = make_layout(a.B, a.L, a.H, a.D);
    if (a.norm) return launch_bwd_d<128, true, true>(a, pl, ly, stream);
    if (a.out_cols == 64) return launch_bwd_d<128, true>(a, pl, ly, stream);
    if (a.D == 64) return launch_bwd_d<64>(a, pl, ly, stream);
    if (a.D == 128) return launch_bwd_d<128>(a, pl, ly, stream);
    return MEMOROID_ERR_UNSUPPORTED;
}

memoroid_status_t launch_fwd(const Args& a, cudaStream_t stream) {
    if (a.norm && a.D != 128) return MEMOROID_ERR_UNSUPPORTED;
    const Plan pl = make_plan(a.B, a.L, a.H);
    if (a.B * a.H * pl.G >= 0x7fffffffLL) return MEMOROID_ERR_UNSUPPORTED;  // one CTA per segment chain
    if (a.D != 64 && a.D != 128) return MEMOROID_ERR_UNSUPPORTED;
    if (cudaMemsetAsync(a.workspace, 0, kHeaderBytes, stream) != cudaSuccess) return MEMOROID_ERR_CUDA;
    const Layout ly = make_layout(a.B, a.L, a.H, a.D);
    if (a.norm) return launch_fwd_d<128, true>(a, pl, ly, stream);
    if (a.D == 64) return launch_fwd_d<64>(a, pl, ly, stream);
    if (a.D == 128) return launch_fwd_d<128>(a, pl, ly, stream);
    return MEMOROID_ERR_UNSUPPORTED;
}

}  // namespace la
}  // namespace memoroid

