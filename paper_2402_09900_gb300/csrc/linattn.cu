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
// Parallel structure: each CTA owns one (tape, head, segment) and walks the
// segment's tiles in order, carrying the state in TMEM.  Segments start from
// a zero state; a carry kernel then folds the segment end states in tape
// order, and a fix-up kernel adds each segment's incoming state to the outputs
// of its steps before its first start.  The reset makes the fold exact: a
// start inside a segment cuts every dependence on earlier segments.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"
#include "ptx.cuh"

namespace memoroid {
namespace la {

using namespace ptx;

constexpr int T = 128;         // steps per tile = the M of the tile contractions
constexpr int kThreads = 256;  // 8 warps: warp w reads TMEM lane quarter w % 4, column half w / 4
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
    size_t meta, seg_decay, seg_state, total;
};

Layout make_layout(int64_t B, int64_t L, int64_t H, int64_t D) {
    const Plan pl = make_plan(B, L, H);
    Layout ly;
    size_t off = kHeaderBytes;
    ly.meta = off;
    off = align_up(off + static_cast<size_t>(B * H * pl.n_tiles) * sizeof(TileMeta), 256);
    ly.seg_decay = off;
    off = align_up(off + static_cast<size_t>(B * H * pl.G) * sizeof(float), 256);
    ly.seg_state = off;
    off = align_up(off + static_cast<size_t>(B * H * pl.G) * D * D * sizeof(float), 256);
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
            // gamma = 0 gives a weight of at most 2^-126 instead of 0
            l = fmaxf(log2f(g), -126.f);
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

// Copies rows [0, nvalid) of a [T x D] bf16 tile (row r at src + r * row_stride
// elements) into the core-matrix layout with 16-byte cp.async; rows past
// nvalid are zero-filled.  32 consecutive chunks of a warp cover 8 rows x 4
// chunks: 64 contiguous global bytes per row, conflict-free shared stores.
template <int D>
__device__ __forceinline__ void load_tile_async(uint32_t dst, const uint16_t* __restrict__ src, int64_t row_stride,
                                                int nvalid, int tid) {
    constexpr int CPR = D / 8;
    constexpr int NCH = T * CPR;
#pragma unroll
    for (int e = tid; e < NCH; e += kThreads) {
        const int blk = e >> 5, ln = e & 31;
        const int rg = blk / (CPR / 4), cq = blk % (CPR / 4);
        const int r = rg * 8 + (ln & 7), c = cq * 4 + (ln >> 3);
        const bool ok = r < nvalid;
        const uint16_t* s = src + (ok ? static_cast<int64_t>(r) * row_stride + c * 8 : 0);
        cp_async16(dst + rg * (D * 16) + c * 128 + (ln & 7) * 16, s, ok);
    }
}

__device__ __forceinline__ void load_meta_async(uint32_t dst, const TileMeta* src, int tid) {
    constexpr int N = sizeof(TileMeta) / 16;
    if (tid < N) cp_async16(dst + tid * 16, reinterpret_cast<const unsigned char*>(src) + tid * 16, true);
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
    static constexpr bool PM_IN_Q = TILE >= PM;  // d = 128: the masked scores overwrite Q
    static constexpr int STAGE = 3 * TILE;       // Q, K, V
    static constexpr int OFF_PM = PM_IN_Q ? 0 : 2 * STAGE;
    static constexpr int OFF_SB = 2 * STAGE + (PM_IN_Q ? 0 : PM);
    static constexpr int OFF_META = OFF_SB + D * D * 2;
    static constexpr int OFF_BAR = OFF_META + 4 * static_cast<int>(sizeof(TileMeta));
    static constexpr int BYTES = OFF_BAR + 32;
    // TMEM columns: scores P, intra output, inter output, state S
    static constexpr uint32_t COL_P = 0, COL_YA = 128, COL_YI = 128 + D, COL_S = 128 + 2 * D;
    static constexpr uint32_t TMEM_COLS = 512;
    static_assert(COL_S + D <= TMEM_COLS, "tensor memory budget");
};

struct FwdParams {
    const uint16_t* q;
    const uint16_t* k;
    const uint16_t* v;
    const float* S0;
    float* y;
    const TileMeta* meta;
    float* seg_state;
    float* seg_decay;
    uint32_t* hdr;
    int64_t B, L, H, n_tiles, tps;
    int G;
    uint64_t wait_ns;
};

// Thread -> (row, first column) of a D x D state accumulator in TMEM.  With
// M = 128 the row is the TMEM lane; with M = 64 rows 16q..16q+15 sit in lanes
// 32q..32q+15 and the upper 16 lanes of each quarter hold nothing.
template <int D>
__device__ __forceinline__ int state_row(int quarter, int lane) {
    if (D == 128) return 32 * quarter + lane;
    return lane < 16 ? 16 * quarter + lane : -1;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) fwd_kernel(const FwdParams p) {
    using S = FwdSmem<D>;
    extern __shared__ __align__(1024) unsigned char smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int quarter = warp & 3, half = warp >> 2;
    const int64_t bh = blockIdx.x / p.G;
    const int g = static_cast<int>(blockIdx.x % p.G);
    const int64_t b = bh / p.H, h = bh % p.H;
    const int64_t tile0 = static_cast<int64_t>(g) * p.tps;
    const int nt = static_cast<int>(min(p.tps, p.n_tiles - tile0));
    const int64_t row_stride = p.H * D;  // elements between consecutive steps of one head

    uint64_t* bar1 = reinterpret_cast<uint64_t*>(smem + S::OFF_BAR);
    uint64_t* bar2 = bar1 + 1;
    uint32_t* tslot = reinterpret_cast<uint32_t*>(bar1 + 2);
    TileMeta* metas = reinterpret_cast<TileMeta*>(smem + S::OFF_META);
    const uint32_t sbase = smem_addr(smem);
    const uint32_t sSb = sbase + S::OFF_SB;
    const TileMeta* gmeta = p.meta + bh * p.n_tiles + tile0;

    auto stage_q = [&](int s) { return sbase + s * S::STAGE; };
    auto stage_k = [&](int s) { return sbase + s * S::STAGE + S::TILE; };
    auto stage_v = [&](int s) { return sbase + s * S::STAGE + 2 * S::TILE; };
    auto stage_pm = [&](int s) { return S::PM_IN_Q ? stage_q(s) : sbase + S::OFF_PM; };
    auto issue_tile = [&](int c, int s) {
        const int64_t t0 = (tile0 + c) * T;
        const int nvalid = static_cast<int>(min(static_cast<int64_t>(T), p.L - t0));
        const int64_t off = ((b * p.L + t0) * p.H + h) * D;
        load_tile_async<D>(stage_q(s), p.q + off, row_stride, nvalid, tid);
        load_tile_async<D>(stage_k(s), p.k + off, row_stride, nvalid, tid);
        load_tile_async<D>(stage_v(s), p.v + off, row_stride, nvalid, tid);
    };

    if (tid == 0) {
        mbar_init(bar1, 1);
        mbar_init(bar2, 1);
        fence_mbar_init();
    }
    if (warp == 0) tc::alloc(tslot, S::TMEM_COLS);

    issue_tile(0, 0);
    load_meta_async(smem_addr(&metas[0]), gmeta, tid);
    if (nt > 1) load_meta_async(smem_addr(&metas[1]), gmeta + 1, tid);
    cp_async_commit();
    cp_async_wait<0>();
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tm = *tslot;

    const int srow = state_row<D>(quarter, lane);
    constexpr int SC = D / 2;  // state columns per thread
    const uint32_t lane_base = tm + (static_cast<uint32_t>(32 * quarter) << 16);

    // ---- incoming state: S0 for the first segment of a tape ----
    bool have_prev = false, have_state = false;
    if (g == 0 && p.S0 != nullptr && metas[0].first_start != 0) {
        have_prev = true;
        const bool scale = metas[0].has_start == 0;
        have_state = scale;
        const float a0 = metas[0].a;
        const float* s0 = p.S0 + bh * D * D;
#pragma unroll
        for (int cc = 0; cc < SC / 16; ++cc) {
            const int j0 = half * SC + cc * 16;
            float v[16];
            if (srow >= 0) {
#pragma unroll
                for (int x = 0; x < 16; x += 4) {
                    const float4 f = *reinterpret_cast<const float4*>(s0 + srow * D + j0 + x);
                    v[x] = f.x;
                    v[x + 1] = f.y;
                    v[x + 2] = f.z;
                    v[x + 3] = f.w;
                }
                uint4 w0, w1;
                w0.x = pack_bf16x2(v[0], v[1]);
                w0.y = pack_bf16x2(v[2], v[3]);
                w0.z = pack_bf16x2(v[4], v[5]);
                w0.w = pack_bf16x2(v[6], v[7]);
                w1.x = pack_bf16x2(v[8], v[9]);
                w1.y = pack_bf16x2(v[10], v[11]);
                w1.z = pack_bf16x2(v[12], v[13]);
                w1.w = pack_bf16x2(v[14], v[15]);
                *reinterpret_cast<uint4*>(smem + S::OFF_SB + core_off(srow, j0, D)) = w0;
                *reinterpret_cast<uint4*>(smem + S::OFF_SB + core_off(srow, j0 + 8, D)) = w1;
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

    constexpr uint32_t ID_QS = tc::idesc_bf16(128, D, false, true);
    constexpr uint32_t ID_QK = tc::idesc_bf16(128, T, false, false);
    constexpr uint32_t ID_PV = tc::idesc_bf16(128, D, false, true);
    constexpr uint32_t ID_KV = tc::idesc_bf16(D, D, true, true);

    float aprod = 1.f;
    bool failed = false;
    for (int c = 0; c < nt; ++c) {
        const int s = c & 1;
        const TileMeta& mc = metas[c & 3];
        if (c + 1 < nt) {
            issue_tile(c + 1, s ^ 1);
            if (c + 2 < nt) load_meta_async(smem_addr(&metas[(c + 2) & 3]), gmeta + c + 2, tid);
        }
        cp_async_commit();
        cp_async_wait<1>();
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        tc::fence_after();

        // ---- P = Q K^T and (with an incoming state) Y_inter = Q S_prev ----
        if (tid == 0) {
            const uint32_t sq = stage_q(s), sk = stage_k(s);
            if (have_prev) {
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk)
                    tc::mma(tm + S::COL_YI, desc_kmajor(sq, D, kk), desc_mnmajor(sSb, D, kk), ID_QS, kk > 0);
            }
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                tc::mma(tm + S::COL_P, desc_kmajor(sq, D, kk), desc_kmajor(sk, D, kk), ID_QK, kk > 0);
            tc::commit(bar1);
        }
        bool ok = wait_mbar(bar1, c & 1, p.wait_ns);
        if (__syncthreads_or(!ok)) {
            failed = true;
            break;
        }
        tc::fence_after();

        // ---- mask: Pm[t][r] = [seg_t <= r <= t] exp2(lam2_t - lam2_r) P[t][r] ----
        {
            const int t = 32 * quarter + lane;
            const float lt = mc.lam2[t];
            const int st = mc.seg[t];
            unsigned char* pm = smem + (stage_pm(s) - sbase);
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
                const int r0 = half * 64 + cc * 16;
                float v[16];
                tc::ld16(lane_base + S::COL_P + r0, v);
#pragma unroll
                for (int x = 0; x < 16; ++x) {
                    const int r = r0 + x;
                    const bool in = r <= t && r >= st;
                    v[x] = in ? v[x] * exp2f(lt - mc.lam2[r]) : 0.f;
                }
                uint4 w0, w1;
                w0.x = pack_bf16x2(v[0], v[1]);
                w0.y = pack_bf16x2(v[2], v[3]);
                w0.z = pack_bf16x2(v[4], v[5]);
                w0.w = pack_bf16x2(v[6], v[7]);
                w1.x = pack_bf16x2(v[8], v[9]);
                w1.y = pack_bf16x2(v[10], v[11]);
                w1.z = pack_bf16x2(v[12], v[13]);
                w1.w = pack_bf16x2(v[14], v[15]);
                *reinterpret_cast<uint4*>(pm + core_off(t, r0, T)) = w0;
                *reinterpret_cast<uint4*>(pm + core_off(t, r0 + 8, T)) = w1;
            }
        }
        // ---- K~[r] = exp2(lam2_end - lam2_r) K[r] for rows of the last episode ----
        {
            unsigned char* kt = smem + (stage_k(s) - sbase);
            const float lend = mc.lam2[T - 1];
            const int ls = mc.last_start;
            constexpr int NCH = T * D / 8;
#pragma unroll
            for (int e = tid; e < NCH; e += kThreads) {
                // e enumerates 16-byte chunks in memory order: a row group of 8
                // rows holds D chunks, 8 per core matrix, one per row
                const int r = (e / D) * 8 + (e & 7);
                const float w = r >= ls ? exp2f(lend - mc.lam2[r]) : 0.f;
                if (w != 1.f) {
                    uint4 u = *reinterpret_cast<uint4*>(kt + e * 16);
                    float2 f;
                    f = unpack_bf16x2(u.x);
                    u.x = pack_bf16x2(f.x * w, f.y * w);
                    f = unpack_bf16x2(u.y);
                    u.y = pack_bf16x2(f.x * w, f.y * w);
                    f = unpack_bf16x2(u.z);
                    u.z = pack_bf16x2(f.x * w, f.y * w);
                    f = unpack_bf16x2(u.w);
                    u.w = pack_bf16x2(f.x * w, f.y * w);
                    *reinterpret_cast<uint4*>(kt + e * 16) = u;
                }
            }
        }
        tc::fence_smem_to_async();
        tc::fence_before();
        __syncthreads();
        tc::fence_after();

        // ---- Y_intra = Pm V and S = a S + K~^T V ----
        if (tid == 0) {
            const uint32_t spm = stage_pm(s), sk = stage_k(s), sv = stage_v(s);
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_YA, desc_kmajor(spm, T, kk), desc_mnmajor(sv, D, kk), ID_PV, kk > 0);
            const bool acc = have_state && mc.has_start == 0;
#pragma unroll
            for (int kk = 0; kk < T / 16; ++kk)
                tc::mma(tm + S::COL_S, desc_mnmajor(sk, D, kk), desc_mnmajor(sv, D, kk), ID_KV, acc || kk > 0);
            tc::commit(bar2);
            aprod *= mc.a;
        }
        ok = wait_mbar(bar2, c & 1, p.wait_ns);
        if (__syncthreads_or(!ok)) {
            failed = true;
            break;
        }
        tc::fence_after();

        // ---- y = Y_intra + w_in * Y_inter ----
        {
            const int t = 32 * quarter + lane;
            const int64_t tg = (tile0 + c) * T + t;
            const bool valid = tg < p.L;
            const float w_in = (have_prev && mc.seg[t] < 0) ? exp2f(mc.lam2[t]) : 0.f;
            float* yrow = p.y + ((b * p.L + tg) * p.H + h) * D;
#pragma unroll
            for (int cc = 0; cc < D / 2 / 16; ++cc) {
                const int j0 = half * (D / 2) + cc * 16;
                float ya[16];
                tc::ld16(lane_base + S::COL_YA + j0, ya);
                if (have_prev) {
                    float yi[16];
                    tc::ld16(lane_base + S::COL_YI + j0, yi);
#pragma unroll
                    for (int x = 0; x < 16; ++x) ya[x] = fmaf(w_in, yi[x], ya[x]);
                }
                if (valid) {
#pragma unroll
                    for (int x = 0; x < 16; x += 4)
                        *reinterpret_cast<float4*>(yrow + j0 + x) = make_float4(ya[x], ya[x + 1], ya[x + 2], ya[x + 3]);
                }
            }
        }
        // ---- state: bf16 copy for the next tile, decay by the next tile's a ----
        if (c + 1 < nt) {
            const TileMeta& mn = metas[(c + 1) & 3];
            const bool scale = mn.has_start == 0 && mn.a != 1.f;
            const float an = mn.a;
#pragma unroll
            for (int cc = 0; cc < SC / 16; ++cc) {
                const int j0 = half * SC + cc * 16;
                float v[16];
                tc::ld16(lane_base + S::COL_S + j0, v);
                if (srow >= 0) {
                    uint4 w0, w1;
                    w0.x = pack_bf16x2(v[0], v[1]);
                    w0.y = pack_bf16x2(v[2], v[3]);
                    w0.z = pack_bf16x2(v[4], v[5]);
                    w0.w = pack_bf16x2(v[6], v[7]);
                    w1.x = pack_bf16x2(v[8], v[9]);
                    w1.y = pack_bf16x2(v[10], v[11]);
                    w1.z = pack_bf16x2(v[12], v[13]);
                    w1.w = pack_bf16x2(v[14], v[15]);
                    *reinterpret_cast<uint4*>(smem + S::OFF_SB + core_off(srow, j0, D)) = w0;
                    *reinterpret_cast<uint4*>(smem + S::OFF_SB + core_off(srow, j0 + 8, D)) = w1;
                }
                if (scale) {
#pragma unroll
                    for (int x = 0; x < 16; ++x) v[x] *= an;
                    tc::st16(lane_base + S::COL_S + j0, v);
                }
            }
        } else {
            float* dst = p.seg_state + (bh * p.G + g) * D * D;
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
        tc::fence_before();
        have_prev = true;
        have_state = true;
    }
    if (failed) {
        if (tid == 0) record_error(p.hdr, DEV_MMA_TIMEOUT);
        cp_async_wait<0>();
    }
    if (tid == 0) p.seg_decay[bh * p.G + g] = failed ? 0.f : aprod;
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 0) tc::dealloc(tm, S::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// kernel 3: fold the segment end states in tape order (elementwise over dk x dv)
// ---------------------------------------------------------------------------
// On exit slot g holds the true state at the end of segment g, i.e. the
// incoming state of segment g + 1:  C_{g+1} = A_g C_g + S_loc_g, C_1 = S_loc_0.
__global__ void __launch_bounds__(256) carry_fwd_kernel(float* __restrict__ seg_state,
                                                        const float* __restrict__ seg_decay, float* __restrict__ S_last,
                                                        int G, int64_t DD) {
    const int64_t bh = blockIdx.y;
    const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (e >= DD) return;
    float* st = seg_state + bh * G * DD + e;
    float prev = st[0];
    for (int g = 1; g < G; ++g) {
        prev = fmaf(seg_decay[bh * G + g], prev, st[static_cast<int64_t>(g) * DD]);
        st[static_cast<int64_t>(g) * DD] = prev;
    }
    if (S_last != nullptr) S_last[bh * DD + e] = prev;
}

// ---------------------------------------------------------------------------
// kernel 4: add each segment's incoming state to its steps before its first start
// ---------------------------------------------------------------------------
//   y_t += (prod_{j = segment begin}^{t} gamma_j) C_g^T q_t
template <int D>
__global__ void __launch_bounds__(kThreads, 1) fix_fwd_kernel(const uint16_t* __restrict__ q, float* __restrict__ y,
                                                             const TileMeta* __restrict__ meta,
                                                             const float* __restrict__ seg_state, int64_t L, int64_t H,
                                                             int64_t n_tiles, int64_t tps, int G) {
    extern __shared__ __align__(16) float qs[];  // [T][D] fp32
    constexpr int NG = kThreads / D;
    const int tid = threadIdx.x, grp = tid / D, j = tid % D;
    const int64_t bh = blockIdx.x / (G - 1);
    const int g = static_cast<int>(blockIdx.x % (G - 1)) + 1;
    const int64_t b = bh / H, h = bh % H;
    const float* C = seg_state + (bh * G + g - 1) * D * D;
    float cj[D];
#pragma unroll
    for (int i = 0; i < D; ++i) cj[i] = C[i * D + j];
    const int64_t tile0 = static_cast<int64_t>(g) * tps;
    const int64_t tile_end = min(n_tiles, tile0 + tps);
    float cum = 1.f;
    for (int64_t tile = tile0; tile < tile_end; ++tile) {
        const TileMeta* m = meta + bh * n_tiles + tile;
        const int64_t t0 = tile * T;
        const int nvalid = static_cast<int>(min(static_cast<int64_t>(T), L - t0));
        const int hs = m->has_start;
        const int nfix = hs ? min(m->first_start, nvalid) : nvalid;
        __syncthreads();
        for (int e = tid; e < nfix * (D / 8); e += kThreads) {
            const int r = e / (D / 8), c8 = e % (D / 8);
            const uint4 u = *reinterpret_cast<const uint4*>(q + ((b * L + t0 + r) * H + h) * D + c8 * 8);
            float2 f0 = unpack_bf16x2(u.x), f1 = unpack_bf16x2(u.y), f2 = unpack_bf16x2(u.z), f3 = unpack_bf16x2(u.w);
            float4* dst = reinterpret_cast<float4*>(qs + r * D + c8 * 8);
            dst[0] = make_float4(f0.x, f0.y, f1.x, f1.y);
            dst[1] = make_float4(f2.x, f2.y, f3.x, f3.y);
        }
        __syncthreads();
        for (int r = grp; r < nfix; r += NG) {
            const float w = cum * exp2f(m->lam2[r]);
            float acc = 0.f;
            const float4* qr = reinterpret_cast<const float4*>(qs + r * D);
#pragma unroll
            for (int i4 = 0; i4 < D / 4; ++i4) {
                const float4 qq = qr[i4];
                acc = fmaf(cj[4 * i4], qq.x, acc);
                acc = fmaf(cj[4 * i4 + 1], qq.y, acc);
                acc = fmaf(cj[4 * i4 + 2], qq.z, acc);
                acc = fmaf(cj[4 * i4 + 3], qq.w, acc);
            }
            float* yp = y + ((b * L + t0 + r) * H + h) * D + j;
            *yp = fmaf(w, acc, *yp);
        }
        if (hs) break;
        cum *= m->a;
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {
template <typename K>
cudaError_t set_smem(K kernel, int bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

template <int D>
memoroid_status_t launch_fwd_d(const Args& a, const Plan& pl, const Layout& ly, cudaStream_t stream) {
    unsigned char* ws = static_cast<unsigned char*>(a.workspace);
    TileMeta* meta = reinterpret_cast<TileMeta*>(ws + ly.meta);
    float* seg_decay = reinterpret_cast<float*>(ws + ly.seg_decay);
    float* seg_state = reinterpret_cast<float*>(ws + ly.seg_state);
    uint32_t* hdr = reinterpret_cast<uint32_t*>(ws);

    const int64_t n_meta_warps = a.B * a.H * pl.n_tiles;
    const int64_t meta_blocks = (n_meta_warps * 32 + 255) / 256;
    meta_kernel<<<static_cast<unsigned>(meta_blocks), 256, 0, stream>>>(a.gamma, a.gamma_per_step, a.start, a.B,
                                                                         a.L, a.H, pl.n_tiles, meta);
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;

    FwdParams p;
    p.q = static_cast<const uint16_t*>(a.q);
    p.k = static_cast<const uint16_t*>(a.k);
    p.v = static_cast<const uint16_t*>(a.v);
    p.S0 = a.S0;
    p.y = a.y;
    p.meta = meta;
    p.seg_state = seg_state;
    p.seg_decay = seg_decay;
    p.hdr = hdr;
    p.B = a.B;
    p.L = a.L;
    p.H = a.H;
    p.n_tiles = pl.n_tiles;
    p.tps = pl.tps;
    p.G = static_cast<int>(pl.G);
    p.wait_ns = debug_knobs().wait_ns;
    if (set_smem(fwd_kernel<D>, FwdSmem<D>::BYTES) != cudaSuccess) return MEMOROID_ERR_CUDA;
    fwd_kernel<D><<<static_cast<unsigned>(a.B * a.H * pl.G), kThreads, FwdSmem<D>::BYTES, stream>>>(p);
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;

    const int64_t DD = static_cast<int64_t>(D) * D;
    if (pl.G > 1 || a.S_last != nullptr) {
        dim3 grid(static_cast<unsigned>((DD + 255) / 256), static_cast<unsigned>(a.B * a.H));
        carry_fwd_kernel<<<grid, 256, 0, stream>>>(seg_state, seg_decay, a.S_last, static_cast<int>(pl.G), DD);
        if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    }
    if (pl.G > 1) {
        const int fix_smem = T * D * static_cast<int>(sizeof(float));
        if (set_smem(fix_fwd_kernel<D>, fix_smem) != cudaSuccess) return MEMOROID_ERR_CUDA;
        fix_fwd_kernel<D><<<static_cast<unsigned>(a.B * a.H * (pl.G - 1)), kThreads, fix_smem, stream>>>(
            p.q, a.y, meta, seg_state, a.L, a.H, pl.n_tiles, pl.tps, static_cast<int>(pl.G));
        if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    }
    return MEMOROID_OK;
}
}  // namespace

size_t workspace_bytes(int64_t B, int64_t L, int64_t H, int64_t D) { return make_layout(B, L, H, D).total; }

int kernels_per_call(int64_t B, int64_t L, int64_t H, int backward, int with_S_last) {
    (void)backward;
    if (B == 0 || L == 0 || H == 0) return 0;
    const Plan pl = make_plan(B, L, H);
    int n = 2;
    if (pl.G > 1 || with_S_last) ++n;
    if (pl.G > 1) ++n;
    return n;
}

memoroid_status_t launch_fwd(const Args& a, cudaStream_t stream) {
    if (cudaMemsetAsync(a.workspace, 0, kHeaderBytes, stream) != cudaSuccess) return MEMOROID_ERR_CUDA;
    const Plan pl = make_plan(a.B, a.L, a.H);
    const Layout ly = make_layout(a.B, a.L, a.H, a.D);
    if (a.D == 64) return launch_fwd_d<64>(a, pl, ly, stream);
    if (a.D == 128) return launch_fwd_d<128>(a, pl, ly, stream);
    return MEMOROID_ERR_UNSUPPORTED;
}

}  // namespace la
}  // namespace memoroid
