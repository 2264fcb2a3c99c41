// linattn_norm.cu -- the paper's Linear Transformer memoroid with its feature
// map and normalizer (Appendix "Linear Transformer"): the pair state
//   (X, x) . (X', x') = (X + X', x + x'),  f(o) = (phi(k) v^T, phi(k)),
//   y = X^T phi(q) / (x^T phi(q)),  phi(z) = 1 + ELU(z),
// decayed by gamma_t and reset at begin flags like the decayed memoroid of
// linattn.cu (gamma = 1 is the paper's model).
//
// Both halves of the state are one decayed outer-product state: with
//   q' = [phi(q), 0],  k' = [phi(k), 0],  v' = [v, 1, 1, 0]   (width 128)
// the state S' = sum decay k' v'^T holds X in its first d columns and x in
// columns d and d + 1, and y' = S'^T q' holds the numerator X^T phi(q) and
// the normalizer x^T phi(q).  So the tensor-core kernels of linattn.cu at
// d = 128 compute both, and this file adds the element-wise steps around
// them: building q', k', v' (and the padded states), the division, and in
// the backward the upstream gradient of the pair,
//   dy' = [g, hi, lo, 0],  g = bf16(dy / den),  hi + lo = -(g . y),
// then the chain rule through phi.  The gradient with respect to q is a
// difference of two large terms, X g and x (g . y), that cancel exactly at an
// episode's first step; so the normalizer term is formed from the bf16 values
// the tensor cores will use and carried as a pair of bf16 numbers (the second
// ones column of v'), which keeps the difference exact for the rounded
// upstream g.  The backward also works in another basis of the same bilinear
// form: phi(q) . phi(k) = phi(q) . psi(k) + sigma(q) with psi = phi - 1 = ELU
// and sigma(q) = sum_i phi(q)_i, i.e.
//   q'' = [phi(q), sigma_hi, sigma_lo, 0],  k'' = [psi(k), 1, 1, 0]
// (sigma as a bf16 pair).  bf16 holds psi(k) with a relative error where
// phi(k) = 1 + psi(k) loses the low bits of psi(k) next to the 1, and dq sums
// phi(k) against the cancelling terms above, so the rounding of phi(k) was
// the largest error in dq for nearly constant features (unit-norm keys).  In
// this basis the state S'' = sum decay k'' v'^T has the incoming (X, x) in its
// first d rows and sum decay v'^T in rows d and d + 1; dphi(q)_i = dq''_i +
// dq''_d (folded in the kernel), dq = dphi(q) (.) phi'(q), dk = dk''[:d] (.)
// phi'(k): for 64-channel heads the kernels' epilogues apply phi' (from the
// raw q and k tiles) and write the caller's gradients, otherwise a chain-rule
// pass does.  Heads of width d <= 120 (a multiple of 8) are supported.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"

namespace memoroid {
namespace lnorm {

namespace {

constexpr int kW = 128;  // width of the padded operands and states
constexpr int kCtas = 152 * 8;

// phi(z) = 1 + ELU(z), rounded to bf16 right after, so the SFU exponential
// (__expf, a few ulp of fp32) is exact enough; the fused forward of linattn.cu
// computes the same expression
__device__ __forceinline__ float phi(float z) { return z > 0.f ? 1.f + z : __expf(z); }
// phi'(z), also by the SFU exponential: the fused kernels' epilogues compute the
// same expression, so both paths give the same gradients bit for bit
__device__ __forceinline__ float dphi(float z) { return z > 0.f ? 1.f : __expf(z); }

struct Buffers {
    __nv_bfloat16 *q, *k, *v;  // [R, 128]
    float* y;                   // fwd: y' [R, 128]; bwd: dy' [R, 128]
    float *dq, *dk, *dv;        // bwd: [R, 128]
    float *S0, *S1, *S2;        // [B*H, 128, 128]: incoming state, outgoing state (or its gradient), dS0
    void* la;                   // the linear-attention workspace (at offset 0, so its header is ours)
    size_t la_bytes;
};

size_t la_bytes(int64_t B, int64_t L, int64_t H) { return align_up(la::workspace_bytes(B, L, H, kW), 256); }

Buffers carve(void* ws, int64_t B, int64_t L, int64_t H, bool backward) {
    unsigned char* p = static_cast<unsigned char*>(ws);
    const size_t R = static_cast<size_t>(B * L * H);
    Buffers b{};
    b.la = p;
    b.la_bytes = la_bytes(B, L, H);
    size_t o = b.la_bytes;
    auto take = [&](size_t bytes) {
        void* r = p + o;
        o = align_up(o + bytes, 256);
        return r;
    };
    b.q = static_cast<__nv_bfloat16*>(take(R * kW * 2));
    b.k = static_cast<__nv_bfloat16*>(take(R * kW * 2));
    b.v = static_cast<__nv_bfloat16*>(take(R * kW * 2));
    b.y = static_cast<float*>(take(R * kW * 4));
    if (backward) {
        b.dq = static_cast<float*>(take(R * kW * 4));
        b.dk = static_cast<float*>(take(R * kW * 4));
        b.dv = static_cast<float*>(take(R * kW * 4));
    }
    b.S0 = static_cast<float*>(take(static_cast<size_t>(B * H) * kW * kW * 4));
    b.S1 = static_cast<float*>(take(static_cast<size_t>(B * H) * kW * kW * 4));
    if (backward) b.S2 = static_cast<float*>(take(static_cast<size_t>(B * H) * kW * kW * 4));
    return b;
}

size_t total_bytes(int64_t B, int64_t L, int64_t H) {
    const size_t R = static_cast<size_t>(B * L * H);
    size_t o = la_bytes(B, L, H);
    const size_t st = static_cast<size_t>(B * H) * kW * kW * 4;
    for (size_t bytes : {R * kW * 2, R * kW * 2, R * kW * 2, R * kW * 4, R * kW * 4, R * kW * 4, R * kW * 4, st, st, st})
        o = align_up(o + bytes, 256);
    return o;
}

// psi(z) = ELU(z) = phi(z) - 1, rounded to bf16 right after (as phi)
__device__ __forceinline__ float psi(float z) { return z > 0.f ? z : __expf(z) - 1.f; }

// Forward: q' = [phi(q), 0], k' = [phi(k), 0], v' = [v, 1, 1, 0].  Backward
// (the basis above): q'' = [phi(q), sigma_hi, sigma_lo, 0], k'' = [psi(k), 1,
// 1, 0], v'.  One thread per 16-byte chunk (8 columns) of a padded row, the
// 16 chunks of a row in 16 consecutive lanes; sigma = unit sums of the bf16
// phi values in column order, then a fixed butterfly over the row's first 8
// chunks (the association the in-kernel construction of 64-channel heads
// uses, so both give the same bits), plus the sum of chunks 8.. (d > 64).
__global__ void __launch_bounds__(256) prep_kernel(const uint4* __restrict__ q, const uint4* __restrict__ k,
                                                   const uint4* __restrict__ v, int64_t R, int d, int backward,
                                                   uint4* __restrict__ qp, uint4* __restrict__ kp,
                                                   uint4* __restrict__ vp) {
    constexpr int CH = kW / 8;  // chunks per padded row
    const int in_chunks = d / 8;
    const int64_t n = R * CH;
    const int lane = threadIdx.x & 31;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    // warp-uniform loop: every lane takes part in the shuffles
    for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31); base < n; base += stride) {
        const int64_t g = base + lane;
        const bool live = g < n;
        const int c = static_cast<int>(g & (CH - 1));
        const int64_t r = g >> 4;
        uint4 oq = make_uint4(0u, 0u, 0u, 0u), ok = oq, ov = oq;
        float su = 0.f;
        if (live && c < in_chunks) {
            const int64_t src = r * in_chunks + c;
            oq = q[src];
            ok = k[src];
            ov = v[src];
            __nv_bfloat162* hq = reinterpret_cast<__nv_bfloat162*>(&oq);
            __nv_bfloat162* hk = reinterpret_cast<__nv_bfloat162*>(&ok);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float2 fq = __bfloat1622float2(hq[e]), fk = __bfloat1622float2(hk[e]);
                hq[e] = __floats2bfloat162_rn(phi(fq.x), phi(fq.y));
                hk[e] = backward ? __floats2bfloat162_rn(psi(fk.x), psi(fk.y))
                                 : __floats2bfloat162_rn(phi(fk.x), phi(fk.y));
                const float2 pq = __bfloat1622float2(hq[e]);
                su += pq.x;
                su += pq.y;
            }
        } else if (live && c == in_chunks) {
            reinterpret_cast<__nv_bfloat162*>(&ov)[0] = __floats2bfloat162_rn(1.f, 1.f);  // columns d, d + 1 of v'
            if (backward) reinterpret_cast<__nv_bfloat162*>(&ok)[0] = __floats2bfloat162_rn(1.f, 1.f);
        }
        su += __shfl_xor_sync(0xffffffffu, su, 1);
        su += __shfl_xor_sync(0xffffffffu, su, 2);
        su += __shfl_xor_sync(0xffffffffu, su, 4);
        // chunks 8.. (d > 64); for d <= 64 their sum is +0, which leaves the bits as they are
        const float sg = su + __shfl_xor_sync(0xffffffffu, su, 8);
        if (backward && live && c == in_chunks) {
            const float hi = __bfloat162float(__float2bfloat16_rn(sg));
            reinterpret_cast<__nv_bfloat162*>(&oq)[0] = __floats2bfloat162_rn(hi, sg - hi);
        }
        if (live) {
            qp[g] = oq;
            kp[g] = ok;
            vp[g] = ov;
        }
    }
}

// padded state from (S [d, d], z [d]) per (tape, head): S' = [[S, z, z2], [0]]
// with z2 = z (a state) or 0 (the gradient of an outgoing state, read from
// column d only); null inputs give zeros.  A gradient (dup = 0) is the one of
// the backward's basis, where the outgoing state is S''[:d] + S''[d]: its row d
// holds the column sums of rows 0..d-1 (summed in row order).
__global__ void __launch_bounds__(256) pad_state_kernel(const float* __restrict__ S, const float* __restrict__ z,
                                                        int64_t BH, int d, int dup, float* __restrict__ Sp) {
    const int64_t n = BH * kW * kW;
    for (int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; g < n;
         g += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int j = static_cast<int>(g % kW), i = static_cast<int>((g / kW) % kW);
        const int64_t m = g / (kW * kW);
        float val = 0.f;
        if (i < d && j < d && S != nullptr) val = S[(m * d + i) * d + j];
        else if (i < d && (j == d || (dup && j == d + 1)) && z != nullptr) val = z[m * d + i];
        else if (!dup && i == d && j < d && S != nullptr) {
            for (int i2 = 0; i2 < d; ++i2) val += S[(m * d + i2) * d + j];
        } else if (!dup && i == d && j == d && z != nullptr) {
            for (int i2 = 0; i2 < d; ++i2) val += z[m * d + i2];
        }
        Sp[g] = val;
    }
}

// (S, z) from a padded state: z = column d (a state), or columns d + d + 1
// (the gradient of an incoming state, whose z feeds both columns)
__global__ void __launch_bounds__(256) unpad_state_kernel(const float* __restrict__ Sp, int64_t BH, int d, int both,
                                                          float* __restrict__ S, float* __restrict__ z) {
    const int64_t n = BH * d * (d + 1);
    for (int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; g < n;
         g += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int j = static_cast<int>(g % (d + 1)), i = static_cast<int>((g / (d + 1)) % d);
        const int64_t m = g / (static_cast<int64_t>(d) * (d + 1));
        const float* row = Sp + (m * kW + i) * kW;
        if (j < d) {
            if (S != nullptr) S[(m * d + i) * d + j] = row[j];
        } else if (z != nullptr) {
            z[m * d + i] = both ? row[d] + row[d + 1] : row[d];
        }
    }
}

// y = y'[:d] / y'[d], den = y'[d]: one warp per row (lane l holds columns 4l..4l+3)
__global__ void __launch_bounds__(256) divide_kernel(const float4* __restrict__ yp, int64_t R, int d,
                                                     float* __restrict__ y, float* __restrict__ den) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    for (int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; r < R; r += nw) {
        const float4 a = yp[r * (kW / 4) + lane];
        // d is a multiple of 8: column d is component 0 of lane d / 4
        const float dn = __shfl_sync(0xffffffffu, a.x, d >> 2);
        const float inv = 1.f / dn;
        const float comp[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int j = 4 * lane + e;
            if (j < d) y[r * d + j] = comp[e] * inv;
        }
        if (lane == 0 && den != nullptr) den[r] = dn;
    }
}

__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// dy' = [g, hi, lo, 0] with g = bf16(dy / den) and hi + lo = -(g . y) (both
// bf16), written in bf16 (every value is one already) as the backward's
// tensor-core operand: one warp per row, lane l holding columns 4l .. 4l + 3
__global__ void __launch_bounds__(256) upstream_kernel(const float* __restrict__ dy, const float* __restrict__ y,
                                                       const float* __restrict__ den, int64_t R, int d,
                                                       uint2* __restrict__ dyp) {
    const int lane = threadIdx.x & 31;
    const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    for (int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; r < R; r += nw) {
        float g[4], dot = 0.f;
        const float inv = 1.f / den[r];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int j = 4 * lane + e;
            g[e] = 0.f;
            if (j < d) {
                g[e] = bf16_round(dy[r * d + j] * inv);
                dot = fmaf(g[e], y[r * d + j], dot);
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
        const float hi = bf16_round(-dot), lo = bf16_round(-dot - hi);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int j = 4 * lane + e;
            if (j == d) g[e] = hi;
            if (j == d + 1) g[e] = lo;
        }
        __nv_bfloat162 w0 = __floats2bfloat162_rn(g[0], g[1]), w1 = __floats2bfloat162_rn(g[2], g[3]);
        dyp[r * (kW / 4) + lane] = make_uint2(*reinterpret_cast<uint32_t*>(&w0), *reinterpret_cast<uint32_t*>(&w1));
    }
}

// dq = dq''[:d] (.) phi'(q) (dq'' with its sum channel already folded in),
// dk = dk''[:d] (.) phi'(k) (psi' = phi'), dv = dv'[:d] from
// padded gradients with rows of w4 float4s: one thread per 4 columns (16-byte
// loads and stores; 32-bit index arithmetic)
__global__ void __launch_bounds__(256) chain_kernel(const float4* __restrict__ dqp, const float4* __restrict__ dkp,
                                                    const float4* __restrict__ dvp, const uint2* __restrict__ q,
                                                    const uint2* __restrict__ k, uint32_t R, uint32_t d4, uint32_t w4,
                                                    float4* __restrict__ dq, float4* __restrict__ dk,
                                                    float4* __restrict__ dv) {
    const uint32_t n = R * d4;
    for (uint32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < n; g += gridDim.x * blockDim.x) {
        const uint32_t r = g / d4, c = g - r * d4;
        const uint32_t pp = r * w4 + c;
        const uint2 qb = q[g], kb = k[g];
        const float2 q0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qb.x));
        const float2 q1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qb.y));
        const float2 k0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kb.x));
        const float2 k1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kb.y));
        const float4 a = dqp[pp], bb = dkp[pp];
        dq[g] = make_float4(a.x * dphi(q0.x), a.y * dphi(q0.y), a.z * dphi(q1.x), a.w * dphi(q1.y));
        dk[g] = make_float4(bb.x * dphi(k0.x), bb.y * dphi(k0.y), bb.z * dphi(k1.x), bb.w * dphi(k1.y));
        dv[g] = dvp[pp];
    }
}

unsigned grid_for(int64_t n, int per_thread = 1) {
    const int64_t want = (n / per_thread + 255) / 256;
    return static_cast<unsigned>(want < 1 ? 1 : (want > kCtas ? kCtas : want));
}

}  // namespace

size_t workspace_bytes(int64_t B, int64_t L, int64_t H) { return total_bytes(B, L, H); }

int kernels_per_call(int64_t B, int64_t L, int64_t H, int64_t d, int backward, int with_dgamma_per_head,
                     int with_states) {
    if (B == 0 || L == 0 || H == 0) return 0;
    // prep, the linear-attention call, then the divide (forward) or the upstream
    // gradient and the chain rule (backward); with states: their padding and
    // unpadding.  64-channel heads (in the forward with y 16-byte aligned) run the
    // fused kernels: the forward is the linear-attention call alone, the backward
    // the upstream gradient and that call (operands built and the chain rule
    // applied in the kernels).
    const bool pad = debug_knobs().lnorm_padded != 0;
    const bool fused = d == 64 && !pad;
    // the backward hands its bf16 upstream gradient to the linear-attention call,
    // which then skips its own bf16 copy
    const int base = la::kernels_per_call(B, L, H, backward, with_dgamma_per_head) +
                     (backward ? (fused ? 1 : 3) - 1 : (fused ? 0 : 2));
    return base + (with_states ? (backward ? 3 : 2) : 0);
}

memoroid_status_t launch(const Args& a, cudaStream_t s) {
    const int64_t R = a.B * a.L * a.H, BH = a.B * a.H;
    const Buffers b = carve(a.workspace, a.B, a.L, a.H, a.backward);
    // the forward of 64-channel heads applies phi, the padding and the division
    // inside the tensor-core kernel (la::Args::norm); everything else goes
    // through the padded operands
    // (the backward of 64-channel heads also builds its operands in the kernels)
    // (the kernels' TMA stores write y, or dq, dk and dv, straight to the caller's
    // arrays: y must be 16-byte aligned, as the gradients always are)
    const bool fused = debug_knobs().lnorm_padded == 0 && a.d == 64 &&
                       (a.backward || (reinterpret_cast<uintptr_t>(a.y) & 15u) == 0);
    if (!fused)
        prep_kernel<<<grid_for(R * 16), 256, 0, s>>>(static_cast<const uint4*>(a.q), static_cast<const uint4*>(a.k),
                                                     static_cast<const uint4*>(a.v), R, static_cast<int>(a.d),
                                                     a.backward ? 1 : 0, reinterpret_cast<uint4*>(b.q),
                                                     reinterpret_cast<uint4*>(b.k), reinterpret_cast<uint4*>(b.v));
    // incoming state and (backward) outgoing-state gradient in the padded layout
    const bool s_in = a.S0 != nullptr || a.z0 != nullptr;
    const bool g_in = a.backward && (a.dS_last != nullptr || a.dz_last != nullptr);
    if (s_in)
        pad_state_kernel<<<grid_for(BH * kW * kW), 256, 0, s>>>(a.S0, a.z0, BH, static_cast<int>(a.d), 1, b.S0);
    if (g_in)
        pad_state_kernel<<<grid_for(BH * kW * kW), 256, 0, s>>>(a.dS_last, a.dz_last, BH, static_cast<int>(a.d), 0,
                                                                b.S1);
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    la::Args l{};
    l.q = b.q;
    l.k = b.k;
    l.v = b.v;
    l.gamma = a.gamma;
    l.gamma_per_step = a.gamma_per_step;
    l.start = a.start;
    l.S0 = s_in ? b.S0 : nullptr;
    l.B = a.B;
    l.L = a.L;
    l.H = a.H;
    l.D = kW;
    l.workspace = b.la;
    l.workspace_bytes = b.la_bytes;
    if (!a.backward) {
        l.S_last = (a.S_last != nullptr || a.z_last != nullptr) ? b.S1 : nullptr;
        if (fused) {
            l.q = a.q;
            l.k = a.k;
            l.v = a.v;
            l.y = a.y;
            l.den = a.den;
            l.norm = 1;
        } else {
            l.y = b.y;
        }
        const memoroid_status_t st = la::launch_fwd(l, s);
        if (st != MEMOROID_OK) return st;
        if (!fused)
            divide_kernel<<<grid_for(R * 32), 256, 0, s>>>(reinterpret_cast<const float4*>(b.y), R,
                                                           static_cast<int>(a.d), a.y, a.den);
        if (l.S_last != nullptr)
            unpad_state_kernel<<<grid_for(BH * a.d * (a.d + 1)), 256, 0, s>>>(b.S1, BH, static_cast<int>(a.d), 0,
                                                                               a.S_last, a.z_last);
        return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
    }
    upstream_kernel<<<grid_for(R * 32), 256, 0, s>>>(a.grad_y, a.y, a.den, R, static_cast<int>(a.d),
                                                     reinterpret_cast<uint2*>(b.y));
    if (cudaGetLastError() != cudaSuccess) return MEMOROID_ERR_CUDA;
    l.grad_y16 = reinterpret_cast<const uint16_t*>(b.y);  // bf16 [R, 128] in the fp32 buffer's first half
    l.dS_last = g_in ? b.S1 : nullptr;
    // heads of up to 64 channels need only the first 64 columns of dq', dk', dv'
    const int64_t wout = a.d <= 64 ? 64 : kW;
    l.out_cols = a.d <= 64 ? 64 : 0;
    l.fold_col = a.d;  // dphi(q)_i = dq''_i + dq''_d
    l.dq = b.dq;
    l.dk = b.dk;
    l.dv = b.dv;
    if (fused) {
        // the kernels build the operands from q, k, v and apply the chain rule
        // through phi in their epilogues, writing the caller's gradients
        l.q = a.q;
        l.k = a.k;
        l.v = a.v;
        l.norm = 1;
        l.dq = a.dq;
        l.dk = a.dk;
        l.dv = a.dv;
    }
    l.dgamma = a.dgamma;
    l.dS0 = (a.dS0 != nullptr || a.dz0 != nullptr) ? b.S2 : nullptr;
    const memoroid_status_t st = la::launch_bwd(l, s);
    if (st != MEMOROID_OK) return st;
    if (!fused)
        chain_kernel<<<grid_for(R * a.d / 4), 256, 0, s>>>(
            reinterpret_cast<const float4*>(b.dq), reinterpret_cast<const float4*>(b.dk),
            reinterpret_cast<const float4*>(b.dv), static_cast<const uint2*>(a.q), static_cast<const uint2*>(a.k),
            static_cast<uint32_t>(R), static_cast<uint32_t>(a.d / 4), static_cast<uint32_t>(wout / 4),
            reinterpret_cast<float4*>(a.dq), reinterpret_cast<float4*>(a.dk), reinterpret_cast<float4*>(a.dv));
    if (l.dS0 != nullptr)
        unpad_state_kernel<<<grid_for(BH * a.d * (a.d + 1)), 256, 0, s>>>(b.S2, BH, static_cast<int>(a.d), 1, a.dS0,
                                                                           a.dz0);
    return cudaGetLastError() == cudaSuccess ? MEMOROID_OK : MEMOROID_ERR_CUDA;
}

}  // namespace lnorm
}  // namespace memoroid
