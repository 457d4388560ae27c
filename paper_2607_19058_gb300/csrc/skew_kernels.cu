// Device kernels of libskewadam (sm_103a).
//
// One SkewAdam step (paper Sec. 3, Eq. 1, Algorithm 1) as seven grouped launches in
// stream order, each over an item table of (tensor, tile) pairs:
//   k_sumsq      phase A, strip tiles: per-row and per-column sums of g^2 of a
//                factored matrix (Eq. 1), column partials per row tile (no atomics);
//   k_rowsq      phase A, whole-row tiles of factored matrices 512 to 4096 wide:
//                chunks of whole rows bulk-copied into a shared-memory ring; R_i
//                formed in the tile (Eq. 1), per-column partials of g^2 and of
//                g^2 / R_i (or M^2 / R_i after the momentum update, stored here),
//                from which the finalize forms sum(U^2) by the bilinear identity;
//   k_finalize   R / C moving averages (strip path) or C (row path), 1/sqrt(C_j),
//                mean(R); on the row path also sum(U^2) and the clip factor, or the
//                tensor is queued for phase B when the 1/sqrt(eps) clamp may bind;
//   k_rms        phase B, strip and flat tiles: momentum / exact second-moment
//                update, U up to its scalar and a compensated sum(U^2) per tile;
//                the last tile forms RMS(U) and the clip factor (Sec. 3);
//   k_fallback   phase B of the queued row-path tensors (element by element);
//   k_apply      phase C, strip and flat tiles: x = w (1 - lr*lambda) - lr*kappa*U
//                in fp32 and the dithered bf16 write-back (Philox-4x32-10);
//   k_apply_rows phase C, whole-row tiles: the same on bulk-copied rows of W and
//                G (or the new M).
// The reconstructed second moment of a factored matrix is never formed:
// 1/sqrt(max(R_i C_j / Rbar, eps)) = min(a_i * b_j, 1/sqrt(eps)) with
// a_i = 1/sqrt(R_i / Rbar) per row and b_j = 1/sqrt(C_j) per column.
//
// The per-step scalars are a kernel parameter (StepArgs, constant bank). Values
// produced by an earlier launch of the same step are read with L2-only (.cg)
// loads. When no element of a tile can reach the clamp (all but degenerate
// tiles), phase C takes a clamp-free path. Every wait on a bulk copy is bounded
// and reports a copy that does not land through the status word.
#include <cuda_runtime.h>
#include <type_traits>
#include <stdint.h>

#include "skew_plan.h"

namespace skew {
namespace {

constexpr uint32_t kAll = 0xFFFFFFFFu;

// Resident CTAs per SM each kernel is compiled for (register budget 64K / (256 * n)).
#ifndef SKEW_MINB_SUMSQ
#define SKEW_MINB_SUMSQ 4
#endif
#ifndef SKEW_MINB_RMS
#define SKEW_MINB_RMS 2
#endif
#ifndef SKEW_MINB_APPLY
#define SKEW_MINB_APPLY 2
#endif
constexpr int kSmemFloats = kVecPerThread * kThreads;  // row scales of the tallest tile
constexpr int kStripCols = 8 * 32;                     // widest column strip

// ---------------------------------------------------------------------------
// Memory access helpers
// ---------------------------------------------------------------------------
// L2 eviction policies for 16-byte accesses (created once per thread).
struct Pol {
    uint64_t keep;  // evict_last: gradient between its first and last pass
    uint64_t drop;  // evict_first: streamed once (weights, last gradient read)
    __device__ Pol() {
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep));
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(drop));
    }
};

__device__ __forceinline__ uint4 ld16_hint(const void *p, uint64_t pol) {
    uint4 u;
    asm volatile("ld.global.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
                 : "=r"(u.x), "=r"(u.y), "=r"(u.z), "=r"(u.w)
                 : "l"(p), "l"(pol));
    return u;
}

__device__ __forceinline__ void st16_hint(void *p, uint4 u, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1,%2,%3,%4}, %5;" ::"l"(p), "r"(u.x), "r"(u.y), "r"(u.z),
                 "r"(u.w), "l"(pol));
}

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float(uint32_t(h) << 16); }

__device__ __forceinline__ void unpack_bf8(uint4 u, float (&o)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        o[2 * q] = __uint_as_float(w[q] << 16);
        o[2 * q + 1] = __uint_as_float(w[q] & 0xFFFF0000u);
    }
}

// The same eight values as four (even, odd) pairs for the packed FP32x2 unit.
__device__ __forceinline__ void unpack_bf8x2(uint4 u, float2 (&o)[4]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) o[q] = make_float2(__uint_as_float(w[q] << 16), __uint_as_float(w[q] & 0xFFFF0000u));
}

__device__ __forceinline__ float2 neg2(float2 a) { return make_float2(-a.x, -a.y); }

// Eight bf16 values (scalar path: elements >= valid read as 0).
__device__ __forceinline__ void load_bf8_scalar(const uint16_t *p, int valid, float (&o)[8]) {
#pragma unroll
    for (int c = 0; c < 8; ++c) o[c] = c < valid ? bf16_to_f32(p[c]) : 0.f;
}

// Elements e0 .. e0+7 of a weight or gradient array on the scalar path (elements
// >= valid read as 0): bf16, or fp32 for a tensor kept in fp32 (its array pointer
// then addresses floats).
__device__ __forceinline__ void load8_elem(const uint16_t *base, bool f32, int64_t e0, int valid, float (&o)[8]) {
    if (f32) {
        const float *p = reinterpret_cast<const float *>(base) + e0;
#pragma unroll
        for (int c = 0; c < 8; ++c) o[c] = c < valid ? p[c] : 0.f;
    } else {
        load_bf8_scalar(base + e0, valid, o);
    }
}

// Eight fp32 values; `cg` reads through L2 only (values an earlier phase wrote).
template <bool VEC>
__device__ __forceinline__ void load_f8(const float *p, int valid, float (&o)[8], bool cg) {
    if (VEC) {
        float4 a, b;
        if (cg) {
            a = __ldcg(reinterpret_cast<const float4 *>(p));
            b = __ldcg(reinterpret_cast<const float4 *>(p + 4));
        } else {
            a = *reinterpret_cast<const float4 *>(p);
            b = *reinterpret_cast<const float4 *>(p + 4);
        }
        o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
        o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
    } else {
#pragma unroll
        for (int c = 0; c < 8; ++c) o[c] = c < valid ? (cg ? __ldcg(p + c) : p[c]) : 0.f;
    }
}

template <bool VEC>
__device__ __forceinline__ void store_f8(float *p, int valid, const float (&o)[8]) {
    if (VEC) {
        *reinterpret_cast<float4 *>(p) = make_float4(o[0], o[1], o[2], o[3]);
        *reinterpret_cast<float4 *>(p + 4) = make_float4(o[4], o[5], o[6], o[7]);
    } else {
#pragma unroll
        for (int c = 0; c < 8; ++c)
            if (c < valid) p[c] = o[c];
    }
}

// ---------------------------------------------------------------------------
// Dither: Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) -- ten rounds of
// two 32x32 multiplies whose high halves are xored with the other counter
// words and the round key; the key advances by two Weyl constants per round.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                               uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
        const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
        c0 = hi1 ^ c1 ^ k0;
        c1 = lo1;
        c2 = hi0 ^ c3 ^ k1;
        c3 = lo0;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return make_uint4(c0, c1, c2, c3);
}

// Dither key of one tensor at one step: tensor id, low 32 bits of the step and
// the two halves of the seed (kept in registers by the hot loops).
struct Dith {
    uint32_t tid, step, k0, k1;
    uint64_t base;  // dither index of the tile's tensor element 0
};

__device__ __forceinline__ Dith dith_of(const StepArgs &A, const TensorDev &T) {
    return Dith{T.tid, A.step_lo, A.seed_lo, A.seed_hi, T.base};
}

// The 16-bit dithers of the eight elements idx0 .. idx0+7 (idx0 a multiple of 8):
// counter (idx0/8 lo, idx0/8 hi, tensor id, step lo), key (seed lo, seed hi);
// element k takes half (k & 1) of word k >> 1.
__device__ __forceinline__ void dither8(uint64_t idx0, const Dith &d, uint32_t (&r)[8]) {
    const uint64_t blk = (idx0 + d.base) >> 3;
    const uint4 o = philox4x32_10((uint32_t)blk, (uint32_t)(blk >> 32), d.tid, d.step, d.k0, d.k1);
    const uint32_t w[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        r[2 * q] = w[q] & 0xFFFFu;
        r[2 * q + 1] = w[q] >> 16;
    }
}

__device__ __forceinline__ uint32_t dither1(uint64_t idx, const Dith &d) {
    idx += d.base;
    const uint64_t blk = idx >> 3;
    const uint4 o = philox4x32_10((uint32_t)blk, (uint32_t)(blk >> 32), d.tid, d.step, d.k0, d.k1);
    const uint32_t k = (uint32_t)(idx & 7);
    const uint32_t w = k < 2 ? o.x : k < 4 ? o.y : k < 6 ? o.z : o.w;
    return (w >> (16 * (k & 1))) & 0xFFFFu;
}

// Dithered rounding to bf16: add the 16-bit draw to the fp32 bit pattern and
// keep the top half (unbiased stochastic rounding); NaN -> canonical quiet NaN.
__device__ __forceinline__ uint32_t sr_bf16(float x, uint32_t r) {
    const uint32_t b = __float_as_uint(x);
    if (x != x) return 0x7FC0u | ((b >> 16) & 0x8000u);
    return (b + r) >> 16;
}

// The gradient scale gamma of the step (the trainer's global gradient-norm clip, Sec. 4
// training setup, App. A Table 9): the step sees gamma * G. It enters only through the
// moving-average increments, (1 - beta2) gamma^2 on g^2 and (1 - beta1) gamma on g, and
// the update coefficient of momentum-free tensors (U = coef * gamma * g / D; set_clip),
// so no kernel reads the gradient more than without it. With gamma = 1 every product
// below is exact and the step is bit for bit the unscaled one.
struct GScale {
    float c1, c2;  // (1 - beta1) gamma, (1 - beta2) gamma^2
    float gam;
};

__device__ __forceinline__ GScale grad_scale(const StepArgs &A) {
    if (!A.gscale) return GScale{A.c1, A.c2, 1.f};
    const float g = __ldg(A.gscale);
    return GScale{A.c1 * g, A.c2 * (g * g), g};
}

// a_i = 1/sqrt(R_i / Rbar), with Rbar = rbar_s * 2^-rbar_e (rbar_s in [1,2)); +inf if Rbar == 0.
__device__ __forceinline__ float row_scale(float Ri, float rbar_s, int rbar_e) {
    if (rbar_s == 0.f) return __int_as_float(0x7F800000);
    return __frsqrt_rn(__fdiv_rn(ldexpf(Ri, rbar_e), rbar_s));
}

// ---------------------------------------------------------------------------
// Reductions
// ---------------------------------------------------------------------------
// Error-free sum (Knuth's TwoSum): s + e == a + b exactly.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bp = s - a;
    e = (a - (s - bp)) + (b - bp);
}

// TwoSum on both lanes of a pair (packed FP32x2 adds; same results as two_sum).
__device__ __forceinline__ void two_sum2(float2 a, float2 b, float2 &s, float2 &e) {
    s = __fadd2_rn(a, b);
    const float2 bp = __fadd2_rn(s, neg2(a));
    e = __fadd2_rn(__fadd2_rn(a, neg2(__fadd2_rn(s, neg2(bp)))), __fadd2_rn(b, neg2(bp)));
}

// The value of a compensated (hi, lo) pair in fp64. Once an infinite term has
// entered, TwoSum's error term is NaN (inf - inf) while hi carries the sum
// (+-inf, or NaN for inf - inf), so a non-finite hi is the value on its own.
__device__ __forceinline__ double pair_value(float hi, float lo) {
    return isfinite(hi) ? (double)hi + (double)lo : (double)hi;
}

// The same, rounded to fp32.
__device__ __forceinline__ float pair_f(float hi, float lo) { return isfinite(hi) ? hi + lo : hi; }

// Compensated accumulator: the running sum is hi + lo.
struct Acc2 {
    float hi = 0.f, lo = 0.f;
    __device__ __forceinline__ void add(float v) {
        float s, e;
        two_sum(hi, v, s, e);
        hi = s;
        lo += e;
    }
};

// Sum of the squares of eight values by a balanced tree (exact doubling when equal).
__device__ __forceinline__ float sumsq8(const float (&u)[8]) {
    const float p01 = fmaf(u[0], u[0], u[1] * u[1]);
    const float p23 = fmaf(u[2], u[2], u[3] * u[3]);
    const float p45 = fmaf(u[4], u[4], u[5] * u[5]);
    const float p67 = fmaf(u[6], u[6], u[7] * u[7]);
    return (p01 + p23) + (p45 + p67);
}

// CTA-wide compensated sum of (hi, lo) pairs; result valid in thread 0.
__device__ float2 block_sum2(Acc2 a, float2 *red) {
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const float h = __shfl_xor_sync(kAll, a.hi, o), l = __shfl_xor_sync(kAll, a.lo, o);
        float s, e;
        two_sum(a.hi, h, s, e);
        a.hi = s;
        a.lo += l + e;
    }
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = make_float2(a.hi, a.lo);
    __syncthreads();
    Acc2 r;
    if (threadIdx.x == 0) {
        for (int k = 0; k < kThreads / 32; ++k) {
            float s, e;
            two_sum(r.hi, red[k].x, s, e);
            r.hi = s;
            r.lo += red[k].y + e;
        }
    }
    return make_float2(r.hi, r.lo);
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kAll, v, o);
    return v;
}

// Deterministic CTA-wide fp64 sum (fixed shuffle tree, then warp 0 over the 8 warp sums).
__device__ double block_sum_d(double v, double *red) {
    v = warp_sum_d(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    double r = 0.0;
    if (w == 0) {
        r = l < kThreads / 32 ? red[l] : 0.0;
        r = warp_sum_d(r);
    }
    return r;  // valid in thread 0
}

// Counter increment that publishes this CTA's (barrier-ordered) writes and, for
// the CTA that sees the final count, acquires every other CTA's.
__device__ __forceinline__ uint32_t atom_add_acq_rel(uint32_t *p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// Shared scratch of a CTA.
struct Smem {
    float colred[kThreads * 8];  // column partials of a sum-of-squares tile
    float2 red2[kThreads / 32];
    double redd[kThreads / 32];
    int last;
};

// Row scales a_i of a factored tile's rows and column scales b_j of its strip.
struct Meta {
    float rows[kSmemFloats];
    float cols[kStripCols];
    float red[2 * kThreads / 32];  // per-warp maxima of the row / column scales
};

// Geometry of a factored tile: LC lanes along a row, RG row groups, 16 rows per thread.
struct FactTile {
    uint32_t LC, RG, lane, rg, s, rt;
    int64_t col0, row0;
    int valid;
    bool act;
    __device__ FactTile(const TensorDev &T, uint32_t tile) {
        LC = 1u << T.lcl;
        RG = kThreads >> T.lcl;
        s = tile % T.strips;
        rt = tile / T.strips;
        lane = threadIdx.x & (LC - 1);
        rg = threadIdx.x >> T.lcl;
        col0 = int64_t(s) * 8 * LC + 8 * lane;
        act = col0 < T.m;
        valid = act ? (int)min(int64_t(8), T.m - col0) : 0;
        row0 = int64_t(rt) * T.tile_rows + rg;
    }
};

// A scale for the clamp-free test: NaN counts as +inf, so that a tile holding a
// NaN scale never takes the clamp-free path.
__device__ __forceinline__ float nan_to_inf(float v) { return v == v ? v : __int_as_float(0x7F800000); }

// a_i of the tile's rows and b_j of its strip (R, 1/sqrt(C), mean(R) read from L2).
// Returns (the same value in every thread) whether no element of the tile can
// reach the clamp: max_i a_i * max_j b_j <= 1/sqrt(eps), all scales finite. Then
// min(a_i * b_j, 1/sqrt(eps)) = a_i * b_j for every element (rounding is monotone).
__device__ bool fill_meta(const TensorDev &T, const TensorScal &S, uint32_t tile, float ce, Meta &meta) {
    const uint32_t s = tile % T.strips, rt = tile / T.strips, width = 8u << T.lcl;
    const float rbar_s = __ldcg(&S.rbar_s);
    const int rbar_e = __ldcg(&S.rbar_e);
    float ma = 0.f, mb = 0.f;
    for (uint32_t r = threadIdx.x; r < T.tile_rows; r += kThreads) {
        const int64_t i = int64_t(rt) * T.tile_rows + r;
        const float a = i < T.n ? row_scale(__ldcg(T.R + i), rbar_s, rbar_e) : 0.f;
        meta.rows[r] = a;
        ma = fmaxf(ma, nan_to_inf(a));
    }
    for (uint32_t c = threadIdx.x; c < width; c += kThreads) {
        const int64_t j = int64_t(s) * width + c;
        const float b = j < T.m ? __ldcg(T.bsc + j) : 0.f;
        meta.cols[c] = b;
        mb = fmaxf(mb, nan_to_inf(b));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        ma = fmaxf(ma, __shfl_xor_sync(kAll, ma, o));
        mb = fmaxf(mb, __shfl_xor_sync(kAll, mb, o));
    }
    if ((threadIdx.x & 31) == 0) {
        meta.red[threadIdx.x >> 5] = ma;
        meta.red[kThreads / 32 + (threadIdx.x >> 5)] = mb;
    }
    __syncthreads();
    ma = mb = 0.f;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) {
        ma = fmaxf(ma, meta.red[w]);
        mb = fmaxf(mb, meta.red[kThreads / 32 + w]);
    }
    return ma * mb <= ce;
}

// ---------------------------------------------------------------------------
// Phase A: per-row / per-column sums of g^2 (Eq. 1).
// ---------------------------------------------------------------------------
// Adds the squares of one row-vector to the column partials; returns the row's
// sum over the LC lanes that share the row.
__device__ __forceinline__ float sumsq_row(const float (&g)[8], float (&col)[8], uint32_t LC) {
    float rs = 0.f;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        const float q = g[c] * g[c];
        col[c] += q;
        rs += q;
    }
    for (uint32_t o = LC >> 1; o; o >>= 1) rs += __shfl_xor_sync(kAll, rs, o);
    return rs;
}

template <bool VEC>
__device__ void sumsq_tile(const TensorDev &T, uint32_t tile, Smem &sm, const Pol &pol) {
    const FactTile F(T, tile);
    const uint16_t *__restrict__ g_ = T.g;
    float *__restrict__ rowp = T.rowp + int64_t(F.s) * T.n;
    const int64_t n = T.n, m = T.m, row0 = F.row0, RG = F.RG, col0 = F.col0;
    const uint32_t LC = F.LC;
    const bool act = F.act, lane0 = F.lane == 0;
    float col[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if constexpr (VEC) {
        constexpr int KCH = 8;  // row-vectors requested before the first is used
#pragma unroll 1
        for (int k0 = 0; k0 < kVecPerThread; k0 += KCH) {
            uint4 raw[KCH];
#pragma unroll
            for (int q = 0; q < KCH; ++q) {
                const int64_t i = row0 + (k0 + q) * RG;
                raw[q] = (act && i < n) ? ld16_hint(g_ + i * m + col0, pol.keep) : make_uint4(0, 0, 0, 0);
            }
            if (LC == 32) {
                // each lane holds partial sums of 8 rows; a transposed butterfly leaves
                // lane L with the full sum of row 4*b4 + 2*b3 + b2 (bits of L)
                float rs[KCH];
#pragma unroll
                for (int q = 0; q < KCH; ++q) {
                    float g[8];
                    unpack_bf8(raw[q], g);
                    float acc = 0.f;
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const float sq = g[c] * g[c];
                        col[c] += sq;
                        acc += sq;
                    }
                    rs[q] = acc;
                }
                const uint32_t ln = threadIdx.x & 31;
                const bool b4 = ln & 16, b3 = ln & 8, b2 = ln & 4;
                float v4[4], v2[2];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float keep = b4 ? rs[q + 4] : rs[q], send = b4 ? rs[q] : rs[q + 4];
                    v4[q] = keep + __shfl_xor_sync(kAll, send, 16);
                }
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    const float keep = b3 ? v4[q + 2] : v4[q], send = b3 ? v4[q] : v4[q + 2];
                    v2[q] = keep + __shfl_xor_sync(kAll, send, 8);
                }
                float v1 = (b2 ? v2[1] : v2[0]) + __shfl_xor_sync(kAll, b2 ? v2[0] : v2[1], 4);
                v1 += __shfl_xor_sync(kAll, v1, 2);
                v1 += __shfl_xor_sync(kAll, v1, 1);
                const int qs = (b4 ? 4 : 0) + (b3 ? 2 : 0) + (b2 ? 1 : 0);
                const int64_t i = row0 + (k0 + qs) * RG;
                if ((ln & 3) == 0 && i < n) rowp[i] = v1;
            } else {
#pragma unroll
                for (int q = 0; q < KCH; ++q) {
                    const int64_t i = row0 + (k0 + q) * RG;
                    float g[8];
                    unpack_bf8(raw[q], g);
                    const float rs = sumsq_row(g, col, LC);
                    if (lane0 && i < n) rowp[i] = rs;
                }
            }
        }
    } else {
        for (int k = 0; k < kVecPerThread; ++k) {
            const int64_t i = row0 + k * RG;
            float g[8];
            if (act && i < n)
                load8_elem(g_, T.f32, i * m + col0, F.valid, g);
            else
#pragma unroll
                for (int c = 0; c < 8; ++c) g[c] = 0.f;
            const float rs = sumsq_row(g, col, LC);
            if (lane0 && i < n) rowp[i] = rs;
        }
    }
#pragma unroll
    for (int c = 0; c < 8; ++c) sm.colred[threadIdx.x * 8 + c] = col[c];
    __syncthreads();
    const uint32_t width = 8 * LC;
    for (uint32_t cc = threadIdx.x; cc < width; cc += kThreads) {
        float acc = 0.f;
        for (uint32_t r = 0; r < F.RG; ++r) acc += sm.colred[r * width + cc];
        const int64_t j = int64_t(F.s) * width + cc;
        if (j < m) T.colp[int64_t(F.rt) * m + j] = acc;
    }
}

// ---------------------------------------------------------------------------
// Row path, phase A (k_rowsq): whole-row tiles of a momentum-free factored
// matrix. With a_i = sqrt(Rbar / R_i) and b_j = 1/sqrt(C_j), and no element at
// the clamp, sum_ij (g_ij a_i b_j)^2 = Rbar * sum_j (1 / C_j) * P_j with
// P_j = sum_i g_ij^2 / R_i. A tile holds whole rows, so it forms R_i (Eq. 1)
// itself and adds g_ij^2 / R_i into per-column partials of P; the column
// finalize then gives C_j and sum(U^2) without phase B re-reading G.
// Each chunk (kRowChunkBytes of consecutive rows, contiguous in memory) is
// brought to shared memory by one bulk copy completing on an mbarrier; the
// CTA keeps kRowStages chunks in flight.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t *b, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)), "r"(bytes) : "memory");
}

// One poll; the thread may be suspended for up to about kMbarSuspendNs while the
// phase is incomplete (a hint to the hardware).
constexpr uint32_t kMbarSuspendNs = 2000;

__device__ __forceinline__ bool mbar_try_wait(uint64_t *b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(b)), "r"(parity), "n"(kMbarSuspendNs)
        : "memory");
    return ok != 0;
}

// Polls of one mbarrier wait before it gives up (about two seconds at the
// suspend hint): a copy that never lands ends the tile with a status word
// instead of hanging the GPU.
constexpr uint32_t kMbarPolls = 1u << 20;

__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity) {
    for (uint32_t i = 0; i < kMbarPolls; ++i)
        if (mbar_try_wait(b, parity)) return true;
    return false;
}

// After a wait gave up (status bit 2): one thread waits for chunks [c, issued_end) of a
// ring of `stages` slots that are still in flight, so that the CTA does not leave while
// a bulk copy may still write into its shared memory. Each gets up to eight more
// rounds of polls (about sixteen seconds); a copy still outstanding after that is
// recorded as status bit 4 and the CTA leaves anyway.
__device__ __noinline__ void drain_copies(uint32_t *err, uint64_t *full, uint32_t stages, uint32_t c,
                                          uint32_t issued_end) {
    atomicOr(err, 2u);
    for (uint32_t k = c; k < issued_end; ++k) {
        bool landed = false;
        for (int round = 0; round < 8 && !landed; ++round) landed = mbar_wait(&full[k % stages], (k / stages) & 1u);
        if (!landed) atomicOr(err, 4u);
    }
}

// Bulk copy global -> shared of `bytes` (multiple of 16, both ends 16-byte
// aligned), completing on mbarrier `bar`, with an L2 eviction policy.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}

// Orders this thread's earlier generic-proxy accesses of shared memory before
// its later async-proxy (bulk copy) accesses.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }

// Threads of the row-path kernels (256 or 512).
#ifndef SKEW_ROW_THREADS
#define SKEW_ROW_THREADS 256
#endif
constexpr int kRowThreads = SKEW_ROW_THREADS;

struct RowSmem {
    uint4 buf[kRowStages][kRowChunkBytes / 16];  // the chunk ring (first member: 16-byte aligned)
    uint64_t full[kRowStages];                   // one mbarrier per ring slot
    float part[kRowThreads / 32][8];             // per-warp row partial sums of the chunk
    float inv[32];                               // 1 / R_i of the chunk's rows (0: no contribution)
    int fail;
};

// Rows `i` of chunk `c` of row tile `tile`: [i0, i0 + rows).
struct RowChunk {
    int64_t i0;
    uint32_t rows;
};

__device__ __forceinline__ RowChunk row_chunk(const TensorDev &T, uint32_t tile, uint32_t c) {
    const int64_t i0 = int64_t(tile) * T.rt_rows + int64_t(c) * T.cr;
    const int64_t left = T.n - i0;
    return RowChunk{i0, left <= 0 ? 0u : (uint32_t)min(left, (int64_t)T.cr)};
}

// Sum of N values p[0], p[stride], ..., p[(N - 1) stride] (N a power of two) by a
// balanced tree.
template <int N>
__device__ __forceinline__ float tree_sum(const float *p, int stride) {
    if constexpr (N == 1) {
        return p[0];
    } else {
        return tree_sum<N / 2>(p, stride) + tree_sum<N / 2>(p + (N / 2) * stride, stride);
    }
}

// Sum over a warp of K per-lane values, transposed: lane L ends with the total
// of value j(L) (K = 8: j = 4*b4 + 2*b3 + b2 of L's bits; K = 4: j = 2*b4 + b3;
// K = 2: j = b4), held by the lanes whose low 2, 3 or 4 bits are zero.
template <int K>
__device__ __forceinline__ float warp_sum_transposed(const float (&x)[K], int &j) {
    const uint32_t ln = threadIdx.x & 31;
    const bool b4 = ln & 16, b3 = ln & 8, b2 = ln & 4;
    if constexpr (K == 8) {
        float v4[4], v2[2];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float keep = b4 ? x[q + 4] : x[q], send = b4 ? x[q] : x[q + 4];
            v4[q] = keep + __shfl_xor_sync(kAll, send, 16);
        }
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const float keep = b3 ? v4[q + 2] : v4[q], send = b3 ? v4[q] : v4[q + 2];
            v2[q] = keep + __shfl_xor_sync(kAll, send, 8);
        }
        float v1 = (b2 ? v2[1] : v2[0]) + __shfl_xor_sync(kAll, b2 ? v2[0] : v2[1], 4);
        v1 += __shfl_xor_sync(kAll, v1, 2);
        v1 += __shfl_xor_sync(kAll, v1, 1);
        j = (b4 ? 4 : 0) + (b3 ? 2 : 0) + (b2 ? 1 : 0);
        return v1;
    } else if constexpr (K == 2) {
        float v1 = (b4 ? x[1] : x[0]) + __shfl_xor_sync(kAll, b4 ? x[0] : x[1], 16);
        v1 += __shfl_xor_sync(kAll, v1, 8);
        v1 += __shfl_xor_sync(kAll, v1, 4);
        v1 += __shfl_xor_sync(kAll, v1, 2);
        v1 += __shfl_xor_sync(kAll, v1, 1);
        j = b4 ? 1 : 0;
        return v1;
    } else {
        float v2[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const float keep = b4 ? x[q + 2] : x[q], send = b4 ? x[q] : x[q + 2];
            v2[q] = keep + __shfl_xor_sync(kAll, send, 16);
        }
        float v1 = (b3 ? v2[1] : v2[0]) + __shfl_xor_sync(kAll, b3 ? v2[0] : v2[1], 8);
        v1 += __shfl_xor_sync(kAll, v1, 4);
        v1 += __shfl_xor_sync(kAll, v1, 2);
        v1 += __shfl_xor_sync(kAll, v1, 1);
        j = (b4 ? 2 : 0) + (b3 ? 1 : 0);
        return v1;
    }
}

// Issues the bulk copy of chunk c of the tile into ring slot c % kRowStages.
__device__ __forceinline__ void row_issue(const TensorDev &T, uint32_t tile, uint32_t c, RowSmem &sm, uint64_t pol) {
    const RowChunk ch = row_chunk(T, tile, c);
    const uint32_t bytes = ch.rows * (uint32_t)T.m * 2u;
    const int st = c % kRowStages;
    mbar_expect_tx(&sm.full[st], bytes);
    bulk_g2s(sm.buf[st], T.g + ch.i0 * T.m, bytes, &sm.full[st], pol);
}

// Thread layout of a row-path kernel with TPB threads on rows of V = m / 8
// 16-byte vectors: NV vectors per thread per row (V > TPB), or RPP rows side by side
// (V < TPB); a thread owns vectors vi, vi + TPB, ... of row-in-pass rp.
template <int TPB, int V>
struct RowLayout {
    static constexpr int NV = V > TPB ? V / TPB : 1;
    static constexpr int RPP = V < TPB ? TPB / V : 1;
    static constexpr int WPR = (V < TPB ? V : TPB) / 32;  // warps per row-in-pass
    int rp, vi;
    __device__ RowLayout() : rp(threadIdx.x / (V < TPB ? V : TPB)), vi(threadIdx.x % (V < TPB ? V : TPB)) {}
};

// k_rowsq on TPB threads, rows of m = 8 V: chunks of CS = 2048 / V rows (32 KB),
// K = CS / RPP rows per thread per chunk.
template <int TPB, int V>
__device__ void rowsq_tile(const StepArgs &A, const TensorDev &T, TensorScal &S, uint32_t tile, RowSmem &sm) {
    using L = RowLayout<TPB, V>;
    constexpr int NV = L::NV, RPP = L::RPP, WPR = L::WPR;
    constexpr int CS = 2048 / V;
    constexpr int K = CS / RPP;
    static_assert(K == 4 || K == 8, "rows per thread per chunk");
    static_assert(CS <= 32, "chunk rows");
    const L lay;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    const uint32_t nch = (uint32_t)min((int64_t)(T.rt_rows / T.cr), (T.n - int64_t(tile) * T.rt_rows + T.cr - 1) / T.cr);
    if (threadIdx.x == 0) {
        for (int st = 0; st < kRowStages; ++st) mbar_init(&sm.full[st], 1);
        fence_mbar_init();
        sm.fail = 0;
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (uint32_t c = 0; c < nch && c < (uint32_t)kRowStages; ++c) row_issue(T, tile, c, sm, pol);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const float b2 = A.b2, c2 = grad_scale(A).c2, inv_m = 1.0f / (float)(8 * V);  // m is a power of two: exact
    // per column pair: sums of g^2, the compensated (hi, lo) sum of g^2 / R_i and its open fp32 part
    float2 cs[NV][4], ph[NV][4], pl[NV][4], t[NV][4];
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int q = 0; q < 4; ++q) cs[v][q] = ph[v][q] = pl[v][q] = t[v][q] = make_float2(0.f, 0.f);
    double rsum = 0.0;                       // threads < CS: sum of the R of this chunk-row position
    float rmin = __int_as_float(0x7F800000);  // threads < CS: smallest positive R of it
    bool zero_row = false;

    // the tile's rows and R, held in registers (the stores to R in the loop could
    // otherwise make the compiler reload them from the descriptor every chunk)
    const int64_t row0 = int64_t(tile) * T.rt_rows, n = T.n;
    const uint32_t cr = T.cr;
    float *__restrict__ Rg = T.R;
    uint32_t c = 0;
    for (; c < nch; ++c) {
        const int st = c % kRowStages;
        const uint32_t par = (c / kRowStages) & 1u;
        const int64_t ci0 = row0 + int64_t(c) * cr;
        const RowChunk ch{ci0, (uint32_t)min(n - ci0, (int64_t)cr)};
        float rp = 0.f;
        if (tid < (int)ch.rows) rp = __ldcg(Rg + ch.i0 + tid);
        const bool ok = mbar_wait(&sm.full[st], par);
        const uint4 *buf = sm.buf[st];
        // a full chunk (every chunk but a tensor's last) needs no row bound checks
        const bool full = ch.rows == (uint32_t)CS;
        // pass 1: row sums and column sums of g^2 (rows lay.rp + RPP k of the chunk)
        float rs[K];
        auto pass1 = [&](auto full_c) {
#pragma unroll
            for (int k = 0; k < K; ++k) {
                const int r = lay.rp + RPP * k;
                float2 r2 = make_float2(0.f, 0.f);
                if (decltype(full_c)::value || r < (int)ch.rows) {
#pragma unroll
                    for (int v = 0; v < NV; ++v) {
                        float2 g[4];
                        unpack_bf8x2(buf[r * V + v * TPB + lay.vi], g);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {  // g^2 into the column and row sums, one rounding each
                            cs[v][q] = __ffma2_rn(g[q], g[q], cs[v][q]);
                            r2 = __ffma2_rn(g[q], g[q], r2);
                        }
                    }
                }
                rs[k] = r2.x + r2.y;
            }
        };
        if (full)
            pass1(std::true_type{});
        else
            pass1(std::false_type{});
        int j;
        const float tot = warp_sum_transposed<K>(rs, j);
        if ((lane & (K == 8 ? 3 : 7)) == 0) sm.part[warp][j] = tot;
        if (__syncthreads_or(!ok)) break;  // every slot before this one has landed
        // slot of chunk c - 1 is free (its pass 2 preceded this barrier): refill it
        // (from warp 1: warp 0 forms the chunk's row scales, which the CTA waits for)
        if (tid == 32 && c >= 1 && c - 1 + kRowStages < nch) {
            fence_proxy_async_smem();
            row_issue(T, tile, c - 1 + kRowStages, sm, pol);
        }
        float Rn = 0.f, sum = 0.f;
        if (tid < (int)ch.rows) {  // chunk row r = tid: row-in-pass r % RPP, its k = r / RPP
            const int w0 = (tid % RPP) * WPR, kr = tid / RPP;
            sum = tree_sum<WPR>(&sm.part[w0][kr], 8);
            Rn = fmaf(b2, rp, c2 * (sum * inv_m));
            sm.inv[tid] = Rn > 0.f && Rn < __int_as_float(0x7F800000) ? __frcp_rn(Rn) : 0.f;
        }
        __syncthreads();
        if (tid < (int)ch.rows) {  // the row's R and the tile's statistics, off the barrier's path
            Rg[ch.i0 + tid] = Rn;
            rsum += (double)Rn;
            if (Rn > 0.f && Rn < __int_as_float(0x7F800000))
                rmin = fminf(rmin, Rn);
            else if (!(Rn == 0.f && sum == 0.f))
                zero_row = true;  // content in a row with R_i == 0, or a non-finite R_i
        }
        // pass 2: P_j += g^2 / R_i, summed in fp32 over four chunks (at most 4 K rows)
        // per column, then folded into (hi, lo)
        auto pass2 = [&](auto full_c) {
#pragma unroll
            for (int k = 0; k < K; ++k) {
                const int r = lay.rp + RPP * k;
                if (decltype(full_c)::value || r < (int)ch.rows) {
                    const float iv = sm.inv[r];
                    const float2 iv2 = make_float2(iv, iv);
#pragma unroll
                    for (int v = 0; v < NV; ++v) {
                        float2 g[4];
                        unpack_bf8x2(buf[r * V + v * TPB + lay.vi], g);
#pragma unroll
                        for (int q = 0; q < 4; ++q) t[v][q] = __ffma2_rn(__fmul2_rn(g[q], g[q]), iv2, t[v][q]);
                    }
                }
            }
        };
        if (full)
            pass2(std::true_type{});
        else
            pass2(std::false_type{});
        if ((c & 3u) == 3u || c + 1 == nch) {
#pragma unroll
            for (int v = 0; v < NV; ++v)
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float2 s2, e2;
                    two_sum2(ph[v][q], t[v][q], s2, e2);
                    ph[v][q] = s2;
                    pl[v][q] = __fadd2_rn(pl[v][q], e2);
                    t[v][q] = make_float2(0.f, 0.f);
                }
        }
    }
    if (c < nch) {
        // A chunk did not land in time: record it, wait (bounded) for the copies in
        // flight and drop the tile. Issued so far: chunks [0, kRowStages) by the
        // prologue and chunk k - 1 + kRowStages at each iteration k in [1, c); chunks
        // before c have landed.
        if (tid == 0)
            drain_copies(A.err, sm.full, kRowStages, c, min(nch, c == 0 ? (uint32_t)kRowStages : c + kRowStages - 1));
        return;
    }
    // per-tile partials, (sum of g^2, sum of g^2 / R_i) per column (the RPP threads that
    // share a column vector are added in row-in-pass order; the compensated sum of
    // g^2 / R_i is rounded to fp32 once), the tile's sum and smallest positive R
    const int64_t base = int64_t(tile) * 8 * V;
    if constexpr (RPP == 1) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int64_t col = 8 * int64_t(v * TPB + lay.vi);
            float4 *pp4 = reinterpret_cast<float4 *>(T.pp + base + col);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                pp4[q] = make_float4(cs[v][q].x, pair_f(ph[v][q].x, pl[v][q].x), cs[v][q].y,
                                     pair_f(ph[v][q].y, pl[v][q].y));
        }
    } else {
        // the ring is free (every chunk consumed before the last barrier): stage there
        float *mcs = reinterpret_cast<float *>(sm.buf[0]);        // [TPB][8]
        float2 *mpp = reinterpret_cast<float2 *>(sm.buf[1]);      // [TPB][8] (hi, lo)
        __syncthreads();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            mcs[tid * 8 + 2 * q] = cs[0][q].x;
            mcs[tid * 8 + 2 * q + 1] = cs[0][q].y;
            mpp[tid * 8 + 2 * q] = make_float2(ph[0][q].x, pl[0][q].x);
            mpp[tid * 8 + 2 * q + 1] = make_float2(ph[0][q].y, pl[0][q].y);
        }
        __syncthreads();
        for (int e = tid; e < 8 * V; e += TPB) {  // column e = 8 vi + q
            const int vi = e >> 3, q = e & 7;
            float cc = 0.f;
            Acc2 pq;
#pragma unroll
            for (int r = 0; r < RPP; ++r) {
                cc += mcs[(r * V + vi) * 8 + q];
                const float2 h = mpp[(r * V + vi) * 8 + q];
                pq.add(h.x);
                pq.lo += h.y;
            }
            T.pp[base + e] = make_float2(cc, pair_f(pq.hi, pq.lo));
        }
    }
    if (zero_row) atomicOr(&S.zflag, 1u);
    if (warp == 0) {  // CS <= 32: the chunk-row positions are lanes of warp 0
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            rsum += __shfl_xor_sync(kAll, rsum, o);
            rmin = fminf(rmin, __shfl_xor_sync(kAll, rmin, o));
        }
        if (lane == 0) {
            T.rsum[tile] = rsum;
            T.rmin[tile] = rmin;
        }
    }
}

// sum_{r < cnt} p[r * stride] (values an earlier launch wrote), added in order
// r = 0, 1, ...; the loads are issued eight at a time ahead of the adds.
template <typename V>
__device__ __forceinline__ V strided_sum(const V *p, int64_t stride, uint32_t cnt) {
    V s = V(0);
    uint32_t r = 0;
    for (; r + 8 <= cnt; r += 8) {
        V v[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) v[q] = __ldcg(p + int64_t(r + q) * stride);
#pragma unroll
        for (int q = 0; q < 8; ++q) s += v[q];
    }
    for (; r < cnt; ++r) s += __ldcg(p + int64_t(r) * stride);
    return s;
}

// mean(R) and its [1, 2) mantissa / exponent split (used by the row scales).
__device__ void set_rbar(TensorScal &S, double rbar) {
    S.rbar = rbar;
    if (rbar > 0.0) {
        int e;
        const double fr = frexp(rbar, &e);  // rbar = fr * 2^e, fr in [0.5, 1)
        S.rbar_s = (float)(2.0 * fr);       // in [1, 2]
        S.rbar_e = 1 - e;                   // rbar * 2^(1-e) = 2 fr
    } else {
        S.rbar_s = 0.f;
        S.rbar_e = 0;
    }
}

// From s = sum of (U / coef)^2: sum(U^2), RMS(U), the clip factor
// kappa = 1 / max(1, RMS / d) (Sec. 3 update clipping) and lr * kappa * coef.
__device__ void set_clip(const StepArgs &A, const TensorDev &T, TensorScal &S, double s) {
    // a momentum-free tensor's U is coef * gamma * g / D (M already carries gamma)
    const double coef = T.momentum ? A.coef_mom : A.coef_plain * (double)grad_scale(A).gam;
    const double su2 = s * coef * coef;
    const double rms = sqrt(su2 / (double)T.numel);
    const double kappa = 1.0 / fmax(1.0, rms / (double)A.clip_d);
    S.sumsq = su2;
    S.rms = rms;
    S.kappa = kappa;
    S.coefC = (float)((double)A.lr * kappa * coef);
}

// Row path, finalize item `local` (kFinChunk columns): C_j, 1/sqrt(C_j) and the
// chunk's sum of P_j / C_j. The last item of the tensor forms mean(R) and, when
// no element can reach the clamp (max_i a_i^2 * max_j b_j^2 <= 1/eps over rows and
// columns that hold gradient), sum(U^2) = coef^2 * mean(R) * sum_j P_j / C_j and
// the clip factor; otherwise it queues the tensor for phase B. P_j and the sums
// of P_j / C_j are compensated fp32 (hi, lo) pairs: fp64 arithmetic runs at a
// small fraction of the fp32 rate here, and every term is non-negative, so a
// pair keeps the sum to about fp64 accuracy and each quotient to one fp32 rounding.
__device__ void phase_F_row(const StepArgs &A, uint32_t t, uint32_t local, Smem &sm) {
    const TensorDev &T = A.tensors[t];
    TensorScal &S = A.scal[t];
    const float inf = __int_as_float(0x7F800000);
    // the item's fci columns, kFinChunk / fci threads per column: thread tid adds the
    // tiles r = sl, sl + tpc, ... of column cix (consecutive threads, consecutive columns)
    const int fci = (int)T.fci, tpc = kFinChunk / fci;
    const int cix = threadIdx.x % fci, sl = threadIdx.x / fci;
    const int64_t j = int64_t(local) * fci + cix;
    float cs = 0.f;  // this thread's tiles: sum of g^2 (in tile order) and, compensated, of g^2 / R_i
    Acc2 pa;
    if (j < T.m) {
        const float2 *p = T.pp + j;
        uint32_t r = sl;
        // loads issued 32 (then 16) at a time ahead of the adds, which go in tile order
        for (; r + 31 * tpc < T.rtiles; r += 32 * tpc) {
            float2 v[32];
#pragma unroll
            for (int q = 0; q < 32; ++q) v[q] = __ldcg(p + int64_t(r + q * tpc) * T.m);
#pragma unroll
            for (int q = 0; q < 32; ++q) {
                cs += v[q].x;
                pa.add(v[q].y);
            }
        }
        for (; r + 15 * tpc < T.rtiles; r += 16 * tpc) {
            float2 v[16];
#pragma unroll
            for (int q = 0; q < 16; ++q) v[q] = __ldcg(p + int64_t(r + q * tpc) * T.m);
#pragma unroll
            for (int q = 0; q < 16; ++q) {
                cs += v[q].x;
                pa.add(v[q].y);
            }
        }
        for (; r < T.rtiles; r += tpc) {
            const float2 v = __ldcg(p + int64_t(r) * T.m);
            cs += v.x;
            pa.add(v.y);
        }
    }
    // the column's tpc parts in slice order
    float *red = sm.colred;  // [3][kFinChunk]: sum g^2, hi, lo
    red[threadIdx.x] = cs;
    red[kFinChunk + threadIdx.x] = pa.hi;
    red[2 * kFinChunk + threadIdx.x] = pa.lo;
    __syncthreads();
    Acc2 contrib;
    float cmin = inf;
    if (sl == 0 && j < T.m) {
        const float Cold = __ldcg(T.C + j);
        for (int k = 1; k < tpc; ++k) {
            cs += red[k * fci + cix];
            pa.add(red[kFinChunk + k * fci + cix]);
            pa.lo += red[2 * kFinChunk + k * fci + cix];
        }
        const float P = pair_f(pa.hi, pa.lo);
        const float mean = __fdiv_rn(cs, (float)T.n);
        const float Cn = fmaf(A.b2, Cold, grad_scale(A).c2 * mean);
        T.C[j] = Cn;
        T.bsc[j] = __frsqrt_rn(Cn);
        if (P > 0.f) {
            if (Cn > 0.f && Cn < inf) {
                contrib.add(__fdiv_rn(P, Cn));
                cmin = Cn;
            } else {
                atomicOr(&S.zflag, 1u);  // gradient in a column whose C_j is 0 or not finite
            }
        } else if (!(P == 0.f)) {
            atomicOr(&S.zflag, 1u);  // NaN
        }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) cmin = fminf(cmin, __shfl_xor_sync(kAll, cmin, o));
    __syncthreads();  // the column parts in colred are consumed
    if ((threadIdx.x & 31) == 0) sm.colred[threadIdx.x >> 5] = cmin;
    const float2 cs2 = block_sum2(contrib, sm.red2);  // its barriers also publish colred
    if (threadIdx.x == 0) {
        for (int w = 0; w < kThreads / 32; ++w) cmin = fminf(cmin, sm.colred[w]);
        T.fsum[local] = pair_value(cs2.x, cs2.y);
        T.fmin[local] = cmin;
        sm.last = (atom_add_acq_rel(&S.cntF, 1u) == T.nfc - 1);
    }
    __syncthreads();
    if (!sm.last) return;
    // Last item of the tensor: the whole CTA sums the row tiles' R sums and minima and
    // the items' sums and minima (thread k takes entries k, k + kThreads, ...; then a
    // fixed shuffle tree: the same order every step).
    double rs = 0.0, fs = 0.0;
    float rmn = inf, cmn = inf;
    for (uint32_t r = threadIdx.x; r < T.rtiles; r += kThreads) {
        rs += __ldcg(T.rsum + r);
        rmn = fminf(rmn, __ldcg(T.rmin + r));
    }
    for (uint32_t f = threadIdx.x; f < T.nfc; f += kThreads) {
        fs += __ldcg(T.fsum + f);
        cmn = fminf(cmn, __ldcg(T.fmin + f));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        rmn = fminf(rmn, __shfl_xor_sync(kAll, rmn, o));
        cmn = fminf(cmn, __shfl_xor_sync(kAll, cmn, o));
    }
    if ((threadIdx.x & 31) == 0) {  // colred was last read before the barrier above
        sm.colred[threadIdx.x >> 5] = rmn;
        sm.colred[kThreads / 32 + (threadIdx.x >> 5)] = cmn;
    }
    rs = block_sum_d(rs, sm.redd);  // its barriers also publish the minima
    fs = block_sum_d(fs, sm.redd);
    if (threadIdx.x == 0) {
        for (int w = 0; w < kThreads / 32; ++w) {
            rmn = fminf(rmn, sm.colred[w]);
            cmn = fminf(cmn, sm.colred[kThreads / 32 + w]);
        }
        const double rbar = rs / (double)T.n;
        set_rbar(S, rbar);
        const double a2 = rmn < inf ? rbar / (double)rmn : 0.0;  // max_i a_i^2 over rows with R_i > 0
        const double b2 = cmn < inf ? 1.0 / (double)cmn : 0.0;   // max_j b_j^2 over columns holding gradient
        const double ce2 = (double)A.ce * (double)A.ce;
        if (__ldcg(&S.zflag) == 0u && a2 * b2 <= ce2 * (1.0 - 1e-6)) {
            set_clip(A, T, S, fs * rbar);
        } else {
            S.fallback = 1u;
            const uint32_t q = atomicAdd(A.fb, 1u);
            A.fb[1 + q] = t;
        }
    }
}

// ---------------------------------------------------------------------------
// Phase F: factor EMAs, 1/sqrt(C_j), mean(R) (Eq. 1).
// ---------------------------------------------------------------------------
__device__ void phase_F(const StepArgs &A, uint32_t t, uint32_t local, Smem &sm) {
    const TensorDev &T = A.tensors[t];
    TensorScal &S = A.scal[t];
    if (T.rowpath) {
        phase_F_row(A, t, local, sm);
        return;
    }
    if (local < T.nfr) {
        const int64_t i = int64_t(local) * kFinChunk + threadIdx.x;
        double rd = 0.0;
        if (threadIdx.x < kFinChunk && i < T.n) {
            const float rs = strided_sum(T.rowp + i, T.n, T.strips);
            const float mean = __fdiv_rn(rs, (float)T.m);
            const float Rn = fmaf(A.b2, T.R[i], grad_scale(A).c2 * mean);
            T.R[i] = Rn;
            rd = (double)Rn;
        }
        rd = block_sum_d(rd, sm.redd);
        if (threadIdx.x == 0) T.rsum[local] = rd;
    } else {
        const int64_t j = int64_t(local - T.nfr) * kFinChunk + threadIdx.x;
        if (threadIdx.x < kFinChunk && j < T.m) {
            const float cs = strided_sum(T.colp + j, T.m, T.rowtiles);
            const float mean = __fdiv_rn(cs, (float)T.n);
            const float Cn = fmaf(A.b2, T.C[j], grad_scale(A).c2 * mean);
            T.C[j] = Cn;
            T.bsc[j] = __frsqrt_rn(Cn);
        }
    }
    // The last finalize item of the tensor forms mean(R) from the row items' partial sums.
    __syncthreads();
    if (threadIdx.x == 0) sm.last = (atom_add_acq_rel(&S.cntF, 1u) == T.nfr + T.nfc - 1);
    __syncthreads();
    if (!sm.last) return;
    double s = 0.0;  // the CTA sums the row items' partials (fixed partition and tree)
    for (uint32_t f = threadIdx.x; f < T.nfr; f += kThreads) s += __ldcg(T.rsum + f);
    s = block_sum_d(s, sm.redd);
    if (threadIdx.x == 0) set_rbar(S, s / (double)T.n);
}

// ---------------------------------------------------------------------------
// Phase B: second moment / momentum update and sum(U^2) (Algorithm 1).
// ---------------------------------------------------------------------------
// U (up to its scalar) of one row-vector of a factored tile, squared and summed into acc.
__device__ __forceinline__ void rms_row(const float (&y)[8], float a, const float (&b)[8], int valid, float ce,
                                        Acc2 &acc) {
    float u[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) u[c] = c < valid ? y[c] * fminf(a * b[c], ce) : 0.f;
    acc.add(sumsq8(u));
}

template <bool VEC, bool MOM>
__device__ Acc2 rms_fact_tile(const StepArgs &A, const TensorDev &T, uint32_t tile, const Meta &meta,
                              const Pol &pol) {
    const FactTile F(T, tile);
    Acc2 acc;
    if (!F.act) return acc;
    const uint16_t *__restrict__ g_ = T.g;
    float *__restrict__ M_ = T.M;
    const int64_t n = T.n, m = T.m, row0 = F.row0, RG = F.RG, col0 = F.col0;
    const int valid = F.valid;
    const float b1 = A.b1, c1 = grad_scale(A).c1, ce = A.ce;
    const bool mnew = MOM && T.rowpath;  // phase B of a queued row-path tensor: M is already new
    const float *rows = meta.rows + F.rg;
    float b[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) b[c] = meta.cols[F.lane * 8 + c];
    if constexpr (VEC) {
        // row-vectors requested together: eight when only g streams, four with the momentum
        constexpr int KCH = MOM ? 4 : 8;
#pragma unroll 1
        for (int k0 = 0; k0 < kVecPerThread; k0 += KCH) {
            uint4 graw[KCH];
            float4 mraw[MOM ? KCH : 1][2];
#pragma unroll
            for (int q = 0; q < KCH; ++q) {
                const int64_t i = row0 + (k0 + q) * RG;
                const int64_t e0 = (i < n ? i : 0) * m + col0;
                if (i < n) graw[q] = ld16_hint(g_ + e0, MOM ? pol.drop : pol.keep);
                if (MOM && i < n) {
                    mraw[MOM ? q : 0][0] = *reinterpret_cast<const float4 *>(M_ + e0);
                    mraw[MOM ? q : 0][1] = *reinterpret_cast<const float4 *>(M_ + e0 + 4);
                }
            }
#pragma unroll
            for (int q = 0; q < KCH; ++q) {
                const int64_t i = row0 + (k0 + q) * RG;
                if (i < n) {
                    float y[8];
                    unpack_bf8(graw[q], y);
                    if (MOM) {
                        const float4 m0 = mraw[MOM ? q : 0][0], m1 = mraw[MOM ? q : 0][1];
                        const float mm[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
                        if (mnew) {  // the row path already stored this step's momentum
#pragma unroll
                            for (int c = 0; c < 8; ++c) y[c] = mm[c];
                        } else {
#pragma unroll
                            for (int c = 0; c < 8; ++c) y[c] = fmaf(b1, mm[c], c1 * y[c]);
                            store_f8<true>(M_ + i * m + col0, 8, y);
                        }
                    }
                    rms_row(y, rows[(k0 + q) * RG], b, 8, ce, acc);
                }
            }
        }
    } else {
        for (int k = 0; k < kVecPerThread; ++k) {
            const int64_t i = row0 + k * RG;
            if (i >= n) break;
            float y[8];
            load8_elem(g_, T.f32, i * m + col0, valid, y);
            if (MOM) {
                float mm[8];
                load_f8<false>(M_ + i * m + col0, valid, mm, false);
                if (mnew) {
#pragma unroll
                    for (int c = 0; c < 8; ++c) y[c] = mm[c];
                } else {
#pragma unroll
                    for (int c = 0; c < 8; ++c) y[c] = fmaf(b1, mm[c], c1 * y[c]);
                    store_f8<false>(M_ + i * m + col0, valid, y);
                }
            }
            rms_row(y, rows[k * RG], b, valid, ce, acc);
        }
    }
    return acc;
}

template <bool VEC>
__device__ Acc2 rms_full_tile(const StepArgs &A, const TensorDev &T, uint32_t tile, const Pol &pol) {
    const GScale gsc = grad_scale(A);
    Acc2 acc;
    for (int k = 0; k < kFlatVecPerThread; ++k) {
        const int64_t e0 = 8 * (int64_t(tile) * kThreads * kFlatVecPerThread + int64_t(k) * kThreads + threadIdx.x);
        if (e0 >= T.numel) break;
        const int valid = (int)min(int64_t(8), T.numel - e0);
        float g[8], v[8], y[8];
        if (VEC)
            unpack_bf8(ld16_hint(T.g + e0, pol.drop), g);
        else
            load8_elem(T.g, T.f32, e0, valid, g);
        load_f8<VEC>(T.v + e0, valid, v, false);
#pragma unroll
        for (int c = 0; c < 8; ++c) v[c] = fmaf(A.b2, v[c], gsc.c2 * (g[c] * g[c]));
        store_f8<VEC>(T.v + e0, valid, v);
        if (T.momentum) {
            float mm[8];
            load_f8<VEC>(T.M + e0, valid, mm, false);
#pragma unroll
            for (int c = 0; c < 8; ++c) y[c] = fmaf(A.b1, mm[c], gsc.c1 * g[c]);
            store_f8<VEC>(T.M + e0, valid, y);
        } else {
#pragma unroll
            for (int c = 0; c < 8; ++c) y[c] = g[c];
        }
        float u[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) u[c] = c < valid ? y[c] * fminf(__frsqrt_rn(v[c]), A.ce) : 0.f;
        acc.add(sumsq8(u));
    }
    return acc;
}

__device__ void phase_B(const StepArgs &A, uint32_t t, uint32_t local, Smem &sm, const Meta &meta, const Pol &pol) {
    const TensorDev &T = A.tensors[t];
    TensorScal &S = A.scal[t];
    Acc2 acc;
    if (T.kind == kKindFactored) {
        if (T.vec)
            acc = T.momentum ? rms_fact_tile<true, true>(A, T, local, meta, pol)
                             : rms_fact_tile<true, false>(A, T, local, meta, pol);
        else
            acc = T.momentum ? rms_fact_tile<false, true>(A, T, local, meta, pol)
                             : rms_fact_tile<false, false>(A, T, local, meta, pol);
    } else {
        acc = T.vec ? rms_full_tile<true>(A, T, local, pol) : rms_full_tile<false>(A, T, local, pol);
    }
    const float2 tsum = block_sum2(acc, sm.red2);
    if (threadIdx.x == 0) {
        T.u2[local] = tsum;
        sm.last = (atom_add_acq_rel(&S.cntB, 1u) == T.ntiles - 1);
    }
    __syncthreads();
    if (!sm.last) return;
    // Last tile of the tensor: sum(U^2), RMS, clip factor (fixed summation order).
    double s = 0.0;
    for (uint32_t k = threadIdx.x; k < T.ntiles; k += kThreads) {
        const float2 p = __ldcg(T.u2 + k);
        s += pair_value(p.x, p.y);
    }
    s = block_sum_d(s, sm.redd);
    if (threadIdx.x == 0) set_clip(A, T, S, s);
}

// ---------------------------------------------------------------------------
// Phase C: decoupled decay, clipped update, dithered bf16 write-back.
// ---------------------------------------------------------------------------
// x of eight elements -> dithered bf16, stored at w + e0 (16-byte store when VEC).
template <bool VEC>
__device__ __forceinline__ void write8(uint16_t *__restrict__ w, const Dith &d, int64_t e0, int valid, bool aligned8,
                                       const float (&x)[8], const Pol &pol) {
    uint32_t r[8];
    if (VEC) {
        dither8((uint64_t)e0, d, r);
        uint32_t o[4];
        // a NaN anywhere makes the sum NaN (so does Inf - Inf): only then test per element
        const float any = ((x[0] + x[1]) + (x[2] + x[3])) + ((x[4] + x[5]) + (x[6] + x[7]));
        if (any == any) {
#pragma unroll
            for (int q = 0; q < 4; ++q)  // top halves of (bits + draw) of the two elements
                o[q] = __byte_perm(__float_as_uint(x[2 * q]) + r[2 * q], __float_as_uint(x[2 * q + 1]) + r[2 * q + 1],
                                   0x7632);
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q)
                o[q] = sr_bf16(x[2 * q], r[2 * q]) | (sr_bf16(x[2 * q + 1], r[2 * q + 1]) << 16);
        }
        st16_hint(w + e0, make_uint4(o[0], o[1], o[2], o[3]), pol.drop);
    } else {
        if (aligned8) dither8((uint64_t)e0, d, r);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            if (c < valid) {
                const uint32_t rc = aligned8 ? r[c] : dither1((uint64_t)(e0 + c), d);
                w[e0 + c] = (uint16_t)sr_bf16(x[c], rc);
            }
        }
    }
}

// Scalar-path write-back of elements e0 .. e0+valid-1: the dithered bf16 rounding,
// or for a tensor kept in fp32 the fp32 value x itself.
__device__ __forceinline__ void store8_elem(const TensorDev &T, uint16_t *w, const Dith &d, int64_t e0, int valid,
                                            const float (&x)[8], const Pol &pol) {
    if (T.f32) {
        float *p = reinterpret_cast<float *>(w) + e0;
#pragma unroll
        for (int c = 0; c < 8; ++c)
            if (c < valid) p[c] = x[c];
    } else {
        write8<false>(w, d, e0, valid, ((e0 + d.base) & 7) == 0, x, pol);
    }
}

// FAST: no element of the tile reaches the clamp (fill_meta), so the update is
// (-lr*kappa*coef * a_i) * b_j * y, one multiply and one fma per element.
template <bool VEC, bool MOM, bool FAST>
__device__ void apply_fact_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t tile,
                                const Meta &meta, const Pol &pol) {
    const FactTile F(T, tile);
    if (!F.act) return;
    const uint16_t *__restrict__ g_ = T.g;
    const float *__restrict__ M_ = T.M;
    uint16_t *__restrict__ w_ = T.w;
    const int64_t n = T.n, m = T.m, row0 = F.row0, RG = F.RG, col0 = F.col0;
    const int valid = F.valid;
    const Dith d = dith_of(A, T);
    const float coefC = __ldcg(&S.coefC);
    const float wdf = T.decay ? A.wdf : 1.0f;
    const float ce = A.ce;
    const float *rows = meta.rows + F.rg;
    float b[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) b[c] = meta.cols[F.lane * 8 + c];
    if constexpr (VEC) {
        constexpr int KCH = 4;  // row-vectors (with their weights) requested together
#pragma unroll 1
        for (int k0 = 0; k0 < kVecPerThread; k0 += KCH) {
            uint4 wraw[KCH], graw[MOM ? 1 : KCH];
            float4 mraw[MOM ? KCH : 1][2];
#pragma unroll
            for (int q = 0; q < KCH; ++q) {
                const int64_t i = row0 + (k0 + q) * RG;
                const int64_t e0 = (i < n ? i : 0) * m + col0;
                if (i < n) {
                    if (MOM) {
                        mraw[MOM ? q : 0][0] = __ldcg(reinterpret_cast<const float4 *>(M_ + e0));
                        mraw[MOM ? q : 0][1] = __ldcg(reinterpret_cast<const float4 *>(M_ + e0 + 4));
                    } else {
                        graw[MOM ? 0 : q] = ld16_hint(g_ + e0, pol.drop);
                    }
                    wraw[q] = ld16_hint(w_ + e0, pol.drop);
                }
            }
#pragma unroll
            for (int q = 0; q < KCH; ++q) {
                const int64_t i = row0 + (k0 + q) * RG;
                if (i < n) {
                    float y[8], w[8], x[8];
                    if (MOM) {
                        const float4 m0 = mraw[MOM ? q : 0][0], m1 = mraw[MOM ? q : 0][1];
                        y[0] = m0.x; y[1] = m0.y; y[2] = m0.z; y[3] = m0.w;
                        y[4] = m1.x; y[5] = m1.y; y[6] = m1.z; y[7] = m1.w;
                    } else {
                        unpack_bf8(graw[MOM ? 0 : q], y);
                    }
                    unpack_bf8(wraw[q], w);
                    const float a = rows[(k0 + q) * RG];
                    if constexpr (FAST) {
                        const float ca = -coefC * a;
                        const float2 ca2 = make_float2(ca, ca), wdf2 = make_float2(wdf, wdf);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 xx = __ffma2_rn(__fmul2_rn(ca2, make_float2(b[2 * q], b[2 * q + 1])),
                                                         make_float2(y[2 * q], y[2 * q + 1]),
                                                         __fmul2_rn(make_float2(w[2 * q], w[2 * q + 1]), wdf2));
                            x[2 * q] = xx.x;
                            x[2 * q + 1] = xx.y;
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < 8; ++c) x[c] = fmaf(-coefC, y[c] * fminf(a * b[c], ce), w[c] * wdf);
                    }
                    write8<true>(w_, d, i * m + col0, 8, true, x, pol);
                }
            }
        }
    } else {
        for (int k = 0; k < kVecPerThread; ++k) {
            const int64_t i = row0 + k * RG;
            if (i >= n) break;
            const int64_t e0 = i * m + col0;
            float y[8], w[8], x[8];
            if (MOM)
                load_f8<false>(M_ + e0, valid, y, true);
            else
                load8_elem(g_, T.f32, e0, valid, y);
            load8_elem(w_, T.f32, e0, valid, w);
            const float a = rows[k * RG];
#pragma unroll
            for (int c = 0; c < 8; ++c) x[c] = fmaf(-coefC, y[c] * fminf(a * b[c], ce), w[c] * wdf);
            store8_elem(T, w_, d, e0, valid, x, pol);
        }
    }
}

template <bool VEC>
__device__ void apply_full_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t tile,
                                const Pol &pol) {
    const float coefC = __ldcg(&S.coefC);
    const float wdf = T.decay ? A.wdf : 1.0f;
    for (int k = 0; k < kFlatVecPerThread; ++k) {
        const int64_t e0 = 8 * (int64_t(tile) * kThreads * kFlatVecPerThread + int64_t(k) * kThreads + threadIdx.x);
        if (e0 >= T.numel) break;
        const int valid = (int)min(int64_t(8), T.numel - e0);
        float y[8], v[8], w[8], x[8];
        if (T.momentum)
            load_f8<VEC>(T.M + e0, valid, y, true);
        else if (VEC)
            unpack_bf8(ld16_hint(T.g + e0, pol.drop), y);
        else
            load8_elem(T.g, T.f32, e0, valid, y);
        load_f8<VEC>(T.v + e0, valid, v, true);
        if (VEC)
            unpack_bf8(ld16_hint(T.w + e0, pol.drop), w);
        else
            load8_elem(T.w, T.f32, e0, valid, w);
#pragma unroll
        for (int c = 0; c < 8; ++c) x[c] = fmaf(-coefC, y[c] * fminf(__frsqrt_rn(v[c]), A.ce), w[c] * wdf);
        const Dith dd = dith_of(A, T);  // on the vector path e0 and base are multiples of 8
        if (VEC)
            write8<true>(T.w, dd, e0, valid, true, x, pol);
        else
            store8_elem(T, T.w, dd, e0, valid, x, pol);
    }
}

// ---------------------------------------------------------------------------
// Row path, phase C (k_apply_rows): the row tiles of k_rowsq. A chunk is CA
// whole rows of W and the same rows of G, one bulk copy each into a ring slot
// (W in the first half, G in the second); the column scales b_j of a thread's
// 8*NV columns stay in registers and the tile's row scales a_i in shared memory.
// Per element the arithmetic, the dither index and the rounding are those of
// apply_fact_tile, so the result is the same bit for bit.
// ---------------------------------------------------------------------------
struct ApplyRowSmem {
    uint4 buf[kRowStages][kRowChunkBytes / 16];  // [W rows | G rows] per slot
    uint64_t full[kRowStages];
    float a[kRowChunks * 32];                    // row scales a_i of the tile (at_rows <= 1024)
    float red[2 * kRowThreads / 32];
};

// Chunk c of the phase-C tile (or half tile) whose first row is r0. A half tile is 16 of
// the phase-A chunks' rows, i.e. whole phase-C chunks, so only the matrix's end cuts one.
__device__ __forceinline__ void apply_row_issue(const TensorDev &T, int64_t r0, uint32_t c, uint32_t ca,
                                                ApplyRowSmem &sm, uint64_t pol) {
    const int64_t i0 = r0 + int64_t(c) * ca;
    const uint32_t rows = (uint32_t)min((int64_t)ca, T.n - i0);
    const uint32_t bytes = rows * (uint32_t)T.m * 2u;
    const int st = c % kRowStages;
    mbar_expect_tx(&sm.full[st], 2u * bytes);
    bulk_g2s(sm.buf[st], T.w + i0 * T.m, bytes, &sm.full[st], pol);
    bulk_g2s(sm.buf[st] + kRowChunkBytes / 32, T.g + i0 * T.m, bytes, &sm.full[st], pol);
}

// CA = 1024 / V rows per chunk (16 KB of W, 16 KB of G), KA = CA / RPP rows per thread.
template <int TPB, int V, bool FAST>
__device__ void apply_rows_body(const StepArgs &A, const TensorDev &T, int64_t r0,
                                const float (&b)[RowLayout<TPB, V>::NV][8], float coefC, ApplyRowSmem &sm,
                                uint32_t nch, uint64_t pol) {
    using L = RowLayout<TPB, V>;
    constexpr int NV = L::NV, RPP = L::RPP;
    constexpr int CA = 1024 / V, KA = CA / RPP;
    const L lay;
    const int tid = threadIdx.x;
    const int64_t m = 8 * V;
    uint16_t *__restrict__ w_ = T.w;
    const Dith d = dith_of(A, T);
    const float wdf = T.decay ? A.wdf : 1.0f;
    const float ce = A.ce;
    const float2 wdf2 = make_float2(wdf, wdf);
    const Pol sp;
    for (uint32_t c = 0; c < nch; ++c) {
        const int st = c % kRowStages;
        const int64_t i0 = r0 + int64_t(c) * CA;
        const int rows = (int)min((int64_t)CA, T.n - i0);
        const bool ok = mbar_wait(&sm.full[st], (c / kRowStages) & 1u);
        const uint4 *bw = sm.buf[st];
        const uint4 *bg = sm.buf[st] + kRowChunkBytes / 32;
#pragma unroll
        for (int k = 0; k < KA; ++k) {
            const int r = lay.rp + RPP * k;
            if (r < rows) {
                const float a = sm.a[c * CA + r];
                const float cr = -coefC * a;
                const float2 cr2 = make_float2(cr, cr);
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    float y[8], w[8], x[8];
                    unpack_bf8(bg[r * V + v * TPB + lay.vi], y);
                    unpack_bf8(bw[r * V + v * TPB + lay.vi], w);
                    if constexpr (FAST) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 xx =
                                __ffma2_rn(__fmul2_rn(cr2, make_float2(b[v][2 * q], b[v][2 * q + 1])),
                                           make_float2(y[2 * q], y[2 * q + 1]),
                                           __fmul2_rn(make_float2(w[2 * q], w[2 * q + 1]), wdf2));
                            x[2 * q] = xx.x;
                            x[2 * q + 1] = xx.y;
                        }
                    } else {
#pragma unroll
                        for (int q = 0; q < 8; ++q) x[q] = fmaf(-coefC, y[q] * fminf(a * b[v][q], ce), w[q] * wdf);
                    }
                    write8<true>(w_, d, (i0 + r) * m + 8 * (v * TPB + lay.vi), 8, true, x, sp);
                }
            }
        }
        // every thread is done with slot st: refill it with chunk c + kRowStages
        if (__syncthreads_or(!ok)) {
            if (tid == 0)  // chunks [0, c + kRowStages) were issued
                drain_copies(A.err, sm.full, kRowStages, c, min(nch, c + kRowStages));
            return;
        }
        if (tid == 0 && c + kRowStages < nch) {
            fence_proxy_async_smem();
            apply_row_issue(T, r0, c + kRowStages, CA, sm, pol);
        }
    }
}

template <int TPB, int V>
__device__ void apply_rows_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t item,
                                ApplyRowSmem &sm) {
    using L = RowLayout<TPB, V>;
    constexpr int NV = L::NV;
    constexpr int CA = 1024 / V;
    const L lay;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    // a whole tile, or one half of it (the step's last tiles run as halves)
    const uint32_t trows = (item & kHalfTile) ? T.at_rows / 2 : T.at_rows;
    const int64_t r0 = int64_t(item & kTileMask) * T.at_rows + ((item & kSecondHalf) ? trows : 0);
    if (r0 >= T.n) return;  // the second half of a matrix's short last tile
    const uint32_t rows_t = (uint32_t)min((int64_t)trows, T.n - r0);
    const uint32_t nch = (rows_t + CA - 1) / CA;
    if (threadIdx.x == 0) {
        for (int st = 0; st < kRowStages; ++st) mbar_init(&sm.full[st], 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (uint32_t c = 0; c < nch && c < (uint32_t)kRowStages; ++c) apply_row_issue(T, r0, c, CA, sm, pol);
    // row scales of the tile, column scales of this thread's columns, and the clamp test
    const float rbar_s = __ldcg(&S.rbar_s);
    const int rbar_e = __ldcg(&S.rbar_e);
    float ma = 0.f, mb = 0.f;
    for (uint32_t r = threadIdx.x; r < rows_t; r += TPB) {
        const float a = row_scale(__ldcg(T.R + r0 + r), rbar_s, rbar_e);
        sm.a[r] = a;
        ma = fmaxf(ma, nan_to_inf(a));
    }
    float b[NV][8];
#pragma unroll
    for (int v = 0; v < NV; ++v) {
        const float *p = T.bsc + 8 * (v * TPB + lay.vi);
        const float4 b0 = __ldcg(reinterpret_cast<const float4 *>(p));
        const float4 b1 = __ldcg(reinterpret_cast<const float4 *>(p + 4));
        b[v][0] = b0.x; b[v][1] = b0.y; b[v][2] = b0.z; b[v][3] = b0.w;
        b[v][4] = b1.x; b[v][5] = b1.y; b[v][6] = b1.z; b[v][7] = b1.w;
#pragma unroll
        for (int k = 0; k < 8; ++k) mb = fmaxf(mb, nan_to_inf(b[v][k]));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        ma = fmaxf(ma, __shfl_xor_sync(kAll, ma, o));
        mb = fmaxf(mb, __shfl_xor_sync(kAll, mb, o));
    }
    if ((threadIdx.x & 31) == 0) {
        sm.red[threadIdx.x >> 5] = ma;
        sm.red[TPB / 32 + (threadIdx.x >> 5)] = mb;
    }
    __syncthreads();
    ma = mb = 0.f;
#pragma unroll
    for (int w = 0; w < TPB / 32; ++w) {
        ma = fmaxf(ma, sm.red[w]);
        mb = fmaxf(mb, sm.red[TPB / 32 + w]);
    }
    const float coefC = __ldcg(&S.coefC);
    if (ma * mb <= A.ce)
        apply_rows_body<TPB, V, true>(A, T, r0, b, coefC, sm, nch, pol);
    else
        apply_rows_body<TPB, V, false>(A, T, r0, b, coefC, sm, nch, pol);
}

// ---------------------------------------------------------------------------
// Row path with momentum (backbone matrices, and experts under the momentum
// variants). Phase A runs on whole rows as in k_rowsq and, in the same pass,
// applies Algorithm 1's momentum update M <- b1 M + (1 - b1) g to a copy of the
// rows of M made beside those of G, storing the new M. With U_ij = coef M_ij a_i b_j
// and no element at the clamp, sum(U^2) = coef^2 * mean(R) * sum_j Q_j / C_j with
// Q_j = sum_i M_ij^2 / R_i, accumulated here where the momentum-free path
// accumulates P_j. Phase C then reads the new M where it would read G. A chunk
// is CS = kMomGBytes / (2 m) rows: 16 KB of G (or W in phase C) and the same rows
// of M (32 KB) in one slot of a 2-slot ring, one bulk copy each. A row whose R_i
// is 0 or not finite sends the tensor to phase B (its momentum may still be
// nonzero), where M is used as already updated.
// ---------------------------------------------------------------------------
constexpr int kMomStages = 2;
constexpr int kMomSlot16 = 3 * kMomGBytes / 16;  // 16-byte words per slot: 16 KB bf16 | 32 KB fp32

struct MomRowSmem {
    uint4 buf[kMomStages][kMomSlot16];  // [G rows | M rows] per slot
    uint64_t full[kMomStages];
    float part[kRowThreads / 32][8];
    float inv[32];
    int fail;
};

// Issues the bulk copies of chunk c of row tile `tile` (rows of x = G in phase A,
// W in phase C, and the same rows of M) into ring slot c % kMomStages.
__device__ __forceinline__ void mom_issue(const TensorDev &T, const uint16_t *x, uint32_t tile, uint32_t c,
                                          uint4 (*buf)[kMomSlot16], uint64_t *full, uint64_t pol) {
    const RowChunk ch = row_chunk(T, tile, c);
    const uint32_t bx = ch.rows * (uint32_t)T.m * 2u;
    const int st = c % kMomStages;
    mbar_expect_tx(&full[st], 3u * bx);
    bulk_g2s(buf[st], x + ch.i0 * T.m, bx, &full[st], pol);
    bulk_g2s(buf[st] + kMomGBytes / 16, T.M + ch.i0 * T.m, 2u * bx, &full[st], pol);
}

// k_rowsq for momentum tensors on TPB threads, rows of m = 8 V: chunks of CS = 1024 / V
// rows, K = CS / RPP rows per thread per chunk.
template <int TPB, int V>
__device__ void rowsq_mom_tile(const StepArgs &A, const TensorDev &T, TensorScal &S, uint32_t tile, MomRowSmem &sm) {
    using L = RowLayout<TPB, V>;
    constexpr int NV = L::NV, RPP = L::RPP, WPR = L::WPR;
    constexpr int CS = 1024 / V;
    constexpr int K = CS / RPP;
    static_assert(K == 2 || K == 4, "rows per thread per chunk");
    const L lay;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    const uint32_t nch = (uint32_t)min((int64_t)kMomChunks, (T.n - int64_t(tile) * T.rt_rows + T.cr - 1) / T.cr);
    if (threadIdx.x == 0) {
        for (int st = 0; st < kMomStages; ++st) mbar_init(&sm.full[st], 1);
        fence_mbar_init();
        sm.fail = 0;
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (uint32_t c = 0; c < nch && c < (uint32_t)kMomStages; ++c) mom_issue(T, T.g, tile, c, sm.buf, sm.full, pol);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const GScale gsc = grad_scale(A);
    const float b1 = A.b1, c1 = gsc.c1, b2 = A.b2, c2 = gsc.c2, inv_m = 1.0f / (float)(8 * V);  // exact
    const float2 b12 = make_float2(b1, b1), c12 = make_float2(c1, c1);
    // per column pair: sums of g^2, the compensated (hi, lo) sum of M^2 / R_i and its open fp32 part
    float2 cs[NV][4], ph[NV][4], pl[NV][4], t[NV][4];
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int q = 0; q < 4; ++q) cs[v][q] = ph[v][q] = pl[v][q] = t[v][q] = make_float2(0.f, 0.f);
    double rsum = 0.0;
    float rmin = __int_as_float(0x7F800000);
    bool zero_row = false;

    uint32_t c = 0;
    for (; c < nch; ++c) {
        const int st = c % kMomStages;
        const uint32_t par = (c / kMomStages) & 1u;
        const RowChunk ch = row_chunk(T, tile, c);
        float rp = 0.f;
        if (tid < (int)ch.rows) rp = __ldcg(T.R + ch.i0 + tid);
        const bool ok = mbar_wait(&sm.full[st], par);
        const uint4 *bg = sm.buf[st];
        const float4 *bm = reinterpret_cast<const float4 *>(sm.buf[st] + kMomGBytes / 16);
        // pass 1: row sums and column sums of g^2
        float rs[K];
#pragma unroll
        for (int k = 0; k < K; ++k) {
            const int r = lay.rp + RPP * k;
            float2 r2 = make_float2(0.f, 0.f);
            if (r < (int)ch.rows) {
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    float2 g[4];
                    unpack_bf8x2(bg[r * V + v * TPB + lay.vi], g);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        cs[v][q] = __ffma2_rn(g[q], g[q], cs[v][q]);
                        r2 = __ffma2_rn(g[q], g[q], r2);
                    }
                }
            }
            rs[k] = r2.x + r2.y;
        }
        int j;
        const float tot = warp_sum_transposed<K>(rs, j);
        if ((lane & (K == 4 ? 7 : 15)) == 0) sm.part[warp][j] = tot;
        if (__syncthreads_or(!ok)) break;  // every slot before this one has landed
        // refill from warp 1: warp 0 forms the chunk's row scales, which the CTA waits for
        if (tid == 32 && c >= 1 && c - 1 + kMomStages < nch) {
            fence_proxy_async_smem();
            mom_issue(T, T.g, tile, c - 1 + kMomStages, sm.buf, sm.full, pol);
        }
        float Rn = 0.f;
        if (tid < (int)ch.rows) {
            const int w0 = (tid % RPP) * WPR, kr = tid / RPP;
            Rn = fmaf(b2, rp, c2 * (tree_sum<WPR>(&sm.part[w0][kr], 8) * inv_m));
            sm.inv[tid] = Rn > 0.f && Rn < __int_as_float(0x7F800000) ? __frcp_rn(Rn) : 0.f;
        }
        __syncthreads();
        if (tid < (int)ch.rows) {  // the row's R and the tile's statistics, off the barrier's path
            T.R[ch.i0 + tid] = Rn;
            rsum += (double)Rn;
            if (Rn > 0.f && Rn < __int_as_float(0x7F800000))
                rmin = fminf(rmin, Rn);
            else
                zero_row = true;  // R_i == 0 or not finite: its momentum may still be nonzero
        }
        // pass 2: M <- b1 M + (1 - b1) g (stored), Q_j += M^2 / R_i
#pragma unroll
        for (int k = 0; k < K; ++k) {
            const int r = lay.rp + RPP * k;
            if (r < (int)ch.rows) {
                const float iv = sm.inv[r];
                const float2 iv2 = make_float2(iv, iv);
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int vec = v * TPB + lay.vi;
                    float2 g[4];
                    unpack_bf8x2(bg[r * V + vec], g);
                    const float4 m0 = bm[2 * (r * V + vec)], m1 = bm[2 * (r * V + vec) + 1];
                    const float2 mo[4] = {make_float2(m0.x, m0.y), make_float2(m0.z, m0.w), make_float2(m1.x, m1.y),
                                          make_float2(m1.z, m1.w)};
                    float2 mn[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        mn[q] = __ffma2_rn(b12, mo[q], __fmul2_rn(c12, g[q]));
                        t[v][q] = __ffma2_rn(__fmul2_rn(mn[q], mn[q]), iv2, t[v][q]);
                    }
                    float4 *dst = reinterpret_cast<float4 *>(T.M + (ch.i0 + r) * T.m + 8 * vec);
                    dst[0] = make_float4(mn[0].x, mn[0].y, mn[1].x, mn[1].y);
                    dst[1] = make_float4(mn[2].x, mn[2].y, mn[3].x, mn[3].y);
                }
            }
        }
        if ((c & 3u) == 3u || c + 1 == nch) {
#pragma unroll
            for (int v = 0; v < NV; ++v)
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float2 s2, e2;
                    two_sum2(ph[v][q], t[v][q], s2, e2);
                    ph[v][q] = s2;
                    pl[v][q] = __fadd2_rn(pl[v][q], e2);
                    t[v][q] = make_float2(0.f, 0.f);
                }
        }
    }
    if (c < nch) {
        // a chunk did not land in time: as in rowsq_tile
        if (tid == 0)
            drain_copies(A.err, sm.full, kMomStages, c, min(nch, c == 0 ? (uint32_t)kMomStages : c + kMomStages - 1));
        return;
    }
    const int64_t base = int64_t(tile) * 8 * V;
    if constexpr (RPP == 1) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int64_t col = 8 * int64_t(v * TPB + lay.vi);
            float4 *pp4 = reinterpret_cast<float4 *>(T.pp + base + col);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                pp4[q] = make_float4(cs[v][q].x, pair_f(ph[v][q].x, pl[v][q].x), cs[v][q].y,
                                     pair_f(ph[v][q].y, pl[v][q].y));
        }
    } else {
        // the ring is free (every chunk consumed before the last barrier): stage there
        float *mcs = reinterpret_cast<float *>(sm.buf[0]);    // [TPB][8]
        float2 *mpp = reinterpret_cast<float2 *>(sm.buf[1]);  // [TPB][8] (hi, lo)
        __syncthreads();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            mcs[tid * 8 + 2 * q] = cs[0][q].x;
            mcs[tid * 8 + 2 * q + 1] = cs[0][q].y;
            mpp[tid * 8 + 2 * q] = make_float2(ph[0][q].x, pl[0][q].x);
            mpp[tid * 8 + 2 * q + 1] = make_float2(ph[0][q].y, pl[0][q].y);
        }
        __syncthreads();
        for (int e = tid; e < 8 * V; e += TPB) {  // column e = 8 vi + q
            const int vi = e >> 3, q = e & 7;
            float cc = 0.f;
            Acc2 pq;
#pragma unroll
            for (int r = 0; r < RPP; ++r) {
                cc += mcs[(r * V + vi) * 8 + q];
                const float2 h = mpp[(r * V + vi) * 8 + q];
                pq.add(h.x);
                pq.lo += h.y;
            }
            T.pp[base + e] = make_float2(cc, pair_f(pq.hi, pq.lo));
        }
    }
    if (zero_row) atomicOr(&S.zflag, 1u);
    if (warp == 0) {  // CS <= 32: the chunk-row positions are lanes of warp 0
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            rsum += __shfl_xor_sync(kAll, rsum, o);
            rmin = fminf(rmin, __shfl_xor_sync(kAll, rmin, o));
        }
        if (lane == 0) {
            T.rsum[tile] = rsum;
            T.rmin[tile] = rmin;
        }
    }
}

struct MomApplySmem {
    uint4 buf[kMomStages][kMomSlot16];  // [W rows | M rows] per slot
    uint64_t full[kMomStages];
    float a[kRowChunks * 32];           // row scales a_i of the tile (at_rows <= 1024)
    float red[2 * kRowThreads / 32];
};

// Phase C of a momentum row tile: as apply_rows_body with y = the new M (Algorithm 1,
// backbone branch: U = coef M / D).
template <int TPB, int V, bool FAST>
__device__ void apply_rows_mom_body(const StepArgs &A, const TensorDev &T, uint32_t tile,
                                    const float (&b)[RowLayout<TPB, V>::NV][8], float coefC, MomApplySmem &sm,
                                    uint32_t nch, uint64_t pol) {
    using L = RowLayout<TPB, V>;
    constexpr int NV = L::NV, RPP = L::RPP;
    constexpr int CA = 1024 / V, KA = CA / RPP;
    const L lay;
    const int tid = threadIdx.x;
    const int64_t m = 8 * V;
    uint16_t *__restrict__ w_ = T.w;
    const Dith d = dith_of(A, T);
    const float wdf = T.decay ? A.wdf : 1.0f;
    const float ce = A.ce;
    const float2 wdf2 = make_float2(wdf, wdf);
    const Pol sp;
    for (uint32_t c = 0; c < nch; ++c) {
        const int st = c % kMomStages;
        const int64_t i0 = int64_t(tile) * T.at_rows + int64_t(c) * CA;
        const int rows = (int)min((int64_t)CA, T.n - i0);
        const bool ok = mbar_wait(&sm.full[st], (c / kMomStages) & 1u);
        const uint4 *bw = sm.buf[st];
        const float4 *bm = reinterpret_cast<const float4 *>(sm.buf[st] + kMomGBytes / 16);
#pragma unroll
        for (int k = 0; k < KA; ++k) {
            const int r = lay.rp + RPP * k;
            if (r < rows) {
                const float a = sm.a[c * CA + r];
                const float cr = -coefC * a;
                const float2 cr2 = make_float2(cr, cr);
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int vec = v * TPB + lay.vi;
                    float w[8], x[8];
                    unpack_bf8(bw[r * V + vec], w);
                    const float4 m0 = bm[2 * (r * V + vec)], m1 = bm[2 * (r * V + vec) + 1];
                    const float y[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
                    if constexpr (FAST) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float2 xx =
                                __ffma2_rn(__fmul2_rn(cr2, make_float2(b[v][2 * q], b[v][2 * q + 1])),
                                           make_float2(y[2 * q], y[2 * q + 1]),
                                           __fmul2_rn(make_float2(w[2 * q], w[2 * q + 1]), wdf2));
                            x[2 * q] = xx.x;
                            x[2 * q + 1] = xx.y;
                        }
                    } else {
#pragma unroll
                        for (int q = 0; q < 8; ++q) x[q] = fmaf(-coefC, y[q] * fminf(a * b[v][q], ce), w[q] * wdf);
                    }
                    write8<true>(w_, d, (i0 + r) * m + 8 * vec, 8, true, x, sp);
                }
            }
        }
        // every thread is done with slot st: refill it with chunk c + kMomStages
        if (__syncthreads_or(!ok)) {
            if (tid == 0) drain_copies(A.err, sm.full, kMomStages, c, min(nch, c + kMomStages));
            return;
        }
        if (tid == 0 && c + kMomStages < nch) {
            fence_proxy_async_smem();
            mom_issue(T, T.w, tile, c + kMomStages, sm.buf, sm.full, pol);
        }
    }
}

template <int TPB, int V>
__device__ void apply_rows_mom_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t tile,
                                    MomApplySmem &sm) {
    using L = RowLayout<TPB, V>;
    constexpr int NV = L::NV;
    const L lay;
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    const int64_t r0 = int64_t(tile) * T.at_rows;
    const uint32_t rows_t = (uint32_t)min((int64_t)T.at_rows, T.n - r0);
    const uint32_t nch = (rows_t + T.cr - 1) / T.cr;
    if (threadIdx.x == 0) {
        for (int st = 0; st < kMomStages; ++st) mbar_init(&sm.full[st], 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0)
        for (uint32_t c = 0; c < nch && c < (uint32_t)kMomStages; ++c) mom_issue(T, T.w, tile, c, sm.buf, sm.full, pol);
    const float rbar_s = __ldcg(&S.rbar_s);
    const int rbar_e = __ldcg(&S.rbar_e);
    float ma = 0.f, mb = 0.f;
    for (uint32_t r = threadIdx.x; r < rows_t; r += TPB) {
        const float a = row_scale(__ldcg(T.R + r0 + r), rbar_s, rbar_e);
        sm.a[r] = a;
        ma = fmaxf(ma, nan_to_inf(a));
    }
    float b[NV][8];
#pragma unroll
    for (int v = 0; v < NV; ++v) {
        const float *p = T.bsc + 8 * (v * TPB + lay.vi);
        const float4 b0 = __ldcg(reinterpret_cast<const float4 *>(p));
        const float4 b1 = __ldcg(reinterpret_cast<const float4 *>(p + 4));
        b[v][0] = b0.x; b[v][1] = b0.y; b[v][2] = b0.z; b[v][3] = b0.w;
        b[v][4] = b1.x; b[v][5] = b1.y; b[v][6] = b1.z; b[v][7] = b1.w;
#pragma unroll
        for (int k = 0; k < 8; ++k) mb = fmaxf(mb, nan_to_inf(b[v][k]));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        ma = fmaxf(ma, __shfl_xor_sync(kAll, ma, o));
        mb = fmaxf(mb, __shfl_xor_sync(kAll, mb, o));
    }
    if ((threadIdx.x & 31) == 0) {
        sm.red[threadIdx.x >> 5] = ma;
        sm.red[TPB / 32 + (threadIdx.x >> 5)] = mb;
    }
    __syncthreads();
    ma = mb = 0.f;
#pragma unroll
    for (int w = 0; w < TPB / 32; ++w) {
        ma = fmaxf(ma, sm.red[w]);
        mb = fmaxf(mb, sm.red[TPB / 32 + w]);
    }
    const float coefC = __ldcg(&S.coefC);
    if (ma * mb <= A.ce)
        apply_rows_mom_body<TPB, V, true>(A, T, tile, b, coefC, sm, nch, pol);
    else
        apply_rows_mom_body<TPB, V, false>(A, T, tile, b, coefC, sm, nch, pol);
}

// ---------------------------------------------------------------------------
// Kernels: one tile / item per CTA. The per-step parameters are a kernel
// parameter (constant bank), so the dither keys and step scalars are uniform
// operands of every warp.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads, SKEW_MINB_SUMSQ)
    k_sumsq(const __grid_constant__ StepArgs A, const uint2 *__restrict__ items) {
    __shared__ Smem sm;
    const Pol pol;
    const uint2 it = items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    if (T.vec)
        sumsq_tile<true>(T, it.y, sm, pol);
    else
        sumsq_tile<false>(T, it.y, sm, pol);
}

// Row path, phase A: one row tile per CTA (dynamic shared memory: RowSmem).
__global__ void __launch_bounds__(kRowThreads, 512 / kRowThreads)
    k_rowsq(const __grid_constant__ StepArgs A, const uint2 *__restrict__ items) {
    extern __shared__ uint4 dyn_smem[];
    RowSmem &sm = *reinterpret_cast<RowSmem *>(dyn_smem);
    const uint2 it = items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    TensorScal &S = A.scal[it.x];
    if (T.momentum) {
        MomRowSmem &ms = *reinterpret_cast<MomRowSmem *>(dyn_smem);
        switch (T.m) {
            case 4096: rowsq_mom_tile<kRowThreads, 512>(A, T, S, it.y, ms); break;
            case 2048: rowsq_mom_tile<kRowThreads, 256>(A, T, S, it.y, ms); break;
            case 1024: rowsq_mom_tile<kRowThreads, 128>(A, T, S, it.y, ms); break;
            default: rowsq_mom_tile<kRowThreads, 64>(A, T, S, it.y, ms); break;  // 512
        }
        return;
    }
    switch (T.m) {
        case 4096: rowsq_tile<kRowThreads, 512>(A, T, S, it.y, sm); break;
        case 2048: rowsq_tile<kRowThreads, 256>(A, T, S, it.y, sm); break;
        case 1024: rowsq_tile<kRowThreads, 128>(A, T, S, it.y, sm); break;
        default: rowsq_tile<kRowThreads, 64>(A, T, S, it.y, sm); break;  // 512
    }
}

// Row path, phase C: one row tile per CTA (dynamic shared memory: ApplyRowSmem).
__global__ void __launch_bounds__(kRowThreads, 512 / kRowThreads)
    k_apply_rows(const __grid_constant__ StepArgs A, const uint2 *__restrict__ items) {
    extern __shared__ uint4 dyn_smem[];
    ApplyRowSmem &sm = *reinterpret_cast<ApplyRowSmem *>(dyn_smem);
    const uint2 it = items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    const TensorScal &S = A.scal[it.x];
    if (T.momentum) {
        MomApplySmem &ms = *reinterpret_cast<MomApplySmem *>(dyn_smem);
        switch (T.m) {
            case 4096: apply_rows_mom_tile<kRowThreads, 512>(A, T, S, it.y, ms); break;
            case 2048: apply_rows_mom_tile<kRowThreads, 256>(A, T, S, it.y, ms); break;
            case 1024: apply_rows_mom_tile<kRowThreads, 128>(A, T, S, it.y, ms); break;
            default: apply_rows_mom_tile<kRowThreads, 64>(A, T, S, it.y, ms); break;  // 512
        }
        return;
    }
    switch (T.m) {
        case 4096: apply_rows_tile<kRowThreads, 512>(A, T, S, it.y, sm); break;
        case 2048: apply_rows_tile<kRowThreads, 256>(A, T, S, it.y, sm); break;
        case 1024: apply_rows_tile<kRowThreads, 128>(A, T, S, it.y, sm); break;
        default: apply_rows_tile<kRowThreads, 64>(A, T, S, it.y, sm); break;  // 512
    }
}

// Phase B of the row-path tensors whose finalize found that a clamp may bind
// (queued in A.fb): the CTAs of this grid split each such tensor's tiles.
__global__ void __launch_bounds__(kThreads, 2) k_fallback(const __grid_constant__ StepArgs A) {
    __shared__ Smem sm;
    __shared__ Meta meta;
    const Pol pol;
    const uint32_t cnt = __ldcg(A.fb);
    for (uint32_t q = 0; q < cnt; ++q) {
        const uint32_t t = __ldcg(A.fb + 1 + q);
        const TensorDev &T = A.tensors[t];
        for (uint32_t tile = blockIdx.x; tile < T.ntiles; tile += gridDim.x) {
            (void)fill_meta(T, A.scal[t], tile, A.ce, meta);
            phase_B(A, t, tile, sm, meta, pol);
            __syncthreads();
        }
    }
}

__global__ void __launch_bounds__(kThreads) k_finalize(const __grid_constant__ StepArgs A, const uint2 *__restrict__ items) {
    __shared__ Smem sm;
    const uint2 it = items[blockIdx.x];
    phase_F(A, it.x, it.y, sm);
}

__global__ void __launch_bounds__(kThreads, SKEW_MINB_RMS)
    k_rms(const __grid_constant__ StepArgs A, const uint2 *__restrict__ items) {
    __shared__ Smem sm;
    __shared__ Meta meta;
    const Pol pol;
    const uint2 it = items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    if (T.kind == kKindFactored) (void)fill_meta(T, A.scal[it.x], it.y, A.ce, meta);
    phase_B(A, it.x, it.y, sm, meta, pol);
}

__global__ void __launch_bounds__(kThreads, SKEW_MINB_APPLY)
    k_apply(const __grid_constant__ StepArgs A, const uint2 *__restrict__ items) {
    __shared__ Meta meta;
    const Pol pol;
    const uint2 it = items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    const TensorScal &S = A.scal[it.x];
    if (T.kind == kKindFactored) {
        const bool fast = fill_meta(T, S, it.y, A.ce, meta);
        if (T.vec) {
            if (T.momentum) {
                if (fast)
                    apply_fact_tile<true, true, true>(A, T, S, it.y, meta, pol);
                else
                    apply_fact_tile<true, true, false>(A, T, S, it.y, meta, pol);
            } else {
                if (fast)
                    apply_fact_tile<true, false, true>(A, T, S, it.y, meta, pol);
                else
                    apply_fact_tile<true, false, false>(A, T, S, it.y, meta, pol);
            }
        } else {
            if (T.momentum)
                apply_fact_tile<false, true, false>(A, T, S, it.y, meta, pol);
            else
                apply_fact_tile<false, false, false>(A, T, S, it.y, meta, pol);
        }
    } else {
        if (T.vec)
            apply_full_tile<true>(A, T, S, it.y, pol);
        else
            apply_full_tile<false>(A, T, S, it.y, pol);
    }
}

// Self-test of the bounded wait: one thread waits, exactly as the row kernels wait for
// a chunk, on an mbarrier phase that nothing completes (no arrival, no transaction);
// the wait gives up after kMbarPolls polls and the timeout lands in the status word.
__global__ void k_wait_selftest(uint32_t *err) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
        if (!mbar_wait(&bar, 0u)) atomicOr(err, 2u);
    }
}

}  // namespace

int launch_wait_selftest(uint32_t *err, void *stream) {
    k_wait_selftest<<<1, 32, 0, (cudaStream_t)stream>>>(err);
    return (int)cudaGetLastError();
}

int launch_phases(const StepArgs &A, const LaunchPlan &L, void *stream, void *const *ev) {
    cudaStream_t s = (cudaStream_t)stream;
    auto mark = [&](int k) {
        if (ev) cudaEventRecord((cudaEvent_t)ev[k], s);
    };
    mark(0);
    if (L.nA) k_sumsq<<<L.nA, kThreads, 0, s>>>(A, L.itemsA);
    mark(1);
    if (L.nR) {
        constexpr size_t kSm = sizeof(RowSmem) > sizeof(MomRowSmem) ? sizeof(RowSmem) : sizeof(MomRowSmem);
        const cudaError_t e = cudaFuncSetAttribute(k_rowsq, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSm);
        if (e != cudaSuccess) return (int)e;
        k_rowsq<<<L.nR, kRowThreads, kSm, s>>>(A, L.itemsR);
    }
    mark(2);
    if (L.nF) k_finalize<<<L.nF, kThreads, 0, s>>>(A, L.itemsF);
    mark(3);
    if (L.nB) k_rms<<<L.nB, kThreads, 0, s>>>(A, L.itemsB);
    mark(4);
    if (L.nFB) k_fallback<<<L.nFB, kThreads, 0, s>>>(A);
    mark(5);
    if (L.nC) k_apply<<<L.nC, kThreads, 0, s>>>(A, L.itemsC);
    mark(6);
    if (L.nCR) {
        constexpr size_t kSm =
            sizeof(ApplyRowSmem) > sizeof(MomApplySmem) ? sizeof(ApplyRowSmem) : sizeof(MomApplySmem);
        const cudaError_t e = cudaFuncSetAttribute(k_apply_rows, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSm);
        if (e != cudaSuccess) return (int)e;
        k_apply_rows<<<L.nCR, kRowThreads, kSm, s>>>(A, L.itemsCR);
    }
    mark(7);
    return (int)cudaGetLastError();
}

}  // namespace skew
