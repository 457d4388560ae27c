// Device kernels of libskewadam (sm_103a).
//
// One SkewAdam step (paper Sec. 3, Eq. 1, Algorithm 1) over every tensor of a
// handle, as four grouped launches over device-side item tables:
//   k_sumsq    : per-row and per-column sums of g^2 of every factored matrix
//                (Eq. 1), 16-byte bf16 loads, warp-shuffle row sums, column
//                partials reduced across the CTA in shared memory and written
//                per row tile (deterministic: no float atomics);
//   k_finalize : R <- b2 R + (1-b2) mean_c(G^2), C <- b2 C + (1-b2) mean_r(G^2),
//                1/sqrt(C_j) per column, and mean(R) by the last item of a tensor;
//   k_rms      : the tier's momentum / exact second moment update, U up to its
//                scalar coefficient, and sum(U^2) per tile; the last tile of a
//                tensor forms RMS(U) and the clip factor (Sec. 3 update clipping);
//   k_apply    : x = w (1 - lr*lambda) - lr*kappa*U in fp32 and the dithered
//                bf16 write-back with a Philox-4x32-10 counter hash.
// The reconstructed second moment of a factored matrix is never formed:
// 1/sqrt(max(R_i C_j / Rbar, eps)) = min(a_i * b_j, 1/sqrt(eps)) with
// a_i = 1/sqrt(R_i / Rbar) per row and b_j = 1/sqrt(C_j) per column.
#include <cuda_runtime.h>
#include <stdint.h>

#include "skew_plan.h"

namespace skew {
namespace {

constexpr uint32_t kAll = 0xFFFFFFFFu;
constexpr int kSmemFloats = kVecPerThread * kThreads;  // row scales of the tallest tile

// ---------------------------------------------------------------------------
// Small helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float(uint32_t(h) << 16); }

// Eight bf16 values at p (16-byte aligned when VEC) -> fp32; lanes >= valid read as 0.
template <bool VEC>
__device__ __forceinline__ void load_bf8(const uint16_t *p, int valid, float (&o)[8]) {
    if (VEC) {
        const uint4 u = *reinterpret_cast<const uint4 *>(p);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            o[2 * q] = __uint_as_float(w[q] << 16);
            o[2 * q + 1] = __uint_as_float(w[q] & 0xFFFF0000u);
        }
    } else {
#pragma unroll
        for (int c = 0; c < 8; ++c) o[c] = c < valid ? bf16_to_f32(p[c]) : 0.f;
    }
}

template <bool VEC>
__device__ __forceinline__ void load_f8(const float *p, int valid, float (&o)[8]) {
    if (VEC) {
        const float4 a = *reinterpret_cast<const float4 *>(p);
        const float4 b = *reinterpret_cast<const float4 *>(p + 4);
        o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
        o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
    } else {
#pragma unroll
        for (int c = 0; c < 8; ++c) o[c] = c < valid ? p[c] : 0.f;
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

// Philox-4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32
// multiplies whose high halves are xored with the other counter words and the
// round key; the key advances by two Weyl constants between rounds.
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

// The 16-bit dithers of the eight elements idx0 .. idx0+7 (idx0 a multiple of 8):
// counter (idx0/8 lo, idx0/8 hi, tensor id, step lo), key (seed lo, seed hi);
// element k takes half (k & 1) of word k >> 1.
__device__ __forceinline__ void dither8(uint64_t idx0, uint32_t tid, const StepArgs &A, uint32_t (&r)[8]) {
    const uint64_t blk = idx0 >> 3;
    const uint4 o = philox4x32_10((uint32_t)blk, (uint32_t)(blk >> 32), tid, A.step_lo, A.seed_lo, A.seed_hi);
    const uint32_t w[4] = {o.x, o.y, o.z, o.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        r[2 * q] = w[q] & 0xFFFFu;
        r[2 * q + 1] = w[q] >> 16;
    }
}

__device__ __forceinline__ uint32_t dither1(uint64_t idx, uint32_t tid, const StepArgs &A) {
    const uint64_t blk = idx >> 3;
    const uint4 o = philox4x32_10((uint32_t)blk, (uint32_t)(blk >> 32), tid, A.step_lo, A.seed_lo, A.seed_hi);
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

// a_i = 1/sqrt(R_i / Rbar), with Rbar = rbar_s * 2^-rbar_e (rbar_s in [1,2)); +inf if Rbar == 0.
__device__ __forceinline__ float row_scale(float Ri, float rbar_s, int rbar_e) {
    if (rbar_s == 0.f) return __int_as_float(0x7F800000);
    return __frsqrt_rn(__fdiv_rn(ldexpf(Ri, rbar_e), rbar_s));
}

// Error-free sum (Knuth's TwoSum): s + e == a + b exactly.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bp = s - a;
    e = (a - (s - bp)) + (b - bp);
}

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

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kAll, v, o);
    return v;
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

// Geometry of a factored tile: LC lanes along a row, RG row groups, 16 rows per thread.
struct FactTile {
    uint32_t LC, RG, lane, rg;
    int64_t col0, row0;
    int valid;
    bool act;
    __device__ FactTile(const TensorDev &T, uint32_t tile) {
        LC = 1u << T.lcl;
        RG = kThreads >> T.lcl;
        const uint32_t s = tile % T.strips, rt = tile / T.strips;
        lane = threadIdx.x & (LC - 1);
        rg = threadIdx.x >> T.lcl;
        col0 = int64_t(s) * 8 * LC + 8 * lane;
        act = col0 < T.m;
        valid = act ? (int)min(int64_t(8), T.m - col0) : 0;
        row0 = int64_t(rt) * T.tile_rows + rg;
    }
};

// ---------------------------------------------------------------------------
// Phase 1: per-row / per-column sums of g^2 (Eq. 1).
// ---------------------------------------------------------------------------
template <bool VEC>
__device__ void sumsq_tile(const TensorDev &T, uint32_t tile, float *sm) {
    const FactTile F(T, tile);
    const uint32_t s = tile % T.strips, rt = tile / T.strips;
    float col[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
    for (int k = 0; k < kVecPerThread; ++k) {
        const int64_t i = F.row0 + int64_t(k) * F.RG;
        float g[8];
        if (F.act && i < T.n)
            load_bf8<VEC>(T.g + i * T.m + F.col0, F.valid, g);
        else
#pragma unroll
            for (int c = 0; c < 8; ++c) g[c] = 0.f;
        float rs = 0.f;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const float q = g[c] * g[c];
            col[c] += q;
            rs += q;
        }
        for (uint32_t o = F.LC >> 1; o; o >>= 1) rs += __shfl_xor_sync(kAll, rs, o);
        if (F.lane == 0 && i < T.n) T.rowp[int64_t(s) * T.n + i] = rs;
    }
#pragma unroll
    for (int c = 0; c < 8; ++c) sm[threadIdx.x * 8 + c] = col[c];
    __syncthreads();
    const uint32_t width = 8 * F.LC;
    for (uint32_t cc = threadIdx.x; cc < width; cc += kThreads) {
        float acc = 0.f;
        for (uint32_t r = 0; r < F.RG; ++r) acc += sm[r * width + cc];
        const int64_t j = int64_t(s) * width + cc;
        if (j < T.m) T.colp[int64_t(rt) * T.m + j] = acc;
    }
}

__global__ void __launch_bounds__(kThreads) k_sumsq(StepArgs A) {
    __shared__ float sm[kThreads * 8];
    const uint2 it = A.items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    if (T.vec)
        sumsq_tile<true>(T, it.y, sm);
    else
        sumsq_tile<false>(T, it.y, sm);
}

// ---------------------------------------------------------------------------
// Phase 2: factor EMAs, 1/sqrt(C_j), mean(R) (Eq. 1).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) k_finalize(StepArgs A) {
    __shared__ double red[kThreads / 32];
    __shared__ int last;
    const uint2 it = A.items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    TensorScal &S = A.scal[it.x];
    if (it.y < T.nfr) {
        const int64_t i = int64_t(it.y) * kFinChunk + threadIdx.x;
        double rd = 0.0;
        if (i < T.n) {
            float rs = 0.f;
            for (uint32_t s = 0; s < T.strips; ++s) rs += T.rowp[int64_t(s) * T.n + i];
            const float mean = __fdiv_rn(rs, (float)T.m);
            const float Rn = fmaf(A.b2, T.R[i], A.c2 * mean);
            T.R[i] = Rn;
            rd = (double)Rn;
        }
        rd = block_sum_d(rd, red);
        if (threadIdx.x == 0) T.rsum[it.y] = rd;
    } else {
        const int64_t j = int64_t(it.y - T.nfr) * kFinChunk + threadIdx.x;
        if (j < T.m) {
            float cs = 0.f;
            for (uint32_t r = 0; r < T.rowtiles; ++r) cs += T.colp[int64_t(r) * T.m + j];
            const float mean = __fdiv_rn(cs, (float)T.n);
            const float Cn = fmaf(A.b2, T.C[j], A.c2 * mean);
            T.C[j] = Cn;
            T.bsc[j] = __frsqrt_rn(Cn);
        }
    }
    // The last finalize item of the tensor forms mean(R) from the row items' partial sums.
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t done = atomicAdd(&S.cntF, 1u);
        last = (done == T.nfr + T.nfc - 1);
    }
    __syncthreads();
    if (last && threadIdx.x == 0) {
        __threadfence();
        double s = 0.0;
        for (uint32_t f = 0; f < T.nfr; ++f) s += __ldcg(T.rsum + f);
        const double rbar = s / (double)T.n;
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
}

// ---------------------------------------------------------------------------
// Phase 3: second moment / momentum update and sum(U^2) (Algorithm 1).
// ---------------------------------------------------------------------------
template <bool VEC>
__device__ Acc2 rms_fact_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t tile, float *sm) {
    const FactTile F(T, tile);
    const uint32_t rt = tile / T.strips;
    for (uint32_t r = threadIdx.x; r < T.tile_rows; r += kThreads) {
        const int64_t i = int64_t(rt) * T.tile_rows + r;
        sm[r] = i < T.n ? row_scale(T.R[i], S.rbar_s, S.rbar_e) : 0.f;
    }
    __syncthreads();
    float b[8];
    if (F.act)
        load_f8<VEC>(T.bsc + F.col0, F.valid, b);
    Acc2 acc;
    if (!F.act) return acc;
#pragma unroll 2
    for (int k = 0; k < kVecPerThread; ++k) {
        const int64_t i = F.row0 + int64_t(k) * F.RG;
        if (i >= T.n) break;
        const int64_t e0 = i * T.m + F.col0;
        float y[8];
        load_bf8<VEC>(T.g + e0, F.valid, y);
        if (T.momentum) {
            float mm[8];
            load_f8<VEC>(T.M + e0, F.valid, mm);
#pragma unroll
            for (int c = 0; c < 8; ++c) y[c] = fmaf(A.b1, mm[c], A.c1 * y[c]);
            store_f8<VEC>(T.M + e0, F.valid, y);
        }
        const float a = sm[F.rg + k * F.RG];
        float u[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) u[c] = c < F.valid ? y[c] * fminf(a * b[c], A.ce) : 0.f;
        acc.add(sumsq8(u));
    }
    return acc;
}

template <bool VEC>
__device__ Acc2 rms_full_tile(const StepArgs &A, const TensorDev &T, uint32_t tile) {
    Acc2 acc;
    for (int k = 0; k < kVecPerThread; ++k) {
        const int64_t e0 = 8 * (int64_t(tile) * kThreads * kVecPerThread + int64_t(k) * kThreads + threadIdx.x);
        if (e0 >= T.numel) break;
        const int valid = (int)min(int64_t(8), T.numel - e0);
        float g[8], v[8], y[8];
        load_bf8<VEC>(T.g + e0, valid, g);
        load_f8<VEC>(T.v + e0, valid, v);
#pragma unroll
        for (int c = 0; c < 8; ++c) v[c] = fmaf(A.b2, v[c], A.c2 * (g[c] * g[c]));
        store_f8<VEC>(T.v + e0, valid, v);
        if (T.momentum) {
            float mm[8];
            load_f8<VEC>(T.M + e0, valid, mm);
#pragma unroll
            for (int c = 0; c < 8; ++c) y[c] = fmaf(A.b1, mm[c], A.c1 * g[c]);
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

__global__ void __launch_bounds__(kThreads) k_rms(StepArgs A) {
    __shared__ float sm[kSmemFloats];
    __shared__ float2 red[kThreads / 32];
    __shared__ double redd[kThreads / 32];
    __shared__ int last;
    const uint2 it = A.items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    TensorScal &S = A.scal[it.x];
    Acc2 acc;
    if (T.kind == kKindFactored)
        acc = T.vec ? rms_fact_tile<true>(A, T, S, it.y, sm) : rms_fact_tile<false>(A, T, S, it.y, sm);
    else
        acc = T.vec ? rms_full_tile<true>(A, T, it.y) : rms_full_tile<false>(A, T, it.y);
    const float2 tsum = block_sum2(acc, red);
    if (threadIdx.x == 0) {
        T.u2[it.y] = tsum;
        __threadfence();
        const uint32_t done = atomicAdd(&S.cntB, 1u);
        last = (done == T.ntiles - 1);
    }
    __syncthreads();
    if (!last) return;
    // Last tile of the tensor: sum(U^2), RMS, clip factor (fixed summation order).
    __threadfence();
    double s = 0.0;
    for (uint32_t k = threadIdx.x; k < T.ntiles; k += kThreads) {
        const float2 p = __ldcg(T.u2 + k);
        s += (double)p.x + (double)p.y;
    }
    s = block_sum_d(s, redd);
    if (threadIdx.x == 0) {
        const double coef = T.momentum ? A.coef_mom : A.coef_plain;
        const double su2 = s * coef * coef;
        const double rms = sqrt(su2 / (double)T.numel);
        const double kappa = 1.0 / fmax(1.0, rms / (double)A.clip_d);
        S.sumsq = su2;
        S.rms = rms;
        S.kappa = kappa;
        S.coefC = (float)((double)A.lr * kappa * coef);
    }
}

// ---------------------------------------------------------------------------
// Phase 4: decoupled decay, clipped update, dithered bf16 write-back.
// ---------------------------------------------------------------------------
template <bool VEC>
__device__ __forceinline__ void write8(const StepArgs &A, const TensorDev &T, int64_t e0, int valid, bool aligned8,
                                       const float (&x)[8]) {
    if (VEC) {
        uint32_t r[8];
        dither8((uint64_t)e0, T.tid, A, r);
        uint32_t o[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) o[q] = sr_bf16(x[2 * q], r[2 * q]) | (sr_bf16(x[2 * q + 1], r[2 * q + 1]) << 16);
        *reinterpret_cast<uint4 *>(T.w + e0) = make_uint4(o[0], o[1], o[2], o[3]);
    } else {
        uint32_t r[8];
        if (aligned8) dither8((uint64_t)e0, T.tid, A, r);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            if (c < valid) {
                const uint32_t rc = aligned8 ? r[c] : dither1((uint64_t)(e0 + c), T.tid, A);
                T.w[e0 + c] = (uint16_t)sr_bf16(x[c], rc);
            }
        }
    }
}

template <bool VEC>
__device__ void apply_fact_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t tile, float *sm) {
    const FactTile F(T, tile);
    const uint32_t rt = tile / T.strips;
    for (uint32_t r = threadIdx.x; r < T.tile_rows; r += kThreads) {
        const int64_t i = int64_t(rt) * T.tile_rows + r;
        sm[r] = i < T.n ? row_scale(T.R[i], S.rbar_s, S.rbar_e) : 0.f;
    }
    __syncthreads();
    if (!F.act) return;
    float b[8];
    load_f8<VEC>(T.bsc + F.col0, F.valid, b);
    const float coefC = S.coefC;
    const float wdf = T.decay ? A.wdf : 1.0f;
#pragma unroll 2
    for (int k = 0; k < kVecPerThread; ++k) {
        const int64_t i = F.row0 + int64_t(k) * F.RG;
        if (i >= T.n) break;
        const int64_t e0 = i * T.m + F.col0;
        float y[8], w[8], x[8];
        if (T.momentum)
            load_f8<VEC>(T.M + e0, F.valid, y);
        else
            load_bf8<VEC>(T.g + e0, F.valid, y);
        load_bf8<VEC>(T.w + e0, F.valid, w);
        const float a = sm[F.rg + k * F.RG];
#pragma unroll
        for (int c = 0; c < 8; ++c) x[c] = fmaf(-coefC, y[c] * fminf(a * b[c], A.ce), w[c] * wdf);
        write8<VEC>(A, T, e0, F.valid, (e0 & 7) == 0, x);
    }
}

template <bool VEC>
__device__ void apply_full_tile(const StepArgs &A, const TensorDev &T, const TensorScal &S, uint32_t tile) {
    const float coefC = S.coefC;
    const float wdf = T.decay ? A.wdf : 1.0f;
    for (int k = 0; k < kVecPerThread; ++k) {
        const int64_t e0 = 8 * (int64_t(tile) * kThreads * kVecPerThread + int64_t(k) * kThreads + threadIdx.x);
        if (e0 >= T.numel) break;
        const int valid = (int)min(int64_t(8), T.numel - e0);
        float y[8], v[8], w[8], x[8];
        if (T.momentum)
            load_f8<VEC>(T.M + e0, valid, y);
        else
            load_bf8<VEC>(T.g + e0, valid, y);
        load_f8<VEC>(T.v + e0, valid, v);
        load_bf8<VEC>(T.w + e0, valid, w);
#pragma unroll
        for (int c = 0; c < 8; ++c) x[c] = fmaf(-coefC, y[c] * fminf(__frsqrt_rn(v[c]), A.ce), w[c] * wdf);
        write8<VEC>(A, T, e0, valid, true, x);
    }
}

__global__ void __launch_bounds__(kThreads) k_apply(StepArgs A) {
    __shared__ float sm[kSmemFloats];
    const uint2 it = A.items[blockIdx.x];
    const TensorDev &T = A.tensors[it.x];
    const TensorScal &S = A.scal[it.x];
    if (T.kind == kKindFactored) {
        if (T.vec)
            apply_fact_tile<true>(A, T, S, it.y, sm);
        else
            apply_fact_tile<false>(A, T, S, it.y, sm);
    } else {
        if (T.vec)
            apply_full_tile<true>(A, T, S, it.y);
        else
            apply_full_tile<false>(A, T, S, it.y);
    }
}

}  // namespace

const char *const kKernelNames[kNumKernels] = {"k_sumsq", "k_finalize", "k_rms", "k_apply"};

int launch_step(const LaunchPlan &P, const StepArgs &A0, void *stream) {
    cudaStream_t s = (cudaStream_t)stream;
    StepArgs A = A0;
    auto mark = [&](int k) {
        if (P.events) cudaEventRecord((cudaEvent_t)P.events[k], s);
    };
    mark(0);
    if (P.nA) {
        A.items = P.itemsA;
        k_sumsq<<<P.nA, kThreads, 0, s>>>(A);
    }
    mark(1);
    if (P.nF) {
        A.items = P.itemsF;
        k_finalize<<<P.nF, kThreads, 0, s>>>(A);
    }
    mark(2);
    if (P.nBC) {
        A.items = P.itemsBC;
        k_rms<<<P.nBC, kThreads, 0, s>>>(A);
    }
    mark(3);
    if (P.nBC) k_apply<<<P.nBC, kThreads, 0, s>>>(A);
    mark(4);
    return (int)cudaGetLastError();
}

}  // namespace skew
