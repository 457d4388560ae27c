// skew_step_tensor_noalloc: a SkewAdam step over one tensor that allocates nothing.
//
// The regular path (skew_create / skew_bind / skew_step) needs a caller-allocated
// workspace for its scratch: row / column partial sums, per-tile sums of U^2,
// per-tensor scalars and the tile tables. Some callers cannot allocate device
// memory at the point where they step the optimizer -- for example code that
// runs while a framework's caching allocator owns every free byte, plugins that
// are handed only pre-sized buffers, or runtimes that forbid cudaMalloc after
// start-up. For them this entry point keeps the scratch in a fixed array
// compiled into the library (g_scratch below, SKEW_NOALLOC_SCRATCH_BYTES bytes
// in the device memory of every GPU that loads the library, held until the
// process exits) and launches the same kernels as skew_step.
//
// The array's address is a device address that host code cannot name
// directly: the host-side symbol is only a stand-in. Every call looks it up
// with cudaGetSymbolAddress for the current device (cheap once the module is
// loaded; a cached address could go stale after cudaDeviceReset).
//
// The array's first bytes hold a status word of its own: the bounded waits of
// the whole-row kernels set it when a copy does not land, every call leaves it
// as it is, and skew_noalloc_sync_status reads and clears it.
#include <cuda_runtime.h>

#include <cmath>

#include "skew_plan.h"
#include "skewadam.h"

namespace skew {
namespace {

static __device__ __align__(256) unsigned char g_scratch[SKEW_NOALLOC_SCRATCH_BYTES];

// Offset of the status word in the array (kept apart from any call's scratch layout).
constexpr size_t kErrOffset = 0;
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// The array's device address on the current device, or null.
unsigned char *scratch_base() {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess) return nullptr;
    return static_cast<unsigned char *>(p);
}

struct SetupTables {
    uint2 *A;
    uint32_t nA;
    uint2 *R;
    uint32_t nR;
    uint2 *F;
    uint32_t nF;
    uint2 *B;
    uint32_t nB;
    uint2 *C;
    uint32_t nC;
    uint2 *CR;
    uint32_t nCR;
};

// Writes the descriptor, clears the scalars and the phase-B queue (the step's
// completion counters must start at zero) and fills the item tables of one tensor.
__global__ void k_noalloc_setup(TensorDev td, TensorDev *dst, TensorScal *scal, uint32_t *fb, SetupTables tb) {
    const uint32_t stride = gridDim.x * blockDim.x;
    const uint32_t i0 = blockIdx.x * blockDim.x + threadIdx.x;
    if (i0 == 0) {
        *dst = td;
        *scal = TensorScal{};
        fb[0] = 0u;
    }
    for (uint32_t i = i0; i < tb.nA; i += stride) tb.A[i] = make_uint2(0, i);
    for (uint32_t i = i0; i < tb.nR; i += stride) tb.R[i] = make_uint2(0, i);
    for (uint32_t i = i0; i < tb.nF; i += stride) tb.F[i] = make_uint2(0, i);
    for (uint32_t i = i0; i < tb.nB; i += stride) tb.B[i] = make_uint2(0, i);
    for (uint32_t i = i0; i < tb.nC; i += stride) tb.C[i] = make_uint2(0, i);
    for (uint32_t i = i0; i < tb.nCR; i += stride) tb.CR[i] = make_uint2(0, i);
}

}  // namespace
}  // namespace skew

using namespace skew;

extern "C" int skew_step_tensor_noalloc(void *weight, const void *grad, int32_t ndim, int64_t rows, int64_t cols,
                                        int32_t tier, uint32_t flags, const skew_hparams_t *hp, void *state,
                                        size_t state_bytes, uint32_t tensor_id, int64_t step, float lr, uint64_t seed,
                                        void *stream) {
    // ---- arguments (same rules as skew_create / skew_step) ------------------
    if (!hp || !weight || !grad || !state) return SKEW_EINVAL;
    if (((uintptr_t)weight & 1) || ((uintptr_t)grad & 1)) return SKEW_EINVAL;
    if (((uintptr_t)state & 3)) return SKEW_EINVAL;
    if (ndim != 1 && ndim != 2) return SKEW_EINVAL;
    if (tier < SKEW_TIER_BACKBONE || tier > SKEW_TIER_ROUTER) return SKEW_EINVAL;
    if (flags & ~(SKEW_F_NO_DECAY | SKEW_F_FP32)) return SKEW_EINVAL;
    const bool f32 = (flags & SKEW_F_FP32) != 0;
    if (f32 && (((uintptr_t)weight | (uintptr_t)grad) & 3)) return SKEW_EINVAL;
    const skew_hparams_t H = *hp;
    if (!std::isfinite(H.beta1) || H.beta1 < 0.f || H.beta1 >= 1.f) return SKEW_EINVAL;
    if (!std::isfinite(H.beta2) || H.beta2 < 0.f || H.beta2 >= 1.f) return SKEW_EINVAL;
    if (!std::isfinite(H.eps) || !(H.eps > 0.f)) return SKEW_EINVAL;
    if (!std::isfinite(H.clip_d) || !(H.clip_d > 0.f)) return SKEW_EINVAL;
    if (!std::isfinite(H.weight_decay) || H.weight_decay < 0.f) return SKEW_EINVAL;
    if (H.policy < SKEW_POLICY_TIERED || H.policy > SKEW_POLICY_ADAFACTOR) return SKEW_EINVAL;
    if (step < 1) return SKEW_EINVAL;
    if (!std::isfinite(lr) || lr < 0.f) return SKEW_EINVAL;
    const int64_t n = rows, m = ndim == 2 ? cols : 1;
    if (n < 1 || m < 1 || n > (int64_t(1) << 40) || m > (int64_t(1) << 40) || n > (int64_t(1) << 62) / m)
        return SKEW_EINVAL;
    const int64_t numel = n * m;

    // ---- tier policy (as the planner's, Sec. 3 "The tiers" / Table 3) -------------
    uint32_t kind, momentum, decay;
    resolve_policy(ndim, tier, H.policy, flags, kind, momentum, decay);

    // ---- caller's state: [M][v][R][C] of this tensor, exactly the closed form -----
    const int64_t state_floats = (momentum ? numel : 0) + (kind == kKindFull ? numel : n + m);
    if (state_bytes != size_t(state_floats) * 4) return SKEW_EINVAL;
    float *sf = reinterpret_cast<float *>(state);
    float *M = momentum ? sf : nullptr;
    float *after_m = sf + (momentum ? numel : 0);
    float *v = kind == kKindFull ? after_m : nullptr;
    float *R = kind == kKindFactored ? after_m : nullptr;
    float *Cc = kind == kKindFactored ? after_m + n : nullptr;

    // ---- tile geometry and item counts (the planner's, plan_geometry) ---------------
    const bool wg_aligned = !f32 && (((uintptr_t)weight | (uintptr_t)grad) & 15) == 0;  // row tiles: bf16 only
    const int64_t tiles64 = kind == kKindFactored ? ((m + 255) / 256) * ((n + 255) / 256)
                                                  : (numel + kFlatTileElems - 1) / kFlatTileElems;
    if (tiles64 > (int64_t(1) << 31)) return SKEW_EINVAL;
    const TileGeom G = plan_geometry(kind, momentum, wg_aligned, n, m, numel);
    const bool fact = kind == kKindFactored, row = fact && G.rowpath;
    const uint32_t nA = fact && !row ? G.ntiles : 0, nR = row ? G.rtiles : 0, nF = fact ? G.nfr + G.nfc : 0;
    const uint32_t nB = row ? 0 : G.ntiles, nC = row ? 0 : G.ntiles, nCR = row ? G.atiles : 0;

    // ---- scratch layout inside the fixed array --------------------------------------
    size_t off = align256(kErrOffset + 16);  // the status word comes first
    const size_t o_scal = off;   off = align256(off + sizeof(TensorScal));
    const size_t o_fb = off;     off = align256(off + 8);
    const size_t o_err = kErrOffset;
    const size_t o_tens = off;   off = align256(off + sizeof(TensorDev));
    const size_t o_iA = off;     off = align256(off + sizeof(uint2) * nA);
    const size_t o_iR = off;     off = align256(off + sizeof(uint2) * nR);
    const size_t o_iF = off;     off = align256(off + sizeof(uint2) * nF);
    const size_t o_iB = off;     off = align256(off + sizeof(uint2) * nB);
    const size_t o_iC = off;     off = align256(off + sizeof(uint2) * nC);
    const size_t o_iCR = off;    off = align256(off + sizeof(uint2) * nCR);
    size_t o_rowp = 0, o_colp = 0, o_bsc = 0, o_rsum = 0, o_pp = 0, o_rmin = 0, o_fsum = 0, o_fmin = 0;
    if (fact && !row) {
        o_rowp = off; off = align256(off + 4 * size_t(G.strips) * n);
        o_colp = off; off = align256(off + 4 * size_t(G.rowtiles) * m);
        o_bsc = off;  off = align256(off + 4 * size_t(m));
        o_rsum = off; off = align256(off + 8 * size_t(G.nfr));
    } else if (row) {
        o_pp = off;   off = align256(off + 8 * size_t(G.rtiles) * m);
        o_bsc = off;  off = align256(off + 4 * size_t(m));
        o_rsum = off; off = align256(off + 8 * size_t(G.rtiles));
        o_rmin = off; off = align256(off + 4 * size_t(G.rtiles));
        o_fsum = off; off = align256(off + 8 * size_t(G.nfc));
        o_fmin = off; off = align256(off + 4 * size_t(G.nfc));
    }
    const size_t o_u2 = off;     off = align256(off + 8 * size_t(G.ntiles));
    if (off > SKEW_NOALLOC_SCRATCH_BYTES) return SKEW_ETOOBIG;  // too large for the fixed array

    // ---- device address of the fixed array on the current device ---------------------
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return SKEW_ECUDA;
    unsigned char *const base = scratch_base();
    if (!base) return SKEW_ECUDA;  // the array's device address is unknown

    TensorDev td{};
    td.w = (uint16_t *)weight;
    td.g = (const uint16_t *)grad;
    td.M = M;
    td.v = v;
    td.R = R;
    td.C = Cc;
    td.rowp = fact && !row ? (float *)(base + o_rowp) : nullptr;
    td.colp = fact && !row ? (float *)(base + o_colp) : nullptr;
    td.bsc = fact ? (float *)(base + o_bsc) : nullptr;
    td.rsum = fact ? (double *)(base + o_rsum) : nullptr;
    td.pp = row ? (float2 *)(base + o_pp) : nullptr;
    td.rmin = row ? (float *)(base + o_rmin) : nullptr;
    td.fsum = row ? (double *)(base + o_fsum) : nullptr;
    td.fmin = row ? (float *)(base + o_fmin) : nullptr;
    td.u2 = (float2 *)(base + o_u2);
    td.n = n;
    td.m = m;
    td.numel = numel;
    td.tid = tensor_id;
    td.kind = kind;
    td.momentum = momentum;
    td.decay = decay;
    auto al16 = [](const void *p) { return ((uintptr_t)p & 15) == 0; };
    bool vec = !f32 && al16(td.w) && al16(td.g) && (!td.M || al16(td.M));
    vec = kind == kKindFull ? (vec && numel % 8 == 0 && al16(td.v)) : (vec && m % 8 == 0);
    td.vec = vec ? 1 : 0;
    td.f32 = f32 ? 1u : 0u;
    td.lcl = G.lcl;
    td.strips = G.strips;
    td.rowtiles = G.rowtiles;
    td.tile_rows = G.tile_rows;
    td.ntiles = G.ntiles;
    td.nfr = G.nfr;
    td.nfc = G.nfc;
    td.rowpath = G.rowpath;
    td.cr = G.cr;
    td.rt_rows = G.rt_rows;
    td.rtiles = G.rtiles;
    td.at_rows = G.at_rows;
    td.atiles = G.atiles;
    td.fci = G.fci;

    // ---- per-step scalars, as skew_step forms them ------------------------------------
    const StepCoefs k = step_coefs(H, step);
    StepArgs a{};
    a.tensors = (const TensorDev *)(base + o_tens);
    a.scal = (TensorScal *)(base + o_scal);
    a.err = (uint32_t *)(base + o_err);
    a.fb = (uint32_t *)(base + o_fb);
    a.b1 = H.beta1;
    a.b2 = k.b2;
    a.c1 = (float)(1.0 - (double)H.beta1);
    a.c2 = k.c2;
    a.ce = (float)(1.0 / std::sqrt((double)H.eps));
    a.wdf = (float)(1.0 - (double)lr * (double)H.weight_decay);
    a.lr = lr;
    a.clip_d = H.clip_d;
    a.coef_mom = k.coef_mom;
    a.coef_plain = k.coef_plain;
    a.step_lo = (uint32_t)(uint64_t)step;
    a.seed_lo = (uint32_t)seed;
    a.seed_hi = (uint32_t)(seed >> 32);

    uint32_t nFB = 0;
    if (row) {  // the phase-B launch a queued row-path tensor gets (as skew_bind sizes it)
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return SKEW_ECUDA;
        nFB = (uint32_t)(2 * (sms > 0 ? sms : 1));
    }

    cudaStream_t s = (cudaStream_t)stream;
    SetupTables tb{(uint2 *)(base + o_iA), nA, (uint2 *)(base + o_iR), nR, (uint2 *)(base + o_iF), nF,
                   (uint2 *)(base + o_iB), nB, (uint2 *)(base + o_iC), nC, (uint2 *)(base + o_iCR), nCR};
    k_noalloc_setup<<<8, 256, 0, s>>>(td, (TensorDev *)(base + o_tens), (TensorScal *)(base + o_scal),
                                      (uint32_t *)(base + o_fb), tb);
    e = cudaGetLastError();
    if (e != cudaSuccess) return SKEW_ECUDA;
    const LaunchPlan lp{nA,
                        nR,
                        nF,
                        nB,
                        nFB,
                        nC,
                        nCR,
                        (const uint2 *)(base + o_iA),
                        (const uint2 *)(base + o_iR),
                        (const uint2 *)(base + o_iF),
                        (const uint2 *)(base + o_iB),
                        (const uint2 *)(base + o_iC),
                        (const uint2 *)(base + o_iCR)};
    e = (cudaError_t)launch_phases(a, lp, stream, nullptr);
    if (e != cudaSuccess) return SKEW_ECUDA;
    return SKEW_OK;
}

extern "C" int skew_noalloc_sync_status(void *stream) {
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaStreamSynchronize(s) != cudaSuccess) return SKEW_ECUDA;
    unsigned char *const base = scratch_base();
    if (!base) return SKEW_ECUDA;
    uint32_t word = 0;
    if (cudaMemcpy(&word, base + kErrOffset, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return SKEW_ECUDA;
    if (!word) return SKEW_OK;
    if (cudaMemsetAsync(base + kErrOffset, 0, 4, s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
        return SKEW_ECUDA;
    return SKEW_ETIMEOUT;
}

extern "C" int skew_noalloc_selftest_wait_timeout(void *stream) {
    unsigned char *const base = scratch_base();
    if (!base) return SKEW_ECUDA;
    return launch_wait_selftest(reinterpret_cast<uint32_t *>(base + kErrOffset), stream) == (int)cudaSuccess
               ? SKEW_OK
               : SKEW_ECUDA;
}
