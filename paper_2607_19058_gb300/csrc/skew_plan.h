// Internal layout shared by the host planner (skew_host.cpp), the no-alloc
// entry point (skew_noalloc.cu) and the device kernels (skew_kernels.cu) of
// libskewadam. Not part of the public ABI.
#pragma once

#include <math.h>
#include <stdint.h>
#include <vector_types.h>

#include "skewadam.h"

namespace skew {

// Every kernel runs 256-thread CTAs; a thread owns 8 consecutive bf16 elements
// (one 16-byte vector) of up to kVecPerThread rows (strip tiles: 64 Ki elements)
// or of kFlatVecPerThread flat vectors (full-second-moment tiles: 8 Ki elements,
// so that the router and the vectors, small, spread over many CTAs).
constexpr int kThreads = 256;
constexpr int kVecPerThread = 32;
constexpr int kFlatVecPerThread = 4;
constexpr int64_t kFlatTileElems = int64_t(kThreads) * kFlatVecPerThread * 8;
constexpr int kFinChunk = 256;  // rows / columns per finalize item

// Row-tile path (phase A on whole rows, no phase B unless a clamp may bind):
// a chunk is kRowChunkBytes of consecutive whole rows of the bf16 gradient,
// copied to shared memory by one bulk copy; a phase-A row tile is kRowChunks
// chunks (kRowChunksWide for 4096-wide matrices of at least 2048 rows, whose
// tiles then pay their ring ramp and column partials half as often; shorter
// matrices keep more, smaller tiles, which measured faster); a phase-C row tile
// is always the rows of kRowChunks chunks; the CTA keeps kRowStages chunks in flight.
constexpr int kRowChunkBytes = 32768;
constexpr int kRowChunks = 32;
constexpr int kRowChunksWide = 64;
constexpr int kRowStages = 3;
// Momentum tensors on the row path: a chunk holds kMomGBytes of bf16 rows (G in
// phase A, W in phase C) and the same rows of fp32 M; a row tile is kMomChunks chunks.
// Phase C on the row path: the last kApplyTailSplit tiles of a step (two waves of the
// kernel's two CTAs per SM on GB300's 152 SMs) run as two half tiles each, so that the
// launch's last wave ends sooner. An item's tile field then carries kHalfTile, plus
// kSecondHalf for the second half (results do not depend on the split).
constexpr uint32_t kApplyTailSplit = 2u * 2u * 152u;
constexpr uint32_t kHalfTile = 1u << 31, kSecondHalf = 1u << 30, kTileMask = kSecondHalf - 1u;
constexpr int kMomGBytes = 16384;
constexpr int kMomChunks = 64;

enum Kind : uint32_t { kKindFull = 0, kKindFactored = 1 };

// Tier policy of one tensor (Sec. 3 "The tiers", Algorithm 1, the Table 3
// variants, and the Adafactor comparator of Sec. 5 / App. A): a vector keeps the exact
// second moment; the router too unless the variant factors it; every other matrix
// is factored (Eq. 1). Momentum: the backbone; experts under "+ momentum on
// experts" and "uniform"; the router under "uniform"; nothing under Adafactor.
// Weight decay: every tier but the router, unless the caller exempts the tensor.
inline void resolve_policy(int ndim, int tier, int policy, uint32_t flags, uint32_t &kind, uint32_t &momentum,
                           uint32_t &decay) {
    const bool router_factored = policy == SKEW_POLICY_FACTORED_ROUTER || policy == SKEW_POLICY_UNIFORM ||
                                 policy == SKEW_POLICY_ADAFACTOR;
    kind = (ndim == 1 || (tier == SKEW_TIER_ROUTER && !router_factored)) ? kKindFull : kKindFactored;
    if (policy == SKEW_POLICY_ADAFACTOR)
        momentum = 0;
    else if (tier == SKEW_TIER_BACKBONE)
        momentum = 1;
    else if (tier == SKEW_TIER_EXPERT)
        momentum = (policy == SKEW_POLICY_EXPERT_MOMENTUM || policy == SKEW_POLICY_UNIFORM);
    else
        momentum = (policy == SKEW_POLICY_UNIFORM);
    decay = (tier != SKEW_TIER_ROUTER) && !(flags & SKEW_F_NO_DECAY);
}

// Second-moment decay (fp32, with 1 - beta2 formed from it in fp64) and the update
// coefficients of step t: sqrt(1 - beta2^t) / (1 - beta1^t) with momentum and
// sqrt(1 - beta2^t) without (Algorithm 1's bias corrections). The Adafactor
// comparator anneals the decay, beta2_t = 1 - t^-0.8, and has no bias correction.
struct StepCoefs {
    float b2, c2;
    double coef_mom, coef_plain;
};

inline StepCoefs step_coefs(const skew_hparams_t &H, int64_t step) {
    const double t = (double)step;
    StepCoefs c;
    if (H.policy == SKEW_POLICY_ADAFACTOR) {
        c.b2 = (float)(1.0 - pow(t, -0.8));
        c.c2 = (float)(1.0 - (double)c.b2);
        c.coef_mom = c.coef_plain = 1.0;
    } else {
        const double s2 = sqrt(1.0 - pow((double)H.beta2, t));
        c.b2 = H.beta2;
        c.c2 = (float)(1.0 - (double)H.beta2);
        c.coef_mom = s2 / (1.0 - pow((double)H.beta1, t));
        c.coef_plain = s2;
    }
    return c;
}

// Tile geometry of one tensor (shared by every entry point, so that the same
// tensor is always cut the same way and results are bit-identical).
struct TileGeom {
    uint32_t lcl = 0, strips = 1, rowtiles = 1, tile_rows = 0, ntiles = 0, nfr = 0, nfc = 0;
    uint32_t rowpath = 0, cr = 0, rt_rows = 0, rtiles = 0;
    uint32_t at_rows = 0, atiles = 0;  // row path: phase-C row tiles (momentum tensors: the phase-A tiles)
    uint32_t fci = 0;  // row path: columns per finalize item (kFinChunk / fci threads per column)
};

// `kind`, `momentum` as resolved by the tier policy; `wg_aligned`: weight and
// gradient pointers are 16-byte aligned. Counts fit 32 bits for n, m <= 2^40
// and n*m <= 2^62 only when the caller has checked the tile count (planner).
inline TileGeom plan_geometry(uint32_t kind, uint32_t momentum, bool wg_aligned, int64_t n, int64_t m, int64_t numel) {
    TileGeom g;
    if (kind == kKindFactored) {
        const int64_t vecs = (m + 7) / 8;  // 8-column groups per row
        uint32_t lc = 1;
        while (lc < 32 && lc < vecs) {
            lc <<= 1;
            ++g.lcl;
        }
        g.strips = (uint32_t)((m + 8 * lc - 1) / (8 * lc));
        g.tile_rows = (uint32_t)(kVecPerThread * (kThreads / lc));
        g.rowtiles = (uint32_t)((n + g.tile_rows - 1) / g.tile_rows);
        g.ntiles = g.strips * g.rowtiles;
        g.nfc = (uint32_t)((m + kFinChunk - 1) / kFinChunk);
        // Whole-row phases A and C: factored matrices of width 512, 1024, 2048
        // or 4096 (64 to 512 16-byte vectors per row), with or without momentum.
        g.rowpath = (wg_aligned && (m == 512 || m == 1024 || m == 2048 || m == 4096)) ? 1u : 0u;
        if (g.rowpath) {
            g.cr = (uint32_t)((momentum ? kMomGBytes : kRowChunkBytes) / (2 * m));
            g.rt_rows = g.cr * (momentum ? kMomChunks : m == 4096 && n >= 2048 ? kRowChunksWide : kRowChunks);
            g.rtiles = (uint32_t)((n + g.rt_rows - 1) / g.rt_rows);
            g.at_rows = momentum ? g.rt_rows : g.cr * kRowChunks;
            g.atiles = (uint32_t)((n + g.at_rows - 1) / g.at_rows);
            g.nfr = 0;
            // tall matrices: up to 8 threads share a column, each adding every 8th tile
            uint32_t tpc = 1;
            while (tpc < 8 && g.rtiles >= 64u * tpc) tpc <<= 1;
            g.fci = (uint32_t)(kFinChunk / tpc);
            g.nfc = (uint32_t)((m + g.fci - 1) / g.fci);
        } else {
            g.nfr = (uint32_t)((n + kFinChunk - 1) / kFinChunk);
        }
    } else {
        g.rowtiles = (uint32_t)((numel + kFlatTileElems - 1) / kFlatTileElems);
        g.ntiles = g.rowtiles;
    }
    return g;
}

// Device descriptor of one tensor (lives in the workspace).
struct TensorDev {
    uint16_t *w;        // bf16 weights, n*m, row-major (borrowed)
    const uint16_t *g;  // bf16 gradient (borrowed)
    float *M;           // momentum (numel) or null
    float *v;           // exact second moment (numel) or null
    float *R;           // row factor (n) or null
    float *C;           // column factor (m) or null
    float *rowp;        // strip path: row partials [strips][n]
    float *colp;        // strip path: column partials of g^2 [rowtiles][m]
    float *bsc;         // factored: 1/sqrt(C_j) [m]
    double *rsum;       // factored: sums of R per finalize-row item [nfr] / per row tile [rtiles]
    float2 *pp;         // row path: per row tile and column, (sum of g^2, sum of g^2 / R_i) [rtiles][m]
    float *rmin;        // row path: smallest positive R_i per row tile [rtiles]
    double *fsum;       // row path: sum of P_j / C_j per finalize item [nfc]
    float *fmin;        // row path: smallest C_j with P_j > 0 per finalize item [nfc]
    float2 *u2;         // per tile sum of (U / coef)^2 as a (hi, lo) pair [ntiles]
    int64_t n, m, numel;
    uint32_t tid;       // dither tensor id
    uint64_t base;      // dither index of element 0 (a matrix of a stacked tensor: its offset)
    uint32_t kind, momentum, decay;
    uint32_t vec;       // 1: 16-byte vector loads / stores are legal (bf16 tensors only)
    uint32_t f32;       // 1: weights and gradient are fp32 (w, g then address floats; no dither)
    uint32_t lcl;       // factored: log2 of lanes along a row (LC)
    uint32_t strips;    // factored: column strips of 8*LC columns
    uint32_t rowtiles;  // factored: row tiles of tile_rows rows; full: flat tiles
    uint32_t tile_rows; // factored: rows per tile = 32 * (256 / LC)
    uint32_t ntiles;    // update tiles of this tensor
    uint32_t nfr, nfc;  // factored: finalize items over rows / columns
    uint32_t rowpath;   // 1: whole-row phase A (k_rowsq) and the bilinear sum of U^2
    uint32_t cr;        // row path: rows per chunk
    uint32_t rt_rows;   // row path: rows per phase-A row tile
    uint32_t rtiles;    // row path: phase-A row tiles
    uint32_t fci;       // row path: columns per finalize item
    uint32_t at_rows;   // row path: rows per phase-C row tile (<= 1024)
    uint32_t atiles;    // row path: phase-C row tiles
};

// Per-tensor scalars of the current step (zeroed at the start of every step).
struct TensorScal {
    double rbar;        // mean(R)
    double sumsq;       // sum over the tensor of U^2
    double rms;         // RMS(U)
    double kappa;       // 1 / max(1, RMS / d)
    float rbar_s;       // mean(R) * 2^rbar_e, in [1, 2); 0 if mean(R) == 0
    int32_t rbar_e;
    float coefC;        // lr * kappa * coef, the factor applied to (y / D)
    uint32_t cntF;      // finalize items done
    uint32_t cntB;      // update-RMS tiles done
    uint32_t fallback;  // row path: 1 if sum(U^2) needs phase B (a clamp may bind)
    uint32_t zflag;     // row path: a row with R_i == 0 holds a nonzero gradient
    uint32_t pad;
};
static_assert(sizeof(TensorScal) == 64, "TensorScal layout");

// Per-step parameters, passed by value to every kernel (a kernel parameter).
struct StepArgs {
    const TensorDev *tensors;
    TensorScal *scal;
    uint32_t *err;         // sticky status word (nonzero: a bounded wait gave up)
    uint32_t *fb;          // [0]: row-path tensors that need phase B, [1..]: their ids
    float b1, b2, c1, c2;  // beta1, beta2, 1-beta1, 1-beta2 (fp32)
    float ce;              // 1 / sqrt(eps), fp32
    float wdf;             // 1 - lr * lambda, fp32
    float lr;
    float clip_d;
    double coef_mom;       // sqrt(1-beta2^t) / (1-beta1^t)
    double coef_plain;     // sqrt(1-beta2^t)
    uint32_t step_lo;
    uint32_t seed_lo, seed_hi;
    const float *gscale;   // device pointer to the step's gradient scale gamma (the trainer's
                           // global-norm clip factor), or null for gamma = 1
};

// The phases of one step: item lists (tensor, local tile / item) in device
// memory and their lengths.
//   A  strip-tile sums of squares (strip-path factored tensors)
//   R  row-tile sums of squares and bilinear partials (row-path tensors)
//   F  finalize items (rows and columns; columns only on the row path)
//   B  update-RMS tiles (strip-path factored and full tensors)
//   FB phase B of the row-path tensors whose finalize asked for it (nFB CTAs)
//   C  apply strip tiles (tensors not on the row path)
//   CR apply row tiles (row-path tensors)
struct LaunchPlan {
    uint32_t nA, nR, nF, nB, nFB, nC, nCR;
    const uint2 *itemsA, *itemsR, *itemsF, *itemsB, *itemsC, *itemsCR;
};

constexpr int kLaunches = 7;

// Enqueues the phases of `L` as grouped launches (A, R, F, B, FB, C, CR; empty
// ones skipped) on `stream`, each given the step parameters by value. If `ev` is
// not null it holds kLaunches + 1 cudaEvent_t, recorded before the first launch
// and after each of the seven. Returns a cudaError_t value.
int launch_phases(const StepArgs &A, const LaunchPlan &L, void *stream, void *const *ev);

// Enqueues the bounded-wait self-test (one thread waits on an mbarrier phase that
// never completes and records the timeout in *err). Returns a cudaError_t value.
int launch_wait_selftest(uint32_t *err, void *stream);

}  // namespace skew
