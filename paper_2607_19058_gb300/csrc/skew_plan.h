// Internal layout shared by the host planner (skew_host.cpp) and the device
// kernels (skew_kernels.cu) of libskewadam. Not part of the public ABI.
#pragma once

#include <stdint.h>
#include <vector_types.h>

namespace skew {

// Every kernel runs 256-thread CTAs; a thread owns 8 consecutive bf16 elements
// (one 16-byte vector) of up to kVecPerThread rows (factored tiles) or flat
// vectors (full-second-moment tiles). A tile is therefore 32 Ki elements.
constexpr int kThreads = 256;
constexpr int kVecPerThread = 32;
constexpr int64_t kFlatTileElems = int64_t(kThreads) * kVecPerThread * 8;
constexpr int kFinChunk = 256;  // rows / columns per finalize item

enum Kind : uint32_t { kKindFull = 0, kKindFactored = 1 };

// Device descriptor of one tensor (lives in the workspace).
struct TensorDev {
    uint16_t *w;        // bf16 weights, n*m, row-major (borrowed)
    const uint16_t *g;  // bf16 gradient (borrowed)
    float *M;           // momentum (numel) or null
    float *v;           // exact second moment (numel) or null
    float *R;           // row factor (n) or null
    float *C;           // column factor (m) or null
    float *rowp;        // factored: row partials [strips][n]
    float *colp;        // factored: column partials [rowtiles][m]
    float *bsc;         // factored: 1/sqrt(C_j) [m]
    double *rsum;       // factored: per finalize-row-item sum of R [nfr]
    float2 *u2;         // per tile sum of (U / coef)^2 as a (hi, lo) pair [ntiles]
    int64_t n, m, numel;
    uint32_t tid;       // dither tensor id
    uint32_t kind, momentum, decay;
    uint32_t vec;       // 1: 16-byte vector loads / stores are legal
    uint32_t lcl;       // factored: log2 of lanes along a row (LC)
    uint32_t strips;    // factored: column strips of 8*LC columns
    uint32_t rowtiles;  // factored: row tiles of tile_rows rows; full: flat tiles
    uint32_t tile_rows; // factored: rows per tile = 16 * (256 / LC)
    uint32_t ntiles;    // update tiles of this tensor
    uint32_t nfr, nfc;  // factored: finalize items over rows / columns
};

// Per-tensor scalars of the current step (zeroed at the start of every step).
struct TensorScal {
    double rbar;      // mean(R)
    double sumsq;     // sum over the tensor of U^2
    double rms;       // RMS(U)
    double kappa;     // 1 / max(1, RMS / d)
    float rbar_s;     // mean(R) * 2^rbar_e, in [1, 2); 0 if mean(R) == 0
    int32_t rbar_e;
    float coefC;      // lr * kappa * coef, the factor applied to (y / D)
    uint32_t cntF;    // finalize items done
    uint32_t cntB;    // update-RMS tiles done
    uint32_t pad[3];
};
static_assert(sizeof(TensorScal) == 64, "TensorScal layout");

// Per-step parameters, passed by value to every kernel (a kernel parameter).
struct StepArgs {
    const TensorDev *tensors;
    TensorScal *scal;
    float b1, b2, c1, c2;  // beta1, beta2, 1-beta1, 1-beta2 (fp32)
    float ce;              // 1 / sqrt(eps), fp32
    float wdf;             // 1 - lr * lambda, fp32
    float lr;
    float clip_d;
    double coef_mom;       // sqrt(1-beta2^t) / (1-beta1^t)
    double coef_plain;     // sqrt(1-beta2^t)
    uint32_t step_lo;
    uint32_t seed_lo, seed_hi;
};

// The four phases of a set of tensors: item lists (tensor, local tile / item)
// in device memory and their lengths.
struct LaunchPlan {
    uint32_t nA, nF, nBC;
    const uint2 *itemsA, *itemsF, *itemsBC;
};

// Enqueues the phases of `L` as four grouped launches (A, F, B, C) on `stream`,
// each given the step parameters A by value. If `ev` is not null it holds five
// cudaEvent_t, recorded before the first launch and after each of the four.
// Returns a cudaError_t value.
int launch_phases(const StepArgs &A, const LaunchPlan &L, void *stream, void *const *ev);

}  // namespace skew
