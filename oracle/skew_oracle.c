/*
 * SkewAdam CPU oracle -- TEST INFRASTRUCTURE, NOT PART OF THE PRODUCT.
 *
 * A plain, slow, fp64 restatement of one SkewAdam optimizer step, written from
 * the paper ("Where Should Optimizer State Live? Tiered State Allocation for
 * Memory-Efficient MoE Training"):
 *   - factored second moment: Sec. 3 "Factored second moments", Eq. 1;
 *   - tier policy: Sec. 3 "The tiers", Fig. 1; ablation variants: Table 3;
 *   - per-tensor step: Algorithm 1;
 *   - update clipping, bf16 write-back with dithered rounding and the
 *     decoupled weight decay: Sec. 3 "Update clipping and low-precision
 *     updates" (and its footnote), Sec. 5 "Limitations";
 *   - closed-form state size: Sec. 3 "Memory model", Eq. 2, App. B (Table 5).
 *
 * Only the test suite, the package smoke check and the benchmark's CPU-baseline
 * leg may load this file's library. It shares no code, header or constant
 * table with the CUDA library: the Philox-4x32-10 generator below is written
 * from its published definition (Salmon, Moraes, Dror, Shaw, "Parallel random
 * numbers: as easy as 1, 2, 3", SC'11).
 *
 * Arithmetic: every step is evaluated in double precision (built without
 * floating-point contraction, so x86 and Arm hosts agree bit for bit); state is
 * stored as fp32 (the memory model counts 4 bytes per state element); weights
 * and gradients are bf16 bit patterns, or fp32 for tensors kept in fp32 (App. A:
 * "fp32 norms and router"), whose new weight is the fp32 value x itself with no
 * dithered cast. Each stored fp32 value is the round-to-nearest-even conversion
 * of the fp64 expression.
 *
 * Readings taken where the paper is silent or loose (each is listed in the
 * design notes with its reason):
 *   - epsilon clamps the reconstructed second moment elementwise,
 *     D = sqrt(max(Vhat, eps)), on the factored path as on the full one, and a
 *     factored tensor whose row mean Rbar is exactly 0 has Vhat = 0;
 *   - R and C store the row / column MEANS of G*G (Eq. 1), Vhat = R C^T / Rbar;
 *   - the RMS of the update is taken over the whole tensor, before clipping,
 *     and the clip threshold d generalises the paper's d = 1;
 *   - weight decay is decoupled and lr-scaled, w <- w (1 - lr*lambda), fused
 *     into the fp32 expression ahead of the rounded cast; the router is exempt;
 *   - the dither is 16-bit integer stochastic rounding of the fp32 bit
 *     pattern (x + U(-ulp/2, ulp/2) rounded to nearest, with the exact bf16
 *     ulp of x), with a counter-based Philox-4x32-10 draw per element.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Philox-4x32-10 (Salmon et al., SC'11).                                    */
/* Each round multiplies counter words 0 and 2 by two fixed odd constants,  */
/* and forms the new counter from the high/low halves of the products mixed */
/* (xor) with the other two words and the round key. The key is bumped by   */
/* the two Weyl constants (golden ratio and sqrt(3)-1 in 32-bit fixed       */
/* point) between rounds.                                                    */
/* ------------------------------------------------------------------------ */
#define SO_PHILOX_M0 0xD2511F53u
#define SO_PHILOX_M1 0xCD9E8D57u
#define SO_PHILOX_W0 0x9E3779B9u
#define SO_PHILOX_W1 0xBB67AE85u

void so_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4])
{
    uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += SO_PHILOX_W0;
            k1 += SO_PHILOX_W1;
        }
        uint64_t p0 = (uint64_t)SO_PHILOX_M0 * (uint64_t)c0;
        uint64_t p1 = (uint64_t)SO_PHILOX_M1 * (uint64_t)c2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t n0 = hi1 ^ c1 ^ k0;
        uint32_t n1 = lo1;
        uint32_t n2 = hi0 ^ c3 ^ k1;
        uint32_t n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/*
 * The 16-bit dither of element `idx` (row-major flat index) of tensor `tid` at
 * step `step` under `seed`. One Philox block serves the eight elements that
 * share idx >> 3:
 *   key     = (low 32 bits of seed, high 32 bits of seed)
 *   counter = (low 32 of idx>>3, high 32 of idx>>3, tid, low 32 of step)
 *   r       = 16-bit half (idx & 1) of output word ((idx & 7) >> 1).
 */
uint16_t so_dither16(uint64_t seed, int64_t step, uint32_t tid, uint64_t idx)
{
    uint64_t blk = idx >> 3;
    uint32_t ctr[4] = {(uint32_t)blk, (uint32_t)(blk >> 32), tid, (uint32_t)(uint64_t)step};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t o[4];
    so_philox4x32_10(ctr, key, o);
    unsigned k = (unsigned)(idx & 7u);
    return (uint16_t)((o[k >> 1] >> (16u * (k & 1u))) & 0xFFFFu);
}

static uint32_t so_f32_bits(float x)
{
    uint32_t b;
    memcpy(&b, &x, 4);
    return b;
}

static double so_bf16_to_double(uint16_t h)
{
    uint32_t b = (uint32_t)h << 16;
    float f;
    memcpy(&f, &b, 4);
    return (double)f;
}

/*
 * Dithered rounding of an fp32 value to bf16 (Sec. 3, Algorithm 1 last step):
 * adding a uniform integer r in [0, 2^16) to the fp32 bit pattern and keeping
 * the top 16 bits rounds the magnitude up with probability (low 16 bits)/2^16,
 * i.e. adds noise of one bf16 ulp width and rounds to nearest. A carry out of
 * the largest finite exponent gives +-Inf; Inf stays Inf; NaN becomes the
 * canonical quiet NaN with the sign kept.
 */
uint16_t so_sr_bf16(float x, uint16_t r)
{
    uint32_t b = so_f32_bits(x);
    if (isnan(x))
        return (uint16_t)(0x7FC0u | ((b >> 16) & 0x8000u));
    return (uint16_t)((b + (uint32_t)r) >> 16);
}

/* ------------------------------------------------------------------------ */
/* Tier policy (Sec. 3 "The tiers", Algorithm 1, Table 3 variants).          */
/* ------------------------------------------------------------------------ */
enum { SO_TIER_BACKBONE = 0, SO_TIER_EXPERT = 1, SO_TIER_ROUTER = 2 };
enum { SO_POLICY_TIERED = 0, SO_POLICY_EXPERT_MOMENTUM = 1, SO_POLICY_FACTORED_ROUTER = 2, SO_POLICY_UNIFORM = 3,
       SO_POLICY_ADAFACTOR = 4 };
enum { SO_KIND_FULL = 0, SO_KIND_FACTORED = 1 };

/*
 * kind:     a vector (ndim 1) keeps the full second moment (Algorithm 1, "W is
 *           a vector"); the router keeps it too unless the variant factors it
 *           (Table 3 "factored router", "uniform"); every other matrix is
 *           factored (Eq. 1).
 * momentum: backbone tensors carry fp32 momentum; experts only under the
 *           "+ momentum on experts" and "uniform" variants; the router only
 *           under "uniform".
 * The Adafactor comparator (Sec. 5 and its footnote, App. A "no momentum")
 * factors every matrix, the router too, and keeps no momentum anywhere.
 * decay:    every tier but the router ("no weight decay" for the router),
 *           unless the caller exempts the tensor.
 * Returns 0, or -1 for an unknown tier / policy / ndim.
 */
int so_resolve(int ndim, int tier, int policy, int no_decay, int *kind, int *momentum, int *decay)
{
    if (ndim != 1 && ndim != 2) return -1;
    if (tier < 0 || tier > 2 || policy < 0 || policy > 4) return -1;
    int k;
    if (ndim == 1)
        k = SO_KIND_FULL;
    else if (tier == SO_TIER_ROUTER && policy != SO_POLICY_FACTORED_ROUTER && policy != SO_POLICY_UNIFORM &&
             policy != SO_POLICY_ADAFACTOR)
        k = SO_KIND_FULL;
    else
        k = SO_KIND_FACTORED;
    int mo;
    if (policy == SO_POLICY_ADAFACTOR)
        mo = 0;
    else if (tier == SO_TIER_BACKBONE)
        mo = 1;
    else if (tier == SO_TIER_EXPERT)
        mo = (policy == SO_POLICY_EXPERT_MOMENTUM || policy == SO_POLICY_UNIFORM);
    else
        mo = (policy == SO_POLICY_UNIFORM);
    *kind = k;
    *momentum = mo;
    *decay = (tier != SO_TIER_ROUTER) && !no_decay;
    return 0;
}

/*
 * Closed-form optimizer-state size in bytes (Eq. 2 plus the full v of vector
 * tensors, Table 5): 4 bytes per momentum element, per full-v element and per
 * entry of the factored R (n) and C (m) vectors. A 1-D tensor of length L is
 * passed as n = L, m = 1.
 */
int64_t so_state_bytes(int ntensors, const int32_t *ndim, const int64_t *n, const int64_t *m,
                       const int32_t *tier, int32_t policy)
{
    int64_t floats = 0;
    for (int k = 0; k < ntensors; ++k) {
        int kind, mo, dec;
        if (so_resolve(ndim[k], tier[k], policy, 0, &kind, &mo, &dec) != 0) return -1;
        int64_t numel = n[k] * m[k];
        if (mo) floats += numel;
        if (kind == SO_KIND_FULL)
            floats += numel;
        else
            floats += n[k] + m[k];
    }
    return 4 * floats;
}

/*
 * beta^t by binary exponentiation with plain IEEE multiplies, so that the
 * result is the same on every host (no libm pow, whose last bit may differ
 * between platforms).
 */
static double so_powi(double b, int64_t t)
{
    double r = 1.0, p = b;
    while (t > 0) {
        if (t & 1) r *= p;
        p *= p;
        t >>= 1;
    }
    return r;
}

/* ------------------------------------------------------------------------ */
/* One SkewAdam step for one tensor (Algorithm 1).                           */
/* ------------------------------------------------------------------------ */
typedef struct {
    uint16_t *w;        /* bf16 bits, n*m, updated in place                      */
    const uint16_t *g;  /* bf16 bits, n*m                                        */
    float *M;           /* fp32 momentum, n*m (momentum tensors) or NULL         */
    float *v;           /* fp32 full second moment, n*m (full kind) or NULL      */
    float *R;           /* fp32 row statistic, n (factored kind) or NULL         */
    float *C;           /* fp32 column statistic, m (factored kind) or NULL      */
    int64_t n, m;       /* rows and columns; a vector of length L is n=L, m=1    */
    int32_t kind;       /* SO_KIND_FULL or SO_KIND_FACTORED                       */
    int32_t momentum;   /* 1: keeps fp32 momentum                                */
    int32_t decay;      /* 1: weight decay applies                               */
    uint32_t tid;       /* tensor id fed to the dither                           */
    uint64_t idx0;      /* dither index of element 0: 0, or for matrix e of a    */
                        /* stacked (E, n, m) tensor e*n*m (its flat offset)      */
    float *wf;          /* fp32 tensor: weights (then w and g are unused), or NULL */
    const float *gf;    /* fp32 tensor: gradient                                 */
} so_tensor_t;

/* Gradient element e as a double (bf16 bits or fp32). */
static double so_grad(const so_tensor_t *T, int64_t e)
{
    return T->gf ? (double)T->gf[e] : so_bf16_to_double(T->g[e]);
}

typedef struct {
    double beta1, beta2, eps, clip_d, weight_decay;
    int32_t annealed;   /* 1: the Adafactor comparator's decay beta2_t = 1 - t^-0.8 */
                        /* (as an fp32 value) and no bias correction; beta2 unused  */
    double gscale;      /* the trainer's global gradient-norm clip factor of this   */
                        /* step (Sec. 4 training setup, App. A Table 9: clip 1.0):  */
                        /* the step sees gscale * G, formed in fp64; 1 = no clip    */
} so_hparams_t;

/*
 * Applies one step to one tensor. `t` is the global 1-based step, `lr` the
 * scheduled learning rate. Optional outputs (NULL to skip): x_out[n*m] the
 * fp32 value before the dithered cast, r_out[n*m] the 16-bit dither, and
 * stats_out[4] = {Rbar, sum of U^2, RMS(U), clip factor kappa}.
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int so_tensor_step(const so_tensor_t *T, const so_hparams_t *hp, int64_t t, double lr, uint64_t seed,
                   float *x_out, uint16_t *r_out, double *stats_out)
{
    if (!T || !hp || t < 1 || T->n < 1 || T->m < 1) return -1;
    const int64_t n = T->n, m = T->m, numel = n * m;
    const double b1 = hp->beta1;
    double b2 = hp->beta2;
    double bc1 = 1.0 - so_powi(b1, t);           /* 1 - beta1^t        */
    double s2 = sqrt(1.0 - so_powi(b2, t));      /* sqrt(1 - beta2^t)  */
    if (hp->annealed) {                          /* Adafactor: beta2_t = 1 - t^-0.8, no correction */
        b2 = (double)(float)(1.0 - pow((double)t, -0.8));
        bc1 = 1.0;
        s2 = 1.0;
    }

    double *U = (double *)malloc((size_t)numel * sizeof(double));
    if (!U) return -1;
    double rbar = 0.0;

    /* Second moment: full (Algorithm 1, full branch) or factored (Eq. 1). */
    if (T->kind == SO_KIND_FULL) {
        for (int64_t e = 0; e < numel; ++e) {
            double g = hp->gscale * so_grad(T, e);
            T->v[e] = (float)(b2 * (double)T->v[e] + (1.0 - b2) * g * g);
        }
    } else {
        double *rs = (double *)calloc((size_t)n, sizeof(double));
        double *cs = (double *)calloc((size_t)m, sizeof(double));
        if (!rs || !cs) { free(rs); free(cs); free(U); return -1; }
        for (int64_t i = 0; i < n; ++i)
            for (int64_t j = 0; j < m; ++j) {
                double g = hp->gscale * so_grad(T, i * m + j);
                rs[i] += g * g;
                cs[j] += g * g;
            }
        for (int64_t i = 0; i < n; ++i)   /* R <- b2 R + (1-b2) mean over columns */
            T->R[i] = (float)(b2 * (double)T->R[i] + (1.0 - b2) * (rs[i] / (double)m));
        for (int64_t j = 0; j < m; ++j)   /* C <- b2 C + (1-b2) mean over rows    */
            T->C[j] = (float)(b2 * (double)T->C[j] + (1.0 - b2) * (cs[j] / (double)n));
        double rsum = 0.0;
        for (int64_t i = 0; i < n; ++i) rsum += (double)T->R[i];
        rbar = rsum / (double)n;          /* Rbar = mean(R)                       */
        free(rs);
        free(cs);
    }

    /* Preconditioned update (Algorithm 1, momentum / no-momentum branches). */
    for (int64_t i = 0; i < n; ++i)
        for (int64_t j = 0; j < m; ++j) {
            const int64_t e = i * m + j;
            double g = hp->gscale * so_grad(T, e);
            double vhat;
            if (T->kind == SO_KIND_FULL)
                vhat = (double)T->v[e];
            else
                vhat = rbar > 0.0 ? (double)T->R[i] * (double)T->C[j] / rbar : 0.0;
            double D = sqrt(fmax(vhat, hp->eps));
            if (T->momentum) {
                T->M[e] = (float)(b1 * (double)T->M[e] + (1.0 - b1) * g);
                U[e] = (s2 / bc1) * (double)T->M[e] / D;
            } else {
                U[e] = s2 * g / D;
            }
        }

    /* Update clipping: U <- U / max(1, RMS(U)/d). */
    double su2 = 0.0;
    for (int64_t e = 0; e < numel; ++e) su2 += U[e] * U[e];
    const double rho = sqrt(su2 / (double)numel);
    const double kappa = 1.0 / fmax(1.0, rho / hp->clip_d);

    /* Decoupled weight decay fused ahead of the dithered bf16 cast (an fp32
     * tensor stores x itself). */
    const double lam = T->decay ? hp->weight_decay : 0.0;
    for (int64_t e = 0; e < numel; ++e) {
        double w = T->wf ? (double)T->wf[e] : so_bf16_to_double(T->w[e]);
        float x = (float)(w * (1.0 - lr * lam) - lr * kappa * U[e]);
        uint16_t r = 0;
        if (T->wf) {
            T->wf[e] = x;
        } else {
            r = so_dither16(seed, t, T->tid, T->idx0 + (uint64_t)e);
            T->w[e] = so_sr_bf16(x, r);
        }
        if (x_out) x_out[e] = x;
        if (r_out) r_out[e] = r;
    }
    if (stats_out) {
        stats_out[0] = rbar;
        stats_out[1] = su2;
        stats_out[2] = rho;
        stats_out[3] = kappa;
    }
    free(U);
    return 0;
}

/* Array helpers for the test harness (same definitions, element by element). */
void so_dither16_array(uint64_t seed, int64_t step, uint32_t tid, uint64_t idx0, int64_t count, uint16_t *out)
{
    for (int64_t k = 0; k < count; ++k) out[k] = so_dither16(seed, step, tid, idx0 + (uint64_t)k);
}

void so_sr_bf16_array(const float *x, const uint16_t *r, int64_t count, uint16_t *out)
{
    for (int64_t k = 0; k < count; ++k) out[k] = so_sr_bf16(x[k], r[k]);
}

/*
 * A whole step over a list of tensors: every tensor is independent, so this
 * is the per-tensor step applied in order. Returns 0 or the first error.
 */
int so_step(so_tensor_t *tensors, int ntensors, const so_hparams_t *hp, int64_t t, double lr, uint64_t seed)
{
    for (int k = 0; k < ntensors; ++k) {
        int rc = so_tensor_step(&tensors[k], hp, t, lr, seed, NULL, NULL, NULL);
        if (rc) return rc;
    }
    return 0;
}
