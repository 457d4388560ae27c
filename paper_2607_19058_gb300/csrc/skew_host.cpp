// Host side of libskewadam: validation, tier policy, state / workspace layout,
// descriptor and tile tables, and the C ABI declared in include/skewadam.h.
//
// The tier policy follows Sec. 3 "The tiers" and Algorithm 1 (vectors keep the
// exact second moment; the router keeps it and no weight decay; backbone keeps
// fp32 momentum), with the Table 3 variants selected by skew_hparams_t.policy.
// The state layout realises Eq. 2 (plus the vectors' full v, Table 5) with no
// padding, so skew_state_bytes() is the closed form exactly.
#include "skewadam.h"
#include "skew_plan.h"

#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <algorithm>
#include <cstring>
#include <new>
#include <string>
#include <vector>

using namespace skew;

namespace {

// One matrix or vector stepped on its own (a stacked descriptor gives several).
struct TPlan {
    void *w = nullptr;        // its bf16 weights and gradient
    const void *g = nullptr;
    uint32_t tid = 0;         // the descriptor's index: the dither's tensor id
    uint64_t base = 0;        // dither index of its element 0 within the descriptor
    int kind = 0, momentum = 0, decay = 0, vec = 0;
    int64_t n = 0, m = 0, numel = 0;
    int64_t moff = -1, voff = -1, roff = -1, coff = -1;  // floats into the state
    uint32_t lcl = 0, strips = 1, rowtiles = 1, tile_rows = 0, ntiles = 0, nfr = 0, nfc = 0;
    uint32_t rowpath = 0, cr = 0, rt_rows = 0, rtiles = 0, at_rows = 0, atiles = 0, fci = 0;
    uint32_t f32 = 0;         // SKEW_F_FP32: fp32 weights and gradient
    // bytes into the workspace
    size_t ws_rowp = 0, ws_colp = 0, ws_bsc = 0, ws_rsum = 0, ws_u2 = 0, ws_pp = 0, ws_rmin = 0, ws_fsum = 0, ws_fmin = 0;
};

thread_local std::string g_create_err;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace

struct skew_handle {
    std::vector<skew_param_desc_t> desc;
    skew_hparams_t hp{};
    std::vector<TPlan> t;                  // matrices / vectors in descriptor order
    std::vector<uint32_t> first, count;    // per descriptor: its first plan and how many
    size_t state_bytes = 0, ws_bytes = 0;
    size_t ws_scal = 0, ws_fb = 0, ws_err = 0, ws_tab = 0, ws_tab_end = 0;
    size_t ws_tens = 0, ws_itemsA = 0, ws_itemsR = 0, ws_itemsF = 0, ws_itemsB = 0, ws_itemsC = 0, ws_itemsCR = 0;
    std::vector<uint2> itemsA, itemsR, itemsF, itemsB, itemsC, itemsCR;  // per phase, tensors in order
    uint32_t n_rowpath = 0;  // tensors on the row path
    uint32_t fb_ctas = 0;    // CTAs of the row path's phase-B launch (set at bind)
    char *state = nullptr, *ws = nullptr;
    bool bound = false;
    std::string err;
    // per-launch timing (skew_profile_begin / skew_profile_end)
    std::vector<cudaEvent_t> prof_ev;
    int32_t prof_max = 0, prof_used = 0;
    ~skew_handle() {
        for (cudaEvent_t e : prof_ev) cudaEventDestroy(e);
    }
};

// What the profiler times per step: the grouped launches (an empty phase times ~0).
constexpr int kProfLaunches = kLaunches;
const char *const kProfNames[kProfLaunches] = {"k_sumsq", "k_rowsq",  "k_finalize", "k_rms",
                                               "k_fallback", "k_apply", "k_apply_rows"};

static int fail(skew_handle_t *h, int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (h)
        h->err = buf;
    else
        g_create_err = buf;
    return code;
}

static int cuda_fail(skew_handle_t *h, cudaError_t e, const char *what) {
    return fail(h, SKEW_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Tier policy: (kind, momentum, decay) of one tensor (resolve_policy).
static void resolve(int ndim, int tier, int policy, uint32_t flags, TPlan &p) {
    uint32_t kind, momentum, decay;
    resolve_policy(ndim, tier, policy, flags, kind, momentum, decay);
    p.kind = (int)kind;
    p.momentum = (int)momentum;
    p.decay = (int)decay;
}

// Tile geometry (plan_geometry): strip tiles of (tile_rows rows) x (8*LC
// columns) or flat tiles of kFlatTileElems elements, and for the row path whole-row tiles.
static void geometry(TPlan &p, bool wg_aligned) {
    const TileGeom g = plan_geometry(p.kind, p.momentum, wg_aligned, p.n, p.m, p.numel);
    p.lcl = g.lcl;
    p.strips = g.strips;
    p.rowtiles = g.rowtiles;
    p.tile_rows = g.tile_rows;
    p.ntiles = g.ntiles;
    p.nfr = g.nfr;
    p.nfc = g.nfc;
    p.rowpath = g.rowpath;
    p.cr = g.cr;
    p.rt_rows = g.rt_rows;
    p.rtiles = g.rtiles;
    p.at_rows = g.at_rows;
    p.atiles = g.atiles;
    p.fci = g.fci;
}

extern "C" {

int skew_create(const skew_param_desc_t *params, int32_t n_params, const skew_hparams_t *hp, skew_handle_t **out) {
    g_create_err.clear();
    if (!out) return fail(nullptr, SKEW_EINVAL, "out is NULL");
    *out = nullptr;
    if (!hp) return fail(nullptr, SKEW_EINVAL, "hp is NULL");
    if (n_params < 0 || (n_params > 0 && !params)) return fail(nullptr, SKEW_EINVAL, "bad parameter list");
    const skew_hparams_t H = *hp;
    auto finite = [](float x) { return std::isfinite(x); };
    if (!finite(H.beta1) || H.beta1 < 0.f || H.beta1 >= 1.f) return fail(nullptr, SKEW_EINVAL, "beta1 must be in [0,1)");
    if (!finite(H.beta2) || H.beta2 < 0.f || H.beta2 >= 1.f) return fail(nullptr, SKEW_EINVAL, "beta2 must be in [0,1)");
    if (!finite(H.eps) || !(H.eps > 0.f)) return fail(nullptr, SKEW_EINVAL, "eps must be finite and > 0");
    if (!finite(H.clip_d) || !(H.clip_d > 0.f)) return fail(nullptr, SKEW_EINVAL, "clip_d must be finite and > 0");
    if (!finite(H.weight_decay) || H.weight_decay < 0.f) return fail(nullptr, SKEW_EINVAL, "weight_decay must be finite and >= 0");
    if (H.policy < SKEW_POLICY_TIERED || H.policy > SKEW_POLICY_ADAFACTOR) return fail(nullptr, SKEW_EINVAL, "unknown policy %d", H.policy);

    skew_handle *h = new (std::nothrow) skew_handle();
    if (!h) return fail(nullptr, SKEW_ENOMEM, "out of host memory");
    try {
        h->hp = H;
        h->desc.assign(params, params + n_params);
        h->first.assign(n_params, 0);
        h->count.assign(n_params, 0);
    } catch (...) {
        delete h;
        return fail(nullptr, SKEW_ENOMEM, "out of host memory");
    }
    const int64_t kMaxExtent = int64_t(1) << 40;
    for (int32_t k = 0; k < n_params; ++k) {
        const skew_param_desc_t &d = params[k];
        TPlan p;
        if (!d.weight || !d.grad) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: null weight or grad", k); }
        if (((uintptr_t)d.weight & 1) || ((uintptr_t)d.grad & 1)) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: bf16 pointers must be 2-byte aligned", k); }
        if (d.ndim < 1 || d.ndim > 3) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: ndim must be 1, 2 or 3", k); }
        if (d.tier < SKEW_TIER_BACKBONE || d.tier > SKEW_TIER_ROUTER) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: unknown tier %d", k, d.tier); }
        if (d.flags & ~(SKEW_F_NO_DECAY | SKEW_F_FP32)) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: unknown flags", k); }
        if ((d.flags & SKEW_F_FP32) && (((uintptr_t)d.weight | (uintptr_t)d.grad) & 3)) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: fp32 pointers must be 4-byte aligned", k); }
        if (d.ndim == 3 ? d.stack < 1 : d.stack != 0) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: stack must be >= 1 when ndim == 3 and 0 otherwise", k); }
        const int64_t E = d.ndim == 3 ? (int64_t)d.stack : 1;
        p.n = d.shape[0];
        p.m = d.ndim >= 2 ? d.shape[1] : 1;
        if (p.n < 1 || p.m < 1 || p.n > kMaxExtent || p.m > kMaxExtent) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: extents must be in [1, 2^40]", k); }
        if (p.n > (int64_t(1) << 62) / p.m || p.n * p.m > (int64_t(1) << 62) / E) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: too many elements", k); }
        p.numel = p.n * p.m;
        resolve(d.ndim == 3 ? 2 : d.ndim, d.tier, H.policy, d.flags, p);  // every matrix of a stack is a matrix
        // tiles are indexed with 32 bits: at most 2^31 per matrix
        const int64_t tiles64 = p.kind == kKindFactored ? ((p.m + 255) / 256) * ((p.n + 255) / 256)
                                                        : (p.numel + kFlatTileElems - 1) / kFlatTileElems;
        if (tiles64 > (int64_t(1) << 31)) { delete h; return fail(nullptr, SKEW_EINVAL, "tensor %d: too many elements", k); }
        try {
            h->first[k] = (uint32_t)h->t.size();
            h->count[k] = (uint32_t)E;
            const int64_t esize = (d.flags & SKEW_F_FP32) ? 4 : 2;  // bytes per weight / gradient element
            for (int64_t e = 0; e < E; ++e) {
                TPlan q = p;
                q.w = (char *)d.weight + e * p.numel * esize;
                q.g = (const char *)d.grad + e * p.numel * esize;
                q.tid = (uint32_t)k;
                q.base = (uint64_t)(e * p.numel);
                q.f32 = (d.flags & SKEW_F_FP32) ? 1u : 0u;
                // whole-row tiles and 16-byte vectors are for bf16 rows
                geometry(q, !q.f32 && (((uintptr_t)q.w | (uintptr_t)q.g) & 15) == 0);
                h->n_rowpath += q.rowpath;
                h->t.push_back(q);
            }
        } catch (...) {
            delete h;
            return fail(nullptr, SKEW_ENOMEM, "out of host memory");
        }
    }
    const int32_t n_plans = (int32_t)h->t.size();

    // State layout (fp32 offsets): [momentum arrays][full v arrays][R arrays][C arrays].
    // Arrays whose length is a multiple of 4 come first in each group so that as
    // many as possible start on a 16-byte boundary; there is no padding.
    int64_t off = 0;
    for (int pass = 0; pass < 2; ++pass)
        for (auto &p : h->t)
            if (p.momentum && ((p.numel % 4 == 0) == (pass == 0))) { p.moff = off; off += p.numel; }
    for (int pass = 0; pass < 2; ++pass)
        for (auto &p : h->t)
            if (p.kind == kKindFull && ((p.numel % 4 == 0) == (pass == 0))) { p.voff = off; off += p.numel; }
    for (auto &p : h->t)
        if (p.kind == kKindFactored) { p.roff = off; off += p.n; }
    for (auto &p : h->t)
        if (p.kind == kKindFactored) { p.coff = off; off += p.m; }
    h->state_bytes = size_t(off) * 4;

    // Item tables: every factored tensor's tiles (phase A), finalize items
    // (phase F) and every tensor's tiles (phases B and C), tensors in order.
    try {
        for (int q = 0; q < n_plans; ++q) {
            const TPlan &p = h->t[q];
            if (p.kind == kKindFactored) {
                if (p.rowpath)
                    for (uint32_t i = 0; i < p.rtiles; ++i) h->itemsR.push_back(make_uint2(q, i));
                else
                    for (uint32_t i = 0; i < p.ntiles; ++i) h->itemsA.push_back(make_uint2(q, i));
                for (uint32_t i = 0; i < p.nfr + p.nfc; ++i) h->itemsF.push_back(make_uint2(q, i));
            }
            if (p.rowpath) {
                for (uint32_t i = 0; i < p.atiles; ++i) h->itemsCR.push_back(make_uint2(q, i));
            } else {
                for (uint32_t i = 0; i < p.ntiles; ++i) h->itemsB.push_back(make_uint2(q, i));
                for (uint32_t i = 0; i < p.ntiles; ++i) h->itemsC.push_back(make_uint2(q, i));
            }
        }
        // the last phase-C row tiles of momentum-free matrices run as two half tiles each
        // (tiles of momentum matrices and tile indices past the mask keep whole tiles)
        std::vector<uint2> tail;
        const size_t ncr = h->itemsCR.size(), nsplit = std::min<size_t>(ncr, kApplyTailSplit);
        for (size_t k = ncr - nsplit; k < ncr; ++k) {
            const uint2 it = h->itemsCR[k];
            if (!h->t[it.x].momentum && it.y <= kTileMask) {
                tail.push_back(make_uint2(it.x, it.y | kHalfTile));
                tail.push_back(make_uint2(it.x, it.y | kHalfTile | kSecondHalf));
            } else {
                tail.push_back(it);
            }
        }
        h->itemsCR.resize(ncr - nsplit);
        h->itemsCR.insert(h->itemsCR.end(), tail.begin(), tail.end());
    } catch (...) {
        delete h;
        return fail(nullptr, SKEW_ENOMEM, "out of host memory");
    }

    // Workspace layout (bytes, 256-aligned regions). The scalars and the row
    // path's phase-B queue ([count][tensor ids]) are zeroed every step.
    size_t w = 0;
    h->ws_scal = w;
    w = align_up(w + sizeof(TensorScal) * n_plans, 256);
    h->ws_fb = w;
    w = align_up(w + 4 * (size_t(h->n_rowpath) + 1), 256);
    h->ws_err = w;
    w = align_up(w + 16, 256);
    h->ws_tab = w;
    h->ws_tens = w;
    w = align_up(w + sizeof(TensorDev) * n_plans, 256);
    auto table = [&](size_t &at, const std::vector<uint2> &v) {
        at = w;
        w = align_up(w + sizeof(uint2) * v.size(), 256);
    };
    table(h->ws_itemsA, h->itemsA);
    table(h->ws_itemsR, h->itemsR);
    table(h->ws_itemsF, h->itemsF);
    table(h->ws_itemsB, h->itemsB);
    table(h->ws_itemsC, h->itemsC);
    table(h->ws_itemsCR, h->itemsCR);
    h->ws_tab_end = w;
    for (auto &p : h->t) {
        if (p.kind == kKindFactored && !p.rowpath) {
            p.ws_rowp = w; w = align_up(w + 4 * size_t(p.strips) * p.n, 256);
            p.ws_colp = w; w = align_up(w + 4 * size_t(p.rowtiles) * p.m, 256);
            p.ws_bsc = w;  w = align_up(w + 4 * size_t(p.m), 256);
            p.ws_rsum = w; w = align_up(w + 8 * size_t(p.nfr), 256);
        } else if (p.kind == kKindFactored) {
            p.ws_pp = w;   w = align_up(w + 8 * size_t(p.rtiles) * p.m, 256);
            p.ws_bsc = w;  w = align_up(w + 4 * size_t(p.m), 256);
            p.ws_rsum = w; w = align_up(w + 8 * size_t(p.rtiles), 256);
            p.ws_rmin = w; w = align_up(w + 4 * size_t(p.rtiles), 256);
            p.ws_fsum = w; w = align_up(w + 8 * size_t(p.nfc), 256);
            p.ws_fmin = w; w = align_up(w + 4 * size_t(p.nfc), 256);
        }
        p.ws_u2 = w;
        w = align_up(w + 8 * size_t(p.ntiles), 256);
    }
    h->ws_bytes = w;
    *out = h;
    return SKEW_OK;
}

int skew_destroy(skew_handle_t *h) {
    delete h;
    return SKEW_OK;
}

size_t skew_state_bytes(const skew_handle_t *h) { return h ? h->state_bytes : 0; }

size_t skew_workspace_bytes(const skew_handle_t *h) { return h ? h->ws_bytes : 0; }

int32_t skew_num_tensors(const skew_handle_t *h) { return h ? (int32_t)h->desc.size() : 0; }

int64_t skew_launches_per_step(const skew_handle_t *h) {
    if (!h) return 0;
    return int64_t(!h->itemsA.empty()) + int64_t(!h->itemsR.empty()) + int64_t(!h->itemsF.empty()) +
           int64_t(!h->itemsB.empty()) + int64_t(h->n_rowpath > 0) + int64_t(!h->itemsC.empty()) +
           int64_t(!h->itemsCR.empty());
}

const char *skew_last_error(const skew_handle_t *h) { return h ? h->err.c_str() : g_create_err.c_str(); }

int skew_tensor_info(const skew_handle_t *h, int32_t tid, skew_tensor_info_t *out) {
    if (!h || !out) return SKEW_EINVAL;
    if (tid < 0 || tid >= (int32_t)h->desc.size()) return fail(const_cast<skew_handle_t *>(h), SKEW_EINVAL, "tid %d out of range", tid);
    const TPlan &p = h->t[h->first[tid]];  // a stack's matrices share kind, shape and path; arrays follow on
    out->kind = p.kind;
    out->momentum = p.momentum;
    out->decay = p.decay;
    out->vectorized = p.vec;
    out->rows = p.n;
    out->cols = p.m;
    out->numel = p.numel * (int64_t)h->count[tid];
    out->m_offset = p.moff;
    out->v_offset = p.voff;
    out->r_offset = p.roff;
    out->c_offset = p.coff;
    out->rowpath = (int32_t)p.rowpath;
    out->stack = h->desc[tid].ndim == 3 ? (int32_t)h->count[tid] : 0;
    return SKEW_OK;
}

int skew_bind(skew_handle_t *h, void *state, size_t state_bytes, void *workspace, size_t workspace_bytes, void *stream) {
    if (!h) return SKEW_EINVAL;
    if (state_bytes != h->state_bytes) return fail(h, SKEW_EINVAL, "state buffer is %zu bytes, need exactly %zu", state_bytes, h->state_bytes);
    if (workspace_bytes != h->ws_bytes) return fail(h, SKEW_EINVAL, "workspace is %zu bytes, need exactly %zu", workspace_bytes, h->ws_bytes);
    if ((h->state_bytes && !state) || (h->ws_bytes && !workspace)) return fail(h, SKEW_EINVAL, "null device buffer");
    if (((uintptr_t)state & 255) || ((uintptr_t)workspace & 255)) return fail(h, SKEW_EINVAL, "state and workspace must be 256-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    h->state = (char *)state;
    h->ws = (char *)workspace;
    h->bound = false;

    // Host image of [TensorDev table][item tables].
    std::vector<char> img;
    try {
        img.assign(h->ws_tab_end - h->ws_tab, 0);
    } catch (...) {
        return fail(h, SKEW_ENOMEM, "out of host memory");
    }
    TensorDev *td = reinterpret_cast<TensorDev *>(img.data() + (h->ws_tens - h->ws_tab));
    float *sf = reinterpret_cast<float *>(state);
    auto al16 = [](const void *p) { return ((uintptr_t)p & 15) == 0; };
    for (size_t k = 0; k < h->t.size(); ++k) {
        TPlan &p = h->t[k];
        TensorDev &T = td[k];
        T.w = (uint16_t *)p.w;
        T.g = (const uint16_t *)p.g;
        T.M = p.moff >= 0 ? sf + p.moff : nullptr;
        T.v = p.voff >= 0 ? sf + p.voff : nullptr;
        T.R = p.roff >= 0 ? sf + p.roff : nullptr;
        T.C = p.coff >= 0 ? sf + p.coff : nullptr;
        const bool fact = p.kind == kKindFactored, row = fact && p.rowpath;
        T.rowp = fact && !row ? (float *)(h->ws + p.ws_rowp) : nullptr;
        T.colp = fact && !row ? (float *)(h->ws + p.ws_colp) : nullptr;
        T.bsc = fact ? (float *)(h->ws + p.ws_bsc) : nullptr;
        T.rsum = fact ? (double *)(h->ws + p.ws_rsum) : nullptr;
        T.pp = row ? (float2 *)(h->ws + p.ws_pp) : nullptr;
        T.rmin = row ? (float *)(h->ws + p.ws_rmin) : nullptr;
        T.fsum = row ? (double *)(h->ws + p.ws_fsum) : nullptr;
        T.fmin = row ? (float *)(h->ws + p.ws_fmin) : nullptr;
        T.u2 = (float2 *)(h->ws + p.ws_u2);
        T.n = p.n;
        T.m = p.m;
        T.numel = p.numel;
        T.tid = p.tid;
        T.base = p.base;
        T.kind = p.kind;
        T.momentum = p.momentum;
        T.decay = p.decay;
        bool vec = !p.f32 && al16(T.w) && al16(T.g) && (!T.M || al16(T.M));
        if (p.kind == kKindFull)
            vec = vec && (p.numel % 8 == 0) && al16(T.v);
        else
            vec = vec && (p.m % 8 == 0);
        p.vec = vec ? 1 : 0;
        T.vec = p.vec;
        T.f32 = p.f32;
        T.lcl = p.lcl;
        T.strips = p.strips;
        T.rowtiles = p.rowtiles;
        T.tile_rows = p.tile_rows;
        T.ntiles = p.ntiles;
        T.nfr = p.nfr;
        T.nfc = p.nfc;
        T.rowpath = p.rowpath;
        T.cr = p.cr;
        T.rt_rows = p.rt_rows;
        T.rtiles = p.rtiles;
        T.at_rows = p.at_rows;
        T.atiles = p.atiles;
        T.fci = p.fci;
    }
    auto put = [&](size_t at, const std::vector<uint2> &v) {
        if (!v.empty()) std::memcpy(img.data() + (at - h->ws_tab), v.data(), v.size() * sizeof(uint2));
    };
    put(h->ws_itemsA, h->itemsA);
    put(h->ws_itemsR, h->itemsR);
    put(h->ws_itemsF, h->itemsF);
    put(h->ws_itemsB, h->itemsB);
    put(h->ws_itemsC, h->itemsC);
    put(h->ws_itemsCR, h->itemsCR);

    cudaError_t e;
    if (!img.empty()) {
        e = cudaMemcpyAsync(h->ws + h->ws_tab, img.data(), img.size(), cudaMemcpyHostToDevice, s);
        if (e != cudaSuccess) return cuda_fail(h, e, "upload of descriptor tables");
        // the pageable source may be freed on return only once the copy has been staged
        e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_fail(h, e, "upload of descriptor tables");
    }
    if (h->state_bytes) {
        e = cudaMemsetAsync(state, 0, h->state_bytes, s);
        if (e != cudaSuccess) return cuda_fail(h, e, "zero-fill of the state");
    }
    if (h->ws_bytes) {
        e = cudaMemsetAsync(h->ws + h->ws_scal, 0, h->ws_tab - h->ws_scal, s);
        if (e != cudaSuccess) return cuda_fail(h, e, "zero-fill of the scalars");
    }
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(h, e, "bind");
    // the row path's phase-B launch: two CTAs per SM split a queued tensor's tiles
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess || (e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return cuda_fail(h, e, "device query");
    h->fb_ctas = (uint32_t)(2 * (sms > 0 ? sms : 1));

    h->bound = true;
    return SKEW_OK;
}

int skew_step(skew_handle_t *h, int64_t step, float lr, uint64_t seed, void *stream) {
    return skew_step_scaled(h, step, lr, seed, nullptr, stream);
}

int skew_step_scaled(skew_handle_t *h, int64_t step, float lr, uint64_t seed, const float *grad_scale, void *stream) {
    if (!h) return SKEW_EINVAL;
    if ((uintptr_t)grad_scale & 3) return fail(h, SKEW_EINVAL, "grad_scale must be a 4-byte aligned device pointer");
    if (!h->bound) return fail(h, SKEW_ESTATE, "skew_step before skew_bind");
    if (step < 1) return fail(h, SKEW_EINVAL, "step must be >= 1 (got %lld)", (long long)step);
    if (!std::isfinite(lr) || lr < 0.f) return fail(h, SKEW_EINVAL, "lr must be finite and >= 0");
    if (h->t.empty()) return SKEW_OK;
    cudaStream_t s = (cudaStream_t)stream;
    const skew_hparams_t &H = h->hp;
    const StepCoefs k = step_coefs(H, step);

    StepArgs a{};
    a.tensors = reinterpret_cast<const TensorDev *>(h->ws + h->ws_tens);
    a.scal = reinterpret_cast<TensorScal *>(h->ws + h->ws_scal);
    a.err = reinterpret_cast<uint32_t *>(h->ws + h->ws_err);
    a.fb = reinterpret_cast<uint32_t *>(h->ws + h->ws_fb);
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
    a.gscale = grad_scale;

    cudaEvent_t *ev = nullptr;
    if (h->prof_used < h->prof_max) {
        ev = h->prof_ev.data() + size_t(h->prof_used) * (kProfLaunches + 1);
        ++h->prof_used;
    }
    cudaError_t e = cudaMemsetAsync(h->ws + h->ws_scal, 0, h->ws_fb + 4 - h->ws_scal, s);
    if (e != cudaSuccess) return cuda_fail(h, e, "reset of per-step scalars");
    auto items = [&](size_t at) { return reinterpret_cast<const uint2 *>(h->ws + at); };
    const LaunchPlan L{(uint32_t)h->itemsA.size(), (uint32_t)h->itemsR.size(), (uint32_t)h->itemsF.size(),
                       (uint32_t)h->itemsB.size(), h->n_rowpath ? h->fb_ctas : 0u, (uint32_t)h->itemsC.size(),
                       (uint32_t)h->itemsCR.size(), items(h->ws_itemsA), items(h->ws_itemsR), items(h->ws_itemsF),
                       items(h->ws_itemsB), items(h->ws_itemsC), items(h->ws_itemsCR)};
    e = (cudaError_t)launch_phases(a, L, s, reinterpret_cast<void *const *>(ev));
    if (e != cudaSuccess) return cuda_fail(h, e, "kernel launch");
    return SKEW_OK;
}

int skew_profile_begin(skew_handle_t *h, int32_t max_steps) {
    if (!h || max_steps < 0 || max_steps > (1 << 20)) return SKEW_EINVAL;
    for (cudaEvent_t e : h->prof_ev) cudaEventDestroy(e);
    h->prof_ev.clear();
    h->prof_max = h->prof_used = 0;
    try {
        h->prof_ev.resize(size_t(max_steps) * (kProfLaunches + 1), nullptr);
    } catch (...) {
        return fail(h, SKEW_ENOMEM, "out of host memory");
    }
    for (auto &ev : h->prof_ev) {
        cudaError_t e = cudaEventCreate(&ev);
        if (e != cudaSuccess) {
            ev = nullptr;
            return cuda_fail(h, e, "event create");
        }
    }
    h->prof_max = max_steps;
    return SKEW_OK;
}

int skew_profile_end(skew_handle_t *h, double *ms, int64_t cap, int32_t *n_steps, int32_t *n_kernels) {
    if (!h || (cap > 0 && !ms)) return SKEW_EINVAL;
    int rc = SKEW_OK;
    int64_t w = 0;
    for (int32_t st = 0; st < h->prof_used; ++st) {
        cudaEvent_t *ev = h->prof_ev.data() + size_t(st) * (kProfLaunches + 1);
        for (int k = 0; k < kProfLaunches; ++k) {
            float t = 0.f;
            cudaError_t e = cudaEventSynchronize(ev[k + 1]);
            if (e == cudaSuccess) e = cudaEventElapsedTime(&t, ev[k], ev[k + 1]);
            if (e != cudaSuccess && rc == SKEW_OK) rc = cuda_fail(h, e, "event timing");
            if (w < cap) ms[w] = t;
            ++w;
        }
    }
    if (n_steps) *n_steps = h->prof_used;
    if (n_kernels) *n_kernels = kProfLaunches;
    for (cudaEvent_t e : h->prof_ev) cudaEventDestroy(e);
    h->prof_ev.clear();
    h->prof_max = h->prof_used = 0;
    return rc;
}

const char *skew_kernel_name(int32_t k) { return (k >= 0 && k < kProfLaunches) ? kProfNames[k] : ""; }

int skew_sync_status(skew_handle_t *h, void *stream) {
    if (!h) return SKEW_EINVAL;
    if (!h->bound) return fail(h, SKEW_ESTATE, "not bound");
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(h, e, "stream synchronize");
    uint32_t word = 0;
    e = cudaMemcpy(&word, h->ws + h->ws_err, 4, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(h, e, "status read");
    if (word) {
        cudaMemset(h->ws + h->ws_err, 0, 4);
        return fail(h, SKEW_ETIMEOUT, "device wait gave up (status 0x%x)", word);
    }
    return SKEW_OK;
}

int skew_selftest_wait_timeout(skew_handle_t *h, void *stream) {
    if (!h) return SKEW_EINVAL;
    if (!h->bound) return fail(h, SKEW_ESTATE, "not bound");
    const cudaError_t e = (cudaError_t)launch_wait_selftest(reinterpret_cast<uint32_t *>(h->ws + h->ws_err), stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "kernel launch");
    return SKEW_OK;
}

int skew_tensor_scalars(skew_handle_t *h, int32_t tid, double out[4], void *stream) {
    return skew_matrix_scalars(h, tid, 0, out, stream);
}

int skew_matrix_scalars(skew_handle_t *h, int32_t tid, int32_t e, double out[4], void *stream) {
    if (!h || !out) return SKEW_EINVAL;
    if (tid < 0 || tid >= (int32_t)h->desc.size()) return fail(h, SKEW_EINVAL, "tid %d out of range", tid);
    if (e < 0 || e >= (int32_t)h->count[tid]) return fail(h, SKEW_EINVAL, "matrix %d of tensor %d out of range", e, tid);
    if (!h->bound) return fail(h, SKEW_ESTATE, "not bound");
    const size_t k = h->first[tid] + (uint32_t)e;
    cudaError_t err = cudaStreamSynchronize((cudaStream_t)stream);
    if (err != cudaSuccess) return cuda_fail(h, err, "stream synchronize");
    TensorScal sc;
    err = cudaMemcpy(&sc, h->ws + h->ws_scal + sizeof(TensorScal) * k, sizeof sc, cudaMemcpyDeviceToHost);
    if (err != cudaSuccess) return cuda_fail(h, err, "scalar read");
    out[0] = sc.rbar;
    out[1] = sc.sumsq;
    out[2] = sc.rms;
    out[3] = sc.kappa;
    return SKEW_OK;
}

}  // extern "C"
