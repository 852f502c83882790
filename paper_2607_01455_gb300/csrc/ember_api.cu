// Host side of the C ABI declared in include/ember.h: argument checks,
// workspace layout and kernel dispatch.  Every check runs before anything is
// launched, so a rejected call leaves the GPU untouched.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "ember_internal.h"

namespace ember {

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

Layout make_layout(int64_t V, int64_t D, int64_t max_sparse_N)
{
    Layout L{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        const size_t at = off;
        off = align_up(off + (bytes ? bytes : 1), 256);
        return at;
    };
    const size_t nstate = (size_t)((D + kStateCols - 1) / kStateCols);
    L.scalars = take(sizeof(DevScalars));
    L.rsum_part = take(sizeof(float) * kRsumParts);
    L.csum_part = take(sizeof(double) * nstate);
    L.colpart = take(sizeof(float) * (size_t)kPartRows * (size_t)D);
    if (max_sparse_N > 0) {
        const size_t N = (size_t)max_sparse_N;
        const size_t Npad = (N + kSortTile - 1) / kSortTile * kSortTile;
        const size_t nslices = (size_t)((D + kThreads - 1) / kThreads);
        L.sp_keys = take(sizeof(uint64_t) * Npad);
        L.sp_rank = take(sizeof(int32_t) * Npad);
        L.sp_sorted = take(sizeof(uint64_t) * N);
        L.sp_tilecnt = take(sizeof(int32_t) * 2 * (Npad / kSortTile));
        L.sp_perm = take(sizeof(int32_t) * N);
        L.sp_segidx = take(sizeof(int32_t) * N);
        L.sp_uniq = take(sizeof(int32_t) * N);
        L.sp_segoff = take(sizeof(int32_t) * (N + 1));
        L.sp_slot = take(sizeof(int32_t) * (size_t)V);
        L.sp_single = take(sizeof(int32_t) * N);
        L.sp_rowpart = take(sizeof(float) * N * nslices);
        L.sp_carry = take(sizeof(float) * 2 * (size_t)kSparseCtas * (size_t)D);
        L.sp_bounds = take(sizeof(int32_t) * ((size_t)kSparseCtas + 1));
        L.sp_rows = take(sizeof(float) * N * (size_t)D);
    }
    L.lm_colpart = take(sizeof(float) * (size_t)lmhead_row_blocks(V) * (size_t)D);
    L.lm_rowpart = take(sizeof(float) * (size_t)lmhead_col_blocks(D) * (size_t)V);
    L.total = off;
    return L;
}

}  // namespace ember

using namespace ember;

static bool is_aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

static bool hparams_ok(const ember_hparams &hp)
{
    return hp.beta2 >= 0.0 && hp.beta2 < 1.0 && isfinite(hp.eps) && hp.eps >= 0.0 &&
           (hp.maximize == 0 || hp.maximize == 1) &&
           (hp.bias_correction == 0 || hp.bias_correction == 1) &&
           hp.variant >= EMBER_VARIANT_FULL && hp.variant <= EMBER_VARIANT_COL;
}

extern "C" {

void ember_hparams_default(ember_hparams *hp)
{
    if (!hp)
        return;
    hp->beta2 = 0.999;
    hp->eps = 1e-8;
    hp->maximize = 0;
    hp->bias_correction = 1;
    hp->variant = EMBER_VARIANT_FULL;
}

ember_status ember_create(int64_t V, int64_t D, const ember_hparams *hp, ember_wdtype wdtype,
                          ember_handle **out)
{
    if (!out)
        return EMBER_ERR_INVALID_ARG;
    *out = nullptr;
    if (V < 1 || D < 1 || V > (int64_t(1) << 62) / D)
        return EMBER_ERR_INVALID_ARG;
    if (D > INT32_MAX || V > INT32_MAX)
        return EMBER_ERR_UNSUPPORTED;
    if (wdtype != EMBER_F32 && wdtype != EMBER_BF16)
        return EMBER_ERR_DTYPE;
    ember_hparams h;
    if (hp)
        h = *hp;
    else
        ember_hparams_default(&h);
    if (!hparams_ok(h))
        return EMBER_ERR_INVALID_ARG;
    ColMap m;
    if (!choose_colmap(D, true, &m))  // wider rows than one CTA holds
        return EMBER_ERR_UNSUPPORTED;
    ember_handle *e = (ember_handle *)calloc(1, sizeof(ember_handle));
    if (!e)
        return EMBER_ERR_INVALID_ARG;
    e->V = V;
    e->D = D;
    e->hp = h;
    e->wdtype = wdtype;
    e->wait_ns = kDefaultWaitNs;
    *out = e;
    return EMBER_OK;
}

void ember_destroy(ember_handle *h) { free(h); }

int ember_column_panels(const ember_handle *h, int vector_path)
{
    ColMap m;
    if (!h || !choose_colmap(h->D, vector_path != 0, &m))
        return 0;
    return m.npanels;
}

int ember_dense_step_launches(const ember_handle *h, int vector_path)
{
    if (!h)
        return 0;
    return dense_step_launches(h->V, h->D, h->wdtype == EMBER_BF16, h->hp.variant, vector_path != 0);
}

size_t ember_state_numel(const ember_handle *h)
{
    return h ? (size_t)(h->V + h->D) : 0;
}

size_t ember_workspace_bytes(const ember_handle *h, int64_t max_sparse_N)
{
    if (!h || max_sparse_N < 0 || max_sparse_N > INT32_MAX / 2)
        return 0;
    return make_layout(h->V, h->D, max_sparse_N).total;
}

ember_status ember_bind_workspace(ember_handle *h, void *workspace, size_t bytes,
                                  int64_t max_sparse_N, void *stream)
{
    if (!h || !workspace || max_sparse_N < 0 || max_sparse_N > INT32_MAX / 2)
        return EMBER_ERR_INVALID_ARG;
    if (!is_aligned(workspace, 256))
        return EMBER_ERR_ALIGNMENT;
    const Layout L = make_layout(h->V, h->D, max_sparse_N);
    if (bytes < L.total)
        return EMBER_ERR_WORKSPACE;
    int dev = 0;
    cudaDeviceProp prop;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess)
        return EMBER_ERR_CUDA;
    if (prop.major != 10 || prop.minor != 3)
        return EMBER_ERR_UNSUPPORTED;
    if (cudaMemsetAsync((unsigned char *)workspace + L.scalars, 0, sizeof(DevScalars),
                        (cudaStream_t)stream) != cudaSuccess)
        return EMBER_ERR_CUDA;
    // the sparse step expects an all-zero slot map and leaves it all-zero
    if (max_sparse_N > 0 &&
        cudaMemsetAsync((unsigned char *)workspace + L.sp_slot, 0, sizeof(int32_t) * (size_t)h->V,
                        (cudaStream_t)stream) != cudaSuccess)
        return EMBER_ERR_CUDA;
    h->ws = (unsigned char *)workspace;
    h->ws_bytes = bytes;
    h->ws_max_N = max_sparse_N;
    return EMBER_OK;
}

ember_status ember_step_dense(ember_handle *h, void *W, const float *G, float *state, float lr,
                              int64_t t, void *stream)
{
    if (!h || !W || !G || !state)
        return EMBER_ERR_INVALID_ARG;
    if (t < 1 || !isfinite(lr))
        return EMBER_ERR_INVALID_ARG;
    const size_t wsz = h->wdtype == EMBER_BF16 ? 2 : 4;
    if (!is_aligned(W, wsz) || !is_aligned(G, 4) || !is_aligned(state, 4))
        return EMBER_ERR_ALIGNMENT;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;

    DenseArgs a{};
    a.V = h->V;
    a.D = h->D;
    a.wbf16 = h->wdtype == EMBER_BF16;
    a.W = W;
    a.G = G;
    a.r = state;
    a.c = state + h->V;
    a.beta2 = h->hp.beta2;
    a.one_minus_beta2 = 1.0 - h->hp.beta2;
    a.inv_bc = h->hp.bias_correction ? 1.0 / (1.0 - pow(h->hp.beta2, (double)t)) : 1.0;
    a.lr_signed = h->hp.maximize ? lr : -lr;
    a.eps = (float)h->hp.eps;
    a.variant = h->hp.variant;
    a.ws = h->ws;
    a.lay = make_layout(h->V, h->D, h->ws_max_N);
    a.stream = (cudaStream_t)stream;
    a.trace = (h->n_trace >= 4) ? h->trace : nullptr;
    a.wait_ns = h->wait_ns;
    const bool vec4 = (h->D % 4 == 0) && is_aligned(W, 4 * wsz) && is_aligned(G, 16);
    if (!choose_colmap(h->D, vec4, &a.map))
        return EMBER_ERR_UNSUPPORTED;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_step_dense_from_host(ember_handle *h, void *W, const float *G_host, float *G_stage,
                                        float *state, float lr, int64_t t, void *stream)
{
    if (!h || !W || !G_host || !G_stage || !state)
        return EMBER_ERR_INVALID_ARG;
    if (t < 1 || !isfinite(lr))
        return EMBER_ERR_INVALID_ARG;
    if (h->hp.variant == EMBER_VARIANT_ROW)
        return EMBER_ERR_UNSUPPORTED;
    const size_t wsz = h->wdtype == EMBER_BF16 ? 2 : 4;
    if (!is_aligned(W, wsz) || !is_aligned(G_host, 4) || !is_aligned(G_stage, 4) || !is_aligned(state, 4))
        return EMBER_ERR_ALIGNMENT;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;
    // the GPU must be able to address G_host
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, G_host) != cudaSuccess) {
        cudaGetLastError();
        return EMBER_ERR_INVALID_ARG;
    }
    const float *G_dev = static_cast<const float *>(attr.devicePointer);
    if (attr.type == cudaMemoryTypeUnregistered || !G_dev)
        return EMBER_ERR_INVALID_ARG;

    DenseArgs a{};
    a.V = h->V;
    a.D = h->D;
    a.wbf16 = h->wdtype == EMBER_BF16;
    a.W = W;
    a.G = G_dev;
    a.G_stage = G_stage;
    a.r = state;
    a.c = state + h->V;
    a.beta2 = h->hp.beta2;
    a.one_minus_beta2 = 1.0 - h->hp.beta2;
    a.inv_bc = h->hp.bias_correction ? 1.0 / (1.0 - pow(h->hp.beta2, (double)t)) : 1.0;
    a.lr_signed = h->hp.maximize ? lr : -lr;
    a.eps = (float)h->hp.eps;
    a.variant = h->hp.variant;
    a.ws = h->ws;
    a.lay = make_layout(h->V, h->D, h->ws_max_N);
    a.stream = (cudaStream_t)stream;
    a.trace = (h->n_trace >= 4) ? h->trace : nullptr;
    a.wait_ns = h->wait_ns;
    const bool vec4 = (h->D % 4 == 0) && is_aligned(W, 4 * wsz) && is_aligned(G_dev, 16) &&
                      is_aligned(G_stage, 16);
    if (!choose_colmap(h->D, vec4, &a.map))
        return EMBER_ERR_UNSUPPORTED;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

static ember_status check_lmhead(const ember_handle *h, const void *dlogits, const void *hidden, int64_t T,
                                 const float *G)
{
    if (!dlogits || !hidden || !G || T < 1 || T > INT32_MAX)
        return EMBER_ERR_INVALID_ARG;
    if (h->V % 8 != 0 || h->D % 8 != 0 || h->V > INT32_MAX)
        return EMBER_ERR_UNSUPPORTED;
    if (!is_aligned(dlogits, 16) || !is_aligned(hidden, 16) || !is_aligned(G, 16))
        return EMBER_ERR_ALIGNMENT;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;
    return EMBER_OK;
}

ember_status ember_lmhead_grad(ember_handle *h, const void *dlogits, const void *hidden, int64_t T, float *G,
                               void *stream)
{
    if (!h)
        return EMBER_ERR_INVALID_ARG;
    const ember_status st = check_lmhead(h, dlogits, hidden, T, G);
    if (st != EMBER_OK)
        return st;
    const Layout L = make_layout(h->V, h->D, h->ws_max_N);
    LmArgs lm{h->V, h->D, T, dlogits, hidden, G, h->wait_ns};
    DevScalars *sc = reinterpret_cast<DevScalars *>(h->ws + L.scalars);
    const cudaError_t e = launch_lmhead_grad(lm, reinterpret_cast<float *>(h->ws + L.lm_colpart),
                                             reinterpret_cast<float *>(h->ws + L.lm_rowpart), &sc->flags,
                                             (cudaStream_t)stream);
    return e == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_step_lmhead(ember_handle *h, void *W, const void *dlogits, const void *hidden, int64_t T,
                               float *G, float *state, float lr, int64_t t, void *stream)
{
    if (!h || !W || !state)
        return EMBER_ERR_INVALID_ARG;
    if (t < 1 || !isfinite(lr))
        return EMBER_ERR_INVALID_ARG;
    const ember_status st = check_lmhead(h, dlogits, hidden, T, G);
    if (st != EMBER_OK)
        return st;
    const size_t wsz = h->wdtype == EMBER_BF16 ? 2 : 4;
    if (!is_aligned(W, wsz) || !is_aligned(state, 4))
        return EMBER_ERR_ALIGNMENT;

    LmArgs lm{h->V, h->D, T, dlogits, hidden, G, h->wait_ns};
    DenseArgs a{};
    a.V = h->V;
    a.D = h->D;
    a.wbf16 = h->wdtype == EMBER_BF16;
    a.W = W;
    a.G = G;
    a.r = state;
    a.c = state + h->V;
    a.beta2 = h->hp.beta2;
    a.one_minus_beta2 = 1.0 - h->hp.beta2;
    a.inv_bc = h->hp.bias_correction ? 1.0 / (1.0 - pow(h->hp.beta2, (double)t)) : 1.0;
    a.lr_signed = h->hp.maximize ? lr : -lr;
    a.eps = (float)h->hp.eps;
    a.variant = h->hp.variant;
    a.ws = h->ws;
    a.lay = make_layout(h->V, h->D, h->ws_max_N);
    a.stream = (cudaStream_t)stream;
    a.trace = (h->n_trace >= 4) ? h->trace : nullptr;
    a.wait_ns = h->wait_ns;
    a.lm = &lm;
    const bool vec4 = is_aligned(W, 4 * wsz);  // D % 8 == 0 and G 16-byte aligned already
    if (!choose_colmap(h->D, vec4, &a.map))
        return EMBER_ERR_UNSUPPORTED;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

// ---- row-sharded dense step ----

static bool shard_plan(const ember_handle *h, int shard, int nshards, ShardArgs *p)
{
    if (!h || nshards < 1 || nshards > kMaxShards || shard < 0 || shard >= nshards)
        return false;
    const int nparts = dense_parts(h->V, h->D);
    const int cap = (nparts + nshards - 1) / nshards;
    int b0 = shard * cap, b1 = (shard + 1) * cap;
    if (b0 > nparts)
        b0 = nparts;
    if (b1 > nparts)
        b1 = nparts;
    p->cta_begin = b0;
    p->cta_end = b1;
    p->row_base = (int64_t)b0 * h->V / nparts;
    return true;
}

int64_t ember_shard_rows(const ember_handle *h, int shard, int nshards, int64_t *row0)
{
    ShardArgs p{};
    if (!shard_plan(h, shard, nshards, &p))
        return -1;
    const int nparts = dense_parts(h->V, h->D);
    const int64_t r1 = (int64_t)p.cta_end * h->V / nparts;
    if (row0)
        *row0 = p.row_base;
    return r1 - p.row_base;
}

size_t ember_shard_scale_bytes(const ember_handle *h) { return h ? (size_t)(h->D + 1) : 0; }

size_t ember_shard_exchange_bytes(const ember_handle *h)
{
    return h ? sizeof(unsigned long long) * (size_t)(h->D + 1) : 0;
}

// Checks shared by the three phases; fills the plan and the common step
// arguments.  G_shard / W_shard are checked only when given (non-null).
static ember_status shard_common(ember_handle *h, int shard, int nshards, const void *W_shard, const float *G_shard,
                                 const float *state, ShardArgs *p, DenseArgs *a)
{
    if (!h || !state)
        return EMBER_ERR_INVALID_ARG;
    if (!shard_plan(h, shard, nshards, p))
        return EMBER_ERR_INVALID_ARG;
    if (h->hp.variant == EMBER_VARIANT_ROW)
        return EMBER_ERR_UNSUPPORTED;  // the row-only step has its own one-pass kernel
    // every shard must take the same vector path as the whole-table step
    const size_t wsz = h->wdtype == EMBER_BF16 ? 2 : 4;
    const bool vec4 = h->D % 4 == 0;
    if (!is_aligned(state, 4) || (G_shard && !is_aligned(G_shard, vec4 ? 16 : 4)) ||
        (W_shard && !is_aligned(W_shard, vec4 ? 4 * wsz : wsz)))
        return EMBER_ERR_ALIGNMENT;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;
    a->V = h->V;
    a->D = h->D;
    a->wbf16 = h->wdtype == EMBER_BF16;
    a->G = G_shard;
    a->r = const_cast<float *>(state);
    a->c = const_cast<float *>(state) + h->V;
    a->beta2 = h->hp.beta2;
    a->one_minus_beta2 = 1.0 - h->hp.beta2;
    a->eps = (float)h->hp.eps;
    a->variant = h->hp.variant;
    a->ws = h->ws;
    a->lay = make_layout(h->V, h->D, h->ws_max_N);
    a->trace = nullptr;
    a->wait_ns = h->wait_ns;
    if (!choose_colmap(h->D, vec4, &a->map))
        return EMBER_ERR_UNSUPPORTED;
    if (a->map.npanels != 1)
        return EMBER_ERR_UNSUPPORTED;  // a shard's rows must fit one CTA whole
    return EMBER_OK;
}

ember_status ember_shard_reduce(ember_handle *h, int shard, int nshards, const float *G_shard, float *state,
                                unsigned char *scales, void *stream)
{
    ShardArgs p{};
    DenseArgs a{};
    if (!scales)
        return EMBER_ERR_INVALID_ARG;
    const ember_status st = shard_common(h, shard, nshards, nullptr, G_shard, state, &p, &a);
    if (st != EMBER_OK)
        return st;
    if (p.cta_end > p.cta_begin && !G_shard)
        return EMBER_ERR_INVALID_ARG;
    p.phase = 1;
    p.scales = scales;
    a.shard = &p;
    a.inv_bc = 1.0;
    a.stream = (cudaStream_t)stream;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_shard_pack(ember_handle *h, int shard, int nshards, const unsigned char *scales,
                              unsigned long long *sums, void *stream)
{
    ShardArgs p{};
    DenseArgs a{};
    if (!h || !scales || !sums)
        return EMBER_ERR_INVALID_ARG;
    if (!is_aligned(sums, 8))
        return EMBER_ERR_ALIGNMENT;
    // the state is not touched by this phase; any aligned non-null pointer
    // passes the shared checks
    const ember_status st = shard_common(h, shard, nshards, nullptr, nullptr, reinterpret_cast<float *>(sums), &p,
                                         &a);
    if (st != EMBER_OK)
        return st;
    p.phase = 2;
    p.scales = const_cast<unsigned char *>(scales);
    p.sums = sums;
    a.shard = &p;
    a.inv_bc = 1.0;
    a.stream = (cudaStream_t)stream;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_shard_update(ember_handle *h, int shard, int nshards, void *W_shard, const float *G_shard,
                                float *state, const unsigned char *scales, const unsigned long long *sums, float lr,
                                int64_t t, void *stream)
{
    if (t < 1 || !isfinite(lr))
        return EMBER_ERR_INVALID_ARG;
    if (!scales || !sums)
        return EMBER_ERR_INVALID_ARG;
    if (!is_aligned(sums, 8))
        return EMBER_ERR_ALIGNMENT;
    ShardArgs p{};
    DenseArgs a{};
    a.W = W_shard;
    const ember_status st = shard_common(h, shard, nshards, W_shard, G_shard, state, &p, &a);
    if (st != EMBER_OK)
        return st;
    if (p.cta_end > p.cta_begin && (!W_shard || !G_shard))
        return EMBER_ERR_INVALID_ARG;
    p.phase = 3;
    p.scales = const_cast<unsigned char *>(scales);
    p.sums = const_cast<unsigned long long *>(sums);
    a.shard = &p;
    a.inv_bc = h->hp.bias_correction ? 1.0 / (1.0 - pow(h->hp.beta2, (double)t)) : 1.0;
    a.lr_signed = h->hp.maximize ? lr : -lr;
    a.stream = (cudaStream_t)stream;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_step_sparse(ember_handle *h, void *W, const void *ids, ember_idtype idtype,
                               int64_t N, const float *rows, float *state, float lr, int64_t t,
                               void *stream)
{
    if (!h || !W || !state || N < 0 || (N > 0 && (!ids || !rows)))
        return EMBER_ERR_INVALID_ARG;
    if (t < 1 || !isfinite(lr))
        return EMBER_ERR_INVALID_ARG;
    if (idtype != EMBER_I32 && idtype != EMBER_I64)
        return EMBER_ERR_DTYPE;
    const size_t wsz = h->wdtype == EMBER_BF16 ? 2 : 4;
    const size_t isz = idtype == EMBER_I64 ? 8 : 4;
    if (!is_aligned(W, wsz) || !is_aligned(state, 4) || (N > 0 && (!is_aligned(ids, isz) ||
                                                                  !is_aligned(rows, 4))))
        return EMBER_ERR_ALIGNMENT;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;
    if (N > h->ws_max_N)
        return EMBER_ERR_WORKSPACE;

    SparseArgs a{};
    a.V = h->V;
    a.D = h->D;
    a.N = N;
    a.wbf16 = h->wdtype == EMBER_BF16;
    a.ids64 = idtype == EMBER_I64;
    a.W = W;
    a.ids = ids;
    a.rows = rows;
    a.r = state;
    a.c = state + h->V;
    a.beta2 = h->hp.beta2;
    a.one_minus_beta2 = 1.0 - h->hp.beta2;
    a.inv_bc = h->hp.bias_correction ? 1.0 / (1.0 - pow(h->hp.beta2, (double)t)) : 1.0;
    a.lr_signed = h->hp.maximize ? lr : -lr;
    a.eps = (float)h->hp.eps;
    a.variant = h->hp.variant;
    a.ws = h->ws;
    a.lay = make_layout(h->V, h->D, h->ws_max_N);
    a.stream = (cudaStream_t)stream;
    a.trace = h->n_trace > 0 ? h->trace : nullptr;
    a.n_trace = h->n_trace;
    const bool vec4 = (h->D % 4 == 0) && is_aligned(W, 4 * wsz) && (N == 0 || is_aligned(rows, 16));
    if (!choose_colmap(h->D, vec4, &a.map))
        return EMBER_ERR_UNSUPPORTED;
    return launch_sparse_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_sparse_unique(ember_handle *h, const void *ids, ember_idtype idtype, int64_t N,
                                 int32_t *uniq, int32_t *counts, int32_t *n_unique, void *stream)
{
    if (!h || N < 0 || (N > 0 && (!ids || !uniq || !counts)) || !n_unique)
        return EMBER_ERR_INVALID_ARG;
    if (idtype != EMBER_I32 && idtype != EMBER_I64)
        return EMBER_ERR_DTYPE;
    const size_t isz = idtype == EMBER_I64 ? 8 : 4;
    if ((N > 0 && (!is_aligned(ids, isz) || !is_aligned(uniq, 4) || !is_aligned(counts, 4))) ||
        !is_aligned(n_unique, 4))
        return EMBER_ERR_ALIGNMENT;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;
    if (N > h->ws_max_N)
        return EMBER_ERR_WORKSPACE;
    SparseArgs a{};
    a.V = h->V;
    a.D = h->D;
    a.N = N;
    a.ids64 = idtype == EMBER_I64;
    a.ids = ids;
    a.ws = h->ws;
    a.lay = make_layout(h->V, h->D, h->ws_max_N);
    a.stream = (cudaStream_t)stream;
    return launch_sparse_unique(a, uniq, counts, n_unique) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}

ember_status ember_get_device_status(ember_handle *h, void *stream)
{
    if (!h)
        return EMBER_ERR_INVALID_ARG;
    if (!h->ws)
        return EMBER_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    const Layout L = make_layout(h->V, h->D, h->ws_max_N);
    DevScalars *sc = reinterpret_cast<DevScalars *>(h->ws + L.scalars);
    unsigned flags = 0;
    if (cudaMemcpyAsync(&flags, &sc->flags, sizeof flags, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return EMBER_ERR_CUDA;
    if (flags && (cudaMemsetAsync(&sc->flags, 0, sizeof(unsigned), s) != cudaSuccess ||
                  cudaStreamSynchronize(s) != cudaSuccess))
        return EMBER_ERR_CUDA;
    if (flags & kFlagTimeout)
        return EMBER_ERR_TIMEOUT;
    if (flags & kFlagIdRange)
        return EMBER_ERR_ID_OUT_OF_RANGE;
    return EMBER_OK;
}

ember_status ember_set_wait_limit_ns(ember_handle *h, uint64_t ns)
{
    if (!h)
        return EMBER_ERR_INVALID_ARG;
    h->wait_ns = ns ? ns : kDefaultWaitNs;
    return EMBER_OK;
}

ember_status ember_set_trace_events(ember_handle *h, void *const *events, int n)
{
    if (!h || n < 0 || n > kMaxTraceEvents || (n > 0 && !events))
        return EMBER_ERR_INVALID_ARG;
    for (int k = 0; k < n; ++k)
        if (!events[k])
            return EMBER_ERR_INVALID_ARG;
    h->n_trace = events ? n : 0;
    for (int k = 0; k < h->n_trace; ++k)
        h->trace[k] = (cudaEvent_t)events[k];
    return EMBER_OK;
}

const char *ember_status_string(ember_status s)
{
    switch (s) {
    case EMBER_OK: return "ok";
    case EMBER_ERR_INVALID_ARG: return "invalid argument";
    case EMBER_ERR_ALIGNMENT: return "misaligned pointer";
    case EMBER_ERR_DTYPE: return "unknown dtype";
    case EMBER_ERR_WORKSPACE: return "workspace missing or too small";
    case EMBER_ERR_CUDA: return "CUDA error";
    case EMBER_ERR_ID_OUT_OF_RANGE: return "token id outside [0, V) skipped";
    case EMBER_ERR_TIMEOUT: return "bounded device wait gave up";
    case EMBER_ERR_UNSUPPORTED: return "unsupported device or size";
    }
    return "unknown status";
}

int ember_abi_version(void) { return EMBER_ABI_VERSION; }

}  // extern "C"
