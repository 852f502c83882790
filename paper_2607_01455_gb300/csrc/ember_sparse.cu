// Sparse Ember step (Section 2.2 of "Token Geometry", arXiv 2607.01455) for
// sm_103a.
//
// An embedding table's gradient is nonzero only on the rows of the token ids
// in the batch; a token seen k times receives the sum of its k
// per-occurrence rows (appendix "The Fisher is proportional to inverse
// frequency squared": g_i = (1/B) sum_k h_{i,k}).  The step equals the dense
// step of Algorithm 1 on that V x D gradient:
//   - every row of r decays (r_i <- beta2 r_i + (1-beta2) mean_j g_ij^2 with
//     g_i = 0 for rows not in the batch);
//   - the column statistics divide by V;
//   - only the touched rows of W change.
//
// Kernels, in launch order:
//   sort      k_sp_tile_sort, k_sp_rank, k_sp_scatter: the N keys
//             (id << 32 | occurrence) in ascending order, without atomics on
//             floating-point data: 1024-key tiles are bitonic-sorted in shared
//             memory, then every key's global rank is its rank in its tile
//             plus its lower bound in every other tile (integer atomics, so
//             the rank is exact and the order deterministic).
//   dedup     k_sp_heads, k_sp_segments: run heads, the distinct ids
//             (ascending), where each id's run starts, and a V-entry map from
//             a touched row to its distinct-id index.
//   segsum    k_sp_chunks, k_sp_carry: the summed gradient row of every
//             distinct id, adding its occurrences in increasing occurrence
//             order; per (id, column slice) sums of g^2; per-CTA column sums
//             of g^2.  The sorted occurrences are cut into chunks of 32 so the
//             work is even however skewed the id counts are (a Zipf head id
//             can own thousands of occurrences); a run that crosses chunk
//             boundaries is summed piecewise and its pieces are added in
//             chunk order by k_sp_carry.
//   rows      k_sp_vpass: r for all V rows, the sums of new r per CTA, and the
//             touched-row map cleared for the next step.
//   state     the dense step's column/normaliser pass.
//   apply     k_sp_apply: the update of the touched rows only.
#include <cuda_runtime.h>
#include <stdint.h>

#include "ember_device.cuh"
#include "ember_internal.h"

namespace ember {
namespace {

using namespace dev;

constexpr uint64_t kPad = ~0ull;
constexpr int kKeysPerThread = kSortTile / kSortThreads;

template <typename IdT>
__global__ void __launch_bounds__(kSortThreads)
k_sp_tile_sort(const IdT *__restrict__ ids, int64_t N, int64_t V, uint64_t *__restrict__ keys,
               int32_t *__restrict__ rank, DevScalars *sc)
{
    __shared__ uint64_t s[kSortTile];
    const int64_t base = (int64_t)blockIdx.x * kSortTile;
    bool bad = false;
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int i = threadIdx.x + q * kSortThreads;
        const int64_t k = base + i;
        uint64_t key = kPad;
        if (k < N) {
            int64_t id = (int64_t)ids[k];
            if (id < 0 || id >= V) {  // skipped: sorts after every valid id
                bad = true;
                id = V;
            }
            key = ((uint64_t)id << 32) | (uint64_t)k;
        }
        s[i] = key;
    }
    if (bad)
        atomicOr(&sc->flags, kFlagIdRange);
    __syncthreads();
    for (int lk = 1; (1 << lk) <= kSortTile; ++lk) {
        for (int lj = lk - 1; lj >= 0; --lj) {
            const int j = 1 << lj;
#pragma unroll
            for (int q = 0; q < kSortTile / 2 / kSortThreads; ++q) {
                const int p = threadIdx.x + q * kSortThreads;  // pair index
                const int i = ((p >> lj) << (lj + 1)) | (p & (j - 1));
                const int l = i + j;
                const bool up = ((i >> lk) & 1) == 0;
                const uint64_t a = s[i], b = s[l];
                if ((a > b) == up) {
                    s[i] = b;
                    s[l] = a;
                }
            }
            __syncthreads();
        }
    }
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int i = threadIdx.x + q * kSortThreads;
        keys[base + i] = s[i];
        rank[base + i] = i;
    }
}

// CTA (own, other): add to each key of tile `own` the number of keys of tile
// `other` below it.  Keys are unique, so the ranks form a permutation.
__global__ void __launch_bounds__(kSortThreads)
k_sp_rank(const uint64_t *__restrict__ keys, int32_t *__restrict__ rank)
{
    const int own = blockIdx.x, other = blockIdx.y;
    if (own == other)
        return;
    __shared__ uint64_t s[kSortTile];
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int i = threadIdx.x + q * kSortThreads;
        s[i] = keys[(int64_t)other * kSortTile + i];
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int64_t at = (int64_t)own * kSortTile + threadIdx.x + q * kSortThreads;
        const uint64_t x = keys[at];
        if (x == kPad)
            continue;
        int lo = 0, hi = kSortTile;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (s[mid] < x)
                lo = mid + 1;
            else
                hi = mid;
        }
        if (lo)
            atomicAdd(&rank[at], lo);
    }
}

__global__ void k_sp_scatter(const uint64_t *__restrict__ keys, const int32_t *__restrict__ rank,
                             int64_t npad, uint64_t *__restrict__ sorted)
{
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < npad;
         q += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t x = keys[q];
        if (x != kPad)
            sorted[rank[q]] = x;
    }
}

__device__ __forceinline__ int block_sum_int(int x, int *sh)
{
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        x += __shfl_xor_sync(0xffffffffu, x, o);
    if (lane == 0)
        sh[w] = x;
    __syncthreads();
    int t = 0;
    for (int q = 0; q < (int)(blockDim.x >> 5); ++q)
        t += sh[q];
    __syncthreads();
    return t;
}

// Per tile of the sorted keys: number of run heads and of valid ids.
__global__ void __launch_bounds__(kSortThreads)
k_sp_heads(const uint64_t *__restrict__ sorted, int64_t N, int64_t V, int32_t *__restrict__ tilecnt)
{
    __shared__ int sh[kSortThreads / 32];
    const int64_t p0 = (int64_t)blockIdx.x * kSortTile + (int64_t)threadIdx.x * kKeysPerThread;
    int nh = 0, nv = 0;
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int64_t p = p0 + q;
        if (p < N) {
            const uint64_t id = sorted[p] >> 32;
            if ((int64_t)id < V) {
                ++nv;
                nh += (p == 0 || (sorted[p - 1] >> 32) != id);
            }
        }
    }
    nh = block_sum_int(nh, sh);
    nv = block_sum_int(nv, sh);
    if (threadIdx.x == 0) {
        tilecnt[2 * blockIdx.x] = nh;
        tilecnt[2 * blockIdx.x + 1] = nv;
    }
}

// Distinct ids and their runs.  Thread t of tile b owns sorted positions
// kSortTile b + 4 t .. + 3; an exclusive scan of run heads numbers the ids.
__global__ void __launch_bounds__(kSortThreads)
k_sp_segments(const uint64_t *__restrict__ sorted, int64_t N, int64_t V,
              const int32_t *__restrict__ tilecnt, int32_t *__restrict__ uniq,
              int32_t *__restrict__ segoff, int32_t *__restrict__ perm, int32_t *__restrict__ segidx,
              int32_t *__restrict__ slot, DevScalars *sc)
{
    __shared__ int pre[2];
    __shared__ int wsum[kSortThreads / 32];
    __shared__ int sh[kSortThreads / 32];
    if (threadIdx.x == 0) {
        int a = 0, b = 0;
        for (int t = 0; t < (int)blockIdx.x; ++t) {
            a += tilecnt[2 * t];
            b += tilecnt[2 * t + 1];
        }
        pre[0] = a;
        pre[1] = b;
    }
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int64_t p0 = (int64_t)blockIdx.x * kSortTile + (int64_t)threadIdx.x * kKeysPerThread;
    uint64_t key[kKeysPerThread];
    bool valid[kKeysPerThread], head[kKeysPerThread];
    int nh = 0, nv = 0;
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int64_t p = p0 + q;
        valid[q] = head[q] = false;
        key[q] = kPad;
        if (p < N) {
            key[q] = sorted[p];
            const uint64_t id = key[q] >> 32;
            valid[q] = (int64_t)id < V;
            head[q] = valid[q] && (p == 0 || (sorted[p - 1] >> 32) != id);
        }
        nh += head[q];
        nv += valid[q];
    }
    // exclusive scan of nh over the block
    int x = nh;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o)
            x += y;
    }
    if (lane == 31)
        wsum[w] = x;
    __syncthreads();
    int before = 0;
    for (int q = 0; q < w; ++q)
        before += wsum[q];
    int run = pre[0] + before + x - nh;  // heads before my first position
#pragma unroll
    for (int q = 0; q < kKeysPerThread; ++q) {
        const int64_t p = p0 + q;
        if (head[q]) {
            const int id = (int)(key[q] >> 32);
            uniq[run] = id;
            segoff[run] = (int)p;
            slot[id] = run + 1;
            ++run;
        }
        if (valid[q]) {
            segidx[p] = run - 1;
            perm[p] = (int)(key[q] & 0xffffffffu);
        }
    }
    const int tot_h = block_sum_int(nh, sh);
    const int tot_v = block_sum_int(nv, sh);
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) {
        const int U = pre[0] + tot_h;
        const int nvalid = pre[1] + tot_v;
        sc->n_unique = U;
        sc->n_valid = nvalid;
        segoff[U] = nvalid;
    }
}

// Sum the occurrences of each run.  CTA b works on column slice b % NS
// (kThreads vector columns) of chunks b / NS, b / NS + nw, ...
template <int VEC>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_sp_chunks(const float *__restrict__ rows, const int32_t *__restrict__ perm,
            const int32_t *__restrict__ segidx, const int32_t *__restrict__ segoff,
            const DevScalars *__restrict__ sc, float *__restrict__ S, float *__restrict__ rowpart,
            float *__restrict__ carry, float *__restrict__ colpart, int D, int NS)
{
    using F = typename Vec<VEC>::F;
    constexpr int R = 16;
    constexpr int kWarps = kThreads / 32;
    __shared__ float rp[kChunk][kWarps];
    __shared__ int fin[kChunk];
    const int DV = D / VEC;
    const int sigma = blockIdx.x % NS;
    const int w = blockIdx.x / NS;
    const int nw = gridDim.x / NS;
    const int col = sigma * kThreads + threadIdx.x;
    const bool active = col < DV;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n_valid = sc->n_valid;
    const int nchunks = (n_valid + kChunk - 1) / kChunk;
    float colacc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e)
        colacc[e] = 0.f;

    for (int q = w; w < nw && q < nchunks; q += nw) {
        const int p0 = q * kChunk;
        const int p1 = min(p0 + kChunk, n_valid);
        int nfin = 0;
        int cur = segidx[p0];
        F acc = zero_vec<VEC>();
        auto flush = [&](int u) {
            const bool before = segoff[u] < p0;
            const bool after = segoff[u + 1] > p1;
            if (!before && !after) {
                float ps = 0.f;
                if (active) {
                    *reinterpret_cast<F *>(S + (int64_t)u * D + (int64_t)col * VEC) = acc;
#pragma unroll
                    for (int e = 0; e < VEC; ++e) {
                        const float a = comp(acc, e);
                        colacc[e] += a * a;
                        ps += a * a;
                    }
                }
#pragma unroll
                for (int o = 16; o >= 1; o >>= 1)
                    ps += __shfl_xor_sync(0xffffffffu, ps, o);
                if (lane == 0)
                    rp[nfin][warp] = ps;
                if (threadIdx.x == 0)
                    fin[nfin] = u;
                ++nfin;
            } else if (active) {
                const int which = before ? 0 : 1;  // piece at the chunk's start / end
                *reinterpret_cast<F *>(carry + ((int64_t)2 * q + which) * D + (int64_t)col * VEC) = acc;
            }
        };
        for (int pb = p0; pb < p1; pb += R) {
            F v[R];
            int uu[R];
#pragma unroll
            for (int k = 0; k < R; ++k) {
                const int p = pb + k;
                uu[k] = -1;
                v[k] = zero_vec<VEC>();
                if (p < p1) {
                    uu[k] = segidx[p];
                    if (active)
                        v[k] = load_g<VEC>(rows + (int64_t)perm[p] * D + (int64_t)col * VEC);
                }
            }
#pragma unroll
            for (int k = 0; k < R; ++k) {
                if (uu[k] < 0)
                    break;
                if (uu[k] != cur) {
                    flush(cur);
                    acc = zero_vec<VEC>();
                    cur = uu[k];
                }
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    set_comp(acc, e, comp(acc, e) + comp(v[k], e));
            }
        }
        flush(cur);
        __syncthreads();
        if (threadIdx.x < nfin) {
            float s = 0.f;
            for (int k = 0; k < kWarps; ++k)
                s += rp[threadIdx.x][k];
            rowpart[(int64_t)fin[threadIdx.x] * NS + sigma] = s;
        }
        __syncthreads();
    }
    float *out = colpart + (int64_t)blockIdx.x * D;
    for (int j = threadIdx.x; j < D; j += kThreads)
        out[j] = 0.f;
    __syncthreads();
    if (active && w < nw)
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            out[col * VEC + e] = colacc[e];
}

// Runs cut by chunk boundaries: add their pieces in chunk order.
template <int VEC>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_sp_carry(const int32_t *__restrict__ segoff, const DevScalars *__restrict__ sc,
           const float *__restrict__ carry, float *__restrict__ S, float *__restrict__ rowpart,
           float *__restrict__ colpart, int D, int NS)
{
    using F = typename Vec<VEC>::F;
    constexpr int kWarps = kThreads / 32;
    __shared__ float red[kWarps];
    const int DV = D / VEC;
    const int sigma = blockIdx.x % NS;
    const int w = blockIdx.x / NS;
    const int nw = gridDim.x / NS;
    const int col = sigma * kThreads + threadIdx.x;
    const bool active = col < DV;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int U = sc->n_unique;
    float colacc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e)
        colacc[e] = 0.f;

    for (int u = w; w < nw && u < U; u += nw) {
        const int s0 = segoff[u], s1 = segoff[u + 1];
        const int q0 = s0 / kChunk, q1 = (s1 - 1) / kChunk;
        if (q0 == q1)
            continue;
        float ps = 0.f;
        if (active) {
            const int64_t off = (int64_t)col * VEC;
            // pieces in chunk order: the end piece of chunk q0, then the start
            // pieces of q0+1 .. q1, eight loads in flight at a time
            F acc = load_g<VEC>(carry + ((int64_t)2 * q0 + 1) * D + off);
            constexpr int kB = 8;
            for (int qb = q0 + 1; qb <= q1; qb += kB) {
                F v[kB];
#pragma unroll
                for (int k = 0; k < kB; ++k)
                    v[k] = (qb + k <= q1) ? load_g<VEC>(carry + ((int64_t)2 * (qb + k)) * D + off)
                                          : zero_vec<VEC>();
#pragma unroll
                for (int k = 0; k < kB; ++k)
#pragma unroll
                    for (int e = 0; e < VEC; ++e)
                        set_comp(acc, e, comp(acc, e) + comp(v[k], e));
            }
            *reinterpret_cast<F *>(S + (int64_t)u * D + off) = acc;
#pragma unroll
            for (int e = 0; e < VEC; ++e) {
                const float a = comp(acc, e);
                colacc[e] += a * a;
                ps += a * a;
            }
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            ps += __shfl_xor_sync(0xffffffffu, ps, o);
        if (lane == 0)
            red[warp] = ps;
        __syncthreads();
        if (threadIdx.x == 0) {
            float s = 0.f;
            for (int k = 0; k < kWarps; ++k)
                s += red[k];
            rowpart[(int64_t)u * NS + sigma] = s;
        }
        __syncthreads();
    }
    float *out = colpart + (int64_t)blockIdx.x * D;
    for (int j = threadIdx.x; j < D; j += kThreads)
        out[j] = 0.f;
    __syncthreads();
    if (active && w < nw)
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            out[col * VEC + e] = colacc[e];
}

// Row second moment of all V rows: untouched rows see a zero gradient row.
__global__ void __launch_bounds__(kThreads)
k_sp_vpass(float *__restrict__ r, int32_t *__restrict__ slot, const float *__restrict__ rowpart,
           int NS, int64_t V, int D, double beta2, double one_minus_beta2,
           double *__restrict__ rsum_part)
{
    __shared__ double sh[kThreads / 32];
    double rsum = 0.0;
    for (int64_t i = (int64_t)blockIdx.x * kThreads + threadIdx.x; i < V;
         i += (int64_t)gridDim.x * kThreads) {
        const int s = slot[i];
        double mean_row = 0.0;
        if (s) {
            const int64_t u = s - 1;
            float tot = 0.f;
            for (int k = 0; k < NS; ++k)
                tot += rowpart[u * NS + k];
            mean_row = (double)tot / (double)D;
            slot[i] = 0;
        }
        const float rn = (float)(beta2 * (double)r[i] + one_minus_beta2 * mean_row);
        r[i] = rn;
        rsum += (double)rn;
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
    if ((threadIdx.x & 31) == 0)
        sh[threadIdx.x >> 5] = rsum;
    __syncthreads();
    if (threadIdx.x == 0) {
        double s = 0.0;
        for (int k = 0; k < kThreads / 32; ++k)
            s += sh[k];
        rsum_part[blockIdx.x] = s;
    }
}

// The update of the touched rows: W[uniq[u]] from the summed row S[u].
template <int VEC, int CPT, int R, bool BF16>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_sp_apply(void *__restrict__ W, const float *__restrict__ S, const int32_t *__restrict__ uniq,
           const float *__restrict__ r, const float *__restrict__ c,
           const DevScalars *__restrict__ sc, int D, int tpr, float inv_bc, float eps,
           float lr_signed, int variant)
{
    using F = typename Vec<VEC>::F;
    using WT = typename WRaw<BF16, VEC>::T;
    extern __shared__ float cs[];
    const int DV = D / VEC;
    const int tid = threadIdx.x;
    const int rg = kThreads / tpr;
    const int g = tid / tpr;
    const int l = tid - g * tpr;
    const int U = sc->n_unique;
    const float inv_s = (variant == EMBER_VARIANT_FULL) ? sc->inv_s : 1.f;
    for (int j = tid; j < D; j += kThreads)
        cs[j] = (variant == EMBER_VARIANT_ROW) ? 1.f : sqrtf(c[j] * inv_bc * inv_s);
    __syncthreads();

    const int64_t stride = (int64_t)gridDim.x * rg * R;
    for (int64_t ub = ((int64_t)blockIdx.x * rg + g) * R; ub < U; ub += stride) {
        F gv[R][CPT];
        WT wr[R][CPT];
        int64_t row[R];
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t u = ub + k;
            row[k] = (u < U) ? (int64_t)uniq[u] : -1;
#pragma unroll
            for (int cc = 0; cc < CPT; ++cc) {
                const int col = l + cc * tpr;
                if (u < U && col < DV) {
                    gv[k][cc] = load_g<VEC>(S + u * D + (int64_t)col * VEC);
                    wr[k][cc] = load_w<BF16, VEC>(W, row[k] * D + (int64_t)col * VEC);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < R; ++k) {
            if (row[k] < 0)
                continue;
            const float rs = (variant == EMBER_VARIANT_COL) ? 1.f : sqrtf(__ldg(r + row[k]) * inv_bc);
#pragma unroll
            for (int cc = 0; cc < CPT; ++cc) {
                const int col = l + cc * tpr;
                if (col >= DV)
                    continue;
                float wv[VEC];
                unpack_w(wr[k][cc], wv);
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const float den = fmaf(rs, cs[col * VEC + e], eps);
                    const float u = comp(gv[k][cc], e) / den;
                    wv[e] = fmaf(lr_signed, u, wv[e]);
                }
                store_w<BF16, VEC>(W, row[k] * D + (int64_t)col * VEC, wv);
            }
        }
    }
}

struct Tracer {
    const cudaEvent_t *ev;
    int n, next;
    cudaStream_t s;
    void mark()
    {
        if (ev && next < n)
            cudaEventRecord(ev[next], s);
        ++next;
    }
};

// Sort the ids and number their runs (or record zero runs when N == 0).
void launch_sort_dedup(const SparseArgs &a, Tracer &tr)
{
    unsigned char *ws = a.ws;
    const Layout &L = a.lay;
    DevScalars *sc = reinterpret_cast<DevScalars *>(ws + L.scalars);
    auto *keys = reinterpret_cast<uint64_t *>(ws + L.sp_keys);
    auto *rank = reinterpret_cast<int32_t *>(ws + L.sp_rank);
    auto *sorted = reinterpret_cast<uint64_t *>(ws + L.sp_sorted);
    auto *tilecnt = reinterpret_cast<int32_t *>(ws + L.sp_tilecnt);
    auto *perm = reinterpret_cast<int32_t *>(ws + L.sp_perm);
    auto *segidx = reinterpret_cast<int32_t *>(ws + L.sp_segidx);
    auto *uniq = reinterpret_cast<int32_t *>(ws + L.sp_uniq);
    auto *segoff = reinterpret_cast<int32_t *>(ws + L.sp_segoff);
    auto *slot = reinterpret_cast<int32_t *>(ws + L.sp_slot);
    if (a.N > 0) {
        const int T = (int)((a.N + kSortTile - 1) / kSortTile);
        const int64_t npad = (int64_t)T * kSortTile;
        if (a.ids64)
            k_sp_tile_sort<int64_t><<<T, kSortThreads, 0, a.stream>>>(
                static_cast<const int64_t *>(a.ids), a.N, a.V, keys, rank, sc);
        else
            k_sp_tile_sort<int32_t><<<T, kSortThreads, 0, a.stream>>>(
                static_cast<const int32_t *>(a.ids), a.N, a.V, keys, rank, sc);
        tr.mark();
        if (T > 1) {
            k_sp_rank<<<dim3(T, T), kSortThreads, 0, a.stream>>>(keys, rank);
            tr.mark();
        }
        const int nsc = (int)((npad + kThreads - 1) / kThreads);
        k_sp_scatter<<<nsc, kThreads, 0, a.stream>>>(keys, rank, npad, sorted);
        tr.mark();
        k_sp_heads<<<T, kSortThreads, 0, a.stream>>>(sorted, a.N, a.V, tilecnt);
        tr.mark();
        k_sp_segments<<<T, kSortThreads, 0, a.stream>>>(sorted, a.N, a.V, tilecnt, uniq, segoff, perm,
                                                        segidx, slot, sc);
        tr.mark();
    } else {
        // no ids: zero distinct ids and zero valid occurrences
        cudaMemsetAsync(&sc->n_unique, 0, 2 * sizeof(int32_t), a.stream);
    }
}

// Distinct ids, their counts and U to caller buffers.
__global__ void k_sp_export(const int32_t *__restrict__ uniq, const int32_t *__restrict__ segoff,
                            const DevScalars *__restrict__ sc, int64_t N, int32_t *__restrict__ uniq_out,
                            int32_t *__restrict__ counts_out, int32_t *__restrict__ n_unique_out)
{
    const int U = sc->n_unique;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < N;
         u += (int64_t)gridDim.x * blockDim.x) {
        if (u < U) {
            uniq_out[u] = uniq[u];
            counts_out[u] = segoff[u + 1] - segoff[u];
        }
    }
    if (blockIdx.x == 0 && threadIdx.x == 0)
        *n_unique_out = U;
}

template <int VEC, int CPT>
cudaError_t launch_sparse_t(const SparseArgs &a)
{
    constexpr int R = (8 / CPT) < 1 ? 1 : (8 / CPT);
    unsigned char *ws = a.ws;
    const Layout &L = a.lay;
    DevScalars *sc = reinterpret_cast<DevScalars *>(ws + L.scalars);
    auto *perm = reinterpret_cast<int32_t *>(ws + L.sp_perm);
    auto *segidx = reinterpret_cast<int32_t *>(ws + L.sp_segidx);
    auto *uniq = reinterpret_cast<int32_t *>(ws + L.sp_uniq);
    auto *segoff = reinterpret_cast<int32_t *>(ws + L.sp_segoff);
    auto *slot = reinterpret_cast<int32_t *>(ws + L.sp_slot);
    auto *rowpart = reinterpret_cast<float *>(ws + L.sp_rowpart);
    auto *carry = reinterpret_cast<float *>(ws + L.sp_carry);
    auto *S = reinterpret_cast<float *>(ws + L.sp_rows);
    auto *colpart = reinterpret_cast<float *>(ws + L.colpart);
    auto *rsum_part = reinterpret_cast<double *>(ws + L.rsum_part);
    auto *csum_part = reinterpret_cast<double *>(ws + L.csum_part);
    const int D = (int)a.D;
    const int DV = D / VEC;
    const int NS = (DV + kThreads - 1) / kThreads;
    Tracer tr{a.trace, a.n_trace, 0, a.stream};

    tr.mark();
    launch_sort_dedup(a, tr);
    const int G = kGridCtas;
    k_sp_chunks<VEC><<<G, kThreads, 0, a.stream>>>(a.rows, perm, segidx, segoff, sc, S, rowpart, carry,
                                                   colpart, D, NS);
    tr.mark();
    k_sp_carry<VEC><<<G, kThreads, 0, a.stream>>>(segoff, sc, carry, S, rowpart, colpart + (int64_t)G * D,
                                                  D, NS);
    tr.mark();
    const int64_t vb = (a.V + kThreads - 1) / kThreads;
    const int GV = (int)(vb < kGridCtas ? vb : kGridCtas);
    k_sp_vpass<<<GV, kThreads, 0, a.stream>>>(a.r, slot, rowpart, NS, a.V, D, a.beta2, a.one_minus_beta2,
                                              rsum_part);
    tr.mark();
    launch_state(colpart, 2 * G, rsum_part, GV, a.c, csum_part, sc, a.V, D, a.beta2, a.one_minus_beta2,
                 a.inv_bc, a.stream);
    tr.mark();
    const size_t cs_bytes = (size_t)D * sizeof(float);
    if (a.wbf16)
        k_sp_apply<VEC, CPT, R, true><<<G, kThreads, cs_bytes, a.stream>>>(
            a.W, S, uniq, a.r, a.c, sc, D, a.map.tpr, (float)a.inv_bc, a.eps, a.lr_signed, a.variant);
    else
        k_sp_apply<VEC, CPT, R, false><<<G, kThreads, cs_bytes, a.stream>>>(
            a.W, S, uniq, a.r, a.c, sc, D, a.map.tpr, (float)a.inv_bc, a.eps, a.lr_signed, a.variant);
    tr.mark();
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_sparse_step(const SparseArgs &a)
{
    if (a.map.vec == 4) {
        switch (a.map.cpt) {
        case 1: return launch_sparse_t<4, 1>(a);
        case 2: return launch_sparse_t<4, 2>(a);
        case 4: return launch_sparse_t<4, 4>(a);
        case 8: return launch_sparse_t<4, 8>(a);
        }
    } else {
        switch (a.map.cpt) {
        case 1: return launch_sparse_t<1, 1>(a);
        case 2: return launch_sparse_t<1, 2>(a);
        case 4: return launch_sparse_t<1, 4>(a);
        case 8: return launch_sparse_t<1, 8>(a);
        }
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_sparse_unique(const SparseArgs &a, int32_t *uniq_out, int32_t *counts_out,
                                 int32_t *n_unique_out)
{
    Tracer tr{nullptr, 0, 0, a.stream};
    launch_sort_dedup(a, tr);
    const DevScalars *sc = reinterpret_cast<const DevScalars *>(a.ws + a.lay.scalars);
    const int32_t *uniq = reinterpret_cast<const int32_t *>(a.ws + a.lay.sp_uniq);
    const int32_t *segoff = reinterpret_cast<const int32_t *>(a.ws + a.lay.sp_segoff);
    int64_t nb = (a.N + kThreads - 1) / kThreads;
    if (nb < 1)
        nb = 1;
    if (nb > 4 * kGridCtas)
        nb = 4 * kGridCtas;
    k_sp_export<<<(int)nb, kThreads, 0, a.stream>>>(uniq, segoff, sc, a.N, uniq_out, counts_out,
                                                     n_unique_out);
    // the touched-row map must be all-zero again before the next step
    int32_t *slot = reinterpret_cast<int32_t *>(a.ws + a.lay.sp_slot);
    cudaMemsetAsync(slot, 0, sizeof(int32_t) * (size_t)a.V, a.stream);
    return cudaGetLastError();
}

}  // namespace ember
