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
//             the rank is exact and the order deterministic).  The same
//             searches find the run heads: a key heads its id's run unless
//             some tile holds a smaller key of the same id, which is then the
//             key just below it in that tile.  The scatter counts the heads
//             and the valid ids of every tile of sorted positions.
//   dedup     k_sp_segments: the distinct ids (ascending), where each id's
//             run starts, and a V-entry map from a touched row to its
//             distinct-id index.
//   segsum    k_sp_segsum, k_sp_carry: the summed gradient row of every
//             distinct id, adding its occurrences in increasing occurrence
//             order (compensated fp32 sums); per (id, column slice) sums of
//             g^2; per-CTA column sums
//             of g^2.  Each worker owns a contiguous, equal share of the
//             sorted occurrences, so the work is even however skewed the id
//             counts are (a Zipf head id can own thousands of occurrences);
//             a run that crosses worker boundaries leaves one piece per
//             worker, which k_sp_carry adds in worker order.
//   state     the dense step's column/normaliser pass, whose launch also runs
//             the row pass: r for all V rows, the sums of new r per CTA, and
//             the touched-row map cleared for the next step.
//   apply     k_sp_apply: the update of the touched rows only (once per
//             column panel for tables wider than a CTA holds).
//
// Every kernel after the first is launched with programmatic dependent
// launch and waits (griddepcontrol.wait) before it reads earlier results.
#include <cuda_runtime.h>
#include <stdint.h>

#include "ember_device.cuh"
#include "ember_internal.h"

namespace ember {
namespace {

using namespace dev;

constexpr uint64_t kPad = ~0ull;
// Bit of a key's rank word set when the key is not the head of its id's run
// (ranks stay below 2^30: N <= INT32_MAX / 2).
constexpr int kNotHead = 1 << 30;
constexpr int kKeysPerThread = kSortTile / kSortThreads;

// keys a <= b afterwards when `up`, a >= b otherwise
__device__ __forceinline__ void cmp_swap(uint64_t &a, uint64_t &b, bool up)
{
    if ((a > b) == up) {
        const uint64_t x = a;
        a = b;
        b = x;
    }
}

__device__ __forceinline__ uint64_t shfl_xor_u64(uint64_t x, int m)
{
    const uint32_t lo = __shfl_xor_sync(0xffffffffu, (uint32_t)x, m);
    const uint32_t hi = __shfl_xor_sync(0xffffffffu, (uint32_t)(x >> 32), m);
    return ((uint64_t)hi << 32) | lo;
}

// Bitonic sort of one tile of kSortTile keys, thread t holding keys
// 4t .. 4t + 3.  For the compare-exchange of keys i and i ^ j at merge size
// k, both holders keep min or max by the same rule: the lower index of the
// pair keeps the min when the block (i & k) sorts ascending.  Partners at
// distance 1 or 2 are in the same thread, distance 4 .. 64 in the same warp
// (shuffles), and only distances 128 .. 512 go through shared memory.
template <typename IdT>
__global__ void __launch_bounds__(kSortThreads)
k_sp_tile_sort(const IdT *__restrict__ ids, int64_t N, int64_t V, uint64_t *__restrict__ keys,
               int32_t *__restrict__ rank, int32_t *__restrict__ tilecnt, DevScalars *sc)
{
    static_assert(kSortTile == 4 * kSortThreads, "four keys per thread");
    __shared__ uint64_t s[kSortTile];
    const int64_t base = (int64_t)blockIdx.x * kSortTile;
    const int t = threadIdx.x;
    grid_dep_wait();  // first kernel of a step: returns at once
    grid_dep_launch();
    bool bad = false;
    uint64_t key[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int64_t k = base + 4 * t + q;
        key[q] = kPad;
        if (k < N) {
            int64_t id = (int64_t)ids[k];
            if (id < 0 || id >= V) {  // skipped: sorts after every valid id
                bad = true;
                id = V;
            }
            key[q] = ((uint64_t)id << 32) | (uint64_t)k;
        }
    }
    if (bad)
        atomicOr(&sc->flags, kFlagIdRange);

    for (int k = 2; k <= kSortTile; k <<= 1) {
        for (int j = k >> 1; j > 0; j >>= 1) {
            if (j >= 128) {  // partner in another warp
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    s[4 * t + q] = key[q];
                __syncthreads();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int i = 4 * t + q;
                    const uint64_t o = s[i ^ j];
                    const bool keep_min = ((i & j) == 0) == ((i & k) == 0);
                    key[q] = keep_min ? (key[q] < o ? key[q] : o) : (key[q] > o ? key[q] : o);
                }
                __syncthreads();
            } else if (j >= 4) {  // partner in this warp
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int i = 4 * t + q;
                    const uint64_t o = shfl_xor_u64(key[q], j >> 2);
                    const bool keep_min = ((i & j) == 0) == ((i & k) == 0);
                    key[q] = keep_min ? (key[q] < o ? key[q] : o) : (key[q] > o ? key[q] : o);
                }
            } else {  // partner in this thread: pairs (0,1),(2,3) or (0,2),(1,3)
                const bool up = ((4 * t) & k) == 0;  // for k >= 4 the same for all four keys
                if (j == 1) {
                    cmp_swap(key[0], key[1], k == 2 ? (((4 * t) & 2) == 0) : up);
                    cmp_swap(key[2], key[3], k == 2 ? (((4 * t + 2) & 2) == 0) : up);
                } else {
                    cmp_swap(key[0], key[2], up);
                    cmp_swap(key[1], key[3], up);
                }
            }
        }
    }
    // rank within the tile, and kNotHead where the key before it in the
    // tile has the same id; the scatter's counts of this tile start at zero
#pragma unroll
    for (int q = 0; q < 4; ++q)
        s[4 * t + q] = key[q];
    if (t < 2)
        tilecnt[2 * blockIdx.x + t] = 0;
    __syncthreads();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int i = 4 * t + q;
        const bool same = i > 0 && (s[i - 1] >> 32) == (key[q] >> 32);
        keys[base + i] = key[q];
        rank[base + i] = i | (same ? kNotHead : 0);
    }
}

// CTA (own, other): add to each key of tile `own` the number of keys of tile
// `other` below it.  Keys are unique, so the ranks form a permutation.  A key
// whose lower bound in `other` follows a key of the same id is not the head
// of its id's run.
__global__ void __launch_bounds__(kSortThreads)
k_sp_rank(const uint64_t *__restrict__ keys, int32_t *__restrict__ rank)
{
    const int own = blockIdx.x, other = blockIdx.y;
    grid_dep_wait();  // tile-sorted keys
    grid_dep_launch();
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
        if (lo) {
            atomicAdd(&rank[at], lo);
            if ((s[lo - 1] >> 32) == (x >> 32))
                atomicOr(&rank[at], kNotHead);
        }
    }
}

// Keys to their sorted positions, and per tile of sorted positions the
// number of run heads and of valid ids (counted per warp, then one integer
// atomic per tile a warp touches).  npad is a multiple of the warp size, so
// every lane of a warp takes the same iterations.
__global__ void k_sp_scatter(const uint64_t *__restrict__ keys, const int32_t *__restrict__ rank,
                             int64_t npad, int64_t V, uint64_t *__restrict__ sorted, int32_t *__restrict__ tilecnt)
{
    grid_dep_wait();  // ranks
    grid_dep_launch();
    const int lane = threadIdx.x & 31;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < npad;
         q += (int64_t)gridDim.x * blockDim.x) {
        const uint64_t x = keys[q];
        const int rk = rank[q];
        const bool real = x != kPad;
        const int pos = rk & ~kNotHead;
        if (real)
            sorted[pos] = x;
        const bool valid = real && (int64_t)(x >> 32) < V;
        const bool head = valid && !(rk & kNotHead);
        const int tile = real ? pos / kSortTile : -1;
        const unsigned peers = __match_any_sync(0xffffffffu, tile);
        const int nh = __popc(__ballot_sync(0xffffffffu, head) & peers);
        const int nv = __popc(__ballot_sync(0xffffffffu, valid) & peers);
        if (real && lane == __ffs(peers) - 1) {
            if (nh)
                atomicAdd(&tilecnt[2 * tile], nh);
            if (nv)
                atomicAdd(&tilecnt[2 * tile + 1], nv);
        }
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

// Distinct ids and their runs.  Thread t of tile b owns sorted positions
// kSortTile b + 4 t .. + 3; an exclusive scan of run heads numbers the ids.
__global__ void __launch_bounds__(kSortThreads)
k_sp_segments(const uint64_t *__restrict__ sorted, int64_t N, int64_t V,
              const int32_t *__restrict__ tilecnt, int32_t *__restrict__ uniq,
              int32_t *__restrict__ segoff, int32_t *__restrict__ perm, int32_t *__restrict__ segidx,
              int32_t *__restrict__ slot, int32_t *__restrict__ single, DevScalars *sc)
{
    __shared__ int pre[2];
    __shared__ int wsum[kSortThreads / 32];
    __shared__ int sh[kSortThreads / 32];
    grid_dep_wait();  // per-tile counts
    grid_dep_launch();
    {
        // run heads and valid ids of the tiles before this one: a thread per
        // tile, then the block's sums (one trip to L2, not one per tile)
        int a = 0, b = 0;
        for (int t = threadIdx.x; t < (int)blockIdx.x; t += kSortThreads) {
            a += tilecnt[2 * t];
            b += tilecnt[2 * t + 1];
        }
        a = block_sum_int(a, sh);
        b = block_sum_int(b, sh);
        if (threadIdx.x == 0) {
            pre[0] = a;
            pre[1] = b;
        }
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
            // an id seen once: its summed row is that occurrence's row
            const bool once = p + 1 >= N || (sorted[p + 1] >> 32) != (uint64_t)id;
            single[run] = once ? (int)(key[q] & 0xffffffffu) : -1;
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

// Workers split the sorted occurrences into contiguous ranges of equal
// cost, cost(p) = p + segidx[p]: one unit per occurrence row read and one
// per summed row written (runs are numbered in order, so the cost rises by
// one or two per position).  Worker w owns [first(w), first(w + 1)), where
// first(w) is the smallest position whose cost reaches T(w) = w C / nw and
// C = n_valid + U.
__device__ __forceinline__ int64_t cost_target(int w, int nw, int64_t C)
{
    return ((int64_t)w * C) / nw;
}

// Smallest p in [0, n_valid] with p + segidx[p] >= T (position n_valid
// counts as reaching every target).  Block-wide 256-way search: each round
// probes kThreads evenly spaced positions and keeps the one interval that
// holds the answer.
__device__ int block_first_reaching(const int32_t *__restrict__ segidx, int n_valid, int64_t T)
{
    __shared__ int lo_hi[2];
    int lo = 0, hi = n_valid;  // answer in [lo, hi]
    while (lo < hi) {
        const int64_t len = hi - lo;
        const int t = threadIdx.x;
        const int p = lo + (int)((len * t) / kThreads);
        const bool reached = (int64_t)p + segidx[p] >= T;  // p < hi <= n_valid
        const int below = __syncthreads_count(!reached);  // probes before the answer
        if (t == 0) {
            int nlo = lo, nhi = hi;
            if (below > 0)
                nlo = lo + (int)((len * (below - 1)) / kThreads) + 1;
            if (below < kThreads)
                nhi = lo + (int)((len * below) / kThreads);
            lo_hi[0] = nlo;
            lo_hi[1] = nhi;
        }
        __syncthreads();
        lo = lo_hi[0];
        hi = lo_hi[1];
        __syncthreads();
    }
    return lo;
}

// Worker whose range holds sorted position p of run u.
__device__ __forceinline__ int worker_of(int p, int u, int nw, int64_t C)
{
    const int64_t c = (int64_t)p + u;
    int w = (int)((c * nw) / C);
    while (w + 1 < nw && cost_target(w + 1, nw, C) <= c)
        ++w;
    while (w > 0 && cost_target(w, nw, C) > c)
        --w;
    return w;
}

// Sum the occurrences of each run.  CTA b works on column slice b % NS
// (kThreads vector columns) of the sorted positions of worker b / NS, adding
// each run's rows in increasing occurrence order with a running sum that
// crosses the worker's whole range.  A run that starts before the range or
// ends after it leaves its piece in the carry buffer (slot 0: the range's
// first run, slot 1: its last run); k_sp_carry adds the pieces in worker
// order.  Completed runs are written to S with their sum of g^2 per slice.
template <int VEC>
__global__ void __launch_bounds__(kThreads, kSparseCtasPerSm)
k_sp_segsum(const float *__restrict__ rows, const int32_t *__restrict__ perm,
            const int32_t *__restrict__ segidx, const DevScalars *__restrict__ sc,
            float *__restrict__ S, float *__restrict__ rowpart, float *__restrict__ carry,
            float *__restrict__ colpart, int32_t *__restrict__ bounds, int D, int NS,
            float *__restrict__ r, const int32_t *__restrict__ slot, int64_t V, EmaPair ema,
            float *__restrict__ rsum_part)
{
    using F = typename Vec<VEC>::F;
    constexpr int R = 8;  // rows in flight per thread
    constexpr int kWarps = kThreads / 32;
    constexpr int kFin = 128;  // completed runs buffered before their g^2 sums are written
    constexpr int kIdxWindow = 1024;
    __shared__ float rp[kFin][kWarps];
    __shared__ int fin[kFin];
    __shared__ int sperm[kIdxWindow];
    __shared__ int sseg[kIdxWindow];
    const int DV = D / VEC;
    const int sigma = blockIdx.x % NS;
    const int w = blockIdx.x / NS;
    const int nw = gridDim.x / NS;
    const int col = sigma * kThreads + threadIdx.x;
    const bool active = col < DV;
    // threads past the row's end load its last vector (and discard the sums)
    const float *src = rows + (int64_t)(active ? col : DV - 1) * VEC;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    grid_dep_wait();  // runs and occurrence order from the dedup kernels
    grid_dep_launch();
    const int n_valid = sc->n_valid;
    float colacc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e)
        colacc[e] = 0.f;
    // the occurrence rows stream through once: evict them first, so that
    // the summed rows written here stay in L2 for the update that reads them
    const uint64_t pol_rows = policy_evict_first();
    const uint64_t pol_sums = policy_evict_last();

    const bool worker = w < nw && n_valid > 0;
    int p0 = 0, p1 = 0;
    if (worker) {
        const int64_t C = (int64_t)n_valid + sc->n_unique;
        p0 = block_first_reaching(segidx, n_valid, cost_target(w, nw, C));
        p1 = (w + 1 == nw) ? n_valid : block_first_reaching(segidx, n_valid, cost_target(w + 1, nw, C));
        if (sigma == 0 && threadIdx.x == 0) {
            bounds[w] = p0;
            if (w + 1 == nw)
                bounds[nw] = n_valid;
        }
        if (p0 == p1 && active) {
            // an empty range holds no piece of the run that spans it
            const F z = zero_vec<VEC>();
            *reinterpret_cast<F *>(carry + ((int64_t)2 * w) * D + (int64_t)col * VEC) = z;
            *reinterpret_cast<F *>(carry + ((int64_t)2 * w + 1) * D + (int64_t)col * VEC) = z;
        }
    }
    int nfin = 0;
    auto drain = [&]() {  // uniform: all threads call it together
        __syncthreads();
        if (threadIdx.x < nfin) {
            float t = 0.f;
            for (int k = 0; k < kWarps; ++k)
                t += rp[threadIdx.x][k];
            rowpart[(int64_t)fin[threadIdx.x] * NS + sigma] = t;
        }
        __syncthreads();
        nfin = 0;
    };
    if (p0 < p1) {
        // Only the range's first run can have started before it and only
        // its last run can continue after it; decide both once, here.
        const int u_first = segidx[p0];
        const int u_last = segidx[p1 - 1];
        const bool first_cut = p0 > 0 && segidx[p0 - 1] == u_first;
        const bool last_cut = p1 < n_valid && segidx[p1] == u_last;
        int cur = u_first;
        int len = 0;  // occurrences of `cur` seen in this range
        // Per-id sums in occurrence order, compensated (Kahan): `acc` is the
        // running sum, `cmp` the part of it that rounding added, so the sum
        // stays within about an ulp even over thousands of duplicates.
        F acc = zero_vec<VEC>();
        F cmp = zero_vec<VEC>();
        auto flush = [&](int u) {
#pragma unroll
            for (int e = 0; e < VEC; ++e)
                set_comp(acc, e, comp(acc, e) - comp(cmp, e));
            const bool before = first_cut && u == u_first;
            const bool after = last_cut && u == u_last;
            if (!before && !after) {
                float ps = 0.f;
                if (active) {
                    // an id seen once needs no summed row: the apply reads its occurrence row
                    if (len > 1)
                        store_g_hint<VEC>(S + (int64_t)u * D + (int64_t)col * VEC, acc, pol_sums);
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
                if (nfin == kFin)
                    drain();
            } else if (active) {
                const int which = before ? 0 : 1;
                *reinterpret_cast<F *>(carry + ((int64_t)2 * w + which) * D + (int64_t)col * VEC) = acc;
            }
        };
        // The range's occurrence and run indices go to shared memory a
        // window at a time, so each batch of rows costs one trip to HBM.
        for (int wb = p0; wb < p1; wb += kIdxWindow) {
            const int we = (wb + kIdxWindow < p1) ? wb + kIdxWindow : p1;
            __syncthreads();  // the previous window's indices are no longer read
            for (int p = wb + threadIdx.x; p < we; p += kThreads) {
                sperm[p - wb] = perm[p];
                sseg[p - wb] = segidx[p];
            }
            __syncthreads();
            for (int pb = wb; pb < we; pb += R) {
                // R rows in flight; only the window's last batch is partial
                const int nb = (we - pb < R) ? we - pb : R;
                const int *bp = sperm + (pb - wb);
                F v[R];
                if (nb == R) {
#pragma unroll
                    for (int k = 0; k < R; ++k)
                        v[k] = load_g_hint<VEC>(src + (int64_t)bp[k] * D, pol_rows);
                } else {
#pragma unroll
                    for (int k = 0; k < R; ++k)
                        v[k] = (k < nb) ? load_g_hint<VEC>(src + (int64_t)bp[k] * D, pol_rows) : zero_vec<VEC>();
                }
#pragma unroll
                for (int k = 0; k < R; ++k) {
                    if (k >= nb)
                        break;
                    const int u = sseg[pb - wb + k];
                    if (u != cur) {
                        flush(cur);
                        acc = zero_vec<VEC>();
                        cmp = zero_vec<VEC>();
                        cur = u;
                        len = 0;
                    }
                    ++len;
#pragma unroll
                    for (int e = 0; e < VEC; ++e) {
                        const float y = comp(v[k], e) - comp(cmp, e);
                        const float t = comp(acc, e) + y;
                        set_comp(cmp, e, (t - comp(acc, e)) - y);
                        set_comp(acc, e, t);
                    }
                }
            }
        }
        flush(cur);
    }
    if (nfin > 0)
        drain();
    float *out = colpart + (int64_t)blockIdx.x * D;
    for (int j = threadIdx.x; j < D; j += kThreads)
        out[j] = 0.f;
    __syncthreads();
    if (active && worker)
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            out[col * VEC + e] = colacc[e];

    // The rows outside the batch: r_i <- beta2 r_i (their g is 0), this CTA's
    // share of the table, kRowBatch rows per thread at a time with their map
    // entries loaded together; the touched rows are left to the state pass.
    // The CTA's fp32 sum of the decayed r goes to rsum_part[blockIdx.x].
    {
        const int64_t i0 = (int64_t)blockIdx.x * V / gridDim.x, i1 = (int64_t)(blockIdx.x + 1) * V / gridDim.x;
        float rsum = 0.f;
        for (int64_t ib = i0 + threadIdx.x; ib < i1; ib += (int64_t)kThreads * kRowBatch) {
            int sl[kRowBatch];
            float rr[kRowBatch];
#pragma unroll
            for (int k = 0; k < kRowBatch; ++k) {
                const int64_t i = ib + (int64_t)k * kThreads;
                sl[k] = (i < i1) ? slot[i] : 1;
                rr[k] = (i < i1) ? r[i] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < kRowBatch; ++k) {
                if (sl[k] != 0)
                    continue;
                const float rn = ema_pair(ema, rr[k], 0.f);
                r[ib + (int64_t)k * kThreads] = rn;
                rsum += rn;
            }
        }
        __shared__ float rsh[kThreads / 32];
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
        if (lane == 0)
            rsh[warp] = rsum;
        __syncthreads();
        if (threadIdx.x == 0) {
            float t = 0.f;
            for (int q = 0; q < kThreads / 32; ++q)
                t += rsh[q];
            rsum_part[blockIdx.x] = t;
        }
    }
}

// Runs cut by worker boundaries.  CTA b handles boundary bd = b / NS + 1
// (position first(bd)) on slice b % NS: if the run holding that position
// started inside the previous worker's range, this CTA adds the run's
// pieces -- the previous worker's last piece, then the first pieces of the
// following workers up to the one holding the run's end -- in worker order.
template <int VEC>
__global__ void __launch_bounds__(kThreads, kSparseCtasPerSm)
k_sp_carry(const int32_t *__restrict__ segidx, const int32_t *__restrict__ segoff,
           const int32_t *__restrict__ bounds, const DevScalars *__restrict__ sc,
           const float *__restrict__ carry, float *__restrict__ S, float *__restrict__ rowpart,
           float *__restrict__ colpart, int D, int NS, int nw)
{
    using F = typename Vec<VEC>::F;
    constexpr int kWarps = kThreads / 32;
    __shared__ float red[kWarps];
    const int DV = D / VEC;
    const int sigma = blockIdx.x % NS;
    const int bd = blockIdx.x / NS + 1;
    const int col = sigma * kThreads + threadIdx.x;
    const bool active = col < DV;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    grid_dep_wait();  // carry pieces from k_sp_segsum
    grid_dep_launch();
    const int n_valid = sc->n_valid;
    float colacc[VEC];
#pragma unroll
    for (int e = 0; e < VEC; ++e)
        colacc[e] = 0.f;
    bool mine = false;
    int u = 0, w0 = 0, w1 = 0;
    if (bd < nw && n_valid > 0) {
        const int p = bounds[bd];
        if (p < n_valid) {
            u = segidx[p];
            const int s0 = segoff[u], s1 = segoff[u + 1];
            w0 = bd - 1;
            mine = s0 < p && s0 >= bounds[w0];
            const int64_t C = (int64_t)n_valid + sc->n_unique;
            w1 = worker_of(s1 - 1, u, nw, C);
        }
    }
    if (mine) {
        float ps = 0.f;
        if (active) {
            const int64_t off = (int64_t)col * VEC;
            F acc = load_g<VEC>(carry + ((int64_t)2 * w0 + 1) * D + off);
            F cmp = zero_vec<VEC>();  // compensated (Kahan) sum, as in k_sp_segsum
            constexpr int kB = 8;
            for (int qb = w0 + 1; qb <= w1; qb += kB) {
                F v[kB];
#pragma unroll
                for (int k = 0; k < kB; ++k) {
                    // workers with an empty range wrote zero pieces
                    const int q = qb + k;
                    v[k] = (q <= w1) ? load_g<VEC>(carry + ((int64_t)2 * q) * D + off) : zero_vec<VEC>();
                }
#pragma unroll
                for (int k = 0; k < kB; ++k)
#pragma unroll
                    for (int e = 0; e < VEC; ++e) {
                        const float y = comp(v[k], e) - comp(cmp, e);
                        const float t = comp(acc, e) + y;
                        set_comp(cmp, e, (t - comp(acc, e)) - y);
                        set_comp(acc, e, t);
                    }
            }
#pragma unroll
            for (int e = 0; e < VEC; ++e)
                set_comp(acc, e, comp(acc, e) - comp(cmp, e));
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
            float t = 0.f;
            for (int k = 0; k < kWarps; ++k)
                t += red[k];
            rowpart[(int64_t)u * NS + sigma] = t;
        }
    }
    // CTA b of this kernel and CTA b of k_sp_segsum share worker bd - 1 and
    // slice sigma: add this run's column sums to that CTA's partial row
    // (its value plus this one, in that order)
    if (active && mine) {
        float *out = colpart + (int64_t)blockIdx.x * D;
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            out[col * VEC + e] += colacc[e];
    }
}

// The update of the touched rows: W[uniq[u]] from the summed row S[u].
// Three CTAs per SM (two for the widest rows): each CTA has only a few rows,
// so more of them are kept in flight at once.  D columns from row stride ld
// (a column panel of a wider table: W, S, rows and c point at its first
// column).
constexpr int apply_ctas_per_sm(int cpt) { return cpt >= 8 ? 2 : cpt >= 4 ? 4 : 3; }
template <int VEC, int CPT, int R, bool BF16>
__global__ void __launch_bounds__(kThreads, apply_ctas_per_sm(CPT))
k_sp_apply(void *__restrict__ W, const float *__restrict__ S, const float *__restrict__ rows,
           const int32_t *__restrict__ uniq, const int32_t *__restrict__ single,
           const float *__restrict__ r, const float *__restrict__ c,
           const DevScalars *__restrict__ sc, int D, int ld, int tpr, float inv_bc, float eps,
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
    grid_dep_wait();  // s, c, r and the summed rows
    grid_dep_launch();
    const int U = sc->n_unique;
    const float inv_s = (variant == EMBER_VARIANT_FULL) ? sc->inv_s : 1.f;
    for (int j = tid; j < D; j += kThreads)
        cs[j] = (variant == EMBER_VARIANT_ROW) ? 1.f : sqrtf(c[j] * inv_bc * inv_s);
    __syncthreads();

    // the summed rows, the W rows and the written W are touched for the last
    // time in the step
    const uint64_t pol = policy_evict_first();
    const int64_t stride = (int64_t)gridDim.x * rg * R;
    const int64_t ub0 = ((int64_t)blockIdx.x * rg + g) * R;
    // row ids (and, for ids seen once, the occurrence row) of the next
    // iteration are loaded while this one's rows are in flight
    int64_t next[R];
    int nsingle[R];
#pragma unroll
    for (int k = 0; k < R; ++k) {
        next[k] = (ub0 + k < U) ? (int64_t)uniq[ub0 + k] : -1;
        nsingle[k] = (ub0 + k < U) ? single[ub0 + k] : -1;
    }
    for (int64_t ub = ub0; ub < U; ub += stride) {
        F gv[R][CPT];
        WT wr[R][CPT];
        int64_t row[R];
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t u = ub + k;
            row[k] = next[k];
            const float *src = (nsingle[k] >= 0) ? rows + (int64_t)nsingle[k] * ld : S + u * ld;
#pragma unroll
            for (int cc = 0; cc < CPT; ++cc) {
                const int col = l + cc * tpr;
                if (row[k] >= 0 && col < DV) {
                    gv[k][cc] = load_g_hint<VEC>(src + (int64_t)col * VEC, pol);
                    wr[k][cc] = load_w_hint<BF16, VEC>(W, row[k] * ld + (int64_t)col * VEC, pol);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t un = ub + stride + k;
            next[k] = (un < U) ? (int64_t)uniq[un] : -1;
            nsingle[k] = (un < U) ? single[un] : -1;
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
                    const float u = update_ratio(comp(gv[k][cc], e), den);
                    wv[e] = fmaf(lr_signed, u, wv[e]);
                }
                store_w_hint<BF16, VEC>(W, row[k] * ld + (int64_t)col * VEC, wv, pol);
            }
        }
    }
}

struct Tracer {
    const cudaEvent_t *ev;
    int n, next;
    cudaStream_t s;
    bool launched = false;  // a kernel of this step is already on the stream
    void mark()
    {
        if (ev && next < n)
            cudaEventRecord(ev[next], s);
        ++next;
    }
    // programmatic dependent launch for every kernel after the first,
    // unless events are recorded between the kernels
    bool pdl()
    {
        const bool p = launched && ev == nullptr;
        launched = true;
        return p;
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
    auto *single = reinterpret_cast<int32_t *>(ws + L.sp_single);
    if (a.N > 0) {
        const int T = (int)((a.N + kSortTile - 1) / kSortTile);
        const int64_t npad = (int64_t)T * kSortTile;
        if (a.ids64)
            launch_k(k_sp_tile_sort<int64_t>, dim3(T), dim3(kSortThreads), 0, a.stream, tr.pdl(),
                     static_cast<const int64_t *>(a.ids), a.N, a.V, keys, rank, tilecnt, sc);
        else
            launch_k(k_sp_tile_sort<int32_t>, dim3(T), dim3(kSortThreads), 0, a.stream, tr.pdl(),
                     static_cast<const int32_t *>(a.ids), a.N, a.V, keys, rank, tilecnt, sc);
        tr.mark();
        if (T > 1) {
            launch_k(k_sp_rank, dim3(T, T), dim3(kSortThreads), 0, a.stream, tr.pdl(), keys, rank);
            tr.mark();
        }
        const int nsc = (int)((npad + kThreads - 1) / kThreads);
        launch_k(k_sp_scatter, dim3(nsc), dim3(kThreads), 0, a.stream, tr.pdl(), keys, rank, npad, a.V, sorted,
                 tilecnt);
        tr.mark();
        launch_k(k_sp_segments, dim3(T), dim3(kSortThreads), 0, a.stream, tr.pdl(), sorted, a.N, a.V,
                 tilecnt, uniq, segoff, perm, segidx, slot, single, sc);
        tr.mark();
    } else {
        // no ids: zero distinct ids and zero valid occurrences
        cudaMemsetAsync(&sc->n_unique, 0, 2 * sizeof(int32_t), a.stream);
        tr.launched = false;  // the next kernel follows the memset in plain stream order
    }
}

// Distinct ids, their counts and U to caller buffers.
__global__ void k_sp_export(const int32_t *__restrict__ uniq, const int32_t *__restrict__ segoff,
                            const DevScalars *__restrict__ sc, int64_t N, int32_t *__restrict__ uniq_out,
                            int32_t *__restrict__ counts_out, int32_t *__restrict__ n_unique_out)
{
    grid_dep_wait();
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
    constexpr int R = (4 / CPT) < 1 ? 1 : (4 / CPT);
    unsigned char *ws = a.ws;
    const Layout &L = a.lay;
    DevScalars *sc = reinterpret_cast<DevScalars *>(ws + L.scalars);
    auto *perm = reinterpret_cast<int32_t *>(ws + L.sp_perm);
    auto *segidx = reinterpret_cast<int32_t *>(ws + L.sp_segidx);
    auto *uniq = reinterpret_cast<int32_t *>(ws + L.sp_uniq);
    auto *segoff = reinterpret_cast<int32_t *>(ws + L.sp_segoff);
    auto *slot = reinterpret_cast<int32_t *>(ws + L.sp_slot);
    auto *single = reinterpret_cast<int32_t *>(ws + L.sp_single);
    auto *rowpart = reinterpret_cast<float *>(ws + L.sp_rowpart);
    auto *carry = reinterpret_cast<float *>(ws + L.sp_carry);
    auto *bounds = reinterpret_cast<int32_t *>(ws + L.sp_bounds);
    auto *S = reinterpret_cast<float *>(ws + L.sp_rows);
    auto *colpart = reinterpret_cast<float *>(ws + L.colpart);
    auto *rsum_part = reinterpret_cast<float *>(ws + L.rsum_part);
    auto *csum_part = reinterpret_cast<float *>(ws + L.csum_part);
    const int D = (int)a.D;
    const int DV = D / VEC;
    const int NS = (DV + kThreads - 1) / kThreads;
    Tracer tr{a.trace, a.n_trace, 0, a.stream};

    tr.mark();
    launch_sort_dedup(a, tr);
    const int G = kSparseCtas;
    const int nw = G / NS;
    const StepConsts kc = make_consts(a.beta2, a.one_minus_beta2, a.V, a.D, a.inv_bc);
    launch_k(k_sp_segsum<VEC>, dim3(G), dim3(kThreads), 0, a.stream, tr.pdl(), a.rows, perm, segidx, sc, S,
             rowpart, carry, colpart, bounds, D, NS, a.r, slot, a.V, kc.ema, rsum_part);
    tr.mark();
    launch_k(k_sp_carry<VEC>, dim3(G), dim3(kThreads), 0, a.stream, tr.pdl(), segidx, segoff, bounds, sc,
             carry, S, rowpart, colpart, D, NS, nw);
    tr.mark();
    // the touched rows' r and the column pass in one launch; the per-CTA
    // sums of r follow the segment-sum CTAs' sums of the decayed rows
    const int64_t ub = (a.N + kStateThreads - 1) / kStateThreads;
    const int GU = (int)(ub < kRsumParts - G ? ub : kRsumParts - G);
    // (segment-sum CTA b writes only the columns of its slice b % NS)
    launch_state(colpart, G, rsum_part, G + GU, a.c, csum_part, sc, a.V, D, kc, a.stream, tr.pdl(), a.r, slot, rowpart,
                 NS, GU, uniq, G, NS, kThreads * VEC);
    tr.mark();
    // one launch per column panel (one unless D is wider than a CTA's row)
    const int np = a.map.npanels, pw = a.map.pw;
    const size_t cs_bytes = (size_t)pw * sizeof(float);
    const int GA = kSms * apply_ctas_per_sm(CPT);
    for (int q = 0; q < np; ++q) {
        const int64_t c0 = (int64_t)q * pw;
        const int dq = (q + 1 < np) ? pw : (int)(a.D - c0);
        void *Wq = static_cast<unsigned char *>(a.W) + c0 * (a.wbf16 ? 2 : 4);
        const float *rq = a.rows ? a.rows + c0 : nullptr;
        if (a.wbf16)
            launch_k(k_sp_apply<VEC, CPT, R, true>, dim3(GA), dim3(kThreads), cs_bytes, a.stream, tr.pdl(), Wq,
                     S + c0, rq, uniq, single, a.r, a.c + c0, sc, dq, (int)a.D, a.map.tpr, (float)a.inv_bc, a.eps,
                     a.lr_signed, a.variant);
        else
            launch_k(k_sp_apply<VEC, CPT, R, false>, dim3(GA), dim3(kThreads), cs_bytes, a.stream, tr.pdl(), Wq,
                     S + c0, rq, uniq, single, a.r, a.c + c0, sc, dq, (int)a.D, a.map.tpr, (float)a.inv_bc, a.eps,
                     a.lr_signed, a.variant);
    }
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
    launch_k(k_sp_export, dim3((int)nb), dim3(kThreads), 0, a.stream, tr.pdl(), uniq, segoff, sc, a.N,
             uniq_out, counts_out, n_unique_out);
    // the touched-row map must be all-zero again before the next step
    int32_t *slot = reinterpret_cast<int32_t *>(a.ws + a.lay.sp_slot);
    cudaMemsetAsync(slot, 0, sizeof(int32_t) * (size_t)a.V, a.stream);
    return cudaGetLastError();
}

}  // namespace ember
