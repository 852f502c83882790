// Dense Ember step (Algorithm 1 of "Token Geometry", arXiv 2607.01455,
// Section 2.1) for sm_103a.
//
// The step needs two passes over the fp32 gradient G: the update of any
// element needs chat_j and s, which depend on every row of G (Section 2.3
// builds both statistics from sums of g^2).  The work is:
//
//   reduce  one read of G.  Per row: sum_j g^2 and the row EMA
//           r_i <- beta2 r_i + (1-beta2) mean_j g^2 (Algorithm 1's row second
//           moment), written once.  Per CTA: column sums of g^2 over its rows
//           and the sum of its new r values, written to the workspace.
//   state   O(D * CTAs) work: per column the exact fixed-point total of the
//           per-CTA partial sums (ember_device.cuh), the column EMA
//           c_j <- beta2 c_j + (1-beta2) mean_i g^2; then mean(rhat),
//           mean(chat) and s = sqrt(mean rhat * mean chat) (the
//           geometric-mean normaliser).
//   apply   reads G and W, writes W:
//           W_ij <- W_ij - lr g_ij / (sqrt(rhat_i) sqrt(chat_j / s) + eps),
//           the factored preconditioner applied as a row scale times a
//           column scale, never stored (Section 2.3).
//
// By default the three parts run as ONE cooperative launch (k_dense_fused):
// every CTA reduces its rows, a grid barrier, the CTAs share the column
// groups, a second grid barrier, then every CTA forms s itself (the same
// arithmetic in every CTA) and updates its rows.  The barriers replace two
// kernel boundaries, which is what small and mid-size tables pay for most.
// The three-kernel form (k_reduce_dense, k_state_dense, k_apply_dense) runs
// the same device code on the same CTA grid and gives the same bits; it
// serves the steps that need more than one launch anyway (column panels,
// the LM-head step, row shards, a gradient in host memory), traced steps,
// and devices where the cooperative grid does not fit.
//
// Bandwidth: 4VD bytes (reduce) + 4VD + 2 w VD bytes (apply), w = bytes per
// weight.  The apply walks each CTA's rows in the reverse order of the
// reduce, so the rows read last by the reduce -- still in L2 -- are the first
// ones it needs.
//
// Determinism: no floating-point atomics.  Every CTA owns a fixed row range
// (a function of V and D only) and every in-CTA sum has a fixed shape; the
// sums across CTAs are exact integer sums, so W and the state are
// bit-identical from run to run and however the partials are grouped (the
// row-sharded step relies on that), as Section 2.3 requires.
//
// The same launcher also runs:
//   - the row-only variant in one pass (k_rowonly_dense), no apply pass;
//   - the LM-head step: the tensor-core kernel of ember_lmhead.cu forms G and
//     its per-tile sums of g^2, the state pass finishes them (row pass from
//     per-column-block sums), then the apply pass;
//   - the three phases of a row-sharded step: the reduce over one shard's
//     CTAs of the whole-table grid (RowSpan) with the shard's largest
//     exponents per column, the fixed-point pack at the all-reduced
//     exponents, and the state pass on the all-reduced totals followed by
//     the shard's apply;
//   - tables wider than a CTA holds (more than 8192 columns, or 2048 without
//     16-byte accesses): the reduce and apply passes once per column panel
//     with the row stride D, the rows' sums of g^2 per panel added up by the
//     state pass, in panel order.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ember_device.cuh"
#include "ember_internal.h"

namespace ember {
namespace {

using namespace dev;

// ---------------------------------------------------------------------------
// Reduce: one read of G.  VEC columns per access, CPT accesses per thread per
// row, R rows per row group per iteration.  The CTA's rows are those of CTA
// span.cta_base + cta of a grid of span.nparts over the table; its column
// partial goes to colpart_row, the sum of its new r to *rsum_out.
// STAGE: G is read from host memory the GPU can address (over the
// Grace-Blackwell chip-to-chip link) and every element is also written to
// G_stage in HBM for the apply pass.
// D is the number of columns this launch covers and ld the row stride of G
// and colpart: a column panel of a wider table has D < ld, and then each
// row's sum of g^2 over the panel goes to rowpart[i] instead of into r.
// ---------------------------------------------------------------------------
// Column partial of a CTA from its row groups' sums: every group's sums side
// by side in rg x D floats of shared memory, then each column added over
// the groups in order 0 .. rg-1 -- the same float sums as a running total
// over the groups, with one barrier instead of one per group.
template <int VEC, int CPT>
__device__ __forceinline__ void combine_row_groups(const float (&acc)[CPT][VEC], float *colsh, float *out, int D,
                                                   int DV, int tpr, int rg, int g, int l)
{
#pragma unroll
    for (int c = 0; c < CPT; ++c) {
        const int col = l + c * tpr;
        if (col < DV)
#pragma unroll
            for (int e = 0; e < VEC; ++e)
                colsh[(size_t)g * D + col * VEC + e] = acc[c][e];
    }
    __syncthreads();
    for (int j = threadIdx.x; j < D; j += kThreads) {
        float t = colsh[j];
        for (int q = 1; q < rg; ++q)
            t += colsh[(size_t)q * D + j];
        out[j] = t;
    }
}

template <int VEC, int CPT, int R, bool STAGE, bool KEEP = false>
__device__ __forceinline__ void reduce_rows(const float *__restrict__ G, float *__restrict__ r,
                                            float *__restrict__ colpart_row, float *__restrict__ rsum_out,
                                            int64_t V, int D, int ld, int tpr, const StepConsts &kc,
                                            float *__restrict__ G_stage, float *__restrict__ rowpart,
                                            RowSpan span, int cta,
                                            float *__restrict__ comb, typename Vec<VEC>::F *__restrict__ keep,
                                            float *__restrict__ keep_r = nullptr)
{
    using F = typename Vec<VEC>::F;
    constexpr int kWarps = kThreads / 32;
    const int DV = D / VEC;
    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int rg = kThreads / tpr;           // row groups
    const int g = tid / tpr;                 // this thread's row group
    const int l = tid - g * tpr;             // position within the row
    const int wpg = tpr >> 5;                // warps per row group
    const int64_t row0 = (int64_t)(span.cta_base + cta) * V / span.nparts;
    const int64_t row1 = (int64_t)(span.cta_base + cta + 1) * V / span.nparts;

    // per-warp row sums of up to kRowBuf rows, finalised together
    constexpr int kRowBuf = 128;
    __shared__ float red[kWarps][kRowBuf];
    __shared__ float rsum_sh[kWarps];

    float acc[CPT][VEC];
#pragma unroll
    for (int c = 0; c < CPT; ++c)
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            acc[c][e] = 0.f;
    float rsum = 0.f;

    const int rows_per_it = rg * R;                 // rows of one iteration
    const int its_per_buf = kRowBuf / rows_per_it;  // >= 1: rg * R <= 128
    int64_t buf_base = row0;
    int nbuf = 0;  // iterations held in the buffer
    int it = 0;    // iteration index (the slot of the kept G)
    for (int64_t base = row0; base < row1; base += rows_per_it, ++it) {
        F v[R][CPT];
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = base + (int64_t)g * R + k;
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col = l + c * tpr;
                const bool in = i < row1 && col < DV;
                if constexpr (STAGE) {
                    const int64_t idx = (i - span.row_base) * ld + (int64_t)col * VEC;
                    v[k][c] = in ? *reinterpret_cast<const F *>(G + idx) : zero_vec<VEC>();
                    if (in)
                        *reinterpret_cast<F *>(G_stage + idx) = v[k][c];
                } else {
                    v[k][c] = in ? load_g<VEC>(G + (i - span.row_base) * ld + (int64_t)col * VEC)
                                 : zero_vec<VEC>();
                }
                if constexpr (KEEP)  // this thread's slot of the iteration, read back by the update
                    keep[((it * R + k) * CPT + c) * kThreads + tid] = v[k][c];
            }
        }
        // squares and per-row partial sums
        float rp[R];
#pragma unroll
        for (int k = 0; k < R; ++k) {
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < CPT; ++c)
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const float x = comp(v[k][c], e);
                    const float x2 = x * x;
                    set_comp(v[k][c], e, x2);
                    s += x2;
                }
            rp[k] = s;
        }
        // column sums: pairwise over the R rows of this iteration, then into acc
#pragma unroll
        for (int w = R / 2; w >= 1; w >>= 1)
#pragma unroll
            for (int k = 0; k < w; ++k)
#pragma unroll
                for (int c = 0; c < CPT; ++c)
#pragma unroll
                    for (int e = 0; e < VEC; ++e)
                        set_comp(v[k][c], e, comp(v[k][c], e) + comp(v[k + w][c], e));
#pragma unroll
        for (int c = 0; c < CPT; ++c)
#pragma unroll
            for (int e = 0; e < VEC; ++e)
                acc[c][e] += comp(v[0][c], e);

        // row sums within the warp; buffered until the cross-warp step
        int row_in_warp;
        const float tot = warp_sum_transposed<R>(rp, lane, row_in_warp);
        if ((lane & (32 / R - 1)) == 0)
            red[warp][nbuf * rows_per_it + g * R + row_in_warp] = tot;
        ++nbuf;
        if (nbuf == its_per_buf || base + rows_per_it >= row1) {
            __syncthreads();
            // row buf_base + q: sum of its row group's warps, in warp order
            for (int q = tid; q < nbuf * rows_per_it; q += kThreads) {
                const int64_t i = buf_base + q;
                if (i < row1) {
                    const int gq = (q % rows_per_it) / R;
                    float sum = 0.f;
                    for (int k = 0; k < wpg; ++k)
                        sum += red[gq * wpg + k][q];
                    if (rowpart) {
                        rowpart[i] = sum;
                        continue;
                    }
                    const float rn = ema_pair(kc.ema, r[i], sum * kc.inv_D);
                    r[i] = rn;
                    if (keep_r)  // the one-launch step's update reads it back here
                        keep_r[i - row0] = rn;
                    rsum += rn;
                }
            }
            __syncthreads();
            buf_base += (int64_t)nbuf * rows_per_it;
            nbuf = 0;
        }
    }

    // column partial of this CTA: row groups combined in order 0 .. rg-1
    if (rg == 1) {
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
            const int col = l + c * tpr;
            if (col < DV)
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    colpart_row[col * VEC + e] = acc[c][e];
        }
    } else {
        combine_row_groups<VEC, CPT>(acc, comb, colpart_row, D, DV, tpr, rg, g, l);  // rg x D floats
    }

    // sum of the new r values of this CTA (fp32): fixed butterfly per warp,
    // warps in order
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
    if (lane == 0)
        rsum_sh[warp] = rsum;
    __syncthreads();
    if (tid == 0 && rowpart == nullptr) {
        float s = 0.f;
        for (int q = 0; q < kWarps; ++q)
            s += rsum_sh[q];
        *rsum_out = s;
    }
}

// ---------------------------------------------------------------------------
// Apply: the update of the CTA's rows, walked from the last iteration block
// to the first.  The column scales live in shared memory (D floats): cs[j] =
// sqrt(chat_j / s) (FULL), sqrt(chat_j) (COL) or 1 (ROW).  D columns from row
// stride ld, as in the reduce: W, G and c point at the first column of the
// panel.  r and c are read through L2 (they may have been written earlier in
// the same launch).
// ---------------------------------------------------------------------------
template <int VEC, int CPT, int R, bool BF16>
__device__ __forceinline__ void apply_rows(void *__restrict__ W, const float *__restrict__ G,
                                           const float *__restrict__ r, const float *__restrict__ c,
                                           float inv_s_full, int64_t V, int D, int ld, int tpr, float inv_bc,
                                           float eps, float lr_signed, int variant, RowSpan span, int cta)
{
    using F = typename Vec<VEC>::F;
    using WT = typename WRaw<BF16, VEC>::T;
    extern __shared__ float cs[];  // D column scales
    const int DV = D / VEC;
    const int tid = threadIdx.x;
    const int rg = kThreads / tpr;
    const int g = tid / tpr;
    const int l = tid - g * tpr;
    const int64_t row0 = (int64_t)(span.cta_base + cta) * V / span.nparts;
    const int64_t row1 = (int64_t)(span.cta_base + cta + 1) * V / span.nparts;
    const int64_t step = (int64_t)rg * R;
    const int64_t nblocks = (row1 - row0 + step - 1) / step;

    const float inv_s = (variant == EMBER_VARIANT_FULL) ? inv_s_full : 1.f;
    for (int j = tid; j < D; j += kThreads)
        cs[j] = (variant == EMBER_VARIANT_ROW) ? 1.f : sqrtf(__ldcg(c + j) * inv_bc * inv_s);
    __syncthreads();

    for (int64_t b = nblocks - 1; b >= 0; --b) {
        const int64_t base = row0 + b * step;
        F gv[R][CPT];
        WT wr[R][CPT];
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = base + (int64_t)g * R + k;
#pragma unroll
            for (int cc = 0; cc < CPT; ++cc) {
                const int col = l + cc * tpr;
                if (i < row1 && col < DV) {
                    const int64_t idx = (i - span.row_base) * ld + (int64_t)col * VEC;
                    gv[k][cc] = load_g<VEC>(G + idx);
                    wr[k][cc] = load_w<BF16, VEC>(W, idx);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = base + (int64_t)g * R + k;
            if (i >= row1)
                continue;
            const float rs = (variant == EMBER_VARIANT_COL) ? 1.f : sqrtf(__ldcg(r + i) * inv_bc);
#pragma unroll
            for (int cc = 0; cc < CPT; ++cc) {
                const int col = l + cc * tpr;
                if (col >= DV)
                    continue;
                float w[VEC];
                unpack_w(wr[k][cc], w);
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const float den = fmaf(rs, cs[col * VEC + e], eps);
                    const float u = update_ratio(comp(gv[k][cc], e), den);
                    w[e] = fmaf(lr_signed, u, w[e]);
                }
                store_w<BF16, VEC>(W, (i - span.row_base) * ld + (int64_t)col * VEC, w);
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Column pass of one group of kStateCols = 32 columns, by a whole CTA of
// kStateThreads threads: lane l of every warp owns column j0 + l.
// Source: the partial rows colpart[b * D + j], b < nparts (warp w reads rows
// w, w + 8, ...; the column's total is their exact fixed-point sum at the
// largest key among them), or, with `sums` set, the totals already formed
// elsewhere (the all-reduce of a row-sharded step) at scales[j].
// Writes c_j <- beta2 c_j + (1 - beta2) total_j / V and csum_part[group] =
// the fp32 sum of the group's new c (a fixed butterfly).
// ---------------------------------------------------------------------------
struct ColSource {
    const float *colpart;                 // [nparts][D]
    int nparts;
    const unsigned long long *sums;       // nullptr, or [D] totals
    const unsigned char *scales;          // their scale exponents
    // partial row b holds nonzero sums only in columns [s pcols, (s + 1) pcols)
    // of slice s = b % pstride (the sparse step's segment-sum CTAs); pstride
    // 1: every row covers every column
    int pstride = 1, pcols = 0;
};

constexpr int kStateWarps = kStateThreads / 32;
// partial rows per warp held in registers by the column pass (the dense
// step's 304 and the sparse step's 456 rows fit; more, as the LM-head step
// has, take two passes through L2)
constexpr int kRegParts = 64;
static_assert(kRegParts * kStateWarps >= kGridCtas, "the dense step's partial rows fit the register path");

__device__ __forceinline__ void column_group(const ColSource &src, int group, float *__restrict__ c,
                                             float *__restrict__ csum_part, int D, const StepConsts &kc)
{
    __shared__ unsigned emax_sh[kStateWarps][32];
    __shared__ unsigned long long ssum_sh[kStateWarps][32];
    const int lane = threadIdx.x & 31;
    const int w = threadIdx.x >> 5;
    const int j = group * kStateCols + lane;
    const float c_old = (w == 0 && j < D) ? __ldcg(c + j) : 0.f;  // loaded with the partials
    // the partial rows of this group's slice: b = sigma + p pstride, p < np
    // (the other rows are zero in these columns and add nothing)
    const int sigma = (src.pstride > 1) ? (group * kStateCols) / src.pcols : 0;
    const int np = (src.nparts - sigma + src.pstride - 1) / src.pstride;
    unsigned long long S = 0;
    unsigned E = 0;
    if (src.sums == nullptr && np <= kRegParts * kStateWarps) {
        // up to kRegParts partial rows per warp: one trip to L2, the values
        // kept in registers for both the largest key and the sum
        // (in chunks of 8, the chunks past this warp's last row skipped)
        constexpr int kChunk = 8;
        const int kv = (np - w + kStateWarps - 1) / kStateWarps;  // this warp's rows
        float v[kRegParts];
        unsigned e = 0;
#pragma unroll
        for (int k0 = 0; k0 < kRegParts; k0 += kChunk) {
            if (k0 >= kv)
                break;
#pragma unroll
            for (int k = k0; k < k0 + kChunk; ++k) {
                const int p = w + k * kStateWarps;
                v[k] = (p < np && j < D) ? __ldcg(src.colpart + (int64_t)(sigma + p * src.pstride) * D + j) : 0.f;
            }
        }
#pragma unroll
        for (int k0 = 0; k0 < kRegParts; k0 += kChunk) {
            if (k0 >= kv)
                break;
#pragma unroll
            for (int k = k0; k < k0 + kChunk; ++k)
                e = max(e, fx_key(v[k]));
        }
        emax_sh[w][lane] = e;
        __syncthreads();
#pragma unroll
        for (int q = 0; q < kStateWarps; ++q)
            E = max(E, emax_sh[q][lane]);
        unsigned long long s = 0;
#pragma unroll
        for (int k0 = 0; k0 < kRegParts; k0 += kChunk) {
            if (k0 >= kv)
                break;
#pragma unroll
            for (int k = k0; k < k0 + kChunk; ++k)
                s += fx_of(v[k], E);
        }
        ssum_sh[w][lane] = s;
        __syncthreads();
        if (w == 0)
#pragma unroll
            for (int q = 0; q < kStateWarps; ++q)
                S += ssum_sh[q][lane];
    } else if (src.sums == nullptr) {
        constexpr int kBatch = 16;
        // pass 1: the largest key of the column (loads batched for latency)
        unsigned e = 0;
        if (j < D)
            for (int p0 = w; p0 < np; p0 += kBatch * kStateWarps) {
                float v[kBatch];
#pragma unroll
                for (int k = 0; k < kBatch; ++k) {
                    const int p = p0 + k * kStateWarps;
                    v[k] = (p < np) ? __ldcg(src.colpart + (int64_t)(sigma + p * src.pstride) * D + j) : 0.f;
                }
#pragma unroll
                for (int k = 0; k < kBatch; ++k)
                    e = max(e, fx_key(v[k]));
            }
        emax_sh[w][lane] = e;
        __syncthreads();
#pragma unroll
        for (int q = 0; q < kStateWarps; ++q)
            E = max(E, emax_sh[q][lane]);
        // pass 2: the exact total (the partials are still in L2)
        unsigned long long s = 0;
        if (j < D)
            for (int p0 = w; p0 < np; p0 += kBatch * kStateWarps) {
                float v[kBatch];
#pragma unroll
                for (int k = 0; k < kBatch; ++k) {
                    const int p = p0 + k * kStateWarps;
                    v[k] = (p < np) ? __ldcg(src.colpart + (int64_t)(sigma + p * src.pstride) * D + j) : 0.f;
                }
#pragma unroll
                for (int k = 0; k < kBatch; ++k)
                    s += fx_of(v[k], E);
            }
        ssum_sh[w][lane] = s;
        __syncthreads();
        if (w == 0)
#pragma unroll
            for (int q = 0; q < kStateWarps; ++q)
                S += ssum_sh[q][lane];
    } else if (w == 0 && j < D) {
        S = src.sums[j];
        E = src.scales[j];
    }
    if (w == 0) {
        float cn = 0.f;
        if (j < D) {
            const float m = fx_value(S, E) * kc.inv_V;
            cn = ema_pair(kc.ema, c_old, m);
            c[j] = cn;
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            cn += __shfl_xor_sync(0xffffffffu, cn, o);
        if (lane == 0)
            csum_part[group] = cn;
    }
    __syncthreads();  // the shared buffers are reused by the next group
}

// Exact fixed-point total of n fp32 values load(0) .. load(n-1) (>= 0), by a
// whole CTA of kStateThreads threads; every thread gets the result.  The
// loader reads global memory through L2 (the values were written by other
// CTAs) or another CTA's shared memory in a cluster.
template <int NT = kStateThreads, typename Load>
__device__ float block_fx_total(Load load, int n)
{
    constexpr int kNW = NT / 32;  // warps
    __shared__ unsigned ek[kNW];
    __shared__ unsigned long long ss[kNW];
    const int lane = threadIdx.x & 31;
    const int w = threadIdx.x >> 5;
    // each thread's first value is loaded once and kept for the second pass
    const float first = ((int)threadIdx.x < n) ? load(threadIdx.x) : 0.f;
    unsigned e = fx_key(first);
    for (int b = threadIdx.x + NT; b < n; b += NT)
        e = max(e, fx_key(load(b)));
    e = __reduce_max_sync(0xffffffffu, e);
    if (lane == 0)
        ek[w] = e;
    __syncthreads();
    unsigned E = 0;
#pragma unroll
    for (int q = 0; q < kNW; ++q)
        E = max(E, ek[q]);
    unsigned long long s = fx_of(first, E);  // 0 for a zero
    for (int b = threadIdx.x + NT; b < n; b += NT)
        s += fx_of(load(b), E);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        s += shfl_xor_u64(s, o);
    if (lane == 0)
        ss[w] = s;
    __syncthreads();
    unsigned long long S = 0;
#pragma unroll
    for (int q = 0; q < kNW; ++q)
        S += ss[q];
    __syncthreads();
    return fx_value(S, E);
}

// The normaliser from the total of r (r_total, over the whole table) and the
// per-group sums of the new c (load(q), q < ngroups), by a whole CTA of NT
// threads; every thread gets it.  The group sums are added in a fixed order
// (thread t takes groups t, t + NT, ... in order, then a fixed butterfly,
// then the warps in order), so every CTA that runs this forms the same bits,
// and for up to 256 groups CTAs of 256 and 512 threads form the same sums
// (each thread holds at most one group; the extra warps add zeros).
struct Norm {
    float s, rbar, cbar, inv_s;
};
template <int NT = kStateThreads, typename Load>
__device__ Norm normaliser(float r_total, Load load, int ngroups, const StepConsts &kc)
{
    constexpr int kNW = NT / 32;  // warps
    __shared__ float part[kNW];
    const int lane = threadIdx.x & 31;
    const int w = threadIdx.x >> 5;
    float csum = 0.f;
    for (int q = threadIdx.x; q < ngroups; q += NT)
        csum += load(q);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        csum += __shfl_xor_sync(0xffffffffu, csum, o);
    if (lane == 0)
        part[w] = csum;
    __syncthreads();
    csum = 0.f;
    for (int q = 0; q < kNW; ++q)
        csum += part[q];
    __syncthreads();
    Norm n;
    n.rbar = (r_total * kc.inv_bc) * kc.inv_V;
    n.cbar = (csum * kc.inv_bc) * kc.inv_D;
    // the square roots taken apart: their product stays in range where
    // rbar * cbar would underflow
    n.s = sqrtf(n.rbar) * sqrtf(n.cbar);
    n.inv_s = (n.s > 0.f) ? 1.f / n.s : 0.f;
    return n;
}

// ---------------------------------------------------------------------------
// Kernels of the three-launch form.
// ---------------------------------------------------------------------------
template <int VEC, int CPT, int R, bool STAGE>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_reduce_dense(const float *__restrict__ G, float *__restrict__ r, float *__restrict__ colpart,
               float *__restrict__ rsum_part, int64_t V, int D, int ld, int tpr, StepConsts kc,
               float *__restrict__ G_stage, float *__restrict__ rowpart, RowSpan span)
{
    grid_dep_wait();    // the first kernel of a step: returns at once
    grid_dep_launch();  // the state pass may start launching now; it waits for this grid
    extern __shared__ float comb_sh[];  // rg x D floats: the row groups' column sums
    reduce_rows<VEC, CPT, R, STAGE>(G, r, colpart + (int64_t)blockIdx.x * ld, rsum_part + blockIdx.x, V, D, ld,
                                    tpr, kc, G_stage, rowpart, span, blockIdx.x, comb_sh,
                                    nullptr);
}

// Column EMA and normaliser.  The first ngroups CTAs each own one group of
// 32 columns (column_group).  For the sparse and LM-head steps and a dense
// step in column panels the remaining CTAs also do the row pass: r for every
// row (rows outside a sparse batch see a zero gradient row, touched rows take
// their sum of g^2 per column slice from `rowpart`) and the sum of the new r
// per CTA.  The last CTA to finish forms mean(rhat), mean(chat) and s; the
// sum of r over the table is the exact fixed-point total of the nrsum per-CTA
// sums, or, in a row-sharded step, comes with the exchanged totals.
struct RowPass {
    float *r;               // r[V], updated
    int32_t *slot;          // sparse step: touched-row map, cleared here
    const float *rowpart;   // per (distinct id, slice) sums of g^2, or per (slice, row)
    int nslices;
    int nrow_ctas;          // 0 for the dense step
    const int32_t *uniq;    // sparse step: the distinct ids (U of them, sc->n_unique)
    int rsum_base;          // index of this launch's first per-CTA sum of r in rsum_part
};

__global__ void __launch_bounds__(kStateThreads)
k_state_dense(ColSource src, float *__restrict__ rsum_part, int nrsum, float *__restrict__ c,
              float *__restrict__ csum_part, DevScalars *sc, int64_t V, int D, StepConsts kc, RowPass rowp)
{
    constexpr int kW = kStateWarps;
    const int lane = threadIdx.x & 31;
    const int w = threadIdx.x >> 5;
    const int ngroups = (int)gridDim.x - rowp.nrow_ctas;
    __shared__ float part[kW];
    __shared__ bool am_last;
    // GB300 runs fp64 at a small fraction of its fp32 rate: everything here
    // is fp32 (the EMAs with float-pair coefficients, sums of at most a few
    // thousand values per CTA in fixed trees, the normaliser) or integer
    // (the fixed-point totals).
    grid_dep_wait();  // column partials and row sums of the earlier passes
    grid_dep_launch();

    if ((int)blockIdx.x < ngroups) {
        column_group(src, blockIdx.x, c, csum_part, D, kc);
    } else {
        const int rb = (int)blockIdx.x - ngroups;
        const int64_t stride = (int64_t)rowp.nrow_ctas * kStateThreads;
        // Every row of the table: the row EMA (ema_pair), then the CTA's sum
        // of the new r in fp32 (thread, warp butterfly, warps in order).
        const float inv_Df = kc.inv_D;
        const EmaPair &ema = kc.ema;
        float rsum = 0.f;
        if (rowp.slot == nullptr) {
            // every row: per-column-block sums, slice-major, in block order
            float tsum = 0.f;
            for (int64_t i = (int64_t)rb * kStateThreads + threadIdx.x; i < V; i += stride) {
                float tot = 0.f;
#pragma unroll 8
                for (int k = 0; k < rowp.nslices; ++k)
                    tot += __ldcg(rowp.rowpart + (int64_t)k * V + i);
                const float rn = ema_pair(ema, rowp.r[i], tot * inv_Df);
                rowp.r[i] = rn;
                tsum += rn;
            }
            rsum = tsum;
        } else {
            // sparse step: the touched rows only (the segment-sum kernel has
            // decayed every other row): each adds its sums of g^2 per slice
            const int64_t U = sc->n_unique;
            for (int64_t u = (int64_t)rb * kStateThreads + threadIdx.x; u < U; u += stride) {
                const int64_t i = rowp.uniq[u];
                float tot = 0.f;
                for (int q = 0; q < rowp.nslices; ++q)
                    tot += rowp.rowpart[u * rowp.nslices + q];
                const float rn = ema_pair(ema, rowp.r[i], tot * inv_Df);
                rowp.r[i] = rn;
                rowp.slot[i] = 0;
                rsum += rn;
            }
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
        if (lane == 0)
            part[w] = rsum;
        __syncthreads();
        if (threadIdx.x == 0) {
            float t = 0.f;
            for (int q = 0; q < kW; ++q)
                t += part[q];
            rsum_part[rowp.rsum_base + rb] = t;
        }
    }
    if (threadIdx.x == 0) {
        __threadfence();
        const unsigned t = atomicAdd(&sc->ticket, 1u);
        am_last = (t == gridDim.x - 1);
    }
    __syncthreads();
    if (!am_last)
        return;
    __threadfence();
    // this thread's first group sum of c, loaded together with the sums of r
    const float c_first = ((int)threadIdx.x < ngroups) ? __ldcg(csum_part + threadIdx.x) : 0.f;
    const float r_total = (src.sums != nullptr)
                              ? fx_value(src.sums[D], src.scales[D])
                              : block_fx_total([&](int b) { return __ldcg(rsum_part + b); }, nrsum);
    const Norm n = normaliser(
        r_total, [&](int q) { return q == (int)threadIdx.x ? c_first : __ldcg(csum_part + q); }, ngroups, kc);
    if (threadIdx.x == 0) {
        sc->s = n.s;
        sc->rbar = n.rbar;
        sc->cbar = n.cbar;
        sc->inv_s = n.inv_s;
        sc->ticket = 0u;
    }
}

template <int VEC, int CPT, int R, bool BF16>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_apply_dense(void *__restrict__ W, const float *__restrict__ G, const float *__restrict__ r,
              const float *__restrict__ c, const DevScalars *__restrict__ sc, int64_t V, int D, int ld, int tpr,
              float inv_bc, float eps, float lr_signed, int variant, RowSpan span)
{
    // While the state pass finishes: pull this thread's first rows of G and
    // W (the last iteration block, walked first) towards L2.
    {
        const int rg = kThreads / tpr;
        const int g = threadIdx.x / tpr;
        const int l = threadIdx.x - g * tpr;
        const int DV = D / VEC;
        const int64_t row0 = (int64_t)(span.cta_base + blockIdx.x) * V / span.nparts;
        const int64_t row1 = (int64_t)(span.cta_base + blockIdx.x + 1) * V / span.nparts;
        const int64_t step = (int64_t)rg * R;
        const int64_t nblocks = (row1 - row0 + step - 1) / step;
        if (nblocks > 0) {
            const int64_t base = row0 + (nblocks - 1) * step;
            for (int k = 0; k < R; ++k) {
                const int64_t i = base + (int64_t)g * R + k;
                for (int cc = 0; cc < CPT; ++cc) {
                    const int col = l + cc * tpr;
                    if (i < row1 && col < DV) {
                        const int64_t idx = (i - span.row_base) * ld + (int64_t)col * VEC;
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(G + idx));
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(static_cast<const char *>(W) +
                                                                       idx * (BF16 ? 2 : 4)));
                    }
                }
            }
        }
    }
    grid_dep_wait();  // c, s (state pass) and r (reduce pass)
    grid_dep_launch();
    apply_rows<VEC, CPT, R, BF16>(W, G, r, c, __ldcg(&sc->inv_s), V, D, ld, tpr, inv_bc, eps, lr_signed, variant,
                                  span, blockIdx.x);
}

// ---------------------------------------------------------------------------
// Small tables in one launch: one thread-block cluster of nparts <= 16 CTAs
// (the same CTA grid and row ranges as the three-launch form).  Each CTA
//   - starts copying its rows of W into shared memory (cp.async) and loads
//     the old c;
//   - reduces its rows with reduce_rows, keeping every element of G it loads
//     in a thread-private slot of shared memory, and leaves its column
//     partial and its sum of r in its own shared memory;
//   - cluster barrier; then reads every CTA's partials through distributed
//     shared memory and forms, for ALL columns, the column totals, the new c
//     and the normaliser itself (the same integer totals, EMA and fixed
//     summation order as column_group / block_fx_total / normaliser, hence
//     the same bits as the three-launch form);
//   - updates its rows from the kept G and W.
// G is read from HBM once (4VD + 2wVD bytes in all, not 8VD + 2wVD), and the
// only synchronisation is the cluster's hardware barrier, so the step is a
// single short launch.  Used when the kept G and W fit shared memory.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cluster_barrier()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive() { asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

// A float of CTA `rank`'s shared memory at the address `local` has in this CTA.
__device__ __forceinline__ float ld_dsmem(const float *local, unsigned rank)
{
    uint32_t a = (uint32_t)__cvta_generic_to_shared(local), ra;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(rank));
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(ra) : "memory");
    return v;
}

struct SmallArgs {
    void *W;
    const float *G;
    float *r, *c;
    DevScalars *sc;
    int64_t V;
    int D, tpr, nits;
    StepConsts kc;
    float eps, lr_signed;
    int variant;
};


// Shared memory of k_dense_cluster, from the dynamic base: kept G, kept W
// (one 16- or 8-byte slot per thread, per row and access of each reduce
// iteration), then D floats of the column partial, (256 / tpr) x D floats of
// the row groups' sums, D floats each of the old c and the new c (then the
// column scales), ceil(D/32) floats, and the new r of the CTA's rows.
template <int CPT, int R, bool BF16>
__host__ __device__ constexpr size_t small_slots(int nits) { return (size_t)nits * R * CPT * kThreads; }

}  // namespace

// Whether a dense step of this table runs as one cluster launch: the vector
// path, one column panel, at most kMaxClusterCtas CTAs, and the kept G and W
// (every slot of the CTA's reduce iterations) within kSmallSmemMax of shared
// memory.  *nits: reduce iterations per CTA; *smem: dynamic shared memory.
bool small_table_plan(int64_t V, int64_t D, bool wbf16, const ColMap &m, int *nits, size_t *smem)
{
    const int nparts = dense_parts(V, D);
    if (m.vec != 4 || m.npanels != 1 || nparts > kMaxClusterCtas)
        return false;
    const int R1 = reduce_rows_per_thread(V, D, m);
    const int rows_per_it = (kThreads / m.tpr) * R1;
    const int64_t rows = (V + nparts - 1) / nparts;
    const int64_t n = (rows + rows_per_it - 1) / rows_per_it;
    const size_t slots = (size_t)n * R1 * m.cpt * kThreads;
    // kept G and W, then D floats each of the column partial, the old c and
    // the new c, rg x D floats of row-group sums, the group sums of c and
    // the new r of the CTA's rows
    const size_t bytes = slots * (16 + (wbf16 ? 8 : 16)) +
                         (size_t)(3 + kThreads / m.tpr) * D * sizeof(float) +
                         (size_t)((D + kStateCols - 1) / kStateCols) * sizeof(float) + (size_t)rows * sizeof(float);
    if (bytes > kSmallSmemMax)
        return false;
    *nits = (int)n;
    *smem = bytes;
    return true;
}

int dense_step_launches(int64_t V, int64_t D, bool wbf16, int variant, bool vec4)
{
    ColMap m;
    if (!choose_colmap(D, vec4, &m))
        return 0;
    int nits = 0;
    size_t sm = 0;
    if (m.npanels == 1 && variant == EMBER_VARIANT_ROW)
        return 2;  // the one-pass row-only kernel and the column state
    if (variant != EMBER_VARIANT_ROW && small_table_plan(V, D, wbf16, m, &nits, &sm))
        return 1;
    return 2 * m.npanels + 1;
}

namespace {

template <int CPT, int R, bool BF16>
__global__ void __launch_bounds__(kThreads, 1)
k_dense_cluster(SmallArgs a)
{
    constexpr int VEC = 4;
    using F = float4;
    using WT = typename WRaw<BF16, VEC>::T;
    extern __shared__ __align__(16) unsigned char sm_dyn[];
    const size_t nslot = small_slots<CPT, R, BF16>(a.nits);
    F *keepG = reinterpret_cast<F *>(sm_dyn);
    WT *keepW = reinterpret_cast<WT *>(sm_dyn + nslot * 16);
    float *cpart = reinterpret_cast<float *>(sm_dyn + nslot * (16 + sizeof(WT)));
    float *comb = cpart + a.D;  // (256 / tpr) x D floats
    float *cold = comb + (size_t)(kThreads / a.tpr) * a.D;
    float *cnew = cold + a.D;
    float *csum_sh = cnew + a.D;
    float *rnew = csum_sh + (a.D + kStateCols - 1) / kStateCols;  // the new r of this CTA's rows
    __shared__ float rsum_own;

    const int D = a.D, DV = D / VEC, tid = threadIdx.x;
    const int tpr = a.tpr, rg = kThreads / tpr, g = tid / tpr, l = tid - g * tpr;
    const unsigned nb = gridDim.x;
    const unsigned cta = blockIdx.x;  // the grid is one cluster: the rank in it
    const RowSpan span{0, (int)nb, 0};
    const int64_t row0 = (int64_t)cta * a.V / nb, row1 = (int64_t)(cta + 1) * a.V / nb;
    const int rows_per_it = rg * R;

    // this CTA's rows of W into its slots, while G is reduced
    for (int it = 0; it < a.nits; ++it)
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = row0 + (int64_t)it * rows_per_it + (int64_t)g * R + k;
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col = l + c * tpr;
                if (i < row1 && col < DV) {
                    WT *dst = keepW + ((it * R + k) * CPT + c) * kThreads + tid;
                    const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst);
                    if constexpr (BF16)
                        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(d),
                                     "l"(static_cast<const unsigned short *>(a.W) + i * D + (int64_t)col * VEC)
                                     : "memory");
                    else
                        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d),
                                     "l"(static_cast<const float *>(a.W) + i * D + (int64_t)col * VEC)
                                     : "memory");
                }
            }
        }
    asm volatile("cp.async.commit_group;" ::: "memory");
    for (int j = tid; j < D; j += kThreads)
        cold[j] = a.c[j];

    reduce_rows<VEC, CPT, R, false, true>(a.G, a.r, cpart, &rsum_own, a.V, D, D, tpr, a.kc, nullptr, nullptr, span,
                                          cta, comb, keepG, rnew);
    cluster_barrier();  // every CTA's partials are in its shared memory

    // the column pass for every column, as column_group forms it
    const int lane = tid & 31, w = tid >> 5;
    const int ngroups = (D + kStateCols - 1) / kStateCols;
    for (int q = w; q < ngroups; q += kThreads / 32) {
        const int j = q * kStateCols + lane;
        float v[kMaxClusterCtas];
        unsigned E = 0;
#pragma unroll
        for (int b = 0; b < kMaxClusterCtas; ++b) {
            v[b] = (b < (int)nb && j < D) ? ld_dsmem(cpart + j, b) : 0.f;
            E = max(E, fx_key(v[b]));
        }
        unsigned long long S = 0;
#pragma unroll
        for (int b = 0; b < kMaxClusterCtas; ++b)
            S += fx_of(v[b], E);
        float cn = 0.f;
        if (j < D) {
            const float m = fx_value(S, E) * a.kc.inv_V;
            cn = ema_pair(a.kc.ema, cold[j], m);
            cnew[j] = cn;
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            cn += __shfl_xor_sync(0xffffffffu, cn, o);
        if (lane == 0)
            csum_sh[q] = cn;
    }
    const float r_total = block_fx_total<kThreads>([&](int b) { return ld_dsmem(&rsum_own, b); }, (int)nb);
    cluster_arrive();  // done reading the other CTAs' shared memory
    const Norm n = normaliser<kThreads>(r_total, [&](int q) { return csum_sh[q]; }, ngroups, a.kc);
    if (cta == 0) {
        for (int j = tid; j < D; j += kThreads)
            a.c[j] = cnew[j];
        if (tid == 0) {
            a.sc->s = n.s;
            a.sc->rbar = n.rbar;
            a.sc->cbar = n.cbar;
            a.sc->inv_s = n.inv_s;
        }
    }

    // the update, as apply_rows forms it, from the kept G and W
    const float inv_bc = a.kc.inv_bc;
    const float inv_s = (a.variant == EMBER_VARIANT_FULL) ? n.inv_s : 1.f;
    float *cs = cnew;  // the column scales replace the new c (already written out)
    __syncthreads();
    for (int j = tid; j < D; j += kThreads)
        cs[j] = (a.variant == EMBER_VARIANT_ROW) ? 1.f : sqrtf(cnew[j] * inv_bc * inv_s);
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
    for (int it = 0; it < a.nits; ++it)
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = row0 + (int64_t)it * rows_per_it + (int64_t)g * R + k;
            if (i >= row1)
                continue;
            const float rs = (a.variant == EMBER_VARIANT_COL) ? 1.f : sqrtf(rnew[i - row0] * inv_bc);
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col = l + c * tpr;
                if (col >= DV)
                    continue;
                const int slot = ((it * R + k) * CPT + c) * kThreads + tid;
                const F gv = keepG[slot];
                float wv[VEC];
                unpack_w(keepW[slot], wv);
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const float den = fmaf(rs, cs[col * VEC + e], a.eps);
                    const float u = update_ratio(comp(gv, e), den);
                    wv[e] = fmaf(a.lr_signed, u, wv[e]);
                }
                store_w<BF16, VEC>(a.W, i * D + (int64_t)col * VEC, wv);
            }
        }
    cluster_wait();  // no CTA leaves while another may still read its shared memory
}

// Row-only Ember in one pass (variant ROW: vtil_ij = rhat_i, the "row-only"
// row of the Section 2.1 ablation table).  The update of row i needs only
// r_i, which depends on row i alone, so a CTA reads each row of G once,
// finishes its sum of g^2 and its r_i, and updates the row of W from the
// gradient still in registers: 4VD + 2wVD bytes instead of the full
// preconditioner's 8VD + 2wVD.  Column sums of g^2 are still accumulated so
// that c (part of the same V + D state) is maintained by the state pass.
//
// With ASYNC (16-byte column slices), each thread copies its own elements of
// the next iteration's rows into shared memory with cp.async while the
// current rows are reduced and updated, so the two barriers of each
// iteration no longer leave HBM without requests.  A thread reads back only
// what it copied itself: the copies need no barrier.
template <int CPT, int R, bool BF16>
constexpr size_t rowonly_stage_bytes() { return (size_t)2 * R * CPT * kThreads * (16 + (BF16 ? 8 : 16)); }

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async8(void *smem, const void *gmem)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_prev() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

template <int VEC, int CPT, int R, bool BF16, bool ASYNC>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_rowonly_dense(void *__restrict__ W, const float *__restrict__ G, float *__restrict__ r,
                float *__restrict__ colpart, float *__restrict__ rsum_part, int64_t V, int D, int tpr,
                StepConsts kc, float eps, float lr_signed)
{
    static_assert(!ASYNC || VEC == 4, "the staged copies move 16-byte slices");
    using F = typename Vec<VEC>::F;
    using WT = typename WRaw<BF16, VEC>::T;
    constexpr int kWarps = kThreads / 32;
    const int DV = D / VEC;
    const int tid = threadIdx.x;
    const int lane = tid & 31;
    const int warp = tid >> 5;
    const int rg = kThreads / tpr;
    const int g = tid / tpr;
    const int l = tid - g * tpr;
    const int wpg = tpr >> 5;
    const int64_t row0 = (int64_t)blockIdx.x * V / gridDim.x;
    const int64_t row1 = (int64_t)(blockIdx.x + 1) * V / gridDim.x;
    __shared__ float red[kWarps][R];
    __shared__ float rs_sh[kThreads / 32 * R];  // sqrt(rhat) of this iteration's rows
    __shared__ float rsum_sh[kWarps];
    // ASYNC: two stages of [R][CPT][kThreads] slices of G, then of W; the
    // column-sum combine buffer (D floats) follows
    extern __shared__ __align__(16) unsigned char ro_dyn[];
    constexpr int kWB = BF16 ? 8 : 16;
    constexpr size_t kStageG = (size_t)2 * R * CPT * kThreads * 16;
    auto sg_at = [&](int buf, int k, int c) {
        return ro_dyn + ((size_t)((buf * R + k) * CPT + c) * kThreads + tid) * 16;
    };
    auto sw_at = [&](int buf, int k, int c) {
        return ro_dyn + kStageG + ((size_t)((buf * R + k) * CPT + c) * kThreads + tid) * kWB;
    };
    grid_dep_wait();
    grid_dep_launch();
    auto stage = [&](int64_t base, int buf) {  // one commit group per call
        if constexpr (ASYNC) {
#pragma unroll
            for (int k = 0; k < R; ++k) {
                const int64_t i = base + (int64_t)g * R + k;
#pragma unroll
                for (int c = 0; c < CPT; ++c) {
                    const int col = l + c * tpr;
                    if (i < row1 && col < DV) {
                        const int64_t idx = i * D + (int64_t)col * VEC;
                        cp_async16(sg_at(buf, k, c), G + idx);
                        if constexpr (BF16)
                            cp_async8(sw_at(buf, k, c), static_cast<const unsigned short *>(W) + idx);
                        else
                            cp_async16(sw_at(buf, k, c), static_cast<const float *>(W) + idx);
                    }
                }
            }
            cp_async_commit();
        }
    };
    int buf = 0;
    if (ASYNC && row0 < row1)
        stage(row0, 0);

    float acc[CPT][VEC];
#pragma unroll
    for (int c = 0; c < CPT; ++c)
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            acc[c][e] = 0.f;
    float rsum = 0.f;
    const int rows_per_it = rg * R;
    for (int64_t base = row0; base < row1; base += rows_per_it) {
        F v[R][CPT];
        WT wr[R][CPT];
        if constexpr (ASYNC) {
            // the next iteration's copies go out, this one's have landed
            if (base + rows_per_it < row1)
                stage(base + rows_per_it, buf ^ 1);
            else
                cp_async_commit();
            cp_async_wait_prev();
        }
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = base + (int64_t)g * R + k;
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col = l + c * tpr;
                const bool in = i < row1 && col < DV;
                if constexpr (ASYNC) {
                    v[k][c] = in ? *reinterpret_cast<const F *>(sg_at(buf, k, c)) : zero_vec<VEC>();
                    if (in)
                        wr[k][c] = *reinterpret_cast<const WT *>(sw_at(buf, k, c));
                } else {
                    v[k][c] = in ? load_g<VEC>(G + i * D + (int64_t)col * VEC) : zero_vec<VEC>();
                    if (in)
                        wr[k][c] = load_w<BF16, VEC>(W, i * D + (int64_t)col * VEC);
                }
            }
        }
        buf ^= 1;
        float rp[R];
#pragma unroll
        for (int k = 0; k < R; ++k) {
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < CPT; ++c)
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const float x = comp(v[k][c], e);
                    s = fmaf(x, x, s);
                    acc[c][e] = fmaf(x, x, acc[c][e]);
                }
            rp[k] = s;
        }
        int row_in_warp;
        const float tot = warp_sum_transposed<R>(rp, lane, row_in_warp);
        if ((lane & (32 / R - 1)) == 0)
            red[warp][row_in_warp] = tot;
        __syncthreads();
        if (l < R) {
            const int64_t i = base + (int64_t)g * R + l;
            float rsv = 0.f;
            if (i < row1) {
                float sum = 0.f;
                for (int q = 0; q < wpg; ++q)
                    sum += red[g * wpg + q][l];
                const float rn = ema_pair(kc.ema, r[i], sum * kc.inv_D);
                r[i] = rn;
                rsum += rn;
                rsv = sqrtf(rn * kc.inv_bc);
            }
            rs_sh[g * R + l] = rsv;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const int64_t i = base + (int64_t)g * R + k;
            if (i >= row1)
                continue;
            const float den = rs_sh[g * R + k] + eps;
#pragma unroll
            for (int c = 0; c < CPT; ++c) {
                const int col = l + c * tpr;
                if (col >= DV)
                    continue;
                float w[VEC];
                unpack_w(wr[k][c], w);
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    w[e] = fmaf(lr_signed, update_ratio(comp(v[k][c], e), den), w[e]);
                store_w<BF16, VEC>(W, i * D + (int64_t)col * VEC, w);
            }
        }
    }

    // column partial of this CTA: row groups combined in order 0 .. rg-1
    float *out = colpart + (int64_t)blockIdx.x * D;
    if (rg == 1) {
#pragma unroll
        for (int c = 0; c < CPT; ++c) {
            const int col = l + c * tpr;
            if (col < DV)
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    out[col * VEC + e] = acc[c][e];
        }
    } else {
        float *colsh = reinterpret_cast<float *>(ro_dyn + (ASYNC ? rowonly_stage_bytes<CPT, R, BF16>() : 0));
        combine_row_groups<VEC, CPT>(acc, colsh, out, D, DV, tpr, rg, g, l);  // rg x D floats
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
    if (lane == 0)
        rsum_sh[warp] = rsum;
    __syncthreads();
    if (tid == 0) {
        float t = 0.f;
        for (int q = 0; q < kWarps; ++q)
            t += rsum_sh[q];
        rsum_part[blockIdx.x] = t;
    }
}

// ---------------------------------------------------------------------------
// Row-sharded step, phases 1 and 2 (after the shard's reduce launch, whose
// ncta partial rows sit in the shard's workspace).
//   k_shard_scales: per column (and, at index D, for the per-CTA sums of r)
//       the largest key among the shard's partials -> scales[0..D].
//   k_shard_pack: per column the fixed-point sum of the shard's partials at
//       the all-reduced scales -> sums[0..D].
// One thread per column; the partial rows are read with coalesced loads.
// ---------------------------------------------------------------------------
__global__ void k_shard_scales(const float *__restrict__ colpart, const float *__restrict__ rsum_part, int ncta,
                               int D, unsigned char *__restrict__ scales)
{
    grid_dep_wait();
    grid_dep_launch();
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j <= D; j += gridDim.x * blockDim.x) {
        unsigned e = 0;
        for (int b = 0; b < ncta; ++b)
            e = max(e, fx_key(j < D ? __ldcg(colpart + (int64_t)b * D + j) : __ldcg(rsum_part + b)));
        scales[j] = (unsigned char)e;
    }
}

__global__ void k_shard_pack(const float *__restrict__ colpart, const float *__restrict__ rsum_part, int ncta,
                             int D, const unsigned char *__restrict__ scales, unsigned long long *__restrict__ sums)
{
    grid_dep_wait();
    grid_dep_launch();
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j <= D; j += gridDim.x * blockDim.x) {
        const unsigned E = scales[j];
        unsigned long long s = 0;
        for (int b = 0; b < ncta; ++b)
            s += fx_of(j < D ? __ldcg(colpart + (int64_t)b * D + j) : __ldcg(rsum_part + b), E);
        sums[j] = s;
    }
}

// R1: rows per thread of the reduce pass, reduce_rows_per_thread(V, D, map)
template <int VEC, int CPT, int R1>
cudaError_t launch_dense_t(const DenseArgs &a)
{
    constexpr int R3 = (8 / CPT) < 1 ? 1 : (8 / CPT);
    const int nparts = dense_parts(a.V, a.D);
    const int D = (int)a.D;
    DevScalars *sc = reinterpret_cast<DevScalars *>(a.ws + a.lay.scalars);
    float *rsum_part = reinterpret_cast<float *>(a.ws + a.lay.rsum_part);
    float *csum_part = reinterpret_cast<float *>(a.ws + a.lay.csum_part);
    const StepConsts kc = make_consts(a.beta2, a.one_minus_beta2, a.V, a.D, a.inv_bc);
    float *colpart = reinterpret_cast<float *>(a.ws + a.lay.colpart);
    const int rg = kThreads / a.map.tpr;
    // column panels (one unless D is wider than a CTA's row): columns
    // [q pw, q pw + cols(q)) with row stride D
    const int np = a.map.npanels;
    const int pw = a.map.pw;
    const int ld = (int)a.D;
    auto cols = [&](int q) { return (q + 1 < np) ? pw : (int)(a.D - (int64_t)q * pw); };
    const size_t shmem = (rg > 1) ? (size_t)rg * pw * sizeof(float) : 0;  // the row groups' column sums

    // With tracing, events sit between the kernels and each launch simply
    // follows the previous one; without, kernels 2 and 3 use programmatic
    // dependent launch.
    const bool pdl = (a.trace == nullptr);
    cudaError_t e;
    RowSpan span{0, nparts, 0};
    if (a.shard) {
        // one phase of a row-sharded step: the shard's own CTAs of the
        // whole-table grid, so each per-CTA partial equals the unsharded one
        const ShardArgs &sh = *a.shard;
        if (np != 1)
            return cudaErrorInvalidValue;  // refused by the entry points
        const int ncta = sh.cta_end - sh.cta_begin;
        span = RowSpan{sh.cta_begin, nparts, sh.row_base};
        const int nthr = 256;
        const int nblk = (D + 1 + nthr - 1) / nthr;
        if (sh.phase == 1) {
            if (ncta > 0) {
                e = launch_k(k_reduce_dense<VEC, CPT, R1, false>, dim3(ncta), dim3(kThreads), shmem, a.stream, false,
                             a.G, a.r, colpart, rsum_part, a.V, D, ld, a.map.tpr, kc,
                             nullptr, nullptr, span);
                if (e != cudaSuccess)
                    return e;
            }
            e = launch_k(k_shard_scales, dim3(nblk), dim3(nthr), 0, a.stream, false, colpart, rsum_part, ncta, D,
                         sh.scales);
            return e != cudaSuccess ? e : cudaGetLastError();
        }
        if (sh.phase == 2) {
            e = launch_k(k_shard_pack, dim3(nblk), dim3(nthr), 0, a.stream, false, colpart, rsum_part, ncta, D,
                         sh.scales, sh.sums);
            return e != cudaSuccess ? e : cudaGetLastError();
        }
        const ColSource src{nullptr, 0, sh.sums, sh.scales};
        e = launch_k(k_state_dense, dim3((D + kStateCols - 1) / kStateCols), dim3(kStateThreads), 0, a.stream,
                     false, src, rsum_part, 0, a.c, csum_part, sc, a.V, D, kc,
                     RowPass{nullptr, nullptr, nullptr, 0, 0, nullptr, 0});
        if (e != cudaSuccess || ncta == 0)
            return e != cudaSuccess ? e : cudaGetLastError();
        const size_t cs_bytes = (size_t)D * sizeof(float);
        if (a.wbf16)
            e = launch_k(k_apply_dense<VEC, CPT, R3, true>, dim3(ncta), dim3(kThreads), cs_bytes, a.stream, pdl,
                         a.W, a.G, a.r, a.c, sc, a.V, D, ld, a.map.tpr, kc.inv_bc, a.eps, a.lr_signed,
                         a.variant, span);
        else
            e = launch_k(k_apply_dense<VEC, CPT, R3, false>, dim3(ncta), dim3(kThreads), cs_bytes, a.stream, pdl,
                         a.W, a.G, a.r, a.c, sc, a.V, D, ld, a.map.tpr, kc.inv_bc, a.eps, a.lr_signed,
                         a.variant, span);
        return e != cudaSuccess ? e : cudaGetLastError();
    }
    if (a.variant == EMBER_VARIANT_ROW && !a.lm && np == 1) {
        // one pass over G and W, then the column state; no apply pass
        constexpr int RR = (4 / CPT) < 1 ? 1 : (4 / CPT);
        constexpr bool kAsync = VEC == 4;
        if (a.trace)
            cudaEventRecord(a.trace[0], a.stream);
        if (a.wbf16) {
            auto *k = k_rowonly_dense<VEC, CPT, RR, true, kAsync>;
            const size_t sm = shmem + (kAsync ? rowonly_stage_bytes<CPT, RR, true>() : 0);
            e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            if (e == cudaSuccess)
                e = launch_k(k, dim3(nparts), dim3(kThreads), sm, a.stream, false, a.W, a.G, a.r, colpart,
                             rsum_part, a.V, D, a.map.tpr, kc, a.eps,
                             a.lr_signed);
        } else {
            auto *k = k_rowonly_dense<VEC, CPT, RR, false, kAsync>;
            const size_t sm = shmem + (kAsync ? rowonly_stage_bytes<CPT, RR, false>() : 0);
            e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            if (e == cudaSuccess)
                e = launch_k(k, dim3(nparts), dim3(kThreads), sm, a.stream, false, a.W, a.G, a.r, colpart,
                             rsum_part, a.V, D, a.map.tpr, kc, a.eps,
                             a.lr_signed);
        }
        if (e != cudaSuccess)
            return e;
        if (a.trace)
            cudaEventRecord(a.trace[1], a.stream);
        e = launch_state(colpart, nparts, rsum_part, nparts, a.c, csum_part, sc, a.V, D, kc, a.stream, pdl, nullptr, nullptr, nullptr, 0, 0);
        if (e != cudaSuccess)
            return e;
        if (a.trace) {
            cudaEventRecord(a.trace[2], a.stream);
            cudaEventRecord(a.trace[3], a.stream);
        }
        return cudaGetLastError();
    }
    if constexpr (VEC == 4) {
        int nits = 0;
        size_t sm = 0;
        if (!a.lm && !a.G_stage && !a.trace && small_table_plan(a.V, a.D, a.wbf16 != 0, a.map, &nits, &sm)) {
            // a small table: the whole step in one cluster launch, the kept
            // G and W in shared memory
            auto *k = a.wbf16 ? k_dense_cluster<CPT, R1, true> : k_dense_cluster<CPT, R1, false>;
            e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            if (e == cudaSuccess && nparts > 8)
                e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
            if (e != cudaSuccess)
                return e;
            SmallArgs sa{a.W, a.G, a.r, a.c, sc, a.V, D, a.map.tpr, nits, kc, a.eps, a.lr_signed, a.variant};
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(nparts);
            cfg.blockDim = dim3(kThreads);
            cfg.dynamicSmemBytes = sm;
            cfg.stream = a.stream;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = nparts;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            e = cudaLaunchKernelEx(&cfg, k, sa);
            return e != cudaSuccess ? e : cudaGetLastError();
        }
    }
    if (a.lm) {
        // G comes from the LM-head kernel, which also leaves the sums of g^2
        // per 128-row block (columns) and per 256-column block (rows); the
        // state pass finishes both, then the apply pass reads G once.
        float *lm_col = reinterpret_cast<float *>(a.ws + a.lay.lm_colpart);
        float *lm_row = reinterpret_cast<float *>(a.ws + a.lay.lm_rowpart);
        if (a.trace)
            cudaEventRecord(a.trace[0], a.stream);
        e = launch_lmhead_grad(*a.lm, lm_col, lm_row, &sc->flags, a.stream);
        if (e != cudaSuccess)
            return e;
        if (a.trace)
            cudaEventRecord(a.trace[1], a.stream);
        // plain stream order after the tensor-core kernel: launched early,
        // the state grid made the step slower (measured 0.1-0.3 ms)
        const int64_t vb = (a.V + kStateThreads - 1) / kStateThreads;
        const int nrow_ctas = (int)(vb < kMaxRowCtas ? vb : kMaxRowCtas);
        e = launch_state(lm_col, lmhead_row_blocks(a.V), rsum_part, nrow_ctas, a.c, csum_part, sc, a.V, D,
                         kc, a.stream, false, a.r, nullptr, lm_row,
                         lmhead_col_blocks(a.D), nrow_ctas);
        if (e != cudaSuccess)
            return e;
    } else {
        // with several column panels each reduce launch leaves its rows' sums
        // of g^2 over the panel in rowpart[q][V] (the LM-head step's region),
        // and the state pass adds them up per row in panel order
        float *rowpart = (np > 1) ? reinterpret_cast<float *>(a.ws + a.lay.lm_rowpart) : nullptr;
        if (a.trace)
            cudaEventRecord(a.trace[0], a.stream);
        for (int q = 0; q < np; ++q) {
            const int64_t c0 = (int64_t)q * pw;
            float *rp = rowpart ? rowpart + (int64_t)q * a.V : nullptr;
            if (a.G_stage)
                e = launch_k(k_reduce_dense<VEC, CPT, R1, true>, dim3(nparts), dim3(kThreads), shmem, a.stream,
                             pdl && q > 0, a.G + c0, a.r, colpart + c0, rsum_part, a.V, cols(q), ld, a.map.tpr,
                             kc, a.G_stage + c0, rp, span);
            else
                e = launch_k(k_reduce_dense<VEC, CPT, R1, false>, dim3(nparts), dim3(kThreads), shmem, a.stream,
                             pdl && q > 0, a.G + c0, a.r, colpart + c0, rsum_part, a.V, cols(q), ld, a.map.tpr,
                             kc, nullptr, rp, span);
            if (e != cudaSuccess)
                return e;
        }
        if (a.trace)
            cudaEventRecord(a.trace[1], a.stream);
        if (np == 1) {
            e = launch_state(colpart, nparts, rsum_part, nparts, a.c, csum_part, sc, a.V, D, kc, a.stream, pdl, nullptr, nullptr, nullptr, 0, 0);
        } else {
            const int64_t vb = (a.V + kStateThreads - 1) / kStateThreads;
            const int nrow_ctas = (int)(vb < kMaxRowCtas ? vb : kMaxRowCtas);
            e = launch_state(colpart, nparts, rsum_part, nrow_ctas, a.c, csum_part, sc, a.V, D, kc, a.stream, pdl, a.r, nullptr, rowpart, np, nrow_ctas);
        }
        if (e != cudaSuccess)
            return e;
    }
    // the apply pass reads the staged copy, or the G the LM-head kernel wrote;
    // panels from the last (the reduce pass's last rows, still in L2)
    const float *Gd = a.lm ? a.lm->G : a.G_stage ? a.G_stage : a.G;
    if (a.trace)
        cudaEventRecord(a.trace[2], a.stream);
    const size_t cs_bytes = (size_t)pw * sizeof(float);
    for (int q = np - 1; q >= 0; --q) {
        const int64_t c0 = (int64_t)q * pw;
        void *Wq = static_cast<unsigned char *>(a.W) + c0 * (a.wbf16 ? 2 : 4);
        if (a.wbf16)
            e = launch_k(k_apply_dense<VEC, CPT, R3, true>, dim3(nparts), dim3(kThreads), cs_bytes,
                         a.stream, pdl, Wq, Gd + c0, a.r, a.c + c0, sc, a.V, cols(q), ld, a.map.tpr,
                         kc.inv_bc, a.eps, a.lr_signed, a.variant, span);
        else
            e = launch_k(k_apply_dense<VEC, CPT, R3, false>, dim3(nparts), dim3(kThreads), cs_bytes,
                         a.stream, pdl, Wq, Gd + c0, a.r, a.c + c0, sc, a.V, cols(q), ld, a.map.tpr,
                         kc.inv_bc, a.eps, a.lr_signed, a.variant, span);
        if (e != cudaSuccess)
            return e;
    }
    if (a.trace)
        cudaEventRecord(a.trace[3], a.stream);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_state(const float *colpart, int nparts, float *rsum_part, int nrsum, float *c,
                         float *csum_part, DevScalars *sc, int64_t V, int D, const StepConsts &kc,
                         cudaStream_t stream, bool pdl, float *r_rows, int32_t *slot, const float *rowpart,
                         int nslices, int nrow_ctas, const int32_t *uniq, int rsum_base, int pstride, int pcols)
{
    const int ngroups = (D + kStateCols - 1) / kStateCols;
    RowPass rp{r_rows, slot, rowpart, nslices, nrow_ctas, uniq, rsum_base};
    const ColSource src{colpart, nparts, nullptr, nullptr, pstride, pcols};
    return launch_k(k_state_dense, dim3(ngroups + nrow_ctas), dim3(kStateThreads), 0, stream, pdl, src,
                    rsum_part, nrsum, c, csum_part, sc, V, D, kc, rp);
}

bool choose_colmap(int64_t D, bool vec4_ok, ColMap *m)
{
    if (D < 1 || D > kMaxCols)
        return false;
    const int vec = (vec4_ok && D % 4 == 0) ? 4 : 1;
    // equal panels of at most kThreads * 8 accesses, widths a multiple of vec
    const int64_t maxw = (int64_t)kThreads * 8 * vec;
    const int64_t np = (D + maxw - 1) / maxw;
    const int64_t pw = ((D + np - 1) / np + vec - 1) / vec * vec;
    m->npanels = (int)((D + pw - 1) / pw);
    m->pw = (int)pw;
    const int64_t DV = pw / vec;
    for (int tpr = 32; tpr <= kThreads; tpr *= 2) {
        const int64_t need = (DV + tpr - 1) / tpr;
        if (need <= 4 || tpr == kThreads) {
            int cpt = 1;
            while (cpt < need)
                cpt *= 2;
            if (cpt > 8)
                return false;
            m->vec = vec;
            m->tpr = tpr;
            m->cpt = cpt;
            return true;
        }
    }
    return false;
}

cudaError_t launch_dense_step(const DenseArgs &a)
{
    if (a.map.vec == 4) {
        const bool half = reduce_rows_per_thread(a.V, a.D, a.map) == 8;
        switch (a.map.cpt) {
        case 1: return half ? launch_dense_t<4, 1, 8>(a) : launch_dense_t<4, 1, 16>(a);
        case 2: return launch_dense_t<4, 2, 8>(a);
        case 4: return launch_dense_t<4, 4, 4>(a);
        case 8: return launch_dense_t<4, 8, 2>(a);
        }
    } else {
        const bool half = reduce_rows_per_thread(a.V, a.D, a.map) == 8;
        switch (a.map.cpt) {
        case 1: return half ? launch_dense_t<1, 1, 8>(a) : launch_dense_t<1, 1, 16>(a);
        case 2: return launch_dense_t<1, 2, 8>(a);
        case 4: return launch_dense_t<1, 4, 4>(a);
        case 8: return launch_dense_t<1, 8, 2>(a);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace ember
