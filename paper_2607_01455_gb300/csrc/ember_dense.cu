// Dense Ember step (Algorithm 1 of "Token Geometry", arXiv 2607.01455,
// Section 2.1) for sm_103a.
//
// The step needs two passes over the fp32 gradient G: the update of any
// element needs chat_j and s, which depend on every row of G (Section 2.3
// builds both statistics from sums of g^2).  The passes are:
//
//   reduce  (k_reduce_dense)  one read of G.  Per row: sum_j g^2, the row EMA
//           r_i <- beta2 r_i + (1-beta2) mean_j g^2 (Algorithm 1's row second
//           moment), written once.  Per CTA: column sums of g^2 over its rows
//           and the sum of its new r values, written to the workspace.
//   state   (k_state_dense)   O(D * CTAs) work: column sums in a fixed order,
//           the column EMA c_j <- beta2 c_j + (1-beta2) mean_i g^2, then the
//           last CTA forms mean(rhat), mean(chat) and s = sqrt(mean rhat *
//           mean chat) (the geometric-mean normaliser).
//   apply   (k_apply_dense)   reads G and W, writes W:
//           W_ij <- W_ij - lr g_ij / (sqrt(rhat_i) sqrt(chat_j / s) + eps),
//           the factored preconditioner applied as a row scale times a
//           column scale, never stored (Section 2.3).
//
// Bandwidth: 4VD bytes (reduce) + 4VD + 2 w VD bytes (apply), w = bytes per
// weight.  The apply pass walks each CTA's rows in the reverse order of the
// reduce pass, so the rows read last by the reduce pass -- still in L2 --
// are the first ones it needs.
//
// Determinism: no floating-point atomics.  Every CTA owns a fixed row range
// (a function of V only), every in-CTA sum has a fixed shape, and the
// cross-CTA sums run in CTA order, so W and the state are bit-identical
// from run to run, as Section 2.3 requires.
//
// The same launcher also runs:
//   - the row-only variant in one pass (k_rowonly_dense), no apply pass;
//   - the LM-head step: the tensor-core kernel of ember_lmhead.cu forms G and
//     its per-tile sums of g^2, the state pass finishes them (row pass from
//     per-column-block sums), then the apply pass;
//   - the two phases of a row-sharded step: the reduce pass or the apply
//     pass over one shard's CTAs of the whole-table grid (RowSpan), and the
//     state pass on every shard's gathered partials.
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

// Pass 1: one read of G.  Template: VEC columns per access, CPT accesses per
// thread per row, R rows per row group per iteration.
// STAGE: G is read from host memory the GPU can address (over the
// Grace-Blackwell chip-to-chip link) and every element is also written to
// G_stage in HBM for the apply pass.
// D is the number of columns this launch covers and ld the row stride of G
// and colpart: a column panel of a wider table has D < ld, and then each
// row's sum of g^2 over the panel goes to rowpart[i] instead of into r.
template <int VEC, int CPT, int R, bool STAGE>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_reduce_dense(const float *__restrict__ G, float *__restrict__ r,
               float *__restrict__ colpart, double *__restrict__ rsum_part,
               int64_t V, int D, int ld, int tpr, double beta2, double one_minus_beta2,
               float *__restrict__ G_stage, float *__restrict__ rowpart, RowSpan span)
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
    const int64_t row0 = (int64_t)(span.cta_base + blockIdx.x) * V / span.nparts;
    const int64_t row1 = (int64_t)(span.cta_base + blockIdx.x + 1) * V / span.nparts;

    grid_dep_wait();    // the first kernel of a step: returns at once
    grid_dep_launch();  // the state pass may start launching now; it waits for this grid

    // per-warp row sums of up to kRowBuf rows, finalised together
    constexpr int kRowBuf = 128;
    __shared__ float red[kWarps][kRowBuf];
    __shared__ double rsum_sh[kWarps];

    float acc[CPT][VEC];
#pragma unroll
    for (int c = 0; c < CPT; ++c)
#pragma unroll
        for (int e = 0; e < VEC; ++e)
            acc[c][e] = 0.f;
    double rsum = 0.0;

    const int rows_per_it = rg * R;               // rows of one iteration
    const int its_per_buf = kRowBuf / rows_per_it;  // >= 1: rg * R <= 128
    int64_t buf_base = row0;
    int nbuf = 0;  // iterations held in the buffer
    for (int64_t base = row0; base < row1; base += rows_per_it) {
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
                    const double mean_row = (double)sum / (double)D;
                    const float rn = (float)(beta2 * (double)r[i] + one_minus_beta2 * mean_row);
                    r[i] = rn;
                    rsum += (double)rn;
                }
            }
            __syncthreads();
            buf_base += (int64_t)nbuf * rows_per_it;
            nbuf = 0;
        }
    }

    // column partial of this CTA: row groups combined in order 0 .. rg-1
    float *out = colpart + (int64_t)blockIdx.x * ld;
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
        extern __shared__ float colsh[];  // D floats
        for (int q = 0; q < rg; ++q) {
            if (g == q) {
#pragma unroll
                for (int c = 0; c < CPT; ++c) {
                    const int col = l + c * tpr;
                    if (col < DV)
#pragma unroll
                        for (int e = 0; e < VEC; ++e)
                            colsh[col * VEC + e] = (q == 0) ? acc[c][e] : colsh[col * VEC + e] + acc[c][e];
                }
            }
            __syncthreads();
        }
        for (int j = tid; j < D; j += kThreads)
            out[j] = colsh[j];
    }

    // sum of the new r values of this CTA: fixed butterfly per warp, warps in order
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
    if (lane == 0)
        rsum_sh[warp] = rsum;
    __syncthreads();
    if (tid == 0 && rowpart == nullptr) {
        double s = 0.0;
        for (int q = 0; q < kWarps; ++q)
            s += rsum_sh[q];
        rsum_part[blockIdx.x] = s;
    }
}

// beta2 r + (1 - beta2) m in fp32, each coefficient carried as a float pair
// hi + lo (hi the coefficient rounded to fp32, lo the rest): within about an
// ulp of the fp64 value, and the fixed point stays at r = m, which rounding
// beta2 and 1 - beta2 to single floats would shift by about 1e-5 of r at
// beta2 = 0.999.  With m = 0 (a row outside a sparse batch) it is the
// correctly rounded product beta2 r in all but near-tie cases.
struct EmaPair {
    float bh, bl, ah, al;
};
__device__ __forceinline__ EmaPair make_ema_pair(double beta2, double one_minus_beta2)
{
    EmaPair e;
    e.bh = (float)beta2;
    e.bl = (float)(beta2 - (double)e.bh);
    e.ah = (float)one_minus_beta2;
    e.al = (float)(one_minus_beta2 - (double)e.ah);
    return e;
}
__device__ __forceinline__ float ema_pair(const EmaPair &e, float r, float m)
{
    return fmaf(e.bh, r, fmaf(e.bl, r, fmaf(e.ah, m, e.al * m)));
}

// Pass 2: column EMA and the normaliser.  The first nstate CTAs each own
// columns [32x, 32x + 32); warp w sums the partials of CTAs w, w+8, ... in
// order.  For the sparse step the remaining CTAs also do the row pass: r for
// every row (rows outside the batch see a zero gradient row, touched rows
// take their sum of g^2 per column slice from `rowpart`) and the sum of the
// new r per CTA.  The last CTA to finish forms mean(rhat), mean(chat) and s.
struct RowPass {
    float *r;               // r[V], updated (sparse step only)
    int32_t *slot;          // touched-row map, cleared here
    const float *rowpart;   // per (distinct id, slice) sums of g^2
    int nslices;
    int nrow_ctas;          // 0 for the dense step
};

__global__ void __launch_bounds__(kStateThreads)
k_state_dense(const float *__restrict__ colpart, int nparts, double *__restrict__ rsum_part,
              int nrsum, float *__restrict__ c, double *__restrict__ csum_part, DevScalars *sc,
              int64_t V, int D, double beta2, double one_minus_beta2, double inv_bc, RowPass rowp)
{
    constexpr int kW = kStateThreads / 32;
    const int lane = threadIdx.x & 31;
    const int w = threadIdx.x >> 5;
    const int nstate = (int)gridDim.x - rowp.nrow_ctas;
    __shared__ float part[kW][32];
    __shared__ double part_last[kW][2];
    __shared__ bool am_last;
    // GB300 runs fp64 at a small fraction of its fp32 rate, and a single
    // fp64 pipe op per row or column showed up in this kernel's time: the
    // per-CTA work is fp32 (the EMAs with float-pair coefficients, sums of
    // at most a few thousand values per CTA in fixed trees), and only the
    // sums across CTAs and the normaliser run in fp64.
    const double inv_D = 1.0 / (double)D, inv_V = 1.0 / (double)V;
    const EmaPair ema = make_ema_pair(beta2, one_minus_beta2);
    grid_dep_wait();  // column partials and row sums of the earlier passes
    grid_dep_launch();

    if ((int)blockIdx.x < nstate) {
        const int j = blockIdx.x * kStateCols + lane;
        // rows w, w + 8, w + 16, ...: 32 loads in flight, summed pairwise
        // within the batch, then across batches and warps in order
        constexpr int kBatch = 32;
        float acc = 0.f;
        if (j < D)
            for (int b0 = w; b0 < nparts; b0 += kBatch * kW) {
                float v[kBatch];
#pragma unroll
                for (int k = 0; k < kBatch; ++k) {
                    const int b = b0 + k * kW;
                    v[k] = (b < nparts) ? __ldcg(colpart + (int64_t)b * D + j) : 0.f;
                }
#pragma unroll
                for (int h = kBatch / 2; h >= 1; h >>= 1)
#pragma unroll
                    for (int k = 0; k < h; ++k)
                        v[k] += v[k + h];
                acc += v[0];
            }
        part[w][lane] = acc;
        __syncthreads();
        if (w == 0) {
            float tot = 0.f;
#pragma unroll
            for (int q = 0; q < kW; ++q)
                tot += part[q][lane];
            float cn = 0.f;
            if (j < D) {
                const float cnew = ema_pair(ema, c[j], tot * (float)inv_V);
                c[j] = cnew;
                cn = cnew;
            }
#pragma unroll
            for (int o = 16; o >= 1; o >>= 1)
                cn += __shfl_xor_sync(0xffffffffu, cn, o);
            if (lane == 0)
                csum_part[blockIdx.x] = (double)cn;
        }
    } else {
        const int rb = (int)blockIdx.x - nstate;
        const int64_t stride = (int64_t)rowp.nrow_ctas * kStateThreads;
        // Every row of the table: the row EMA (ema_pair), then the CTA's sum
        // of the new r in fp32 (thread, warp butterfly, warps in order).
        const float inv_Df = (float)inv_D;
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
            // sparse step: kRowBatch rows per thread at a time, their map
            // entries and r loaded together; rows outside the batch's ids
            // decay, touched rows add their sums of g^2
            for (int64_t i0 = (int64_t)rb * kStateThreads + threadIdx.x; i0 < V; i0 += stride * kRowBatch) {
                int sl[kRowBatch];
                float rr[kRowBatch];
#pragma unroll
                for (int k = 0; k < kRowBatch; ++k) {
                    const int64_t i = i0 + k * stride;
                    sl[k] = (i < V) ? rowp.slot[i] : 0;
                    rr[k] = (i < V) ? rowp.r[i] : 0.f;
                }
                float tsum = 0.f;
#pragma unroll
                for (int k = 0; k < kRowBatch; ++k) {
                    const int64_t i = i0 + k * stride;
                    if (i >= V)
                        break;
                    float mean_row = 0.f;
                    if (sl[k]) {
                        const int64_t u = sl[k] - 1;
                        float tot = 0.f;
                        for (int q = 0; q < rowp.nslices; ++q)
                            tot += rowp.rowpart[u * rowp.nslices + q];
                        mean_row = tot * inv_Df;
                        rowp.slot[i] = 0;
                    }
                    const float rn = ema_pair(ema, rr[k], mean_row);
                    rowp.r[i] = rn;
                    tsum += rn;
                }
                rsum += tsum;
            }
        }
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1)
            rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
        if (lane == 0)
            part[w][0] = rsum;
        __syncthreads();
        if (threadIdx.x == 0) {
            float t = 0.f;
            for (int q = 0; q < kW; ++q)
                t += part[q][0];
            rsum_part[rb] = (double)t;
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
    // The last CTA: thread t sums entries t, t + 256, ... in order (all its
    // loads in flight at once), then a fixed butterfly per warp and the
    // warps in order.
    double csum = 0.0, rsum = 0.0;
    for (int b = threadIdx.x; b < nstate; b += kStateThreads)
        csum += __ldcg(csum_part + b);
    for (int b = threadIdx.x; b < nrsum; b += kStateThreads)
        rsum += __ldcg(rsum_part + b);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        csum += __shfl_xor_sync(0xffffffffu, csum, o);
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
    }
    if (lane == 0) {
        part_last[w][0] = csum;
        part_last[w][1] = rsum;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        csum = 0.0;
        rsum = 0.0;
        for (int q = 0; q < kW; ++q) {
            csum += part_last[q][0];
            rsum += part_last[q][1];
        }
        const double rbar = rsum * inv_bc * inv_V;
        const double cbar = csum * inv_bc * inv_D;
        const double s = sqrt(rbar * cbar);
        sc->s = s;
        sc->rbar = rbar;
        sc->cbar = cbar;
        sc->inv_s = (s > 0.0) ? (float)(1.0 / s) : 0.f;
        sc->ticket = 0u;
    }
}

// Pass 3: the update.  Same row ranges and column mapping as pass 1; each
// CTA walks its rows from the last iteration block to the first.  The
// column scales live in shared memory (D floats).  D columns from row stride
// ld, as in pass 1: W, G and c point at the first column of the panel.
template <int VEC, int CPT, int R, bool BF16>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
k_apply_dense(void *__restrict__ W, const float *__restrict__ G, const float *__restrict__ r,
              const float *__restrict__ c, const DevScalars *__restrict__ sc,
              int64_t V, int D, int ld, int tpr, float inv_bc, float eps, float lr_signed, int variant,
              RowSpan span)
{
    using F = typename Vec<VEC>::F;
    using WT = typename WRaw<BF16, VEC>::T;
    extern __shared__ float cs[];  // D column scales
    const int DV = D / VEC;
    const int tid = threadIdx.x;
    const int rg = kThreads / tpr;
    const int g = tid / tpr;
    const int l = tid - g * tpr;
    const int64_t row0 = (int64_t)(span.cta_base + blockIdx.x) * V / span.nparts;
    const int64_t row1 = (int64_t)(span.cta_base + blockIdx.x + 1) * V / span.nparts;
    const int64_t step = (int64_t)rg * R;
    const int64_t nblocks = (row1 - row0 + step - 1) / step;

    // While the state pass finishes: pull this thread's first rows of G and
    // W (the last iteration block, walked first) towards L2.
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
    grid_dep_wait();  // c, s (state pass) and r (reduce pass)
    grid_dep_launch();

    // column scale sqrt(chat_j / s) (FULL), sqrt(chat_j) (COL) or 1 (ROW)
    const float inv_s = (variant == EMBER_VARIANT_FULL) ? sc->inv_s : 1.f;
    for (int j = tid; j < D; j += kThreads)
        cs[j] = (variant == EMBER_VARIANT_ROW) ? 1.f : sqrtf(c[j] * inv_bc * inv_s);
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
            const float rs = (variant == EMBER_VARIANT_COL) ? 1.f : sqrtf(__ldg(r + i) * inv_bc);
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
                    const float u = comp(gv[k][cc], e) / den;
                    w[e] = fmaf(lr_signed, u, w[e]);
                }
                store_w<BF16, VEC>(W, (i - span.row_base) * ld + (int64_t)col * VEC, w);
            }
        }
    }
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
                float *__restrict__ colpart, double *__restrict__ rsum_part, int64_t V, int D, int tpr,
                double beta2, double one_minus_beta2, float inv_bc, float eps, float lr_signed)
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
    __shared__ double rsum_sh[kWarps];
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
    double rsum = 0.0;
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
                const double mean_row = (double)sum / (double)D;
                const float rn = (float)(beta2 * (double)r[i] + one_minus_beta2 * mean_row);
                r[i] = rn;
                rsum += (double)rn;
                rsv = sqrtf(rn * inv_bc);
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
                    w[e] = fmaf(lr_signed, comp(v[k][c], e) / den, w[e]);
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
        for (int q = 0; q < rg; ++q) {
            if (g == q) {
#pragma unroll
                for (int c = 0; c < CPT; ++c) {
                    const int col = l + c * tpr;
                    if (col < DV)
#pragma unroll
                        for (int e = 0; e < VEC; ++e)
                            colsh[col * VEC + e] = (q == 0) ? acc[c][e] : colsh[col * VEC + e] + acc[c][e];
                }
            }
            __syncthreads();
        }
        for (int j = tid; j < D; j += kThreads)
            out[j] = colsh[j];
    }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1)
        rsum += __shfl_xor_sync(0xffffffffu, rsum, o);
    if (lane == 0)
        rsum_sh[warp] = rsum;
    __syncthreads();
    if (tid == 0) {
        double t = 0.0;
        for (int q = 0; q < kWarps; ++q)
            t += rsum_sh[q];
        rsum_part[blockIdx.x] = t;
    }
}

// Row-sharded step: copy the per-CTA partials of every shard's exchange
// block (CTA b is entry b % cap of shard b / cap) into the workspace layout
// of the whole-table step, in CTA order.
__global__ void k_shard_unpack(const unsigned char *__restrict__ blocks, size_t block_bytes, size_t block_rsum,
                               int cap, int nparts, int D, float *__restrict__ colpart,
                               double *__restrict__ rsum_part)
{
    grid_dep_wait();
    grid_dep_launch();
    const int64_t total = (int64_t)nparts * D;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total;
         q += (int64_t)gridDim.x * blockDim.x) {
        const int b = (int)(q / D);
        const int j = (int)(q - (int64_t)b * D);
        const float *src = reinterpret_cast<const float *>(blocks + (size_t)(b / cap) * block_bytes);
        colpart[q] = src[(int64_t)(b % cap) * D + j];
    }
    for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < nparts; b += gridDim.x * blockDim.x)
        rsum_part[b] = reinterpret_cast<const double *>(blocks + (size_t)(b / cap) * block_bytes + block_rsum)[b % cap];
}

template <int VEC, int CPT>
cudaError_t launch_dense_t(const DenseArgs &a)
{
    constexpr int R1 = (16 / CPT) < 1 ? 1 : (16 / CPT);
    constexpr int R3 = (8 / CPT) < 1 ? 1 : (8 / CPT);
    const int nparts = dense_parts(a.V);
    const int D = (int)a.D;
    DevScalars *sc = reinterpret_cast<DevScalars *>(a.ws + a.lay.scalars);
    double *rsum_part = reinterpret_cast<double *>(a.ws + a.lay.rsum_part);
    double *csum_part = reinterpret_cast<double *>(a.ws + a.lay.csum_part);
    float *colpart = reinterpret_cast<float *>(a.ws + a.lay.colpart);
    const int rg = kThreads / a.map.tpr;
    // column panels (one unless D is wider than a CTA's row): columns
    // [q pw, q pw + cols(q)) with row stride D
    const int np = a.map.npanels;
    const int pw = a.map.pw;
    const int ld = (int)a.D;
    auto cols = [&](int q) { return (q + 1 < np) ? pw : (int)(a.D - (int64_t)q * pw); };
    const size_t shmem = (rg > 1) ? (size_t)pw * sizeof(float) : 0;

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
        if (sh.phase == 1) {
            if (ncta == 0)
                return cudaSuccess;
            float *bcol = static_cast<float *>(sh.block);
            double *brsum = reinterpret_cast<double *>(static_cast<unsigned char *>(sh.block) + sh.block_rsum);
            e = launch_k(k_reduce_dense<VEC, CPT, R1, false>, dim3(ncta), dim3(kThreads), shmem, a.stream, false,
                         a.G, a.r, bcol, brsum, a.V, D, ld, a.map.tpr, a.beta2, a.one_minus_beta2, nullptr,
                         nullptr, span);
            return e != cudaSuccess ? e : cudaGetLastError();
        }
        e = launch_k(k_shard_unpack, dim3(kGridCtas), dim3(kThreads), 0, a.stream, false,
                     static_cast<const unsigned char *>(sh.blocks), sh.block_bytes, sh.block_rsum, sh.cap, nparts, D,
                     colpart, rsum_part);
        if (e != cudaSuccess)
            return e;
        e = launch_state(colpart, nparts, rsum_part, nparts, a.c, csum_part, sc, a.V, D, a.beta2,
                         a.one_minus_beta2, a.inv_bc, a.stream, pdl, nullptr, nullptr, nullptr, 0, 0);
        if (e != cudaSuccess || ncta == 0)
            return e != cudaSuccess ? e : cudaGetLastError();
        const size_t cs_bytes = (size_t)D * sizeof(float);
        if (a.wbf16)
            e = launch_k(k_apply_dense<VEC, CPT, R3, true>, dim3(ncta), dim3(kThreads), cs_bytes, a.stream, pdl,
                         a.W, a.G, a.r, a.c, sc, a.V, D, ld, a.map.tpr, (float)a.inv_bc, a.eps, a.lr_signed,
                         a.variant, span);
        else
            e = launch_k(k_apply_dense<VEC, CPT, R3, false>, dim3(ncta), dim3(kThreads), cs_bytes, a.stream, pdl,
                         a.W, a.G, a.r, a.c, sc, a.V, D, ld, a.map.tpr, (float)a.inv_bc, a.eps, a.lr_signed,
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
                             rsum_part, a.V, D, a.map.tpr, a.beta2, a.one_minus_beta2, (float)a.inv_bc, a.eps,
                             a.lr_signed);
        } else {
            auto *k = k_rowonly_dense<VEC, CPT, RR, false, kAsync>;
            const size_t sm = shmem + (kAsync ? rowonly_stage_bytes<CPT, RR, false>() : 0);
            e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            if (e == cudaSuccess)
                e = launch_k(k, dim3(nparts), dim3(kThreads), sm, a.stream, false, a.W, a.G, a.r, colpart,
                             rsum_part, a.V, D, a.map.tpr, a.beta2, a.one_minus_beta2, (float)a.inv_bc, a.eps,
                             a.lr_signed);
        }
        if (e != cudaSuccess)
            return e;
        if (a.trace)
            cudaEventRecord(a.trace[1], a.stream);
        e = launch_state(colpart, nparts, rsum_part, nparts, a.c, csum_part, sc, a.V, D, a.beta2,
                         a.one_minus_beta2, a.inv_bc, a.stream, pdl, nullptr, nullptr, nullptr, 0, 0);
        if (e != cudaSuccess)
            return e;
        if (a.trace) {
            cudaEventRecord(a.trace[2], a.stream);
            cudaEventRecord(a.trace[3], a.stream);
        }
        return cudaGetLastError();
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
                         a.beta2, a.one_minus_beta2, a.inv_bc, a.stream, false, a.r, nullptr, lm_row,
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
                             a.beta2, a.one_minus_beta2, a.G_stage + c0, rp, span);
            else
                e = launch_k(k_reduce_dense<VEC, CPT, R1, false>, dim3(nparts), dim3(kThreads), shmem, a.stream,
                             pdl && q > 0, a.G + c0, a.r, colpart + c0, rsum_part, a.V, cols(q), ld, a.map.tpr,
                             a.beta2, a.one_minus_beta2, nullptr, rp, span);
            if (e != cudaSuccess)
                return e;
        }
        if (a.trace)
            cudaEventRecord(a.trace[1], a.stream);
        if (np == 1) {
            e = launch_state(colpart, nparts, rsum_part, nparts, a.c, csum_part, sc, a.V, D, a.beta2,
                             a.one_minus_beta2, a.inv_bc, a.stream, pdl, nullptr, nullptr, nullptr, 0, 0);
        } else {
            const int64_t vb = (a.V + kStateThreads - 1) / kStateThreads;
            const int nrow_ctas = (int)(vb < kMaxRowCtas ? vb : kMaxRowCtas);
            e = launch_state(colpart, nparts, rsum_part, nrow_ctas, a.c, csum_part, sc, a.V, D, a.beta2,
                             a.one_minus_beta2, a.inv_bc, a.stream, pdl, a.r, nullptr, rowpart, np, nrow_ctas);
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
                         (float)a.inv_bc, a.eps, a.lr_signed, a.variant, span);
        else
            e = launch_k(k_apply_dense<VEC, CPT, R3, false>, dim3(nparts), dim3(kThreads), cs_bytes,
                         a.stream, pdl, Wq, Gd + c0, a.r, a.c + c0, sc, a.V, cols(q), ld, a.map.tpr,
                         (float)a.inv_bc, a.eps, a.lr_signed, a.variant, span);
        if (e != cudaSuccess)
            return e;
    }
    if (a.trace)
        cudaEventRecord(a.trace[3], a.stream);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_state(const float *colpart, int nparts, double *rsum_part, int nrsum, float *c,
                         double *csum_part, DevScalars *sc, int64_t V, int D, double beta2,
                         double one_minus_beta2, double inv_bc, cudaStream_t stream, bool pdl,
                         float *r_rows, int32_t *slot, const float *rowpart, int nslices, int nrow_ctas)
{
    const int nstate = (D + kStateCols - 1) / kStateCols;
    RowPass rp{r_rows, slot, rowpart, nslices, nrow_ctas};
    return launch_k(k_state_dense, dim3(nstate + nrow_ctas), dim3(kStateThreads), 0, stream, pdl, colpart,
                    nparts, rsum_part, nrsum, c, csum_part, sc, V, D, beta2, one_minus_beta2, inv_bc, rp);
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
        switch (a.map.cpt) {
        case 1: return launch_dense_t<4, 1>(a);
        case 2: return launch_dense_t<4, 2>(a);
        case 4: return launch_dense_t<4, 4>(a);
        case 8: return launch_dense_t<4, 8>(a);
        }
    } else {
        switch (a.map.cpt) {
        case 1: return launch_dense_t<1, 1>(a);
        case 2: return launch_dense_t<1, 2>(a);
        case 4: return launch_dense_t<1, 4>(a);
        case 8: return launch_dense_t<1, 8>(a);
        }
    }
    return cudaErrorInvalidValue;
}

}  // namespace ember
