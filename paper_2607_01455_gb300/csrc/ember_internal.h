// Internal declarations shared by the CUDA translation units of libember.
// Not installed; the public ABI is include/ember.h.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "ember.h"

namespace ember {

// Streaming kernels (row/column reduction, apply) run a persistent grid of
// kGridCtas CTAs of kThreads threads: two co-resident CTAs on each of the
// GB300's 152 SMs.  Each CTA owns one contiguous range of rows, the same
// range in the reduction and in the apply pass.  The grid is a constant, not
// a device query, so results depend on (V, D) only and are bit-identical on
// every run and every device.
constexpr int kThreads = 256;
constexpr int kCtasPerSm = 2;
constexpr int kSms = 152;
constexpr int kGridCtas = kSms * kCtasPerSm;
// The sparse step's segment sums run three smaller CTAs per SM.
constexpr int kSparseCtasPerSm = 3;
constexpr int kSparseCtas = kSms * kSparseCtasPerSm;
constexpr int kPartRows = kSparseCtas > kGridCtas ? kSparseCtas : kGridCtas;

// The state pass reduces 32 columns per CTA of kStateThreads threads (16
// warps, so that each warp adds few per-CTA partial rows).  Its row pass runs
// up to kMaxRowCtas CTAs: about one row per thread for the LM-head step (whose
// rows each sum ceil(D/256) slices) and for a dense step in column panels
// (one slice per panel), and kRowBatch rows per thread for the sparse step
// (whose untouched rows only decay).
constexpr int kStateCols = 32;
constexpr int kStateThreads = 512;
constexpr int kMaxRowCtas = 1024;
constexpr int kRowBatch = 8;
constexpr int kRsumParts = kMaxRowCtas > kGridCtas ? kMaxRowCtas : kGridCtas;

// Bits of the sticky device flag.
constexpr unsigned kFlagIdRange = 1u << 0;
constexpr unsigned kFlagTimeout = 1u << 1;

// Scalars that live in the workspace.  `ticket` counts finished CTAs of the
// state pass and is returned to zero by the last one.
struct DevScalars {
    double s;          // geometric-mean normaliser sqrt(mean rhat * mean chat)
    double rbar;       // mean over rows of rhat
    double cbar;       // mean over columns of chat
    float inv_s;       // 1/s in fp32, 0 when s == 0
    unsigned ticket;
    unsigned flags;    // sticky device error bits (kFlag*)
    int32_t n_unique;  // sparse step: number of distinct valid ids
    int32_t n_valid;   // sparse step: number of ids inside [0, V)
};

// Sparse step: ids are sorted in tiles of kSortTile keys by kSortThreads
// threads.
constexpr int kSortTile = 1024;
constexpr int kSortThreads = 256;

// Workspace layout (byte offsets, each 256-byte aligned).
struct Layout {
    size_t scalars;     // DevScalars
    size_t rsum_part;   // float[kRsumParts]            sum of new r per CTA
    size_t csum_part;   // float[ceil(D/32)]            sum of new c per 32-column group
    size_t colpart;     // float[kPartRows * D]     column sums of g^2 per CTA
    // sparse step (present when max_sparse_N > 0); N = max_sparse_N,
    // Npad = N rounded up to kSortTile
    size_t sp_keys;     // uint64[Npad]  (id << 32 | occurrence), sorted within tiles
    size_t sp_rank;     // int32[Npad]   global rank of each tile-sorted key
    size_t sp_sorted;   // uint64[N]     keys in (id, occurrence) order
    size_t sp_tilecnt;  // int32[2 * Npad / kSortTile]  heads and valid ids per tile
    size_t sp_perm;     // int32[N]      occurrence index at each sorted position
    size_t sp_segidx;   // int32[N]      distinct-id index at each sorted position
    size_t sp_uniq;     // int32[N]      distinct ids, ascending
    size_t sp_segoff;   // int32[N + 1]  first sorted position of each distinct id
    size_t sp_slot;     // int32[V]      1 + distinct-id index of a touched row, else 0
    size_t sp_single;   // int32[N]      occurrence index of an id seen once, else -1
    size_t sp_rowpart;  // float[N * ceil(D / kThreads)]  sum g^2 per (distinct id, slice)
    size_t sp_carry;    // float[2 * kSparseCtas * D]  partial sums of runs cut by worker ranges
    size_t sp_bounds;   // int32[kSparseCtas + 1]  first sorted position of each worker range
    size_t sp_rows;     // float[N * D]  summed gradient row of each distinct id seen twice or more
    // LM-head step (the gradient formed here on the tensor cores)
    size_t lm_colpart;  // float[ceil(V/128) * D]  sums of g^2 over each 128-row block
    size_t lm_rowpart;  // float[ceil(D/256) * V]  sums of g^2 over each 256-column block
                        // (a dense step in column panels: over each panel)
    size_t total;
};

Layout make_layout(int64_t V, int64_t D, int64_t max_sparse_N);

// Column mapping of a V x D row-major table onto the CTA: `vec` consecutive
// columns per access, `tpr` threads per row, `cpt` accesses per thread per row.
// A CTA holds kThreads x 8 accesses of one row: 8192 columns with 16-byte
// accesses, 2048 with 4-byte ones.  Wider tables are split into column
// panels of equal width (the last one may be narrower), each run as a
// table of `pw` columns with row stride D; the row sums of g^2 then come
// from per-panel partial sums.  kMaxCols bounds D.
constexpr int kMaxCols = 65536;
struct ColMap {
    int vec;      // 4 (16-byte fp32 accesses) or 1
    int tpr;      // threads per row: 32 .. kThreads, a power of two
    int cpt;      // accesses per thread per row: 1, 2, 4 or 8
    int npanels;  // column panels: 1 when a CTA holds a whole row
    int pw;       // panel width in columns (a multiple of vec); D when npanels == 1
};

bool choose_colmap(int64_t D, bool vec4_ok, ColMap *m);

// Small tables run the whole dense step as one thread-block cluster launch
// (see ember_dense.cu); the plan and the launch count of a dense step.
constexpr int kMaxClusterCtas = 16;  // a non-portable cluster size past 8
constexpr size_t kSmallSmemMax = 200 << 10;
bool small_table_plan(int64_t V, int64_t D, bool wbf16, const ColMap &m, int *nits, size_t *smem);
int dense_step_launches(int64_t V, int64_t D, bool wbf16, int variant, bool vec4);

// LM-head gradient G = dlogits^T hidden (T tokens, bf16 inputs, fp32 G).
struct LmArgs {
    int64_t V, D, T;
    const void *dlogits;  // T x V bf16
    const void *hidden;   // T x D bf16
    float *G;             // V x D fp32, written
    uint64_t wait_ns;     // limit of the kernel's main-loop waits (0: the default)
};

int lmhead_row_blocks(int64_t V);
int lmhead_col_blocks(int64_t D);
// Forms G and the per-tile sums of g^2 (colpart: [row blocks][D], rowpart:
// [column blocks][V]); a bounded wait that gives up sets kFlagTimeout in *flags.
cudaError_t launch_lmhead_grad(const LmArgs &a, float *colpart, float *rowpart, unsigned *flags,
                               cudaStream_t stream);

// Rows a launch of the reduce or apply kernel covers: its CTA b is CTA
// cta_base + b of a grid of nparts over the whole table (row range
// [(cta_base+b) V / nparts, (cta_base+b+1) V / nparts)), and the G and W
// pointers hold rows from row_base on.  The whole-table step uses
// {0, nparts, 0}; a row shard uses its own CTAs of the same grid, so every
// per-CTA partial is the one the whole-table step would form.
struct RowSpan {
    int cta_base;
    int nparts;
    int64_t row_base;
};

// Row-sharded dense step (see ember_shard_reduce / ember_shard_pack /
// ember_shard_update).
constexpr int kMaxShards = 4096;
struct ShardArgs {
    int phase;                        // 1: reduce, local exponents; 2: pack at the global
                                      // exponents; 3: state pass and apply
    int cta_begin, cta_end;           // this shard's CTAs of the whole-table grid
    int64_t row_base;                 // first row this shard holds
    unsigned char *scales;            // D + 1 exponents: phase 1 out, phases 2 and 3 in (all-reduced by max)
    unsigned long long *sums;         // D + 1 fixed-point totals: phase 2 out, phase 3 in (all-reduced by sum)
};

struct DenseArgs {
    int64_t V, D;
    int wbf16;
    void *W;
    const float *G;
    float *r;      // state[0, V)
    float *c;      // state[V, V + D)
    double beta2, one_minus_beta2, inv_bc;
    float lr_signed;  // -lr for descent, +lr for ascent
    float eps;
    int variant;
    unsigned char *ws;
    Layout lay;
    ColMap map;
    cudaStream_t stream;
    const cudaEvent_t *trace;  // nullptr, or events[0..3] to record at kernel boundaries
    float *G_stage;            // nullptr, or the HBM copy the reduce pass writes of a host-resident G
    const LmArgs *lm;          // nullptr, or: G is formed by the LM-head kernel instead of read
    const ShardArgs *shard;    // nullptr, or: one phase of a row-sharded step
    uint64_t wait_ns;          // limit of every bounded wait inside a kernel
};

// CTAs of the dense step's reduce and apply grids for a V x D table: one
// per kMinCtaElems elements of G (so that a table of up to 16 x 4096
// elements has at most 16 CTAs and can run as one cluster launch), at most
// kGridCtas and at most one per row.  A function of (V, D) only, so the
// per-CTA partial sums -- and the results -- are the same on every run and
// device.
constexpr int64_t kMinCtaElems = 4096;
inline int dense_parts(int64_t V, int64_t D)
{
    int64_t n = (V * D + kMinCtaElems - 1) / kMinCtaElems;
    if (n > kGridCtas)
        n = kGridCtas;
    if (n > V)
        n = V;
    return (int)(n < 1 ? 1 : n);
}

// Rows a thread of the reduce pass takes per iteration (its rows in flight):
// 16 / cpt, halved for rows of one access per thread when a CTA's rows fit
// in half an iteration, so that on a small table every thread reduces (and,
// in the one-launch step, updates) half as many rows.  A function of (V, D)
// and the column map only, like the grid: every form of the step forms the
// same per-CTA partials.
inline int reduce_rows_per_thread(int64_t V, int64_t D, const ColMap &m)
{
    const int r = (16 / m.cpt) < 1 ? 1 : 16 / m.cpt;
    if (m.cpt != 1)
        return r;
    const int nparts = dense_parts(V, D);
    const int64_t rows = (V + nparts - 1) / nparts;
    return rows <= (int64_t)(kThreads / m.tpr) * (r / 2) ? r / 2 : r;
}

// Default limit of a bounded wait inside a kernel (grid barriers, mbarrier
// waits): 2 s of wall time.
constexpr uint64_t kDefaultWaitNs = 2000000000ull;

cudaError_t launch_dense_step(const DenseArgs &a);

// beta2 r + (1 - beta2) m is formed in fp32 with each coefficient carried as
// a float pair hi + lo (hi the coefficient rounded to fp32, lo the rest),
// computed once on the host.  See ema_pair() in ember_dense.cu.
struct EmaPair {
    float bh, bl, ah, al;
};

// Constants of one step, rounded to fp32 on the host: the EMA coefficients,
// 1/D, 1/V and the bias-correction factor 1/(1 - beta2^t) (1 without it).
// GB300 runs fp64 at a small fraction of its fp32 rate, so the kernels keep
// fp64 out of their latency-bound parts.
struct StepConsts {
    EmaPair ema;
    float inv_D, inv_V, inv_bc;
};
// beta2 r + (1 - beta2) m in fp32 with the coefficients carried as float
// pairs: within about an ulp of the fp64 value, and the fixed point stays
// at r = m, which rounding beta2 and 1 - beta2 to single floats would shift
// by about 1e-5 of r at beta2 = 0.999.  With m = 0 (a row outside a sparse
// batch) it is the correctly rounded product beta2 r in all but near-tie
// cases.
__device__ __forceinline__ float ema_pair(const EmaPair &e, float r, float m)
{
    return fmaf(e.bh, r, fmaf(e.bl, r, fmaf(e.ah, m, e.al * m)));
}

inline StepConsts make_consts(double beta2, double one_minus_beta2, int64_t V, int64_t D, double inv_bc)
{
    StepConsts k;
    k.ema.bh = (float)beta2;
    k.ema.bl = (float)(beta2 - (double)k.ema.bh);
    k.ema.ah = (float)one_minus_beta2;
    k.ema.al = (float)(one_minus_beta2 - (double)k.ema.ah);
    k.inv_D = (float)(1.0 / (double)D);
    k.inv_V = (float)(1.0 / (double)V);
    k.inv_bc = (float)inv_bc;
    return k;
}

// Column EMA and normaliser; with nrow_ctas > 0 the same launch also runs a
// row pass: r from per-slice sums of g^2, taken from rowpart[u][nslices] for
// the touched rows of the sparse step, or, with slot == nullptr, from
// rowpart[nslices][V] for every row.
// Column totals are exact fixed-point sums of the nparts partial rows
// (ember_device.cuh); the normaliser's sum of r likewise over the nrsum
// per-CTA sums in rsum_part.
// For the sparse step (slot set) the row pass covers only the U touched rows
// uniq[0..U) (the segment-sum kernel decays the others) and writes its
// per-CTA sums of r from rsum_part[rsum_base] on.
cudaError_t launch_state(const float *colpart, int nparts, float *rsum_part, int nrsum, float *c,
                         float *csum_part, DevScalars *sc, int64_t V, int D, const StepConsts &k,
                         cudaStream_t stream, bool pdl, float *r_rows, int32_t *slot, const float *rowpart,
                         int nslices, int nrow_ctas, const int32_t *uniq = nullptr, int rsum_base = 0,
                         int pstride = 1, int pcols = 0);

struct SparseArgs {
    int64_t V, D, N;
    int wbf16;
    int ids64;
    void *W;
    const void *ids;
    const float *rows;
    float *r;
    float *c;
    double beta2, one_minus_beta2, inv_bc;
    float lr_signed;
    float eps;
    int variant;
    unsigned char *ws;
    Layout lay;
    ColMap map;
    cudaStream_t stream;
    const cudaEvent_t *trace;  // nullptr, or events to record at kernel boundaries
    int n_trace;
};

cudaError_t launch_sparse_step(const SparseArgs &a);

// Sort and dedup only; then copy the distinct ids, their counts and U out.
cudaError_t launch_sparse_unique(const SparseArgs &a, int32_t *uniq_out, int32_t *counts_out,
                                 int32_t *n_unique_out);

constexpr int kMaxTraceEvents = 16;

// Launch `kernel` on `stream`.  With pdl = true the launch may begin while
// the previous kernel on the stream is still finishing (programmatic
// dependent launch); every kernel launched this way calls grid_dep_wait()
// before it reads anything an earlier kernel wrote.
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                     cudaStream_t stream, bool pdl, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = pdl ? attr : nullptr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

}  // namespace ember

struct ember_handle {
    int64_t V, D;
    ember_hparams hp;
    ember_wdtype wdtype;
    unsigned char *ws;
    size_t ws_bytes;
    int64_t ws_max_N;
    cudaEvent_t trace[ember::kMaxTraceEvents];
    int n_trace;
    uint64_t wait_ns;  // limit of the bounded waits inside kernels (ember_set_wait_limit_ns)
};
