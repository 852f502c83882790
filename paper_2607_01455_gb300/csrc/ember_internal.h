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

// The state pass reduces 32 columns per CTA.
constexpr int kStateCols = 32;
constexpr int kStateThreads = 256;

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

// Workspace layout (byte offsets, each 256-byte aligned).
struct Layout {
    size_t scalars;     // DevScalars
    size_t rsum_part;   // double[kGridCtas]            sum of new r per CTA
    size_t csum_part;   // double[ceil(D/32)]           sum of new c per state CTA
    size_t colpart;     // float[kGridCtas * D]         column sums of g^2 per CTA
    // sparse step (present when max_sparse_N > 0)
    size_t sp_keys;     // uint64[N]  (id << 32 | occurrence), tile-sorted
    size_t sp_sorted;   // uint64[N]  globally sorted keys
    size_t sp_head;     // int32[N + 1] run-head flags / offsets scratch
    size_t sp_uniq;     // int32[N]   distinct ids, ascending
    size_t sp_segoff;   // int32[N + 1] start of each distinct id's run in sp_sorted
    size_t sp_tilecnt;  // int32[ceil(N / tile) + 1] per-tile counts
    size_t sp_rows;     // float[N * D] summed gradient rows, one per distinct id
    size_t total;
};

Layout make_layout(int64_t V, int64_t D, int64_t max_sparse_N);

// Column mapping of a V x D row-major table onto the CTA: `vec` consecutive
// columns per access, `tpr` threads per row, `cpt` accesses per thread per row.
struct ColMap {
    int vec;   // 4 (16-byte fp32 accesses) or 1
    int tpr;   // threads per row: 32 .. kThreads, a power of two
    int cpt;   // accesses per thread per row: 1, 2, 4 or 8
};

bool choose_colmap(int64_t D, bool vec4_ok, ColMap *m);

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
};

cudaError_t launch_dense_step(const DenseArgs &a);

constexpr int kMaxTraceEvents = 16;

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
};
