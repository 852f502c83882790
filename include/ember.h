/*
 * ember.h -- C ABI of the Ember optimizer step for V x D token tables
 * (embedding tables and LM heads), GB300 (sm_103a) CUDA implementation.
 *
 * Ember is Algorithm 1 of "Token Geometry" (arXiv 2607.01455, Section 2.1).
 * For a table W (V rows = tokens, D columns = features) and its gradient g
 * at step t it keeps only two fp32 vectors, r (V) and c (D), and does:
 *
 *   r <- beta2 r + (1-beta2) mean_j g_ij^2          (row second moment)
 *   c <- beta2 c + (1-beta2) mean_i g_ij^2          (column second moment)
 *   rhat = r / (1-beta2^t),  chat = c / (1-beta2^t) (bias correction)
 *   s = sqrt(mean_i rhat_i * mean_j chat_j)         (geometric-mean normaliser)
 *   W_ij <- W_ij - lr * g_ij / (sqrt(rhat_i chat_j / s) + eps)
 *
 * The V x D preconditioner rhat chat^T / s is never stored: it is applied as
 * a per-row and a per-column scaling, as Section 2.3 prescribes.  The sparse step (Section 2.2) takes the token ids of a
 * batch and one gradient row per occurrence; it equals the dense step on the
 * V x D gradient whose row u is the sum of the rows of every occurrence of u.
 *
 * Conventions shared by every entry point:
 *   - Device pointers are CUDA device (or managed) addresses on the current
 *     device; every array is row-major and contiguous.  The library allocates
 *     and frees no device memory at run time: W, G, ids, rows, the state and
 *     the workspace belong to the caller.  The one exception is a static
 *     10 MiB scratch array in the library's device code, present on every
 *     GPU that loads the library until the process exits, which only
 *     ember_step_dense_noalloc uses.
 *   - "stream" is a cudaStream_t passed as void* (NULL = the legacy default
 *     stream).  Steps are asynchronous on that stream.  Errors the host can
 *     see are returned at once and nothing is launched; errors only the GPU
 *     can see (an id outside [0, V), a bounded wait that gave up) set a
 *     sticky flag in the workspace that ember_get_device_status() reads.
 *   - A handle is not thread-safe; use one handle per table and do not run
 *     two steps of one handle concurrently on different streams (they share
 *     the workspace).
 *   - Results are deterministic: the same inputs give bit-identical W and
 *     state on every run.  No floating-point atomics are used; every sum is
 *     taken in a fixed order or, across CTAs, exactly in 64-bit fixed point
 *     (the deterministic, atomic-free reduction that Section 2.3 asks for).
 *   - Waits inside kernels are bounded (the mbarrier waits of the LM-head
 *     kernel): a wait that runs past the handle's limit (2 s by default,
 *     ember_set_wait_limit_ns) sets EMBER_ERR_TIMEOUT in the sticky device
 *     flag and the kernel returns early, after the copies and matrix
 *     operations it has issued complete; the step is then incomplete.
 */
#ifndef EMBER_H
#define EMBER_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define EMBER_ABI_VERSION 2

typedef enum {
    EMBER_OK = 0,
    EMBER_ERR_INVALID_ARG = 1,     /* null pointer, bad size, t < 1, beta2 outside [0,1), ... */
    EMBER_ERR_ALIGNMENT = 2,       /* a pointer is not aligned to its element size */
    EMBER_ERR_DTYPE = 3,           /* unknown weight or id type */
    EMBER_ERR_WORKSPACE = 4,       /* no workspace bound, or too small for this call */
    EMBER_ERR_CUDA = 5,            /* a CUDA runtime call or a kernel launch failed */
    EMBER_ERR_ID_OUT_OF_RANGE = 6, /* device flag: a token id was outside [0, V) and was skipped */
    EMBER_ERR_TIMEOUT = 7,         /* device flag: a bounded wait inside a kernel gave up */
    EMBER_ERR_UNSUPPORTED = 8      /* the GPU is not sm_103 or the size is beyond a stated limit */
} ember_status;

typedef enum { EMBER_F32 = 0, EMBER_BF16 = 1 } ember_wdtype;  /* storage type of W */
typedef enum { EMBER_I32 = 0, EMBER_I64 = 1 } ember_idtype;   /* storage type of token ids */

/* Preconditioner.  FULL is Algorithm 1.  ROW (vtil_ij = rhat_i, a V-float
 * state in use) and COL (vtil_ij = chat_j) are the "row-only" and "col-only"
 * rows of the ablation table in Section 2.1; both keep the same V + D state
 * layout so that a handle can switch between them. */
typedef enum {
    EMBER_VARIANT_FULL = 0,
    EMBER_VARIANT_ROW = 1,
    EMBER_VARIANT_COL = 2
} ember_variant;

typedef struct {
    double beta2;        /* second-moment decay, in [0, 1).  Default 0.999 (Algorithm 1). */
    double eps;          /* added to sqrt(vtil), >= 0.  Default 1e-8 (Algorithm 1). */
    int maximize;        /* 0 (default): W -= lr u, descending a loss whose gradient is G.
                            1: W += lr u, ascending a reward, as Algorithm 1 is printed. */
    int bias_correction; /* 1 (default): divide by 1 - beta2^t.  0: the ablation of the
                            appendix "Ablations" (rhat = r, chat = c). */
    int variant;         /* ember_variant; default EMBER_VARIANT_FULL */
} ember_hparams;

typedef struct ember_handle ember_handle;

/* Fill *hp with the defaults of Algorithm 1: beta2 = 0.999, eps = 1e-8,
 * descent, bias correction on, full preconditioner. */
void ember_hparams_default(ember_hparams *hp);

/* Create a host-side handle for one V x D table whose weights are stored as
 * wdtype.  hp == NULL takes the defaults.  Validates V >= 1, D >= 1,
 * V * D < 2^62, 0 <= beta2 < 1, eps >= 0 (finite) and the enums
 * (EMBER_ERR_INVALID_ARG), and V < 2^31, D <= 65536 (EMBER_ERR_UNSUPPORTED).
 * Touches no GPU.  On success *out owns a handle to free with
 * ember_destroy().
 *   Tables whose rows a CTA cannot hold whole (D > 8192 on the 16-byte
 * vector path, D > 2048 on the scalar one) are processed in column panels
 * of equal width: one reduce and one apply launch per panel, each row's sum
 * of g^2 added up from per-panel partial sums in panel order.  Every step
 * accepts them except the row-sharded one and ember_step_dense_noalloc. */
ember_status ember_create(int64_t V, int64_t D, const ember_hparams *hp,
                          ember_wdtype wdtype, ember_handle **out);

/* Free the host handle (never device memory).  NULL is ignored. */
void ember_destroy(ember_handle *h);

/* Column panels the dense, LM-head and sparse steps of this handle run in
 * (see ember_create): 1 when a CTA holds a whole row, more for wider
 * tables; each panel costs one reduce and one apply launch (one apply
 * launch for the sparse and LM-head steps).  vector_path = 1 for pointers
 * that take the 16-byte path (D % 4 == 0, W, G and rows 16-byte aligned,
 * 8-byte for bf16 W), 0 for the scalar path.  Host only.  Returns 0 for a
 * NULL handle. */
int ember_column_panels(const ember_handle *h, int vector_path);

/* Kernel launches one ember_step_dense of this handle makes without trace
 * events: 1 for a small table (one cluster launch), 2 for the row-only
 * variant (its one-pass kernel and the column state), otherwise 2 per
 * column panel plus the state pass.  vector_path as for
 * ember_column_panels.  Host only; 0 for a NULL handle. */
int ember_dense_step_launches(const ember_handle *h, int vector_path);

/* Number of fp32 values of optimizer state: exactly V + D (Algorithm 1
 * keeps r in R^V and c in R^D).  The caller's state buffer holds r in
 * [0, V) followed by c in [V, V + D).  A new table starts from all zeros
 * (Algorithm 1 initialises r_0 = 0 and c_0 = 0). */
size_t ember_state_numel(const ember_handle *h);

/* Bytes of device workspace the steps of this handle need when sparse steps
 * carry at most max_sparse_N ids (0 if only dense steps are used).  Returns
 * 0 for a NULL handle or a negative max_sparse_N.  The workspace holds
 * per-block partial sums (among them the LM-head step's per-tile sums of
 * g^2, V*D*4*(1/128 + 1/256) bytes, always reserved), the sort buffers of
 * the sparse step, the summed gradient rows of the sparse step (up to
 * max_sparse_N x D fp32), a V-entry map of touched rows and a few scalars.
 * It is not optimizer state, but the steps leave the touched-row map zeroed
 * for the next one: the caller must not write to the workspace after binding
 * it, nor touch it while a step is in flight. */
size_t ember_workspace_bytes(const ember_handle *h, int64_t max_sparse_N);

/* Give the handle its device workspace (256-byte aligned, at least
 * ember_workspace_bytes(h, max_sparse_N) bytes) and clear the sticky device
 * flag with a memset on `stream`.  Rebinding replaces the previous
 * workspace. */
ember_status ember_bind_workspace(ember_handle *h, void *workspace, size_t bytes,
                                  int64_t max_sparse_N, void *stream);

/* One dense Ember step (Algorithm 1) at step number t >= 1.
 *   W:     V x D, wdtype, updated in place.
 *   G:     V x D fp32 gradient of the loss (of the reward when maximize = 1).
 *   state: V + D fp32 (r then c), updated in place.
 *   lr:    step size alpha, applied in fp32 (any finite value).
 * W and G must be 4-byte (bf16 W: 2-byte) aligned; with D % 4 == 0 and
 * 16-byte aligned W, G and state the vectorised kernels run, otherwise a
 * scalar path gives the same results more slowly.
 *   A small table (V * D <= 65536 on the vector path, whose rows a CTA
 * covers in a few passes) runs as one launch of a thread-block cluster of
 * up to 16 CTAs that keeps G and W in shared memory and reads G from HBM
 * once; every other table runs as three launches (reduce, column
 * statistics and normaliser, update), chained with programmatic dependent
 * launch.  Both forms run the same arithmetic on the same CTA row
 * ranges and give the same bits.  Graph capture works for both. */
ember_status ember_step_dense(ember_handle *h, void *W, const float *G, float *state,
                              float lr, int64_t t, void *stream);

/* The dense step with the gradient in host memory (Grace-Blackwell systems).
 * Same update as ember_step_dense.  The reduce pass reads G_host directly
 * over the chip-to-chip link -- no copy engine -- and writes each element to
 * G_stage (device, V x D fp32, caller-owned) as it goes; the state and apply
 * passes then read G_stage from HBM.  G_host must be addressable by the GPU:
 * pinned (cudaHostAlloc / cudaHostRegister), managed or device memory;
 * unregistered host memory returns EMBER_ERR_INVALID_ARG.  The row-only
 * variant is not offered here (EMBER_ERR_UNSUPPORTED).  Afterwards G_stage
 * holds a copy of G. */
ember_status ember_step_dense_from_host(ember_handle *h, void *W, const float *G_host, float *G_stage,
                                        float *state, float lr, int64_t t, void *stream);

/* The dense step for callers that cannot give the library any device
 * memory: hosts whose allocator offers plugins no allocation hook,
 * optimizer loops under a fully reserved memory budget, and code paths
 * where a cudaMalloc would synchronise the device mid-step.  The paper has
 * no counterpart; this is an interface convenience.
 *   Same arguments, same kernels and same results as ember_step_dense, but
 * no workspace is bound or used: the scratch (column and row-sum partials,
 * scalars) lives in a 10 MiB array inside the library, present on every GPU
 * that loads the library until the process exits.  Nothing is allocated.
 * Every table whose rows a CTA holds whole fits (D <= 8192 needs 9.97 MB);
 * a table processed in column panels (see ember_create) returns
 * EMBER_ERR_WORKSPACE.
 *   The first call on each device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current and caches it with the
 * device's current CUDA context; it is looked up again if the context
 * changes (after a cudaDeviceReset, for instance).  Make the first call on
 * a device before any stream capture.  All calls on a device share the one
 * array and each starts by zeroing its scalars, so calls that overlap on
 * the GPU (two streams, two handles, two threads) race and must be
 * serialised by the caller.  A timeout of a bounded wait is reported by
 * the sticky flag in the array, which the next call clears: this entry
 * point has no workspace for ember_get_device_status to read. */
ember_status ember_step_dense_noalloc(ember_handle *h, void *W, const float *G, float *state,
                                      float lr, int64_t t, void *stream);

/* The gradient of an LM head (output embedding) W = V x D, formed on the
 * tensor cores: G = dlogits^T hidden, i.e. G[v][d] = sum_t dlogits[t][v]
 * hidden[t][d], the sum over the T tokens of the outer product of each
 * token's output-side error (softmax minus one-hot) and its hidden state
 * (appendix "Decomposing the Squared Gradient").  bf16 products, fp32
 * accumulation.
 *   dlogits: T x V bfloat16, row-major, device (any 1/T scaling applied).
 *   hidden:  T x D bfloat16, row-major, device.
 *   T:       tokens, 1 <= T <= 2^31 - 1.
 *   G:       V x D fp32, row-major, device, written (caller-owned).
 * Requires V % 8 == 0 and D % 8 == 0 (rows of dlogits and hidden a multiple
 * of 16 bytes; EMBER_ERR_UNSUPPORTED otherwise) and 16-byte aligned
 * dlogits, hidden and G (EMBER_ERR_ALIGNMENT).  Uses the bound workspace;
 * the optimizer state is untouched.  A bounded wait inside the kernel that
 * gives up sets EMBER_ERR_TIMEOUT in the device flag. */
ember_status ember_lmhead_grad(ember_handle *h, const void *dlogits, const void *hidden, int64_t T,
                               float *G, void *stream);

/* One dense Ember step (Algorithm 1) of an LM head whose gradient is formed
 * here: G = dlogits^T hidden exactly as ember_lmhead_grad (G is written, the
 * same bits), then the step of ember_step_dense on that G.  The kernel that
 * forms G also writes, from the registers that hold each finished 128 x 256
 * tile, the tile's sums of g^2 along its rows and along its columns (the
 * fused deterministic reduction of Section 2.3, moved into the producer of
 * G); the state pass finishes those sums in a fixed order and the apply pass
 * reads G once, so the step moves 8VD + 2wVD bytes of G and W instead of
 * 12VD (bf16 W).  Results are bit-identical from run to run; they match
 * ember_step_dense on the same G to rounding (the sums of g^2 are grouped
 * differently).  Every variant is accepted.  Requirements: those of
 * ember_lmhead_grad and of ember_step_dense. */
ember_status ember_step_lmhead(ember_handle *h, void *W, const void *dlogits, const void *hidden,
                               int64_t T, float *G, float *state, float lr, int64_t t, void *stream);

/* Row-sharded dense step (Section 2.3: the statistics are sums of g^2, so
 * a table whose rows are spread over ranks needs only small per-rank sums
 * exchanged before the update: one value per column and one for the sum of
 * r).  A step is three calls per shard with two all-reduces between them:
 *
 *   ember_shard_reduce (every shard)  the reduction pass over the shard's
 *       rows: updates r for those rows, keeps the shard's per-CTA partial
 *       sums in its workspace, and writes `scales`: for each column (and, at
 *       index D, for the sums of r) the largest fp32 exponent among the
 *       shard's partials, one byte each;
 *   the caller all-reduces `scales` with MAX (uint8, D + 1 bytes:
 *       ember_shard_scale_bytes);
 *   ember_shard_pack (every shard)  writes `sums`: each column's (and the r
 *       sums') partials added in 64-bit fixed point at the all-reduced
 *       exponent, one uint64 each;
 *   the caller all-reduces `sums` with SUM (uint64/int64, 8 (D + 1) bytes:
 *       ember_shard_exchange_bytes, 64 KiB at D = 8192);
 *   ember_shard_update (every shard)  the column EMA and normaliser from the
 *       totals (every shard forms the same c and s), then the update of the
 *       shard's rows of W.
 *
 * Integer sums do not depend on how the partials are grouped, and the
 * whole-table steps form the same fixed-point totals from the same per-CTA
 * partials (shards are cut at the whole-table step's CTA row ranges), so W,
 * r and c come out bit-identical to ember_step_dense for any number of
 * shards (the paper's "bitwise identical" requirement of Section 2.3).
 *
 *   shard, nshards: 0 <= shard < nshards <= 4096.  Shards past the table's
 *       last CTA hold no rows (their calls still take part: their scales
 *       and sums are zero, and the update maintains c).
 *   G_shard, W_shard: the shard's rows (ember_shard_rows), row-major,
 *       device memory; with D % 4 == 0 they must be 16-byte aligned (8-byte
 *       for bf16 W) so that every shard takes the whole-table step's
 *       vector path (EMBER_ERR_ALIGNMENT otherwise).
 *   state: a full V + D buffer per shard; only the shard's rows of r and all
 *       of c are read and written.
 *   scales: device, D + 1 bytes.  sums: device, D + 1 uint64, 8-byte
 *       aligned.  Both caller-owned.
 * Between a shard's reduce and its update the handle's workspace holds the
 * shard's partials: run no other step of that handle in between.  Variant
 * ROW is not offered (EMBER_ERR_UNSUPPORTED): its one-pass kernel needs no
 * exchange for W and is run per shard with ember_step_dense.  Nor are tables
 * processed in column panels (see ember_create; EMBER_ERR_UNSUPPORTED). */
int64_t ember_shard_rows(const ember_handle *h, int shard, int nshards, int64_t *row0);
size_t ember_shard_scale_bytes(const ember_handle *h);
size_t ember_shard_exchange_bytes(const ember_handle *h);
ember_status ember_shard_reduce(ember_handle *h, int shard, int nshards, const float *G_shard, float *state,
                                unsigned char *scales, void *stream);
ember_status ember_shard_pack(ember_handle *h, int shard, int nshards, const unsigned char *scales,
                              unsigned long long *sums, void *stream);
ember_status ember_shard_update(ember_handle *h, int shard, int nshards, void *W_shard, const float *G_shard,
                                float *state, const unsigned char *scales, const unsigned long long *sums,
                                float lr, int64_t t, void *stream);

/* One sparse Ember step (Section 2.2) at step number t >= 1.
 *   ids:   N token ids of type idtype (duplicates allowed, any order).
 *   rows:  N x D fp32, row k is the gradient contribution of occurrence k
 *          (any 1/batch scaling already applied by the caller).
 *   N:     0 <= N <= the max_sparse_N the workspace was bound for.
 * Equals ember_step_dense on the V x D gradient whose row u is the sum of
 * rows[k] over the k with ids[k] == u, summed in increasing k: every row of
 * r decays by beta2, the column statistics divide by V, and rows of W whose
 * id does not occur are left bit-identical.  An id outside [0, V) is
 * skipped and sets EMBER_ERR_ID_OUT_OF_RANGE in the device flag. */
ember_status ember_step_sparse(ember_handle *h, void *W, const void *ids,
                               ember_idtype idtype, int64_t N, const float *rows,
                               float *state, float lr, int64_t t, void *stream);

/* Token-id dedup alone (the first part of ember_step_sparse, Section 2.2):
 * writes, on `stream`, the distinct ids of ids[0..N) that lie in [0, V) in
 * ascending order to uniq[0..U), how often each occurs to counts[0..U), and
 * U to *n_unique.  uniq and counts hold N int32 each, n_unique one int32;
 * all three are device memory owned by the caller.  Uses the bound
 * workspace (N <= max_sparse_N); leaves the optimizer state untouched.
 * Ids outside [0, V) are skipped and set EMBER_ERR_ID_OUT_OF_RANGE in the
 * device flag. */
ember_status ember_sparse_unique(ember_handle *h, const void *ids, ember_idtype idtype, int64_t N,
                                 int32_t *uniq, int32_t *counts, int32_t *n_unique, void *stream);

/* Synchronise `stream`, return the sticky device flag of this handle's
 * workspace (EMBER_OK if no device error happened since the last call) and
 * clear it. */
ember_status ember_get_device_status(ember_handle *h, void *stream);

/* Kernel-boundary tracing.  events[k] are cudaEvent_t handles owned by the
 * caller (created on the current device); n of them, at most 16.  While set,
 * every step records events[0] on its stream before its first kernel and
 * events[k] after its k-th kernel, so cudaEventElapsedTime(events[k-1],
 * events[k]) is the device time of kernel k.  The dense step launches 3
 * kernels (reduce, state, apply), so it records events[0..3]; the sparse
 * step records one event per kernel it launches, up to n - 1.  Pass
 * events = NULL or n = 0 to stop tracing.  The events are not recorded
 * when n is too small for a step; nothing else changes. */
ember_status ember_set_trace_events(ember_handle *h, void *const *events, int n);

/* Limit, in nanoseconds of wall time, of the bounded waits inside this
 * handle's kernels (the main-loop mbarrier waits of the LM-head kernel; its
 * teardown waits keep 2 s so that copies already issued always complete);
 * 0 restores the default of 2 s.  A short limit makes a wait give up on
 * purpose: the kernel sets EMBER_ERR_TIMEOUT and returns early, which is how
 * the failure path is tested.  Host only. */
ember_status ember_set_wait_limit_ns(ember_handle *h, uint64_t ns);

/* Static description of a status code. */
const char *ember_status_string(ember_status s);

/* EMBER_ABI_VERSION of the compiled library. */
int ember_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* EMBER_H */
