// ember_step_dense_noalloc: the dense step with library-owned scratch.
//
// Some callers cannot hand this library a device workspace:
//   - hosts whose device memory is owned by a framework allocator that
//     gives plugins no allocation hook;
//   - optimizer loops running under a fixed memory budget that is already
//     fully reserved;
//   - code paths where a cudaMalloc would synchronise the device in the
//     middle of a training step.
// For them this entry point runs the very same kernels as ember_step_dense,
// with their scratch (per-CTA column partials, row-sum partials, a few
// scalars) in a file-scope device array instead of a bound workspace.  It allocates nothing: no cudaMalloc, no cudaFree, no allocating
// library call.
//
// The array is kNoAllocScratchBytes (10 MiB) on every GPU that loads the
// library, held until the process exits.  That covers every table a CTA
// holds whole rows of (D <= 8192 needs 9.97 MB); wider tables, which run in
// column panels with per-row partial sums, are refused.
//
// In host code the array's name is only a host-side stand-in; the kernels get
// its device address, looked up with cudaGetSymbolAddress on the first call
// made with a device current.  The address is cached per device together
// with the CUDA context it was looked up in: after a cudaDeviceReset (or any
// teardown and re-creation of the device's context) the module is loaded
// again, the context differs, and the address is looked up again instead of
// reusing a stale one.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>
#include <mutex>
#include <stdint.h>

#include "ember_internal.h"

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(10) << 20;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mutex;
struct ScratchAddr {
    CUcontext ctx;
    unsigned char *ptr;
};
ScratchAddr g_scratch[kMaxDevices] = {};

// The driver's cuCtxGetCurrent, reached through the runtime (no link to
// libcuda needed); nullptr if the driver does not provide it.
PFN_cuCtxGetCurrent_v4000 ctx_get_current_fn()
{
    static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    });
    return fn;
}

// Device address of the scratch array on the current device and context
// (nullptr on error).
unsigned char *scratch_for_current_device()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return nullptr;
    PFN_cuCtxGetCurrent_v4000 get_ctx = ctx_get_current_fn();
    if (!get_ctx)
        return nullptr;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    CUcontext ctx = nullptr;
    if (get_ctx(&ctx) != CUDA_SUCCESS)
        return nullptr;
    if (!ctx || !g_scratch[dev].ptr || g_scratch[dev].ctx != ctx) {
        // the lookup also makes the device's primary context current if no
        // runtime call has yet; the context is read again after it
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
            return nullptr;
        if (get_ctx(&ctx) != CUDA_SUCCESS || !ctx)
            return nullptr;
        g_scratch[dev].ctx = ctx;
        g_scratch[dev].ptr = static_cast<unsigned char *>(p);
    }
    return g_scratch[dev].ptr;
}

bool aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

}  // namespace

extern "C" ember_status ember_step_dense_noalloc(ember_handle *h, void *W, const float *G,
                                                 float *state, float lr, int64_t t, void *stream)
{
    using namespace ember;
    if (!h || !W || !G || !state)
        return EMBER_ERR_INVALID_ARG;
    if (t < 1 || !isfinite(lr))
        return EMBER_ERR_INVALID_ARG;
    const size_t wsz = h->wdtype == EMBER_BF16 ? 2 : 4;
    if (!aligned(W, wsz) || !aligned(G, 4) || !aligned(state, 4))
        return EMBER_ERR_ALIGNMENT;

    // The dense kernels use the workspace's scalars, row-sum partials,
    // column-group sums and the column-sum partials of one CTA grid (at most
    // kGridCtas rows of D floats), nothing after that.
    const Layout lay = make_layout(h->V, h->D, 0);
    const size_t need = lay.colpart + sizeof(float) * (size_t)kGridCtas * (size_t)h->D;
    if (need > kNoAllocScratchBytes)
        return EMBER_ERR_WORKSPACE;

    // a table split into column panels also needs per-row partial sums
    const bool vec4 = (h->D % 4 == 0) && aligned(W, 4 * wsz) && aligned(G, 16);
    ColMap map;
    if (!choose_colmap(h->D, vec4, &map))
        return EMBER_ERR_UNSUPPORTED;
    if (map.npanels != 1)
        return EMBER_ERR_WORKSPACE;

    unsigned char *scratch = scratch_for_current_device();
    if (!scratch)
        return EMBER_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    // every call shares the array: start each one from zeroed scalars
    if (cudaMemsetAsync(scratch + lay.scalars, 0, sizeof(DevScalars), s) != cudaSuccess)
        return EMBER_ERR_CUDA;

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
    a.ws = scratch;
    a.lay = lay;
    a.stream = s;
    a.trace = nullptr;
    a.wait_ns = h->wait_ns;
    a.map = map;
    return launch_dense_step(a) == cudaSuccess ? EMBER_OK : EMBER_ERR_CUDA;
}
