// LM-head gradient on the tensor cores, with the Ember statistics in the
// epilogue.
//
// For an output head the per-token gradient is the outer product of the
// token's softmax error delta_t (V values) and its hidden state h_t (D
// values), and the batch gradient is their sum over the T tokens:
//     G = dlogits^T H,   G[v][d] = sum_t dlogits[t][v] H[t][d]
// (appendix "Decomposing the Squared Gradient").  Algorithm 1 then needs the
// sums of g^2 along every row and every column of G.  This kernel forms G
// tile by tile with tcgen05.mma (bf16 in, fp32 accumulate in tensor memory)
// and, while a finished tile is in registers for its store, also writes the
// tile's per-row and per-column sums of g^2.  The optimizer step then skips
// its reduction pass (one 4VD-byte read of G) and goes straight to the state
// and apply passes: the fused deterministic reduction of Section 2.3, moved
// into the producer of G.
//
// Tiles: a pair of CTAs (a cluster of two, on two SMs) runs
// tcgen05.mma.cta_group::2 on 256 rows of G (vocabulary) x 256 columns
// (features).  Each CTA holds, per pipeline stage of 80 tokens, its own 128
// rows of dlogits and its own 128 columns of H (40 KiB; five stages, 200
// KiB), and its tensor memory holds its 128 rows of the 256 x 256
// accumulator; the even CTA (the leader) issues the MMAs for both.  Halving
// the H each SM stages (the two tensor cores share the halves) is what lets
// 400 tokens of operands be in flight, enough to cover L2 latency.  How they
// are split matters: on the 128256 x 8192 head four stages of 96 ran 4 %
// faster than six of 64 and 3 % faster than three of 128 (two of 192 and
// twelve of 32 far slower), and five of 80, with one G staging block per
// epilogue warp instead of two to make room, 1 % faster again.  A last
// stage past T reads zeros (the tensor map fills them).
//
// Both operands are "MN-major" in memory (dlogits is T x V and H is T x D,
// row-major, so for a fixed token the tile's rows, resp. columns, are
// contiguous): TMA loads 64-element x 80-token boxes with the 128-byte
// swizzle, described to the MMA as MN-major, swizzled, 10 KiB between
// 64-element blocks and 1 KiB between 8-token groups.  Both CTAs' loads of a stage complete on the
// leader's barrier; the leader's MMA completion frees the stage in both.
//
// Tiles are taken in bands of 16 column blocks (all row pairs of a band, then
// the next band), so the CTAs at work at one time share 32 MiB of H at most;
// H is loaded with an evict-last L2 policy, dlogits and G stream.
//
// Warp roles (256 threads per CTA, one CTA per SM, persistent over tiles):
//   warp 0   one thread issues the TMA loads of this CTA's halves
//   warp 1   allocates, with its peer, 512 tensor-memory columns (two
//            accumulators, so the epilogue of one tile overlaps the MMAs of
//            the next); in the leader one thread issues the MMAs
//   warps 4-7  epilogue: warp 4+q reads accumulator lanes 32q..32q+31 (rows
//            of the tile), forms the sums of g^2, and writes each 32 x 32
//            block of G through swizzled shared memory with a TMA store
//            (whole 128-byte lines, clipped at the edges of G)
//
// Determinism: every output element of G, of the per-tile row sums and of
// the per-tile column sums is produced by exactly one tile, in a fixed
// order, whatever the grid; nothing is accumulated across CTAs here.  The
// state pass sums the per-tile partials in a fixed order.
//
// Waits on mbarriers are bounded (the handle's wait limit, 2 s by default, of
// wall time); a wait that gives up sets the sticky timeout flag, stops every
// role, lets the copies and MMAs already issued finish (those teardown waits
// keep the fixed 2 s limit), frees the tensor memory and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "ember_device.cuh"
#include "ember_internal.h"

namespace ember {
namespace {

constexpr int kBM = 128;                    // accumulator rows per CTA (half the pair's UMMA M)
constexpr int kPairM = 2 * kBM;             // UMMA M of the pair
constexpr int kBN = 256;                    // tile columns (UMMA N)
constexpr int kBK = 80;                     // tokens per stage (five MMAs of 16)
constexpr int kUK = 16;                     // K of one kind::f16 MMA
constexpr int kStages = 5;
constexpr int kBox = 64;                    // TMA box: 64 bf16 = 128 bytes, the swizzle span
constexpr int kABytes = kBM * kBK * 2;      // 20 KiB: this CTA's 128 rows of dlogits
constexpr int kBBytes = (kBN / 2) * kBK * 2;  // 20 KiB: this CTA's 128 columns of H
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kBlockBytes = kBox * kBK * 2; // one 64-wide box: 10 KiB
constexpr int kAccCols = kBN;               // fp32 accumulator columns per tile
constexpr int kTmemCols = 2 * kAccCols;     // two accumulators
constexpr int kLmThreads = 256;
constexpr int kEpiWarp0 = 4;
constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s
// Column blocks per band of the tile order (see tile_of).
constexpr int kLmBand = 16;

// Shared memory: stages (1 KiB aligned for the swizzle), G staging, barriers.
struct LmSmemTail {
    uint64_t full[kStages];    // leader: both CTAs' bytes of the stage landed
    uint64_t empty[kStages];   // each CTA: the pair's MMAs of the stage done
    uint64_t tfull[2];         // each CTA: accumulator ready for the epilogue
    uint64_t tempty[2];        // leader: both CTAs' epilogues drained the accumulator
    uint64_t drain;            // leader: every MMA issued has completed
    uint32_t tmem_base;
    int abort;
    float xch[2][4][32];       // per-warp column sums, double-buffered
};
// Epilogue staging of G for the TMA store: per epilogue warp, kStoreBufs
// 32 x 32 fp32 blocks (4 KiB each, 128-byte swizzled rows).
constexpr int kStoreBufs = 1;
constexpr int kStoreBlockBytes = 32 * 32 * 4;
constexpr int kStoreBytes = 4 * kStoreBufs * kStoreBlockBytes;
constexpr size_t kLmSmemBytes = 1024 + (size_t)kStages * kStageBytes + kStoreBytes + sizeof(LmSmemTail);
static_assert(kLmSmemBytes <= 232448, "over the 227 KiB of shared memory a CTA may use");

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t now_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the phase of parity `parity` of `bar` to complete.  Gives up when
// another role has aborted or after limit_ns (the handle's wait limit);
// returns false then.
__device__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort, uint64_t limit_ns)
{
    if (mbar_test(bar, parity))
        return true;
    // try_wait may suspend the thread for a while before it reports "not
    // yet", so the clock and the abort word are checked after every try
    const uint64_t t0 = now_ns();
    for (;;) {
        if (mbar_test(bar, parity))
            return true;
        if (*abort)
            return false;
        if (now_ns() - t0 > limit_ns)
            return false;
    }
}

// Same, for teardown: no abort check, only the fixed limit kWaitNs (the
// copies and MMAs already issued are waited for even when the main-loop
// limit was made short).
__device__ bool mbar_wait_final(uint32_t bar, uint32_t parity)
{
    const uint64_t t0 = now_ns();
    while (!mbar_test(bar, parity))
        if (now_ns() - t0 > kWaitNs)
            return false;
    return true;
}

// L2 eviction policies for the TMA loads (createpolicy; fraction 1.0).
__device__ __forceinline__ uint64_t l2_policy(int kind)
{
    uint64_t p;
    if (kind == 1)
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    else if (kind == 2)
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    else
        asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// G block of 32 columns x 32 rows from shared memory to global, clipped at
// the edges of G by the tensor map; one bulk group per call.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, uint32_t src, int x, int y, uint64_t pol)
{
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group.L2::cache_hint [%0, {%1, %2}], [%3], %4;" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(src), "l"(pol)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Wait until at most N bulk groups of this thread still read shared memory.
template <int N>
__device__ __forceinline__ void tma_store_wait_read()
{
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void tma_store_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor of tcgen05.mma for an MN-major operand
// with the 128-byte swizzle: start address, 10 KiB between 64-element blocks
// along M (or N) ("leading" offset), 1 KiB between groups of 8 rows along K
// ("stride" offset), descriptor version 1, swizzle mode 2 (128 bytes).
__device__ __forceinline__ uint64_t mn_major_sw128_desc(uint32_t saddr)
{
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((kBlockBytes >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((1024 >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator,
// bf16 A and B, both MN-major, N = 256, M = 256 (the pair).
constexpr uint32_t kInstrDesc = (1u << 4)               // D: f32
                                | (1u << 7)             // A: bf16
                                | (1u << 10)            // B: bf16
                                | (1u << 15)            // A MN-major
                                | (1u << 16)            // B MN-major
                                | ((uint32_t)(kBN >> 3) << 17)
                                | ((uint32_t)(kPairM >> 4) << 24);

// 32 consecutive fp32 accumulator columns of this thread's lane.
__device__ __forceinline__ void tmem_load32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int e = 0; e < 32; ++e)
        v[e] = __uint_as_float(r[e]);
}

// Named barrier 1 over the 128 epilogue threads.
__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

// Same barrier with an OR over the threads' flags: every epilogue thread gets
// the same answer, so the four warps always take the same branch.
__device__ __forceinline__ bool epi_bar_any(bool c)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, 1, 128, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)c)
        : "memory");
    return r != 0;
}

__device__ void set_timeout(volatile int *abort, unsigned *flags)
{
    *abort = 1;
    atomicOr(flags, kFlagTimeout);
}

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_id()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_count()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
    return r;
}
// Every thread of every CTA of the cluster: arrive, then wait for all.
__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Address of the same shared-memory variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_rank(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr)
{
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// One 64 x 64 box into this CTA's shared memory; its bytes complete on the
// barrier `bar` (a cluster address: the leader's barrier for both CTAs).
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint32_t bar,
                                            uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
        ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(kInstrDesc), "r"(acc)
        : "memory");
}

// Arrive on the barrier at `bar`'s offset in both CTAs of the pair once the
// MMAs issued so far by this thread have completed.
__device__ __forceinline__ void mma_commit_mc(uint32_t bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
        "h"((uint16_t)3)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// Pair tile gt -> (row block mb of this CTA, column block nb).  Column
// blocks are taken in bands of `band`; within a band the row pairs go in
// order and the column blocks of the band vary fastest, so the CTAs working
// at the same time share few slices of H and few of dlogits.
__device__ __forceinline__ void tile_of(int gt, int nblocks, int mpairs, int band, int rank, int &mb, int &nb)
{
    const int per_band = band * mpairs;
    const int b = gt / per_band;
    const int r = gt - b * per_band;
    const int nb0 = b * band;
    const int w = (nblocks - nb0 < band) ? nblocks - nb0 : band;  // the last band may be narrower
    const int mp = r / w;
    nb = nb0 + (r - mp * w);
    mb = mp * 2 + rank;
}

// G = dlogits^T H, one CTA of a pair.  Outputs:
//   G        V x D fp32, row-major (TMA stores through tm_g)
//   colpart  [ceil(V/128)][D]: sum of g^2 over the 128 rows of each row block
//   rowpart  [ceil(D/256)][V]: sum of g^2 over the 256 columns of each column block
__global__ void __launch_bounds__(kLmThreads, 1)
k_lmhead_grad(const __grid_constant__ CUtensorMap tm_dl, const __grid_constant__ CUtensorMap tm_h,
              const __grid_constant__ CUtensorMap tm_g, float *__restrict__ colpart, float *__restrict__ rowpart,
              unsigned *flags, int V, int D, int T, int band, uint64_t wait_ns)
{
    extern __shared__ unsigned char lm_smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(lm_smem_raw) + 1023) & ~(uintptr_t)1023);
    unsigned char *gstage = smem + (size_t)kStages * kStageBytes;
    LmSmemTail *tail = reinterpret_cast<LmSmemTail *>(gstage + kStoreBytes);
    volatile int *abort = &tail->abort;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int mblocks = (V + kBM - 1) / kBM;
    const int nblocks = (D + kBN - 1) / kBN;
    const int mpairs = (mblocks + 1) / 2;
    const int npair_tiles = mpairs * nblocks;
    const int kblocks = (T + kBK - 1) / kBK;
    const int rank = (int)cluster_rank();
    const bool leader = rank == 0;
    const int gt0 = (int)cluster_id();
    const int gstep = (int)cluster_count();

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_addr(&tail->full[s]), 1);
            mbar_init(smem_addr(&tail->empty[s]), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(smem_addr(&tail->tfull[a]), 1);
            mbar_init(smem_addr(&tail->tempty[a]), 8);  // four epilogue warps in each CTA
        }
        mbar_init(smem_addr(&tail->drain), 1);
        tail->abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_dl)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_h)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_g)) : "memory");
    }
    if (warp == 1) {
        // one warp in each CTA of the pair allocates, together
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_addr(&tail->tmem_base)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    // no peer may signal this CTA's barriers before they are initialised
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = tail->tmem_base;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer (both CTAs) ----------------
        int stage = 0;
        uint32_t phase = 0;
        uint32_t last_parity[kStages];
        bool issued[kStages];
        for (int s = 0; s < kStages; ++s) {
            issued[s] = false;
            last_parity[s] = 0;
        }
        const uint64_t pol_a = l2_policy(0);
        const uint64_t pol_b = l2_policy(1);
        bool ok = true;
        for (int gt = gt0; gt < npair_tiles && ok; gt += gstep) {
            int mb, nb;
            tile_of(gt, nblocks, mpairs, band, rank, mb, nb);
            for (int kb = 0; kb < kblocks; ++kb) {
                // both CTAs' halves of this stage were read by the pair's MMAs
                if (!mbar_wait(smem_addr(&tail->empty[stage]), phase ^ 1u, abort, wait_ns)) {
                    ok = false;
                    break;
                }
                const uint32_t my_full = smem_addr(&tail->full[stage]);
                if (leader)
                    mbar_expect_tx(my_full, 2 * kStageBytes);  // both CTAs' bytes land on the leader's barrier
                const uint32_t bar = mapa_rank(my_full, 0);
                issued[stage] = true;
                last_parity[stage] = phase;
                const uint32_t a_dst = smem_addr(smem + (size_t)stage * kStageBytes);
                const uint32_t b_dst = a_dst + kABytes;
                const int y = kb * kBK;
#pragma unroll
                for (int j = 0; j < kBM / kBox; ++j)
                    tma_load_2d(a_dst + j * kBlockBytes, &tm_dl, mb * kBM + j * kBox, y, bar, pol_a);
#pragma unroll
                for (int j = 0; j < (kBN / 2) / kBox; ++j)
                    tma_load_2d(b_dst + j * kBlockBytes, &tm_h, nb * kBN + rank * (kBN / 2) + j * kBox, y,
                                bar, pol_b);
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
        }
        if (!ok)
            set_timeout(abort, flags);
        // After an abort, copies already issued may still be on their way:
        // the leader waits for the last phase of each stage (both CTAs'
        // bytes complete there; immediate when every stage was consumed)
        // before the pair meets at the final cluster barrier.
        if (leader)
            for (int s = 0; s < kStages; ++s)
                if (issued[s])
                    mbar_wait_final(smem_addr(&tail->full[s]), last_parity[s]);
    } else if (warp == 1 && lane == 0 && leader) {
        // ---------------- MMA issuer (leader only) ----------------
        int stage = 0;
        uint32_t phase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        for (int gt = gt0; gt < npair_tiles && ok; gt += gstep) {
            if (!mbar_wait(smem_addr(&tail->tempty[acc]), acc_phase ^ 1u, abort, wait_ns)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t d_tmem = tmem + (uint32_t)(acc * kAccCols);
            for (int kb = 0; kb < kblocks; ++kb) {
                if (!mbar_wait(smem_addr(&tail->full[stage]), phase, abort, wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a_base = smem_addr(smem + (size_t)stage * kStageBytes);
                const uint32_t b_base = a_base + kABytes;
#pragma unroll
                for (int k = 0; k < kBK / kUK; ++k) {
                    // K step k: token rows 16k .. 16k+15 of every box, 2 KiB further on;
                    // the same offsets address the peer's halves
                    const uint64_t ad = mn_major_sw128_desc(a_base + (uint32_t)(k * kUK * 128));
                    const uint64_t bd = mn_major_sw128_desc(b_base + (uint32_t)(k * kUK * 128));
                    mma_bf16(d_tmem, ad, bd, (kb | k) != 0);
                }
                mma_commit_mc(smem_addr(&tail->empty[stage]));
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok)
                break;
            mma_commit_mc(smem_addr(&tail->tfull[acc]));
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if (!ok)
            set_timeout(abort, flags);
        // every MMA issued above completes before either CTA frees its tensor memory
        mma_commit(smem_addr(&tail->drain));
        mbar_wait_final(smem_addr(&tail->drain), 0);
    } else if (warp >= kEpiWarp0) {
        // ---------------- epilogue (both CTAs) ----------------
        const int q = warp - kEpiWarp0;  // accumulator lanes 32q .. 32q+31
        int acc = 0;
        uint32_t acc_phase = 0;
        int buf = 0;
        int sbuf = 0;
        unsigned char *my_stage = gstage + (size_t)q * kStoreBufs * kStoreBlockBytes;
        const uint64_t pol_g = l2_policy(2);
        for (int gt = gt0; gt < npair_tiles; gt += gstep) {
            int mb, nb;
            tile_of(gt, nblocks, mpairs, band, rank, mb, nb);
            bool fail = !mbar_wait(smem_addr(&tail->tfull[acc]), acc_phase, abort, wait_ns);
            if (fail && !*abort)
                set_timeout(abort, flags);
            fail = fail || *abort;
            if (epi_bar_any(fail))  // all four warps leave together
                break;
            tc_fence_after();
            const int row = mb * kBM + q * 32 + lane;
            float rowsq = 0.f;
#pragma unroll 1
            for (int ch = 0; ch < kBN / 32; ++ch) {
                float v[32];
                tmem_load32(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kAccCols + ch * 32), v);
                const int col0 = nb * kBN + ch * 32;
                const int row0 = mb * kBM + q * 32;
                // G block (32 rows x 32 columns) through shared memory: row
                // `lane` is 128 bytes, its 16-byte pieces in the 128-byte
                // swizzle order; then one TMA store, clipped at V and D
                if (row0 < V) {
                    if (lane == 0)
                        tma_store_wait_read<kStoreBufs - 1>();  // this staging block's previous store has read it
                    __syncwarp();
                    unsigned char *blk = my_stage + sbuf * kStoreBlockBytes + lane * 128;
#pragma unroll
                    for (int c = 0; c < 8; ++c)
                        *reinterpret_cast<float4 *>(blk + ((c ^ (lane & 7)) << 4)) =
                            make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    if (lane == 0)
                        tma_store_2d(&tm_g, smem_addr(my_stage + sbuf * kStoreBlockBytes), col0, row0, pol_g);
                    sbuf = (sbuf + 1 == kStoreBufs) ? 0 : sbuf + 1;
                }
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    v[e] = v[e] * v[e];
                    rowsq += v[e];
                }
                int col_of_lane;
                const float cs = dev::warp_sum_transposed<32>(v, lane, col_of_lane);
                tail->xch[buf][q][col_of_lane] = cs;
                epi_bar();
                if (q == 0 && mb < mblocks && col0 + lane < D)
                    colpart[(int64_t)mb * D + col0 + lane] =
                        ((tail->xch[buf][0][lane] + tail->xch[buf][1][lane]) + tail->xch[buf][2][lane]) +
                        tail->xch[buf][3][lane];
                buf ^= 1;
            }
            if (row < V)
                rowpart[(int64_t)nb * V + row] = rowsq;
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive_cluster(mapa_rank(smem_addr(&tail->tempty[acc]), 0));  // the leader's barrier
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
    }

    if (warp >= kEpiWarp0 && lane == 0)
        tma_store_wait_all();  // the stores of G have completed
    tc_fence_before();
    __syncthreads();
    // neither CTA frees its tensor memory or exits while its peer may still
    // use them (the leader's MMAs write both; arrivals cross the pair)
    cluster_sync();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols)
                     : "memory");
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// G, V x D fp32 row-major, stored as 32 x 32 boxes with the 128-byte swizzle.
bool make_store_map(CUtensorMap *m, float *G, int64_t V, int64_t D)
{
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)V};
    cuuint64_t strides[1] = {(cuuint64_t)D * 4};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, G, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// T x n bf16, row-major, loaded as 64 x 64 boxes with the 128-byte swizzle.
bool make_map(CUtensorMap *m, const void *base, int64_t n, int64_t T)
{
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn)
        return false;
    cuuint64_t dims[2] = {(cuuint64_t)n, (cuuint64_t)T};
    cuuint64_t strides[1] = {(cuuint64_t)n * 2};
    cuuint32_t box[2] = {(cuuint32_t)kBox, (cuuint32_t)kBK};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int lmhead_row_blocks(int64_t V) { return (int)((V + kBM - 1) / kBM); }
int lmhead_col_blocks(int64_t D) { return (int)((D + kBN - 1) / kBN); }

cudaError_t launch_lmhead_grad(const LmArgs &a, float *colpart, float *rowpart, unsigned *flags,
                               cudaStream_t stream)
{
    CUtensorMap tm_dl, tm_h, tm_g;
    if (!make_map(&tm_dl, a.dlogits, a.V, a.T) || !make_map(&tm_h, a.hidden, a.D, a.T) ||
        !make_store_map(&tm_g, a.G, a.V, a.D))
        return cudaErrorInvalidValue;
    // per device and cheap: set on every call
    cudaError_t e = cudaFuncSetAttribute(k_lmhead_grad, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kLmSmemBytes);
    if (e != cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(kLmThreads);
    cfg.dynamicSmemBytes = kLmSmemBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    // persistent: as many pairs as fit on the GPU at once
    cfg.gridDim = dim3(kSms);
    int fit = 0;
    e = cudaOccupancyMaxActiveClusters(&fit, k_lmhead_grad, &cfg);
    if (e != cudaSuccess)
        return e;
    if (fit < 1)
        return cudaErrorInvalidConfiguration;
    const int pairs = (lmhead_row_blocks(a.V) + 1) / 2 * lmhead_col_blocks(a.D);
    const int nclusters = pairs < fit ? pairs : fit;
    cfg.gridDim = dim3(nclusters * 2);
    const int band = kLmBand < lmhead_col_blocks(a.D) ? kLmBand : lmhead_col_blocks(a.D);
    return cudaLaunchKernelEx(&cfg, k_lmhead_grad, tm_dl, tm_h, tm_g, colpart, rowpart, flags, (int)a.V,
                              (int)a.D, (int)a.T, band, a.wait_ns ? a.wait_ns : kDefaultWaitNs);
}

}  // namespace ember
