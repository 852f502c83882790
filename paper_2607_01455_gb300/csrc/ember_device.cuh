// Device helpers shared by the CUDA translation units of libember:
// vector access types, fp32/bf16 loads and stores, warp reductions.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ember {
namespace dev {

// Programmatic dependent launch: wait until the kernels this one depends on
// have completed and their writes are visible (a no-op when launched
// without the attribute), and allow the next kernel to start launching.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;"); }

template <int VEC> struct Vec;
template <> struct Vec<4> { using F = float4; };
template <> struct Vec<1> { using F = float; };

__device__ __forceinline__ float comp(const float4 &v, int e)
{
    return e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
}
__device__ __forceinline__ float comp(const float &v, int) { return v; }
__device__ __forceinline__ void set_comp(float4 &v, int e, float x)
{
    if (e == 0) v.x = x; else if (e == 1) v.y = x; else if (e == 2) v.z = x; else v.w = x;
}
__device__ __forceinline__ void set_comp(float &v, int, float x) { v = x; }

template <int VEC>
__device__ __forceinline__ typename Vec<VEC>::F load_g(const float *p)
{
    if constexpr (VEC == 4)
        return __ldg(reinterpret_cast<const float4 *>(p));
    else
        return __ldg(p);
}

template <int VEC>
__device__ __forceinline__ typename Vec<VEC>::F zero_vec()
{
    if constexpr (VEC == 4)
        return make_float4(0.f, 0.f, 0.f, 0.f);
    else
        return 0.f;
}

// Sum R per-lane values over the 32 lanes of a warp, "transposed": each
// halving step trades half of the values with a partner lane, so the R
// totals cost R-1 + log2(32/R) shuffles instead of 5R.  On return v[0] of
// lane l is the warp total of value index `row` (lanes whose low
// log2(32/R) bits differ hold the same total).  The addition tree is fixed,
// so the result is the same on every run.
template <int R>
__device__ __forceinline__ float warp_sum_transposed(float (&v)[R], int lane, int &row)
{
    static_assert(R >= 1 && R <= 32 && (R & (R - 1)) == 0, "R must be a power of two <= 32");
    constexpr int kLog = (R >= 32) ? 5 : (R >= 16) ? 4 : (R >= 8) ? 3 : (R >= 4) ? 2 : (R >= 2) ? 1 : 0;
    row = 0;
#pragma unroll
    for (int s = 0; s < kLog; ++s) {
        const int o = 16 >> s;
        const int h = R >> (s + 1);
        const bool hi = (lane & o) != 0;
#pragma unroll
        for (int m = 0; m < h; ++m) {
            const float send = hi ? v[m] : v[m + h];
            const float keep = hi ? v[m + h] : v[m];
            v[m] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
        if (hi)
            row += h;
    }
#pragma unroll
    for (int o = 16 >> kLog; o >= 1; o >>= 1)
        v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
    return v[0];
}

__device__ __forceinline__ float bf16_lo(unsigned u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(unsigned u) { return __uint_as_float(u & 0xFFFF0000u); }
__device__ __forceinline__ unsigned short f2bf(float x)
{
    return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

// Raw weight vectors: kept packed between the load and the update.
template <bool BF16, int VEC> struct WRaw;
template <> struct WRaw<true, 4> { using T = uint2; };
template <> struct WRaw<true, 1> { using T = unsigned short; };
template <> struct WRaw<false, 4> { using T = float4; };
template <> struct WRaw<false, 1> { using T = float; };

template <bool BF16, int VEC>
__device__ __forceinline__ typename WRaw<BF16, VEC>::T load_w(const void *W, int64_t idx)
{
    using T = typename WRaw<BF16, VEC>::T;
    if constexpr (BF16)
        return *reinterpret_cast<const T *>(static_cast<const unsigned short *>(W) + idx);
    else
        return *reinterpret_cast<const T *>(static_cast<const float *>(W) + idx);
}

__device__ __forceinline__ void unpack_w(const uint2 &u, float (&w)[4])
{
    w[0] = bf16_lo(u.x); w[1] = bf16_hi(u.x); w[2] = bf16_lo(u.y); w[3] = bf16_hi(u.y);
}
__device__ __forceinline__ void unpack_w(const unsigned short &u, float (&w)[1])
{
    w[0] = __uint_as_float((unsigned)u << 16);
}
__device__ __forceinline__ void unpack_w(const float4 &f, float (&w)[4])
{
    w[0] = f.x; w[1] = f.y; w[2] = f.z; w[3] = f.w;
}
__device__ __forceinline__ void unpack_w(const float &f, float (&w)[1]) { w[0] = f; }

template <bool BF16, int VEC>
__device__ __forceinline__ void store_w(void *W, int64_t idx, const float (&w)[VEC])
{
    if constexpr (BF16 && VEC == 4) {
        uint2 u;
        u.x = (unsigned)f2bf(w[0]) | ((unsigned)f2bf(w[1]) << 16);
        u.y = (unsigned)f2bf(w[2]) | ((unsigned)f2bf(w[3]) << 16);
        *reinterpret_cast<uint2 *>(static_cast<unsigned short *>(W) + idx) = u;
    } else if constexpr (BF16) {
        static_cast<unsigned short *>(W)[idx] = f2bf(w[0]);
    } else if constexpr (VEC == 4) {
        *reinterpret_cast<float4 *>(static_cast<float *>(W) + idx) = make_float4(w[0], w[1], w[2], w[3]);
    } else {
        static_cast<float *>(W)[idx] = w[0];
    }
}

// L2 eviction-priority policies (createpolicy, fraction 1.0) and loads and
// stores that carry one: evict_first for data touched for the last time in
// a launch, so that it leaves L2 before data still to be reused.
__device__ __forceinline__ uint64_t policy_evict_first()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_last()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

template <int VEC>
__device__ __forceinline__ typename Vec<VEC>::F load_g_hint(const float *p, uint64_t pol)
{
    if constexpr (VEC == 4) {
        float4 v;
        asm volatile("ld.global.nc.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                     : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                     : "l"(p), "l"(pol));
        return v;
    } else {
        float v;
        asm volatile("ld.global.nc.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(p), "l"(pol));
        return v;
    }
}

template <bool BF16, int VEC>
__device__ __forceinline__ typename WRaw<BF16, VEC>::T load_w_hint(const void *W, int64_t idx, uint64_t pol)
{
    if constexpr (BF16 && VEC == 4) {
        uint2 u;
        asm volatile("ld.global.L2::cache_hint.v2.u32 {%0, %1}, [%2], %3;"
                     : "=r"(u.x), "=r"(u.y)
                     : "l"(static_cast<const unsigned short *>(W) + idx), "l"(pol));
        return u;
    } else if constexpr (!BF16 && VEC == 4) {
        float4 v;
        asm volatile("ld.global.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                     : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                     : "l"(static_cast<const float *>(W) + idx), "l"(pol));
        return v;
    } else {
        return load_w<BF16, VEC>(W, idx);
    }
}

template <bool BF16, int VEC>
__device__ __forceinline__ void store_w_hint(void *W, int64_t idx, const float (&w)[VEC], uint64_t pol)
{
    if constexpr (BF16 && VEC == 4) {
        const unsigned x = (unsigned)f2bf(w[0]) | ((unsigned)f2bf(w[1]) << 16);
        const unsigned y = (unsigned)f2bf(w[2]) | ((unsigned)f2bf(w[3]) << 16);
        asm volatile("st.global.L2::cache_hint.v2.u32 [%0], {%1, %2}, %3;" ::"l"(
                         static_cast<unsigned short *>(W) + idx),
                     "r"(x), "r"(y), "l"(pol)
                     : "memory");
    } else if constexpr (!BF16 && VEC == 4) {
        asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(
                         static_cast<float *>(W) + idx),
                     "f"(w[0]), "f"(w[1]), "f"(w[2]), "f"(w[3]), "l"(pol)
                     : "memory");
    } else {
        store_w<BF16, VEC>(W, idx, w);
    }
}

template <int VEC>
__device__ __forceinline__ void store_g_hint(float *p, const typename Vec<VEC>::F &v, uint64_t pol)
{
    if constexpr (VEC == 4)
        asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x), "f"(v.y),
                     "f"(v.z), "f"(v.w), "l"(pol)
                     : "memory");
    else
        asm volatile("st.global.L2::cache_hint.f32 [%0], %1, %2;" ::"l"(p), "f"(v), "l"(pol) : "memory");
}

// The update ratio g / (sqrt(rhat_i) sqrt(chat_j / s) + eps) of Algorithm 1,
// with the fast reciprocal-and-multiply division (within 2 fp32 ulps for a
// denominator below 2^126; the denominator here is a gradient-sized positive
// number).  Every kernel that applies an update uses this one form, so the
// dense, sparse, one-launch and sharded steps stay bitwise identical.
__device__ __forceinline__ float update_ratio(float g, float den) { return __fdividef(g, den); }

__device__ __forceinline__ uint64_t now_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ unsigned ld_acquire(const unsigned *p)
{
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// ---------------------------------------------------------------------------
// Exact sums of non-negative fp32 values in 64-bit fixed point.
//
// The statistics of a step are sums over the whole table of per-CTA fp32
// partial sums (of g^2 per column, of the new r per row block).  Adding
// those partials as integers makes the total independent of how they are
// grouped: the same bits whether one CTA, the state pass or an all-reduce
// across row shards forms it.  The scale is shared by all partials of one
// sum: E, the largest biased fp32 exponent among them, maps the largest
// partial below 2^(24 + kFxShift) = 2^50, so that up to 4096 partials add
// up below 2^62 without overflow.  A partial 2^k times smaller than the
// largest loses its lowest max(0, k - 26) bits; the total is exact to
// within 2^-41 of itself for 304 partials.  NaN or Inf partials (biased
// exponent 255, or a sign bit) make the total NaN or Inf as a float sum
// would.
// ---------------------------------------------------------------------------
constexpr int kFxShift = 26;
constexpr unsigned kFxSpecial = 255u;

// Key of p for the shared scale: its biased exponent (0 for zero and
// subnormals), 255 for NaN, Inf or a negative value.
__device__ __forceinline__ unsigned fx_key(float p)
{
    const unsigned b = __float_as_uint(p);
    return (b >> 23) > 254u ? kFxSpecial : (b >> 23);
}

// p in units of 2^(max(E,1) - 150 - kFxShift), where E >= fx_key(p) is the
// largest key among the values summed.  When E == 255 (some value is NaN,
// Inf or negative) the units change meaning: NaN counts 2^32, +Inf counts 1,
// anything else 0, so that every grouping of the same values gives the
// same total and fx_value() tells NaN from Inf.
__device__ __forceinline__ unsigned long long fx_of(float p, unsigned E)
{
    const unsigned b = __float_as_uint(p);
    if (E >= kFxSpecial)
        return isnan(p) ? (1ull << 32) : (b == 0x7F800000u ? 1ull : 0ull);
    const unsigned ef = b >> 23;
    const unsigned long long M = (b & 0x7FFFFFu) | (ef ? 0x800000u : 0u);
    const int sh = (int)(ef ? ef : 1u) - (int)(E ? E : 1u) + kFxShift;
    if (sh >= 0)
        return M << sh;
    return sh > -32 ? (M >> (unsigned)(-sh)) : 0ull;
}

// The fixed-point total S at scale exponent E as a float: S rounded to
// fp32, then scaled by 2^(max(E,1) - 150 - kFxShift) in two exact steps (the
// total is at least 2^(E - 127) when E >= 1, so neither step underflows
// before the last); NaN or +Inf when E == 255.
__device__ __forceinline__ float fx_value(unsigned long long S, unsigned E)
{
    if (E >= kFxSpecial)
        return (S >> 32) ? __uint_as_float(0x7FC00000u) : __uint_as_float(0x7F800000u);
    const float x = (float)S;  // S < 2^62
    return (x * 0x1p-49f) * __uint_as_float((E ? E : 1u) << 23);  // 2^-49 * 2^(E-127)
}

__device__ __forceinline__ unsigned long long shfl_xor_u64(unsigned long long x, int m)
{
    const unsigned lo = __shfl_xor_sync(0xffffffffu, (unsigned)x, m);
    const unsigned hi = __shfl_xor_sync(0xffffffffu, (unsigned)(x >> 32), m);
    return ((unsigned long long)hi << 32) | lo;
}

}  // namespace dev
}  // namespace ember
