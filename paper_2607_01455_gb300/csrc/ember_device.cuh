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

}  // namespace dev
}  // namespace ember
