// Device-side building blocks shared by the QUASAR kernels (sm_103a):
// mbarrier + 1-D TMA bulk copies (global -> shared), a bounded wait that
// records a timeout instead of spinning forever, and small numeric helpers.
#pragma once

#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "params.h"

namespace quasar {


__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}

// Make barrier initialisation visible to the async (TMA) proxy.
__device__ __forceinline__ void mbar_init_fence()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t global_timer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

// Wait until the barrier phase with the given parity completes, or until
// limit_ns nanoseconds have passed.  Returns false on timeout.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
#pragma unroll 1
        for (int i = 0; i < 32; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (global_timer_ns() - t0 > limit_ns) return false;
    }
}

// The bounded wait of a whole warp, with one outcome for all its lanes.  Each
// lane waits on the barrier itself (so each observes the completed phase and
// the data the copies delivered), and the warp reports a timeout if any
// lane's own limit ran out: no lane takes the failure path while others go
// on to warp-wide shuffles.  Every lane of the warp must call it.
__device__ __forceinline__ bool warp_wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns)
{
    return __all_sync(0xffffffffu, mbar_wait_bounded(bar, parity, limit_ns));
}

// 1-D bulk copy global -> shared, completion counted in bytes on `bar`.
// dst, src and bytes must be multiples of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void record_timeout(unsigned int* status)
{
    atomicOr(status, kStatusTimeout);
}

__device__ __forceinline__ float4 lds128(const void* p)
{
    return *reinterpret_cast<const float4*>(p);
}

__device__ __forceinline__ uint2 lds64(const void* p) { return *reinterpret_cast<const uint2*>(p); }

// Minimum / maximum of x over the lanes of `mask` in one warp reduction (used
// over the whole warp: with a mask per 8-lane segment it ran slower than
// three shuffle steps).  NaN inputs are ignored, as by fminf / fmaxf.
__device__ __forceinline__ float lanes_min(float x, unsigned mask)
{
    float r;
    asm volatile("redux.sync.min.f32 %0, %1, %2;" : "=f"(r) : "f"(x), "r"(mask));
    return r;
}

__device__ __forceinline__ float lanes_max(float x, unsigned mask)
{
    float r;
    asm volatile("redux.sync.max.f32 %0, %1, %2;" : "=f"(r) : "f"(x), "r"(mask));
    return r;
}

// Three-input minimum / maximum (one instruction each on sm_100 and later).
__device__ __forceinline__ float fmin3(float a, float b, float c)
{
    float r;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

__device__ __forceinline__ float fmax3(float a, float b, float c)
{
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

__device__ __forceinline__ float bf16lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16hi(uint32_t x) { return __uint_as_float(x & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&p);
}

// Streaming (evict-first) global stores: every output is written once.
__device__ __forceinline__ void stg_cs(float4* p, float4 v) { __stcs(p, v); }
__device__ __forceinline__ void stg_cs(uint2* p, uint2 v) { __stcs(p, v); }
__device__ __forceinline__ void stg_cs(uint32_t* p, uint32_t v)
{
    __stcs(reinterpret_cast<unsigned int*>(p), v);
}

// 1.5 * 2^23: adding it to a float in [0, 2^22) rounds that float to an
// integer (round-to-nearest-even) in the low mantissa bits.
constexpr float kRoundMagic = 12582912.0f;

// Saliency sums near the bottom of fp32's range: the reconstruction is
// invariant to a common scale of h (Algorithm 1's argmin and Eq. 4's fit), so
// a group (or block) whose sum of h is below 2^-40 is fitted with h scaled by a
// power of two s = s1 s2, exactly, chosen so that x s lies in [1, 2) for the
// sum x: the products of its moment sums then stay normal.  Two factors,
// because s can exceed the largest float power of two 2^127.
constexpr float kTinySaliency = 9.094947e-13f;  // 2^-40

__device__ __forceinline__ void tiny_scale(float x, float& s1, float& s2)
{
    s1 = 1.0f;
    if (x < 1.17549435e-38f) {  // denormal: first 2^64
        s1 = 18446744073709551616.0f;
        x *= s1;
    }
    const int e = (int)((__float_as_uint(x) >> 23) & 0xFFu) - 127;  // x = 1.f 2^e
    s2 = __uint_as_float((uint32_t)(127 - e) << 23);
}

}  // namespace quasar
