// One AdamW step over a batch of tensors that also takes each tensor's
// absmax of the updated weights: the first half of the fused AdamW + NVFP4
// step (the NVFP4 reconstruction of w' needs the tensor scale of w' before
// any block is processed).  The arithmetic is the integer kernel's fused
// step, element for element: packed fp32, the root as v' rsqrt(v'), the
// quotient by the fast reciprocal, and w' = w + (-(w lr wd) - step m'/den)
// rounded once.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

#include "device_common.cuh"
#include "params.h"

namespace quasar {

// blockIdx.y picks the tensor; each thread takes 4 consecutive elements at a
// time (n is a multiple of 16).  *slot must start at 0.
template <int MAXT>
__global__ void __launch_bounds__(256) k_adamw_amax(const __grid_constant__ AdamwBatch<MAXT> B)
{
    const AdamwItem& it = B.t[blockIdx.y];
    const AdamwHp& hp = B.hp;
    if (it.n == 0) return;
    const float2 beta12 = make_float2(hp.beta1, hp.beta1), c1b2 = make_float2(hp.c1b, hp.c1b);
    const float2 beta22 = make_float2(hp.beta2, hp.beta2), c12 = make_float2(hp.c1, hp.c1);
    const float2 nlrwd2 = make_float2(-hp.lr_wd, -hp.lr_wd);
    const float2 nstep2 = make_float2(-hp.step_size, -hp.step_size);
    const float2 isbc22 = make_float2(hp.isbc2, hp.isbc2), eps2 = make_float2(hp.eps, hp.eps);
    float amax = 0.0f;
    const int64_t n4 = it.n / 4;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float4 w4 = __ldcs(reinterpret_cast<const float4*>(it.w) + i);
        const float4 m4 = __ldcs(reinterpret_cast<const float4*>(it.m) + i);
        const float4 v4 = __ldcs(reinterpret_cast<const float4*>(it.v) + i);
        float2 gv[2];
        if (hp.g_kind == 2) {
            const uint2 gb = __ldcs(reinterpret_cast<const uint2*>(it.g) + i);
            gv[0] = make_float2(bf16lo(gb.x), bf16hi(gb.x));
            gv[1] = make_float2(bf16lo(gb.y), bf16hi(gb.y));
        } else {
            const float4 g4 = __ldcs(reinterpret_cast<const float4*>(it.g) + i);
            gv[0] = make_float2(g4.x, g4.y);
            gv[1] = make_float2(g4.z, g4.w);
        }
        float2 wv[2] = {make_float2(w4.x, w4.y), make_float2(w4.z, w4.w)};
        float2 mv[2] = {make_float2(m4.x, m4.y), make_float2(m4.z, m4.w)};
        float2 hv[2] = {make_float2(v4.x, v4.y), make_float2(v4.z, v4.w)};
#pragma unroll
        for (int pr = 0; pr < 2; ++pr) {
            mv[pr] = __ffma2_rn(mv[pr], beta12, __fmul2_rn(c1b2, gv[pr]));
            hv[pr] = __ffma2_rn(hv[pr], beta22, __fmul2_rn(c12, __fmul2_rn(gv[pr], gv[pr])));
            float2 sq = __fmul2_rn(hv[pr], make_float2(rsqrtf(hv[pr].x), rsqrtf(hv[pr].y)));
            sq.x = hv[pr].x > 0.0f ? sq.x : 0.0f;
            sq.y = hv[pr].y > 0.0f ? sq.y : 0.0f;
            const float2 den = __ffma2_rn(sq, isbc22, eps2);
            const float2 upd = make_float2(__fdividef(mv[pr].x, den.x), __fdividef(mv[pr].y, den.y));
            const float2 t = __ffma2_rn(wv[pr], nlrwd2, __fmul2_rn(nstep2, upd));
            wv[pr] = __fadd2_rn(wv[pr], t);
            amax = fmaxf(amax, fmaxf(fabsf(wv[pr].x), fabsf(wv[pr].y)));
        }
        __stcs(reinterpret_cast<float4*>(it.w) + i, make_float4(wv[0].x, wv[0].y, wv[1].x, wv[1].y));
        __stcs(reinterpret_cast<float4*>(it.m) + i, make_float4(mv[0].x, mv[0].y, mv[1].x, mv[1].y));
        __stcs(reinterpret_cast<float4*>(it.v) + i, make_float4(hv[0].x, hv[0].y, hv[1].x, hv[1].y));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    __shared__ float red[32];
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = amax;
    __syncthreads();
    if (threadIdx.x < 32) {
        amax = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0f;
#pragma unroll
        for (int o = 16; o; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
        if (threadIdx.x == 0 && amax > 0.0f)
            atomicMax(reinterpret_cast<unsigned int*>(it.slot), __float_as_uint(amax));
    }
}

}  // namespace quasar
