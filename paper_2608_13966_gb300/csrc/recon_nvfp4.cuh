// QUASAR for NVFP4 (Sec. 4.2): E2M1 codes, one E4M3 scale per 16-element
// block, one fp32 scale per tensor s_T = amax/(6*448).  For each block and
// each search factor f: sigma = f*amax_b/6, codes on the E2M1 grid of
// |w|/sigma (saturating at 6, ties to even), least-squares slope
// a* = sum h q w / sum h q^2, E4M3 scale e = rne_satfinite(a* / s_T) (the
// nearest E4M3 value is exactly optimal because the error is a symmetric
// quadratic in the scale), error sum h (s_T*e*q - w)^2; keep the lowest.
//
// Decomposition: one lane owns one block (16 elements), so the search needs
// no cross-lane traffic; a warp owns 32 consecutive blocks (512 elements) at
// a time, staged through its own ring of shared-memory buffers filled by 1-D
// TMA bulk copies, exactly as the integer kernel.  A lane reads its block's
// four 16-byte chunks in a lane-rotated order so that each shared-memory
// access of the warp is bank-conflict free.  Arithmetic is packed f32x2, two
// elements per instruction.
//
// Per candidate the codes stay in registers: moments -> a* -> E4M3 scale,
// then the error summed directly, sum h (alpha*q - |w|)^2 (no cancellation,
// so its fp32 error is a few ulps of itself).  Candidates within that bound
// of the best, unless their codes and scale equal the best's (the sum of
// codes never decreases with the scale factor, so equal sums mean equal
// codes), are re-evaluated exactly in float-float arithmetic.
#pragma once

#include <cuda_fp16.h>

#include "device_common.cuh"
#include "params.h"

namespace quasar {

__device__ __forceinline__ float tensor_scale_of(float amax)
{
    return amax > 0.0f ? __fdiv_rn(amax, 2688.0f) : 1.0f;
}

// E4M3 (e4m3fn) round-to-nearest-even with saturation, and its value.
__device__ __forceinline__ uint32_t e4m3_rn_satfinite(float x)
{
    uint16_t r;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %1;" : "=h"(r) : "f"(x));
    return (uint32_t)(r & 0xFFu);
}

__device__ __forceinline__ float e4m3_value(uint32_t bits)
{
    // normal: exponent e - 7 + 127, mantissa m << 20; subnormal (e = 0): m * 2^-9
    const uint32_t b = bits & 0x7Fu;
    const float normal = __uint_as_float((b << 20) + (120u << 23));
    return b < 8u ? (float)b * 0.001953125f : normal;
}

// E2M1 nibble of a value that lies on the signed E2M1 grid.
__device__ __forceinline__ uint32_t e2m1_nibble(float qs)
{
    uint16_t r;
    asm("{\n\t.reg .b8 t;\n\tcvt.rn.satfinite.e2m1x2.f32 t, %1, %1;\n\tcvt.u16.u8 %0, t;\n\t}"
        : "=h"(r)
        : "f"(qs));
    return (uint32_t)(r & 0xFu);
}

// Error-free transformations for the exact comparison (Knuth TwoSum,
// FMA-based TwoProd).
__device__ __forceinline__ void two_sum_f(float a, float b, float& s, float& e)
{
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

__device__ __forceinline__ void two_prod_f(float a, float b, float& p, float& e)
{
    p = __fmul_rn(a, b);
    e = fmaf(a, b, -p);
}

template <int NCH, int MAXT>
__global__ void __launch_bounds__(256) k_recon_nvfp4(const __grid_constant__ Nvfp4Launch<MAXT> Lp)
{
    const Nvfp4Params& p = Lp.p;
    constexpr int KM = NCH * 8;
    constexpr int UNIT = kBlocksPerUnit * 16;
    extern __shared__ __align__(128) unsigned char smem[];

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int S = p.stages;
    unsigned char* ring = smem + (size_t)warp * S * p.stage_bytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)nwarps * S * p.stage_bytes) + warp * (S + 1);

    const int gbytes = p.g_kind == 2 ? 2 : (p.g_kind == 1 ? 4 : 0);
    constexpr uint32_t kVOff = UNIT * 4;
    constexpr uint32_t kGOff = UNIT * 8;

    const int64_t n_units = Lp.n_units;
    // the tensor of a unit (units numbered consecutively across tensors,
    // met by each warp in increasing order)
    auto tensor_of = [&](int64_t u, int& ti) {
        while (ti + 1 < Lp.n_t && u >= Lp.t[ti + 1].unit0) ++ti;
    };
    int ti = 0, ti_s = -1;
    float sT = 1.0f, inv_sT = 1.0f;
    const int64_t first = (int64_t)blockIdx.x * nwarps + warp;
    const int64_t stride = (int64_t)gridDim.x * nwarps;


    if (lane == 0) {
        for (int s = 0; s <= S; ++s) mbar_init(&bars[s], 1);
        mbar_init_fence();
    }
    __syncwarp();

    auto issue = [&](int64_t u, int s) {
        int tj = ti;
        tensor_of(u, tj);
        const Nvfp4Tensor& T = Lp.t[tj];
        const int64_t b0 = (u - T.unit0) * kBlocksPerUnit;
        const int64_t nb = min((int64_t)kBlocksPerUnit, T.n_blocks - b0);
        const uint32_t elems = (uint32_t)(nb * 16);
        unsigned char* st = ring + (size_t)s * p.stage_bytes;
        mbar_arrive_expect_tx(&bars[s], elems * (8u + (uint32_t)gbytes));
        bulk_g2s(st, T.w + b0 * 16, elems * 4u, &bars[s]);
        bulk_g2s(st + kVOff, T.v + b0 * 16, elems * 4u, &bars[s]);
        if (gbytes)
            bulk_g2s(st + kGOff, static_cast<const unsigned char*>(T.g) + b0 * 16 * gbytes,
                     elems * (uint32_t)gbytes, &bars[s]);
    };
    auto fail = [&](int64_t it) {
        if (lane == 0) record_timeout(p.status);
        for (int j = 0; j < S; ++j) {
            const int64_t u = first + (it + j) * stride;
            if (u >= n_units) break;
            mbar_wait_bounded(&bars[(it + j) % S], (uint32_t)(((it + j) / S) & 1), p.timeout_ns);
        }
    };

    if (lane == 0)
        for (int s = 0; s < S; ++s) {
            const int64_t u = first + s * stride;
            if (u < n_units) issue(u, s);
        }
    if (p.force_timeout_ns && blockIdx.x == 0 && warp == 0) {
        if (!warp_wait_bounded(&bars[S], 0, p.force_timeout_ns)) {
            fail(0);
            return;
        }
    }

    const int rot = (lane >> 1) & 3;
    const float ulp = 5.9604645e-8f * p.tie_kappa;
    const float2 beta22 = make_float2(p.beta2, p.beta2);
    const float2 c12 = make_float2(p.c1, p.c1);
    const float2 six2 = make_float2(6.0f, 6.0f), neg12 = make_float2(-1.0f, -1.0f);
    int s_cur = 0;
    uint32_t parity = 0;

    // E2M1 magnitudes of two values y >= 0: the hardware conversion rounds
    // to nearest, ties to the even code, and saturates at 6; converting the
    // pair back through f16x2 gives their values (a goes to the upper half in
    // both conversions, so y.y is passed first)
    auto e2m1_2 = [](float2 y) -> float2 {
        uint32_t hh;
        asm("{\n\t.reg .b8 t;\n\tcvt.rn.satfinite.e2m1x2.f32 t, %1, %2;\n\tcvt.rn.f16x2.e2m1x2 %0, t;\n\t}"
            : "=r"(hh)
            : "f"(y.y), "f"(y.x));
        return __half22float2(*reinterpret_cast<__half2*>(&hh));
    };

    for (int64_t it = 0;; ++it) {
        const int64_t u = first + it * stride;
        if (u >= n_units) break;
        if (!warp_wait_bounded(&bars[s_cur], parity, p.timeout_ns)) {
            fail(it);
            return;
        }
        const unsigned char* st = ring + (size_t)s_cur * p.stage_bytes;

        // element 4*cidx[i] + jj of this lane's block is held at slot 4*i + jj,
        // pairs (slot 2t, 2t+1) in w2[t], h2[t]
        float2 w2[8], h2[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int cidx = (i + rot) & 3;
            const int e = lane * 16 + cidx * 4;
            const float4 w4 = lds128(st + e * 4);
            const float4 v4 = lds128(st + kVOff + e * 4);
            w2[2 * i] = make_float2(w4.x, w4.y);
            w2[2 * i + 1] = make_float2(w4.z, w4.w);
            float2 hA = make_float2(v4.x, v4.y), hB = make_float2(v4.z, v4.w);
            if (p.g_kind) {
                float2 gA, gB;
                if (p.g_kind == 2) {
                    const uint2 gb = lds64(st + kGOff + e * 2);
                    gA = make_float2(bf16lo(gb.x), bf16hi(gb.x));
                    gB = make_float2(bf16lo(gb.y), bf16hi(gb.y));
                } else {
                    const float4 g4 = lds128(st + kGOff + e * 4);
                    gA = make_float2(g4.x, g4.y);
                    gB = make_float2(g4.z, g4.w);
                }
                hA = __ffma2_rn(hA, beta22, __fmul2_rn(c12, __fmul2_rn(gA, gA)));
                hB = __ffma2_rn(hB, beta22, __fmul2_rn(c12, __fmul2_rn(gB, gB)));
            }
            h2[2 * i] = hA;
            h2[2 * i + 1] = hB;
        }
        __syncwarp();
        if (lane == 0) {
            const int64_t un = u + (int64_t)S * stride;
            if (un < n_units) issue(un, s_cur);
        }
        if (++s_cur == S) {
            s_cur = 0;
            parity ^= 1u;
        }

        tensor_of(u, ti);
        const Nvfp4Tensor& T = Lp.t[ti];
        if (ti != ti_s) {  // a new tensor: its scale s_T
            ti_s = ti;
            sT = *T.tensor_scale;
            inv_sT = 1.0f / sT;
        }
        const int64_t blk = (u - T.unit0) * kBlocksPerUnit + lane;
        const bool valid = blk < T.n_blocks;
        const int64_t ebase = blk * 16;

        if (valid && p.g_kind) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int cidx = (i + rot) & 3;
                stg_cs(reinterpret_cast<float4*>(T.v + ebase + cidx * 4),
                       make_float4(h2[2 * i].x, h2[2 * i].y, h2[2 * i + 1].x, h2[2 * i + 1].y));
            }
        }

        if (p.h_mode != kSalEma)  // the fit's saliency: v'^2 or 1
#pragma unroll
            for (int t = 0; t < 8; ++t)
                h2[t] = p.h_mode == kSalEmaSquared ? __fmul2_rn(h2[t], h2[t]) : make_float2(1.0f, 1.0f);

        float2 aw2[8], naw2[8];
        float amax_b = 0.0f;
        float2 SS = make_float2(0.0f, 0.0f);
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            aw2[t] = make_float2(fabsf(w2[t].x), fabsf(w2[t].y));
            naw2[t] = make_float2(-aw2[t].x, -aw2[t].y);
            amax_b = fmaxf(amax_b, fmaxf(aw2[t].x, aw2[t].y));
            SS = __fadd2_rn(SS, h2[t]);
        }
        const float ssb = SS.x + SS.y;
        if (__any_sync(0xffffffffu, ssb < kTinySaliency)) {
            if (ssb == 0.0f) {  // all saliencies zero: h = 1
#pragma unroll
                for (int t = 0; t < 8; ++t) h2[t] = make_float2(1.0f, 1.0f);
            } else if (ssb < kTinySaliency) {
                // near the bottom of the fp32 range: h scaled by a power of two
                float s1, s2;
                tiny_scale(ssb, s1, s2);
                const float2 s12 = make_float2(s1, s1), s22 = make_float2(s2, s2);
#pragma unroll
                for (int t = 0; t < 8; ++t) h2[t] = __fmul2_rn(__fmul2_rn(h2[t], s12), s22);
            }
        }
        const bool zero = !(amax_b > 0.0f);
        const float P1 = zero ? 0.0f : __fdiv_rn(6.0f, amax_b);  // 1/sigma at f = 1

        // ---- candidates: codes in registers, moments, E4M3 scale, direct error
        float Ek[KM];
        uint32_t Kk[KM];
        float Eb = INFINITY;
        int kb = 0;
        uint32_t e_sel = 0;
        float alpha_sel = 0.0f;
#pragma unroll
        for (int k = 0; k < KM; ++k) {
            const float P = P1 * p.invf[k];
            const float2 P2 = make_float2(P, P);
            float2 q2[8];
            float2 S2 = make_float2(0.0f, 0.0f), S3 = S2;
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                float2 y = __fmul2_rn(aw2[t], P2);
                q2[t] = e2m1_2(y);
                const float2 hq = __fmul2_rn(h2[t], q2[t]);
                S2 = __ffma2_rn(hq, q2[t], S2);
                S3 = __ffma2_rn(hq, aw2[t], S3);
            }
            const float s2 = S2.x + S2.y, s3 = S3.x + S3.y;
            // degenerate (every weighted element coded 0): the search scale
            const float x = s2 > 0.0f ? __fdividef(s3, s2) * inv_sT
                                      : amax_b * p.f[k] * (1.0f / 6.0f) * inv_sT;
            const uint32_t e = e4m3_rn_satfinite(x);
            const float alpha = sT * e4m3_value(e);
            const float2 a2 = make_float2(alpha, alpha);
            float2 E2 = make_float2(0.0f, 0.0f);
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const float2 ev = __ffma2_rn(a2, q2[t], naw2[t]);
                E2 = __ffma2_rn(__fmul2_rn(h2[t], ev), ev, E2);
            }
            const float err = k < p.n_clip ? E2.x + E2.y : INFINITY;
            // candidates with equal moments and scale have, to within rounding
            // below the tie margin, equal codes and errors: a key of the three
            Ek[k] = err;
            Kk[k] = (__float_as_uint(s2) * 0x9E3779B1u + __float_as_uint(s3)) ^ e;
            if (err < Eb) {  // strict: ties keep the lower index
                Eb = err;
                kb = k;
                e_sel = e;
                alpha_sel = alpha;
            }
        }
        // contenders: within the direct sums' fp32 error bound of the best
        uint32_t keyb = Kk[0];
#pragma unroll
        for (int k = 1; k < KM; ++k)
            if (k == kb) keyb = Kk[k];
        unsigned set = 0;
#pragma unroll
        for (int k = 0; k < KM; ++k)
            if (k != kb && Ek[k] - Eb <= ulp * (Ek[k] + Eb) && Kk[k] != keyb) set |= 1u << k;

        if (set != 0 && valid && !zero) {
            // exact comparison: sum h (alpha q - |w|)^2 with alpha*q - |w| as an
            // exact pair (TwoProd, TwoSum) and the squares and sum in float pairs
            if (p.stats) atomicAdd(&p.stats[0], 1u);
            set |= 1u << kb;
            float best_h = INFINITY, best_l = 0.0f;
            int bk = -1;
            while (set) {
                const int k = __ffs(set) - 1;
                set &= set - 1;
                const float P = P1 * p.invf[k];
                const float2 P2 = make_float2(P, P);
                float2 S2 = make_float2(0.0f, 0.0f), S3 = S2;
                float2 q2[8];
#pragma unroll
                for (int t = 0; t < 8; ++t) {
                    float2 y = __fmul2_rn(aw2[t], P2);
                    q2[t] = e2m1_2(y);
                    const float2 hq = __fmul2_rn(h2[t], q2[t]);
                    S2 = __ffma2_rn(hq, q2[t], S2);
                    S3 = __ffma2_rn(hq, aw2[t], S3);
                }
                const float s2 = S2.x + S2.y, s3 = S3.x + S3.y;
                const float x = s2 > 0.0f ? __fdividef(s3, s2) * inv_sT
                                          : amax_b * p.f[k] * (1.0f / 6.0f) * inv_sT;
                const uint32_t e = e4m3_rn_satfinite(x);
                const float alpha = sT * e4m3_value(e);
                float eh = 0.0f, el = 0.0f;
#pragma unroll
                for (int t = 0; t < 8; ++t) {
#pragma unroll
                    for (int c2 = 0; c2 < 2; ++c2) {
                        const float q = c2 ? q2[t].y : q2[t].x;
                        const float aw = c2 ? aw2[t].y : aw2[t].x;
                        const float h = c2 ? h2[t].y : h2[t].x;
                        float ph, pl, dh, dl, sh, sl;
                        two_prod_f(alpha, q, ph, pl);
                        two_sum_f(ph, -aw, dh, dl);
                        dl = __fadd_rn(dl, pl);  // alpha q - |w| = dh + dl
                        two_prod_f(dh, dh, sh, sl);
                        sl = fmaf(2.0f * dh, dl, sl);
                        two_prod_f(h, sh, ph, pl);
                        pl = fmaf(h, sl, pl);
                        float t1, t2;
                        two_sum_f(eh, ph, t1, t2);
                        eh = t1;
                        el = __fadd_rn(el, __fadd_rn(t2, pl));
                    }
                }
                if (bk < 0 || eh < best_h || (eh == best_h && el < best_l)) {
                    best_h = eh;
                    best_l = el;
                    bk = k;
                    alpha_sel = alpha;
                    e_sel = e;
                }
            }
            kb = bk;
        }
        if (!valid) continue;
        if (zero) {
            kb = 0;
            e_sel = 0;
            alpha_sel = 0.0f;
        }

        // ---- outputs of the kept candidate
        const float Pb = P1 * p.invf[kb];
        const float2 Pb2 = make_float2(Pb, Pb);
        const float2 as2 = make_float2(alpha_sel, alpha_sel);
        uint64_t pk = 0;  // packed codes: element j's nibble at bit 4j
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int cidx = (i + rot) & 3;
            float2 rv[2];
            uint32_t cw = 0;
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int t = 2 * i + hh;
                float2 y = __fmul2_rn(aw2[t], Pb2);
                const float2 q = e2m1_2(y);
                // the code carries the sign of w (magnitude 0 is stored as +0)
                const float2 qs = make_float2(q.x > 0.0f ? copysignf(q.x, w2[t].x) : 0.0f,
                                              q.y > 0.0f ? copysignf(q.y, w2[t].y) : 0.0f);
                rv[hh] = __fmul2_rn(as2, qs);
                if (T.codes) cw |= (e2m1_nibble(qs.x) | (e2m1_nibble(qs.y) << 8)) << (16 * hh);
            }
            const int64_t e = ebase + cidx * 4;
            if (p.r_bf16) {
                stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + e),
                       make_uint2(pack_bf16x2(rv[0].x, rv[0].y), pack_bf16x2(rv[1].x, rv[1].y)));
            } else {
                stg_cs(reinterpret_cast<float4*>(static_cast<float*>(T.r) + e),
                       make_float4(rv[0].x, rv[0].y, rv[1].x, rv[1].y));
            }
            if (T.codes) {
                if (!p.codes_packed) {
                    stg_cs(reinterpret_cast<uint32_t*>(T.codes + e), cw);
                } else {
                    // bytes q0 q1 q2 q3 -> nibbles q0 | q1 << 4 | q2 << 8 | q3 << 12
                    const uint32_t nib = (cw & 0xFu) | ((cw >> 4) & 0xF0u) | ((cw >> 8) & 0xF00u) |
                                         ((cw >> 12) & 0xF000u);
                    pk |= (uint64_t)nib << (16 * cidx);
                }
            }
        }
        if (T.codes && p.codes_packed) stg_cs(reinterpret_cast<uint2*>(T.codes + blk * 8),
                                             make_uint2((uint32_t)pk, (uint32_t)(pk >> 32)));
        T.scale[blk] = (uint8_t)e_sel;
        if (T.idx) T.idx[blk] = (uint8_t)kb;
    }
}

// Tensor absmax of a batch: blockIdx.y picks the tensor; max |w| over its n
// elements is accumulated into *slot (which must start at 0) as the bit
// pattern of a non-negative float (such patterns order like uints).
// Tensors whose amax is supplied are skipped.
template <int MAXT>
__global__ void __launch_bounds__(256) k_amax(const __grid_constant__ AmaxBatch<MAXT> B)
{
    const AmaxItem& it = B.t[blockIdx.y];
    if (it.amax_in || it.n == 0) return;
    const float* w = it.w;
    const int64_t n = it.n;
    float m = 0.0f;
    const int64_t n4 = n / 4;
    const float4* w4 = reinterpret_cast<const float4*>(w);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float4 x = __ldcs(w4 + i);
        m = fmaxf(m, fmaxf(fmaxf(fabsf(x.x), fabsf(x.y)), fmaxf(fabsf(x.z), fabsf(x.w))));
    }
    for (int64_t i = n4 * 4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        m = fmaxf(m, fabsf(w[i]));
#pragma unroll
    for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    __shared__ float red[32];
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x < 32) {
        m = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0f;
#pragma unroll
        for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
        if (threadIdx.x == 0 && m > 0.0f)
            atomicMax(reinterpret_cast<unsigned int*>(it.slot), __float_as_uint(m));
    }
}

// Zero the absmax slots of a batch before k_amax: those of the tensors whose
// amax is computed, or every slot (all != 0), in one launch.
template <int MAXT>
__global__ void k_amax_init(const __grid_constant__ AmaxBatch<MAXT> B, int all)
{
    for (int i = threadIdx.x; i < B.n_t; i += blockDim.x)
        if (all || !B.t[i].amax_in) *B.t[i].slot = 0.0f;
}

// *slot := s_T of the supplied amax, or of the amax the slot holds.
template <int MAXT>
__global__ void k_amax_to_scale(const __grid_constant__ AmaxBatch<MAXT> B)
{
    for (int i = threadIdx.x; i < B.n_t; i += blockDim.x) {
        const AmaxItem& it = B.t[i];
        const float amax = it.amax_in ? *it.amax_in : *it.slot;
        *it.slot = tensor_scale_of(amax);
    }
}

}  // namespace quasar
