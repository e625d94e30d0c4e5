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
// access of the warp is bank-conflict free.
//
// Exactness: the candidate error is evaluated from moments,
// S_ww - 2*alpha*S3 + alpha^2*S2; candidates within an error bound of the
// best are re-evaluated directly as sum h (alpha*q - |w|)^2, where
// fma(alpha, q, -|w|) rounds once.
#pragma once

#include "device_common.cuh"
#include "params.h"

namespace quasar {

__device__ __forceinline__ float tensor_scale_of(float amax)
{
    return amax > 0.0f ? __fdiv_rn(amax, 2688.0f) : 1.0f;
}

// E2M1 magnitude nearest to y in [0, 6] (ties to even): rounds y on the grid
// spacing of its binade (0.5 below 2, 1 in [2,4), 2 in [4,6]) with a magic
// constant whose ulp is that spacing.
__device__ __forceinline__ float e2m1_mag(float y)
{
    const uint32_t eb = max(__float_as_uint(y), 0x3F800000u) & 0x7F800000u;
    const float M = __uint_as_float(eb + 0x0B400000u);
    return __fsub_rn(__fadd_rn(y, M), M);
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
    const uint32_t e = (bits >> 3) & 0xFu, m = bits & 7u;
    if (e == 0) return (float)m * 0.001953125f;  // m * 2^-9
    return __uint_as_float(((e + 120u) << 23) | (m << 20));
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

template <int NCH>
__global__ void __launch_bounds__(256) k_recon_nvfp4(const Nvfp4Params p)
{
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

    const int64_t n_units = (p.n_blocks + kBlocksPerUnit - 1) / kBlocksPerUnit;
    const int64_t first = (int64_t)blockIdx.x * nwarps + warp;
    const int64_t stride = (int64_t)gridDim.x * nwarps;

    const float amax_t = *p.amax;
    const float sT = tensor_scale_of(amax_t);
    const float inv_sT = 1.0f / sT;
    if (p.write_scale && blockIdx.x == 0 && threadIdx.x == 0) *p.tensor_scale = sT;

    if (lane == 0) {
        for (int s = 0; s <= S; ++s) mbar_init(&bars[s], 1);
        mbar_init_fence();
    }
    __syncwarp();

    auto issue = [&](int64_t u, int s) {
        const int64_t b0 = u * kBlocksPerUnit;
        const int64_t nb = min((int64_t)kBlocksPerUnit, p.n_blocks - b0);
        const uint32_t elems = (uint32_t)(nb * 16);
        unsigned char* st = ring + (size_t)s * p.stage_bytes;
        mbar_arrive_expect_tx(&bars[s], elems * (8u + (uint32_t)gbytes));
        bulk_g2s(st, p.w + b0 * 16, elems * 4u, &bars[s]);
        bulk_g2s(st + kVOff, p.v + b0 * 16, elems * 4u, &bars[s]);
        if (gbytes)
            bulk_g2s(st + kGOff, static_cast<const unsigned char*>(p.g) + b0 * 16 * gbytes,
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
        if (!mbar_wait_bounded(&bars[S], 0, p.force_timeout_ns)) {
            fail(0);
            return;
        }
    }

    const int rot = (lane >> 1) & 3;
    const float ulp = 5.9604645e-8f * p.tie_kappa;
    int s_cur = 0;
    uint32_t parity = 0;

    for (int64_t it = 0;; ++it) {
        const int64_t u = first + it * stride;
        if (u >= n_units) break;
        if (!mbar_wait_bounded(&bars[s_cur], parity, p.timeout_ns)) {
            fail(it);
            return;
        }
        const unsigned char* st = ring + (size_t)s_cur * p.stage_bytes;

        // element 4*cidx[i] + jj of this lane's block is held at slot 4*i + jj
        float w[16], h[16];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int cidx = (i + rot) & 3;
            const int e = lane * 16 + cidx * 4;
            const float4 w4 = lds128(st + e * 4);
            const float4 v4 = lds128(st + kVOff + e * 4);
            w[4 * i + 0] = w4.x; w[4 * i + 1] = w4.y; w[4 * i + 2] = w4.z; w[4 * i + 3] = w4.w;
            h[4 * i + 0] = v4.x; h[4 * i + 1] = v4.y; h[4 * i + 2] = v4.z; h[4 * i + 3] = v4.w;
            if (p.g_kind) {
                float g0, g1, g2, g3;
                if (p.g_kind == 2) {
                    const uint2 gb = lds64(st + kGOff + e * 2);
                    g0 = bf16lo(gb.x); g1 = bf16hi(gb.x); g2 = bf16lo(gb.y); g3 = bf16hi(gb.y);
                } else {
                    const float4 g4 = lds128(st + kGOff + e * 4);
                    g0 = g4.x; g1 = g4.y; g2 = g4.z; g3 = g4.w;
                }
                h[4 * i + 0] = fmaf(p.beta2, h[4 * i + 0], __fmul_rn(p.c1, __fmul_rn(g0, g0)));
                h[4 * i + 1] = fmaf(p.beta2, h[4 * i + 1], __fmul_rn(p.c1, __fmul_rn(g1, g1)));
                h[4 * i + 2] = fmaf(p.beta2, h[4 * i + 2], __fmul_rn(p.c1, __fmul_rn(g2, g2)));
                h[4 * i + 3] = fmaf(p.beta2, h[4 * i + 3], __fmul_rn(p.c1, __fmul_rn(g3, g3)));
            }
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

        const int64_t blk = u * kBlocksPerUnit + lane;
        const bool valid = blk < p.n_blocks;
        const int64_t ebase = blk * 16;

        if (valid && p.g_kind) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int cidx = (i + rot) & 3;
                stg_cs(reinterpret_cast<float4*>(p.v + ebase + cidx * 4),
                       make_float4(h[4 * i], h[4 * i + 1], h[4 * i + 2], h[4 * i + 3]));
            }
        }

        float amax_b = 0.0f, ss = 0.0f;
        float aw[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            aw[j] = fabsf(w[j]);
            amax_b = fmaxf(amax_b, aw[j]);
            ss += h[j];
        }
        if (ss == 0.0f) {
#pragma unroll
            for (int j = 0; j < 16; ++j) h[j] = 1.0f;
        }
        float sww = 0.0f;
#pragma unroll
        for (int j = 0; j < 16; ++j) sww = fmaf(h[j] * aw[j], aw[j], sww);

        const bool zero = !(amax_b > 0.0f);
        const float P1 = zero ? 0.0f : 6.0f / amax_b;  // 1/sigma at f = 1

        // Candidate k: moments, fitted E4M3 scale and error from moments.
        auto candidate = [&](int k, float& alpha, uint32_t& e, float& s2, float& s3) {
            const float P = P1 * p.invf[k];
            s2 = 0.0f;
            s3 = 0.0f;
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float q = e2m1_mag(fminf(aw[j] * P, 6.0f));
                const float hq = __fmul_rn(h[j], q);
                s2 = fmaf(hq, q, s2);
                s3 = fmaf(hq, aw[j], s3);
            }
            const float x = s2 > 0.0f ? __fdividef(s3, s2) * inv_sT
                                      : amax_b * p.f[k] * (1.0f / 6.0f) * inv_sT;
            e = e4m3_rn_satfinite(x);
            alpha = sT * e4m3_value(e);
        };

        // Per candidate: the error from moments and its fp32 error bound.
        float Sk[KM], dSk[KM];
        float Sb = INFINITY, dSb = 0.0f, alpha_sel = 0.0f;
        uint32_t e_sel = 0;
        int kb = 0;
#pragma unroll
        for (int k = 0; k < KM; ++k) {
            float alpha, s2, s3;
            uint32_t e;
            candidate(k, alpha, e, s2, s3);
            const float Sv = k < p.n_clip ? fmaf(alpha, fmaf(alpha, s2, -2.0f * s3), sww) : INFINITY;
            Sk[k] = Sv;
            dSk[k] = ulp * (sww + 2.0f * alpha * s3 + alpha * alpha * s2);
            if (Sv < Sb) {  // strict: ties keep the lower index
                Sb = Sv;
                dSb = dSk[k];
                alpha_sel = alpha;
                e_sel = e;
                kb = k;
            }
        }
        unsigned set = 0;
#pragma unroll
        for (int k = 0; k < KM; ++k)
            if (k != kb && Sk[k] - Sb <= dSb + dSk[k]) set |= 1u << k;

        if (set != 0 && valid && !zero) {
            if (p.stats) atomicAdd(&p.stats[0], 1u);
            set |= 1u << kb;
            float best = INFINITY;
            int bk = -1;
            while (set) {
                const int k = __ffs(set) - 1;
                set &= set - 1;
                float alpha, s2, s3;
                uint32_t e;
                candidate(k, alpha, e, s2, s3);
                const float P = P1 * p.invf[k];
                float t[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const float q = e2m1_mag(fminf(aw[j] * P, 6.0f));
                    const float ej = fmaf(alpha, q, -aw[j]);
                    t[j] = h[j] * (ej * ej);
                }
#pragma unroll
                for (int s = 1; s < 16; s <<= 1)
#pragma unroll
                    for (int j = 0; j + s < 16; j += 2 * s) t[j] += t[j + s];
                if (bk < 0 || t[0] < best) {
                    best = t[0];
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

        const float Pb = P1 * p.invf[kb];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int cidx = (i + rot) & 3;
            float rv[4];
            uint32_t cw = 0;
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
                const int j = 4 * i + jj;
                const float q = zero ? 0.0f : e2m1_mag(fminf(aw[j] * Pb, 6.0f));
                const float qs = q > 0.0f ? copysignf(q, w[j]) : 0.0f;
                rv[jj] = alpha_sel * qs;
                cw |= e2m1_nibble(qs) << (8 * jj);
            }
            const int64_t e = ebase + cidx * 4;
            if (p.r_bf16) {
                stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.r) + e),
                       make_uint2(pack_bf16x2(rv[0], rv[1]), pack_bf16x2(rv[2], rv[3])));
            } else {
                stg_cs(reinterpret_cast<float4*>(static_cast<float*>(p.r) + e),
                       make_float4(rv[0], rv[1], rv[2], rv[3]));
            }
            if (p.codes) stg_cs(reinterpret_cast<uint32_t*>(p.codes + e), cw);
        }
        p.scale[blk] = (uint8_t)e_sel;
        if (p.idx) p.idx[blk] = (uint8_t)kb;
    }
}

// max |w| over n elements, accumulated into *out (which must start at 0) as
// the bit pattern of a non-negative float (such patterns order like uints).
__global__ void __launch_bounds__(256) k_amax(const float* __restrict__ w, int64_t n, unsigned int* out)
{
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
        if (threadIdx.x == 0) atomicMax(out, __float_as_uint(m));
    }
}

// tensor_scale[0] := s_T of the amax it holds.
__global__ void k_amax_to_scale(float* tensor_scale)
{
    *tensor_scale = tensor_scale_of(*tensor_scale);
}

}  // namespace quasar
