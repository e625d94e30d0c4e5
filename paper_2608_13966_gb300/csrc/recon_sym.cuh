// QUASAR with symmetric integer codes: the offset-free closed form of
// Sec. 4.1.2.  For each group and clip factor f: step s_f = f amax / Q
// (amax = max |w| of the group, Q = 2^(bits-1) - 1), codes
// q = clamp(round_half_even(w / s_f), -Q, Q), fit s* = sum h q w / sum h q^2,
// and the candidate whose error sum h (s* q - w)^2 = sum h w^2 - S3^2 / S2
// is lowest is kept (S2 = sum h q^2, S3 = sum h q w).
//
// Layout as the asymmetric kernel: a warp takes 4 groups a unit, 8 lanes a
// group, from a per-warp TMA ring.  Both sums are over non-negative terms
// (h |q|^2 and h |q| |w|), so each carries a small relative error and
// S3^2 / S2 a bound of a few ulps: candidates within the bound of the best
// are compared exactly (float-float direct errors, whole warp), and the
// kept fit needs no refinement.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

#include "device_common.cuh"
#include "params.h"

namespace quasar {
namespace sym {

constexpr float kMagic = 8388608.0f;  // 2^23: adding it rounds to an integer (nearest even)
constexpr float kU = 5.9604645e-8f;

__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e)
{
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

__device__ __forceinline__ void two_prod(float a, float b, float& p, float& e)
{
    p = __fmul_rn(a, b);
    e = fmaf(a, b, -p);
}

__device__ __forceinline__ void ff_acc(float& hi, float& lo, float xh, float xl)
{
    float s, e;
    two_sum(hi, xh, s, e);
    hi = s;
    lo = __fadd_rn(lo, __fadd_rn(e, xl));
}

__device__ __forceinline__ void ff_norm(float& hi, float& lo)
{
    const float s = __fadd_rn(hi, lo);
    lo = __fsub_rn(lo, __fsub_rn(s, hi));
    hi = s;
}

__device__ __forceinline__ void ff_reduce32(float& hi, float& lo)
{
    ff_norm(hi, lo);
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const float oh = __shfl_xor_sync(0xffffffffu, hi, o);
        const float ol = __shfl_xor_sync(0xffffffffu, lo, o);
        ff_acc(hi, lo, oh, ol);
        ff_norm(hi, lo);
    }
    // the float-pair sum is not symmetric in its operands, so lanes can end
    // one rounding apart: every lane takes lane 0's pair, so that decisions
    // taken from it are the same across the warp
    hi = __shfl_sync(0xffffffffu, hi, 0);
    lo = __shfl_sync(0xffffffffu, lo, 0);
}

// |q| = min(round_half_even(|w| P), Q) as a float
__device__ __forceinline__ float code_n(float aw, float P, float Q)
{
    return __fsub_rn(fminf(__fmaf_rn(aw, P, kMagic), kMagic + Q), kMagic);
}

}  // namespace sym

template <int EPL, int MAXT>
__global__ void __launch_bounds__(256, 2) k_recon_sym(const __grid_constant__ IntLaunch<MAXT> Lp)
{
    using namespace sym;
    const IntParams& p = Lp.p;
    constexpr int G = EPL * kLanesPerGroup;
    constexpr int UNIT = kGroupsPerUnit * G;
    constexpr int NCHK = EPL / 4;
    extern __shared__ __align__(128) unsigned char smem[];

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int gs = lane >> 3;
    const int sl = lane & 7;
    const int S = p.stages;
    unsigned char* ring = smem + (size_t)warp * S * p.stage_bytes;
    float* red = reinterpret_cast<float*>(smem + (size_t)nwarps * S * p.stage_bytes +
                                          (size_t)warp * kIntScratchBytes);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)nwarps * S * p.stage_bytes +
                                                 (size_t)nwarps * kIntScratchBytes) +
                     warp * (S + 1);

    const int gbytes = p.g_kind == 2 ? 2 : (p.g_kind == 1 ? 4 : 0);
    constexpr uint32_t kVOff = UNIT * 4;
    constexpr uint32_t kGOff = UNIT * 8;
    const int Qi = (p.qmax - 1) >> 1;  // qmax = 2Q + 1 levels
    const float Q = (float)Qi;
    const int NCH = (p.n_clip + 7) >> 3;

    const int64_t n_units = Lp.n_units;
    auto tensor_of = [&](int64_t u, int& ti) {
        while (ti + 1 < Lp.n_t && u >= Lp.t[ti + 1].unit0) ++ti;
    };
    int ti = 0;
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
        const IntTensor& T = Lp.t[tj];
        const int64_t g0 = (u - T.unit0) * kGroupsPerUnit;
        const int64_t ng = min((int64_t)kGroupsPerUnit, T.n_groups - g0);
        const uint32_t elems = (uint32_t)(ng * G);
        unsigned char* st = ring + (size_t)s * p.stage_bytes;
        mbar_arrive_expect_tx(&bars[s], elems * (8u + (uint32_t)gbytes));
        bulk_g2s(st, T.w + g0 * G, elems * 4u, &bars[s]);
        bulk_g2s(st + kVOff, T.v + g0 * G, elems * 4u, &bars[s]);
        if (gbytes)
            bulk_g2s(st + kGOff, static_cast<const unsigned char*>(T.g) + g0 * G * gbytes,
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

    const float2 beta22 = make_float2(p.beta2, p.beta2);
    const float2 c12 = make_float2(p.c1, p.c1);
    const float2 M2 = make_float2(kMagic, kMagic);
    const float2 cap2 = make_float2(kMagic + Q, kMagic + Q);
    const float2 nM2 = make_float2(-kMagic, -kMagic);
    const float gam = kU * p.tie_kappa;
    int s_cur = 0;
    uint32_t parity = 0;

    for (int64_t it = 0;; ++it) {
        const int64_t u = first + it * stride;
        if (u >= n_units) break;
        if (!warp_wait_bounded(&bars[s_cur], parity, p.timeout_ns)) {
            fail(it);
            return;
        }
        unsigned char* st = ring + (size_t)s_cur * p.stage_bytes;
        float* ws = reinterpret_cast<float*>(st);
        float* hs = reinterpret_cast<float*>(st + kVOff);
        const unsigned char* gsm = st + kGOff;
        tensor_of(u, ti);
        const IntTensor& T = Lp.t[ti];
        const int64_t grp = (u - T.unit0) * kGroupsPerUnit + gs;
        const bool valid = grp < T.n_groups;
        const int64_t gbase = grp * (int64_t)G;

        // ---- pass A: EMA (v' out), the fit's saliency h into the tile,
        // amax and the saliency mass of the group
        float amax = 0.0f, ss = 0.0f;
#pragma unroll
        for (int i = 0; i < NCHK; ++i) {
            const int e = gs * G + i * 32 + sl * 4;
            const float4 w4 = lds128(ws + e);
            float4 h4 = lds128(hs + e);
            if (p.g_kind) {
                float2 gA, gB;
                if (p.g_kind == 2) {
                    const uint2 gb = lds64(gsm + e * 2);
                    gA = make_float2(bf16lo(gb.x), bf16hi(gb.x));
                    gB = make_float2(bf16lo(gb.y), bf16hi(gb.y));
                } else {
                    const float4 g4 = lds128(gsm + e * 4);
                    gA = make_float2(g4.x, g4.y);
                    gB = make_float2(g4.z, g4.w);
                }
                const float2 hA = __ffma2_rn(make_float2(h4.x, h4.y), beta22, __fmul2_rn(c12, __fmul2_rn(gA, gA)));
                const float2 hB = __ffma2_rn(make_float2(h4.z, h4.w), beta22, __fmul2_rn(c12, __fmul2_rn(gB, gB)));
                h4 = make_float4(hA.x, hA.y, hB.x, hB.y);
                if (valid) stg_cs(reinterpret_cast<float4*>(T.v + gbase + sl * 4 + i * 32), h4);
            }
            if (p.h_mode != kSalEma)
                h4 = p.h_mode == kSalEmaSquared
                         ? make_float4(h4.x * h4.x, h4.y * h4.y, h4.z * h4.z, h4.w * h4.w)
                         : make_float4(1.0f, 1.0f, 1.0f, 1.0f);
            *reinterpret_cast<float4*>(hs + e) = h4;
            amax = fmaxf(amax, fmaxf(fmaxf(fabsf(w4.x), fabsf(w4.y)), fmaxf(fabsf(w4.z), fabsf(w4.w))));
            ss += (h4.x + h4.y) + (h4.z + h4.w);
        }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
            ss += __shfl_xor_sync(0xffffffffu, ss, o);
        }
        if (__any_sync(0xffffffffu, ss == 0.0f)) {  // all saliencies zero: h = 1
            if (ss == 0.0f)
#pragma unroll
                for (int i = 0; i < NCHK; ++i)
                    *reinterpret_cast<float4*>(hs + gs * G + i * 32 + sl * 4) = make_float4(1.0f, 1.0f, 1.0f, 1.0f);
        }
        // a sum of saliencies near the bottom of the fp32 range: h scaled by
        // a power of two
        const bool h_tiny = ss > 0.0f && ss < kTinySaliency;
        if (__any_sync(0xffffffffu, h_tiny)) {
            if (h_tiny) {
                float s1, s2;
                tiny_scale(ss, s1, s2);
#pragma unroll 1
                for (int i = 0; i < NCHK; ++i) {
                    float4* hp = reinterpret_cast<float4*>(hs + gs * G + i * 32 + sl * 4);
                    const float4 h4 = *hp;
                    *hp = make_float4(h4.x * s1 * s2, h4.y * s1 * s2, h4.z * s1 * s2, h4.w * s1 * s2);
                }
            }
        }
        __syncwarp();
        const bool flat = !(amax > 0.0f);
        const float R = flat ? 0.0f : __fdividef(Q, amax);  // P = R / f

        // ---- candidates, 8 at a time: S2, S3 per candidate, lane sl owns k = 8 ch + sl
        float Ek[4], dEk[4], S2k[4], S3k[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) Ek[c] = dEk[c] = S2k[c] = S3k[c] = 0.0f;
#pragma unroll 1
        for (int ch = 0; ch < NCH; ++ch) {
            float2 P2[8];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const float P = R * p.invf[ch * 8 + kk];
                P2[kk] = make_float2(P, P);
            }
            float2 A2[8], A3[8];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) A2[kk] = A3[kk] = make_float2(0.0f, 0.0f);
#pragma unroll 1
            for (int i = 0; i < NCHK; ++i) {
                const int e = gs * G + i * 32 + sl * 4;
                const float4 w4 = lds128(ws + e);
                const float4 h4 = lds128(hs + e);
#pragma unroll
                for (int pr = 0; pr < 2; ++pr) {
                    const float2 aw = pr ? make_float2(fabsf(w4.z), fabsf(w4.w)) : make_float2(fabsf(w4.x), fabsf(w4.y));
                    const float2 h = pr ? make_float2(h4.z, h4.w) : make_float2(h4.x, h4.y);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        float2 y = __ffma2_rn(aw, P2[kk], M2);
                        y.x = fminf(y.x, cap2.x);
                        y.y = fminf(y.y, cap2.y);
                        const float2 n = __fadd2_rn(y, nM2);
                        const float2 t = __fmul2_rn(h, n);
                        A2[kk] = __ffma2_rn(t, n, A2[kk]);
                        A3[kk] = __ffma2_rn(t, aw, A3[kk]);
                    }
                }
            }
            // transpose: lane L writes its 8 candidates' (S2, S3) in row L
            // (8-byte columns XOR-swizzled by the row), lane (gs, sl) sums
            // column sl over its group's 8 rows
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
                *reinterpret_cast<float2*>(red + lane * 16 + ((kk ^ sl) << 1)) =
                    make_float2(A2[kk].x + A2[kk].y, A3[kk].x + A3[kk].y);
            __syncwarp();
            float2 x[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) x[j] = *reinterpret_cast<const float2*>(red + (gs * 8 + j) * 16 + ((sl ^ j) << 1));
#pragma unroll
            for (int s2 = 1; s2 < 8; s2 <<= 1)
#pragma unroll
                for (int j = 0; j + s2 < 8; j += 2 * s2) {
                    x[j].x += x[j + s2].x;
                    x[j].y += x[j + s2].y;
                }
            __syncwarp();
            const float S2 = x[0].x, S3 = x[0].y;
            const bool real = ch * 8 + sl < p.n_clip;
            const float E = S2 > 0.0f ? __fdividef(S3 * S3, S2) : 0.0f;
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (c == ch) {
                    Ek[c] = real ? E : -INFINITY;
                    dEk[c] = (3.0f * gam + 4.0f * kU) * E;
                    S2k[c] = S2;
                    S3k[c] = S3;
                }
        }

        // ---- argmax of E (ties: lowest index), contenders
        float Eb = -INFINITY, dEb = 0.0f;
        int kb = 0x7fff;
#pragma unroll
        for (int c = 0; c < 4; ++c)
            if (c < NCH && Ek[c] > Eb) {
                Eb = Ek[c];
                dEb = dEk[c];
                kb = c * 8 + sl;
            }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            const float Eo = __shfl_xor_sync(0xffffffffu, Eb, o);
            const float dEo = __shfl_xor_sync(0xffffffffu, dEb, o);
            const int ko = __shfl_xor_sync(0xffffffffu, kb, o);
            if (Eo > Eb || (Eo == Eb && ko < kb)) {
                Eb = Eo;
                dEb = dEo;
                kb = ko;
            }
        }
        if (kb > 0x7ff) kb = 0;
        float S2b = 0.0f, S3b = 0.0f;
        {
            const int owner = (gs * 8) | (kb & 7);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const float a2 = __shfl_sync(0xffffffffu, S2k[c], owner);
                const float a3 = __shfl_sync(0xffffffffu, S3k[c], owner);
                if ((kb >> 3) == c) {
                    S2b = a2;
                    S3b = a3;
                }
            }
        }
        unsigned my_set = 0;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int k = c * 8 + sl;
            // equal sums bit for bit: a tie, settled by the index as by the
            // exact errors (codes differing only where h = 0 give equal errors)
            const bool twin = S2k[c] == S2b && S3k[c] == S3b;
            if (c < NCH && k != kb && Ek[c] > -INFINITY && !twin && Eb - Ek[c] <= dEb + dEk[c])
                my_set |= 1u << c;
        }
        unsigned set = 0;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const unsigned bal = __ballot_sync(0xffffffffu, (my_set >> c) & 1u);
            set |= ((bal >> (gs * 8)) & 0xFFu) << (c * 8);
        }
        if (set) set |= 1u << kb;

        // the fit; with sum h q^2 = 0 it is the candidate's step s_f
        float a_sel = S2b > 0.0f ? S3b / S2b : 0.0f;
        if (!flat && !(S2b > 0.0f)) a_sel = p.f[kb] * amax / Q;

        // ---- exact comparison: float-float direct errors, whole warp per group
        unsigned todo = __ballot_sync(0xffffffffu, valid && !flat && set != 0 && sl == 0);
        while (todo) {
            const int g = (__ffs(todo) - 1) >> 3;
            todo &= todo - 1;
            const int src = g * 8;
            const float gR = __shfl_sync(0xffffffffu, R, src);
            const float gamax = __shfl_sync(0xffffffffu, amax, src);
            unsigned gset = __shfl_sync(0xffffffffu, set, src);
            if (p.stats && lane == 0) atomicAdd(&p.stats[0], 1u);
            const float* gws = ws + g * G;
            const float* ghs = hs + g * G;
            float best_h = 0.0f, best_l = 0.0f, best_a = 0.0f;
            int best_k = -1;
            while (gset) {
                const int k = __ffs(gset) - 1;
                gset &= gset - 1;
                const float P = gR * p.invf[k];
                float s2h = 0.0f, s2l = 0.0f, s3h = 0.0f, s3l = 0.0f;
#pragma unroll
                for (int m = 0; m < G / 32; ++m) {
                    const int e = lane + 32 * m;
                    const float w = gws[e], h = ghs[e];
                    const float n = code_n(fabsf(w), P, Q);
                    float ph, pl;
                    two_prod(h, n * n, ph, pl);  // n^2 is exact (|n| <= 127)
                    ff_acc(s2h, s2l, ph, pl);
                    two_prod(h * n, fabsf(w), ph, pl);
                    pl = fmaf(fmaf(h, n, -h * n), fabsf(w), pl);
                    ff_acc(s3h, s3l, ph, pl);
                }
                ff_reduce32(s2h, s2l);
                ff_reduce32(s3h, s3l);
                float ah, al;
                if (s2h > 0.0f) {
                    ah = s3h / s2h;
                    float qh, ql;
                    two_prod(ah, s2h, qh, ql);
                    const float rr = __fsub_rn(__fsub_rn(__fadd_rn(__fsub_rn(s3h, qh), s3l), ql), ah * s2l);
                    al = rr / s2h;
                } else {
                    ah = p.f[k] * gamax / Q;
                    al = 0.0f;
                }
                float eh = 0.0f, el = 0.0f;
#pragma unroll
                for (int m = 0; m < G / 32; ++m) {
                    const int e = lane + 32 * m;
                    const float w = gws[e], h = ghs[e];
                    const float q = copysignf(code_n(fabsf(w), P, Q), w);
                    // d = a q - w in float-float
                    float dh, dl, ph, pl;
                    two_prod(ah, q, ph, pl);
                    pl = fmaf(al, q, pl);
                    two_sum(ph, -w, dh, dl);
                    dl = __fadd_rn(dl, pl);
                    ff_norm(dh, dl);
                    float sh, sl2;
                    two_prod(dh, dh, sh, sl2);
                    sl2 = fmaf(2.0f * dh, dl, sl2);
                    float th, tl;
                    two_prod(h, sh, th, tl);
                    tl = fmaf(h, sl2, tl);
                    ff_acc(eh, el, th, tl);
                }
                ff_reduce32(eh, el);
                if (best_k < 0 || eh < best_h || (eh == best_h && el < best_l)) {
                    best_h = eh;
                    best_l = el;
                    best_k = k;
                    best_a = ah;
                }
            }
            if (gs == g) {
                kb = best_k;
                a_sel = best_a;
            }
        }

        // ---- outputs: r = a q, codes q + Q, a, b = -a Q, index
        const float Pk = R * p.invf[kb];
        if (valid) {
            const float2 a2 = make_float2(a_sel, a_sel);
#pragma unroll
            for (int i = 0; i < NCHK; ++i) {
                const float4 w4 = lds128(ws + gs * G + i * 32 + sl * 4);
                const float wv[4] = {w4.x, w4.y, w4.z, w4.w};
                float qv[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) qv[j] = flat ? 0.0f : copysignf(code_n(fabsf(wv[j]), Pk, Q), wv[j]);
                const float2 r0 = __fmul2_rn(a2, make_float2(qv[0], qv[1]));
                const float2 r1 = __fmul2_rn(a2, make_float2(qv[2], qv[3]));
                const int64_t eo = gbase + i * 32 + sl * 4;
                if (p.r_bf16)
                    stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + eo),
                           make_uint2(pack_bf16x2(r0.x, r0.y), pack_bf16x2(r1.x, r1.y)));
                else
                    stg_cs(reinterpret_cast<float4*>(static_cast<float*>(T.r) + eo), make_float4(r0.x, r0.y, r1.x, r1.y));
                if (T.codes && !p.codes_packed) {
                    uint32_t cw = 0;
#pragma unroll
                    for (int j = 0; j < 4; ++j) cw |= (uint32_t)(int)(qv[j] + Q) << (8 * j);
                    stg_cs(reinterpret_cast<uint32_t*>(T.codes + eo), cw);
                }
            }
        }
        if (T.codes && p.codes_packed) {
            // the packed format of the asymmetric kernel: the group's codes
            // as one little-endian bitstream of `bits` bits a code
            uint32_t* wsc = reinterpret_cast<uint32_t*>(red) + gs * 8;
            const uint32_t o = (uint32_t)sl * 4u * (uint32_t)p.bits;
#pragma unroll 1
            for (int i = 0; i < NCHK; ++i) {
                uint32_t pk = 0;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float wv = ws[gs * G + i * 32 + sl * 4 + j];
                    const float q = flat ? 0.0f : copysignf(code_n(fabsf(wv), Pk, Q), wv);
                    pk |= (uint32_t)(int)(q + Q) << (j * p.bits);
                }
                const uint64_t f = (uint64_t)pk << (o & 31u);
                if (sl < p.bits) wsc[sl] = 0u;
                __syncwarp();
                atomicOr(&wsc[o >> 5], (uint32_t)f);
                if ((uint32_t)(f >> 32)) atomicOr(&wsc[(o >> 5) + 1], (uint32_t)(f >> 32));
                __syncwarp();
                if (valid && sl < p.bits)
                    stg_cs(reinterpret_cast<uint32_t*>(T.codes) + grp * (int64_t)(G / 32) * p.bits + i * p.bits + sl,
                           wsc[sl]);
                __syncwarp();
            }
        }
        if (valid && sl == 0) {
            T.a[grp] = flat ? 0.0f : a_sel;
            T.b[grp] = flat ? 0.0f : -a_sel * Q;
            if (T.idx) T.idx[grp] = flat ? 0 : (uint8_t)kb;
        }

        // release the tile (h was written into it: order those writes before
        // the async-proxy copy that refills it)
        __syncwarp();
        if (lane == 0) {
            const int64_t un = u + (int64_t)S * stride;
            if (un < n_units) {
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                issue(un, s_cur);
            }
        }
        if (++s_cur == S) {
            s_cur = 0;
            parity ^= 1u;
        }
    }
}

}  // namespace quasar
