// QUASAR for the Rubin INT3 lookup-table format (App. B).
//
// A block is 8 consecutive rows x 64 consecutive columns (512 weights).  For
// each clip factor f the block's weights get 3-bit indices on the grid of the
// clipped range [c - f rho, c + f rho] (Eq. 1 with qmax = 7), each of the 8
// table entries is the E4M3 rounding of the saliency-weighted mean of its
// weights (Eq. rubin-fit; an index with no weight takes its grid point), and
// the candidate with the lowest weighted error sum h (C_q - w)^2 is kept.
//
// One warp owns one block: lane L holds block elements 16 L .. 16 L + 15
// (row L / 4, columns 16 (L % 4) ..), read once from a per-warp TMA ring.
// An index is a sign s of d = w - c and a magnitude level m = min(floor(|d|
// P), 3).  Per candidate each lane accumulates, for each sign and threshold
// t = 1, 2, 3, the sums of h and of h |d| over its elements with m >= t
// (packed f32x2; the masks [m >= t] come from saturated adds on the floor,
// so no per-index one-hot work); the 12 sums are transposed through shared
// memory, and with the block's per-sign totals they give every index's H_j =
// sum h and X_j = sum h |d|.  Index j's entry is the E4M3 rounding of its
// weighted mean c + s X_j / H_j, and the error is
//   sum h d^2 - sum_j X_j^2 / H_j + sum_j H_j (C_j - mean_j)^2
// (the within-index scatter plus each entry's offset from its mean).  Both
// the entry's rounding and the error carry an fp32 bound.  Candidates within
// the bound of the best, and undecided roundings, are settled exactly
// (float-float sums over the codes, whole warp), so indices, tables and the
// kept candidate equal the exact computation's.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

#include "device_common.cuh"
#include "params.h"

namespace quasar {
namespace lut {

constexpr float kMagic = 8388608.0f;      // 2^23: its ulp is 1
constexpr float kHalfBelow = 8388607.5f;  // 2^23 - 1/2: y - it = floor + 1/2
constexpr float kU = 5.9604645e-8f;       // fp32 unit roundoff

// Signed E4M3: round to nearest even, saturating at 448; magnitude 0 as +0.
__device__ __forceinline__ uint32_t e4m3_encode(float x)
{
    uint16_t r;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %1;" : "=h"(r) : "f"(x));
    const uint32_t b = r & 0xFFu;
    return (b & 0x7Fu) ? b : 0u;
}

__device__ __forceinline__ float e4m3_decode(uint32_t bits)
{
    const uint32_t m = bits & 0x7Fu;
    // normal: exponent e - 7 + 127, mantissa m << 20; subnormal (e = 0): m * 2^-9
    const float mag = m < 8u ? (float)m * 0.001953125f : __uint_as_float((m << 20) + (120u << 23));
    return (bits & 0x80u) ? -mag : mag;
}

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

// (hi, lo) += (xh, xl), lo left unnormalised
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

__device__ __forceinline__ bool ff_less(float ah, float al, float bh, float bl)
{
    return ah < bh || (ah == bh && al < bl);
}

// Signed centred code z = sign(d) (min(floor(|d| P), 3) + 1/2); index z + 7/2.
__device__ __forceinline__ float code_z(float d, float P)
{
    const float y = fminf(__fmaf_rd(fabsf(d), P, kMagic), kMagic + 3.0f);
    return copysignf(__fsub_rn(y, kHalfBelow), d);
}

// [x + b >= 1] for x + b an integer (x on the 2^23 grid): the sum saturated
// to [0, 1]
__device__ __forceinline__ float add_sat(float x, float b)
{
    float r;
    asm("add.rn.sat.f32 %0, %1, %2;" : "=f"(r) : "f"(x), "f"(b));
    return r;
}

// The E4M3 value nearest the float-float x = xh + xl (ties to the even
// mantissa): the rounding of xh, or one of its neighbours.
__device__ __forceinline__ uint32_t e4m3_round_ff(float xh, float xl)
{
    const uint32_t c0 = e4m3_encode(xh);
    uint32_t best = c0;
    float bh, bl;
    two_sum(e4m3_decode(c0), -xh, bh, bl);
    bl = __fsub_rn(bl, xl);
    ff_norm(bh, bl);
    float bd = fabsf(bh);
    const uint32_t mag = c0 & 0x7Fu;
    const uint32_t sgn = (xh < 0.0f) ? 0x80u : 0u;
#pragma unroll
    for (int t = 0; t < 2; ++t) {
        // the neighbours of c0's magnitude on the side of xh's sign (a
        // magnitude 0 neighbour below 0x01 is 0 itself)
        const int m = (int)mag + (t ? 1 : -1);
        if (m < 0 || m > 0x7E) continue;
        const uint32_t c = (m == 0) ? 0u : (sgn | (uint32_t)m);
        float dh, dl;
        two_sum(e4m3_decode(c), -xh, dh, dl);
        dl = __fsub_rn(dl, xl);
        ff_norm(dh, dl);
        const float d = fabsf(dh);
        // nearer, or as near with an even mantissa (the lower one of a tie)
        if (d < bd || (d == bd && ((c & 1u) == 0u) && ((best & 1u) != 0u))) {
            best = c;
            bd = d;
        }
    }
    return best;
}

}  // namespace lut

template <int MAXT>
__global__ void __launch_bounds__(256, 2) k_recon_lut(const __grid_constant__ LutLaunch<MAXT> Lp)
{
    using namespace lut;
    const LutParams& p = Lp.p;
    extern __shared__ __align__(128) unsigned char smem[];

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int S = p.stages;
    unsigned char* ring = smem + (size_t)warp * S * p.stage_bytes;
    unsigned char* scr = smem + (size_t)nwarps * S * p.stage_bytes + (size_t)warp * kLutScratchBytes;
    float* sums = reinterpret_cast<float*>(scr);  // [24][33]
    uint32_t* cbook = reinterpret_cast<uint32_t*>(scr + kLutSumsBytes);  // [32][2]
    float* cerr = reinterpret_cast<float*>(cbook + 2 * kMaxClip);       // [32]
    float* cbnd = cerr + kMaxClip;                                        // [32]
    uint32_t* camb = reinterpret_cast<uint32_t*>(cbnd + kMaxClip);      // [32]
    float* table = reinterpret_cast<float*>(scr + kLutSumsBytes + kLutCandBytes);  // [8]
    // the block's per-sign sums of h and h |d|, and sum h d^2
    float* bconst = table + 8;  // [7]: also the block's sum of h and its range
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)nwarps * S * p.stage_bytes +
                                                 (size_t)nwarps * kLutScratchBytes) +
                     warp * (S + 1);

    const int gbytes = p.g_kind == 2 ? 2 : (p.g_kind == 1 ? 4 : 0);
    constexpr uint32_t kVOff = kLutBlock * 4;
    constexpr uint32_t kGOff = kLutBlock * 8;
    const int K = p.n_clip;

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

    // the 8 row segments of a block, each of w, v and g: lane 0 announces
    // the bytes, lane r copies row r (every lane calls it)
    auto issue = [&](int64_t u, int s) {
        int tj = ti;
        tensor_of(u, tj);
        const LutTensor& T = Lp.t[tj];
        // block row and column (a tensor holds fewer than 2^32 blocks)
        const uint32_t b = (uint32_t)(u - T.unit0);
        const uint32_t nbc = (uint32_t)(T.cols / kLutCols);
        const uint32_t brow = b / nbc;
        const int64_t base = (int64_t)brow * kLutRows * T.cols + (int64_t)(b - brow * nbc) * kLutCols;
        unsigned char* st = ring + (size_t)s * p.stage_bytes;
        if (lane == 0) mbar_arrive_expect_tx(&bars[s], (uint32_t)kLutBlock * (8u + (uint32_t)gbytes));
        __syncwarp();
        if (lane < kLutRows) {
            const int r = lane;
            const int64_t off = base + r * T.cols;
            bulk_g2s(st + r * kLutCols * 4, T.w + off, kLutCols * 4, &bars[s]);
            bulk_g2s(st + kVOff + r * kLutCols * 4, T.v + off, kLutCols * 4, &bars[s]);
            if (gbytes)
                bulk_g2s(st + kGOff + r * kLutCols * gbytes,
                         static_cast<const unsigned char*>(T.g) + off * gbytes,
                         (uint32_t)(kLutCols * gbytes), &bars[s]);
        }
    };
    auto fail = [&](int64_t it) {
        if (lane == 0) record_timeout(p.status);
        for (int j = 0; j < S; ++j) {
            const int64_t u = first + (it + j) * stride;
            if (u >= n_units) break;
            mbar_wait_bounded(&bars[(it + j) % S], (uint32_t)(((it + j) / S) & 1), p.timeout_ns);
        }
    };

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
        const unsigned char* st = ring + (size_t)s_cur * p.stage_bytes;
        tensor_of(u, ti);
        const LutTensor& T = Lp.t[ti];
        const uint32_t b = (uint32_t)(u - T.unit0);
        const uint32_t nbc = (uint32_t)(T.cols / kLutCols);
        const uint32_t brow = b / nbc;
        // the lane's 16 elements: row lane/4 of the block, columns 16 (lane % 4) ..
        const int64_t gofs = ((int64_t)brow * kLutRows + (lane >> 2)) * T.cols +
                             (int64_t)(b - brow * nbc) * kLutCols + (lane & 3) * 16;

        // ---- pass A: w, the saliency EMA (v' out), the fit's saliency h
        float2 w2[8], h2[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int e = lane * 16 + i * 4;
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
                stg_cs(reinterpret_cast<float4*>(T.v + gofs + i * 4), make_float4(hA.x, hA.y, hB.x, hB.y));
            }
            h2[2 * i] = hA;
            h2[2 * i + 1] = hB;
        }
        // the block is in registers: release the stage
        __syncwarp();
        {
            const int64_t un = u + (int64_t)S * stride;
            if (un < n_units) issue(un, s_cur);
        }
        if (++s_cur == S) {
            s_cur = 0;
            parity ^= 1u;
        }
        if (p.h_mode != kSalEma)
#pragma unroll
            for (int t = 0; t < 8; ++t)
                h2[t] = p.h_mode == kSalEmaSquared ? __fmul2_rn(h2[t], h2[t]) : make_float2(1.0f, 1.0f);

        float mn = INFINITY, mx = -INFINITY, ss = 0.0f;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            mn = fminf(mn, fminf(w2[t].x, w2[t].y));
            mx = fmaxf(mx, fmaxf(w2[t].x, w2[t].y));
            ss += h2[t].x + h2[t].y;
        }
        mn = lanes_min(mn, 0xffffffffu);
        mx = lanes_max(mx, 0xffffffffu);
#pragma unroll
        for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        if (ss == 0.0f)  // all saliencies zero: h = 1
#pragma unroll
            for (int t = 0; t < 8; ++t) h2[t] = make_float2(1.0f, 1.0f);
        const float range = mx - mn;
        const bool flat = !(range > 0.0f);
        const float c = 0.5f * (mn + mx);
        const float R = flat ? 0.0f : __fdividef(7.0f, range);
        const float2 nc2 = make_float2(-c, -c);

        // candidate-independent: |d| = |w - c| and the saliency split by the
        // sign of d (a negative zero counts as negative, as the index does);
        // w itself is read again from memory only by the exact look
        float2 ad2[8], hp2[8], hn2[8];
        uint32_t negm = 0;  // bit i: element i has d < 0 (or -0)
        {
            float tp, tn, up, un, sd;
            float2 Tp = make_float2(0.0f, 0.0f), Tn = Tp, Up = Tp, Un = Tp, Sd = Tp;
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const float2 d = __fadd2_rn(w2[t], nc2);
                const bool nx = signbit(d.x), ny = signbit(d.y);
                negm |= (nx ? 1u : 0u) << (2 * t);
                negm |= (ny ? 1u : 0u) << (2 * t + 1);
                ad2[t] = make_float2(fabsf(d.x), fabsf(d.y));
                hp2[t] = make_float2(nx ? 0.0f : h2[t].x, ny ? 0.0f : h2[t].y);
                hn2[t] = make_float2(nx ? h2[t].x : 0.0f, ny ? h2[t].y : 0.0f);
                Tp = __fadd2_rn(Tp, hp2[t]);
                Tn = __fadd2_rn(Tn, hn2[t]);
                const float2 hd = __fmul2_rn(h2[t], ad2[t]);
                Up = __fadd2_rn(Up, make_float2(nx ? 0.0f : hd.x, ny ? 0.0f : hd.y));
                Un = __fadd2_rn(Un, make_float2(nx ? hd.x : 0.0f, ny ? hd.y : 0.0f));
                Sd = __ffma2_rn(hd, ad2[t], Sd);
            }
            tp = Tp.x + Tp.y;
            tn = Tn.x + Tn.y;
            up = Up.x + Up.y;
            un = Un.x + Un.y;
            sd = Sd.x + Sd.y;
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                tp += __shfl_xor_sync(0xffffffffu, tp, o);
                tn += __shfl_xor_sync(0xffffffffu, tn, o);
                up += __shfl_xor_sync(0xffffffffu, up, o);
                un += __shfl_xor_sync(0xffffffffu, un, o);
                sd += __shfl_xor_sync(0xffffffffu, sd, o);
            }
            // one value for every lane, kept in the scratch until the
            // candidates' entries need them
            if (lane == 0) {
                bconst[0] = tp;
                bconst[1] = tn;
                bconst[2] = up;
                bconst[3] = un;
                bconst[4] = sd;
                bconst[5] = ss;
                bconst[6] = range;
            }
        }

        int kb = 0;
        if (!flat) {
            // ---- candidates, four a pass: in two rounds of two, the
            // per-index sums of each (12 rows of the scratch a candidate)
            // summed across lanes, then entries and errors of all four at
            // once (lanes 8 q .. 8 q + 7 candidate k0 + q)
#pragma unroll 1
            for (int k0 = 0; k0 < K; k0 += 4) {
                float tot_a = 0.0f, tot_b = 0.0f;  // the two rounds' row sums
#pragma unroll 1
                for (int kr = k0; kr < min(k0 + 4, K); kr += 2) {
                    const int nk = min(2, K - kr);
#pragma unroll 1
                    for (int kk = 0; kk < nk; ++kk) {
                        const float P = R * p.invf[kr + kk];
                        const float2 P2 = make_float2(P, P);
                        // [l]: threshold m >= l + 1; sums of h (A) and h |d| (X),
                        // by sign.  The masked saliency h [m >= t] is exact, and
                        // so is its product with |d| inside the FMA: every term
                        // is exact.
                        float2 Ap[3], An[3], Xp[3], Xn[3];
#pragma unroll
                        for (int l = 0; l < 3; ++l) Ap[l] = An[l] = Xp[l] = Xn[l] = make_float2(0.0f, 0.0f);
#pragma unroll
                        for (int t = 0; t < 8; ++t) {
                            const float2 y = __ffma2_rd(ad2[t], P2, M2);  // 2^23 + floor(|d| P)
#pragma unroll
                            for (int l = 0; l < 3; ++l) {
                                const float nb = -(kMagic + (float)l);
                                const float2 mk = make_float2(add_sat(y.x, nb), add_sat(y.y, nb));
                                const float2 mp = __fmul2_rn(hp2[t], mk);
                                const float2 mq = __fmul2_rn(hn2[t], mk);
                                Ap[l] = __fadd2_rn(Ap[l], mp);
                                An[l] = __fadd2_rn(An[l], mq);
                                Xp[l] = __ffma2_rn(mp, ad2[t], Xp[l]);
                                Xn[l] = __ffma2_rn(mq, ad2[t], Xn[l]);
                            }
                        }
                        // rows (of this candidate's 12): A+ 0..2, A- 3..5, X+ 6..8,
                        // X- 9..11
                        float* rows = sums + kk * 12 * kLutRow + lane;
#pragma unroll
                        for (int l = 0; l < 3; ++l) {
                            rows[l * kLutRow] = Ap[l].x + Ap[l].y;
                            rows[(3 + l) * kLutRow] = An[l].x + An[l].y;
                            rows[(6 + l) * kLutRow] = Xp[l].x + Xp[l].y;
                            rows[(9 + l) * kLutRow] = Xn[l].x + Xn[l].y;
                        }
                    }
                    __syncwarp();
                    // lane r < 12 nk sums row r
                    if (lane < 12 * nk) {
                        float a0 = 0.0f, a1 = 0.0f, a2 = 0.0f, a3 = 0.0f;
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const float4 v = *reinterpret_cast<const float4*>(sums + lane * kLutRow + 4 * i);
                            a0 += v.x;
                            a1 += v.y;
                            a2 += v.z;
                            a3 += v.w;
                        }
                        const float tot = (a0 + a1) + (a2 + a3);
                        if (kr == k0) tot_a = tot;
                        else tot_b = tot;
                    }
                    __syncwarp();  // the scratch rows are rewritten by the next round
                }
                // lane j < 8 of each group q of 8: index j, sign s (j >= 4:
                // d >= 0), level m; its H = A_m - A_(m+1) and X = X_m - X_(m+1)
                // (A_0, X_0: the sign's totals; A_4 = X_4 = 0)
                const int q4 = lane >> 3;   // candidate k0 + q4
                const int half = q4 & 1;
                const int rb = half * 12;  // the candidate's first row in its round
                const float P = R * p.invf[min(k0 + q4, K - 1)];
                const float sg = __fdividef(1.0f, P);
                const int j = lane & 7;
                const bool pos = j >= 4;
                const int m = pos ? j - 4 : 3 - j;
                const int r0 = rb + (pos ? 0 : 3);
                // a row sum of this lane's round (q4 < 2: the first)
                auto row = [&](int r) {
                    const float va = __shfl_sync(0xffffffffu, tot_a, r);
                    const float vb = __shfl_sync(0xffffffffu, tot_b, r);
                    return q4 < 2 ? va : vb;
                };
                const float sA0 = row(r0 + max(m - 1, 0));
                const float sA1 = row(r0 + min(m, 2));
                const float sX0 = row(6 + r0 + max(m - 1, 0));
                const float sX1 = row(6 + r0 + min(m, 2));
                const float Am = m == 0 ? bconst[pos ? 0 : 1] : sA0;
                const float Am1 = m == 3 ? 0.0f : sA1;
                const float Xm = m == 0 ? bconst[pos ? 2 : 3] : sX0;
                const float Xm1 = m == 3 ? 0.0f : sX1;
                const float H = Am - Am1, X = fmaxf(Xm - Xm1, 0.0f);
                const float sgn = pos ? 1.0f : -1.0f;
                const float gj = fmaf((float)j - 3.5f, sg, c);  // the grid point
                // errors: the cumulative sums are sums of exact nonnegative
                // terms over at most tie_kappa levels (the per-sign totals of
                // h |d| carry one more rounding a term)
                const float dA = gam * (Am + Am1) + kU * H;
                const float dX = (gam + kU) * (Xm + Xm1) + kU * X;
                float mean = gj, q = 0.0f, dq = 0.0f, dm = 4.0f * kU * fabsf(gj);
                if (H > 0.0f) {
                    q = __fdividef(X, H);
                    mean = fmaf(sgn, q, c);
                    dq = __fdividef(dX + q * dA, H) + 2.0f * kU * q;
                    // plus the roundings of w - c (relative u each), of the
                    // quotient's use and of the mean's sum
                    dm = dq + 3.0f * kU * q + 2.0f * kU * fabsf(mean);
                }
                const uint32_t cb = e4m3_encode(mean);
                // an index whose H is not clearly above its error bound may be
                // empty or may hold weights of tiny saliency lost to the
                // differences: its entry is undecided unless nothing on its
                // side reaches its level, and its whole term is bounded below
                const bool thin = !(H > dA) && Am + Am1 > 0.0f;
                const bool amb = thin || e4m3_encode(mean - dm) != e4m3_encode(mean + dm);
                const float dc = e4m3_decode(cb) - mean;
                // the index's error: H (C - mean)^2 - X^2 / H (the scatter
                // term sum h d^2 is added once below)
                const float Sj = H > 0.0f && !thin ? fmaf(H * dc, dc, -X * q) : 0.0f;
                float bj = dA * dc * dc + 2.0f * H * fabsf(dc) * dm + 3.0f * kU * H * dc * dc + dX * q +
                           X * dq + 2.0f * kU * X * q;
                if (amb) {  // the other rounding moves the entry by at most this much
                    const float c1 = e4m3_decode(e4m3_encode(mean - dm)) - mean;
                    const float c2 = e4m3_decode(e4m3_encode(mean + dm)) - mean;
                    bj += H * fabsf(c2 - c1) * (fabsf(c1) + fabsf(c2) + 2.0f * dm);
                }
                bj = thin ? 2.0f * (dA + fabsf(H)) * bconst[6] * bconst[6] : bj;
                const bool live = k0 + q4 < K;
                float E = live ? Sj : 0.0f, dE = live ? bj : 0.0f, aE = live ? fabsf(Sj) : 0.0f;
                uint32_t wb = live ? cb << (8 * (lane & 3)) : 0u;
#pragma unroll
                for (int o = 4; o; o >>= 1) {
                    E += __shfl_xor_sync(0xffffffffu, E, o);
                    dE += __shfl_xor_sync(0xffffffffu, dE, o);
                    aE += __shfl_xor_sync(0xffffffffu, aE, o);
                }
                const float sd = bconst[4];
                E += sd;
                // sum h d^2: its terms' roundings (|d|^2, h times it) and sum
                dE += (gam + 3.0f * kU) * sd + 4.0f * kU * (sd + aE);
#pragma unroll
                for (int o = 2; o; o >>= 1) wb |= __shfl_xor_sync(0xffffffffu, wb, o);
                const uint32_t wb1 = __shfl_sync(0xffffffffu, wb, (lane & 24) | 4);
                const uint32_t ambm = __ballot_sync(0xffffffffu, amb && live);
                if ((lane & 7) == 0 && live) {
                    const int k = k0 + q4;
                    cbook[2 * k] = wb;
                    cbook[2 * k + 1] = wb1;
                    cerr[k] = E;
                    cbnd[k] = dE;
                    camb[k] = (ambm >> (8 * q4)) & 0xFFu;
                }
                __syncwarp();
            }
            __syncwarp();

            // ---- argmin (ties: lowest index); candidates that need an exact look
            float Ek = lane < K ? cerr[lane] : INFINITY;
            const float dEk = lane < K ? cbnd[lane] : 0.0f;
            float Eb = Ek;
            int kk = lane;
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                const float Eo = __shfl_xor_sync(0xffffffffu, Eb, o);
                const int ko = __shfl_xor_sync(0xffffffffu, kk, o);
                if (Eo < Eb || (Eo == Eb && ko < kk)) {
                    Eb = Eo;
                    kk = ko;
                }
            }
            kb = kk;
            const float dEb = __shfl_sync(0xffffffffu, dEk, kb);
            unsigned set = __ballot_sync(0xffffffffu, lane < K && lane != kb && Ek - Eb <= dEk + dEb);
            if (p.stats && lane == 0 && camb[kb]) atomicAdd(&p.stats[2], 1u);

            // a block whose sum of saliencies is near the bottom of the fp32
            // range: its fast sums are not to be trusted; h is scaled by a
            // power of two and every candidate and entry is settled below
            // (ts1 ts2: that power of two, applied where the settling steps
            // read h; 1 otherwise)
            float ts1 = 1.0f, ts2 = 1.0f;
            if (bconst[5] > 0.0f && bconst[5] < kTinySaliency) {
                tiny_scale(bconst[5], ts1, ts2);
                set = (K >= 32) ? 0xFFFFFFFFu : ((1u << K) - 1u);
                if (lane < K) camb[lane] = 0xFFu;
                __syncwarp();
            }

            // index (0..7) of element i for the grid of P
            auto index_of = [&](int i, float P) {
                const float a = (i & 1) ? ad2[i >> 1].y : ad2[i >> 1].x;
                const float mf = fminf(__fmaf_rd(a, P, kMagic) - kMagic, 3.0f);
                const int mi = (int)mf;
                return ((negm >> i) & 1u) ? 3 - mi : 4 + mi;
            };
            // Undecided entries of candidate k from direct per-index sums
            // (fp32, nonnegative exact terms, 16 + 5 levels: relative error
            // within 24 ulps): settled (table updated) unless a rounding is
            // still undecided.
            auto refine = [&](int k) -> bool {
                const float P = R * p.invf[k];
                uint32_t und = camb[k];
                uint32_t w0 = cbook[2 * k], w1 = cbook[2 * k + 1];
                while (und) {
                    const int j = __ffs(und) - 1;
                    und &= und - 1;
                    float Hs = 0.0f, Xs = 0.0f;
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        if (index_of(i, P) == j) {
                            const float hv = ((i & 1) ? hp2[i >> 1].y + hn2[i >> 1].y : hp2[i >> 1].x + hn2[i >> 1].x) * ts1 * ts2;
                            const float av = (i & 1) ? ad2[i >> 1].y : ad2[i >> 1].x;
                            Hs += hv;
                            Xs = fmaf(hv, av, Xs);
                        }
                    }
#pragma unroll
                    for (int o = 16; o; o >>= 1) {
                        Hs += __shfl_xor_sync(0xffffffffu, Hs, o);
                        Xs += __shfl_xor_sync(0xffffffffu, Xs, o);
                    }
                    Hs = __shfl_sync(0xffffffffu, Hs, 0);
                    Xs = __shfl_sync(0xffffffffu, Xs, 0);
                    uint32_t cbj;
                    if (!(Hs > 0.0f)) {
                        // no weight of nonzero saliency: the grid point
                        cbj = e4m3_encode(fmaf((float)j - 3.5f, __fdividef(1.0f, P), c));
                    } else {
                        const float q = Xs / Hs;
                        const float mean = fmaf(j >= 4 ? 1.0f : -1.0f, q, c);
                        // two sums (24 ulps each), the quotient, w - c (an ulp
                        // a term), the mean's sum
                        const float dm = 52.0f * kU * q + 2.0f * kU * fabsf(mean);
                        if (e4m3_encode(mean - dm) != e4m3_encode(mean + dm)) return false;
                        cbj = e4m3_encode(mean);
                    }
                    if (j < 4) w0 = (w0 & ~(0xFFu << (8 * j))) | (cbj << (8 * j));
                    else w1 = (w1 & ~(0xFFu << (8 * (j - 4)))) | (cbj << (8 * (j - 4)));
                }
                __syncwarp();
                if (lane == 0) {
                    cbook[2 * k] = w0;
                    cbook[2 * k + 1] = w1;
                    camb[k] = 0u;
                }
                __syncwarp();
                return true;
            };

            if (set == 0u) {
                // the winner alone: its table must be decided
                if (camb[kb] && !refine(kb)) set = 1u << kb;
            } else {
                set |= 1u << kb;
                bool decided = true;
                for (unsigned s2 = set; s2; s2 &= s2 - 1) {
                    const int k = __ffs(s2) - 1;
                    if (camb[k] && !refine(k)) decided = false;
                }
                if (decided) {
                    // direct fp32 errors sum h (C_q - w)^2 of the candidates
                    // left (terms within 3 ulps, 21 levels: 32 ulps in all)
                    if (p.stats && lane == 0) atomicAdd(&p.stats[3], 1u);
                    float xwv[16];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float4 w4 = __ldg(reinterpret_cast<const float4*>(T.w + gofs + i * 4));
                        xwv[4 * i] = w4.x;
                        xwv[4 * i + 1] = w4.y;
                        xwv[4 * i + 2] = w4.z;
                        xwv[4 * i + 3] = w4.w;
                    }
                    for (unsigned s2 = set; s2; s2 &= s2 - 1) {
                        const int k = __ffs(s2) - 1;
                        const float P = R * p.invf[k];
                        if (lane < 8)
                            table[lane] = e4m3_decode((cbook[2 * k + (lane >> 2)] >> (8 * (lane & 3))) & 0xFFu);
                        __syncwarp();
                        float acc = 0.0f;
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const float hv = ((i & 1) ? hp2[i >> 1].y + hn2[i >> 1].y : hp2[i >> 1].x + hn2[i >> 1].x) * ts1 * ts2;
                            const float df = table[index_of(i, P)] - xwv[i];
                            acc = fmaf(hv * df, df, acc);
                        }
#pragma unroll
                        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                        acc = __shfl_sync(0xffffffffu, acc, 0);
                        __syncwarp();
                        if (lane == 0) {
                            cerr[k] = acc;
                            cbnd[k] = 32.0f * kU * acc;
                        }
                    }
                    __syncwarp();
                    // the argmin again, over the set
                    const bool in = lane < K && ((set >> lane) & 1u);
                    float Ed = in ? cerr[lane] : INFINITY;
                    const float dEd = in ? cbnd[lane] : 0.0f;
                    float Edb = Ed;
                    int kd = lane;
#pragma unroll
                    for (int o = 16; o; o >>= 1) {
                        const float Eo = __shfl_xor_sync(0xffffffffu, Edb, o);
                        const int ko = __shfl_xor_sync(0xffffffffu, kd, o);
                        if (Eo < Edb || (Eo == Edb && ko < kd)) {
                            Edb = Eo;
                            kd = ko;
                        }
                    }
                    kb = kd;
                    const float dEdb = __shfl_sync(0xffffffffu, dEd, kb);
                    set = __ballot_sync(0xffffffffu, in && lane != kb && Ed - Edb <= dEd + dEdb);
                    if (set) set |= 1u << kb;
                }
            }


            // ---- exact look: float-float sums, exact roundings, direct error
            if (set) {
                if (p.stats && lane == 0) atomicAdd(&p.stats[0], 1u);
                // the lane's w again (from memory: this path is rare) and h
                float2 xw[8], xh[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float4 w4 = __ldg(reinterpret_cast<const float4*>(T.w + gofs + i * 4));
                    xw[2 * i] = make_float2(w4.x, w4.y);
                    xw[2 * i + 1] = make_float2(w4.z, w4.w);
                }
#pragma unroll
                for (int t = 0; t < 8; ++t)  // one of the two is 0
                    xh[t] = __fmul2_rn(__fmul2_rn(__fadd2_rn(hp2[t], hn2[t]), make_float2(ts1, ts1)),
                                       make_float2(ts2, ts2));
                float best_h = 0.0f, best_l = 0.0f;
                int best_k = -1;
                uint32_t best_w0 = 0, best_w1 = 0;
                while (set) {
                    const int k = __ffs(set) - 1;
                    set &= set - 1;
                    if (p.stats && lane == 0) atomicAdd(&p.stats[1], 1u);
                    const float P = R * p.invf[k];
                    const float sg = __fdividef(1.0f, P);
                    float zz[16];
#pragma unroll
                    for (int t = 0; t < 8; ++t) {
                        zz[2 * t] = code_z(xw[t].x - c, P);
                        zz[2 * t + 1] = code_z(xw[t].y - c, P);
                    }
                    uint32_t w0 = 0, w1 = 0;
#pragma unroll 1
                    for (int j = 0; j < 8; ++j) {
                        const float zj = (float)j - 3.5f;
                        const float gj = fmaf(zj, sg, c);
                        float Hh = 0.0f, Hl = 0.0f, Wh = 0.0f, Wl = 0.0f;
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            if (zz[i] == zj) {
                                const float hv = (i & 1) ? xh[i >> 1].y : xh[i >> 1].x;
                                const float wv = (i & 1) ? xw[i >> 1].y : xw[i >> 1].x;
                                float eh, el, ph, pl;
                                two_sum(wv, -gj, eh, el);
                                two_prod(hv, eh, ph, pl);
                                pl = fmaf(hv, el, pl);
                                ff_acc(Wh, Wl, ph, pl);
                                ff_acc(Hh, Hl, hv, 0.0f);
                            }
                        }
                        ff_reduce32(Hh, Hl);
                        ff_reduce32(Wh, Wl);
                        uint32_t cb;
                        if (Hh > 0.0f) {
                            // mean = g + W / H in float-float
                            const float qh = Wh / Hh;
                            float ph, pl;
                            two_prod(qh, Hh, ph, pl);
                            const float rr = __fsub_rn(__fsub_rn(__fadd_rn(__fsub_rn(Wh, ph), Wl), pl),
                                                       qh * Hl);
                            const float ql = rr / Hh;
                            float mh, ml;
                            two_sum(gj, qh, mh, ml);
                            ml = __fadd_rn(ml, ql);
                            ff_norm(mh, ml);
                            cb = e4m3_round_ff(mh, ml);
                        } else {
                            cb = e4m3_encode(gj);
                        }
                        if (j < 4) w0 |= cb << (8 * j);
                        else w1 |= cb << (8 * (j - 4));
                    }
                    // direct error sum h (C_q - w)^2
                    float eh = 0.0f, el = 0.0f;
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int q = (int)(zz[i] + 3.5f);
                        const uint32_t cb = ((q < 4 ? w0 : w1) >> (8 * (q & 3))) & 0xFFu;
                        const float hv = (i & 1) ? xh[i >> 1].y : xh[i >> 1].x;
                        const float wv = (i & 1) ? xw[i >> 1].y : xw[i >> 1].x;
                        float dh, dl, sh, sl;
                        two_sum(e4m3_decode(cb), -wv, dh, dl);
                        two_prod(dh, dh, sh, sl);
                        sl = fmaf(2.0f * dh, dl, sl);
                        float th, tl;
                        two_prod(hv, sh, th, tl);
                        tl = fmaf(hv, sl, tl);
                        ff_acc(eh, el, th, tl);
                    }
                    ff_reduce32(eh, el);
                    if (best_k < 0 || ff_less(eh, el, best_h, best_l)) {
                        best_h = eh;
                        best_l = el;
                        best_k = k;
                        best_w0 = w0;
                        best_w1 = w1;
                    }
                }
                kb = best_k;
                if (lane == 0) {
                    cbook[2 * kb] = best_w0;
                    cbook[2 * kb + 1] = best_w1;
                }
                __syncwarp();
            }
        }

        // ---- outputs of the kept candidate: table, indices, r
        uint32_t bw0, bw1;
        if (flat) {
            const uint32_t cb = e4m3_encode(c);
            bw0 = bw1 = cb * 0x01010101u;
        } else {
            bw0 = cbook[2 * kb];
            bw1 = cbook[2 * kb + 1];
        }
        if (lane < 8) table[lane] = e4m3_decode(((lane < 4 ? bw0 : bw1) >> (8 * (lane & 3))) & 0xFFu);
        __syncwarp();
        const float P = flat ? 0.0f : R * p.invf[kb];
        uint32_t q4[4] = {0u, 0u, 0u, 0u};  // the 16 indices, a byte each
        float rv[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float adv = (i & 1) ? ad2[i >> 1].y : ad2[i >> 1].x;
            const float dv = ((negm >> i) & 1u) ? -adv : adv;  // w - c
            const uint32_t q = flat ? 0u : (uint32_t)(int)(code_z(dv, P) + 3.5f);
            q4[i >> 2] |= q << (8 * (i & 3));
            rv[i] = table[q];
        }
        if (p.r_bf16) {
            uint32_t pk[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) pk[i] = pack_bf16x2(rv[2 * i], rv[2 * i + 1]);
            stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + gofs), make_uint2(pk[0], pk[1]));
            stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + gofs + 4), make_uint2(pk[2], pk[3]));
            stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + gofs + 8), make_uint2(pk[4], pk[5]));
            stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + gofs + 12), make_uint2(pk[6], pk[7]));
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                stg_cs(reinterpret_cast<float4*>(static_cast<float*>(T.r) + gofs + 4 * i),
                       make_float4(rv[4 * i], rv[4 * i + 1], rv[4 * i + 2], rv[4 * i + 3]));
        }
        if (T.codes) {
            if (!p.codes_packed) {
#pragma unroll
                for (int i = 0; i < 4; ++i) stg_cs(reinterpret_cast<uint32_t*>(T.codes + gofs) + i, q4[i]);
            } else {
                // 3 bits an index in block order: lane L's 48 bits at bit 48 L;
                // an even lane writes its pair's 12 bytes
                uint64_t bits48 = 0;
#pragma unroll
                for (int i = 0; i < 16; ++i) bits48 |= (uint64_t)((q4[i >> 2] >> (8 * (i & 3))) & 7u) << (3 * i);
                const uint32_t lo = (uint32_t)bits48, hi = (uint32_t)(bits48 >> 32);
                const uint32_t olo = __shfl_down_sync(0xffffffffu, lo, 1);
                const uint32_t ohi = __shfl_down_sync(0xffffffffu, hi, 1);
                if ((lane & 1) == 0) {
                    uint32_t* dst = reinterpret_cast<uint32_t*>(T.codes) + (size_t)b * 48 + (lane >> 1) * 3;
                    stg_cs(dst, lo);
                    stg_cs(dst + 1, (hi & 0xFFFFu) | (olo << 16));
                    stg_cs(dst + 2, (olo >> 16) | (ohi << 16));
                }
            }
        }
        if (lane == 0) {
            stg_cs(reinterpret_cast<uint2*>(T.book + (size_t)b * 8), make_uint2(bw0, bw1));
            if (T.idx) T.idx[b] = (uint8_t)kb;
        }
        __syncwarp();  // table and scratch are reused by the next block
    }
}

}  // namespace quasar
