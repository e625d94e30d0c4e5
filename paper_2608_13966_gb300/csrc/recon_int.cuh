// QUASAR reconstruction with asymmetric integer codes (Algorithm 1; Eq. 1
// code assignment, Eq. 4 weighted least-squares dequantizer, Eq. 3 weighted
// error; saliency EMA of Sec. 4.1.1 / App. A.2), one fused pass over HBM.
//
// Work decomposition.  A "unit" is 4 consecutive groups; one warp owns a unit
// at a time, 8 lanes per group, EPL = G/8 elements per lane.  Lane sl of a
// group holds elements {32*i + 4*sl + j : i < EPL/4, j < 4}, so every
// shared-memory read and global store of the warp is a set of full 128-byte
// segments.  Each warp runs its own ring of `stages` shared-memory buffers
// filled by 1-D TMA bulk copies (cp.async.bulk + mbarrier), so w, g and v are
// read from HBM exactly once and the loads of later units overlap the
// arithmetic of the current one.  The grid is persistent.
//
// Arithmetic per group (fp32):
//   v' = beta2*v + (1-beta2)*g^2 (written back), h = v';
//   min/max -> c, range; d = w - c;
//   per candidate k (codes t = d*P_k + qmax/2, P_k = qmax/(f_k*range),
//   clamped and rounded half-to-even with the 1.5*2^23 trick):
//     S1 = sum h q, S2 = sum h q^2, S3 = sum h q d;
//   common: Ss = sum h, Sd = sum h d, Sdd = sum h d^2;
//   each candidate's three sums are all-reduced over the 8 lanes of the
//   group and lane (k mod 8) keeps candidate k's; it forms
//   D = S2 - S1^2/Ss, N = S3 - S1*Sd/Ss,
//   the fit a = N/D, b = mean(d) - a*mean(q) (+c), and the explained term
//   E = N^2/D.  The weighted error of candidate k is C - E_k with C common,
//   so the argmin of the error is the argmax of E.
//
// Exactness.  E carries fp32 rounding error; candidates whose E lies within
// an error bound of the best (and candidates whose weighted code variance D
// is too small to trust) are re-evaluated exactly: codes recomputed, the fit
// redone in two centred passes, and sum h (a q + b - w)^2 evaluated directly
// with (a, b) rounded to a common power-of-two grid so that a*q + b is exact
// in fp32 and only w's subtraction rounds; per-lane partial sums are combined
// in fp64.  That direct error is what Algorithm 1 compares.
#pragma once

#include "device_common.cuh"
#include "params.h"

namespace quasar {

__device__ __forceinline__ float shx(float x, int m) { return __shfl_xor_sync(0xffffffffu, x, m); }

// Code of one element for one candidate (Eq. 1 in centred form):
// q = clamp(rne(d*P + qmax/2), 0, qmax), returned as a float.
__device__ __forceinline__ float int_code(float d, float P, float H, float qmaxf)
{
    float t = fmaf(d, P, H);
    t = fminf(fmaxf(t, 0.0f), qmaxf);
    const float y = __fadd_rn(t, kRoundMagic);
    return __fsub_rn(y, kRoundMagic);
}

// Round x to a multiple of the power of two U (x*invU is exact).
__device__ __forceinline__ float round_to_grid(float x, float U, float invU)
{
    return rintf(x * invU) * U;
}

// The rare paths below (exact comparison of near-tied candidates, the
// compensated fit) stream the group's w and h = v' again from global memory
// (L2-resident: this warp read them and wrote v' moments ago; each lane
// re-reads only the elements it wrote itself), one pass per sum, so the hot
// loop's per-lane arrays never need an address and stay in registers, and
// these functions need few registers of their own.
struct Chunk {
    float w[4], h[4], d[4];
};

__device__ __forceinline__ Chunk load_chunk(const float* wg, const float* hg, bool h_one, float c,
                                            int i, int sl)
{
    Chunk ch;
    const float4 w4 = __ldcg(reinterpret_cast<const float4*>(wg + i * 32 + sl * 4));
    const float4 h4 = __ldcg(reinterpret_cast<const float4*>(hg + i * 32 + sl * 4));
    ch.w[0] = w4.x; ch.w[1] = w4.y; ch.w[2] = w4.z; ch.w[3] = w4.w;
    ch.h[0] = h4.x; ch.h[1] = h4.y; ch.h[2] = h4.z; ch.h[3] = h4.w;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        if (h_one) ch.h[j] = 1.0f;
        ch.d[j] = ch.w[j] - c;
    }
    return ch;
}

// Error-free transformations (Knuth TwoSum, FMA-based TwoProd).
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

// (hi, lo) += (xh, xl); lo is left unnormalised (a group adds at most 32 terms per lane).
__device__ __forceinline__ void ff_acc(float& hi, float& lo, float xh, float xl)
{
    float sum, err;
    two_sum(hi, xh, sum, err);
    hi = sum;
    lo = __fadd_rn(lo, __fadd_rn(err, xl));
}

// Renormalise so that |lo| <= ulp(hi)/2 (Dekker's Fast2Sum; |hi| >= |lo|).
__device__ __forceinline__ void ff_norm(float& hi, float& lo)
{
    const float s = __fadd_rn(hi, lo);
    lo = __fsub_rn(lo, __fsub_rn(s, hi));
    hi = s;
}

// Sum of a float pair over the 8 lanes of a group (mask m), renormalised.
__device__ __forceinline__ void ff_reduce8(float& hi, float& lo, unsigned m)
{
    ff_norm(hi, lo);
#pragma unroll
    for (int o = 4; o; o >>= 1) {
        const float oh = __shfl_xor_sync(m, hi, o);
        const float ol = __shfl_xor_sync(m, lo, o);
        ff_acc(hi, lo, oh, ol);
        ff_norm(hi, lo);
    }
}

__device__ __forceinline__ bool ff_less(float ah, float al, float bh, float bl)
{
    return ah < bh || (ah == bh && al < bl);
}

// Weighted least-squares fit (Eq. 4) of one candidate on one group, in
// compensated arithmetic, for groups whose fp32 moment fit would miss the
// output tolerance (large weights with an offset near zero, or a badly
// conditioned code variance); the fit is returned as float pairs so that r
// can be formed to full fp32 accuracy.  Centres: mq = the weighted mean code
// rounded to 1/16 (so q - mq and (q - mq)^2 are exact) and mu ~ the weighted
// mean weight (w - mu kept as an exact pair).  The sums of h (q-mq)^2 and
// h (q-mq)(w-mu) are accumulated and combined across lanes as float pairs
// (no fp64: its rate on this part is a small fraction of fp32's); the
// offset is mu - s*mq + mean_h(w - mu - s (q - mq)).
template <int EPL>
__device__ __noinline__ void precise_fit(const float* wg, const float* hg, bool h_one, float c,
                                         int sl, unsigned m, float P, float H, float qmaxf,
                                         float Ss, float mu, float* a_hi, float* a_lo,
                                         float* B_hi, float* B_lo)
{
    float s1 = 0.0f;
#pragma unroll 1
    for (int i = 0; i < EPL / 4; ++i) {
        const Chunk ch = load_chunk(wg, hg, h_one, c, i, sl);
#pragma unroll
        for (int j = 0; j < 4; ++j) s1 = fmaf(ch.h[j], int_code(ch.d[j], P, H, qmaxf), s1);
    }
#pragma unroll
    for (int o = 4; o; o >>= 1) s1 += __shfl_xor_sync(m, s1, o);
    const float mq = rintf(s1 / Ss * 16.0f) * 0.0625f;

    float Dh = 0.0f, Dl = 0.0f, Nh = 0.0f, Nl = 0.0f, A = 0.0f, B = 0.0f;
#pragma unroll 1
    for (int i = 0; i < EPL / 4; ++i) {
        const Chunk ch = load_chunk(wg, hg, h_one, c, i, sl);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float qd = int_code(ch.d[j], P, H, qmaxf) - mq;
            float wh, wl, xh, xl, th, tl, ph, pl;
            two_sum(ch.w[j], -mu, wh, wl);
            two_prod(ch.h[j], qd, xh, xl);
            two_prod(xh, qd, th, tl);
            tl = fmaf(xl, qd, tl);
            ff_acc(Dh, Dl, th, tl);
            two_prod(xh, wh, ph, pl);
            pl = fmaf(xh, wl, fmaf(xl, wh, pl));
            ff_acc(Nh, Nl, ph, pl);
            A = __fadd_rn(A, xh);
            B = fmaf(ch.h[j], wh, B);
        }
    }
    ff_reduce8(Dh, Dl, m);
    ff_reduce8(Nh, Nl, m);
#pragma unroll
    for (int o = 4; o; o >>= 1) {
        A += __shfl_xor_sync(m, A, o);
        B += __shfl_xor_sync(m, B, o);
    }
    // centring corrections (small: mq and mu are close to the weighted means)
    {
        float sum, err;
        two_sum(Dh, -(A * A / Ss), sum, err);
        Dh = sum;
        Dl = __fadd_rn(Dl, err);
        ff_norm(Dh, Dl);
        two_sum(Nh, -(A * B / Ss), sum, err);
        Nh = sum;
        Nl = __fadd_rn(Nl, err);
        ff_norm(Nh, Nl);
    }
    // s = N / D as a float pair: the remainder N - s_hi*D is exact by FMA
    const float shi = Nh / Dh;
    const float rem = __fadd_rn(fmaf(-shi, Dh, Nh), fmaf(-shi, Dl, Nl));
    const float slo = rem / Dh;
    float Rs = 0.0f;
#pragma unroll 1
    for (int i = 0; i < EPL / 4; ++i) {
        const Chunk ch = load_chunk(wg, hg, h_one, c, i, sl);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float qd = int_code(ch.d[j], P, H, qmaxf) - mq;
            float wh, wl;
            two_sum(ch.w[j], -mu, wh, wl);
            const float res = __fadd_rn(fmaf(-shi, qd, wh), fmaf(-slo, qd, wl));
            Rs = fmaf(ch.h[j], res, Rs);
        }
    }
#pragma unroll
    for (int o = 4; o; o >>= 1) Rs += __shfl_xor_sync(m, Rs, o);
    // z = mu - s*mq + mean_h(residual)
    float ph, pl, zh, zl;
    two_prod(shi, mq, ph, pl);
    pl = fmaf(slo, mq, pl);
    two_sum(mu, -ph, zh, zl);
    zl = __fadd_rn(__fsub_rn(zl, pl), Rs / Ss);
    ff_norm(zh, zl);
    *a_hi = shi;
    *a_lo = slo;
    *B_hi = zh;
    *B_lo = zl;
}

// Exact evaluation of one candidate on one group (8 lanes, mask m): codes,
// exact degenerate test, two-pass centred fit, and the direct weighted error
// sum h (a q + b - w)^2 with (a, b) on a common power-of-two grid U so that
// a*q + b is exact and only "- w" rounds; per-lane sums are combined as a
// float pair (err[0] + err[1]).
template <int EPL>
__device__ __noinline__ void segment_exact(const float* wg, const float* hg, bool h_one, int sl,
                                           unsigned m, float P, float H, float qmaxf, float Ss,
                                           float dbar, float c, float step, float* err,
                                           float* a_out, float* bc_out, float* qbar_out,
                                           bool* degenerate)
{
    float s1 = 0.0f;
    int qlo = 1 << 30, qhi = -1;
#pragma unroll 1
    for (int i = 0; i < EPL / 4; ++i) {
        const Chunk ch = load_chunk(wg, hg, h_one, c, i, sl);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float q = int_code(ch.d[j], P, H, qmaxf);
            s1 = fmaf(ch.h[j], q, s1);
            if (ch.h[j] > 0.0f) {
                qlo = min(qlo, (int)q);
                qhi = max(qhi, (int)q);
            }
        }
    }
#pragma unroll
    for (int o = 4; o; o >>= 1) {
        s1 += __shfl_xor_sync(m, s1, o);
        qlo = min(qlo, __shfl_xor_sync(m, qlo, o));
        qhi = max(qhi, __shfl_xor_sync(m, qhi, o));
    }
    float a, bc;
    const float qbar = s1 / Ss;
    *qbar_out = qbar;
    *degenerate = qlo == qhi;
    if (qlo == qhi) {
        // every weighted element shares one code: a = grid step
        a = step;
        bc = dbar - step * (float)qlo;
    } else {
        float dd = 0.0f, nn = 0.0f;
#pragma unroll 1
        for (int i = 0; i < EPL / 4; ++i) {
            const Chunk ch = load_chunk(wg, hg, h_one, c, i, sl);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float dq = int_code(ch.d[j], P, H, qmaxf) - qbar;
                const float hdq = ch.h[j] * dq;
                dd = fmaf(hdq, dq, dd);
                nn = fmaf(hdq, ch.d[j] - dbar, nn);
            }
        }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            dd += __shfl_xor_sync(m, dd, o);
            nn += __shfl_xor_sync(m, nn, o);
        }
        a = nn / dd;
        bc = dbar - a * qbar;
    }
    const float B = bc + c;
    const float mr = fmaxf(fabsf(B), fabsf(fmaf(a, qmaxf, B))) + fabsf(a);
    int er = (int)((__float_as_uint(mr) >> 23) & 0xFF) - 126;  // mr < 2^er
    er = max(er, -100);
    const float U = __uint_as_float((uint32_t)(er - 23 + 127) << 23);
    const float invU = __uint_as_float((uint32_t)(23 - er + 127) << 23);
    const float ag = round_to_grid(a, U, invU);
    const float Bg = round_to_grid(B, U, invU);
    // per-chunk pairwise sums, then pairwise over chunks
    float part[EPL / 4];
#pragma unroll
    for (int i = 0; i < EPL / 4; ++i) {
        const Chunk ch = load_chunk(wg, hg, h_one, c, i, sl);
        float t[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float e = fmaf(ag, int_code(ch.d[j], P, H, qmaxf), Bg) - ch.w[j];
            t[j] = ch.h[j] * (e * e);
        }
        part[i] = (t[0] + t[1]) + (t[2] + t[3]);
    }
#pragma unroll
    for (int s = 1; s < EPL / 4; s <<= 1)
#pragma unroll
        for (int i = 0; i + s < EPL / 4; i += 2 * s) part[i] += part[i + s];
    float eh = part[0], el = 0.0f;
    ff_reduce8(eh, el, m);
    err[0] = eh;
    err[1] = el;
    *a_out = a;
    *bc_out = bc;
}

template <int EPL, int NCH>
__global__ void __launch_bounds__(256) k_recon_int(const IntParams p)
{
    constexpr int G = EPL * kLanesPerGroup;
    constexpr int UNIT = kGroupsPerUnit * G;
    extern __shared__ __align__(128) unsigned char smem[];

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int gs = lane >> 3;
    const int sl = lane & 7;
    const unsigned seg_mask = 0xFFu << (gs * 8);

    const int S = p.stages;
    unsigned char* ring = smem + (size_t)warp * S * p.stage_bytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)nwarps * S * p.stage_bytes) + warp * (S + 1);

    const int gbytes = p.g_kind == 2 ? 2 : (p.g_kind == 1 ? 4 : 0);
    constexpr uint32_t kVOff = UNIT * 4;
    constexpr uint32_t kGOff = UNIT * 8;

    const int64_t n_units = (p.n_groups + kGroupsPerUnit - 1) / kGroupsPerUnit;
    const int64_t first = (int64_t)blockIdx.x * nwarps + warp;
    const int64_t stride = (int64_t)gridDim.x * nwarps;

    if (lane == 0) {
        for (int s = 0; s <= S; ++s) mbar_init(&bars[s], 1);
        mbar_init_fence();
    }
    __syncwarp();

    auto issue = [&](int64_t u, int s) {
        const int64_t g0 = u * kGroupsPerUnit;
        const int64_t ng = min((int64_t)kGroupsPerUnit, p.n_groups - g0);
        const uint32_t elems = (uint32_t)(ng * G);
        unsigned char* st = ring + (size_t)s * p.stage_bytes;
        mbar_arrive_expect_tx(&bars[s], elems * (8u + (uint32_t)gbytes));
        bulk_g2s(st, p.w + g0 * G, elems * 4u, &bars[s]);
        bulk_g2s(st + kVOff, p.v + g0 * G, elems * 4u, &bars[s]);
        if (gbytes)
            bulk_g2s(st + kGOff, static_cast<const unsigned char*>(p.g) + g0 * G * gbytes,
                     elems * (uint32_t)gbytes, &bars[s]);
    };

    // Drain the copies still in flight from iteration `it` on, then leave.
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
        // Failure-path hook: a barrier nothing ever arrives on.
        if (!mbar_wait_bounded(&bars[S], 0, p.force_timeout_ns)) {
            fail(0);
            return;
        }
    }

    const float qmaxf = (float)p.qmax;
    const float H = 0.5f * qmaxf;
    // The hot loop accumulates codes centred on Hc = floor(qmax/2): subtracting
    // the rounding constant plus Hc (exact) yields q - Hc directly and keeps the
    // moment sums well conditioned.
    const float Hc = (float)(p.qmax >> 1);
    const float magic_c = kRoundMagic + Hc;
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

        float w[EPL], h[EPL];
#pragma unroll
        for (int i = 0; i < EPL / 4; ++i) {
            const int e = gs * G + i * 32 + sl * 4;
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

        const int64_t grp = u * kGroupsPerUnit + gs;
        const bool valid = grp < p.n_groups;
        const int64_t gbase = grp * (int64_t)G;

        if (valid && p.g_kind) {
#pragma unroll
            for (int i = 0; i < EPL / 4; ++i)
                stg_cs(reinterpret_cast<float4*>(p.v + gbase + i * 32 + sl * 4),
                       make_float4(h[4 * i], h[4 * i + 1], h[4 * i + 2], h[4 * i + 3]));
        }

        // ---- group range and saliency mass ----
        float mn = w[0], mx = w[0], ss = 0.0f;
#pragma unroll
        for (int j = 0; j < EPL; ++j) {
            mn = fminf(mn, w[j]);
            mx = fmaxf(mx, w[j]);
            ss += h[j];
        }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            mn = fminf(mn, shx(mn, o));
            mx = fmaxf(mx, shx(mx, o));
            ss += shx(ss, o);
        }
        const bool h_one = ss == 0.0f;
        if (h_one) {  // all saliencies zero: fit with h = 1
#pragma unroll
            for (int j = 0; j < EPL; ++j) h[j] = 1.0f;
            ss = (float)G;
        }
        // where the rare paths find h again: v' as just written, or v itself
        const float* hsrc = p.v;
        const float range = mx - mn;
        const bool flat = !(range > 0.0f);
        const float c = 0.5f * (mn + mx);
        const float R = flat ? 0.0f : qmaxf / range;

        float d[EPL];
        float sd = 0.0f, sdd = 0.0f;
#pragma unroll
        for (int j = 0; j < EPL; ++j) {
            d[j] = w[j] - c;
            const float hd = h[j] * d[j];
            sd += hd;
            sdd = fmaf(hd, d[j], sdd);
        }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            sd += shx(sd, o);
            sdd += shx(sdd, o);
        }
        const float inv_ss = 1.0f / ss;
        const float dbar = sd * inv_ss;
        // Cauchy-Schwarz bound of sum h |q d| / qmax, for the error bound on N.
        const float habsd = sqrtf(ss * sdd);
        const float ulp = 5.9604645e-8f * p.tie_kappa;

        // ---- candidate search: this lane owns candidates ch*8 + sl ----
        // Candidate loop (rolled, to keep the code small): the three
        // per-candidate sums are all-reduced over the 8 lanes of the group and
        // lane (k mod 8) keeps the totals of candidate k.
        float T1k[NCH], T2k[NCH], T3k[NCH];
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) T1k[ch] = T2k[ch] = T3k[ch] = 0.0f;
#pragma unroll 1
        for (int k = 0; k < NCH * 8; ++k) {
            const float P = R * p.invf[k];
            float s1 = 0.0f, s2 = 0.0f, s3 = 0.0f;
#pragma unroll
            for (int j = 0; j < EPL; ++j) {
                float t = fmaf(d[j], P, H);
                t = fminf(fmaxf(t, 0.0f), qmaxf);
                const float q = __fsub_rn(__fadd_rn(t, kRoundMagic), magic_c);  // q - Hc
                const float hq = __fmul_rn(h[j], q);
                s1 = __fadd_rn(s1, hq);
                s2 = fmaf(hq, q, s2);
                s3 = fmaf(hq, d[j], s3);
            }
#pragma unroll
            for (int o = 4; o; o >>= 1) {
                s1 += shx(s1, o);
                s2 += shx(s2, o);
                s3 += shx(s3, o);
            }
            if ((k & 7) == sl) {
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch)
                    if ((k >> 3) == ch) {
                        T1k[ch] = s1;
                        T2k[ch] = s2;
                        T3k[ch] = s3;
                    }
            }
        }
        float Ek[NCH], dEk[NCH], ak[NCH], bk[NCH], condk[NCH];
        bool suspk[NCH];
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) {
            const float T[3] = {T1k[ch], T2k[ch], T3k[ch]};
            const int k = ch * 8 + sl;
            const float qbar = T[0] * inv_ss;  // mean of q - Hc
            const float D = T[1] - T[0] * qbar;
            const float N = T[2] - T[0] * dbar;
            const bool susp = !(D > 1e-3f * T[1]);
            const float a = N / D;
            const float E = susp ? 0.0f : N * a;
            const float dN = ulp * qmaxf * habsd;
            const float dD = ulp * T[1];
            const bool real = k < p.n_clip;
            Ek[ch] = real && !susp ? E : -INFINITY;
            dEk[ch] = 2.0f * fabsf(a) * dN + a * a * dD;
            ak[ch] = a;
            bk[ch] = dbar - a * (qbar + Hc);
            condk[ch] = T[1] / D + (fabsf(T[2]) + fabsf(T[0] * dbar)) / fabsf(N);
            suspk[ch] = real && susp;
        }

        // ---- argmax of E over the group (ties: lowest index) ----
        float Eb = -INFINITY, dEb = 0.0f;
        int kb = 0x7fff;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch)
            if (Ek[ch] > Eb) {  // strict: keeps the lower k of this lane
                Eb = Ek[ch];
                dEb = dEk[ch];
                kb = ch * 8 + sl;
            }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            const float Eo = shx(Eb, o);
            const float dEo = shx(dEb, o);
            const int ko = __shfl_xor_sync(0xffffffffu, kb, o);
            if (Eo > Eb || (Eo == Eb && ko < kb)) {
                Eb = Eo;
                dEb = dEo;
                kb = ko;
            }
        }
        if (kb > 0x7ff) kb = 0;  // every candidate suspicious: the exact path picks

        // Fit of the winner and its weighted code sum, from its owner lane.
        float a_sel = 0.0f, bc_sel = 0.0f, cond_sel = 0.0f, T1b = 0.0f;
        {
            const int owner = (gs * 8) | (kb & 7);
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) {
                const float av = __shfl_sync(0xffffffffu, ak[ch], owner);
                const float bv = __shfl_sync(0xffffffffu, bk[ch], owner);
                const float cv = __shfl_sync(0xffffffffu, condk[ch], owner);
                const float t1 = __shfl_sync(0xffffffffu, T1k[ch], owner);
                if ((kb >> 3) == ch) {
                    a_sel = av;
                    bc_sel = bv;
                    cond_sel = cv;
                    T1b = t1;
                }
            }
        }
        // Candidates that need an exact comparison: within the fp32 error
        // bound of the winner.  (Equal fp32 moments do not prove equal codes:
        // an element of tiny saliency can change the error without changing
        // the rounded moments, so such candidates are compared exactly too.)
        unsigned my_set = 0;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) {
            const int k = ch * 8 + sl;
            const bool contender = k != kb && Ek[ch] > -INFINITY && Eb - Ek[ch] <= dEb + dEk[ch];
            if (contender || suspk[ch]) my_set |= 1u << ch;
        }
        unsigned set = 0;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) {
            const unsigned bal = __ballot_sync(0xffffffffu, (my_set >> ch) & 1u);
            set |= ((bal >> (gs * 8)) & 0xFFu) << (ch * 8);
        }

        float qbar_sel = T1b * inv_ss + Hc;
        bool deg_sel = false;
        const bool need_exact = valid && !flat && (set != 0 || Eb == -INFINITY);
        if (need_exact) {
            if (p.stats && sl == 0) atomicAdd(&p.stats[0], 1u);
            unsigned todo = set | (Eb == -INFINITY ? 0u : 1u << kb);
            if (Eb == -INFINITY) todo |= (p.n_clip >= 32) ? 0xFFFFFFFFu : ((1u << p.n_clip) - 1u);
            float best_eh = 0.0f, best_el = 0.0f;
            int best_k = -1;
            float best_a = 0.0f, best_bc = 0.0f, best_qbar = 0.0f;
            bool best_deg = false;
            while (todo) {
                const int k = __ffs(todo) - 1;
                todo &= todo - 1;
                const float P = R * p.invf[k];
                const float step = p.f[k] * range / qmaxf;
                float err[2];
                float a_k, bc_k, qbar_k;
                bool deg_k;
                segment_exact<EPL>(p.w + gbase, hsrc + gbase, h_one, sl, seg_mask, P, H, qmaxf, ss,
                                   dbar, c, step, err, &a_k, &bc_k, &qbar_k, &deg_k);
                if (best_k < 0 || ff_less(err[0], err[1], best_eh, best_el)) {
                    best_eh = err[0];
                    best_el = err[1];
                    best_k = k;
                    best_a = a_k;
                    best_bc = bc_k;
                    best_qbar = qbar_k;
                    best_deg = deg_k;
                }
            }
            kb = best_k;
            a_sel = best_a;
            bc_sel = best_bc;
            qbar_sel = best_qbar;
            deg_sel = best_deg;
            cond_sel = 1.0f;
        }
        float Bsel = bc_sel + c;
        // fp32 error estimate of the fit: the line passes through the weighted
        // centroid, so b, and every level a*q + b, errs by a few ulp of
        // |w| + a*qbar.  Compared with half the output tolerance 1e-7 + 1e-5|x|
        // at the offset and at the level closest to zero.
        const float est_b = 2.3841858e-07f * (fabsf(c) + 0.5f * range) * (1.0f + qbar_sel);
        const float q0 = fminf(fmaxf(rintf(-Bsel / a_sel), 0.0f), qmaxf);
        const float rmin = fminf(fabsf(Bsel), fabsf(fmaf(a_sel, q0, Bsel)));
        const bool need_precise = valid && !flat && !deg_sel &&
                                  (!(cond_sel <= p.refit_cond) ||
                                   est_b > 0.5f * (1e-7f + 1e-5f * rmin));
        float a_lo = 0.0f, B_lo = 0.0f;
        if (need_precise) {
            if (p.stats && sl == 0) atomicAdd(&p.stats[1], 1u);
            precise_fit<EPL>(p.w + gbase, hsrc + gbase, h_one, c, sl, seg_mask, R * p.invf[kb], H,
                             qmaxf, ss, c + dbar, &a_sel, &a_lo, &Bsel, &B_lo);
        }

        // ---- outputs of the kept candidate ----
        if (!valid) continue;
        const float Pb = R * p.invf[kb];
#pragma unroll
        for (int i = 0; i < EPL / 4; ++i) {
            float rv[4];
            uint32_t cw = 0;
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
                const int j = 4 * i + jj;
                if (flat) {
                    rv[jj] = w[j];
                } else {
                    float t = fmaf(d[j], Pb, H);
                    t = fminf(fmaxf(t, 0.0f), qmaxf);
                    const float y = __fadd_rn(t, kRoundMagic);
                    const float q = __fsub_rn(y, kRoundMagic);
                    // a_lo, B_lo are zero unless the compensated fit ran
                    rv[jj] = fmaf(a_sel, q, Bsel) + fmaf(a_lo, q, B_lo);
                    cw |= (__float_as_uint(y) & 0xFFu) << (8 * jj);
                }
            }
            const int64_t e = gbase + i * 32 + sl * 4;
            if (p.r_bf16) {
                stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.r) + e),
                       make_uint2(pack_bf16x2(rv[0], rv[1]), pack_bf16x2(rv[2], rv[3])));
            } else {
                stg_cs(reinterpret_cast<float4*>(static_cast<float*>(p.r) + e),
                       make_float4(rv[0], rv[1], rv[2], rv[3]));
            }
            if (p.codes) stg_cs(reinterpret_cast<uint32_t*>(p.codes + e), cw);
        }
        if (sl == 0) {
            p.a[grp] = flat ? 0.0f : a_sel;
            p.b[grp] = flat ? w[0] : Bsel;
            if (p.idx) p.idx[grp] = flat ? 0 : (uint8_t)kb;
        }
    }
}

}  // namespace quasar
