// QUASAR reconstruction with asymmetric integer codes (Algorithm 1; Eq. 1
// code assignment, Eq. 4 weighted least-squares dequantizer, Eq. 3 weighted
// error; saliency EMA of Sec. 4.1.1 / App. A.2), one fused pass over HBM.
//
// Work decomposition.  A "unit" is 4 consecutive groups; one warp owns a unit
// at a time, 8 lanes per group, EPL = G/8 elements per lane.  Lane sl of a
// group handles elements {32*i + 4*sl + j : i < EPL/4, j < 4}, so every
// 16-byte shared-memory access of the warp is bank-conflict free and every
// global store covers whole 128-byte segments.  Each warp runs its own ring
// of `stages` shared-memory tiles filled by 1-D TMA bulk copies
// (cp.async.bulk + mbarrier), so w, g and v are read from HBM exactly once,
// and the loads of later units overlap the arithmetic of the current one.
// The tile stays in shared memory while the unit is processed, and the
// passes below stream it from there (rolled loops: small code, few
// registers).  The grid is persistent.
//
// Per group (fp32):
//   pass A  v' = beta2*v + (1-beta2)*g^2 (written back; kept in the tile as
//           the saliency h), min/max -> c, range, sum h;
//   pass B  for 8 candidates at a time, codes q = clamp(rne(d*P_k + qmax/2))
//           with d = w - c and P_k = qmax/(f_k*range) (the 1.5*2^23 rounding
//           trick; codes are accumulated centred on Hc = floor(qmax/2)), and
//           the sums S1 = sum h q, S2 = sum h q^2, S3 = sum h q d; packed
//           f32x2 arithmetic, two elements per instruction;
//   reduce  the 8 lanes' partial sums are transposed through shared memory
//           so that lane sl owns candidate sl of the chunk;
//   fit     D = S2 - S1^2/Ss, N = S3 - S1*Sd/Ss, a = N/D, b = mean(d) -
//           a*mean(q) (+c), explained E = N^2/D: the weighted error of
//           candidate k is C - E_k with C common, so argmin error = argmax E;
//   pass C  codes of the kept candidate, r = a*q + b, outputs.
//
// Exactness.  E carries fp32 rounding error; candidates whose E lies within
// an error bound of the best (and candidates whose weighted code variance D
// is too small to trust) are re-evaluated exactly, and fits whose fp32
// rounding could miss the output tolerance are recomputed in compensated
// (float-float) arithmetic.  Both are rare; they are deferred to the end of
// the unit and done by the whole warp on one group at a time.
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

// ---------------------------------------------------------------- float pairs

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

// (hi, lo) += (xh, xl); lo is left unnormalised (at most 8 terms per lane).
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

// Sum of a float pair over the 32 lanes of the warp, renormalised.
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
}

__device__ __forceinline__ bool ff_less(float ah, float al, float bh, float bl)
{
    return ah < bh || (ah == bh && al < bl);
}

__device__ __forceinline__ float wsum32(float x)
{
#pragma unroll
    for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// ------------------------------------------------- whole-warp group helpers
//
// One group, evaluated by all 32 lanes (lane L takes elements L + 32m) from
// the tile in shared memory: w at ws, saliency h at hs (or 1 if h_one).

// True when candidates with scale factors Pa and Pb give the same codes on
// every element of the group (whole warp).
template <int G>
__device__ bool coop_same_codes(const float* ws, float c, float Pa, float Pb, float H, float qmaxf)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    bool same = true;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const float d = ws[lane + 32 * m] - c;
        same &= int_code(d, Pa, H, qmaxf) == int_code(d, Pb, H, qmaxf);
    }
    return __all_sync(0xffffffffu, same);
}

// Exact evaluation of one candidate: codes, exact degenerate test (all
// weighted elements on one code), two-pass centred fit, and the direct error
// sum h (a q + b - w)^2 with (a, b) rounded to a common power-of-two grid U so
// that a*q + b is exact and only "- w" rounds; lanes combine as a float pair.
template <int G>
__device__ void coop_exact(const float* ws, const float* hs, bool h_one, float c, float P,
                           float H, float qmaxf, float Ss, float dbar, float step, float* err_hi,
                           float* err_lo, float* a_out, float* bc_out, bool* degenerate)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    float s1 = 0.0f;
    int qlo = 1 << 30, qhi = -1;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = h_one ? 1.0f : hs[e];
        const float q = int_code(ws[e] - c, P, H, qmaxf);
        s1 = fmaf(h, q, s1);
        if (h > 0.0f) {
            qlo = min(qlo, (int)q);
            qhi = max(qhi, (int)q);
        }
    }
    s1 = wsum32(s1);
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        qlo = min(qlo, __shfl_xor_sync(0xffffffffu, qlo, o));
        qhi = max(qhi, __shfl_xor_sync(0xffffffffu, qhi, o));
    }
    const float qbar = s1 / Ss;
    *degenerate = qlo == qhi;
    float a, bc;
    if (qlo == qhi) {
        a = step;  // every weighted element shares one code
        bc = dbar - step * (float)qlo;
    } else {
        float dd = 0.0f, nn = 0.0f;
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const int e = lane + 32 * m;
            const float h = h_one ? 1.0f : hs[e];
            const float d = ws[e] - c;
            const float dq = int_code(d, P, H, qmaxf) - qbar;
            const float hdq = h * dq;
            dd = fmaf(hdq, dq, dd);
            nn = fmaf(hdq, d - dbar, nn);
        }
        a = wsum32(nn) / wsum32(dd);
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
    float t[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = h_one ? 1.0f : hs[e];
        const float w = ws[e];
        const float ev = fmaf(ag, int_code(w - c, P, H, qmaxf), Bg) - w;
        t[m] = h * (ev * ev);
    }
#pragma unroll
    for (int s = 1; s < M; s <<= 1)
#pragma unroll
        for (int m = 0; m + s < M; m += 2 * s) t[m] += t[m + s];
    float eh = t[0], el = 0.0f;
    ff_reduce32(eh, el);
    *err_hi = eh;
    *err_lo = el;
    *a_out = a;
    *bc_out = bc;
}

// Weighted least-squares fit (Eq. 4) of one candidate in compensated
// arithmetic, for groups whose fp32 fit could miss the output tolerance
// (large weights with an offset or a level near zero, or badly conditioned
// code variance).  Centres: mq = the weighted mean code rounded to 1/16 (so
// q - mq and (q - mq)^2 are exact) and mu ~ the weighted mean weight (w - mu
// kept as an exact pair).  The sums of h (q-mq)^2 and h (q-mq)(w-mu) are
// accumulated and combined across lanes as float pairs (no fp64: its rate on
// this part is a small fraction of fp32's); the offset is
// mu - s*mq + mean_h(w - mu - s (q - mq)).  Returns the fit as float pairs.
template <int G>
__device__ void coop_precise(const float* ws, const float* hs, bool h_one, float c, float P,
                             float H, float qmaxf, float Ss, float mu, float* a_hi, float* a_lo,
                             float* B_hi, float* B_lo)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    float s1 = 0.0f;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = h_one ? 1.0f : hs[e];
        s1 = fmaf(h, int_code(ws[e] - c, P, H, qmaxf), s1);
    }
    const float mq = rintf(wsum32(s1) / Ss * 16.0f) * 0.0625f;

    float Dh = 0.0f, Dl = 0.0f, Nh = 0.0f, Nl = 0.0f, A = 0.0f, B = 0.0f;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = h_one ? 1.0f : hs[e];
        const float w = ws[e];
        const float qd = int_code(w - c, P, H, qmaxf) - mq;
        float wh, wl, xh, xl, th, tl, ph, pl;
        two_sum(w, -mu, wh, wl);
        two_prod(h, qd, xh, xl);
        two_prod(xh, qd, th, tl);
        tl = fmaf(xl, qd, tl);
        ff_acc(Dh, Dl, th, tl);
        two_prod(xh, wh, ph, pl);
        pl = fmaf(xh, wl, fmaf(xl, wh, pl));
        ff_acc(Nh, Nl, ph, pl);
        A = __fadd_rn(A, xh);
        B = fmaf(h, wh, B);
    }
    ff_reduce32(Dh, Dl);
    ff_reduce32(Nh, Nl);
    A = wsum32(A);
    B = wsum32(B);
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
    const float slo = __fadd_rn(fmaf(-shi, Dh, Nh), fmaf(-shi, Dl, Nl)) / Dh;
    float Rs = 0.0f;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = h_one ? 1.0f : hs[e];
        const float w = ws[e];
        const float qd = int_code(w - c, P, H, qmaxf) - mq;
        float wh, wl;
        two_sum(w, -mu, wh, wl);
        Rs = fmaf(h, __fadd_rn(fmaf(-shi, qd, wh), fmaf(-slo, qd, wl)), Rs);
    }
    Rs = wsum32(Rs);
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

// ------------------------------------------------------------------ kernel

template <int EPL, int NCH>
__global__ void __launch_bounds__(256) k_recon_int(const IntParams p)
{
    constexpr int G = EPL * kLanesPerGroup;
    constexpr int UNIT = kGroupsPerUnit * G;
    constexpr int NCHK = EPL / 4;  // 16-byte chunks per lane and group
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
    // Pass B accumulates codes centred on Hc = floor(qmax/2): subtracting the
    // rounding constant plus Hc (exact) yields q - Hc directly and keeps the
    // moment sums well conditioned.
    const float Hc = (float)(p.qmax >> 1);
    const float2 H2 = make_float2(H, H);
    const float2 magic2 = make_float2(kRoundMagic, kRoundMagic);
    const float2 nmagic_c2 = make_float2(-(kRoundMagic + Hc), -(kRoundMagic + Hc));
    const float ulp = 5.9604645e-8f * p.tie_kappa;
    const float2 beta22 = make_float2(p.beta2, p.beta2);
    const float2 c12 = make_float2(p.c1, p.c1);
    int s_cur = 0;
    uint32_t parity = 0;

    for (int64_t it = 0;; ++it) {
        const int64_t u = first + it * stride;
        if (u >= n_units) break;
        if (!mbar_wait_bounded(&bars[s_cur], parity, p.timeout_ns)) {
            fail(it);
            return;
        }
        unsigned char* st = ring + (size_t)s_cur * p.stage_bytes;
        const float* ws = reinterpret_cast<const float*>(st);
        float* hs = reinterpret_cast<float*>(st + kVOff);
        const unsigned char* gsm = st + kGOff;

        const int64_t grp = u * kGroupsPerUnit + gs;
        const bool valid = grp < p.n_groups;
        const int64_t gbase = grp * (int64_t)G;

        // ---- pass A: saliency EMA (h kept in the tile), range, saliency mass
        float mn = INFINITY, mx = -INFINITY, ss = 0.0f;
#pragma unroll
        for (int i = 0; i < NCHK; ++i) {
            const int e = gs * G + i * 32 + sl * 4;
            const float4 w4 = lds128(ws + e);
            float4 h4 = lds128(hs + e);
            if (p.g_kind) {
                float g0, g1, g2, g3;
                if (p.g_kind == 2) {
                    const uint2 gb = lds64(gsm + e * 2);
                    g0 = bf16lo(gb.x); g1 = bf16hi(gb.x); g2 = bf16lo(gb.y); g3 = bf16hi(gb.y);
                } else {
                    const float4 g4 = lds128(gsm + e * 4);
                    g0 = g4.x; g1 = g4.y; g2 = g4.z; g3 = g4.w;
                }
                const float2 gA = make_float2(g0, g1), gB = make_float2(g2, g3);
                const float2 hA = __ffma2_rn(make_float2(h4.x, h4.y), beta22,
                                             __fmul2_rn(c12, __fmul2_rn(gA, gA)));
                const float2 hB = __ffma2_rn(make_float2(h4.z, h4.w), beta22,
                                             __fmul2_rn(c12, __fmul2_rn(gB, gB)));
                h4 = make_float4(hA.x, hA.y, hB.x, hB.y);
                *reinterpret_cast<float4*>(hs + e) = h4;
                if (valid) stg_cs(reinterpret_cast<float4*>(p.v + gbase + i * 32 + sl * 4), h4);
            }
            mn = fminf(fminf(fminf(mn, w4.x), fminf(w4.y, w4.z)), w4.w);
            mx = fmaxf(fmaxf(fmaxf(mx, w4.x), fmaxf(w4.y, w4.z)), w4.w);
            ss += (h4.x + h4.y) + (h4.z + h4.w);
        }
#pragma unroll
        for (int o = 4; o; o >>= 1) {
            mn = fminf(mn, shx(mn, o));
            mx = fmaxf(mx, shx(mx, o));
            ss += shx(ss, o);
        }
        const bool h_one = ss == 0.0f;  // all saliencies zero: fit with h = 1
        if (h_one) ss = (float)G;
        const float range = mx - mn;
        const bool flat = !(range > 0.0f);
        const float c = 0.5f * (mn + mx);
        // approximate divisions (<= 2 ulp) are enough here: R scales the code
        // positions (margins are measured against the clipping range), and
        // the fit of the kept candidate is rechecked below
        const float R = flat ? 0.0f : __fdividef(qmaxf, range);
        const float inv_ss = __fdividef(1.0f, ss);
        const float2 nc2 = make_float2(-c, -c);

        // ---- pass B + reduction + fit, 8 candidates at a time
        float Ek[NCH], dEk[NCH], ak[NCH], bk[NCH], T1k[NCH], T2k[NCH], T3k[NCH];
        bool suspk[NCH];
        float sd = 0.0f, sdd = 0.0f;
#pragma unroll 1
        for (int ch = 0; ch < NCH; ++ch) {
            float2 P2[8];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const float P = R * p.invf[ch * 8 + kk];
                P2[kk] = make_float2(P, P);
            }
            float2 A1[8], A2[8], A3[8];
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) A1[kk] = A2[kk] = A3[kk] = make_float2(0.0f, 0.0f);
            float2 SD = make_float2(0.0f, 0.0f), SDD = make_float2(0.0f, 0.0f);
#pragma unroll 1
            for (int i = 0; i < NCHK; ++i) {
                const int e = gs * G + i * 32 + sl * 4;
                const float4 w4 = lds128(ws + e);
                const float4 h4 = h_one ? make_float4(1.0f, 1.0f, 1.0f, 1.0f) : lds128(hs + e);
                const float2 d[2] = {__fadd2_rn(make_float2(w4.x, w4.y), nc2),
                                     __fadd2_rn(make_float2(w4.z, w4.w), nc2)};
                const float2 h[2] = {make_float2(h4.x, h4.y), make_float2(h4.z, h4.w)};
                float2 hd[2];
#pragma unroll
                for (int pr = 0; pr < 2; ++pr) {
                    hd[pr] = __fmul2_rn(h[pr], d[pr]);
                    SD = __fadd2_rn(SD, hd[pr]);
                    SDD = __ffma2_rn(hd[pr], d[pr], SDD);
                }
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)
#pragma unroll
                    for (int pr = 0; pr < 2; ++pr) {
                        float2 t = __ffma2_rn(d[pr], P2[kk], H2);
                        t.x = fminf(fmaxf(t.x, 0.0f), qmaxf);
                        t.y = fminf(fmaxf(t.y, 0.0f), qmaxf);
                        const float2 q = __fadd2_rn(__fadd2_rn(t, magic2), nmagic_c2);  // q - Hc
                        const float2 hq = __fmul2_rn(h[pr], q);
                        A1[kk] = __fadd2_rn(A1[kk], hq);
                        A2[kk] = __ffma2_rn(hq, q, A2[kk]);
                        A3[kk] = __ffma2_rn(q, hd[pr], A3[kk]);
                    }
            }
            // transpose through shared memory: lane L writes row L, lane
            // (gs, sl) sums columns sl*4.. of the 8 rows of its group
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
                *reinterpret_cast<float4*>(red + lane * 36 + kk * 4) =
                    make_float4(A1[kk].x + A1[kk].y, A2[kk].x + A2[kk].y, A3[kk].x + A3[kk].y, 0.0f);
            __syncwarp();
            float3 T = make_float3(0.0f, 0.0f, 0.0f);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float4 x = *reinterpret_cast<const float4*>(red + (gs * 8 + j) * 36 + sl * 4);
                T.x += x.x;
                T.y += x.y;
                T.z += x.z;
            }
            __syncwarp();
            if (ch == 0) {
                sd = SD.x + SD.y;
                sdd = SDD.x + SDD.y;
#pragma unroll
                for (int o = 4; o; o >>= 1) {
                    sd += shx(sd, o);
                    sdd += shx(sdd, o);
                }
            }
            const float dbar = sd * inv_ss;
            const float habsd = sqrtf(ss * sdd);  // >= sum h |d| (Cauchy-Schwarz)
            const int k = ch * 8 + sl;
            const float qbar = T.x * inv_ss;  // mean of q - Hc
            const float D = T.y - T.x * qbar;
            const float N = T.z - T.x * dbar;
            const bool susp = !(D > 1e-3f * T.y);
            const float a = __fdividef(N, D);
            const float E = susp ? 0.0f : N * a;
            const float dN = ulp * qmaxf * habsd;
            const float dD = ulp * T.y;
            const bool real = k < p.n_clip;
#pragma unroll
            for (int cc = 0; cc < NCH; ++cc)
                if (cc == ch) {
                    Ek[cc] = real && !susp ? E : -INFINITY;
                    dEk[cc] = 2.0f * fabsf(a) * dN + a * a * dD;
                    ak[cc] = a;
                    bk[cc] = dbar - a * (qbar + Hc);
                    suspk[cc] = real && susp;
                    T1k[cc] = T.x;
                    T2k[cc] = T.y;
                    T3k[cc] = T.z;
                }
        }
        const float dbar = sd * inv_ss;

        // ---- argmax of E over the group (ties: lowest index)
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

        // winner's fit and sums, from its owner lane
        float a_sel = 0.0f, bc_sel = 0.0f, T1b = 0.0f, T2b = 0.0f, T3b = 0.0f;
        {
            const int owner = (gs * 8) | (kb & 7);
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) {
                const float av = __shfl_sync(0xffffffffu, ak[ch], owner);
                const float bv = __shfl_sync(0xffffffffu, bk[ch], owner);
                const float t1 = __shfl_sync(0xffffffffu, T1k[ch], owner);
                const float t2 = __shfl_sync(0xffffffffu, T2k[ch], owner);
                const float t3 = __shfl_sync(0xffffffffu, T3k[ch], owner);
                if ((kb >> 3) == ch) {
                    a_sel = av;
                    bc_sel = bv;
                    T1b = t1;
                    T2b = t2;
                    T3b = t3;
                }
            }
        }
        // Candidates needing an exact comparison: within the fp32 error bound
        // of the winner.  Those whose sums equal the winner's bit for bit
        // ("twins") almost always have the winner's codes -- equal codes give
        // equal errors, and the lower index is kept, as Algorithm 1's argmin
        // does -- but an element of tiny saliency can differ without moving the
        // sums, so twins are first checked code by code (cheaply, deferred).
        unsigned my_set = 0, my_twin = 0;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) {
            const int k = ch * 8 + sl;
            const bool twin = T1k[ch] == T1b && T2k[ch] == T2b && T3k[ch] == T3b;
            const bool contender = k != kb && Ek[ch] > -INFINITY && Eb - Ek[ch] <= dEb + dEk[ch];
            if (contender || suspk[ch]) my_set |= 1u << ch;
            if (contender && twin && !suspk[ch]) my_twin |= 1u << ch;
        }
        unsigned set = 0, twins = 0;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) {
            const unsigned bal = __ballot_sync(0xffffffffu, (my_set >> ch) & 1u);
            set |= ((bal >> (gs * 8)) & 0xFFu) << (ch * 8);
            const unsigned balt = __ballot_sync(0xffffffffu, (my_twin >> ch) & 1u);
            twins |= ((balt >> (gs * 8)) & 0xFFu) << (ch * 8);
        }
        if (Eb == -INFINITY) set = (p.n_clip >= 32) ? 0xFFFFFFFFu : ((1u << p.n_clip) - 1u);
        else if (set) set |= 1u << kb;

        float Bsel = bc_sel + c, a_lo = 0.0f, B_lo = 0.0f;
        float qbar_sel = T1b * inv_ss + Hc;
        bool deg_sel = false;

        // ---- deferred exact comparisons: the whole warp takes one group at a time
        unsigned todo = __ballot_sync(0xffffffffu, valid && !flat && set != 0 && sl == 0);
        if (todo) __syncwarp();  // h written by other lanes is read below
        while (todo) {
            const int g = (__ffs(todo) - 1) >> 3;
            todo &= todo - 1;
            const int src = g * 8;
            const float gc = __shfl_sync(0xffffffffu, c, src);
            const float grange = __shfl_sync(0xffffffffu, range, src);
            const float gR = __shfl_sync(0xffffffffu, R, src);
            const float gss = __shfl_sync(0xffffffffu, ss, src);
            const float gdbar = __shfl_sync(0xffffffffu, dbar, src);
            const bool gh_one = __shfl_sync(0xffffffffu, (int)h_one, src) != 0;
            unsigned gset = __shfl_sync(0xffffffffu, set, src);
            const unsigned gtwins = __shfl_sync(0xffffffffu, twins, src);
            const int gkb0 = __shfl_sync(0xffffffffu, kb, src);
            const float* gws = ws + g * G;
            const float* ghs = hs + g * G;
            unsigned tw = gtwins;
            while (tw) {
                const int k = __ffs(tw) - 1;
                tw &= tw - 1;
                if (coop_same_codes<G>(gws, gc, gR * p.invf[k], gR * p.invf[gkb0], H, qmaxf))
                    gset &= ~(1u << k);
            }
            if (gset == (1u << gkb0)) continue;  // only the winner left
            if (p.stats && lane == 0) atomicAdd(&p.stats[0], 1u);
            float best_h = 0.0f, best_l = 0.0f, ga = 0.0f, gB = 0.0f;
            int best_k = -1;
            bool gdeg = false;
            while (gset) {
                const int k = __ffs(gset) - 1;
                gset &= gset - 1;
                float eh, el, a_k, bc_k;
                bool deg_k;
                coop_exact<G>(gws, ghs, gh_one, gc, gR * p.invf[k], H, qmaxf, gss, gdbar,
                              p.f[k] * grange / qmaxf, &eh, &el, &a_k, &bc_k, &deg_k);
                if (best_k < 0 || ff_less(eh, el, best_h, best_l)) {
                    best_h = eh;
                    best_l = el;
                    best_k = k;
                    ga = a_k;
                    gB = bc_k + gc;
                    gdeg = deg_k;
                }
            }
            if (gs == g) {
                kb = best_k;
                a_sel = ga;
                Bsel = gB;
                deg_sel = gdeg;
                qbar_sel = -1.0f;  // recomputed by the refit below
            }
        }

        // ---- pass R: two-pass weighted least-squares fit (Eq. 4) of the kept
        // candidate, centred on a short approximation m of its weighted mean
        // code (q - m exact) and on the weighted mean weight; the offset is
        // assembled in compensated arithmetic and kept as a float pair.
        const float Pk = R * p.invf[kb];
        const bool refit = !flat && !deg_sel;
        float kap = 0.0f;
        {
            const float2 Pk2 = make_float2(Pk, Pk);
            float qm = qbar_sel;
            // winner changed in the exact pass: its mean code again (warp-uniform
            // branch, the reduction below shuffles across all lanes)
            if (__any_sync(0xffffffffu, qm < 0.0f)) {
                float s1 = 0.0f;
#pragma unroll 1
                for (int i = 0; i < NCHK; ++i) {
                    const int e = gs * G + i * 32 + sl * 4;
                    const float4 w4 = lds128(ws + e);
                    const float4 h4 = h_one ? make_float4(1.0f, 1.0f, 1.0f, 1.0f) : lds128(hs + e);
                    s1 = fmaf(h4.x, int_code(w4.x - c, Pk, H, qmaxf), s1);
                    s1 = fmaf(h4.y, int_code(w4.y - c, Pk, H, qmaxf), s1);
                    s1 = fmaf(h4.z, int_code(w4.z - c, Pk, H, qmaxf), s1);
                    s1 = fmaf(h4.w, int_code(w4.w - c, Pk, H, qmaxf), s1);
                }
#pragma unroll
                for (int o = 4; o; o >>= 1) s1 += shx(s1, o);
                if (qm < 0.0f) qm = s1 * inv_ss;
            }
            const float m = rintf(qm);  // integer: q - m is exact and magic + m too
            const float2 nm2 = make_float2(-(kRoundMagic + m), -(kRoundMagic + m));
            const float2 ndbar2 = make_float2(-dbar, -dbar);
            float2 D2 = make_float2(0.0f, 0.0f), N2 = D2, A2 = D2, B2s = D2, W2 = D2;
#pragma unroll 1
            for (int i = 0; i < NCHK; ++i) {
                const int e = gs * G + i * 32 + sl * 4;
                const float4 w4 = lds128(ws + e);
                const float4 h4 = h_one ? make_float4(1.0f, 1.0f, 1.0f, 1.0f) : lds128(hs + e);
#pragma unroll
                for (int pr = 0; pr < 2; ++pr) {
                    const float2 wv = pr ? make_float2(w4.z, w4.w) : make_float2(w4.x, w4.y);
                    const float2 hv = pr ? make_float2(h4.z, h4.w) : make_float2(h4.x, h4.y);
                    const float2 d = __fadd2_rn(wv, nc2);
                    float2 t = __ffma2_rn(d, Pk2, H2);
                    t.x = fminf(fmaxf(t.x, 0.0f), qmaxf);
                    t.y = fminf(fmaxf(t.y, 0.0f), qmaxf);
                    const float2 dq = __fadd2_rn(__fadd2_rn(t, magic2), nm2);  // q - m, exact
                    const float2 wd = __fadd2_rn(d, ndbar2);
                    const float2 hdq = __fmul2_rn(hv, dq);
                    D2 = __ffma2_rn(hdq, dq, D2);
                    N2 = __ffma2_rn(hdq, wd, N2);
                    A2 = __fadd2_rn(A2, hdq);
                    B2s = __ffma2_rn(hv, wd, B2s);
                    W2 = __ffma2_rn(__fmul2_rn(hv, wd), wd, W2);
                }
            }
            float Dr = D2.x + D2.y, Nr = N2.x + N2.y, Ar = A2.x + A2.y, Br = B2s.x + B2s.y;
            float Wr = W2.x + W2.y;
#pragma unroll
            for (int o = 4; o; o >>= 1) {
                Dr += shx(Dr, o);
                Nr += shx(Nr, o);
                Ar += shx(Ar, o);
                Br += shx(Br, o);
                Wr += shx(Wr, o);
            }
            if (refit) {
                const float Aq = Ar * inv_ss;  // mean of q - m
                const float Bw = Br * inv_ss;  // mean of d - dbar
                const float Nc = Nr - Ar * Bw, Dc = Dr - Ar * Aq;
                const float an = Nc / Dc;
                // b = (c + dbar + Bw) - a * (m + Aq), as a float pair
                float mu_h, mu_l, p_h, p_l, bh, bl;
                two_sum(c, dbar, mu_h, mu_l);
                two_prod(an, m, p_h, p_l);
                two_sum(mu_h, -p_h, bh, bl);
                bl = __fadd_rn(bl, __fsub_rn(__fadd_rn(mu_l, Bw), fmaf(an, Aq, p_l)));
                ff_norm(bh, bl);
                a_sel = an;
                Bsel = bh;
                B_lo = bl;
                // conditioning of the slope: rounding in the sums moves a by
                // about ulp * (sum |h dq wd| / |Nc| + sum h dq^2 / Dc), and
                // sum |h dq wd| <= sqrt(Dr Wr) (Cauchy-Schwarz)
                kap = __fdividef(sqrtf(Dr * Wr), fabsf(Nc)) + __fdividef(Dr, Dc);
            }
        }

        // ---- output accuracy check.  The refit's error at any level is at most
        // about est = fit_ulps * ulp * (|a| qmax kap + |c| + range) (fit_ulps
        // calibrated against the oracle with a margin).  The offset b (fp32)
        // and a level written in fp32 must meet tol(x) = 1e-7 + 1e-5|x|.  A
        // level written in bf16 is exact when no bf16 rounding midpoint lies
        // within est of it, and within the tolerance band when est <= tol.
        // Groups that could miss get the compensated (float-float) fit.
        bool prec;
        {
            const float est = p.fit_ulps * 5.9604645e-8f * (fabsf(a_sel) * qmaxf * kap + fabsf(c) + range);
            prec = est > 1e-7f + 1e-5f * fabsf(Bsel);
            if (!p.r_bf16) {
                const float q0 = fminf(fmaxf(rintf(__fdividef(-Bsel, a_sel)), 0.0f), qmaxf);
                const float rmin = fminf(fabsf(Bsel), fabsf(fmaf(a_sel, q0, Bsel)));
                prec |= est > 1e-7f + 1e-5f * rmin;
            } else {
                for (int q = sl; q <= p.qmax; q += kLanesPerGroup) {
                    const float rq = fmaf(a_sel, (float)q, Bsel);
                    if (est > 1e-7f + 1e-5f * fabsf(rq)) {
                        const uint32_t bits = __float_as_uint(rq);
                        const int dmid = abs((int)(bits & 0xFFFFu) - 0x8000);  // fp32 ulps to the midpoint
                        const float ulp32 =
                            __uint_as_float(max(bits & 0x7F800000u, 0x0C000000u) - 0x0B800000u);
                        prec |= (float)dmid * ulp32 < 1.5f * est;
                    }
                }
            }
            prec = prec || est != est;  // NaN sums: take the careful path
        }
        {
            // one decision per group: any lane of the segment that flagged
            const unsigned flag = __ballot_sync(0xffffffffu, prec);
            prec = ((flag >> (gs * kLanesPerGroup)) & 0xFFu) != 0;
        }
        todo = __ballot_sync(0xffffffffu, valid && refit && prec && sl == 0);
        if (todo) __syncwarp();
        while (todo) {
            const int g = (__ffs(todo) - 1) >> 3;
            todo &= todo - 1;
            const int src = g * 8;
            const float gc = __shfl_sync(0xffffffffu, c, src);
            const float gR = __shfl_sync(0xffffffffu, R, src);
            const float gss = __shfl_sync(0xffffffffu, ss, src);
            const float gdbar = __shfl_sync(0xffffffffu, dbar, src);
            const bool gh_one = __shfl_sync(0xffffffffu, (int)h_one, src) != 0;
            const int gkb = __shfl_sync(0xffffffffu, kb, src);
            if (p.stats && lane == 0) atomicAdd(&p.stats[1], 1u);
            float ga, ga_lo, gB, gB_lo;
            coop_precise<G>(ws + g * G, hs + g * G, gh_one, gc, gR * p.invf[gkb], H, qmaxf, gss,
                            gc + gdbar, &ga, &ga_lo, &gB, &gB_lo);
            if (gs == g) {
                a_sel = ga;
                a_lo = ga_lo;
                Bsel = gB;
                B_lo = gB_lo;
            }
        }

        // ---- pass C: outputs of the kept candidate
        if (valid) {
            const float Pb = R * p.invf[kb];
            const float2 Pb2 = make_float2(Pb, Pb);
            const float2 a2 = make_float2(a_sel, a_sel), B2 = make_float2(Bsel, Bsel);
            const float2 alo2 = make_float2(a_lo, a_lo), Blo2 = make_float2(B_lo, B_lo);
            const bool comp = a_lo != 0.0f || B_lo != 0.0f;
            const float2 nmagic2 = make_float2(-kRoundMagic, -kRoundMagic);
#pragma unroll 1
            for (int i = 0; i < NCHK; ++i) {
                const int e = gs * G + i * 32 + sl * 4;
                const float4 w4 = lds128(ws + e);
                float2 rv[2];
                uint32_t cw = 0;
#pragma unroll
                for (int pr = 0; pr < 2; ++pr) {
                    const float2 wv = pr ? make_float2(w4.z, w4.w) : make_float2(w4.x, w4.y);
                    float2 t = __ffma2_rn(__fadd2_rn(wv, nc2), Pb2, H2);
                    t.x = fminf(fmaxf(t.x, 0.0f), qmaxf);
                    t.y = fminf(fmaxf(t.y, 0.0f), qmaxf);
                    const float2 y = __fadd2_rn(t, magic2);
                    const float2 q = __fadd2_rn(y, nmagic2);
                    rv[pr] = __ffma2_rn(a2, q, B2);
                    // a_lo, B_lo are nonzero only where the compensated fit ran
                    if (comp) rv[pr] = __fadd2_rn(rv[pr], __ffma2_rn(alo2, q, Blo2));
                    if (flat) rv[pr] = wv;
                    if (p.codes)
                        cw |= ((__float_as_uint(y.x) & 0xFFu) | ((__float_as_uint(y.y) & 0xFFu) << 8))
                              << (16 * pr);
                }
                const int64_t eo = gbase + i * 32 + sl * 4;
                if (p.r_bf16) {
                    stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.r) + eo),
                           make_uint2(pack_bf16x2(rv[0].x, rv[0].y), pack_bf16x2(rv[1].x, rv[1].y)));
                } else {
                    stg_cs(reinterpret_cast<float4*>(static_cast<float*>(p.r) + eo),
                           make_float4(rv[0].x, rv[0].y, rv[1].x, rv[1].y));
                }
                if (p.codes) stg_cs(reinterpret_cast<uint32_t*>(p.codes + eo), flat ? 0u : cw);
            }
            if (sl == 0) {
                p.a[grp] = flat ? 0.0f : a_sel;
                p.b[grp] = flat ? ws[gs * G] : Bsel;
                if (p.idx) p.idx[grp] = flat ? 0 : (uint8_t)kb;
            }
        }

        // release the tile: all lanes are done with it; order our generic
        // writes to it before the async-proxy copy that refills it
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
