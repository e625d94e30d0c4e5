// QUASAR reconstruction with asymmetric integer codes (Algorithm 1; Eq. 1
// code assignment, Eq. 4 weighted least-squares dequantizer, Eq. 3 weighted
// error; saliency EMA of Sec. 4.1.1 / App. A.2), one fused pass over HBM.
//
// Work decomposition.  A "unit" is 8 consecutive groups; one warp owns a unit
// at a time, 4 lanes per group, EPL = G/4 elements per lane.  Lane sl of
// group gs holds the group's 16-byte chunks {i ^ swz : i < EPL/4} at element
// offset 4 sl within each 16-element span (swz a per-group XOR, so that the
// groups one shared-memory access phase covers hit different banks).  The
// CTA runs one ring of tile slots (one unit each) filled by 1-D TMA bulk
// copies (cp.async.bulk + mbarrier); each slot carries the sequence number of
// the unit loading into it, warp j takes the CTA's units j, j + warps, ...
// and, done with a tile, issues the copy of the unit that many slots ahead
// into the same slot.  w, g and v are read from HBM exactly once, and the
// loads of later units overlap the arithmetic of the current ones.  After
// pass A the tile's gradient region is the warp's transpose scratch.  The
// grid is persistent.
//
// Codes.  With d = (w - min) - rho (the offset from the group's centre,
// formed without rounding the centre itself: w - min and the half range are
// exact wherever the group lies far from zero), P = qmax / (f * range) and
// J = (qmax - 1)/2, Eq. 1's code is q = zeta + J + 1 with
//     zeta = clamp(floor(d P), -(J+1), J),
// which equals clamp(round(d P + qmax/2), 0, qmax) except at exact rounding
// ties (d P an integer), which lie inside the checker's margin exemption.
// floor is one FMA rounded toward -inf onto the unit grid at 1.5 * 2^23 (the
// product is exact inside the FMA), so y = M + zeta with M = 1.5 * 2^23.  The
// clamp is applied to d instead, once per set of candidates: for a set whose
// factors satisfy J f_max < tau < (J + 1) f_min (with a margin the host
// checks), clamping |d| at tau * range / qmax gives every candidate of the
// set its clamped code bit for bit (a set of one always has such a tau).
//
// Per group (fp32):
//   pass A  v' = beta2*v + (1-beta2)*g^2 (written back; kept in the tile as
//           the saliency h), min/max -> range, sum h, sum h w -> mu;
//   pass B  for the 8 candidates of a single chunk at once (4 at a time with
//           more chunks), the codes and the moments about a
//           centre zeta0 shared by the candidates of an 8-candidate chunk
//           (the code of the weighted mean, from mu): S1 = sum h (zeta -
//           zeta0), S2 = sum h (zeta - zeta0)^2, S3 = sum h (zeta - zeta0) e,
//           e = w - mu (plus the candidate-independent sum h e, sum h e^2);
//   reduce  the 4 lanes' partial sums are transposed through the scratch so
//           that lane sl owns candidate sl of each 4-candidate quad;
//   select  D = S2 - S1^2/Ss, N = S3 - S1*Se/Ss: the weighted error of
//           candidate k is C - N^2/D with C common, so argmin error =
//           argmax E = N^2/D; the winner's fit is a = N/D with the offset
//           from the weighted means, taken from the same centred sums;
//   pass C  codes of the kept candidate, r = a*zeta + B, outputs (b = B -
//           a*(J+1) is the offset of the paper's r = a*q + b).
//
// Exactness.  E carries fp32 rounding error; candidates whose E lies within
// an error bound of the best (and candidates whose weighted code variance D
// is too small to trust) are re-evaluated exactly, and fits whose fp32
// rounding could miss the output tolerance are recomputed in compensated
// (float-float) arithmetic.  Both are rare; they are deferred to the end of
// the unit's selection and done by the whole warp on one group at a time.
#pragma once

#include <type_traits>

#include "device_common.cuh"
#include "params.h"

namespace quasar {

__device__ __forceinline__ float shx(float x, int m) { return __shfl_xor_sync(0xffffffffu, x, m); }

// 1.5 * 2^23: in [2^23, 2^24) fp32 values are spaced 1, so fl_rd(x + M) =
// M + floor(x) for |x| < 2^22.
constexpr float kGridMagic = 12582912.0f;

// Offset of an element from its group's centre, d = (w - mn) - rho.
__device__ __forceinline__ float centred(float w, float nmn, float nrho)
{
    return __fadd_rn(__fadd_rn(w, nmn), nrho);
}

// Code q in [0, qmax] of an offset d for the scale P: M + floor(d P) clamped
// to [ylo, yhi] = [M - J - 1, M + J], minus ylo (exact).
__device__ __forceinline__ float int_code_q(float d, float P, float ylo, float yhi)
{
    return __fsub_rn(fminf(fmaxf(__fmaf_rd(d, P, kGridMagic), ylo), yhi), ylo);
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

__device__ __forceinline__ float wsum32(float x)
{
#pragma unroll
    for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// (hi, lo) + x*K as a renormalised pair: moves an offset between two code
// origins (q = 0 and zeta = 0, q = zeta + K).
__device__ __forceinline__ void ff_add_prod(float& hi, float& lo, float xh, float xl, float K)
{
    float ph, pl, sh, se;
    two_prod(xh, K, ph, pl);
    two_sum(hi, ph, sh, se);
    lo = __fadd_rn(__fadd_rn(lo, se), fmaf(xl, K, pl));
    hi = sh;
    ff_norm(hi, lo);
}

// ------------------------------------------------- whole-warp group helpers
//
// One group, evaluated by all 32 lanes (lane L takes elements L + 32m) from
// the tile in shared memory: w at ws, saliency h at hs.

// The code geometry of one group.
struct GroupGeom {
    float nmn, nrho;  // -min, -rho: d = (w - min) - rho
    float ylo, yhi;   // code clamp on the grid M + zeta
};

// True when candidates with scale factors Pa and Pb give the same codes on
// every element of the group (whole warp).
template <int G>
__device__ bool coop_same_codes(const float* ws, const GroupGeom& gq, float Pa, float Pb)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    bool same = true;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const float d = centred(ws[lane + 32 * m], gq.nmn, gq.nrho);
        same &= int_code_q(d, Pa, gq.ylo, gq.yhi) == int_code_q(d, Pb, gq.ylo, gq.yhi);
    }
    return __all_sync(0xffffffffu, same);
}

// The direct error sum h (a q + B - w)^2 of one candidate for the fit
// (a, bc), bc the offset at q = 0 of w - cref, with (a, B) rounded to a
// common power-of-two grid U so that a*q + B is exact and only "- w" rounds;
// lanes combine as a float pair.  Far from zero (|centre| >= 2 range) the
// residual is formed about an anchor A at the centre, a q + (B - A) - (w - A),
// with w - A exact: the grid then follows the group's range rather than its
// magnitude, and the rounded fit stays a tiny fraction of a level from the
// given one (the error's excess is second order in that distance).
template <int G>
__device__ void coop_error(const float* ws, const float* hs, const GroupGeom& gq, float P,
                           float Jp1, float cref, float a, float bc, float* err_hi, float* err_lo)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    const float range = -2.0f * gq.nrho;
    const float A = fabsf(cref) >= 2.0f * range ? cref : 0.0f;
    const float B = bc + (cref - A);  // offset at q = 0 of w - A
    const float mr = fmaxf(fabsf(B), fabsf(fmaf(a, 2.0f * Jp1, B))) + fabsf(a);
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
        const float h = hs[e];
        const float w = ws[e];
        const float q = int_code_q(centred(w, gq.nmn, gq.nrho), P, gq.ylo, gq.yhi);
        const float ev = fmaf(ag, q, Bg) - (w - A);
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
}

// Exact evaluation of one candidate: codes q, exact degenerate test (all
// weighted elements on one code), two-pass centred fit, and the direct error
// sum h (a q + B - w)^2 with (a, B) rounded to a common power-of-two grid U
// so that a*q + B is exact and only "- w" rounds; lanes combine as a float
// pair (coop_error).  dbar is the weighted mean of w - cref.  Returns the fit
// as (a, Bz) with r = a zeta + Bz (offset at zeta = 0, i.e. q = J + 1), and a
// condition estimate kap of the slope (see the tier-2 trigger in the kernel).
template <int G>
__device__ void coop_exact(const float* ws, const float* hs, const GroupGeom& gq, float P,
                           float Jp1, float Ss, float dbar, float step, float cref, float* err_hi,
                           float* err_lo, float* a_out, float* Bz_out, float* kap_out,
                           bool* degenerate)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    float s1 = 0.0f;
    int qlo = 1 << 30, qhi = -1;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = hs[e];
        const float q = int_code_q(centred(ws[e], gq.nmn, gq.nrho), P, gq.ylo, gq.yhi);
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
    float a, bc, kap = 1.0f;
    if (qlo == qhi) {
        a = step;  // every weighted element shares one code
        bc = dbar - step * (float)qlo;
    } else {
        float dd = 0.0f, nn = 0.0f, ww = 0.0f;
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const int e = lane + 32 * m;
            const float h = hs[e];
            const float w = ws[e];
            const float dq = int_code_q(centred(w, gq.nmn, gq.nrho), P, gq.ylo, gq.yhi) - qbar;
            const float hdq = h * dq;
            const float wd = (w - cref) - dbar;
            dd = fmaf(hdq, dq, dd);
            nn = fmaf(hdq, wd, nn);
            ww = fmaf(h * wd, wd, ww);
        }
        dd = wsum32(dd);
        nn = wsum32(nn);
        ww = wsum32(ww);
        a = nn / dd;
        bc = dbar - a * qbar;
        kap = sqrtf(dd * ww) / fabsf(nn) + 1.0f;
    }
    coop_error<G>(ws, hs, gq, P, Jp1, cref, a, bc, err_hi, err_lo);
    *a_out = a;
    *Bz_out = fmaf(a, Jp1, bc + cref);
    *kap_out = kap;
}

// Weighted least-squares fit (Eq. 4) of one candidate in compensated
// arithmetic, for groups whose fp32 fit could miss the output tolerance
// (large weights with an offset or a level near zero, or badly conditioned
// code variance).  Centres: mq = the weighted mean code rounded to 1/16 (so
// q - mq and (q - mq)^2 are exact) and mu ~ the weighted mean weight (w - mu
// kept as an exact pair).  The sums of h (q-mq)^2 and h (q-mq)(w-mu) are
// accumulated and combined across lanes as float pairs (no fp64: its rate on
// this part is a small fraction of fp32's); the offset is
// mu - s*mq + mean_h(w - mu - s (q - mq)).  Returns the fit as float pairs,
// with the offset Bz at the code origin zeta = 0 (q = J + 1, r = a zeta + Bz).
template <int G>
__device__ void coop_precise(const float* ws, const float* hs, const GroupGeom& gq, float P,
                             float Jp1, float Ss, float mu, float* a_hi, float* a_lo,
                             float* Bz_hi, float* Bz_lo)
{
    constexpr int M = G / 32;
    const int lane = threadIdx.x & 31;
    float s1 = 0.0f;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        s1 = fmaf(hs[e], int_code_q(centred(ws[e], gq.nmn, gq.nrho), P, gq.ylo, gq.yhi), s1);
    }
    const float mq = rintf(wsum32(s1) / Ss * 16.0f) * 0.0625f;

    float Dh = 0.0f, Dl = 0.0f, Nh = 0.0f, Nl = 0.0f, A = 0.0f, B = 0.0f;
#pragma unroll
    for (int m = 0; m < M; ++m) {
        const int e = lane + 32 * m;
        const float h = hs[e];
        const float w = ws[e];
        const float qd = int_code_q(centred(w, gq.nmn, gq.nrho), P, gq.ylo, gq.yhi) - mq;
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
        const float h = hs[e];
        const float w = ws[e];
        const float qd = int_code_q(centred(w, gq.nmn, gq.nrho), P, gq.ylo, gq.yhi) - mq;
        float wh, wl;
        two_sum(w, -mu, wh, wl);
        Rs = fmaf(h, __fadd_rn(fmaf(-shi, qd, wh), fmaf(-slo, qd, wl)), Rs);
    }
    Rs = wsum32(Rs);
    // offset at the code origin zeta = 0, i.e. q = J + 1: mu + s*(J + 1 - mq)
    // + mean residual
    float ph, pl, zh, zl;
    two_prod(shi, Jp1 - mq, ph, pl);  // J + 1 - mq is exact (both multiples of 1/16)
    pl = fmaf(slo, Jp1 - mq, pl);
    two_sum(mu, ph, zh, zl);
    zl = __fadd_rn(__fadd_rn(zl, pl), Rs / Ss);
    ff_norm(zh, zl);
    *a_hi = shi;
    *a_lo = slo;
    *Bz_hi = zh;
    *Bz_lo = zl;
}

// ------------------------------------------------------------------ kernel

// Wait until the tile of sequence number t is the one in flight into a slot
// (its sequence word, written before the copy is issued), or until limit_ns
// has passed; the same outcome for every lane of the warp.
__device__ __forceinline__ bool warp_wait_seq(const volatile int* seq, int t, uint64_t limit_ns)
{
    bool ok = *seq == t;
    if (!__all_sync(0xffffffffu, ok)) {
        const uint64_t t0 = global_timer_ns();
        for (;;) {
#pragma unroll 1
            for (int i = 0; i < 32 && !ok; ++i) ok = *seq == t;
            if (ok || global_timer_ns() - t0 > limit_ns) break;
        }
        ok = __all_sync(0xffffffffu, ok);
    }
    return ok;
}

// Two CTAs per SM: 8-warp CTAs, 6-warp ones for the AdamW-fused variant.
// VAR: the variants of the options (a saliency other than v', packed codes);
// without it they compile out of the common kernel.
// SS: candidates per clamp set (4, 2 or 1; with a single chunk also 8, or 3:
// the sets 0-2, 3-5 and 6-7): the host picks the largest size whose sets all
// admit a cap (see the header comment); every size gives the same codes.
template <int EPL, int NCH, int MAXT, bool ADAM, bool VAR, int SS>
__global__ void __launch_bounds__(ADAM ? 192 : 256, 2)
    k_recon_int(const __grid_constant__ IntLaunch<MAXT> Lp)
{
    static_assert(SS == 1 || SS == 2 || SS == 4 || ((SS == 3 || SS == 8) && NCH == 1),
                  "clamp sets of 1, 2 or 4 candidates, or of 8 or 3-3-2 in a single chunk");
    // candidates a sweep of pass B over the tile: all 8 of the chunk with
    // one chunk (the loads, offsets and loop shared by 8), a quad with more
    // (whose other live state leaves no room for 8 sets of sums)
    constexpr int QW = NCH == 1 ? 8 : 4;
    // clamp sets a sweep, and the set of the sweep's candidate kk (its first
    // slot is kq + set * SS)
    constexpr int NSETS = SS == 3 ? 3 : QW / SS;
    auto set_of = [](int kk) { return SS == 3 ? (kk < 3 ? 0 : (kk < 6 ? 1 : 2)) : kk / SS; };
    const IntParams& p = Lp.p;
    constexpr int G = EPL * kIntLanes;
    constexpr int UNIT = kIntGroups * G;
    constexpr int NCHK = EPL / 4;  // 16-byte chunks per lane and group
    // chunk i of a lane is the group's chunk i ^ (gs & SWZ): the two (or
    // four) groups a shared-memory access phase covers then hit different
    // banks
    constexpr int SWZ = NCHK >= 4 ? 3 : (NCHK >= 2 ? 1 : 0);
    extern __shared__ __align__(128) unsigned char smem[];

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    const int gs = lane >> 2;
    const int sl = lane & 3;
    const int swz = gs & SWZ;

    // the CTA's ring: S tile slots, a full barrier each (and one spare for
    // the failure hook), and the sequence number of the tile each slot is
    // loading or holding
    const int S = p.stages;
    unsigned char* ring = smem;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)S * p.stage_bytes);
    volatile int* seq = reinterpret_cast<volatile int*>(bars + S + 1);

    const int gbytes = p.g_kind == 2 ? 2 : (p.g_kind == 1 ? 4 : 0);
    // stage: w | v | m (fused AdamW only) | g, then the transpose scratch
    constexpr uint32_t kVOff = UNIT * 4;
    constexpr uint32_t kMOff = UNIT * 8;
    constexpr uint32_t kGOff = UNIT * (ADAM ? 12 : 8);

    // tiles: the CTA takes units blockIdx.x + t * gridDim.x, t = 0 .. nt-1,
    // and warp w the tiles t = w, w + nwarps, ...; tile t goes to slot t % S
    const int64_t n_units = Lp.n_units;
    const int nt = n_units > (int64_t)blockIdx.x
                       ? (int)((n_units - 1 - (int64_t)blockIdx.x) / gridDim.x + 1)
                       : 0;
    auto unit_of = [&](int t) { return (int64_t)blockIdx.x + (int64_t)t * gridDim.x; };
    // the tensor of a unit: units are numbered consecutively across the
    // launch's tensors, and each warp meets them in increasing order
    auto tensor_of = [&](int64_t u, int& ti) {
        while (ti + 1 < Lp.n_t && u >= Lp.t[ti + 1].unit0) ++ti;
    };
    int ti = 0;

    // (the unit issued is after the one being processed, or the first ones:
    // its tensor index is found from ti onwards)
    auto issue = [&](int t, int s) {
        const int64_t u = unit_of(t);
        int tj = ti;
        tensor_of(u, tj);
        const IntTensor& T = Lp.t[tj];
        const int64_t g0 = (u - T.unit0) * kIntGroups;
        const int64_t ng = min((int64_t)kIntGroups, T.n_groups - g0);
        const uint32_t elems = (uint32_t)(ng * G);
        unsigned char* st = ring + (size_t)s * p.stage_bytes;
        seq[s] = t;
        mbar_arrive_expect_tx(&bars[s], elems * ((ADAM ? 12u : 8u) + (uint32_t)gbytes));
        bulk_g2s(st, T.w + g0 * G, elems * 4u, &bars[s]);
        bulk_g2s(st + kVOff, T.v + g0 * G, elems * 4u, &bars[s]);
        if constexpr (ADAM) bulk_g2s(st + kMOff, T.m + g0 * G, elems * 4u, &bars[s]);
        if (gbytes)
            bulk_g2s(st + kGOff, static_cast<const unsigned char*>(T.g) + g0 * G * gbytes,
                     elems * (uint32_t)gbytes, &bars[s]);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s <= S; ++s) mbar_init(&bars[s], 1);
        for (int s = 0; s < S; ++s) seq[s] = -1;
        mbar_init_fence();
        for (int s = 0; s < S && s < nt; ++s) issue(s, s);
    }
    __syncthreads();

    // Record the failure and wait (bounded) until every tile issued into
    // the ring has landed, then leave.  (A copy that never lands is given up
    // on, and the CTA then exits with it still in flight.)
    auto fail = [&]() {
        if (lane == 0) record_timeout(p.status);
        for (int s = 0; s < S; ++s) {
            const int ts = seq[s];
            if (ts >= 0) mbar_wait_bounded(&bars[s], (uint32_t)((ts / S) & 1), p.timeout_ns);
        }
    };

    if constexpr (SS > 1)  // which kernel ran, for the tuning counters
        if (p.stats && threadIdx.x == 0) atomicAdd(&p.stats[3], 1u);

    if (p.force_timeout_ns && blockIdx.x == 0 && warp == 0) {
        // Failure-path hook: a barrier nothing ever arrives on.
        if (!warp_wait_bounded(&bars[S], 0, p.force_timeout_ns)) {
            fail();
            return;
        }
    }

    const float qmaxf = (float)p.qmax;
    const int J = p.qmax >> 1;
    const float Jp1 = (float)(J + 1);
    const float ylo = kGridMagic - Jp1, yhi = kGridMagic + (float)J;
    const float2 Mg2 = make_float2(kGridMagic, kGridMagic);
    const float2 nMg2 = make_float2(-kGridMagic, -kGridMagic);
    const float ulp = 5.9604645e-8f * p.tie_kappa;
    const float2 beta22 = make_float2(p.beta2, p.beta2);
    const float2 c12 = make_float2(p.c1, p.c1);
    const float2 beta12 = make_float2(p.beta1, p.beta1), c1b2 = make_float2(p.c1b, p.c1b);
    const float2 nlrwd2 = make_float2(-p.lr_wd, -p.lr_wd);
    const float2 nstep2 = make_float2(-p.step_size, -p.step_size);
    const float2 isbc22 = make_float2(p.isbc2, p.isbc2), eps2 = make_float2(p.eps, p.eps);
    const unsigned gmask = 0xFu << (gs * kIntLanes);  // this group's lanes

    int slot = warp;  // t % S (nwarps < S)
    uint32_t parity = 0;  // (t / S) & 1
    for (int t = warp; t < nt; t += nwarps) {
        if (!warp_wait_seq(seq + slot, t, p.timeout_ns) ||
            !warp_wait_bounded(&bars[slot], parity, p.timeout_ns)) {
            fail();
            return;
        }
        const int64_t u = unit_of(t);
        unsigned char* st = ring + (size_t)slot * p.stage_bytes;
        float* ws = reinterpret_cast<float*>(st);
        float* hs = reinterpret_cast<float*>(st + kVOff);
        const unsigned char* gsm = st + kGOff;
        // transpose scratch (the gradient region, free once pass A is done)
        float* red = reinterpret_cast<float*>(st + kGOff);

        tensor_of(u, ti);
        const IntTensor& T = Lp.t[ti];
        const int64_t grp = (u - T.unit0) * kIntGroups + gs;
        const bool valid = grp < T.n_groups;
        const int64_t gbase = grp * (int64_t)G;
        const float* gws = ws + gs * G;  // this lane's group in the tile
        float* ghs = hs + gs * G;
        auto eoff = [&](int i) { return 16 * (i ^ swz) + 4 * sl; };  // chunk i of this lane

        // ---- pass A: saliency EMA (h kept in the tile), range, saliency mass
        // and weighted sum of w (a centre for the moments).  The fused variant
        // first takes one AdamW step and keeps w' in the tile, so everything
        // after this pass reconstructs the updated weights.
        float mn = INFINITY, mx = -INFINITY, ss = 0.0f, sw = 0.0f;
        {
            float* vout = T.v + gbase;
            float* wout = const_cast<float*>(T.w) + gbase;
            float* mout = T.m + gbase;
            auto pass_a = [&](auto gk) {
                constexpr int GK = decltype(gk)::value;
                float2 SS2 = make_float2(0.0f, 0.0f), SW = SS2;
// two chunks an iteration: the loop stays small in the instruction cache
#pragma unroll 2
                for (int i = 0; i < NCHK; ++i) {
                    const int eo = eoff(i);
                    const int e = gs * G + eo;
                    float4 w4 = lds128(ws + e);
                    float4 h4 = lds128(hs + e);
                    if constexpr (ADAM) {
                        float2 gv[2];
                        if constexpr (GK == 2) {
                            const uint2 gb = lds64(gsm + e * 2);
                            gv[0] = make_float2(bf16lo(gb.x), bf16hi(gb.x));
                            gv[1] = make_float2(bf16lo(gb.y), bf16hi(gb.y));
                        } else {
                            const float4 g4 = lds128(gsm + e * 4);
                            gv[0] = make_float2(g4.x, g4.y);
                            gv[1] = make_float2(g4.z, g4.w);
                        }
                        const float4 m4 = lds128(reinterpret_cast<const float*>(st + kMOff) + e);
                        float2 wv[2] = {make_float2(w4.x, w4.y), make_float2(w4.z, w4.w)};
                        float2 mv[2] = {make_float2(m4.x, m4.y), make_float2(m4.z, m4.w)};
                        float2 hv[2] = {make_float2(h4.x, h4.y), make_float2(h4.z, h4.w)};
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr) {
                            mv[pr] = __ffma2_rn(mv[pr], beta12, __fmul2_rn(c1b2, gv[pr]));
                            hv[pr] = __ffma2_rn(hv[pr], beta22,
                                                __fmul2_rn(c12, __fmul2_rn(gv[pr], gv[pr])));
                            // sqrt(v') as v' * rsqrt(v') (v' = 0 gives 0) and the
                            // quotient by the fast reciprocal: each within 2 ulps,
                            // small beside the ulp of w that w' is rounded to
                            float2 sq = __fmul2_rn(hv[pr], make_float2(rsqrtf(hv[pr].x),
                                                                       rsqrtf(hv[pr].y)));
                            sq.x = hv[pr].x > 0.0f ? sq.x : 0.0f;
                            sq.y = hv[pr].y > 0.0f ? sq.y : 0.0f;
                            const float2 den = __ffma2_rn(sq, isbc22, eps2);
                            const float2 upd = make_float2(__fdividef(mv[pr].x, den.x),
                                                           __fdividef(mv[pr].y, den.y));
                            // the decrement is formed first and added once, so
                            // w' is w + t rounded a single time
                            const float2 t2 = __ffma2_rn(wv[pr], nlrwd2, __fmul2_rn(nstep2, upd));
                            wv[pr] = __fadd2_rn(wv[pr], t2);
                        }
                        w4 = make_float4(wv[0].x, wv[0].y, wv[1].x, wv[1].y);
                        h4 = make_float4(hv[0].x, hv[0].y, hv[1].x, hv[1].y);
                        *reinterpret_cast<float4*>(ws + e) = w4;
                        *reinterpret_cast<float4*>(hs + e) = h4;
                        if (valid) {
                            stg_cs(reinterpret_cast<float4*>(wout + eo), w4);
                            stg_cs(reinterpret_cast<float4*>(mout + eo),
                                   make_float4(mv[0].x, mv[0].y, mv[1].x, mv[1].y));
                            stg_cs(reinterpret_cast<float4*>(vout + eo), h4);
                        }
                    } else if constexpr (GK != 0) {
                        float2 gA, gB;
                        if constexpr (GK == 2) {
                            const uint2 gb = lds64(gsm + e * 2);
                            gA = make_float2(bf16lo(gb.x), bf16hi(gb.x));
                            gB = make_float2(bf16lo(gb.y), bf16hi(gb.y));
                        } else {
                            const float4 g4 = lds128(gsm + e * 4);
                            gA = make_float2(g4.x, g4.y);
                            gB = make_float2(g4.z, g4.w);
                        }
                        const float2 hA = __ffma2_rn(make_float2(h4.x, h4.y), beta22,
                                                     __fmul2_rn(c12, __fmul2_rn(gA, gA)));
                        const float2 hB = __ffma2_rn(make_float2(h4.z, h4.w), beta22,
                                                     __fmul2_rn(c12, __fmul2_rn(gB, gB)));
                        h4 = make_float4(hA.x, hA.y, hB.x, hB.y);
                        *reinterpret_cast<float4*>(hs + e) = h4;
                        if (valid) stg_cs(reinterpret_cast<float4*>(vout + eo), h4);
                    }
                    mn = fmin3(fmin3(mn, w4.x, w4.y), w4.z, w4.w);
                    mx = fmax3(fmax3(mx, w4.x, w4.y), w4.z, w4.w);
                    const float2 hA = make_float2(h4.x, h4.y), hB = make_float2(h4.z, h4.w);
                    SS2 = __fadd2_rn(SS2, __fadd2_rn(hA, hB));
                    SW = __ffma2_rn(hA, make_float2(w4.x, w4.y), SW);
                    SW = __ffma2_rn(hB, make_float2(w4.z, w4.w), SW);
                }
                ss = SS2.x + SS2.y;
                sw = SW.x + SW.y;
            };
            if (p.g_kind == 2) pass_a(std::integral_constant<int, 2>{});
            else if (ADAM || p.g_kind == 1) pass_a(std::integral_constant<int, 1>{});
            else pass_a(std::integral_constant<int, 0>{});
            if (VAR && p.h_mode != kSalEma) {
                // the fit's saliency is v'^2 or 1: rewrite h in the tile (v'
                // went out already) and take its sums again
                float2 SS2 = make_float2(0.0f, 0.0f), SW = SS2;
#pragma unroll 1
                for (int i = 0; i < NCHK; ++i) {
                    const int e = gs * G + eoff(i);
                    const float4 w4 = lds128(ws + e);
                    float4 h4 = lds128(hs + e);
                    h4 = p.h_mode == kSalEmaSquared
                             ? make_float4(h4.x * h4.x, h4.y * h4.y, h4.z * h4.z, h4.w * h4.w)
                             : make_float4(1.0f, 1.0f, 1.0f, 1.0f);
                    *reinterpret_cast<float4*>(hs + e) = h4;
                    const float2 hA = make_float2(h4.x, h4.y), hB = make_float2(h4.z, h4.w);
                    SS2 = __fadd2_rn(SS2, __fadd2_rn(hA, hB));
                    SW = __ffma2_rn(hA, make_float2(w4.x, w4.y), SW);
                    SW = __ffma2_rn(hB, make_float2(w4.z, w4.w), SW);
                }
                ss = SS2.x + SS2.y;
                sw = SW.x + SW.y;
            }
        }
#pragma unroll
        for (int o = 2; o; o >>= 1) {
            mn = fminf(mn, shx(mn, o));
            mx = fmaxf(mx, shx(mx, o));
            ss += shx(ss, o);
            sw += shx(sw, o);
        }
        // all saliencies zero: the group is fitted with h = 1 (the tile's h
        // is overwritten; v' has been written out already)
        const bool h_one = ss == 0.0f;
        if (__any_sync(0xffffffffu, h_one)) {
            if (h_one)
#pragma unroll
                for (int i = 0; i < NCHK; ++i)
                    *reinterpret_cast<float4*>(ghs + eoff(i)) = make_float4(1.0f, 1.0f, 1.0f, 1.0f);
        }
        // a sum of saliencies near the bottom of the fp32 range: h scaled by
        // a power of two in the tile, and its sums taken again
        const bool h_tiny = !h_one && ss < kTinySaliency;
        if (__any_sync(0xffffffffu, h_tiny)) {
            float s1 = 1.0f, s2 = 1.0f;
            tiny_scale(ss, s1, s2);
            float2 SS2 = make_float2(0.0f, 0.0f), SW = SS2;
            if (h_tiny) {
#pragma unroll 1
                for (int i = 0; i < NCHK; ++i) {
                    const float4 w4 = lds128(gws + eoff(i));
                    float4 h4 = lds128(ghs + eoff(i));
                    h4 = make_float4(h4.x * s1 * s2, h4.y * s1 * s2, h4.z * s1 * s2, h4.w * s1 * s2);
                    *reinterpret_cast<float4*>(ghs + eoff(i)) = h4;
                    const float2 hA = make_float2(h4.x, h4.y), hB = make_float2(h4.z, h4.w);
                    SS2 = __fadd2_rn(SS2, __fadd2_rn(hA, hB));
                    SW = __ffma2_rn(hA, make_float2(w4.x, w4.y), SW);
                    SW = __ffma2_rn(hB, make_float2(w4.z, w4.w), SW);
                }
            }
            float ss2 = SS2.x + SS2.y, sw2 = SW.x + SW.y;
#pragma unroll
            for (int o = 2; o; o >>= 1) {
                ss2 += shx(ss2, o);
                sw2 += shx(sw2, o);
            }
            if (h_tiny) {
                ss = ss2;
                sw = sw2;
            }
        }
        // the gradient region becomes the transpose scratch: every lane is
        // past pass A, and the h rewrites above are visible to all lanes
        __syncwarp();
        const float range = mx - mn;
        const bool flat = !(range > 0.0f);
        const float rho = 0.5f * range;
        GroupGeom gq;
        gq.nmn = -mn;
        gq.nrho = -rho;
        gq.ylo = ylo;
        gq.yhi = yhi;
        const float cref = mn + rho;  // the centre, rounded (an anchor only)
        if (h_one) ss = (float)G;
        const float inv_ss = __fdividef(1.0f, ss);
        // mu: approximate weighted mean of w (only a centre for the sums)
        const float mu = h_one ? cref : sw * inv_ss;
        // approximate divisions (<= 2 ulp) are enough here: R scales the code
        // positions (margins are measured against the clipping range), and
        // the accuracy of the kept fit is checked below
        const float R = flat ? 0.0f : __fdividef(qmaxf, range);
        const float2 nmn2 = make_float2(-mn, -mn), nrho2 = make_float2(-rho, -rho);
        const float2 nmu2 = make_float2(-mu, -mu);
        // the weighted mean's offset from the centre, for the chunks' centres
        const float dmu = centred(mu, -mn, -rho);

        // ---- pass B + reduction + candidate errors, 8 candidates a chunk,
        // QW a sweep over the tile.  Codes from d = (w - mn) - rho; moments
        // about the chunk's centre code zeta0 and, for S3, e = w - mu.  Lane
        // sl owns candidates 8 ch + 4 qd + sl.
        float Ek[NCH][2], dEk[NCH][2], T1k[NCH][2], T2k[NCH][2], T3k[NCH][2], Y0k[NCH];
        bool suspk[NCH][2];
        float se = 0.0f, see = 0.0f;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch) {
            // centre: the code of the weighted mean for the chunk's mean 1/f
            const float y0 = fminf(fmaxf(__fmaf_rd(dmu, R * p.invfc[ch], kGridMagic), ylo), yhi);
            const float2 nY02 = make_float2(-y0, -y0);
            Y0k[ch] = y0;
            float2 SE = make_float2(0.0f, 0.0f), SEE = make_float2(0.0f, 0.0f);
            float4 xq[2];
#pragma unroll
            for (int sw = 0; sw < 8 / QW; ++sw) {
                const int kq = ch * 8 + sw * QW;
                float2 A1[QW], A2[QW], A3[QW];
#pragma unroll
                for (int kk = 0; kk < QW; ++kk) A1[kk] = A2[kk] = A3[kk] = make_float2(0.0f, 0.0f);
                if ((ch == 0 && sw == 0) || kq < p.n_clip) {
                    float2 P2[QW];
#pragma unroll
                    for (int kk = 0; kk < QW; ++kk) {
                        const float P = R * p.invf[kq + kk];
                        P2[kk] = make_float2(P, P);
                    }
                    float cp[NSETS];
#pragma unroll
                    for (int s = 0; s < NSETS; ++s) cp[s] = p.cap[kq + s * SS] * range;
// rolled: a compact unit loop keeps the careful paths' code from evicting it
// from the instruction cache when they run
#pragma unroll 1
                    for (int i = 0; i < NCHK; ++i) {
                        const int e = eoff(i);
                        const float4 w4 = lds128(gws + e);
                        const float4 h4 = lds128(ghs + e);
#pragma unroll
                        for (int pr = 0; pr < 2; ++pr) {
                            const float2 wv = pr ? make_float2(w4.z, w4.w) : make_float2(w4.x, w4.y);
                            const float2 h = pr ? make_float2(h4.z, h4.w) : make_float2(h4.x, h4.y);
                            const float2 d = __fadd2_rn(__fadd2_rn(wv, nmn2), nrho2);
                            const float2 ev = __fadd2_rn(wv, nmu2);
                            if (ch == 0 && sw == 0) {
                                const float2 he = __fmul2_rn(h, ev);
                                SE = __fadd2_rn(SE, he);
                                SEE = __ffma2_rn(he, ev, SEE);
                            }
                            float2 dc[NSETS];
#pragma unroll
                            for (int s = 0; s < NSETS; ++s)
                                dc[s] = make_float2(fminf(fmaxf(d.x, -cp[s]), cp[s]),
                                                    fminf(fmaxf(d.y, -cp[s]), cp[s]));
#pragma unroll
                            for (int kk = 0; kk < QW; ++kk) {
                                const float2 y = __ffma2_rd(dc[set_of(kk)], P2[kk], Mg2);
                                const float2 zc = __fadd2_rn(y, nY02);  // zeta - zeta0, exact
                                const float2 t2 = __fmul2_rn(h, zc);
                                A1[kk] = __ffma2_rn(h, zc, A1[kk]);
                                A2[kk] = __ffma2_rn(t2, zc, A2[kk]);
                                A3[kk] = __ffma2_rn(t2, ev, A3[kk]);
                            }
                        }
                    }
                }
                // transpose each quad through the scratch: lane L writes row L
                // (its sums of candidate kk in 16-byte column kk ^ ((L >> 1) &
                // 3)), and lane (gs, sl) sums column sl of its group's 4 rows
                // (each group starting at another row, so that an access
                // phase's two groups read rows of both parities: no bank
                // conflicts)
#pragma unroll
                for (int q4 = 0; q4 < QW / 4; ++q4) {
                    __syncwarp();
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const int c = q4 * 4 + kk;
                        *reinterpret_cast<float4*>(red + lane * 16 + ((kk ^ ((lane >> 1) & 3)) << 2)) =
                            make_float4(A1[c].x + A1[c].y, A2[c].x + A2[c].y, A3[c].x + A3[c].y, 0.0f);
                    }
                    __syncwarp();
                    float4 x[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int row = gs * 4 + ((j + gs) & 3);
                        x[j] = *reinterpret_cast<const float4*>(red + row * 16 + ((sl ^ ((row >> 1) & 3)) << 2));
                    }
                    xq[sw * (QW / 4) + q4] = make_float4((x[0].x + x[1].x) + (x[2].x + x[3].x),
                                                         (x[0].y + x[1].y) + (x[2].y + x[3].y),
                                                         (x[0].z + x[1].z) + (x[2].z + x[3].z), 0.0f);
                }
            }
            if (ch == 0) {
                se = SE.x + SE.y;
                see = SEE.x + SEE.y;
#pragma unroll
                for (int o = 2; o; o >>= 1) {
                    se += shx(se, o);
                    see += shx(see, o);
                }
            }
            // candidates 8 ch + 4 qd + sl: E = N^2/D and a bound dE on its fp32
            // error.  The sums are accumulated over tie_kappa levels at most,
            // so each is within tie_kappa ulps of the sum of its terms'
            // magnitudes: sum h zc^2 = S2, sum |h zc e| <= sqrt(S2 * sum h e^2).
            const float ebar = se * inv_ss;
#pragma unroll
            for (int qd = 0; qd < 2; ++qd) {
                const float T1 = xq[qd].x, T2 = xq[qd].y, T3 = xq[qd].z;
                const float zbar = T1 * inv_ss;
                const float D = T2 - T1 * zbar;
                const float N = T3 - T1 * ebar;
                const float a = __fdividef(N, D);
                // a near-degenerate code variance, or a non-finite E (sums
                // near the denormal range): left to the exact comparison
                const bool susp = !(D > 1e-3f * T2) || !(N * a < INFINITY);
                const float E = susp ? 0.0f : N * a;
                const float s2e = fmaxf(T2 * see, 1e-37f);
                const float dN = ulp * (s2e * rsqrtf(s2e) * 1.001f + fabsf(T1 * ebar));
                const float dD = ulp * (T2 + fabsf(T1 * zbar));
                const bool real = ch * 8 + qd * 4 + sl < p.n_clip;
                Ek[ch][qd] = real && !susp ? E : -INFINITY;
                dEk[ch][qd] = 2.0f * fabsf(a) * dN + a * a * dD;
                suspk[ch][qd] = real && susp;
                T1k[ch][qd] = T1;
                T2k[ch][qd] = T2;
                T3k[ch][qd] = T3;
            }
        }
        const float ebar = se * inv_ss;

        // ---- argmax of E over the group (ties: lowest index)
        float Eb = -INFINITY, dEb = 0.0f;
        int kb = 0x7fff;
        if constexpr (NCH == 1) {
            // the max of integer keys, E's bits (E >= 0 orders like them) with
            // the low 3 replaced by 7 - k; a candidate out of the running
            // (E = -inf) has key 0.  Two candidates within 7 ulps of each other
            // are both within the tie bound below (dE is at least 2 tie_kappa
            // ulps of E, since sqrt(S2 sum h e^2) >= |N|, and the host's
            // tie_kappa is at least 12), so whichever the key picks, the exact
            // comparison settles them.
            uint32_t key = 0;
#pragma unroll
            for (int qd = 0; qd < 2; ++qd) {
                const uint32_t k = (uint32_t)(qd * 4 + sl);
                const uint32_t kq = Ek[0][qd] >= 0.0f ? ((__float_as_uint(Ek[0][qd]) & ~7u) | (7u - k)) : 0u;
                key = max(key, kq);
            }
#pragma unroll
            for (int o = 2; o; o >>= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, o));
            const int kk = 7 - (int)(key & 7u);
            const int owner = (gs * 4) | (kk & 3);
            const float Eo0 = __shfl_sync(0xffffffffu, Ek[0][0], owner);
            const float Eo1 = __shfl_sync(0xffffffffu, Ek[0][1], owner);
            const float dEo0 = __shfl_sync(0xffffffffu, dEk[0][0], owner);
            const float dEo1 = __shfl_sync(0xffffffffu, dEk[0][1], owner);
            if (key != 0u) {
                Eb = kk & 4 ? Eo1 : Eo0;
                dEb = kk & 4 ? dEo1 : dEo0;
                kb = kk;
            }
        } else {
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                for (int qd = 0; qd < 2; ++qd)
                    if (Ek[ch][qd] > Eb) {  // strict: keeps the lower k of this lane
                        Eb = Ek[ch][qd];
                        dEb = dEk[ch][qd];
                        kb = ch * 8 + qd * 4 + sl;
                    }
#pragma unroll
            for (int o = 2; o; o >>= 1) {
                const float Eo = shx(Eb, o);
                const float dEo = shx(dEb, o);
                const int ko = __shfl_xor_sync(0xffffffffu, kb, o);
                if (Eo > Eb || (Eo == Eb && ko < kb)) {
                    Eb = Eo;
                    dEb = dEo;
                    kb = ko;
                }
            }
        }
        if (kb > 0x7ff) kb = 0;  // every candidate suspicious: the exact path picks

        // the sums of candidate k, from its owner lane (every lane of a group
        // names the same k)
        auto sums_of = [&](int k, float& t1, float& t2, float& t3) {
            const int owner = (gs * 4) | (k & 3);
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                for (int qd = 0; qd < 2; ++qd) {
                    const float a1 = __shfl_sync(0xffffffffu, T1k[ch][qd], owner);
                    const float a2 = __shfl_sync(0xffffffffu, T2k[ch][qd], owner);
                    const float a3 = __shfl_sync(0xffffffffu, T3k[ch][qd], owner);
                    if ((k >> 2) == ch * 2 + qd) {
                        t1 = a1;
                        t2 = a2;
                        t3 = a3;
                    }
                }
        };
        float T1b = 0.0f, T2b = 0.0f, T3b = 0.0f;
        sums_of(kb, T1b, T2b, T3b);
        // Candidates needing an exact comparison: within the fp32 error bound
        // of the winner.  Those whose sums, about the winner's centre code
        // (their chunk's or another chunk's with the same centre), equal the
        // winner's bit for bit ("twins") almost always have the winner's
        // codes -- equal codes give equal errors, and the lower index is
        // kept, as Algorithm 1's argmin does -- but an element of tiny
        // saliency can differ without moving the sums, so twins are first
        // checked code by code (cheaply, deferred) -- unless every saliency
        // of the group is too large for that.  Between two factors every
        // element's code moves away from the centre or stays, and a moving
        // element has |d| >= range f / q_max (f the smaller factor), so a
        // code difference moves T3 - (c - mu) T1 by at least h_min range f /
        // q_max, less the roundings of e, d and c (every term has the sign of
        // the move: e - (c - mu) is d up to those roundings).  Bitwise-equal
        // sums bound that change by twice their fp32 errors, ulp sqrt(T2 see)
        // and |c - mu| ulp sqrt(Ss T2); a larger bound leaves the codes
        // equal (up to elements of zero saliency, which move no error).
        float y0w = Y0k[0];
#pragma unroll
        for (int ch = 1; ch < NCH; ++ch)
            if ((kb >> 3) == ch) y0w = Y0k[ch];
        bool twinf[NCH][2];
        bool anytwin = false;
#pragma unroll
        for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
            for (int qd = 0; qd < 2; ++qd) {
                const int k = ch * 8 + qd * 4 + sl;
                twinf[ch][qd] = k != kb && Y0k[ch] == y0w && T1k[ch][qd] == T1b &&
                                T2k[ch][qd] == T2b && T3k[ch][qd] == T3b;
                anytwin |= twinf[ch][qd];
            }
        // the bound (only where a warp has twins): the group's smallest
        // saliency, from the tile (the fit's h, 1 for all-zero groups).
        // Built for 16 or more candidates, where twins are common (with 8
        // they are rare and the code costs more than it saves).
        constexpr bool kCertify = NCH >= 2 && !ADAM;
        float twin_q = INFINITY, twin_h = 0.0f, twin_e = 0.0f;
        if (kCertify && __any_sync(0xffffffffu, anytwin)) {
            float hmn = INFINITY;
#pragma unroll 1
            for (int i = 0; i < NCHK; ++i) {
                const float4 h4 = lds128(ghs + eoff(i));
                hmn = fmin3(fmin3(hmn, h4.x, h4.y), h4.z, h4.w);
            }
#pragma unroll
            for (int o = 2; o; o >>= 1) hmn = fminf(hmn, shx(hmn, o));
            const float t2s = fmaxf(T2b * see, 0.0f), t2w = fmaxf(ss * T2b, 0.0f);
            twin_q = 2.0f * ulp * (sqrtf(t2s) + fabsf(cref - mu) * sqrtf(t2w)) * qmaxf;
            twin_h = hmn * range;
            twin_e = hmn * qmaxf * (8.0f * 5.9604645e-8f) * (range + fabsf(cref));
        }
        unsigned set = 0, twins = 0;
        if constexpr (!kCertify) {
            // contenders first; the twins among them only where a warp has any
            bool cont[NCH][2];
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                for (int qd = 0; qd < 2; ++qd) {
                    const int k = ch * 8 + qd * 4 + sl;
                    cont[ch][qd] = k != kb && Ek[ch][qd] > -INFINITY &&
                                   Eb - Ek[ch][qd] <= dEb + dEk[ch][qd];
                    const unsigned bal = __ballot_sync(0xffffffffu, cont[ch][qd] || suspk[ch][qd]);
                    set |= ((bal >> (gs * 4)) & 0xFu) << (ch * 8 + qd * 4);
                }
            if (__any_sync(0xffffffffu, set != 0u)) {
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                    for (int qd = 0; qd < 2; ++qd) {
                        const unsigned balt =
                            __ballot_sync(0xffffffffu, cont[ch][qd] && twinf[ch][qd] && !suspk[ch][qd]);
                        twins |= ((balt >> (gs * 4)) & 0xFu) << (ch * 8 + qd * 4);
                    }
            }
        } else {
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                for (int qd = 0; qd < 2; ++qd) {
                    const int k = ch * 8 + qd * 4 + sl;
                    const bool twin = twinf[ch][qd];
                    // a twin whose codes are certainly the winner's: as the winner
                    const bool sure = twin && twin_h * fminf(p.f[k], p.f[kb]) - twin_e > twin_q;
                    const bool contender = k != kb && !sure && Ek[ch][qd] > -INFINITY &&
                                           Eb - Ek[ch][qd] <= dEb + dEk[ch][qd];
                    const unsigned bal = __ballot_sync(0xffffffffu, contender || suspk[ch][qd]);
                    set |= ((bal >> (gs * 4)) & 0xFu) << (ch * 8 + qd * 4);
                    const unsigned balt = __ballot_sync(0xffffffffu, contender && twin && !suspk[ch][qd]);
                    twins |= ((balt >> (gs * 4)) & 0xFu) << (ch * 8 + qd * 4);
                }
        }
        if (Eb == -INFINITY) set = (p.n_clip >= 32) ? 0xFFFFFFFFu : ((1u << p.n_clip) - 1u);
        else if (set) set |= 1u << kb;

        // the kept fit: r = a zeta + Bz (a = a_sel + a_lo, Bz = Bz + Bz_lo); kap
        // estimates the conditioning of its slope
        float a_sel = 0.0f, Bz = 0.0f, kap_sel = 0.0f;
        float Bz_lo = 0.0f, a_lo = 0.0f;
        bool deg_sel = false;

        // ---- deferred exact comparisons: the whole warp takes one group at a time
        unsigned todo = __ballot_sync(0xffffffffu, valid && !flat && set != 0 && sl == 0);
        while (todo) {
            const int g = (__ffs(todo) - 1) >> 2;
            todo &= todo - 1;
            const int src = g * 4;
            GroupGeom ggq;
            ggq.nmn = __shfl_sync(0xffffffffu, gq.nmn, src);
            ggq.nrho = __shfl_sync(0xffffffffu, gq.nrho, src);
            ggq.ylo = ylo;
            ggq.yhi = yhi;
            const float grange = __shfl_sync(0xffffffffu, range, src);
            const float gR = __shfl_sync(0xffffffffu, R, src);
            const float gss = __shfl_sync(0xffffffffu, ss, src);
            const float gcref = __shfl_sync(0xffffffffu, cref, src);
            // the weighted mean of w - cref
            const float gdbar = __shfl_sync(0xffffffffu, (mu - cref) + ebar, src);
            unsigned gset = __shfl_sync(0xffffffffu, set, src);
            const unsigned gtwins = __shfl_sync(0xffffffffu, twins, src);
            int gw = __shfl_sync(0xffffffffu, kb, src);  // the winner
            const float* tws = ws + g * G;
            const float* ths = hs + g * G;
            float gy0[NCH];
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) gy0[ch] = __shfl_sync(0xffffffffu, Y0k[ch], src);
            if (p.stats && lane == 0) atomicAdd(&p.stats[2], 1u);
            auto same_codes = [&](int k) {
                if (p.stats && lane == 0) atomicAdd(&p.stats[6], 1u);
                return coop_same_codes<G>(tws, ggq, gR * p.invf[k], gR * p.invf[gw]);
            };
            // Codes move monotonically with 1/f, element by element (the
            // factors decrease with k), so two candidates with equal codes
            // share them with every candidate between them: the highest twin
            // settles all twins when its codes are the winner's.
            const bool mono = p.monotone != 0;
            unsigned tw = gtwins;
            if (tw && mono) {
                const int khi = 31 - __clz(tw);
                tw &= ~(1u << khi);
                if (same_codes(khi)) {
                    gset &= ~((2u << khi) - (2u << gw));  // (gw, khi]
                    tw = 0;
                }
            }
            while (tw) {
                const int k = __ffs(tw) - 1;
                tw &= tw - 1;
                if (same_codes(k)) gset &= ~(1u << k);
            }
            // Contenders about another centre code (their sums are not
            // comparable with the winner's): first whether they share the
            // winner's codes -- below the winner, lowest first, such a
            // candidate becomes the winner; above it, highest first, it
            // drops out (with monotone codes, so does everything between it
            // and the winner).
            auto other_centres = [&]() {
                float y0g = gy0[0];
#pragma unroll
                for (int ch = 1; ch < NCH; ++ch)
                    if ((gw >> 3) == ch) y0g = gy0[ch];
                unsigned m = 0;
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch)
                    if (gy0[ch] != y0g) m |= 0xFFu << (8 * ch);
                return m;
            };
            if (NCH > 1) {
                const unsigned cmask = other_centres();
                unsigned lo = gset & cmask & ((1u << gw) - 1u);
                while (lo) {
                    const int k = __ffs(lo) - 1;
                    lo &= lo - 1;
                    if (same_codes(k)) {
                        gset &= ~(mono ? (2u << gw) - (2u << k) : 1u << gw);  // (k, gw]
                        gw = k;
                        break;
                    }
                }
                unsigned hi = gset & cmask & ~((2u << gw) - 1u);
                while (hi) {
                    const int k = 31 - __clz(hi);
                    hi &= ~(1u << k);
                    if (same_codes(k)) {
                        gset &= ~(mono ? (2u << k) - (2u << gw) : 1u << k);  // (gw, k]
                        if (mono) break;
                    }
                }
            }
            if (gset == (1u << gw)) {  // only the winner left
                if (gs == g) kb = gw;
                continue;
            }
            if (p.stats && lane == 0) atomicAdd(&p.stats[0], 1u);
            float best_h = 0.0f, best_l = 0.0f, ga = 0.0f, gB = 0.0f, gkap = 0.0f;
            int best_k = -1;
            bool gdeg = false;
            // the quick error pass only where every candidate left has the
            // winner's centre code: candidates about different centres can
            // have equal codes with unequal sums, and only the two-pass fit, a
            // function of the codes alone, then gives them bitwise-equal
            // errors, so that the lower index is kept
            const bool one_chunk = (gset & other_centres()) == 0u;
            const float gebar = __shfl_sync(0xffffffffu, ebar, src);
            const float gsee = __shfl_sync(0xffffffffu, see, src);
            while (gset) {
                const int k = __ffs(gset) - 1;
                gset &= gset - 1;
                // the candidate's own fit from its centred sums, where its
                // fp32 error (fit_ulps ulps times the slope's condition kap)
                // moves the error sum by less than 1e-9 of itself (second
                // order: (rel. fit error)^2 times explained over residual
                // variance): then one error pass settles it; otherwise (and
                // for nearly degenerate code variance) the two-pass fit
                float k1 = 0.0f, k2 = 0.0f, k3 = 0.0f, y0k = gy0[0];
                {
                    const int owner = src | (k & 3);
#pragma unroll
                    for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                        for (int qd = 0; qd < 2; ++qd) {
                            const float a1 = __shfl_sync(0xffffffffu, T1k[ch][qd], owner);
                            const float a2 = __shfl_sync(0xffffffffu, T2k[ch][qd], owner);
                            const float a3 = __shfl_sync(0xffffffffu, T3k[ch][qd], owner);
                            if ((k >> 2) == ch * 2 + qd) {
                                k1 = a1;
                                k2 = a2;
                                k3 = a3;
                                y0k = gy0[ch];
                            }
                        }
                }
                const float Dk = k2 - k1 * (k1 / gss), Nk = k3 - k1 * gebar;
                const float ak = Nk / Dk, Exk = Nk * ak;
                const float kapk = sqrtf(k2 * gsee) / fabsf(Nk) + k2 / Dk;
                const float rel = p.fit_ulps * 5.9604645e-8f * kapk;
                const bool quick =
                    one_chunk && Dk > 1e-3f * k2 && rel * rel * Exk < 1e-9f * (gsee - Exk);
                float eh, el, a_k = 0.0f, B_k = 0.0f, kap_k = 0.0f;
                bool deg_k = false;
                if (p.stats && lane == 0) atomicAdd(&p.stats[quick ? 5 : 4], 1u);
                if (quick) {
                    // offset at q = 0 of w - cref: mean(w - cref) - a (mean zeta + J + 1)
                    const float bck = gdbar - ak * ((y0k - kGridMagic) + k1 / gss + Jp1);
                    coop_error<G>(tws, ths, ggq, gR * p.invf[k], Jp1, gcref, ak, bck, &eh, &el);
                } else {
                    coop_exact<G>(tws, ths, ggq, gR * p.invf[k], Jp1, gss, gdbar,
                                  p.f[k] * grange / qmaxf, gcref, &eh, &el, &a_k, &B_k, &kap_k, &deg_k);
                }
                if (best_k < 0 || ff_less(eh, el, best_h, best_l)) {
                    best_h = eh;
                    best_l = el;
                    best_k = k;
                    ga = a_k;
                    gB = B_k;
                    gkap = kap_k;
                    gdeg = deg_k;
                }
            }
            if (gs == g) {
                kb = best_k;
                a_sel = ga;
                Bz = gB;
                kap_sel = gkap;
                deg_sel = gdeg;
            }
        }

        // ---- the fit (Eq. 4) from the kept candidate's centred sums: codes
        // about its chunk's centre zeta0, weights about mu
        sums_of(kb, T1b, T2b, T3b);
        float y0b = Y0k[0];
#pragma unroll
        for (int ch = 1; ch < NCH; ++ch)
            if ((kb >> 3) == ch) y0b = Y0k[ch];
        if (!deg_sel) {
            // T1 = sum h (zeta - zeta0) (small); sum h (w - mu) = Se
            const float Aq = T1b * inv_ss;
            const float Nc = T3b - T1b * ebar, Dc = T2b - T1b * Aq;
            // the quotient from the fast reciprocal and one correction
            // (the remainder Nc - q Dc is exact by FMA): within an ulp
            const float q0 = __fdividef(Nc, Dc);
            const float an = fmaf(fmaf(-q0, Dc, Nc), __fdividef(1.0f, Dc), q0);
            // Bz = (mu + ebar) - a (zeta0 + Aq), as a float pair
            const float z0 = y0b - kGridMagic;  // exact
            float p_h, p_l, bh, bl;
            two_prod(an, z0, p_h, p_l);
            two_sum(mu, -p_h, bh, bl);
            bl = __fadd_rn(bl, __fsub_rn(ebar, fmaf(an, Aq, p_l)));
            ff_norm(bh, bl);
            a_sel = an;
            Bz = bh;
            Bz_lo = bl;
            const float dse = fmaxf(T2b * see, 1e-37f);
            kap_sel = __fdividef(dse * rsqrtf(dse), fabsf(Nc)) + __fdividef(T2b, Dc);
        }

        // ---- output accuracy check.  The fp32 fit's error at level q is at
        // most about est(q) = fit_ulps * ulp * (|a| kap (|q - qbar| + 1) + |c|
        // + |mu| + sqrt(see / Ss)): the slope's relative error (kap ulps)
        // times the level's distance from the weighted mean code qbar, plus
        // the error of the weighted mean itself, of the order of ulps of the
        // weighted mean |w| (at most |mu| + sqrt(see / Ss)) or, far from
        // zero, of the centre c.  fit_ulps is calibrated against the oracle
        // with a margin.  The slope a, the offset b (fp32) and a level
        // written in fp32 must meet tol(x) = 1e-7 + 1e-5|x|.  A level written
        // in bf16 is exact when no bf16 rounding midpoint lies within est of
        // it, and within the tolerance band when est <= tol.  Groups that
        // could miss get the compensated fit.
        const bool refit = !flat && !deg_sel;
        bool prec;
        {
            const float uf = p.fit_ulps * 5.9604645e-8f;
            const float ea = uf * fabsf(a_sel) * kap_sel;
            // (plus half an ulp of Bz: pass C may fold Bz's low part into it;
            // the square root as x rsqrt(x), within 2 ulps: immaterial beside
            // the margin in fit_ulps)
            const float sv = fmaxf(see * inv_ss, 1e-37f);
            const float ec = uf * (fabsf(cref) + fabsf(mu) + sv * rsqrtf(sv)) +
                             0.5f * 5.9604645e-8f * fabsf(Bz);
            // the weighted mean code (q = zeta + J + 1)
            const float qbar = (y0b - kGridMagic) + T1b * inv_ss + Jp1;
            const float b0 = fmaf(-a_sel, Jp1, Bz);  // offset at q = 0
            prec = fmaf(ea, fabsf(qbar) + 1.0f, ec) > 1e-7f + 1e-5f * fabsf(b0);
            prec |= ea > 1e-7f + 1e-5f * fabsf(a_sel);
            for (float qf = (float)sl; qf <= qmaxf; qf += (float)kIntLanes) {
                const float rq = fmaf(a_sel, qf, b0);
                const float est = fmaf(ea, fabsf(qf - qbar) + 1.0f, ec);
                if (est > 1e-7f + 1e-5f * fabsf(rq)) {
                    if (!p.r_bf16) {
                        prec = true;
                    } else {
                        const uint32_t bits = __float_as_uint(rq);
                        const int dmid = abs((int)(bits & 0xFFFFu) - 0x8000);  // fp32 ulps to the midpoint
                        const float ulp32 =
                            __uint_as_float(max(bits & 0x7F800000u, 0x0C000000u) - 0x0B800000u);
                        prec |= (float)dmid * ulp32 < 1.5f * est;
                    }
                }
            }
            const float esum = ea + ec + qbar;
            prec = prec || esum != esum;  // NaN sums: take the careful path
            // one decision per group: any lane of the group that flagged
            prec = (__ballot_sync(0xffffffffu, prec) & gmask) != 0;
        }
        todo = __ballot_sync(0xffffffffu, valid && refit && prec && sl == 0);
        while (todo) {
            const int g = (__ffs(todo) - 1) >> 2;
            todo &= todo - 1;
            const int src = g * 4;
            GroupGeom ggq;
            ggq.nmn = __shfl_sync(0xffffffffu, gq.nmn, src);
            ggq.nrho = __shfl_sync(0xffffffffu, gq.nrho, src);
            ggq.ylo = ylo;
            ggq.yhi = yhi;
            const float gR = __shfl_sync(0xffffffffu, R, src);
            const float gss = __shfl_sync(0xffffffffu, ss, src);
            const float gmu = __shfl_sync(0xffffffffu, mu + ebar, src);
            const int gkb = __shfl_sync(0xffffffffu, kb, src);
            if (p.stats && lane == 0) atomicAdd(&p.stats[1], 1u);
            float ga, ga_lo, gB, gB_lo;
            coop_precise<G>(ws + g * G, hs + g * G, ggq, gR * p.invf[gkb], Jp1, gss, gmu, &ga,
                            &ga_lo, &gB, &gB_lo);
            if (gs == g) {
                a_sel = ga;
                a_lo = ga_lo;
                Bz = gB;
                Bz_lo = gB_lo;
            }
        }

        // ---- pass C: outputs of the kept candidate (its codes recomputed
        // with the clamp of its set, as pass B formed them)
        const float Pk = R * p.invf[kb];
        const float capk = p.cap[kb] * range;
        {
            const float2 a2 = make_float2(a_sel, a_sel), B2 = make_float2(Bz, Bz);
            const float2 alo2 = make_float2(a_lo, a_lo), Blo2 = make_float2(Bz_lo, Bz_lo);
            // the fast path folds Bz's low part into Bz (within the half ulp
            // the accuracy check allows for it); a compensated fit keeps both
            const float Bf = __fadd_rn(Bz, Bz_lo);
            const float2 Bf2 = make_float2(Bf, Bf);
            const float2 Pk2 = make_float2(Pk, Pk);
            const int64_t ebase = gbase;
            // general: codes, fp32 r, zero-range groups (r = w), compensated fits;
            // fast: none of these (and the folded offset)
            auto pass_c = [&](auto general) {
                constexpr bool GEN = decltype(general)::value;
#pragma unroll 2
                for (int i = 0; i < NCHK; ++i) {
                    const int eo = eoff(i);
                    const float4 w4 = lds128(gws + eo);
                    float2 yv[2], zs[2];
#pragma unroll
                    for (int pr = 0; pr < 2; ++pr) {
                        const float2 wv = pr ? make_float2(w4.z, w4.w) : make_float2(w4.x, w4.y);
                        const float2 d = __fadd2_rn(__fadd2_rn(wv, nmn2), nrho2);
                        const float2 dc = make_float2(fminf(fmaxf(d.x, -capk), capk),
                                                      fminf(fmaxf(d.y, -capk), capk));
                        yv[pr] = __ffma2_rd(dc, Pk2, Mg2);
                        zs[pr] = __fadd2_rn(yv[pr], nMg2);  // zeta, exact
                    }
                    float2 rv[2];
#pragma unroll
                    for (int pr = 0; pr < 2; ++pr)
                        rv[pr] = GEN ? __fadd2_rn(__ffma2_rn(a2, zs[pr], B2), __ffma2_rn(alo2, zs[pr], Blo2))
                                     : __ffma2_rn(a2, zs[pr], Bf2);
                    const int64_t ge = ebase + eo;
                    if constexpr (GEN) {
                        if (flat) {
                            rv[0] = make_float2(w4.x, w4.y);
                            rv[1] = make_float2(w4.z, w4.w);
                        }
                        if (T.codes) {
                            // q = y - ylo, an integer in [0, 255]: y and ylo share
                            // a binade, so it is the difference of their bits
                            const uint32_t b0 = __float_as_uint(ylo);
                            uint32_t cw = 0;
#pragma unroll
                            for (int pr = 0; pr < 2; ++pr)
                                cw |= (((__float_as_uint(yv[pr].x) - b0) & 0xFFu) |
                                       (((__float_as_uint(yv[pr].y) - b0) & 0xFFu) << 8))
                                      << (16 * pr);
                            if (flat) cw = 0;
                            if (!(VAR && p.codes_packed) && valid)
                                stg_cs(reinterpret_cast<uint32_t*>(T.codes + ge), cw);
                        }
                    }
                    if (!valid) {
                    } else if (!GEN || p.r_bf16) {
                        stg_cs(reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(T.r) + ge),
                               make_uint2(pack_bf16x2(rv[0].x, rv[0].y), pack_bf16x2(rv[1].x, rv[1].y)));
                    } else {
                        stg_cs(reinterpret_cast<float4*>(static_cast<float*>(T.r) + ge),
                               make_float4(rv[0].x, rv[0].y, rv[1].x, rv[1].y));
                    }
                }
            };
            // lanes of a missing group store nothing (with VAR every lane runs
            // pass C: the packed codes below synchronise the warp)
            const bool gen = !p.r_bf16 || T.codes != nullptr || __any_sync(0xffffffffu, flat || a_lo != 0.0f);
            if (VAR || valid) {
                if (gen) pass_c(std::true_type{});
                else pass_c(std::false_type{});
            }
            if (VAR && T.codes && p.codes_packed) {
                // the deployment format: the group's codes as one little-endian
                // bitstream of `bits` bits a code.  Each 32-code span fills
                // `bits` words; in two steps, each of the 4 lanes ORs a 4-code
                // field (4 bits bits wide) into them in the scratch, and lanes
                // sl and sl + 4 of the span's words are stored.
                uint32_t* wsc = reinterpret_cast<uint32_t*>(red) + gs * 8;
// (codes recomputed from the tile, as pass C forms them: kept registers would
// raise the pressure of the common path)
#pragma unroll 1
                for (int m = 0; m < G / 32; ++m) {
                    __syncwarp();
                    wsc[sl] = 0u;
                    wsc[sl + 4] = 0u;
                    __syncwarp();
#pragma unroll
                    for (int j2 = 0; j2 < 2; ++j2) {
                        const int c0 = 16 * j2 + 4 * sl;  // first code of the field
                        uint32_t pk = 0;
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const float d = centred(gws[32 * m + c0 + j], gq.nmn, gq.nrho);
                            const uint32_t q = flat ? 0u : (uint32_t)int_code_q(d, Pk, ylo, yhi);
                            pk |= q << (j * p.bits);
                        }
                        const uint32_t o = (uint32_t)c0 * (uint32_t)p.bits;
                        const uint64_t f = (uint64_t)pk << (o & 31u);
                        atomicOr(&wsc[o >> 5], (uint32_t)f);
                        if ((uint32_t)(f >> 32)) atomicOr(&wsc[(o >> 5) + 1], (uint32_t)(f >> 32));
                    }
                    __syncwarp();
                    uint32_t* dst = reinterpret_cast<uint32_t*>(T.codes) + grp * (int64_t)(G / 32) * p.bits +
                                    m * p.bits;
                    if (valid && sl < p.bits) stg_cs(dst + sl, wsc[sl]);
                    if (valid && sl + 4 < p.bits) stg_cs(dst + sl + 4, wsc[sl + 4]);
                }
                __syncwarp();
            }
            if (valid && sl == 0) {
                // b = Bz - a*(J + 1): the offset at code 0
                float bh = Bz, bl = Bz_lo;
                ff_add_prod(bh, bl, -a_sel, -a_lo, Jp1);
                T.a[grp] = flat ? 0.0f : a_sel;
                T.b[grp] = flat ? mn : __fadd_rn(bh, bl);
                if (T.idx) T.idx[grp] = flat ? 0 : (uint8_t)kb;
            }
        }

        // release the tile: all lanes are done with it; order our generic
        // writes to it before the async-proxy copy that refills it with the
        // slot's next tile
        __syncwarp();
        if (lane == 0 && t + S < nt) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue(t + S, slot);
        }
        slot += nwarps;
        if (slot >= S) {
            slot -= S;
            parity ^= 1u;
        }
    }
}

}  // namespace quasar
