"""Pins for the oracle's single-candidate helpers that the parity checker uses.

The checker calls these on groups where the GPU and the oracle may
legitimately differ (an element within 1e-6 of a rounding boundary, two
candidates within 1e-6 of each other): it recomputes codes, fits and errors
of the GPU's candidate with them.  Each helper is pinned here against
something other than the oracle: numpy's least-squares solver, a direct
numpy sum of Eq. 3, an enumeration of every E2M1 or E4M3 value, or the
pinned full-algorithm entry points (Algorithm 1, Sec. 4.2, App. B) on the
candidate they kept.
"""
import numpy as np
import pytest

CLIP8 = [1.0, 0.95, 0.9, 0.85, 0.8, 0.75, 0.7, 0.65]
E2M1 = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])


def _f32(x):
    return float(np.float32(x))


def _groups(seed, n, G):
    rng = np.random.default_rng(seed)
    w = (0.02 * rng.standard_t(4, size=(n, G))).astype(np.float32)
    h = np.exp(rng.normal(-14.0, 2.0, size=(n, G))).astype(np.float32)
    return w, h


def _wlstsq(q, w, h, intercept=True):
    """Weighted least squares of w on q (and 1) by numpy's solver."""
    sq = np.sqrt(h.astype(np.float64))
    cols = [q.astype(np.float64)] + ([np.ones(q.size)] if intercept else [])
    A = np.stack(cols, 1) * sq[:, None]
    sol, *_ = np.linalg.lstsq(A, w.astype(np.float64) * sq, rcond=None)
    return sol


def _direct(w, h, r):
    """Eq. 3: sum h (r - w)^2 in fp64."""
    return float(np.sum(h.astype(np.float64) * (r - w.astype(np.float64)) ** 2))


def _e4m3_table(oracle):
    return np.array([oracle.e4m3_value(b) for b in range(0x7F)])


def _e4m3_nearest(table, x):
    """Nearest non-negative finite E4M3 value by enumeration: ties to the even
    bit pattern, above 448 saturating (the format's satfinite rounding)."""
    d = np.abs(table - x)
    best = np.flatnonzero(d == d.min())
    even = [b for b in best if b % 2 == 0]
    return int(even[0] if even else best[0])


def _e2m1_codes(w, sigma):
    """E2M1 codes of a block by enumeration: nearest magnitude of |w|/sigma
    (saturating at 6, ties to the even code index), sign of w, +0 for 0."""
    out = np.zeros(w.size, np.uint8)
    for i, x in enumerate(w.astype(np.float64)):
        y = min(abs(x) / sigma, 6.0)
        d = np.abs(E2M1 - y)
        best = np.flatnonzero(d == d.min())
        even = [m for m in best if m % 2 == 0]
        m = int(even[0] if even else best[0])
        out[i] = (8 if (x < 0 and m != 0) else 0) | m
    return out


def _decode(codes):
    c = codes.astype(np.int64)
    return np.where(c & 8, -1.0, 1.0) * E2M1[c & 7]


# ----------------------------------------------------------- integer codes --

def test_refit_int_is_weighted_least_squares(oracle):
    """qo_refit_int: on the kept codes it reproduces Algorithm 1's (a, b,
    error); on arbitrary codes it is numpy's weighted least-squares line with
    the direct Eq. 3 error; one weighted code gives the grid-step rule D3; all
    saliencies zero give ordinary least squares (D2)."""
    bits, G = 3, 128
    w, h = _groups(41, 12, G)
    O = oracle.recon_int(w, h, G, bits, CLIP8)
    rng = np.random.default_rng(42)
    for g in range(w.shape[0]):
        k = int(O["idx"][g])
        q = O["codes"][G * g:G * (g + 1)]
        s, z, e = oracle.refit_int(w[g], h[g], q, bits, CLIP8[k])
        assert s == pytest.approx(O["a"][g], rel=1e-12)
        assert z == pytest.approx(O["b"][g], rel=1e-12, abs=1e-15)
        assert e == pytest.approx(O["err"][g], rel=1e-12, abs=1e-300)
        qr = rng.integers(0, 8, G).astype(np.uint8)
        s, z, e = oracle.refit_int(w[g], h[g], qr, bits, 0.9)
        a_ref, b_ref = _wlstsq(qr, w[g], h[g])
        assert s == pytest.approx(a_ref, rel=1e-9)
        assert abs(z - b_ref) <= 1e-10 * np.abs(w[g]).max()
        assert e == pytest.approx(_direct(w[g], h[g], a_ref * qr + b_ref), rel=1e-9)
    # D3: every weighted element on one code
    wg, hg = w[0].copy(), h[0].copy()
    q1 = np.full(G, 5, np.uint8)
    f = 0.8
    s, z, e = oracle.refit_int(wg, hg, q1, bits, f)
    wd, hd = wg.astype(np.float64), hg.astype(np.float64)
    step = (wd.max() - wd.min()) * _f32(f) / 7.0
    wbar = np.sum(hd * wd) / np.sum(hd)
    assert s == pytest.approx(step, rel=1e-14)
    assert z == pytest.approx(wbar - 5 * step, rel=1e-12, abs=1e-15)
    assert e == pytest.approx(np.sum(hd * (wd - wbar) ** 2), rel=1e-10)
    # D2: no saliency at all is the unweighted fit
    qr = rng.integers(0, 8, G).astype(np.uint8)
    s, z, e = oracle.refit_int(wg, np.zeros(G, np.float32), qr, bits, 1.0)
    a_ref, b_ref = _wlstsq(qr, wg, np.ones(G))
    assert s == pytest.approx(a_ref, rel=1e-9)
    assert abs(z - b_ref) <= 1e-10 * np.abs(wg).max()


def test_refit_sym_is_least_squares_through_origin(oracle):
    """qo_refit_sym: Algorithm 1's kept (a, error) on the kept symmetric
    codes; numpy's weighted slope through the origin on arbitrary codes; the
    candidate's grid step when every weighted element codes to 0."""
    bits, G = 4, 128
    Q = 7
    w, h = _groups(43, 8, G)
    O = oracle.recon_sym(w.ravel(), h.ravel(), G, bits, CLIP8)
    rng = np.random.default_rng(44)
    for g in range(w.shape[0]):
        k = int(O["idx"][g])
        q = O["codes"][G * g:G * (g + 1)]
        s, e = oracle.refit_sym(w[g], h[g], q, bits, CLIP8[k])
        assert s == pytest.approx(O["a"][g], rel=1e-12)
        assert e == pytest.approx(O["err"][g], rel=1e-12, abs=1e-300)
        qr = rng.integers(0, 2 * Q + 1, G).astype(np.uint8)
        s, e = oracle.refit_sym(w[g], h[g], qr, bits, 0.85)
        qs = qr.astype(np.float64) - Q
        (a_ref,) = _wlstsq(qs, w[g], h[g], intercept=False)
        assert s == pytest.approx(a_ref, rel=1e-9)
        assert e == pytest.approx(_direct(w[g], h[g], a_ref * qs), rel=1e-9)
    wg = w[1]
    s, e = oracle.refit_sym(wg, h[1], np.full(G, Q, np.uint8), bits, 0.75)
    assert s == pytest.approx(_f32(0.75) * np.abs(wg.astype(np.float64)).max() / Q, rel=1e-14)
    assert e == pytest.approx(_direct(wg, h[1], np.zeros(G)), rel=1e-12)


# ------------------------------------------------------------------- NVFP4 --

def _nvfp4_case(seed, n_blocks=48):
    rng = np.random.default_rng(seed)
    w = (0.02 * rng.standard_t(4, size=n_blocks * 16)).astype(np.float32)
    h = np.exp(rng.normal(-14.0, 2.0, n_blocks * 16)).astype(np.float32)
    return w, h


def test_codes_nvfp4_enumeration_and_kept_codes(oracle):
    """qo_codes_nvfp4: the nearest E2M1 value of |w|/sigma for every
    element (enumerated here), sigma = f amax_b / 6 (Sec. 4.2), the sign of
    w with +0 for magnitude 0; and the codes Sec. 4.2's search kept."""
    w, h = _nvfp4_case(51)
    _, sT = oracle.tensor_scale(w)
    O = oracle.recon_nvfp4(w, h, sT, CLIP8)
    for b in range(w.size // 16):
        wb = w[16 * b:16 * (b + 1)]
        amax = np.abs(wb.astype(np.float64)).max()
        for f in (CLIP8[int(O["idx"][b])], 0.7, 1.0):
            q, m = oracle.codes_nvfp4(wb, f)
            ref = _e2m1_codes(wb, _f32(f) * amax / 6.0)
            ok = (q == ref) | (m < 1e-12)
            assert np.all(ok), (b, f)
        q, _ = oracle.codes_nvfp4(wb, CLIP8[int(O["idx"][b])])
        assert np.array_equal(q, O["codes"][16 * b:16 * (b + 1)])
    # the zero block codes to +0 everywhere
    q, _ = oracle.codes_nvfp4(np.zeros(16, np.float32), 0.9)
    assert np.all(q == 0)
    # signed zeros: -0.0 and tiny negatives that round to 0 store +0
    wz = np.array([-0.0, -1e-9, 3.0] + [0.5] * 13, np.float32)
    q, _ = oracle.codes_nvfp4(wz, 1.0)
    assert q[0] == 0 and q[1] == 0 and q[2] == 7


def test_fit_nvfp4_scale_enumerates_e4m3(oracle):
    """qo_fit_nvfp4_scale: among all 127 non-negative E4M3 values the
    returned one minimises Eq. 3 of the given codes (enumerated here), equal
    to the kept scale of Sec. 4.2's search on the kept codes; with no
    weighted nonzero code it is E4M3 of the search scale (rule N4)."""
    tab = _e4m3_table(oracle)
    w, h = _nvfp4_case(52)
    _, sT = oracle.tensor_scale(w)
    sT64 = float(sT)
    O = oracle.recon_nvfp4(w, h, sT, CLIP8)
    rng = np.random.default_rng(53)
    for b in range(w.size // 16):
        wb, hb = w[16 * b:16 * (b + 1)], h[16 * b:16 * (b + 1)]
        k = int(O["idx"][b])
        kept = O["codes"][16 * b:16 * (b + 1)]
        bits, _ = oracle.fit_nvfp4_scale(wb, hb, sT, CLIP8[k], kept)
        assert bits == O["scale"][b]
        qr = rng.integers(0, 16, 16).astype(np.uint8)
        bits, _ = oracle.fit_nvfp4_scale(wb, hb, sT, 0.8, qr)
        q = _decode(qr)
        errs = np.array([_direct(wb, hb, sT64 * e * q) for e in tab])
        assert errs[bits] <= errs.min() * (1 + 1e-12) + 1e-300
        hd = hb.astype(np.float64)
        x = np.sum(hd * q * wb) / np.sum(hd * q * q) / sT64
        if x > 0:
            assert bits == _e4m3_nearest(tab, x)
    wb = w[:16].copy()
    hb = np.zeros(16, np.float32)
    hb[3] = 1.0
    wb[3] = 1e-12 * np.abs(wb).max()   # the one weighted element codes to 0
    bits, _ = oracle.fit_nvfp4_scale(wb, hb, sT, 0.9, oracle.codes_nvfp4(wb, 0.9)[0])
    sigma = _f32(0.9) * np.abs(wb.astype(np.float64)).max() / 6.0
    assert bits == _e4m3_nearest(tab, sigma / sT64)


def test_eval_nvfp4_is_the_direct_error(oracle):
    """qo_eval_nvfp4: Eq. 3 of s_T e q summed directly in numpy, for random
    codes and scale bits, and the kept candidate's error of Sec. 4.2."""
    tab = _e4m3_table(oracle)
    w, h = _nvfp4_case(54, 16)
    _, sT = oracle.tensor_scale(w)
    O = oracle.recon_nvfp4(w, h, sT, CLIP8)
    rng = np.random.default_rng(55)
    for b in range(w.size // 16):
        wb, hb = w[16 * b:16 * (b + 1)], h[16 * b:16 * (b + 1)]
        qr = rng.integers(0, 16, 16).astype(np.uint8)
        sb = int(rng.integers(0, 0x7F))
        e = oracle.eval_nvfp4(wb, hb, sT, qr, sb)
        assert e == pytest.approx(_direct(wb, hb, float(sT) * tab[sb] * _decode(qr)), rel=1e-13)
        e = oracle.eval_nvfp4(wb, hb, sT, O["codes"][16 * b:16 * (b + 1)], int(O["scale"][b]))
        assert e == pytest.approx(O["err"][b], rel=1e-13, abs=1e-300)
    # all saliencies zero: h = 1 (rule D2)
    wb = w[:16]
    e = oracle.eval_nvfp4(wb, np.zeros(16, np.float32), sT, np.zeros(16, np.uint8), 0)
    assert e == pytest.approx(_direct(wb, np.ones(16), np.zeros(16)), rel=1e-13)


# ------------------------------------------------------------ lookup table --

def _signed_e4m3(oracle):
    vals, bits = [], []
    for b in range(0x7F):
        v = oracle.e4m3_value(b)
        vals += [v, -v]
        bits += [b, 0x80 | b]
    return np.array(vals), np.array(bits)


def _lut_case(seed, rows=8, cols=128):
    rng = np.random.default_rng(seed)
    w = (0.02 * rng.standard_t(4, size=(rows, cols))).astype(np.float32)
    h = np.exp(-14.0 + 2.0 * rng.standard_normal((rows, cols))).astype(np.float32)
    return w, h


def test_lut_block_matches_app_b_candidates(oracle):
    """qo_lut_block: per candidate, the error App. B's search reports for
    that candidate, and for the kept candidate its indices and table."""
    w, h = _lut_case(61)
    O = oracle.recon_lut(w, h, CLIP8)
    wb, hb = oracle.lut_blocks(w), oracle.lut_blocks(h)
    qb = oracle.lut_blocks(O["codes"].reshape(w.shape))
    for blk in range(wb.shape[0]):
        for k, f in enumerate(CLIP8):
            q, book, e, _, _ = oracle.lut_block(wb[blk], hb[blk], f)
            assert e == pytest.approx(O["cand_err"][blk][k], rel=1e-13, abs=1e-300)
            if k == O["idx"][blk]:
                assert np.array_equal(q, qb[blk])
                assert np.array_equal(book, O["book"][blk])


def test_lut_fit_is_the_weighted_mean_rounded(oracle):
    """qo_lut_fit (Eq. rubin-fit) on arbitrary indices: each index with
    weight gets the signed E4M3 value that minimises sum h (C - w)^2 over
    every finite E4M3 value (enumerated here); an index with none gets the
    E4M3 value nearest its grid point c - f rho + k 2 f rho / 7 (L3)."""
    vals, vbits = _signed_e4m3(oracle)
    w, h = _lut_case(62)
    wb, hb = oracle.lut_blocks(w), oracle.lut_blocks(h)
    rng = np.random.default_rng(63)
    f = 0.85
    for blk in range(wb.shape[0]):
        q = rng.integers(0, 7, wb.shape[1]).astype(np.uint8)  # index 7 left empty
        book, _ = oracle.lut_fit(wb[blk], hb[blk], f, q)
        wd, hd = wb[blk].astype(np.float64), hb[blk].astype(np.float64)
        for k in range(7):
            sel = q == k
            cost = ((vals[:, None] - wd[sel][None, :]) ** 2 * hd[sel][None, :]).sum(1)
            got = oracle.e4m3s_value(int(book[k]))
            assert ((got - wd[sel]) ** 2 * hd[sel]).sum() <= cost.min() * (1 + 1e-12) + 1e-300
        mn, mx = wd.min(), wd.max()
        c, rho = 0.5 * (mn + mx), 0.5 * (mx - mn)
        grid = c - _f32(f) * rho + 7 * 2.0 * _f32(f) * rho / 7.0
        d = np.abs(vals - grid)
        assert abs(oracle.e4m3s_value(int(book[7])) - grid) == d.min()
    # the kept table of App. B's search on its kept indices
    O = oracle.recon_lut(w, h, CLIP8)
    qb = oracle.lut_blocks(O["codes"].reshape(w.shape))
    for blk in range(wb.shape[0]):
        book, _ = oracle.lut_fit(wb[blk], hb[blk], CLIP8[int(O["idx"][blk])], qb[blk])
        assert np.array_equal(book, O["book"][blk])


def test_lut_eval_is_the_direct_error(oracle):
    """qo_lut_eval: sum h (table[q] - w)^2 summed directly in numpy."""
    w, h = _lut_case(64)
    wb, hb = oracle.lut_blocks(w), oracle.lut_blocks(h)
    rng = np.random.default_rng(65)
    for blk in range(wb.shape[0]):
        q = rng.integers(0, 8, wb.shape[1]).astype(np.uint8)
        book = rng.integers(0, 256, 8).astype(np.uint8)
        book[(book & 0x7F) == 0x7F] = 0x7E               # finite values only
        table = np.array([oracle.e4m3s_value(int(b)) for b in book])
        e = oracle.lut_eval(wb[blk], hb[blk], q, book)
        assert e == pytest.approx(_direct(wb[blk], hb[blk], table[q]), rel=1e-13)
    e = oracle.lut_eval(wb[0], np.zeros(wb.shape[1], np.float32), q, book)
    assert e == pytest.approx(_direct(wb[0], np.ones(wb.shape[1]), table[q]), rel=1e-13)
