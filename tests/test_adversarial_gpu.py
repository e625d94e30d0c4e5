"""GPU against the oracle on inputs that stress the fp32 bounds the kernels
rely on (the code margins, the candidate-error tie bound, the fit error
estimate that decides the compensated fit):

* groups far from zero: centre c with |c| / range from 10 to 1e4, where the
  centre and the weights share their leading bits;
* ranges of a few ulps of the centre (a handful of distinct values);
* saliencies spanning 1e-30 .. 1e3 inside one group;
* exact duplicate weights (two or three distinct values a group);
* 8-bit codes, groups of 256 and 32 candidates on Student-t(2) weights;
* INT2, groups of 64 and 16 candidates (where candidates with the winner's
  sums are certified by the saliency floor or checked code by code).

Every case runs through the C ABI (single-tensor and batch calls) and is
checked with the same acceptance as the other parity tests (Algorithm 1,
Eq. 1, Eq. 3, Eq. 4; Sec. 4.2 for NVFP4)."""
import numpy as np
import pytest
import torch

from paper_2608_13966_gb300 import api
from paper_2608_13966_gb300 import workloads as WL
from tests import checker
from tests import gpu_harness as H

CLIP8 = list(WL.CLIP_8)
CLIP16 = list(WL.CLIP_16)
CLIP32 = [round(1.0 - 0.025 * i, 3) for i in range(32)]


def _lognormal(rng, n):
    return np.exp(-14.0 + 2.0 * rng.standard_normal(n)).astype(np.float32)


def far_from_zero(seed, n_groups, G):
    """Each group: c + range * (t4 values scaled into [-1/2, 1/2]), with
    |c| / range in {10, 100, 1e3, 1e4} and either sign."""
    rng = np.random.default_rng(seed)
    w = np.empty((n_groups, G), np.float32)
    for i in range(n_groups):
        ratio = [1e1, 1e2, 1e3, 1e4][i % 4] * (1 if (i // 4) % 2 == 0 else -1)
        r0 = [1e-2, 1.0, 3e-5][(i // 8) % 3]
        t = rng.standard_t(4, G)
        t = 0.5 * t / np.abs(t).max()
        w[i] = (np.float64(ratio * r0) + r0 * t).astype(np.float32)
    return w.ravel(), _lognormal(rng, n_groups * G)


def few_ulps(seed, n_groups, G):
    """Each group takes values c + k ulp(c), k in 0..4, for c in {1, -3, 1e3, 2^-20}."""
    rng = np.random.default_rng(seed)
    w = np.empty((n_groups, G), np.float32)
    for i in range(n_groups):
        c = np.float32([1.0, -3.0, 1e3, 2.0 ** -20][i % 4])
        k = rng.integers(0, 5, G)
        k[:2] = (0, 4)
        w[i] = c + k.astype(np.float32) * np.spacing(c)
    return w.ravel(), _lognormal(rng, n_groups * G)


def saliency_span(seed, n_groups, G):
    """t4 weights; saliency 10^u, u uniform in [-30, 3], inside every group."""
    rng = np.random.default_rng(seed)
    w = (0.02 * rng.standard_t(4, n_groups * G)).astype(np.float32)
    h = (10.0 ** rng.uniform(-30.0, 3.0, n_groups * G)).astype(np.float32)
    return w, h


def denormal_saliency(seed, n_groups, G):
    """t4 weights; saliency 10^u, u uniform in [-45, -38]: denormal and
    barely normal fp32 values, every group's sum far below the normal range
    of its squares (an EMA of squared gradients that decayed for long)."""
    rng = np.random.default_rng(seed)
    w = (0.02 * rng.standard_t(4, n_groups * G)).astype(np.float32)
    h = (10.0 ** rng.uniform(-45.0, -38.0, n_groups * G)).astype(np.float32)
    return w, h


def duplicates(seed, n_groups, G):
    """Two or three distinct values a group, each repeated."""
    rng = np.random.default_rng(seed)
    w = np.empty((n_groups, G), np.float32)
    for i in range(n_groups):
        vals = (0.02 * rng.standard_t(4, 2 + i % 2)).astype(np.float32)
        w[i] = vals[rng.integers(0, vals.size, G)]
    return w.ravel(), _lognormal(rng, n_groups * G)


def heavy_t2(seed, n_groups, G):
    """Student-t(2) weights (infinite variance), lognormal saliency."""
    rng = np.random.default_rng(seed)
    return (0.02 * rng.standard_t(2, n_groups * G)).astype(np.float32), _lognormal(rng, n_groups * G)


CASES = {
    "far_from_zero": (far_from_zero, 3, 128, CLIP8),
    "few_ulps": (few_ulps, 3, 128, CLIP8),
    "saliency_span": (saliency_span, 3, 128, CLIP8),
    "duplicates": (duplicates, 3, 128, CLIP8),
    "bits8_g256_k32_t2": (heavy_t2, 8, 256, CLIP32),
    "bits2_g64_k32_t2": (heavy_t2, 2, 64, CLIP32),
    "bits4_g32_k8_far": (far_from_zero, 4, 32, CLIP8),
    # 16 candidates: equal-sum candidates are taken as the winner's without a
    # code check when the group's smallest saliency allows it; these inputs
    # have tiny saliencies (the check runs) and repeated values (many equal
    # codes)
    "bits2_g64_k16_span": (saliency_span, 2, 64, CLIP16),
    "bits2_g64_k16_dup": (duplicates, 2, 64, CLIP16),
    "bits2_g64_k16_t2": (heavy_t2, 2, 64, CLIP16),
    "bits3_g128_k8_denorm": (denormal_saliency, 3, 128, CLIP8),
    "bits2_g64_k16_denorm": (denormal_saliency, 2, 64, CLIP16),
}


def _assert(rep, what):
    assert rep["ok"], (what, rep)


@pytest.mark.gpu
@pytest.mark.parametrize("r_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("case", sorted(CASES))
def test_int_adversarial(oracle, case, r_dtype):
    gen, bits, G, clip = CASES[case]
    n_groups = 48 * 3 + 5  # a ragged last unit
    w, h = gen(17, n_groups, G)
    w_t = torch.tensor(w, device="cuda").reshape(n_groups, G)
    v_t = torch.tensor(h, device="cuda").reshape(n_groups, G)
    # no gradient: h = v as given (the EMA is covered elsewhere)
    rep, ema = H.run_int(oracle, w_t, None, v_t, bits=bits, group_size=G, clip=clip,
                         r_dtype=r_dtype)
    _assert(rep, case)
    _assert(ema, case)
    # the same tensor through the batch call, split into two tensors
    rows = n_groups // 2
    items = [(w_t[:rows].clone(), None, v_t[:rows].clone()),
             (w_t[rows:].clone(), None, v_t[rows:].clone())]
    outs = api.recon_int_batch(items, bits=bits, group_size=G, clip=clip, r_dtype=r_dtype,
                               codes=True)
    torch.cuda.synchronize()
    for (wi, _, vi), o in zip(items, outs):
        wh, hh = H._host(wi), H._host(vi)
        O = oracle.recon_int(wh, hh, G, bits, clip)
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        _assert(checker.check_int(oracle, wh, hh, bits, clip, O, gpu, G,
                                  r_dtype == torch.bfloat16), case + " batch")


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["saliency_span", "duplicates", "heavy_t2", "denormal_saliency"])
def test_nvfp4_adversarial(oracle, case):
    gen = {"saliency_span": saliency_span, "duplicates": duplicates, "heavy_t2": heavy_t2,
           "denormal_saliency": denormal_saliency}[case]
    n_rows = 40
    w, h = gen(23, n_rows, 256)
    w_t = torch.tensor(w, device="cuda").reshape(n_rows, 256)
    v_t = torch.tensor(h, device="cuda").reshape(n_rows, 256)
    rep, ema = H.run_nvfp4(oracle, w_t, None, v_t, clip=CLIP8)
    _assert(rep, case)
    _assert(ema, case)


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["saliency_span", "duplicates", "denormal_saliency"])
def test_lut_adversarial(oracle, case):
    """The Rubin lookup table (App. B) on 8x64 blocks of the same inputs."""
    gen = {"saliency_span": saliency_span, "duplicates": duplicates,
           "denormal_saliency": denormal_saliency}[case]
    rows, cols = 24, 320  # 15 blocks
    w, h = gen(29, rows * cols // 64, 64)
    w_t = torch.tensor(w, device="cuda").reshape(rows, cols)
    v_t = torch.tensor(h, device="cuda").reshape(rows, cols)
    out = api.recon_lut_batch([(w_t, None, v_t)], clip=CLIP8, codes=True, r_dtype=torch.float32)[0]
    torch.cuda.synchronize()
    w2, h2 = w.reshape(rows, cols), h.reshape(rows, cols)
    O = oracle.recon_lut(w2, h2, CLIP8)
    gpu = {"r": H._host(out["r"]), "book": out["book"].cpu().numpy(),
           "codes": out["codes"].cpu().numpy(), "idx": out["cand_idx"].cpu().numpy()}
    _assert(checker.check_lut(oracle, w2, h2, CLIP8, O, gpu), case)


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["saliency_span", "denormal_saliency", "far_from_zero"])
def test_sym_adversarial(oracle, case):
    """Symmetric codes (Sec. 4.1.2's closed form) on the same inputs."""
    gen = {"saliency_span": saliency_span, "denormal_saliency": denormal_saliency,
           "far_from_zero": far_from_zero}[case]
    n_groups, G, bits = 149, 128, 4
    w, h = gen(31, n_groups, G)
    w_t = torch.tensor(w, device="cuda").reshape(n_groups, G)
    v_t = torch.tensor(h, device="cuda").reshape(n_groups, G)
    out = api.recon_int_batch([(w_t, None, v_t)], bits=bits, group_size=G, clip=CLIP8, codes=True,
                              symmetric=True, r_dtype=torch.float32)[0]
    torch.cuda.synchronize()
    O = oracle.recon_sym(w, h, G, bits, CLIP8)
    gpu = {"r": H._host(out["r"]), "a": out["a"].cpu().numpy(), "b": out["b"].cpu().numpy(),
           "codes": out["codes"].cpu().numpy().ravel(), "idx": out["cand_idx"].cpu().numpy()}
    _assert(checker.check_sym(oracle, w, h, bits, CLIP8, O, gpu, G, False), case)
