"""GPU parity: the CUDA library (through the C ABI) against the fp64 oracle.

Small cases span several units per warp, several warps per CTA and ragged
tails; the named workloads are the paper-shaped layers at full size.
"""
import json

import numpy as np
import pytest
import torch

from paper_2608_13966_gb300 import workloads as wl
from tests import checker
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

CLIP8 = list(wl.CLIP_8)
CLIP16 = list(wl.CLIP_16)


def _inputs(rows, cols, seed, dist="t4", g_dtype=torch.bfloat16):
    d = wl.random_groups(1, rows * cols, seed=seed, dist=dist, g_dtype=g_dtype, device="cuda")
    return (d["w"].reshape(rows, cols), d["g"].reshape(rows, cols), d["v"].reshape(rows, cols))


def _assert(rep, ema):
    assert ema["ok"], json.dumps(ema)
    assert rep["ok"], json.dumps(rep)


def test_single_matrix_int4(oracle):
    """256x1024 fp32 matrix, INT4, group 128, 8 candidates, fp32 g and r."""
    w_ = wl.workload("single_int4")
    d = wl.make_tensor(w_, w_.tensors[0], device="cuda")
    rep, ema = H.run_int(oracle, d["w"], d["g"], d["v"], bits=4, group_size=128,
                         clip=list(w_.clip), beta2=w_.beta2, r_dtype=torch.float32)
    _assert(rep, ema)


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
@pytest.mark.parametrize("G", [32, 64, 128, 256])
def test_int_bits_groups_ragged(oracle, bits, G):
    # 37 rows x 3 groups: the unit count is not a multiple of the warps
    w, g, v = _inputs(37, 3 * G, seed=bits * 1000 + G)
    rep, ema = H.run_int(oracle, w, g, v, bits=bits, group_size=G, clip=CLIP8)
    _assert(rep, ema)


@pytest.mark.parametrize("K", [1, 5, 8, 13, 16, 32])
def test_int_candidate_counts(oracle, K):
    clip = [round(1.0 - 0.7 * i / max(K - 1, 1), 4) for i in range(K)]
    w, g, v = _inputs(64, 1024, seed=K)
    rep, ema = H.run_int(oracle, w, g, v, bits=3, group_size=128, clip=clip)
    _assert(rep, ema)


def test_int_fp32_gradient_and_output(oracle):
    w, g, v = _inputs(128, 512, seed=77, g_dtype=torch.float32)
    rep, ema = H.run_int(oracle, w, g, v, bits=4, group_size=128, clip=CLIP8,
                         r_dtype=torch.float32)
    _assert(rep, ema)


def test_int_without_gradient_and_optional_outputs(oracle):
    w, _, v = _inputs(64, 512, seed=78)
    v0 = v.clone()
    rep, ema = H.run_int(oracle, w, None, v, bits=3, group_size=128, clip=CLIP8,
                         codes=False, idx=False)
    _assert(rep, ema)
    assert torch.equal(v, v0)


def test_int_degenerate_groups(oracle):
    """Constant groups, all-zero saliency, one salient element, clipped heavy
    tails, exact zeros -- each in its own group of the same launch."""
    G = 128
    w, g, v = _inputs(16, G, seed=79)
    w[0] = 0.0123                       # zero range
    w[1] = -0.5                         # zero range, negative
    v[2] = 0.0; g[2] = 0.0              # all saliency zero
    v[3] = 0.0; g[3] = 0.0; v[3, 17] = 1e-6   # one salient element
    v[4] = 0.0; g[4] = 0.0; v[4, :2] = 1e-6   # two salient elements
    w[5, ::2] = 0.0                     # many exact zeros
    w[6, 5] = 3.0                       # one outlier
    w[7] = torch.linspace(-1, 1, G, device="cuda")  # codes on grid boundaries
    rep, ema = H.run_int(oracle, w, g, v, bits=3, group_size=G, clip=CLIP8)
    _assert(rep, ema)


def test_int_nonfinite_inputs_do_not_fault(oracle):
    w, g, v = _inputs(8, 256, seed=80)
    w[0, 3] = float("nan")
    w[1, 5] = float("inf")
    v[2, 7] = float("nan")
    from paper_2608_13966_gb300 import api
    api.recon_int(w, g, v, bits=3, group_size=128, clip=CLIP8)
    torch.cuda.synchronize()


def test_nvfp4_small_and_degenerate(oracle):
    w, g, v = _inputs(48, 256, seed=81)
    w[0, :16] = 0.0                      # zero block
    v[1, :16] = 0.0; g[1, :16] = 0.0     # zero saliency block
    v[2, :16] = 0.0; g[2, :16] = 0.0; v[2, 3] = 1e-6
    rep, ema = H.run_nvfp4(oracle, w, g, v, clip=CLIP8)
    _assert(rep, ema)


@pytest.mark.parametrize("K", [1, 8, 13, 16, 32])
def test_nvfp4_candidate_counts_supplied_amax(oracle, K):
    clip = [round(1.0 - 0.7 * i / max(K - 1, 1), 4) for i in range(K)]
    w, g, v = _inputs(40, 528, seed=100 + K)     # 1320 blocks: ragged unit count
    rep, ema = H.run_nvfp4(oracle, w, g, v, clip=clip, supply_amax=True,
                           r_dtype=torch.float32)
    _assert(rep, ema)


def _layer(name):
    w_ = wl.workload(name)
    for spec in w_.tensors:
        yield w_, spec, wl.make_tensor(w_, spec, device="cuda")


@pytest.mark.parametrize("name", ["llama_layer_int3", "qwen_layer_int2"])
def test_paper_shaped_layer_int(oracle, name):
    for w_, spec, d in _layer(name):
        rep, ema = H.run_int(oracle, d["w"], d["g"], d["v"], bits=w_.bits,
                             group_size=w_.group, clip=list(w_.clip), beta2=w_.beta2)
        _assert(rep, ema)
        del d
        torch.cuda.empty_cache()


def test_paper_shaped_layer_nvfp4(oracle):
    for w_, spec, d in _layer("llama_layer_nvfp4"):
        rep, ema = H.run_nvfp4(oracle, d["w"], d["g"], d["v"], clip=list(w_.clip),
                               beta2=w_.beta2)
        _assert(rep, ema)
        del d
        torch.cuda.empty_cache()


def test_timeout_path_reports_and_recovers(oracle):
    """A wait on a barrier that nothing signals runs out after 1 ms; the
    kernel records the timeout and returns; the context stays usable."""
    from paper_2608_13966_gb300 import api, quasar
    w, g, v = _inputs(64, 512, seed=82)
    assert quasar.quasar_get_device_status() == quasar.QuasarStatus.OK
    quasar.quasar_debug_force_timeout(1_000_000)
    try:
        api.recon_int(w, g, v, bits=3, group_size=128, clip=CLIP8)
    finally:
        quasar.quasar_debug_force_timeout(0)
    assert quasar.quasar_get_device_status() == quasar.QuasarStatus.ERR_TIMEOUT
    assert quasar.quasar_get_device_status() == quasar.QuasarStatus.OK
    rep, ema = H.run_int(oracle, *_inputs(64, 512, seed=83), bits=3, group_size=128,
                         clip=CLIP8)
    _assert(rep, ema)


def test_int_batch_matches_oracle_and_single_calls(oracle):
    """One launch over tensors of different shapes (group counts that leave
    a partial last unit, a tiny tensor, an empty one) gives, tensor by
    tensor, the oracle's result and bit-for-bit the single-call result."""
    from paper_2608_13966_gb300 import api
    shapes = [(64, 1024), (3, 384), (1, 128), (0, 256), (37, 640), (128, 512)]
    items, copies = [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(max(rows, 1), cols, seed=300 + i)
        w, g, v = w[:rows].contiguous(), g[:rows].contiguous(), v[:rows].contiguous()
        items.append((w, g, v))
        copies.append((w.clone(), g.clone(), v.clone()))
    clip = list(wl.CLIP_8)
    w_h = [H._host(w) for w, _, _ in items]
    g_h = [H._host(g) for _, g, _ in items]
    v_h = [H._host(v) for _, _, v in items]
    outs = api.recon_int_batch(items, bits=3, group_size=128, clip=clip, codes=True)
    singles = [api.recon_int(w, g, v, bits=3, group_size=128, clip=clip, codes=True)
               for (w, g, v) in copies]
    torch.cuda.synchronize()
    for i, (o, s1) in enumerate(zip(outs, singles)):
        for key in ("r", "a", "b", "codes", "cand_idx"):
            assert torch.equal(o[key], s1[key]), (shapes[i], key)
        assert torch.equal(items[i][2], copies[i][2])  # v' identical
        if w_h[i].size == 0:
            continue
        h = oracle.ema(v_h[i], g_h[i], 0.999)
        O = oracle.recon_int(w_h[i], h, 128, 3, clip)
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_int(oracle, w_h[i], h, 3, clip, O, gpu, 128, True)
        ema = checker.check_ema(h, H._host(items[i][2]))
        _assert(rep, ema)


def _set_size(bits, clip):
    """The largest clamp-set size (4, 2 or 1 consecutive candidate slots)
    whose sets all admit one code clamp: J f_max (1 + 1e-3) < (J + 1) f_min
    (1 - 1e-3) on every set, J = (qmax - 1) / 2 (the library's own rule,
    restated to know which kernel should run)."""
    f = [float(np.float32(clip[min(k, len(clip) - 1)])) for k in range(32)]
    J = ((1 << bits) - 1) >> 1
    ok = lambda s, n: J * max(f[s:s + n]) * 1.001 < (J + 1) * min(f[s:s + n]) * 0.999
    # one set of 8 (every slot of each 8) with a single chunk of candidates
    if len(clip) <= 8 and all(ok(s, 8) for s in range(0, 32, 8)):
        return 8
    if all(ok(s, 4) for s in range(0, 32, 4)):
        return 4
    # runs of 3, 3 and 2 of every 8 slots, with a single chunk of candidates
    if len(clip) <= 8 and all(ok(s + o, n) for s in range(0, 32, 8) for o, n in ((0, 3), (3, 3), (6, 2))):
        return 3
    if all(ok(s, 2) for s in range(0, 32, 2)):
        return 2
    return 1


NARROW8 = [1.0, 0.99, 0.98, 0.97, 0.96, 0.95, 0.94, 0.93]
# 16 factors whose INT4 clamp sets hold 2 candidates (4 do not fit; 3-3-2 is
# for a single chunk only)
CLIP16_W = [round(1.0 - 0.03 * i, 4) for i in range(16)]


def _edge_inputs(rows, cols, seed):
    """Ragged t4 weights with the degenerate groups of the edge-case test."""
    w, g, v = _inputs(rows, cols, seed=seed)
    if rows >= 6:
        w[0] = 0.25                                  # zero range
        v[1] = 0.0; g[1] = 0.0                       # all saliency zero
        v[2] = 0.0; g[2] = 0.0; v[2, 17] = 1e-6      # one salient element
        w[3, ::2] = 0.0                              # many exact zeros
        w[4, 5] = 3.0                                # one outlier
        w[5] = torch.linspace(-1, 1, cols, device="cuda")  # codes on grid boundaries
    if rows >= 8:
        w[6] = w[6] * 1e-30                          # tiny range: R near 1e31
        w[7] = w[7] * 1e-3 + 1e3                     # small range far from zero
    return w, g, v


@pytest.mark.parametrize("bits,clip,size", [(1, CLIP8, 8), (2, CLIP8, 8), (3, CLIP8, 4),
                                            (3, CLIP8[:5], 8), (4, NARROW8, 8), (4, CLIP8, 3),
                                            (4, CLIP16_W, 2), (2, wl.CLIP_16, 4), (5, CLIP8, 1)])
@pytest.mark.parametrize("G", [32, 64, 128, 256])
def test_int_hoisted_clamp_equals_per_candidate_clamp(bits, clip, size, G):
    """The batch kernel that clamps |w - c| once per set of 8, 4, 3 or 2
    candidates gives bit for bit the outputs of the kernel that clamps every
    candidate on its own (itself checked against the oracle above), on ragged
    shapes with degenerate groups."""
    from paper_2608_13966_gb300 import api, quasar
    assert _set_size(bits, clip) == size
    shapes = [(37, 3 * G), (8, 2 * G), (1, G)]
    base = [_edge_inputs(r, c, seed=900 + 10 * bits + i) for i, (r, c) in enumerate(shapes)]
    outs = {}
    stats = torch.zeros(8, dtype=torch.int32, device="cuda")
    try:
        for hoist in (True, False):
            quasar.quasar_debug_set_hoist(hoist)
            stats.zero_()
            quasar.quasar_debug_set_stats(stats)
            items = [(w.clone(), g.clone(), v.clone()) for w, g, v in base]
            o = api.recon_int_batch(items, bits=bits, group_size=G, clip=clip, codes=True)
            torch.cuda.synchronize()
            quasar.quasar_debug_set_stats(None)
            outs[hoist] = (o, [v for _, _, v in items])
            # a kernel with sets of several candidates ran exactly when allowed
            assert (int(stats[3]) > 0) == (hoist and size > 1), (hoist, stats.tolist())
    finally:
        quasar.quasar_debug_set_stats(None)
        quasar.quasar_debug_set_hoist(True)
    for i in range(len(shapes)):
        for key in ("r", "a", "b", "codes", "cand_idx"):
            assert torch.equal(outs[True][0][i][key], outs[False][0][i][key]), (shapes[i], key)
        assert torch.equal(outs[True][1][i], outs[False][1][i])


def test_adamw_int_hoisted_clamp_equals_per_candidate_clamp():
    """The fused AdamW + INT3 batch kernel: hoisted and per-candidate clamps
    give the same w', m', v' and outputs bit for bit."""
    from paper_2608_13966_gb300 import api, quasar
    hp = dict(wl.ADAMW_LLAMA_INT3)
    shapes = [(37, 384), (64, 512)]
    base = []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _edge_inputs(rows, cols, seed=950 + i)
        base.append((w, g, wl.first_moment((rows, cols), 950 + i, device="cuda"), v))
    outs = {}
    try:
        for hoist in (True, False):
            quasar.quasar_debug_set_hoist(hoist)
            items = [tuple(t.clone() for t in it) for it in base]
            o = api.adamw_recon_int_batch(items, lr=hp["lr"], beta1=hp["beta1"], beta2=0.999,
                                          eps=hp["eps"], weight_decay=hp["weight_decay"],
                                          step=hp["step"], bits=3, group_size=128, clip=CLIP8,
                                          codes=True)
            torch.cuda.synchronize()
            outs[hoist] = (o, items)
    finally:
        quasar.quasar_debug_set_hoist(True)
    for i in range(len(shapes)):
        for key in ("r", "a", "b", "codes", "cand_idx"):
            assert torch.equal(outs[True][0][i][key], outs[False][0][i][key]), (shapes[i], key)
        for a, b in zip(outs[True][1][i], outs[False][1][i]):
            assert torch.equal(a, b)


def test_nvfp4_batch_matches_oracle_and_single_calls(oracle):
    """One absmax pass, one scale pass and one reconstruction launch over
    tensors of different shapes (one with its amax supplied, a tiny one, an
    empty one) give, tensor by tensor, the oracle's result and bit-for-bit
    the single-call result."""
    from paper_2608_13966_gb300 import api
    shapes = [(48, 512), (3, 48), (0, 64), (37, 528), (1, 16), (64, 1024)]
    items, copies = [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(max(rows, 1), cols, seed=400 + i)
        w, g, v = w[:rows].contiguous(), g[:rows].contiguous(), v[:rows].contiguous()
        amax = w.abs().max().reshape(1).float() if (i == 3 and rows) else None
        items.append((w, g, v, amax))
        copies.append((w.clone(), g.clone(), v.clone(), amax))
    clip = list(wl.CLIP_8)
    hosts = [(H._host(w), H._host(g), H._host(v)) for w, g, v, _ in items]
    outs = api.recon_nvfp4_batch(items, clip=clip, codes=True)
    singles = [api.recon_nvfp4(w, g, v, clip=clip, tensor_amax=amax, codes=True)
               for (w, g, v, amax) in copies]
    torch.cuda.synchronize()
    for i, (o, s1) in enumerate(zip(outs, singles)):
        for key in ("r", "block_scale", "tensor_scale", "codes", "cand_idx"):
            assert torch.equal(o[key], s1[key]), (shapes[i], key)
        assert torch.equal(items[i][2], copies[i][2])  # v' identical
        w_h, g_h, v_h = hosts[i]
        if w_h.size == 0:
            assert float(o["tensor_scale"].cpu()[0]) == 1.0
            continue
        h = oracle.ema(v_h, g_h, 0.999)
        _, s_T = oracle.tensor_scale(w_h)
        O = oracle.recon_nvfp4(w_h, h, s_T, clip)
        gpu = {"r": H._host(o["r"]), "scale": o["block_scale"].cpu().numpy(),
               "tensor_scale": float(o["tensor_scale"].cpu()[0]),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_nvfp4(oracle, w_h, h, clip, s_T, O, gpu, True)
        ema = checker.check_ema(h, H._host(items[i][2]))
        _assert(rep, ema)


def _hp32(hp, beta2):
    """The hyper-parameters as the kernel receives them (fp32 values)."""
    f32 = lambda x: float(np.float32(x))
    return dict(lr=f32(hp["lr"]), beta1=f32(hp["beta1"]), beta2=f32(beta2), eps=f32(hp["eps"]),
                weight_decay=f32(hp["weight_decay"]), step=int(hp["step"]))


def _adamw_case(oracle, shapes, seed0, hp, bits=3, G=128, clip=CLIP8, g_dtype=torch.bfloat16,
                r_dtype=torch.bfloat16):
    """Fused AdamW step + reconstruction over tensors of the given shapes,
    checked tensor by tensor: the AdamW state against the oracle's step, the
    reconstruction against the oracle's Algorithm 1 on the oracle's w', v'."""
    from paper_2608_13966_gb300 import api
    items, hosts = [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(max(rows, 1), cols, seed=seed0 + i, g_dtype=g_dtype)
        m = wl.first_moment((max(rows, 1), cols), seed0 + i, device="cuda")
        w, g, m, v = (t[:rows].contiguous() for t in (w, g, m, v))
        items.append((w, g, m, v))
        hosts.append(tuple(H._host(t) for t in (w, g, m, v)))
    outs = api.adamw_recon_int_batch(items, lr=hp["lr"], beta1=hp["beta1"], beta2=0.999,
                                     eps=hp["eps"], weight_decay=hp["weight_decay"],
                                     step=hp["step"], bits=bits, group_size=G, clip=clip,
                                     r_dtype=r_dtype, codes=True)
    torch.cuda.synchronize()
    for i, (o, (w_h, g_h, m_h, v_h)) in enumerate(zip(outs, hosts)):
        if w_h.size == 0:
            continue
        hp32 = _hp32(hp, 0.999)
        w1, m1, v1 = oracle.adamw(w_h, g_h, m_h, v_h, **hp32)
        w_gpu, _, m_gpu, v_gpu = (H._host(t) for t in items[i])
        st = checker.check_adamw(w_h, g_h, m_h, hp32, w1, m1, v1, w_gpu, m_gpu, v_gpu)
        assert st["ok"], (shapes[i], json.dumps(st))
        O = oracle.recon_int(w1, v1, G, bits, clip)
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_int(oracle, w1, v1, bits, clip, O, gpu, G,
                                r_dtype == torch.bfloat16)
        assert rep["ok"], (shapes[i], json.dumps(rep))


ADAMW_PAPER = dict(wl.ADAMW_LLAMA_INT3)


def test_adamw_recon_int_batch_matches_oracle(oracle):
    """Tensors of different shapes (a partial last unit, a tiny tensor, an
    empty one) at the paper's Llama INT3 learning rate."""
    _adamw_case(oracle, [(64, 1024), (3, 384), (0, 256), (37, 640), (128, 512)], 500,
                ADAMW_PAPER)


@pytest.mark.parametrize("hp", [
    dict(lr=1e-3, beta1=0.9, eps=1e-8, weight_decay=0.1, step=1),    # first step, large lr
    dict(lr=3e-5, beta1=0.0, eps=1e-6, weight_decay=0.0, step=7),    # no momentum, no decay
    dict(lr=0.0, beta1=0.9, eps=1e-8, weight_decay=0.01, step=100),  # w unchanged
])
def test_adamw_recon_int_hyperparameters(oracle, hp):
    _adamw_case(oracle, [(48, 512)], 600, hp)


@pytest.mark.parametrize("bits,G,K", [(2, 64, 16), (4, 256, 8), (8, 32, 5)])
def test_adamw_recon_int_settings(oracle, bits, G, K):
    clip = [round(1.0 - 0.7 * i / max(K - 1, 1), 4) for i in range(K)]
    _adamw_case(oracle, [(40, 4 * G), (7, 2 * G)], 700 + bits, ADAMW_PAPER, bits=bits, G=G,
                clip=clip, g_dtype=torch.float32, r_dtype=torch.float32)


def test_adamw_layer_matches_oracle(oracle):
    """A full Llama-3.1-8B-shaped layer (all seven linear weights) in one
    fused launch, as the training step runs it."""
    from paper_2608_13966_gb300 import api
    w_ = wl.workload("llama_layer_int3_adamw")
    hp = w_.adamw
    ds = [wl.make_tensor(w_, spec, device="cuda") for spec in w_.tensors]
    hosts = [tuple(H._host(d[k]) for k in ("w", "g", "m", "v")) for d in ds]
    outs = api.adamw_recon_int_batch([(d["w"], d["g"], d["m"], d["v"]) for d in ds],
                                     lr=hp["lr"], beta1=hp["beta1"], beta2=w_.beta2,
                                     eps=hp["eps"], weight_decay=hp["weight_decay"],
                                     step=hp["step"], bits=w_.bits, group_size=w_.group,
                                     clip=list(w_.clip), codes=True)
    torch.cuda.synchronize()
    for spec, d, o, (w_h, g_h, m_h, v_h) in zip(w_.tensors, ds, outs, hosts):
        hp32 = _hp32(hp, w_.beta2)
        w1, m1, v1 = oracle.adamw(w_h, g_h, m_h, v_h, **hp32)
        st = checker.check_adamw(w_h, g_h, m_h, hp32, w1, m1, v1, H._host(d["w"]),
                                 H._host(d["m"]), H._host(d["v"]))
        assert st["ok"], (spec.name, json.dumps(st))
        O = oracle.recon_int(w1, v1, w_.group, w_.bits, list(w_.clip))
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_int(oracle, w1, v1, w_.bits, list(w_.clip), O, gpu, w_.group, True)
        assert rep["ok"], (spec.name, json.dumps(rep))


# ------------------------------------------------ variants (quasar_options)

@pytest.mark.parametrize("mode", ["ema_squared", "uniform"])
def test_int_saliency_variants(oracle, mode):
    """h = v'^2 (App. A.3) and h = 1 (the scale-search-only ablation): the
    fit and the search use the variant's h while v is still updated to v'."""
    from paper_2608_13966_gb300 import api
    w, g, v = _inputs(64, 1024, seed=900 + len(mode))
    w_h, g_h, v_h = H._host(w), H._host(g), H._host(v)
    o = api.recon_int_batch([(w, g, v)], bits=3, group_size=128, clip=CLIP8, codes=True,
                            saliency=mode)[0]
    torch.cuda.synchronize()
    v1 = oracle.ema(v_h, g_h, 0.999)
    h = oracle.saliency(v1, mode)
    O = oracle.recon_int(w_h, h, 128, 3, CLIP8)
    gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
           "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
    _assert(checker.check_int(oracle, w_h, h, 3, CLIP8, O, gpu, 128, True),
            checker.check_ema(v1, H._host(v)))


@pytest.mark.parametrize("mode", ["ema_squared", "uniform"])
def test_nvfp4_saliency_variants(oracle, mode):
    from paper_2608_13966_gb300 import api
    w, g, v = _inputs(48, 512, seed=910 + len(mode))
    w_h, g_h, v_h = H._host(w), H._host(g), H._host(v)
    o = api.recon_nvfp4_batch([(w, g, v)], clip=CLIP8, codes=True, saliency=mode)[0]
    torch.cuda.synchronize()
    v1 = oracle.ema(v_h, g_h, 0.999)
    h = oracle.saliency(v1, mode)
    _, s_T = oracle.tensor_scale(w_h)
    O = oracle.recon_nvfp4(w_h, h, s_T, CLIP8)
    gpu = {"r": H._host(o["r"]), "scale": o["block_scale"].cpu().numpy(),
           "tensor_scale": float(o["tensor_scale"].cpu()[0]),
           "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
    _assert(checker.check_nvfp4(oracle, w_h, h, CLIP8, s_T, O, gpu, True),
            checker.check_ema(v1, H._host(v)))


@pytest.mark.parametrize("bits,G", [(1, 32), (2, 64), (3, 128), (3, 32), (4, 256), (5, 128),
                                    (8, 64)])
def test_int_packed_codes(oracle, bits, G):
    """The packed deployment format: read back with the oracle's unpacking,
    the codes pass the same parity check as one-byte codes, and equal the
    one-byte codes of the same call bit for bit.  Tensors with a partial
    last unit and a one-group tensor are included."""
    from paper_2608_13966_gb300 import api
    clip = CLIP8
    shapes = [(37, 3 * G), (1, G), (16, 8 * G)]
    items, copies, hosts = [], [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(rows, cols, seed=950 + 10 * bits + i)
        items.append((w, g, v))
        copies.append((w.clone(), g.clone(), v.clone()))
        hosts.append((H._host(w), H._host(g), H._host(v)))
    packed = api.recon_int_batch(items, bits=bits, group_size=G, clip=clip, codes=True,
                                 packed_codes=True)
    plain = api.recon_int_batch(copies, bits=bits, group_size=G, clip=clip, codes=True)
    torch.cuda.synchronize()
    for (rows, cols), o, o1, (w_h, g_h, v_h) in zip(shapes, packed, plain, hosts):
        n = rows * cols
        assert o["codes"].numel() == n * bits // 8
        q = oracle.unpack_int_codes(o["codes"].cpu().numpy(), bits, n)
        assert np.array_equal(q, o1["codes"].cpu().numpy().ravel())
        h = oracle.ema(v_h, g_h, 0.999)
        O = oracle.recon_int(w_h, h, G, bits, clip)
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": q, "idx": o["cand_idx"].cpu().numpy()}
        _assert(checker.check_int(oracle, w_h, h, bits, clip, O, gpu, G, True),
                checker.check_ema(h, H._host(items[shapes.index((rows, cols))][2])))


def test_nvfp4_packed_codes(oracle):
    from paper_2608_13966_gb300 import api
    shapes = [(48, 512), (3, 48), (1, 16)]
    items, copies, hosts = [], [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(rows, cols, seed=990 + i)
        items.append((w, g, v))
        copies.append((w.clone(), g.clone(), v.clone()))
        hosts.append((H._host(w), H._host(g), H._host(v)))
    packed = api.recon_nvfp4_batch(items, clip=CLIP8, codes=True, packed_codes=True)
    plain = api.recon_nvfp4_batch(copies, clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    for (rows, cols), o, o1, (w_h, g_h, v_h) in zip(shapes, packed, plain, hosts):
        n = rows * cols
        assert o["codes"].numel() == n // 2
        q = oracle.unpack_nvfp4_codes(o["codes"].cpu().numpy())
        assert np.array_equal(q, o1["codes"].cpu().numpy().ravel())
        h = oracle.ema(v_h, g_h, 0.999)
        _, s_T = oracle.tensor_scale(w_h)
        O = oracle.recon_nvfp4(w_h, h, s_T, CLIP8)
        gpu = {"r": H._host(o["r"]), "scale": o["block_scale"].cpu().numpy(),
               "tensor_scale": float(o["tensor_scale"].cpu()[0]), "codes": q,
               "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_nvfp4(oracle, w_h, h, CLIP8, s_T, O, gpu, True)
        assert rep["ok"], json.dumps(rep)


def test_adamw_with_options(oracle):
    """The fused AdamW step with h = v'^2 and packed codes."""
    from paper_2608_13966_gb300 import api
    hp = ADAMW_PAPER
    w, g, v = _inputs(40, 512, seed=1001)
    m = wl.first_moment((40, 512), 1001, device="cuda")
    w_h, g_h, m_h, v_h = (H._host(t) for t in (w, g, m, v))
    o = api.adamw_recon_int_batch([(w, g, m, v)], lr=hp["lr"], beta1=hp["beta1"], beta2=0.999,
                                  eps=hp["eps"], weight_decay=hp["weight_decay"], step=hp["step"],
                                  bits=3, group_size=128, clip=CLIP8, codes=True,
                                  saliency="ema_squared", packed_codes=True)[0]
    torch.cuda.synchronize()
    hp32 = _hp32(hp, 0.999)
    w1, m1, v1 = oracle.adamw(w_h, g_h, m_h, v_h, **hp32)
    st = checker.check_adamw(w_h, g_h, m_h, hp32, w1, m1, v1, H._host(w), H._host(m), H._host(v))
    assert st["ok"], json.dumps(st)
    h = oracle.saliency(v1, "ema_squared")
    O = oracle.recon_int(w1, h, 128, 3, CLIP8)
    q = oracle.unpack_int_codes(o["codes"].cpu().numpy(), 3, w_h.size)
    gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
           "codes": q, "idx": o["cand_idx"].cpu().numpy()}
    rep = checker.check_int(oracle, w1, h, 3, CLIP8, O, gpu, 128, True)
    assert rep["ok"], json.dumps(rep)


# ------------------------------------------------ Rubin INT3 LUT (App. B)

def _lut_run(oracle, shapes, seed0, clip, saliency="ema", packed=False, g_dtype=torch.bfloat16,
             r_dtype=torch.bfloat16, g_none=False):
    from paper_2608_13966_gb300 import api
    items, hosts = [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(rows, cols, seed=seed0 + i, g_dtype=g_dtype)
        if g_none:
            g = None
        items.append((w, g, v))
        hosts.append((H._host(w), None if g is None else H._host(g), H._host(v)))
    outs = api.recon_lut_batch(items, clip=clip, codes=True, saliency=saliency,
                               packed_codes=packed, r_dtype=r_dtype)
    torch.cuda.synchronize()
    for (rows, cols), o, (w_h, g_h, v_h), it in zip(shapes, outs, hosts, items):
        v1 = oracle.ema(v_h, g_h, 0.999) if g_h is not None else v_h
        h = oracle.saliency(v1, saliency)
        w2, h2 = w_h.reshape(rows, cols), h.reshape(rows, cols)
        O = oracle.recon_lut(w2, h2, clip)
        if packed:
            nb = rows * cols // 512
            qb = oracle.unpack_int_codes(o["codes"].cpu().numpy(), 3, nb * 512).reshape(nb, 512)
            # block order -> tensor layout
            codes = qb.reshape(rows // 8, cols // 64, 8, 64).transpose(0, 2, 1, 3).reshape(rows, cols)
        else:
            codes = o["codes"].cpu().numpy()
        gpu = {"r": H._host(o["r"]), "book": o["book"].cpu().numpy(), "codes": codes,
               "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_lut(oracle, w2, h2, clip, O, gpu)
        assert rep["ok"], json.dumps(rep)
        ema = checker.check_ema(v1, H._host(it[2]))
        assert ema["ok"], json.dumps(ema)


def test_lut_batch_shapes(oracle):
    """Several tensors of different block counts, 8 candidates."""
    _lut_run(oracle, [(64, 512), (8, 64), (16, 1024), (24, 192)], 1100, CLIP8)


@pytest.mark.parametrize("K", [1, 5, 16, 32])
def test_lut_candidate_counts(oracle, K):
    clip = [round(1.0 - 0.7 * i / max(K - 1, 1), 4) for i in range(K)]
    _lut_run(oracle, [(32, 512)], 1200 + K, clip)


def test_lut_variants(oracle):
    """fp32 gradient and output, no gradient, h = v'^2, uniform h, packed
    indices."""
    _lut_run(oracle, [(16, 256)], 1300, CLIP8, g_dtype=torch.float32, r_dtype=torch.float32)
    _lut_run(oracle, [(16, 256)], 1301, CLIP8, g_none=True)
    _lut_run(oracle, [(16, 256)], 1302, CLIP8, saliency="ema_squared")
    _lut_run(oracle, [(16, 256)], 1303, CLIP8, saliency="uniform")
    _lut_run(oracle, [(16, 256), (8, 64)], 1304, CLIP8, packed=True)


def test_lut_degenerate_blocks(oracle):
    from paper_2608_13966_gb300 import api
    w, g, v = _inputs(16, 256, seed=1400)
    w[:8, :64] = 0.0123                  # zero range
    v[:8, 64:128] = 0.0
    g[:8, 64:128] = 0.0                  # all saliency zero
    w[8:, :64] = torch.linspace(-1, 1, 512, device="cuda").reshape(8, 64)  # on grid boundaries
    w[8:, 64:128] = 0.0
    w[8, 64] = 1.0                       # one outlier, everything else equal
    w_h, g_h, v_h = H._host(w), H._host(g), H._host(v)
    o = api.recon_lut_batch([(w, g, v)], clip=CLIP8, codes=True)[0]
    torch.cuda.synchronize()
    h = oracle.ema(v_h, g_h, 0.999).reshape(16, 256)
    O = oracle.recon_lut(w_h.reshape(16, 256), h, CLIP8)
    gpu = {"r": H._host(o["r"]), "book": o["book"].cpu().numpy(), "codes": o["codes"].cpu().numpy(),
           "idx": o["cand_idx"].cpu().numpy()}
    rep = checker.check_lut(oracle, w_h.reshape(16, 256), h, CLIP8, O, gpu)
    assert rep["ok"], json.dumps(rep)


def test_lut_paper_shaped_layer(oracle):
    """A full Llama-3.1-8B-shaped layer (7 tensors, 426k blocks) in one launch."""
    from paper_2608_13966_gb300 import api
    w_ = wl.workload("llama_layer_int3")
    ds = [wl.make_tensor(w_, spec, device="cuda") for spec in w_.tensors]
    hosts = [tuple(H._host(d[k]) for k in ("w", "g", "v")) for d in ds]
    outs = api.recon_lut_batch([(d["w"], d["g"], d["v"]) for d in ds], clip=list(w_.clip),
                               codes=True)
    torch.cuda.synchronize()
    for spec, d, o, (w_h, g_h, v_h) in zip(w_.tensors, ds, outs, hosts):
        h = oracle.ema(v_h, g_h, w_.beta2).reshape(spec.rows, spec.cols)
        O = oracle.recon_lut(w_h.reshape(spec.rows, spec.cols), h, list(w_.clip))
        gpu = {"r": H._host(o["r"]), "book": o["book"].cpu().numpy(),
               "codes": o["codes"].cpu().numpy(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_lut(oracle, w_h.reshape(spec.rows, spec.cols), h, list(w_.clip), O, gpu)
        assert rep["ok"], (spec.name, json.dumps(rep))


@pytest.mark.parametrize("hp", [ADAMW_PAPER, dict(lr=1e-3, beta1=0.9, eps=1e-8,
                                                   weight_decay=0.1, step=1)])
def test_adamw_recon_nvfp4_batch_matches_oracle(oracle, hp):
    """AdamW step (w', m', v' and the absmax of w' in one pass), then NVFP4
    reconstruction of w' with h = v': tensor by tensor against the oracle's
    AdamW step followed by its Sec. 4.2 search on the oracle's w', v'."""
    from paper_2608_13966_gb300 import api
    shapes = [(48, 512), (3, 48), (0, 64), (37, 528)]
    items, hosts = [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(max(rows, 1), cols, seed=1500 + i)
        m = wl.first_moment((max(rows, 1), cols), 1500 + i, device="cuda")
        w, g, m, v = (t[:rows].contiguous() for t in (w, g, m, v))
        items.append((w, g, m, v))
        hosts.append(tuple(H._host(t) for t in (w, g, m, v)))
    outs = api.adamw_recon_nvfp4_batch(items, lr=hp["lr"], beta1=hp["beta1"], beta2=0.999,
                                       eps=hp["eps"], weight_decay=hp["weight_decay"],
                                       step=hp["step"], clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    hp32 = _hp32(hp, 0.999)
    for (rows, cols), o, it, (w_h, g_h, m_h, v_h) in zip(shapes, outs, items, hosts):
        if w_h.size == 0:
            assert float(o["tensor_scale"].cpu()[0]) == 1.0
            continue
        w1, m1, v1 = oracle.adamw(w_h, g_h, m_h, v_h, **hp32)
        st = checker.check_adamw(w_h, g_h, m_h, hp32, w1, m1, v1, H._host(it[0]), H._host(it[2]),
                                 H._host(it[3]))
        assert st["ok"], json.dumps(st)
        _, s_T = oracle.tensor_scale(w1)
        O = oracle.recon_nvfp4(w1, v1, s_T, CLIP8)
        gpu = {"r": H._host(o["r"]), "scale": o["block_scale"].cpu().numpy(),
               "tensor_scale": float(o["tensor_scale"].cpu()[0]),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_nvfp4(oracle, w1, v1, CLIP8, s_T, O, gpu, True)
        assert rep["ok"], json.dumps(rep)


# ------------------------------------------------ symmetric integer codes

def _sym_case(oracle, shapes, seed0, bits, G, clip, saliency="ema", packed=False,
              g_dtype=torch.bfloat16, r_dtype=torch.bfloat16, g_none=False):
    from paper_2608_13966_gb300 import api
    items, hosts = [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(rows, cols, seed=seed0 + i, g_dtype=g_dtype)
        if g_none:
            g = None
        items.append((w, g, v))
        hosts.append((H._host(w), None if g is None else H._host(g), H._host(v)))
    outs = api.recon_int_batch(items, bits=bits, group_size=G, clip=clip, codes=True,
                               symmetric=True, saliency=saliency, packed_codes=packed,
                               r_dtype=r_dtype)
    torch.cuda.synchronize()
    for (rows, cols), o, (w_h, g_h, v_h), it in zip(shapes, outs, hosts, items):
        v1 = oracle.ema(v_h, g_h, 0.999) if g_h is not None else v_h
        h = oracle.saliency(v1, saliency)
        O = oracle.recon_sym(w_h, h, G, bits, clip)
        codes = (oracle.unpack_int_codes(o["codes"].cpu().numpy(), bits, w_h.size) if packed
                 else o["codes"].cpu().numpy().ravel())
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": codes, "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_sym(oracle, w_h, h, bits, clip, O, gpu, G, r_dtype == torch.bfloat16)
        assert rep["ok"], json.dumps(rep)
        assert checker.check_ema(v1, H._host(it[2]))["ok"]


@pytest.mark.parametrize("bits,G", [(2, 64), (3, 128), (4, 128), (4, 32), (8, 256)])
def test_sym_bits_groups(oracle, bits, G):
    _sym_case(oracle, [(37, 3 * G), (1, G), (64, 8 * G)], 1600 + bits * 10, bits, G, CLIP8)


@pytest.mark.parametrize("K", [1, 13, 32])
def test_sym_candidate_counts(oracle, K):
    clip = [round(1.0 - 0.7 * i / max(K - 1, 1), 4) for i in range(K)]
    _sym_case(oracle, [(64, 1024)], 1700 + K, 4, 128, clip)


def test_sym_variants(oracle):
    _sym_case(oracle, [(16, 512)], 1800, 4, 128, CLIP8, g_dtype=torch.float32, r_dtype=torch.float32)
    _sym_case(oracle, [(16, 512)], 1801, 4, 128, CLIP8, g_none=True)
    _sym_case(oracle, [(16, 512)], 1802, 3, 128, CLIP8, saliency="ema_squared")
    _sym_case(oracle, [(16, 512)], 1803, 3, 128, CLIP8, saliency="uniform")
    _sym_case(oracle, [(37, 384), (1, 128)], 1804, 3, 128, CLIP8, packed=True)


def test_sym_degenerate_groups(oracle):
    from paper_2608_13966_gb300 import api
    G = 128
    w, g, v = _inputs(8, G, seed=1900)
    w[0] = 0.0                                   # max |w| = 0
    v[1] = 0.0; g[1] = 0.0                       # all saliency zero
    v[2] = 0.0; g[2] = 0.0; v[2, 5] = 1e-6; w[2, 5] = 1e-7   # the only salient element codes to 0
    w[3] = torch.linspace(-1, 1, G, device="cuda")            # many exact half-levels
    w_h, g_h, v_h = H._host(w), H._host(g), H._host(v)
    o = api.recon_int_batch([(w, g, v)], bits=3, group_size=G, clip=CLIP8, codes=True,
                            symmetric=True)[0]
    torch.cuda.synchronize()
    h = oracle.ema(v_h, g_h, 0.999)
    O = oracle.recon_sym(w_h, h, G, 3, CLIP8)
    gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
           "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
    rep = checker.check_sym(oracle, w_h, h, 3, CLIP8, O, gpu, G, True)
    assert rep["ok"], json.dumps(rep)


def test_sym_paper_shaped_layer(oracle):
    """A Llama-3.1-8B-shaped layer, INT4 symmetric, group 128."""
    from paper_2608_13966_gb300 import api
    w_ = wl.workload("llama_layer_int3")
    ds = [wl.make_tensor(w_, spec, device="cuda") for spec in w_.tensors]
    hosts = [tuple(H._host(d[k]) for k in ("w", "g", "v")) for d in ds]
    outs = api.recon_int_batch([(d["w"], d["g"], d["v"]) for d in ds], bits=4, group_size=128,
                               clip=list(w_.clip), codes=True, symmetric=True)
    torch.cuda.synchronize()
    for spec, o, (w_h, g_h, v_h) in zip(w_.tensors, outs, hosts):
        h = oracle.ema(v_h, g_h, w_.beta2)
        O = oracle.recon_sym(w_h, h, 128, 4, list(w_.clip))
        gpu = {"r": H._host(o["r"]), "a": o["a"].cpu().numpy(), "b": o["b"].cpu().numpy(),
               "codes": o["codes"].cpu().numpy().ravel(), "idx": o["cand_idx"].cpu().numpy()}
        rep = checker.check_sym(oracle, w_h, h, 4, list(w_.clip), O, gpu, 128, True)
        assert rep["ok"], (spec.name, json.dumps(rep))


@pytest.mark.parametrize("path", ["nvfp4", "lut", "sym", "adamw"])
def test_timeout_path_of_every_kernel(oracle, path):
    """Each kernel's bounded wait: a barrier nothing arrives at runs out after
    1 ms, the kernel records the timeout and returns, the status reports it
    once, and the next call is correct."""
    from paper_2608_13966_gb300 import api, quasar
    w, g, v = _inputs(64, 512, seed=2000)
    assert quasar.quasar_get_device_status() == quasar.QuasarStatus.OK
    quasar.quasar_debug_force_timeout(1_000_000)
    try:
        if path == "nvfp4":
            api.recon_nvfp4_batch([(w, g, v)], clip=CLIP8)
        elif path == "lut":
            api.recon_lut_batch([(w, g, v)], clip=CLIP8)
        elif path == "sym":
            api.recon_int_batch([(w, g, v)], bits=3, group_size=128, clip=CLIP8, symmetric=True)
        else:
            m = wl.first_moment((64, 512), 2000, device="cuda")
            api.adamw_recon_int_batch([(w, g, m, v)], lr=1e-5, step=1, bits=3, group_size=128,
                                      clip=CLIP8)
    finally:
        quasar.quasar_debug_force_timeout(0)
    assert quasar.quasar_get_device_status() == quasar.QuasarStatus.ERR_TIMEOUT
    assert quasar.quasar_get_device_status() == quasar.QuasarStatus.OK
    rep, ema = H.run_int(oracle, *_inputs(64, 512, seed=2001), bits=3, group_size=128, clip=CLIP8)
    _assert(rep, ema)


def test_adamw_recon_nvfp4_fp32_gradient_and_options(oracle):
    """The AdamW + NVFP4 step with an fp32 gradient, h = v'^2 and packed codes."""
    from paper_2608_13966_gb300 import api
    hp = dict(wl.ADAMW_NVFP4)
    w, g, v = _inputs(40, 512, seed=2100, g_dtype=torch.float32)
    m = wl.first_moment((40, 512), 2100, device="cuda")
    w_h, g_h, m_h, v_h = (H._host(t) for t in (w, g, m, v))
    o = api.adamw_recon_nvfp4_batch([(w, g, m, v)], lr=hp["lr"], beta1=hp["beta1"], beta2=0.999,
                                    eps=hp["eps"], weight_decay=hp["weight_decay"],
                                    step=hp["step"], clip=CLIP8, codes=True,
                                    saliency="ema_squared", packed_codes=True,
                                    r_dtype=torch.float32)[0]
    torch.cuda.synchronize()
    hp32 = _hp32(hp, 0.999)
    w1, m1, v1 = oracle.adamw(w_h, g_h, m_h, v_h, **hp32)
    st = checker.check_adamw(w_h, g_h, m_h, hp32, w1, m1, v1, H._host(w), H._host(m), H._host(v))
    assert st["ok"], json.dumps(st)
    h = oracle.saliency(v1, "ema_squared")
    _, s_T = oracle.tensor_scale(w1)
    O = oracle.recon_nvfp4(w1, h, s_T, CLIP8)
    gpu = {"r": H._host(o["r"]), "scale": o["block_scale"].cpu().numpy(),
           "tensor_scale": float(o["tensor_scale"].cpu()[0]),
           "codes": oracle.unpack_nvfp4_codes(o["codes"].cpu().numpy()),
           "idx": o["cand_idx"].cpu().numpy()}
    rep = checker.check_nvfp4(oracle, w1, h, CLIP8, s_T, O, gpu, False)
    assert rep["ok"], json.dumps(rep)


def test_more_than_one_launch_of_tensors(oracle):
    """300 tensors in one batch call: more than a launch holds (256), so the
    call makes two launches; every tensor matches the oracle."""
    from paper_2608_13966_gb300 import api
    items, hosts = [], []
    for i in range(300):
        w, g, v = _inputs(2, 128, seed=3000 + i)
        items.append((w, g, v))
        hosts.append((H._host(w), H._host(g), H._host(v)))
    outs = api.recon_int_batch(items, bits=3, group_size=128, clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    w_h = np.concatenate([h[0] for h in hosts])
    hh = np.concatenate([oracle.ema(h[2], h[1], 0.999) for h in hosts])
    O = oracle.recon_int(w_h, hh, 128, 3, CLIP8)
    gpu = {"r": np.concatenate([H._host(o["r"]) for o in outs]),
           "a": np.concatenate([o["a"].cpu().numpy() for o in outs]),
           "b": np.concatenate([o["b"].cpu().numpy() for o in outs]),
           "codes": np.concatenate([o["codes"].cpu().numpy().ravel() for o in outs]),
           "idx": np.concatenate([o["cand_idx"].cpu().numpy() for o in outs])}
    rep = checker.check_int(oracle, w_h, hh, 3, CLIP8, O, gpu, 128, True)
    assert rep["ok"], json.dumps(rep)
