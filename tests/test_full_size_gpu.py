"""Parity at full size: every tensor of the 32-layer Llama-3.1-8B-shaped
model (6.98e9 weights resident on the device), reconstructed through the
C-ABI calls and launch configuration that ``bench.py`` times, checked against
the oracle on a seeded sample of groups (blocks) from every tensor, together
with the in-place EMA update of those groups (and, for the fused AdamW
workload, the in-place AdamW step of w and m)."""
import numpy as np
import pytest
import torch

import bench
from paper_2608_13966_gb300 import workloads as WL
from tests import checker

SAMPLES_PER_TENSOR = 48


def _sample(model, unit, seed):
    rng = np.random.default_rng(seed)
    out = []
    for d in model.tensors:
        n_units = d["spec"].numel // unit
        idx = np.sort(rng.choice(n_units, size=min(SAMPLES_PER_TENSOR, n_units), replace=False))
        sel = torch.as_tensor(idx, device="cuda")
        m = d["m"].view(-1, unit)[sel].cpu() if "m" in d else None
        out.append((sel, d["w"].view(-1, unit)[sel].cpu(), d["g"].view(-1, unit)[sel].float().cpu(),
                    d["v"].view(-1, unit)[sel].cpu(), m))
    return out


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["llama_int3", "llama_nvfp4", "llama_int3_adamw"])
def test_full_model_sampled(oracle, name):
    wl = WL.workload(name)
    unit = wl.group if wl.fmt == "int" else 16
    model = bench.Model(wl, torch.device("cuda"))
    samples = _sample(model, unit, seed=1234)
    stream = torch.cuda.Stream()
    step = bench.Step(model, wl, stream)
    with torch.cuda.stream(stream):
        step.run()
    torch.cuda.synchronize()

    bad = []
    f32 = lambda x: float(np.float32(x))
    for d, (sel, w_s, g_s, v_s, m_s) in zip(model.tensors, samples):
        w = w_s.numpy().ravel()
        v_gpu = d["v"].view(-1, unit)[sel].cpu().numpy().ravel()
        if wl.adamw:
            hp = wl.adamw
            hp32 = dict(lr=f32(hp["lr"]), beta1=f32(hp["beta1"]), beta2=f32(wl.beta2),
                        eps=f32(hp["eps"]), weight_decay=f32(hp["weight_decay"]),
                        step=int(hp["step"]))
            g_h, m_h = g_s.numpy().ravel(), m_s.numpy().ravel()
            w, m1, h = oracle.adamw(w, g_h, m_h, v_s.numpy().ravel(), **hp32)
            ema = checker.check_adamw(w_s.numpy().ravel(), g_h, m_h, hp32, w, m1, h,
                                      d["w"].view(-1, unit)[sel].cpu().numpy().ravel(),
                                      d["m"].view(-1, unit)[sel].cpu().numpy().ravel(), v_gpu)
        else:
            h = oracle.ema(v_s.numpy().ravel(), g_s.numpy().ravel(), wl.beta2)
            ema = checker.check_ema(h, v_gpu)
        r = d["r"].view(-1, unit)[sel].float().cpu().numpy().ravel()
        if wl.fmt == "int":
            O = oracle.recon_int(w, h, wl.group, wl.bits, list(wl.clip))
            gpu = {"r": r, "a": d["a"][sel].cpu().numpy(), "b": d["b"][sel].cpu().numpy(),
                   "codes": None, "idx": d["idx"][sel].cpu().numpy()}
            rep = checker.check_int(oracle, w, h, wl.bits, list(wl.clip), O, gpu, wl.group, True)
        else:
            amax = float(d["w"].abs().max().cpu())
            _, s_T = oracle.tensor_scale(np.array([amax], dtype=np.float32))
            O = oracle.recon_nvfp4(w, h, s_T, list(wl.clip))
            gpu = {"r": r, "scale": d["scale"][sel].cpu().numpy(),
                   "tensor_scale": float(d["ts"].cpu()[0]), "codes": None,
                   "idx": d["idx"][sel].cpu().numpy()}
            rep = checker.check_nvfp4(oracle, w, h, list(wl.clip), s_T, O, gpu, True)
        if not (rep["ok"] and ema["ok"]):
            bad.append((d["spec"].name, rep, ema))
    del model
    torch.cuda.empty_cache()
    assert not bad, bad[:3]
