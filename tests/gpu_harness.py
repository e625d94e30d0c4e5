"""Runs the CUDA path and the oracle on the same seeded inputs and checks them.

Inputs are drawn on the GPU (or given), copied to the host BEFORE the call
(the call updates v in place), the CUDA library runs through the C ABI, and
the oracle recomputes everything from the host copies.
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_13966_gb300 import api
from tests import checker


def _host(t):
    return None if t is None else t.detach().float().cpu().numpy().ravel()


def run_int(oracle, w, g, v, *, bits, group_size, clip, beta2=0.999, r_dtype=torch.bfloat16,
            codes=True, idx=True):
    """w, g, v: CUDA tensors [rows, cols].  Returns (int report, ema report)."""
    w_h, g_h, v_h = _host(w), _host(g), _host(v)
    out = api.recon_int(w, g, v, bits=bits, group_size=group_size, clip=clip, beta2=beta2,
                        r_dtype=r_dtype, codes=codes, cand_idx=idx)
    torch.cuda.synchronize()
    gpu = {"r": _host(out["r"]), "a": out["a"].cpu().numpy(), "b": out["b"].cpu().numpy(),
           "codes": out["codes"].cpu().numpy().ravel() if codes else None,
           "idx": out["cand_idx"].cpu().numpy() if idx else None}
    h_ref = oracle.ema(v_h, g_h, beta2) if g is not None else v_h
    O = oracle.recon_int(w_h, h_ref, group_size, bits, clip)
    rep = checker.check_int(oracle, w_h, h_ref, bits, clip, O, gpu, group_size,
                            r_dtype == torch.bfloat16)
    ema = checker.check_ema(h_ref, _host(v))
    return rep, ema


def run_nvfp4(oracle, w, g, v, *, clip, beta2=0.999, r_dtype=torch.bfloat16, codes=True,
              idx=True, supply_amax=False):
    w_h, g_h, v_h = _host(w), _host(g), _host(v)
    amax_t = None
    if supply_amax:
        amax_t = w.abs().max().reshape(1).float()
    out = api.recon_nvfp4(w, g, v, clip=clip, beta2=beta2, tensor_amax=amax_t, r_dtype=r_dtype,
                          codes=codes, cand_idx=idx)
    torch.cuda.synchronize()
    gpu = {"r": _host(out["r"]), "scale": out["block_scale"].cpu().numpy(),
           "tensor_scale": float(out["tensor_scale"].cpu()[0]),
           "codes": out["codes"].cpu().numpy().ravel() if codes else None,
           "idx": out["cand_idx"].cpu().numpy() if idx else None}
    h_ref = oracle.ema(v_h, g_h, beta2) if g is not None else v_h
    _, s_T = oracle.tensor_scale(w_h)
    O = oracle.recon_nvfp4(w_h, h_ref, s_T, clip)
    rep = checker.check_nvfp4(oracle, w_h, h_ref, clip, s_T, O, gpu, r_dtype == torch.bfloat16)
    ema = checker.check_ema(h_ref, _host(v))
    return rep, ema
