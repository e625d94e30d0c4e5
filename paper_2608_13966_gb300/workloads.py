"""Seeded synthetic workloads for the QUASAR reconstruction.

This module only draws random inputs (latent weights ``w``, gradients ``g``,
EMA state ``v``) with the shapes and value distributions of the paper's
models; it holds none of the reconstruction's arithmetic.  The CUDA path
(``quasar``), the benchmark and the tests all take their inputs from here, and
the oracle receives the very same bits copied to the host.

The paper trains Llama-3.1-8B-Instruct and Qwen3 models (Sec. 6.1); their
weights are not available here, so the tensors below are synthetic stand-ins
with the same linear-layer shapes:

* Llama-3.1-8B decoder layer: q 4096x4096, k/v 1024x4096, o 4096x4096,
  gate/up 14336x4096, down 4096x14336 (``nn.Linear`` layout [out, in]).
* Qwen3-8B decoder layer: hidden 4096, 32 query / 8 key-value heads of
  dimension 128, MLP 12288.

Distributions: latent weights are Student-t (heavy-tailed like trained LLM
weights) scaled by 0.02, optionally with a sparse set of x20 outliers; the
STE gradient is N(0, 1e-3^2) (bf16 where the training run keeps it in bf16);
the Adam second moment is lognormal(-14, 2), i.e. values around 1e-6 spread
over several decades.  Student-t(nu) is drawn from its definition,
Z / sqrt(chi2_nu / nu) with chi2_nu the sum of nu squared standard normals.

Every tensor has its own generator seeded with ``seed*1000 + index`` where
``index = 7*layer + j`` (j over q, k, v, o, gate, up, down), and the draws are
taken in the order w, warm-up gradient (first workload only), g, v.  Adam's
first moment m, for the workloads that take an AdamW step, comes from a
generator of its own (seed ``seed*1000 + index + 500000``): N(0, (3e-4)^2),
a smoothed gradient of the gradient's scale.

AdamW workloads use the paper's Llama-3.1-8B INT3 learning rate 2e-5
(Sec. 6.1 setup) and, where the paper gives none, PyTorch's AdamW defaults
(beta1 0.9, eps 1e-8, weight decay 0.01); the step counter is 100, a point
where both bias corrections still differ from 1.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch

LLAMA31_8B_LAYER = (
    ("q_proj", 4096, 4096),
    ("k_proj", 1024, 4096),
    ("v_proj", 1024, 4096),
    ("o_proj", 4096, 4096),
    ("gate_proj", 14336, 4096),
    ("up_proj", 14336, 4096),
    ("down_proj", 4096, 14336),
)

QWEN3_8B_LAYER = (
    ("q_proj", 4096, 4096),
    ("k_proj", 1024, 4096),
    ("v_proj", 1024, 4096),
    ("o_proj", 4096, 4096),
    ("gate_proj", 12288, 4096),
    ("up_proj", 12288, 4096),
    ("down_proj", 4096, 12288),
)

CLIP_8 = tuple(round(1.00 - 0.05 * i, 2) for i in range(8))    # 1.00 ... 0.65
CLIP_16 = tuple(round(1.00 - 0.05 * i, 2) for i in range(16))  # 1.00 ... 0.25
CLIP_PAPER = tuple(round(0.30 + 0.05 * i, 2) for i in range(15))  # 0.30 ... 1.00

# AdamW hyper-parameters of the fused-step workloads
ADAMW_LLAMA_INT3 = {"lr": 2e-5, "beta1": 0.9, "eps": 1e-8, "weight_decay": 0.01, "step": 100}
# the paper's NVFP4 QAD learning rate (Sec. 6.1)
ADAMW_NVFP4 = {"lr": 1e-6, "beta1": 0.9, "eps": 1e-8, "weight_decay": 0.01, "step": 100}


@dataclass(frozen=True)
class TensorSpec:
    name: str
    rows: int
    cols: int
    layer: int
    index: int  # 7*layer + position in the layer

    @property
    def numel(self) -> int:
        return self.rows * self.cols


@dataclass(frozen=True)
class Workload:
    """One benchmark / parity workload."""

    name: str
    fmt: str                  # "int", "nvfp4" or "lut"
    bits: int                 # integer bit width (4 for NVFP4's E2M1 codes)
    group: int                # group size (16 for NVFP4 blocks)
    clip: tuple
    beta2: float
    g_dtype: torch.dtype
    r_dtype: torch.dtype
    with_codes: bool
    tensors: tuple            # TensorSpec, ...
    w_dist: str               # "normal", "t4", "t3_outliers"
    v_dist: str               # "warm_g2" or "lognormal"
    notes: str = ""
    extra: dict = field(default_factory=dict, compare=False)
    adamw: dict = field(default_factory=dict, compare=False)  # AdamW step, if any
    symmetric: bool = False   # symmetric integer codes

    @property
    def numel(self) -> int:
        return sum(t.numel for t in self.tensors)


def _layer_tensors(layout, n_layers: int) -> tuple:
    out = []
    for layer in range(n_layers):
        for j, (name, rows, cols) in enumerate(layout):
            out.append(TensorSpec(f"layers.{layer}.{name}", rows, cols, layer, 7 * layer + j))
    return tuple(out)


def workload(name: str) -> Workload:
    """Named workloads.  ``llama_int{2,3,4}`` / ``llama_nvfp4`` cover the
    32-layer Llama-3.1-8B-shaped model (all linear weights, ~6.98e9)."""
    f32, bf16 = torch.float32, torch.bfloat16
    if name == "single_int4":
        return Workload(name, "int", 4, 128, CLIP_8, 0.999, f32, f32, True,
                        (TensorSpec("matrix", 256, 1024, 0, 0),), "normal", "warm_g2",
                        "single fp32 256x1024, INT4 asymmetric, group 128")
    if name == "llama_layer_int3":
        return Workload(name, "int", 3, 128, CLIP_8, 0.999, bf16, bf16, True,
                        _layer_tensors(LLAMA31_8B_LAYER, 1), "t4", "lognormal",
                        "one Llama-3.1-8B-shaped layer, INT3 group 128")
    if name == "qwen_layer_int2":
        return Workload(name, "int", 2, 64, CLIP_16, 0.999, bf16, bf16, True,
                        _layer_tensors(QWEN3_8B_LAYER, 1), "t3_outliers", "lognormal",
                        "one Qwen3-8B-shaped layer, INT2 group 64, 16 candidates")
    if name == "llama_layer_nvfp4":
        return Workload(name, "nvfp4", 4, 16, CLIP_8, 0.999, bf16, bf16, True,
                        _layer_tensors(LLAMA31_8B_LAYER, 1), "t4", "lognormal",
                        "one Llama-3.1-8B-shaped layer, NVFP4")
    for bits in (2, 3, 4):
        if name == f"llama_int{bits}":
            return Workload(name, "int", bits, 128, CLIP_8, 0.999, bf16, bf16, False,
                            _layer_tensors(LLAMA31_8B_LAYER, 32), "t4", "lognormal",
                            f"all linear weights of a 32-layer Llama-3.1-8B-shaped model, "
                            f"INT{bits} group 128")
    if name == "llama_layer_int3_adamw":
        return Workload(name, "int", 3, 128, CLIP_8, 0.999, bf16, bf16, True,
                        _layer_tensors(LLAMA31_8B_LAYER, 1), "t4", "lognormal",
                        "one Llama-3.1-8B-shaped layer, AdamW step + INT3 group 128",
                        adamw=dict(ADAMW_LLAMA_INT3))
    if name == "llama_int3_adamw":
        return Workload(name, "int", 3, 128, CLIP_8, 0.999, bf16, bf16, False,
                        _layer_tensors(LLAMA31_8B_LAYER, 32), "t4", "lognormal",
                        "AdamW step fused with INT3 group-128 reconstruction of all linear "
                        "weights of a 32-layer Llama-3.1-8B-shaped model",
                        adamw=dict(ADAMW_LLAMA_INT3))
    if name == "llama_layer_nvfp4_adamw":
        return Workload(name, "nvfp4", 4, 16, CLIP_8, 0.999, bf16, bf16, True,
                        _layer_tensors(LLAMA31_8B_LAYER, 1), "t4", "lognormal",
                        "one Llama-3.1-8B-shaped layer, AdamW step + NVFP4",
                        adamw=dict(ADAMW_NVFP4))
    if name == "llama_nvfp4_adamw":
        return Workload(name, "nvfp4", 4, 16, CLIP_8, 0.999, bf16, bf16, False,
                        _layer_tensors(LLAMA31_8B_LAYER, 32), "t4", "lognormal",
                        "AdamW step then NVFP4 reconstruction of all linear weights of a 32-layer "
                        "Llama-3.1-8B-shaped model", adamw=dict(ADAMW_NVFP4))
    if name == "llama_int4_sym":
        return Workload(name, "int", 4, 128, CLIP_8, 0.999, bf16, bf16, False,
                        _layer_tensors(LLAMA31_8B_LAYER, 32), "t4", "lognormal",
                        "all linear weights of a 32-layer Llama-3.1-8B-shaped model, symmetric INT4 "
                        "group 128", symmetric=True)
    if name == "llama_layer_int4_sym":
        return Workload(name, "int", 4, 128, CLIP_8, 0.999, bf16, bf16, True,
                        _layer_tensors(LLAMA31_8B_LAYER, 1), "t4", "lognormal",
                        "one Llama-3.1-8B-shaped layer, symmetric INT4 group 128", symmetric=True)
    if name == "llama_layer_lut":
        return Workload(name, "lut", 3, 512, CLIP_8, 0.999, bf16, bf16, True,
                        _layer_tensors(LLAMA31_8B_LAYER, 1), "t4", "lognormal",
                        "one Llama-3.1-8B-shaped layer, Rubin INT3 lookup table (8x64 blocks)")
    if name == "llama_lut":
        return Workload(name, "lut", 3, 512, CLIP_8, 0.999, bf16, bf16, False,
                        _layer_tensors(LLAMA31_8B_LAYER, 32), "t4", "lognormal",
                        "all linear weights of a 32-layer Llama-3.1-8B-shaped model, Rubin INT3 "
                        "lookup table (8x64 blocks, 8 E4M3 entries)")
    if name == "llama_nvfp4":
        return Workload(name, "nvfp4", 4, 16, CLIP_8, 0.999, bf16, bf16, False,
                        _layer_tensors(LLAMA31_8B_LAYER, 32), "t4", "lognormal",
                        "all linear weights of a 32-layer Llama-3.1-8B-shaped model, NVFP4")
    raise KeyError(name)


WORKLOADS = ("single_int4", "llama_layer_int3", "qwen_layer_int2", "llama_layer_nvfp4",
             "llama_layer_int3_adamw", "llama_layer_nvfp4_adamw", "llama_layer_lut", "llama_int2",
             "llama_int3", "llama_int4", "llama_nvfp4", "llama_int3_adamw", "llama_nvfp4_adamw",
             "llama_lut", "llama_int4_sym", "llama_layer_int4_sym")


def _student_t(gen, shape, nu: int, device) -> torch.Tensor:
    z = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
    chi2 = torch.zeros(shape, device=device, dtype=torch.float32)
    for _ in range(nu):
        x = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        chi2.addcmul_(x, x)
    return z / torch.sqrt(chi2 / nu)


def first_moment(shape, seed: int, device="cpu") -> torch.Tensor:
    """Adam's first moment m ~ N(0, (3e-4)^2), fp32, from its own generator."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed + 500000)
    return (3e-4 * torch.randn(shape, generator=gen, device=device, dtype=torch.float32)).contiguous()


def make_tensor(wl: Workload, spec: TensorSpec, device="cpu", seed: int = 0) -> dict:
    """Draw (w, g, v) for one tensor.  w and v are fp32, g is wl.g_dtype."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed * 1000 + spec.index)
    shape = (spec.rows, spec.cols)

    if wl.w_dist == "normal":
        w = 0.02 * torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
    elif wl.w_dist == "t4":
        w = 0.02 * _student_t(gen, shape, 4, device)
    elif wl.w_dist == "t3_outliers":
        w = 0.02 * _student_t(gen, shape, 3, device)
        mask = torch.rand(shape, generator=gen, device=device) < 0.001
        w = torch.where(mask, w * 20.0, w)
    else:
        raise ValueError(wl.w_dist)

    if wl.v_dist == "warm_g2":
        g_warm = 1e-3 * torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        g = 1e-3 * torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        v = g_warm * g_warm
    elif wl.v_dist == "lognormal":
        g = 1e-3 * torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
        v = torch.exp(-14.0 + 2.0 * torch.randn(shape, generator=gen, device=device,
                                                dtype=torch.float32))
    else:
        raise ValueError(wl.v_dist)

    out = {"w": w.contiguous(), "g": g.to(wl.g_dtype).contiguous(), "v": v.contiguous()}
    if wl.adamw:
        out["m"] = first_moment(shape, seed * 1000 + spec.index, device)
    return out


def random_groups(n_groups: int, group: int, *, seed: int = 0, dist: str = "t4",
                  g_dtype=torch.float32, device="cpu") -> dict:
    """Small flat inputs (n_groups*group elements) for parity cases."""
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    shape = (n_groups * group,)
    if dist == "normal":
        w = 0.02 * torch.randn(shape, generator=gen, device=device)
    elif dist == "t4":
        w = 0.02 * _student_t(gen, shape, 4, device)
    elif dist == "t3_outliers":
        w = 0.02 * _student_t(gen, shape, 3, device)
        mask = torch.rand(shape, generator=gen, device=device) < 0.001
        w = torch.where(mask, w * 20.0, w)
    else:
        raise ValueError(dist)
    g = 1e-3 * torch.randn(shape, generator=gen, device=device)
    v = torch.exp(-14.0 + 2.0 * torch.randn(shape, generator=gen, device=device))
    return {"w": w.contiguous(), "g": g.to(g_dtype).contiguous(), "v": v.contiguous()}
