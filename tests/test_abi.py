"""C-ABI checks that need no GPU: the library builds for sm_103a, loads,
exports every function include/quasar.h declares, and rejects bad arguments
on the host without launching anything."""
import ctypes
import os
import re

import pytest

from paper_2608_13966_gb300 import build as qbuild
from paper_2608_13966_gb300 import quasar as Q

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "quasar.h")

# Fake, 16-byte aligned device addresses: validation must reject before use.
A, B, C, D, E, F = (0x10000000 * (i + 1) for i in range(6))
CLIP = [1.0, 0.9, 0.8]


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(quasar_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    qbuild.build()
    return Q.load(build_if_missing=False)


def test_header_and_binding_agree():
    assert declared_functions() == sorted(Q.PROTOTYPES)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert Q.quasar_version() >= 100


def test_status_strings(lib):
    for st in Q.QuasarStatus:
        assert Q.quasar_status_string(st) == "QUASAR_" + st.name
    assert Q.quasar_status_string(99) == "QUASAR_ERR_UNKNOWN"


def _int(**kw):
    args = dict(w=A, g=B, v=C, beta2=0.999, bits=3, group_size=128, clip=CLIP, rows=4,
                cols=256, r=D, codes=None, a=E, b=F, cand_idx=None, stream=0,
                g_dtype=Q.BF16, r_dtype=Q.BF16)
    args.update(kw)
    return Q.quasar_recon_int(**args)


@pytest.mark.parametrize("kw,expect", [
    (dict(bits=0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(bits=9), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(group_size=100, cols=300), Q.QuasarStatus.ERR_UNSUPPORTED),
    (dict(cols=200), Q.QuasarStatus.ERR_INVALID_ARG),          # cols % group_size
    (dict(beta2=1.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(beta2=-0.1), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(clip=[]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(clip=[1.0] * 33), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(clip=[1.0, 0.0]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(clip=[1.5]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(clip=[float("nan")]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(w=None), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(v=None), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(r=None), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(a=None), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(w=A + 4), Q.QuasarStatus.ERR_INVALID_ARG),           # misaligned
    (dict(g=B + 8), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(codes=D + 8), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(rows=-1), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(rows=1 << 40, cols=1 << 40), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(r_dtype=7), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(r=A + 512), Q.QuasarStatus.ERR_INVALID_ARG),         # r overlaps w
    (dict(a=C + 64), Q.QuasarStatus.ERR_INVALID_ARG),          # a overlaps v
    (dict(cand_idx=B + 16), Q.QuasarStatus.ERR_INVALID_ARG),   # idx overlaps g
    (dict(rows=0), Q.QuasarStatus.OK),                         # empty: no-op
])
def test_int_argument_validation(lib, kw, expect):
    assert _int(**kw) == expect


def _nv(**kw):
    args = dict(w=A, g=B, v=C, beta2=0.999, clip=CLIP, rows=4, cols=256, tensor_amax=None,
                r=D, codes=None, block_scale=E, tensor_scale=F, cand_idx=None, stream=0,
                g_dtype=Q.BF16, r_dtype=Q.BF16)
    args.update(kw)
    return Q.quasar_recon_nvfp4(**args)


@pytest.mark.parametrize("kw,expect", [
    (dict(cols=250), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(block_scale=None), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(tensor_scale=None), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(tensor_scale=F + 2), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(tensor_amax=F), Q.QuasarStatus.ERR_INVALID_ARG),     # amax aliases tensor_scale
    (dict(block_scale=A + 16), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(beta2=2.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(clip=[0.5] * 40), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(w=A + 4), Q.QuasarStatus.ERR_INVALID_ARG),
])
def test_nvfp4_argument_validation(lib, kw, expect):
    assert _nv(**kw) == expect


def test_amax_argument_validation(lib):
    assert Q.quasar_tensor_amax(A, -1, B, stream=0) == Q.QuasarStatus.ERR_INVALID_ARG
    assert Q.quasar_tensor_amax(A, 16, None, stream=0) == Q.QuasarStatus.ERR_INVALID_ARG
    assert Q.quasar_tensor_amax(A + 4, 16, B, stream=0) == Q.QuasarStatus.ERR_INVALID_ARG


def test_product_path_has_no_oracle_dependency():
    """The CUDA library and its binding never reference the oracle."""
    pkg = os.path.join(ROOT, "paper_2608_13966_gb300")
    for dirpath, _, files in os.walk(pkg):
        if "_build" in dirpath:
            continue
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, fn)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", text, re.M), fn
                assert "quasar_oracle" not in text and "qo_" not in text, fn


def _desc(**kw):
    d = dict(w=A, g=B, v=C, r=D, codes=None, a=E, b=F, cand_idx=None, rows=4, cols=256)
    d.update(kw)
    return d


def test_int_batch_argument_validation(lib):
    st = Q.QuasarStatus
    call = lambda items, **kw: Q.quasar_recon_int_batch(
        items, kw.get("beta2", 0.999), kw.get("bits", 3), kw.get("group_size", 128), CLIP, stream=0)
    assert Q.quasar_recon_int_batch([], 0.999, 3, 128, CLIP, stream=0) == st.OK  # nothing to do
    assert call([_desc(rows=0), _desc(cols=0)]) == st.OK                         # all empty
    assert call([_desc(), _desc(g=None)]) == st.ERR_INVALID_ARG                  # mixed gradients
    assert call([_desc(), _desc(a=None)]) == st.ERR_INVALID_ARG                  # bad second tensor
    assert call([_desc(), _desc(cols=200)]) == st.ERR_INVALID_ARG                # cols % group_size
    assert call([_desc(), _desc(r=A)]) == st.ERR_INVALID_ARG                     # output aliases w
    assert call([_desc()], bits=9) == st.ERR_INVALID_ARG
    assert call([_desc()], group_size=48) == st.ERR_UNSUPPORTED
    n = ctypes.c_void_p(None)
    assert Q.load().quasar_recon_int_batch(n, 2, Q.BF16, 0.999, 3, 128, None, 0, Q.BF16, None) == st.ERR_INVALID_ARG


def _ndesc(**kw):
    d = dict(w=A, g=B, v=C, tensor_amax=None, r=D, codes=None, block_scale=E, tensor_scale=F,
             cand_idx=None, rows=4, cols=256)
    d.update(kw)
    return d


def test_nvfp4_batch_argument_validation(lib):
    st = Q.QuasarStatus
    call = lambda items: Q.quasar_recon_nvfp4_batch(items, 0.999, CLIP, stream=0)
    assert call([]) == st.OK
    assert call([_ndesc(), _ndesc(g=None)]) == st.ERR_INVALID_ARG      # mixed gradients
    assert call([_ndesc(), _ndesc(block_scale=None)]) == st.ERR_INVALID_ARG
    assert call([_ndesc(), _ndesc(cols=40)]) == st.ERR_INVALID_ARG     # cols % 16
    assert call([_ndesc(), _ndesc(tensor_scale=None)]) == st.ERR_INVALID_ARG
    assert call([_ndesc(), _ndesc(r=C)]) == st.ERR_INVALID_ARG         # output aliases v


M_ADDR = 0x70000000


def _adesc(**kw):
    d = dict(w=A, g=B, m=M_ADDR, v=C, r=D, codes=None, a=E, b=F, cand_idx=None, rows=4, cols=256)
    d.update(kw)
    return d


@pytest.mark.parametrize("kw,expect", [
    (dict(items=[]), Q.QuasarStatus.OK),
    (dict(items=[_adesc(rows=0, g=None, m=None)]), Q.QuasarStatus.OK),       # empty: no-op
    (dict(items=[_adesc(g=None)]), Q.QuasarStatus.ERR_INVALID_ARG),         # gradient required
    (dict(items=[_adesc(m=None)]), Q.QuasarStatus.ERR_INVALID_ARG),         # m required
    (dict(items=[_adesc(m=M_ADDR + 4)]), Q.QuasarStatus.ERR_INVALID_ARG),   # misaligned m
    (dict(items=[_adesc(m=A + 1024)]), Q.QuasarStatus.ERR_INVALID_ARG),     # m overlaps w
    (dict(items=[_adesc(m=C)]), Q.QuasarStatus.ERR_INVALID_ARG),            # m is v
    (dict(items=[_adesc(g=C + 16)]), Q.QuasarStatus.ERR_INVALID_ARG),       # g overlaps v
    (dict(items=[_adesc(r=M_ADDR + 64)]), Q.QuasarStatus.ERR_INVALID_ARG),  # r overlaps m
    (dict(items=[_adesc(a=M_ADDR)]), Q.QuasarStatus.ERR_INVALID_ARG),       # a overlaps m
    (dict(items=[_adesc(), _adesc(cols=200)]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(lr=-1.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(lr=float("inf")), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(beta1=1.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(beta2=1.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(eps=0.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(weight_decay=-0.1), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(step=0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(bits=0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(group_size=48), Q.QuasarStatus.ERR_UNSUPPORTED),
])
def test_adamw_batch_argument_validation(lib, kw, expect):
    args = dict(items=[_adesc()], lr=1e-5, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0,
                step=1, bits=3, group_size=128)
    args.update(kw)
    items = args.pop("items")
    assert Q.quasar_adamw_recon_int_batch(items, clip=CLIP, stream=0, **args) == expect


def test_options_validation(lib):
    st = Q.QuasarStatus
    ok_opt = Q.options("ema_squared", True)
    call = lambda opt: Q.quasar_recon_int_batch_ex([_desc(rows=0)], 0.999, 3, 128, CLIP, opt, stream=0)
    assert call(None) == st.OK
    assert call(ok_opt) == st.OK
    assert call(Q.options(7)) == st.ERR_INVALID_ARG                  # unknown saliency
    assert call(Q.options("ema", 5)) == st.ERR_INVALID_ARG           # unknown codes layout
    nd = [_ndesc(rows=0)]
    assert Q.quasar_recon_nvfp4_batch_ex(nd, 0.999, CLIP, Q.options(3), stream=0) == st.ERR_INVALID_ARG
    # packed INT3 codes of 4 x 256 weights take 384 bytes: a buffer whose
    # last 16 of them overlap v is rejected (nothing here may pass
    # validation: the addresses are fake)
    assert Q.quasar_recon_int_batch_ex([_desc(codes=C - 368)], 0.999, 3, 128, CLIP,
                                       Q.options("ema", True), stream=0) == st.ERR_INVALID_ARG
    assert Q.quasar_recon_nvfp4_batch_ex([_ndesc(codes=C - 496)], 0.999, CLIP,
                                         Q.options("ema", True), stream=0) == st.ERR_INVALID_ARG


def _ldesc(**kw):
    d = dict(w=A, g=B, v=C, r=D, codes=None, book=E, cand_idx=None, rows=8, cols=128)
    d.update(kw)
    return d


@pytest.mark.parametrize("kw,expect", [
    (dict(items=[]), Q.QuasarStatus.OK),
    (dict(items=[_ldesc(rows=0)]), Q.QuasarStatus.OK),                      # empty: no-op
    (dict(items=[_ldesc(rows=12)]), Q.QuasarStatus.ERR_INVALID_ARG),        # rows % 8
    (dict(items=[_ldesc(cols=96)]), Q.QuasarStatus.ERR_INVALID_ARG),        # cols % 64
    (dict(items=[_ldesc(book=None)]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(items=[_ldesc(book=E + 8)]), Q.QuasarStatus.ERR_INVALID_ARG),     # misaligned
    (dict(items=[_ldesc(book=C + 64)]), Q.QuasarStatus.ERR_INVALID_ARG),    # book overlaps v
    (dict(items=[_ldesc(r=A + 256)]), Q.QuasarStatus.ERR_INVALID_ARG),      # r overlaps w
    (dict(items=[_ldesc(), _ldesc(g=None)]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(items=[_ldesc()], beta2=1.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(items=[_ldesc()], opt=Q.options(9)), Q.QuasarStatus.ERR_INVALID_ARG),
])
def test_lut_argument_validation(lib, kw, expect):
    items = kw.pop("items")
    assert Q.quasar_recon_lut_batch(items, kw.get("beta2", 0.999), CLIP, kw.get("opt"),
                                    stream=0) == expect


def _andesc(**kw):
    d = dict(w=A, g=B, m=M_ADDR, v=C, r=D, codes=None, block_scale=E, tensor_scale=F,
             cand_idx=None, rows=4, cols=256)
    d.update(kw)
    return d


@pytest.mark.parametrize("kw,expect", [
    (dict(items=[]), Q.QuasarStatus.OK),
    (dict(items=[_andesc(g=None)]), Q.QuasarStatus.ERR_INVALID_ARG),       # gradient required
    (dict(items=[_andesc(m=None)]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(items=[_andesc(m=A + 64)]), Q.QuasarStatus.ERR_INVALID_ARG),     # m overlaps w
    (dict(items=[_andesc(r=M_ADDR + 64)]), Q.QuasarStatus.ERR_INVALID_ARG),  # r overlaps m
    (dict(items=[_andesc(cols=40)]), Q.QuasarStatus.ERR_INVALID_ARG),      # cols % 16
    (dict(items=[_andesc(tensor_scale=None)]), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(lr=-1.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(eps=0.0), Q.QuasarStatus.ERR_INVALID_ARG),
    (dict(step=0), Q.QuasarStatus.ERR_INVALID_ARG),
])
def test_adamw_nvfp4_argument_validation(lib, kw, expect):
    args = dict(items=[_andesc()], lr=1e-5, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0,
                step=1)
    args.update(kw)
    items = args.pop("items")
    assert Q.quasar_adamw_recon_nvfp4_batch(items, clip=CLIP, stream=0, **args) == expect


def test_symmetric_option_validation(lib):
    st = Q.QuasarStatus
    sym = Q.options(symmetric=True)
    assert Q.quasar_recon_int_batch_ex([_desc(rows=0)], 0.999, 3, 128, CLIP, sym, stream=0) == st.OK
    assert Q.quasar_recon_int_batch_ex([_desc()], 0.999, 1, 128, CLIP, sym, stream=0) == st.ERR_INVALID_ARG
    assert Q.quasar_recon_int_batch_ex([_desc()], 0.999, 3, 128, CLIP, Q.options(symmetric=2),
                                       stream=0) == st.ERR_INVALID_ARG
    assert Q.quasar_adamw_recon_int_batch([_adesc()], 1e-5, 0.9, 0.999, 1e-8, 0.0, 1, 3, 128, CLIP,
                                          options=sym, stream=0) == st.ERR_UNSUPPORTED
    assert Q.quasar_recon_nvfp4_batch_ex([_ndesc()], 0.999, CLIP, sym, stream=0) == st.ERR_INVALID_ARG
    assert Q.quasar_recon_lut_batch([_ldesc()], 0.999, CLIP, sym, stream=0) == st.ERR_INVALID_ARG
