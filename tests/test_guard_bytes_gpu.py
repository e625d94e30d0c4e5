"""Out-of-bounds writes, checked with guard bytes (compute-sanitizer is not
available): every buffer an entry point writes -- and every input it reads
or updates in place -- lives inside a larger device buffer whose bytes
before and after it hold a known pattern.  After the call the pattern must
be intact, and the interior must hold exactly what the same call returns on
ordinary tensors (those outputs are checked against the oracle by the
parity tests; the integer and NVFP4 interiors are checked against the oracle
here as well).

The shapes are ragged on purpose: group counts that leave the last unit of
a warp partly empty, a single group, a single row, one clip candidate, and
batches of 255, 256 and 257 tensors (one and two launches)."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_13966_gb300 import api, quasar
from paper_2608_13966_gb300 import workloads as WL
from tests import checker
from tests import gpu_harness as H

PAD = 256           # guard bytes on each side (keeps the interior 16-byte aligned)
FILL = 0xA5
CLIP8 = list(WL.CLIP_8)


class Guarded:
    """A device buffer of n bytes with PAD guard bytes on each side."""

    def __init__(self, shape, dtype, init=None):
        self.shape = tuple(shape)
        self.dtype = dtype
        n = int(np.prod(self.shape)) * torch.tensor([], dtype=dtype).element_size()
        self.n = n
        self.buf = torch.full((PAD + n + PAD,), FILL, dtype=torch.uint8, device="cuda")
        self.t = self.buf[PAD:PAD + n].view(dtype).view(self.shape)
        if init is not None:
            self.t.copy_(init)

    def intact(self):
        return bool((self.buf[:PAD] == FILL).all()) and bool((self.buf[PAD + self.n:] == FILL).all())


def _inputs(rows, cols, seed, g_dtype=torch.bfloat16):
    d = WL.random_groups(rows * cols // 16, 16, seed=seed, device="cuda", g_dtype=g_dtype)
    return (d["w"].reshape(rows, cols), d["g"].reshape(rows, cols), d["v"].reshape(rows, cols))


def _damaged(bufs):
    """Indices of the buffers whose guard bytes changed."""
    return [i for i, b in enumerate(bufs) if b is not None and not b.intact()]


# shapes (rows, cols) at group size G: 8-group units left partly empty, one
# group, one row
def _int_shapes(G):
    return [(37, 2 * G), (1, G), (1, 5 * G), (13, 3 * G)]


@pytest.mark.gpu
@pytest.mark.parametrize("bits,G,clip", [(3, 128, CLIP8), (4, 64, CLIP8), (2, 32, [1.0]),
                                         (3, 256, CLIP8[:5])])
def test_recon_int_guards(oracle, bits, G, clip):
    """quasar_recon_int: one tensor, every output and input guarded."""
    for i, (rows, cols) in enumerate(_int_shapes(G)):
        w, g, v = _inputs(rows, cols, seed=3000 + i)
        w_h, g_h, v_h = H._host(w), H._host(g), H._host(v)
        W, Gb, V = Guarded(w.shape, w.dtype, w), Guarded(g.shape, g.dtype, g), Guarded(v.shape, v.dtype, v)
        n_groups = rows * cols // G
        R = Guarded((rows, cols), torch.bfloat16)
        C = Guarded((rows, cols), torch.uint8)
        A = Guarded((n_groups,), torch.float32)
        B = Guarded((n_groups,), torch.float32)
        K = Guarded((n_groups,), torch.uint8)
        st = quasar.quasar_recon_int(W.t, Gb.t, V.t, 0.999, bits, G, clip, rows, cols, R.t, C.t,
                                     A.t, B.t, K.t)
        assert st == quasar.QuasarStatus.OK
        torch.cuda.synchronize()
        assert not _damaged([W, Gb, V, R, C, A, B, K]), (rows, cols)
        h = oracle.ema(v_h, g_h, 0.999)
        O = oracle.recon_int(w_h, h, G, bits, clip)
        gpu = {"r": H._host(R.t), "a": A.t.cpu().numpy(), "b": B.t.cpu().numpy(),
               "codes": C.t.cpu().numpy().ravel(), "idx": K.t.cpu().numpy()}
        rep = checker.check_int(oracle, w_h, h, bits, clip, O, gpu, G, True)
        assert rep["ok"], rep
        assert checker.check_ema(h, H._host(V.t))["ok"]
        assert torch.equal(W.t, w) and torch.equal(Gb.t, g)


def _int_batch_descs(shapes, G, seed, adam=False, packed_bits=0):
    """Guarded buffers and descriptors of a batch; returns (descs, bufs,
    originals) with originals the unguarded input copies."""
    descs, bufs, orig = [], [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(rows, cols, seed=seed + i)
        m = WL.first_moment((rows, cols), seed + i, device="cuda") if adam else None
        n_groups = rows * cols // G
        W, Gb, V = Guarded(w.shape, w.dtype, w), Guarded(g.shape, g.dtype, g), Guarded(v.shape, v.dtype, v)
        M = Guarded(m.shape, m.dtype, m) if adam else None
        R = Guarded((rows, cols), torch.bfloat16)
        C = (Guarded((rows * cols * packed_bits // 8,), torch.uint8) if packed_bits
             else Guarded((rows, cols), torch.uint8))
        A = Guarded((n_groups,), torch.float32)
        B = Guarded((n_groups,), torch.float32)
        K = Guarded((n_groups,), torch.uint8)
        d = {"w": W.t, "g": Gb.t, "v": V.t, "r": R.t, "codes": C.t, "a": A.t, "b": B.t,
             "cand_idx": K.t, "rows": rows, "cols": cols}
        if adam:
            d["m"] = M.t
        descs.append(d)
        bufs.append([W, Gb, V, M, R, C, A, B, K])
        orig.append((w, g, m, v) if adam else (w, g, v))
    return descs, bufs, orig


def _check_batch_against(bufs, outs, orig, adam=False):
    for i, (bb, o) in enumerate(zip(bufs, outs)):
        W, Gb, V, M, R, C, A, B, K = bb
        assert not _damaged(bb), i
        assert torch.equal(R.t, o["r"]) and torch.equal(A.t, o["a"]) and torch.equal(B.t, o["b"])
        assert torch.equal(K.t, o["cand_idx"]) and torch.equal(C.t.view(-1), o["codes"].view(-1))
        if adam:
            w, g, m, v = orig[i]
            assert torch.equal(W.t, w) and torch.equal(M.t, m) and torch.equal(V.t, v)
        else:
            w, g, v = orig[i]
            assert torch.equal(V.t, v) and torch.equal(W.t, w)


@pytest.mark.gpu
@pytest.mark.parametrize("n_tensors", [3, 255, 256, 257])
def test_recon_int_batch_guards(n_tensors):
    """quasar_recon_int_batch over ragged tensors, 255-257 of them (257 is
    two launches): guards intact, outputs equal the ordinary call's."""
    G = 128
    shapes = [(1 + (i * 7) % 5, G * (1 + i % 3)) for i in range(n_tensors)]
    descs, bufs, orig = _int_batch_descs(shapes, G, seed=4000)
    st = quasar.quasar_recon_int_batch(descs, 0.999, 3, G, CLIP8)
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    # the ordinary call updates the original v in place, as the guarded call
    # updated its guarded copy
    outs = api.recon_int_batch(orig, bits=3, group_size=G, clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    _check_batch_against(bufs, outs, orig)


@pytest.mark.gpu
@pytest.mark.parametrize("opt", ["packed", "symmetric", "uniform"])
def test_recon_int_batch_ex_guards(opt):
    G, bits = 64, 3
    shapes = [(13, 3 * G), (1, G), (9, 5 * G)]
    descs, bufs, orig = _int_batch_descs(shapes, G, seed=4100, packed_bits=bits if opt == "packed" else 0)
    o = quasar.options(saliency="uniform" if opt == "uniform" else "ema",
                       packed_codes=opt == "packed", symmetric=opt == "symmetric")
    st = quasar.quasar_recon_int_batch_ex(descs, 0.999, bits, G, CLIP8, o)
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    outs = api.recon_int_batch(orig, bits=bits, group_size=G,
                               clip=CLIP8, codes=True, packed_codes=opt == "packed",
                               symmetric=opt == "symmetric",
                               saliency="uniform" if opt == "uniform" else "ema")
    torch.cuda.synchronize()
    _check_batch_against(bufs, outs, orig)


@pytest.mark.gpu
def test_adamw_recon_int_batch_guards():
    G = 128
    shapes = [(37, 2 * G), (1, G), (5, 3 * G)]
    descs, bufs, orig = _int_batch_descs(shapes, G, seed=4200, adam=True)
    hp = dict(WL.ADAMW_LLAMA_INT3)
    st = quasar.quasar_adamw_recon_int_batch(descs, hp["lr"], hp["beta1"], 0.999, hp["eps"],
                                             hp["weight_decay"], hp["step"], 3, G, CLIP8)
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    # the ordinary call updates the original w, m, v in place, as the
    # guarded call updated their guarded copies
    outs = api.adamw_recon_int_batch(orig, lr=hp["lr"], beta1=hp["beta1"], beta2=0.999, eps=hp["eps"],
                                     weight_decay=hp["weight_decay"], step=hp["step"], bits=3,
                                     group_size=G, clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    _check_batch_against(bufs, outs, orig, adam=True)


def _nvfp4_bufs(rows, cols, seed, adam=False, packed=False, supply_amax=False):
    w, g, v = _inputs(rows, cols, seed)
    m = WL.first_moment((rows, cols), seed, device="cuda") if adam else None
    nb = rows * cols // 16
    W, Gb, V = Guarded(w.shape, w.dtype, w), Guarded(g.shape, g.dtype, g), Guarded(v.shape, v.dtype, v)
    M = Guarded(m.shape, m.dtype, m) if adam else None
    R = Guarded((rows, cols), torch.bfloat16)
    C = Guarded((rows * cols // 2,), torch.uint8) if packed else Guarded((rows, cols), torch.uint8)
    S = Guarded((nb,), torch.uint8)
    T = Guarded((1,), torch.float32)
    K = Guarded((nb,), torch.uint8)
    Am = Guarded((1,), torch.float32, w.abs().max().reshape(1)) if supply_amax else None
    return (w, g, m, v), [W, Gb, V, M, R, C, S, T, K, Am]


def _nvfp4_desc(bufs):
    W, Gb, V, M, R, C, S, T, K, Am = bufs
    d = {"w": W.t, "g": Gb.t, "v": V.t, "tensor_amax": None if Am is None else Am.t, "r": R.t,
         "codes": C.t, "block_scale": S.t, "tensor_scale": T.t, "cand_idx": K.t,
         "rows": W.t.shape[0], "cols": W.t.shape[1]}
    if M is not None:
        d["m"] = M.t
    return d


def _check_nvfp4_against(bufs, o, orig, adam=False):
    W, Gb, V, M, R, C, S, T, K, Am = bufs
    assert not _damaged(bufs)
    assert torch.equal(R.t, o["r"]) and torch.equal(S.t, o["block_scale"])
    assert torch.equal(T.t, o["tensor_scale"]) and torch.equal(K.t, o["cand_idx"])
    assert torch.equal(C.t.view(-1), o["codes"].view(-1))
    w, g, m, v = orig
    assert torch.equal(V.t, v) and torch.equal(W.t, w)
    if adam:
        assert torch.equal(M.t, m)


@pytest.mark.gpu
@pytest.mark.parametrize("supply_amax", [False, True])
def test_recon_nvfp4_guards(oracle, supply_amax):
    """quasar_recon_nvfp4 on ragged single tensors (1 row; 3 blocks; 1 block)."""
    for i, (rows, cols) in enumerate([(37, 48), (1, 16), (1, 48), (7, 1024)]):
        orig, bufs = _nvfp4_bufs(rows, cols, seed=5000 + i, supply_amax=supply_amax)
        W, Gb, V, M, R, C, S, T, K, Am = bufs
        w_h, g_h, v_h = H._host(orig[0]), H._host(orig[1]), H._host(orig[3])
        st = quasar.quasar_recon_nvfp4(W.t, Gb.t, V.t, 0.999, CLIP8, rows, cols,
                                       None if Am is None else Am.t, R.t, C.t, S.t, T.t, K.t)
        assert st == quasar.QuasarStatus.OK
        torch.cuda.synchronize()
        assert not _damaged(bufs), (rows, cols)
        h = oracle.ema(v_h, g_h, 0.999)
        _, s_T = oracle.tensor_scale(w_h)
        O = oracle.recon_nvfp4(w_h, h, s_T, CLIP8)
        gpu = {"r": H._host(R.t), "scale": S.t.cpu().numpy(), "tensor_scale": float(T.t.cpu()[0]),
               "codes": C.t.cpu().numpy().ravel(), "idx": K.t.cpu().numpy()}
        assert checker.check_nvfp4(oracle, w_h, h, CLIP8, s_T, O, gpu, True)["ok"]


@pytest.mark.gpu
@pytest.mark.parametrize("packed", [False, True])
def test_recon_nvfp4_batch_guards(packed):
    shapes = [(37, 48), (1, 16), (9, 256), (2, 1024)]
    origs, bufss = zip(*[_nvfp4_bufs(r, c, 5100 + i, packed=packed) for i, (r, c) in enumerate(shapes)])
    descs = [_nvfp4_desc(b) for b in bufss]
    st = quasar.quasar_recon_nvfp4_batch_ex(descs, 0.999, CLIP8, quasar.options(packed_codes=packed))
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    outs = api.recon_nvfp4_batch([(o[0], o[1], o[3]) for o in origs], clip=CLIP8, codes=True,
                                 packed_codes=packed)
    torch.cuda.synchronize()
    for b, o, og in zip(bufss, outs, origs):
        _check_nvfp4_against(b, o, og)


@pytest.mark.gpu
def test_adamw_recon_nvfp4_batch_guards():
    shapes = [(37, 48), (1, 16), (9, 256)]
    origs, bufss = zip(*[_nvfp4_bufs(r, c, 5200 + i, adam=True) for i, (r, c) in enumerate(shapes)])
    descs = [_nvfp4_desc(b) for b in bufss]
    hp = dict(WL.ADAMW_NVFP4)
    st = quasar.quasar_adamw_recon_nvfp4_batch(descs, hp["lr"], hp["beta1"], 0.999, hp["eps"],
                                               hp["weight_decay"], hp["step"], CLIP8)
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    outs = api.adamw_recon_nvfp4_batch([(o[0], o[1], o[2], o[3]) for o in origs], lr=hp["lr"],
                                       beta1=hp["beta1"], beta2=0.999, eps=hp["eps"],
                                       weight_decay=hp["weight_decay"], step=hp["step"],
                                       clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    for b, o, og in zip(bufss, outs, origs):
        _check_nvfp4_against(b, o, og, adam=True)


@pytest.mark.gpu
def test_recon_lut_batch_guards():
    shapes = [(8, 64), (24, 192), (8, 4096)]
    descs, bufs, orig = [], [], []
    for i, (rows, cols) in enumerate(shapes):
        w, g, v = _inputs(rows, cols, seed=5300 + i)
        nb = rows * cols // 512
        W, Gb, V = Guarded(w.shape, w.dtype, w), Guarded(g.shape, g.dtype, g), Guarded(v.shape, v.dtype, v)
        R = Guarded((rows, cols), torch.bfloat16)
        C = Guarded((rows, cols), torch.uint8)
        Bk = Guarded((nb, 8), torch.uint8)
        K = Guarded((nb,), torch.uint8)
        descs.append({"w": W.t, "g": Gb.t, "v": V.t, "r": R.t, "codes": C.t, "book": Bk.t,
                      "cand_idx": K.t, "rows": rows, "cols": cols})
        bufs.append([W, Gb, V, R, C, Bk, K])
        orig.append((w, g, v))
    st = quasar.quasar_recon_lut_batch(descs, 0.999, CLIP8)
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    outs = api.recon_lut_batch(orig, clip=CLIP8, codes=True)
    torch.cuda.synchronize()
    for bb, o, (w, g, v) in zip(bufs, outs, orig):
        W, Gb, V, R, C, Bk, K = bb
        assert not _damaged(bb)
        assert torch.equal(R.t, o["r"]) and torch.equal(Bk.t, o["book"])
        assert torch.equal(C.t, o["codes"]) and torch.equal(K.t, o["cand_idx"])
        assert torch.equal(V.t, v) and torch.equal(W.t, w)


@pytest.mark.gpu
@pytest.mark.parametrize("n", [16, 4096 + 16, 1 << 20])
def test_tensor_amax_guards(n):
    w = WL.random_groups(n // 16, 16, seed=5400, device="cuda")["w"]
    W = Guarded((n,), torch.float32, w)
    Am = Guarded((1,), torch.float32)
    st = quasar.quasar_tensor_amax(W.t, n, Am.t)
    assert st == quasar.QuasarStatus.OK
    torch.cuda.synchronize()
    assert W.intact() and Am.intact()
    assert float(Am.t.cpu()[0]) == float(w.abs().max().cpu())
