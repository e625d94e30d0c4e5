"""fp64 CPU oracle for the QUASAR reconstruction (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never does, and this
package never imports the CUDA library: the two share no code.

The arithmetic lives in ``quasar_oracle.c`` (plain C, fp64, OpenMP over
groups); this module only compiles it with gcc and marshals numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "quasar_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libquasar_oracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no FMA contraction, so x86 and Arm agree)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-ffp-contract=off", "-fno-fast-math", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i64, i32, f32, f64 = ctypes.c_int64, ctypes.c_int, ctypes.c_float, ctypes.c_double
        lib.qo_ema.argtypes = [P, P, i64, f32, P]
        lib.qo_ema.restype = None
        lib.qo_adamw.argtypes = [P, P, P, P, i64, f64, f64, f64, f64, f64, i64, P, P, P]
        lib.qo_adamw.restype = None
        lib.qo_recon_int.argtypes = [P, P, i64, i32, i32, P, i32] + [P] * 11
        lib.qo_recon_int.restype = i32
        lib.qo_refit_int.argtypes = [P, P, P, i32, i32, f32, P, P]
        lib.qo_refit_int.restype = f64
        lib.qo_codes_int.argtypes = [P, i32, i32, f32, P, P, P]
        lib.qo_codes_int.restype = i32
        lib.qo_tensor_scale.argtypes = [P, i64, P, P]
        lib.qo_tensor_scale.restype = None
        lib.qo_recon_nvfp4.argtypes = [P, P, i64, f32, P, i32] + [P] * 10
        lib.qo_recon_nvfp4.restype = i32
        lib.qo_e2m1_round.argtypes = [f64]
        lib.qo_e2m1_round.restype = i32
        lib.qo_e4m3_round.argtypes = [f64]
        lib.qo_e4m3_round.restype = i32
        lib.qo_e4m3_value.argtypes = [i32]
        lib.qo_e4m3_value.restype = f64
        lib.qo_set_threads.argtypes = [i32]
        lib.qo_set_threads.restype = None
        lib.qo_get_threads.argtypes = []
        lib.qo_get_threads.restype = i32
        lib.qo_codes_nvfp4.argtypes = [P, f32, P, P, P]
        lib.qo_codes_nvfp4.restype = None
        lib.qo_fit_nvfp4_scale.argtypes = [P, P, f32, f32, P, P]
        lib.qo_fit_nvfp4_scale.restype = i32
        lib.qo_eval_nvfp4.argtypes = [P, P, f32, P, i32]
        lib.qo_eval_nvfp4.restype = f64
        lib.qo_recon_sym.argtypes = [P, P, i64, i32, i32, P, i32] + [P] * 8
        lib.qo_recon_sym.restype = i32
        lib.qo_codes_sym.argtypes = [P, i32, i32, f32, P, P]
        lib.qo_codes_sym.restype = None
        lib.qo_refit_sym.argtypes = [P, P, P, i32, i32, f32, P]
        lib.qo_refit_sym.restype = f64
        lib.qo_recon_lut.argtypes = [P, P, i64, i64, i32, i32, P, i32] + [P] * 9
        lib.qo_recon_lut.restype = i32
        lib.qo_lut_block.argtypes = [P, P, i32, f32, P, P, P, P]
        lib.qo_lut_block.restype = f64
        lib.qo_lut_fit.argtypes = [P, P, i32, f32, P, P, P]
        lib.qo_lut_fit.restype = None
        lib.qo_lut_eval.argtypes = [P, P, i32, P, P]
        lib.qo_lut_eval.restype = f64
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def set_threads(n: int) -> None:
    _load().qo_set_threads(int(n))


def get_threads() -> int:
    return int(_load().qo_get_threads())


def ema(v, g, beta2: float) -> np.ndarray:
    """Saliency EMA: fl32(beta2*v + (1-beta2)*g^2) in fp64; g=None: no update."""
    v = _c(v, np.float32).ravel()
    gg = None if g is None else _c(g, np.float32).ravel()
    out = np.empty_like(v)
    _load().qo_ema(_ptr(v), _ptr(gg), v.size, ctypes.c_float(beta2), _ptr(out))
    return out


def saliency(v_prime, mode: str = "ema") -> np.ndarray:
    """The weights h of the fit and the error from the EMA state v':
    "ema" h = v' (Sec. 4.1.1), "ema_squared" h = v'^2 (App. A.3, the
    alternative weighting; the square of an fp32 value is exact in fp64 and
    rounded once where it is stored as fp32 saliency), "uniform" h = 1 (scale
    search without saliency, the Sec. 6.5 ablation)."""
    v = _c(v_prime, np.float32).ravel()
    if mode == "ema":
        return v.copy()
    if mode == "ema_squared":
        return (v.astype(np.float64) * v.astype(np.float64)).astype(np.float32)
    if mode == "uniform":
        return np.ones_like(v)
    raise ValueError(mode)


def pack_int_codes(codes, bits: int) -> np.ndarray:
    """Deployment format of integer codes: one little-endian bitstream of
    `bits` bits a code, element j in bits [j*bits, (j+1)*bits) (byte k holds
    bits 8k .. 8k+7, least significant first).  Groups of group_size*bits/8
    whole bytes follow one another, so the flat tensor is one stream."""
    q = _c(codes, np.uint8).ravel().astype(np.int64)
    assert q.size * bits % 8 == 0
    stream = np.zeros(q.size * bits, np.uint8)
    for b in range(bits):
        stream[b::bits] = (q >> b) & 1
    return np.packbits(stream, bitorder="little")


def unpack_int_codes(packed, bits: int, n: int) -> np.ndarray:
    """Inverse of pack_int_codes for n codes."""
    stream = np.unpackbits(_c(packed, np.uint8).ravel(), bitorder="little")[: n * bits]
    q = np.zeros(n, np.int64)
    for b in range(bits):
        q |= stream[b::bits].astype(np.int64) << b
    return q.astype(np.uint8)


def pack_nvfp4_codes(codes) -> np.ndarray:
    """Two E2M1 codes (4-bit sign|magnitude nibbles) a byte, the even
    element in the low nibble."""
    q = _c(codes, np.uint8).ravel()
    assert q.size % 2 == 0 and np.all(q < 16)
    return (q[0::2] | (q[1::2] << 4)).astype(np.uint8)


def unpack_nvfp4_codes(packed) -> np.ndarray:
    p = _c(packed, np.uint8).ravel()
    out = np.empty(p.size * 2, np.uint8)
    out[0::2] = p & 0xF
    out[1::2] = p >> 4
    return out


def adamw(w, g, m, v, *, lr: float, beta1: float, beta2: float, eps: float, weight_decay: float,
          step: int):
    """One AdamW step in fp64 (stored state rounded to fp32): returns
    (w', m', v') as fp32 arrays."""
    w = _c(w, np.float32).ravel()
    g = _c(g, np.float32).ravel()
    m = _c(m, np.float32).ravel()
    v = _c(v, np.float32).ravel()
    wo, mo, vo = np.empty_like(w), np.empty_like(w), np.empty_like(w)
    _load().qo_adamw(_ptr(w), _ptr(g), _ptr(m), _ptr(v), w.size, float(lr), float(beta1),
                     float(beta2), float(eps), float(weight_decay), int(step), _ptr(wo), _ptr(mo),
                     _ptr(vo))
    return wo, mo, vo


def recon_int(w, h, group_size: int, bits: int, clip) -> dict:
    """Algorithm 1 with asymmetric integer codes, every group of a flat tensor."""
    w = _c(w, np.float32).ravel()
    h = _c(h, np.float32).ravel()
    clip = _c(clip, np.float32).ravel()
    G, K = int(group_size), clip.size
    assert w.size == h.size and w.size % G == 0
    n = w.size // G
    out = dict(
        idx=np.empty(n, np.int32), a=np.empty(n), b=np.empty(n),
        codes=np.empty(w.size, np.uint8), r=np.empty(w.size), err=np.empty(n),
        cand_err=np.empty(n * K), cand_a=np.empty(n * K), cand_b=np.empty(n * K),
        m_round=np.empty(n), m_tie=np.empty(n))
    rc = _load().qo_recon_int(
        _ptr(w), _ptr(h), n, G, int(bits), _ptr(clip), K,
        _ptr(out["idx"]), _ptr(out["a"]), _ptr(out["b"]), _ptr(out["codes"]),
        _ptr(out["r"]), _ptr(out["err"]), _ptr(out["cand_err"]), _ptr(out["cand_a"]),
        _ptr(out["cand_b"]), _ptr(out["m_round"]), _ptr(out["m_tie"]))
    if rc != 0:
        raise ValueError("qo_recon_int: bad arguments")
    for key in ("cand_err", "cand_a", "cand_b"):
        out[key] = out[key].reshape(n, K)
    return out


def codes_int(w_group, bits: int, f: float, with_t: bool = False):
    """Eq. 1 codes and per-element margins of one candidate for one group
    (and the unrounded positions t if with_t)."""
    w = _c(w_group, np.float32).ravel()
    q = np.empty(w.size, np.uint8)
    m = np.empty(w.size)
    t = np.empty(w.size)
    _load().qo_codes_int(_ptr(w), w.size, int(bits), ctypes.c_float(f), _ptr(q), _ptr(m), _ptr(t))
    return (q, m, t) if with_t else (q, m)


def refit_int(w_group, h_group, codes, bits: int, f: float):
    """Eq. 4 fit and Eq. 3 error for given codes; returns (s, z, err)."""
    w = _c(w_group, np.float32).ravel()
    h = _c(h_group, np.float32).ravel()
    q = _c(codes, np.uint8).ravel()
    s = ctypes.c_double()
    z = ctypes.c_double()
    e = _load().qo_refit_int(_ptr(w), _ptr(h), _ptr(q), w.size, int(bits), ctypes.c_float(f),
                             ctypes.byref(s), ctypes.byref(z))
    return s.value, z.value, float(e)


def tensor_scale(w):
    """NVFP4 per-tensor scale: (amax, s_T) as fp32 values."""
    w = _c(w, np.float32).ravel()
    amax = ctypes.c_float()
    sT = ctypes.c_float()
    _load().qo_tensor_scale(_ptr(w), w.size, ctypes.byref(amax), ctypes.byref(sT))
    return np.float32(amax.value), np.float32(sT.value)


def recon_nvfp4(w, h, s_T: float, clip) -> dict:
    """NVFP4 QUASAR (Sec. 4.2) over every 16-element block of a flat tensor."""
    w = _c(w, np.float32).ravel()
    h = _c(h, np.float32).ravel()
    clip = _c(clip, np.float32).ravel()
    K = clip.size
    assert w.size == h.size and w.size % 16 == 0
    n = w.size // 16
    out = dict(
        idx=np.empty(n, np.int32), scale=np.empty(n, np.uint8), codes=np.empty(w.size, np.uint8),
        r=np.empty(w.size), err=np.empty(n), cand_err=np.empty(n * K),
        cand_scale=np.empty(n * K, np.uint8), m_round=np.empty(n), m_scale=np.empty(n),
        m_tie=np.empty(n))
    rc = _load().qo_recon_nvfp4(
        _ptr(w), _ptr(h), n, ctypes.c_float(s_T), _ptr(clip), K,
        _ptr(out["idx"]), _ptr(out["scale"]), _ptr(out["codes"]), _ptr(out["r"]),
        _ptr(out["err"]), _ptr(out["cand_err"]), _ptr(out["cand_scale"]),
        _ptr(out["m_round"]), _ptr(out["m_scale"]), _ptr(out["m_tie"]))
    if rc != 0:
        raise ValueError("qo_recon_nvfp4: bad arguments")
    out["cand_err"] = out["cand_err"].reshape(n, K)
    out["cand_scale"] = out["cand_scale"].reshape(n, K)
    return out


def codes_nvfp4(w_block, f: float, with_y: bool = False):
    """E2M1 codes and per-element boundary margins of one block for factor f
    (and |w|/sigma if with_y)."""
    w = _c(w_block, np.float32).ravel()
    assert w.size == 16
    q = np.empty(16, np.uint8)
    m = np.empty(16)
    y = np.empty(16)
    _load().qo_codes_nvfp4(_ptr(w), ctypes.c_float(f), _ptr(q), _ptr(m), _ptr(y))
    return (q, m, y) if with_y else (q, m)


def fit_nvfp4_scale(w_block, h_block, s_T: float, f: float, codes):
    """Fitted E4M3 scale bits of given codes and the E4M3 boundary margin."""
    w = _c(w_block, np.float32).ravel()
    h = _c(h_block, np.float32).ravel()
    q = _c(codes, np.uint8).ravel()
    m = ctypes.c_double()
    bits = _load().qo_fit_nvfp4_scale(_ptr(w), _ptr(h), ctypes.c_float(s_T), ctypes.c_float(f),
                                      _ptr(q), ctypes.byref(m))
    return int(bits), m.value


def eval_nvfp4(w_block, h_block, s_T: float, codes, scale_bits: int) -> float:
    """Eq. 3 error of a block reconstructed as s_T * E4M3(scale_bits) * q."""
    w = _c(w_block, np.float32).ravel()
    h = _c(h_block, np.float32).ravel()
    q = _c(codes, np.uint8).ravel()
    return float(_load().qo_eval_nvfp4(_ptr(w), _ptr(h), ctypes.c_float(s_T), _ptr(q),
                                       int(scale_bits)))


def e2m1_round(y: float) -> int:
    return int(_load().qo_e2m1_round(float(y)))


def e4m3_round(x: float) -> int:
    return int(_load().qo_e4m3_round(float(x)))


def e4m3_value(bits: int) -> float:
    return float(_load().qo_e4m3_value(int(bits)))


E2M1_MAGNITUDES = (0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0)


# ----------------------------------------------------- Rubin INT3 LUT (App. B)

LUT_BLOCK = (8, 64)  # reading L1: 8 rows x 64 columns, 512 weights


def recon_lut(w, h, clip, block=LUT_BLOCK) -> dict:
    """App. B over a [rows, cols] tensor in blocks of block[0] x block[1]:
    per candidate, Eq. 1 indices with qmax = 7 on the block's clipped range,
    table entries E4M3(weighted mean of each index's weights) (Eq.
    rubin-fit), direct weighted error, argmin.  Returns per block idx, book
    [n_blocks, 8] (E4M3 bits), err, cand_err, margins; per element (tensor
    layout) codes and r."""
    w = _c(w, np.float32)
    h = _c(h, np.float32)
    assert w.ndim == 2 and w.shape == h.shape
    rows, cols = w.shape
    br, bc = block
    clip = _c(clip, np.float32).ravel()
    K = clip.size
    n = (rows // br) * (cols // bc)
    out = dict(idx=np.empty(n, np.int32), book=np.empty(n * 8, np.uint8),
               codes=np.empty(rows * cols, np.uint8), r=np.empty(rows * cols), err=np.empty(n),
               cand_err=np.empty(n * K), m_round=np.empty(n), m_book=np.empty(n),
               m_tie=np.empty(n))
    rc = _load().qo_recon_lut(_ptr(w), _ptr(h), rows, cols, br, bc, _ptr(clip), K,
                              _ptr(out["idx"]), _ptr(out["book"]), _ptr(out["codes"]),
                              _ptr(out["r"]), _ptr(out["err"]), _ptr(out["cand_err"]),
                              _ptr(out["m_round"]), _ptr(out["m_book"]), _ptr(out["m_tie"]))
    if rc != 0:
        raise ValueError("qo_recon_lut: bad arguments")
    out["book"] = out["book"].reshape(n, 8)
    out["cand_err"] = out["cand_err"].reshape(n, K)
    return out


def lut_blocks(x, block=LUT_BLOCK) -> np.ndarray:
    """[rows, cols] -> [n_blocks, br*bc]: each block's elements in row-major
    order, blocks in row-major order."""
    x = np.asarray(x)
    rows, cols = x.shape
    br, bc = block
    return (x.reshape(rows // br, br, cols // bc, bc).transpose(0, 2, 1, 3)
            .reshape(-1, br * bc))


def lut_block(w_block, h_block, f: float):
    """One candidate of one block (block order): (indices, table bits,
    error, index margins, entry margins)."""
    w = _c(w_block, np.float32).ravel()
    h = _c(h_block, np.float32).ravel()
    n = w.size
    q = np.empty(n, np.uint8)
    book = np.empty(8, np.uint8)
    m = np.empty(n)
    bm = np.empty(8)
    e = _load().qo_lut_block(_ptr(w), _ptr(h), n, ctypes.c_float(f), _ptr(q), _ptr(book), _ptr(m),
                             _ptr(bm))
    return q, book, float(e), m, bm


def lut_fit(w_block, h_block, f: float, codes):
    """Table bits (Eq. rubin-fit) of given indices on one block for factor f,
    with each entry's E4M3 boundary margin."""
    w = _c(w_block, np.float32).ravel()
    h = _c(h_block, np.float32).ravel()
    q = _c(codes, np.uint8).ravel()
    book = np.empty(8, np.uint8)
    bm = np.empty(8)
    _load().qo_lut_fit(_ptr(w), _ptr(h), w.size, ctypes.c_float(f), _ptr(q), _ptr(book), _ptr(bm))
    return book, bm


def lut_eval(w_block, h_block, codes, book) -> float:
    """Weighted error of given indices and table on one block."""
    w = _c(w_block, np.float32).ravel()
    h = _c(h_block, np.float32).ravel()
    q = _c(codes, np.uint8).ravel()
    b = _c(book, np.uint8).ravel()
    return float(_load().qo_lut_eval(_ptr(w), _ptr(h), w.size, _ptr(q), _ptr(b)))


def e4m3s_value(bits: int) -> float:
    """Value of signed E4M3 bits (sign bit 0x80)."""
    v = e4m3_value(int(bits) & 0x7F)
    return -v if int(bits) & 0x80 else v


# ------------------------------------------------------ symmetric integer codes

def recon_sym(w, h, group_size: int, bits: int, clip) -> dict:
    """Algorithm 1 with symmetric codes (readings S1, S2): per group and
    candidate, q = clamp(rne(w / s_f), -Q, Q), s_f = f amax / Q, the fit
    s* = sum h q w / sum h q^2, direct error, argmin.  codes are q + Q."""
    w = _c(w, np.float32).ravel()
    h = _c(h, np.float32).ravel()
    clip = _c(clip, np.float32).ravel()
    G, K = int(group_size), clip.size
    assert w.size == h.size and w.size % G == 0
    n = w.size // G
    out = dict(idx=np.empty(n, np.int32), a=np.empty(n), codes=np.empty(w.size, np.uint8),
               r=np.empty(w.size), err=np.empty(n), cand_err=np.empty(n * K), m_round=np.empty(n),
               m_tie=np.empty(n))
    rc = _load().qo_recon_sym(_ptr(w), _ptr(h), n, G, int(bits), _ptr(clip), K, _ptr(out["idx"]),
                              _ptr(out["a"]), _ptr(out["codes"]), _ptr(out["r"]), _ptr(out["err"]),
                              _ptr(out["cand_err"]), _ptr(out["m_round"]), _ptr(out["m_tie"]))
    if rc != 0:
        raise ValueError("qo_recon_sym: bad arguments")
    out["cand_err"] = out["cand_err"].reshape(n, K)
    return out


def codes_sym(w_group, bits: int, f: float):
    """Symmetric codes (q + Q) and boundary margins of one group for factor f."""
    w = _c(w_group, np.float32).ravel()
    q = np.empty(w.size, np.uint8)
    m = np.empty(w.size)
    _load().qo_codes_sym(_ptr(w), w.size, int(bits), ctypes.c_float(f), _ptr(q), _ptr(m))
    return q, m


def refit_sym(w_group, h_group, codes, bits: int, f: float):
    """(s*, error) of given symmetric codes on one group."""
    w = _c(w_group, np.float32).ravel()
    h = _c(h_group, np.float32).ravel()
    q = _c(codes, np.uint8).ravel()
    s = ctypes.c_double()
    e = _load().qo_refit_sym(_ptr(w), _ptr(h), _ptr(q), w.size, int(bits), ctypes.c_float(f),
                             ctypes.byref(s))
    return s.value, float(e)
