"""ctypes binding of ``libquasar.so`` (declared in ``include/quasar.h``).

Functions carry the C names and only marshal arguments: tensors become
device pointers, the clip list becomes a host float array, the stream
becomes its ``cudaStream_t`` handle.  Every step of the reconstruction runs
in the library's CUDA kernels; there is no Python or CPU fallback, and the
module raises at import-time use if the library cannot be loaded.
"""
from __future__ import annotations

import ctypes
import enum
import os
import threading

from . import build as _build

_lib = None
_lock = threading.Lock()


class QuasarStatus(enum.IntEnum):
    OK = 0
    ERR_INVALID_ARG = 1
    ERR_UNSUPPORTED = 2
    ERR_CUDA = 3
    ERR_TIMEOUT = 4


class QuasarError(RuntimeError):
    def __init__(self, status):
        self.status = QuasarStatus(status)
        super().__init__(quasar_status_string(status))


F32, BF16 = 0, 1

# Every function declared in include/quasar.h, with its ctypes prototype.
_P, _I, _I64, _F = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float
PROTOTYPES = {
    "quasar_recon_int": (_I, [_P, _P, _I, _P, _F, _I, _I, _P, _I, _I64, _I64, _P, _I, _P, _P, _P,
                              _P, _P]),
    "quasar_recon_nvfp4": (_I, [_P, _P, _I, _P, _F, _P, _I, _I64, _I64, _P, _P, _I, _P, _P, _P,
                                _P, _P]),
    "quasar_recon_int_batch": (_I, [_P, _I, _I, _F, _I, _I, _P, _I, _I, _P]),
    "quasar_recon_int_batch_ex": (_I, [_P, _I, _I, _F, _I, _I, _P, _I, _I, _P, _P]),
    "quasar_adamw_recon_int_batch": (_I, [_P, _I, _I, _F, _F, _F, _F, _F, _I64, _I, _I, _P, _I,
                                          _I, _P, _P]),
    "quasar_recon_nvfp4_batch": (_I, [_P, _I, _I, _F, _P, _I, _I, _P]),
    "quasar_recon_nvfp4_batch_ex": (_I, [_P, _I, _I, _F, _P, _I, _I, _P, _P]),
    "quasar_recon_lut_batch": (_I, [_P, _I, _I, _F, _P, _I, _I, _P, _P]),
    "quasar_adamw_recon_nvfp4_batch": (_I, [_P, _I, _I, _F, _F, _F, _F, _F, _I64, _P, _I, _I, _P,
                                            _P]),
    "quasar_tensor_amax": (_I, [_P, _I64, _P, _P]),
    "quasar_get_device_status": (_I, [_P]),
    "quasar_debug_force_timeout": (None, [_I64]),
    "quasar_debug_set_stats": (None, [_P]),
    "quasar_debug_set_hoist": (None, [_I]),
    "quasar_status_string": (ctypes.c_char_p, [_I]),
    "quasar_version": (_I, []),
}


def library_path() -> str:
    return os.environ.get("QUASAR_LIBRARY") or _build.LIB


def load(build_if_missing: bool = True):
    """Load libquasar.so (building it first if asked and needed).  The
    environment variable QUASAR_LIBRARY names another build of the same
    library to load instead (no build step then)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if os.environ.get("QUASAR_LIBRARY"):
            path = os.environ["QUASAR_LIBRARY"]
        elif build_if_missing:
            path = _build.build()
        if not os.path.exists(path):
            raise OSError(f"libquasar.so not found at {path}; run paper_2608_13966_gb300.build")
        lib = ctypes.CDLL(path)
        for name, (res, args) in PROTOTYPES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _ptr(x):
    """Device pointer of a tensor, an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _dtype_code(t, default=F32):
    if t is None:
        return default
    if isinstance(t, int):
        return default
    import torch
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _clip_array(clip):
    arr = (ctypes.c_float * len(clip))(*[float(c) for c in clip])
    return arr, len(clip)


def quasar_recon_int(w, g, v, beta2, bits, group_size, clip, rows, cols, r, codes, a, b,
                     cand_idx=None, stream=None, g_dtype=None, r_dtype=None) -> QuasarStatus:
    lib = load()
    carr, nclip = _clip_array(clip)
    gd = g_dtype if g_dtype is not None else _dtype_code(g)
    rd = r_dtype if r_dtype is not None else _dtype_code(r)
    st = lib.quasar_recon_int(_ptr(w), _ptr(g), gd, _ptr(v), beta2, bits, group_size, carr, nclip,
                              rows, cols, _ptr(r), rd, _ptr(codes), _ptr(a), _ptr(b),
                              _ptr(cand_idx), _stream(stream))
    return QuasarStatus(st)


class QuasarIntTensor(ctypes.Structure):
    """quasar_int_tensor: one tensor's buffers (device pointers) and shape."""
    _fields_ = [("w", ctypes.c_void_p), ("g", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("r", ctypes.c_void_p), ("codes", ctypes.c_void_p), ("a", ctypes.c_void_p),
                ("b", ctypes.c_void_p), ("cand_idx", ctypes.c_void_p), ("rows", ctypes.c_int64),
                ("cols", ctypes.c_int64)]


def int_tensor_array(items):
    """A ctypes array of QuasarIntTensor from dicts with keys w, g, v, r,
    codes, a, b, cand_idx (tensors, pointers or None), rows, cols."""
    arr = (QuasarIntTensor * len(items))()
    for i, d in enumerate(items):
        arr[i] = QuasarIntTensor(_ptr(d["w"]), _ptr(d.get("g")), _ptr(d["v"]), _ptr(d["r"]),
                                 _ptr(d.get("codes")), _ptr(d["a"]), _ptr(d["b"]),
                                 _ptr(d.get("cand_idx")), int(d["rows"]), int(d["cols"]))
    return arr


def quasar_recon_int_batch(tensors, beta2, bits, group_size, clip, g_dtype=BF16, r_dtype=BF16,
                           stream=None) -> QuasarStatus:
    """tensors: a ctypes array from int_tensor_array (or a list of dicts)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = int_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_recon_int_batch(ctypes.cast(tensors, ctypes.c_void_p), len(tensors), g_dtype,
                                    beta2, bits, group_size, carr, nclip, r_dtype, _stream(stream))
    return QuasarStatus(st)


# quasar_saliency / quasar_codes_layout
SALIENCY = {"ema": 0, "ema_squared": 1, "uniform": 2}
CODES_U8, CODES_PACKED = 0, 1


class QuasarOptions(ctypes.Structure):
    """quasar_options: variant of the reconstruction (saliency, codes layout,
    integer grid)."""
    _fields_ = [("saliency", ctypes.c_int), ("codes_layout", ctypes.c_int), ("grid", ctypes.c_int)]


def options(saliency="ema", packed_codes=False, symmetric=False):
    """A QuasarOptions; saliency is "ema", "ema_squared", "uniform" or a raw
    integer, packed_codes and symmetric booleans or raw integers (raw values
    pass through unchecked, for the library's own validation)."""
    raw = lambda x: isinstance(x, int) and not isinstance(x, bool)
    sal = SALIENCY[saliency] if isinstance(saliency, str) else int(saliency)
    lay = packed_codes if raw(packed_codes) else (CODES_PACKED if packed_codes else CODES_U8)
    grid = symmetric if raw(symmetric) else (1 if symmetric else 0)
    return QuasarOptions(sal, lay, grid)


def _opt_ptr(opt):
    return None if opt is None else ctypes.cast(ctypes.pointer(opt), ctypes.c_void_p)


def quasar_recon_int_batch_ex(tensors, beta2, bits, group_size, clip, options=None, g_dtype=BF16,
                              r_dtype=BF16, stream=None) -> QuasarStatus:
    """quasar_recon_int_batch with a QuasarOptions (None = defaults)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = int_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_recon_int_batch_ex(ctypes.cast(tensors, ctypes.c_void_p), len(tensors), g_dtype,
                                       beta2, bits, group_size, carr, nclip, r_dtype,
                                       _opt_ptr(options), _stream(stream))
    return QuasarStatus(st)


class QuasarAdamwTensor(ctypes.Structure):
    """quasar_adamw_tensor: one tensor's buffers (device pointers) and shape."""
    _fields_ = [("w", ctypes.c_void_p), ("g", ctypes.c_void_p), ("m", ctypes.c_void_p),
                ("v", ctypes.c_void_p), ("r", ctypes.c_void_p), ("codes", ctypes.c_void_p),
                ("a", ctypes.c_void_p), ("b", ctypes.c_void_p), ("cand_idx", ctypes.c_void_p),
                ("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


def adamw_tensor_array(items):
    """A ctypes array of QuasarAdamwTensor from dicts with keys w, g, m, v,
    r, codes, a, b, cand_idx (tensors, pointers or None), rows, cols."""
    arr = (QuasarAdamwTensor * len(items))()
    for i, d in enumerate(items):
        arr[i] = QuasarAdamwTensor(_ptr(d["w"]), _ptr(d.get("g")), _ptr(d.get("m")), _ptr(d["v"]),
                                   _ptr(d["r"]), _ptr(d.get("codes")), _ptr(d["a"]), _ptr(d["b"]),
                                   _ptr(d.get("cand_idx")), int(d["rows"]), int(d["cols"]))
    return arr


def quasar_adamw_recon_int_batch(tensors, lr, beta1, beta2, eps, weight_decay, step, bits,
                                 group_size, clip, g_dtype=BF16, r_dtype=BF16, options=None,
                                 stream=None) -> QuasarStatus:
    """tensors: a ctypes array from adamw_tensor_array (or a list of dicts)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = adamw_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_adamw_recon_int_batch(ctypes.cast(tensors, ctypes.c_void_p), len(tensors),
                                          g_dtype, lr, beta1, beta2, eps, weight_decay, step,
                                          bits, group_size, carr, nclip, r_dtype,
                                          _opt_ptr(options), _stream(stream))
    return QuasarStatus(st)


class QuasarNvfp4Tensor(ctypes.Structure):
    """quasar_nvfp4_tensor: one tensor's buffers (device pointers) and shape."""
    _fields_ = [("w", ctypes.c_void_p), ("g", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("tensor_amax", ctypes.c_void_p), ("r", ctypes.c_void_p),
                ("codes", ctypes.c_void_p), ("block_scale", ctypes.c_void_p),
                ("tensor_scale", ctypes.c_void_p), ("cand_idx", ctypes.c_void_p),
                ("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


def nvfp4_tensor_array(items):
    """A ctypes array of QuasarNvfp4Tensor from dicts with keys w, g, v,
    tensor_amax, r, codes, block_scale, tensor_scale, cand_idx, rows, cols."""
    arr = (QuasarNvfp4Tensor * len(items))()
    for i, d in enumerate(items):
        arr[i] = QuasarNvfp4Tensor(_ptr(d["w"]), _ptr(d.get("g")), _ptr(d["v"]),
                                   _ptr(d.get("tensor_amax")), _ptr(d["r"]), _ptr(d.get("codes")),
                                   _ptr(d["block_scale"]), _ptr(d["tensor_scale"]),
                                   _ptr(d.get("cand_idx")), int(d["rows"]), int(d["cols"]))
    return arr


def quasar_recon_nvfp4_batch(tensors, beta2, clip, g_dtype=BF16, r_dtype=BF16,
                             stream=None) -> QuasarStatus:
    """tensors: a ctypes array from nvfp4_tensor_array (or a list of dicts)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = nvfp4_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_recon_nvfp4_batch(ctypes.cast(tensors, ctypes.c_void_p), len(tensors), g_dtype,
                                      beta2, carr, nclip, r_dtype, _stream(stream))
    return QuasarStatus(st)


def quasar_recon_nvfp4_batch_ex(tensors, beta2, clip, options=None, g_dtype=BF16, r_dtype=BF16,
                                stream=None) -> QuasarStatus:
    """quasar_recon_nvfp4_batch with a QuasarOptions (None = defaults)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = nvfp4_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_recon_nvfp4_batch_ex(ctypes.cast(tensors, ctypes.c_void_p), len(tensors),
                                         g_dtype, beta2, carr, nclip, r_dtype, _opt_ptr(options),
                                         _stream(stream))
    return QuasarStatus(st)


class QuasarAdamwNvfp4Tensor(ctypes.Structure):
    """quasar_adamw_nvfp4_tensor: one tensor's buffers (device pointers) and shape."""
    _fields_ = [("w", ctypes.c_void_p), ("g", ctypes.c_void_p), ("m", ctypes.c_void_p),
                ("v", ctypes.c_void_p), ("r", ctypes.c_void_p), ("codes", ctypes.c_void_p),
                ("block_scale", ctypes.c_void_p), ("tensor_scale", ctypes.c_void_p),
                ("cand_idx", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


def adamw_nvfp4_tensor_array(items):
    """A ctypes array of QuasarAdamwNvfp4Tensor from dicts with keys w, g, m,
    v, r, codes, block_scale, tensor_scale, cand_idx, rows, cols."""
    arr = (QuasarAdamwNvfp4Tensor * len(items))()
    for i, d in enumerate(items):
        arr[i] = QuasarAdamwNvfp4Tensor(
            _ptr(d["w"]), _ptr(d.get("g")), _ptr(d.get("m")), _ptr(d["v"]), _ptr(d["r"]),
            _ptr(d.get("codes")), _ptr(d["block_scale"]), _ptr(d["tensor_scale"]),
            _ptr(d.get("cand_idx")), int(d["rows"]), int(d["cols"]))
    return arr


def quasar_adamw_recon_nvfp4_batch(tensors, lr, beta1, beta2, eps, weight_decay, step, clip,
                                   g_dtype=BF16, r_dtype=BF16, options=None,
                                   stream=None) -> QuasarStatus:
    """tensors: a ctypes array from adamw_nvfp4_tensor_array (or a list of dicts)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = adamw_nvfp4_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_adamw_recon_nvfp4_batch(ctypes.cast(tensors, ctypes.c_void_p), len(tensors),
                                            g_dtype, lr, beta1, beta2, eps, weight_decay, step,
                                            carr, nclip, r_dtype, _opt_ptr(options),
                                            _stream(stream))
    return QuasarStatus(st)


class QuasarLutTensor(ctypes.Structure):
    """quasar_lut_tensor: one tensor's buffers (device pointers) and shape."""
    _fields_ = [("w", ctypes.c_void_p), ("g", ctypes.c_void_p), ("v", ctypes.c_void_p),
                ("r", ctypes.c_void_p), ("codes", ctypes.c_void_p), ("book", ctypes.c_void_p),
                ("cand_idx", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


def lut_tensor_array(items):
    """A ctypes array of QuasarLutTensor from dicts with keys w, g, v, r,
    codes, book, cand_idx (tensors, pointers or None), rows, cols."""
    arr = (QuasarLutTensor * len(items))()
    for i, d in enumerate(items):
        arr[i] = QuasarLutTensor(_ptr(d["w"]), _ptr(d.get("g")), _ptr(d["v"]), _ptr(d["r"]),
                                 _ptr(d.get("codes")), _ptr(d["book"]), _ptr(d.get("cand_idx")),
                                 int(d["rows"]), int(d["cols"]))
    return arr


def quasar_recon_lut_batch(tensors, beta2, clip, options=None, g_dtype=BF16, r_dtype=BF16,
                           stream=None) -> QuasarStatus:
    """tensors: a ctypes array from lut_tensor_array (or a list of dicts)."""
    lib = load()
    if not isinstance(tensors, ctypes.Array):
        tensors = lut_tensor_array(tensors)
    carr, nclip = _clip_array(clip)
    st = lib.quasar_recon_lut_batch(ctypes.cast(tensors, ctypes.c_void_p), len(tensors), g_dtype,
                                    beta2, carr, nclip, r_dtype, _opt_ptr(options), _stream(stream))
    return QuasarStatus(st)


def quasar_recon_nvfp4(w, g, v, beta2, clip, rows, cols, tensor_amax, r, codes, block_scale,
                       tensor_scale, cand_idx=None, stream=None, g_dtype=None,
                       r_dtype=None) -> QuasarStatus:
    lib = load()
    carr, nclip = _clip_array(clip)
    gd = g_dtype if g_dtype is not None else _dtype_code(g)
    rd = r_dtype if r_dtype is not None else _dtype_code(r)
    st = lib.quasar_recon_nvfp4(_ptr(w), _ptr(g), gd, _ptr(v), beta2, carr, nclip, rows, cols,
                                _ptr(tensor_amax), _ptr(r), rd, _ptr(codes), _ptr(block_scale),
                                _ptr(tensor_scale), _ptr(cand_idx), _stream(stream))
    return QuasarStatus(st)


def quasar_tensor_amax(w, n, amax_out, stream=None) -> QuasarStatus:
    return QuasarStatus(load().quasar_tensor_amax(_ptr(w), n, _ptr(amax_out), _stream(stream)))


def quasar_get_device_status(stream=None) -> QuasarStatus:
    return QuasarStatus(load().quasar_get_device_status(_stream(stream)))


def quasar_debug_force_timeout(nanoseconds: int) -> None:
    load().quasar_debug_force_timeout(int(nanoseconds))


def quasar_debug_set_stats(counters) -> None:
    load().quasar_debug_set_stats(_ptr(counters))


def quasar_debug_set_hoist(enable: bool) -> None:
    load().quasar_debug_set_hoist(1 if enable else 0)


def quasar_status_string(status) -> str:
    return load().quasar_status_string(int(status)).decode()


def quasar_version() -> int:
    return int(load().quasar_version())
