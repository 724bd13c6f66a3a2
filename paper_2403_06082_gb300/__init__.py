"""Python binding of libframequant: the forward pass of a frame-quantized linear layer
(FrameQuant, arXiv 2403.06082) on a GB300 GPU.

Argument marshalling only.  Every function here has the name and the arguments of a C entry
point declared in include/framequant.h; tensors are torch tensors on the GPU (torch provides
device memory and streams), passed to the library as raw pointers.  The computation itself
runs in the library's CUDA kernels; there is no other implementation to fall back to, and a
missing library is an error.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

__all__ = [
    "FQ_BF16", "FQ_FP32_DEBUG", "FQ_ACT_BITS", "FrameQuantError", "Packed", "ld_words", "lib", "lib_path",
    "fq_packed_words", "fq_pack", "fq_workspace_bytes", "fq_linear_forward",
    "fq_linear_forward_sms", "fq_linear_forward_ex", "fq_check",
    "fq_status_str", "EXPORTED", "fq_frame_workspace_bytes", "fq_frame_build",
    "fq_coefficients_workspace_bytes", "fq_coefficients", "fq_quantize_rtn",
    "fq_linear_forward_static", "FQ_STATIC_SCRATCH_BYTES", "Frame", "fq_frame_implicit_bytes",
    "fq_frame_implicit", "fq_implicit_workspace_bytes", "fq_linear_forward_implicit",
    "fq_reconstruct_workspace_bytes", "fq_reconstruct_weight", "fq_dense_workspace_bytes",
    "fq_dense_forward", "fq_static_check", "fq_group_workspace_bytes",
    "fq_linear_forward_group", "Layer", "FQ_MAX_GROUP", "fq_gptq_hessian",
    "fq_gptq_workspace_bytes", "fq_quantize_gptq", "fq_implicit_group_workspace_bytes",
    "fq_linear_forward_implicit_group", "ImplicitLayer", "fq_frame_tiles_bytes", "fq_frame_tile",
]
FQ_MAX_GROUP = 4
FQ_STATIC_SCRATCH_BYTES = 16 << 20

FQ_BF16 = 0
FQ_FP32_DEBUG = 1


def FQ_ACT_BITS(n: int) -> int:
    """Mode flag: round the frame representation of the activations to n-bit integers
    (FQ_BF16 | FQ_ACT_BITS(n), include/framequant.h)."""
    return n << 8
STATUS = {0: "FQ_OK", 1: "FQ_ERR_INVALID_ARG", 2: "FQ_ERR_ALIGNMENT", 3: "FQ_ERR_UNSUPPORTED",
          4: "FQ_ERR_WORKSPACE", 5: "FQ_ERR_CUDA", 6: "FQ_ERR_TIMEOUT",
          7: "FQ_ERR_DEVICE_CHECK"}
EXPORTED = ("fq_packed_words", "fq_pack", "fq_workspace_bytes", "fq_linear_forward",
            "fq_linear_forward_sms", "fq_linear_forward_ex",
            "fq_check", "fq_status_str", "fq_frame_workspace_bytes", "fq_frame_build",
            "fq_coefficients_workspace_bytes", "fq_coefficients", "fq_quantize_rtn",
            "fq_linear_forward_static", "fq_frame_implicit_bytes", "fq_frame_implicit",
            "fq_implicit_workspace_bytes", "fq_linear_forward_implicit",
            "fq_reconstruct_workspace_bytes", "fq_reconstruct_weight", "fq_dense_workspace_bytes",
            "fq_dense_forward", "fq_static_check", "fq_group_workspace_bytes",
            "fq_linear_forward_group", "fq_gptq_hessian", "fq_gptq_workspace_bytes",
            "fq_quantize_gptq", "fq_implicit_group_workspace_bytes",
            "fq_linear_forward_implicit_group", "fq_frame_tiles_bytes", "fq_frame_tile")

_HERE = os.path.dirname(os.path.abspath(__file__))


def lib_path() -> str:
    return os.path.join(_HERE, "libframequant.so")


class FrameQuantError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)}")


class _Packed(ctypes.Structure):
    _fields_ = [("words", ctypes.c_void_p), ("scale_f16", ctypes.c_void_p),
                ("zero_f16", ctypes.c_void_p), ("n_out", ctypes.c_int32), ("n_in", ctypes.c_int32),
                ("ld_words", ctypes.c_int32), ("bits", ctypes.c_int32)]


class _Rotation(ctypes.Structure):
    _fields_ = [("a", ctypes.c_int32), ("b", ctypes.c_int32), ("gauss_a", ctypes.c_void_p),
                ("gauss_b", ctypes.c_void_p), ("perm", ctypes.c_void_p),
                ("signs", ctypes.c_void_p)]


class _Opts(ctypes.Structure):
    _fields_ = [("max_sms", ctypes.c_int32), ("l2_prefetch", ctypes.c_void_p),
                ("l2_prefetch_bytes", ctypes.c_size_t), ("inject_timeout_cycles", ctypes.c_int64)]


class _Layer(ctypes.Structure):
    _fields_ = [("x", ctypes.c_void_p), ("d_in", ctypes.c_int32), ("T_in", ctypes.c_void_p),
                ("C", ctypes.POINTER(_Packed)), ("T_out_t", ctypes.c_void_p),
                ("d_out", ctypes.c_int32), ("gamma", ctypes.c_void_p), ("y", ctypes.c_void_p),
                ("T_in_tiles", ctypes.c_void_p), ("T_out_tiles", ctypes.c_void_p)]


class _ImplLayer(ctypes.Structure):
    _fields_ = [("x", ctypes.c_void_p), ("F_in", ctypes.c_void_p), ("C", ctypes.c_void_p),
                ("F_out", ctypes.c_void_p), ("gamma", ctypes.c_void_p), ("y", ctypes.c_void_p)]


class _Frame(ctypes.Structure):
    _fields_ = [("k", ctypes.c_int32), ("rho", ctypes.c_int32), ("d", ctypes.c_int32),
                ("a", ctypes.c_int32), ("b", ctypes.c_int32), ("Qa", ctypes.c_void_p),
                ("QaT", ctypes.c_void_p), ("Qb", ctypes.c_void_p), ("QbT", ctypes.c_void_p),
                ("perm", ctypes.c_void_p), ("iperm", ctypes.c_void_p),
                ("signs", ctypes.c_void_p), ("ana_tiles", ctypes.c_void_p),
                ("ana_idx", ctypes.c_void_p), ("ana_count", ctypes.c_int32),
                ("syn_tiles", ctypes.c_void_p), ("syn_idx", ctypes.c_void_p),
                ("syn_count", ctypes.c_int32)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libframequant.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        path = lib_path()
        if not os.path.exists(path):
            raise ImportError(f"libframequant.so is missing ({path}); build it with "
                              "`python -m paper_2403_06082_gb300._build`")
        L = ctypes.CDLL(path)
        L.fq_frame_tiles_bytes.restype = ctypes.c_size_t
        L.fq_frame_tiles_bytes.argtypes = [ctypes.c_int, ctypes.c_int]
        L.fq_frame_tile.restype = ctypes.c_int
        L.fq_frame_tile.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                    ctypes.c_size_t, ctypes.c_void_p]
        L.fq_packed_words.restype = ctypes.c_size_t
        L.fq_packed_words.argtypes = [ctypes.c_int, ctypes.c_int]
        L.fq_pack.restype = ctypes.c_int
        L.fq_pack.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                              ctypes.c_int, ctypes.POINTER(_Packed), ctypes.c_void_p,
                              ctypes.c_void_p]
        L.fq_workspace_bytes.restype = ctypes.c_size_t
        L.fq_workspace_bytes.argtypes = [ctypes.c_int] * 6
        L.fq_linear_forward.restype = ctypes.c_int
        L.fq_linear_forward.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
            ctypes.POINTER(_Packed), ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_void_p]
        L.fq_linear_forward_sms.restype = ctypes.c_int
        L.fq_linear_forward_sms.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
            ctypes.POINTER(_Packed), ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_int,
            ctypes.c_void_p]
        L.fq_linear_forward_ex.restype = ctypes.c_int
        L.fq_linear_forward_ex.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
            ctypes.POINTER(_Packed), ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int,
            ctypes.POINTER(_Opts), ctypes.c_void_p]
        L.fq_check.restype = ctypes.c_int
        L.fq_check.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
        L.fq_status_str.restype = ctypes.c_char_p
        L.fq_status_str.argtypes = [ctypes.c_int]
        L.fq_frame_workspace_bytes.restype = ctypes.c_size_t
        L.fq_frame_workspace_bytes.argtypes = [ctypes.c_int] * 5
        L.fq_frame_build.restype = ctypes.c_int
        L.fq_frame_build.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                     ctypes.POINTER(_Rotation), ctypes.c_void_p, ctypes.c_void_p,
                                     ctypes.c_size_t, ctypes.c_void_p]
        L.fq_coefficients_workspace_bytes.restype = ctypes.c_size_t
        L.fq_coefficients_workspace_bytes.argtypes = [ctypes.c_int, ctypes.c_int]
        L.fq_coefficients.restype = ctypes.c_int
        L.fq_coefficients.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                      ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
                                      ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                                      ctypes.c_size_t, ctypes.c_void_p]
        L.fq_linear_forward_static.restype = ctypes.c_int
        L.fq_linear_forward_static.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
            ctypes.POINTER(_Packed), ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p]
        L.fq_group_workspace_bytes.restype = ctypes.c_size_t
        L.fq_group_workspace_bytes.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.POINTER(_Layer)]
        L.fq_linear_forward_group.restype = ctypes.c_int
        L.fq_linear_forward_group.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.POINTER(_Layer),
                                              ctypes.c_void_p, ctypes.c_size_t,
                                              ctypes.POINTER(_Opts), ctypes.c_void_p]
        L.fq_gptq_hessian.restype = ctypes.c_int
        L.fq_gptq_hessian.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                      ctypes.c_void_p]
        L.fq_gptq_workspace_bytes.restype = ctypes.c_size_t
        L.fq_gptq_workspace_bytes.argtypes = [ctypes.c_int, ctypes.c_int]
        L.fq_quantize_gptq.restype = ctypes.c_int
        L.fq_quantize_gptq.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                       ctypes.c_double, ctypes.c_int, ctypes.c_void_p,
                                       ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                       ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
        L.fq_implicit_group_workspace_bytes.restype = ctypes.c_size_t
        L.fq_implicit_group_workspace_bytes.argtypes = [ctypes.c_int, ctypes.c_int,
                                                        ctypes.POINTER(_ImplLayer)]
        L.fq_linear_forward_implicit_group.restype = ctypes.c_int
        L.fq_linear_forward_implicit_group.argtypes = [
            ctypes.c_int, ctypes.c_int, ctypes.POINTER(_ImplLayer), ctypes.c_void_p,
            ctypes.c_size_t, ctypes.c_int, ctypes.c_void_p]
        L.fq_static_check.restype = ctypes.c_int
        L.fq_static_check.argtypes = [ctypes.c_void_p]
        L.fq_frame_implicit_bytes.restype = ctypes.c_size_t
        L.fq_frame_implicit_bytes.argtypes = [ctypes.c_int] * 5
        L.fq_frame_implicit.restype = ctypes.c_int
        L.fq_frame_implicit.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.POINTER(_Rotation), ctypes.c_void_p,
                                        ctypes.c_size_t, ctypes.POINTER(_Frame), ctypes.c_void_p]
        L.fq_implicit_workspace_bytes.restype = ctypes.c_size_t
        L.fq_implicit_workspace_bytes.argtypes = [ctypes.c_int] * 5
        L.fq_linear_forward_implicit.restype = ctypes.c_int
        L.fq_linear_forward_implicit.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.POINTER(_Frame), ctypes.POINTER(_Packed),
            ctypes.POINTER(_Frame), ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
            ctypes.c_size_t, ctypes.c_int, ctypes.c_void_p]
        L.fq_reconstruct_workspace_bytes.restype = ctypes.c_size_t
        L.fq_reconstruct_workspace_bytes.argtypes = [ctypes.c_int] * 4
        L.fq_reconstruct_weight.restype = ctypes.c_int
        L.fq_reconstruct_weight.argtypes = [
            ctypes.c_void_p, ctypes.POINTER(_Packed), ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
        L.fq_dense_workspace_bytes.restype = ctypes.c_size_t
        L.fq_dense_workspace_bytes.argtypes = [ctypes.c_int] * 3
        L.fq_dense_forward.restype = ctypes.c_int
        L.fq_dense_forward.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
        L.fq_quantize_rtn.restype = ctypes.c_int
        L.fq_quantize_rtn.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                      ctypes.c_void_p, ctypes.c_void_p]
        _lib = L
    return _lib


def _ptr(t) -> int | None:
    """Raw device pointer of a dense row-major tensor (the C ABI takes no strides)."""
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("libframequant takes contiguous row-major tensors only")
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def _ok(st: int, where: str) -> None:
    if st != 0:
        raise FrameQuantError(st, where)


def ld_words(n_in: int) -> int:
    """Words per row of the packed layout, 4 * ceil(n_in / 64) (include/framequant.h)."""
    return 4 * (-(-n_in // 64))


@dataclass
class Packed:
    """The packed descriptor of include/framequant.h: device tensors of packed codes (int32 view
    of the uint32 words), fp16 scale and zero (int16 views of the bit patterns), the sizes, the
    row pitch in words and the code width.  fq_pack returns one."""
    words: object
    scale: object
    zero: object
    n_out: int
    n_in: int
    ld_words: int | None = None
    bits: int = 2

    def __post_init__(self):
        if self.ld_words is None:
            self.ld_words = ld_words(self.n_in)

    def _c(self) -> _Packed:
        return _Packed(_ptr(self.words), _ptr(self.scale), _ptr(self.zero), self.n_out,
                       self.n_in, self.ld_words, self.bits)


def fq_frame_tiles_bytes(rows: int, cols: int) -> int:
    return lib().fq_frame_tiles_bytes(rows, cols)


def fq_frame_tile(T, rows: int, cols: int, out, out_bytes: int, stream=None) -> None:
    """Tiled copy of a dense bf16 frame operand (T_in or T_out_t) for Layer.T_in_tiles /
    Layer.T_out_tiles."""
    _ok(lib().fq_frame_tile(_ptr(T), rows, cols, _ptr(out), out_bytes, _stream(stream)),
        "fq_frame_tile")


def fq_packed_words(n_out: int, n_in: int) -> int:
    return lib().fq_packed_words(n_out, n_in)


def fq_pack(codes, scale, zero, n_out: int, n_in: int, words, status=None,
            stream=None) -> Packed:
    """Pack uint8 codes (n_out x n_in) into `words` and return the descriptor, which refers to
    `words`, `scale` and `zero` (fp16 bit patterns, any 16-bit dtype)."""
    pc = _Packed()
    pc.words = _ptr(words)
    _ok(lib().fq_pack(_ptr(codes), _ptr(scale), _ptr(zero), n_out, n_in, ctypes.byref(pc),
                      _ptr(status), _stream(stream)), "fq_pack")
    return Packed(words, scale, zero, pc.n_out, pc.n_in, pc.ld_words, pc.bits)


def fq_workspace_bytes(M: int, d_in: int, n_in: int, n_out: int, d_out: int,
                       mode: int = FQ_BF16) -> int:
    return lib().fq_workspace_bytes(M, d_in, n_in, n_out, d_out, mode)


def fq_linear_forward(x, M: int, d_in: int, T_in, C: Packed, T_out_t, d_out: int, gamma, y,
                      ws, ws_bytes: int, mode: int = FQ_BF16, stream=None) -> None:
    pc = C._c()
    _ok(lib().fq_linear_forward(_ptr(x), M, d_in, _ptr(T_in), ctypes.byref(pc), _ptr(T_out_t),
                                d_out, _ptr(gamma), _ptr(y), _ptr(ws), ws_bytes, mode,
                                _stream(stream)), "fq_linear_forward")


def fq_linear_forward_sms(x, M: int, d_in: int, T_in, C: Packed, T_out_t, d_out: int, gamma,
                          y, ws, ws_bytes: int, max_sms: int, mode: int = FQ_BF16,
                          stream=None) -> None:
    """fq_linear_forward on at most max_sms SMs (0: all), for independent layers run side by
    side on different streams; budgets of concurrent calls must fit the device together."""
    pc = C._c()
    _ok(lib().fq_linear_forward_sms(_ptr(x), M, d_in, _ptr(T_in), ctypes.byref(pc),
                                    _ptr(T_out_t), d_out, _ptr(gamma), _ptr(y), _ptr(ws),
                                    ws_bytes, mode, max_sms, _stream(stream)),
        "fq_linear_forward_sms")


def fq_linear_forward_ex(x, M: int, d_in: int, T_in, C: Packed, T_out_t, d_out: int, gamma, y,
                         ws, ws_bytes: int, mode: int = FQ_BF16, max_sms: int = 0,
                         prefetch=None, stream=None, inject_timeout_cycles: int = 0) -> None:
    """fq_linear_forward with options: an SM budget, a device tensor to warm in L2 while the
    call runs (typically the next layer's T_in; a hint, results do not depend on it), and the
    timeout test hook of include/framequant.h (0 in normal use)."""
    pc = C._c()
    nb = 0 if prefetch is None else prefetch.numel() * prefetch.element_size()
    opts = _Opts(max_sms, _ptr(prefetch), nb, inject_timeout_cycles)
    _ok(lib().fq_linear_forward_ex(_ptr(x), M, d_in, _ptr(T_in), ctypes.byref(pc), _ptr(T_out_t),
                                   d_out, _ptr(gamma), _ptr(y), _ptr(ws), ws_bytes, mode,
                                   ctypes.byref(opts), _stream(stream)), "fq_linear_forward_ex")


def fq_linear_forward_static(x, M: int, d_in: int, T_in, C: Packed, T_out_t, d_out: int, gamma,
                             y, mode: int = FQ_BF16, stream=None) -> None:
    """fq_linear_forward with the library's own device scratch array instead of a workspace
    (for callers that cannot allocate device memory; see include/framequant.h)."""
    pc = C._c()
    _ok(lib().fq_linear_forward_static(_ptr(x), M, d_in, _ptr(T_in), ctypes.byref(pc),
                                       _ptr(T_out_t), d_out, _ptr(gamma), _ptr(y), mode,
                                       _stream(stream)), "fq_linear_forward_static")


@dataclass
class Layer:
    """One layer of fq_linear_forward_group (the arguments of fq_linear_forward)."""
    x: object
    d_in: int
    T_in: object
    C: Packed
    T_out_t: object
    d_out: int
    gamma: object
    y: object
    T_in_tiles: object = None     # fq_frame_tile(T_in, n_in, d_in), or None
    T_out_tiles: object = None    # fq_frame_tile(T_out_t, d_out, n_out), or None


def _layers(layers):
    """C array of fq_layer, and the packed descriptors it points to (kept alive by the caller)."""
    packs = [L.C._c() for L in layers]
    arr = (_Layer * len(layers))()
    for i, (L, pc) in enumerate(zip(layers, packs)):
        arr[i] = _Layer(_ptr(L.x), L.d_in, _ptr(L.T_in), ctypes.pointer(pc), _ptr(L.T_out_t),
                        L.d_out, _ptr(L.gamma), _ptr(L.y), _ptr(L.T_in_tiles),
                        _ptr(L.T_out_tiles))
    return arr, packs


def fq_group_workspace_bytes(M: int, layers) -> int:
    arr, packs = _layers(layers)
    n = lib().fq_group_workspace_bytes(M, len(layers), arr)
    del packs
    return n


def fq_linear_forward_group(M: int, layers, ws, ws_bytes: int, max_sms: int = 0, prefetch=None,
                            stream=None) -> None:
    """The FQ_BF16 forward of independent layers (list of Layer) in one call."""
    arr, packs = _layers(layers)
    nb = 0 if prefetch is None else prefetch.numel() * prefetch.element_size()
    opts = _Opts(max_sms, _ptr(prefetch), nb, 0)
    _ok(lib().fq_linear_forward_group(M, len(layers), arr, _ptr(ws), ws_bytes,
                                      ctypes.byref(opts), _stream(stream)),
        "fq_linear_forward_group")
    del packs


def fq_static_check(stream=None) -> int:
    """Synchronize and return the device status of the last fq_linear_forward_static call on
    the current device; after a timeout it also clears the library scratch array's header."""
    return lib().fq_static_check(_stream(stream))


def fq_check(status_word, stream=None) -> int:
    """Synchronize and return the device status (0 = FQ_OK) at a workspace head or fq_pack
    status word."""
    return lib().fq_check(_ptr(status_word), _stream(stream))


def fq_status_str(status: int) -> str:
    return lib().fq_status_str(status).decode()


# ------------------------------------------------------------------ offline preparation
def fq_frame_workspace_bytes(k: int, rho: int, d: int, a: int = 0, b: int = 0) -> int:
    return lib().fq_frame_workspace_bytes(k, rho, d, a, b)


def fq_frame_build(k: int, rho: int, d: int, rotation, T, ws, ws_bytes: int,
                   stream=None) -> None:
    """rotation: None or (a, b, gauss_a, gauss_b, perm, signs) with host numpy arrays
    (float64, float64, int64, float64)."""
    import numpy as np
    rot = None
    keep = None
    if rotation is not None:
        a, b, ga, gb, perm, signs = rotation
        keep = [np.ascontiguousarray(ga, np.float64), np.ascontiguousarray(gb, np.float64),
                np.ascontiguousarray(perm, np.int64), np.ascontiguousarray(signs, np.float64)]
        rot = _Rotation(a, b, *(k_.ctypes.data for k_ in keep))
    _ok(lib().fq_frame_build(k, rho, d, ctypes.byref(rot) if rot is not None else None,
                             _ptr(T), _ptr(ws), ws_bytes, _stream(stream)), "fq_frame_build")
    del keep


@dataclass
class Frame:
    """A frame in structured form: the device buffer filled by fq_frame_implicit and the C
    descriptor pointing into it (the buffer must stay alive while the frame is used)."""
    buf: object
    c: _Frame

    @property
    def n(self) -> int:
        return self.c.k * self.c.rho

    @property
    def d(self) -> int:
        return self.c.d


def fq_frame_implicit_bytes(k: int, rho: int, d: int, a: int = 0, b: int = 0) -> int:
    return lib().fq_frame_implicit_bytes(k, rho, d, a, b)


def fq_frame_implicit(k: int, rho: int, d: int, rotation, device=None, stream=None) -> Frame:
    """Structured form of the (k, rho, d) frame; rotation as in fq_frame_build.  Allocates the
    device buffer with torch."""
    import numpy as np
    import torch
    a, b = (rotation[0], rotation[1]) if rotation is not None else (0, 0)
    nb = fq_frame_implicit_bytes(k, rho, d, a, b)
    if nb == 0:
        raise FrameQuantError(1, "fq_frame_implicit_bytes")
    buf = torch.empty(nb, dtype=torch.uint8, device=device or "cuda")
    rot, keep = None, None
    if rotation is not None:
        _, _, ga, gb, perm, signs = rotation
        keep = [np.ascontiguousarray(ga, np.float64), np.ascontiguousarray(gb, np.float64),
                np.ascontiguousarray(perm, np.int64), np.ascontiguousarray(signs, np.float64)]
        rot = _Rotation(a, b, *(k_.ctypes.data for k_ in keep))
    c = _Frame()
    _ok(lib().fq_frame_implicit(k, rho, d, ctypes.byref(rot) if rot is not None else None,
                                _ptr(buf), nb, ctypes.byref(c), _stream(stream)),
        "fq_frame_implicit")
    del keep
    return Frame(buf, c)


def fq_implicit_workspace_bytes(M: int, d_in: int, n_in: int, n_out: int, d_out: int) -> int:
    return lib().fq_implicit_workspace_bytes(M, d_in, n_in, n_out, d_out)


def fq_linear_forward_implicit(x, M: int, F_in: Frame, C: Packed, F_out: Frame, gamma, y, ws,
                               ws_bytes: int, max_sms: int = 0, stream=None) -> None:
    pc = C._c()
    _ok(lib().fq_linear_forward_implicit(_ptr(x), M, ctypes.byref(F_in.c), ctypes.byref(pc),
                                         ctypes.byref(F_out.c), _ptr(gamma), _ptr(y), _ptr(ws),
                                         ws_bytes, max_sms, _stream(stream)),
        "fq_linear_forward_implicit")


@dataclass
class ImplicitLayer:
    """One layer of fq_linear_forward_implicit_group."""
    x: object
    F_in: Frame
    C: Packed
    F_out: Frame
    gamma: object
    y: object


def _impl_layers(layers):
    keep = [L.C._c() for L in layers]
    arr = (_ImplLayer * len(layers))()
    for i, (L, pc) in enumerate(zip(layers, keep)):
        arr[i] = _ImplLayer(_ptr(L.x), ctypes.addressof(L.F_in.c), ctypes.addressof(pc),
                            ctypes.addressof(L.F_out.c), _ptr(L.gamma), _ptr(L.y))
    return arr, keep


def fq_implicit_group_workspace_bytes(M: int, layers) -> int:
    arr, keep = _impl_layers(layers)
    n = lib().fq_implicit_group_workspace_bytes(M, len(layers), arr)
    del keep
    return n


def fq_linear_forward_implicit_group(M: int, layers, ws, ws_bytes: int, max_sms: int = 0,
                                     stream=None) -> None:
    arr, keep = _impl_layers(layers)
    _ok(lib().fq_linear_forward_implicit_group(M, len(layers), arr, _ptr(ws), ws_bytes, max_sms,
                                               _stream(stream)),
        "fq_linear_forward_implicit_group")
    del keep


def fq_reconstruct_workspace_bytes(d_in: int, n_in: int, n_out: int, d_out: int) -> int:
    return lib().fq_reconstruct_workspace_bytes(d_in, n_in, n_out, d_out)


def fq_reconstruct_weight(T_in, C: Packed, T_out_t, d_in: int, d_out: int, gamma, W_hat, ws,
                          ws_bytes: int, stream=None) -> None:
    """W_hat = T_out^T diag(gamma) C_hat T_in (bf16 d_out x d_in), include/framequant_dense.h."""
    pc = C._c()
    _ok(lib().fq_reconstruct_weight(_ptr(T_in), ctypes.byref(pc), _ptr(T_out_t), d_in, d_out,
                                    _ptr(gamma), _ptr(W_hat), _ptr(ws), ws_bytes,
                                    _stream(stream)), "fq_reconstruct_weight")


def fq_dense_workspace_bytes(M: int, d_in: int, d_out: int) -> int:
    return lib().fq_dense_workspace_bytes(M, d_in, d_out)


def fq_dense_forward(x, M: int, d_in: int, W_hat, d_out: int, y, ws, ws_bytes: int,
                     stream=None) -> None:
    """y = x W_hat^T on the tensor cores (include/framequant_dense.h)."""
    _ok(lib().fq_dense_forward(_ptr(x), M, d_in, _ptr(W_hat), d_out, _ptr(y), _ptr(ws), ws_bytes,
                               _stream(stream)), "fq_dense_forward")


def fq_gptq_hessian(Z, N: int, n_in: int, H, stream=None) -> None:
    """H = Z^T Z for calibration tokens' frame representations Z (N x n_in, fp64)."""
    _ok(lib().fq_gptq_hessian(_ptr(Z), N, n_in, _ptr(H), _stream(stream)), "fq_gptq_hessian")


def fq_gptq_workspace_bytes(n_out: int, n_in: int) -> int:
    return lib().fq_gptq_workspace_bytes(n_out, n_in)


def fq_quantize_gptq(C, n_out: int, n_in: int, H, codes, scale, zero, gamma=None, ws=None,
                     ws_bytes: int = 0, damp: float = 0.01, clip: bool = False,
                     stream=None) -> None:
    """Frame-domain GPTQ of C (fp64) against H (fp64), include/framequant.h."""
    _ok(lib().fq_quantize_gptq(_ptr(C), n_out, n_in, _ptr(H), damp, int(clip), _ptr(codes),
                               _ptr(scale), _ptr(zero), _ptr(gamma), _ptr(ws), ws_bytes,
                               _stream(stream)), "fq_quantize_gptq")


def fq_coefficients_workspace_bytes(d_out: int, n_in: int) -> int:
    return lib().fq_coefficients_workspace_bytes(d_out, n_in)


def fq_coefficients(W, d_out: int, d_in: int, T_in, n_in: int, T_out, n_out: int, C, ws,
                    ws_bytes: int, stream=None) -> None:
    _ok(lib().fq_coefficients(_ptr(W), d_out, d_in, _ptr(T_in), n_in, _ptr(T_out), n_out,
                              _ptr(C), _ptr(ws), ws_bytes, _stream(stream)), "fq_coefficients")


def fq_quantize_rtn(C, n_out: int, n_in: int, codes, scale, zero, gamma=None,
                    stream=None) -> None:
    _ok(lib().fq_quantize_rtn(_ptr(C), n_out, n_in, _ptr(codes), _ptr(scale), _ptr(zero),
                              _ptr(gamma), _stream(stream)), "fq_quantize_rtn")
