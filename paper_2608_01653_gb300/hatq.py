"""Thin Python binding of libhatq (include/hatq.h): argument marshalling only.

Every computation runs inside libhatq's CUDA kernels (or, for the offline
weight preparation, its host code). PyTorch supplies device memory and the
current stream. There is no CPU fallback: if the library cannot be built or
loaded, or no CUDA device is present, the calls raise.
"""
from __future__ import annotations

import ctypes
import re
from dataclasses import dataclass

import numpy as np

from . import build as _build

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_OVERFLOW, ERR_CUDA, ERR_TIMEOUT = range(6)
DH, WH, TRANSFORM = 0, 1, 2
ACT_NONE, ACT_RELU, ACT_SILU, ACT_GELU = 0, 1, 2, 3
IN_OPERAND, IN_I8, IN_F16 = 0, 1, 2

_ACTS = {"none": ACT_NONE, "relu": ACT_RELU, "silu": ACT_SILU, "gelu": ACT_GELU}
GENERAL_ACTS = ("silu", "gelu")
_FORMS = {"DH": DH, "WH": WH}


class HatqError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"hatq status {status}: {message}")
        self.status = status


class ConvDesc(ctypes.Structure):
    _fields_ = [("c_in", ctypes.c_int), ("c_out", ctypes.c_int), ("kh", ctypes.c_int), ("kw", ctypes.c_int),
                ("stride", ctypes.c_int), ("pad", ctypes.c_int), ("form", ctypes.c_int),
                ("hb_in", ctypes.c_int), ("hb_out", ctypes.c_int)]


class PreparedStruct(ctypes.Structure):
    _fields_ = [("d", ConvDesc), ("act", ctypes.c_int), ("hb_next", ctypes.c_int), ("out_f32", ctypes.c_int),
                ("shift", ctypes.c_int), ("k_pad", ctypes.c_int), ("gather", ctypes.c_int),
                ("s_x", ctypes.c_float), ("s_y", ctypes.c_float),
                ("w_i8", ctypes.c_void_p), ("w_f16", ctypes.c_void_p), ("b_int", ctypes.c_void_p),
                ("mult", ctypes.c_void_p), ("deq", ctypes.c_void_p), ("s_w", ctypes.c_void_p),
                ("opaque", ctypes.c_uint64 * 16),
                ("s_z", ctypes.c_float), ("s_u", ctypes.c_float), ("shift_in", ctypes.c_int),
                ("in_affine", ctypes.c_int), ("mult_in", ctypes.c_longlong), ("lut", ctypes.c_int8 * 256),
                ("in_f16", ctypes.c_int), ("out_f16", ctypes.c_int)]


MAX_TRANSPOSED_CLASSES = 4


class PreparedTransposedStruct(ctypes.Structure):
    _fields_ = [("d", ConvDesc), ("out_pad", ctypes.c_int), ("classes", ctypes.c_int),
                ("pad_y", ctypes.c_int * MAX_TRANSPOSED_CLASSES), ("pad_x", ctypes.c_int * MAX_TRANSPOSED_CLASSES),
                ("sub", PreparedStruct * MAX_TRANSPOSED_CLASSES)]


class PreparedGdnStruct(ctypes.Structure):
    _fields_ = [("c", ctypes.c_int), ("inverse", ctypes.c_int), ("hb_next", ctypes.c_int), ("e", ctypes.c_int),
                ("t", ctypes.c_int), ("shift_in", ctypes.c_int), ("P", ctypes.c_longlong),
                ("mult_in", ctypes.c_longlong), ("s_z", ctypes.c_float), ("s_u", ctypes.c_float),
                ("s_y", ctypes.c_float), ("g_f16", ctypes.c_void_p), ("b_pool", ctypes.c_void_p),
                ("opaque", ctypes.c_uint64 * 16)]


_LIB = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float


def load(build: bool = True) -> ctypes.CDLL:
    """Load libhatq.so (building it in-tree first if it is missing or stale)."""
    global _LIB
    if _LIB is None:
        path = _build.build() if build else _build.LIB
        lib = ctypes.CDLL(path)
        sig = {
            "hatq_prepared_sizes": (_I, [ctypes.POINTER(ConvDesc), ctypes.POINTER(ctypes.c_size_t),
                                         ctypes.POINTER(ctypes.c_size_t)]),
            "hatq_prepare_weights": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _F, _F, _I, _I, _I,
                                          ctypes.POINTER(PreparedStruct), _P]),
            "hatq_prepare_weights_general": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _F, _F, _F, _F, _I, _I,
                                                  ctypes.POINTER(PreparedStruct), _P]),
            "hatq_prepare_weights_general_host": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _F, _F, _F, _F, _I, _I,
                                                       _P, _P, _P, _P, _P, ctypes.POINTER(_I),
                                                       ctypes.POINTER(ctypes.c_longlong), ctypes.POINTER(_I), _P]),
            "hatq_prepare_weights_host": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _F, _F, _I, _I, _I,
                                               _P, _P, _P, _P, _P, _P, ctypes.POINTER(_I)]),
            "hatq_quantize_act": (_I, [_P, _I, _F, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P]),
            "hatq_conv2d_i8": (_I, [_P, _I, _I, _I, ctypes.POINTER(PreparedStruct), _P, _P]),
            "hatq_layer": (_I, [_P, _I, _F, _I, _I, _I, ctypes.POINTER(PreparedStruct), _P, _P,
                                ctypes.c_size_t, _P]),
            "hatq_layer_launches": (_I, [_I, _F, ctypes.POINTER(PreparedStruct)]),
            "hatq_last_error": (ctypes.c_char_p, []),
            "hatq_sync_status": (_I, [_P]),
            "hatq_selftest_wait": (_I, [ctypes.c_ulonglong, _P]),
            "hatq_profile_range": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P]),
            "hatq_select_form": (_I, [_P, _I, _I, _I, ctypes.POINTER(_I), ctypes.POINTER(_I)]),
            "hatq_hadamard_order": (_I, [_I, ctypes.POINTER(_I)]),
            "hatq_hadamard_matrix": (_I, [_I, _P]),
            "hatq_prepare_weights_order": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _F, _F, _I, _I, _I,
                                                ctypes.POINTER(PreparedStruct), _P]),
            "hatq_prepare_weights_order_host": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _F, _F, _I, _I, _I,
                                                     _P, _P, _P, _P, _P, _P, ctypes.POINTER(_I)]),
            "hatq_prepare_order_transform": (_I, [_I, _F, _F, ctypes.POINTER(PreparedStruct), _P]),
            "hatq_prepare_weights_affine": (_I, [ctypes.POINTER(ConvDesc), _P, _P, _I, ctypes.POINTER(PreparedStruct),
                                                 _P]),
            "hatq_quantize_act_affine": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P, _P]),
            "hatq_conv2d_affine": (_I, [_P, _I, _I, _I, ctypes.POINTER(PreparedStruct), _P, _P, _P]),
            "hatq_transposed_sizes": (_I, [ctypes.POINTER(ConvDesc), _I, ctypes.POINTER(ctypes.c_size_t),
                                           ctypes.POINTER(ctypes.c_size_t)]),
            "hatq_prepare_weights_transposed": (_I, [ctypes.POINTER(ConvDesc), _I, _P, _P, _F, _F, _I, _I, _I,
                                                     ctypes.POINTER(PreparedTransposedStruct), _P]),
            "hatq_conv_transpose2d_i8": (_I, [_P, _I, _I, _I, ctypes.POINTER(PreparedTransposedStruct), _P, _P]),
            "hatq_conv2d_i8_subpixel": (_I, [_P, _I, _I, _I, ctypes.POINTER(PreparedStruct), _I, _P, _P]),
            "hatq_layer_noalloc": (_I, [_P, _I, _F, _I, _I, _I, ctypes.POINTER(PreparedStruct), _P, _P]),
            "hatq_prepare_gdn_host": (_I, [_I, _P, _P, _F, _F, _I, _F, _I, _P, _P, ctypes.POINTER(_I),
                                           ctypes.POINTER(ctypes.c_longlong), ctypes.POINTER(_I),
                                           ctypes.POINTER(ctypes.c_longlong), ctypes.POINTER(_I)]),
            "hatq_prepare_gdn": (_I, [_I, _P, _P, _F, _F, _I, _F, _I, ctypes.POINTER(PreparedGdnStruct), _P]),
            "hatq_gdn": (_I, [_P, _I, _I, _I, ctypes.POINTER(PreparedGdnStruct), _P, _P]),
            "hatq_set_operand_format": (_I, [ctypes.POINTER(PreparedStruct), _I, _I]),
            "hatq_version": (_I, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = lib
    return _LIB


def declared_functions(header_path: str | None = None):
    """Names of the functions include/hatq.h declares."""
    import os
    header_path = header_path or os.path.join(_build.INCLUDE, "hatq.h")
    text = open(header_path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hatq_[a-z0-9_]+)\s*\(", text)))


def last_error() -> str:
    return load().hatq_last_error().decode()


def _check(status):
    if status != OK:
        raise HatqError(status, last_error())


def _torch():
    import torch
    if not torch.cuda.is_available():
        raise RuntimeError("libhatq needs a CUDA device; none is available")
    return torch


def _stream(stream):
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def make_desc(c_in, c_out, k, stride, pad, form, hb_in=0, hb_out=0, kw=None) -> ConvDesc:
    form = _FORMS.get(form, form)
    return ConvDesc(c_in, c_out, k, k if kw is None else kw, stride, pad, form, hb_in, hb_out)


def desc_from_spec(spec) -> ConvDesc:
    """A ConvDesc from a layer description with c_in, c_out, k, stride, pad, form, hb_in, hb_out."""
    return make_desc(spec.c_in, spec.c_out, spec.k, spec.stride, spec.pad, spec.form, spec.hb_in, spec.hb_out)


def prepared_sizes(desc: ConvDesc):
    w = ctypes.c_size_t()
    c = ctypes.c_size_t()
    _check(load().hatq_prepared_sizes(ctypes.byref(desc), ctypes.byref(w), ctypes.byref(c)))
    return w.value, c.value


@dataclass
class HostPrepared:
    w_i8: np.ndarray
    w_f16: np.ndarray
    b_int: np.ndarray
    mult: np.ndarray
    deq: np.ndarray
    s_w: np.ndarray
    shift: int


def prepare_weights_host(desc: ConvDesc, w_ohwi, bias, s_x, s_y, act="none", hb_next=0, out_f32=False):
    """hatq_prepare_weights_host: the offline preparation into host arrays."""
    w_elems, ch = prepared_sizes(desc)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    out = HostPrepared(np.zeros(w_elems, np.int8), np.zeros(w_elems, np.uint16), np.zeros(ch, np.int32),
                       np.zeros(ch, np.int32), np.zeros(ch, np.float32), np.zeros(ch, np.float32), 0)
    shift = ctypes.c_int()
    _check(load().hatq_prepare_weights_host(
        ctypes.byref(desc), w.ctypes.data, None if b is None else b.ctypes.data, float(s_x), float(s_y),
        _ACTS.get(act, act), int(hb_next), int(bool(out_f32)), out.w_i8.ctypes.data, out.w_f16.ctypes.data,
        out.b_int.ctypes.data, out.mult.ctypes.data, out.deq.ctypes.data, out.s_w.ctypes.data, ctypes.byref(shift)))
    out.shift = shift.value
    k_pad = w_elems // desc.c_out
    out.w_i8 = out.w_i8.reshape(desc.c_out, k_pad)
    out.w_f16 = out.w_f16.reshape(desc.c_out, k_pad)
    return out


class PreparedLayer:
    """A prepared layer: device buffers (torch tensors) plus the C struct."""

    def __init__(self, desc: ConvDesc, device="cuda"):
        torch = _torch()
        w_elems, ch = prepared_sizes(desc)
        self.desc = desc
        self.w_i8 = torch.zeros(w_elems, dtype=torch.int8, device=device)
        self.w_f16 = torch.zeros(w_elems, dtype=torch.float16, device=device)
        self.b_int = torch.zeros(ch, dtype=torch.int32, device=device)
        self.mult = torch.zeros(ch, dtype=torch.int32, device=device)
        self.deq = torch.zeros(ch, dtype=torch.float32, device=device)
        self.s_w = torch.zeros(ch, dtype=torch.float32, device=device)
        self.struct = PreparedStruct()
        self.struct.w_i8 = self.w_i8.data_ptr()
        self.struct.w_f16 = self.w_f16.data_ptr()
        self.struct.b_int = self.b_int.data_ptr()
        self.struct.mult = self.mult.data_ptr()
        self.struct.deq = self.deq.data_ptr()
        self.struct.s_w = self.s_w.data_ptr()

    @property
    def c_in(self):
        return self.desc.c_in

    @property
    def c_out(self):
        return self.desc.c_out

    @property
    def out_f32(self):
        return bool(self.struct.out_f32)

    @property
    def s_x(self):
        return float(self.struct.s_x)

    @property
    def in_f16(self):
        return bool(self.struct.in_f16)

    @property
    def out_f16(self):
        return bool(self.struct.out_f16)

    @property
    def out_dtype(self):
        """torch dtype name of the layer's output tensor."""
        return "float32" if self.out_f32 else ("float16" if self.out_f16 else "int8")

    @property
    def s_y(self):
        return float(self.struct.s_y)

    def out_shape(self, n, h, w):
        d = self.desc
        return (n, (h + 2 * d.pad - d.kh) // d.stride + 1, (w + 2 * d.pad - d.kw) // d.stride + 1, d.c_out)


def prepare_weights(desc: ConvDesc, w_ohwi, bias, s_x, s_y, act="none", hb_next=0, out_f32=False,
                    stream=None, device="cuda", s_z=None, s_u=None) -> PreparedLayer:
    """hatq_prepare_weights (or, for act 'silu' / 'gelu', hatq_prepare_weights_general
    with preactivation scale s_z and activation scale s_u): offline transform,
    quantize and pack into device buffers."""
    L = PreparedLayer(desc, device)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    bp = None if b is None else b.ctypes.data
    if act in GENERAL_ACTS:
        if out_f32 or s_z is None or s_u is None:
            raise ValueError("a SiLU / GELU layer emits INT8 codes and needs s_z and s_u")
        _check(load().hatq_prepare_weights_general(ctypes.byref(desc), w.ctypes.data, bp, float(s_x), float(s_z),
                                                   float(s_u), float(s_y), _ACTS[act], int(hb_next),
                                                   ctypes.byref(L.struct), _stream(stream)))
        return L
    _check(load().hatq_prepare_weights(ctypes.byref(desc), w.ctypes.data, bp, float(s_x), float(s_y),
                                       _ACTS.get(act, act), int(hb_next), int(bool(out_f32)),
                                       ctypes.byref(L.struct), _stream(stream)))
    return L


def hadamard_order(c: int) -> int:
    """hatq_hadamard_order: m(C) of Eq. supp_hadamard_order."""
    m = ctypes.c_int()
    _check(load().hatq_hadamard_order(int(c), ctypes.byref(m)))
    return m.value


def hadamard_matrix(m: int) -> np.ndarray:
    """hatq_hadamard_matrix: the library's unnormalized H~_m as an int8 [m, m] array."""
    h = np.zeros((m, m), np.int8)
    _check(load().hatq_hadamard_matrix(int(m), h.ctypes.data))
    return h


def order_desc(desc: ConvDesc) -> ConvDesc:
    """The operand descriptor of a DH layer in the paper's order: c_in = hb_in = m(c_in)."""
    m = hadamard_order(desc.c_in)
    return ConvDesc(m, desc.c_out, desc.kh, desc.kw, desc.stride, desc.pad, desc.form, m, 0)


def prepare_weights_order_host(desc: ConvDesc, w_ohwi, bias, s_x, s_y, act="none", hb_next=0, out_f32=False):
    """hatq_prepare_weights_order_host: a paper-order DH layer prepared into host arrays."""
    if desc.form != DH:                             # the library rejects it before touching any buffer
        _check(load().hatq_prepare_weights_order_host(ctypes.byref(desc), None, None, float(s_x), float(s_y), 0, 0,
                                                      0, None, None, None, None, None, None, None))
    dop = order_desc(desc)
    w_elems, ch = prepared_sizes(dop)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    out = HostPrepared(np.zeros(w_elems, np.int8), np.zeros(w_elems, np.uint16), np.zeros(ch, np.int32),
                       np.zeros(ch, np.int32), np.zeros(ch, np.float32), np.zeros(ch, np.float32), 0)
    shift = ctypes.c_int()
    _check(load().hatq_prepare_weights_order_host(
        ctypes.byref(desc), w.ctypes.data, None if b is None else b.ctypes.data, float(s_x), float(s_y),
        _ACTS.get(act, act), int(hb_next), int(bool(out_f32)), out.w_i8.ctypes.data, out.w_f16.ctypes.data,
        out.b_int.ctypes.data, out.mult.ctypes.data, out.deq.ctypes.data, out.s_w.ctypes.data, ctypes.byref(shift)))
    out.shift = shift.value
    out.w_i8 = out.w_i8.reshape(desc.c_out, -1)
    out.w_f16 = out.w_f16.reshape(desc.c_out, -1)
    return out


def prepare_weights_order(desc: ConvDesc, w_ohwi, bias, s_x, s_y, act="none", hb_next=0, out_f32=False,
                          stream=None, device="cuda") -> "PreparedLayer":
    """hatq_prepare_weights_order: a DH layer whose input side takes the paper's
    order m(c_in); the returned layer consumes an operand of m channels."""
    L = PreparedLayer(order_desc(desc), device)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    _check(load().hatq_prepare_weights_order(ctypes.byref(desc), w.ctypes.data, None if b is None else b.ctypes.data,
                                             float(s_x), float(s_y), _ACTS.get(act, act), int(hb_next),
                                             int(bool(out_f32)), ctypes.byref(L.struct), _stream(stream)))
    return L


def prepare_order_transform(c: int, s_in, s_out, stream=None, device="cuda") -> "PreparedLayer":
    """hatq_prepare_order_transform: the activation-side transform into the
    order m(c) as a 1x1 layer (c -> m channels), run with conv2d_i8 or layer."""
    m = hadamard_order(c)
    L = PreparedLayer(ConvDesc(c, m, 1, 1, 1, 0, TRANSFORM, 0, 0), device)
    _check(load().hatq_prepare_order_transform(int(c), float(s_in), float(s_out), ctypes.byref(L.struct),
                                               _stream(stream)))
    return L


def prepare_weights_affine(desc: ConvDesc, w_ohwi, bias, act="none", stream=None, device="cuda") -> "PreparedLayer":
    """hatq_prepare_weights_affine: a layer for dynamic affine activations
    (centred int16 operand, per-input scale, float32 output)."""
    L = PreparedLayer(desc, device)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    _check(load().hatq_prepare_weights_affine(ctypes.byref(desc), w.ctypes.data, None if b is None else b.ctypes.data,
                                              _ACTS.get(act, act), ctypes.byref(L.struct), _stream(stream)))
    return L


def quantize_act_affine(x, hb, y=None, params=None, workspace=None, stream=None):
    """hatq_quantize_act_affine on a CUDA fp16 NHWC tensor: returns (centred
    int16 codes, params = device float[2] holding s and z)."""
    if getattr(x, "dim", lambda: 0)() != 4:
        raise ValueError("x must be a 4-D NHWC tensor")
    _check_tensor(x, "x", "float16")
    n, h, w, c = x.shape
    if y is not None:
        _check_tensor(y, "y", "int16", (n, h, w, c))
    _check_cuda(("x", x), ("y", y))
    torch = _torch()
    if y is None:
        y = torch.empty((n, h, w, c), dtype=torch.int16, device=x.device)
    if params is None:
        params = torch.empty(2, dtype=torch.float32, device=x.device)
    if workspace is None:
        workspace = torch.empty(64, dtype=torch.uint8, device=x.device)
    _check(load().hatq_quantize_act_affine(_ptr(x), n, h, w, c, int(hb), _ptr(y), _ptr(params), _ptr(workspace),
                                           _stream(stream)))
    return y, params


def conv2d_affine(x, L: "PreparedLayer", params, y=None, stream=None):
    """hatq_conv2d_affine: the convolution on centred int16 codes at step params[0]."""
    if getattr(x, "dim", lambda: 0)() != 4 or x.shape[-1] != L.c_in:
        raise ValueError("x must be a 4-D NHWC tensor with the layer's input channels")
    _check_tensor(x, "x", "int16")
    n, h, w, c = x.shape
    if y is not None:
        _check_tensor(y, "y", "float32", L.out_shape(n, h, w))
    _check_cuda(("x", x), ("y", y), ("params", params))
    torch = _torch()
    if y is None:
        y = torch.empty(L.out_shape(n, h, w), dtype=torch.float32, device=x.device)
    _check(load().hatq_conv2d_affine(_ptr(x), n, h, w, ctypes.byref(L.struct), _ptr(params), _ptr(y), _stream(stream)))
    return y


class PreparedTransposed:
    """A prepared transposed convolution: one sub-layer (device buffers + C
    struct) per output parity class, inside the C struct
    hatq_prepared_transposed."""

    def __init__(self, desc: ConvDesc, out_pad: int, device="cuda"):
        torch = _torch()
        self.desc = desc
        self.out_pad = out_pad
        self.struct = PreparedTransposedStruct()
        self.buffers = []
        for cls in range(desc.stride * desc.stride):
            w = ctypes.c_size_t()
            c = ctypes.c_size_t()
            _check(load().hatq_transposed_sizes(ctypes.byref(desc), cls, ctypes.byref(w), ctypes.byref(c)))
            bufs = dict(w_i8=torch.zeros(w.value, dtype=torch.int8, device=device),
                        w_f16=torch.zeros(w.value, dtype=torch.float16, device=device),
                        b_int=torch.zeros(c.value, dtype=torch.int32, device=device),
                        mult=torch.zeros(c.value, dtype=torch.int32, device=device),
                        deq=torch.zeros(c.value, dtype=torch.float32, device=device),
                        s_w=torch.zeros(c.value, dtype=torch.float32, device=device))
            for k, t in bufs.items():
                setattr(self.struct.sub[cls], k, t.data_ptr())
            self.buffers.append(bufs)

    @property
    def c_in(self):
        return self.desc.c_in

    @property
    def out_f32(self):
        return bool(self.struct.sub[0].out_f32)

    def out_shape(self, n, h, w):
        d = self.desc
        return (n, (h - 1) * d.stride - 2 * d.pad + d.kh + self.out_pad,
                (w - 1) * d.stride - 2 * d.pad + d.kw + self.out_pad, d.c_out)


def prepare_weights_transposed(desc: ConvDesc, out_pad, w_ohwi, bias, s_x, s_y, act="none", hb_next=0,
                               out_f32=False, stream=None, device="cuda") -> PreparedTransposed:
    """hatq_prepare_weights_transposed: a transposed convolution (decoder side)
    prepared as one stride-1 sub-layer per output parity class."""
    T = PreparedTransposed(desc, out_pad, device)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    _check(load().hatq_prepare_weights_transposed(ctypes.byref(desc), int(out_pad), w.ctypes.data,
                                                  None if b is None else b.ctypes.data, float(s_x), float(s_y),
                                                  _ACTS.get(act, act), int(hb_next), int(bool(out_f32)),
                                                  ctypes.byref(T.struct), _stream(stream)))
    return T


def conv_transpose2d_i8(x, T: PreparedTransposed, y=None, stream=None):
    """hatq_conv_transpose2d_i8 on the INT8 operand x (NHWC)."""
    n, h, w, c = _check_layer_io(x, IN_OPERAND, T, y)
    torch = _torch()
    if y is None:
        y = torch.empty(T.out_shape(n, h, w), dtype=torch.float32 if T.out_f32 else torch.int8, device=x.device)
    _check(load().hatq_conv_transpose2d_i8(_ptr(x), n, h, w, ctypes.byref(T.struct), _ptr(y), _stream(stream)))
    return y


@dataclass
class HostGdn:
    """hatq_prepare_gdn_host outputs."""
    G: np.ndarray
    B: np.ndarray
    e: int
    P: int
    t: int
    mult_in: int
    shift_in: int


def _gdn_args(c, beta, gamma):
    beta = np.ascontiguousarray(beta, dtype=np.float64).ravel()
    gamma = np.ascontiguousarray(gamma, dtype=np.float64)
    if beta.size != c or gamma.shape != (c, c):
        raise ValueError(f"beta must have {c} entries and gamma be {c} x {c}")
    return beta, gamma


def prepare_gdn_host(c, beta, gamma, s_z, s_u, inverse, s_y, hb_next=0) -> HostGdn:
    """hatq_prepare_gdn_host: the integer GDN / IGDN parameters on the host."""
    beta, gamma = _gdn_args(c, beta, gamma)
    G = np.zeros((c, c), dtype=np.int32)
    B = np.zeros(c, dtype=np.int32)
    e, t, n_in = _I(), _I(), _I()
    P, m_in = ctypes.c_longlong(), ctypes.c_longlong()
    _check(load().hatq_prepare_gdn_host(int(c), beta.ctypes.data, gamma.ctypes.data, float(s_z), float(s_u),
                                        int(bool(inverse)), float(s_y), int(hb_next), G.ctypes.data, B.ctypes.data,
                                        ctypes.byref(e), ctypes.byref(P), ctypes.byref(t), ctypes.byref(m_in),
                                        ctypes.byref(n_in)))
    return HostGdn(G, B, e.value, P.value, t.value, m_in.value, n_in.value)


class PreparedGdn:
    """A prepared GDN / IGDN transition: device G (fp16) and B, and the C
    struct hatq_prepared_gdn."""

    def __init__(self, c, device="cuda"):
        torch = _torch()
        self.c = c
        self.g_f16 = torch.zeros(c * c, dtype=torch.float16, device=device)
        self.b_pool = torch.zeros(c, dtype=torch.int32, device=device)
        self.struct = PreparedGdnStruct()
        self.struct.g_f16 = self.g_f16.data_ptr()
        self.struct.b_pool = self.b_pool.data_ptr()


def prepare_gdn(c, beta, gamma, s_z, s_u, inverse, s_y, hb_next=0, stream=None, device="cuda") -> PreparedGdn:
    """hatq_prepare_gdn: phi_int of GDN (inverse False) or IGDN for c channels
    and the next layer's input transition (block hb_next, scale s_y)."""
    beta, gamma = _gdn_args(c, beta, gamma)
    g = PreparedGdn(c, device)
    _check(load().hatq_prepare_gdn(int(c), beta.ctypes.data, gamma.ctypes.data, float(s_z), float(s_u),
                                   int(bool(inverse)), float(s_y), int(hb_next), ctypes.byref(g.struct),
                                   _stream(stream)))
    return g


def gdn(z, g: PreparedGdn, y=None, stream=None):
    """hatq_gdn on the preactivation codes z (NHWC int8, c channels): the
    next layer's INT8 operand."""
    _check_tensor(z, "z", "int8")
    if z.dim() != 4 or z.shape[-1] != g.c:
        raise ValueError(f"z must be NHWC with {g.c} channels")
    if y is not None:
        _check_tensor(y, "y", "int8", tuple(z.shape))
    _check_cuda(("z", z), ("y", y))
    torch = _torch()
    if y is None:
        y = torch.empty_like(z)
    n, h, w, _ = z.shape
    _check(load().hatq_gdn(_ptr(z), n, h, w, ctypes.byref(g.struct), _ptr(y), _stream(stream)))
    return y


def conv2d_i8_subpixel(x, L: "PreparedLayer", r: int, y=None, stream=None):
    """hatq_conv2d_i8_subpixel: the convolution followed by the sub-pixel
    (depth-to-space) rearrangement with factor r, in the copy-out."""
    n, h, w, c = _check_layer_io(x, IN_OPERAND, L, None)
    _, ho, wo, co = L.out_shape(n, h, w)
    shape = (n, ho * r, wo * r, co // (r * r))
    if y is not None:
        _check_tensor(y, "y", "int8", shape)
    torch = _torch()
    if y is None:
        y = torch.empty(shape, dtype=torch.int8, device=x.device)
    _check(load().hatq_conv2d_i8_subpixel(_ptr(x), n, h, w, ctypes.byref(L.struct), int(r), _ptr(y), _stream(stream)))
    return y


@dataclass
class HostGeneral:
    w_i8: np.ndarray
    b_int: np.ndarray
    mult: np.ndarray
    s_w: np.ndarray
    shift: int
    mult_in: int
    shift_in: int
    lut: np.ndarray


def prepare_weights_general_host(desc: ConvDesc, w_ohwi, bias, s_x, s_z, s_u, s_y, act, hb_next=0) -> HostGeneral:
    """hatq_prepare_weights_general_host: the host half of a SiLU / GELU layer's preparation."""
    w_elems, ch = prepared_sizes(desc)
    w = np.ascontiguousarray(w_ohwi, dtype=np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    w_i8, w_f16 = np.zeros(w_elems, np.int8), np.zeros(w_elems, np.uint16)
    b_int, mult, s_w = np.zeros(ch, np.int32), np.zeros(ch, np.int32), np.zeros(ch, np.float32)
    lut = np.zeros(256, np.int8)
    shift, shift_in, mult_in = ctypes.c_int(), ctypes.c_int(), ctypes.c_longlong()
    _check(load().hatq_prepare_weights_general_host(
        ctypes.byref(desc), w.ctypes.data, None if b is None else b.ctypes.data, float(s_x), float(s_z), float(s_u),
        float(s_y), _ACTS[act], int(hb_next), w_i8.ctypes.data, w_f16.ctypes.data, b_int.ctypes.data,
        mult.ctypes.data, s_w.ctypes.data, ctypes.byref(shift), ctypes.byref(mult_in), ctypes.byref(shift_in),
        lut.ctypes.data))
    return HostGeneral(w_i8.reshape(desc.c_out, -1), b_int, mult, s_w, shift.value, mult_in.value, shift_in.value, lut)


_KIND_DTYPE = {IN_OPERAND: "int8", IN_I8: "int8", IN_F16: "float16"}


def _check_tensor(t, what, dtype=None, shape=None):
    """Shape, dtype, layout and device of a tensor handed to the library: the
    entry points read and write exactly the elements these describe."""
    import torch
    if not isinstance(t, torch.Tensor):
        raise ValueError(f"{what} must be a torch tensor")
    if dtype is not None and t.dtype != getattr(torch, dtype):
        raise ValueError(f"{what} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{what} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous (NHWC, C innermost)")


def _check_cuda(*named):
    for what, t in named:
        if t is not None and not t.is_cuda:
            raise ValueError(f"{what} must be on a CUDA device")


def _check_layer_io(x, x_kind, L, y=None, scratch=None):
    """The input of a layer call (kind, dtype, 4-D NHWC with L.c_in channels)
    and, when given, its output and scratch buffers."""
    if x_kind not in _KIND_DTYPE:
        raise ValueError(f"unknown input kind {x_kind}")
    if getattr(x, "dim", lambda: 0)() != 4:
        raise ValueError("x must be a 4-D NHWC tensor")
    n, h, w, c = x.shape
    if c != L.c_in:
        raise ValueError(f"x has {c} channels, the layer takes {L.c_in}")
    f16_op = x_kind == IN_OPERAND and getattr(L, "in_f16", False)
    _check_tensor(x, "x", "float16" if f16_op else _KIND_DTYPE[x_kind])
    if y is not None:
        _check_tensor(y, "y", getattr(L, "out_dtype", "float32" if L.out_f32 else "int8"), L.out_shape(n, h, w))
    if scratch is not None:
        _check_tensor(scratch, "scratch", "int8")
    _check_cuda(("x", x), ("y", y), ("scratch", scratch))
    return n, h, w, c


def quantize_act(x, x_kind, s_in, hb, s_out, y=None, s_used=None, workspace=None, stream=None):
    """hatq_quantize_act on a CUDA NHWC tensor (int8 codes or fp16 values).
    s_out <= 0 selects the dynamic mode (s_used: 1-element float32 CUDA tensor)."""
    torch = _torch()
    if x_kind not in (IN_I8, IN_F16) or getattr(x, "dim", lambda: 0)() != 4:
        raise ValueError("x must be a 4-D NHWC tensor of kind IN_I8 or IN_F16")
    _check_tensor(x, "x", _KIND_DTYPE[x_kind])
    n, h, w, c = x.shape
    if y is not None:
        _check_tensor(y, "y", "int8", (n, h, w, c))
    _check_cuda(("x", x), ("y", y))
    if y is None:
        y = torch.empty((n, h, w, c), dtype=torch.int8, device=x.device)
    if s_out <= 0:
        if s_used is None:
            s_used = torch.empty(1, dtype=torch.float32, device=x.device)
        if workspace is None:
            workspace = torch.empty(64, dtype=torch.uint8, device=x.device)
    _check(load().hatq_quantize_act(_ptr(x), int(x_kind), float(s_in), n, h, w, c, int(hb), float(s_out), _ptr(y),
                                    _ptr(s_used), _ptr(workspace), _stream(stream)))
    return (y, s_used) if s_out <= 0 else y


def set_operand_format(L: PreparedLayer, in_f16: bool, out_f16: bool):
    """hatq_set_operand_format: the layer's operand (in_f16) and / or its
    output codes (out_f16) stored as fp16 values instead of int8."""
    _check(load().hatq_set_operand_format(ctypes.byref(L.struct), int(bool(in_f16)), int(bool(out_f16))))
    return L


def conv2d_i8(x, L: PreparedLayer, y=None, stream=None):
    """hatq_conv2d_i8: convolution + fused requantize epilogue on the INT8 operand x (NHWC; fp16 codes
    for a layer with in_f16)."""
    n, h, w, c = _check_layer_io(x, IN_OPERAND, L, y)
    torch = _torch()
    if y is None:
        y = torch.empty(L.out_shape(n, h, w), dtype=getattr(torch, L.out_dtype), device=x.device)
    _check(load().hatq_conv2d_i8(_ptr(x), n, h, w, ctypes.byref(L.struct), _ptr(y), _stream(stream)))
    return y


def layer(x, x_kind, s_in, L: PreparedLayer, y=None, scratch=None, stream=None):
    """hatq_layer: input transform/quantize (when needed) + conv in one call."""
    n, h, w, c = _check_layer_io(x, x_kind, L, y, scratch)
    torch = _torch()
    if y is None:
        y = torch.empty(L.out_shape(n, h, w), dtype=getattr(torch, L.out_dtype), device=x.device)
    nbytes = 0
    if layer_launches(x_kind, s_in, L) > 1:
        if scratch is None:
            scratch = torch.empty(n * h * w * c, dtype=torch.int8, device=x.device)
        nbytes = scratch.numel() * scratch.element_size()
    _check(load().hatq_layer(_ptr(x), int(x_kind), float(s_in), n, h, w, ctypes.byref(L.struct), _ptr(y),
                             _ptr(scratch), nbytes, _stream(stream)))
    return y


def layer_launches(x_kind, s_in, L: PreparedLayer) -> int:
    return int(load().hatq_layer_launches(int(x_kind), float(s_in), ctypes.byref(L.struct)))


def sync_status(stream=None):
    _check(load().hatq_sync_status(_stream(stream)))


def profile_range(x, hb: int, stream=None):
    """hatq_profile_range on an NHWC int8 code tensor: returns (maxima [n, 2]
    int32: max|x_k|, max|H~ x_k| per image; expands [n] uint8)."""
    import torch
    if x.dtype != torch.int8 or x.dim() != 4 or not x.is_cuda:
        raise ValueError("x must be a CUDA int8 NHWC tensor")
    x = x.contiguous()
    n, h, w, c = x.shape
    maxima = torch.empty((n, 2), dtype=torch.int32, device=x.device)
    expands = torch.empty((n,), dtype=torch.uint8, device=x.device)
    _check(load().hatq_profile_range(_ptr(x), n, h, w, c, hb, _ptr(maxima), _ptr(expands), _stream(stream)))
    return maxima, expands


def select_form(expands, tau=(4, 5)):
    """hatq_select_form: the DH/WH decision of Eq. layerwise_hadamard_selection
    from the per-image indicators (host array or tensor) and tau_sel given as
    (numerator, denominator). Returns (form 'DH' or 'WH', p_l as a Fraction)."""
    from fractions import Fraction
    e = np.ascontiguousarray(expands.cpu().numpy() if hasattr(expands, "cpu") else expands, dtype=np.uint8).ravel()
    form, count = ctypes.c_int(), ctypes.c_int()
    _check(load().hatq_select_form(e.ctypes.data if e.size else None, int(e.size), int(tau[0]), int(tau[1]),
                                   ctypes.byref(form), ctypes.byref(count)))
    return ("WH" if form.value == WH else "DH"), Fraction(count.value, int(e.size))


def selftest_wait(limit_cycles: int, stream=None):
    """hatq_selftest_wait: make one bounded device wait expire on purpose
    (failure-detection test; the next sync_status() raises ERR_TIMEOUT)."""
    _check(load().hatq_selftest_wait(int(limit_cycles), _stream(stream)))


def version() -> int:
    return int(load().hatq_version())


def layer_noalloc(x, x_kind, s_in, L: PreparedLayer, y=None, stream=None):
    """hatq_layer_noalloc: hatq_layer for callers that cannot allocate device
    memory; the staged INT8 operand lives in the library's fixed device array
    (at most HATQ_NOALLOC_MAX_BYTES bytes, shared by all calls)."""
    n, h, w, c = _check_layer_io(x, x_kind, L, y)
    torch = _torch()
    if y is None:
        y = torch.empty(L.out_shape(n, h, w), dtype=getattr(torch, L.out_dtype), device=x.device)
    _check(load().hatq_layer_noalloc(_ptr(x), int(x_kind), float(s_in), n, h, w, ctypes.byref(L.struct), _ptr(y),
                                     _stream(stream)))
    return y


NOALLOC_MAX_BYTES = 32 << 20
