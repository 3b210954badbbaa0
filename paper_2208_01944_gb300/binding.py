"""Thin ctypes binding of libpalquant.so (include/palquant.h).

Functions keep the C names and argument order.  They only marshal arguments:
device buffers are passed as ``torch.Tensor`` (their ``data_ptr()``) or raw integer
addresses, host arrays as numpy arrays or sequences, streams as ``torch.cuda.Stream``
or raw handles (default: torch's current stream).  A non-OK status raises
:class:`PalquantError`.  Every computation happens in the CUDA library; if it has
not been built, importing this module raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libpalquant.so")

PQ_OK, PQ_EINVAL, PQ_EUNSUPPORTED, PQ_ECUDA, PQ_ETIMEOUT = 0, -1, -2, -3, -4
PQ_CODES_INT8, PQ_CODES_E4M3, PQ_CODES_C16, PQ_CODES_C16P2, PQ_CODES_C32F4 = 0, 1, 2, 3, 4
PQ_LAYER_INPUTS_READY = 1  # pq_layer_desc.flags: the previous kernel on the stream writes neither input nor weights

# Every symbol include/palquant.h declares.
EXPORTS = [
    "palquant_strerror", "palquant_version", "palquant_act_steps_scratch_bytes", "palquant_act_steps",
    "palquant_act_steps_noalloc",
    "palquant_weight_steps", "palquant_epilogue_scales", "palquant_packed_weight_bytes",
    "palquant_pack_weights_host", "palquant_pack_weights", "palquant_pack_weight_codes_host",
    "palquant_unpack_weight_codes_host", "palquant_quantize_act", "palquant_group_conv", "palquant_layer_fused",
    "palquant_quantize_layer_fused",
    "palquant_sync_check", "palquant_set_wait_limit_ns", "palquant_watchdog_selftest", "palquant_conv_plan",
    "palquant_conv2d_f32", "palquant_stem_pool_f32", "palquant_maxpool2d_f32", "palquant_avgpool_f32",
    "palquant_linear_f32",
    "palquant_cyclic_shuffle_module", "palquant_bitsplit_desc", "palquant_bitsplit_scratch_bytes",
    "palquant_bitsplit_pack_weight_codes_host", "palquant_bitsplit_act", "palquant_bitsplit_conv",
    "palquant_pack_weights_odd_host", "palquant_fake_quant_forward", "palquant_fake_quant_scratch_bytes",
    "palquant_fake_quant_backward", "palquant_quantize_act_lu", "palquant_quantize_layer_fused_lu",
]


class PalquantError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {strerror(status)} ({status})")


class LayerDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "N", "H", "W", "G", "Cin_g", "Cout_g", "kh", "kw", "stride", "pad", "bits_a", "bits_w", "bits_out", "relu",
        "code_format", "flags", "wslices")]


class Shuffle(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("shift", ctypes.c_int32), ("perm", ctypes.POINTER(ctypes.c_int32))]


class ConvPlan(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "supported", "mode", "rows_per_tile", "m_tiles", "tile_pitch", "n_block", "n_blocks", "k_chunk", "k_blocks",
        "taps", "weights_resident", "acc_stages", "smem_bytes")] + [("tiles", ctypes.c_int64), ("work_items", ctypes.c_int64),
                                                                     ("pointwise", ctypes.c_int32)]

    def as_dict(self):
        return {name: getattr(self, name) for name, _ in self._fields_}


_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_F32P = ctypes.POINTER(ctypes.c_float)


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run paper_2208_01944_gb300.build.build() (or __graft_entry__.build())")
    L = ctypes.CDLL(LIB_PATH)
    L.palquant_strerror.restype = ctypes.c_char_p
    L.palquant_strerror.argtypes = [_I32]
    L.palquant_version.restype = _I32
    L.palquant_act_steps_scratch_bytes.restype = ctypes.c_size_t
    L.palquant_act_steps_scratch_bytes.argtypes = [_I64, _I32]
    L.palquant_act_steps.restype = _I32
    L.palquant_act_steps.argtypes = [_P, _I64, _I32, _I32, _I32, _I32, _I32, _P, ctypes.c_size_t, _P, _P]
    L.palquant_act_steps_noalloc.restype = _I32
    L.palquant_act_steps_noalloc.argtypes = [_P, _I64, _I32, _I32, _I32, _I32, _I32, _P, _P]
    L.palquant_weight_steps.restype = _I32
    L.palquant_weight_steps.argtypes = [_P, ctypes.POINTER(LayerDesc), _P]
    L.palquant_epilogue_scales.restype = _I32
    L.palquant_epilogue_scales.argtypes = [_I32, _P, _P, ctypes.c_double, _P, Shuffle, _P, _P]
    L.palquant_packed_weight_bytes.restype = ctypes.c_size_t
    L.palquant_packed_weight_bytes.argtypes = [ctypes.POINTER(LayerDesc)]
    L.palquant_pack_weights_host.restype = _I32
    L.palquant_pack_weights_host.argtypes = [_P, ctypes.POINTER(LayerDesc), _P, _P, ctypes.c_size_t]
    L.palquant_pack_weights.restype = _I32
    L.palquant_pack_weights.argtypes = [_P, ctypes.POINTER(LayerDesc), _P, _P, ctypes.c_size_t, _P]
    L.palquant_pack_weight_codes_host.restype = _I32
    L.palquant_pack_weight_codes_host.argtypes = [_P, ctypes.POINTER(LayerDesc), _P, ctypes.c_size_t]
    L.palquant_unpack_weight_codes_host.restype = _I32
    L.palquant_unpack_weight_codes_host.argtypes = [_P, ctypes.POINTER(LayerDesc), _P]
    L.palquant_quantize_act.restype = _I32
    L.palquant_quantize_act.argtypes = [_P, _P, _I64, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P]
    L.palquant_group_conv.restype = _I32
    L.palquant_group_conv.argtypes = [_P, _P, _P, ctypes.POINTER(LayerDesc), _P]
    L.palquant_layer_fused.restype = _I32
    L.palquant_layer_fused.argtypes = [_P, _P, ctypes.POINTER(LayerDesc), _P, _P, Shuffle, _P, _P, _P, _P, _P]
    L.palquant_quantize_layer_fused.restype = _I32
    L.palquant_quantize_layer_fused.argtypes = [_P, _P, _P, ctypes.POINTER(LayerDesc), _P, _P, Shuffle, _P, _P, _P, _P,
                                                _P]
    L.palquant_sync_check.restype = _I32
    L.palquant_sync_check.argtypes = [_P]
    L.palquant_set_wait_limit_ns.restype = _I32
    L.palquant_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
    L.palquant_watchdog_selftest.restype = _I32
    L.palquant_watchdog_selftest.argtypes = [ctypes.c_uint64, _P]
    L.palquant_conv_plan.restype = _I32
    L.palquant_conv_plan.argtypes = [ctypes.POINTER(LayerDesc), ctypes.POINTER(ConvPlan)]
    L.palquant_pack_weights_odd_host.restype = _I32
    L.palquant_pack_weights_odd_host.argtypes = [_P, ctypes.POINTER(LayerDesc), _P, _P, ctypes.c_size_t]
    L.palquant_bitsplit_desc.restype = _I32
    L.palquant_bitsplit_desc.argtypes = [ctypes.POINTER(LayerDesc), _I32, ctypes.POINTER(LayerDesc)]
    L.palquant_bitsplit_scratch_bytes.restype = ctypes.c_size_t
    L.palquant_bitsplit_scratch_bytes.argtypes = [ctypes.POINTER(LayerDesc), _I32]
    L.palquant_bitsplit_pack_weight_codes_host.restype = _I32
    L.palquant_bitsplit_pack_weight_codes_host.argtypes = [_P, ctypes.POINTER(LayerDesc), _I32, _P, ctypes.c_size_t]
    L.palquant_bitsplit_act.restype = _I32
    L.palquant_bitsplit_act.argtypes = [_P, _P, ctypes.c_size_t, ctypes.POINTER(LayerDesc), _I32, _P]
    L.palquant_bitsplit_conv.restype = _I32
    L.palquant_bitsplit_conv.argtypes = [_P, _P, ctypes.c_size_t, _P, _P, ctypes.POINTER(LayerDesc), _I32, _P]
    L.palquant_cyclic_shuffle_module.restype = _I32
    L.palquant_cyclic_shuffle_module.argtypes = [_P, _P, ctypes.POINTER(LayerDesc), _P, _P, _I32, _P, _P, _P, _P]
    for name, args in (("palquant_conv2d_f32", [_P, _P, _P, _I64] + [_I32] * 8 + [_P]),
                       ("palquant_stem_pool_f32", [_P, _P, _P, _P, _I64, _I32, _I32, _I32, _P]),
                       ("palquant_maxpool2d_f32", [_P, _P, _I64] + [_I32] * 6 + [_P]),
                       ("palquant_avgpool_f32", [_P, _P, _I64, _I32, _I32, _I32, _P]),
                       ("palquant_linear_f32", [_P, _P, _P, _I64, _I32, _I32, _P])):
        getattr(L, name).restype = _I32
        getattr(L, name).argtypes = args
    L.palquant_quantize_act_lu.restype = _I32
    L.palquant_quantize_act_lu.argtypes = [_P, _P, _I64, _I32, _I32, _I32, _I32, _I32, _I32, _P, _P, _P]
    L.palquant_quantize_layer_fused_lu.restype = _I32
    L.palquant_quantize_layer_fused_lu.argtypes = list(L.palquant_quantize_layer_fused.argtypes[:1]) + [_P, _P] + \
        list(L.palquant_quantize_layer_fused.argtypes[2:])
    L.palquant_fake_quant_forward.restype = _I32
    L.palquant_fake_quant_forward.argtypes = [_P, _P, _I64, _I32, _I32, _I32, _I32, _P, _P, _P]
    L.palquant_fake_quant_scratch_bytes.restype = ctypes.c_size_t
    L.palquant_fake_quant_scratch_bytes.argtypes = [_I64, _I32, _I32]
    L.palquant_fake_quant_backward.restype = _I32
    L.palquant_fake_quant_backward.argtypes = [_P, _P, _P, _P, _P, _I64, _I32, _I32, _I32, _I32, _P, _P, _P,
                                               ctypes.c_size_t, _P]
    return L


lib = _load()


# ----------------------------------------------------------------- marshalling
def _ptr(obj):
    """Device or host address of a tensor / array / int (None -> NULL)."""
    if obj is None:
        return None
    if isinstance(obj, int):
        return obj
    if isinstance(obj, np.ndarray):
        assert obj.flags["C_CONTIGUOUS"]
        return obj.ctypes.data
    if hasattr(obj, "data_ptr"):
        assert obj.is_contiguous(), "tensors passed to libpalquant must be contiguous"
        return obj.data_ptr()
    raise TypeError(f"cannot pass {type(obj)} as a pointer")


def _stream(stream):
    if stream is None:
        import torch

        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def _check(status: int, where: str):
    if status != PQ_OK:
        raise PalquantError(status, where)


def strerror(status: int) -> str:
    return lib.palquant_strerror(status).decode()


def layer_desc(N, H, W, G, Cin_g, Cout_g, k, stride=1, pad=0, bits_a=2, bits_w=2, bits_out=2, relu=1,
               code_format=PQ_CODES_INT8, kw=None, flags=0) -> LayerDesc:
    return LayerDesc(N, H, W, G, Cin_g, Cout_g, k, k if kw is None else kw, stride, pad, bits_a, bits_w, bits_out,
                     int(relu), code_format, int(flags), 0)


def shuffle(kind=1, shift=1, perm=None):
    """pq_shuffle; the returned pair keeps the permutation array alive."""
    arr = None if perm is None else (ctypes.c_int32 * len(perm))(*[int(v) for v in perm])
    s = Shuffle(kind, shift, ctypes.cast(arr, ctypes.POINTER(ctypes.c_int32)) if arr is not None else None)
    s._keep = arr
    return s


# ------------------------------------------------------------------ the ABI
def palquant_version() -> int:
    return lib.palquant_version()


def palquant_act_steps_scratch_bytes(P: int, G: int) -> int:
    return lib.palquant_act_steps_scratch_bytes(P, G)


def palquant_act_steps(x_dev, N, H, W, G, Cg, bits, scratch_dev, scratch_bytes, stream=None) -> np.ndarray:
    out = np.empty(G, dtype=np.float32)
    _check(lib.palquant_act_steps(_ptr(x_dev), N, H, W, G, Cg, bits, _ptr(scratch_dev), scratch_bytes, _ptr(out),
                                  _stream(stream)), "palquant_act_steps")
    return out


def palquant_act_steps_noalloc(x_dev, N, H, W, G, Cg, bits, stream=None) -> np.ndarray:
    """Per-group activation steps without any device allocation (fixed library scratch)."""
    out = np.empty(G, dtype=np.float32)
    _check(lib.palquant_act_steps_noalloc(_ptr(x_dev), N, H, W, G, Cg, bits, _ptr(out), _stream(stream)),
           "palquant_act_steps_noalloc")
    return out


def palquant_weight_steps(w_host: np.ndarray, d: LayerDesc) -> np.ndarray:
    w = _f32(w_host)
    out = np.empty(d.G, dtype=np.float32)
    _check(lib.palquant_weight_steps(_ptr(w), ctypes.byref(d), _ptr(out)), "palquant_weight_steps")
    return out


def palquant_epilogue_scales(G, s_w, s_a, alpha=1.0, s_next=None, shuf=None):
    s_w, s_a = _f32(s_w), _f32(s_a)
    sn = None if s_next is None else _f32(s_next)
    m_out = np.empty(G, dtype=np.float32)
    m_req = np.empty(G, dtype=np.float32)
    _check(lib.palquant_epilogue_scales(G, _ptr(s_w), _ptr(s_a), float(alpha), _ptr(sn), shuf or shuffle(0, 0),
                                        _ptr(m_out), _ptr(m_req)), "palquant_epilogue_scales")
    return m_out, (m_req if sn is not None else None)


def palquant_packed_weight_bytes(d: LayerDesc) -> int:
    return lib.palquant_packed_weight_bytes(ctypes.byref(d))


def palquant_pack_weights_host(w_host, d: LayerDesc, inv_sw) -> np.ndarray:
    n = palquant_packed_weight_bytes(d)
    if n == 0:
        raise PalquantError(PQ_EUNSUPPORTED, "palquant_packed_weight_bytes")
    out = np.empty(n, dtype=np.uint8)
    w, inv = _f32(w_host), _f32(inv_sw)
    _check(lib.palquant_pack_weights_host(_ptr(w), ctypes.byref(d), _ptr(inv), _ptr(out), n), "palquant_pack_weights_host")
    return out


def palquant_pack_weights(w_host, d: LayerDesc, inv_sw, packed_dev, packed_bytes, stream=None):
    w, inv = _f32(w_host), _f32(inv_sw)
    _check(lib.palquant_pack_weights(_ptr(w), ctypes.byref(d), _ptr(inv), _ptr(packed_dev), packed_bytes,
                                     _stream(stream)), "palquant_pack_weights")


def palquant_pack_weight_codes_host(wq_host, d: LayerDesc) -> np.ndarray:
    n = palquant_packed_weight_bytes(d)
    if n == 0:
        raise PalquantError(PQ_EUNSUPPORTED, "palquant_packed_weight_bytes")
    out = np.empty(n, dtype=np.uint8)
    wq = np.ascontiguousarray(wq_host, dtype=np.int8)
    _check(lib.palquant_pack_weight_codes_host(_ptr(wq), ctypes.byref(d), _ptr(out), n), "palquant_pack_weight_codes_host")
    return out


def palquant_unpack_weight_codes_host(packed_host, d: LayerDesc) -> np.ndarray:
    """[G][Cout_g][kh][kw][Cin_g], or [G][Cout_g][kh][kw][R][Cin_g] with R = d.wslices > 1 weight slices."""
    R = d.wslices if d.wslices > 1 else 1
    shape = (d.G, d.Cout_g, d.kh, d.kw, d.Cin_g) if R == 1 else (d.G, d.Cout_g, d.kh, d.kw, R, d.Cin_g)
    out = np.empty(shape, dtype=np.int8)
    pk = np.ascontiguousarray(packed_host, dtype=np.uint8)
    _check(lib.palquant_unpack_weight_codes_host(_ptr(pk), ctypes.byref(d), _ptr(out)), "palquant_unpack_weight_codes_host")
    return out


def palquant_quantize_act(x_dev, q_dev, N, H, W, G, Cg, bits, inv_s, code_format=PQ_CODES_INT8, stream=None):
    inv = _f32(inv_s)
    _check(lib.palquant_quantize_act(_ptr(x_dev), _ptr(q_dev), N, H, W, G, Cg, bits, code_format, _ptr(inv),
                                     _stream(stream)), "palquant_quantize_act")


def palquant_group_conv(q_dev, w_packed_dev, acc_dev, d: LayerDesc, stream=None):
    _check(lib.palquant_group_conv(_ptr(q_dev), _ptr(w_packed_dev), _ptr(acc_dev), ctypes.byref(d), _stream(stream)),
           "palquant_group_conv")


def palquant_layer_fused(q_dev, w_packed_dev, d: LayerDesc, m_out, m_req=None, shuf=None, shortcut_dev=None,
                         acc_out_dev=None, y_out_dev=None, q_out_dev=None, stream=None):
    mo = None if m_out is None else _f32(m_out)
    mr = None if m_req is None else _f32(m_req)
    _check(lib.palquant_layer_fused(_ptr(q_dev), _ptr(w_packed_dev), ctypes.byref(d), _ptr(mo), _ptr(mr),
                                    shuf or shuffle(1, 1), _ptr(shortcut_dev), _ptr(acc_out_dev), _ptr(y_out_dev),
                                    _ptr(q_out_dev), _stream(stream)), "palquant_layer_fused")


def palquant_quantize_layer_fused(x_dev, inv_s, w_packed_dev, d: LayerDesc, m_out, m_req=None, shuf=None,
                                  shortcut_dev=None, acc_out_dev=None, y_out_dev=None, q_out_dev=None, stream=None):
    inv = _f32(inv_s)
    mo = None if m_out is None else _f32(m_out)
    mr = None if m_req is None else _f32(m_req)
    _check(lib.palquant_quantize_layer_fused(_ptr(x_dev), _ptr(inv), _ptr(w_packed_dev), ctypes.byref(d), _ptr(mo),
                                             _ptr(mr), shuf or shuffle(1, 1), _ptr(shortcut_dev), _ptr(acc_out_dev),
                                             _ptr(y_out_dev), _ptr(q_out_dev), _stream(stream)),
           "palquant_quantize_layer_fused")


def palquant_cyclic_shuffle_module(q_dev, w_packed_dev, d: LayerDesc, m_out, m_req=None, shift=1, x_dev=None,
                                   z_out_dev=None, q_out_dev=None, stream=None):
    mo = None if m_out is None else _f32(m_out)
    mr = None if m_req is None else _f32(m_req)
    _check(lib.palquant_cyclic_shuffle_module(_ptr(q_dev), _ptr(w_packed_dev), ctypes.byref(d), _ptr(mo), _ptr(mr),
                                              int(shift), _ptr(x_dev), _ptr(z_out_dev), _ptr(q_out_dev),
                                              _stream(stream)), "palquant_cyclic_shuffle_module")


def palquant_sync_check(stream=None) -> int:
    return lib.palquant_sync_check(_stream(stream))


def palquant_set_wait_limit_ns(ns: int):
    _check(lib.palquant_set_wait_limit_ns(int(ns)), "palquant_set_wait_limit_ns")


def palquant_watchdog_selftest(limit_ns: int, stream=None) -> int:
    return lib.palquant_watchdog_selftest(int(limit_ns), _stream(stream))


def palquant_conv_plan(d: LayerDesc) -> ConvPlan:
    plan = ConvPlan()
    st = lib.palquant_conv_plan(ctypes.byref(d), ctypes.byref(plan))
    if st not in (PQ_OK, PQ_EUNSUPPORTED):
        raise PalquantError(st, "palquant_conv_plan")
    return plan


# Full-precision layers around the PalQuant body (first and last layers of a network).
def palquant_conv2d_f32(x_dev, w_dev, y_dev, N, H, W, Cin, Cout, k, stride, pad, relu=False, stream=None):
    _check(lib.palquant_conv2d_f32(_ptr(x_dev), _ptr(w_dev), _ptr(y_dev), N, H, W, Cin, Cout, k, stride, pad,
                                   int(bool(relu)), _stream(stream)), "palquant_conv2d_f32")


def palquant_stem_pool_f32(x_dev, w_dev, stem_dev, pool_dev, N, H, W, Cout, stream=None):
    """7x7/2 stem + ReLU and 3x3/2 max pooling in one pass; stem_dev may be None."""
    _check(lib.palquant_stem_pool_f32(_ptr(x_dev), _ptr(w_dev), _ptr(stem_dev) if stem_dev is not None else None,
                                      _ptr(pool_dev), N, H, W, Cout, _stream(stream)), "palquant_stem_pool_f32")


def palquant_maxpool2d_f32(x_dev, y_dev, N, H, W, C, k, stride, pad, stream=None):
    _check(lib.palquant_maxpool2d_f32(_ptr(x_dev), _ptr(y_dev), N, H, W, C, k, stride, pad, _stream(stream)),
           "palquant_maxpool2d_f32")


def palquant_avgpool_f32(x_dev, y_dev, N, H, W, C, stream=None):
    _check(lib.palquant_avgpool_f32(_ptr(x_dev), _ptr(y_dev), N, H, W, C, _stream(stream)), "palquant_avgpool_f32")


def palquant_linear_f32(x_dev, w_dev, y_dev, N, Cin, Cout, stream=None):
    _check(lib.palquant_linear_f32(_ptr(x_dev), _ptr(w_dev), _ptr(y_dev), N, Cin, Cout, _stream(stream)),
           "palquant_linear_f32")


# Bit-level decomposition (Eq. 4): the baseline PalQuant is compared with.
def palquant_bitsplit_desc(d: LayerDesc, bits_b: int) -> LayerDesc:
    out = LayerDesc()
    _check(lib.palquant_bitsplit_desc(ctypes.byref(d), bits_b, ctypes.byref(out)), "palquant_bitsplit_desc")
    return out


def palquant_bitsplit_scratch_bytes(d: LayerDesc, bits_b: int) -> int:
    return lib.palquant_bitsplit_scratch_bytes(ctypes.byref(d), bits_b)


def palquant_bitsplit_pack_weight_codes_host(wq_host, d: LayerDesc, bits_b: int) -> np.ndarray:
    n = palquant_packed_weight_bytes(palquant_bitsplit_desc(d, bits_b))
    out = np.empty(n, dtype=np.uint8)
    wq = np.ascontiguousarray(wq_host, dtype=np.int8)
    _check(lib.palquant_bitsplit_pack_weight_codes_host(_ptr(wq), ctypes.byref(d), bits_b, _ptr(out), n),
           "palquant_bitsplit_pack_weight_codes_host")
    return out


def palquant_bitsplit_act(q_dev, xs_dev, xs_bytes, d: LayerDesc, bits_b: int, stream=None):
    _check(lib.palquant_bitsplit_act(_ptr(q_dev), _ptr(xs_dev), xs_bytes, ctypes.byref(d), bits_b, _stream(stream)),
           "palquant_bitsplit_act")


def palquant_bitsplit_conv(q_dev, xs_dev, xs_bytes, w_packed_dev, acc_dev, d: LayerDesc, bits_b: int, stream=None):
    _check(lib.palquant_bitsplit_conv(_ptr(q_dev), _ptr(xs_dev), xs_bytes, _ptr(w_packed_dev), _ptr(acc_dev),
                                      ctypes.byref(d), bits_b, _stream(stream)), "palquant_bitsplit_conv")


def palquant_pack_weights_odd_host(w_host, d: LayerDesc, u) -> np.ndarray:
    """The paper's odd-level weight quantiser (clip range [-u, u]) and packing."""
    n = palquant_packed_weight_bytes(d)
    if n == 0:
        raise PalquantError(PQ_EUNSUPPORTED, "palquant_packed_weight_bytes")
    out = np.empty(n, dtype=np.uint8)
    w, uu = _f32(w_host), _f32(u)
    _check(lib.palquant_pack_weights_odd_host(_ptr(w), ctypes.byref(d), _ptr(uu), _ptr(out), n),
           "palquant_pack_weights_odd_host")
    return out


# ---------------------------------------------------------------- quantisation-aware training
def palquant_fake_quant_forward(x_dev, xhat_dev, P, G, Cg, bits, kind, l, u, stream=None) -> None:
    """Fake quantisation with learned per-group bounds (Eq. 2-3); kind 0 activations, 1 weights."""
    lf, uf = _f32(l), _f32(u)
    _check(lib.palquant_fake_quant_forward(_ptr(x_dev), _ptr(xhat_dev), P, G, Cg, bits, kind, _ptr(lf), _ptr(uf),
                                           _stream(stream)), "palquant_fake_quant_forward")


def palquant_fake_quant_scratch_bytes(P, G, Cg) -> int:
    return lib.palquant_fake_quant_scratch_bytes(P, G, Cg)


def palquant_fake_quant_backward(x_dev, dy_dev, dx_dev, dl_dev, du_dev, P, G, Cg, bits, kind, l, u, scratch_dev,
                                 scratch_bytes, stream=None) -> None:
    """Straight-through backward: dx (fp32) and the per-group gradients of l and u (G doubles each, device)."""
    lf, uf = _f32(l), _f32(u)
    _check(lib.palquant_fake_quant_backward(_ptr(x_dev), _ptr(dy_dev), _ptr(dx_dev), _ptr(dl_dev), _ptr(du_dev), P, G,
                                            Cg, bits, kind, _ptr(lf), _ptr(uf), _ptr(scratch_dev), scratch_bytes,
                                            _stream(stream)), "palquant_fake_quant_backward")


# ---------------------------------------------------------------- learned bounds at inference
def palquant_quantize_act_lu(x_dev, q_dev, N, H, W, G, Cg, bits, l, u, code_format=PQ_CODES_INT8, stream=None):
    """Activation codes with learned per-group bounds l < u (the training forward's codes)."""
    lf, uf = _f32(l), _f32(u)
    _check(lib.palquant_quantize_act_lu(_ptr(x_dev), _ptr(q_dev), N, H, W, G, Cg, bits, code_format, _ptr(lf),
                                        _ptr(uf), _stream(stream)), "palquant_quantize_act_lu")


def palquant_quantize_layer_fused_lu(x_dev, l, u, w_packed_dev, d: LayerDesc, m_out, m_req=None, shuf=None,
                                     shortcut_dev=None, acc_out_dev=None, y_out_dev=None, q_out_dev=None,
                                     stream=None):
    """Quantise-on-load with learned per-group bounds l < u, then the layer."""
    lf, uf = _f32(l), _f32(u)
    mo = None if m_out is None else _f32(m_out)
    mr = None if m_req is None else _f32(m_req)
    _check(lib.palquant_quantize_layer_fused_lu(_ptr(x_dev), _ptr(lf), _ptr(uf), _ptr(w_packed_dev), ctypes.byref(d),
                                                _ptr(mo), _ptr(mr), shuf or shuffle(1, 1), _ptr(shortcut_dev),
                                                _ptr(acc_out_dev), _ptr(y_out_dev), _ptr(q_out_dev), _stream(stream)),
           "palquant_quantize_layer_fused_lu")
