"""PalQuant CPU oracle -- test infrastructure only.

A plain, slow, obviously correct CPU statement of the PalQuant layer (Hu et al.,
arXiv 2208.01944): group-wise activation quantisation (Sec. 3.2, Eq. 2), the
B-bit group convolution of parallel low-precision quantisation (Sec. 4.1), the
de-quantising rescale with the output scale alpha (Sec. 3.2), the cyclic
permutation of the cyclic shuffle (Sec. 4.2, Eq. 6-8) and requantisation for the
next layer.  The arithmetic lives in ``palquant_oracle.c`` (int64 nested loops,
fp32 decisions made exactly as written there); this module only builds that file
with gcc and marshals numpy arrays to it.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It imports nothing from the GPU library and
the GPU library imports nothing from it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "palquant_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

# Compiler flags: no contraction of a*b+c into fused multiply-adds and no fast
# math, so every fp32 decision is one IEEE round-to-nearest operation.
CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC", "-shared"]


def build(force: bool = False, src: str = _SRC, out: str = _SO) -> str:
    """Compile the oracle C file into a shared library (gcc) and return its path."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, src, "-lm"])
        os.replace(tmp, out)
    return out


_I64 = ctypes.c_int64
_I32 = ctypes.c_int
_P = ctypes.c_void_p


def _declare(lib):
    lib.oracle_num_threads.restype = _I32
    lib.oracle_set_num_threads.argtypes = [_I32]
    lib.oracle_quantize_act.argtypes = [_P, _P, _I64, _I64, _I64, _I32, _I32, _I32, _P]
    lib.oracle_quantize_weights.argtypes = [_P, _P, _I32, _I32, _I32, _I32, _I32, _I32, _P]
    lib.oracle_group_conv.restype = _I64
    lib.oracle_group_conv.argtypes = [_P, _P, _P, _I64, _I64, _I64] + [_I32] * 7
    lib.oracle_group_conv_pixels.argtypes = [_P, _P, _P, _P, _I64, _I64, _I64, _I64] + [_I32] * 7
    lib.oracle_group_perm.restype = _I32
    lib.oracle_group_perm.argtypes = [_I32, _I32, _I32, _P, _P]
    lib.oracle_epilogue.restype = _I32
    lib.oracle_epilogue.argtypes = [_P, _I64, _I32, _I32, _P, _P, _I32, _I32, _P, _P, _I32, _I32, _P, _P, _P]
    lib.oracle_act_step.argtypes = [_P, _I64, _I64, _I64, _I32, _I32, _I32, _P]
    lib.oracle_weight_step.argtypes = [_P, _I32, _I64, _I32, _P]
    lib.oracle_inv_step.restype = ctypes.c_float
    lib.oracle_inv_step.argtypes = [ctypes.c_float]
    lib.oracle_epilogue_scales.restype = _I32
    lib.oracle_epilogue_scales.argtypes = [_I32, _P, _P, ctypes.c_double, _P, _I32, _I32, _P, _P, _P]
    lib.oracle_quantize_weights_odd.argtypes = [_P, _P, _I32, _I64, _I32, _P]
    lib.oracle_fake_quant_fwd.argtypes = [_P, _P, _I64, _I32, _I64, _I32, _I32, _P, _P]
    lib.oracle_quantize_act_lu.argtypes = [_P, _P, _I64, _I32, _I64, _I32, _P, _P]
    lib.oracle_fake_quant_bwd.argtypes = [_P, _P, _P, _P, _P, _I64, _I32, _I64, _I32, _I32, _P, _P]
    lib.oracle_conv2d_f32.argtypes = [_P, _P, _P, _I64, _I64, _I64, _I32, _I32, _I32, _I32, _I32, _I32]
    lib.oracle_maxpool_f32.argtypes = [_P, _P, _I64, _I64, _I64, _I32, _I32, _I32, _I32]
    lib.oracle_avgpool_f32.argtypes = [_P, _P, _I64, _I64, _I64, _I32]
    lib.oracle_linear_f32.argtypes = [_P, _P, _P, _I64, _I32, _I32]
    return lib


def lib():
    """The loaded oracle library (built on first use)."""
    global _lib
    with _lock:
        if _lib is None:
            _lib = _declare(ctypes.CDLL(build()))
        return _lib


def load_variant(path: str):
    """Load another build of the oracle source (used by the mutation tests)."""
    return _declare(ctypes.CDLL(path))


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return a.ctypes.data


def _f32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32))


def out_dim(n: int, k: int, s: int, p: int) -> int:
    return (n + 2 * p - k) // s + 1


def num_threads(L=None) -> int:
    return (L or lib()).oracle_num_threads()


def set_num_threads(n: int, L=None) -> None:
    (L or lib()).oracle_set_num_threads(int(n))


def quantize_act(x: np.ndarray, G: int, bits: int, inv_s, L=None) -> np.ndarray:
    """Eq. 2 per group: codes = clamp(rint(x * inv_s[g]), 0, 2^bits - 1); x is NHWC fp32."""
    L = L or lib()
    x = _f32(x)
    N, H, W, C = x.shape
    assert C % G == 0
    inv_s = _f32(inv_s)
    assert inv_s.shape == (G,)
    q = np.empty(x.shape, dtype=np.uint8)
    L.oracle_quantize_act(_ptr(x), _ptr(q), N, H, W, G, C // G, bits, _ptr(inv_s))
    return q


def quantize_weights(w: np.ndarray, bits: int, inv_sw, L=None) -> np.ndarray:
    """Signed codes clamp(rint(w * inv_sw[g]), -2^(b-1), 2^(b-1)-1); w is [G,Cout_g,kh,kw,Cin_g]."""
    L = L or lib()
    w = _f32(w)
    G, Co, kh, kw, Ci = w.shape
    inv_sw = _f32(inv_sw)
    assert inv_sw.shape == (G,)
    wq = np.empty(w.shape, dtype=np.int8)
    L.oracle_quantize_weights(_ptr(w), _ptr(wq), G, Co, kh, kw, Ci, bits, _ptr(inv_sw))
    return wq


def group_conv(q: np.ndarray, wq: np.ndarray, stride: int, pad: int, L=None) -> np.ndarray:
    """B-bit group convolution (Sec. 4.1) in int64: returns acc [N,Ho,Wo,G*Cout_g]."""
    L = L or lib()
    q = np.ascontiguousarray(q, dtype=np.uint8)
    wq = np.ascontiguousarray(wq, dtype=np.int8)
    N, H, W, C = q.shape
    G, Co, kh, kw, Ci = wq.shape
    assert C == G * Ci
    Ho, Wo = out_dim(H, kh, stride, pad), out_dim(W, kw, stride, pad)
    acc = np.empty((N, Ho, Wo, G * Co), dtype=np.int64)
    L.oracle_group_conv(_ptr(q), _ptr(wq), _ptr(acc), N, H, W, G, Ci, Co, kh, kw, stride, pad)
    return acc


def group_conv_pixels(q: np.ndarray, wq: np.ndarray, stride: int, pad: int, pix: np.ndarray, L=None) -> np.ndarray:
    """The group convolution at selected output pixels (flat index (n*Ho+oh)*Wo+ow)."""
    L = L or lib()
    q = np.ascontiguousarray(q, dtype=np.uint8)
    wq = np.ascontiguousarray(wq, dtype=np.int8)
    pix = np.ascontiguousarray(pix, dtype=np.int64)
    N, H, W, C = q.shape
    G, Co, kh, kw, Ci = wq.shape
    acc = np.empty((pix.shape[0], G * Co), dtype=np.int64)
    L.oracle_group_conv_pixels(_ptr(q), _ptr(wq), _ptr(acc), _ptr(pix), pix.shape[0], N, H, W, G, Ci, Co, kh, kw, stride, pad)
    return acc


def group_perm(G: int, kind: int = 1, shift: int = 1, perm=None, L=None) -> np.ndarray:
    """Destination group of every source group (Eq. 6 for kind 1, shift 1)."""
    L = L or lib()
    p = None if perm is None else np.ascontiguousarray(perm, dtype=np.int32)
    dst = np.empty(G, dtype=np.int32)
    rc = L.oracle_group_perm(G, kind, shift, _ptr(p), _ptr(dst))
    if rc != 0:
        raise ValueError("shuffle spec is not a permutation")
    return dst


def epilogue(acc: np.ndarray, G: int, m_out, m_req=None, kind: int = 1, shift: int = 1, perm=None,
             shortcut: np.ndarray | None = None, relu: bool = True, bits_out: int = 2, L=None):
    """Rescale, optional shortcut add, ReLU, output permutation and requantisation.

    acc is [..., G*Cout_g] int64; returns (acc_out int32, y_out fp32, q_out uint8) in the
    permuted channel order (q_out is None when m_req is None)."""
    L = L or lib()
    acc = np.ascontiguousarray(acc, dtype=np.int64)
    shape = acc.shape
    C = shape[-1]
    Co = C // G
    npix = acc.size // C
    m_out = _f32(m_out)
    m_req_a = None if m_req is None else _f32(m_req)
    p = None if perm is None else np.ascontiguousarray(perm, dtype=np.int32)
    sc = None if shortcut is None else _f32(shortcut)
    if sc is not None:
        assert sc.shape == shape
    acc_out = np.empty(shape, dtype=np.int32)
    y_out = np.empty(shape, dtype=np.float32)
    q_out = None if m_req_a is None else np.empty(shape, dtype=np.uint8)
    rc = L.oracle_epilogue(_ptr(acc), npix, G, Co, _ptr(m_out), _ptr(m_req_a), kind, shift, _ptr(p), _ptr(sc),
                           int(bool(relu)), bits_out, _ptr(acc_out), _ptr(y_out), _ptr(q_out))
    if rc != 0:
        raise ValueError("oracle epilogue rejected its input (|acc| >= 2^24 or bad shuffle)")
    return acc_out, y_out, q_out


def act_step(x: np.ndarray, G: int, bits: int, L=None) -> np.ndarray:
    """LSQ step initialisation per group: 2*mean(x_g)/sqrt(2^b-1), mean in double."""
    L = L or lib()
    x = _f32(x)
    N, H, W, C = x.shape
    s = np.empty(G, dtype=np.float32)
    L.oracle_act_step(_ptr(x), N, H, W, G, C // G, bits, _ptr(s))
    return s


def weight_step(w: np.ndarray, bits: int, L=None) -> np.ndarray:
    """LSQ step initialisation per group: 2*mean|w_g|/sqrt(2^(b-1)-1), mean in double."""
    L = L or lib()
    w = _f32(w)
    G = w.shape[0]
    s = np.empty(G, dtype=np.float32)
    L.oracle_weight_step(_ptr(w), G, w.size // G, bits, _ptr(s))
    return s


def inv_step(s) -> np.ndarray:
    """fl(1/s) computed in double, the multiplier both implementations use."""
    L = lib()
    return np.array([L.oracle_inv_step(float(v)) for v in np.asarray(s, dtype=np.float32)], dtype=np.float32)


def epilogue_scales(s_w, s_a, s_next=None, alpha: float = 1.0, kind: int = 1, shift: int = 1, perm=None, L=None):
    """(m_out, m_req): fl(s_w s_a alpha) and fl(s_w s_a alpha / s_next[dst(g)])."""
    L = L or lib()
    s_w, s_a = _f32(s_w), _f32(s_a)
    G = s_w.shape[0]
    sn = None if s_next is None else _f32(s_next)
    p = None if perm is None else np.ascontiguousarray(perm, dtype=np.int32)
    m_out = np.empty(G, dtype=np.float32)
    m_req = np.empty(G, dtype=np.float32)
    rc = L.oracle_epilogue_scales(G, _ptr(s_w), _ptr(s_a), float(alpha), _ptr(sn), kind, shift, _ptr(p), _ptr(m_out), _ptr(m_req))
    if rc != 0:
        raise ValueError("bad shuffle spec")
    return m_out, (m_req if sn is not None else None)


def layer(x_codes: np.ndarray, wq: np.ndarray, stride: int, pad: int, m_out, m_req=None, kind: int = 1,
          shift: int = 1, perm=None, shortcut=None, relu: bool = True, bits_out: int = 2, L=None):
    """One PalQuant layer on codes: group conv then the epilogue.  Returns (acc, y, q)."""
    G = wq.shape[0]
    acc = group_conv(x_codes, wq, stride, pad, L=L)
    return epilogue(acc, G, m_out, m_req, kind, shift, perm, shortcut, relu, bits_out, L=L)


# ---------------------------------------------------------------------------
# Full-precision layers around the PalQuant body (the paper keeps the first and
# last layers in full precision, Sec. 5).  Fixed summation orders, see the C file.
# ---------------------------------------------------------------------------
def conv2d_f32(x: np.ndarray, w: np.ndarray, stride: int, pad: int, relu: bool = False, L=None) -> np.ndarray:
    """NHWC fp32 convolution, w [Cout,k,k,Cin]; fmaf over (kh, kw, ci) in order."""
    L = L or lib()
    x, w = _f32(x), _f32(w)
    N, H, W, Ci = x.shape
    Co, k, k2, Ci2 = w.shape
    assert k == k2 and Ci == Ci2
    Ho, Wo = out_dim(H, k, stride, pad), out_dim(W, k, stride, pad)
    y = np.empty((N, Ho, Wo, Co), dtype=np.float32)
    L.oracle_conv2d_f32(_ptr(x), _ptr(w), _ptr(y), N, H, W, Ci, Co, k, stride, pad, int(bool(relu)))
    return y


def maxpool_f32(x: np.ndarray, k: int, stride: int, pad: int, L=None) -> np.ndarray:
    L = L or lib()
    x = _f32(x)
    N, H, W, C = x.shape
    y = np.empty((N, out_dim(H, k, stride, pad), out_dim(W, k, stride, pad), C), dtype=np.float32)
    L.oracle_maxpool_f32(_ptr(x), _ptr(y), N, H, W, C, k, stride, pad)
    return y


def avgpool_f32(x: np.ndarray, L=None) -> np.ndarray:
    L = L or lib()
    x = _f32(x)
    N, H, W, C = x.shape
    y = np.empty((N, C), dtype=np.float32)
    L.oracle_avgpool_f32(_ptr(x), _ptr(y), N, H, W, C)
    return y


def linear_f32(x: np.ndarray, w: np.ndarray, L=None) -> np.ndarray:
    L = L or lib()
    x, w = _f32(x), _f32(w)
    N, Ci = x.shape
    Co = w.shape[0]
    assert w.shape == (Co, Ci)
    y = np.empty((N, Co), dtype=np.float32)
    L.oracle_linear_f32(_ptr(x), _ptr(w), _ptr(y), N, Ci, Co)
    return y


# ---------------------------------------------------------------------------
# Cyclic shuffle module (Sec. 4.2, Eq. 9-10): Y = CyclicPermute(X) by Eq. 8,
# Z = X + Conv1x1(Y) with the 1x1 convolution a PalQuant group convolution.
# ---------------------------------------------------------------------------
def permute_groups(t: np.ndarray, G: int, shift: int = 1, L=None) -> np.ndarray:
    """Eq. 8 on the channel axis of an NHWC tensor: Y[..., pi(i) block] = X[..., i block],
    pi(i) = (i + shift) mod G (Eq. 6 for shift 1)."""
    dst = group_perm(G, 1, shift, L=L)
    C = t.shape[-1]
    Cg = C // G
    y = np.empty_like(t)
    for i in range(G):
        y[..., dst[i] * Cg:(dst[i] + 1) * Cg] = t[..., i * Cg:(i + 1) * Cg]
    return y


def cyclic_shuffle_module(x: np.ndarray, q: np.ndarray, wq: np.ndarray, m_out, m_req=None, shift: int = 1,
                          relu: bool = False, bits_out: int = 2, L=None):
    """Z = X + Conv1x1(CyclicPermute(X)) on a quantised layer: the codes q of X are
    permuted by Eq. 8, convolved by the 1x1 group convolution wq [G, C_g, 1, 1, C_g],
    rescaled by m_out and added to the fp32 X (Eq. 10), optional ReLU; with m_req, the
    codes of Z for the next layer (requantised from the sum).  Returns (z, codes or None)."""
    G = wq.shape[0]
    y = permute_groups(q, G, shift, L=L)
    acc = group_conv(y, wq, 1, 0, L=L)
    _, z, codes = epilogue(acc, G, m_out, m_req, 0, 0, None, x, relu, bits_out, L=L)
    return z, codes


# ---------------------------------------------------------------------------
# Bit-level decomposition (Sec. 3.3, Eq. 4): an M-bit layer run as G^2 B-bit
# products, G = ceil(M / B), shifted and summed:
#   Y = sum_i sum_j X_i W_j^T 2^((i + j) B)
# with X_i, W_j the B-bit slices of the M-bit codes.
# ---------------------------------------------------------------------------
def bit_slices_act(q: np.ndarray, bits_m: int, bits_b: int) -> list:
    """Unsigned M-bit codes -> [X_0, ..., X_{G-1}], x = sum_i X_i 2^(i B), X_i in [0, 2^B - 1]."""
    G = -(-bits_m // bits_b)
    q = np.asarray(q).astype(np.int64)
    return [((q >> (i * bits_b)) & ((1 << bits_b) - 1)).astype(np.uint8) for i in range(G)]


def bit_slices_weights(wq: np.ndarray, bits_m: int, bits_b: int) -> list:
    """Signed M-bit codes -> [W_0, ..., W_{G-1}], w = sum_j W_j 2^(j B): the lower slices
    unsigned in [0, 2^B - 1], the top slice the signed remainder (two's complement)."""
    G = -(-bits_m // bits_b)
    w = np.asarray(wq).astype(np.int64)
    out = []
    for j in range(G):
        if j < G - 1:
            out.append(((w >> (j * bits_b)) & ((1 << bits_b) - 1)).astype(np.int8))
        else:
            out.append((w >> (j * bits_b)).astype(np.int8))  # arithmetic shift keeps the sign
    return out


def bitsplit_conv(q: np.ndarray, wq: np.ndarray, stride: int, pad: int, bits_m: int, bits_b: int, L=None) -> np.ndarray:
    """Eq. 4: the M-bit convolution as G^2 B-bit convolutions, each shifted by 2^((i+j)B)
    and summed (int64)."""
    xs = bit_slices_act(q, bits_m, bits_b)
    ws = bit_slices_weights(wq, bits_m, bits_b)
    acc = None
    for i, xi in enumerate(xs):
        for j, wj in enumerate(ws):
            part = group_conv(xi, wj, stride, pad, L=L) << ((i + j) * bits_b)
            acc = part if acc is None else acc + part
    return acc


def quantize_weights_odd(w: np.ndarray, bits: int, u, L=None) -> np.ndarray:
    """The paper's weight quantiser (Eq. 2, Eq. 3's weight form): odd integer codes
    2 x_q - (2^b - 1), x_q = clamp(rint((w + u[g]) * fl((2^b-1) / (2 u[g]))), 0, 2^b - 1)."""
    L = L or lib()
    w = _f32(w)
    u = _f32(u)
    G = w.shape[0]
    assert u.shape == (G,)
    wq = np.empty(w.shape, dtype=np.int8)
    L.oracle_quantize_weights_odd(_ptr(w), _ptr(wq), G, w.size // G, bits, _ptr(u))
    return wq


def fake_quant_forward(x: np.ndarray, G: int, bits: int, kind: int, l, u, L=None) -> np.ndarray:
    """Quantisation-aware training forward (Eq. 2-3 with learned bounds l, u per
    group; kind 0 activations in [0, 1], kind 1 weights in [-1, 1]).  x: [..., G*Cg]."""
    L = L or lib()
    x = _f32(x)
    l, u = _f32(l), _f32(u)
    C = x.shape[-1]
    assert C % G == 0 and l.shape == (G,) and u.shape == (G,)
    out = np.empty_like(x)
    L.oracle_fake_quant_fwd(_ptr(x), _ptr(out), x.size // C, G, C // G, bits, kind, _ptr(l), _ptr(u))
    return out


def fake_quant_backward(x: np.ndarray, dy: np.ndarray, G: int, bits: int, kind: int, l, u, L=None):
    """Its straight-through backward: (dx fp32, dl [G] float64, du [G] float64)."""
    L = L or lib()
    x, dy = _f32(x), _f32(dy)
    l, u = _f32(l), _f32(u)
    assert x.shape == dy.shape
    C = x.shape[-1]
    assert C % G == 0 and l.shape == (G,) and u.shape == (G,)
    dx = np.empty_like(x)
    dl = np.empty(G, dtype=np.float64)
    du = np.empty(G, dtype=np.float64)
    L.oracle_fake_quant_bwd(_ptr(x), _ptr(dy), _ptr(dx), _ptr(dl), _ptr(du), x.size // C, G, C // G, bits, kind,
                            _ptr(l), _ptr(u))
    return dx, dl, du


def quantize_act_lu(x: np.ndarray, G: int, bits: int, l, u, L=None) -> np.ndarray:
    """Inference codes with learned per-group bounds l < u (Eq. 2): the training
    forward's x_q, x_q = rint(clamp((x - l) * fl(1/fl(u - l)), 0, 1) * (2^b - 1)).
    x: [..., G*Cg] fp32 -> uint8 codes of the same shape."""
    L = L or lib()
    x = _f32(x)
    l, u = _f32(l), _f32(u)
    C = x.shape[-1]
    assert C % G == 0 and l.shape == (G,) and u.shape == (G,)
    q = np.empty(x.shape, dtype=np.uint8)
    L.oracle_quantize_act_lu(_ptr(x), _ptr(q), x.size // C, G, C // G, bits, _ptr(l), _ptr(u))
    return q
