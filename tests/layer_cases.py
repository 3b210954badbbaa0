"""Shared set-up of PalQuant layer parity cases: seeded inputs, oracle-side
calibration and reference outputs, and the GPU run through the C ABI."""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

import oracle
from paper_2208_01944_gb300 import synth


@dataclass
class Case:
    N: int
    H: int
    W: int
    G: int
    Cin: int
    Cout: int
    k: int
    stride: int = 1
    pad: int = 0
    bits: int = 2
    kind: int = 1
    shift: int = 1
    perm: tuple | None = None
    relu: bool = True
    shortcut: bool = False
    seed: int = 0
    bits_out: int | None = None

    @property
    def Ho(self):
        return (self.H + 2 * self.pad - self.k) // self.stride + 1

    @property
    def Wo(self):
        return (self.W + 2 * self.pad - self.k) // self.stride + 1

    @property
    def bo(self):
        return self.bits if self.bits_out is None else self.bits_out

    def __str__(self):
        return (f"N{self.N}_{self.H}x{self.W}_G{self.G}_c{self.Cin}-{self.Cout}_k{self.k}s{self.stride}p{self.pad}"
                f"_b{self.bits}_sh{self.kind}{'_sc' if self.shortcut else ''}{'' if self.relu else '_norelu'}")


def prepare(c: Case, sample_pix: np.ndarray | None = None):
    """Inputs and oracle results.  With sample_pix, the oracle evaluates only those
    output pixels (flat indices); otherwise all of them."""
    gen = synth.generator(c.seed)
    x = synth.half_normal((c.N, c.H, c.W, c.G * c.Cin), gen)
    w = synth.he_weights(c.G, c.Cout, c.k, c.k, c.Cin, gen)
    shortcut = synth.normal((c.N, c.Ho, c.Wo, c.G * c.Cout), gen) if c.shortcut else None
    s_a = oracle.act_step(x, c.G, c.bits)
    s_w = oracle.weight_step(w, c.bits)
    inv_s, inv_sw = oracle.inv_step(s_a), oracle.inv_step(s_w)
    q = oracle.quantize_act(x, c.G, c.bits, inv_s)
    wq = oracle.quantize_weights(w, c.bits, inv_sw)
    if sample_pix is None:
        acc = oracle.group_conv(q, wq, c.stride, c.pad).reshape(-1, c.G * c.Cout)
    else:
        acc = oracle.group_conv_pixels(q, wq, c.stride, c.pad, sample_pix)
    sc = None if shortcut is None else shortcut.reshape(-1, c.G * c.Cout)
    if sc is not None and sample_pix is not None:
        sc = np.ascontiguousarray(sc[sample_pix])
    # Next layer's steps: calibrated on this layer's (sampled) rescaled output.
    m_out, _ = oracle.epilogue_scales(s_w, s_a, None, 1.0, c.kind, c.shift, c.perm)
    _, y0, _ = oracle.epilogue(acc, c.G, m_out, None, c.kind, c.shift, c.perm, sc, True, c.bo)
    y_grp = y0.reshape(-1, c.G, c.Cout)
    s_next = (2.0 * y_grp.astype(np.float64).mean(axis=(0, 2)) / np.sqrt((1 << c.bo) - 1)).astype(np.float32)
    s_next = np.where(s_next > 0, s_next, np.float32(1.0)).astype(np.float32)
    m_out, m_req = oracle.epilogue_scales(s_w, s_a, s_next, 1.0, c.kind, c.shift, c.perm)
    a_ref, y_ref, q_ref = oracle.epilogue(acc, c.G, m_out, m_req, c.kind, c.shift, c.perm, sc, c.relu, c.bo)
    return dict(x=x, w=w, shortcut=shortcut, s_a=s_a, s_w=s_w, inv_s=inv_s, inv_sw=inv_sw, q=q, wq=wq,
                m_out=m_out, m_req=m_req, acc_ref=a_ref, y_ref=y_ref, q_ref=q_ref)


def c16_to_nhwc(a: np.ndarray, N: int, H: int, W: int, C: int) -> np.ndarray:
    """Channel-blocked codes [N][C/16][H][W][16] -> NHWC (a pure permutation of bytes)."""
    return np.ascontiguousarray(a.reshape(N, C // 16, H, W, 16).transpose(0, 2, 3, 1, 4).reshape(N, H, W, C))


def c16p2_to_nhwc(a: np.ndarray, N: int, H: int, W: int, C: int) -> np.ndarray:
    """Packed channel-blocked 2-bit codes (little-endian 32-bit word per position and
    16-channel block, code of channel c at bits 2 (c % 16)) -> NHWC, one code per byte."""
    words = np.ascontiguousarray(a).view(np.uint32).reshape(N, C // 16, H, W)
    codes = (words[..., None] >> (2 * np.arange(16, dtype=np.uint32))) & 3
    return np.ascontiguousarray(codes.astype(np.uint8).transpose(0, 2, 3, 1, 4).reshape(N, H, W, C))


def c32f4_to_nhwc(a: np.ndarray, N: int, H: int, W: int, C: int) -> np.ndarray:
    """FP4 nibble codes [N][C/32][H][W][16 bytes], channel 2i of a block in the low
    nibble of byte i and 2i+1 in the high nibble -> NHWC, one code per byte."""
    b = np.ascontiguousarray(a).reshape(N, C // 32, H, W, 16)
    codes = np.stack([b & 15, b >> 4], axis=-1).reshape(N, C // 32, H, W, 32)
    return np.ascontiguousarray(codes.astype(np.uint8).transpose(0, 2, 3, 1, 4).reshape(N, H, W, C))


def to_format(codes_nhwc: np.ndarray, fmt: int) -> np.ndarray:
    """NHWC codes -> the given code format's bytes (0 NHWC, 2 channel-blocked, 3 packed
    2-bit, 4 FP4 nibbles)."""
    N, H, W, C = codes_nhwc.shape
    if fmt == 4:
        blk = codes_nhwc.reshape(N, H, W, C // 32, 16, 2).transpose(0, 3, 1, 2, 4, 5).astype(np.uint8)
        return np.ascontiguousarray(blk[..., 0] | (blk[..., 1] << 4)).reshape(-1)
    blk = codes_nhwc.reshape(N, H, W, C // 16, 16).transpose(0, 3, 1, 2, 4)
    if fmt == 2:
        return np.ascontiguousarray(blk).reshape(-1)
    if fmt == 3:
        w = (blk.astype(np.uint32) << (2 * np.arange(16, dtype=np.uint32))).sum(axis=-1).astype(np.uint32)
        return np.ascontiguousarray(w).view(np.uint8).reshape(-1)
    return np.ascontiguousarray(codes_nhwc).reshape(-1)


def from_format(raw: np.ndarray, fmt: int, N: int, H: int, W: int, C: int) -> np.ndarray:
    if fmt == 2:
        return c16_to_nhwc(raw, N, H, W, C)
    if fmt == 3:
        return c16p2_to_nhwc(raw, N, H, W, C)
    if fmt == 4:
        return c32f4_to_nhwc(raw, N, H, W, C)
    return np.ascontiguousarray(raw).reshape(N, H, W, C)


def code_bytes(n_codes: int, fmt: int) -> int:
    """Bytes of n_codes codes in a code format."""
    return n_codes // {3: 4, 4: 2}.get(fmt, 1)


def run_gpu(c: Case, ref: dict, outputs=("acc", "y", "q"), fmt: int = 0):
    """Quantise and run the fused layer on the GPU through the C ABI.  fmt is the
    code format of the activation and output codes (0 NHWC, 2 channel-blocked);
    returned codes are always NHWC."""
    import torch

    from paper_2208_01944_gb300 import binding as B

    dev = torch.device("cuda:0")
    x = torch.from_numpy(ref["x"]).to(dev)
    nq = code_bytes(x.numel(), fmt)
    q = torch.empty(nq, dtype=torch.uint8, device=dev)
    B.palquant_quantize_act(x, q, c.N, c.H, c.W, c.G, c.Cin, c.bits, ref["inv_s"], code_format=fmt)
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin, c.Cout, c.k, c.stride, c.pad, c.bits, c.bits, c.bo, int(c.relu),
                     code_format=fmt)
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    B.palquant_pack_weights(ref["w"], d, ref["inv_sw"], wp, nbytes)
    shape = (c.N, c.Ho, c.Wo, c.G * c.Cout)
    acc = torch.full(shape, -7, dtype=torch.int32, device=dev) if "acc" in outputs else None
    y = torch.full(shape, float("nan"), dtype=torch.float32, device=dev) if "y" in outputs else None
    nqo = code_bytes(int(np.prod(shape)), fmt)
    qo = torch.full((nqo,), 255, dtype=torch.uint8, device=dev) if "q" in outputs else None
    sc = None if ref["shortcut"] is None else torch.from_numpy(ref["shortcut"]).to(dev)
    B.palquant_layer_fused(q, wp, d, ref["m_out"], ref["m_req"], B.shuffle(c.kind, c.shift, c.perm), sc, acc, y, qo)
    st = B.palquant_sync_check()
    assert st == B.PQ_OK, B.strerror(st)
    qh = from_format(q.cpu().numpy(), fmt, c.N, c.H, c.W, c.G * c.Cin)
    out = dict(q=qh)
    if acc is not None:
        out["acc"] = acc.cpu().numpy().reshape(-1, c.G * c.Cout)
    if y is not None:
        out["y"] = y.cpu().numpy().reshape(-1, c.G * c.Cout)
    if qo is not None:
        qoh = from_format(qo.cpu().numpy(), fmt, c.N, c.Ho, c.Wo, c.G * c.Cout)
        out["q_out"] = qoh.reshape(-1, c.G * c.Cout)
    return out


def assert_layer_parity(c: Case, ref: dict, got: dict, pix: np.ndarray | None = None):
    """Bit-exact codes and int32 sums; fp32 outputs within 1e-5 relative (and report exactness)."""
    assert np.array_equal(got["q"], ref["q"]), "activation codes differ"
    sel = (lambda a: a) if pix is None else (lambda a: a[pix])
    if "acc" in got:
        diff = np.argwhere(sel(got["acc"]) != ref["acc_ref"])
        assert diff.size == 0, f"int32 sums differ at {diff[:5].tolist()} ({len(diff)} elements)"
    if "q_out" in got:
        diff = np.argwhere(sel(got["q_out"]) != ref["q_ref"])
        assert diff.size == 0, f"requantised codes differ at {diff[:5].tolist()} ({len(diff)} elements)"
    if "y" in got:
        yg, yr = sel(got["y"]), ref["y_ref"]
        G, Co = c.G, c.Cout
        # tolerance scale per destination channel: max(|y_ref|, m_out of its source group)
        scale = np.maximum(np.abs(yr), float(np.min(ref["m_out"])))
        err = np.abs(yg.astype(np.float64) - yr.astype(np.float64))
        assert np.all(np.isfinite(yg)), "non-finite fp32 outputs"
        assert np.all(err <= 1e-5 * scale), f"fp32 outputs beyond 1e-5 relative: max {np.max(err / scale):.3g}"
