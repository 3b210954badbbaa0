"""Bit-level decomposition (Sec. 3.3, Eq. 4) on the GPU: the M-bit layer computed as the
G^2 shifted B-bit slice products in one tensor-core pass (each activation slice stored
and read once, meeting the Gw weight slices as extra taps) equals the oracle's M-bit
convolution (and its own decomposition) exactly."""
import numpy as np
import pytest
import torch

import oracle
from paper_2208_01944_gb300 import synth

pytestmark = pytest.mark.gpu


def _to_fmt(q, fmt):
    if fmt == 2:
        N, H, W, C = q.shape
        return np.ascontiguousarray(q.reshape(N, H, W, C // 16, 16).transpose(0, 3, 1, 2, 4))
    return q


@pytest.mark.parametrize("fmt", [0, 2], ids=["nhwc", "c16"])
@pytest.mark.parametrize("M,Bb,shape", [
    (4, 2, (2, 9, 11, 64, 32, 3, 1, 1)),
    (4, 2, (1, 14, 14, 128, 64, 1, 1, 0)),
    (4, 2, (2, 10, 10, 32, 48, 3, 2, 1)),
    (3, 2, (1, 7, 9, 96, 16, 3, 1, 1)),
    (4, 1, (1, 6, 6, 32, 32, 3, 1, 1)),
    (6, 3, (1, 8, 8, 64, 32, 3, 1, 1)),
], ids=lambda v: str(v))
def test_bitsplit_conv_matches_oracle(M, Bb, shape, fmt):
    from paper_2208_01944_gb300 import binding as B

    N, H, W, C, Co, k, s, p = shape
    gen = synth.generator(M * 100 + sum(shape))
    q = synth.random_codes((N, H, W, C), M, gen)
    wq = synth.random_codes((1, Co, k, k, C), M, gen, signed=True)
    ref = oracle.group_conv(q, wq, s, p)
    assert np.array_equal(ref, oracle.bitsplit_conv(q, wq, s, p, M, Bb))
    d = B.layer_desc(N, H, W, 1, C, Co, k, s, p, M, M, 2, 0, code_format=fmt)
    t = B.palquant_bitsplit_desc(d, Bb)
    wp = torch.from_numpy(B.palquant_bitsplit_pack_weight_codes_host(wq, d, Bb)).cuda()
    qd = torch.from_numpy(_to_fmt(q, fmt)).cuda()
    nbytes = B.palquant_bitsplit_scratch_bytes(d, Bb)
    assert nbytes == N * H * W * t.Cin_g
    xs = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    acc = torch.full(ref.shape, -7, dtype=torch.int32, device="cuda")
    B.palquant_bitsplit_conv(qd, xs, nbytes, wp, acc, d, Bb)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), ref)
    # the slices in the scratch buffer are the oracle's, each stored once
    Ga = -(-M // Bb)
    assert t.Cin_g == Ga * C and t.wslices == Ga
    got = xs.cpu().numpy()
    slices = oracle.bit_slices_act(q, M, Bb)
    want = np.concatenate([slices[i] for i in range(Ga)], axis=-1)
    assert np.array_equal(got.reshape(want.shape) if fmt == 0 else got, _to_fmt(want, fmt).ravel() if fmt == 2 else want)
