"""Pins of the oracle's bit-level decomposition (Sec. 3.3, Eq. 4) -- no GPU.

Eq. 4 is an exact identity: the M-bit convolution equals the sum over the G^2 pairs of
B-bit slice convolutions shifted by 2^((i+j)B).  The slices are checked against their
definition (reconstruction and ranges) and the decomposed convolution against torch's
float64 convolution of the M-bit codes.
"""
import numpy as np
import pytest

import oracle
from paper_2208_01944_gb300 import synth

from test_oracle_pins import torch_group_conv_f64


@pytest.mark.parametrize("M,B", [(4, 2), (6, 2), (8, 2), (4, 1), (5, 2), (8, 4)])
def test_slices_reconstruct_and_stay_in_range(M, B):
    gen = synth.generator(M * 10 + B)
    q = synth.random_codes((3, 4, 5, 8), M, gen)
    wq = synth.random_codes((2, 3, 3, 3, 4), M, gen, signed=True)
    G = -(-M // B)
    xs = oracle.bit_slices_act(q, M, B)
    ws = oracle.bit_slices_weights(wq, M, B)
    assert len(xs) == len(ws) == G
    assert np.array_equal(sum(x.astype(np.int64) << (i * B) for i, x in enumerate(xs)), q.astype(np.int64))
    assert np.array_equal(sum(w.astype(np.int64) << (j * B) for j, w in enumerate(ws)), wq.astype(np.int64))
    for x in xs:
        assert x.min() >= 0 and x.max() <= (1 << B) - 1
    for w in ws[:-1]:
        assert w.min() >= 0 and w.max() <= (1 << B) - 1
    top = M - (G - 1) * B  # bits of the signed top slice
    assert ws[-1].min() >= -(1 << (top - 1)) and ws[-1].max() <= (1 << (top - 1)) - 1


def test_hand_case_eq4():
    # x = 13 = 0b1101 -> slices (1, 3); w = -6 = ...1010 -> slices (2, -2) at B = 2
    q = np.array([13], dtype=np.uint8).reshape(1, 1, 1, 1)
    w = np.array([-6], dtype=np.int8).reshape(1, 1, 1, 1, 1)
    assert [int(v.ravel()[0]) for v in oracle.bit_slices_act(q, 4, 2)] == [1, 3]
    assert [int(v.ravel()[0]) for v in oracle.bit_slices_weights(w, 4, 2)] == [2, -2]
    assert int(oracle.bitsplit_conv(q, w, 1, 0, 4, 2).ravel()[0]) == -78


@pytest.mark.parametrize("M,B,G,k,s,p", [(4, 2, 1, 3, 1, 1), (4, 2, 2, 3, 2, 1), (8, 2, 1, 1, 1, 0), (6, 2, 3, 3, 1, 0)])
def test_eq4_equals_the_M_bit_convolution(M, B, G, k, s, p):
    gen = synth.generator(M + 7 * G + k)
    q = synth.random_codes((2, 7, 6, G * 8), M, gen)
    wq = synth.random_codes((G, 5, k, k, 8), M, gen, signed=True)
    got = oracle.bitsplit_conv(q, wq, s, p, M, B)
    assert np.array_equal(got, oracle.group_conv(q, wq, s, p))
    assert np.array_equal(got.astype(np.float64), torch_group_conv_f64(q, wq, s, p))
