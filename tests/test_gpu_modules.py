"""The cyclic shuffle module (Sec. 4.2, Eq. 9-10) on the GPU against the oracle:
Z = X + Conv1x1(CyclicPermute(X)) with the 1x1 PalQuant group convolution, fp32 Z and
Z's codes bit for bit, in both code layouts."""
import numpy as np
import pytest
import torch

import oracle
from layer_cases import c16_to_nhwc
from paper_2208_01944_gb300 import synth

pytestmark = pytest.mark.gpu

CASES = [  # N, H, W, G, Cg, shift, relu
    (2, 7, 9, 2, 32, 1, False),
    (1, 14, 14, 4, 64, 1, False),
    (3, 5, 11, 3, 96, 1, True),
    (2, 16, 16, 4, 32, -1, False),
    (64, 14, 14, 2, 128, 1, False),
]


@pytest.mark.parametrize("fmt", [0, 2], ids=["nhwc", "c16"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: "N%dx%dx%d_G%dx%d_sh%d%s" % (c[:6] + ("_relu" if c[6] else "",)))
def test_cyclic_shuffle_module_matches_oracle(case, fmt):
    from paper_2208_01944_gb300 import binding as B

    N, H, W, G, Cg, shift, relu = case
    gen = synth.generator(sum(case[:5]))
    x = synth.normal((N, H, W, G * Cg), gen)
    w = synth.he_weights(G, Cg, 1, 1, Cg, gen)
    s_a = oracle.act_step(np.abs(x), G, 2)
    inv_s = oracle.inv_step(s_a)
    s_w = oracle.weight_step(w, 2)
    inv_sw = oracle.inv_step(s_w)
    q = oracle.quantize_act(x, G, 2, inv_s)
    wq = oracle.quantize_weights(w, 2, inv_sw)
    # the conv of group g reads input group pi^-1(g): its multiplier uses that group's step
    src = [(g - shift) % G for g in range(G)]
    m_out = np.array([np.float32(np.float64(s_w[g]) * np.float64(s_a[src[g]])) for g in range(G)], np.float32)
    inv_next = (np.arange(G, dtype=np.float32) * np.float32(0.25) + np.float32(0.9))
    z_ref, q_ref = oracle.cyclic_shuffle_module(x, q, wq, m_out, inv_next, shift, relu, 2)
    d = B.layer_desc(N, H, W, G, Cg, Cg, 1, 1, 0, 2, 2, 2, int(relu), code_format=fmt)
    qd = torch.empty((N, H, W, G * Cg), dtype=torch.uint8, device="cuda")
    xd = torch.from_numpy(x).cuda()
    B.palquant_quantize_act(xd, qd, N, H, W, G, Cg, 2, inv_s, code_format=fmt)
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    B.palquant_pack_weights(w, d, inv_sw, wp, nbytes)
    z = torch.full((N, H, W, G * Cg), float("nan"), device="cuda")
    qo = torch.full((N, H, W, G * Cg), 255, dtype=torch.uint8, device="cuda")
    B.palquant_cyclic_shuffle_module(qd, wp, d, m_out, inv_next, shift, xd, z, qo)
    assert B.palquant_sync_check() == B.PQ_OK
    assert np.array_equal(z.cpu().numpy(), z_ref)
    got = qo.cpu().numpy()
    if fmt == 2:
        got = c16_to_nhwc(got, N, H, W, G * Cg)
    assert np.array_equal(got, q_ref)


def test_module_rejects_non_1x1():
    from paper_2208_01944_gb300 import binding as B

    for d in [B.layer_desc(1, 8, 8, 2, 32, 32, 3, 1, 1), B.layer_desc(1, 8, 8, 2, 32, 64, 1, 1, 0),
              B.layer_desc(1, 8, 8, 2, 32, 32, 1, 2, 0)]:
        with pytest.raises(B.PalquantError) as e:
            B.palquant_cyclic_shuffle_module(16, 16, d, [1.0, 1.0], [1.0, 1.0], 1, 16, 16, None)
        assert e.value.status == B.PQ_EINVAL


@pytest.mark.parametrize("G", [2, 3, 4])
def test_prop1_chained_modules_reach_every_group(G):
    """Prop. 1 on the device: G - 1 cyclic shuffle modules chained through the library
    (each module's fp32 output quantised by the library for the next) spread one
    non-zero input group to every group; every intermediate tensor bit for bit
    against the oracle's chain."""
    from paper_2208_01944_gb300 import binding as B

    Cg, N, H, W = 32, 1, 4, 6
    wq = np.ones((G, Cg, 1, 1, Cg), dtype=np.int8)
    m_out = np.full(G, 0.1, np.float32)
    inv = np.ones(G, np.float32)
    d = B.layer_desc(N, H, W, G, Cg, Cg, 1, 1, 0, 2, 2, 2, 0, code_format=2)
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).cuda()
    for s in range(G):
        x = np.zeros((N, H, W, G * Cg), dtype=np.float32)
        x[..., s * Cg:(s + 1) * Cg] = 2.0
        xd = torch.from_numpy(x).cuda()
        for k in range(1, G):
            q_ref = oracle.quantize_act(x, G, 2, inv)
            x, _ = oracle.cyclic_shuffle_module(x, q_ref, wq, m_out, None, 1)
            qd = torch.empty((N, H, W, G * Cg), dtype=torch.uint8, device="cuda")
            B.palquant_quantize_act(xd, qd, N, H, W, G, Cg, 2, inv, code_format=2)
            zd = torch.empty_like(xd)
            B.palquant_cyclic_shuffle_module(qd, wp, d, m_out, None, 1, xd, zd, None)
            assert B.palquant_sync_check() == B.PQ_OK
            assert np.array_equal(zd.cpu().numpy(), x), (G, s, k)
            live = {g for g in range(G) if np.any(x[..., g * Cg:(g + 1) * Cg] != 0)}
            assert live == {(s + j) % G for j in range(k + 1)}, (G, s, k, live)
            xd = zd
