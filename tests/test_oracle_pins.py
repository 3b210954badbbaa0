"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test checks the oracle against something other than itself: hand-worked values of
Eq. 2, the two-line notation of Eq. 7, an independent float64 library convolution, a
brute-force dequantised convolution, closed forms and invariants.
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2208_01944_gb300 import synth, workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def torch_group_conv_f64(q, wq, stride, pad):
    """Independent check: torch's float64 grouped convolution on the integer codes."""
    G, Co, kh, kw, Ci = wq.shape
    x = torch.from_numpy(q.astype(np.float64)).permute(0, 3, 1, 2)
    w = torch.from_numpy(wq.astype(np.float64)).reshape(G * Co, kh, kw, Ci).permute(0, 3, 1, 2)
    y = F.conv2d(x, w, stride=stride, padding=pad, groups=G)
    return y.permute(0, 2, 3, 1).numpy()


# --------------------------------------------------------------------- Eq. 2
def test_quantizer_hand_cases():
    for bits, x, want in _rows("quantizer_cases.txt"):
        bits, x, want = int(bits), float(x), int(want)
        arr = np.full((1, 1, 1, 1), x, dtype=np.float32)
        got = oracle.quantize_act(arr, 1, bits, [1.0])[0, 0, 0, 0]
        assert got == want, (bits, x, got, want)


def test_quantizer_nan_inf():
    arr = np.array([np.nan, np.inf, -np.inf], dtype=np.float32).reshape(1, 1, 1, 3)
    got = oracle.quantize_act(arr, 1, 2, [1.0]).ravel()
    assert list(got) == [0, 3, 0]


def test_quantizer_range_and_monotone():
    gen = synth.generator(1)
    x = synth.normal((2, 5, 7, 12), gen, 3.0)
    for bits in (2, 3, 4):
        q = oracle.quantize_act(x, 3, bits, [0.7, 1.3, 2.1])
        assert q.min() >= 0 and q.max() <= (1 << bits) - 1
        # monotone within a group along sorted values
        for g, inv in enumerate([0.7, 1.3, 2.1]):
            xs = x[..., g * 4:(g + 1) * 4].ravel()
            qs = q[..., g * 4:(g + 1) * 4].ravel()
            order = np.argsort(xs, kind="stable")
            assert np.all(np.diff(qs[order].astype(int)) >= 0)


def test_quantizer_per_group_steps():
    # each group uses its own step: x = 1 everywhere, steps 1, 1/2, 1/3 -> codes 1, 2, 3
    x = np.ones((1, 2, 2, 6), dtype=np.float32)
    q = oracle.quantize_act(x, 3, 2, [1.0, 2.0, 3.0])
    assert (q[..., 0:2] == 1).all() and (q[..., 2:4] == 2).all() and (q[..., 4:6] == 3).all()


def test_weight_quantizer_hand_cases():
    w = np.array([0.0, 0.5, 0.6, -0.5, -1.5, -2.6, 1.49, 7.0, -9.0], dtype=np.float32).reshape(1, 1, 1, 1, 9)
    assert list(oracle.quantize_weights(w, 2, [1.0]).ravel()) == [0, 0, 1, 0, -2, -2, 1, 1, -2]
    assert list(oracle.quantize_weights(w, 4, [1.0]).ravel()) == [0, 0, 1, 0, -2, -3, 1, 7, -8]


# --------------------------------------------------------------- Sec. 4.1 conv
CONV_CASES = [
    # N, H, W, G, Ci, Co, k, stride, pad
    (1, 5, 7, 1, 3, 2, 3, 1, 1),
    (2, 6, 5, 2, 4, 3, 3, 1, 1),
    (1, 7, 7, 3, 2, 5, 3, 2, 1),
    (2, 8, 6, 4, 3, 2, 1, 1, 0),
    (1, 9, 8, 2, 5, 4, 1, 2, 0),
    (1, 6, 6, 2, 3, 3, 3, 1, 0),
    (1, 7, 5, 2, 2, 2, 5, 1, 2),
]


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("bits", [2, 4])
def test_group_conv_equals_float64_library_conv(case, bits):
    N, H, W, G, Ci, Co, k, s, p = case
    gen = synth.generator(hash(case) % 1000 + bits)
    q = synth.random_codes((N, H, W, G * Ci), bits, gen)
    wq = synth.random_codes((G, Co, k, k, Ci), bits, gen, signed=True)
    acc = oracle.group_conv(q, wq, s, p)
    ref = torch_group_conv_f64(q, wq, s, p)
    assert acc.shape == ref.shape
    assert np.array_equal(acc.astype(np.float64), ref)


def test_group_conv_pixels_match_full():
    gen = synth.generator(5)
    q = synth.random_codes((2, 9, 7, 3 * 4), 2, gen)
    wq = synth.random_codes((3, 5, 3, 3, 4), 2, gen, signed=True)
    full = oracle.group_conv(q, wq, 2, 1)
    pix = np.array([0, 3, 7, 11, 12, 19, 31, 39], dtype=np.int64)
    got = oracle.group_conv_pixels(q, wq, 2, 1, pix)
    assert np.array_equal(got, full.reshape(-1, full.shape[-1])[pix])


def test_dequantized_bruteforce_conv():
    """Brute-force float64 conv of the dequantised tensors equals s_w s_a acc (Sec. 3.2)."""
    N, H, W, G, Ci, Co, k, s, p = 1, 4, 5, 2, 2, 3, 3, 1, 1
    gen = synth.generator(9)
    x = synth.half_normal((N, H, W, G * Ci), gen)
    w = synth.he_weights(G, Co, k, k, Ci, gen)
    s_a = oracle.act_step(x, G, 2)
    s_w = oracle.weight_step(w, 2)
    q = oracle.quantize_act(x, G, 2, oracle.inv_step(s_a))
    wq = oracle.quantize_weights(w, 2, oracle.inv_step(s_w))
    acc = oracle.group_conv(q, wq, s, p)
    Ho, Wo = oracle.out_dim(H, k, s, p), oracle.out_dim(W, k, s, p)
    for n in range(N):
        for oh in range(Ho):
            for ow in range(Wo):
                for g in range(G):
                    for co in range(Co):
                        tot = 0.0
                        for kh in range(k):
                            for kw in range(k):
                                ih, iw = oh * s - p + kh, ow * s - p + kw
                                if 0 <= ih < H and 0 <= iw < W:
                                    for ci in range(Ci):
                                        xa = float(s_a[g]) * float(q[n, ih, iw, g * Ci + ci])
                                        wb = float(s_w[g]) * float(wq[g, co, kh, kw, ci])
                                        tot += xa * wb
                        want = float(s_w[g]) * float(s_a[g]) * float(acc[n, oh, ow, g * Co + co])
                        assert abs(tot - want) <= 1e-12 * max(1.0, abs(want))


def test_G1_is_ordinary_quantized_conv():
    gen = synth.generator(3)
    q = synth.random_codes((2, 6, 6, 8), 2, gen)
    wq = synth.random_codes((1, 5, 3, 3, 8), 2, gen, signed=True)
    acc = oracle.group_conv(q, wq, 1, 1)
    x = torch.from_numpy(q.astype(np.float64)).permute(0, 3, 1, 2)
    w = torch.from_numpy(wq[0].astype(np.float64)).permute(0, 3, 1, 2)
    ref = F.conv2d(x, w, padding=1).permute(0, 2, 3, 1).numpy()
    assert np.array_equal(acc.astype(np.float64), ref)


def test_1x1_is_matmul():
    gen = synth.generator(4)
    G, Ci, Co = 3, 6, 4
    q = synth.random_codes((2, 3, 5, G * Ci), 2, gen)
    wq = synth.random_codes((G, Co, 1, 1, Ci), 2, gen, signed=True)
    acc = oracle.group_conv(q, wq, 1, 0)
    X = q.reshape(-1, G, Ci).astype(np.float64)
    for g in range(G):
        ref = X[:, g, :] @ wq[g, :, 0, 0, :].astype(np.float64).T
        assert np.array_equal(acc.reshape(-1, G * Co)[:, g * Co:(g + 1) * Co].astype(np.float64), ref)


@pytest.mark.parametrize("bits", [2, 4])
def test_all_max_codes_closed_form(bits):
    """All activation codes at Qp, all weight codes at -2^(b-1): acc = taps_in_bounds * Cin * Qp * w."""
    N, H, W, G, Ci, Co, k, s, p = 1, 5, 6, 2, 7, 3, 3, 1, 1
    qp, wmin = (1 << bits) - 1, -(1 << (bits - 1))
    q = np.full((N, H, W, G * Ci), qp, dtype=np.uint8)
    wq = np.full((G, Co, k, k, Ci), wmin, dtype=np.int8)
    acc = oracle.group_conv(q, wq, s, p)
    for oh in range(H):
        for ow in range(W):
            rows = sum(1 for kh in range(k) if 0 <= oh - p + kh < H)
            cols = sum(1 for kw in range(k) if 0 <= ow - p + kw < W)
            assert (acc[0, oh, ow] == rows * cols * Ci * qp * wmin).all()


# --------------------------------------------------------- Sec. 4.2, Eq. 6-8
def _two_line_blocks():
    rows = _rows("cyclic_perm_two_line.txt")
    out = {}
    i = 0
    while i < len(rows):
        G = int(rows[i][0].split("=")[1])
        out[G] = ([int(v) for v in rows[i + 1]], [int(v) for v in rows[i + 2]])
        i += 3
    return out


def test_cyclic_perm_two_line_notation():
    for G, (top, bottom) in _two_line_blocks().items():
        assert top == list(range(G))
        assert list(oracle.group_perm(G, 1, 1)) == bottom


@pytest.mark.parametrize("G", [1, 2, 3, 4, 5, 8])
def test_cyclic_perm_is_G_cycle(G):
    pi = oracle.group_perm(G, 1, 1)
    assert sorted(pi) == list(range(G))  # bijection
    # Prop. 1: pi is a G-cycle, so pi^G = id and no smaller power is the identity (G > 1)
    cur = np.arange(G)
    for step in range(1, G + 1):
        cur = pi[cur]
        if step < G and G > 1:
            assert not np.array_equal(cur, np.arange(G))
    assert np.array_equal(cur, np.arange(G))
    # the orbit of group 0 visits every group
    orbit, g = set(), 0
    for _ in range(G):
        orbit.add(int(g))
        g = pi[g]
    assert orbit == set(range(G))


def test_bad_permutation_rejected():
    with pytest.raises(ValueError):
        oracle.group_perm(3, 3, 0, [0, 0, 1])
    with pytest.raises(ValueError):
        oracle.group_perm(3, 3, 0, [0, 1, 3])


@pytest.mark.parametrize("G", [2, 3, 4])
def test_epilogue_remap_is_roll_on_group_axis(G):
    """Eq. 8, Y[:, pi(i)] = X[:, i] with pi(i) = i + 1 mod G, equals torch.roll(+1) over groups."""
    gen = synth.generator(G)
    Co = 3
    acc = torch.randint(-50, 50, (2, 3, 4, G * Co), generator=gen).numpy().astype(np.int64)
    m_out = np.linspace(0.1, 0.3, G).astype(np.float32)
    m_req = np.linspace(0.05, 0.2, G).astype(np.float32)
    a0, y0, q0 = oracle.epilogue(acc, G, m_out, m_req, kind=0)
    a1, y1, q1 = oracle.epilogue(acc, G, m_out, m_req, kind=1, shift=1)
    for ref, got in ((a0, a1), (y0, y1), (q0, q1)):
        t = torch.from_numpy(ref).reshape(2, 3, 4, G, Co)
        rolled = torch.roll(t, shifts=1, dims=3).reshape(ref.shape).numpy()
        assert np.array_equal(rolled, got)
    # the inverse permutation (shift -1) restores the source order
    inv = oracle.group_perm(G, 1, -1)
    fwd = oracle.group_perm(G, 1, 1)
    assert np.array_equal(inv[fwd], np.arange(G))
    restored = a1.reshape(2, 3, 4, G, Co)[..., fwd, :].reshape(acc.shape)
    assert np.array_equal(restored, a0)


def test_epilogue_hand_cases():
    # G = 2, Cout_g = 2, one pixel; channel order (g0c0, g0c1, g1c0, g1c1)
    acc = np.array([[10, -4, 7, 100]], dtype=np.int64)
    m_out = [0.25, 0.5]
    m_req = [0.125, 0.0625]
    a, y, q = oracle.epilogue(acc, 2, m_out, m_req, kind=1, shift=1, relu=True, bits_out=2)
    # group 0 -> destination group 1 (channels 2, 3); group 1 -> destination group 0
    assert list(a[0]) == [7, 100, 10, -4]
    assert list(y[0]) == [3.5, 50.0, 2.5, 0.0]
    # codes: 7/16 = 0.4375 -> 0; 100/16 = 6.25 -> 6 -> clamp 3; 10/8 = 1.25 -> 1; -4/8 -> 0
    assert list(q[0]) == [0, 3, 1, 0]
    a, y, q = oracle.epilogue(acc, 2, m_out, m_req, kind=0, relu=False, bits_out=4)
    assert list(y[0]) == [2.5, -1.0, 3.5, 50.0]
    # rint half-to-even: 10/8 = 1.25 -> 1; 100/16 = 6.25 -> 6
    assert list(q[0]) == [1, 0, 0, 6]


def test_epilogue_shortcut_requant_from_sum():
    acc = np.array([[4, -8]], dtype=np.int64)  # G = 1, Cout_g = 2
    sc = np.array([[0.5, 1.0]], dtype=np.float32)
    a, y, q = oracle.epilogue(acc, 1, [0.25], [2.0], kind=0, shortcut=sc, relu=True, bits_out=2)
    # y = acc*0.25 + sc = [1.5, -1.0] -> relu [1.5, 0]; q = rint(y*2) = [3, 0]
    assert list(y[0]) == [1.5, 0.0]
    assert list(q[0]) == [3, 0]


def test_epilogue_rejects_large_acc():
    with pytest.raises(ValueError):
        oracle.epilogue(np.array([[1 << 24]], dtype=np.int64), 1, [1.0], [1.0], kind=0)


def test_epilogue_scales_hand_case():
    m_out, m_req = oracle.epilogue_scales([0.5, 2.0], [0.25, 4.0], s_next=[1.0, 0.5], kind=1, shift=1)
    # dst(0) = 1, dst(1) = 0
    assert list(m_out) == [0.125, 8.0]
    assert list(m_req) == [0.25, 8.0]


# ------------------------------------------------- LSQ step initialisation
def test_act_step_half_normal_closed_form():
    """E|N(0,1)| = sqrt(2/pi), so the step is 2 sqrt(2/pi) / sqrt(Qp) (statistical)."""
    gen = synth.generator(11)
    x = synth.half_normal((4, 64, 64, 2 * 16), gen)
    s = oracle.act_step(x, 2, 2)
    want = 2.0 * math.sqrt(2.0 / math.pi) / math.sqrt(3.0)
    assert np.allclose(s, want, rtol=5e-3)
    # exact on a constant tensor: mean = c
    c = np.full((1, 2, 2, 4), 1.5, dtype=np.float32)
    assert np.allclose(oracle.act_step(c, 2, 2), 2 * 1.5 / math.sqrt(3.0), rtol=1e-7)


def test_weight_step_gaussian_closed_form():
    gen = synth.generator(12)
    fan_in = 64 * 9
    w = synth.he_weights(4, 64, 3, 3, 64, gen)
    s = oracle.weight_step(w, 2)
    want = 2.0 * math.sqrt(2.0 / fan_in) * math.sqrt(2.0 / math.pi) / 1.0  # Qp_w = 1 at b = 2
    assert np.allclose(s, want, rtol=1e-2)
    s4 = oracle.weight_step(w, 4)
    assert np.allclose(s4, want / math.sqrt(7.0), rtol=1e-2)


def test_inv_step_rounding():
    assert oracle.inv_step([0.5, 4.0])[0] == 2.0
    v = oracle.inv_step([3.0])[0]
    assert v == np.float32(1.0 / 3.0)


# ------------------------------------------------------- Appendix B BitOps
def test_bitops_table1():
    for net, method, bw, ba, G, want in _rows("table1_bitops.txt"):
        bw, ba, G, want = int(bw), int(ba), int(G), float(want) * 1e9
        blocks = (2, 2, 2, 2) if net == "resnet18" else (3, 4, 6, 3)
        if method == "lsq":
            got = workloads.bitops(workloads.resnet_convs(blocks), bw, ba)
            assert abs(got - want) / want < 3e-3, (net, bw, got, want)
        else:
            # PalQuant: channels expanded G times, G-group convolutions, plus the 1x1
            # group convolution of a cyclic shuffle module at the start of stages 2-4.
            got = workloads.bitops(workloads.resnet_convs(blocks, G, G, shuffle_module_stages=(1, 2, 3)), bw, ba)
            assert abs(got - want) / want < 6e-3, (net, G, got, want)


def test_layer_op_counts():
    c1 = workloads.CONFIG1
    assert c1.int_ops == 2 * 64 * 56 * 56 * 4 * 64 * 9 * 64
    assert abs(c1.int_ops - 59.19e9) / 59.19e9 < 1e-3
    assert abs(workloads.CONFIG4.int_ops - 3.70e9) / 3.70e9 < 2e-3


@pytest.mark.parametrize("G,Co", [(2, 3), (4, 2), (3, 5)])
def test_epilogue_channel_shuffle_is_shufflenet_transpose(G, Co):
    """The channel shuffle (ShuffleNet's reshape to [G, C/G], transpose, flatten) that the
    paper pairs with the cyclic shuffle (Sec. 4.3), written with torch's reshape/transpose."""
    gen = synth.generator(G * 7 + Co)
    acc = torch.randint(-50, 50, (2, 3, G * Co), generator=gen).numpy().astype(np.int64)
    a0, y0, _ = oracle.epilogue(acc, G, np.full(G, 0.5, np.float32), kind=0)
    a2, y2, _ = oracle.epilogue(acc, G, np.full(G, 0.5, np.float32), kind=2)
    for ref, got in ((a0, a2), (y0, y2)):
        t = torch.from_numpy(ref).reshape(2, 3, G, Co).transpose(2, 3).reshape(ref.shape).numpy()
        assert np.array_equal(t, got)


# ------------------------------------------------ the paper's odd weight levels
def test_odd_weight_levels_hand_cases():
    # b = 2, u = 1: k = 3 / 2; t = (w + 1) * 1.5
    w = np.array([-2.0, -1.0, -0.5, -1.0 / 3.0, 0.0, 0.2, 1.0 / 3.0, 0.5, 1.0, 5.0], dtype=np.float32)
    got = oracle.quantize_weights_odd(w.reshape(1, 1, 1, 1, -1), 2, [1.0]).ravel()
    # t: -1.5 0 0.75 1.0 1.5 1.8 2.0 2.25 3 9 -> x_q 0 0 1 1 2 2 2 2 3 3 -> 2 x_q - 3
    assert list(got) == [-3, -3, -1, -1, 1, 1, 1, 1, 3, 3]


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_odd_weight_levels_range_and_monotone(bits):
    gen = synth.generator(bits + 100)
    w = synth.normal((2, 4, 3, 3, 16), gen, 0.3)
    u = np.array([0.4, 0.7], np.float32)
    wq = oracle.quantize_weights_odd(w, bits, u)
    qp = (1 << bits) - 1
    assert np.all(np.abs(wq) <= qp) and np.all(wq % 2 != 0)  # odd levels in [-Qp, Qp]
    for g in range(2):
        order = np.argsort(w[g].ravel(), kind="stable")
        assert np.all(np.diff(wq[g].ravel()[order].astype(int)) >= 0)
        # outside the clip range the extreme levels
        assert np.all(wq[g][w[g] >= u[g]] == qp) and np.all(wq[g][w[g] <= -u[g]] == -qp)
