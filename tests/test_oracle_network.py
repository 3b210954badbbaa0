"""Pins of the oracle's full-precision layers and of its ResNet-18-shaped network (no GPU).

The full-precision layers (the paper keeps the first and last layer in full precision,
Sec. 5) are checked against torch's float64 routines within the fp32 rounding bound of
their fixed summation order, exactly where every partial sum is representable, and max
pooling exactly.  The network's wiring (which tensor feeds which layer, strides, the
shortcut source, the direction of the permutation, which steps requantise what) is
re-derived block by block from the oracle's own codes with torch's float64 grouped
convolution.  Planted mistakes in the C source must fail these pins.
"""
import os
import subprocess

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
import oracle.resnet as R
from paper_2208_01944_gb300 import synth

EPS = np.finfo(np.float32).eps


def _nchw(x):
    return torch.from_numpy(np.asarray(x, dtype=np.float64)).permute(0, 3, 1, 2)


def _nhwc(t):
    return t.permute(0, 2, 3, 1).numpy()


def conv_ref(x, w, stride, pad):
    """float64 convolution and the sum of |terms| per output (rounding bound)."""
    wt = torch.from_numpy(np.asarray(w, dtype=np.float64)).permute(0, 3, 1, 2)
    y = F.conv2d(_nchw(x), wt, stride=stride, padding=pad)
    mag = F.conv2d(_nchw(np.abs(x)), wt.abs(), stride=stride, padding=pad)
    return _nhwc(y), _nhwc(mag)


# ------------------------------------------------------------ full-precision layers
@pytest.mark.parametrize("shape,k,s,p", [((2, 17, 15, 3), 7, 2, 3), ((1, 9, 9, 5), 3, 1, 1), ((1, 8, 6, 4), 3, 2, 0)])
def test_conv2d_f32_within_rounding_bound(shape, k, s, p, L=None):
    gen = synth.generator(3)
    x = synth.normal(shape, gen)
    w = synth.normal((16, k, k, shape[3]), gen, 0.3)
    y = oracle.conv2d_f32(x, w, s, p, L=L)
    ref, mag = conv_ref(x, w, s, p)
    n = k * k * shape[3]
    assert y.shape == ref.shape
    assert np.all(np.abs(y - ref) <= n * EPS * mag + 1e-30)


def test_conv2d_f32_exact_on_small_integers(L=None):
    gen = synth.generator(4)
    x = synth.random_codes((1, 9, 11, 3), 4, gen).astype(np.float32) - 7.0
    w = synth.random_codes((16, 7, 7, 3), 3, gen, signed=True).astype(np.float32)
    y = oracle.conv2d_f32(x, w, 2, 3, L=L)
    ref, _ = conv_ref(x, w, 2, 3)
    assert np.array_equal(y.astype(np.float64), ref)
    yr = oracle.conv2d_f32(x, w, 2, 3, relu=True, L=L)
    assert np.array_equal(yr.astype(np.float64), np.maximum(ref, 0.0))


def test_maxpool_exact(L=None):
    gen = synth.generator(5)
    x = synth.normal((2, 11, 9, 6), gen)
    y = oracle.maxpool_f32(x, 3, 2, 1, L=L)
    ref = _nhwc(F.max_pool2d(_nchw(x), 3, 2, 1))
    assert np.array_equal(y.astype(np.float64), ref)
    # all-negative input: the padding is not a zero tap
    y = oracle.maxpool_f32(-np.abs(x) - 1.0, 3, 2, 1, L=L)
    assert np.all(y < 0)


def test_avgpool(L=None):
    gen = synth.generator(6)
    x = synth.normal((3, 7, 7, 5), gen)
    y = oracle.avgpool_f32(x, L=L)
    ref = np.asarray(x, dtype=np.float64).mean(axis=(1, 2))
    bound = 49 * EPS * np.abs(x).astype(np.float64).sum(axis=(1, 2)) / 49 + EPS * np.abs(ref)
    assert np.all(np.abs(y - ref) <= bound)
    xi = np.arange(2 * 2 * 2 * 3, dtype=np.float32).reshape(2, 2, 2, 3)
    assert np.array_equal(oracle.avgpool_f32(xi, L=L), xi.astype(np.float64).mean(axis=(1, 2)).astype(np.float32))


def test_linear(L=None):
    gen = synth.generator(7)
    x = synth.normal((3, 50), gen)
    w = synth.normal((7, 50), gen)
    y = oracle.linear_f32(x, w, L=L)
    ref = x.astype(np.float64) @ w.astype(np.float64).T
    mag = np.abs(x).astype(np.float64) @ np.abs(w).astype(np.float64).T
    assert np.all(np.abs(y - ref) <= 50 * EPS * mag)
    xi = np.arange(6, dtype=np.float32).reshape(2, 3)
    wi = np.array([[1, 0, 0], [0, 2, -1]], dtype=np.float32)
    assert np.array_equal(oracle.linear_f32(xi, wi, L=L), np.array([[0, 0], [3, 3]], dtype=np.float32))


# ------------------------------------------------------------ network wiring
G, BITS, WIDTHS = 2, 2, (32, 32, 32, 32)


@pytest.fixture(scope="module")
def net():
    x, params = synth.resnet18_inputs(2, 32, 32, G, WIDTHS, 10, seed=1)
    steps = R.calibrate(x, params, G, BITS)
    return x, params, steps, R.forward(x, params, G, BITS, steps)


def torch_group_conv_f64(q, wq, stride, pad):
    Gg, Co, kh, kw, Ci = wq.shape
    xt = _nchw(q)
    w = torch.from_numpy(wq.astype(np.float64)).reshape(Gg * Co, kh, kw, Ci).permute(0, 3, 1, 2)
    return _nhwc(F.conv2d(xt, w, stride=stride, padding=pad, groups=Gg))


def test_network_shapes_and_code_ranges(net):
    x, params, steps, r = net
    assert r["stem"].shape == (2, 16, 16, 64) and r["pool"].shape == (2, 8, 8, 64)
    assert r["s4b2.out"].shape == (2, 1, 1, 64) and r["logits"].shape == (2, 10)
    for k, v in r.items():
        if k.endswith("codes"):
            assert v.dtype == np.uint8 and v.max() <= 3
    # every step positive and finite
    for k, v in steps.items():
        assert np.all(np.isfinite(v)) and np.all(v > 0), k


def test_network_blocks_rederived_with_float64_library(net):
    """Each block recomputed from the oracle's own block input: torch float64 grouped
    convolution of the integer codes (exact), one fp32 multiply by the multiplier, the
    shortcut add, ReLU and Eq. 8's roll on the group axis."""
    x, params, steps, r = net
    stem = conv_ref(x, params["stem"], 2, 3)[0]
    assert np.allclose(r["stem"], np.maximum(stem, 0), rtol=1e-5, atol=1e-5)
    X = r["pool"]
    blocks = [("s1b1", 1, False), ("s1b2", 1, False), ("s2b1", 2, True), ("s2b2", 1, False),
              ("s3b1", 2, True), ("s3b2", 1, False), ("s4b1", 2, True), ("s4b2", 1, False)]
    for i, (b, stride, down) in enumerate(blocks):
        Q = r[b + ".in_codes"]
        assert np.array_equal(Q, oracle.quantize_act(X, G, BITS, oracle.inv_step(steps[b + ".in"])))
        f32 = lambda a, m: (a.astype(np.float32).reshape(*a.shape[:-1], G, -1) *
                            np.asarray(m, np.float32)[:, None]).reshape(a.shape)
        sw1, sin, smid = steps[b + ".conv1.w"], steps[b + ".in"], steps[b + ".mid"]
        wq1 = oracle.quantize_weights(params[b + ".conv1"], BITS, oracle.inv_step(sw1))
        acc1 = torch_group_conv_f64(Q, wq1, stride, 1)
        m_req1 = (np.float64(sw1) * np.float64(sin) / np.float64(smid)).astype(np.float32)
        t1 = f32(acc1, m_req1)
        q1 = np.clip(np.rint(t1), 0, 3).astype(np.uint8)
        assert np.array_equal(q1, r[b + ".mid_codes"]), b
        if down:
            swd = steps[b + ".down.w"]
            wqd = oracle.quantize_weights(params[b + ".down"], BITS, oracle.inv_step(swd))
            accd = torch_group_conv_f64(Q, wqd, stride, 0)
            S = f32(accd, (np.float64(swd) * np.float64(sin)).astype(np.float32))
            assert np.array_equal(S, r[b + ".down"]), b
        else:
            S = X
        sw2 = steps[b + ".conv2.w"]
        wq2 = oracle.quantize_weights(params[b + ".conv2"], BITS, oracle.inv_step(sw2))
        acc2 = torch_group_conv_f64(q1, wq2, 1, 1)
        y = np.maximum(f32(acc2, (np.float64(sw2) * np.float64(smid)).astype(np.float32)) + S, np.float32(0))
        rolled = np.roll(y.reshape(*y.shape[:-1], G, -1), 1, axis=-2).reshape(y.shape)
        assert np.array_equal(rolled, r[b + ".out"]), b
        if i + 1 < len(blocks):
            nxt = blocks[i + 1][0]
            want = oracle.quantize_act(r[b + ".out"], G, BITS, oracle.inv_step(steps[nxt + ".in"]))
            assert np.array_equal(want, r[b + ".out_codes"]), b
        X = r[b + ".out"]
    ref = X.astype(np.float64).mean(axis=(1, 2)) @ params["fc"].astype(np.float64).T
    assert np.allclose(r["logits"], ref, rtol=1e-4, atol=1e-4)


def test_calibrated_steps_follow_lsq_init(net):
    x, params, steps, r = net
    assert np.array_equal(steps["s1b1.in"], oracle.act_step(r["pool"], G, BITS))
    assert np.array_equal(steps["s2b1.in"], oracle.act_step(r["s1b2.out"], G, BITS))
    assert np.array_equal(steps["s3b1.conv1.w"], oracle.weight_step(params["s3b1.conv1"], BITS))


# ------------------------------------------------------------ planted mistakes
SRC = os.path.join(os.path.dirname(oracle.__file__), "palquant_oracle.c")
MUTATIONS = {
    "conv_kernel_flipped": ("const float* wp = w + (((int64_t)co * k + kh) * k + kw) * Cin;",
                            "const float* wp = w + (((int64_t)co * k + kw) * k + kh) * Cin;"),
    "conv_pad_ignored": ("const int64_t ih = oh * s - p + kh;\n                        if (ih < 0 || ih >= H) continue;\n                        for (int kw",
                         "const int64_t ih = oh * s + kh;\n                        if (ih < 0 || ih >= H) continue;\n                        for (int kw"),
    "conv_relu_dropped": ("if (relu) acc = fmaxf(acc, 0.0f);\n                    y[", "y["),
    "maxpool_zero_start": ("float m = -INFINITY;", "float m = 0.0f;"),
    "avgpool_wrong_count": ("y[n * C + c] = acc / (float)(H * W);", "y[n * C + c] = acc / (float)(H);"),
    "linear_transposed": ("acc = fmaf(x[n * Cin + i], w[(int64_t)o * Cin + i], acc);",
                          "acc = fmaf(x[n * Cin + i], w[(int64_t)i * Cout + o], acc);"),
}


def _fp32_pins_pass(L) -> bool:
    try:
        test_conv2d_f32_within_rounding_bound((1, 9, 9, 5), 3, 1, 1, L=L)
        test_conv2d_f32_within_rounding_bound((2, 17, 15, 3), 7, 2, 3, L=L)
        test_conv2d_f32_exact_on_small_integers(L=L)
        test_maxpool_exact(L=L)
        test_avgpool(L=L)
        test_linear(L=L)
        return True
    except AssertionError:
        return False


def test_unmutated_fp32_oracle_passes():
    assert _fp32_pins_pass(oracle.lib())


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_fp32_mutation_is_caught(name, tmp_path):
    old, new = MUTATIONS[name]
    src = open(SRC).read()
    assert old in src, name
    path = tmp_path / "mut.c"
    path.write_text(src.replace(old, new, 1))
    so = oracle.build(force=True, src=str(path), out=str(tmp_path / "libmut.so"))
    assert not _fp32_pins_pass(oracle.load_variant(so)), f"mutation {name} not caught"


# ------------------------------------------------------------ cyclic shuffle module (Eq. 9-10)
def test_permute_groups_is_eq8():
    x = np.arange(2 * 3 * 12, dtype=np.float32).reshape(2, 3, 12)
    y = oracle.permute_groups(x, 4, 1)
    # Y[:, pi(i)] = X[:, i] with pi(i) = (i + 1) mod 4: group 0 lands in group 1, group 3 in group 0
    assert np.array_equal(y[..., 3:6], x[..., 0:3]) and np.array_equal(y[..., 0:3], x[..., 9:12])
    assert np.array_equal(y, np.roll(x.reshape(2, 3, 4, 3), 1, axis=2).reshape(x.shape))
    assert np.array_equal(oracle.permute_groups(y, 4, -1), x)


@pytest.mark.parametrize("G,Cg", [(2, 32), (4, 16), (3, 32)])
def test_cyclic_shuffle_module_rederived(G, Cg):
    """Z = X + Conv1x1(CyclicPermute(X)) recomputed with numpy's roll and torch's
    float64 grouped convolution of the integer codes (exact), one fp32 multiply and
    one fp32 add."""
    gen = synth.generator(G * Cg)
    x = synth.half_normal((2, 5, 6, G * Cg), gen)
    q = oracle.quantize_act(x, G, 2, np.full(G, 1.7, np.float32))
    wq = synth.random_codes((G, Cg, 1, 1, Cg), 2, gen, signed=True)
    m_out = (np.arange(G, dtype=np.float32) + 1) * np.float32(0.03)
    inv_next = np.full(G, 1.3, np.float32)
    z, codes = oracle.cyclic_shuffle_module(x, q, wq, m_out, inv_next, 1)
    rolled = np.roll(q.reshape(2, 5, 6, G, Cg), 1, axis=3).reshape(q.shape)
    acc = torch_group_conv_f64(rolled, wq, 1, 0)
    y = (acc.astype(np.float32).reshape(2, 5, 6, G, Cg) * m_out[:, None]).reshape(acc.shape)
    assert np.array_equal(z, y + x)
    assert np.array_equal(codes, oracle.quantize_act(z, G, 2, inv_next))


@pytest.mark.parametrize("G", [2, 3, 4, 5])
def test_prop1_G_minus_1_modules_reach_every_group(G):
    """Prop. 1: after G-1 cyclic shuffle modules every group holds information from
    every group.  Only group s of the input is non-zero and all weights are positive:
    after k modules exactly the groups s, s+1, ..., s+k (mod G) are non-zero."""
    Cg = 16
    wq = np.ones((G, Cg, 1, 1, Cg), dtype=np.int8)
    m_out = np.full(G, 0.1, np.float32)  # large enough that a reached group quantises to a non-zero code
    inv = np.ones(G, np.float32)
    for s in range(G):
        x = np.zeros((1, 2, 2, G * Cg), dtype=np.float32)
        x[..., s * Cg:(s + 1) * Cg] = 2.0
        for k in range(1, G):
            q = oracle.quantize_act(x, G, 2, inv)
            x, _ = oracle.cyclic_shuffle_module(x, q, wq, m_out, None, 1)
            live = {g for g in range(G) if np.any(x[..., g * Cg:(g + 1) * Cg] != 0)}
            assert live == {(s + j) % G for j in range(k + 1)}, (G, s, k, live)


# ------------------------------------------- the paper's placement (Sec. 4.3)
@pytest.fixture(scope="module")
def net_paper():
    x, params = synth.resnet18_inputs(2, 32, 32, G, WIDTHS, 10, seed=5, cyclic_modules=True)
    steps = R.calibrate(x, params, G, BITS, placement="paper")
    return x, params, steps, R.forward(x, params, G, BITS, steps, placement="paper")


def test_paper_placement_rederived_with_float64_library(net_paper):
    """The paper's placement re-derived stage by stage from the oracle's own tensors:
    the cyclic shuffle module at each stage's start (Eq. 9-10: torch float64 1x1
    grouped convolution of the group-rolled codes, one fp32 multiply, + X, no ReLU),
    no permutation inside the stage, and the channel shuffle (ShuffleNet's
    reshape/transpose) after the add and ReLU of each stage's last block."""
    x, params, steps, r = net_paper
    f32 = lambda a, m: (a.astype(np.float32).reshape(*a.shape[:-1], G, -1) *
                        np.asarray(m, np.float32)[:, None]).reshape(a.shape)
    X = r["pool"]
    for k in range(1, 5):
        csm = f"s{k}.csm"
        Q = r[csm + ".in_codes"]
        assert np.array_equal(Q, oracle.quantize_act(X, G, BITS, oracle.inv_step(steps[csm + ".in"]))), csm
        swc = steps[csm + ".w"]
        wqc = oracle.quantize_weights(params[csm], BITS, oracle.inv_step(swc))
        rolled_q = np.roll(Q.reshape(*Q.shape[:-1], G, -1), 1, axis=-2).reshape(Q.shape)  # Eq. 8
        accc = torch_group_conv_f64(rolled_q, wqc, 1, 0)
        src = [(g - 1) % G for g in range(G)]
        m_c = (np.float64(swc) * np.float64(np.asarray(steps[csm + ".in"])[src])).astype(np.float32)
        Z = f32(accc, m_c) + X
        assert np.array_equal(Z, r[csm + ".out"]), csm
        for b, stride, down, last in ((f"s{k}b1", 1 if k == 1 else 2, k > 1, False), (f"s{k}b2", 1, False, True)):
            Qb = r[b + ".in_codes"]
            Xb = Z if not last else r[f"s{k}b1.out"]
            assert np.array_equal(Qb, oracle.quantize_act(Xb, G, BITS, oracle.inv_step(steps[b + ".in"]))), b
            sw1, sin, smid = steps[b + ".conv1.w"], steps[b + ".in"], steps[b + ".mid"]
            wq1 = oracle.quantize_weights(params[b + ".conv1"], BITS, oracle.inv_step(sw1))
            acc1 = torch_group_conv_f64(Qb, wq1, stride, 1)
            q1 = np.clip(np.rint(f32(acc1, (np.float64(sw1) * np.float64(sin) / np.float64(smid)).astype(np.float32))),
                         0, 3).astype(np.uint8)
            assert np.array_equal(q1, r[b + ".mid_codes"]), b
            if down:
                swd = steps[b + ".down.w"]
                wqd = oracle.quantize_weights(params[b + ".down"], BITS, oracle.inv_step(swd))
                S = f32(torch_group_conv_f64(Qb, wqd, stride, 0), (np.float64(swd) * np.float64(sin)).astype(np.float32))
            else:
                S = Xb
            sw2 = steps[b + ".conv2.w"]
            wq2 = oracle.quantize_weights(params[b + ".conv2"], BITS, oracle.inv_step(sw2))
            acc2 = torch_group_conv_f64(q1, wq2, 1, 1)
            y = np.maximum(f32(acc2, (np.float64(sw2) * np.float64(smid)).astype(np.float32)) + S, np.float32(0))
            if last:  # ShuffleNet's channel shuffle: [G, Cg] -> [Cg, G]
                y = np.swapaxes(y.reshape(*y.shape[:-1], G, -1), -1, -2).reshape(y.shape)
            assert np.array_equal(y, r[b + ".out"]), b
        X = r[f"s{k}b2.out"]
    ref = X.astype(np.float64).mean(axis=(1, 2)) @ params["fc"].astype(np.float64).T
    assert np.allclose(r["logits"], ref, rtol=1e-4, atol=1e-4)

