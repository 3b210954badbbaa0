"""Pins of the oracle's quantisation-aware training forward / backward (Sec. 3.2
Eq. 2-3, Sec. 5: learned bounds l, u and the straight-through estimator).

The forward is pinned by hand cases and by the structure of its output levels; the
backward by what the straight-through estimator means: with the rounding passed
through, the gradients are those of the unrounded quantiser c * clip((x - l) / (u - l),
0, 1), which central differences in float64 give independently of the oracle's
formulas; and by the invariances of Eq. 2's normalisation ((x - l) / (u - l) does not
change when x, l, u are shifted together or scaled together).
"""
import numpy as np
import pytest

import oracle


def test_forward_hand_cases():
    # l = 0, u = 4, b = 2 (Qp = 3): t = x / 4, x_q = rint(3 t) (half to even)
    x = np.array([[0.5, 1.0, 2.0, 3.5, 4.0, 5.0, -1.0, np.nan, np.inf, -np.inf]], np.float32)
    codes = np.array([0, 1, 2, 3, 3, 3, 0, 0, 3, 0], np.float32)  # 0.375 -> 0, 0.75 -> 1, 1.5 -> 2, 2.625 -> 3
    a = oracle.fake_quant_forward(x, 1, 2, 0, [0.0], [4.0])
    np.testing.assert_array_equal(a[0], (codes / np.float32(3)).astype(np.float32))
    w = oracle.fake_quant_forward(x, 1, 2, 1, [0.0], [4.0])
    np.testing.assert_array_equal(w[0], (np.float32(2) * (codes / np.float32(3) - np.float32(0.5))).astype(np.float32))
    # a non-zero lower bound shifts the grid: l = -2, u = 2, b = 1 (Qp = 1): x_q = rint((x + 2) / 4)
    x2 = np.array([[-3.0, -2.0, -0.5, 0.0, 0.5, 2.0]], np.float32)
    a2 = oracle.fake_quant_forward(x2, 1, 1, 0, [-2.0], [2.0])
    np.testing.assert_array_equal(a2[0], [0, 0, 0, 0, 1, 1])  # t = 0.375 -> 0, t = 0.5 -> 0 (even), 0.625 -> 1


def test_forward_levels_monotone_and_groups():
    rng = np.random.default_rng(3)
    G, Cg, bits = 3, 8, 3
    l = np.array([-0.5, 0.0, 0.25], np.float32)
    u = np.array([1.5, 2.0, 0.75], np.float32)
    x = rng.normal(0.5, 1.0, size=(40, G * Cg)).astype(np.float32)
    qp = (1 << bits) - 1
    for kind in (0, 1):
        y = oracle.fake_quant_forward(x, G, bits, kind, l, u)
        lev = (y + 1.0) / 2.0 if kind else y
        k = np.rint(lev.astype(np.float64) * qp)
        assert np.all(np.abs(lev * qp - k) < 1e-5) and k.min() >= 0 and k.max() <= qp
        # per group: monotone non-decreasing in x, saturating at the bounds
        for g in range(G):
            xs, ys = x[:, g * Cg:(g + 1) * Cg].ravel(), y[:, g * Cg:(g + 1) * Cg].ravel()
            order = np.argsort(xs, kind="stable")
            assert np.all(np.diff(ys[order]) >= 0)
            lo, hi = (-1.0, 1.0) if kind else (0.0, 1.0)
            assert np.all(ys[xs <= l[g]] == lo) and np.all(ys[xs >= u[g]] == hi)


def _unrounded_loss(x, dy, G, kind, l, u):
    """sum(dy * c * clip((x - l) / (u - l), 0, 1)) in float64: the quantiser with
    the rounding taken out, which the straight-through estimator differentiates."""
    c = 2.0 if kind else 1.0
    C = x.shape[-1]
    Cg = C // G
    tot = 0.0
    for g in range(G):
        xs = x[..., g * Cg:(g + 1) * Cg].astype(np.float64)
        t = np.clip((xs - l[g]) / (u[g] - l[g]), 0.0, 1.0)
        tot += float(np.sum(dy[..., g * Cg:(g + 1) * Cg].astype(np.float64) * c * t))
    return tot


@pytest.mark.parametrize("kind", [0, 1])
def test_backward_matches_central_differences(kind):
    rng = np.random.default_rng(11 + kind)
    G, Cg, bits = 2, 16, 2
    l = np.array([-0.25, 0.5], np.float64)
    u = np.array([1.75, 1.5], np.float64)
    x = rng.uniform(-1.0, 2.5, size=(6, G * Cg)).astype(np.float32)
    # keep every element away from the clip corners, where the derivative jumps
    for g in range(G):
        sl = x[:, g * Cg:(g + 1) * Cg]
        t = (sl.astype(np.float64) - l[g]) / (u[g] - l[g])
        sl[np.abs(t) < 1e-2] += np.float32(0.05)
        sl[np.abs(t - 1.0) < 1e-2] += np.float32(0.05)
    dy = rng.normal(size=x.shape).astype(np.float32)
    dx, dl, du = oracle.fake_quant_backward(x, dy, G, bits, kind, l.astype(np.float32), u.astype(np.float32))
    h = 1e-6
    for g in range(G):
        lp, lm = l.copy(), l.copy()
        lp[g] += h
        lm[g] -= h
        num_dl = (_unrounded_loss(x, dy, G, kind, lp, u) - _unrounded_loss(x, dy, G, kind, lm, u)) / (2 * h)
        up, um = u.copy(), u.copy()
        up[g] += h
        um[g] -= h
        num_du = (_unrounded_loss(x, dy, G, kind, l, up) - _unrounded_loss(x, dy, G, kind, l, um)) / (2 * h)
        assert abs(dl[g] - num_dl) <= 1e-6 * (1 + abs(num_dl))
        assert abs(du[g] - num_du) <= 1e-6 * (1 + abs(num_du))
    # dx: the derivative of the unrounded map per element (c / (u - l) inside, 0 outside)
    c = 2.0 if kind else 1.0
    for g in range(G):
        xs = x[:, g * Cg:(g + 1) * Cg].astype(np.float64)
        t = (xs - l[g]) / (u[g] - l[g])
        ref = np.where((t > 0) & (t < 1), dy[:, g * Cg:(g + 1) * Cg] * c / (u[g] - l[g]), 0.0)
        np.testing.assert_allclose(dx[:, g * Cg:(g + 1) * Cg], ref, rtol=2e-7, atol=0)


@pytest.mark.parametrize("kind", [0, 1])
def test_backward_shift_and_scale_invariance(kind):
    """(x - l) / (u - l) is unchanged by x, l, u -> x + d, l + d, u + d and by
    x, l, u -> a x, a l, a u, so sum(dx) + dl + du = 0 and
    sum(x dx) + l dl + u du = 0 per group."""
    rng = np.random.default_rng(5 + kind)
    G, Cg = 4, 8
    l = np.array([0.0, -1.0, 0.5, 2.0], np.float32)
    u = np.array([1.0, 1.0, 4.5, 2.5], np.float32)
    x = rng.uniform(-2.0, 5.0, size=(50, G * Cg)).astype(np.float32)
    dy = rng.normal(size=x.shape).astype(np.float32)
    dx, dl, du = oracle.fake_quant_backward(x, dy, G, 3, kind, l, u)
    for g in range(G):
        d = dx[:, g * Cg:(g + 1) * Cg].astype(np.float64)
        xs = x[:, g * Cg:(g + 1) * Cg].astype(np.float64)
        scale = np.sum(np.abs(d)) + abs(dl[g]) + abs(du[g])
        assert abs(np.sum(d) + dl[g] + du[g]) <= 1e-6 * scale
        scale2 = np.sum(np.abs(xs * d)) + abs(l[g] * dl[g]) + abs(u[g] * du[g])
        assert abs(np.sum(xs * d) + float(l[g]) * dl[g] + float(u[g]) * du[g]) <= 1e-6 * scale2


def test_backward_hand_case_and_outside_zero():
    x = np.array([[0.5, 1.0, 2.0, 3.5, 4.0, 5.0, -1.0, np.nan]], np.float32)
    dy = np.ones_like(x)
    dx, dl, du = oracle.fake_quant_backward(x, dy, 1, 2, 0, [0.0], [4.0])
    np.testing.assert_array_equal(dx[0], [0.25, 0.25, 0.25, 0.25, 0, 0, 0, 0])  # t = 1 is outside (strict)
    assert dl[0] == (0.5 + 1 + 2 + 3.5 - 4 * 4) / 16.0   # sum(x - u) / r^2 over the four inside elements
    assert du[0] == -(0.5 + 1 + 2 + 3.5) / 16.0


def test_inference_codes_with_learned_bounds():
    """Eq. 2 with l, u at inference: hand cases (a negative lower bound shifts code 0
    below x = 0), and the codes equal the training forward's x_q (x_hat * (2^b - 1))."""
    x = np.array([[-3.0, -2.0, -1.0, 0.0, 0.5, 1.0, 2.0, 3.0, np.nan]], np.float32)
    # l = -2, u = 2, b = 2: t = (x + 2) / 4, x_q = rint(3 t): 0, 0, 0.75 -> 1, 1.5 -> 2, 1.875 -> 2, 2.25 -> 2, 3, 3, 0
    np.testing.assert_array_equal(oracle.quantize_act_lu(x, 1, 2, [-2.0], [2.0])[0], [0, 0, 1, 2, 2, 2, 3, 3, 0])
    rng = np.random.default_rng(9)
    G, Cg = 3, 16
    l = np.array([-0.75, 0.0, 0.5], np.float32)
    u = np.array([1.25, 3.0, 0.625], np.float32)
    xs = rng.uniform(-1.5, 3.5, size=(64, G * Cg)).astype(np.float32)
    for bits in (1, 2, 3, 4, 8):
        q = oracle.quantize_act_lu(xs, G, bits, l, u)
        xh = oracle.fake_quant_forward(xs, G, bits, 0, l, u)
        qp = (1 << bits) - 1
        assert q.max() <= qp
        np.testing.assert_array_equal(np.rint(xh.astype(np.float64) * qp).astype(np.uint8), q)
