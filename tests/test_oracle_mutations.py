"""Planted mistakes in the oracle are caught by its pins (no GPU).

Each case rebuilds a copy of the oracle's C source with one plausible mistake (a wrong
index, a dropped term, a wrong rounding or sign) in a temporary directory and checks that
at least one pin fails on it.  This shows the pins constrain every part of the oracle.
"""
import os
import subprocess

import numpy as np
import pytest

import oracle
from paper_2208_01944_gb300 import synth

from test_oracle_pins import torch_group_conv_f64

SRC = os.path.join(os.path.dirname(oracle.__file__), "palquant_oracle.c")

MUTATIONS = {
    # kh and kw swapped in the weight index
    "weight_tap_transposed": ("* sh->kh + r) * sh->kw + s)", "* sh->kh + s) * sh->kw + r)"),
    # padding not subtracted from the input row
    "pad_dropped_rows": ("oh * sh->stride - sh->pad + r", "oh * sh->stride + r"),
    # group offset of the input channels dropped
    "group_offset_dropped": ("iw) * Cin + (int64_t)g * sh->Cin_g", "iw) * Cin"),
    # weights read as unsigned bytes
    "weight_sign_lost": ("(int64_t)wp[ci]", "(int64_t)(uint8_t)wp[ci]"),
    # round half away from zero instead of half to even
    "round_half_away": ("float r = rintf(t);               /* round half to even */",
                        "float r = roundf(t);"),
    # clamp one level too high
    "clamp_off_by_one": ("r = fminf(r, (float)qmax);\n    return", "r = fminf(r, (float)(qmax + 1));\n    return"),
    # permutation in the wrong direction
    "perm_direction": ("dst[g] = (int32_t)((((g + shift) % G) + G) % G);", "dst[g] = (int32_t)((((g - shift) % G) + G) % G);"),
    # requantisation from the rescaled output instead of the accumulator
    "requant_from_y": ("float t = (shortcut ? y : af) * m_req[g];", "float t = y * m_req[g];"),
    # the shortcut added after the ReLU
    "shortcut_after_relu": ("if (shortcut) y = y + shortcut[p * C + src];\n                if (relu) y = fmaxf(y, 0.0f);",
                            "if (relu) y = fmaxf(y, 0.0f);\n                if (shortcut) y = y + shortcut[p * C + src];"),
    # channel shuffle as the identity instead of ShuffleNet's transpose
    "channel_shuffle_identity": ("if (kind == 2) return (int64_t)co * G + g;",
                                 "if (kind == 2) return (int64_t)g * Cout_g + co;"),
    # odd weight levels without the factor 2
    "odd_levels_unscaled": ("wq[g * per_group + i] = (int8_t)(2 * (int)r - qp);",
                            "wq[g * per_group + i] = (int8_t)((int)r - qp);"),
    # the clip range shifted by u twice
    "odd_levels_shift": ("float t = (w[g * per_group + i] + u[g]) * k;", "float t = (w[g * per_group + i] + 2.0f * u[g]) * k;"),
    # quantisation-aware training: weights de-quantised without the factor 2
    "qat_weight_factor": ("xhat[i] = kind ? 2.0f * (v - 0.5f) : v;", "xhat[i] = kind ? (v - 0.5f) : v;"),
    # rounding half up instead of half to even
    "qat_round_half_up": ("float xq = rintf(xn * qp);", "float xq = floorf(xn * qp + 0.5f);"),
    # the straight-through gradient also at the clip bounds
    "qat_inside_inclusive": ("if (t > 0.0f && t < 1.0f) {", "if (t >= 0.0f && t <= 1.0f) {"),
    # the gradient of u with the wrong sign
    "qat_du_sign": ("du[g] = -c / (rd * rd) * sb;", "du[g] = c / (rd * rd) * sb;"),
    # the gradient of l measured from the wrong bound
    "qat_dl_bound": ("sa += (double)dy[i] * ((double)x[i] - (double)u[g]);",
                     "sa += (double)dy[i] * ((double)x[i] - (double)l[g]);"),
    # the input gradient without the de-quantisation factor
    "qat_dx_factor": ("const float k = (float)c * inv_r;", "const float k = inv_r;"),
    # step from the mean without the factor 2
    "act_step_factor": ("s_out[g] = (float)(2.0 * mean / sqrt(qp));\n    }\n}\n\nvoid oracle_weight_step",
                        "s_out[g] = (float)(mean / sqrt(qp));\n    }\n}\n\nvoid oracle_weight_step"),
}


def _pins_pass(L) -> bool:
    """Run a compact set of the pins against an oracle build; True if all hold."""
    import math

    try:
        # Eq. 2 hand cases
        x = np.array([0.5, 1.5, 2.5, 3.7, -0.3, 1e6], dtype=np.float32).reshape(1, 1, 1, 6)
        if list(oracle.quantize_act(x, 1, 2, [1.0], L=L).ravel()) != [0, 2, 2, 3, 0, 3]:
            return False
        # library convolution on codes
        for (N, H, W, G, Ci, Co, k, s, p) in [(2, 6, 5, 2, 4, 3, 3, 1, 1), (1, 7, 7, 3, 2, 5, 3, 2, 1)]:
            gen = synth.generator(7)
            q = synth.random_codes((N, H, W, G * Ci), 2, gen)
            wq = synth.random_codes((G, Co, k, k, Ci), 2, gen, signed=True)
            if not np.array_equal(oracle.group_conv(q, wq, s, p, L=L).astype(np.float64), torch_group_conv_f64(q, wq, s, p)):
                return False
        # Eq. 6 two-line notation
        if list(oracle.group_perm(4, 1, 1, L=L)) != [1, 2, 3, 0]:
            return False
        # epilogue hand cases
        acc = np.array([[10, -4, 7, 100]], dtype=np.int64)
        a, y, qq = oracle.epilogue(acc, 2, [0.25, 0.5], [0.125, 0.0625], kind=1, shift=1, relu=True, L=L)
        if list(y[0]) != [3.5, 50.0, 2.5, 0.0] or list(qq[0]) != [0, 3, 1, 0]:
            return False
        a, y, qq = oracle.epilogue(np.array([[4, -8]], dtype=np.int64), 1, [0.25], [2.0], kind=0,
                                   shortcut=np.array([[0.5, 1.0]], dtype=np.float32), relu=True, L=L)
        if list(y[0]) != [1.5, 0.0] or list(qq[0]) != [3, 0]:
            return False
        # the paper's odd weight levels
        wo = np.array([-2.0, -0.5, 0.0, 0.5, 1.0], np.float32).reshape(1, 1, 1, 1, -1)
        if list(oracle.quantize_weights_odd(wo, 2, [1.0], L=L).ravel()) != [-3, -1, 1, 1, 3]:
            return False
        # channel shuffle: ShuffleNet's reshape / transpose
        acc = np.arange(12, dtype=np.int64).reshape(1, 12)
        _, y2, _ = oracle.epilogue(acc, 3, [1.0, 1.0, 1.0], None, kind=2, relu=False, L=L)
        if list(y2[0]) != [float(v) for v in np.arange(12).reshape(3, 4).T.ravel()]:
            return False
        # quantisation-aware training: forward hand cases (both kinds, a shifted grid)
        xq = np.array([[0.5, 1.0, 2.0, 3.5, 4.0, 5.0, -1.0]], np.float32)
        third = np.float32(1) / np.float32(3)
        if list(oracle.fake_quant_forward(xq, 1, 2, 0, [0.0], [4.0], L=L)[0]) != \
                [0.0, third, np.float32(2) / np.float32(3), 1.0, 1.0, 1.0, 0.0]:
            return False
        if list(oracle.fake_quant_forward(xq, 1, 2, 1, [0.0], [4.0], L=L)[0][[0, 3, 6]]) != [-1.0, 1.0, -1.0]:
            return False
        if list(oracle.fake_quant_forward(np.array([[-0.5, 0.0, 0.5]], np.float32), 1, 1, 0, [-2.0], [2.0],
                                          L=L)[0]) != [0.0, 0.0, 1.0]:
            return False
        # backward hand cases (the bound t = 1 is outside; weights carry the factor 2)
        dx, dl, du = oracle.fake_quant_backward(xq, np.ones_like(xq), 1, 2, 0, [0.0], [4.0], L=L)
        if list(dx[0]) != [0.25, 0.25, 0.25, 0.25, 0.0, 0.0, 0.0] or dl[0] != -9.0 / 16 or du[0] != -7.0 / 16:
            return False
        dx, dl, du = oracle.fake_quant_backward(xq, np.ones_like(xq), 1, 2, 1, [0.0], [4.0], L=L)
        if list(dx[0][:4]) != [0.5] * 4 or dl[0] != -18.0 / 16 or du[0] != -14.0 / 16:
            return False
        # constant-tensor step closed form
        c = np.full((1, 2, 2, 4), 1.5, dtype=np.float32)
        if not np.allclose(oracle.act_step(c, 2, 2, L=L), 2 * 1.5 / math.sqrt(3.0), rtol=1e-7):
            return False
        return True
    except ValueError:
        return False


def test_unmutated_oracle_passes():
    assert _pins_pass(oracle.lib())


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_mutation_is_caught(name, tmp_path):
    old, new = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique in the oracle source"
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src.replace(old, new))
    so = str(tmp_path / "libmutant.so")
    subprocess.check_call(["gcc", *oracle.CFLAGS, "-o", so, str(mutated), "-lm"])
    assert not _pins_pass(oracle.load_variant(so)), f"pins did not catch mutation {name}"
